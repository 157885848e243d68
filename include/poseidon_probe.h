/*
 * poseidon_probe.h -- measurement tooling shipped beside libposeidon.so in
 * libposeidon_probe.so; not part of the library's contract and with no
 * counterpart in the paper.
 */
#ifndef POSEIDON_PROBE_H
#define POSEIDON_PROBE_H
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/*
 * Runs a kernel made of the makespan kernels' relaxation,
 * max(pred + edge, clock) + weight, in independent chains on every SM of
 * the current device, twice, and reports the second run: *ops = int32
 * operations executed (3 per relaxation), *ms = its duration (CUDA events
 * on `stream`, a cudaStream_t; NULL = legacy default stream).  ops / ms is
 * the measured INT32 rate the ALU-bound kernels are compared with.
 * Synchronises the stream; takes a 4-byte stream-ordered allocation.
 * Returns 0, or the cudaError_t of the failing call (cudaErrorInvalidValue
 * for a NULL output pointer).
 */
int poseidon_probe_int32(void *stream, int64_t *ops, double *ms);

#ifdef __cplusplus
}
#endif
#endif /* POSEIDON_PROBE_H */
