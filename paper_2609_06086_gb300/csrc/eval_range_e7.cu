// Instantiation unit of the eval kernel family (see eval_kernel.cuh):
// Eager 1F1B with M < 2S-1 (unrolled per (S, M)), S = 13.
#include "eval_kernel.cuh"

namespace pos {

pos_status eval_eager_short_13_13(const EvalParams &p, cudaStream_t s) {
    return launch_eval_range<13, 13, kPathEagerUnrolled, 2>(p, s);
}

}  // namespace pos
