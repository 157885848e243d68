// Instantiation unit of the Interleaved 1F1B eval kernels (interleaved.cuh):
// pairs (N, V) by index in interleaved_order.h.
#include "interleaved.cuh"

namespace pos {

pos_status eval_il_0_11(const EvalParams &p, cudaStream_t s) {
    return launch_il_range<0, 11, 4>(p, s);
}

}  // namespace pos
