// Instantiation unit of the eval kernel family (see eval_kernel.cuh):
// Eager 1F1B with M < 2S-1 (level programs).
#include "eval_kernel.cuh"

namespace pos {

pos_status eval_eager_short_2_8(const EvalParams &p, cudaStream_t s) {
    return launch_eval_range<2, 8, kPathEagerShort, 4>(p, s);
}

pos_status eval_eager_short_9_12(const EvalParams &p, cudaStream_t s) {
    return launch_eval_range<9, 12, kPathEagerShort, 2>(p, s);
}

pos_status eval_eager_short_13_16(const EvalParams &p, cudaStream_t s) {
    return launch_eval_range<13, 16, kPathEagerShort, 2>(p, s);
}

}  // namespace pos
