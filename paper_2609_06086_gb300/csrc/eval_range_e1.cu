// Instantiation unit of the eval kernel family (see eval_kernel.cuh):
// Eager 1F1B with M >= 2S-1.
#include "eval_kernel.cuh"

namespace pos {

pos_status eval_eager_1_6(const EvalParams &p, cudaStream_t s) {
    return launch_eval_range<1, 6, kPathEager, 4>(p, s);
}

pos_status eval_eager_7_10(const EvalParams &p, cudaStream_t s) {
    return launch_eval_range<7, 10, kPathEager, 3>(p, s);
}

}  // namespace pos
