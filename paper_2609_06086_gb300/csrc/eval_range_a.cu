// Instantiation unit of the eval kernel family (see eval_kernel.cuh).
#include "eval_kernel.cuh"

namespace pos {

pos_status eval_fast_1_4(const EvalParams &p, cudaStream_t s) {
    return launch_eval_range<1, 4, kPathFast, 6>(p, s);
}

pos_status eval_fast_5_8(const EvalParams &p, cudaStream_t s) {
    return launch_eval_range<5, 8, kPathFast, 4>(p, s);
}

}  // namespace pos
