// Instantiation unit of the eval kernel family (see eval_kernel.cuh).
#include "eval_kernel.cuh"

namespace pos {

pos_status eval_fast_9_12(const EvalParams &p, cudaStream_t s) {
    return launch_eval_range<9, 12, kPathFast, 3>(p, s);
}

}  // namespace pos
