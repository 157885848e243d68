// Instantiation unit of the eval kernel family (see eval_kernel.cuh).
#include "eval_kernel.cuh"

namespace pos {

pos_status eval_fast_13_16(const EvalParams &p, cudaStream_t s) {
    return launch_eval_range<13, 16, kPathFast, 3>(p, s);
}

}  // namespace pos
