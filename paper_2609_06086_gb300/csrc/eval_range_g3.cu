// Instantiation unit of the eval kernel family (see eval_kernel.cuh).
#include "eval_kernel.cuh"

namespace pos {

pos_status eval_generic_13_14(const EvalParams &p, cudaStream_t s) {
    return launch_eval_range<13, 14, kPathGeneric, 3>(p, s);
}

}  // namespace pos
