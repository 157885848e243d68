// Instantiation unit of the eval kernel family (see eval_kernel.cuh).
#include "eval_kernel.cuh"

namespace pos {

pos_status eval_generic_2_8(const EvalParams &p, cudaStream_t s) {
    return launch_eval_range<2, 8, kPathGeneric, 4>(p, s);
}

}  // namespace pos
