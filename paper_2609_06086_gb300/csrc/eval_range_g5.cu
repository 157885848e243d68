// Instantiation unit of the eval kernel family (see eval_kernel.cuh).
#include "eval_kernel.cuh"

namespace pos {

pos_status eval_generic_16_16(const EvalParams &p, cudaStream_t s) {
    return launch_eval_range<16, 16, kPathGeneric, 2>(p, s);
}

}  // namespace pos
