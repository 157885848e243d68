// Instantiation unit of the search leaf kernel (see search_kernels.cuh).
#include "search_kernels.cuh"

namespace pos {

pos_status launch_leaf_15_15(int S, bool fast, const LeafParams &p, int grid, cudaStream_t s) {
    switch (S) {
        case 15:
            return fast ? launch_leaf_t<15, kPathFast>(p, grid, s)
                        : launch_leaf_t<15, kPathGeneric>(p, grid, s);
        default:
            return fail(POS_EINVAL, "stage count outside this unit");
    }
}

}  // namespace pos
