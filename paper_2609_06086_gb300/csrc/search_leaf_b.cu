// Instantiation unit of the search leaf kernel (see search_kernels.cuh).
#include "search_kernels.cuh"

namespace pos {

pos_status launch_leaf_7_10(int S, bool fast, const LeafParams &p, int grid, cudaStream_t s) {
    switch (S) {
        case 7:
            return fast ? launch_leaf_t<7, kPathFast>(p, grid, s)
                        : launch_leaf_t<7, kPathGeneric>(p, grid, s);
        case 8:
            return fast ? launch_leaf_t<8, kPathFast>(p, grid, s)
                        : launch_leaf_t<8, kPathGeneric>(p, grid, s);
        case 9:
            return fast ? launch_leaf_t<9, kPathFast>(p, grid, s)
                        : launch_leaf_t<9, kPathGeneric>(p, grid, s);
        case 10:
            return fast ? launch_leaf_t<10, kPathFast>(p, grid, s)
                        : launch_leaf_t<10, kPathGeneric>(p, grid, s);
        default:
            return fail(POS_EINVAL, "stage count outside this unit");
    }
}

}  // namespace pos
