// Instantiation unit of the search leaf kernel (see search_kernels.cuh).
#include "search_kernels.cuh"

namespace pos {

pos_status launch_leaf_1_6(int S, bool fast, const LeafParams &p, int grid, cudaStream_t s) {
    switch (S) {
        case 1:
            return fast ? launch_leaf_t<1, kPathFast>(p, grid, s)
                        : launch_leaf_t<1, kPathFast>(p, grid, s);
        case 2:
            return fast ? launch_leaf_t<2, kPathFast>(p, grid, s)
                        : launch_leaf_t<2, kPathGeneric>(p, grid, s);
        case 3:
            return fast ? launch_leaf_t<3, kPathFast>(p, grid, s)
                        : launch_leaf_t<3, kPathGeneric>(p, grid, s);
        case 4:
            return fast ? launch_leaf_t<4, kPathFast>(p, grid, s)
                        : launch_leaf_t<4, kPathGeneric>(p, grid, s);
        case 5:
            return fast ? launch_leaf_t<5, kPathFast>(p, grid, s)
                        : launch_leaf_t<5, kPathGeneric>(p, grid, s);
        case 6:
            return fast ? launch_leaf_t<6, kPathFast>(p, grid, s)
                        : launch_leaf_t<6, kPathGeneric>(p, grid, s);
        default:
            return fail(POS_EINVAL, "stage count outside this unit");
    }
}

}  // namespace pos
