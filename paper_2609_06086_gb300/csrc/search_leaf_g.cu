// Instantiation unit of the search leaf kernel (see search_kernels.cuh):
// Eager 1F1B (fast path and level programs), S = 1..8.
#include "search_kernels.cuh"

namespace pos {

pos_status launch_leaf_eager_1_8(int S, int path, const LeafParams &p, int grid,
                                   cudaStream_t s) {
    switch (S) {
        case 1:
            return launch_leaf_s<1, true>(path, p, grid, s);
        case 2:
            return launch_leaf_s<2, true>(path, p, grid, s);
        case 3:
            return launch_leaf_s<3, true>(path, p, grid, s);
        case 4:
            return launch_leaf_s<4, true>(path, p, grid, s);
        case 5:
            return launch_leaf_s<5, true>(path, p, grid, s);
        case 6:
            return launch_leaf_s<6, true>(path, p, grid, s);
        case 7:
            return launch_leaf_s<7, true>(path, p, grid, s);
        case 8:
            return launch_leaf_s<8, true>(path, p, grid, s);
        default:
            return fail(POS_EINVAL, "stage count outside this unit");
    }
}

}  // namespace pos
