// Instantiation unit of the search leaf kernel (see search_kernels.cuh):
// 1F1B (fast and short paths), S = 1..6.
#include "search_kernels.cuh"

namespace pos {

pos_status launch_leaf_1f1b_1_6(int S, int path, const LeafParams &p, int grid,
                                   cudaStream_t s) {
    switch (S) {
        case 1:
            return launch_leaf_s<1, false>(path, p, grid, s);
        case 2:
            return launch_leaf_s<2, false>(path, p, grid, s);
        case 3:
            return launch_leaf_s<3, false>(path, p, grid, s);
        case 4:
            return launch_leaf_s<4, false>(path, p, grid, s);
        case 5:
            return launch_leaf_s<5, false>(path, p, grid, s);
        case 6:
            return launch_leaf_s<6, false>(path, p, grid, s);
        default:
            return fail(POS_EINVAL, "stage count outside this unit");
    }
}

}  // namespace pos
