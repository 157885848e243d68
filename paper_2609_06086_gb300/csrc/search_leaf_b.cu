// Instantiation unit of the search leaf kernel (see search_kernels.cuh):
// 1F1B (fast and short paths), S = 7..10.
#include "search_kernels.cuh"

namespace pos {

pos_status launch_leaf_1f1b_7_10(int S, int path, const LeafParams &p, int grid,
                                   cudaStream_t s) {
    switch (S) {
        case 7:
            return launch_leaf_s<7, false>(path, p, grid, s);
        case 8:
            return launch_leaf_s<8, false>(path, p, grid, s);
        case 9:
            return launch_leaf_s<9, false>(path, p, grid, s);
        case 10:
            return launch_leaf_s<10, false>(path, p, grid, s);
        default:
            return fail(POS_EINVAL, "stage count outside this unit");
    }
}

}  // namespace pos
