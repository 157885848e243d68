// Instantiation unit of the search leaf kernel (see search_kernels.cuh):
// 1F1B (fast and short paths), S = 11..12.
#include "search_kernels.cuh"

namespace pos {

pos_status launch_leaf_1f1b_11_12(int S, int path, const LeafParams &p, int grid,
                                   cudaStream_t s) {
    switch (S) {
        case 11:
            return launch_leaf_s<11, false>(path, p, grid, s);
        case 12:
            return launch_leaf_s<12, false>(path, p, grid, s);
        default:
            return fail(POS_EINVAL, "stage count outside this unit");
    }
}

}  // namespace pos
