// Instantiation unit of the search leaf kernel (see search_kernels.cuh):
// 1F1B (fast and short paths), S = 15..15.
#include "search_kernels.cuh"

namespace pos {

pos_status launch_leaf_1f1b_15_15(int S, int path, const LeafParams &p, int grid,
                                   cudaStream_t s) {
    switch (S) {
        case 15:
            return launch_leaf_s<15, false>(path, p, grid, s);
        default:
            return fail(POS_EINVAL, "stage count outside this unit");
    }
}

}  // namespace pos
