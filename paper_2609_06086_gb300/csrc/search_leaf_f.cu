// Instantiation unit of the search leaf kernel (see search_kernels.cuh):
// 1F1B (fast and short paths), S = 16..16.
#include "search_kernels.cuh"

namespace pos {

pos_status launch_leaf_1f1b_16_16(int S, int path, const LeafParams &p, int grid,
                                   cudaStream_t s) {
    switch (S) {
        case 16:
            return launch_leaf_s<16, false>(path, p, grid, s);
        default:
            return fail(POS_EINVAL, "stage count outside this unit");
    }
}

}  // namespace pos
