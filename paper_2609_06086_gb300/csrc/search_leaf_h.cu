// Instantiation unit of the search leaf kernel (see search_kernels.cuh):
// Eager 1F1B (fast path and level programs), S = 9..12.
#include "search_kernels.cuh"

namespace pos {

pos_status launch_leaf_eager_9_12(int S, int path, const LeafParams &p, int grid,
                                   cudaStream_t s) {
    switch (S) {
        case 9:
            return launch_leaf_s<9, true>(path, p, grid, s);
        case 10:
            return launch_leaf_s<10, true>(path, p, grid, s);
        case 11:
            return launch_leaf_s<11, true>(path, p, grid, s);
        case 12:
            return launch_leaf_s<12, true>(path, p, grid, s);
        default:
            return fail(POS_EINVAL, "stage count outside this unit");
    }
}

}  // namespace pos
