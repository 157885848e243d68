// Instantiation unit of the search leaf kernel (see search_kernels.cuh):
// Eager 1F1B (fast path and level programs), S = 13..14.
#include "search_kernels.cuh"

namespace pos {

pos_status launch_leaf_eager_13_14(int S, int path, const LeafParams &p, int grid,
                                   cudaStream_t s) {
    switch (S) {
        case 13:
            return launch_leaf_s<13, true>(path, p, grid, s);
        case 14:
            return launch_leaf_s<14, true>(path, p, grid, s);
        default:
            return fail(POS_EINVAL, "stage count outside this unit");
    }
}

}  // namespace pos
