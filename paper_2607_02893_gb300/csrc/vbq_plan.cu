// vbq_plan.cu — host-side choice of the kernel for a small batch (2..4 rows).
#include "vbq_kernels.h"

namespace vbq {

// Batches of 2..GEMV1_MAX_B rows run on the table kernel (two rows per launch,
// the two-vector variant sharing every lookup address and masked code between
// its rows, plus a one-vector launch for an odd count) or on the tensor cores,
// whichever the layout's width mix makes cheaper. Cost per million groups of
// each width (1, 2, 4, 8 bits), in microseconds, measured on a GB300 on
// 16384 x 16384: one row on the table kernel, two rows on it, and up to 8 rows
// on the tensor cores. Tables win for 1- and 2-bit groups, the tensor cores for
// 4- and 8-bit ones from 3 rows on.
constexpr double COST_ONE[4] = {5.33, 7.02, 9.98, 14.0};
constexpr double COST_PAIR[4] = {8.62, 11.8, 16.3, 27.5};
constexpr double COST_MMA[4] = {18.7, 20.3, 20.3, 27.0};

bool tables_for_batch(const LayoutView& L, int B) {
    double tab = 0.0, mma = 0.0;
    for (int w = 0; w < 4; ++w) {
        tab += (double)L.items[w] * ((B / 2) * COST_PAIR[w] + (B % 2) * COST_ONE[w]);
        mma += (double)L.items[w] * COST_MMA[w];
    }
    return tab <= mma;
}

}  // namespace vbq
