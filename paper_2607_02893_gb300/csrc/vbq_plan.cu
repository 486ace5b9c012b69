// vbq_plan.cu — host-side choice of the kernel for a small batch (2..4 rows).
#include "vbq_kernels.h"

namespace vbq {

// Batches of 2..GEMV1_MAX_B rows run on the table kernel (two rows per launch,
// the two-vector variant sharing every lookup address and masked code between
// its rows, plus a one-vector launch for an odd count) or on the tensor cores,
// whichever the layout's width mix makes cheaper. Cost per million groups of
// each width (1, 2, 4, 8 bits), in microseconds, measured on a GB300 on
// 16384 x 16384 matrices of one width: one row on the table kernel, two rows
// on it, and up to 8 rows on the tensor cores. The tensor cores take items in
// tiles of 16 from each (column, width) bucket of a unit, so a bucket leaves
// about 6 item slots of its last tile idle (fitted to the mixed distribution:
// 16384 x 16384 at 8 rows, 80 us measured, 82 us modelled).
constexpr double COST_ONE[4] = {5.33, 7.02, 9.98, 14.0};
constexpr double COST_PAIR[4] = {8.62, 11.8, 16.3, 27.5};
constexpr double COST_MMA[4] = {14.7, 17.5, 17.8, 24.5};
constexpr double MMA_IDLE_PER_BUCKET = 6.0;

bool tables_for_batch(const LayoutView& L, int B) {
    const double buckets = (double)L.units * L.C;
    double tab = 0.0, mma = 0.0;
    for (int w = 0; w < 4; ++w) {
        if (L.items[w] == 0) continue;
        tab += (double)L.items[w] * ((B / 2) * COST_PAIR[w] + (B % 2) * COST_ONE[w]);
        mma += ((double)L.items[w] + MMA_IDLE_PER_BUCKET * buckets) * COST_MMA[w];
    }
    return tab <= mma;
}

}  // namespace vbq
