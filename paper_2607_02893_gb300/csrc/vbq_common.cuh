// vbq_common.cuh — device layout of a packed VBQ matrix, shared by the CUDA
// kernels of this library (pack, dequant, GEMV).
//
// Layout (chosen for GB300; the paper fixes only "64*b bits per group on byte
// boundaries", §1 and §6):
//
//   * Rows are cut into row blocks of RB = 128 rows; the K/64 group columns
//     into slabs of C columns (C in 4..32, chosen per matrix at pack time so
//     that there are enough blocks for every SM). A (row block, slab) pair is
//     a "unit", numbered u = rb * S + s with S = slabs per row.
//   * For each unit a width map holds a 2-bit width code per (column, row):
//     code w means b = 1 << w. Column c of unit u occupies 8 32-bit words
//     map[(u*C + c)*8 + j], word j holding rows 16j .. 16j+15 (2 bits each,
//     row r at bits 2*(r%16)).
//   * Each width b has its own item stream. An item is one group (64 codes)
//     of width b; within a unit the items of width b are ordered by
//     (column, row), and units follow each other in unit order. Item i of
//     width index w starts at byte 8*b*i of payload[w] and its FP16 scale is
//     scales[w][i]. ustart[u*4 + w] is the index of the unit's first item of
//     width index w (ustart has units+1 rows; the last row holds the totals).
//   * Inside an item, code j of the group (column 64*col + j) occupies bits
//     [j*b, j*b + b) of the item's little-endian bytes.
//
// The map gives, per unit, every item's (column, row) without storing row or
// column indices per item: kernels rebuild the item list of a unit in shared
// memory from the map (build_item_list below).
#pragma once

#include <cstdint>
#include <cuda_runtime.h>
#include <cuda_fp16.h>

namespace vbq {

constexpr int RB = 128;          // rows per row block
constexpr int GROUP = 64;        // weights per group (§3.1)
constexpr int MAX_C = 32;        // max group columns per slab
constexpr int MAP_WORDS = RB / 16;   // map words per column
constexpr int MAX_BATCH = 16;

struct LayoutView {
    const uint32_t* map;
    const uint32_t* ustart;
    const uint8_t* payload[4];
    const uint16_t* scales[4];
    int64_t N, K;
    int G, C, S, nrb, units;
};

__host__ __device__ inline int width_of(int w) { return 1 << w; }

// Rows and columns actually present in unit (rb, s).
__host__ __device__ inline int unit_rows(const LayoutView& L, int rb) {
    int64_t r = L.N - (int64_t)rb * RB;
    return r < RB ? (int)r : RB;
}
__host__ __device__ inline int unit_cols(const LayoutView& L, int s) {
    int c = L.G - s * L.C;
    return c < L.C ? c : L.C;
}

// Shared-memory item list of one unit. list[i] = (column << 8) | row, with
// the items of width index w at [wbase[w], wbase[w] + wcount[w]) in
// (column, row) order. colbase must have room for MAX_C * 4 ints.
struct ItemList {
    uint16_t* list;
    int* colbase;     // [MAX_C][4] scratch
    int* wcount;      // [4]
    int* wbase;       // [4]
};

// Rebuild the item list of a unit from its width map (already in shared memory
// as map_s[c*8 + j]). All threads of the block must call it; blockDim.x must be
// a multiple of 32.
__device__ inline void build_item_list(const uint32_t* map_s, int rows, int cols, ItemList il) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
    // pass 1: per (column, width) counts
    for (int c = warp; c < cols; c += nwarps) {
        int cnt0 = 0, cnt1 = 0, cnt2 = 0, cnt3 = 0;
        for (int chunk = 0; chunk < RB / 32; ++chunk) {
            int r = chunk * 32 + lane;
            uint32_t code = (map_s[c * MAP_WORDS + (r >> 4)] >> (2 * (r & 15))) & 3u;
            bool valid = r < rows;
            cnt0 += __popc(__ballot_sync(0xffffffffu, valid && code == 0));
            cnt1 += __popc(__ballot_sync(0xffffffffu, valid && code == 1));
            cnt2 += __popc(__ballot_sync(0xffffffffu, valid && code == 2));
            cnt3 += __popc(__ballot_sync(0xffffffffu, valid && code == 3));
        }
        if (lane == 0) {
            il.colbase[c * 4 + 0] = cnt0;
            il.colbase[c * 4 + 1] = cnt1;
            il.colbase[c * 4 + 2] = cnt2;
            il.colbase[c * 4 + 3] = cnt3;
        }
    }
    __syncthreads();
    if (threadIdx.x < 4) {
        int w = threadIdx.x, tot = 0;
        for (int c = 0; c < cols; ++c) tot += il.colbase[c * 4 + w];
        il.wcount[w] = tot;
    }
    __syncthreads();
    if (threadIdx.x < 4) {
        int w = threadIdx.x, base = 0;
        for (int v = 0; v < w; ++v) base += il.wcount[v];
        il.wbase[w] = base;
        for (int c = 0; c < cols; ++c) {
            int n = il.colbase[c * 4 + w];
            il.colbase[c * 4 + w] = base;
            base += n;
        }
    }
    __syncthreads();
    // pass 2: scatter (column, row) entries
    const uint32_t lt = (1u << lane) - 1u;
    for (int c = warp; c < cols; c += nwarps) {
        int run0 = il.colbase[c * 4 + 0], run1 = il.colbase[c * 4 + 1];
        int run2 = il.colbase[c * 4 + 2], run3 = il.colbase[c * 4 + 3];
        for (int chunk = 0; chunk < RB / 32; ++chunk) {
            int r = chunk * 32 + lane;
            uint32_t code = (map_s[c * MAP_WORDS + (r >> 4)] >> (2 * (r & 15))) & 3u;
            bool valid = r < rows;
            uint32_t m0 = __ballot_sync(0xffffffffu, valid && code == 0);
            uint32_t m1 = __ballot_sync(0xffffffffu, valid && code == 1);
            uint32_t m2 = __ballot_sync(0xffffffffu, valid && code == 2);
            uint32_t m3 = __ballot_sync(0xffffffffu, valid && code == 3);
            if (valid) {
                int pos;
                if (code == 0) pos = run0 + __popc(m0 & lt);
                else if (code == 1) pos = run1 + __popc(m1 & lt);
                else if (code == 2) pos = run2 + __popc(m2 & lt);
                else pos = run3 + __popc(m3 & lt);
                il.list[pos] = (uint16_t)((c << 8) | r);
            }
            run0 += __popc(m0); run1 += __popc(m1); run2 += __popc(m2); run3 += __popc(m3);
        }
    }
    __syncthreads();
}

}  // namespace vbq
