// vbq_common.cuh — device layout of a packed VBQ matrix, shared by the CUDA
// kernels of this library (pack, dequant, products).
//
// Layout (chosen for GB300; the paper fixes only "64*b bits per group, packed
// on byte boundaries", §1 and §6):
//
//   * Rows are cut into row blocks of RB = 128 rows; the K/64 group columns
//     into slabs of C columns (C in 1..16, chosen per matrix at pack time). A
//     (row block, slab) pair is a "unit", numbered slab-major:
//     u = s * nrb + rb, so consecutive units share the same activations.
//   * Every unit is one contiguous, 16-byte aligned blob (so a kernel can copy
//     it into shared memory in one sweep):
//         UnitHeader (48 bytes)
//         payload of width index w = 0..3 (b = 1 << w), each padded to 16 bytes
//         FP16 scales of each width, each padded to 16 bytes
//         row bytes of each width (row within the row block), padded to 16
//         column ends: uint16 cend[w][c] = index (within width w) of the
//         first item after column c
//         task table: one 16-byte TaskDesc per warp task of the batch-1
//         product (see TaskDesc), in the balanced order of balance_tasks
//         (vbq_pack.cu)
//     Blob u starts at byte 16 * blob_off[u] of the layout's blob area.
//   * When a row has several slabs, the batch-1 product adds every slab's row
//     partials into y with atomics, and y needs no zeroing by the caller: the
//     block that owns slab 0 of a row block zeroes those rows first and then
//     sets that row block's flag to the current call's epoch; blocks adding
//     other slabs wait for the flag. With the SwiGLU epilogue it also resets
//     the row block's slab count, and the block whose addition brings the
//     count to S applies the epilogue to the finished rows. The epoch lives on the device (the last
//     block of a call advances it), so graph replays stay correct. Calls that
//     share a layout must not overlap on the GPU.
//   * Within a unit the groups ("items") of one width are ordered by
//     (column, row); item i of width index w has its 8*b payload bytes at
//     payload_w + 8*b*i, its scale at scales_w[i], its row at rows_w[i].
//   * Item formats (code j = the group's weight at column 64*col + j):
//       b = 1: 8 bytes, bit j of the little-endian 64-bit word is code j;
//       b = 2: 16 bytes as two bit planes: bytes 0-7 hold bit 0 of every code
//              (bit j = code j's low bit), bytes 8-15 bit 1;
//       b = 4: 32 bytes, code j at bits [4j, 4j+4) (little-endian);
//       b = 8: 64 bytes, byte j is code j.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>
#include <cuda_fp16.h>

namespace vbq {

constexpr int RB = 128;          // rows per row block
constexpr int GROUP = 64;        // weights per group (§3.1)
constexpr int MAX_C = 16;        // max group columns per slab
constexpr int MAX_BATCH = 16;
constexpr int MAX_UNIT_ITEMS = RB * MAX_C;
constexpr uint32_t MAX_BLOB_BYTES = 41 * 1024;   // a unit blob fits one shared-memory stage

struct UnitHeader {
    uint16_t n[4];        // items per width index
    uint16_t pay16[4];    // payload offsets within the blob, in 16-byte units
    uint16_t sc16[4];     // scale offsets
    uint16_t row16[4];    // row-byte offsets
    uint16_t cc16;        // column-end offset (uint16 [4][C])
    uint16_t size16;      // blob size in 16-byte units
    uint16_t ntask;       // warp tasks of the batch-1 product
    uint16_t task16;      // task-table offset (TaskDesc [ntask])
    uint16_t pad[4];
};
static_assert(sizeof(UnitHeader) == 48, "header is 48 bytes");

// One warp task of the batch-1 product, built at pack time so that a warp
// needs nothing else to run it: up to 32 consecutive items of one width (64
// for 1 bit, lane l holding the adjacent items 2l and 2l + 1), their byte
// offsets within the blob, and the columns they lie in, given as masks over
// the lanes. A width can have no items in some columns, so several column
// ends can fall on one item.
//   32-item tasks: lane l's item lies in column
//     c0 + popc(M1 & lanes <= l) + 2 popc(M2 & lanes <= l),
//     M1 and M2 holding the binary digits of the number of column ends at
//     each item (at most 3; the packer ends a task early before an item with
//     more).
//   1-bit tasks: bit l of M1 marks a column end at item 2l and bit l of M2 one
//     at item 2l + 1 (at most one each; a task ends early before an item with
//     more). Tasks start on an even item so that a lane's pair is one 16-byte
//     load; a task that has to begin on an odd item starts one item early
//     with that first item switched off (skip bit), c0 being the column of
//     its second item.
//   x: scale byte offset of the first item (bits 0-15), c0 (16-19), count - 1
//      (20-25), width index (26-27), skip (28)
//   y: M1   z: M2
//   w: payload byte offset of the first item (bits 0-15), row-byte offset (16-31)
struct __align__(16) TaskDesc {
    uint32_t x, y, z, w;
};
static_assert(sizeof(TaskDesc) == 16, "16-byte task descriptors");
constexpr int TASK_SPAN1 = 64;   // items per 1-bit task
constexpr int TASK_SPAN = 32;    // items per 2-, 4- and 8-bit task
constexpr int MAX_UNIT_TASKS = 2 * MAX_UNIT_ITEMS / TASK_SPAN;   // a bound the task cuts never exceed

// The tasks of one unit from its column ends ce[w][c] (w = width index, c <
// cols): widths 8, 4, 2, 1 bit in that order, each cut into spans of at most
// TASK_SPAN (TASK_SPAN1) items, a span ending early before an item on which
// more column ends fall than its masks can count. Writes the descriptors when
// out is not null (h gives the blob offsets) and returns their number.
__host__ __device__ inline int unit_tasks(const uint16_t (*ce)[MAX_C], int cols, const UnitHeader* h,
                                          TaskDesc* out) {
    int nt = 0;
    for (int w = 3; w >= 0; --w) {
        const int span = w == 0 ? TASK_SPAN1 : TASK_SPAN, maxm = w == 0 ? 1 : 3;
        const int n = cols > 0 ? ce[w][cols - 1] : 0;
        int st = 0;                     // first item of the next task
        while (st < n) {
            const int i0 = w == 0 ? (st & ~1) : st, skip = st - i0;
            int end = i0 + span < n ? i0 + span : n;
            uint32_t m1 = 0, m2 = 0;
            int c0 = 0;                 // ends are nondecreasing: c0 = the first column ending after st
            while (c0 < cols && ce[w][c0] <= st) ++c0;
            for (int c = c0; c < cols && ce[w][c] < end;) {
                const int e = ce[w][c], p = e - i0;
                int mult = 0;
                while (c < cols && ce[w][c] == e) { ++mult; ++c; }
                if (mult > maxm) { end = e; break; }
                if (w == 0) {
                    if (p & 1) m2 |= 1u << (p >> 1);
                    else m1 |= 1u << (p >> 1);
                } else {
                    if (mult & 1) m1 |= 1u << p;
                    if (mult & 2) m2 |= 1u << p;
                }
            }
            if (out) {
                const uint32_t b = 1u << w;
                TaskDesc d;
                d.x = (uint32_t)(h->sc16[w] * 16 + 2 * i0) | ((uint32_t)c0 << 16) |
                      ((uint32_t)(end - i0 - 1) << 20) | ((uint32_t)w << 26) | ((uint32_t)skip << 28);
                d.y = m1;
                d.z = m2;
                d.w = (uint32_t)(h->pay16[w] * 16 + 8 * b * i0) | ((uint32_t)(h->row16[w] * 16 + i0) << 16);
                out[nt] = d;
            }
            ++nt;
            st = end;
        }
    }
    return nt;
}


struct LayoutView {
    const uint8_t* blobs;       // blob area
    const uint32_t* blob_off;   // units + 1 offsets, in 16-byte units
    uint32_t* ctl;              // [0..1] 64-bit call counter (see call_epoch), [2 + rb] y-zeroed flags,
                                // [2 + nrb + rb] slabs added (SwiGLU epilogue, see swiglu_row_block)
    int64_t N, K;
    int G, C, S, nrb, units;
    int max_blob16;             // largest blob, in 16-byte units
    int64_t items[4];           // groups per width index (1, 2, 4, 8 bits): host-side launch choices
    int single_w;               // the width index of every group when the matrix has one width (the
                                // fixed recipe's projections, §3.4), else -1
};

// One product of a chain (a sequence of batch-1 products run by one
// persistent kernel, in order): its layout, activation vector and output.
// Before product i touches x or y, products wait_from .. wait_hi - 1 must be
// complete (wait_from == wait_hi: no wait; wait_hi <= i). Block p takes the
// balanced share of virtual block (p - rot) mod P, so products with fewer
// units than blocks land on different blocks.
struct ChainItem {
    LayoutView L;
    const uint16_t* x;
    float* y;
    int wait_from;
    int wait_hi;
    int rot;
};

__host__ __device__ inline int width_of(int w) { return 1 << w; }
__host__ __device__ inline int unit_rb(const LayoutView& L, int u) { return u % L.nrb; }
__host__ __device__ inline int unit_slab(const LayoutView& L, int u) { return u / L.nrb; }

// Rows and columns actually present in unit (rb, s).
__host__ __device__ inline int unit_rows(const LayoutView& L, int rb) {
    int64_t r = L.N - (int64_t)rb * RB;
    return r < RB ? (int)r : RB;
}
__host__ __device__ inline int unit_cols(const LayoutView& L, int s) {
    int c = L.G - s * L.C;
    return c < L.C ? c : L.C;
}

// Sizes of the blob parts, given the item counts of a unit.
__host__ __device__ inline uint32_t pad16(uint32_t bytes) { return (bytes + 15u) / 16u; }

// A unit of a single-width matrix (every group at width index w, n = rows x
// cols items in (column, row) order) starts with its header, payload and
// scales; this is that prefix's length in 16-byte units (make_header lays the
// blob out so).
__host__ __device__ inline uint32_t single_prefix16(uint32_t n, int w) {
    return (uint32_t)(sizeof(UnitHeader) / 16) + pad16(n * 8u * (1u << w)) + pad16(n * 2u);
}

__host__ __device__ inline UnitHeader make_header(const uint32_t n[4], int C, int ntask) {
    UnitHeader h{};
    uint32_t off = sizeof(UnitHeader) / 16;
    for (int w = 0; w < 4; ++w) { h.n[w] = (uint16_t)n[w]; h.pay16[w] = (uint16_t)off; off += pad16(n[w] * 8u * (1u << w)); }
    for (int w = 0; w < 4; ++w) { h.sc16[w] = (uint16_t)off; off += pad16(n[w] * 2u); }
    for (int w = 0; w < 4; ++w) { h.row16[w] = (uint16_t)off; off += pad16(n[w]); }
    h.cc16 = (uint16_t)off;
    off += pad16(8u * (uint32_t)C);
    h.ntask = (uint16_t)ntask;
    h.task16 = (uint16_t)off;
    off += (uint32_t)ntask;
    h.size16 = (uint16_t)off;
    return h;
}

// ---------------------------------------------------------------------------
// Item formats: pack 64 codes (64 bytes, one per code) into an item, and back.
// ---------------------------------------------------------------------------

template <int B>
__device__ __forceinline__ void pack_item(const uint8_t* __restrict__ src, uint8_t* __restrict__ dst) {
    uint32_t cw[16];
    const uint4* p = reinterpret_cast<const uint4*>(src);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        uint4 v = p[q];
        cw[4 * q] = v.x; cw[4 * q + 1] = v.y; cw[4 * q + 2] = v.z; cw[4 * q + 3] = v.w;
    }
    auto code = [&](int j) -> uint32_t { return (cw[j >> 2] >> (8 * (j & 3))) & 0xffu; };
    if (B == 1 || B == 2) {
        uint64_t plane[2] = {0, 0};
#pragma unroll
        for (int j = 0; j < GROUP; ++j) {
            const uint64_t c = code(j);
            plane[0] |= (c & 1ull) << j;
            if (B == 2) plane[1] |= ((c >> 1) & 1ull) << j;
        }
        if (B == 1) {
            *reinterpret_cast<uint2*>(dst) = make_uint2((uint32_t)plane[0], (uint32_t)(plane[0] >> 32));
        } else {
            *reinterpret_cast<uint4*>(dst) = make_uint4((uint32_t)plane[0], (uint32_t)(plane[0] >> 32),
                                                        (uint32_t)plane[1], (uint32_t)(plane[1] >> 32));
        }
    } else if (B == 4) {
        uint32_t o[8];
#pragma unroll
        for (int t = 0; t < 8; ++t) {
            uint32_t w = 0;
#pragma unroll
            for (int i = 0; i < 8; ++i) w |= code(8 * t + i) << (4 * i);
            o[t] = w;
        }
        uint4* d = reinterpret_cast<uint4*>(dst);
        d[0] = make_uint4(o[0], o[1], o[2], o[3]);
        d[1] = make_uint4(o[4], o[5], o[6], o[7]);
    } else {
        uint4* d = reinterpret_cast<uint4*>(dst);
#pragma unroll
        for (int q = 0; q < 4; ++q) d[q] = make_uint4(cw[4 * q], cw[4 * q + 1], cw[4 * q + 2], cw[4 * q + 3]);
    }
}

// Code j of an item of width B held in 2*B words.
template <int B>
__device__ __forceinline__ uint32_t item_code(const uint32_t* w, int j) {
    if (B == 1) return (w[j >> 5] >> (j & 31)) & 1u;
    if (B == 2) return ((w[j >> 5] >> (j & 31)) & 1u) | (((w[2 + (j >> 5)] >> (j & 31)) & 1u) << 1);
    if (B == 4) return (w[j >> 3] >> (4 * (j & 7))) & 0xfu;
    return (w[j >> 2] >> (8 * (j & 3))) & 0xffu;
}

// Load an item of width B (8-byte aligned for B = 1, 16-byte otherwise) into 2*B words.
template <int B>
__device__ __forceinline__ void load_item(const uint8_t* __restrict__ src, uint32_t* w) {
    if (B == 1) {
        uint2 v = *reinterpret_cast<const uint2*>(src);
        w[0] = v.x; w[1] = v.y;
    } else {
#pragma unroll
        for (int q = 0; q < B / 2; ++q) {
            uint4 v = reinterpret_cast<const uint4*>(src)[q];
            w[4 * q] = v.x; w[4 * q + 1] = v.y; w[4 * q + 2] = v.z; w[4 * q + 3] = v.w;
        }
    }
}

// Level L_b(u): 2u - 1 for b = 1, u - 2^(b-1) otherwise.
template <int B>
__device__ __forceinline__ int level_of(uint32_t u) {
    return B == 1 ? (int)(2 * u) - 1 : (int)u - (1 << (B - 1));
}

// Column of item i of width w, given its column-end table cend (C entries,
// nondecreasing) and a lower bound c0 on the answer.
__device__ __forceinline__ int column_of(const uint16_t* cend, int cols, int c0, int i) {
    int c = c0;
    while (c < cols - 1 && (int)cend[c] <= i) ++c;
    return c;
}

}  // namespace vbq
