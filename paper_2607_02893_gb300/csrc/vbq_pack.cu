// vbq_pack.cu — kernels that build the packed layout described in
// vbq_common.cuh (the export step of §6) and unpack it again.
#include "vbq_kernels.h"

namespace vbq {
namespace {

__device__ __forceinline__ int width_index(uint32_t b) {
    return b == 1 ? 0 : b == 2 ? 1 : b == 4 ? 2 : b == 8 ? 3 : -1;
}

// One thread per group: width in {1,2,4,8} (bit 0 of err) and every code < 2^b (bit 1).
__global__ void validate_kernel(const uint8_t* __restrict__ codes, const uint8_t* __restrict__ widths,
                                int64_t ngroups, uint32_t* err) {
    uint32_t flags = 0;
    for (int64_t gi = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; gi < ngroups;
         gi += (int64_t)gridDim.x * blockDim.x) {
        uint32_t b = widths[gi];
        if (width_index(b) < 0) { flags |= 1u; continue; }
        if (b == 8) continue;
        const uint4* p = reinterpret_cast<const uint4*>(codes + gi * GROUP);
        uint32_t hi = 0;
        uint32_t m = 0xffu & ~((1u << b) - 1u);
        m = m | (m << 8) | (m << 16) | (m << 24);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            uint4 v = p[q];
            hi |= (v.x & m) | (v.y & m) | (v.z & m) | (v.w & m);
        }
        if (hi) flags |= 2u;
    }
    if (flags) atomicOr(err, flags);
}

// One block per unit (slab-major numbering), one thread per row: item counts
// per width and the number of warp tasks the unit's column ends give
// (unit_tasks), as counts[5u .. 5u + 4].
__global__ void __launch_bounds__(RB) count_kernel(const uint8_t* __restrict__ widths, int64_t N, int G, int C,
                                                   int nrb, uint32_t* __restrict__ counts) {
    __shared__ uint32_t wcnt[RB / 32][4];
    __shared__ uint16_t ce[4][MAX_C];
    const int u = blockIdx.x, rb = u % nrb, s = u / nrb;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t row = (int64_t)rb * RB + threadIdx.x;
    const bool valid = row < N;
    const int c0 = s * C, cols = min(C, G - c0);
    uint32_t run[4] = {0, 0, 0, 0};
    for (int c = 0; c < cols; ++c) {
        const int w = valid ? width_index(widths[row * G + c0 + c]) & 3 : 0;
#pragma unroll
        for (int v = 0; v < 4; ++v) {
            const uint32_t m = __ballot_sync(0xffffffffu, valid && w == v);
            if (lane == 0) wcnt[warp][v] = __popc(m);
        }
        __syncthreads();
#pragma unroll
        for (int v = 0; v < 4; ++v) {
            for (int pw = 0; pw < RB / 32; ++pw) run[v] += wcnt[pw][v];
            if (threadIdx.x == 0) ce[v][c] = (uint16_t)run[v];
        }
        __syncthreads();
    }
    if (threadIdx.x == 0) {
        for (int v = 0; v < 4; ++v) counts[(int64_t)u * 5 + v] = run[v];
        counts[(int64_t)u * 5 + 4] = (uint32_t)unit_tasks(ce, cols, nullptr, nullptr);
    }
}

// One block per unit, one thread per row (RB threads). Walks the unit's columns
// in order; each row's group is ranked among the column's groups of the same
// width (rows in increasing order) and written as the next item of that
// width: payload, scale and row byte. Also writes the header (prepared on the
// host) and the per-column counts.
// The batch-1 kernel deals a unit's task k to warp (k + rotation) mod tw of its
// team (tw = 16 or 8) and a block's warps meet at the end of its last unit, so
// the table is written in an order that balances those warps: tasks by
// decreasing cost, each to the least-loaded of 16 bins that still has a
// position (bin b holds positions b, b + 16, ...; the first nt % 16 bins one
// more than the rest, so the positions are exactly 0 .. nt - 1; bins b and
// b + 8 together are a warp's share when tw = 8). The costs are the batch-1
// kernel's measured time per group and width (COST_ONE in vbq_plan.cu: 5.33,
// 7.02, 9.98, 14.0 units for 1, 2, 4, 8 bits) times a task's items: a task
// costs its full span even when shorter, since idle lanes repeat its first
// item. The order does not change any result: every group has its own slot.
__device__ void balance_tasks(TaskDesc* t, int nt) {
    if (nt <= 1 || nt > MAX_UNIT_TASKS) return;
    constexpr int BINS = 16;
    constexpr uint32_t cost_w[4] = {341, 225, 319, 448};     // 64 x 5.33, 32 x 7.02, 32 x 9.98, 32 x 14.0
    constexpr int by_cost[4] = {3, 0, 2, 1};                  // 8, 1, 4, 2 bits
    TaskDesc in[MAX_UNIT_TASKS];
    for (int k = 0; k < nt; ++k) in[k] = t[k];
    uint32_t load[BINS];
    int cnt[BINS];
    for (int b = 0; b < BINS; ++b) { load[b] = 0; cnt[b] = 0; }
    const int base = nt / BINS, extra = nt % BINS;
    for (int oi = 0; oi < 4; ++oi) {
        const uint32_t w = (uint32_t)by_cost[oi];
        for (int k = 0; k < nt; ++k) {
            if (((in[k].x >> 26) & 3u) != w) continue;
            int best = -1;
            for (int b = 0; b < BINS; ++b)
                if (cnt[b] < base + (b < extra ? 1 : 0) && (best < 0 || load[b] < load[best])) best = b;
            t[best + BINS * cnt[best]] = in[k];
            load[best] += cost_w[w];
            ++cnt[best];
        }
    }
}

__global__ void __launch_bounds__(RB) scatter_kernel(const uint8_t* __restrict__ codes,
                                                     const uint8_t* __restrict__ widths,
                                                     const uint16_t* __restrict__ scales,
                                                     const UnitHeader* __restrict__ headers,
                                                     LayoutView L, uint8_t* __restrict__ blobs) {
    __shared__ uint32_t wcnt[RB / 32][4];
    const int u = blockIdx.x, rb = unit_rb(L, u), s = unit_slab(L, u);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int rows = unit_rows(L, rb), cols = unit_cols(L, s);
    const int r = threadIdx.x;
    const bool valid = r < rows;
    const int64_t row = (int64_t)rb * RB + r;
    const int c0 = s * L.C;
    uint8_t* blob = blobs + (int64_t)L.blob_off[u] * 16;
    const UnitHeader h = headers[u];
    if (threadIdx.x < sizeof(UnitHeader) / 4)
        reinterpret_cast<uint32_t*>(blob)[threadIdx.x] = reinterpret_cast<const uint32_t*>(&headers[u])[threadIdx.x];
    uint16_t* cend = reinterpret_cast<uint16_t*>(blob + h.cc16 * 16);
    __shared__ uint16_t ce_s[4][MAX_C];
    uint32_t run[4] = {0, 0, 0, 0};
    const uint32_t lt = (1u << lane) - 1u;
    for (int c = 0; c < cols; ++c) {
        int w = 0;
        if (valid) w = width_index(widths[row * L.G + c0 + c]) & 3;
        uint32_t m[4];
#pragma unroll
        for (int v = 0; v < 4; ++v) m[v] = __ballot_sync(0xffffffffu, valid && w == v);
        if (lane == 0) {
#pragma unroll
            for (int v = 0; v < 4; ++v) wcnt[warp][v] = __popc(m[v]);
        }
        __syncthreads();
        if (valid) {
            uint32_t item = run[w] + __popc(m[w] & lt);
            for (int pw = 0; pw < warp; ++pw) item += wcnt[pw][w];
            const uint8_t* src = codes + row * L.K + (int64_t)(c0 + c) * GROUP;
            const uint16_t sc = scales[row * L.G + c0 + c];
            uint8_t* pay = blob + h.pay16[w] * 16;
            switch (w) {
                case 0: pack_item<1>(src, pay + item * 8); break;
                case 1: pack_item<2>(src, pay + item * 16); break;
                case 2: pack_item<4>(src, pay + item * 32); break;
                default: pack_item<8>(src, pay + item * 64); break;
            }
            reinterpret_cast<uint16_t*>(blob + h.sc16[w] * 16)[item] = sc;
            (blob + h.row16[w] * 16)[item] = (uint8_t)r;
        }
#pragma unroll
        for (int v = 0; v < 4; ++v) {
            uint32_t tot = 0;
            for (int pw = 0; pw < RB / 32; ++pw) tot += wcnt[pw][v];
            run[v] += tot;
            if (threadIdx.x == 0) {
                cend[v * L.C + c] = (uint16_t)run[v];
                ce_s[v][c] = (uint16_t)run[v];
            }
        }
        __syncthreads();
    }
    // the batch-1 product's warp tasks (the count was planned on the host from
    // the same column ends), in the dealing's balanced order
    if (threadIdx.x == 0) {
        TaskDesc* tasks = reinterpret_cast<TaskDesc*>(blob + h.task16 * 16);
        const int nt = unit_tasks(ce_s, cols, &h, tasks);
        balance_tasks(tasks, nt);
    }
}

// Unpack one item of width B into codes_out (64 bytes) and/or w_out
// (64 floats = s * L_B(u)).
template <int B>
__device__ __forceinline__ void unpack_item(const uint8_t* __restrict__ src, float s,
                                            uint8_t* codes_out, float* w_out) {
    uint32_t w[2 * B];
    load_item<B>(src, w);
#pragma unroll
    for (int q = 0; q < 16; ++q) {
        uint32_t packed = 0;
        float f[4];
#pragma unroll
        for (int t = 0; t < 4; ++t) {
            const uint32_t u = item_code<B>(w, 4 * q + t);
            packed |= u << (8 * t);
            f[t] = s * (float)level_of<B>(u);
        }
        if (codes_out) reinterpret_cast<uint32_t*>(codes_out)[q] = packed;
        if (w_out) reinterpret_cast<float4*>(w_out)[q] = make_float4(f[0], f[1], f[2], f[3]);
    }
}

constexpr int DQ_THREADS = 256;

__global__ void __launch_bounds__(DQ_THREADS) dequant_kernel(LayoutView L, uint8_t* codes_out,
                                                             uint8_t* widths_out, uint16_t* scales_out,
                                                             float* w_out) {
    __shared__ UnitHeader h;
    const int u = blockIdx.x, rb = unit_rb(L, u), s = unit_slab(L, u);
    const int cols = unit_cols(L, s);
    const uint8_t* blob = L.blobs + (int64_t)L.blob_off[u] * 16;
    if (threadIdx.x == 0) h = *reinterpret_cast<const UnitHeader*>(blob);
    __syncthreads();
    const uint16_t* cend = reinterpret_cast<const uint16_t*>(blob + h.cc16 * 16);
    const int total = h.n[0] + h.n[1] + h.n[2] + h.n[3];
    for (int i = threadIdx.x; i < total; i += blockDim.x) {
        int w = 0, j = i;
        while (w < 3 && j >= h.n[w]) { j -= h.n[w]; ++w; }
        const int c = column_of(cend + w * L.C, cols, 0, j);
        const int r = (blob + h.row16[w] * 16)[j];
        const uint16_t sbits = reinterpret_cast<const uint16_t*>(blob + h.sc16[w] * 16)[j];
        const float sf = __half2float(__ushort_as_half(sbits));
        const int64_t row = (int64_t)rb * RB + r;
        const int64_t gcol = (int64_t)s * L.C + c;
        uint8_t* co = codes_out ? codes_out + row * L.K + gcol * GROUP : nullptr;
        float* wo = w_out ? w_out + row * L.K + gcol * GROUP : nullptr;
        const uint8_t* pay = blob + h.pay16[w] * 16;
        if (co || wo) {
            switch (w) {
                case 0: unpack_item<1>(pay + j * 8, sf, co, wo); break;
                case 1: unpack_item<2>(pay + j * 16, sf, co, wo); break;
                case 2: unpack_item<4>(pay + j * 32, sf, co, wo); break;
                default: unpack_item<8>(pay + j * 64, sf, co, wo); break;
            }
        }
        if (widths_out) widths_out[row * L.G + gcol] = (uint8_t)(1 << w);
        if (scales_out) scales_out[row * L.G + gcol] = sbits;
    }
}

}  // namespace

cudaError_t launch_validate(const uint8_t* codes, const uint8_t* widths, int64_t N, int64_t K,
                            uint32_t* err_flags, cudaStream_t s) {
    const int64_t ngroups = N * (K / GROUP);
    int64_t blocks = (ngroups + 255) / 256;
    if (blocks > 152 * 32) blocks = 152 * 32;
    validate_kernel<<<(unsigned)blocks, 256, 0, s>>>(codes, widths, ngroups, err_flags);
    return cudaGetLastError();
}

cudaError_t launch_count(const uint8_t* widths, int64_t N, int G, int C, int nrb, int units,
                         uint32_t* counts, cudaStream_t s) {
    count_kernel<<<units, RB, 0, s>>>(widths, N, G, C, nrb, counts);
    return cudaGetLastError();
}

cudaError_t launch_scatter(const uint8_t* codes, const uint8_t* widths, const uint16_t* scales,
                           const UnitHeader* headers, const LayoutView& L, uint8_t* blobs, cudaStream_t s) {
    scatter_kernel<<<L.units, RB, 0, s>>>(codes, widths, scales, headers, L, blobs);
    return cudaGetLastError();
}

cudaError_t launch_dequant(const LayoutView& L, uint8_t* codes_out, uint8_t* widths_out,
                           uint16_t* scales_out, float* w_out, cudaStream_t s) {
    dequant_kernel<<<L.units, DQ_THREADS, 0, s>>>(L, codes_out, widths_out, scales_out, w_out);
    return cudaGetLastError();
}

}  // namespace vbq
