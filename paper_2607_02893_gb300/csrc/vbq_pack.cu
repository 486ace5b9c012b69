// vbq_pack.cu — kernels that build and unpack the packed layout described in
// vbq_common.cuh (the export step of §6 and its inverse).
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

// One block per unit, one thread per row: item counts per width index.
__global__ void count_kernel(const uint8_t* __restrict__ widths, int64_t N, int G, int C, int S,
                             uint32_t* __restrict__ counts) {
    __shared__ uint32_t cnt[4];
    const int u = blockIdx.x, rb = u / S, s = u % S;
    if (threadIdx.x < 4) cnt[threadIdx.x] = 0;
    __syncthreads();
    const int64_t row = (int64_t)rb * RB + threadIdx.x;
    const int c0 = s * C, cols = min(C, G - c0);
    uint32_t local[4] = {0, 0, 0, 0};
    if (row < N) {
        for (int c = 0; c < cols; ++c) {
            int w = width_index(widths[row * G + c0 + c]);
            local[w & 3] += 1;
        }
    }
    for (int w = 0; w < 4; ++w)
        if (local[w]) atomicAdd(&cnt[w], local[w]);
    __syncthreads();
    if (threadIdx.x < 4) counts[u * 4 + threadIdx.x] = cnt[threadIdx.x];
}

// Pack the 64 codes of one group (64 bytes at src) at width b into 8*b bytes at dst.
template <int B>
__device__ __forceinline__ void pack_group(const uint8_t* __restrict__ src, uint8_t* __restrict__ dst) {
    constexpr int WORDS = B;          // 64*B bits = B 64-bit words
    uint64_t acc[WORDS];
#pragma unroll
    for (int i = 0; i < WORDS; ++i) acc[i] = 0;
    const uint4* p = reinterpret_cast<const uint4*>(src);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        uint4 v = p[q];
        uint32_t wv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int t = 0; t < 4; ++t) {
#pragma unroll
            for (int byte = 0; byte < 4; ++byte) {
                const int j = q * 16 + t * 4 + byte;
                const uint64_t code = (wv[t] >> (8 * byte)) & 0xffu;
                const int bit = j * B;
                acc[bit >> 6] |= code << (bit & 63);
            }
        }
    }
    if (B == 1) {
        *reinterpret_cast<uint64_t*>(dst) = acc[0];
    } else {
        uint4* d = reinterpret_cast<uint4*>(dst);
#pragma unroll
        for (int i = 0; i < WORDS / 2; ++i) {
            uint4 o;
            o.x = (uint32_t)acc[2 * i]; o.y = (uint32_t)(acc[2 * i] >> 32);
            o.z = (uint32_t)acc[2 * i + 1]; o.w = (uint32_t)(acc[2 * i + 1] >> 32);
            d[i] = o;
        }
    }
}

// One block per unit, one thread per row (RB threads). Walks the unit's columns
// in order, ranks each row's group among the column's groups of the same
// width (rows in increasing order), writes the map, the packed item and its
// scale.
__global__ void __launch_bounds__(RB) scatter_kernel(const uint8_t* __restrict__ codes,
                                                     const uint8_t* __restrict__ widths,
                                                     const uint16_t* __restrict__ scales,
                                                     LayoutView L, uint32_t* __restrict__ map,
                                                     uint8_t* p0, uint8_t* p1, uint8_t* p2, uint8_t* p3,
                                                     uint16_t* s0, uint16_t* s1, uint16_t* s2, uint16_t* s3) {
    __shared__ uint32_t wcnt[RB / 32][4];
    const int u = blockIdx.x, rb = u / L.S, s = u % L.S;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int rows = unit_rows(L, rb), cols = unit_cols(L, s);
    const int r = threadIdx.x;
    const bool valid = r < rows;
    const int64_t row = (int64_t)rb * RB + r;
    const int c0 = s * L.C;
    uint32_t run[4];
#pragma unroll
    for (int w = 0; w < 4; ++w) run[w] = L.ustart[u * 4 + w];
    const uint32_t lt = (1u << lane) - 1u;
    for (int c = 0; c < L.C; ++c) {
        // map words for this column (unused columns and rows stay zero)
        int w = 0;
        if (valid && c < cols) w = width_index(widths[row * L.G + c0 + c]) & 3;
        uint32_t mylo = (lane < 16) ? ((uint32_t)w << (2 * (lane & 15))) : 0u;
        uint32_t myhi = (lane >= 16) ? ((uint32_t)w << (2 * (lane & 15))) : 0u;
        uint32_t wlo = __reduce_or_sync(0xffffffffu, mylo);
        uint32_t whi = __reduce_or_sync(0xffffffffu, myhi);
        if (lane == 0) {
            uint32_t* mw = map + ((int64_t)u * L.C + c) * MAP_WORDS + warp * 2;
            mw[0] = wlo;
            mw[1] = whi;
        }
        if (c >= cols) continue;        // uniform across the block
        const bool has = valid;
        uint32_t m[4];
#pragma unroll
        for (int v = 0; v < 4; ++v) m[v] = __ballot_sync(0xffffffffu, has && w == v);
        if (lane == 0) {
#pragma unroll
            for (int v = 0; v < 4; ++v) wcnt[warp][v] = __popc(m[v]);
        }
        __syncthreads();
        if (has) {
            uint32_t item = run[w] + __popc(m[w] & lt);
            for (int pw = 0; pw < warp; ++pw) item += wcnt[pw][w];
            const uint8_t* src = codes + row * L.K + (int64_t)(c0 + c) * GROUP;
            const uint16_t sc = scales[row * L.G + c0 + c];
            switch (w) {
                case 0: pack_group<1>(src, p0 + (int64_t)item * 8); s0[item] = sc; break;
                case 1: pack_group<2>(src, p1 + (int64_t)item * 16); s1[item] = sc; break;
                case 2: pack_group<4>(src, p2 + (int64_t)item * 32); s2[item] = sc; break;
                default: pack_group<8>(src, p3 + (int64_t)item * 64); s3[item] = sc; break;
            }
        }
#pragma unroll
        for (int v = 0; v < 4; ++v) {
            uint32_t tot = 0;
            for (int pw = 0; pw < RB / 32; ++pw) tot += wcnt[pw][v];
            run[v] += tot;
        }
        __syncthreads();
    }
}

// Unpack one item (64 codes of width B at src) into codes_out (64 bytes),
// and optionally w_out (64 floats = s * L_B(u)).
template <int B>
__device__ __forceinline__ void unpack_group(const uint8_t* __restrict__ src, float s,
                                             uint8_t* codes_out, float* w_out) {
    uint64_t acc[B];
    if (B == 1) {
        acc[0] = *reinterpret_cast<const uint64_t*>(src);
    } else {
        const uint4* p = reinterpret_cast<const uint4*>(src);
#pragma unroll
        for (int i = 0; i < B / 2; ++i) {
            uint4 v = p[i];
            acc[2 * i] = (uint64_t)v.x | ((uint64_t)v.y << 32);
            acc[2 * i + 1] = (uint64_t)v.z | ((uint64_t)v.w << 32);
        }
    }
    constexpr uint32_t MASK = (1u << B) - 1u;
#pragma unroll
    for (int q = 0; q < 16; ++q) {
        uint32_t packed = 0;
        float f[4];
#pragma unroll
        for (int t = 0; t < 4; ++t) {
            const int j = q * 4 + t;
            const int bit = j * B;
            const uint32_t u = (uint32_t)(acc[bit >> 6] >> (bit & 63)) & MASK;
            packed |= u << (8 * t);
            const int lv = (B == 1) ? (int)(2 * u) - 1 : (int)u - (1 << (B - 1));
            f[t] = s * (float)lv;
        }
        if (codes_out) reinterpret_cast<uint32_t*>(codes_out)[q] = packed;
        if (w_out) reinterpret_cast<float4*>(w_out)[q] = make_float4(f[0], f[1], f[2], f[3]);
    }
}

constexpr int DQ_THREADS = 256;

__global__ void __launch_bounds__(DQ_THREADS) dequant_kernel(LayoutView L, uint8_t* codes_out,
                                                             uint8_t* widths_out, uint16_t* scales_out,
                                                             float* w_out) {
    __shared__ uint32_t map_s[MAX_C * MAP_WORDS];
    __shared__ uint16_t list_s[RB * MAX_C];
    __shared__ int colbase_s[MAX_C * 4];
    __shared__ int wcount_s[4], wbase_s[4];
    const int u = blockIdx.x, rb = u / L.S, s = u % L.S;
    const int rows = unit_rows(L, rb), cols = unit_cols(L, s);
    for (int i = threadIdx.x; i < cols * MAP_WORDS; i += blockDim.x)
        map_s[i] = L.map[(int64_t)u * L.C * MAP_WORDS + i];
    __syncthreads();
    ItemList il{list_s, colbase_s, wcount_s, wbase_s};
    build_item_list(map_s, rows, cols, il);
    const int total = wbase_s[3] + wcount_s[3];
    for (int i = threadIdx.x; i < total; i += blockDim.x) {
        int w = (i >= wbase_s[3]) ? 3 : (i >= wbase_s[2]) ? 2 : (i >= wbase_s[1]) ? 1 : 0;
        const uint32_t e = list_s[i];
        const int c = e >> 8, r = e & 0xff;
        const int64_t item = (int64_t)L.ustart[u * 4 + w] + (i - wbase_s[w]);
        const int64_t row = (int64_t)rb * RB + r;
        const int64_t gcol = (int64_t)s * L.C + c;
        const uint16_t sbits = L.scales[w][item];
        const float sf = __half2float(__ushort_as_half(sbits));
        uint8_t* co = codes_out ? codes_out + row * L.K + gcol * GROUP : nullptr;
        float* wo = w_out ? w_out + row * L.K + gcol * GROUP : nullptr;
        if (co || wo) {
            switch (w) {
                case 0: unpack_group<1>(L.payload[0] + item * 8, sf, co, wo); break;
                case 1: unpack_group<2>(L.payload[1] + item * 16, sf, co, wo); break;
                case 2: unpack_group<4>(L.payload[2] + item * 32, sf, co, wo); break;
                default: unpack_group<8>(L.payload[3] + item * 64, sf, co, wo); break;
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

cudaError_t launch_count(const uint8_t* widths, int64_t N, int G, int C, int S, int nrb,
                         uint32_t* counts, cudaStream_t s) {
    count_kernel<<<nrb * S, RB, 0, s>>>(widths, N, G, C, S, counts);
    return cudaGetLastError();
}

cudaError_t launch_scatter(const uint8_t* codes, const uint8_t* widths, const uint16_t* scales,
                           const LayoutView& L, uint32_t* map, uint8_t* const payload[4],
                           uint16_t* const scales_out[4], cudaStream_t s) {
    scatter_kernel<<<L.units, RB, 0, s>>>(codes, widths, scales, L, map, payload[0], payload[1],
                                          payload[2], payload[3], scales_out[0], scales_out[1],
                                          scales_out[2], scales_out[3]);
    return cudaGetLastError();
}

cudaError_t launch_dequant(const LayoutView& L, uint8_t* codes_out, uint8_t* widths_out,
                           uint16_t* scales_out, float* w_out, cudaStream_t s) {
    dequant_kernel<<<L.units, DQ_THREADS, 0, s>>>(L, codes_out, widths_out, scales_out, w_out);
    return cudaGetLastError();
}

}  // namespace vbq
