// vbq_gemv.cu — fused dequantise-and-multiply y = W x over the packed layout
// (§6: "loads the packed low-bit bytes for a group, expands them ... in
// registers using the per-group scale, and accumulates the matrix-vector
// product").
//
// One block per unit (row block x slab). The block stages the slab's x in
// shared memory as fp32, rebuilds the unit's item list from the width map,
// then each thread takes whole items: it loads the item's 8*b bytes, expands
// each code to its level, accumulates level * x in fp32, applies the group
// scale once, and adds the group's contribution to the row's shared-memory
// partial sum. Row partials go to y directly (one slab per row) or are added
// into a zeroed y (several slabs).
#include "vbq_kernels.h"

namespace vbq {
namespace {

constexpr int GEMV_THREADS = 256;

template <int B, int NB>
__device__ __forceinline__ void dot_item(const uint8_t* __restrict__ src, const float* __restrict__ xs,
                                         int xstride, int nb, float* acc) {
    uint64_t wv[B];
    if (B == 1) {
        wv[0] = __ldg(reinterpret_cast<const unsigned long long*>(src));
    } else {
        const uint4* p = reinterpret_cast<const uint4*>(src);
#pragma unroll
        for (int i = 0; i < B / 2; ++i) {
            uint4 v = __ldg(p + i);
            wv[2 * i] = (uint64_t)v.x | ((uint64_t)v.y << 32);
            wv[2 * i + 1] = (uint64_t)v.z | ((uint64_t)v.w << 32);
        }
    }
    constexpr uint32_t MASK = (1u << B) - 1u;
#pragma unroll
    for (int j = 0; j < GROUP; ++j) {
        const int bit = j * B;
        const uint32_t u = (uint32_t)(wv[bit >> 6] >> (bit & 63)) & MASK;
        const float lv = (B == 1) ? (float)(int)(2 * u - 1) : (float)((int)u - (1 << (B - 1)));
#pragma unroll
        for (int q = 0; q < NB; ++q)
            if (q < nb) acc[q] = fmaf(lv, xs[q * xstride + j], acc[q]);
    }
}

template <int NB>
__global__ void __launch_bounds__(GEMV_THREADS) gemv_kernel(LayoutView L, const uint16_t* __restrict__ X,
                                                            float* __restrict__ Y, int nb) {
    extern __shared__ float4 smem_f4[];
    float* xs = reinterpret_cast<float*>(smem_f4);                 // [NB][C*64]
    __shared__ uint32_t map_s[MAX_C * MAP_WORDS];
    __shared__ uint16_t list_s[RB * MAX_C];
    __shared__ int colbase_s[MAX_C * 4];
    __shared__ int wcount_s[4], wbase_s[4];
    __shared__ float ys[NB][RB];

    const int u = blockIdx.x, rb = u / L.S, s = u % L.S;
    const int rows = unit_rows(L, rb), cols = unit_cols(L, s);
    const int xstride = L.C * GROUP;
    const int64_t k0 = (int64_t)s * L.C * GROUP;

    for (int i = threadIdx.x; i < cols * MAP_WORDS; i += blockDim.x)
        map_s[i] = L.map[(int64_t)u * L.C * MAP_WORDS + i];
    for (int i = threadIdx.x; i < nb * cols * GROUP; i += blockDim.x) {
        const int q = i / (cols * GROUP), k = i - q * cols * GROUP;
        const uint32_t bits = X[(int64_t)q * L.K + k0 + k];
        xs[q * xstride + k] = __uint_as_float(bits << 16);
    }
    for (int i = threadIdx.x; i < NB * RB; i += blockDim.x) (&ys[0][0])[i] = 0.f;
    __syncthreads();
    ItemList il{list_s, colbase_s, wcount_s, wbase_s};
    build_item_list(map_s, rows, cols, il);

    const int total = wbase_s[3] + wcount_s[3];
    for (int i = threadIdx.x; i < total; i += blockDim.x) {
        const int w = (i >= wbase_s[3]) ? 3 : (i >= wbase_s[2]) ? 2 : (i >= wbase_s[1]) ? 1 : 0;
        const uint32_t e = list_s[i];
        const int c = e >> 8, r = e & 0xff;
        const int64_t item = (int64_t)L.ustart[u * 4 + w] + (i - wbase_s[w]);
        const float sf = __half2float(__ushort_as_half(L.scales[w][item]));
        float acc[NB];
#pragma unroll
        for (int q = 0; q < NB; ++q) acc[q] = 0.f;
        const float* xc = xs + c * GROUP;
        switch (w) {
            case 0: dot_item<1, NB>(L.payload[0] + item * 8, xc, xstride, nb, acc); break;
            case 1: dot_item<2, NB>(L.payload[1] + item * 16, xc, xstride, nb, acc); break;
            case 2: dot_item<4, NB>(L.payload[2] + item * 32, xc, xstride, nb, acc); break;
            default: dot_item<8, NB>(L.payload[3] + item * 64, xc, xstride, nb, acc); break;
        }
#pragma unroll
        for (int q = 0; q < NB; ++q)
            if (q < nb) atomicAdd(&ys[q][r], sf * acc[q]);
    }
    __syncthreads();
    const bool direct = (L.S == 1);
    for (int i = threadIdx.x; i < nb * rows; i += blockDim.x) {
        const int q = i / rows, r = i - q * rows;
        float* dst = Y + (int64_t)q * L.N + (int64_t)rb * RB + r;
        if (direct) *dst = ys[q][r];
        else atomicAdd(dst, ys[q][r]);
    }
}

template <int NB>
cudaError_t launch_nb(const LayoutView& L, const uint16_t* X, float* Y, int B, cudaStream_t s) {
    const size_t dyn = (size_t)NB * L.C * GROUP * sizeof(float);
    static bool attr_set = false;           // per process; the attribute is per function
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(gemv_kernel<NB>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)(NB * MAX_C * GROUP * sizeof(float)));
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    gemv_kernel<NB><<<L.units, GEMV_THREADS, dyn, s>>>(L, X, Y, B);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_gemv(const LayoutView& L, const uint16_t* X, float* Y, int B, cudaStream_t s) {
    if (B <= 1) return launch_nb<1>(L, X, Y, B, s);
    if (B <= 2) return launch_nb<2>(L, X, Y, B, s);
    if (B <= 4) return launch_nb<4>(L, X, Y, B, s);
    if (B <= 8) return launch_nb<8>(L, X, Y, B, s);
    return launch_nb<16>(L, X, Y, B, s);
}

}  // namespace vbq
