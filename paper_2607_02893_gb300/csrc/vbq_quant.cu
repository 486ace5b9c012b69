// vbq_quant.cu — per-group quantisation of a dense FP32 matrix into codes and
// FP16 scales (§3.1), the export step before vbq_pack:
//   b >= 2 (Eq. 1): s = FP16(max|w| / qmax), qmax = 2^(b-1) - 1;
//                   q = clip(round(w / s), -qmax, qmax) with round-half-even
//                   of the exact quotient; u = q + 2^(b-1) (s = 0: every
//                   u = 2^(b-1));
//   b = 1         : s = FP16(mean|w|), the sum of |w| taken as a balanced
//                   fp64 tree over neighbouring weights; u = [w >= 0].
// FP16(v) rounds to nearest even and saturates above 65504. The results are
// those of the fp64 formulas (the library's definition), computed without
// fp64 arithmetic in the common case (fp64 runs at a small fraction of the
// fp32 rate on this GPU):
//   - a code: an estimate k = rint(|w| * (1/s)) is within one of the answer,
//     and the thresholds (k -+ 1/2) s are exact fp32 numbers (2k + 1 has at
//     most 10 significant bits, the FP16 s at most 11), so comparing |w| with
//     them gives the correctly rounded quotient, ties included; an fp64
//     quotient rounds to the same integer (with a 24-bit w and an 11-bit s
//     it cannot land on a half-integer the exact quotient misses);
//   - the scale of Eq. 1: the same argument for max|w| / qmax against the
//     FP16 midpoints (fp64 rounding of the quotient never reaches one);
//   - the 1-bit mean: exact integer arithmetic when the fp64 tree is exact
//     (see one_bit_scale), else the fp64 tree itself.
//
// One warp per group, two weights per lane (one 8-byte load; a warp reads the
// group's 256 bytes in one coalesced request), several groups per warp in
// flight.
#include "vbq_kernels.h"

namespace vbq {
namespace {

constexpr int QTHREADS = 256;            // 8 warps per block
constexpr int QGROUPS = 8;               // groups in flight per warp

// FP16 bits of RN(S * 2^P) (S >= 0 an exact integer below 2^53), values
// above 65504 saturating to 65504: integer round-half-even at the FP16
// quantum of the value's binade (2^-24 in the subnormal range).
__device__ __forceinline__ uint32_t fp16_bits_of_scaled(unsigned long long S, int P) {
    if (S == 0) return 0u;
    const int n = 63 - __clzll((long long)S);           // S in [2^n, 2^(n+1))
    int qe = max(n + P - 10, -24);                       // quantum exponent
    const int r = qe - P;                                // bits below the quantum
    unsigned long long mant;
    if (r <= 0) {
        mant = S << (-r);                                // exact (r >= n - 10 >= -10)
    } else if (r >= n + 2) {
        mant = 0;                                        // below half a quantum
    } else {
        mant = S >> r;
        const unsigned long long rem = S & ((1ull << r) - 1), half = 1ull << (r - 1);
        if (rem > half || (rem == half && (mant & 1))) mant += 1;
    }
    if (mant >= 2048) { mant >>= 1; qe += 1; }           // carry out of the 11-bit significand
    if (mant < 1024) return (uint32_t)mant;              // subnormal (qe == -24) or zero
    const int e = qe + 10;
    if (e > 15) return 0x7BFFu;
    return (uint32_t)(((e + 15) << 10) | (int)(mant - 1024));
}

// FP16 bits of RN(m / qmax) for m >= 0 (or +inf), qmax in {1, 7, 127},
// saturating above 65504. An fp32 estimate gives a candidate within one FP16
// step; the midpoints
// to its neighbours times qmax are exact fp32 numbers (at most 12 + 7
// significant bits), so comparing m with them settles the rounding exactly.
__device__ __forceinline__ uint32_t fp16_bits_of_quotient(float m, int qmax) {
    if (m > 65504.f * (float)qmax) return 0x7BFFu;       // exact product; also m = +inf
    // candidate: m times fl(1 / qmax), within 2^-23 of the quotient, so its
    // FP16 rounding is at most one step off
    const float inv = qmax == 1 ? 1.f : qmax == 7 ? (1.f / 7.f) : (1.f / 127.f);
    uint32_t c = (uint32_t)__half_as_ushort(__float2half_rn(m * inv));
    const float cv = __half2float(__ushort_as_half((uint16_t)c));
    if (c < 0x7BFFu) {
        const float hu = 0.5f * (cv + __half2float(__ushort_as_half((uint16_t)(c + 1))));
        const float tu = hu * (float)qmax;
        if (m > tu || (m == tu && (c & 1u))) return c + 1;
    }
    if (c > 0u) {
        const float hd = 0.5f * (cv + __half2float(__ushort_as_half((uint16_t)(c - 1))));
        const float td = hd * (float)qmax;
        if (m < td || (m == td && (c & 1u))) return c - 1;
    }
    return c;
}

__device__ __forceinline__ uint32_t fp16_bits_sat(double s) {   // s >= 0 (or +inf)
    if (s > 65504.0) return 0x7BFFu;
    return (uint32_t)__half_as_ushort(__double2half(s));
}

// 1 / x to within about 2^-22 relative for a normal x (the hardware
// reciprocal approximation): an estimate only; the callers' exact checks
// absorb its error.
__device__ __forceinline__ float rcp_estimate(float x) {
    float r;
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
    return r;
}

// round-half-even(a / sf) for a >= 0 (finite or +inf) and sf > 0, capped at
// qmax, given k = rint of an estimate of the quotient that is within one of
// the answer: the thresholds (k -+ 1/2) sf are exact, so comparing a with
// them settles the rounding, ties included.
__device__ __noinline__ int code_magnitude_exact(float a, float sf, float hs, float k, int qmax) {
    const float base = k * sf;                  // exact
    const float up = base + hs, lo = base - hs; // exact: (k + 1/2) s and (k - 1/2) s
    int q = (int)k;
    if (a > up) q += 1;
    else if (a < lo) q -= 1;
    else if (a == up) q += q & 1;              // tie between k and k + 1: the even one
    else if (a == lo) q -= q & 1;              // tie between k - 1 and k
    return min(q, qmax);
}
// The same with r an estimate of 1 / sf within 2^-22 relative: t = fl(a * r)
// is within (a / sf) 2^-21 <= 2^-13 of the quotient (up to the 256 cap), so
// when t is at least 0.0005 away from a half-integer, rint(t) is the answer;
// otherwise (rarely) the exact thresholds decide.
__device__ __forceinline__ int code_magnitude(float a, float sf, float hs, float r, int qmax) {
    const float t = fminf(a * r, 256.f);
    const float k = rintf(t);
    if (fabsf(t - k) <= 0.4995f) return min((int)k, qmax);
    return code_magnitude_exact(a, sf, hs, k, qmax);   // near a half-integer (rare)
}

// The 1-bit scale FP16(mean |w|) of a group held two weights per lane, with
// the mean's sum taken as the balanced fp64 tree over neighbouring weights.
// When every nonzero |w| is a multiple of 2^L (L the smallest ulp exponent)
// and the largest ulp exponent is at most L + 23, all partial sums of that
// tree are multiples of 2^L below 2^(L + 53): the fp64 tree is exact, and the
// exact integer sum S = sum |w| / 2^L (below 2^53) gives FP16(S * 2^(L - 6))
// directly. Otherwise (a spread over 23 binades, or an infinity) the fp64
// tree is evaluated as written.
__device__ __noinline__ uint32_t one_bit_scale_exact(float a0, float a1) {
    const uint32_t b0 = __float_as_uint(a0), b1 = __float_as_uint(a1);
    const int e0 = (int)(b0 >> 23), e1 = (int)(b1 >> 23);           // biased exponents (a >= 0)
    // ulp exponents of nonzero values (subnormals share the smallest normal's)
    const int u0 = max(e0, 1) - 150, u1 = max(e1, 1) - 150;
    const int lo = min(b0 ? u0 : 1000, b1 ? u1 : 1000), hi = max(b0 ? u0 : -1000, b1 ? u1 : -1000);
    const int L = __reduce_min_sync(0xffffffffu, lo), H = __reduce_max_sync(0xffffffffu, hi);
    const bool finite = __all_sync(0xffffffffu, e0 < 255 && e1 < 255);
    if (L == 1000) return 0u;                                        // all zero
    if (finite && H - L <= 23) {
        const unsigned long long m0 = b0 ? (unsigned long long)((b0 & 0x7FFFFFu) | (e0 ? 0x800000u : 0u)) << (u0 - L) : 0ull;
        const unsigned long long m1 = b1 ? (unsigned long long)((b1 & 0x7FFFFFu) | (e1 ? 0x800000u : 0u)) << (u1 - L) : 0ull;
        unsigned long long S = m0 + m1;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) S += __shfl_xor_sync(0xffffffffu, S, off);
        return fp16_bits_of_scaled(S, L - 6);
    }
    double p = (double)a0 + (double)a1;                              // leaves of the pairwise tree
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) p += __shfl_xor_sync(0xffffffffu, p, off);
    return fp16_bits_sat(p * (1.0 / GROUP));                         // exact division by 64
}

// The same scale, first from an fp32 tree of the same shape: its sum is
// within 6 * 2^-24 (depth times unit roundoff) of the exact sum of the
// non-negative |w|, so its FP16 rounding is the exact mean's unless an FP16
// midpoint lies within 2^-20 of the fp32 mean; only then (rarely) the exact
// evaluation runs. Warp-uniform: every lane holds the same fp32 sum.
__device__ __forceinline__ uint32_t one_bit_scale(float a0, float a1) {
    float t = a0 + a1;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) t += __shfl_xor_sync(0xffffffffu, t, off);
    if (isinf(t)) return 0x7BFFu;                      // the exact mean is far above 65504 too
    const float mean = t * (1.f / GROUP);              // exact
    uint32_t c = min((uint32_t)__half_as_ushort(__float2half_rn(mean)), 0x7BFFu);
    const float cv = __half2float(__ushort_as_half((uint16_t)c)), err = mean * 0x1p-20f;
    bool near = false;
    if (c < 0x7BFFu) near |= fabsf(mean - 0.5f * (cv + __half2float(__ushort_as_half((uint16_t)(c + 1))))) <= err;
    if (c > 0u) near |= fabsf(mean - 0.5f * (cv + __half2float(__ushort_as_half((uint16_t)(c - 1))))) <= err;
    return near ? one_bit_scale_exact(a0, a1) : c;
}

// Width in {1, 2, 4, 8} for every group (bit 0) and no NaN weight (bit 1):
// 16-byte loads over w and the widths as flat arrays.
__global__ void quant_validate_kernel(const float* __restrict__ w, const uint8_t* __restrict__ widths,
                                      int64_t nweights, int64_t ngroups, uint32_t* err) {
    uint32_t flags = 0;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x, t0 = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t n4 = nweights / 4;                    // K % 64 == 0, so a whole number of float4
    const float4* w4 = reinterpret_cast<const float4*>(w);
    for (int64_t i = t0; i < n4; i += 4 * stride) {
        float4 v[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) v[j] = i + j * stride < n4 ? __ldcs(w4 + i + j * stride) : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int j = 0; j < 4; ++j)
            if (isnan(v[j].x) || isnan(v[j].y) || isnan(v[j].z) || isnan(v[j].w)) flags |= 2u;
    }
    for (int64_t gi = t0; gi < ngroups; gi += stride) {
        const uint32_t b = widths[gi];
        if (b != 1 && b != 2 && b != 4 && b != 8) flags |= 1u;
    }
    if (flags) atomicOr(err, flags);
}

__global__ void __launch_bounds__(QTHREADS) quantize_kernel(const float* __restrict__ w,
                                                            const uint8_t* __restrict__ widths, int64_t ngroups,
                                                            uint8_t* __restrict__ codes, uint16_t* __restrict__ scales) {
    const int lane = threadIdx.x & 31;
    const int64_t warps = (int64_t)gridDim.x * (QTHREADS >> 5);
    for (int64_t g0 = ((int64_t)blockIdx.x * (QTHREADS >> 5) + (threadIdx.x >> 5)) * QGROUPS; g0 < ngroups;
         g0 += warps * QGROUPS) {
        float2 v[QGROUPS];
        uint32_t bw[QGROUPS];
#pragma unroll
        for (int j = 0; j < QGROUPS; ++j) {     // loads first: QGROUPS groups in flight
            const int64_t gi = g0 + j < ngroups ? g0 + j : g0;
            v[j] = __ldcs(reinterpret_cast<const float2*>(w + gi * GROUP) + lane);
            bw[j] = widths[gi];
        }
#pragma unroll
        for (int j = 0; j < QGROUPS; ++j) {
            const int64_t gi = g0 + j;
            if (gi >= ngroups) break;           // warp-uniform
            const float a0 = fabsf(v[j].x), a1 = fabsf(v[j].y);
            uint32_t sbits, u0, u1;
            if (bw[j] == 1) {
                sbits = one_bit_scale(a0, a1);
                u0 = v[j].x >= 0.f;
                u1 = v[j].y >= 0.f;
            } else {
                const int qmax = (1 << (bw[j] - 1)) - 1, z = 1 << (bw[j] - 1);
                float m = fmaxf(a0, a1);
#pragma unroll
                for (int off = 16; off > 0; off >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));
                sbits = fp16_bits_of_quotient(m, qmax);
                const float sf = __half2float(__ushort_as_half((uint16_t)sbits));
                if (sf == 0.f) {
                    u0 = u1 = (uint32_t)z;
                } else {
                    const float r = rcp_estimate(sf), hs = 0.5f * sf;
                    const int q0 = code_magnitude(a0, sf, hs, r, qmax), q1 = code_magnitude(a1, sf, hs, r, qmax);
                    u0 = (uint32_t)(z + (v[j].x < 0.f ? -q0 : q0));
                    u1 = (uint32_t)(z + (v[j].y < 0.f ? -q1 : q1));
                }
            }
            reinterpret_cast<uint16_t*>(codes + gi * GROUP)[lane] = (uint16_t)(u0 | (u1 << 8));
            if (lane == 0) scales[gi] = (uint16_t)sbits;
        }
    }
}

int grid_for(int64_t ngroups, int warps_per_block, int per_warp) {
    int dev = 0, sms = 148;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t need = (ngroups + (int64_t)warps_per_block * per_warp - 1) / ((int64_t)warps_per_block * per_warp);
    const int64_t cap = (int64_t)sms * 8;       // 8 blocks of 8 warps per SM
    return (int)(need < cap ? (need > 0 ? need : 1) : cap);
}

}  // namespace

cudaError_t launch_quant_validate(const float* w, const uint8_t* widths, int64_t N, int64_t K, uint32_t* err,
                                  cudaStream_t s) {
    const int64_t ngroups = N * (K / GROUP);
    quant_validate_kernel<<<grid_for(N * K / 4, QTHREADS, 4), QTHREADS, 0, s>>>(w, widths, N * K, ngroups, err);
    return cudaGetLastError();
}

cudaError_t launch_quantize(const float* w, const uint8_t* widths, int64_t N, int64_t K, uint8_t* codes,
                            uint16_t* scales, cudaStream_t s) {
    const int64_t ngroups = N * (K / GROUP);
    quantize_kernel<<<grid_for(ngroups, QTHREADS / 32, QGROUPS), QTHREADS, 0, s>>>(w, widths, ngroups, codes, scales);
    return cudaGetLastError();
}

}  // namespace vbq
