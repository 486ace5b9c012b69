// vbq_soft.cu — the training-time soft-quantised forward (§3.2 differentiable
// bit selection; Alg. 1's weight step): per group of 64 weights, the convex
// combination of its four candidate reconstructions (§3.1: Eq. 1 at 2, 4 and 8
// bits, sign times absmean at 1 bit) under pi = softmax((l + e) / tau), the
// group's expected width sum_k pi_k B_k and its hardened width B_argmax l.
//
// A warp takes 16 consecutive groups at a time, two weights of every group per
// lane (8-byte loads: each group's 256 bytes in one request). max|w| and
// sum|w| of the 16 groups are reduced together across the lanes so that lane j
// ends with group j's (31 shuffles per quantity for the 16 groups, a balanced
// tree of depth 6 per group). Lane j then evaluates group j's selection and
// scales once and hands them to the warp through shared memory. The integer decisions of Eq. 1 are those of a float32
// framework: s = max|w| / qmax is a correctly rounded quotient (__fdiv_rn), and
// every code is rint of the correctly rounded quotient w / s, clipped. That
// code is found from t = |w| * fl(1/s), two roundings within 2^-16 of the
// exact quotient for quotients up to 127: rint(t) is the code whenever t is
// at least 2^-15 from a half-integer (the correctly rounded quotient, within
// 2^-17 of the exact one, is then on the same side of it); otherwise, and for
// scales outside [2^-125, 2^125] (whose reciprocal is not a normal float),
// the IEEE quotient is taken. The arithmetic around the decisions uses
// explicitly rounded operations (no contraction), so it is fixed by this
// source. HBM-bound in intent: 4 bytes in and 4 out per weight, 16 or 32 in
// and 5 out per group.
#include <cstdint>
#include <cuda_runtime.h>

#include "vbq_kernels.h"

namespace vbq {
namespace {

constexpr int SQ_THREADS = 256;
constexpr int SQ_WARPS = SQ_THREADS / 32;
constexpr int SQ_BATCH = 16;             // groups per warp pass: lanes j and j + 16 own group j's terms

// Per-group terms, written by the group's owner lane, read by the warp.
struct __align__(16) GroupTerms {
    float mean, s2, s4, s8;              // 1-bit magnitude; the 2/4/8-bit scales
    float r2, r4, r8, pad;               // fl(1/s), or 0 where the quotient must be divided out
    float pi0, pi1, pi2, pi3;            // the selection
};

// The reciprocal of a scale when t = |w| * fl(1/s) may stand in for the
// quotient (s in [2^-125, 2^125]: fl(1/s) normal); 0 otherwise.
__device__ __forceinline__ float rcp_or_zero(float s) {
    return (s >= 0x1p-125f && s <= 0x1p125f) ? __frcp_rn(s) : 0.f;
}

// s * clip(rint(fl(x / s)), -qmax, qmax) for s > 0, with the code decided from
// t = |x| * r as above (r = rcp_or_zero(s)); 0 for s = 0 (an all-zero group).
__device__ __forceinline__ float recon(float x, float s, float r, float qmax) {
    if (s == 0.f) return 0.f;
    const float a = fabsf(x);
    float q = rintf(__fmul_rn(a, r));
    // t within 2^-15 of a half-integer: |t - rint(t)| > 1/2 - 2^-15 (exact: |t| < 2^23)
    if (r == 0.f || fabsf(__fsub_rn(__fmul_rn(a, r), q)) > 0.5f - 0x1p-15f) q = rintf(__fdiv_rn(a, s));
    return __fmul_rn(s, copysignf(fminf(q, qmax), x));
}

// Reduction of 16 per-lane vectors over the 32 lanes: afterwards m[0] (s[0])
// of lanes j and j + 16 is the maximum (sum) over all lanes of entry j. The
// first level adds lanes l and l ^ 16 entry by entry (both get the same
// bits); then a transposing butterfly: at each level a lane keeps the half of
// its entries whose group index has its lane bit and sends the other half to
// its partner, so n entries take n/2 shuffles per quantity.
template <int N>
__device__ __forceinline__ void reduce_level(float (&m)[SQ_BATCH], float (&s)[SQ_BATCH], int lane) {
    constexpr int H = N / 2;
    const bool hi = lane & H;
#pragma unroll
    for (int i = 0; i < H; ++i) {
        const float ms = hi ? m[i] : m[i + H], mk = hi ? m[i + H] : m[i];
        const float ss = hi ? s[i] : s[i + H], sk = hi ? s[i + H] : s[i];
        m[i] = fmaxf(mk, __shfl_xor_sync(0xffffffffu, ms, H));
        s[i] = __fadd_rn(sk, __shfl_xor_sync(0xffffffffu, ss, H));
    }
}

__global__ void __launch_bounds__(SQ_THREADS) soft_quant_kernel(const float* __restrict__ w,
                                                                const float* __restrict__ logits,
                                                                const float* __restrict__ gumbel, float tau,
                                                                int64_t groups, float* __restrict__ w_soft,
                                                                float* __restrict__ exp_bits,
                                                                uint8_t* __restrict__ hard) {
    __shared__ GroupTerms terms[SQ_WARPS][SQ_BATCH];
    const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
    const int64_t warp0 = ((int64_t)blockIdx.x * SQ_THREADS + threadIdx.x) >> 5;
    const int64_t nwarps = ((int64_t)gridDim.x * SQ_THREADS) >> 5;
    for (int64_t g0 = warp0 * SQ_BATCH; g0 < groups; g0 += nwarps * SQ_BATCH) {
        const int nb = (int)(groups - g0 < SQ_BATCH ? groups - g0 : SQ_BATCH);
        float2 v[SQ_BATCH];
        float m[SQ_BATCH], sm[SQ_BATCH];
#pragma unroll
        for (int j = 0; j < SQ_BATCH; ++j) {
            v[j] = j < nb ? reinterpret_cast<const float2*>(w + (g0 + j) * GROUP)[lane] : make_float2(0.f, 0.f);
            const float a0 = fabsf(v[j].x), a1 = fabsf(v[j].y);
            m[j] = fmaxf(a0, a1);
            sm[j] = __fadd_rn(a0, a1);
        }
#pragma unroll
        for (int j = 0; j < SQ_BATCH; ++j) {
            m[j] = fmaxf(m[j], __shfl_xor_sync(0xffffffffu, m[j], 16));
            sm[j] = __fadd_rn(sm[j], __shfl_xor_sync(0xffffffffu, sm[j], 16));
        }
        reduce_level<16>(m, sm, lane);
        reduce_level<8>(m, sm, lane);
        reduce_level<4>(m, sm, lane);
        reduce_level<2>(m, sm, lane);
        if (lane < nb) {
            // group g0 + lane: its selection pi = softmax((l + e) / tau), widths and scales
            // (lanes 16.. hold the same sums as lanes 0.. and stay idle here)
            const int64_t g = g0 + lane;
            const float mx = m[0];
            const float4 l = reinterpret_cast<const float4*>(logits)[g];
            const float4 e = gumbel ? reinterpret_cast<const float4*>(gumbel)[g] : make_float4(0.f, 0.f, 0.f, 0.f);
            const float z0 = __fdiv_rn(__fadd_rn(l.x, e.x), tau), z1 = __fdiv_rn(__fadd_rn(l.y, e.y), tau);
            const float z2 = __fdiv_rn(__fadd_rn(l.z, e.z), tau), z3 = __fdiv_rn(__fadd_rn(l.w, e.w), tau);
            const float zm = fmaxf(fmaxf(z0, z1), fmaxf(z2, z3));
            const float p0 = expf(__fsub_rn(z0, zm)), p1 = expf(__fsub_rn(z1, zm));
            const float p2 = expf(__fsub_rn(z2, zm)), p3 = expf(__fsub_rn(z3, zm));
            const float S = __fadd_rn(__fadd_rn(p0, p1), __fadd_rn(p2, p3));
            GroupTerms t;
            t.pi0 = __fdiv_rn(p0, S); t.pi1 = __fdiv_rn(p1, S); t.pi2 = __fdiv_rn(p2, S); t.pi3 = __fdiv_rn(p3, S);
            t.mean = __fmul_rn(sm[0], 1.f / GROUP);                // exact: a power of two
            t.s2 = mx;                                            // qmax 1
            t.s4 = __fdiv_rn(mx, 7.f);
            t.s8 = __fdiv_rn(mx, 127.f);
            t.r2 = rcp_or_zero(t.s2); t.r4 = rcp_or_zero(t.s4); t.r8 = rcp_or_zero(t.s8);
            t.pad = 0.f;
            terms[wib][lane] = t;
            if (exp_bits)
                exp_bits[g] = __fadd_rn(__fadd_rn(__fadd_rn(t.pi0, __fmul_rn(2.f, t.pi1)), __fmul_rn(4.f, t.pi2)),
                                        __fmul_rn(8.f, t.pi3));
            if (hard) {                                           // the first maximum of the logits
                int k = 0;
                float best = l.x;
                if (l.y > best) { k = 1; best = l.y; }
                if (l.z > best) { k = 2; best = l.z; }
                if (l.w > best) k = 3;
                hard[g] = (uint8_t)(1u << k);
            }
        }
        __syncwarp();
#pragma unroll
        for (int j = 0; j < SQ_BATCH; ++j) {
            if (j < nb) {
                const GroupTerms& t = terms[wib][j];
                const float4 a = *reinterpret_cast<const float4*>(&t.mean);
                const float4 r = *reinterpret_cast<const float4*>(&t.r2);
                const float4 p = *reinterpret_cast<const float4*>(&t.pi0);
                float out[2];
                const float xs[2] = {v[j].x, v[j].y};
#pragma unroll
                for (int i = 0; i < 2; ++i) {
                    const float x = xs[i];
                    const float r1 = x >= 0.f ? a.x : -a.x;      // sign(0) = +1
                    const float r2 = recon(x, a.y, r.x, 1.f), r4 = recon(x, a.z, r.y, 7.f),
                                r8 = recon(x, a.w, r.z, 127.f);
                    out[i] = __fadd_rn(__fadd_rn(__fadd_rn(__fmul_rn(p.x, r1), __fmul_rn(p.y, r2)),
                                                 __fmul_rn(p.z, r4)),
                                       __fmul_rn(p.w, r8));
                }
                reinterpret_cast<float2*>(w_soft + (g0 + j) * GROUP)[lane] = make_float2(out[0], out[1]);
            }
        }
        __syncwarp();                    // the terms are read before the next pass rewrites them
    }
}

}  // namespace

cudaError_t launch_soft_quant(const float* w, const float* logits, const float* gumbel, float tau, int64_t N,
                              int64_t K, float* w_soft, float* exp_bits, uint8_t* hard, cudaStream_t s) {
    const int64_t groups = N * (K / GROUP);
    int sms = 0;
    const int err = device_sms(&sms);
    if (err != 0) return (cudaError_t)err;
    const int64_t per_block = (int64_t)SQ_WARPS * SQ_BATCH;
    const int64_t want = (groups + per_block - 1) / per_block;
    const int64_t cap = (int64_t)sms * 4;                        // 4 blocks of 8 warps per SM, grid-stride beyond
    const int grid = (int)(want < cap ? want : cap);
    soft_quant_kernel<<<grid, SQ_THREADS, 0, s>>>(w, logits, gumbel, tau, groups, w_soft, exp_bits, hard);
    return cudaGetLastError();
}

}  // namespace vbq
