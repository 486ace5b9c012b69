// vbq_soft.cu — the training-time soft-quantised forward (§3.2 differentiable
// bit selection; Alg. 1's weight step): per group of 64 weights, the convex
// combination of its four candidate reconstructions (§3.1: Eq. 1 at 2, 4 and 8
// bits, sign times absmean at 1 bit) under pi = softmax((l + e) / tau), the
// group's expected width sum_k pi_k B_k and its hardened width B_argmax l.
//
// One warp per group, two weights per lane (one 8-byte load: the warp reads
// the group's 256 bytes in one request). max|w| and sum|w| by butterfly
// shuffles (every lane ends with the same bits: each level adds the same two
// values). Every lane evaluates the selection, so no broadcast is needed. The
// integer decisions of Eq. 1 are taken with IEEE float32 operations, as a
// float32 framework takes them: s = max|w| / qmax and w / s are correctly
// rounded quotients (__fdiv_rn), rounded half to even (rintf) and clipped. The
// arithmetic around them uses explicitly rounded operations (no contraction),
// so it is fixed by this source. HBM-bound in intent: 4 bytes in and 4 out
// per weight, 16 or 32 in and 5 out per group.
#include <cstdint>
#include <cuda_runtime.h>

#include "vbq_kernels.h"

namespace vbq {
namespace {

constexpr int SQ_THREADS = 256;

// s * clip(round(x / s), -qmax, qmax); 0 for a zero scale (an all-zero group).
__device__ __forceinline__ float recon(float x, float s, float qmax) {
    if (s == 0.f) return 0.f;
    const float q = fminf(fmaxf(rintf(__fdiv_rn(x, s)), -qmax), qmax);
    return __fmul_rn(s, q);
}

__global__ void __launch_bounds__(SQ_THREADS) soft_quant_kernel(const float* __restrict__ w,
                                                                const float* __restrict__ logits,
                                                                const float* __restrict__ gumbel, float tau,
                                                                int64_t groups, float* __restrict__ w_soft,
                                                                float* __restrict__ exp_bits,
                                                                uint8_t* __restrict__ hard) {
    const int lane = threadIdx.x & 31;
    const int64_t warp0 = ((int64_t)blockIdx.x * SQ_THREADS + threadIdx.x) >> 5;
    const int64_t nwarps = ((int64_t)gridDim.x * SQ_THREADS) >> 5;
    for (int64_t g = warp0; g < groups; g += nwarps) {
        const float2 v = reinterpret_cast<const float2*>(w + g * GROUP)[lane];
        const float a0 = fabsf(v.x), a1 = fabsf(v.y);
        float mx = fmaxf(a0, a1), sm = __fadd_rn(a0, a1);
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
            sm = __fadd_rn(sm, __shfl_xor_sync(0xffffffffu, sm, o));
        }
        const float mean = __fmul_rn(sm, 1.f / GROUP);          // exact: a power of two
        // selection: pi = softmax((l + e) / tau)
        const float4 l = reinterpret_cast<const float4*>(logits)[g];
        const float4 e = gumbel ? reinterpret_cast<const float4*>(gumbel)[g] : make_float4(0.f, 0.f, 0.f, 0.f);
        const float z0 = __fdiv_rn(__fadd_rn(l.x, e.x), tau), z1 = __fdiv_rn(__fadd_rn(l.y, e.y), tau);
        const float z2 = __fdiv_rn(__fadd_rn(l.z, e.z), tau), z3 = __fdiv_rn(__fadd_rn(l.w, e.w), tau);
        const float zm = fmaxf(fmaxf(z0, z1), fmaxf(z2, z3));
        const float p0 = expf(__fsub_rn(z0, zm)), p1 = expf(__fsub_rn(z1, zm));
        const float p2 = expf(__fsub_rn(z2, zm)), p3 = expf(__fsub_rn(z3, zm));
        const float S = __fadd_rn(__fadd_rn(p0, p1), __fadd_rn(p2, p3));
        const float pi0 = __fdiv_rn(p0, S), pi1 = __fdiv_rn(p1, S), pi2 = __fdiv_rn(p2, S), pi3 = __fdiv_rn(p3, S);
        // scales of the 2-, 4- and 8-bit candidates (qmax 1, 7, 127)
        const float s4 = __fdiv_rn(mx, 7.f), s8 = __fdiv_rn(mx, 127.f);
        float out[2];
        const float xs[2] = {v.x, v.y};
#pragma unroll
        for (int i = 0; i < 2; ++i) {
            const float x = xs[i];
            const float r1 = x >= 0.f ? mean : -mean;             // sign(0) = +1
            const float r2 = recon(x, mx, 1.f), r4 = recon(x, s4, 7.f), r8 = recon(x, s8, 127.f);
            out[i] = __fadd_rn(__fadd_rn(__fadd_rn(__fmul_rn(pi0, r1), __fmul_rn(pi1, r2)), __fmul_rn(pi2, r4)),
                               __fmul_rn(pi3, r8));
        }
        reinterpret_cast<float2*>(w_soft + g * GROUP)[lane] = make_float2(out[0], out[1]);
        if (lane == 0) {
            if (exp_bits)
                exp_bits[g] = __fadd_rn(__fadd_rn(__fadd_rn(pi0, __fmul_rn(2.f, pi1)), __fmul_rn(4.f, pi2)),
                                        __fmul_rn(8.f, pi3));
            if (hard) {                                           // the first maximum of the logits
                int k = 0;
                float best = l.x;
                if (l.y > best) { k = 1; best = l.y; }
                if (l.z > best) { k = 2; best = l.z; }
                if (l.w > best) k = 3;
                hard[g] = (uint8_t)(1u << k);
            }
        }
    }
}

}  // namespace

cudaError_t launch_soft_quant(const float* w, const float* logits, const float* gumbel, float tau, int64_t N,
                              int64_t K, float* w_soft, float* exp_bits, uint8_t* hard, cudaStream_t s) {
    const int64_t groups = N * (K / GROUP);
    int sms = 0;
    const int err = device_sms(&sms);
    if (err != 0) return (cudaError_t)err;
    const int64_t want = (groups + SQ_THREADS / 32 - 1) / (SQ_THREADS / 32);
    const int64_t cap = (int64_t)sms * 8;                        // 8 blocks of 8 warps per SM, grid-stride beyond
    const int grid = (int)(want < cap ? want : cap);
    soft_quant_kernel<<<grid, SQ_THREADS, 0, s>>>(w, logits, gumbel, tau, groups, w_soft, exp_bits, hard);
    return cudaGetLastError();
}

}  // namespace vbq
