// vbq_kernels.h — launchers of the library's CUDA kernels (internal; called by
// the C ABI in vbq_api.cu). Each returns the cudaError_t of its launch.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>
#include "vbq_common.cuh"

namespace vbq {

// Pack-time kernels (vbq_pack.cu).
cudaError_t launch_validate(const uint8_t* codes, const uint8_t* widths, int64_t N, int64_t K,
                            uint32_t* err_flags, cudaStream_t s);
cudaError_t launch_count(const uint8_t* widths, int64_t N, int G, int C, int nrb, int units,
                         uint32_t* counts, cudaStream_t s);
cudaError_t launch_scatter(const uint8_t* codes, const uint8_t* widths, const uint16_t* scales,
                           const UnitHeader* headers, const LayoutView& L, uint8_t* blobs, cudaStream_t s);
cudaError_t launch_dequant(const LayoutView& L, uint8_t* codes_out, uint8_t* widths_out,
                           uint16_t* scales_out, float* w_out, cudaStream_t s);

// Quantisation (vbq_quant.cu): validation (bit 0 of err: a width outside
// {1,2,4,8}; bit 1: a NaN weight), then codes and FP16 scales per group.
cudaError_t launch_quant_validate(const float* w, const uint8_t* widths, int64_t N, int64_t K, uint32_t* err,
                                  cudaStream_t s);
cudaError_t launch_quantize(const float* w, const uint8_t* widths, int64_t N, int64_t K, uint8_t* codes,
                            uint16_t* scales, cudaStream_t s);

// Training-time soft-quantised forward (vbq_soft.cu): w_soft (N x K), and per
// group the expected width (exp_bits, may be null) and the hardened width
// (hard, may be null). gumbel may be null (no noise).
cudaError_t launch_soft_quant(const float* w, const float* logits, const float* gumbel, float tau, int64_t N,
                              int64_t K, float* w_soft, float* exp_bits, uint8_t* hard, cudaStream_t s);

// Batches of 2..GEMV1_MAX_B rows may run on the batch-1 table kernel, two
// rows per launch; tables_for_batch (vbq_plan.cu) says whether the layout's
// width mix makes that cheaper than the tensor-core kernel.
constexpr int GEMV1_MAX_B = 4;
bool tables_for_batch(const LayoutView& L, int B);

// Products (vbq_gemv.cu). Y is B x N, overwritten (no zeroing needed).
cudaError_t launch_gemv(const LayoutView& L, const uint16_t* X, float* Y, int B, cudaStream_t s);

// How a batch-1 launch orders itself against the previous kernel on its
// stream (programmatic dependent launch):
//   DEP_BEFORE       lets the next kernel launch at once, then waits for the
//                    previous kernel before touching x, y or control words
//                    (every product call: x may be the previous output);
//   DEP_GROUP_FIRST  waits first, then lets the next kernel launch, so the
//                    rest of a group starts only after earlier stream work;
//   DEP_GROUP_NEXT   lets the next kernel launch and works without waiting
//                    (its inputs predate the group), then waits for the
//                    previous kernel before it completes, so kernels still
//                    complete in stream order.
enum Dep : int { DEP_BEFORE = 0, DEP_GROUP_FIRST = 1, DEP_GROUP_NEXT = 2 };

// count independent batch-1 products (distinct layouts and outputs) as one
// group: launch i > 0 overlaps the tail of launch i - 1.
cudaError_t launch_gemv_group(const LayoutView* const* Ls, const uint16_t* const* xs, float* const* ys, int count,
                              cudaStream_t s);

// Batch 1 on a gate-up matrix whose rows alternate (gate i, up i) with the
// SwiGLU epilogue: y (N floats) as launch_gemv writes it, and h (N/2 BF16 bit
// patterns) = silu(gate) * up. Uses the layout's slab counts (control words
// 2 + nrb ..) when a row spans several slabs.
cudaError_t launch_gemv_swiglu(const LayoutView& L, const uint16_t* x, float* y, uint16_t* h, cudaStream_t s);

// Batch 1 whose activations are h_k = silu(gu[2k]) * gu[2k + 1], computed in
// fp32 while the activation tables are built (gu: 2K floats, the y of a
// gate-up product with alternating rows); h never reaches memory.
cudaError_t launch_gemv_swiglu_in(const LayoutView& L, const float* gu, float* y, cudaStream_t s);

// A chain of count batch-1 products in one persistent launch of blocks
// blocks (every product's ChainItem::rot computed for that count). cctl:
// 3 + count zero-initialised words owned by the chain (call counter, one
// completion count per product, then the count of blocks that have zeroed
// their split-K rows).
cudaError_t launch_chain(const ChainItem* items, int count, uint32_t* cctl, int blocks, cudaStream_t s);
int device_sms(int* sms);   // the current device's SM count (0 on success)

// Batch 1 with the split-K control words in a fixed device array (no
// allocation anywhere); usable for layouts with at most STATIC_CTL_WORDS - 2
// row blocks.
constexpr int STATIC_CTL_WORDS = 2 + 8192;
cudaError_t launch_gemv1_static(const LayoutView& L, const uint16_t* x, float* y, cudaStream_t s);

// Batch 2..16 on the tensor cores (vbq_gemm.cu); Y is B x N, overwritten.
cudaError_t launch_gemm_small(const LayoutView& L, const uint16_t* X, float* Y, int B, cudaStream_t s);

// Bounded-wait report: synchronise s, read and clear the device status words
// of both product files (nonzero when some wait gave up); and the self-test
// that makes one wait run out after limit_ns.
cudaError_t read_device_status(uint32_t* status, cudaStream_t s);
cudaError_t read_device_status_gemm(uint32_t* status);
cudaError_t launch_selftest_timeout(unsigned long long limit_ns, cudaStream_t s);

}  // namespace vbq
