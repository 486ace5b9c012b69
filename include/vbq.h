/*
 * vbq.h — C ABI of the VBQ packed-weight GEMV library for GB300 (sm_103a).
 *
 * VBQ ("Variable Bit-width Quantization", arXiv 2607.02893) stores a weight
 * matrix W (N x K, row-major) as contiguous groups of 64 weights along K
 * (§3.1). Each group g of row n has its own width b[n][g] in {1, 2, 4, 8}
 * (§3.2, the candidate set) and one FP16 scale s[n][g] (§3.1). A group
 * holds 64 integer codes u of b bits each; its weights are s * L_b(u) with
 *     L_1(u) = 2u - 1                       (sign times the absmean scale, §3.1)
 *     L_b(u) = u - 2^(b-1)   for b >= 2     (the symmetric grid of Eq. 1)
 * (the paper fixes the values, not the bit encoding; offset binary is this
 * library's encoding and code 0 of a b >= 2 group decodes to -2^(b-1)).
 *
 * The library implements the inference step of §6: a fused dequantise-and-
 * multiply y = W x that streams the packed codes and never writes wide
 * weights to memory, for one activation vector (vbq_gemv) or a small batch
 * of 2..16 (vbq_gemm_small). Activations are BF16, accumulation and outputs
 * FP32.
 *
 * Conventions for every call:
 *   - Pointers documented as "device" point to CUDA device memory of the
 *     current device; "host" pointers to host memory.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *     stream). Work is enqueued on it and the call returns without waiting,
 *     unless the call says otherwise.
 *   - Every call returns a vbq_status_t. Arguments are validated before any
 *     work is enqueued; on an error nothing is enqueued and outputs are
 *     untouched. Nothing aborts or throws across the ABI. vbq_last_error()
 *     gives a human-readable detail of the calling thread's last error.
 *   - Device arrays must be 16-byte aligned (VBQ_ERR_ALIGN otherwise).
 *   - The library keeps per-device state for the life of the process (each
 *     kernel's shared-memory limit, set once per device; the device address
 *     of vbq_gemv_static's array). A device reset (cudaDeviceReset), or
 *     anything else that destroys and recreates the device's primary
 *     context, invalidates that state: do not call the library on that
 *     device afterwards in the same process.
 *   - Activations (BF16) must be finite with magnitude below 2^64; larger
 *     values may overflow inside the kernels' scaled arithmetic.
 */
#ifndef VBQ_H
#define VBQ_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef int vbq_status_t;

enum {
    VBQ_OK              = 0,
    VBQ_ERR_ARG         = -1,  /* null pointer, bad flag or bad count          */
    VBQ_ERR_SHAPE       = -2,  /* N < 1, K < 64 or K not a multiple of 64      */
    VBQ_ERR_WIDTH       = -3,  /* a bit-width outside {1, 2, 4, 8}              */
    VBQ_ERR_CODE_RANGE  = -4,  /* a code >= 2^b of its group                    */
    VBQ_ERR_ALIGN       = -5,  /* a device pointer not 16-byte aligned          */
    VBQ_ERR_CUDA        = -6,  /* a CUDA runtime call or launch failed          */
    VBQ_ERR_UNSUPPORTED = -7,  /* batch outside 1..16, or a size over a limit   */
    VBQ_ERR_TIMEOUT     = -8,  /* a bounded device wait gave up                 */
    VBQ_ERR_NOMEM       = -9   /* device or host allocation failed              */
};

/* Opaque packed matrix: host descriptor plus one device allocation. */
typedef struct vbq_layout vbq_layout;

/*
 * vbq_quantize — quantise a dense matrix group by group (§3.1), the step that
 * produces vbq_pack's inputs (§6 export).
 *
 *   w           device, N x K float32, row-major. +-inf allowed, NaN is
 *               VBQ_ERR_ARG.
 *   bitwidths   device, N x (K/64) uint8, each in {1, 2, 4, 8}
 *               (VBQ_ERR_WIDTH otherwise).
 *   N, K        K % 64 == 0, N * K <= 2^40.
 *   codes_out   device, N x K uint8: the codes vbq_pack takes.
 *   scales_out  device, N x (K/64) FP16 bit patterns.
 *   stream      stream for the device work.
 *
 * Per group of 64 weights w_j at width b (FP16() rounds to nearest even and
 * saturates above 65504 to 65504):
 *   b >= 2 (Eq. 1): qmax = 2^(b-1) - 1, s = FP16(max_j |w_j| / qmax) with the
 *          quotient in fp64; q_j = clip(round(w_j / s), -qmax, qmax), round
 *          half to even of the exact quotient; u_j = q_j + 2^(b-1). A group
 *          whose s is 0 gets u_j = 2^(b-1).
 *   b = 1  (absmean sign rule): s = FP16(mean_j |w_j|), the sum of |w_j| in
 *          fp64 as a balanced pairwise tree over neighbouring weights
 *          ((|w_0| + |w_1|) + (|w_2| + |w_3|), ...); u_j = 1 if w_j >= 0
 *          (including -0), else 0.
 * So codes and scales are a pure function of w and the widths. The call
 * validates widths and NaNs on the device first and synchronises `stream`
 * (outputs are untouched on an error), then enqueues the quantisation and
 * returns without waiting. It allocates a 4-byte temporary.
 */
vbq_status_t vbq_quantize(const float* w, const uint8_t* bitwidths, int64_t N, int64_t K,
                          uint8_t* codes_out, uint16_t* scales_out, void* stream);

/*
 * vbq_soft_quant — the training-time soft-quantised forward of one matrix
 * (§3.2, differentiable bit selection; the weight step of Alg. 1). Per group g
 * of 64 weights along K:
 *   pi_g      = softmax((l_g + e_g) / tau) over the candidates B = {1, 2, 4, 8};
 *   w_soft    = sum_k pi_gk * w_hat^(B_k), the candidate reconstructions of §3.1
 *               (Eq. 1 with s = max|w| / (2^(b-1) - 1) at 2, 4 and 8 bits;
 *               sign(w) * mean|w| at 1 bit, sign(0) = +1; a zero scale gives 0);
 *   exp_bits  = sum_k pi_gk B_k (the mean over groups is Alg. 1's b-bar);
 *   hard      = B_argmax_k l_gk (the first maximum; Alg. 1's hardened width).
 * The reconstructions' integer decisions are float32 operations, as a float32
 * training framework takes them: s and w / s are correctly rounded float32
 * quotients, rounded half to even, then clipped. The rest is float32 with a few
 * ulps of rounding (w_soft within (eps + 2^-20) sum_k pi_k |w_hat_k| and
 * exp_bits within (eps + 2^-20) exp_bits, eps = 2^-20 (1 + max_k |z_k|),
 * z = (l + e) / tau).
 *
 *   w            device, N x K float32, finite (not checked).
 *   logits       device, N x (K/64) x 4 float32, finite.
 *   gumbel       device, N x (K/64) x 4 float32 noise e, or NULL for none.
 *   tau          the temperature, > 0 and finite (VBQ_ERR_ARG otherwise); the
 *                quotients (l + e) / tau must stay finite in float32 (the paper
 *                anneals tau from 5.0 to 0.5), or pi is undefined.
 *   N, K         K % 64 == 0 (VBQ_ERR_SHAPE), N * K <= 2^40.
 *   w_soft       device, N x K float32; overwritten.
 *   exp_bits     device, N x (K/64) float32, or NULL.
 *   hard_widths  device, N x (K/64) uint8, or NULL.
 * Enqueued on `stream`; allocates nothing.
 */
vbq_status_t vbq_soft_quant(const float* w, const float* logits, const float* gumbel, float tau, int64_t N,
                            int64_t K, float* w_soft, float* exp_bits, uint8_t* hard_widths, void* stream);

/*
 * vbq_pack — build the packed device layout of one matrix (§6: the export
 * step that turns per-group codes into packed storage; §3.1 groups of 64).
 *
 *   codes        N x K uint8, row-major; codes[n*K + k] < 2^b of its group.
 *   bitwidths    N x (K/64) uint8, each in {1, 2, 4, 8}.
 *   scales_fp16  N x (K/64) IEEE half bit patterns.
 *   N, K         rows and columns of W; K % 64 == 0 (callers zero-pad K, as
 *                the paper pads MLP intermediates, §6).
 *   src_on_device  0: the three arrays are host memory; 1: device memory.
 *   stream       stream for the device work.
 *   out          receives the new layout on VBQ_OK.
 *
 * Validates shape, widths and code ranges (VBQ_ERR_SHAPE / _WIDTH /
 * _CODE_RANGE) before building anything. The layout owns its device memory
 * until vbq_free. This call synchronises `stream` (it reads back counts to
 * size the allocation) and may allocate temporary device memory.
 */
vbq_status_t vbq_pack(const uint8_t* codes, const uint8_t* bitwidths,
                      const uint16_t* scales_fp16, int64_t N, int64_t K,
                      int src_on_device, void* stream, vbq_layout** out);

/*
 * vbq_packed_bytes — storage of a layout in bytes (§1, §6 storage accounting).
 *   payload  packed codes: sum over groups of 64*b/8 (exactly; no padding).
 *   scales   2 bytes per group.
 *   meta     everything else the layout keeps on the device (width map, item
 *            offsets, alignment padding).
 * Any output pointer may be NULL.
 */
vbq_status_t vbq_packed_bytes(const vbq_layout* layout, size_t* payload,
                              size_t* scales, size_t* meta);

/* vbq_layout_shape — N and K of a layout (either pointer may be NULL). */
vbq_status_t vbq_layout_shape(const vbq_layout* layout, int64_t* N, int64_t* K);

/*
 * vbq_dequant — unpack a layout back to per-group form (inverse of vbq_pack;
 * the weights of §3.1 rebuilt from storage). All outputs are device arrays
 * and any of them may be NULL:
 *   codes_out      N x K uint8 codes (bit-exact copy of what was packed).
 *   bitwidths_out  N x (K/64) uint8 widths.
 *   scales_out     N x (K/64) FP16 bit patterns.
 *   w_out          N x K float: s * L_b(u).
 */
vbq_status_t vbq_dequant(const vbq_layout* layout, uint8_t* codes_out,
                         uint8_t* bitwidths_out, uint16_t* scales_out,
                         float* w_out, void* stream);

/*
 * vbq_gemv — y = W x for one activation vector (§6, fused dequantise-and-
 * multiply; batch 1 decode).
 *   x  device, K BF16 bit patterns.
 *   y  device, N floats; overwritten.
 * Per output, |y - y_exact| stays within 2e-3 * sum_k |w_nk x_k| + 1e-5.
 * Groups of one row block are summed in a varying order, so repeated calls can
 * differ in the last bits. When a row spans several slabs of the layout, the
 * call uses a split-K workspace
 * owned by the layout: calls that share a layout must not overlap on the GPU
 * (issue them on one stream, or order them with events). The kernel is
 * launched with programmatic dependent launch: it may start loading weights
 * before the previous kernel on the stream has finished, and reads x only
 * after it has.
 */
vbq_status_t vbq_gemv(const vbq_layout* layout, const uint16_t* x, float* y,
                      void* stream);

/*
 * vbq_gemm_small — Y = X W^T for a small batch (§6 product for B = 1..16).
 *   X  device, B x K BF16 bit patterns, row-major.
 *   Y  device, B x N floats, row-major; overwritten.
 *   B  1..16 (VBQ_ERR_UNSUPPORTED otherwise).
 * Same accuracy statement as vbq_gemv; the summation order is not fixed (results
 * can differ in the last bits between calls). For B = 2..4 the library picks,
 * from the layout's group count per width, the cheaper of two paths: the
 * batch-1 table kernel, two rows per launch (both rows share every lookup
 * address and decoded code) and a single row for an odd count, each row
 * computed as vbq_gemv computes it; or the tensor cores (chosen for layouts
 * heavy in 4- and 8-bit groups). For B >= 5 the product runs on the tensor
 * cores:
 * activations are scaled per (row, group column) by a power of two into fp16
 * range (values below 2^-14 of that scale lose low bits), weights enter as
 * exact levels, products and fp32 accumulation as in vbq_gemv. Y needs no
 * zeroing; the same split-K workspace and ordering rules as vbq_gemv apply
 * (calls sharing a layout must not overlap on the GPU), and the kernels are
 * launched the same way.
 */
vbq_status_t vbq_gemm_small(const vbq_layout* layout, const uint16_t* X, float* Y,
                            int B, void* stream);

/*
 * vbq_gemv_swiglu — the MLP's gate-up product with its SwiGLU epilogue fused
 * in (§4: the models' MLPs are SwiGLU; §6: the fused kernels stream the
 * packed gate and up projections, and zero-padded intermediates are inert
 * because silu(0) * u = 0).
 *   layout  a gate-up matrix whose rows alternate: row 2i is the gate
 *           projection of feature i, row 2i + 1 its up projection (N even,
 *           VBQ_ERR_SHAPE otherwise). Any layout from vbq_pack with even N.
 *   x       device, K BF16 bit patterns.
 *   y       device, N floats; overwritten with W x (rows interleaved as in W),
 *           exactly as vbq_gemv writes it. It is also the kernel's
 *           accumulator when a row spans several slabs.
 *   h       device, N/2 BF16 bit patterns; overwritten with
 *           h_i = silu(y_2i) * y_2i+1, silu(z) = z / (1 + e^-z), evaluated in
 *           fp32 on the kernel's y and rounded to nearest even. This is the
 *           down projection's input.
 * Accuracy: y as vbq_gemv; h within the error that the bound on y implies
 * (|d silu/dz| <= 1.1) plus its BF16 rounding. One launch: when a row spans
 * several slabs, each row block's outputs are written by the block that adds
 * its last slab. Same ordering rules as vbq_gemv (calls sharing a layout must
 * not overlap on the GPU; the kernel is launched with programmatic dependent
 * launch).
 */
vbq_status_t vbq_gemv_swiglu(const vbq_layout* layout, const uint16_t* x, float* y, uint16_t* h,
                             void* stream);

/*
 * vbq_gemv_swiglu_in — the MLP's down projection applied to the SwiGLU of a
 * gate-up product, y = W h with h_k = silu(gu[2k]) * gu[2k+1] (§4 SwiGLU
 * MLPs; §6 fused packed products, padded features inert since
 * silu(0) * u = 0). h is computed in fp32 as the kernel stages its
 * activations and never reaches memory.
 *   layout  the down projection, N x K.
 *   gu      device, 2K floats: gate and up of feature k at 2k and 2k + 1, i.e.
 *           the y of a vbq_gemv over a gate-up matrix whose rows alternate.
 *   y       device, N floats; overwritten.
 * Per output, |y - y_exact| stays within 2e-3 * sum_k |w_nk h_k| + 1e-5, with
 * h and y_exact exact functions of gu (h's fp32 evaluation adds a few ulps).
 * Same ordering rules as vbq_gemv; gu is read only after the previous kernel
 * on the stream has finished, so it may be that kernel's output.
 */
vbq_status_t vbq_gemv_swiglu_in(const vbq_layout* layout, const float* gu, float* y, void* stream);

/*
 * vbq_gemv_group — count independent batch-1 products y_i = W_i x_i (§6
 * product, several matrices). (The paper has no counterpart; this is an
 * execution mode for products that do not feed one another, such as the
 * projections of one decode step that read the same input.)
 *   layouts, xs, ys  host arrays of count pointers: layouts, device x_i (K_i
 *                    BF16 bit patterns), device y_i (N_i floats, overwritten).
 *   count            >= 0; 0 does nothing.
 * Product i runs exactly as vbq_gemv(layouts[i], xs[i], ys[i]) and satisfies
 * its accuracy statement, but the launches overlap: launch i > 0 starts
 * without waiting for launch i - 1 and waits for it only before completing.
 * So no x_i may be written by another product of the same group, the layouts
 * must be distinct and the outputs must not overlap (a repeated layout or
 * output is VBQ_ERR_ARG; overlap of distinct output ranges is not checked).
 * Work enqueued on the stream before the call is complete before any product
 * reads its inputs, and work enqueued after it sees every output (it must
 * order itself after the group's last kernel as after any kernel).
 */
vbq_status_t vbq_gemv_group(const vbq_layout* const* layouts, const uint16_t* const* xs, float* const* ys,
                            int count, void* stream);

/*
 * vbq_chain_* — a decode chain: count batch-1 products y_i = W_i x_i run in
 * order by one persistent kernel launch (§6 products, one per projection of
 * a decode step). (The paper has no counterpart; this is an execution mode.)
 *
 * vbq_chain_create fixes the chain's layouts, inputs and outputs:
 *   layouts, xs, ys  host arrays of count pointers: distinct layouts, device
 *                    x_i (K_i BF16 bit patterns), device y_i (N_i floats,
 *                    overwritten, distinct; overlap of distinct output ranges
 *                    is not checked). The layouts must outlive the chain.
 *   waits            host array of count flags, or NULL for all 1. waits[i] = 1:
 *                    product i reads x_i only after every earlier product has
 *                    completed, as when x_i derives from earlier outputs (the
 *                    default; the results equal those of count vbq_gemv calls
 *                    in order). waits[i] = 2: product i has the dependencies
 *                    of product i - 1 and does not depend on it, as when
 *                    products read the same input (a decode step's Q, K and V,
 *                    or gate and up): it may run alongside product i - 1, and a
 *                    later product with waits = 1 waits for both. waits[i] = 0:
 *                    product i does not depend on earlier products of the
 *                    chain. Since no y_i is an input of the chain, a product
 *                    may zero its own y_i early.
 *   count            1 .. 2^20.
 *   out              receives the chain on VBQ_OK.
 * It allocates a small device buffer (descriptors and completion counts) and
 * synchronises the device.
 *
 * vbq_chain_run launches the chain on `stream`: one block per SM, which
 * streams its share of every product's packed weights back to back, across
 * product boundaries (weights never depend on activations), and waits for
 * earlier products only before it reads x_i. Each y_i satisfies the
 * accuracy statement of vbq_gemv. x_i must not be written by the chain's own
 * products. Runs of one chain, and products on its layouts, must not overlap
 * on the GPU (order them on one stream); the launch uses programmatic
 * dependent launch like vbq_gemv. It can be captured in a CUDA graph.
 *
 * vbq_chain_free releases a chain (NULL is accepted).
 */
typedef struct vbq_chain vbq_chain;
vbq_status_t vbq_chain_create(const vbq_layout* const* layouts, const uint16_t* const* xs, float* const* ys,
                              const int* waits, int count, vbq_chain** out);
vbq_status_t vbq_chain_run(const vbq_chain* chain, void* stream);
vbq_status_t vbq_chain_free(vbq_chain* chain);

/*
 * vbq_gemv_static — vbq_gemv for callers that must not allocate device memory.
 * (The paper has no counterpart; this is an operational variant.)
 *
 * Some callers cannot call cudaMalloc where they run products: a serving loop
 * that must stay inside a memory budget fixed at start-up, or a host framework
 * whose allocator must own every device byte (an allocation outside it would
 * break its accounting). This entry point allocates nothing, on the device or
 * the host.
 * It runs the same batch-1 kernel as vbq_gemv, but keeps the kernel's split-K
 * control words (a call counter and one flag per row block) in a fixed array
 * inside this library instead of in the layout.
 *
 *   layout  a layout with at most 8192 row blocks of 128 rows (N <= 1048576);
 *           larger layouts give VBQ_ERR_UNSUPPORTED.
 *   x, y    as in vbq_gemv (device, 16-byte aligned; y is overwritten).
 *
 * The array (32 KB) is a static device variable: every GPU that loads the
 * library holds it until the process exits. The first call on a device looks
 * up the array's address with that device current. Every call on a device shares the
 * array and leaves its contents for the next call: each call adds the same
 * amount to the counter, whatever its grid, so the epoch its flags carry only
 * grows and flags left behind never match a later call. Calls that overlap on
 * the GPU race on the array: order them on one stream. Nothing is enqueued
 * besides the kernel.
 */
vbq_status_t vbq_gemv_static(const vbq_layout* layout, const uint16_t* x, float* y,
                             void* stream);

/*
 * vbq_device_status — report (and clear) a bounded wait that gave up.
 * (The paper has no counterpart; this is the library's failure report.)
 *
 * Every wait inside the product kernels (a copy landing in shared memory, a
 * hand-over between warps, another block's split-K flag) is bounded to about
 * one second. A wait that runs out records VBQ_ERR_TIMEOUT in a device word,
 * lets its block finish without further writes to y and without leaving
 * copies in flight, so the CUDA context stays usable; the affected y is
 * undefined. This call synchronises `stream`, then reads and clears the word.
 *
 *   Returns VBQ_OK, VBQ_ERR_TIMEOUT (some product since the last call gave
 *   up), or VBQ_ERR_CUDA.
 */
vbq_status_t vbq_device_status(void* stream);

/*
 * vbq_selftest_timeout — exercise the bounded-wait path on the device.
 * (The paper has no counterpart; this is a test of vbq_device_status.)
 *
 * Launches one block whose thread 0 waits on a shared-memory barrier that
 * nothing completes, with the wait bounded to limit_us microseconds
 * (1..1000000, else VBQ_ERR_ARG). Afterwards vbq_device_status reports
 * VBQ_ERR_TIMEOUT. Nothing faults and nothing hangs: the block returns when
 * its limit runs out.
 */
vbq_status_t vbq_selftest_timeout(int limit_us, void* stream);

/* vbq_free — release a layout and its device memory (NULL is accepted). */
vbq_status_t vbq_free(vbq_layout* layout);

/* vbq_status_string — static name of a status code. */
const char* vbq_status_string(vbq_status_t status);

/* vbq_last_error — detail of the calling thread's last failed call ("" if none). */
const char* vbq_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* VBQ_H */
