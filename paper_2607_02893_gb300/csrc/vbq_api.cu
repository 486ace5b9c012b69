// vbq_api.cu — the C ABI declared in include/vbq.h: argument validation,
// layout planning and allocation, and kernel dispatch on the caller's stream.
#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <vector>

#include "../../include/vbq.h"
#include "vbq_kernels.h"

struct vbq_layout {
    vbq::LayoutView view;     // device pointers and shape, passed to kernels
    void* base = nullptr;     // the one device allocation
    size_t alloc_bytes = 0;
    size_t payload_bytes = 0, scale_bytes = 0, meta_bytes = 0;
    int device = 0;
};

struct vbq_chain {
    void* base = nullptr;             // one device allocation: the items, then the control words
    vbq::ChainItem* items = nullptr;
    uint32_t* cctl = nullptr;
    int count = 0, blocks = 0, device = 0;
};

namespace {

thread_local char g_err[512] = "";

vbq_status_t fail(vbq_status_t st, const char* fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof(g_err), fmt, ap);
    va_end(ap);
    return st;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

size_t round_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

// Device buffers that vbq_pack frees on every exit path.
struct TempBuffers {
    std::vector<void*> ptrs;
    ~TempBuffers() {
        for (void* p : ptrs) cudaFree(p);
    }
    cudaError_t alloc(void** p, size_t bytes) {
        cudaError_t e = cudaMalloc(p, bytes);
        if (e == cudaSuccess) ptrs.push_back(*p);
        return e;
    }
};

#define VBQ_CUDA(call)                                                                     \
    do {                                                                                   \
        cudaError_t e_ = (call);                                                           \
        if (e_ != cudaSuccess)                                                             \
            return fail(e_ == cudaErrorMemoryAllocation ? VBQ_ERR_NOMEM : VBQ_ERR_CUDA,    \
                        "%s: %s (%s:%d)", #call, cudaGetErrorString(e_), __FILE__, __LINE__); \
    } while (0)

vbq_status_t check_layout(const vbq_layout* L) {
    if (!L) return fail(VBQ_ERR_ARG, "layout is NULL");
    if (!L->base) return fail(VBQ_ERR_ARG, "layout has no device storage");
    return VBQ_OK;
}

}  // namespace

extern "C" {

const char* vbq_status_string(vbq_status_t st) {
    switch (st) {
        case VBQ_OK: return "VBQ_OK";
        case VBQ_ERR_ARG: return "VBQ_ERR_ARG";
        case VBQ_ERR_SHAPE: return "VBQ_ERR_SHAPE";
        case VBQ_ERR_WIDTH: return "VBQ_ERR_WIDTH";
        case VBQ_ERR_CODE_RANGE: return "VBQ_ERR_CODE_RANGE";
        case VBQ_ERR_ALIGN: return "VBQ_ERR_ALIGN";
        case VBQ_ERR_CUDA: return "VBQ_ERR_CUDA";
        case VBQ_ERR_UNSUPPORTED: return "VBQ_ERR_UNSUPPORTED";
        case VBQ_ERR_TIMEOUT: return "VBQ_ERR_TIMEOUT";
        case VBQ_ERR_NOMEM: return "VBQ_ERR_NOMEM";
        default: return "VBQ_ERR_UNKNOWN";
    }
}

const char* vbq_last_error(void) { return g_err; }

vbq_status_t vbq_soft_quant(const float* w, const float* logits, const float* gumbel, float tau, int64_t N,
                            int64_t K, float* w_soft, float* exp_bits, uint8_t* hard_widths, void* stream) {
    g_err[0] = 0;
    if (!w || !logits || !w_soft) return fail(VBQ_ERR_ARG, "w, logits and w_soft must be non-NULL");
    if (!(tau > 0.f) || tau == INFINITY) return fail(VBQ_ERR_ARG, "tau must be positive and finite");
    if (N < 1 || K < vbq::GROUP || K % vbq::GROUP != 0)
        return fail(VBQ_ERR_SHAPE, "need N >= 1 and K a positive multiple of 64 (N=%lld K=%lld)",
                    (long long)N, (long long)K);
    if (N > (1LL << 40) / K) return fail(VBQ_ERR_UNSUPPORTED, "N x K above 2^40 weights");
    if (!aligned16(w) || !aligned16(logits) || !aligned16(gumbel) || !aligned16(w_soft) || !aligned16(exp_bits) ||
        !aligned16(hard_widths))
        return fail(VBQ_ERR_ALIGN, "device arrays must be 16-byte aligned");
    VBQ_CUDA(vbq::launch_soft_quant(w, logits, gumbel, tau, N, K, w_soft, exp_bits, hard_widths,
                                    static_cast<cudaStream_t>(stream)));
    return VBQ_OK;
}

vbq_status_t vbq_pack(const uint8_t* codes, const uint8_t* bitwidths, const uint16_t* scales_fp16,
                      int64_t N, int64_t K, int src_on_device, void* stream, vbq_layout** out) {
    g_err[0] = 0;
    if (!out) return fail(VBQ_ERR_ARG, "out is NULL");
    *out = nullptr;
    if (!codes || !bitwidths || !scales_fp16) return fail(VBQ_ERR_ARG, "codes, bitwidths and scales must be non-NULL");
    if (src_on_device != 0 && src_on_device != 1) return fail(VBQ_ERR_ARG, "src_on_device must be 0 or 1");
    if (N < 1 || K < vbq::GROUP || K % vbq::GROUP != 0)
        return fail(VBQ_ERR_SHAPE, "need N >= 1 and K a positive multiple of 64 (N=%lld K=%lld)",
                    (long long)N, (long long)K);
    if (N > (1LL << 31) - 1 || K / vbq::GROUP > (1LL << 20))
        return fail(VBQ_ERR_UNSUPPORTED, "N or K too large (N=%lld K=%lld)", (long long)N, (long long)K);
    if (src_on_device && !(aligned16(codes) && aligned16(bitwidths) && aligned16(scales_fp16)))
        return fail(VBQ_ERR_ALIGN, "device inputs must be 16-byte aligned");

    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const int64_t G = K / vbq::GROUP;
    const size_t ncodes = (size_t)N * (size_t)K, ngroups = (size_t)N * (size_t)G;
    TempBuffers tmp;

    const uint8_t* d_codes = codes;
    const uint8_t* d_widths = bitwidths;
    const uint16_t* d_scales = scales_fp16;
    if (!src_on_device) {
        void *pc, *pw, *ps;
        VBQ_CUDA(tmp.alloc(&pc, ncodes));
        VBQ_CUDA(tmp.alloc(&pw, ngroups));
        VBQ_CUDA(tmp.alloc(&ps, ngroups * 2));
        VBQ_CUDA(cudaMemcpyAsync(pc, codes, ncodes, cudaMemcpyHostToDevice, s));
        VBQ_CUDA(cudaMemcpyAsync(pw, bitwidths, ngroups, cudaMemcpyHostToDevice, s));
        VBQ_CUDA(cudaMemcpyAsync(ps, scales_fp16, ngroups * 2, cudaMemcpyHostToDevice, s));
        d_codes = static_cast<uint8_t*>(pc);
        d_widths = static_cast<uint8_t*>(pw);
        d_scales = static_cast<uint16_t*>(ps);
    }

    // 1. validation on the device
    void* d_err;
    VBQ_CUDA(tmp.alloc(&d_err, sizeof(uint32_t)));
    VBQ_CUDA(cudaMemsetAsync(d_err, 0, sizeof(uint32_t), s));
    VBQ_CUDA(vbq::launch_validate(d_codes, d_widths, N, K, static_cast<uint32_t*>(d_err), s));
    uint32_t h_err = 0;
    VBQ_CUDA(cudaMemcpyAsync(&h_err, d_err, sizeof(uint32_t), cudaMemcpyDeviceToHost, s));
    VBQ_CUDA(cudaStreamSynchronize(s));
    if (h_err & 1u) return fail(VBQ_ERR_WIDTH, "a bit-width is not in {1,2,4,8}");
    if (h_err & 2u) return fail(VBQ_ERR_CODE_RANGE, "a code is >= 2^b for its group's width");

    // 2. plan: row blocks x slabs. Take the widest slab (C in 16..1) that gives
    // at least half as many units as SMs and whose largest unit blob fits a
    // stage. (Wider units cost less per group than the imbalance they leave:
    // measured on 1B- and 9B-class shapes, 4096^2 takes 5.8 us with C = 16
    // against 6.6 us with C = 4, the width a 3-units-per-SM rule picks.)
    int dev = 0, sms = 0;
    VBQ_CUDA(cudaGetDevice(&dev));
    VBQ_CUDA(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
    const int64_t nrb = (N + vbq::RB - 1) / vbq::RB;
    std::vector<uint32_t> counts;
    std::vector<vbq::UnitHeader> headers;
    int C = 0;
    int64_t S = 0, units = 0;
    uint32_t max16 = 0;
    for (int cand : {16, 8, 4, 2, 1}) {
        if (cand > vbq::MAX_C || (cand > G && cand != 1)) continue;
        const int64_t Sc = (G + cand - 1) / cand, uc = nrb * Sc;
        const bool last = (cand == 1);
        if (!last && 2 * uc < sms) continue;          // fewer units than half the SMs: narrower slabs
        if (uc > (1LL << 31) - 2) return fail(VBQ_ERR_UNSUPPORTED, "too many units");
        void* dc = nullptr;
        VBQ_CUDA(tmp.alloc(&dc, (size_t)uc * 5 * sizeof(uint32_t)));
        VBQ_CUDA(vbq::launch_count(d_widths, N, (int)G, cand, (int)nrb, (int)uc, static_cast<uint32_t*>(dc), s));
        std::vector<uint32_t> cnt((size_t)uc * 5);
        VBQ_CUDA(cudaMemcpyAsync(cnt.data(), dc, cnt.size() * sizeof(uint32_t), cudaMemcpyDeviceToHost, s));
        VBQ_CUDA(cudaStreamSynchronize(s));
        std::vector<vbq::UnitHeader> hd((size_t)uc);
        uint32_t m16 = 0;
        for (int64_t u = 0; u < uc; ++u) {
            hd[u] = vbq::make_header(&cnt[u * 5], cand, (int)cnt[u * 5 + 4]);
            m16 = std::max<uint32_t>(m16, hd[u].size16);
        }
        if (m16 * 16u > vbq::MAX_BLOB_BYTES && !last) continue;
        if (m16 * 16u > vbq::MAX_BLOB_BYTES) return fail(VBQ_ERR_UNSUPPORTED, "unit blob too large");
        C = cand; S = Sc; units = uc; max16 = m16;
        counts.swap(cnt);
        headers.swap(hd);
        break;
    }
    if (C == 0) return fail(VBQ_ERR_UNSUPPORTED, "no slab width fits");
    uint64_t real_items[4] = {0, 0, 0, 0};
    std::vector<uint32_t> blob_off((size_t)units + 1);
    uint64_t off16 = 0;
    for (int64_t u = 0; u < units; ++u) {
        blob_off[u] = (uint32_t)off16;
        off16 += headers[u].size16;
        for (int w = 0; w < 4; ++w) real_items[w] += counts[u * 5 + w];
        if (off16 > 0xffffffffull) return fail(VBQ_ERR_UNSUPPORTED, "layout too large");
    }
    blob_off[units] = (uint32_t)off16;
    const uint64_t total_items = real_items[0] + real_items[1] + real_items[2] + real_items[3];
    if (total_items != ngroups) return fail(VBQ_ERR_CUDA, "item count mismatch (%llu vs %llu)",
                                            (unsigned long long)total_items, (unsigned long long)ngroups);
    size_t payload_bytes = 0;
    for (int w = 0; w < 4; ++w) payload_bytes += (size_t)real_items[w] * 8 * (1u << w);
    const size_t scale_bytes = (size_t)ngroups * 2;

    // 3. one device allocation: blob area (+ slack), then the blob offsets
    const size_t blob_bytes = (size_t)off16 * 16 + 256;
    const size_t off_at = round_up(blob_bytes, 256);
    const size_t ctl_at = round_up(off_at + blob_off.size() * 4, 256);
    // control words: call counter, zeroed-row flags, SwiGLU slab counts
    const size_t alloc_bytes = ctl_at + (2 + 2 * (size_t)nrb) * sizeof(uint32_t);
    void* d_headers = nullptr;
    VBQ_CUDA(tmp.alloc(&d_headers, headers.size() * sizeof(vbq::UnitHeader)));
    VBQ_CUDA(cudaMemcpyAsync(d_headers, headers.data(), headers.size() * sizeof(vbq::UnitHeader),
                             cudaMemcpyHostToDevice, s));

    vbq_layout* L = new (std::nothrow) vbq_layout();
    if (!L) return fail(VBQ_ERR_NOMEM, "host allocation failed");
    cudaError_t e = cudaMalloc(&L->base, alloc_bytes);
    if (e != cudaSuccess) {
        delete L;
        return fail(VBQ_ERR_NOMEM, "cudaMalloc(%zu): %s", alloc_bytes, cudaGetErrorString(e));
    }
    auto bail = [&](vbq_status_t st, const char* what, cudaError_t err) {
        cudaFree(L->base);
        delete L;
        return fail(st, "%s: %s", what, cudaGetErrorString(err));
    };
    uint8_t* base = static_cast<uint8_t*>(L->base);
    L->alloc_bytes = alloc_bytes;
    L->payload_bytes = payload_bytes;
    L->scale_bytes = scale_bytes;
    L->meta_bytes = alloc_bytes - payload_bytes - scale_bytes;
    L->device = dev;
    vbq::LayoutView& V = L->view;
    V.blobs = base;
    V.blob_off = reinterpret_cast<uint32_t*>(base + off_at);
    V.ctl = reinterpret_cast<uint32_t*>(base + ctl_at);
    V.N = N;
    V.K = K;
    V.G = (int)G;
    V.C = C;
    V.S = (int)S;
    V.nrb = (int)nrb;
    V.units = (int)units;
    for (int w = 0; w < 4; ++w) V.items[w] = (int64_t)real_items[w];
    V.max_blob16 = (int)max16;
    V.single_w = -1;
    for (int w = 0, present = 0; w < 4; ++w)
        if (real_items[w]) V.single_w = present++ ? -2 : w;
    if (V.single_w < 0) V.single_w = -1;

    if ((e = cudaMemsetAsync(L->base, 0, alloc_bytes, s)) != cudaSuccess) return bail(VBQ_ERR_CUDA, "memset", e);
    if ((e = cudaMemcpyAsync(base + off_at, blob_off.data(), blob_off.size() * 4, cudaMemcpyHostToDevice, s)) !=
        cudaSuccess)
        return bail(VBQ_ERR_CUDA, "offset copy", e);
    if ((e = vbq::launch_scatter(d_codes, d_widths, d_scales, static_cast<const vbq::UnitHeader*>(d_headers), V,
                                 base, s)) != cudaSuccess)
        return bail(VBQ_ERR_CUDA, "scatter launch", e);
    if ((e = cudaStreamSynchronize(s)) != cudaSuccess) return bail(VBQ_ERR_CUDA, "pack", e);
    *out = L;
    return VBQ_OK;
}

vbq_status_t vbq_packed_bytes(const vbq_layout* L, size_t* payload, size_t* scales, size_t* meta) {
    vbq_status_t st = check_layout(L);
    if (st) return st;
    if (payload) *payload = L->payload_bytes;
    if (scales) *scales = L->scale_bytes;
    if (meta) *meta = L->meta_bytes;
    return VBQ_OK;
}

vbq_status_t vbq_layout_shape(const vbq_layout* L, int64_t* N, int64_t* K) {
    vbq_status_t st = check_layout(L);
    if (st) return st;
    if (N) *N = L->view.N;
    if (K) *K = L->view.K;
    return VBQ_OK;
}

vbq_status_t vbq_quantize(const float* w, const uint8_t* bitwidths, int64_t N, int64_t K, uint8_t* codes_out,
                          uint16_t* scales_out, void* stream) {
    g_err[0] = 0;
    if (!w || !bitwidths || !codes_out || !scales_out)
        return fail(VBQ_ERR_ARG, "w, bitwidths, codes_out and scales_out must be non-NULL");
    if (N < 1 || K < vbq::GROUP || K % vbq::GROUP != 0)
        return fail(VBQ_ERR_SHAPE, "need N >= 1 and K a positive multiple of 64 (N=%lld K=%lld)",
                    (long long)N, (long long)K);
    if (N > (1LL << 40) / K) return fail(VBQ_ERR_UNSUPPORTED, "N x K above 2^40 weights");
    if (!aligned16(w) || !aligned16(bitwidths) || !aligned16(codes_out) || !aligned16(scales_out))
        return fail(VBQ_ERR_ALIGN, "device arrays must be 16-byte aligned");
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    // the flag word is a stream-ordered allocation (no device-wide sync on free)
    void* d_err = nullptr;
    VBQ_CUDA(cudaMallocAsync(&d_err, sizeof(uint32_t), s));
    uint32_t h_err = 0;
    cudaError_t e = cudaMemsetAsync(d_err, 0, sizeof(uint32_t), s);
    if (e == cudaSuccess) e = vbq::launch_quant_validate(w, bitwidths, N, K, static_cast<uint32_t*>(d_err), s);
    if (e == cudaSuccess) e = cudaMemcpyAsync(&h_err, d_err, sizeof(uint32_t), cudaMemcpyDeviceToHost, s);
    const cudaError_t ef = cudaFreeAsync(d_err, s);
    if (e == cudaSuccess) e = ef;
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    VBQ_CUDA(e);
    if (h_err & 1u) return fail(VBQ_ERR_WIDTH, "a bit-width is not in {1,2,4,8}");
    if (h_err & 2u) return fail(VBQ_ERR_ARG, "a weight is NaN");
    VBQ_CUDA(vbq::launch_quantize(w, bitwidths, N, K, codes_out, scales_out, s));
    return VBQ_OK;
}

vbq_status_t vbq_dequant(const vbq_layout* L, uint8_t* codes_out, uint8_t* bitwidths_out,
                         uint16_t* scales_out, float* w_out, void* stream) {
    g_err[0] = 0;
    vbq_status_t st = check_layout(L);
    if (st) return st;
    if (!aligned16(codes_out) || !aligned16(bitwidths_out) || !aligned16(scales_out) || !aligned16(w_out))
        return fail(VBQ_ERR_ALIGN, "outputs must be 16-byte aligned");
    if (!codes_out && !bitwidths_out && !scales_out && !w_out) return VBQ_OK;
    VBQ_CUDA(vbq::launch_dequant(L->view, codes_out, bitwidths_out, scales_out, w_out,
                                 static_cast<cudaStream_t>(stream)));
    return VBQ_OK;
}

static vbq_status_t run_product(const vbq_layout* L, const uint16_t* X, float* Y, int B, void* stream) {
    g_err[0] = 0;
    vbq_status_t st = check_layout(L);
    if (st) return st;
    if (!X || !Y) return fail(VBQ_ERR_ARG, "x and y must be non-NULL");
    if (B < 1 || B > vbq::MAX_BATCH) return fail(VBQ_ERR_UNSUPPORTED, "batch %d outside 1..16", B);
    if (!aligned16(X) || !aligned16(Y)) return fail(VBQ_ERR_ALIGN, "x and y must be 16-byte aligned");
    VBQ_CUDA(vbq::launch_gemv(L->view, X, Y, B, static_cast<cudaStream_t>(stream)));
    return VBQ_OK;
}

vbq_status_t vbq_gemv(const vbq_layout* L, const uint16_t* x, float* y, void* stream) {
    return run_product(L, x, y, 1, stream);
}

vbq_status_t vbq_gemm_small(const vbq_layout* L, const uint16_t* X, float* Y, int B, void* stream) {
    return run_product(L, X, Y, B, stream);
}

vbq_status_t vbq_gemv_group(const vbq_layout* const* layouts, const uint16_t* const* xs, float* const* ys,
                            int count, void* stream) {
    g_err[0] = 0;
    if (count < 0) return fail(VBQ_ERR_ARG, "count %d is negative", count);
    if (count == 0) return VBQ_OK;
    if (!layouts || !xs || !ys) return fail(VBQ_ERR_ARG, "layouts, xs and ys must be non-NULL arrays");
    std::vector<const vbq::LayoutView*> views((size_t)count);
    std::vector<const void*> seen_l((size_t)count), seen_y((size_t)count);
    for (int i = 0; i < count; ++i) {
        if (!layouts[i]) return fail(VBQ_ERR_ARG, "layout %d is NULL", i);
        if (!layouts[i]->base) return fail(VBQ_ERR_ARG, "layout %d has no device storage", i);
        if (!xs[i] || !ys[i]) return fail(VBQ_ERR_ARG, "x and y of product %d must be non-NULL", i);
        if (!aligned16(xs[i]) || !aligned16(ys[i]))
            return fail(VBQ_ERR_ALIGN, "x and y of product %d must be 16-byte aligned", i);
        views[i] = &layouts[i]->view;
        seen_l[i] = layouts[i];
        seen_y[i] = ys[i];
    }
    // the products of a group may run at the same time: layouts (their split-K
    // control words) and outputs must all be distinct
    std::sort(seen_l.begin(), seen_l.end());
    std::sort(seen_y.begin(), seen_y.end());
    if (std::adjacent_find(seen_l.begin(), seen_l.end()) != seen_l.end())
        return fail(VBQ_ERR_ARG, "a layout appears twice in one group");
    if (std::adjacent_find(seen_y.begin(), seen_y.end()) != seen_y.end())
        return fail(VBQ_ERR_ARG, "an output appears twice in one group");
    VBQ_CUDA(vbq::launch_gemv_group(views.data(), xs, ys, count, static_cast<cudaStream_t>(stream)));
    return VBQ_OK;
}

vbq_status_t vbq_gemv_swiglu(const vbq_layout* L, const uint16_t* x, float* y, uint16_t* h, void* stream) {
    g_err[0] = 0;
    vbq_status_t st = check_layout(L);
    if (st) return st;
    if (!x || !y || !h) return fail(VBQ_ERR_ARG, "x, y and h must be non-NULL");
    if (!aligned16(x) || !aligned16(y) || !aligned16(h)) return fail(VBQ_ERR_ALIGN, "x, y and h must be 16-byte aligned");
    if (L->view.N % 2 != 0)
        return fail(VBQ_ERR_SHAPE, "a gate-up matrix has an even number of rows (N=%lld)", (long long)L->view.N);
    VBQ_CUDA(vbq::launch_gemv_swiglu(L->view, x, y, h, static_cast<cudaStream_t>(stream)));
    return VBQ_OK;
}

vbq_status_t vbq_gemv_swiglu_in(const vbq_layout* L, const float* gu, float* y, void* stream) {
    g_err[0] = 0;
    vbq_status_t st = check_layout(L);
    if (st) return st;
    if (!gu || !y) return fail(VBQ_ERR_ARG, "gu and y must be non-NULL");
    if (!aligned16(gu) || !aligned16(y)) return fail(VBQ_ERR_ALIGN, "gu and y must be 16-byte aligned");
    VBQ_CUDA(vbq::launch_gemv_swiglu_in(L->view, gu, y, static_cast<cudaStream_t>(stream)));
    return VBQ_OK;
}

vbq_status_t vbq_gemv_static(const vbq_layout* L, const uint16_t* x, float* y, void* stream) {
    g_err[0] = 0;
    vbq_status_t st = check_layout(L);
    if (st) return st;
    if (!x || !y) return fail(VBQ_ERR_ARG, "x and y must be non-NULL");
    if (!aligned16(x) || !aligned16(y)) return fail(VBQ_ERR_ALIGN, "x and y must be 16-byte aligned");
    if (L->view.nrb > vbq::STATIC_CTL_WORDS - 2)
        return fail(VBQ_ERR_UNSUPPORTED, "vbq_gemv_static supports at most %d row blocks of 128 rows (N <= %d); "
                    "this layout has %d", vbq::STATIC_CTL_WORDS - 2, (vbq::STATIC_CTL_WORDS - 2) * vbq::RB,
                    L->view.nrb);
    VBQ_CUDA(vbq::launch_gemv1_static(L->view, x, y, static_cast<cudaStream_t>(stream)));
    return VBQ_OK;
}

vbq_status_t vbq_chain_create(const vbq_layout* const* layouts, const uint16_t* const* xs, float* const* ys,
                              const int* waits, int count, vbq_chain** out) {
    g_err[0] = 0;
    if (!out) return fail(VBQ_ERR_ARG, "out is NULL");
    *out = nullptr;
    if (count < 1 || count > (1 << 20)) return fail(VBQ_ERR_ARG, "count %d outside 1..2^20", count);
    if (!layouts || !xs || !ys) return fail(VBQ_ERR_ARG, "layouts, xs and ys must be non-NULL arrays");
    std::vector<vbq::ChainItem> items((size_t)count);
    std::vector<const void*> seen_l((size_t)count), seen_y((size_t)count);
    int sms = 0;
    if (vbq::device_sms(&sms) != 0 || sms < 1) return fail(VBQ_ERR_CUDA, "cannot read the device's SM count");
    int64_t units_before = 0;
    int last_wait = 0;                // products before it are complete once it is
    for (int i = 0; i < count; ++i) {
        if (!layouts[i] || !layouts[i]->base) return fail(VBQ_ERR_ARG, "layout %d is NULL or empty", i);
        if (!xs[i] || !ys[i]) return fail(VBQ_ERR_ARG, "x and y of product %d must be non-NULL", i);
        if (!aligned16(xs[i]) || !aligned16(ys[i]))
            return fail(VBQ_ERR_ALIGN, "x and y of product %d must be 16-byte aligned", i);
        if (waits && (waits[i] < 0 || waits[i] > 2)) return fail(VBQ_ERR_ARG, "waits[%d] must be 0, 1 or 2", i);
        vbq::ChainItem& it = items[(size_t)i];
        it.L = layouts[i]->view;
        it.x = xs[i];
        it.y = ys[i];
        const int w = waits ? waits[i] : 1;
        if (w == 2 && i > 0) {          // the same dependencies as the product before
            it.wait_from = items[(size_t)i - 1].wait_from;
            it.wait_hi = items[(size_t)i - 1].wait_hi;
        } else if (w != 0) {            // every product since the last waiting one (itself after the rest)
            it.wait_from = last_wait;
            it.wait_hi = i;
            last_wait = i;
        } else {
            it.wait_from = it.wait_hi = i;
        }
        it.rot = (int)(units_before % sms);
        units_before += it.L.units;
        seen_l[i] = layouts[i];
        seen_y[i] = ys[i];
    }
    std::sort(seen_l.begin(), seen_l.end());
    std::sort(seen_y.begin(), seen_y.end());
    if (std::adjacent_find(seen_l.begin(), seen_l.end()) != seen_l.end())
        return fail(VBQ_ERR_ARG, "a layout appears twice in one chain");
    if (std::adjacent_find(seen_y.begin(), seen_y.end()) != seen_y.end())
        return fail(VBQ_ERR_ARG, "an output appears twice in one chain");
    const size_t items_bytes = round_up(items.size() * sizeof(vbq::ChainItem), 256);
    // control words: call counter, a completion count per product, the zeroing count
    const size_t bytes = items_bytes + (3 + (size_t)count) * sizeof(uint32_t);
    vbq_chain* C = new (std::nothrow) vbq_chain();
    if (!C) return fail(VBQ_ERR_NOMEM, "host allocation failed");
    cudaError_t e = cudaMalloc(&C->base, bytes);
    if (e != cudaSuccess) {
        delete C;
        return fail(VBQ_ERR_NOMEM, "cudaMalloc(%zu): %s", bytes, cudaGetErrorString(e));
    }
    C->items = static_cast<vbq::ChainItem*>(C->base);
    C->cctl = reinterpret_cast<uint32_t*>(static_cast<uint8_t*>(C->base) + items_bytes);
    C->count = count;
    C->blocks = sms;
    cudaGetDevice(&C->device);
    if ((e = cudaMemset(C->base, 0, bytes)) == cudaSuccess)
        e = cudaMemcpy(C->items, items.data(), items.size() * sizeof(vbq::ChainItem), cudaMemcpyHostToDevice);
    if (e != cudaSuccess) {
        cudaFree(C->base);
        delete C;
        return fail(VBQ_ERR_CUDA, "chain set-up: %s", cudaGetErrorString(e));
    }
    *out = C;
    return VBQ_OK;
}

vbq_status_t vbq_chain_run(const vbq_chain* C, void* stream) {
    g_err[0] = 0;
    if (!C || !C->base) return fail(VBQ_ERR_ARG, "chain is NULL or empty");
    VBQ_CUDA(vbq::launch_chain(C->items, C->count, C->cctl, C->blocks, static_cast<cudaStream_t>(stream)));
    return VBQ_OK;
}

vbq_status_t vbq_chain_free(vbq_chain* C) {
    if (!C) return VBQ_OK;
    cudaError_t e = C->base ? cudaFree(C->base) : cudaSuccess;
    delete C;
    if (e != cudaSuccess) return fail(VBQ_ERR_CUDA, "cudaFree: %s", cudaGetErrorString(e));
    return VBQ_OK;
}

vbq_status_t vbq_device_status(void* stream) {
    g_err[0] = 0;
    uint32_t word = 0;
    VBQ_CUDA(vbq::read_device_status(&word, static_cast<cudaStream_t>(stream)));
    if (word) return fail(VBQ_ERR_TIMEOUT, "a bounded device wait gave up (status word 0x%x)", word);
    return VBQ_OK;
}

vbq_status_t vbq_selftest_timeout(int limit_us, void* stream) {
    g_err[0] = 0;
    if (limit_us < 1 || limit_us > 1000000) return fail(VBQ_ERR_ARG, "limit_us must be in 1..1000000, got %d", limit_us);
    VBQ_CUDA(vbq::launch_selftest_timeout(1000ull * (unsigned long long)limit_us, static_cast<cudaStream_t>(stream)));
    return VBQ_OK;
}

vbq_status_t vbq_free(vbq_layout* L) {
    if (!L) return VBQ_OK;
    cudaError_t e = L->base ? cudaFree(L->base) : cudaSuccess;
    delete L;
    if (e != cudaSuccess) return fail(VBQ_ERR_CUDA, "cudaFree: %s", cudaGetErrorString(e));
    return VBQ_OK;
}

}  // extern "C"
