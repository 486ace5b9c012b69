// vbq_device.cuh — device helpers shared by the product kernels of this
// library: shared-memory access by 32-bit shared address, reductions, the
// bounded mbarrier waits and TMA bulk copies of unit blobs, the split-K flag
// wait.
#pragma once

#include <cstdint>
#include <mutex>
#include <cuda_runtime.h>
#include <cuda_fp16.h>

#include "vbq_common.cuh"

namespace vbq {
namespace {

// Host side, per kernel: its dynamic shared-memory limit is a per-device
// property of the function, set once on every device it is launched on, and
// the device's SM count sizes the persistent grids. Host threads may launch
// concurrently, so this state is read and written under a lock.
struct LaunchPrep {
    static constexpr int MAX_DEVICES = 64;
    std::mutex mu;
    bool ready[MAX_DEVICES] = {};
    int sms[MAX_DEVICES] = {};

    template <class Kernel>
    cudaError_t get(Kernel kernel, size_t smem, int* sms_out) {
        int dev = 0;
        cudaError_t e = cudaGetDevice(&dev);
        if (e != cudaSuccess) return e;
        if (dev < 0 || dev >= MAX_DEVICES) return cudaErrorInvalidDevice;
        std::lock_guard<std::mutex> lock(mu);
        if (!ready[dev]) {
            if ((e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)) !=
                cudaSuccess)
                return e;
            if ((e = cudaDeviceGetAttribute(&sms[dev], cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
            ready[dev] = true;
        }
        *sms_out = sms[dev];
        return cudaSuccess;
    }
};

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

template <int OFF>
__device__ __forceinline__ float lds_f32(uint32_t addr) {
    float v;
    asm("ld.shared.f32 %0, [%1+%2];" : "=f"(v) : "r"(addr), "n"(OFF));
    return v;
}

__device__ __forceinline__ void sts_f32(uint32_t addr, float v) {
    asm volatile("st.shared.f32 [%0], %1;" :: "r"(addr), "f"(v) : "memory");
}
// Store only when pred is true (a predicated store: the code around it stays
// one basic block).
__device__ __forceinline__ void sts_f32_if(uint32_t addr, float v, bool pred) {
    asm volatile("{\n\t.reg .pred p;\n\tsetp.ne.u32 p, %2, 0;\n\t@p st.shared.f32 [%0], %1;\n\t}"
                 :: "r"(addr), "f"(v), "r"((uint32_t)pred) : "memory");
}
__device__ __forceinline__ void sts_zero4(uint32_t addr) {
    asm volatile("st.shared.v4.u32 [%0], {%1, %1, %1, %1};" :: "r"(addr), "r"(0u) : "memory");
}
__device__ __forceinline__ float4 lds_f32x4(uint32_t addr) {
    float4 v;
    asm("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];"
                 : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w) : "r"(addr));
    return v;
}

__device__ __forceinline__ uint32_t lds_u8(uint32_t addr) {
    uint32_t v;
    asm("ld.shared.u8 %0, [%1];" : "=r"(v) : "r"(addr));
    return v;
}
__device__ __forceinline__ uint32_t lds_u16(uint32_t addr) {
    uint32_t v;
    asm("ld.shared.u16 %0, [%1];" : "=r"(v) : "r"(addr));
    return v;
}
__device__ __forceinline__ float lds_f32r(uint32_t addr) {
    float v;
    asm("ld.shared.f32 %0, [%1];" : "=f"(v) : "r"(addr));
    return v;
}
__device__ __forceinline__ float2 lds_f32x2(uint32_t addr) {
    float2 v;
    asm("ld.shared.v2.f32 {%0, %1}, [%2];" : "=f"(v.x), "=f"(v.y) : "r"(addr));
    return v;
}

__device__ __forceinline__ uint4 lds_u32x4(uint32_t addr) {
    uint4 v;
    asm("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr));
    return v;
}

__device__ __forceinline__ uint2 lds_u32x2(uint32_t addr) {
    uint2 v;
    asm("ld.shared.v2.u32 {%0, %1}, [%2];" : "=r"(v.x), "=r"(v.y) : "r"(addr));
    return v;
}

__device__ __forceinline__ uint32_t lds_u32(uint32_t addr) {
    uint32_t v;
    asm("ld.shared.u32 %0, [%1];" : "=r"(v) : "r"(addr));
    return v;
}

__device__ __forceinline__ float2 f2(float a, float b) { return make_float2(a, b); }

// y += v on a shared-memory float (32-bit shared address) / a global float.
__device__ __forceinline__ void red_shared(uint32_t addr, float v) {
    asm volatile("red.shared.add.f32 [%0], %1;" :: "r"(addr), "f"(v) : "memory");
}
__device__ __forceinline__ void red_global(float* p, float v) {
    asm volatile("red.global.add.f32 [%0], %1;" :: "l"(p), "f"(v) : "memory");
}

// Bring the 128-byte line holding p into L2 (no value is read: safe before
// griddepcontrol.wait, since a later write by the previous grid updates the
// line in L2, where coherence is kept).
__device__ __forceinline__ void prefetch_l2(const void* p) {
    asm volatile("prefetch.global.L2 [%0];" :: "l"(p));
}

// Order this thread's earlier writes (and those it has observed) before its
// later ones, GPU-wide: the release half of __threadfence, without waiting for
// sequential consistency.
// Release store / acquire load at GPU scope: the split-K zeroed-row flags.
// A warp's zero stores, ordered before lane 0 by the warp barrier, are visible
// to whoever acquires the flag; the acquiring lanes order the warp's later
// additions after it by another warp barrier.
__device__ __forceinline__ void st_release_gpu(uint32_t* p, uint32_t v) {
    asm volatile("st.release.gpu.global.u32 [%0], %1;" :: "l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ uint32_t ld_acquire_gpu(const uint32_t* p) {
    uint32_t v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

// Acquire-release add at GPU scope (returns the old value), and a relaxed
// GPU-scope load of two floats (read at L2, never a stale L1 line).
__device__ __forceinline__ uint32_t atom_add_acq_rel_gpu(uint32_t* p, uint32_t v) {
    uint32_t old;
    asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
    return old;
}
__device__ __forceinline__ float2 ld_relaxed_gpu_f32x2(const float* p) {
    float2 v;
    asm volatile("ld.relaxed.gpu.global.v2.f32 {%0, %1}, [%2];" : "=f"(v.x), "=f"(v.y) : "l"(p) : "memory");
    return v;
}

// Shared-memory words at CTA scope: a release addition (no reply) and an
// acquire load.
__device__ __forceinline__ void red_release_cta_shared_add(uint32_t addr, uint32_t v) {
    asm volatile("red.release.cta.shared::cta.add.u32 [%0], %1;" :: "r"(addr), "r"(v) : "memory");
}
__device__ __forceinline__ uint32_t ld_acquire_cta_shared(uint32_t addr) {
    uint32_t v;
    asm volatile("ld.acquire.cta.shared::cta.u32 %0, [%1];" : "=r"(v) : "r"(addr) : "memory");
    return v;
}

// Release reduction at GPU scope (no reply): a chain's per-product completion counts.
__device__ __forceinline__ void red_release_gpu_add(uint32_t* p, uint32_t v) {
    asm volatile("red.release.gpu.global.add.u32 [%0], %1;" :: "l"(p), "r"(v) : "memory");
}

// Split-K call counter, control words 0-1 (one 64-bit word): every call adds
// exactly 2^CALL_SHIFT in all, split over its blocks, so (counter >>
// CALL_SHIFT) counts the calls before this one; a block that reads it while
// other blocks of the same call have already added their shares still sees
// fewer than 2^CALL_SHIFT of them. The call's epoch (the value its zeroed-row
// flags carry) is that count + 1. The additions need no reply, so no block
// waits on them before it exits.
constexpr int CALL_SHIFT = 20;
__device__ __forceinline__ unsigned long long call_count_raw(const uint32_t* ctl) {
    unsigned long long c;
    asm volatile("ld.volatile.global.u64 %0, [%1];" : "=l"(c) : "l"(ctl) : "memory");
    return c;
}
__device__ __forceinline__ uint32_t epoch_of(unsigned long long c) { return (uint32_t)(c >> CALL_SHIFT) + 1u; }
__device__ __forceinline__ uint32_t call_epoch(const uint32_t* ctl) { return epoch_of(call_count_raw(ctl)); }
__device__ __forceinline__ void call_done(uint32_t* ctl) {     // one thread per block, once per call
    const unsigned long long q = (1ull << CALL_SHIFT) / gridDim.x;
    const unsigned long long share = blockIdx.x == 0 ? (1ull << CALL_SHIFT) - q * (gridDim.x - 1) : q;
    asm volatile("red.relaxed.gpu.global.add.u64 [%0], %1;" :: "l"(ctl), "l"(share) : "memory");
}
__device__ __forceinline__ float half_bits(uint32_t bits) { return __half2float(__ushort_as_half((uint16_t)bits)); }

// ---------------------------------------------------------------------------
// Unit blobs arrive by TMA bulk copy; roles hand stages over through
// mbarriers. Every wait is bounded: after about a second (or as soon as another
// role has given up) the waiting role records VBQ_DEVICE_TIMEOUT in
// g_device_status, raises the block's abort flag and skips the rest of its
// work; the copier lets every copy it started land before the block exits.
// ---------------------------------------------------------------------------

__device__ uint32_t g_device_status;     // one word per translation unit (internal linkage)
constexpr uint32_t VBQ_DEVICE_TIMEOUT = 1u;
constexpr unsigned long long WAIT_LIMIT_NS = 1000000000ull;

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" :: "r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void fence_barrier_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ unsigned long long global_ns() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile("{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\tselp.u32 %0, 1, 0, p;\n\t}"
                 : "=r"(ok) : "r"(bar), "r"(parity) : "memory");
    return ok != 0;
}
// try_wait that lets the hardware suspend the thread for up to `hint` ns while
// the phase is incomplete (it resumes as soon as the phase completes), so a
// waiting warp issues a handful of instructions per wait instead of spinning.
constexpr uint32_t SUSPEND_HINT_NS = 20000;
__device__ __forceinline__ bool mbar_try_wait_sleep(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile("{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\tselp.u32 %0, 1, 0, p;\n\t}"
                 : "=r"(ok) : "r"(bar), "r"(parity), "n"(SUSPEND_HINT_NS) : "memory");
    return ok != 0;
}
__device__ __forceinline__ int lds_volatile(uint32_t addr) {
    int v;
    asm volatile("ld.volatile.shared.u32 %0, [%1];" : "=r"(v) : "r"(addr) : "memory");
    return v;
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" :: "r"(bar) : "memory");
}
// Wait until the barrier's phase with this parity completes. False when the
// wait ran out or the block's abort flag (shared address abort_addr) is up.
// A role off the critical path passes nap_ns > 0 to sleep between polls.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, uint32_t abort_addr, uint32_t nap_ns) {
    if (mbar_try_wait(bar, parity)) return true;
    const unsigned long long t0 = global_ns();
    while (!mbar_try_wait_sleep(bar, parity)) {
        if (nap_ns) __nanosleep(nap_ns);
        if (lds_volatile(abort_addr) || global_ns() - t0 > WAIT_LIMIT_NS) return false;
    }
    return true;
}
// mbar_wait by a whole warp, with one verdict for all lanes (the roles' code
// after a wait uses full-warp shuffles and must not diverge on it).
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, uint32_t abort_addr, uint32_t nap_ns = 0) {
    return __all_sync(0xffffffffu, mbar_wait(bar, parity, abort_addr, nap_ns));
}
// Plain bounded wait (no abort flag), for the copier's final drain.
__device__ __forceinline__ bool mbar_wait_bounded(uint32_t bar, uint32_t parity) {
    const unsigned long long t0 = global_ns();
    while (!mbar_try_wait_sleep(bar, parity)) {
        if (global_ns() - t0 > WAIT_LIMIT_NS) return false;
    }
    return true;
}
__device__ __forceinline__ void raise_abort(int* abort_flag) {
    atomicOr(&g_device_status, VBQ_DEVICE_TIMEOUT);
    *reinterpret_cast<volatile int*>(abort_flag) = 1;
}
// One thread: expect `bytes` on the barrier and start the bulk copy.
__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" :: "r"(bar), "r"(bytes) : "memory");
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                 :: "r"(dst), "l"(src), "r"(bytes), "r"(bar) : "memory");
}

__device__ __forceinline__ void issue_unit(const LayoutView& L, int u, uint32_t dst, uint32_t bar) {
    const uint32_t o0 = L.blob_off[u], o1 = L.blob_off[u + 1];
    bulk_load(dst, L.blobs + (int64_t)o0 * 16, (o1 - o0) * 16, bar);
}

// Split-K: true once every row block this block adds a slab s > 0 into has
// been zeroed in this call (flag == epoch), within the wait limit. A whole warp:
// lane i watches units u_begin + i, + 32, ..., so one round trip covers them
// all; the flags are read with acquire loads.
__device__ __forceinline__ bool split_k_flags_ready(const LayoutView& L, uint32_t epoch, int u_begin, int u_end,
                                                    int lane) {
    bool seen = true;
    const unsigned long long t0 = global_ns();
    for (int u = u_begin + lane; u < u_end && seen; u += 32) {
        if (u >= L.nrb) {               // slab > 0
            const uint32_t* f = L.ctl + 2 + (u % L.nrb);
            while (!(seen = ld_acquire_gpu(f) == epoch))
                if (global_ns() - t0 > WAIT_LIMIT_NS) break;
        }
    }
    __syncwarp();                       // every lane's later additions after every acquire
    return __all_sync(0xffffffffu, seen);
}

}  // namespace
}  // namespace vbq
