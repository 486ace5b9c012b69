// vbq_gemv.cu — fused dequantise-and-multiply y = W x over the packed layout
// (§6: load the packed low-bit bytes of a group, expand them in registers with
// the group's scale, accumulate the matrix-vector product; the wide weights
// never reach memory).
//
// Batch 1 (gemv1_kernel): a persistent grid of three blocks per SM. Block p
// owns a contiguous range of units in slab-major order, so consecutive units
// share their activations. Unit blobs stream into two shared-memory stages
// with cp.async (the next unit loads while the current one is computed).
// Per slab the block stages x as fp32 and builds, for every 4 consecutive
// weights of a group column, the 16 subset sums of their activations (a
// lookup table indexed by 4 code bits). Per unit, the four widths are split
// into warp tasks:
//   b = 1  one table lookup per 4 weights: S = sum of x over set bits, and
//          the group's dot product is 2S - X (L_1(u) = 2u - 1, X = sum of x);
//   b = 2  the two bit planes use the same tables: S0 + 2 S1 - 2X;
//   b = 4  codes are masked in place and read as exact denormal floats
//          against activations pre-scaled per code slot (packed f32x2 FMAs);
//          8X (summed in the same order) is subtracted for the zero level;
//   b = 8  same with a byte permute and 2^23 + 128.
// X is summed from the tables in the same order as the lookups, so a group
// whose codes are all at the zero level contributes exactly 0. Each group's
// fp32 dot product is scaled once by its FP16 scale and added to its row's
// shared-memory partial; a unit's rows then go to y directly (one slab per
// row) or through the layout's split-K workspace (several slabs).
//
// Batch 2..16 (gemm_kernel<NB>): one block per unit, one thread per group,
// plain fp32 FMAs per code and per activation row.
#include <cstddef>
#include <mutex>

#include "vbq_kernels.h"

namespace vbq {
namespace {

constexpr int THREADS = 256;
constexpr int WARPS = THREADS / 32;
constexpr int XQ = 20;                   // floats per 16-code quarter of x (16 + 4 pad: quarters use other banks)
constexpr int XH = 36;                   // floats per 32-code half of the pre-scaled x (32 + 4 pad)
constexpr int LUT_COL_BYTES = 1088;      // 16 tables x 64 bytes + 64: neighbouring columns use other banks
constexpr int COLARR_BYTES = MAX_UNIT_ITEMS + 64;
constexpr int STAGE_BYTES = MAX_BLOB_BYTES;   // holds the largest unit blob (the packer guarantees it)

struct __align__(16) Tables {
    uint8_t lut[MAX_C * LUT_COL_BYTES];  // column c, nibble j, entry m at c*1088 + j*64 + m*4
    float xs[MAX_C * 4 * XQ];            // x as fp32; quarter (c, q) at (c*4 + q) * XQ
    float x4s[MAX_C * 2 * XH];           // x pre-scaled per 4-bit nibble slot (see dot4_half); half (c, h) at (c*2 + h) * XH
    float2 x4z[MAX_C][2];                // per column and half: sums of x * 2^-100, even / odd codes
    float xlut[MAX_C];                   // per column: sum of the all-ones entries, in lookup order
    float ys[2][RB];                     // row partials of the current and the previous unit
    unsigned long long bar[2];           // one mbarrier per stage
    alignas(16) uint8_t colarr[2][COLARR_BYTES];       // column of every item of the last two units (16-byte stores)
    uint32_t epoch;                      // this call's epoch (split-K y zeroing)
    int flag_ok;
};
static_assert(offsetof(Tables, colarr) % 16 == 0, "colarr takes 16-byte stores");
static_assert(offsetof(Tables, bar) % 8 == 0, "mbarriers are 8-byte aligned");
static_assert(offsetof(Tables, lut) == 0, "tables start at the aligned base");
static_assert(RB <= THREADS, "one thread per row writes a unit's rows");

constexpr size_t GEMV1_SMEM = 128 /* alignment slack */ + 2 * STAGE_BYTES + sizeof(Tables);
// three blocks per SM: 3 x (GEMV1_SMEM + 1 KB reserved per block) must fit in 228 KB
static_assert(3 * (GEMV1_SMEM + 1024) <= 228 * 1024, "three blocks per SM");

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

template <int OFF>
__device__ __forceinline__ float lds_f32(uint32_t addr) {
    float v;
    asm("ld.shared.f32 %0, [%1+%2];" : "=f"(v) : "r"(addr), "n"(OFF));
    return v;
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

__device__ __forceinline__ uint32_t lds_u32(uint32_t addr) {
    uint32_t v;
    asm("ld.shared.u32 %0, [%1];" : "=r"(v) : "r"(addr));
    return v;
}

__device__ __forceinline__ float2 f2(float a, float b) { return make_float2(a, b); }

// Byte offset of nibble I (0..7) of w, scaled by 4 (a table entry is 4 bytes).
template <int I>
__device__ __forceinline__ uint32_t nib4(uint32_t w) {
    return (I == 0 ? (w << 2) : (w >> (4 * I - 2))) & 0x3Cu;
}

// Sum over the 16 nibbles of a 64-bit bit plane (words lo, hi) of the table
// entries they select; tb = shared address of the column's tables. The 16
// lookups are added as a balanced tree (pairs, then pairs of pairs), the same
// tree that builds xlut.
__device__ __forceinline__ float tree16(const float* v) {
    const float a0 = v[0] + v[1], a1 = v[2] + v[3], a2 = v[4] + v[5], a3 = v[6] + v[7];
    const float a4 = v[8] + v[9], a5 = v[10] + v[11], a6 = v[12] + v[13], a7 = v[14] + v[15];
    return ((a0 + a1) + (a2 + a3)) + ((a4 + a5) + (a6 + a7));
}

__device__ __forceinline__ float plane_sum(uint32_t tb, uint32_t lo, uint32_t hi) {
    float v[16];
    v[0] = lds_f32<0>(nib4<0>(lo) | tb);
    v[1] = lds_f32<64>(nib4<1>(lo) | tb);
    v[2] = lds_f32<128>(nib4<2>(lo) | tb);
    v[3] = lds_f32<192>(nib4<3>(lo) | tb);
    v[4] = lds_f32<256>(nib4<4>(lo) | tb);
    v[5] = lds_f32<320>(nib4<5>(lo) | tb);
    v[6] = lds_f32<384>(nib4<6>(lo) | tb);
    v[7] = lds_f32<448>(nib4<7>(lo) | tb);
    v[8] = lds_f32<512>(nib4<0>(hi) | tb);
    v[9] = lds_f32<576>(nib4<1>(hi) | tb);
    v[10] = lds_f32<640>(nib4<2>(hi) | tb);
    v[11] = lds_f32<704>(nib4<3>(hi) | tb);
    v[12] = lds_f32<768>(nib4<4>(hi) | tb);
    v[13] = lds_f32<832>(nib4<5>(hi) | tb);
    v[14] = lds_f32<896>(nib4<6>(hi) | tb);
    v[15] = lds_f32<960>(nib4<7>(hi) | tb);
    return tree16(v);
}

// 4-bit, half a group per lane (32 codes: four words of LSB-first nibbles).
// Codes are masked in place: (w & 0xF << 4i) read as a float is exactly
// u * 2^(4i - 149) for nibbles whose top bit is at most bit 23 (a set bit 23 is
// the implicit leading one of a normal number, which keeps the value linear in
// u). The top two nibbles are shifted down first. Activations come pre-scaled
// per nibble slot (x4s[j] = x_j * 2^(49 - e_j), e_j the slot's shift), so each
// product is exactly u * x * 2^-100. Two f32x2 chains (words 0, 2 and 1, 3)
// add even codes in .x and odd codes in .y; x4z holds the same sums of x.
__device__ __forceinline__ float2 dot4_half(uint4 v, uint32_t xa) {
    float2 ca = f2(0.f, 0.f), cb = f2(0.f, 0.f);
    const uint32_t words[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int t = 0; t < 4; ++t) {
        const uint32_t w = words[t], w2 = w >> 24;
        const float4 xa4 = lds_f32x4(xa + t * 32), xb4 = lds_f32x4(xa + t * 32 + 16);
        float2& c = (t & 1) ? cb : ca;
        c = __ffma2_rn(f2(__uint_as_float(w & 0xFu), __uint_as_float(w & 0xF0u)), f2(xa4.x, xa4.y), c);
        c = __ffma2_rn(f2(__uint_as_float(w & 0xF00u), __uint_as_float(w & 0xF000u)), f2(xa4.z, xa4.w), c);
        c = __ffma2_rn(f2(__uint_as_float(w & 0xF0000u), __uint_as_float(w & 0xF00000u)), f2(xb4.x, xb4.y), c);
        c = __ffma2_rn(f2(__uint_as_float(w2 & 0xFu), __uint_as_float(w2 & 0xF0u)), f2(xb4.z, xb4.w), c);
    }
    return __fadd2_rn(ca, cb);
}

// 8-bit, a quarter group per lane (16 codes): codes expand to exact floats
// 2^23 + u by a byte permute, 2^23 + 128 is subtracted exactly, packed f32x2
// FMAs accumulate in two chains.
__device__ __forceinline__ float dot8_quarter(uint4 v, uint32_t xa) {
    const float2 off = f2(-8388736.f, -8388736.f);          // -(2^23 + 128)
    const uint32_t M = 0x4B000000u;
    float2 ca = f2(0.f, 0.f), cb = f2(0.f, 0.f);
    const uint32_t words[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int t = 0; t < 4; ++t) {
        const uint32_t w = words[t];
        const float4 x4 = lds_f32x4(xa + t * 16);
        const float2 l0 = __fadd2_rn(f2(__uint_as_float(__byte_perm(w, M, 0x7540)),
                                        __uint_as_float(__byte_perm(w, M, 0x7541))), off);
        const float2 l1 = __fadd2_rn(f2(__uint_as_float(__byte_perm(w, M, 0x7542)),
                                        __uint_as_float(__byte_perm(w, M, 0x7543))), off);
        ca = __ffma2_rn(l0, f2(x4.x, x4.y), ca);
        cb = __ffma2_rn(l1, f2(x4.z, x4.w), cb);
    }
    return (ca.x + ca.y) + (cb.x + cb.y);
}

__device__ __forceinline__ uint32_t ld_volatile(const uint32_t* p) {
    return *reinterpret_cast<const volatile uint32_t*>(p);
}
__device__ __forceinline__ void st_volatile(uint32_t* p, uint32_t v) {
    *reinterpret_cast<volatile uint32_t*>(p) = v;
}

__device__ __forceinline__ float half_bits(uint32_t bits) { return __half2float(__ushort_as_half((uint16_t)bits)); }

// ---------------------------------------------------------------------------
// Unit blobs arrive by TMA bulk copy, completion tracked by one mbarrier per
// stage. Every wait is bounded: after about a second the block records
// VBQ_DEVICE_TIMEOUT in g_device_status and stops.
// ---------------------------------------------------------------------------

__device__ uint32_t g_device_status;
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
// Wait until the barrier's phase with this parity completes; false on timeout.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity) {
    if (mbar_try_wait(bar, parity)) return true;
    const unsigned long long t0 = global_ns();
    while (!mbar_try_wait(bar, parity)) {
        if (global_ns() - t0 > WAIT_LIMIT_NS) return false;
    }
    return true;
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

// Fill colarr[cb + a .. cb + e) with column c: bytes up to a 16-byte boundary,
// 16-byte stores in between, bytes after.
__device__ __forceinline__ void fill_run(uint32_t cb, int a, int e, int c) {
    const uint32_t b4 = 0x01010101u * (uint32_t)c;
    const int a16 = min((a + 15) & ~15, e), e16 = max(e & ~15, a16);
    for (int i = a; i < a16; ++i) asm volatile("st.shared.u8 [%0], %1;" :: "r"(cb + i), "r"(c) : "memory");
    for (int i = a16; i < e16; i += 16)
        asm volatile("st.shared.v4.u32 [%0], {%1, %1, %1, %1};" :: "r"(cb + i), "r"(b4) : "memory");
    for (int i = e16; i < e; ++i) asm volatile("st.shared.u8 [%0], %1;" :: "r"(cb + i), "r"(c) : "memory");
}

// Split-K: true once every row block this block adds a slab s > 0 into has
// been zeroed in this call (flag == epoch), within the wait limit. Thread 0
// only; ends with an acquire fence.
__device__ __forceinline__ bool split_k_flags_ready(const LayoutView& L, uint32_t epoch, int u_begin, int u_end,
                                                    int s0, int rb0) {
    bool seen = true;
    const unsigned long long t0 = global_ns();
    int s2 = s0, rb2 = rb0;
    for (int u = u_begin; u < u_end && seen; ++u) {
        if (s2 > 0) {
            while (!(seen = ld_volatile(L.ctl + 2 + rb2) == epoch))
                if (global_ns() - t0 > WAIT_LIMIT_NS) break;
        }
        if (++rb2 == L.nrb) { rb2 = 0; ++s2; }
    }
    asm volatile("fence.acq_rel.gpu;" ::: "memory");
    return seen;
}

// A finished unit's row partials ys (row block rbw) go to y: stored when the
// row has one slab, added otherwise; ys is zeroed for reuse.
__device__ __forceinline__ void write_rows(const LayoutView& L, float* y, float* ys, int rbw, int tid) {
    if (tid >= RB) return;
    const int rows = min(RB, (int)(L.N - (int64_t)rbw * RB));
    const float v = ys[tid];
    ys[tid] = 0.f;
    if (tid < rows) {
        float* dst = y + (int64_t)rbw * RB + tid;
        if (L.S == 1) *dst = v;
        else atomicAdd(dst, v);
    }
}

__global__ void __launch_bounds__(THREADS, 3) gemv1_kernel(LayoutView L, const uint16_t* __restrict__ x,
                                                           float* __restrict__ y) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    // stages and tables on a 128-byte boundary: lookups OR a nibble offset into table addresses
    unsigned char* base = smem_raw + ((128u - (smem_u32(smem_raw) & 127u)) & 127u);
    Tables& T = *reinterpret_cast<Tables*>(base + 2 * STAGE_BYTES);
    const uint32_t stage0 = smem_u32(base);
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int P = gridDim.x, p = blockIdx.x;
    const int u_begin = (int)((int64_t)L.units * p / P), u_end = (int)((int64_t)L.units * (p + 1) / P);
    if (u_begin >= u_end) return;

    const uint32_t bar0 = smem_u32(&T.bar[0]);
    if (tid == 0) {
        mbar_init(bar0, 1);
        mbar_init(bar0 + 8, 1);
        fence_barrier_init();
    }
    __syncthreads();
    if (tid == 0) {
        issue_unit(L, u_begin, stage0, bar0);
        if (u_begin + 1 < u_end) issue_unit(L, u_begin + 1, stage0 + STAGE_BYTES, bar0 + 8);
    }
    // Weights never depend on earlier work in the stream, so their first copies
    // are in flight before this grid waits for its predecessor (programmatic
    // dependent launch); x, y and the workspace are touched only after the wait.
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    asm volatile("griddepcontrol.wait;" ::: "memory");
    if (L.S > 1) {
        // split-K: this call's epoch; zero y for the row blocks whose slab 0 this
        // block owns (units u < nrb) and publish them
        if (tid == 0) T.epoch = ld_volatile(L.ctl) + 1u;
        const int z_end = min(u_end, L.nrb);
        for (int u = u_begin; u < z_end; ++u) {
            float* dst = y + (int64_t)u * RB;
            const int rows = min(RB, (int)(L.N - (int64_t)u * RB));
            for (int r = tid; r < rows; r += THREADS) dst[r] = 0.f;
        }
        __syncthreads();
        if (tid == 0 && u_begin < z_end) {
            __threadfence();
            for (int u = u_begin; u < z_end; ++u) st_volatile(L.ctl + 2 + u, T.epoch);
        }
    }
    for (int i = tid; i < 2 * RB; i += THREADS) (&T.ys[0][0])[i] = 0.f;

    const uint32_t lut0 = smem_u32(T.lut), xs0 = smem_u32(T.xs), x4s0 = smem_u32(T.x4s);
    const uint32_t x4z0 = smem_u32(T.x4z), xlut0 = smem_u32(T.xlut), cola0 = smem_u32(&T.colarr[0][0]);
    const int s0 = u_begin / L.nrb, rb0 = u_begin - s0 * L.nrb;
    int s = s0, rb = rb0, prev_rb = rb0;
    int cur_slab = -1;
    bool ok = true;
    bool checked = L.S == 1;            // split-K zeroing flags verified (or not needed)
    for (int k = u_begin; k < u_end; ++k) {
        const int j = k - u_begin, buf = j & 1;
        const unsigned char* blob = base + buf * STAGE_BYTES;
        const uint32_t sblob = stage0 + buf * STAGE_BYTES;
        const int cols = min(L.C, L.G - s * L.C);
        float* ys = T.ys[buf];
        const uint32_t cola = cola0 + buf * COLARR_BYTES;

        if (s != cur_slab) {            // activations of a new slab: x, tables, X sums
            const int64_t k0 = (int64_t)s * L.C * GROUP;
            __syncthreads();            // nobody still reads the old tables
            for (int i = tid; i < cols * 32; i += THREADS) {
                const uint32_t two = __ldg(reinterpret_cast<const uint32_t*>(x + k0) + i);
                const float xa = __uint_as_float(two << 16), xb = __uint_as_float(two & 0xFFFF0000u);
                const int kk = 2 * i, c = kk >> 6, jj = kk & 63;
                *reinterpret_cast<float2*>(&T.xs[(c * 4 + (jj >> 4)) * XQ + (jj & 15)]) = f2(xa, xb);
                // 4-bit slot shifts: nibble slots 0..5 of a word keep their place, 6 and 7 come down by 24
                const int slot = jj & 7, e = slot < 6 ? 4 * slot : 4 * (slot - 6);
                *reinterpret_cast<float2*>(&T.x4s[(c * 2 + (jj >> 5)) * XH + (jj & 31)]) =
                    f2(xa * __uint_as_float((uint32_t)(127 + 49 - e) << 23),
                       xb * __uint_as_float((uint32_t)(127 + 49 - e - 4) << 23));
            }
            __syncthreads();
            for (int pj = tid; pj < cols * 16; pj += THREADS) {
                const int c = pj >> 4, jn = pj & 15;
                const float4 xv = *reinterpret_cast<const float4*>(&T.xs[(c * 4 + (jn >> 2)) * XQ + 4 * (jn & 3)]);
                const float t3 = xv.x + xv.y, t12 = xv.w + xv.z;
                float4* dst = reinterpret_cast<float4*>(T.lut + c * LUT_COL_BYTES + jn * 64);
                dst[0] = make_float4(0.f, xv.x, xv.y, t3);
                dst[1] = make_float4(xv.z, xv.z + xv.x, xv.z + xv.y, xv.z + t3);
                dst[2] = make_float4(xv.w, xv.w + xv.x, xv.w + xv.y, xv.w + t3);
                dst[3] = make_float4(t12, t12 + xv.x, t12 + xv.y, t12 + t3);
            }
            __syncthreads();
            if (tid < cols) {
                const float* t = reinterpret_cast<const float*>(T.lut + tid * LUT_COL_BYTES);
                float v[16];
#pragma unroll
                for (int jn = 0; jn < 16; ++jn) v[jn] = t[jn * 16 + 15];
                T.xlut[tid] = tree16(v);
                // X for the 4-bit zero level, summed as dot4_half accumulates
#pragma unroll
                for (int hh = 0; hh < 2; ++hh) {
                    float2 ca = f2(0.f, 0.f), cb = f2(0.f, 0.f);
                    for (int t4 = 0; t4 < 4; ++t4) {
                        float2& cc = (t4 & 1) ? cb : ca;
                        for (int e = 0; e < 8; e += 2) {
                            const int jj = 32 * hh + 8 * t4 + e;
                            const float* xq = &T.xs[(tid * 4 + (jj >> 4)) * XQ + (jj & 15)];
                            cc = __ffma2_rn(f2(xq[0], xq[1]), f2(0x1p-100f, 0x1p-100f), cc);
                        }
                    }
                    T.x4z[tid][hh] = __fadd2_rn(ca, cb);
                }
            }
            cur_slab = s;
        }

        ok = mbar_wait(bar0 + 8 * buf, (j >> 1) & 1);   // unit k's blob has landed (each thread waits)
        const UnitHeader h = *reinterpret_cast<const UnitHeader*>(blob);
        const int n0 = h.n[0], n1 = h.n[1], n2 = h.n[2], n3 = h.n[3];
        const uint32_t cb1 = (n0 + 15) & ~15, cb2 = cb1 + ((n1 + 15) & ~15), cb3 = cb2 + ((n2 + 15) & ~15);
        if (ok && tid < 4 * cols) {     // one thread per (width, column) run
            const uint16_t* cend = reinterpret_cast<const uint16_t*>(blob + h.cc16 * 16);
            const int w = tid / cols, c = tid - w * cols;
            const int a = c == 0 ? 0 : cend[w * L.C + c - 1], e = cend[w * L.C + c];
            const uint32_t cb = cola + (w == 0 ? 0u : w == 1 ? cb1 : w == 2 ? cb2 : cb3);
            fill_run(cb, a, e, c);
        }
        if (!checked && j == 1 && tid == 0) T.flag_ok = split_k_flags_ready(L, T.epoch, u_begin, u_end, s0, rb0);
        // one barrier per unit: unit k's column array is complete and every warp
        // has finished unit k-1, whose stage, rows and partials are now free
        if (!__syncthreads_and(ok)) break;
        if (j >= 1) {
            if (!checked) {
                checked = true;
                if (!T.flag_ok) { ok = false; break; }
            }
            if (tid == 0 && k + 1 < u_end) issue_unit(L, k + 1, stage0 + (buf ^ 1) * STAGE_BYTES, bar0 + 8 * (buf ^ 1));
            write_rows(L, y, T.ys[buf ^ 1], prev_rb, tid);
        }

        // warp tasks: 16 four-bit groups (two lanes each), 8 eight-bit groups
        // (four lanes each), 32 two-bit groups, 64 one-bit groups (two per lane)
        const int t4 = (n2 + 15) >> 4, t8 = (n3 + 7) >> 3, t2 = (n1 + 31) >> 5, t1 = (n0 + 63) >> 6;
        const int ntask = t4 + t8 + t2 + t1;
        for (int t = warp; t < ntask; t += WARPS) {
            if (t < t4) {                                   // 4-bit: two lanes per group, one half each
                // lanes l and l+16 share group l%16; the half is swizzled so that a
                // quarter-warp reads 8 distinct 16-byte bank groups
                const int e = lane & 15, hh = ((e >> 2) + (lane >> 4)) & 1;
                const int i = t * 16 + e;
                float part = 0.f;
                if (i < n2) {
                    const uint4 v = lds_u32x4(sblob + h.pay16[2] * 16 + i * 32 + hh * 16);
                    const int c = lds_u8(cola + cb2 + i);
                    const float2 acc = dot4_half(v, x4s0 + (c * 2 + hh) * XH * 4);
                    const float2 z = lds_f32x2(x4z0 + (c * 2 + hh) * 8);
                    part = (acc.x - 8.f * z.x) + (acc.y - 8.f * z.y);
                }
                part += __shfl_xor_sync(0xffffffffu, part, 16);
                if (i < n2 && lane < 16) {
                    const int r = lds_u8(sblob + h.row16[2] * 16 + i);
                    atomicAdd(&ys[r], (half_bits(lds_u16(sblob + h.sc16[2] * 16 + 2 * i)) * 0x1p100f) * part);
                }
            } else if (t < t4 + t8) {                       // 8-bit: four lanes per group, one quarter each
                // lane 8k + e takes quarter ((e >> 1) + k) % 4 of group e: a quarter-warp
                // reads 8 distinct 16-byte bank groups
                const int e = lane & 7, q = ((e >> 1) + (lane >> 3)) & 3;
                const int i = (t - t4) * 8 + e;
                float part = 0.f;
                if (i < n3) {
                    const uint4 v = lds_u32x4(sblob + h.pay16[3] * 16 + i * 64 + q * 16);
                    const int c = lds_u8(cola + cb3 + i);
                    part = dot8_quarter(v, xs0 + (c * 4 + q) * XQ * 4);
                }
                part += __shfl_xor_sync(0xffffffffu, part, 8);
                part += __shfl_xor_sync(0xffffffffu, part, 16);
                if (i < n3 && lane < 8) {
                    const int r = lds_u8(sblob + h.row16[3] * 16 + i);
                    atomicAdd(&ys[r], half_bits(lds_u16(sblob + h.sc16[3] * 16 + 2 * i)) * part);
                }
            } else if (t < t4 + t8 + t2) {                  // 2-bit: one group per lane
                const int i = (t - t4 - t8) * 32 + lane;
                if (i < n1) {
                    const uint4 pl = lds_u32x4(sblob + h.pay16[1] * 16 + i * 16);
                    const int c = lds_u8(cola + cb1 + i);
                    const uint32_t tb = lut0 + c * LUT_COL_BYTES;
                    const float s0 = plane_sum(tb, pl.x, pl.y);
                    const float s1 = plane_sum(tb, pl.z, pl.w);
                    const int r = lds_u8(sblob + h.row16[1] * 16 + i);
                    atomicAdd(&ys[r], half_bits(lds_u16(sblob + h.sc16[1] * 16 + 2 * i)) *
                                          (s0 + 2.f * (s1 - lds_f32r(xlut0 + 4 * c))));
                }
            } else {                                        // 1-bit: two groups per lane
                const int i = (t - t4 - t8 - t2) * 64 + 2 * lane;
                if (i < n0) {
                    const uint4 v = lds_u32x4(sblob + h.pay16[0] * 16 + i * 8);
                    const uint32_t rows2 = lds_u16(sblob + h.row16[0] * 16 + i);
                    const uint32_t sc2 = lds_u32(sblob + h.sc16[0] * 16 + 2 * i);
                    const uint32_t cols2 = lds_u16(cola + i);
                    const int ca = cols2 & 0xff;
                    const float suma = plane_sum(lut0 + ca * LUT_COL_BYTES, v.x, v.y);
                    if (i + 1 < n0) {
                        const int cb = cols2 >> 8;
                        const float sumb = plane_sum(lut0 + cb * LUT_COL_BYTES, v.z, v.w);
                        atomicAdd(&ys[rows2 >> 8], half_bits(sc2 >> 16) * (2.f * sumb - lds_f32r(xlut0 + 4 * cb)));
                    }
                    atomicAdd(&ys[rows2 & 0xff], half_bits(sc2) * (2.f * suma - lds_f32r(xlut0 + 4 * ca)));
                }
            }
        }
        prev_rb = rb;
        if (++rb == L.nrb) { rb = 0; ++s; }
    }
    if (ok) {                           // the last unit's rows
        if (!checked && tid == 0) T.flag_ok = split_k_flags_ready(L, T.epoch, u_begin, u_end, s0, rb0);
        __syncthreads();
        if (!checked && !T.flag_ok) ok = false;
        else write_rows(L, y, T.ys[(u_end - 1 - u_begin) & 1], prev_rb, tid);
    }
    if (!ok) {
        // a copy or a flag never arrived: record it, give the outstanding copies a
        // bounded time to land, and stop
        if (tid == 0) {
            atomicOr(&g_device_status, VBQ_DEVICE_TIMEOUT);
            mbar_wait(bar0, 0);
            mbar_wait(bar0 + 8, 0);
        }
    }
    if (L.S > 1 && tid == 0) {
        // the last block of the call advances the epoch for the next call
        __threadfence();
        if (atomicAdd(L.ctl + 1, 1u) == gridDim.x - 1) {
            st_volatile(L.ctl + 1, 0u);
            st_volatile(L.ctl, T.epoch);
        }
    }
}

// ---------------------------------------------------------------------------
// Batch 2..16: one block per unit, one thread per group.
// ---------------------------------------------------------------------------

template <int B, int NB>
__device__ __forceinline__ void dot_item(const uint8_t* __restrict__ src, const float* __restrict__ xs,
                                         int xstride, int nb, float* acc) {
    uint32_t w[2 * B];
    load_item<B>(src, w);
#pragma unroll
    for (int j = 0; j < GROUP; ++j) {
        const float lv = (float)level_of<B>(item_code<B>(w, j));
#pragma unroll
        for (int q = 0; q < NB; ++q)
            if (q < nb) acc[q] = fmaf(lv, xs[q * xstride + j], acc[q]);
    }
}

template <int NB>
__global__ void __launch_bounds__(THREADS) gemm_kernel(LayoutView L, const uint16_t* __restrict__ X,
                                                       float* __restrict__ Y, int nb) {
    extern __shared__ float4 smem_f4[];
    float* xs = reinterpret_cast<float*>(smem_f4);                 // [NB][C*64]
    __shared__ UnitHeader h;
    __shared__ float ys[NB][RB];

    const int u = blockIdx.x, rb = unit_rb(L, u), s = unit_slab(L, u);
    const int rows = unit_rows(L, rb), cols = unit_cols(L, s);
    const int xstride = L.C * GROUP;
    const int64_t k0 = (int64_t)s * L.C * GROUP;
    const uint8_t* blob = L.blobs + (int64_t)L.blob_off[u] * 16;

    if (threadIdx.x == 0) h = *reinterpret_cast<const UnitHeader*>(blob);
    for (int i = threadIdx.x; i < nb * cols * GROUP; i += blockDim.x) {
        const int q = i / (cols * GROUP), k = i - q * cols * GROUP;
        const uint32_t bits = X[(int64_t)q * L.K + k0 + k];
        xs[q * xstride + k] = __uint_as_float(bits << 16);
    }
    for (int i = threadIdx.x; i < NB * RB; i += blockDim.x) (&ys[0][0])[i] = 0.f;
    __syncthreads();
    const uint16_t* cend = reinterpret_cast<const uint16_t*>(blob + h.cc16 * 16);
    const int total = h.n[0] + h.n[1] + h.n[2] + h.n[3];
    for (int i = threadIdx.x; i < total; i += blockDim.x) {
        int w = 0, j = i;
        while (w < 3 && j >= h.n[w]) { j -= h.n[w]; ++w; }
        const int c = column_of(cend + w * L.C, cols, 0, j);
        const int r = blob[h.row16[w] * 16 + j];
        const float sf = __half2float(__ushort_as_half(reinterpret_cast<const uint16_t*>(blob + h.sc16[w] * 16)[j]));
        const uint8_t* pay = blob + h.pay16[w] * 16;
        float acc[NB];
#pragma unroll
        for (int q = 0; q < NB; ++q) acc[q] = 0.f;
        const float* xc = xs + c * GROUP;
        switch (w) {
            case 0: dot_item<1, NB>(pay + j * 8, xc, xstride, nb, acc); break;
            case 1: dot_item<2, NB>(pay + j * 16, xc, xstride, nb, acc); break;
            case 2: dot_item<4, NB>(pay + j * 32, xc, xstride, nb, acc); break;
            default: dot_item<8, NB>(pay + j * 64, xc, xstride, nb, acc); break;
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
    static bool attr_set = false;           // the attribute is per function; set once per process
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(gemm_kernel<NB>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)(NB * MAX_C * GROUP * sizeof(float)));
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    gemm_kernel<NB><<<L.units, THREADS, dyn, s>>>(L, X, Y, B);
    return cudaGetLastError();
}

int g_sms = 0;

cudaError_t launch_gemv1(const LayoutView& L, const uint16_t* x, float* y, cudaStream_t s) {
    static bool attr_set = false;
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(gemv1_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)GEMV1_SMEM);
        if (e != cudaSuccess) return e;
        int dev = 0;
        if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
        if ((e = cudaDeviceGetAttribute(&g_sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
        attr_set = true;
    }
    const int grid = L.units < 3 * g_sms ? L.units : 3 * g_sms;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(THREADS);
    cfg.dynamicSmemBytes = GEMV1_SMEM;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cudaError_t e = cudaLaunchKernelEx(&cfg, gemv1_kernel, L, x, y);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace

// ---------------------------------------------------------------------------
// Batch 1 with the split-K control words in a fixed device array instead of
// the layout's own allocation (for callers that cannot allocate device
// memory; see vbq_gemv_static in vbq.h). Every call on a device shares the
// array: word 0 is the call epoch, word 1 the count of finished blocks
// (cleared on the stream before every launch), words 2.. the per-row-block
// zeroed flags. Epochs only grow, so flags left by earlier calls never match
// the current one. Calls that overlap on the GPU race on the array.
// ---------------------------------------------------------------------------

static __device__ __align__(256) uint32_t g_static_ctl[STATIC_CTL_WORDS];

cudaError_t launch_gemv1_static(const LayoutView& L, const uint16_t* x, float* y, cudaStream_t s) {
    constexpr int MAX_DEVICES = 64;
    static std::mutex mu;
    static uint32_t* addr[MAX_DEVICES] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= MAX_DEVICES) return cudaErrorInvalidDevice;
    uint32_t* ctl;
    {
        std::lock_guard<std::mutex> lock(mu);
        if (!addr[dev]) {       // once per device, with that device current
            void* p = nullptr;
            if ((e = cudaGetSymbolAddress(&p, g_static_ctl)) != cudaSuccess) return e;
            addr[dev] = static_cast<uint32_t*>(p);
        }
        ctl = addr[dev];
    }
    if ((e = cudaMemsetAsync(ctl + 1, 0, sizeof(uint32_t), s)) != cudaSuccess) return e;
    LayoutView Ls = L;
    Ls.ctl = ctl;
    return launch_gemv1(Ls, x, y, s);
}

cudaError_t launch_gemv(const LayoutView& L, const uint16_t* X, float* Y, int B, cudaStream_t s) {
    if (B <= 1) return launch_gemv1(L, X, Y, s);
    if (B <= 2) return launch_nb<2>(L, X, Y, B, s);
    if (B <= 4) return launch_nb<4>(L, X, Y, B, s);
    if (B <= 8) return launch_nb<8>(L, X, Y, B, s);
    return launch_nb<16>(L, X, Y, B, s);
}

}  // namespace vbq
