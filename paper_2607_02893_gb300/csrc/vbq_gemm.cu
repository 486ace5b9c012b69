// vbq_gemm.cu — batched product Y = X W^T for 2..16 activation rows (§6's
// fused dequantise-and-multiply, several tokens at once) on the tensor cores.
//
// With B activation rows every decoded weight is used B times, so the product
// is a dense contraction over dequantised tiles: here mma.sync m16n8k16 with
// fp16 operands and fp32 accumulators. The operands are arranged so that the
// packed bits go into A fragments with masks and byte permutes only:
//
//   A (16 x 16 per k-step) = sixteen items (groups) of one width and one
//       column: lane (g, t) decodes items g and g + 8, holding each item's
//       weights 16t + rho (low half) and 16t + 8 + rho (high half) in register
//       rho. Any fixed assignment of the 64 weights of a group to the MMA's k
//       positions gives the same sum, as long as B uses the same one; this
//       one lets every width expand with one or two instructions per register
//       into exact fp16 denormals u * 2^-24. One more packed fp16 subtraction
//       (a fused 2u - 1 for one bit) turns u * 2^-24 into L(u) * 2^-24,
//       exactly (every value is an integer times the smallest fp16 denormal,
//       and fp16 arithmetic keeps denormals).
//   B (16 x 8 per k-step) = activations: column n = batch row n (8 per MMA;
//       two MMAs per k-step for more than 8 rows; rows >= B are zero),
//       pre-scaled per (batch row, group column) by 2^(24 - E), E set from the
//       largest |x| of that column so every value stays in fp16 range; built
//       once per slab into shared memory, one fragment set per column and lane.
//   D (16 x 8) = item x batch row: sum over the group of L(u) * x * 2^-E.
//       Every product is exact, so a group whose codes all sit at the zero
//       level gives exactly 0.
//
// The epilogue scales D by the item's FP16 scale and 2^E and adds it to the
// stage's row partials of that batch row; for up to 8 batch rows on layouts
// of 16-column units it stores it instead into the item's own (row, column)
// slot, which the consumers sum per row after the unit (no shared-memory float
// additions, which this GPU runs as compare-and-swap loops). The kernel
// around it is the batch-1 pipeline: one persistent block per SM, a copier
// warp streaming unit blobs by TMA bulk copies into shared-memory stages and
// writing row partials to Y (in the slot form the consumers write Y), consumer
// warps in teams, two mbarriers per stage, split-K y zeroing by epoch-tagged
// flags (see vbq_gemv.cu).
#include <cstddef>

#include "vbq_kernels.h"
#include "vbq_device.cuh"

namespace vbq {
namespace {

constexpr int NCWB = 16;                 // consumer warps
constexpr int NCTB = 32 * NCWB;
constexpr int GB_THREADS = 32 * (NCWB + 1);
constexpr int STAGE_BYTES_B = MAX_BLOB_BYTES;
// Row partials of one batch row take RB + 4 floats: each batch row starts on
// a 16-byte boundary (the flush moves 4 rows per lane), and the same row of
// eight batch rows (the eight lane groups of an epilogue store) falls in
// banks 4 apart.
constexpr int YS_STRIDE = RB + 4;
static_assert(YS_STRIDE % 4 == 0 && RB == 32 * 4, "a warp flushes a batch row's 128 partials 4 per lane");
// Stages and consumer teams. With row partials, NB = 8 leaves room for four
// stages and up to two teams (a team's next blob lands while it works on the
// current one); NB = 16 for three stages and one team. The slot form (SL, NB =
// 8 only) stores into slots (one per row, group column and batch row: each row
// of a unit has exactly one group per column) instead of adding into row
// partials: shared-memory float additions are compare-and-swap loops on this
// GPU (about 7 instructions and 2.6 times a plain store each, measured), and
// they were a third of the kernel's time. The slots take 64 KB, the room of a
// fourth stage, and one team flushes them after every unit, so the slot form
// pays on wide units only; NB = 16 would need 128 KB and keeps the row partials.
constexpr int SLOT_MIN_C = 16;          // the slot form for units of at least this many columns
template <int NB, bool SL> struct Pipe {
    static_assert(!SL || NB == 8, "slots for 8 batch rows only");
    static constexpr int stages = NB == 8 && !SL ? 4 : 3, max_teams = NB == 8 && !SL ? 2 : 1;
};
static_assert(Pipe<8, false>::stages % Pipe<8, false>::max_teams == 0 && Pipe<16, false>::stages % Pipe<16, false>::max_teams == 0,
              "each team's units use stages no other team uses");
static_assert(STAGE_BYTES_B % 256 == 0, "stage alignment");

// Shared-memory tables of the batched kernel; NB = 8 or 16 A rows: the
// slab's activation tables, then the pipeline's state (SL: the slot form).
template <int NB>
struct __align__(16) ActTables {
    uint32_t xfr[MAX_C][NB / 4][32][4];  // activation (B) fragments (fp16x2) per column, register quad and lane: a warp's
                                         // 16-byte loads of one quad read 512 contiguous bytes
    uint16_t xb[NB][MAX_C * GROUP];      // the slab's activations (BF16 bits), rows >= B zero
    float e2[MAX_C][16];                 // per column and batch row: 2^E (0 for absent rows)
    float fx[MAX_C][16];                 // per column and batch row: 2^(24 - E), the activations' prescale
};
template <int NB, bool SL>
struct __align__(16) TablesB : ActTables<NB> {
    float ys[SL ? 1 : Pipe<NB, SL>::stages][NB][YS_STRIDE];   // row partials of each stage, per batch row
    float sl[SL ? RB * MAX_C * 8 : 4];                        // SL: the current unit's slots (slot_index)
    unsigned long long full[Pipe<NB, SL>::stages];            // blob landed
    unsigned long long empty[Pipe<NB, SL>::stages];           // the unit's team is done
    int abort;
    uint32_t sk_ok;                                           // SL: the copier's split-K flag check, passed on
};

template <int NB, bool SL>
constexpr size_t gemmb_smem() { return 256 + (size_t)Pipe<NB, SL>::stages * STAGE_BYTES_B + sizeof(TablesB<NB, SL>); }
static_assert(gemmb_smem<16, false>() <= 227 * 1024 && gemmb_smem<8, false>() <= 227 * 1024 &&
              gemmb_smem<8, true>() <= 227 * 1024, "one block per SM");

// Slot of row r, group column c and batch row b (NB = 8): a row's 16 columns x
// 8 batch rows are 128 contiguous floats, its columns XOR-swizzled by the row's
// low bits, so the 8-byte stores of four items of one column (a half-warp of
// the epilogue) fall in four distinct groups of 8 banks when their rows differ
// in their low two bits.
__host__ __device__ constexpr uint32_t slot_index(uint32_t r, uint32_t c, uint32_t b) {
    return r * (MAX_C * 8) + ((c ^ (r & (MAX_C - 1))) << 3) + b;
}


__device__ __forceinline__ void consumer_sync_b() {
    asm volatile("bar.sync 1, %0;" :: "n"(NCTB) : "memory");
}

__device__ __forceinline__ void mma16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
    asm("mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
                 : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
                 : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// The same with a zero accumulator (the first k-step of a tile).
__device__ __forceinline__ void mma16816_z(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
    asm("mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%10,%10,%10,%10};"
                 : "=f"(d[0]), "=f"(d[1]), "=f"(d[2]), "=f"(d[3])
                 : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1), "f"(0.f));
}

__device__ __forceinline__ float bf16_bits(uint32_t b) { return __uint_as_float(b << 16); }

// y[0..3] += v as one vector reduction (16-byte aligned address).
__device__ __forceinline__ void red_global_v4(float* p, float4 v) {
    asm volatile("red.global.add.v4.f32 [%0], {%1, %2, %3, %4};" :: "l"(p), "f"(v.x), "f"(v.y), "f"(v.z), "f"(v.w)
                 : "memory");
}

__device__ __forceinline__ void sts_f32x2(uint32_t addr, float2 v) {
    asm volatile("st.shared.v2.f32 [%0], {%1, %2};" :: "r"(addr), "f"(v.x), "f"(v.y) : "memory");
}

// red_shared at a constant offset of OFF floats from addr.
template <int OFF>
__device__ __forceinline__ void red_shared_off(uint32_t addr, float v) {
    asm volatile("red.shared.add.f32 [%0+%2], %1;" :: "r"(addr), "f"(v), "n"(OFF * 4) : "memory");
}

// Per slab: E and the activation fragments of every column.
// Consumer threads only (ct = 0 .. NCTB-1); starts and ends with a consumer barrier.
// Kept out of line: inlined, it changed the register allocation of the tile
// loops (measured up to 20% slower on all-4-bit matrices).
// The slab's activations are first staged in shared memory with every thread's
// 16-byte loads in flight at once (the table build is on the path of every
// unit of the slab, so its latency counts, not its instructions).
template <int NB>
__device__ __noinline__ void build_tables_b(ActTables<NB>& T, const LayoutView& L, const uint16_t* __restrict__ X, int B, int s,
                               int ct) {
    constexpr int ROW_CHUNKS = MAX_C * GROUP / 8;                 // 16-byte chunks of one staged row
    constexpr int PER = NB * ROW_CHUNKS / NCTB;
    static_assert(PER * NCTB == NB * ROW_CHUNKS, "whole chunks per consumer thread");
    const int cols = min(L.C, L.G - s * L.C);
    const int64_t k0 = (int64_t)s * L.C * GROUP;
    consumer_sync_b();                   // nobody still reads the old tables
    {
        uint4 v[PER];
#pragma unroll
        for (int i = 0; i < PER; ++i) {
            const int q = ct + i * NCTB, b = q / ROW_CHUNKS, o = q - b * ROW_CHUNKS;
            v[i] = make_uint4(0u, 0u, 0u, 0u);
            if (b < B && o < cols * (GROUP / 8))
                v[i] = __ldg(reinterpret_cast<const uint4*>(X + (int64_t)b * L.K + k0) + o);
        }
#pragma unroll
        for (int i = 0; i < PER; ++i) *reinterpret_cast<uint4*>(&T.xb[0][0] + (size_t)(ct + i * NCTB) * 8) = v[i];
    }
    consumer_sync_b();
    // two threads per (column, batch row < NB): the largest |x| of the column's 64
    // values, as BF16 magnitude bits (ordered like the magnitudes), and from
    // its exponent ex: E = ex + 11, so |x| * 2^(24 - E) < 2^14 fits fp16.
    // E is held in [-100, 127] so that 2^E and 2^(24 - E) stay normal floats
    // (a column of values below 2^-111 then keeps fewer fp16 bits, far below
    // the accuracy bound's absolute term; values of 2^116 and more overflow).
    {
        const int pr = ct >> 1, c = pr / NB, b = pr % NB;         // c < 256 / NB, every column of the slab
        uint32_t m = 0;
        if (c < cols) {
            const uint4* src = reinterpret_cast<const uint4*>(&T.xb[b][c * GROUP + 32 * (ct & 1)]);
            uint32_t m2 = 0;
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const uint4 w = src[q];
                m2 = __vmaxu2(m2, __vmaxu2(w.x & 0x7FFF7FFFu, w.y & 0x7FFF7FFFu));
                m2 = __vmaxu2(m2, __vmaxu2(w.z & 0x7FFF7FFFu, w.w & 0x7FFF7FFFu));
            }
            m = max(m2 & 0xFFFFu, m2 >> 16);
        }
        m = max(m, __shfl_xor_sync(0xffffffffu, m, 1));
        const int ef = (int)(m >> 7);                             // biased exponent of max |x| (0: zero or subnormal)
        const int E = min(max(ef - 127 + 11, -100), 127);
        if (c < cols && (ct & 1) == 0) {
            T.e2[c][b] = b < B ? __uint_as_float((uint32_t)(127 + E) << 23) : 0.f;
            T.fx[c][b] = __uint_as_float((uint32_t)(127 + 24 - E) << 23);
        }
    }
    consumer_sync_b();
    // Activation fragments: register r of lane (g, t) for column c. NB = 16:
    // k-step s = r / 4, q = r % 4 -> (batch row g + 8 (q & 1), half h = q >> 1);
    // NB = 8: s = r / 2, h = r % 2, batch row g. Register pair (rho = 2s + h):
    // the row's activations at weights 16t + rho (low) and 16t + 8 + rho (high)
    // of the column.
    for (int p = ct; p < cols * 32 * NB; p += NCTB) {
        const int r = p % NB, l = (p / NB) & 31, c = p / (NB * 32);
        const int g = l >> 2, t = l & 3;
        int s2, h, row;
        if (NB == 16) { s2 = r >> 2; h = (r >> 1) & 1; row = g + 8 * (r & 1); }
        else { s2 = r >> 1; h = r & 1; row = g; }
        const int rho = 2 * s2 + h;
        const float f = T.fx[c][row];
        const uint16_t* xr = &T.xb[row][c * GROUP + 16 * t + rho];
        const __half2 hv = __floats2half2_rn(bf16_bits(xr[0]) * f, bf16_bits(xr[8]) * f);
        T.xfr[c][r >> 2][l][r & 3] = *reinterpret_cast<const uint32_t*>(&hv);
    }
    consumer_sync_b();
}

// Weight fragments (8 registers, u * 2^-24 per half) of lane t's 16 weights of one item.
__device__ __forceinline__ void bfrag_1(uint2 w, int t, uint32_t (&b)[8]) {
    const uint32_t word = t < 2 ? w.x : w.y;
    const uint32_t lo = 2u * (t & 1), sel = lo | (lo << 4) | ((lo + 1) << 8) | ((lo + 1) << 12);
    const uint32_t W = __byte_perm(word, word, sel);          // field bits 0-7 at 0-7, 8-15 at 16-23
#pragma unroll
    for (int r = 0; r < 8; ++r) b[r] = (W >> r) & 0x00010001u;
}
__device__ __forceinline__ void bfrag_2(uint4 w, int t, uint32_t (&b)[8]) {
    const uint32_t lo = 2u * (t & 1), sel = lo | (lo << 4) | ((lo + 1) << 8) | ((lo + 1) << 12);
    const uint32_t W0 = __byte_perm(t < 2 ? w.x : w.y, t < 2 ? w.x : w.y, sel);   // bit plane 0
    const uint32_t W1 = __byte_perm(t < 2 ? w.z : w.w, t < 2 ? w.z : w.w, sel);   // bit plane 1
    b[0] = (W0 & 0x00010001u) | ((W1 << 1) & 0x00020002u);
#pragma unroll
    for (int r = 1; r < 8; ++r) b[r] = ((W0 >> r) & 0x00010001u) | ((W1 >> (r - 1)) & 0x00020002u);
}
__device__ __forceinline__ void bfrag_4(uint2 w, uint32_t (&b)[8]) {   // w = words 2t, 2t+1 of the item
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const uint32_t V = __byte_perm(w.x, w.y, q | (q << 4) | ((4 + q) << 8) | ((4 + q) << 12));
        b[2 * q] = V & 0x000F000Fu;
        b[2 * q + 1] = (V >> 4) & 0x000F000Fu;
    }
}
__device__ __forceinline__ void bfrag_8(uint4 w, uint32_t (&b)[8]) {   // w = words 4t .. 4t+3 of the item
    const uint32_t words[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int r = 0; r < 8; ++r) {
        const uint32_t q = r & 3;
        b[r] = __byte_perm(words[r >> 2], words[2 + (r >> 2)], q | (q << 4) | ((4 + q) << 8) | ((4 + q) << 12)) &
               0x00FF00FFu;
    }
}

// u * 2^-24 -> L(u) * 2^-24 in both halves: 2u - 1 for one bit, u - z otherwise.
template <int W>
__device__ __forceinline__ void to_levels(uint32_t (&b)[8]) {
    if (W == 0) {
        const __half2 two = __floats2half2_rn(2.f, 2.f), m1 = __halves2half2(__ushort_as_half(0x8001u), __ushort_as_half(0x8001u));
#pragma unroll
        for (int r = 0; r < 8; ++r) {
            const __half2 v = __hfma2(*reinterpret_cast<const __half2*>(&b[r]), two, m1);
            b[r] = *reinterpret_cast<const uint32_t*>(&v);
        }
    } else {
        constexpr unsigned short zb = W == 1 ? 2 : W == 2 ? 8 : 128;   // z * 2^-24 as fp16 bits (a denormal)
        const __half2 z = __halves2half2(__ushort_as_half(zb), __ushort_as_half(zb));
#pragma unroll
        for (int r = 0; r < 8; ++r) {
            const __half2 v = __hsub2(*reinterpret_cast<const __half2*>(&b[r]), z);
            b[r] = *reinterpret_cast<const uint32_t*>(&v);
        }
    }
}

// The lane's 16 weights of item ig (positions 16t .. 16t + 15) as 8 fp16x2
// registers of u * 2^-24 (register rho: weights 16t + rho and 16t + 8 + rho);
// pay is the item's width's payload.
template <int W>
__device__ __forceinline__ void item_frag(uint32_t pay, int ig, int t, uint32_t (&b)[8]) {
    if (W == 0) bfrag_1(lds_u32x2(pay + ig * 8), t, b);
    else if (W == 1) bfrag_2(lds_u32x4(pay + ig * 16), t, b);
    else if (W == 2) bfrag_4(lds_u32x2(pay + ig * 32 + 8 * t), b);
    else bfrag_8(lds_u32x4(pay + ig * 64 + 16 * t), b);
}

// ---------------------------------------------------------------------------
// The weights as the MMA's A operand (16 items of one (column, width) bucket
// as its 16 rows) and the activations as its B operand (8 batch rows as its
// 8 columns; two such MMAs per k-step for NB = 16). Lane (g, t) decodes items
// g and g + 8 of a tile, and D gives it batch rows 2t and 2t + 1 (and 8 + 2t,
// 9 + 2t) of both, so a tile covers 16 items with 4 (8) MMAs and 4 (8)
// shared-memory additions per lane. The k order is the one above: in k-step s,
// A register (row, h) holds weights 16t + 2s + h and 16t + 8 + 2s + h, the
// activation table's register for batch row g, k-step s and half h (NB = 8:
// register 2s + h; NB = 16: 4s + 2h + n for the batch rows 8n + g), read here
// as B's two registers.
// ---------------------------------------------------------------------------
struct Tile16In {
    uint32_t bg[8], bh[8];       // levels of the lane's items g and g + 8 (fp16x2, u * 2^-24)
    float sg, sh;                // their FP16 scales
    uint32_t ag, ah;             // their row partials of batch row 2t (2t + 1 is YS_STRIDE floats on)
    bool og, oh;                 // the items exist
};

template <int W, bool SL>
__device__ __forceinline__ void tile16_in(Tile16In& ti, uint32_t pay, uint32_t scb, uint32_t rwb, int i0, int nv,
                                          uint32_t yst, int c, int g, int t) {
    const int ig = i0 + min(g, nv - 1), ih = i0 + min(g + 8, nv - 1);    // valid items past the end
    item_frag<W>(pay, ig, t, ti.bg);
    item_frag<W>(pay, ih, t, ti.bh);
    ti.sg = half_bits(lds_u16(scb + 2 * ig));
    ti.sh = half_bits(lds_u16(scb + 2 * ih));
    const uint32_t rg = lds_u8(rwb + ig), rh = lds_u8(rwb + ih);
    if constexpr (SL) {             // yst: the slots plus the lane's batch rows 2t, 2t + 1
        ti.ag = yst + 4 * slot_index(rg, (uint32_t)c, 0);
        ti.ah = yst + 4 * slot_index(rh, (uint32_t)c, 0);
    } else {
        ti.ag = yst + 4 * rg;
        ti.ah = yst + 4 * rh;
    }
    ti.og = g < nv;
    ti.oh = g + 8 < nv;
    to_levels<W>(ti.bg);
    to_levels<W>(ti.bh);
}

template <int NB>
__device__ __forceinline__ void tile16_mma(const uint32_t (&xb)[NB], const Tile16In& ti, float (&d)[NB / 2]) {
#pragma unroll
    for (int s2 = 0; s2 < 4; ++s2) {
        const uint32_t a[4] = {ti.bg[2 * s2], ti.bh[2 * s2], ti.bg[2 * s2 + 1], ti.bh[2 * s2 + 1]};
#pragma unroll
        for (int n = 0; n < NB / 8; ++n) {
            float (&dn)[4] = *reinterpret_cast<float (*)[4]>(&d[4 * n]);
            const uint32_t b0 = NB == 8 ? xb[2 * s2] : xb[4 * s2 + n];
            const uint32_t b1 = NB == 8 ? xb[2 * s2 + 1] : xb[4 * s2 + 2 + n];
            if (s2 == 0) mma16816_z(dn, a, b0, b1);
            else mma16816(dn, a, b0, b1);
        }
    }
}

// D (items g, g + 8 x batch rows 2t, 2t + 1, and 8 + 2t, 9 + 2t) times the
// items' scales and the batch rows' 2^E, into the row partials.
template <int NB, bool SL>
__device__ __forceinline__ void tile16_out(const Tile16In& ti, const float (&d)[NB / 2], const float2 (&e2)[NB / 8]) {
    const float2 vg = __fmul2_rn(__fmul2_rn(f2(d[0], d[1]), f2(ti.sg, ti.sg)), e2[0]);
    const float2 vh = __fmul2_rn(__fmul2_rn(f2(d[2], d[3]), f2(ti.sh, ti.sh)), e2[0]);
    if constexpr (SL) {                     // each (row, column) once per unit: stored, not added
        if (ti.og) sts_f32x2(ti.ag, vg);
        if (ti.oh) sts_f32x2(ti.ah, vh);
        return;
    }
    if (ti.og) {
        red_shared(ti.ag, vg.x);
        red_shared_off<YS_STRIDE>(ti.ag, vg.y);
    }
    if (ti.oh) {
        red_shared(ti.ah, vh.x);
        red_shared_off<YS_STRIDE>(ti.ah, vh.y);
    }
    if constexpr (NB == 16) {
        const float2 wg = __fmul2_rn(__fmul2_rn(f2(d[4], d[5]), f2(ti.sg, ti.sg)), e2[1]);
        const float2 wh = __fmul2_rn(__fmul2_rn(f2(d[6], d[7]), f2(ti.sh, ti.sh)), e2[1]);
        if (ti.og) {
            red_shared_off<8 * YS_STRIDE>(ti.ag, wg.x);
            red_shared_off<9 * YS_STRIDE>(ti.ag, wg.y);
        }
        if (ti.oh) {
            red_shared_off<8 * YS_STRIDE>(ti.ah, wh.x);
            red_shared_off<9 * YS_STRIDE>(ti.ah, wh.y);
        }
    }
}

// Tiles k0 .. k1-1 (16 items each) of one (column, width W) bucket [bs, be);
// pay / scb / rwb: the width's payload, scales and row bytes.
template <int NB, int W, bool SL>
__device__ __forceinline__ void run_tiles16(const uint32_t (&xb)[NB], const float2 (&e2)[NB / 8], uint32_t pay,
                                            uint32_t scb, uint32_t rwb, int bs, int be, int k0, int k1, uint32_t yst,
                                            int c, int g, int t) {
    for (int k = k0; k < k1; ++k) {
        const int i0 = bs + 16 * k;
        Tile16In ti;
        tile16_in<W, SL>(ti, pay, scb, rwb, i0, min(16, be - i0), yst, c, g, t);
        float d[NB / 2];
        tile16_mma<NB>(xb, ti, d);
        tile16_out<NB, SL>(ti, d, e2);
    }
}

// One consumer warp's share of a unit: tiles of 16 items of one (column,
// width) bucket, in (column, width) order; warp wt of a team of tw warps takes
// a contiguous run of them.
template <int NB, bool SL>
__device__ __forceinline__ void consume_unit_b16(const ActTables<NB>& T, uint32_t sblob, int C, int cols, uint32_t ys,
                                                 int wt, int tw, int lane) {
    const int g = lane >> 2, t = lane & 3;
    // the lane's batch row 2t: in the row partials, or (NB = 8) in the slots
    const uint32_t yst = SL ? ys + 8u * (uint32_t)t : ys + 4u * (uint32_t)(2 * t * YS_STRIDE);
    const uint4 h0 = lds_u32x4(sblob), h1 = lds_u32x4(sblob + 16), h2 = lds_u32x4(sblob + 32);
    const uint32_t cc = sblob + (h2.x & 0xFFFF) * 16;
    int start[4], end[4], ntile[4], nt_col = 0;
#pragma unroll
    for (int w = 0; w < 4; ++w) {
        const int e = lane < cols ? (int)lds_u16(cc + 2 * (w * C + lane)) : 0;
        int a = __shfl_up_sync(0xffffffffu, e, 1);
        if (lane == 0) a = 0;
        start[w] = a;
        end[w] = e;
        ntile[w] = lane < cols ? (e - a + 15) >> 4 : 0;
        nt_col += ntile[w];
    }
    int incl = nt_col;                   // tiles of columns 0..lane
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int v = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += v;
    }
    const int total = __shfl_sync(0xffffffffu, incl, 31);
    const int lg_tw = __popc(tw - 1);                  // tw is a power of two
    const int ta = (total * wt) >> lg_tw, tb = (total * (wt + 1)) >> lg_tw;
    if (ta >= tb) return;
    const uint32_t pay[4] = {sblob + (h0.z & 0xFFFF) * 16, sblob + (h0.z >> 16) * 16, sblob + (h0.w & 0xFFFF) * 16,
                             sblob + (h0.w >> 16) * 16};
    const uint32_t scb[4] = {sblob + (h1.x & 0xFFFF) * 16, sblob + (h1.x >> 16) * 16, sblob + (h1.y & 0xFFFF) * 16,
                             sblob + (h1.y >> 16) * 16};
    const uint32_t rwb[4] = {sblob + (h1.z & 0xFFFF) * 16, sblob + (h1.z >> 16) * 16, sblob + (h1.w & 0xFFFF) * 16,
                             sblob + (h1.w >> 16) * 16};
    for (int c = __popc(__ballot_sync(0xffffffffu, incl <= ta)); c < cols; ++c) {
        const int c_end = __shfl_sync(0xffffffffu, incl, c), c_begin = c_end - __shfl_sync(0xffffffffu, nt_col, c);
        if (c_begin >= tb) break;
        // the column's activation fragments (the table's NB registers per lane)
        uint32_t xb[NB];
#pragma unroll
        for (int r = 0; r < NB; r += 4) {
            const uint4 v = *reinterpret_cast<const uint4*>(&T.xfr[c][r >> 2][lane][0]);
            xb[r] = v.x; xb[r + 1] = v.y; xb[r + 2] = v.z; xb[r + 3] = v.w;
        }
        float2 e2[NB / 8];
#pragma unroll
        for (int n = 0; n < NB / 8; ++n) e2[n] = f2(T.e2[c][8 * n + 2 * t], T.e2[c][8 * n + 2 * t + 1]);
        int tile0 = c_begin;
#pragma unroll
        for (int w = 0; w < 4; ++w) {
            const int nt = __shfl_sync(0xffffffffu, ntile[w], c);
            const int k0 = max(ta - tile0, 0), k1 = min(tb - tile0, nt);
            if (k0 < k1) {
                const int bs = __shfl_sync(0xffffffffu, start[w], c), be = __shfl_sync(0xffffffffu, end[w], c);
                if (w == 0) run_tiles16<NB, 0, SL>(xb, e2, pay[0], scb[0], rwb[0], bs, be, k0, k1, yst, c, g, t);
                else if (w == 1) run_tiles16<NB, 1, SL>(xb, e2, pay[1], scb[1], rwb[1], bs, be, k0, k1, yst, c, g, t);
                else if (w == 2) run_tiles16<NB, 2, SL>(xb, e2, pay[2], scb[2], rwb[2], bs, be, k0, k1, yst, c, g, t);
                else run_tiles16<NB, 3, SL>(xb, e2, pay[3], scb[3], rwb[3], bs, be, k0, k1, yst, c, g, t);
            }
            tile0 += nt;
        }
    }
}

// NB = 8: the team's flush of a finished unit from its slots. Thread ct takes
// row r = ct / 4 and batch rows 2q, 2q + 1 (q = ct % 4), sums the row's slots
// over the unit's columns in column order, and stores the sums into Y (one
// slab) or adds them (split-K). A half-warp's 8-byte loads (four rows, four
// batch-row pairs) fall in distinct banks when the rows differ in their low
// two bits, which four consecutive rows do.
__device__ __forceinline__ void flush_slots(const float* sl, const LayoutView& L, float* __restrict__ Y, int B,
                                            int rb, int cols, int ct) {
    const int r = ct >> 2, q = ct & 3;
    const int rows = min(RB, (int)(L.N - (int64_t)rb * RB));
    if (r >= rows || 2 * q >= B) return;
    const uint32_t row = smem_u32(sl) + 4u * ((uint32_t)r * (MAX_C * 8) + 2u * q);
    const uint32_t sw = (uint32_t)r & (MAX_C - 1);            // column c sits at (c ^ sw) * 8 floats (slot_index)
    float2 acc = lds_f32x2(row + ((0u ^ sw) << 5));
    for (int c = 1; c < cols; ++c) acc = __fadd2_rn(acc, lds_f32x2(row + (((uint32_t)c ^ sw) << 5)));
    float* y0 = Y + (int64_t)(2 * q) * L.N + (int64_t)rb * RB + r;
    if (L.S == 1) {
        y0[0] = acc.x;
        if (2 * q + 1 < B) y0[L.N] = acc.y;
    } else {
        red_global(y0, acc.x);
        if (2 * q + 1 < B) red_global(y0 + L.N, acc.y);
    }
}

template <int NB, bool SL>
__global__ void __launch_bounds__(GB_THREADS, 1) gemmb_kernel(LayoutView L, const uint16_t* __restrict__ X,
                                                              float* __restrict__ Y, int B) {
    constexpr int NST = Pipe<NB, SL>::stages;
    extern __shared__ __align__(16) unsigned char smem_raw[];
    unsigned char* base = smem_raw + ((256u - (smem_u32(smem_raw) & 255u)) & 255u);
    TablesB<NB, SL>& T = *reinterpret_cast<TablesB<NB, SL>*>(base + (size_t)NST * STAGE_BYTES_B);
    const uint32_t stage0 = smem_u32(base);
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int P = gridDim.x, p = blockIdx.x;
    const int per = L.units / P, extra = L.units - per * P;
    const int u_begin = p * per + min(p, extra), u_end = u_begin + per + (p < extra ? 1 : 0);
    const int n_units = u_end - u_begin;
    if (n_units <= 0) return;
    const int s0 = u_begin / L.nrb, rb0 = u_begin - s0 * L.nrb;
    // Teams as in the batch-1 kernel, at most Pipe<NB, SL>::max_teams: unit j uses
    // stage j % stages and goes to team j % teams, and teams divides stages, so
    // each team waits the phases of its own stages in order (a parity wait that
    // skipped a phase could match an older completed one).
    const int lg_teams = Pipe<NB, SL>::max_teams == 2 && n_units >= 4 ? 1 : 0;
    const int teams = 1 << lg_teams, tw = NCWB >> lg_teams;

    const uint32_t full0 = smem_u32(&T.full[0]), empty0 = smem_u32(&T.empty[0]);
    const uint32_t abort_addr = smem_u32(&T.abort);
    if (tid == 0) {
        for (int i = 0; i < NST; ++i) {
            mbar_init(full0 + 8 * i, 1);
            mbar_init(empty0 + 8 * i, tw);
        }
        T.abort = 0;
        T.sk_ok = 0;
        fence_barrier_init();
    }
    if constexpr (!SL)
        for (int i = tid; i < NST * NB * YS_STRIDE; i += GB_THREADS) (&T.ys[0][0][0])[i] = 0.f;
    __syncthreads();
    if (tid == 0) {
        const int first = n_units < NST ? n_units : NST;
        for (int j = 0; j < first; ++j) issue_unit(L, u_begin + j, stage0 + j * STAGE_BYTES_B, full0 + 8 * j);
    }
    {   // the first slab's activations into L2 while waiting for the previous grid
        const int64_t k0 = (int64_t)s0 * L.C * GROUP;
        const int lines = (min(L.C, L.G - s0 * L.C) * GROUP * 2 + 127) / 128;
        for (int q = tid - 32; q >= 0 && q < lines * B; q += GB_THREADS - 32)
            prefetch_l2(X + (int64_t)(q / lines) * L.K + k0 + (int64_t)(q % lines) * 64);
    }
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    asm volatile("griddepcontrol.wait;" ::: "memory");

    if (warp == 0) {
        // ---- copier: split-K zeroing, then per unit: rows out, next copy in ----
        // (whole row blocks move 4 rows per lane when every batch row of Y
        // starts on a 16-byte boundary)
        const bool vec = (L.N & 3) == 0;
        uint32_t epoch = 0;
        if (L.S > 1) {
            // the call count's load is in flight while the warp zeroes (the zeros
            // do not depend on it; the flags do)
            const unsigned long long count = call_count_raw(L.ctl);
            const int z_end = min(u_end, L.nrb);
            for (int u = u_begin; u < z_end; ++u) {
                const int rows = min(RB, (int)(L.N - (int64_t)u * RB));
                for (int b = 0; b < B; ++b) {
                    float* yr = Y + (int64_t)b * L.N + (int64_t)u * RB;
                    if (vec && rows == RB) reinterpret_cast<float4*>(yr)[lane] = make_float4(0.f, 0.f, 0.f, 0.f);
                    else
                        for (int r = lane; r < rows; r += 32) yr[r] = 0.f;
                }
            }
            __syncwarp();
            epoch = epoch_of(count);
            // release stores, one unit per lane in parallel: the warp's zeros
            // (ordered by __syncwarp) before each flag
            for (int u = u_begin + lane; u < z_end; u += 32) st_release_gpu(L.ctl + 2 + u, epoch);
        }
        bool dead = false;
        if (L.S > 1 && !split_k_flags_ready(L, epoch, u_begin, u_end, lane)) {
            // a row block this block adds into was never zeroed in time
            dead = true;
            if (lane == 0) raise_abort(&T.abort);
        }
        // NB = 8: the consumers write Y; they add only after these flags (and
        // this warp's own zeroing), passed on by a release
        if (SL && L.S > 1 && lane == 0) red_release_cta_shared_add(smem_u32(&T.sk_ok), dead ? 0x10000u : 1u);
        int st = 0, rbw = rb0, issued = n_units < NST ? n_units : NST;
        uint32_t par = 0;
        for (int j = 0; j < n_units; ++j) {
            // units here take microseconds: nap between polls, except on the
            // block's last unit, whose rows end the block
            if (!dead && !warp_wait(empty0 + 8 * st, par, abort_addr, j + 1 < n_units ? 1024 : 0)) {
                dead = true;
                if (lane == 0) raise_abort(&T.abort);
            }
            if (!dead && !SL) {
                const int rows = min(RB, (int)(L.N - (int64_t)rbw * RB));
                for (int b = 0; b < B; ++b) {
                    const uint32_t ysb = smem_u32(&T.ys[st][b][0]) + 16u * lane;
                    float* yr = Y + (int64_t)b * L.N + (int64_t)rbw * RB + 4 * lane;
                    const float4 v = lds_f32x4(ysb);
                    sts_zero4(ysb);
                    if (vec && rows == RB) {
                        if (L.S == 1) *reinterpret_cast<float4*>(yr) = v;
                        else red_global_v4(yr, v);
                    } else {
                        const float vv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            if (4 * lane + i < rows) {
                                if (L.S == 1) yr[i] = vv[i];
                                else red_global(yr + i, vv[i]);
                            }
                        }
                    }
                }
                __syncwarp();
            }
            if (!dead && j + NST < n_units) {
                if (lane == 0) issue_unit(L, u_begin + j + NST, stage0 + st * STAGE_BYTES_B, full0 + 8 * st);
                ++issued;
            }
            if (++st == NST) { st = 0; par ^= 1; }
            if (++rbw == L.nrb) rbw = 0;
        }
        if (dead && lane == 0) {
            for (int i = 0; i < NST && i < issued; ++i) {
                const int jl = i + ((issued - 1 - i) / NST) * NST;
                mbar_wait_bounded(full0 + 8 * i, (uint32_t)((jl / NST) & 1));
            }
        }
        if (L.S > 1 && lane == 0) call_done(L.ctl);      // this block's share of the call count
    } else {
        // ---- consumers: team `team` takes units j = team, team + teams, ... ----
        const int cw = warp - 1, ct = tid - 32, team = cw / tw, wt = cw - team * tw;
        const int s_last = (u_end - 1) / L.nrb;
        bool dead = false, sk_seen = L.S == 1;
        int cur = s0, rbj = rb0 + team, sj = s0;
        while (rbj >= L.nrb) { rbj -= L.nrb; ++sj; }
        build_tables_b(T, L, X, B, s0, ct);
        for (int j = team; j < n_units; j += teams) {
            while (cur < sj) build_tables_b(T, L, X, B, ++cur, ct);
            const int st = j % NST;                      // NST is a compile-time constant
            const uint32_t par = (uint32_t)(j / NST) & 1u;
            const int cols = min(L.C, L.G - sj * L.C);
            if (!dead && !warp_wait(full0 + 8 * st, par, abort_addr)) { dead = true; if (lane == 0) raise_abort(&T.abort); }
            if (!dead) {
                consume_unit_b16<NB, SL>(T, stage0 + st * STAGE_BYTES_B, L.C, cols,
                                         SL ? smem_u32(&T.sl[0]) : smem_u32(&T.ys[st][0][0]), wt, tw, lane);
                __syncwarp();
                if (lane == 0) mbar_arrive(empty0 + 8 * st);
            }
            if constexpr (SL) {
                // every warp's slot stores, then the unit's rows out; the next
                // unit's stores only after every thread's reads
                consumer_sync_b();
                if (!sk_seen && !dead) {
                    // split-K: after the copier's flag check (bounded wait)
                    uint32_t g = 0;
                    const unsigned long long w0 = global_ns();
                    while ((g = ld_acquire_cta_shared(smem_u32(&T.sk_ok))) == 0u && !lds_volatile(abort_addr) &&
                           global_ns() - w0 < WAIT_LIMIT_NS)
                        __nanosleep(32);
                    if (g != 1u) {
                        dead = true;
                        if (lane == 0) raise_abort(&T.abort);
                    }
                    sk_seen = true;
                }
                if (!dead) flush_slots(T.sl, L, Y, B, rbj, cols, ct);
                consumer_sync_b();
            }
            rbj += teams;
            while (rbj >= L.nrb) { rbj -= L.nrb; ++sj; }
        }
        while (cur < s_last) build_tables_b(T, L, X, B, ++cur, ct);
    }
}

template <int NB, bool SL>
cudaError_t launch_gemmb(const LayoutView& L, const uint16_t* X, float* Y, int B, cudaStream_t s) {
    static LaunchPrep prep;
    int sms = 0;
    cudaError_t e = prep.get(gemmb_kernel<NB, SL>, gemmb_smem<NB, SL>(), &sms);
    if (e != cudaSuccess) return e;
    const int grid = L.units < sms ? L.units : sms;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(GB_THREADS);
    cfg.dynamicSmemBytes = gemmb_smem<NB, SL>();
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, gemmb_kernel<NB, SL>, L, X, Y, B);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_gemm_small(const LayoutView& L, const uint16_t* X, float* Y, int B, cudaStream_t s) {
    if (B > 8) return launch_gemmb<16, false>(L, X, Y, B, s);
    // slots where units are wide: their per-unit flush and barriers are then
    // small against a unit's tiles; narrow units keep two teams and four stages
    return L.C >= SLOT_MIN_C ? launch_gemmb<8, true>(L, X, Y, B, s) : launch_gemmb<8, false>(L, X, Y, B, s);
}

cudaError_t read_device_status_gemm(uint32_t* status) {
    cudaError_t e = cudaMemcpyFromSymbol(status, g_device_status, sizeof(uint32_t));
    if (e != cudaSuccess) return e;
    const uint32_t zero = 0;
    return cudaMemcpyToSymbol(g_device_status, &zero, sizeof(uint32_t));
}

}  // namespace vbq
