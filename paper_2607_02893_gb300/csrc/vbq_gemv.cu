// vbq_gemv.cu — fused dequantise-and-multiply y = W x over the packed layout
// (§6: load the packed low-bit bytes of a group, expand them in registers with
// the group's scale, accumulate the matrix-vector product; the wide weights
// never reach memory).
//
// Batch 1 (gemv1_kernel): one persistent block per SM, warp-specialised.
//   warp 0 (copier)    streams unit blobs into NSTAGE shared-memory stages with
//                      TMA bulk copies and, once a unit is consumed, sums its
//                      slots per row into y and starts the copy of a later unit
//                      into the freed stage;
//   warps 1.. (NCW)    consumers, in 1 or 2 teams (2 from 4 units per block
//                      on): unit j goes to team j % teams, whose warps split
//                      the unit's warp tasks (a table the packer stores in
//                      the blob: each task's items, their offsets and
//                      columns) and store each group's scaled dot product in
//                      the stage's (row, column) slot.
// The roles hand stages to one another through two mbarriers per stage
// (full: blob landed; empty: the unit's team is done), so no block-wide
// barrier sits in the steady state and up to NSTAGE units are in flight per
// SM. Block p owns a contiguous range of units in
// slab-major order, so consecutive units share their activations; on a slab
// change the consumer warps rebuild, under a named barrier of their own, the
// per-slab activation tables: x as fp32 and, for every 4 consecutive weights of
// a group column, the 16 signed sums of their activations (a lookup table
// indexed by 4 code bits: bit i set adds x_i, clear subtracts it). Per width:
//   b = 1  one table lookup per 4 weights; L_1(u) = 2u - 1 is the sign the
//          table applies, so the group's dot product is the sum T of its 16
//          lookups; two groups per lane, their sums added as f32x2 pairs;
//   b = 2  the two bit planes use the same tables: with u = b0 + 2 b1,
//          L_2(u) = b0 + 2 b1 - 2 = (2 b0 - 1) / 2 + (2 b1 - 1) - 1/2, so the
//          dot product is T0 / 2 + T1 - X / 2 (X = sum of x);
//   b = 4  codes are masked in place and read as exact denormal floats
//          against activations pre-scaled per code slot (packed f32x2 FMAs);
//          8X (summed in the same order) is subtracted for the zero level;
//   b = 8  same with a byte permute and 2^23 + 128.
// X is summed from the tables in the same order as the lookups (and entry
// 15 - m is exactly -entry m), so a group whose codes are all at the zero
// level contributes exactly 0. Each group's
// fp32 dot product is scaled once by its FP16 scale and stored in its
// (row, column) slot; the copier sums a row's slots in a fixed order and
// writes y directly (one slab per row) or through atomics (several slabs).
//
// The same kernel takes two activation vectors per launch (NX = 2, batches of
// 2..4 as one or two launches): the second vector's tables sit a fixed
// distance after the first's, so each lookup address, masked code and level
// serves both. Batches of 5..16 run on the tensor cores in vbq_gemm.cu.
//
// Two more instantiations fuse a SwiGLU MLP's nonlinearity into the products
// (the paper's models use SwiGLU MLPs, §4; zero-padded intermediates are inert,
// §6): MODE_SWIGLU_EPI, on a gate-up matrix whose rows alternate, also writes
// h = silu(gate) * up in BF16 (the copier computes it from a row pair's sums
// when a row has one slab, otherwise the block whose addition completes a row
// block's slab count reads the finished rows back); MODE_SWIGLU_IN, on the
// down projection, builds its activation tables from h_k = silu(gu[2k]) *
// gu[2k + 1] of the gate-up product's fp32 output, so h never reaches memory.
#include <cstddef>
#include <mutex>

#include "vbq_kernels.h"
#include "vbq_device.cuh"
#include <cuda_bf16.h>

namespace vbq {
namespace {

constexpr int NCW = 16;                  // consumer warps of the batch-1 kernel
constexpr int NCT = 32 * NCW;            // consumer threads
constexpr int NCOPY = 2;                 // copier warps of the batch-1 kernel (unit j: copier j % 2)
constexpr int G1_THREADS = 32 * (NCW + NCOPY);
constexpr int CH_THREADS = 32 * (NCW + 1);    // the chain kernel: one copier warp
constexpr int XQ = 20;                   // floats per 16-code quarter of x (16 + 4 pad: quarters use other banks)
constexpr int XH = 36;                   // floats per 32-code half of the pre-scaled x (32 + 4 pad)
constexpr int LUT_COL_BYTES = 1280;      // 16 tables x 64 bytes (+64 for odd columns), columns on 256-byte boundaries
constexpr int STAGE_BYTES = MAX_BLOB_BYTES;   // holds the largest unit blob (the packer guarantees it)
static_assert(STAGE_BYTES % 256 == 0, "stages keep the tables 256-byte aligned");
static_assert(LUT_COL_BYTES % 256 == 0 && 64 + 16 * 64 <= LUT_COL_BYTES, "column tables: 256-byte aligned, room for the odd shift");

// What a launch does around the product (a template argument, so the plain
// product's code carries none of the others'): MODE_PLAIN y = W x;
// MODE_SWIGLU_EPI also writes h = silu(gate) * up in BF16 from a gate-up
// product whose rows alternate (NX = 1); MODE_SWIGLU_IN takes as activations
// h_k = silu(gu[2k]) * gu[2k + 1] of a gate-up output gu (NX = 1).
enum Mode : int { MODE_PLAIN = 0, MODE_SWIGLU_EPI = 1, MODE_SWIGLU_IN = 2 };

// One kernel serves NX = 1 or 2 activation vectors (batch rows) per launch.
// With two, every table lookup address serves both: the second vector's
// tables sit a fixed distance after the first's, reached by the load's
// immediate offset. Per vector (byte strides between the vectors' copies):
constexpr int LUT_BYTES = MAX_C * LUT_COL_BYTES;          // nibble lookup tables
constexpr int XS_FLOATS = MAX_C * 4 * XQ;                 // x as fp32
constexpr int X4S_FLOATS = MAX_C * 2 * XH;                // pre-scaled 4-bit slots
constexpr int SLOT_FLOATS = RB * MAX_C;                   // (row, column) slots of a unit
static_assert(LUT_BYTES % 256 == 0, "the second vector's tables keep the byte-merge alignment");

// Stages and consumer teams per vector count. Unit j uses stage j % nstage and
// goes to team j % teams; with nstage a multiple of every team count, each
// stage serves one team only, and that team waits the stage's phases in order
// (a parity wait never skips a phase). Two teams give each team two stages,
// so its next blob lands while it works on the current one; two vectors'
// tables leave room for two stages and one team.
template <int NX> struct Geo {
    static constexpr int nstage = NX == 1 ? 4 : 2;
    static constexpr int max_teams = NX == 1 ? 2 : 1;
    static_assert((nstage & (nstage - 1)) == 0, "power-of-two stage count");
    static_assert(nstage % max_teams == 0 && nstage / max_teams >= 2, "each team owns at least two stages");
};
static_assert(NCW == 16, "teams of 16 or 8 warps: task steps are powers of two (masks, no division)");

template <int NX>
struct __align__(16) TablesT {
    uint8_t lut[NX * LUT_BYTES];         // vector v, column c, nibble j, entry m at v*LUT_BYTES + c*1280 + (c&1)*64 + j*64 + m*4
    float xs[NX * XS_FLOATS];            // x as fp32; quarter (c, q) at (c*4 + q) * XQ
    float x4s[NX * X4S_FLOATS];          // x pre-scaled per 4-bit nibble slot (see dot4_half); half (c, h) at (c*2 + h) * XH
    float2 x4z[NX][MAX_C][2];            // per column and half: sums of x * 2^-100, even / odd codes
    float xlut[NX][MAX_C];               // per column: sum of the all-ones entries, in lookup order
    float slots[Geo<NX>::nstage][NX][SLOT_FLOATS];   // per stage and vector: one value per (row, column) (see slot_addr)
    unsigned long long full[Geo<NX>::nstage];        // blob landed (TMA transaction count)
    unsigned long long empty[Geo<NX>::nstage];       // the unit's team is done (one arrival per team warp)
    uint32_t sk_ok;                      // split-K: copiers whose flag checks passed (+1 each; 0x10000 on failure)
    int abort;                           // set by any role whose wait ran out
};
template <int NX> struct TablesCheck {
    using T = TablesT<NX>;
    static_assert(offsetof(T, full) % 8 == 0, "mbarriers are 8-byte aligned");
    static_assert(offsetof(T, lut) == 0, "tables start at the aligned base");
    static_assert(offsetof(T, x4z) % 16 == 0 && offsetof(T, xs) % 16 == 0 && offsetof(T, x4s) % 16 == 0 &&
                  offsetof(T, slots) % 16 == 0, "16-byte table reads");
    static constexpr bool ok = true;
};
static_assert(TablesCheck<1>::ok && TablesCheck<2>::ok, "table layout");
static_assert(RB % 32 == 0, "the copier flushes rows a warp at a time");
static_assert(MAX_C <= 32, "a warp holds a unit's column ends one per lane");

template <int NX>
constexpr size_t gemv1_smem() { return 256 /* alignment slack */ + (size_t)Geo<NX>::nstage * STAGE_BYTES + sizeof(TablesT<NX>); }
static_assert(gemv1_smem<1>() <= 227 * 1024 && gemv1_smem<2>() <= 227 * 1024, "one block per SM");

// The 16 table entries that a 64-bit bit plane (words lo, hi) selects from a
// column's tables at tb (256-byte aligned): nibble p of the plane picks entry
// m at tb + sh + 64 p + 4 m, where sh is 64 for odd columns and 0 for even
// ones (odd columns sit in the other half of the banks, so a warp whose lanes
// straddle two columns reads without bank conflicts). Even and odd nibbles are
// masked into the bytes of two words as 4 m + sh (sh4 = sh in every byte); a
// byte permute then merges one such byte with the upper bytes of tb, so every
// lookup address costs one instruction.
__device__ __forceinline__ uint32_t col_shift4(int c) { return (uint32_t)(c & 1) * 0x40404040u; }

// Every (row, column) of a unit holds exactly one group, so each group's
// scaled dot product has a slot of its own and is stored, not added: no
// shared-memory atomics, and the row sums are taken later in a fixed order.
// Row r's 16 slots are 64 contiguous bytes; column c sits at position
// c ^ ((r >> 1) & 15), so a warp storing one column for up to 32 consecutive
// rows touches 32 distinct banks.
static_assert(MAX_C == 16, "16 slots per row");
__device__ __forceinline__ uint32_t slot_addr(uint32_t slots, uint32_t r, int c) {
    return slots + (r << 6) + (((uint32_t)c ^ ((r >> 1) & 15u)) << 2);
}
__device__ __forceinline__ void plane_entries(uint32_t tb, uint32_t sh4, uint32_t lo, uint32_t hi, float (&v)[16]) {
    const uint32_t M = 0x3C3C3C3Cu;
    const uint32_t le = ((lo << 2) & M) | sh4, lo_ = ((lo >> 2) & M) | sh4;
    const uint32_t he = ((hi << 2) & M) | sh4, ho = ((hi >> 2) & M) | sh4;
    v[0] = lds_f32<0>(__byte_perm(le, tb, 0x7650));
    v[1] = lds_f32<64>(__byte_perm(lo_, tb, 0x7650));
    v[2] = lds_f32<128>(__byte_perm(le, tb, 0x7651));
    v[3] = lds_f32<192>(__byte_perm(lo_, tb, 0x7651));
    v[4] = lds_f32<256>(__byte_perm(le, tb, 0x7652));
    v[5] = lds_f32<320>(__byte_perm(lo_, tb, 0x7652));
    v[6] = lds_f32<384>(__byte_perm(le, tb, 0x7653));
    v[7] = lds_f32<448>(__byte_perm(lo_, tb, 0x7653));
    v[8] = lds_f32<512>(__byte_perm(he, tb, 0x7650));
    v[9] = lds_f32<576>(__byte_perm(ho, tb, 0x7650));
    v[10] = lds_f32<640>(__byte_perm(he, tb, 0x7651));
    v[11] = lds_f32<704>(__byte_perm(ho, tb, 0x7651));
    v[12] = lds_f32<768>(__byte_perm(he, tb, 0x7652));
    v[13] = lds_f32<832>(__byte_perm(ho, tb, 0x7652));
    v[14] = lds_f32<896>(__byte_perm(he, tb, 0x7653));
    v[15] = lds_f32<960>(__byte_perm(ho, tb, 0x7653));
}

// Sums of a (in .x) and of b (in .y) as balanced trees (pairs, then pairs of
// pairs: the order the all-ones column sums xlut use), with f32x2 adds.
__device__ __forceinline__ float2 tree16x2(const float (&a)[16], const float (&b)[16]) {
    float2 p[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) p[i] = __fadd2_rn(f2(a[2 * i], b[2 * i]), f2(a[2 * i + 1], b[2 * i + 1]));
    const float2 q0 = __fadd2_rn(p[0], p[1]), q1 = __fadd2_rn(p[2], p[3]);
    const float2 q2 = __fadd2_rn(p[4], p[5]), q3 = __fadd2_rn(p[6], p[7]);
    return __fadd2_rn(__fadd2_rn(q0, q1), __fadd2_rn(q2, q3));
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

// Two activation vectors: the same 16 lookups of a plane, each address
// reading the first vector's entry (.x) and the second's, LUT_BYTES further
// (.y).
template <int OFF>
__device__ __forceinline__ float2 lds_pair(uint32_t a) { return f2(lds_f32<OFF>(a), lds_f32<OFF + LUT_BYTES>(a)); }
__device__ __forceinline__ void plane_entries2(uint32_t tb, uint32_t sh4, uint32_t lo, uint32_t hi, float2 (&v)[16]) {
    const uint32_t M = 0x3C3C3C3Cu;
    const uint32_t le = ((lo << 2) & M) | sh4, lo_ = ((lo >> 2) & M) | sh4;
    const uint32_t he = ((hi << 2) & M) | sh4, ho = ((hi >> 2) & M) | sh4;
    v[0] = lds_pair<0>(__byte_perm(le, tb, 0x7650));
    v[1] = lds_pair<64>(__byte_perm(lo_, tb, 0x7650));
    v[2] = lds_pair<128>(__byte_perm(le, tb, 0x7651));
    v[3] = lds_pair<192>(__byte_perm(lo_, tb, 0x7651));
    v[4] = lds_pair<256>(__byte_perm(le, tb, 0x7652));
    v[5] = lds_pair<320>(__byte_perm(lo_, tb, 0x7652));
    v[6] = lds_pair<384>(__byte_perm(le, tb, 0x7653));
    v[7] = lds_pair<448>(__byte_perm(lo_, tb, 0x7653));
    v[8] = lds_pair<512>(__byte_perm(he, tb, 0x7650));
    v[9] = lds_pair<576>(__byte_perm(ho, tb, 0x7650));
    v[10] = lds_pair<640>(__byte_perm(he, tb, 0x7651));
    v[11] = lds_pair<704>(__byte_perm(ho, tb, 0x7651));
    v[12] = lds_pair<768>(__byte_perm(he, tb, 0x7652));
    v[13] = lds_pair<832>(__byte_perm(ho, tb, 0x7652));
    v[14] = lds_pair<896>(__byte_perm(he, tb, 0x7653));
    v[15] = lds_pair<960>(__byte_perm(ho, tb, 0x7653));
}
// Sums of 16 pairs in the order tree16x2 adds each of its two operands.
__device__ __forceinline__ float2 tree16_pairs(const float2 (&a)[16]) {
    float2 p[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) p[i] = __fadd2_rn(a[2 * i], a[2 * i + 1]);
    const float2 q0 = __fadd2_rn(p[0], p[1]), q1 = __fadd2_rn(p[2], p[3]);
    const float2 q2 = __fadd2_rn(p[4], p[5]), q3 = __fadd2_rn(p[6], p[7]);
    return __fadd2_rn(__fadd2_rn(q0, q1), __fadd2_rn(q2, q3));
}
// dot4_half for two vectors: the masked codes are shared, each vector's
// pre-scaled slots are X4S_FLOATS after the previous one's.
__device__ __forceinline__ void dot4_half2(uint4 v, uint32_t xa, float2& r0, float2& r1) {
    float2 ca = f2(0.f, 0.f), cb = f2(0.f, 0.f), da = f2(0.f, 0.f), db = f2(0.f, 0.f);
    const uint32_t words[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int t = 0; t < 4; ++t) {
        const uint32_t w = words[t], w2 = w >> 24;
        const float4 xa4 = lds_f32x4(xa + t * 32), xb4 = lds_f32x4(xa + t * 32 + 16);
        const float4 ya4 = lds_f32x4(xa + 4 * X4S_FLOATS + t * 32), yb4 = lds_f32x4(xa + 4 * X4S_FLOATS + t * 32 + 16);
        const float2 u0 = f2(__uint_as_float(w & 0xFu), __uint_as_float(w & 0xF0u));
        const float2 u1 = f2(__uint_as_float(w & 0xF00u), __uint_as_float(w & 0xF000u));
        const float2 u2 = f2(__uint_as_float(w & 0xF0000u), __uint_as_float(w & 0xF00000u));
        const float2 u3 = f2(__uint_as_float(w2 & 0xFu), __uint_as_float(w2 & 0xF0u));
        float2& c = (t & 1) ? cb : ca;
        float2& d = (t & 1) ? db : da;
        c = __ffma2_rn(u0, f2(xa4.x, xa4.y), c);
        c = __ffma2_rn(u1, f2(xa4.z, xa4.w), c);
        c = __ffma2_rn(u2, f2(xb4.x, xb4.y), c);
        c = __ffma2_rn(u3, f2(xb4.z, xb4.w), c);
        d = __ffma2_rn(u0, f2(ya4.x, ya4.y), d);
        d = __ffma2_rn(u1, f2(ya4.z, ya4.w), d);
        d = __ffma2_rn(u2, f2(yb4.x, yb4.y), d);
        d = __ffma2_rn(u3, f2(yb4.z, yb4.w), d);
    }
    r0 = __fadd2_rn(ca, cb);
    r1 = __fadd2_rn(da, db);
}
// dot8_quarter for two vectors (levels shared; each vector's fp32 x is
// XS_FLOATS after the previous one's). Returns (vector 0, vector 1).
__device__ __forceinline__ float2 dot8_quarter2(uint4 v, uint32_t xa) {
    const float2 off = f2(-8388736.f, -8388736.f);          // -(2^23 + 128)
    const uint32_t M = 0x4B000000u;
    float2 ca = f2(0.f, 0.f), cb = f2(0.f, 0.f), da = f2(0.f, 0.f), db = f2(0.f, 0.f);
    const uint32_t words[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int t = 0; t < 4; ++t) {
        const uint32_t w = words[t];
        const float4 x4 = lds_f32x4(xa + t * 16), y4 = lds_f32x4(xa + 4 * XS_FLOATS + t * 16);
        const float2 l0 = __fadd2_rn(f2(__uint_as_float(__byte_perm(w, M, 0x7540)),
                                        __uint_as_float(__byte_perm(w, M, 0x7541))), off);
        const float2 l1 = __fadd2_rn(f2(__uint_as_float(__byte_perm(w, M, 0x7542)),
                                        __uint_as_float(__byte_perm(w, M, 0x7543))), off);
        ca = __ffma2_rn(l0, f2(x4.x, x4.y), ca);
        cb = __ffma2_rn(l1, f2(x4.z, x4.w), cb);
        da = __ffma2_rn(l0, f2(y4.x, y4.y), da);
        db = __ffma2_rn(l1, f2(y4.z, y4.w), db);
    }
    return f2((ca.x + ca.y) + (cb.x + cb.y), (da.x + da.y) + (db.x + db.y));
}

// Consumer warps only (named barrier 1).
__device__ __forceinline__ void consumer_sync() {
    asm volatile("bar.sync 1, %0;" :: "n"(NCT) : "memory");
}

// silu(g) * u with silu(z) = z / (1 + e^-z), in fp32 with explicitly rounded
// operations (no contraction), so every call site gives the same bits.
// silu(0) * u = 0: zero-padded features stay inert.
__device__ __forceinline__ float swiglu_f32(float g, float u) {
    return __fmul_rn(__fdiv_rn(g, __fadd_rn(1.f, expf(-g))), u);
}

// The 4-bit zero-level sum of half a group's activations (32 of them), as
// (even, odd) code slots times 2^-100, in the order dot4_half accumulates.
__device__ __forceinline__ float2 zero_level_sum4(const float (&xh)[32]) {
    float2 ca = f2(0.f, 0.f), cb = f2(0.f, 0.f);
#pragma unroll
    for (int t4 = 0; t4 < 4; ++t4) {
        float2& cc = (t4 & 1) ? cb : ca;
#pragma unroll
        for (int e = 0; e < 8; e += 2)
            cc = __ffma2_rn(f2(xh[8 * t4 + e], xh[8 * t4 + e + 1]), f2(0x1p-100f, 0x1p-100f), cc);
    }
    return __fadd2_rn(ca, cb);
}

// Activations of slab s (per vector, for NX vectors stored K apart): x as fp32,
// the pre-scaled x of the 4-bit slots, the nibble lookup tables, and the
// per-column sums in lookup order. Consumer threads only (ct = 0 .. NCT-1):
// threads 0 .. 16 MAX_C - 1 one per (column, 4 weights), each reading its 4
// activations from global memory (L2); the next 2 MAX_C threads one per
// (column, half) for the 4-bit zero-level sums, reading their 32 activations
// at the same time. So the whole build is one phase between two consumer
// barriers. The column sum of the all-ones entries (xlut) is added over the
// column's half-warp in the pairs tree16x2 uses.
static_assert(NCT >= 16 * MAX_C + 2 * MAX_C, "threads for the tables and the zero-level sums");
template <int NX, int MODE>
__device__ void build_tables(TablesT<NX>& T, const LayoutView& L, const uint16_t* __restrict__ x,
                             const float* __restrict__ gu, int s, int ct) {
    const int cols = min(L.C, L.G - s * L.C);
    consumer_sync();                // nobody still reads the old tables
    if (ct < cols * 16) {
        const int c = ct >> 4, jn = ct & 15, jj = 4 * jn;
#pragma unroll
        for (int v = 0; v < NX; ++v) {
            float* xs = T.xs + v * XS_FLOATS;
            float* x4s = T.x4s + v * X4S_FLOATS;
            float x0, x1, x2, x3;
            if constexpr (MODE == MODE_SWIGLU_IN) {
                // SwiGLU input: activation k is silu(gu[2k]) * gu[2k + 1]
                const float4* src = reinterpret_cast<const float4*>(gu + 2 * ((int64_t)s * L.C * GROUP + c * GROUP + jj));
                const float4 a = __ldg(src), b = __ldg(src + 1);
                x0 = swiglu_f32(a.x, a.y);
                x1 = swiglu_f32(a.z, a.w);
                x2 = swiglu_f32(b.x, b.y);
                x3 = swiglu_f32(b.z, b.w);
            } else {
                const uint16_t* xg = x + (int64_t)v * L.K + (int64_t)s * L.C * GROUP;
                const uint2 four = __ldg(reinterpret_cast<const uint2*>(xg + c * GROUP + jj));
                x0 = __uint_as_float(four.x << 16);
                x1 = __uint_as_float(four.x & 0xFFFF0000u);
                x2 = __uint_as_float(four.y << 16);
                x3 = __uint_as_float(four.y & 0xFFFF0000u);
            }
            *reinterpret_cast<float4*>(&xs[(c * 4 + (jj >> 4)) * XQ + (jj & 15)]) = make_float4(x0, x1, x2, x3);
            // 4-bit slot shifts: nibble slots 0..5 of a word keep their place, 6 and 7 come down by 24
            float p4[4];
            const float xv4[4] = {x0, x1, x2, x3};
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int slot = (jj + i) & 7, e = slot < 6 ? 4 * slot : 4 * (slot - 6);
                p4[i] = xv4[i] * __uint_as_float((uint32_t)(127 + 49 - e) << 23);
            }
            *reinterpret_cast<float4*>(&x4s[(c * 2 + (jj >> 5)) * XH + (jj & 31)]) = make_float4(p4[0], p4[1], p4[2], p4[3]);
            // entry m = sum_i (2 m_i - 1) x_i (code bit i of the nibble picks +x_i or
            // -x_i), as p[m & 3] + q[m >> 2]; entry 15 - m is exactly -entry m
            const float a = x0 + x1, b = x0 - x1, cc = x2 + x3, d = x2 - x3;
            float4* dst = reinterpret_cast<float4*>(T.lut + v * LUT_BYTES + c * LUT_COL_BYTES + (c & 1) * 64 + jn * 64);
            dst[0] = make_float4(-a + -cc, b + -cc, -b + -cc, a + -cc);
            dst[1] = make_float4(-a + d, b + d, -b + d, a + d);
            dst[2] = make_float4(-a + -d, b + -d, -b + -d, a + -d);
            dst[3] = make_float4(-a + cc, b + cc, -b + cc, a + cc);
            // xlut: balanced tree over the column's 16 all-ones entries (xor 1, 2, 4, 8
            // pair them as tree16x2 pairs the lookups)
            const unsigned half = (ct & 16) ? 0xFFFF0000u : 0x0000FFFFu;
            float sv = a + cc;
            sv += __shfl_xor_sync(half, sv, 1);
            sv += __shfl_xor_sync(half, sv, 2);
            sv += __shfl_xor_sync(half, sv, 4);
            sv += __shfl_xor_sync(half, sv, 8);
            if (jn == 0) T.xlut[v][c] = sv;
        }
    } else if (MODE != MODE_SWIGLU_IN && ct >= 16 * MAX_C && ct < 16 * MAX_C + cols * 2) {
        // X for the 4-bit zero level of half hh of column c, summed as
        // dot4_half accumulates (threads the lookup tables leave idle)
        const int z = ct - 16 * MAX_C, c = z >> 1, hh = z & 1;     // c < cols, hh < 2
#pragma unroll
        for (int v = 0; v < NX; ++v) {
            const uint16_t* xg = x + (int64_t)v * L.K + (int64_t)s * L.C * GROUP;
            const uint4* src = reinterpret_cast<const uint4*>(xg + c * GROUP + 32 * hh);
            float xh[32];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const uint4 w = __ldg(src + q);
                const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    xh[8 * q + 2 * i] = __uint_as_float(ws[i] << 16);
                    xh[8 * q + 2 * i + 1] = __uint_as_float(ws[i] & 0xFFFF0000u);
                }
            }
            T.x4z[v][c][hh] = zero_level_sum4(xh);
        }
    }
    if constexpr (MODE == MODE_SWIGLU_IN) {
        // SwiGLU input: the activations exist only once the table threads have
        // computed them, so the zero-level sums read them back from xs after a
        // barrier (the same values the lookups and products use)
        consumer_sync();
        if (ct >= 16 * MAX_C && ct < 16 * MAX_C + cols * 2) {
            const int z = ct - 16 * MAX_C, c = z >> 1, hh = z & 1;
            float xh[32];
#pragma unroll
            for (int q = 0; q < 2; ++q) {
                const uint32_t a = smem_u32(T.xs) + ((c * 4 + 2 * hh + q) * XQ) * 4;
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const float4 f = lds_f32x4(a + 16 * i);
                    xh[16 * q + 4 * i] = f.x;
                    xh[16 * q + 4 * i + 1] = f.y;
                    xh[16 * q + 4 * i + 2] = f.z;
                    xh[16 * q + 4 * i + 3] = f.w;
                }
            }
            T.x4z[0][c][hh] = zero_level_sum4(xh);
        }
    }
    consumer_sync();
}

// One warp task (a TaskDesc built at pack time: items, their blob offsets and
// columns), for the per-width bodies below. Lanes past the task's last item
// redo its first item (always present) and store nothing, so every body is
// branch-free.
struct Task {
    uint32_t pay, sc;           // shared addresses of the lane's (first) item: payload, scale
    uint32_t r, r2;             // the rows of its item(s) within the unit
    bool on, on2;               // the lane's item (1 bit: its first and second item) is stored
    int c, c2;                  // their columns
};

// 32-item tasks: lane l takes item l.
__device__ __forceinline__ Task task32(uint32_t sblob, uint4 d, int lane, int bytes_per_item) {
    Task t;
    const int cnt = (int)((d.x >> 20) & 63u) + 1;
    const uint32_t le = (2u << lane) - 1u;
    t.on = lane < cnt;
    const int ii = t.on ? lane : 0;
    t.c = (int)((d.x >> 16) & 15u) + __popc(d.y & le) + 2 * __popc(d.z & le);
    t.pay = sblob + (d.w & 0xFFFFu) + ii * bytes_per_item;
    t.sc = sblob + (d.x & 0xFFFFu) + 2 * ii;
    t.r = lds_u8(sblob + (d.w >> 16) + ii);
    t.r2 = t.r;
    t.on2 = false;
    t.c2 = t.c;
    return t;
}

// 1-bit tasks: lane l takes items 2l and 2l + 1 (one 16-byte payload load, one
// 2-byte row load, one 4-byte scale load); the first item is off in a task
// that starts one item early (skip bit).
__device__ __forceinline__ Task task64(uint32_t sblob, uint4 d, int lane) {
    Task t;
    const int cnt = (int)((d.x >> 20) & 63u) + 1;
    const uint32_t le = (2u << lane) - 1u, lt = (1u << lane) - 1u;
    const int j = 2 * lane;
    t.on = j < cnt && !(lane == 0 && (d.x >> 28));
    t.on2 = j + 1 < cnt;
    const int ii = j < cnt ? j : 0;
    t.c = (int)((d.x >> 16) & 15u) + __popc(d.y & le) + __popc(d.z & lt);
    t.c2 = t.c + (int)((d.z >> lane) & 1u);
    t.pay = sblob + (d.w & 0xFFFFu) + ii * 8;
    t.sc = sblob + (d.x & 0xFFFFu) + 2 * ii;
    const uint32_t rows2 = lds_u16(sblob + (d.w >> 16) + ii);
    t.r = rows2 & 0xffu;
    t.r2 = rows2 >> 8;
    return t;
}

// The per-width bodies: each group's scaled dot product (per activation
// vector) into its (row, column) slot of the stage.
template <int NX>
__device__ __forceinline__ void body4(const TablesT<NX>& T, const Task& t, uint32_t slots, int lane) {
    constexpr uint32_t SLOT_V = SLOT_FLOATS * 4;      // bytes between the vectors' slot arrays
    // halves in the order (lane >> 2) & 1 first, so each quarter-warp's
    // 16-byte loads fall in 8 distinct bank groups
    const int c = t.c;
    const int h0 = (lane >> 2) & 1;
    const uint4 va = lds_u32x4(t.pay + h0 * 16), vb = lds_u32x4(t.pay + (h0 ^ 1) * 16);
    const uint32_t xa = smem_u32(T.x4s) + (c * 2 + h0) * XH * 4, xb = smem_u32(T.x4s) + (c * 2 + (h0 ^ 1)) * XH * 4;
    const uint32_t sa = slot_addr(slots, t.r, c);
    const float scl = half_bits(lds_u16(t.sc)) * 0x1p100f;
    if constexpr (NX == 1) {
        const float2 aa = dot4_half(va, xa), ab = dot4_half(vb, xb);
        const float4 z = lds_f32x4(smem_u32(T.x4z) + c * 16);     // (even, odd) of half 0, then of half 1
        const float part = ((aa.x + ab.x) - 8.f * (z.x + z.z)) + ((aa.y + ab.y) - 8.f * (z.y + z.w));
        sts_f32_if(sa, scl * part, t.on);
    } else {
        float2 aa0, aa1, ab0, ab1;
        dot4_half2(va, xa, aa0, aa1);
        dot4_half2(vb, xb, ab0, ab1);
        const float4 z0 = lds_f32x4(smem_u32(T.x4z) + c * 16), z1 = lds_f32x4(smem_u32(T.x4z) + MAX_C * 16 + c * 16);
        const float p0 = ((aa0.x + ab0.x) - 8.f * (z0.x + z0.z)) + ((aa0.y + ab0.y) - 8.f * (z0.y + z0.w));
        const float p1 = ((aa1.x + ab1.x) - 8.f * (z1.x + z1.z)) + ((aa1.y + ab1.y) - 8.f * (z1.y + z1.w));
        sts_f32_if(sa, scl * p0, t.on);
        sts_f32_if(sa + SLOT_V, scl * p1, t.on);
    }
}

template <int NX>
__device__ __forceinline__ void body8(const TablesT<NX>& T, const Task& t, uint32_t slots, int lane) {
    constexpr uint32_t SLOT_V = SLOT_FLOATS * 4;
    // quarter (k + (lane >> 1)) & 3 in step k: conflict-free 16-byte loads
    const int c = t.c;
    const int q0 = lane >> 1;
    const uint32_t sa = slot_addr(slots, t.r, c);
    const float scl = half_bits(lds_u16(t.sc));
    if constexpr (NX == 1) {
        float part = 0.f;
#pragma unroll
        for (int step = 0; step < 4; ++step) {
            const int q = (step + q0) & 3;
            const uint4 v = lds_u32x4(t.pay + q * 16);
            part += dot8_quarter(v, smem_u32(T.xs) + (c * 4 + q) * XQ * 4);
        }
        sts_f32_if(sa, scl * part, t.on);
    } else {
        float p0 = 0.f, p1 = 0.f;
#pragma unroll
        for (int step = 0; step < 4; ++step) {
            const int q = (step + q0) & 3;
            const uint4 v = lds_u32x4(t.pay + q * 16);
            const float2 dd = dot8_quarter2(v, smem_u32(T.xs) + (c * 4 + q) * XQ * 4);
            p0 += dd.x;
            p1 += dd.y;
        }
        sts_f32_if(sa, scl * p0, t.on);
        sts_f32_if(sa + SLOT_V, scl * p1, t.on);
    }
}

template <int NX>
__device__ __forceinline__ void body2(const TablesT<NX>& T, const Task& t, uint32_t slots) {
    constexpr uint32_t SLOT_V = SLOT_FLOATS * 4;
    const int c = t.c;
    const uint4 pl = lds_u32x4(t.pay);
    const uint32_t tb = smem_u32(T.lut) + c * LUT_COL_BYTES;
    const uint32_t sa = slot_addr(slots, t.r, c);
    const float scl = half_bits(lds_u16(t.sc));
    // T0 / 2 + T1 - X / 2: for an all-zero-level group (b0 = 0, b1 = 1) T0 = -X
    // and T1 = X exactly, and X - X / 2 is exact, so the result is exactly 0
    if constexpr (NX == 1) {
        float va[16], vb[16];
        plane_entries(tb, col_shift4(c), pl.x, pl.y, va);
        plane_entries(tb, col_shift4(c), pl.z, pl.w, vb);
        const float2 sp = tree16x2(va, vb);
        sts_f32_if(sa, scl * ((0.5f * sp.x + sp.y) - 0.5f * lds_f32r(smem_u32(T.xlut) + 4 * c)), t.on);
    } else {
        float2 pv[16];
        plane_entries2(tb, col_shift4(c), pl.x, pl.y, pv);
        const float2 s0 = tree16_pairs(pv);                       // plane 0, both vectors
        plane_entries2(tb, col_shift4(c), pl.z, pl.w, pv);
        const float2 s1 = tree16_pairs(pv);                       // plane 1
        const uint32_t xl = smem_u32(T.xlut) + 4 * c;
        sts_f32_if(sa, scl * ((0.5f * s0.x + s1.x) - 0.5f * lds_f32r(xl)), t.on);
        sts_f32_if(sa + SLOT_V, scl * ((0.5f * s0.y + s1.y) - 0.5f * lds_f32r(xl + 4 * MAX_C)), t.on);
    }
}

template <int NX>
__device__ __forceinline__ void body1(const TablesT<NX>& T, const Task& t, uint32_t slots) {
    constexpr uint32_t SLOT_V = SLOT_FLOATS * 4;
    const int ca = t.c, cb = t.c2;
    const uint4 v = lds_u32x4(t.pay);
    const uint32_t sc2 = lds_u32(t.sc);
    const uint32_t sb = slot_addr(slots, t.r2, cb), sa = slot_addr(slots, t.r, ca);
    const float scb = half_bits(sc2 >> 16), sca = half_bits(sc2);
    if constexpr (NX == 1) {
        float va[16], vb[16];
        plane_entries(smem_u32(T.lut) + ca * LUT_COL_BYTES, col_shift4(ca), v.x, v.y, va);
        plane_entries(smem_u32(T.lut) + cb * LUT_COL_BYTES, col_shift4(cb), v.z, v.w, vb);
        const float2 sp = tree16x2(va, vb);
        sts_f32_if(sb, scb * sp.y, t.on2);
        sts_f32_if(sa, sca * sp.x, t.on);
    } else {
        float2 pv[16];
        plane_entries2(smem_u32(T.lut) + ca * LUT_COL_BYTES, col_shift4(ca), v.x, v.y, pv);
        const float2 sx = tree16_pairs(pv);                       // first item, both vectors
        sts_f32_if(sa, sca * sx.x, t.on);
        sts_f32_if(sa + SLOT_V, sca * sx.y, t.on);
        plane_entries2(smem_u32(T.lut) + cb * LUT_COL_BYTES, col_shift4(cb), v.z, v.w, pv);
        const float2 sy = tree16_pairs(pv);                       // second item
        sts_f32_if(sb, scb * sy.x, t.on2);
        sts_f32_if(sb + SLOT_V, scb * sy.y, t.on2);
    }
}

// One consumer warp's share of a unit (blob at shared address sblob): tasks
// t0, t0 + tstep, ... of the unit's task table (written at pack time in an
// order that balances the warps of this deal). Each group's result goes to its
// slot in the stage's slot array at shared address slots.
template <int NX>
__device__ __forceinline__ void consume_unit(const TablesT<NX>& T, uint32_t sblob, uint32_t slots, int t0, int tstep,
                                             int lane) {
    const uint32_t hw = lds_u32(sblob + offsetof(UnitHeader, ntask));     // ntask | task16 << 16
    const int ntask = (int)(hw & 0xFFFFu);
    const uint32_t tasks = sblob + (hw >> 16) * 16;
    for (int k = t0; k < ntask; k += tstep) {
        const uint4 d = lds_u32x4(tasks + k * 16);
        const uint32_t w = (d.x >> 26) & 3u;
        if (w == 0) body1<NX>(T, task64(sblob, d, lane), slots);
        else if (w == 1) body2<NX>(T, task32(sblob, d, lane, 16), slots);
        else if (w == 2) body4<NX>(T, task32(sblob, d, lane, 32), slots, lane);
        else body8<NX>(T, task32(sblob, d, lane, 64), slots, lane);
    }
}

// Single-width units (every group of the matrix at width index W, items in
// (column, row) order, n = rows x cols of them): warp task k covers items
// SPAN k .. SPAN k + SPAN - 1 (64 at one bit, two per lane; 32 otherwise),
// and every item's column and row follow from its index, so the unit's task
// table, row bytes and column ends are neither read nor copied.
__device__ __forceinline__ void item_pos(int i, int rows, int& c, uint32_t& r) {
    if (rows == RB) {
        c = i >> 7;
        r = (uint32_t)(i & (RB - 1));
    } else {
        c = i / rows;
        r = (uint32_t)(i - c * rows);
    }
}
static_assert(RB == 128, "item_pos shifts by log2(RB)");

template <int NX, int W>
__device__ __forceinline__ void consume_single_w(const TablesT<NX>& T, uint32_t sblob, uint32_t slots, int t0,
                                                 int tstep, int lane, int rows) {
    const int n = (int)lds_u16(sblob + offsetof(UnitHeader, n) + 2 * W);
    const uint32_t pay = sblob + lds_u16(sblob + offsetof(UnitHeader, pay16) + 2 * W) * 16;
    const uint32_t sc = sblob + lds_u16(sblob + offsetof(UnitHeader, sc16) + 2 * W) * 16;
    constexpr int SPAN = W == 0 ? TASK_SPAN1 : TASK_SPAN, BPI = 8 << W;
    const int ntask = (n + SPAN - 1) / SPAN;
    for (int k = t0; k < ntask; k += tstep) {
        const int cnt = min(SPAN, n - SPAN * k);
        Task t;
        if (W == 0) {
            // lane l: items 2l and 2l + 1 (an even first item: one 16-byte payload
            // load, one 4-byte scale load); past the end, the task's first pair
            const int j = 2 * lane;
            t.on = j < cnt;
            t.on2 = j + 1 < cnt;
            const int ii = SPAN * k + (t.on ? j : 0);
            item_pos(ii, rows, t.c, t.r);
            if (t.on2 && (int)t.r + 1 == rows) { t.c2 = t.c + 1; t.r2 = 0; }
            else { t.c2 = t.c; t.r2 = t.on2 ? t.r + 1 : t.r; }
            t.pay = pay + ii * 8;
            t.sc = sc + 2 * ii;
            body1<NX>(T, t, slots);
        } else {
            t.on = lane < cnt;
            t.on2 = false;
            const int ii = SPAN * k + (t.on ? lane : 0);
            item_pos(ii, rows, t.c, t.r);
            t.c2 = t.c;
            t.r2 = t.r;
            t.pay = pay + ii * BPI;
            t.sc = sc + 2 * ii;
            if (W == 1) body2<NX>(T, t, slots);
            else if (W == 2) body4<NX>(T, t, slots, lane);
            else body8<NX>(T, t, slots, lane);
        }
    }
}

template <int NX>
__device__ __forceinline__ void consume_single(const TablesT<NX>& T, uint32_t sblob, uint32_t slots, int t0, int tstep,
                                               int lane, int rows, int w) {
    if (w == 0) consume_single_w<NX, 0>(T, sblob, slots, t0, tstep, lane, rows);
    else if (w == 1) consume_single_w<NX, 1>(T, sblob, slots, t0, tstep, lane, rows);
    else if (w == 2) consume_single_w<NX, 2>(T, sblob, slots, t0, tstep, lane, rows);
    else consume_single_w<NX, 3>(T, sblob, slots, t0, tstep, lane, rows);
}

// A unit's copy: the whole blob, or for a single-width matrix (SW) only the
// header, payload and scales at its start.
template <bool SW>
__device__ __forceinline__ void issue_unit_g1(const LayoutView& L, int u, uint32_t dst, uint32_t bar) {
    if constexpr (SW) {
        const int rb = u % L.nrb, sl = u / L.nrb;
        const int rows = min(RB, (int)(L.N - (int64_t)rb * RB)), cols = min(L.C, L.G - sl * L.C);
        bulk_load(dst, L.blobs + (int64_t)L.blob_off[u] * 16, single_prefix16((uint32_t)(rows * cols), L.single_w) * 16u,
                  bar);
    } else {
        issue_unit(L, u, dst, bar);
    }
}

// SwiGLU epilogue of a gate-up product whose rows alternate (row 2i the gate
// of feature i, row 2i + 1 its up projection): h_i = silu(g_i) * u_i, rounded
// to BF16 (to nearest even), the input format of the down projection.
__device__ __forceinline__ uint16_t swiglu_bf16(float g, float u) {
    return __bfloat16_as_ushort(__float2bfloat16_rn(swiglu_f32(g, u)));
}

// Several slabs per row: after adding a unit's rows into y, the copier adds 1
// to its row block's slab count (reset by the zeroing owner of slab 0 before
// it publishes its flag) with an acquire-release RMW by lane 0, ordered after
// the warp's additions by the preceding __syncwarp. The RMW's reply is read one
// unit later, so its round trip overlaps the next unit. The adder whose RMW
// brings the count to S writes the row block's 64 outputs: its lane 0 has
// acquired every slab's additions, and the warp barrier (which orders memory
// among the warp's lanes) passes them on to the lanes' GPU-scope loads.
__device__ __forceinline__ void swiglu_rows(const LayoutView& L, const float* y, uint16_t* h, int rb, int lane) {
    const int rows = min(RB, (int)(L.N - (int64_t)rb * RB));
    const float* yr = y + (int64_t)rb * RB;
    uint16_t* hr = h + (int64_t)rb * (RB / 2);
    for (int p = lane; 2 * p < rows; p += 32) {
        const float2 gu = ld_relaxed_gpu_f32x2(yr + 2 * p);
        hr[p] = swiglu_bf16(gu.x, gu.y);
    }
}

// Split-K for one copier: true once every row block it adds into (units
// u_begin + j for j = cp, cp + step, ... below n) has been zeroed in this call
// (flag == epoch), within the wait limit. Copier 0 zeroes this block's own
// slab-0 rows, so it skips those; the others wait for them like any other.
// Lane i watches the copier's units i, i + 32, ...; acquire loads.
__device__ __forceinline__ bool copier_flags_ready(const LayoutView& L, uint32_t epoch, int u_begin, int n, int cp,
                                                   int step, int lane) {
    bool seen = true;
    const unsigned long long t0 = global_ns();
    for (int j = cp + step * lane; j < n && seen; j += 32 * step) {
        const int u = u_begin + j;
        if (u >= L.nrb || cp != 0) {
            const uint32_t* f = L.ctl + 2 + (u % L.nrb);
            while (!(seen = ld_acquire_gpu(f) == epoch))
                if (global_ns() - t0 > WAIT_LIMIT_NS) break;
        }
    }
    __syncwarp();                       // every lane's later additions after every acquire
    return __all_sync(0xffffffffu, seen);
}

// Consumer warps of one team (named barrier 2 + team; tw warps).
__device__ __forceinline__ void team_sync(int team, int tw) {
    asm volatile("bar.sync %0, %1;" :: "r"(2 + team), "r"(32 * tw) : "memory");
}

// A team's cooperative flush of a finished unit: warp wt of tw takes rows
// [wt * 128 / tw, (wt + 1) * 128 / tw), tw / 4 lanes per row, each lane
// summing 64 / tw of the row's 16 slots (16-byte chunks; absent columns hold
// 0), then the row's lanes added by xor shuffles in a fixed order. Rows are
// stored when the matrix has one slab and added otherwise.
template <int NX>
__device__ __forceinline__ void team_flush(const TablesT<NX>& T, const LayoutView& L, float* __restrict__ y, int st,
                                           int rb, int wt, int tw, int lane) {
    const int lpr = tw >> 2;                    // lanes per row: 4 (16 warps) or 2 (8 warps)
    const int rpw = 32 / lpr;                   // rows per warp
    const int r = wt * rpw + lane / lpr, part = lane % lpr;
    const int rows = min(RB, (int)(L.N - (int64_t)rb * RB));
    const int chunks = 4 / lpr;                 // 16-byte chunks per lane
#pragma unroll
    for (int v = 0; v < NX; ++v) {
        const uint32_t ra = smem_u32(T.slots[st][v]) + (uint32_t)r * 64;
        float sum = 0.f;
        for (int k = 0; k < chunks; ++k) {
            const float4 a = lds_f32x4(ra + ((part * chunks + k) << 4));
            sum += (a.x + a.y) + (a.z + a.w);
        }
        for (int o = 1; o < lpr; o <<= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
        if (part == 0 && r < rows) {
            float* yr = y + (int64_t)v * L.N + (int64_t)rb * RB + r;
            if (L.S == 1) *yr = sum;
            else red_global(yr, sum);
        }
    }
}

// NX activation vectors x (NX x K, row-major) and outputs y (NX x N). SW: the
// matrix has a single width (L.single_w >= 0; see consume_single).
template <int NX, int MODE, bool SW = false>
__global__ void __launch_bounds__(G1_THREADS, 1) gemv1_kernel(LayoutView L, const uint16_t* __restrict__ x,
                                                              float* __restrict__ y, int dep,
                                                              uint16_t* __restrict__ h,
                                                              const float* __restrict__ gu) {
    static_assert(MODE == MODE_PLAIN || NX == 1, "the SwiGLU forms take one activation vector");
    constexpr int NSTAGE = Geo<NX>::nstage;
    static_assert(NSTAGE % NCOPY == 0, "each stage belongs to one copier");
    // each team flushes its own last unit (the copiers would add a hand-off
    // at the very end of the block); the SwiGLU epilogue stays with the copiers
    constexpr bool COOP = MODE != MODE_SWIGLU_EPI;
    extern __shared__ __align__(16) unsigned char smem_raw[];
    // stages and tables on a 256-byte boundary: lookups merge a byte into table addresses
    unsigned char* base = smem_raw + ((256u - (smem_u32(smem_raw) & 255u)) & 255u);
    TablesT<NX>& T = *reinterpret_cast<TablesT<NX>*>(base + (size_t)NSTAGE * STAGE_BYTES);
    const uint32_t stage0 = smem_u32(base);
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int P = gridDim.x, p = blockIdx.x;
    // balanced contiguous split of the units over the blocks
    const int per = L.units / P, extra = L.units - per * P;
    const int u_begin = p * per + min(p, extra), u_end = u_begin + per + (p < extra ? 1 : 0);
    const int n_units = u_end - u_begin;
    if (n_units <= 0) return;
    const int s0 = u_begin / L.nrb, rb0 = u_begin - s0 * L.nrb;
    // more units per block -> more teams: each warp then covers more groups per
    // unit (less per-unit overhead); few units -> whole-block teams (less latency)
    // two teams once the block has 4 units: each team then has NSTAGE / 2
    // stages, so its next blob lands while it works on the current one
    const int lg_teams = Geo<NX>::max_teams == 2 && n_units >= 4 ? 1 : 0;
    const int teams = 1 << lg_teams, tw = NCW >> lg_teams;

    const uint32_t full0 = smem_u32(&T.full[0]), empty0 = smem_u32(&T.empty[0]);
    const uint32_t abort_addr = smem_u32(&T.abort);
    if (tid == 0) {
        for (int i = 0; i < NSTAGE; ++i) {
            mbar_init(full0 + 8 * i, 1);
            mbar_init(empty0 + 8 * i, tw);
        }
        T.abort = 0;
        T.sk_ok = 0;
        fence_barrier_init();
    }
    // slots no group of a unit writes (rows past N, columns past the last
    // slab's) must read as zero; the copier re-zeroes every slot it sums
    for (int i = tid; i < NSTAGE * NX * SLOT_FLOATS; i += G1_THREADS) (&T.slots[0][0][0])[i] = 0.f;
    __syncthreads();
    if (tid == 0) {
        const int first = n_units < NSTAGE ? n_units : NSTAGE;
        for (int j = 0; j < first; ++j) issue_unit_g1<SW>(L, u_begin + j, stage0 + j * STAGE_BYTES, full0 + 8 * j);
    }
    // Weights never depend on earlier work in the stream, so the first copies
    // are in flight before this grid waits for its predecessor (programmatic
    // dependent launch); x, y and the control words are read only after. The
    // first slab's activations are prefetched into L2 meanwhile.
    {
        const int64_t k0 = (int64_t)s0 * L.C * GROUP;
        if constexpr (MODE == MODE_SWIGLU_IN) {      // 8 bytes (a gate-up pair) per activation
            const int lines = (min(L.C, L.G - s0 * L.C) * GROUP * 8 + 127) / 128;
            if (tid >= 32 * NCOPY && tid - 32 * NCOPY < lines) prefetch_l2(gu + 2 * k0 + (int64_t)(tid - 32 * NCOPY) * 32);
        } else {
            const int lines = (min(L.C, L.G - s0 * L.C) * GROUP * 2 + 127) / 128;
            if (tid >= 32 * NCOPY && tid - 32 * NCOPY < NX * lines) {
                const int v = (tid - 32 * NCOPY) / lines, ln = (tid - 32 * NCOPY) - v * lines;
                prefetch_l2(x + (int64_t)v * L.K + k0 + (int64_t)ln * 64);
            }
        }
    }
    // Ordering against the previous kernel on the stream (see Dep):
    if (dep != DEP_GROUP_FIRST) asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    if (dep != DEP_GROUP_NEXT) asm volatile("griddepcontrol.wait;" ::: "memory");
    if (dep == DEP_GROUP_FIRST) asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

    if (warp < NCOPY) {
        // ---- copiers: split-K zeroing, then per unit j = cp, cp + NCOPY, ...:
        // rows out, next copy in (copier cp owns the stages s = cp mod NCOPY) ----
        const int cp = warp;
        uint32_t epoch = 0;
        if (L.S > 1) {
            // the call count's load is in flight while copier 0 zeroes (the
            // zeros do not depend on it; the flags it publishes do)
            const unsigned long long count = call_count_raw(L.ctl);
            if (cp == 0) {
                // zero y for the row blocks whose slab 0 this block owns (units
                // u < nrb) and publish them
                const int z_end = min(u_end, L.nrb);
                for (int u = u_begin; u < z_end; ++u) {
                    const int rows = min(RB, (int)(L.N - (int64_t)u * RB));
#pragma unroll
                    for (int v = 0; v < NX; ++v) {
                        float* dst = y + (int64_t)v * L.N + (int64_t)u * RB;
                        for (int r = lane; r < rows; r += 32) dst[r] = 0.f;
                    }
                }
                __syncwarp();
            }
            epoch = epoch_of(count);
            if (cp == 0) {
                const int z_end = min(u_end, L.nrb);
                // release stores, one unit per lane in parallel: the warp's zeros
                // (ordered by __syncwarp) before each flag
                for (int u = u_begin + lane; u < z_end; u += 32) {
                    if (MODE == MODE_SWIGLU_EPI) L.ctl[2 + L.nrb + u] = 0u;     // SwiGLU slab count, before the flag's release
                    st_release_gpu(L.ctl + 2 + u, epoch);
                }
            }
        }
        bool dead = false;
        // a row block this copier adds into that was never zeroed in time (the
        // other copiers also wait for copier 0's zeroing of this block's own rows)
        if (L.S > 1 && !copier_flags_ready(L, epoch, u_begin, n_units, cp, NCOPY, lane)) {
            dead = true;
            if (lane == 0) raise_abort(&T.abort);
        }
        // the flags this warp acquired, passed on to the consumers' final flush
        if (L.S > 1 && lane == 0) red_release_cta_shared_add(smem_u32(&T.sk_ok), dead ? 0x10000u : 1u);
        int jdone = -1;                 // the last unit this copier flushed (and refilled after)
        int pend_rb = -1;               // SwiGLU: row block whose slab count's reply is pending
        uint32_t pend_count = 0;        // (lane 0) that count before this copier's addition
        for (int j = cp; j < n_units; j += NCOPY) {
            if (COOP && j >= n_units - teams) break;          // each team flushes its last unit itself
            const int st = j & (NSTAGE - 1);
            const uint32_t par = (uint32_t)(j / NSTAGE) & 1u;
            const int u = u_begin + j, rbw = u % L.nrb, sw = u / L.nrb;
            // nap between polls, except on the block's last units, whose rows end the block
            if (!dead && !warp_wait(empty0 + 8 * st, par, abort_addr, j + NCOPY < n_units ? 256 : 0)) {
                dead = true;
                if (lane == 0) raise_abort(&T.abort);
            }
            if (!dead) {
                const int rows = min(RB, (int)(L.N - (int64_t)rbw * RB));
                // the stage's next unit rewrites every slot this one wrote unless it
                // has fewer columns (the last, partial slab): zero only then
                const int cols = min(L.C, L.G - sw * L.C);
                const int un = u + NSTAGE;
                const bool rezero = j + NSTAGE < n_units && min(L.C, L.G - (un / L.nrb) * L.C) < cols;
#pragma unroll
                for (int v = 0; v < NX; ++v)            // per vector: its slots into its row of y
#pragma unroll
                for (int q = 0; q < RB / 32; ++q) {
                    const uint32_t sl = smem_u32(T.slots[st][v]);
                    float* yr = y + (int64_t)v * L.N + (int64_t)rbw * RB;
                    // row r's 16 slots as four 16-byte chunks, chunk (k + (lane >> 1)) & 3
                    // at step k (each quarter-warp touches 8 distinct bank groups);
                    // summed as a tree
                    const int r = lane + 32 * q;
                    const uint32_t ra = sl + (uint32_t)r * 64;
                    float4 a4[4];
#pragma unroll
                    for (int k = 0; k < 4; ++k) a4[k] = lds_f32x4(ra + (((k + (lane >> 1)) & 3) << 4));
                    if (rezero) {
#pragma unroll
                        for (int k = 0; k < 4; ++k) sts_zero4(ra + (((k + (lane >> 1)) & 3) << 4));
                    }
                    const float sum = (((a4[0].x + a4[0].y) + (a4[0].z + a4[0].w)) + ((a4[1].x + a4[1].y) + (a4[1].z + a4[1].w))) +
                                      (((a4[2].x + a4[2].y) + (a4[2].z + a4[2].w)) + ((a4[3].x + a4[3].y) + (a4[3].z + a4[3].w)));
                    if (r < rows) {
                        if (L.S == 1) yr[r] = sum;
                        else red_global(yr + r, sum);
                    }
                    if (MODE == MODE_SWIGLU_EPI && L.S == 1) {
                        // the row is complete: gate (even row) and up (odd row) sit in
                        // neighbouring lanes
                        const float up = __shfl_xor_sync(0xffffffffu, sum, 1);
                        if (!(lane & 1) && r < rows) h[((int64_t)rbw * RB + r) >> 1] = swiglu_bf16(sum, up);
                    }
                }
                __syncwarp();
                if (j + NSTAGE < n_units && lane == 0)
                    issue_unit_g1<SW>(L, u_begin + j + NSTAGE, stage0 + st * STAGE_BYTES, full0 + 8 * st);
                jdone = j;
                if (MODE == MODE_SWIGLU_EPI && L.S > 1) {
                    // SwiGLU: count this unit's slab, then act on the previous unit's count
                    uint32_t count = 0;
                    if (lane == 0) count = atom_add_acq_rel_gpu(L.ctl + 2 + L.nrb + rbw, 1u);
                    if (pend_rb >= 0 && __shfl_sync(0xffffffffu, pend_count, 0) + 1u == (uint32_t)L.S) {
                        __syncwarp();
                        swiglu_rows(L, y, h, pend_rb, lane);
                    }
                    pend_rb = rbw;
                    pend_count = count;
                }
            }
        }
        if (MODE == MODE_SWIGLU_EPI && L.S > 1 && pend_rb >= 0) {
            if (__shfl_sync(0xffffffffu, pend_count, 0) + 1u == (uint32_t)L.S) {
                __syncwarp();
                swiglu_rows(L, y, h, pend_rb, lane);
            }
        }
        if (dead && lane == 0) {
            // let every copy this copier's stages received land before the block
            // exits: units below NSTAGE were issued at the start, and each flushed
            // unit j issued j + NSTAGE, so the last unit issued into stage i is the
            // largest k = i mod NSTAGE below both n_units and jdone + NSTAGE + 1;
            // wait for it with its parity (a completed phase returns at once)
            const int kmax = min(n_units - 1, max(jdone + NSTAGE, NSTAGE - 1));
            for (int i = cp; i < NSTAGE; i += NCOPY) {
                if (i > kmax) continue;
                const int k = kmax - ((kmax - i) % NSTAGE);
                mbar_wait_bounded(full0 + 8 * i, (uint32_t)((k / NSTAGE) & 1));
            }
        }
        if (cp == 0 && L.S > 1 && lane == 0) call_done(L.ctl);      // this block's share of the call count
        // a grouped product that started without waiting completes only after
        // its predecessor, so completion stays in stream order
        if (cp == 0 && dep == DEP_GROUP_NEXT && lane == 0) asm volatile("griddepcontrol.wait;" ::: "memory");
    } else {
        // ---- consumers: team `team` takes units j = team, team + teams, ... ----
        const int cw = warp - NCOPY, ct = tid - 32 * NCOPY, team = cw / tw, wt = cw - team * tw;
        const int s_last = (u_end - 1) / L.nrb;
        bool dead = false;
        int cur = s0;
        int rbj = rb0 + team, sj = s0;                  // row block and slab of unit j
        while (rbj >= L.nrb) { rbj -= L.nrb; ++sj; }
        build_tables<NX, MODE>(T, L, x, gu, s0, ct);
        for (int j = team; j < n_units; j += teams) {
            // every consumer warp rebuilds the tables at every slab boundary of the
            // block's range, in order (the rebuild's named barrier waits for all)
            while (cur < sj) build_tables<NX, MODE>(T, L, x, gu, ++cur, ct);
            const int st = j & (NSTAGE - 1);
            const uint32_t par = (uint32_t)(j / NSTAGE) & 1u;
            if (!dead && !warp_wait(full0 + 8 * st, par, abort_addr)) { dead = true; if (lane == 0) raise_abort(&T.abort); }
            if (!dead) {
                // the deal rotates by 5 warps from unit to unit (coprime with tw), so a
                // warp's bins differ from unit to unit
                const int t0 = (wt - 5 * (j >> lg_teams)) & (tw - 1);
                if constexpr (SW)
                    consume_single<NX>(T, stage0 + st * STAGE_BYTES, smem_u32(T.slots[st][0]), t0, tw, lane,
                                       min(RB, (int)(L.N - (int64_t)rbj * RB)), L.single_w);
                else
                    consume_unit<NX>(T, stage0 + st * STAGE_BYTES, smem_u32(T.slots[st][0]), t0, tw, lane);
                __syncwarp();
                if (!(COOP && j >= n_units - teams) && lane == 0) mbar_arrive(empty0 + 8 * st);
            }
            if (COOP && j >= n_units - teams) {
                // the team's last unit: every warp of the team flushes 128 / tw of its rows
                team_sync(team, tw);
                if (L.S > 1) {
                    // split-K: after the copiers' flag checks (bounded wait)
                    uint32_t g = 0;
                    const unsigned long long w0 = global_ns();
                    while ((g = ld_acquire_cta_shared(smem_u32(&T.sk_ok))) < (uint32_t)NCOPY &&
                           !lds_volatile(abort_addr) && global_ns() - w0 < WAIT_LIMIT_NS)
                        __nanosleep(32);
                    if (g != (uint32_t)NCOPY) {
                        dead = true;
                        if (lane == 0) raise_abort(&T.abort);
                    }
                }
                if (!dead) team_flush<NX>(T, L, y, st, rbj, wt, tw, lane);
            }
            rbj += teams;
            while (rbj >= L.nrb) { rbj -= L.nrb; ++sj; }
        }
        while (cur < s_last) build_tables<NX, MODE>(T, L, x, gu, ++cur, ct);   // boundaries past this team's last unit
    }
}

// ---------------------------------------------------------------------------
// Chains: a sequence of batch-1 products in one persistent launch (one block
// per SM). The chain keeps its own control words and never touches its
// layouts' split-K words. Weights never depend on activations, so each block's copier
// streams the unit blobs of its share of every product back to back, across
// product boundaries, while a product that waits for earlier ones (a decode
// chain: each input derives from earlier outputs) reads its x only once their
// completion counts say so (the consumers wait before building the product's
// tables). Each block adds 1 to a product's count (a release reduction) after
// its last write of that product's y, including blocks that hold none of its
// units; in launch e (1-based, from the chain's call counter) a product is
// complete once its count reaches e * P. A block with units of a product adds
// to its count only after flushing units its consumers computed after that
// product's wait, so a count at e * P implies that every earlier product the
// product waited for is complete too.
// ---------------------------------------------------------------------------

// Units [ub, ue) of product i that block p owns.
__device__ __forceinline__ void chain_range(const ChainItem* items, int i, int p, int P, int& ub, int& ue) {
    const int units = items[i].L.units;
    int q = p - items[i].rot;
    if (q < 0) q += P;
    const int per = units / P, extra = units - per * P;
    ub = q * per + min(q, extra);
    ue = ub + per + (q < extra ? 1 : 0);
}

// A position in a block's unit sequence: unit u of product i, whose range ends at ue.
struct ChainCursor {
    int i, u, ue;
};

// Move to the next unit of the block's sequence (products in order, empty
// ranges skipped); false past the end.
__device__ __forceinline__ bool chain_next(const ChainItem* items, int count, int p, int P, ChainCursor& c) {
    if (++c.u < c.ue) return true;
    while (++c.i < count) {
        chain_range(items, c.i, p, P, c.u, c.ue);
        if (c.u < c.ue) return true;
    }
    c.i = count;
    c.u = c.ue = 0;
    return false;
}

// True once products from .. to - 1 are complete (count >= target, compared
// modulo 2^32), within the wait limit. A whole warp: lane l watches products
// from + l, from + l + 32, ...; the counts are read with acquire loads.
__device__ __forceinline__ bool chain_deps_ready(const uint32_t* done, int from, int to, uint32_t target, int lane) {
    bool seen = true;
    const unsigned long long t0 = global_ns();
    for (int j = from + lane; j < to && seen; j += 32) {
        while (!(seen = (int)(ld_acquire_gpu(done + j) - target) >= 0)) {
            if (global_ns() - t0 > WAIT_LIMIT_NS) break;
            __nanosleep(32);            // a light backoff: two pollers per block share the count's L2 line
        }
    }
    __syncwarp();
    return __all_sync(0xffffffffu, seen);
}

// When the copier's issue position enters a new (product, slab), bring that
// slab's activations into L2 (a prefetch reads no value, so it is safe however
// far ahead of the product's dependencies it runs): lane l the l-th 128-byte
// line of the slab's x.
__device__ __forceinline__ void chain_prefetch_x(const ChainItem* items, const ChainCursor& c, int& pf_i, int& pf_s,
                                                 int lane) {
    const int nrb = items[c.i].L.nrb, s = c.u / nrb;
    if (c.i == pf_i && s == pf_s) return;
    pf_i = c.i;
    pf_s = s;
    const int C = items[c.i].L.C, G = items[c.i].L.G;
    const int lines = min(C, G - s * C);                // 64 BF16 activations = one line per group column
    if (lane < lines) prefetch_l2(items[c.i].x + ((int64_t)s * C + lane) * GROUP);
}

__global__ void __launch_bounds__(CH_THREADS, 1) gemv_chain_kernel(const ChainItem* __restrict__ items, int count,
                                                                   uint32_t* __restrict__ cctl) {
    constexpr int NSTAGE = Geo<1>::nstage;
    // one team: every consumer warp works on every unit (a chain's products are
    // serialised, so a unit's latency is what counts; with two teams a block
    // holding one unit of a product computes it on half its warps)
    constexpr int TW = NCW;
    extern __shared__ __align__(16) unsigned char smem_raw[];
    unsigned char* base = smem_raw + ((256u - (smem_u32(smem_raw) & 255u)) & 255u);
    TablesT<1>& T = *reinterpret_cast<TablesT<1>*>(base + (size_t)NSTAGE * STAGE_BYTES);
    const uint32_t stage0 = smem_u32(base);
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int P = gridDim.x, p = blockIdx.x;
    uint32_t* done = cctl + 2;

    const uint32_t full0 = smem_u32(&T.full[0]), empty0 = smem_u32(&T.empty[0]);
    const uint32_t abort_addr = smem_u32(&T.abort);
    if (tid == 0) {
        for (int i = 0; i < NSTAGE; ++i) {
            mbar_init(full0 + 8 * i, 1);
            mbar_init(empty0 + 8 * i, TW);
        }
        T.abort = 0;
        fence_barrier_init();
    }
    for (int i = tid; i < NSTAGE * SLOT_FLOATS; i += CH_THREADS) (&T.slots[0][0][0])[i] = 0.f;
    __syncthreads();
    // the copier's issue position, and the first copies (weights only: before
    // the wait for the previous kernel)
    ChainCursor is{-1, 0, 0};
    int issued = 0, pf_i = -1, pf_s = -1;
    if (warp == 0) {
        while (issued < NSTAGE && chain_next(items, count, p, P, is)) {
            if (lane == 0) issue_unit(items[is.i].L, is.u, stage0 + issued * STAGE_BYTES, full0 + 8 * issued);
            chain_prefetch_x(items, is, pf_i, pf_s, lane);
            ++issued;
        }
    }
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    asm volatile("griddepcontrol.wait;" ::: "memory");
    const uint32_t target = call_epoch(cctl) * (uint32_t)P;
    uint32_t* zeroed = cctl + 2 + count;
    // Split-K for the whole chain at once: every block zeroes the rows of the
    // slab-0 units it owns in every product whose rows span several slabs (no
    // y is an input of the chain, so this may run ahead of any product), then
    // counts itself in `zeroed`; a copier adds into y only once every block
    // has (one grid-wide wait per launch instead of flags per product).
    for (int i = warp; i < count; i += CH_THREADS / 32) {
        const LayoutView& Li = items[i].L;
        if (Li.S > 1) {
            int ub, ue;
            chain_range(items, i, p, P, ub, ue);
            float* y = items[i].y;
            const int z_end = min(ue, Li.nrb);
            for (int u = ub; u < z_end; ++u) {
                const int rows = min(RB, (int)(Li.N - (int64_t)u * RB));
                for (int r = lane; r < rows; r += 32) y[(int64_t)u * RB + r] = 0.f;
            }
        }
    }
    __syncthreads();
    if (tid == 0) red_release_gpu_add(zeroed, 1u);

    if (warp == 0) {
        // ---- copier: per product, split-K zeroing, then per unit rows out and
        // the next copy of the block's sequence in; then the product's count ----
        bool dead = false, zero_seen = false;
        int st = 0;
        uint32_t par = 0;
        for (int i = 0; i < count; ++i) {
            const LayoutView L = items[i].L;
            float* y = items[i].y;
            int ub, ue;
            chain_range(items, i, p, P, ub, ue);
            if (ub < ue) {
                // no dependency wait here: y's values come from units the consumers
                // compute only after the product's dependencies
                if (!dead && L.S > 1 && !zero_seen) {
                    if (!chain_deps_ready(zeroed, 0, 1, target, lane)) {
                        dead = true;
                        if (lane == 0) raise_abort(&T.abort);
                    }
                    zero_seen = true;
                }
                for (int u = ub; u < ue; ++u) {
                    if (!dead && !warp_wait(empty0 + 8 * st, par, abort_addr, 0)) {
                        dead = true;
                        if (lane == 0) raise_abort(&T.abort);
                    }
                    if (!dead) {
                        const int rb = u % L.nrb;
                        const int rows = min(RB, (int)(L.N - (int64_t)rb * RB));
                        const uint32_t sl = smem_u32(T.slots[st][0]);
                        float* yr = y + (int64_t)rb * RB;
#pragma unroll
                        for (int q = 0; q < RB / 32; ++q) {
                            const int r = lane + 32 * q;
                            const uint32_t ra = sl + (uint32_t)r * 64;
                            float4 a[4];
#pragma unroll
                            for (int k = 0; k < 4; ++k) a[k] = lds_f32x4(ra + (((k + (lane >> 1)) & 3) << 4));
#pragma unroll
                            for (int k = 0; k < 4; ++k) sts_zero4(ra + (((k + (lane >> 1)) & 3) << 4));
                            const float sum = (((a[0].x + a[0].y) + (a[0].z + a[0].w)) + ((a[1].x + a[1].y) + (a[1].z + a[1].w))) +
                                              (((a[2].x + a[2].y) + (a[2].z + a[2].w)) + ((a[3].x + a[3].y) + (a[3].z + a[3].w)));
                            if (r < rows) {
                                if (L.S == 1) yr[r] = sum;
                                else red_global(yr + r, sum);
                            }
                        }
                        __syncwarp();
                        if (chain_next(items, count, p, P, is)) {      // the unit NSTAGE ahead, into the freed stage
                            if (lane == 0) issue_unit(items[is.i].L, is.u, stage0 + st * STAGE_BYTES, full0 + 8 * st);
                            chain_prefetch_x(items, is, pf_i, pf_s, lane);
                            ++issued;
                        }
                    }
                    if (++st == NSTAGE) { st = 0; par ^= 1; }
                }
            }
            // this block is done with product i (its writes of y, ordered before
            // the release by the warp barrier); every block counts every product
            __syncwarp();
            if (lane == 0) red_release_gpu_add(done + i, 1u);
        }
        if (dead && lane == 0) {
            for (int i = 0; i < NSTAGE && i < issued; ++i) {
                const int jl = i + ((issued - 1 - i) / NSTAGE) * NSTAGE;   // last unit issued into stage i
                mbar_wait_bounded(full0 + 8 * i, (uint32_t)((jl / NSTAGE) & 1));
            }
        }
        if (lane == 0) call_done(cctl);
    } else {
        // ---- consumers: every warp takes part in every unit, rebuilding the
        // tables at every (product, slab) boundary of the block's sequence ----
        const int wt = warp - 1, ct = tid - 32;
        bool dead = false;
        ChainCursor c{-1, 0, 0};
        int tb_i = -1, tb_s = -1;
        LayoutView L = items[0].L;
        const uint16_t* x = items[0].x;
        for (int j = 0; chain_next(items, count, p, P, c); ++j) {
            const bool new_product = c.i != tb_i;
            if (new_product) {
                L = items[c.i].L;
                x = items[c.i].x;
                const int wf = items[c.i].wait_from, wh = items[c.i].wait_hi;
                // the first consumer warp waits for the product's dependencies; the
                // table build's barrier holds the others until it is through
                if (ct < 32 && !dead && wf < wh && !chain_deps_ready(done, wf, wh, target, lane)) {
                    dead = true;
                    if (lane == 0) raise_abort(&T.abort);
                }
            }
            const int sj = c.u / L.nrb;
            if (new_product || sj != tb_s) {
                build_tables<1, MODE_PLAIN>(T, L, x, nullptr, sj, ct);
                tb_i = c.i;
                tb_s = sj;
            }
            {
                const int st = j & (NSTAGE - 1);
                const uint32_t par = (uint32_t)(j / NSTAGE) & 1u;
                if (!dead && !warp_wait(full0 + 8 * st, par, abort_addr)) { dead = true; if (lane == 0) raise_abort(&T.abort); }
                if (!dead) {
                    // the deal rotates by 5 warps from unit to unit
                    const int t0 = (wt - 5 * j) & (TW - 1);
                    consume_unit<1>(T, stage0 + st * STAGE_BYTES, smem_u32(T.slots[st][0]), t0, TW, lane);
                    __syncwarp();
                    if (lane == 0) mbar_arrive(empty0 + 8 * st);
                }
            }
        }
    }
}

template <int NX, int MODE = MODE_PLAIN, bool SW = false>
cudaError_t launch_gemv1(const LayoutView& L, const uint16_t* x, float* y, cudaStream_t s, int dep,
                         uint16_t* h = nullptr, const float* gu = nullptr) {
    static LaunchPrep prep;
    int sms = 0;
    cudaError_t e = prep.get(gemv1_kernel<NX, MODE, SW>, gemv1_smem<NX>(), &sms);
    if (e != cudaSuccess) return e;
    const int grid = L.units < sms ? L.units : sms;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(G1_THREADS);
    cfg.dynamicSmemBytes = gemv1_smem<NX>();
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, gemv1_kernel<NX, MODE, SW>, L, x, y, dep, h, gu);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace

int device_sms(int* sms) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(sms, cudaDevAttrMultiProcessorCount, dev);
    return (int)e;
}

cudaError_t launch_chain(const ChainItem* items, int count, uint32_t* cctl, int blocks, cudaStream_t s) {
    static LaunchPrep prep;
    int sms = 0;
    const cudaError_t pe = prep.get(gemv_chain_kernel, gemv1_smem<1>(), &sms);
    if (pe != cudaSuccess) return pe;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(blocks);
    cfg.blockDim = dim3(CH_THREADS);
    cfg.dynamicSmemBytes = gemv1_smem<1>();
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    const cudaError_t e = cudaLaunchKernelEx(&cfg, gemv_chain_kernel, items, count, cctl);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Batch 1 with the split-K control words in a fixed device array instead of
// the layout's own allocation (for callers that cannot allocate device
// memory; see vbq_gemv_static in vbq.h). Every call on a device shares the
// array: words 0-1 the call counter (each call adds exactly 2^CALL_SHIFT,
// whatever its grid), words 2.. the per-row-block zeroed flags. Epochs only
// grow, so flags left by earlier calls never match the current one. Calls
// that overlap on the GPU race on the array.
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
    LayoutView Ls = L;
    Ls.ctl = ctl;
    return launch_gemv1<1>(Ls, x, y, s, DEP_BEFORE);
}

// ---------------------------------------------------------------------------
// Failure report of the bounded waits, and its self-test.
// ---------------------------------------------------------------------------

namespace {

// One block: thread 0 waits on a barrier that nothing completes, bounded to
// limit_ns, and records the timeout the way the product kernels do.
__global__ void selftest_timeout_kernel(unsigned long long limit_ns) {
    __shared__ __align__(8) unsigned long long bar;
    const uint32_t b = smem_u32(&bar);
    if (threadIdx.x == 0) {
        mbar_init(b, 1);
        fence_barrier_init();
        const unsigned long long t0 = global_ns();
        bool done = false;
        while (!(done = mbar_try_wait_sleep(b, 0))) {
            if (global_ns() - t0 > limit_ns) break;
        }
        if (!done) atomicOr(&g_device_status, VBQ_DEVICE_TIMEOUT);
    }
}

}  // namespace

cudaError_t read_device_status(uint32_t* status, cudaStream_t s) {
    cudaError_t e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return e;
    uint32_t mine = 0, gemm = 0;
    if ((e = cudaMemcpyFromSymbol(&mine, g_device_status, sizeof(uint32_t))) != cudaSuccess) return e;
    const uint32_t zero = 0;
    if ((e = cudaMemcpyToSymbol(g_device_status, &zero, sizeof(uint32_t))) != cudaSuccess) return e;
    if ((e = read_device_status_gemm(&gemm)) != cudaSuccess) return e;
    *status = mine | gemm;
    return cudaSuccess;
}

cudaError_t launch_selftest_timeout(unsigned long long limit_ns, cudaStream_t s) {
    selftest_timeout_kernel<<<1, 32, 0, s>>>(limit_ns);
    return cudaGetLastError();
}


cudaError_t launch_gemv_group(const LayoutView* const* Ls, const uint16_t* const* xs, float* const* ys, int count,
                              cudaStream_t s) {
    for (int i = 0; i < count; ++i) {
        const int dep = count == 1 ? DEP_BEFORE : i == 0 ? DEP_GROUP_FIRST : DEP_GROUP_NEXT;
        const cudaError_t e = launch_gemv1<1>(*Ls[i], xs[i], ys[i], s, dep);
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

cudaError_t launch_gemv_swiglu(const LayoutView& L, const uint16_t* x, float* y, uint16_t* h, cudaStream_t s) {
    return launch_gemv1<1, MODE_SWIGLU_EPI>(L, x, y, s, DEP_BEFORE, h);
}

cudaError_t launch_gemv_swiglu_in(const LayoutView& L, const float* gu, float* y, cudaStream_t s) {
    return launch_gemv1<1, MODE_SWIGLU_IN>(L, nullptr, y, s, DEP_BEFORE, nullptr, gu);
}

cudaError_t launch_gemv(const LayoutView& L, const uint16_t* X, float* Y, int B, cudaStream_t s) {
    if (B > 1 && (B > GEMV1_MAX_B || !tables_for_batch(L, B))) return launch_gemm_small(L, X, Y, B, s);
    int b = 0;
    for (; b + 2 <= B; b += 2) {
        const cudaError_t e = launch_gemv1<2>(L, X + (int64_t)b * L.K, Y + (int64_t)b * L.N, s, DEP_BEFORE);
        if (e != cudaSuccess) return e;
    }
    if (B == 1 && L.single_w >= 0) return launch_gemv1<1, MODE_PLAIN, true>(L, X, Y, s, DEP_BEFORE);
    if (b < B) return launch_gemv1<1>(L, X + (int64_t)b * L.K, Y + (int64_t)b * L.N, s, DEP_BEFORE);
    return cudaSuccess;
}

}  // namespace vbq
