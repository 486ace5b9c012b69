"""Checks that pin the CPU oracle to the paper and to plain mathematics.

Each pin takes the oracle module as an argument so that the same checks can
be run against deliberately broken copies of it (see test_oracle.py): every
plausible mistake must trip at least one pin.
"""

from __future__ import annotations

import os
from fractions import Fraction

import numpy as np

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


class PinFailed(AssertionError):
    pass


def _check(cond, msg):
    if not cond:
        raise PinFailed(msg)


def load_eq1_examples():
    rows = []
    with open(os.path.join(GOLDEN, "eq1_examples.txt")) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            name, b, pairs, sbits, codes, zcode = [p.strip() for p in line.split("|")]
            idx, vals = [], []
            for tok in pairs.split():
                i, v = tok.split(":")
                idx.append(int(i))
                vals.append(float(v))
            rows.append(dict(name=name, b=int(b), idx=idx, vals=vals,
                             sbits=int(sbits, 16),
                             codes=[int(c) for c in codes.split()], zcode=int(zcode)))
    return rows


def pin_eq1_golden(O):
    """Hand-worked Eq. 1 / 1-bit examples: scale bits and codes."""
    for ex in load_eq1_examples():
        w = np.zeros(64)
        w[ex["idx"]] = ex["vals"]
        codes, s = O.quantize_group(w, ex["b"])
        _check(int(np.float16(s).view(np.uint16)) == ex["sbits"],
               f"{ex['name']}: scale bits {int(np.float16(s).view(np.uint16)):04x} != {ex['sbits']:04x}")
        exp = np.full(64, ex["zcode"], dtype=np.int64)
        exp[ex["idx"]] = ex["codes"]
        _check(np.array_equal(codes.astype(np.int64), exp), f"{ex['name']}: codes {codes} != {exp}")


def pin_level_grid(O):
    """Eq. 1's reconstruction grid: integer, uniform step 1, symmetric, zero at the
    midpoint code; the quantiser's codes 1 .. 2^b-1 span -qmax .. qmax. 1 bit: +-1."""
    for b in (2, 4, 8):
        qmax = (1 << (b - 1)) - 1
        z = 1 << (b - 1)
        lv = [int(O.level(b, u)) for u in range(1 << b)]
        _check(lv[z] == 0, f"b={b}: midpoint code is not the zero level")
        _check(all(lv[u + 1] - lv[u] == 1 for u in range(len(lv) - 1)), f"b={b}: grid step")
        _check(lv[1] == -qmax and lv[(1 << b) - 1] == qmax, f"b={b}: emitted range")
        _check(all(lv[z + k] == -lv[z - k] for k in range(1, qmax + 1)), f"b={b}: symmetry")
    _check(int(O.level(1, 1)) == 1 and int(O.level(1, 0)) == -1, "1-bit polarity")


def pin_grid_roundtrip(O, seed=1):
    """Weights already on an Eq. 1 grid (power-of-two scale, a group containing
    +-qmax) are reproduced exactly by quantise -> dequantise; a constant-magnitude
    group at 1 bit too."""
    rng = np.random.default_rng(seed)
    for b in (1, 2, 4, 8):
        n, k = 3, 128
        widths = np.full((n, k // 64), b, dtype=np.uint8)
        if b == 1:
            mag = 2.0 ** rng.integers(-8, 2, size=(n, k // 64))
            sign = np.where(rng.random((n, k)) < 0.5, -1.0, 1.0)
            w = sign * np.repeat(mag, 64, axis=1)
        else:
            qmax = (1 << (b - 1)) - 1
            q = rng.integers(-qmax, qmax + 1, size=(n, k))
            q[:, ::64] = qmax                          # each group contains +qmax
            s = 2.0 ** rng.integers(-10, 0, size=(n, k // 64))
            w = np.repeat(s, 64, axis=1) * q
        codes, scales = O.quantize(w, widths)
        _check(np.array_equal(O.dequant(codes, widths, scales), w), f"b={b}: grid roundtrip")


def pin_quantizer_invariants(O, seed=2):
    rng = np.random.default_rng(seed)
    for b in (2, 4, 8):
        qmax = (1 << (b - 1)) - 1
        for _ in range(20):
            w = rng.normal(0, rng.uniform(0.01, 3.0), size=64)
            codes, s = O.quantize_group(w, b)
            q = codes.astype(np.int64) - (1 << (b - 1))
            _check(np.all(np.abs(q) <= qmax), f"b={b}: |q| > qmax")
            sf = float(s)
            err = np.abs(w - sf * q)
            _check(np.all(err <= sf / 2 * (1 + 1e-9) + 1e-12), f"b={b}: error above s/2")
            imax = int(np.argmax(np.abs(w)))
            _check(abs(int(q[imax])) == qmax, f"b={b}: max-magnitude weight not at +-qmax")
            # idempotence: quantising the reconstruction gives the same codes and scale
            wh = sf * q
            c2, s2 = O.quantize_group(wh, b)
            _check(np.array_equal(c2, codes) and float(s2) == sf, f"b={b}: not idempotent")
    for _ in range(10):
        w = rng.normal(0, 1, size=64)
        codes, s = O.quantize_group(w, 1)
        _check(np.array_equal(codes, (w >= 0).astype(np.uint8)), "1-bit codes != sign")
        _check(float(s) == float(np.float16(np.mean(np.abs(w)))), "1-bit scale != mean|w|")


def pin_one_bit_mean_order(O):
    """The 1-bit scale is FP16(mean |w|) (§3.1) with the mean summed as a
    balanced fp64 tree. Hand-derived case where the order decides the FP16 bits:
    w0 = 1 + 2^-11 (the FP16 midpoint between 1 and 1 + 2^-10, times 64 later)
    and 63 weights of 2^-54. Exactly, sum = 1 + 2^-11 + 63 * 2^-54, above the
    midpoint, so FP16(sum / 64) = 2^-6 (1 + 2^-10) = 0x2401. The tree loses
    the first 2^-54 (w0 + w1 rounds to w0), and (w0 + w1) + (w2 + w3) is a tie
    that rounds to even (w0); then it adds 2^-52, 2^-51, 2^-50 and 2^-49
    exactly: 1 + 2^-11 + 15 * 2^-52, still above the midpoint: 0x2401. A
    left-to-right sum loses every 2^-54 (each is below half an ulp of 1),
    lands on the midpoint and rounds to even: 0x2400."""
    w = np.full(64, 2.0 ** -54)
    w[0] = 1.0 + 2.0 ** -11
    codes, s = O.quantize_group(w, 1)
    _check(int(np.float16(s).view(np.uint16)) == 0x2401, f"1-bit mean order: scale {np.float16(s)}")
    _check(np.array_equal(codes, np.ones(64, np.uint8)), "1-bit mean order: codes")
    _check(O.pairwise_sum([1.0, 2.0, 3.0]) == 6.0 and O.pairwise_sum([]) == 0.0, "pairwise_sum edge cases")


def pin_group_size_one(O, seed=3):
    """§3.1: with one weight per group every width reconstructs w exactly
    (unrounded scale)."""
    rng = np.random.default_rng(seed)
    for w0 in rng.normal(0, 1, size=50):
        for b in (1, 2, 4, 8):
            codes, s = O.quantize_group(np.array([w0]), b, fp16_scale=False)
            wh = s * int(O.level(b, int(codes[0])))
            _check(abs(wh - w0) <= 4e-16 * abs(w0), f"b={b}: G=1 not exact ({wh} vs {w0})")


def pin_integer_gemv(O, seed=4):
    """All-8-bit, unit scales, small integer x: y is an exact integer product,
    checked against an int64 matmul; and with power-of-two scales and mixed
    widths against exact rational arithmetic on a tiny case."""
    rng = np.random.default_rng(seed)
    n, k = 37, 256
    codes = rng.integers(0, 256, size=(n, k)).astype(np.uint8)
    widths = np.full((n, k // 64), 8, dtype=np.uint8)
    scales = np.ones((n, k // 64), dtype=np.float16)
    x = rng.integers(-8, 9, size=(2, k))
    y, a = O.gemv(codes, widths, scales, x.astype(np.float64))
    exp = (codes.astype(np.int64) - 128) @ x.T.astype(np.int64)
    _check(np.array_equal(y, exp.T.astype(np.float64)), "integer all-8-bit GEMV")
    _check(np.array_equal(a, (np.abs(codes.astype(np.int64) - 128) @ np.abs(x.T)).T.astype(np.float64)),
           "integer all-8-bit bound term")


def pin_exact_rational(O, seed=5):
    """Tiny mixed-width case: the fp64 product equals the exact rational sum of
    the dequantised weights times x to within fp64 rounding."""
    rng = np.random.default_rng(seed)
    n, k = 5, 192
    widths = rng.choice(np.array([1, 2, 4, 8], np.uint8), size=(n, k // 64))
    codes = (rng.integers(0, 256, size=(n, k)) & ((1 << np.repeat(widths, 64, axis=1).astype(np.int64)) - 1)).astype(np.uint8)
    scales = (np.abs(rng.normal(0, 0.02, size=(n, k // 64))) + 1e-4).astype(np.float16)
    x = rng.normal(0, 1, size=k).astype(np.float32)
    w = O.dequant(codes, widths, scales)
    y, _ = O.gemv(codes, widths, scales, x)
    for r in range(n):
        exact = sum((Fraction(float(w[r, j])) * Fraction(float(x[j])) for j in range(k)), Fraction(0))
        mag = sum(abs(Fraction(float(w[r, j])) * Fraction(float(x[j]))) for j in range(k))
        _check(abs(Fraction(float(y[0, r])) - exact) <= mag * Fraction(1, 2 ** 45), f"row {r}: fp64 sum")
    # one-hot activations pick out single dequantised weights: checks group indexing
    for j in (0, 63, 64, 130, 191):
        e = np.zeros(k)
        e[j] = 1.0
        yj, _ = O.gemv(codes, widths, scales, e)
        g = j // 64
        for r in range(n):
            b = int(widths[r, g])
            expect = float(scales[r, g]) * int(O.level(b, int(codes[r, j])))
            _check(yj[0, r] == expect, f"one-hot column {j} row {r}")


def pin_enumerated_codes(O):
    """Brute force over every code at every position of one group: with a one-hot
    x the product returns s * level, and for each width the 2^b results form the
    uniform grid s * (-2^(b-1) .. 2^(b-1)-1) (b >= 2) or {-s, +s} (b = 1)."""
    s = np.float16(0.375)
    for b in (1, 2, 4, 8):
        ncode = 1 << b
        z = (1 << (b - 1)) if b > 1 else 1
        n = ncode * 64
        codes = np.full((n, 64), z, dtype=np.uint8)
        for pos in range(64):
            for u in range(ncode):
                codes[pos * ncode + u, pos] = u
        widths = np.full((n, 1), b, dtype=np.uint8)
        scales = np.full((n, 1), s, dtype=np.float16)
        for pos in (0, 1, 31, 63):
            e = np.zeros(64)
            e[pos] = 1.0
            y, _ = O.gemv(codes, widths, scales, e)
            got = y[0, pos * ncode:(pos + 1) * ncode]
            if b == 1:
                _check(list(got) == [-0.375, 0.375], f"b=1 pos {pos}: {got}")
            else:
                expect = [0.375 * (u - (1 << (b - 1))) for u in range(ncode)]
                _check(list(got) == expect, f"b={b} pos {pos}")


def pin_swiglu(O):
    """SwiGLU (§4 models; §6 silu(0) * u = 0) by closed forms and identities:
    silu(0) = 0, silu(1) = e / (1 + e), silu(z) - silu(-z) = z (the sigmoid's
    symmetry), silu(z) -> z for large z and -> 0 for very negative z; the
    pairing puts gate on even rows and up on odd rows; the slope bound the
    tolerance uses holds on a dense grid."""
    import math
    _check(float(O.silu(0.0)) == 0.0, "silu(0)")
    _check(abs(float(O.silu(1.0)) - math.e / (1.0 + math.e)) <= 1e-16, "silu(1)")
    z = np.linspace(-30, 30, 6001)
    _check(np.allclose(O.silu(z) - O.silu(-z), z, rtol=0, atol=1e-13), "silu odd part")
    _check(float(O.silu(60.0)) == 60.0 and abs(float(O.silu(-60.0))) < 1e-20, "silu tails")
    _check(np.isfinite(O.silu(np.array([-1000.0, 1000.0]))).all(), "silu overflow")
    h = O.swiglu(np.array([[2.0, 3.0, -1.0, 5.0, 0.0, 7.0]]))
    exp = [2.0 / (1.0 + math.exp(-2.0)) * 3.0, -1.0 / (1.0 + math.exp(1.0)) * 5.0, 0.0]
    _check(np.allclose(h[0], exp, rtol=1e-15, atol=0), f"swiglu pairing {h}")
    d = np.diff(O.silu(np.linspace(-20, 20, 400001))) / 1e-4
    _check(np.abs(d).max() <= O.SILU_SLOPE_MAX and np.abs(d).max() > 1.09, "silu slope bound")
    y = np.array([[1.5, -2.0, 0.25, 4.0]])
    a = np.abs(y) + 1.0
    _check(O.swiglu_within_bound(O.swiglu(y), y, a).all(), "bound admits the exact value")
    _check(not O.swiglu_within_bound(O.swiglu(y) + 0.1, y, a).any(), "bound rejects a gross error")


def pin_payload_accounting(O, seed=6):
    rng = np.random.default_rng(seed)
    n, k = 7, 320
    widths = rng.choice(np.array([1, 2, 4, 8], np.uint8), size=(n, k // 64))
    codes = (rng.integers(0, 256, size=(n, k)) & ((1 << np.repeat(widths, 64, axis=1).astype(np.int64)) - 1)).astype(np.uint8)
    buf = O.pack_lsb(codes, widths)
    _check(len(buf) == sum(64 * int(b) // 8 for b in widths.ravel()), "packed length")
    _check(O.payload_bytes(widths) == len(buf), "payload_bytes")
    _check(O.scale_bytes(widths) == 2 * n * (k // 64), "scale bytes")
    _check(np.array_equal(O.unpack_lsb(buf, widths), codes), "pack/unpack roundtrip")


def pin_soft_quant(O):
    """The training-time soft forward (§3.2, Alg. 1) by closed forms and by the
    export quantiser: equal logits give pi = 1/4 and an expected width of
    (1 + 2 + 4 + 8) / 4 = 3.75; a dominant logit selects that candidate's
    reconstruction, which is the weight itself for a group on its grid with a
    power-of-two scale; e is added to l and tau divides both; the hardened
    width is the first maximum's candidate; and the float32 reconstructions
    agree with the (separately pinned) fp64 quantiser wherever no quotient
    lies near a rounding tie."""
    B = (1, 2, 4, 8)
    _check(tuple(O.CANDIDATES) == B, f"candidates {O.CANDIDATES}")
    rng = np.random.default_rng(31)
    # equal logits: uniform selection
    w = rng.normal(0, 0.02, (3, 128)).astype(np.float32)
    lg = np.full((3, 2, 4), 0.7, np.float32)
    ws, eb, hard, pi = O.soft_quant_forward(w, lg, None, 0.9)
    _check(np.allclose(pi, 0.25, rtol=0, atol=1e-15), "equal logits -> pi = 1/4")
    _check(np.allclose(eb, 3.75, rtol=0, atol=1e-14), f"expected width {eb}")
    for r in range(3):
        for j in range(2):
            wg = w[r, 64 * j:64 * j + 64]
            mean = sum(O.reconstruct_fp32(wg, b) for b in B) / 4.0
            _check(np.allclose(ws[r, 64 * j:64 * j + 64], mean, rtol=1e-13, atol=0), "uniform mixture")
    # a dominant logit selects its candidate; on-grid groups reconstruct exactly
    for kk, b in enumerate(B[1:], start=1):
        qmax = (1 << (b - 1)) - 1
        q = rng.integers(-qmax, qmax + 1, size=64)
        q[5], q[40] = qmax, -qmax
        wg = (q * 2.0 ** -9).astype(np.float32)[None, :]
        lg1 = np.zeros((1, 1, 4), np.float32)
        lg1[0, 0, kk] = 60.0
        ws1, eb1, hard1, _ = O.soft_quant_forward(wg, lg1, None, 1.0)
        _check(np.allclose(ws1[0], wg[0].astype(np.float64), rtol=1e-20, atol=1e-24),
               f"dominant {b}-bit logit on its grid")
        _check(abs(eb1[0, 0] - b) < 1e-20 * 8 + 1e-22, f"dominant {b}-bit expected width {eb1}")
        _check(int(hard1[0, 0]) == b, f"hardened {hard1}")
    # exact ties of the float32 quotient round half to even: at 4 bits with
    # max|w| = 7 * 2^-6 the scale is 2^-6, and w = (k + 1/2) 2^-6 lands on k + 1/2
    halves = [0.5, 1.5, 2.5, 3.5, 4.5, 5.5, 6.5, -0.5, -1.5, -2.5, -6.5]
    want_q = [0, 2, 2, 4, 4, 6, 6, 0, -2, -2, -6]          # by hand: the even neighbour
    wt = np.zeros(64, np.float32)
    wt[:len(halves)] = np.array(halves) * 2.0 ** -6
    wt[63] = 7 * 2.0 ** -6
    rt = O.reconstruct_fp32(wt, 4)
    _check(np.array_equal(rt[:len(halves)], np.array(want_q, dtype=np.float64) * 2.0 ** -6),
           f"ties to even: {rt[:len(halves)] / 2.0 ** -6}")
    # 1 bit: a constant-magnitude group reconstructs exactly, sign(0) = +1
    wc = np.where(rng.random(64) < 0.5, -0.03, 0.03).astype(np.float32)
    wc[7] = 0.0
    r1 = O.reconstruct_fp32(wc, 1)
    m = float(np.abs(wc.astype(np.float64)).sum()) / 64
    _check(r1[7] == m and np.allclose(np.abs(r1), m, rtol=0, atol=0), "1-bit sign * mean")
    _check(np.array_equal(np.sign(r1[wc != 0]), np.sign(wc[wc != 0])), "1-bit signs")
    # noise is added to the logits, tau divides both, and a shift cancels
    l2 = rng.normal(0, 2, (2, 3, 4)).astype(np.float32)
    e2 = rng.gumbel(size=(2, 3, 4)).astype(np.float32)
    p_a = O.soft_select(l2, e2, 0.5)
    p_b = O.soft_select(l2.astype(np.float64) + e2, None, 0.5)
    p_c = O.soft_select((l2.astype(np.float64) + e2) / 0.5 + 3.0, None, 1.0)
    _check(np.allclose(p_a, p_b, rtol=1e-14, atol=0) and np.allclose(p_a, p_c, rtol=1e-12, atol=0),
           "softmax of (l + e) / tau")
    _check(np.allclose(p_a.sum(-1), 1.0, atol=1e-15), "pi sums to 1")
    z = (l2.astype(np.float64) + e2) / 0.5
    ratio = p_a[..., 3] / p_a[..., 0]
    _check(np.allclose(ratio, np.exp(z[..., 3] - z[..., 0]), rtol=1e-12), "pi ratio = exp(z3 - z0)")
    # hardened widths: the first maximum
    lh = np.array([[[1, 3, 3, 0], [5, 5, 5, 5], [0, 0, 0, 1], [-1, -2, -3, -0.5]]], np.float32)
    _, _, hh, _ = O.soft_quant_forward(np.zeros((1, 256), np.float32), lh, None, 1.0)
    _check(hh[0].tolist() == [2, 1, 8, 8], f"hardened widths {hh}")
    # float32 reconstructions against the fp64 export quantiser (unrounded scale)
    agree = 0
    for _ in range(200):
        wg = (rng.normal(0, 0.02, 64) * np.exp(rng.normal(0, 1))).astype(np.float32)
        for b in (2, 4, 8):
            qmax = (1 << (b - 1)) - 1
            s64 = float(np.max(np.abs(wg.astype(np.float64)))) / qmax
            frac = np.abs(wg.astype(np.float64) / s64)
            if np.min(np.abs(frac - np.floor(frac) - 0.5)) < 1e-5:
                continue                    # a quotient near a tie: the precisions may differ
            codes, _ = O.quantize_group(wg.astype(np.float64), b, fp16_scale=False)
            q_ref = codes.astype(np.int64) - (1 << (b - 1))
            rec = O.reconstruct_fp32(wg, b)
            s32 = float(np.float32(np.max(np.abs(wg)) / np.float32(qmax)))
            _check(np.array_equal(np.rint(rec / s32).astype(np.int64), q_ref), f"{b}-bit codes vs the quantiser")
            agree += 1
    _check(agree > 400, f"only {agree} comparisons")


def pin_soft_bound(O):
    """The acceptance bound of a float32 soft forward (soft_quant_within_bound,
    §3.2 / Alg. 1's weight step) against values derived by hand.

    Hand-worked group: all 64 weights equal c = 2^-4, equal logits, no noise,
    tau = 1. Then z = (l + e) / tau = 0, so pi_k = 1/4 exactly and the bound's
    eps = 2^-20 (1 + max|z|) + 2^-20 = 2^-19. Every reconstruction is c up to
    float32 rounding of its scale (1 bit: mean|w| = c; 2 bits: s = c / 1, q = 1;
    4 and 8 bits: q = 7 and 127 against s = c / 7, c / 127), so
    sum_k pi_k |w_hat_k| = c within 2^-22 relatively and the expected width is
    (1 + 2 + 4 + 8) / 4 = 3.75. A weight error of eps c / 2 is inside the bound
    and one of 4 eps c outside it; the same for the expected width with 3.75
    in place of c. The forward's own output is admitted, and a weight moved by
    a quarter of its 4-bit step under a dominant 4-bit logit is rejected."""
    c = 2.0 ** -4
    w = np.full((1, 64), c, np.float32)
    lg = np.zeros((1, 1, 4), np.float32)
    eps = 2.0 ** -19                                    # by hand, from z = 0
    ws, eb, _, pi = O.soft_quant_forward(w, lg, None, 1.0)
    _check(np.array_equal(pi[0, 0], np.full(4, 0.25)), f"pi {pi[0, 0]}")
    _check(abs(eb[0, 0] - 3.75) < 1e-15, f"expected width {eb[0, 0]}")
    _check(np.allclose(ws, c, rtol=2.0 ** -22, atol=0), "reconstructions all c")
    ok_w, ok_b = O.soft_quant_within_bound(ws, eb, w, lg, None, 1.0)
    _check(ok_w.all() and ok_b.all(), "bound admits the forward's own output")
    for j in (0, 17, 63):
        for sgn in (1.0, -1.0):
            near = ws.copy()
            near[0, j] += sgn * 0.5 * eps * c
            far = ws.copy()
            far[0, j] += sgn * 4.0 * eps * c
            okn, _ = O.soft_quant_within_bound(near, eb, w, lg, None, 1.0)
            okf, _ = O.soft_quant_within_bound(far, eb, w, lg, None, 1.0)
            _check(okn.all(), f"eps c / 2 at weight {j} admitted")
            _check(not okf[0, j] and okf.sum() == 63, f"4 eps c at weight {j} rejected, the rest admitted")
    _, okb = O.soft_quant_within_bound(ws, eb + 0.5 * eps * 3.75, w, lg, None, 1.0)
    _check(okb.all(), "expected width off by eps 3.75 / 2 admitted")
    _, okb = O.soft_quant_within_bound(ws, eb - 4.0 * eps * 3.75, w, lg, None, 1.0)
    _check(not okb.any(), "expected width off by 4 eps 3.75 rejected")
    # a quarter step: dominant 4-bit logit, random group; the 4-bit step is s =
    # max|w| / 7 and pi_4 is 1 to within e^-40
    rng = np.random.default_rng(37)
    wr = rng.normal(0, 0.02, (1, 128)).astype(np.float32)
    lr = np.zeros((1, 2, 4), np.float32)
    lr[0, :, 2] = 40.0
    ws2, eb2, _, _ = O.soft_quant_forward(wr, lr, None, 1.0)
    ok_w, ok_b = O.soft_quant_within_bound(ws2, eb2, wr, lr, None, 1.0)
    _check(ok_w.all() and ok_b.all(), "bound admits the forward's own output (dominant 4 bits)")
    s4 = float(np.max(np.abs(wr[0, 64:]))) / 7.0
    moved = ws2.copy()
    moved[0, 64 + 9] += 0.25 * s4
    okm, _ = O.soft_quant_within_bound(moved, eb2, wr, lr, None, 1.0)
    _check(not okm[0, 64 + 9] and okm.sum() == 127, "a quarter 4-bit step rejected")
    # the noise enters z: e = 1000 on the 4-bit candidate and l = 0 give z =
    # (0, 0, 1000, 0), pi = (0, 0, 1, 0) and eps = 2^-20 (1 + 1000) + 2^-20 =
    # 1002 2^-20 (by hand); an error of eps |w_hat_4| / 2 is admitted
    ge = np.zeros((1, 2, 4), np.float32)
    ge[0, :, 2] = 1000.0
    ws3, eb3, _, _ = O.soft_quant_forward(wr, np.zeros((1, 2, 4), np.float32), ge, 1.0)
    rec4 = O.reconstruct_fp32(wr[0, :64], 4)
    j = int(np.argmax(np.abs(rec4)))
    half = ws3.copy()
    half[0, j] += 0.5 * 1002 * 2.0 ** -20 * abs(rec4[j])
    okh, _ = O.soft_quant_within_bound(half, eb3, wr, np.zeros((1, 2, 4), np.float32), ge, 1.0)
    _check(okh.all(), "eps from z with the noise: eps |w_hat| / 2 admitted")
    over = ws3.copy()
    over[0, j] += 4.0 * 1002 * 2.0 ** -20 * abs(rec4[j])
    oko, _ = O.soft_quant_within_bound(over, eb3, wr, np.zeros((1, 2, 4), np.float32), ge, 1.0)
    _check(not oko[0, j], "eps from z with the noise: 4 eps |w_hat| rejected")


ALL_PINS = [pin_eq1_golden, pin_level_grid, pin_grid_roundtrip, pin_quantizer_invariants,
            pin_one_bit_mean_order, pin_group_size_one, pin_integer_gemv, pin_exact_rational, pin_enumerated_codes,
            pin_swiglu, pin_soft_quant, pin_soft_bound, pin_payload_accounting]
