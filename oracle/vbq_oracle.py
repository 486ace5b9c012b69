"""CPU oracle for VBQ per-group variable bit-width weights (fp64, numpy).

TEST INFRASTRUCTURE. Only tests/, __graft_entry__.smoke() and bench.py's CPU
baseline leg may import or call this module. The CUDA library never uses it,
and this module imports nothing from the CUDA package.

What it defines (paper: "Variable Bit-width Quantization", arXiv 2607.02893):

* Groups: a weight matrix W (N x K, row-major) is cut into contiguous groups of
  G = 64 weights along K (§3.1); group g of row n covers columns [64g, 64g+64).
  Each group has its own width b in {1, 2, 4, 8} (§3.2, the candidate set) and
  one scale s (§3.1), stored as FP16.
* Quantiser, b >= 2 (§3.1, Eq. 1): s = max|w| / (2^(b-1) - 1) and
  w_hat = s * clip(round(w / s), -(2^(b-1) - 1), 2^(b-1) - 1).
* Quantiser, b = 1 (§3.1): w_hat = sign(w) * mean|w| over the group.
* Packed storage: each group holds 64*b bits (§1, §6: "aligned byte
  boundaries"), i.e. 8*b bytes, plus its scale.
* The inference product (§6): y = W_hat x with the weights never widened in
  memory; here simply the plain dense definition in fp64.
* The training-time soft-quantised forward (§3.2, Alg. 1): per group, the
  convex combination of the four candidate reconstructions under
  pi = softmax((l + e) / tau), the expected width and the hardened width.
* SwiGLU on a gate-up product (the models' MLP, §4; §6 relies on
  silu(0) * u = 0): h = silu(gate) * up with silu(z) = z / (1 + exp(-z)),
  gate and up rows alternating (row 2i gate i, row 2i + 1 up i), fp64.

Readings of points the paper leaves open (each also listed in the design notes):

* Code encoding (never given in the paper): b >= 2 stores the integer
  q in [-(2^(b-1)-1), 2^(b-1)-1] as offset binary u = q + 2^(b-1), so
  L_b(u) = u - 2^(b-1). The code u = 0 (q = -2^(b-1)) is never produced by
  the quantiser but is decoded by the same line. b = 1 stores u = 1 for
  +mean|w| and u = 0 for -mean|w|, so L_1(u) = 2u - 1.
* round() breaks ties to even (round-half-to-even).
* sign(0) = +1 (one bit cannot encode zero).
* The scale is computed in fp64, rounded to FP16 (round to nearest even),
  and the codes are computed with the rounded scale; clip absorbs overshoot.
  Scales above 65504 saturate to 65504. The 1-bit mean sums |w| in fp64 as a
  balanced pairwise tree over neighbouring weights (pairwise_sum), then
  divides by the group size. NaN weights are rejected; +-inf quantise like
  any value above the saturated scale.
* An all-zero group (or one whose scale rounds to 0) gets s = 0 and codes
  u = 2^(b-1) (b >= 2) or u = 1 (b = 1); it dequantises to zeros.
* Activations are BF16; the reference product is exact-input fp64:
  y[b, n] = sum_k f64(w_hat[n, k]) * f64(x[b, k]), with the error-scale term
  A[b, n] = sum_k |w_hat[n, k] * x[b, k]|.
"""

from __future__ import annotations

import numpy as np

GROUP = 64
WIDTHS = (1, 2, 4, 8)
FP16_MAX = 65504.0


# ---------------------------------------------------------------------------
# Level map (§3.1, Eq. 1 and the 1-bit sign rule; encoding as read above)
# ---------------------------------------------------------------------------

def level(b: int, u):
    """Integer level L_b(u) of code u at width b (scalar or integer array)."""
    u = np.asarray(u, dtype=np.int64)
    if b == 1:
        return 2 * u - 1
    if b in (2, 4, 8):
        return u - (1 << (b - 1))
    raise ValueError(f"width {b} not in {WIDTHS}")


def check_inputs(codes: np.ndarray, widths: np.ndarray, scales: np.ndarray) -> None:
    n, k = codes.shape
    if k % GROUP:
        raise ValueError("K must be a multiple of 64")
    if widths.shape != (n, k // GROUP) or scales.shape != (n, k // GROUP):
        raise ValueError("widths/scales must be N x K/64")
    if not np.isin(widths, WIDTHS).all():
        raise ValueError("widths must be in {1,2,4,8}")
    wide = np.repeat(widths.astype(np.int64), GROUP, axis=1)
    if (codes.astype(np.int64) >= (np.int64(1) << wide)).any():
        raise ValueError("code out of range for its group's width")


def dequant(codes: np.ndarray, widths: np.ndarray, scales_fp16: np.ndarray) -> np.ndarray:
    """Dense fp64 W_hat[n, k] = f64(s[n, k // 64]) * L_{b[n, k // 64]}(codes[n, k])."""
    codes = np.asarray(codes, dtype=np.uint8)
    widths = np.asarray(widths, dtype=np.uint8)
    scales = np.asarray(scales_fp16, dtype=np.float16)
    check_inputs(codes, widths, scales)
    n, k = codes.shape
    w = np.empty((n, k), dtype=np.float64)
    for g in range(k // GROUP):
        cols = slice(g * GROUP, (g + 1) * GROUP)
        s = scales[:, g].astype(np.float64)
        lv = np.zeros((n, GROUP), dtype=np.int64)
        for b in WIDTHS:
            rows = widths[:, g] == b
            if rows.any():
                lv[rows] = level(b, codes[rows, cols])
        w[:, cols] = s[:, None] * lv.astype(np.float64)
    return w


def gemv(codes: np.ndarray, widths: np.ndarray, scales_fp16: np.ndarray, x: np.ndarray):
    """y = W_hat x for a batch of activation rows.

    x: (B, K) or (K,) float array holding the (BF16-representable) activations.
    Returns (y, A), both (B, N) fp64, A[b, n] = sum_k |w_hat[n, k] * x[b, k]|.
    """
    w = dequant(codes, widths, scales_fp16)
    x = np.atleast_2d(np.asarray(x, dtype=np.float64))
    if x.shape[1] != w.shape[1]:
        raise ValueError("x has the wrong length")
    y = np.empty((x.shape[0], w.shape[0]), dtype=np.float64)
    a = np.empty_like(y)
    for bi in range(x.shape[0]):
        prod = w * x[bi][None, :]
        y[bi] = prod.sum(axis=1)
        a[bi] = np.abs(prod).sum(axis=1)
    return y, a


def within_bound(y, y_ref, a_ref, rel: float = 2e-3, floor: float = 1e-5) -> np.ndarray:
    """Acceptance test of a computed y: |y - y_ref| <= rel * A + floor, elementwise."""
    return np.abs(np.asarray(y, np.float64) - y_ref) <= rel * a_ref + floor


# ---------------------------------------------------------------------------
# SwiGLU on a gate-up product (§4 models; §6: zero-padded intermediates are
# inert because silu(0) * u = 0)
# ---------------------------------------------------------------------------

SILU_SLOPE_MAX = 1.1        # max |d silu / dz| (about 1.0998, at z near 2.4)


def silu(z):
    """silu(z) = z * sigmoid(z) = z / (1 + exp(-z)), fp64."""
    z = np.asarray(z, dtype=np.float64)
    with np.errstate(over="ignore"):
        return z / (1.0 + np.exp(-z))


def swiglu(y):
    """h = silu(gate) * up for a gate-up product whose rows alternate: row 2i
    is gate i, row 2i + 1 is up i. y: (B, N) with N even -> h: (B, N / 2)."""
    y = np.atleast_2d(np.asarray(y, dtype=np.float64))
    if y.shape[1] % 2:
        raise ValueError("a gate-up product has an even number of rows")
    return silu(y[:, 0::2]) * y[:, 1::2]


def swiglu_error_bound(y_ref, a_ref, rel: float = 2e-3, floor: float = 1e-5) -> np.ndarray:
    """Largest |silu(g') u' - silu(g) u| over gate-up values g', u' that are
    within the product bound of within_bound from the exact g, u: with eg, eu
    those bounds, 1.1 eg (|u| + eu) + |silu(g)| eu (mean value theorem on silu,
    whose slope is at most 1.1 in magnitude). Shape (B, N / 2)."""
    y_ref = np.atleast_2d(y_ref)
    a_ref = np.atleast_2d(a_ref)
    g, u = y_ref[:, 0::2], y_ref[:, 1::2]
    eg, eu = rel * a_ref[:, 0::2] + floor, rel * a_ref[:, 1::2] + floor
    return SILU_SLOPE_MAX * eg * (np.abs(u) + eu) + np.abs(silu(g)) * eu


def swiglu_within_bound(h, y_ref, a_ref, rel: float = 2e-3, floor: float = 1e-5) -> np.ndarray:
    """True where h (rounded to BF16 by the kernel) is within the error that
    follows from a gate-up product within within_bound (swiglu_error_bound),
    plus the BF16 rounding of the result (2^-8 relative, here 2^-7 for the
    fp32 evaluation as well)."""
    h_ref = swiglu(y_ref)
    e = swiglu_error_bound(y_ref, a_ref, rel, floor)
    tol = e * (1.0 + 2.0 ** -7) + 2.0 ** -7 * np.abs(h_ref)
    return np.abs(np.atleast_2d(h) - h_ref) <= tol


# ---------------------------------------------------------------------------
# Quantiser (§3.1, Eq. 1 and the 1-bit absmean rule)
# ---------------------------------------------------------------------------

def _to_fp16_scale(s: float) -> np.float16:
    if s > FP16_MAX:
        return np.float16(FP16_MAX)
    return np.float16(s)


def pairwise_sum(v) -> float:
    """fp64 sum of v as a balanced tree over neighbours: (v0 + v1), (v2 + v3),
    ... then pairs of those, and so on (an odd element is carried up a level).
    The paper fixes the mean of the 1-bit rule, not a summation order; this is
    the order the quantiser uses, written out."""
    level = [float(t) for t in v]
    if not level:
        return 0.0
    while len(level) > 1:
        nxt = [level[i] + level[i + 1] for i in range(0, len(level) - 1, 2)]
        if len(level) % 2:
            nxt.append(level[-1])
        level = nxt
    return level[0]


def quantize_group(w, b: int, fp16_scale: bool = True):
    """Quantise one group of weights at width b.

    Returns (codes uint8[len(w)], scale) where scale is np.float16 if
    fp16_scale else the unrounded fp64 value. NaN weights are rejected.
    """
    w = np.asarray(w, dtype=np.float64)
    if np.isnan(w).any():
        raise ValueError("NaN weight")
    if b == 1:
        s = pairwise_sum(np.abs(w)) / w.size if w.size else 0.0
        s_used = _to_fp16_scale(s) if fp16_scale else s
        codes = (w >= 0).astype(np.uint8)          # sign(0) = +1
        return codes, s_used
    if b not in (2, 4, 8):
        raise ValueError(f"width {b} not in {WIDTHS}")
    qmax = (1 << (b - 1)) - 1
    z = 1 << (b - 1)
    m = float(np.max(np.abs(w))) if w.size else 0.0
    s = m / qmax
    s_used = _to_fp16_scale(s) if fp16_scale else s
    sf = float(s_used)
    if sf == 0.0:
        return np.full(w.shape, z, dtype=np.uint8), s_used
    q = np.clip(np.round(w / sf), -qmax, qmax).astype(np.int64)   # np.round: ties to even
    return (q + z).astype(np.uint8), s_used


def quantize(w: np.ndarray, widths: np.ndarray):
    """Quantise an N x K matrix with per-group widths; returns (codes, scales_fp16)."""
    w = np.asarray(w, dtype=np.float64)
    n, k = w.shape
    widths = np.asarray(widths, dtype=np.uint8)
    if k % GROUP or widths.shape != (n, k // GROUP):
        raise ValueError("bad shapes")
    codes = np.empty((n, k), dtype=np.uint8)
    scales = np.empty((n, k // GROUP), dtype=np.float16)
    for r in range(n):
        for g in range(k // GROUP):
            c, s = quantize_group(w[r, g * GROUP:(g + 1) * GROUP], int(widths[r, g]))
            codes[r, g * GROUP:(g + 1) * GROUP] = c
            scales[r, g] = s
    return codes, scales


# ---------------------------------------------------------------------------
# Training-time soft quantisation (§3.2 differentiable bit selection, Alg. 1)
# ---------------------------------------------------------------------------

CANDIDATES = (1, 2, 4, 8)          # the candidate widths B_k, in the order of the logits


def reconstruct_fp32(w_group, b: int) -> np.ndarray:
    """The reconstruction of one group at width b as a float32 training forward
    computes it (§3.1): b >= 2, s = max|w| / (2^(b-1) - 1) and
    s * clip(round(w / s)) (Eq. 1); b = 1, sign(w) * mean|w| (sign(0) = +1).
    The integer decisions (the codes) are taken in float32, as the framework
    evaluating Eq. 1 on float32 weights takes them: s and w / s are float32
    quotients, rounded half to even. The values are returned in fp64 (s * q is
    exact there; the 1-bit mean is the fp64 pairwise sum / 64). A group whose
    float32 s is 0 reconstructs as 0."""
    w32 = np.asarray(w_group, dtype=np.float32)
    if not np.isfinite(w32).all():
        raise ValueError("non-finite weight")
    if b == 1:
        mean = pairwise_sum(np.abs(w32.astype(np.float64))) / w32.size
        return np.where(w32 >= 0, 1.0, -1.0) * mean
    if b not in (2, 4, 8):
        raise ValueError(f"width {b} not in {WIDTHS}")
    qmax = np.float32((1 << (b - 1)) - 1)
    s = np.float32(np.max(np.abs(w32)) / qmax)
    if s == 0:
        return np.zeros(w32.shape, dtype=np.float64)
    t = (w32 / s).astype(np.float32)
    q = np.clip(np.rint(t), -qmax, qmax)          # np.rint: ties to even
    return q.astype(np.float64) * float(s)


def soft_select(logits, gumbel, tau: float) -> np.ndarray:
    """pi = softmax((l + e) / tau) over the last axis (the 4 candidates), fp64;
    gumbel may be None (no noise)."""
    z = np.asarray(logits, dtype=np.float64)
    if gumbel is not None:
        z = z + np.asarray(gumbel, dtype=np.float64)
    z = z / tau
    z = z - z.max(axis=-1, keepdims=True)
    p = np.exp(z)
    return p / p.sum(axis=-1, keepdims=True)


def soft_quant_forward(w, logits, gumbel, tau: float):
    """The soft-quantised forward of one matrix (§3.2, Alg. 1's weight step):
    per group g, pi_g = softmax((l_g + e_g) / tau), w_soft = sum_k pi_gk *
    w_hat^(B_k) (reconstruct_fp32), the group's expected width sum_k pi_gk B_k
    (whose mean over groups is Alg. 1's b-bar), and the hardened width
    B_argmax_k l_gk (the first maximum on ties; Alg. 1's return).
    w: N x K, logits and gumbel: N x (K/64) x 4 (gumbel may be None).
    Returns (w_soft N x K, exp_bits N x G, hard N x G uint8, pi N x G x 4)."""
    w = np.asarray(w, dtype=np.float32)
    n, k = w.shape
    g = k // GROUP
    logits = np.asarray(logits, dtype=np.float32)
    if k % GROUP or logits.shape != (n, g, 4):
        raise ValueError("bad shapes")
    pi = soft_select(logits, gumbel, tau)
    cand = np.array(CANDIDATES, dtype=np.float64)
    exp_bits = (pi * cand).sum(axis=-1)
    hard = np.array(CANDIDATES, dtype=np.uint8)[np.argmax(logits, axis=-1)]   # argmax: the first maximum
    w_soft = np.empty((n, k), dtype=np.float64)
    for r in range(n):
        for j in range(g):
            wg = w[r, j * GROUP:(j + 1) * GROUP]
            acc = np.zeros(GROUP)
            for kk, b in enumerate(CANDIDATES):
                acc += pi[r, j, kk] * reconstruct_fp32(wg, b)
            w_soft[r, j * GROUP:(j + 1) * GROUP] = acc
    return w_soft, exp_bits, hard, pi


def soft_quant_within_bound(w_soft, exp_bits, w, logits, gumbel, tau: float):
    """Acceptance of a float32 evaluation of soft_quant_forward: per group,
    eps = 2^-20 (1 + max_k |z_k|) with z = (l + e) / tau bounds the relative
    error of each pi_k (z's float32 rounding moves each pi_k by at most
    2 max|dz| relatively, plus exp and the normalisation's roundings, with a
    factor 2 to spare). Then |dw_soft| <= (eps + 2^-20) sum_k pi_k |w_hat_k|
    (each w_hat_k within 2^-21 relatively, the 4-term float32 sum within
    2^-22) and |d exp_bits| <= (eps + 2^-20) sum_k pi_k B_k.
    Returns (ok_w N x K, ok_bits N x G)."""
    w = np.asarray(w, dtype=np.float32)
    n, k = w.shape
    g = k // GROUP
    ref_w, ref_b, _, pi = soft_quant_forward(w, logits, gumbel, tau)
    z = np.asarray(logits, dtype=np.float64)
    if gumbel is not None:
        z = z + np.asarray(gumbel, dtype=np.float64)
    z = z / tau
    eps = 2.0 ** -20 * (1.0 + np.abs(z).max(axis=-1)) + 2.0 ** -20          # N x G
    mag = np.zeros((n, k))
    for r in range(n):
        for j in range(g):
            wg = w[r, j * GROUP:(j + 1) * GROUP]
            for kk, b in enumerate(CANDIDATES):
                mag[r, j * GROUP:(j + 1) * GROUP] += pi[r, j, kk] * np.abs(reconstruct_fp32(wg, b))
    tol_w = np.repeat(eps, GROUP, axis=1) * mag
    ok_w = np.abs(np.asarray(w_soft, dtype=np.float64) - ref_w) <= tol_w
    ok_b = np.abs(np.asarray(exp_bits, dtype=np.float64) - ref_b) <= eps * ref_b
    return ok_w, ok_b


# ---------------------------------------------------------------------------
# Storage accounting (§1, §6: each group packs 64*b bits plus its FP16 scale)
# ---------------------------------------------------------------------------

def payload_bytes(widths: np.ndarray) -> int:
    """Packed code bytes: sum over groups of 64*b/8."""
    return int(np.asarray(widths, dtype=np.int64).sum()) * GROUP // 8


def scale_bytes(widths: np.ndarray) -> int:
    return 2 * int(np.asarray(widths).size)


def pack_lsb(codes: np.ndarray, widths: np.ndarray) -> bytes:
    """Plain reference packing: groups in row-major order, each group's 64 codes
    LSB-first into 8*b bytes. Used to check the storage accounting."""
    out = bytearray()
    n, k = codes.shape
    for r in range(n):
        for g in range(k // GROUP):
            b = int(widths[r, g])
            acc = 0
            for i in range(GROUP):
                acc |= int(codes[r, g * GROUP + i]) << (i * b)
            out += acc.to_bytes(8 * b, "little")
    return bytes(out)


def unpack_lsb(buf: bytes, widths: np.ndarray) -> np.ndarray:
    n, g = widths.shape
    codes = np.empty((n, g * GROUP), dtype=np.uint8)
    pos = 0
    for r in range(n):
        for j in range(g):
            b = int(widths[r, j])
            acc = int.from_bytes(buf[pos:pos + 8 * b], "little")
            pos += 8 * b
            mask = (1 << b) - 1
            for i in range(GROUP):
                codes[r, j * GROUP + i] = (acc >> (i * b)) & mask
    if pos != len(buf):
        raise ValueError("trailing bytes")
    return codes
