"""vbq_quantize (the §3.1 per-group quantiser on the GPU) against the oracle's
quantiser: codes and FP16 scale bits must be identical, for random weights at
every width mix and for groups built to sit on the rounding decisions (exact
ties of Eq. 1's round, their fp32 neighbours, scales that round to zero or
saturate, signed zeros, infinities, fp32 subnormals, and the 1-bit mean whose
FP16 bits depend on the summation order)."""

import numpy as np
import pytest
import torch

import oracle
import paper_2607_02893_gb300 as vbq
import synth
from synth import gen

pytestmark = pytest.mark.gpu

DEV = "cuda"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2607_02893_gb300 import build
    build.build()
    vbq.load()
    torch.cuda.init()


def _gpu_quantize(w: np.ndarray, widths: np.ndarray):
    wd = torch.from_numpy(np.ascontiguousarray(w, dtype=np.float32)).to(DEV)
    bd = torch.from_numpy(np.ascontiguousarray(widths, dtype=np.uint8)).to(DEV)
    codes, scales = vbq.vbq_quantize(wd, bd)
    torch.cuda.synchronize()
    return codes.cpu().numpy(), scales.cpu().numpy().view(np.uint16)


def _assert_same(w: np.ndarray, widths: np.ndarray, rows=None):
    codes, scales = _gpu_quantize(w, widths)
    if rows is None:
        rows = np.arange(w.shape[0])
    rc, rs = oracle.quantize(w[rows].astype(np.float64), widths[rows])
    rs = rs.view(np.uint16)
    bad_s = np.argwhere(scales[rows] != rs)
    assert bad_s.size == 0, f"{len(bad_s)} scales differ, first (row, group) {bad_s[:3].tolist()}: " \
                            f"{[(hex(scales[rows][tuple(i)]), hex(rs[tuple(i)])) for i in bad_s[:3]]}"
    bad_c = np.argwhere(codes[rows] != rc)
    assert bad_c.size == 0, f"{len(bad_c)} codes differ, first (row, col) {bad_c[:3].tolist()}: " \
                            f"{[(int(codes[rows][tuple(i)]), int(rc[tuple(i)])) for i in bad_c[:3]]}"
    return codes, scales


@pytest.mark.parametrize("shape,dist", [
    ((37, 320), synth.DIST_MAIN), ((256, 4096), synth.DIST_MLP0), ((1000, 64), synth.DIST_HEAD),
    ((5, 64 * 37), synth.DIST_ALL1), ((64, 1024), synth.DIST_ALL2), ((64, 1024), synth.DIST_ALL4),
    ((64, 1024), synth.DIST_ALL8), ((1, 64), synth.DIST_MAIN)], ids=lambda v: str(v))
def test_random_weights_bit_exact(shape, dist):
    n, k = shape
    rng = gen.rng_for([90, n, k])
    w = gen.draw_dense_weights(n, k, rng)
    widths = gen.draw_widths(n, k // 64, dist, rng)
    _assert_same(w, widths)


def _tie_group(b: int, s16: np.float16, rng) -> np.ndarray:
    """A group whose FP16 scale is exactly s16 (its largest weight is qmax * s)
    and whose other weights sit on Eq. 1's decisions: exact ties (k + 1/2) s,
    their fp32 neighbours, exact multiples k s, zeros of both signs."""
    qmax = (1 << (b - 1)) - 1
    s = np.float32(s16)
    w = np.zeros(64, np.float32)
    w[0] = np.float32(qmax) * s
    vals = []
    for kk in range(0, qmax):              # (qmax - 1/2) s stays below the maximum qmax s
        t = np.float32((kk + 0.5) * float(s))
        vals += [t, np.nextafter(t, np.float32(np.inf)), np.nextafter(t, np.float32(-np.inf)),
                 np.float32(kk * float(s))]
    vals += [np.float32(0.0), np.float32(-0.0)]
    vals = np.array(vals, np.float32)
    pick = rng.choice(len(vals), size=63, replace=len(vals) < 63)
    w[1:] = vals[pick] * np.where(rng.random(63) < 0.5, -1, 1).astype(np.float32)
    if rng.random() < 0.5:
        w[0] = -w[0]
    return w


@pytest.mark.parametrize("b", [2, 4, 8])
def test_eq1_ties_and_neighbours(b):
    rng = gen.rng_for([91, b])
    scales16 = [np.float16(0.25), np.float16(0.1), np.float16(3.0e-2), np.float16(1.0),
                np.float16(6.0e-8), np.float16(3 * 2.0 ** -24), np.float16(1.5e-5),     # subnormal FP16 scales
                np.float16(1000.0), np.float16(0.0999755859375)]
    groups = [_tie_group(b, s, rng) for s in scales16 for _ in range(6)]
    w = np.stack(groups).reshape(len(groups) // 2, 128)
    widths = np.full((w.shape[0], 2), b, np.uint8)
    _assert_same(w, widths)


def test_scale_extremes_and_special_values():
    rows = []
    z = np.zeros(64, np.float32)
    rows.append(z)                                        # all zero: s = 0
    g = z.copy(); g[5] = 1e-30; rows.append(g)            # scale rounds to 0 in FP16
    g = z.copy(); g[1] = 2.0 ** -25 * 7; rows.append(g)   # scale near the FP16 subnormal threshold
    g = z.copy(); g[0] = 1e30; g[1] = -3e29; g[2] = 5.0; rows.append(g)   # saturated scale
    g = z.copy(); g[3] = np.inf; g[4] = -1.0; rows.append(g)               # +inf
    g = z.copy(); g[3] = -np.inf; g[9] = 2.0; rows.append(g)               # -inf
    g = np.full(64, -0.0, np.float32); rows.append(g)     # negative zeros
    g = np.full(64, 1e-45, np.float32); g[::2] = -1e-45; rows.append(g)   # fp32 subnormals
    g = np.full(64, np.float32(65504.0 * 127)); g[1::2] *= -1; rows.append(g)
    w = np.stack(rows)
    for b in (1, 2, 4, 8):
        widths = np.full((w.shape[0], 1), b, np.uint8)
        _assert_same(w, widths)


def test_one_bit_mean_summation_order():
    w = np.full((2, 64), 2.0 ** -54, np.float32)
    w[0, 0] = 1.0 + 2.0 ** -11                # the order decides: 0x2401 (tree) vs 0x2400 (left to right)
    w[1] = gen.draw_dense_weights(1, 64, gen.rng_for([92]))[0]
    widths = np.ones((2, 1), np.uint8)
    codes, scales = _assert_same(w, widths)
    assert scales[0, 0] == 0x2401


def test_one_bit_spread_around_the_exact_path():
    """1-bit groups whose ulp exponents span 21..26 binades, on both sides of
    the switch between the kernel's exact integer sum and its fp64 tree."""
    rng = gen.rng_for([95])
    rows = []
    for spread in range(21, 27):
        for _ in range(8):
            big = np.float32(rng.uniform(1, 2)) * np.float32(2.0 ** rng.integers(-10, 4))
            g = np.abs(rng.normal(0, 1, 64)).astype(np.float32) * big
            g[rng.integers(64)] = np.float32(float(big) * 2.0 ** -spread * rng.uniform(1, 2))
            g *= np.where(rng.random(64) < 0.5, -1, 1).astype(np.float32)
            rows.append(g)
    w = np.stack(rows)
    _assert_same(w, np.ones((w.shape[0], 1), np.uint8))


def test_errors_leave_outputs_untouched():
    w = torch.zeros((4, 128), dtype=torch.float32, device=DEV)
    widths = torch.full((4, 2), 4, dtype=torch.uint8, device=DEV)
    codes = torch.full((4, 128), 0xAB, dtype=torch.uint8, device=DEV)
    scales = torch.full((4, 2), 0x1234, dtype=torch.int16, device=DEV)
    w[2, 77] = float("nan")
    with pytest.raises(vbq.VbqError) as ei:
        vbq.vbq_quantize(w, widths, codes, scales)
    assert ei.value.name == "VBQ_ERR_ARG"
    w[2, 77] = 0.0
    widths[3, 1] = 3
    with pytest.raises(vbq.VbqError) as ei:
        vbq.vbq_quantize(w, widths, codes, scales)
    assert ei.value.name == "VBQ_ERR_WIDTH"
    torch.cuda.synchronize()
    assert bool((codes == 0xAB).all()) and bool((scales == 0x1234).all())


def test_quantize_pack_dequant_gemv_roundtrip():
    n, k = 300, 2048
    rng = gen.rng_for([93])
    w = gen.draw_dense_weights(n, k, rng)
    widths = gen.draw_widths(n, k // 64, synth.DIST_MAIN, rng)
    wd = torch.from_numpy(w).to(DEV)
    bd = torch.from_numpy(widths).to(DEV)
    codes, scales = vbq.vbq_quantize(wd, bd)
    lay = vbq.vbq_pack(codes, bd, scales)
    c2 = torch.empty_like(codes)
    s2 = torch.empty_like(scales)
    vbq.vbq_dequant(lay, codes_out=c2, scales_out=s2)
    torch.cuda.synchronize()
    assert torch.equal(c2, codes) and torch.equal(s2, scales)
    x_bits = gen.draw_x_bf16(1, k, rng)
    x = torch.from_numpy(x_bits.view(np.int16)).to(DEV)
    y = torch.empty(n, dtype=torch.float32, device=DEV)
    vbq.vbq_gemv(lay, x, y)
    torch.cuda.synchronize()
    rc, rs = oracle.quantize(w.astype(np.float64), widths)
    y_ref, a_ref = oracle.gemv(rc, widths, rs, gen.bf16_bits_to_f32(x_bits).astype(np.float64))
    assert oracle.within_bound(y.cpu().numpy()[None, :], y_ref, a_ref).all()


def test_full_size_sampled_rows():
    """The 14336 x 4096 MLP shape of the 9B stack at full size; 48 sampled rows
    against the oracle, and the whole result packs (every code in range)."""
    n, k = 14336, 4096
    rng = gen.rng_for([94])
    w = gen.draw_dense_weights(n, k, rng)
    widths = gen.draw_widths(n, k // 64, synth.DIST_MAIN, rng)
    rows = np.sort(rng.choice(n, size=48, replace=False))
    rows[-1] = n - 1
    codes, scales = _assert_same(w, widths, rows=rows)
    lay = vbq.vbq_pack(torch.from_numpy(codes).to(DEV), torch.from_numpy(widths).to(DEV),
                       torch.from_numpy(scales.view(np.int16)).to(DEV))
    assert vbq.vbq_layout_shape(lay) == (n, k)
