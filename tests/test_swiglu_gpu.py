"""Parity of the fused gate-up product with its SwiGLU epilogue
(vbq_gemv_swiglu, through the C ABI) with the CPU oracle.

The gate-up matrix's rows alternate (row 2i gate i, row 2i + 1 up i). Every
output y must satisfy the product bound of vbq_gemv, and every h_i =
silu(y_2i) * y_2i+1 (BF16) the bound oracle.swiglu_within_bound derives from
it. Shapes cover one slab per row (the epilogue in the copier's flush) and
several slabs (the epilogue by the block that adds a row block's last slab),
ragged last row blocks, repeated calls on one layout, the zero-padded
features the paper relies on (silu(0) * u = 0), and the full-size gate-up
matrices of the three stacks in a captured graph, as bench.py runs them."""

import numpy as np
import pytest
import torch

import oracle
import paper_2607_02893_gb300 as vbq
import synth
from synth import gen
from vbq_cases import Matrix, bits_to_i16, scales_to_i16

pytestmark = pytest.mark.gpu

DEV = "cuda"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2607_02893_gb300 import build
    build.build()
    vbq.load()
    torch.cuda.init()


def _run(layout, x_bits, n, stream=None):
    x = bits_to_i16(x_bits).to(DEV)
    y = torch.full((n,), float("nan"), dtype=torch.float32, device=DEV)
    h = torch.full((n // 2,), -1, dtype=torch.int16, device=DEV)       # 0xFFFF: a NaN pattern
    vbq.vbq_gemv_swiglu(layout, x, y, h, stream=stream)
    torch.cuda.synchronize()
    return y.cpu().numpy(), h.cpu().numpy().view(np.uint16)


def _check(y, h_bits, codes, widths, scales, x):
    y_ref, a_ref = oracle.gemv(codes, widths, scales, x[None, :])
    ok_y = oracle.within_bound(y[None, :], y_ref, a_ref)
    h = gen.bf16_bits_to_f32(h_bits)[None, :]
    ok_h = oracle.swiglu_within_bound(h, y_ref, a_ref)
    if not (ok_y.all() and ok_h.all()):
        bad = np.argwhere(~ok_h[0])[:5].ravel()
        h_ref = oracle.swiglu(y_ref)[0]
        raise AssertionError(f"{int((~ok_y).sum())} y and {int((~ok_h).sum())} h outside the bound; "
                             f"first h: {[(int(i), float(h[0, i]), float(h_ref[i])) for i in bad]}")


# (rows, K): one slab per row for (20000, 1024) and (9728, 768) (16 or 12
# group columns, enough row blocks for the SMs); several slabs otherwise;
# 600 and 1000 rows end in a ragged row block; (2, 64) is a single feature.
SHAPES = [(2, 64), (256, 768), (600, 2048), (1000, 64 * 37), (4096, 768), (20000, 1024), (9728, 768)]


@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: f"{s[0]}x{s[1]}")
@pytest.mark.parametrize("dist", ["main", "mlp0"])
def test_swiglu_parity(shape, dist):
    n, k = shape
    d = {"main": synth.DIST_MAIN, "mlp0": synth.DIST_MLP0}[dist]
    m = Matrix(n, k, dist=d, seed_path=(90, n, k))
    layout = vbq.vbq_pack(*m.device_args(DEV))
    y, h = _run(layout, m.x_bits[0], n)
    _check(y, h, m.codes.numpy(), m.widths, m.scales, m.x()[0])


def test_swiglu_repeated_and_mixed_calls():
    # the slab counts are reset by every call; plain products on the same
    # layout leave them alone
    m = Matrix(1000, 2048, seed_path=(90, 1, 0), batch=3)
    layout = vbq.vbq_pack(*m.device_args(DEV))
    codes = m.codes.numpy()
    for b in (0, 1, 1, 2):
        y, h = _run(layout, m.x_bits[b], m.n)
        _check(y, h, codes, m.widths, m.scales, m.x()[b])
        yp = torch.empty(m.n, dtype=torch.float32, device=DEV)
        vbq.vbq_gemv(layout, bits_to_i16(m.x_bits[b]).to(DEV), yp)
        torch.cuda.synchronize()
        y_ref, a_ref = oracle.gemv(codes, m.widths, m.scales, m.x()[b][None, :])
        assert oracle.within_bound(yp.cpu().numpy()[None, :], y_ref, a_ref).all()


@pytest.mark.parametrize("k", [768, 4096])
def test_zero_padded_features_are_inert(k):
    # features whose gate and up rows hold only zero-level codes (a padded
    # channel, §6): g = 0 exactly, so h = silu(0) * u = 0 exactly, and the other
    # features are unaffected
    n = 1024
    m = Matrix(n, k, dist=(0.0, 0.3, 0.4, 0.3), seed_path=(90, 2, k))
    codes = m.codes.numpy().copy()
    pad = np.arange(n // 2) % 3 == 0
    pad_rows = np.flatnonzero(np.repeat(pad, 2))
    zl = (1 << (m.widths.astype(np.int64) - 1)).astype(np.uint8)          # the zero level per group
    codes[pad_rows] = np.repeat(zl[pad_rows], 64, axis=1)
    layout = vbq.vbq_pack(torch.from_numpy(codes).to(DEV), torch.from_numpy(m.widths).to(DEV),
                          scales_to_i16(m.scales).to(DEV))
    y, h = _run(layout, m.x_bits[0], n)
    assert np.all(y[pad_rows] == 0.0)
    assert np.all((h[pad] & 0x7FFF) == 0)                                  # +0 or -0
    _check(y, h, codes, m.widths, m.scales, m.x()[0])


def test_swiglu_rejects_bad_arguments():
    m = Matrix(257, 128, seed_path=(90, 3, 0))
    odd = vbq.vbq_pack(*m.device_args(DEV))
    x = bits_to_i16(m.x_bits[0]).to(DEV)
    y = torch.empty(258, dtype=torch.float32, device=DEV)
    h = torch.empty(136, dtype=torch.int16, device=DEV)
    with pytest.raises(vbq.VbqError) as e:
        vbq.vbq_gemv_swiglu(odd, x, y, h)
    assert e.value.name == "VBQ_ERR_SHAPE"
    m2 = Matrix(256, 128, seed_path=(90, 3, 1))
    even = vbq.vbq_pack(*m2.device_args(DEV))
    with pytest.raises(vbq.VbqError) as e:
        vbq.vbq_gemv_swiglu(even, x, y, h[1:])
    assert e.value.name == "VBQ_ERR_ALIGN"
    with pytest.raises(vbq.VbqError) as e:
        vbq.vbq_gemv_swiglu(even, x, y, None)
    assert e.value.name == "VBQ_ERR_ARG"


@pytest.mark.parametrize("name", ["stack131m-fused", "stack1b-fused", "stack9b-fused"])
def test_gate_up_fullsize_graph(name):
    # every layer's full-size gate-up matrix with its epilogue, captured in one
    # graph on one stream and replayed twice; sampled features checked against
    # the oracle row pair by row pair
    work = synth.workload(name, 1)
    specs = [s for s in work.mats if s.name.endswith("gate_up")][:4]
    rng = np.random.default_rng(11)
    inps = [gen.matrix_inputs(s, 1) for s in specs]
    lays, xs, ys, hs = [], [], [], []
    for s, inp in zip(specs, inps):
        wd = torch.from_numpy(inp["widths"]).to(DEV)
        codes = gen.codes_torch(wd, inp["key"], s.k, device=DEV)
        lays.append(vbq.vbq_pack(codes, wd, scales_to_i16(inp["scales"]).to(DEV)))
        del codes
        xs.append(bits_to_i16(inp["x_bits"][0]).to(DEV))
        ys.append(torch.empty(s.n, dtype=torch.float32, device=DEV))
        hs.append(torch.empty(s.n // 2, dtype=torch.int16, device=DEV))
    stream = torch.cuda.Stream()

    def step():
        for lay, x, y, h in zip(lays, xs, ys, hs):
            vbq.vbq_gemv_swiglu(lay, x, y, h, stream=stream)

    with torch.cuda.stream(stream):
        step()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        step()
    for _ in range(2):
        g.replay()
    torch.cuda.synchronize()
    for s, inp, y, h in zip(specs, inps, ys, hs):
        feats = sorted({0, s.n // 2 - 1, *(int(f) for f in rng.integers(0, s.n // 2, size=6))})
        rows = [r for f in feats for r in (2 * f, 2 * f + 1)]
        codes = np.concatenate([gen.codes_torch(inp["widths"], inp["key"], s.k, row0=r, nrows=1,
                                                device="cpu").numpy() for r in rows])
        x = gen.bf16_bits_to_f32(inp["x_bits"][:1])
        y_ref, a_ref = oracle.gemv(codes, inp["widths"][rows], inp["scales"][rows], x)
        yg = y.cpu().numpy()[rows][None, :]
        hg = gen.bf16_bits_to_f32(h.cpu().numpy().view(np.uint16)[feats])[None, :]
        assert oracle.within_bound(yg, y_ref, a_ref).all(), s.name
        assert oracle.swiglu_within_bound(hg, y_ref, a_ref).all(), s.name


# ---------------------------------------------------------------------------
# vbq_gemv_swiglu_in: the down projection reading the gate-up output, h in fp32
# inside the kernel (never stored)
# ---------------------------------------------------------------------------

def _gate_up_vector(k, seed):
    return gen.draw_gate_up(k, gen.rng_for((89, k, seed)))


def _run_in(layout, gu, n):
    g = torch.from_numpy(gu).to(DEV)
    y = torch.full((n,), float("nan"), dtype=torch.float32, device=DEV)
    vbq.vbq_gemv_swiglu_in(layout, g, y)
    torch.cuda.synchronize()
    return y.cpu().numpy()


def _assert_down(y, codes, widths, scales, gu, rows=None):
    h_ref = oracle.swiglu(gu[None, :])
    y_ref, a_ref = oracle.gemv(codes, widths, scales, h_ref)
    got = y[None, :] if rows is None else y[rows][None, :]
    ok = oracle.within_bound(got, y_ref, a_ref)
    assert ok.all(), f"{int((~ok).sum())} outputs outside the bound"


# (rows, K): K = 64 is one group; 2048 / 5632 / 14336 the intermediate widths of
# the three stacks' down projections (several slabs); 300 rows a ragged block
SHAPES_IN = [(64, 64), (768, 2048), (300, 64 * 37), (2048, 5632), (1000, 1024)]


@pytest.mark.parametrize("shape", SHAPES_IN, ids=lambda s: f"{s[0]}x{s[1]}")
@pytest.mark.parametrize("dist", ["main", "mlp0"])
def test_swiglu_in_parity(shape, dist):
    n, k = shape
    d = {"main": synth.DIST_MAIN, "mlp0": synth.DIST_MLP0}[dist]
    m = Matrix(n, k, dist=d, seed_path=(89, n, k))
    layout = vbq.vbq_pack(*m.device_args(DEV))
    gu = _gate_up_vector(k, 0)
    _assert_down(_run_in(layout, gu, n), m.codes.numpy(), m.widths, m.scales, gu)


def test_swiglu_in_fullsize_9b_down_sampled():
    # the 9B stack's down projection (4096 x 14336), sampled rows
    m = Matrix(4096, 14336, seed_path=(89, 9, 0), codes_device=DEV)
    layout = vbq.vbq_pack(*m.device_args(DEV))
    gu = _gate_up_vector(14336, 1)
    y = _run_in(layout, gu, m.n)
    rows = sorted({0, 4095, *(int(r) for r in np.random.default_rng(3).integers(0, 4096, size=10))})
    _assert_down(y, m.rows_codes_cpu(rows), m.widths[rows], m.scales[rows], gu, rows)


@pytest.mark.parametrize("b", [2, 4, 8])
def test_swiglu_in_all_zero_level_exact(b):
    # the zero-level sums use the same fp32 activations as the lookups and
    # products, in the same order: a matrix of zero-level codes gives exactly 0
    n, k = 256, 2048
    codes = np.full((n, k), 1 << (b - 1), np.uint8)
    widths = np.full((n, k // 64), b, np.uint8)
    m = Matrix(n, k, seed_path=(89, b, 1))
    layout = vbq.vbq_pack(torch.from_numpy(codes).to(DEV), torch.from_numpy(widths).to(DEV),
                          scales_to_i16(m.scales).to(DEV))
    y = _run_in(layout, _gate_up_vector(k, 2), n)
    assert float(np.abs(y).max()) == 0.0


def test_swiglu_in_padded_features_only():
    # every feature padded (gate = up = 0): h = 0, so y = 0 exactly
    m = Matrix(512, 1024, seed_path=(89, 4, 0))
    layout = vbq.vbq_pack(*m.device_args(DEV))
    y = _run_in(layout, np.zeros(2048, np.float32), 512)
    assert float(np.abs(y).max()) == 0.0


def test_swiglu_in_rejects_bad_arguments():
    m = Matrix(256, 128, seed_path=(89, 5, 0))
    layout = vbq.vbq_pack(*m.device_args(DEV))
    gu = torch.zeros(260, dtype=torch.float32, device=DEV)
    y = torch.empty(256, dtype=torch.float32, device=DEV)
    with pytest.raises(vbq.VbqError) as e:
        vbq.vbq_gemv_swiglu_in(layout, gu[1:], y)
    assert e.value.name == "VBQ_ERR_ALIGN"
    with pytest.raises(vbq.VbqError) as e:
        vbq.vbq_gemv_swiglu_in(layout, None, y)
    assert e.value.name == "VBQ_ERR_ARG"


@pytest.mark.parametrize("name", ["stack131m-fused", "stack1b-fused"])
def test_mlp_chain_graph(name):
    # layer 1's MLP as bench.py's fused_swiglu_in mode runs it: gate-up product
    # (vbq_gemv), then the down projection on its output (vbq_gemv_swiglu_in),
    # captured in one graph. The oracle computes the whole chain from the
    # inputs; the bound on the down output adds the gate-up error carried
    # through |W_down| (swiglu_error_bound, plus 2^-20 |h| for h's fp32
    # evaluation) to the product bound.
    work = synth.workload(name, 1)
    gs, ds = [s for s in work.mats if s.name == "l1.gate_up"][0], [s for s in work.mats if s.name == "l1.down"][0]
    ig, idn = gen.matrix_inputs(gs, 1), gen.matrix_inputs(ds, 1)
    mats, lays = [], []
    for s, inp in ((gs, ig), (ds, idn)):
        codes = gen.codes_torch(inp["widths"], inp["key"], s.k, device="cpu")
        mats.append(codes)
        lays.append(vbq.vbq_pack(codes.to(DEV), torch.from_numpy(inp["widths"]).to(DEV),
                                 scales_to_i16(inp["scales"]).to(DEV)))
    lay_g, lay_d = lays
    x = bits_to_i16(ig["x_bits"][0]).to(DEV)
    ygu = torch.empty(gs.n, dtype=torch.float32, device=DEV)
    y = torch.empty(ds.n, dtype=torch.float32, device=DEV)
    stream = torch.cuda.Stream()

    def step():
        vbq.vbq_gemv(lay_g, x, ygu, stream=stream)
        vbq.vbq_gemv_swiglu_in(lay_d, ygu, y, stream=stream)

    with torch.cuda.stream(stream):
        step()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        step()
    for _ in range(2):
        g.replay()
    torch.cuda.synchronize()
    xg = gen.bf16_bits_to_f32(ig["x_bits"][:1])
    y_gu, a_gu = oracle.gemv(mats[0].numpy(), ig["widths"], ig["scales"], xg)
    h_ref = oracle.swiglu(y_gu)
    e_h = oracle.swiglu_error_bound(y_gu, a_gu) + 2.0 ** -20 * np.abs(h_ref)
    w_d = np.abs(oracle.dequant(mats[1].numpy(), idn["widths"], idn["scales"]))
    y_ref, a_ref = oracle.gemv(mats[1].numpy(), idn["widths"], idn["scales"], h_ref)
    carried = (w_d @ e_h[0])[None, :]
    tol = 2e-3 * (a_ref + carried) + carried + 1e-5
    got = y.cpu().numpy()[None, :]
    assert (np.abs(got - y_ref) <= tol).all()
