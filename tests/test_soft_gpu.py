"""Parity of the training-time soft-quantised forward (vbq_soft_quant,
through the C ABI) with the CPU oracle.

Hardened widths must match bit-exactly; w_soft and the expected widths must
be within the float32 bound oracle.soft_quant_within_bound derives. Cases:
several shapes, temperatures at both ends of the paper's anneal (5.0 and
0.5), with and without Gumbel noise, exact half-way ties of the float32
quotients (a different rounding decision would move a weight by a whole
step), all-zero and dominant-logit groups, optional outputs, argument
errors, and a full-size 4096 x 14336 matrix (sampled rows)."""

import numpy as np
import pytest
import torch

import oracle
import paper_2607_02893_gb300 as vbq
from synth import gen

pytestmark = pytest.mark.gpu

DEV = "cuda"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2607_02893_gb300 import build
    build.build()
    vbq.load()
    torch.cuda.init()


def _run(w, logits, gumbel, tau):
    d = lambda a: None if a is None else torch.from_numpy(np.ascontiguousarray(a)).to(DEV)
    ws, eb, hw = vbq.vbq_soft_quant(d(w), d(logits), tau, gumbel=d(gumbel))
    torch.cuda.synchronize()
    return ws.cpu().numpy(), eb.cpu().numpy(), hw.cpu().numpy()


def _check(w, logits, gumbel, tau, ws, eb, hw, rows=None):
    if rows is not None:
        w, logits, ws, eb, hw = w[rows], logits[rows], ws[rows], eb[rows], hw[rows]
        gumbel = None if gumbel is None else gumbel[rows]
    _, _, hard_ref, _ = oracle.soft_quant_forward(w, logits, gumbel, tau)
    assert np.array_equal(hw, hard_ref), "hardened widths"
    ok_w, ok_b = oracle.soft_quant_within_bound(ws, eb, w, logits, gumbel, tau)
    assert ok_w.all(), f"{int((~ok_w).sum())} soft weights outside the bound"
    assert ok_b.all(), f"{int((~ok_b).sum())} expected widths outside the bound"


@pytest.mark.parametrize("shape", [(1, 64), (3, 128), (257, 1024), (64, 4096)], ids=lambda s: f"{s[0]}x{s[1]}")
@pytest.mark.parametrize("tau", [5.0, 0.5])
@pytest.mark.parametrize("noise", [True, False])
def test_soft_parity(shape, tau, noise):
    n, k = shape
    w, lg, gb = gen.draw_soft_inputs(n, k, gen.rng_for((70, n, k)))
    g = gb if noise else None
    ws, eb, hw = _run(w, lg, g, tau)
    _check(w, lg, g, tau, ws, eb, hw)


def test_soft_ties_zero_groups_and_dominant_logits():
    rng = gen.rng_for((70, 1, 1))
    n, k = 8, 256
    w, lg, gb = gen.draw_soft_inputs(n, k, rng)
    # exact half-way quotients: row r holds max|w| = qmax * 2^-6 in every group
    # and otherwise (j + 1/2) 2^-6 with |j + 1/2| < qmax, so at the width of
    # that qmax the scale is 2^-6 and every such quotient is a tie
    for r, qmax in ((0, 1), (1, 7), (2, 127)):
        row = ((np.arange(k) % (2 * qmax)) - qmax + 0.5).astype(np.float32) * np.float32(2.0 ** -6)
        row[::64] = qmax * 2.0 ** -6
        w[r] = row
    w[3] = 0.0                                     # all-zero groups
    w[4, :64] = -0.0
    lg[5] = 0.0
    lg[5, :, 3] = 40.0                             # a dominant logit
    lg[6] = 1.25                                   # all equal: ties to the first
    ws, eb, hw = _run(w, lg, gb, 0.7)
    _check(w, lg, gb, 0.7, ws, eb, hw)
    assert np.all(ws[3] == 0.0) and np.all(ws[4, :64] == 0.0)
    assert np.all(hw[6] == 1) and np.all(hw[5] == 8)


def test_soft_optional_outputs_and_repeat():
    n, k = 40, 512
    w, lg, gb = gen.draw_soft_inputs(n, k, gen.rng_for((70, 2, 0)))
    d = lambda a: torch.from_numpy(a).to(DEV)
    ws1, _, _ = vbq.vbq_soft_quant(d(w), d(lg), 1.3, gumbel=d(gb), exp_bits=False, hard_widths=False)
    ws2, eb2, hw2 = vbq.vbq_soft_quant(d(w), d(lg), 1.3, gumbel=d(gb))
    torch.cuda.synchronize()
    assert torch.equal(ws1, ws2), "w_soft does not depend on the optional outputs (and is deterministic)"
    _check(w, lg, gb, 1.3, ws2.cpu().numpy(), eb2.cpu().numpy(), hw2.cpu().numpy())


def test_soft_rejects_bad_arguments():
    w = torch.zeros((2, 128), device=DEV)
    lg = torch.zeros((2, 2, 4), device=DEV)
    for tau in (0.0, -1.0, float("inf"), float("nan")):
        with pytest.raises(vbq.VbqError) as e:
            vbq.vbq_soft_quant(w, lg, tau)
        assert e.value.name == "VBQ_ERR_ARG"
    with pytest.raises(vbq.VbqError) as e:
        vbq.vbq_soft_quant(torch.zeros((2, 96), device=DEV), lg, 1.0)
    assert e.value.name == "VBQ_ERR_SHAPE"
    with pytest.raises(vbq.VbqError) as e:
        vbq.vbq_soft_quant(w, lg, 1.0, w_soft=torch.zeros(2 * 128 + 1, device=DEV)[1:].view(2, 128))
    assert e.value.name == "VBQ_ERR_ALIGN"


def test_soft_fullsize_sampled():
    # the 9B stack's down projection shape, 4096 x 14336 (58.7M weights)
    n, k = 4096, 14336
    w, lg, gb = gen.draw_soft_inputs(n, k, gen.rng_for((70, 9, 0)))
    ws, eb, hw = _run(w, lg, gb, 0.5)
    rows = sorted({0, n - 1, *(int(r) for r in np.random.default_rng(4).integers(0, n, size=6))})
    _check(w, lg, gb, 0.5, ws, eb, hw, rows)


def test_soft_extreme_scales_and_near_ties():
    # The codes come from |w| * fl(1/s) unless that product is within 2^-15 of
    # a half-integer or s lies outside [2^-125, 2^125]; then from the IEEE
    # quotient. Groups here: max|w| near 1e-37, so the 8-bit scale is a float32
    # subnormal and the 4-bit one below 2^-125 (the weights themselves stay
    # mostly normal: the bound is relative, and subnormal weights would lose
    # relative precision in any float32 evaluation); scales so large that
    # fl(1/s) would be subnormal; zeros of both signs; and quotients placed a
    # few ulps and about 2^-14 from half-integers at each width (either
    # decision there moves a weight by a whole step).
    rng = gen.rng_for((70, 3, 0))
    n, k = 6, 64 * 8
    w = np.zeros((n, k), dtype=np.float32)
    w[0] = (rng.standard_normal(k) * 3e-38).astype(np.float32)          # 8-bit scale subnormal
    w[1] = (rng.standard_normal(k) * 1e35).astype(np.float32)          # sum|w| stays finite in float32
    w[1, ::64] = np.float32(3.0e38)                                       # s = max|w| above 2^125
    w[2, 1::2] = -0.0
    w[2, ::2] = rng.standard_normal(k // 2).astype(np.float32)
    for r, qmax in ((3, 1), (4, 7), (5, 127)):
        s = np.float32(np.float32(1.0) / np.float32(qmax))                # max|w| = 1 in every group
        j = (np.arange(k) % (2 * qmax)) - qmax
        half = ((j + 0.5) * s).astype(np.float32)
        ulps = rng.integers(-3, 4, size=k)
        near = np.nextafter(half, np.where(ulps >= 0, np.float32(np.inf), np.float32(-np.inf)))
        for _ in range(2):
            near = np.where(np.abs(ulps) > 1, np.nextafter(near, np.where(ulps >= 0, np.inf, -np.inf)).astype(np.float32), near)
        off = (half + np.float32(2.0 ** -14) * s * np.where(np.arange(k) % 3 == 0, 1, -1)).astype(np.float32)
        row = np.where(np.arange(k) % 2 == 0, near, off).astype(np.float32)
        row[::64] = np.float32(1.0)
        w[r] = np.clip(row, -1.0, 1.0)
    lg = rng.standard_normal((n, k // 64, 4)).astype(np.float32)
    ws, eb, hw = _run(w, lg, None, 0.8)
    _check(w, lg, None, 0.8, ws, eb, hw)
    assert np.isfinite(ws).all()
