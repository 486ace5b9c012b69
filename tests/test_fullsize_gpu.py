"""Full-size parity: every matrix of the benchmarked stacks and the roofline
sweep, run through the C ABI in the launch configuration bench.py times (one
stream, all GEMVs of a stack captured in one CUDA graph and replayed), with
sampled rows checked against the CPU oracle row by row."""

import numpy as np
import pytest
import torch

import oracle
import paper_2607_02893_gb300 as vbq
import synth
from synth import gen
from vbq_cases import bits_to_i16, scales_to_i16

pytestmark = pytest.mark.gpu

DEV = "cuda"
ROWS_PER_MATRIX = 6


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2607_02893_gb300 import build
    build.build()
    vbq.load()
    torch.cuda.init()


def _sample_rows(n, rng):
    rows = {0, n - 1}
    rows.update(int(r) for r in rng.integers(0, n, size=ROWS_PER_MATRIX))
    return sorted(rows)


def _oracle_rows(spec, inp, rows, batch):
    codes = np.concatenate([gen.codes_torch(inp["widths"], inp["key"], spec.k, row0=r, nrows=1,
                                            device="cpu").numpy() for r in rows])
    x = gen.bf16_bits_to_f32(inp["x_bits"][:batch])
    return oracle.gemv(codes, inp["widths"][rows], inp["scales"][rows], x)


def _pack(spec, inp):
    wd = torch.from_numpy(inp["widths"]).to(DEV)
    codes = gen.codes_torch(wd, inp["key"], spec.k, device=DEV)
    lay = vbq.vbq_pack(codes, wd, scales_to_i16(inp["scales"]).to(DEV))
    del codes
    return lay


@pytest.mark.parametrize("name", ["single768", "stack131m", "stack1b", "stack9b",
                                  "stack131m-fused", "stack1b-fused", "stack9b-fused",
                                  "stack131m-recipe", "stack1b-recipe", "stack9b-recipe"])
def test_stack_fullsize_sampled(name):
    work = synth.workload(name, 1)
    rng = np.random.default_rng(7)
    inps = [gen.matrix_inputs(spec, 1) for spec in work.mats]
    lays = [_pack(spec, inp) for spec, inp in zip(work.mats, inps)]
    xs = [bits_to_i16(inp["x_bits"]).to(DEV) for inp in inps]
    ys = [torch.empty(spec.n, dtype=torch.float32, device=DEV) for spec in work.mats]
    st = torch.cuda.Stream()

    def run():
        for lay, x, y in zip(lays, xs, ys):
            vbq.vbq_gemv(lay, x[0], y, stream=st)

    with torch.cuda.stream(st):
        run()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=st):
        run()
    for y in ys:
        y.fill_(float("nan"))
    torch.cuda.synchronize()
    with torch.cuda.stream(st):
        g.replay()
        g.replay()
    torch.cuda.synchronize()
    bad = []
    for spec, inp, y in zip(work.mats, inps, ys):
        rows = _sample_rows(spec.n, rng)
        y_ref, a_ref = _oracle_rows(spec, inp, rows, 1)
        got = y.cpu().numpy()[rows][None, :]
        ok = oracle.within_bound(got, y_ref, a_ref)
        if not ok.all():
            bad.append((spec.name, int((~ok).sum())))
    assert not bad, f"outputs outside the bound: {bad[:10]}"


@pytest.mark.parametrize("n", [4096, 8192, 16384])
@pytest.mark.parametrize("dist", ["all1", "all2", "all4", "all8", "mixed"])
def test_sweep_fullsize_sampled(n, dist):
    spec = synth.workload(f"sweep:{n}:{dist}", 16).mats[0]
    inp = gen.matrix_inputs(spec, 16)
    lay = _pack(spec, inp)
    rng = np.random.default_rng(n)
    rows = _sample_rows(n, rng)
    X = bits_to_i16(inp["x_bits"]).to(DEV)
    for batch in (1, 2, 4, 8, 16):
        Y = torch.full((batch, n), float("nan"), dtype=torch.float32, device=DEV)
        if batch == 1:
            vbq.vbq_gemv(lay, X[0], Y[0])
        else:
            vbq.vbq_gemm_small(lay, X[:batch].contiguous(), Y, batch)
        torch.cuda.synchronize()
        y_ref, a_ref = _oracle_rows(spec, inp, rows, batch)
        got = Y.cpu().numpy()[:, rows]
        ok = oracle.within_bound(got, y_ref, a_ref)
        assert ok.all(), f"sweep {n} {dist} batch {batch}: {int((~ok).sum())} outside the bound"
