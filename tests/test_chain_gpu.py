"""Parity of the persistent chain (vbq_chain_create / vbq_chain_run through
the C ABI) with the CPU oracle.

A chain runs its products in order in one launch, streaming weights across
product boundaries. Every y_i must satisfy the product bound of vbq_gemv.
Covered: products of one and several slabs, ragged row blocks, products with
fewer units than blocks, every product waiting (the default), mixed waits
and products sharing their predecessor's dependencies, repeated runs (the completion counts and split-K epochs carry over),
plain products on the same layouts between runs, graph capture, and the
full-size stacks as bench.py runs them (sampled rows)."""

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


SHAPES = [(768, 768), (1, 64), (129, 832), (300, 4096), (1000, 2048), (257, 64 * 37), (4096, 1024),
          (20000, 1024), (64, 64 * 200)]


def _mats(seed):
    return [Matrix(n, k, seed_path=(80 + seed, n, k)) for n, k in SHAPES]


def _check(ms, ys):
    for m, y in zip(ms, ys):
        y_ref, a_ref = oracle.gemv(m.codes.numpy(), m.widths, m.scales, m.x()[:1])
        ok = oracle.within_bound(y.cpu().numpy()[None, :], y_ref, a_ref)
        assert ok.all(), f"{m.n}x{m.k}: {int((~ok).sum())} outputs outside the bound"


WAITS = {"all": None, "mixed": [i % 2 for i in range(len(SHAPES))], "none": [0] * len(SHAPES),
         # decode-step style: products that read the same input share their
         # dependencies (waits 2), the next one waits for all of them
         "grouped": [1, 2, 2, 1, 2, 1, 0, 2, 1]}


@pytest.mark.parametrize("waits", sorted(WAITS))
def test_chain_parity(waits):
    ms = _mats(0)
    lays = [vbq.vbq_pack(*m.device_args(DEV)) for m in ms]
    xs = [bits_to_i16(m.x_bits[0]).to(DEV) for m in ms]
    ys = [torch.full((m.n,), float("nan"), dtype=torch.float32, device=DEV) for m in ms]
    w = WAITS[waits]
    chain = vbq.Chain(lays, xs, ys, w)
    for _ in range(3):
        for y in ys:
            y.fill_(float("nan"))
        chain.run()
        torch.cuda.synchronize()
        _check(ms, ys)
    vbq.vbq_device_status()
    chain.free()


def test_chain_runs_between_plain_products():
    # runs of a chain and vbq_gemv calls on the same layouts share their
    # split-K control words: each keeps the other's epochs valid
    ms = _mats(1)
    lays = [vbq.vbq_pack(*m.device_args(DEV)) for m in ms]
    xs = [bits_to_i16(m.x_bits[0]).to(DEV) for m in ms]
    ys = [torch.empty(m.n, dtype=torch.float32, device=DEV) for m in ms]
    chain = vbq.Chain(lays, xs, ys)
    for _ in range(2):
        chain.run()
        torch.cuda.synchronize()
        _check(ms, ys)
        yp = [torch.empty(m.n, dtype=torch.float32, device=DEV) for m in ms]
        for lay, x, y in zip(lays, xs, yp):
            vbq.vbq_gemv(lay, x, y)
        torch.cuda.synchronize()
        _check(ms, yp)
    vbq.vbq_device_status()


def test_chain_rejects_bad_arguments():
    ms = _mats(2)[:2]
    lays = [vbq.vbq_pack(*m.device_args(DEV)) for m in ms]
    xs = [bits_to_i16(m.x_bits[0]).to(DEV) for m in ms]
    ys = [torch.empty(m.n, dtype=torch.float32, device=DEV) for m in ms]
    for args, name in [((lays[:1] * 2, xs, ys), "VBQ_ERR_ARG"),          # a layout twice
                       ((lays, xs, [ys[0], ys[0]]), "VBQ_ERR_ARG"),       # an output twice
                       ((lays, xs, ys, [1, 3]), "VBQ_ERR_ARG"),           # a bad wait flag
                       ((lays, [xs[0][1:], xs[1]], ys), "VBQ_ERR_ALIGN")]:
        with pytest.raises(vbq.VbqError) as e:
            vbq.Chain(*args)
        assert e.value.name == name
    with pytest.raises(ValueError):
        vbq.Chain(lays, xs[:1], ys)


@pytest.mark.parametrize("name", ["stack131m", "stack1b", "stack9b", "stack9b-fused"])
def test_chain_fullsize_graph(name):
    # the whole stack as one chain (every product waiting), captured in a graph
    # and replayed three times, as bench.py's chain mode runs it
    work = synth.workload(name, 1)
    rng = np.random.default_rng(5)
    inps = [gen.matrix_inputs(spec, 1) for spec in work.mats]
    lays, xs, ys = [], [], []
    for spec, inp in zip(work.mats, inps):
        wd = torch.from_numpy(inp["widths"]).to(DEV)
        codes = gen.codes_torch(wd, inp["key"], spec.k, device=DEV)
        lays.append(vbq.vbq_pack(codes, wd, scales_to_i16(inp["scales"]).to(DEV)))
        del codes
        xs.append(bits_to_i16(inp["x_bits"][0]).to(DEV))
        ys.append(torch.full((spec.n,), float("nan"), dtype=torch.float32, device=DEV))
    chain = vbq.Chain(lays, xs, ys)
    stream = torch.cuda.Stream()
    with torch.cuda.stream(stream):
        chain.run(stream=stream)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        chain.run(stream=stream)
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    vbq.vbq_device_status()
    for spec, inp, y in zip(work.mats, inps, ys):
        rows = sorted({0, spec.n - 1, *(int(r) for r in rng.integers(0, spec.n, size=4))})
        codes = np.concatenate([gen.codes_torch(inp["widths"], inp["key"], spec.k, row0=r, nrows=1,
                                                device="cpu").numpy() for r in rows])
        x = gen.bf16_bits_to_f32(inp["x_bits"][:1])
        y_ref, a_ref = oracle.gemv(codes, inp["widths"][rows], inp["scales"][rows], x)
        ok = oracle.within_bound(y.cpu().numpy()[rows][None, :], y_ref, a_ref)
        assert ok.all(), f"{spec.name}: {int((~ok).sum())} of {len(rows)} sampled outputs outside the bound"
    chain.free()
