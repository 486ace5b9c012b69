"""Full-row parity at full size: every output row of the ~9B stack's LM head
(128256 x 4096) and of one 14336 x 4096 MLP matrix, and the first and last
row of every 128-row block of every matrix of the ~9B stack, against the CPU
oracle. The GPU side runs the whole stack as bench.py times it (one stream,
captured in a CUDA graph, replayed); the oracle runs on every host core, in
row chunks, in processes started with spawn (no CUDA state is inherited)."""

import multiprocessing as mp
import os

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
CHUNK = 2048


def _oracle_rows(task):
    """Worker: (workload name, matrix index, sorted row list) -> (matrix index,
    rows, y_ref, a_ref); rows are taken in contiguous runs."""
    name, mi, rows = task
    os.environ["OMP_NUM_THREADS"] = "1"
    torch.set_num_threads(1)
    spec = synth.workload(name, 1).mats[mi]
    inp = gen.matrix_inputs(spec, 1)
    rows = np.asarray(rows, dtype=np.int64)
    cuts = np.flatnonzero(np.diff(rows) != 1) + 1
    codes = np.concatenate([gen.codes_torch(inp["widths"], inp["key"], spec.k, row0=int(run[0]), nrows=len(run),
                                            device="cpu").numpy() for run in np.split(rows, cuts)])
    x = gen.bf16_bits_to_f32(inp["x_bits"][:1])
    y_ref, a_ref = oracle.gemv(codes, inp["widths"][rows], inp["scales"][rows], x)
    return mi, rows, y_ref[0], a_ref[0]


@pytest.fixture(scope="module")
def stack9b_outputs():
    from paper_2607_02893_gb300 import build
    build.build()
    vbq.load()
    work = synth.workload("stack9b", 1)
    inps = [gen.matrix_inputs(spec, 1) for spec in work.mats]
    lays, xs, ys = [], [], []
    for spec, inp in zip(work.mats, inps):
        wd = torch.from_numpy(inp["widths"]).to(DEV)
        codes = gen.codes_torch(wd, inp["key"], spec.k, device=DEV)
        lays.append(vbq.vbq_pack(codes, wd, scales_to_i16(inp["scales"]).to(DEV)))
        del codes
        xs.append(bits_to_i16(inp["x_bits"][0]).to(DEV))
        ys.append(torch.full((spec.n,), float("nan"), dtype=torch.float32, device=DEV))
    st = torch.cuda.Stream()

    def run():
        for lay, x, y in zip(lays, xs, ys):
            vbq.vbq_gemv(lay, x, y, stream=st)

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
    out = [y.cpu().numpy() for y in ys]
    for lay in lays:
        lay.free()
    del ys, xs
    torch.cuda.empty_cache()
    return work, out


def _check(tasks, outs):
    bad = []
    with mp.get_context("spawn").Pool(min(len(tasks), os.cpu_count() or 1)) as pool:
        for mi, rows, y_ref, a_ref in pool.imap_unordered(_oracle_rows, tasks):
            ok = oracle.within_bound(outs[mi][rows], y_ref, a_ref)
            if not ok.all():
                bad.append((mi, int((~ok).sum()), int(rows[np.argmin(ok)])))
    return bad


def test_fullrow_head_and_mlp(stack9b_outputs):
    work, outs = stack9b_outputs
    names = [m.name for m in work.mats]
    tasks = []
    for mi in (names.index("head"), names.index("l3.gate")):
        n = work.mats[mi].n
        tasks += [("stack9b", mi, list(range(r0, min(n, r0 + CHUNK)))) for r0 in range(0, n, CHUNK)]
    bad = _check(tasks, outs)
    assert not bad, f"(matrix, outputs outside the bound, first bad row): {bad[:10]}"


def test_fullrow_block_edges_every_matrix(stack9b_outputs):
    work, outs = stack9b_outputs
    tasks = []
    for mi, spec in enumerate(work.mats):
        rows = sorted({r for b in range(0, spec.n, 128) for r in (b, min(spec.n, b + 128) - 1)})
        for c0 in range(0, len(rows), CHUNK):
            tasks.append(("stack9b", mi, rows[c0:c0 + CHUNK]))
    bad = _check(tasks, outs)
    assert not bad, f"(matrix, outputs outside the bound, first bad row): {bad[:10]}"
