"""Benchmark: batch-1 VBQ decode GEMV over a synthetic decoder linear stack.

One step = one token through every linear layer of the stack, each a packed
VBQ GEMV run by libvbq.so on one stream, replayed from a CUDA graph. The
headline (default workload stack9b) is layer-serial: one GEMV per projection
(Q, K, V, O, gate, up, down per layer, then the LM head), each launch ordered
after the previous one. Weights are random-but-seeded (synthetic) with the
per-projection width distributions of the workload; every GEMV has its own
resident BF16 activation vector.

`modes` reports, for a stack workload at batch 1, companions measured in the
same run: `grouped_by_input` (the headline's products in decode order, those
that read the same input, Q/K/V and gate/up, issued as one vbq_gemv_group),
`fused` (the <stack>-fused workload: QKV and gate-up as single matrices, 4
GEMVs per layer), `fused_swiglu` (the same with the gate-up product's SwiGLU
epilogue in its kernel, vbq_gemv_swiglu, whose BF16 output is the down
projection's input: the MLP as one dependent chain), `fused_swiglu_in` (the
same chain with the SwiGLU applied by the down projection as it stages its
activations from the gate-up product's fp32 output, vbq_gemv_swiglu_in),
`chain` (the headline's products as one vbq_chain_run: one
persistent launch per step, every product still waiting for all earlier
ones, weights streamed across product boundaries), `chain_by_input` (the same
chain where a product that reads the same input as its predecessor, K and V
after Q, up after gate, waits only for what that predecessor waits for),
`chain_fused` (the same for
the fused workload), `chain_independent` (the headline's products as one
chain without waits: independent products in one persistent launch, the
kernel's streaming upper bound), `grouped` (all of the headline's layouts as one
vbq_gemv_group per step: independent products whose launches overlap, the
streaming upper bound) and `cublas_bf16` (dense BF16 weights of the same
shapes through torch.mv, i.e. cuBLAS, as a reference point), `recipe` (the
fixed recipe's widths on the same shapes, layer-serial), and for the ~9B stack
`stack1b` (the ~1B stack, layer-serial as the headline) and `batch16_mlp`
(vbq_gemm_small at batch 16 on the 14336x4096 MLP shape); and, on the
workload's largest non-head matrix, `quantize` (vbq_quantize, the export-time
quantiser) and `soft_quant` (vbq_soft_quant, the training-time soft forward).

Printed JSON line (rank 0):
  value         algorithmic HBM GB/s of the whole step: sum over GEMVs of
                (packed payload + FP16 scales + x + y bytes) / step time.
  roofline      the GEMV kernel (the only kernel of the step): per-launch
                algorithmic bytes / CUDA-event launch duration, against the
                measured copy bandwidth; `traffic` is the DRAM bytes per launch
                modelled from committed one-launch ncu captures per matrix
                shape (each launch's algorithmic bytes times its shape's
                DRAM/algorithmic ratio), reported only while the kernel
                sources still hash to the captured ones.
  e2e           the same metric with the step's activations copied in from
                pinned host memory and the head's logits copied back, inside
                the timed region.
  cpu_baseline  the CPU oracle (numpy fp64) on a bounded row sample of the
                same stack, one process per host core (and on one core).

Workloads smaller than three times L2 are replicated (every copy packed
separately) so that each step streams its weights from HBM; a step is then one
pass over all copies, and tokens/s counts one token per copy.

`--impl reference` times the CPU oracle alone on the same workload (rank 0).
"""

from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = ("batch-1 decode GEMV achieved HBM GB/s (% of ~8 TB/s) and layer-stack tokens/s")
NOMINAL_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=300)
    p.add_argument("--warmup", type=int, default=10)
    p.add_argument("--impl", default="ours", choices=["ours", "reference"])
    p.add_argument("--workload", default="stack9b")
    p.add_argument("--batch", type=int, default=1)
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--sweep", action="store_true",
                   help="print the roofline sweep (N = K in 4096/8192/16384, batch 1..16, five width "
                        "distributions) as one JSON line instead of the stack benchmark")
    p.add_argument("--no-modes", action="store_true",
                   help="skip the fused, grouped and cuBLAS BF16 companion measurements")
    p.add_argument("--event-ring", type=int, default=4)
    return p.parse_args()


def measured_peak():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


# the sources that define the batch-1 GEMV kernel's code (the profiled kernel)
GEMV_SOURCES = ("vbq_common.cuh", "vbq_device.cuh", "vbq_gemv.cu")


def kernel_source_hash() -> str:
    """sha256 over the CUDA sources that define the GEMV kernel (sorted by name)."""
    h = hashlib.sha256()
    for name in sorted(GEMV_SOURCES):
        f = os.path.join(ROOT, "paper_2607_02893_gb300", "csrc", name)
        h.update(name.encode())
        with open(f, "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()


TRAFFIC_PROFILE = os.path.join(ROOT, "profiles", "gemv1_dram_traffic_by_shape.md")


def shape_traffic_ratios():
    """DRAM bytes over algorithmic bytes of one batch-1 GEMV launch per matrix
    shape, from the committed per-shape ncu captures (one launch each, a small
    replicated workload per shape): {(n, k): ratio}, or None when the file is
    absent or the GEMV kernel's sources changed since the captures."""
    try:
        kv, ratios = {}, {}
        with open(TRAFFIC_PROFILE) as f:
            for line in f:
                line = line.strip()
                if line.startswith("shape:"):
                    n, k, dram, alg = line.split(":", 1)[1].split()[:4]
                    ratios[(int(n), int(k))] = float(dram) / float(alg)
                elif line.startswith("source_sha256:"):
                    kv["source_sha256"] = line.split(":", 1)[1].strip()
        if kv.get("source_sha256") != kernel_source_hash() or not ratios:
            return None
        return ratios
    except Exception:
        return None


def profiled_traffic(mats, nbytes, batch: int):
    """DRAM bytes per launch of the step, modelled from the per-shape captures:
    each launch's algorithmic bytes times its shape's measured DRAM/algorithmic
    ratio (the nearest captured shape by weight count where the exact shape
    was not captured), averaged over the step's launches. None at batch > 1,
    without captures, or after a kernel change."""
    ratios = shape_traffic_ratios()
    if batch != 1 or ratios is None:
        return None
    total = 0.0
    for spec, nb in zip(mats, nbytes):
        key = (spec.n, spec.k)
        if key not in ratios:
            key = min(ratios, key=lambda nk: abs(np.log(nk[0] * nk[1] / (spec.n * spec.k))))
        total += ratios[key] * nb
    return total / len(nbytes)


def algorithmic_bytes(widths: np.ndarray, n: int, k: int, batch: int) -> int:
    """Packed payload + FP16 scales + BF16 x + FP32 y bytes of one product."""
    payload = int(widths.astype(np.int64).sum()) * 8
    return payload + 2 * widths.size + 2 * k * batch + 4 * n * batch


# ---------------------------------------------------------------------------
# clocks sampler (nvidia-smi during the timed region)
# ---------------------------------------------------------------------------

class ClockSampler:
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.QUERY}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if not self.proc:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.thread.join(timeout=2)
        sm, smax, reasons = [], 0.0, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax = max(smax, float(parts[2]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": smax, "reasons": sorted(reasons),
                "samples": len(sm)}


# ---------------------------------------------------------------------------
# CPU oracle leg
# ---------------------------------------------------------------------------

ORACLE_WEIGHTS_PER_S = 2.5e7     # rough single-core rate of the numpy oracle, for sizing samples


def oracle_block(spec, batch: int, rows: int, seed: int):
    """Time the oracle on a random contiguous block of `rows` rows of one matrix.

    Returns (seconds, algorithmic bytes of the block)."""
    import oracle
    from synth import gen
    rng = np.random.default_rng(seed)
    inp = gen.matrix_inputs(spec, batch)
    r = max(1, min(rows, spec.n))
    row0 = int(rng.integers(0, spec.n - r + 1))
    codes = gen.codes_torch(inp["widths"], inp["key"], spec.k, row0=row0, nrows=r,
                            device="cpu").numpy()
    w, s = inp["widths"][row0:row0 + r], inp["scales"][row0:row0 + r]
    x = gen.bf16_bits_to_f32(inp["x_bits"])
    t0 = time.perf_counter()
    oracle.gemv(codes, w, s, x)
    return time.perf_counter() - t0, algorithmic_bytes(w, r, spec.k, batch)


def host_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count() or 1


def _oracle_worker(q, barrier, workload, batch, blocks, rounds, rank):
    """One host process of the parallel oracle legs (spawned: no CUDA state is
    inherited). Prepares its row blocks first (untimed: input generation is
    not the oracle), then per round waits for every process at the barrier and
    runs the oracle on its next block, reporting (round, start, end, bytes)."""
    os.environ["OMP_NUM_THREADS"] = "1"
    import oracle
    import synth
    from synth import gen
    try:
        import torch
        torch.set_num_threads(1)
    except Exception:
        pass
    work = synth.workload(workload, batch)
    prepared = []
    for mi, rows, seed in blocks:
        spec = work.mats[mi]
        rng = np.random.default_rng(seed)
        inp = gen.matrix_inputs(spec, batch)
        r = max(1, min(rows, spec.n))
        row0 = int(rng.integers(0, spec.n - r + 1))
        codes = gen.codes_torch(inp["widths"], inp["key"], spec.k, row0=row0, nrows=r, device="cpu").numpy()
        w, sc = inp["widths"][row0:row0 + r], inp["scales"][row0:row0 + r]
        prepared.append((codes, w, sc, gen.bf16_bits_to_f32(inp["x_bits"]),
                         algorithmic_bytes(w, r, spec.k, batch), r))
    for rd in range(rounds):
        codes, w, sc, x, nb, r = prepared[rd % len(prepared)]
        barrier.wait()
        t0 = time.perf_counter()
        oracle.gemv(codes, w, sc, x)
        q.put((rd, rank, t0, time.perf_counter(), nb, r))


def oracle_parallel(work, workload: str, batch: int, cores: int, rounds: int, block_s: float, seed: int):
    """The oracle, unchanged, on `cores` host processes at once: in each round
    every process runs one random row block (about block_s seconds of work),
    the blocks cycling through the workload's matrices. Returns per round
    (wall seconds from the first start to the last end, algorithmic bytes,
    rows)."""
    import multiprocessing as mp
    ctx = mp.get_context("spawn")
    m = len(work.mats)
    q, barrier = ctx.Queue(), ctx.Barrier(cores)
    procs = []
    for p in range(cores):
        blocks = []
        for rd in range(min(rounds, 8)):
            mi = (rd * cores + p) % m
            rows = max(1, int(block_s * ORACLE_WEIGHTS_PER_S / work.mats[mi].k))
            blocks.append((mi, rows, seed + rd * cores + p))
        pr = ctx.Process(target=_oracle_worker, args=(q, barrier, workload, batch, blocks, rounds, p))
        pr.start()
        procs.append(pr)
    got = [q.get(timeout=600) for _ in range(rounds * cores)]
    for pr in procs:
        pr.join(timeout=60)
    out = []
    for rd in range(rounds):
        rs = [g for g in got if g[0] == rd]
        out.append((max(g[3] for g in rs) - min(g[2] for g in rs), sum(g[4] for g in rs), sum(g[5] for g in rs)))
    return out


def oracle_leg(work, batch: int, budget_s: float, seed: int = 0):
    """The oracle on one row block of every matrix, about `budget_s` seconds of
    oracle time in all. Block sizes follow the rate measured so far on this
    host; matrices are revisited (new random blocks) until the budget is met."""
    m = len(work.mats)
    t, nb, rows_done, weights, i = 0.0, 0, 0, 0, 0
    rate = ORACLE_WEIGHTS_PER_S
    while i < m or t < 0.9 * budget_s:
        spec = work.mats[i % m]
        target = (budget_s - t) / max(1, m - i) if i < m else min(0.5, budget_s - t)
        rows = max(1, int(max(target, 0.002) * rate / spec.k))
        dt, b = oracle_block(spec, batch, rows, seed + i)
        r = min(rows, spec.n)
        t += dt
        nb += b
        rows_done += r
        weights += r * spec.k
        rate = weights / max(t, 1e-9)
        i += 1
    frac = rows_done / sum(mm.n for mm in work.mats)
    return t, nb, frac


# ---------------------------------------------------------------------------
# GPU leg
# ---------------------------------------------------------------------------

def setup_stack(work, batch, dev, min_bytes: int = 0):
    """Pack every matrix of the workload, as many copies of the whole workload
    as it takes to stream at least min_bytes per pass. Returns per GEMV:
    layouts, device activations, outputs, algorithmic bytes, host activations;
    and the number of copies."""
    import torch
    import paper_2607_02893_gb300 as vbq
    from synth import gen
    inps = [gen.matrix_inputs(spec, batch) for spec in work.mats]
    once = sum(algorithmic_bytes(inp["widths"], spec.n, spec.k, batch) for spec, inp in zip(work.mats, inps))
    copies = max(1, -(-min_bytes // once))
    layouts, xs, ys, nbytes, host_x = [], [], [], [], []
    for _ in range(copies):
        for spec, inp in zip(work.mats, inps):
            wd = torch.from_numpy(inp["widths"]).to(dev)
            codes = gen.codes_torch(wd, inp["key"], spec.k, device=dev)
            sc = torch.from_numpy(inp["scales"].view(np.uint16).astype(np.int16)).to(dev)
            layouts.append(vbq.vbq_pack(codes, wd, sc))
            del codes, wd, sc
            xb = inp["x_bits"].astype(np.uint16).view(np.int16)
            host_x.append(xb)
            xs.append(torch.from_numpy(xb.copy()).to(dev))
            ys.append(torch.empty((batch, spec.n), dtype=torch.float32, device=dev))
            nbytes.append(algorithmic_bytes(inp["widths"], spec.n, spec.k, batch))
    torch.cuda.synchronize()
    return layouts, xs, ys, nbytes, host_x, copies


def max_over_ranks(vals, device=None):
    """Element-wise maximum of vals over the ranks of the default process group
    (the values themselves on a single process)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return [float(v) for v in vals]
    t = torch.tensor([float(v) for v in vals], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(v) for v in t.cpu()]


def job_throughput(step_bytes: int, copies: int, batch: int, world: int, ms_max: float):
    """Whole-job GB/s and tokens/s: every rank streams its own replica of the
    step, so the job moves world times the bytes in the slowest rank's time."""
    gbs = step_bytes * world / (ms_max * 1e-3) / 1e9
    tok_s = batch * copies * world / (ms_max * 1e-3)
    return gbs, tok_s


def time_graph(torch, stream, fn, steps: int, warmup: int) -> float:
    """ms per replay of fn captured as one CUDA graph on stream."""
    with torch.cuda.stream(stream):
        fn()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        fn()
    with torch.cuda.stream(stream):
        for _ in range(warmup):
            g.replay()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    with torch.cuda.stream(stream):
        for _ in range(steps):
            g.replay()
    e1.record(stream)
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / steps


def companion_modes(args, work, layouts, xs, ys, step_bytes, copies, stream, dev, l2):
    """The fused, grouped and cuBLAS BF16 companions of a batch-1 stack."""
    import torch
    import paper_2607_02893_gb300 as vbq
    import synth
    steps, warm = max(20, args.steps // 2), args.warmup
    out = {}

    def entry(ms, nbytes, cp, launches, note):
        return {"ms_per_step": round(ms, 4), "value": round(nbytes / (ms * 1e-3) / 1e9, 1), "unit": "GB/s",
                "tokens_per_s": round(cp / (ms * 1e-3), 1), "gemvs_per_step": launches, "note": note}

    x0 = [x[0] for x in xs]
    y0 = [y[0] for y in ys]
    ms = time_graph(torch, stream, lambda: vbq.vbq_gemv_group(layouts, x0, y0, stream=stream), steps, warm)
    out["grouped"] = entry(ms, step_bytes, copies, len(layouts),
                           "the headline layouts as one vbq_gemv_group per step (independent products, "
                           "overlapping launches): the streaming upper bound")
    # the headline's chain in one persistent launch: every product still waits
    # for all earlier ones before it touches x and y (layer-serial), but the
    # weights stream across product boundaries
    chain = vbq.Chain(layouts, x0, y0)
    ms = time_graph(torch, stream, lambda: chain.run(stream=stream), steps, warm)
    out["chain"] = entry(ms, step_bytes, copies, len(layouts),
                         "the headline's products as one vbq_chain_run per step (one persistent launch; every "
                         "product waits for all earlier ones, as layer-serial; weights stream across products)")
    chain.free()
    chain = vbq.Chain(layouts, x0, y0, [0] * len(layouts))
    ms = time_graph(torch, stream, lambda: chain.run(stream=stream), steps, warm)
    out["chain_independent"] = entry(ms, step_bytes, copies, len(layouts),
                                     "the headline's products as one vbq_chain_run with no waits (independent "
                                     "products in one persistent launch): the kernel's streaming upper bound")
    chain.free()
    # the decode step's own dependencies: K and V read Q's input, up reads
    # gate's, so they share their predecessor's dependencies (waits 2)
    by_input = [2 if m.name.rpartition(".")[2] in ("k", "v", "up") else 1 for m in work.mats] * copies
    if 2 in by_input:
        chain = vbq.Chain(layouts, x0, y0, by_input)
        ms = time_graph(torch, stream, lambda: chain.run(stream=stream), steps, warm)
        out["chain_by_input"] = entry(ms, step_bytes, copies, len(layouts),
                                      "the headline's products as one vbq_chain_run with the decode step's "
                                      "dependencies: Q, K, V wait for the previous layer, O for Q, K and V, gate "
                                      "and up for O, down for gate and up")
        chain.free()
    # the decode order with products that read the same input issued as one
    # group: per layer (Q, K, V) together, O, (gate, up) together, down
    names = [m.name for m in work.mats] * copies
    steps_list, i = [], 0
    while i < len(names):
        proj = names[i].rpartition(".")[2]
        span = 3 if proj == "q" else 2 if proj == "gate" else 1
        steps_list.append(list(range(i, i + span)))
        i += span
    if any(len(st) > 1 for st in steps_list):
        def by_input():
            for st in steps_list:
                if len(st) == 1:
                    vbq.vbq_gemv(layouts[st[0]], x0[st[0]], y0[st[0]], stream=stream)
                else:
                    xin = x0[st[0]]
                    vbq.vbq_gemv_group([layouts[j] for j in st], [xin] * len(st), [y0[j] for j in st], stream=stream)
        ms = time_graph(torch, stream, by_input, steps, warm)
        out["grouped_by_input"] = entry(ms, step_bytes, copies, len(layouts),
                                        "the headline's products in decode order, those that read the same input "
                                        "(Q, K, V; gate, up) issued as one vbq_gemv_group: "
                                        f"{len(steps_list)} dependent steps per token")
    name = args.workload
    if name in ("stack131m", "stack1b", "stack9b"):
        fwork = synth.workload(name + "-fused", 1)
        flays, fxs, fys, fnb, _, fcp = setup_stack(fwork, 1, dev, min_bytes=3 * l2)
        ms = time_graph(torch, stream,
                        lambda: [vbq.vbq_gemv(l, x[0], y[0], stream=stream) for l, x, y in zip(flays, fxs, fys)],
                        steps, warm)
        out["fused"] = entry(ms, sum(fnb), fcp, len(flays),
                             "workload " + name + "-fused: QKV and gate-up as single matrices, layer-serial")
        fchain = vbq.Chain(flays, [x[0] for x in fxs], [y[0] for y in fys])
        ms = time_graph(torch, stream, lambda: fchain.run(stream=stream), steps, warm)
        out["chain_fused"] = entry(ms, sum(fnb), fcp, len(flays),
                                   "workload " + name + "-fused as one vbq_chain_run per step (every product "
                                   "waits for all earlier ones)")
        fchain.free()
        # the same chain with the MLP's SwiGLU fused into the products, so the
        # down projection consumes the gate-up product: (a) as the gate-up
        # kernel's epilogue (vbq_gemv_swiglu writes BF16 h, the down
        # projection reads it); (b) in the down projection's activation
        # staging (vbq_gemv_swiglu_in reads the gate-up product's fp32 output)
        calls, prev = [], None
        for i, nm in enumerate([m.name for m in fwork.mats] * fcp):
            proj = nm.rpartition(".")[2]
            if proj == "gate_up":
                prev = (i, torch.empty(flays[i].N // 2, dtype=torch.int16, device=dev))
                calls.append((i, "gate_up", prev))
            elif proj == "down" and prev is not None:
                calls.append((i, "down", prev))
                prev = None
            else:
                calls.append((i, "gemv", None))

        def swiglu_chain(epilogue):
            for i, kind, link in calls:
                if kind == "gate_up" and epilogue:
                    vbq.vbq_gemv_swiglu(flays[i], fxs[i][0], fys[i][0], link[1], stream=stream)
                elif kind == "down" and epilogue:
                    vbq.vbq_gemv(flays[i], link[1], fys[i][0], stream=stream)
                elif kind == "down":
                    vbq.vbq_gemv_swiglu_in(flays[i], fys[link[0]][0], fys[i][0], stream=stream)
                else:
                    vbq.vbq_gemv(flays[i], fxs[i][0], fys[i][0], stream=stream)
        ms = time_graph(torch, stream, lambda: swiglu_chain(True), steps, warm)
        out["fused_swiglu"] = entry(ms, sum(fnb), fcp, len(flays),
                                    "workload " + name + "-fused with vbq_gemv_swiglu for gate-up (SwiGLU "
                                    "epilogue in the product kernel, BF16 h) feeding the down projection, "
                                    "layer-serial")
        ms = time_graph(torch, stream, lambda: swiglu_chain(False), steps, warm)
        out["fused_swiglu_in"] = entry(ms, sum(fnb), fcp, len(flays),
                                       "workload " + name + "-fused, the down projection as vbq_gemv_swiglu_in on "
                                       "the gate-up product's fp32 output (SwiGLU while staging activations, h "
                                       "never stored), layer-serial")
        del flays, fxs, fys
        torch.cuda.empty_cache()
        rwork = synth.workload(name + "-recipe", 1)
        rlays, rxs, rys, rnb, _, rcp = setup_stack(rwork, 1, dev, min_bytes=3 * l2)
        ms = time_graph(torch, stream,
                        lambda: [vbq.vbq_gemv(l, x[0], y[0], stream=stream) for l, x, y in zip(rlays, rxs, rys)],
                        steps, warm)
        out["recipe"] = entry(ms, sum(rnb), rcp, len(rlays),
                              "workload " + name + "-recipe: the fixed recipe's widths (§3.4; layer-0 MLP "
                              "4-bit, other projections 2-bit, head tiered per row, mean 1.18 bits), "
                              "layer-serial, same shapes as the headline")
        del rlays, rxs, rys
        torch.cuda.empty_cache()
    # the ~1B layer stack, layer-serial as the headline, and a batch of 16 on
    # the ~9B stack's 14336x4096 MLP shape
    if name == "stack9b":
        peak, _ = measured_peak()
        w1 = synth.workload("stack1b", 1)
        l1, x1, y1, nb1, _, cp1 = setup_stack(w1, 1, dev, min_bytes=3 * l2)
        ms = time_graph(torch, stream,
                        lambda: [vbq.vbq_gemv(l, x[0], y[0], stream=stream) for l, x, y in zip(l1, x1, y1)],
                        steps, warm)
        e1 = entry(ms, sum(nb1), cp1, len(l1), "workload stack1b (~1B stack, 155 GEMVs per token), layer-serial "
                   "as the headline" + (f"; packed {cp1} times to exceed 3x L2" if cp1 > 1 else ""))
        e1["frac"] = round(e1["value"] / peak, 4)
        out["stack1b"] = e1
        del l1, x1, y1
        torch.cuda.empty_cache()
        wb = synth.workload("matrix:14336:4096:main", 16)
        lb, xb, yb, nbb, _, cpb = setup_stack(wb, 16, dev, min_bytes=3 * l2)
        ms = time_graph(torch, stream,
                        lambda: [vbq.vbq_gemm_small(l, x, y, 16, stream=stream) for l, x, y in zip(lb, xb, yb)],
                        steps, warm)
        eb = entry(ms, sum(nbb), cpb * 16, len(lb), "vbq_gemm_small, batch 16, on 14336x4096 (main width mix), "
                   f"{cpb} packed copies cycled; value counts payload + scales + 16 x and 16 y per product")
        eb["frac"] = round(eb["value"] / peak, 4)
        eb["us_per_product"] = round(ms * 1e3 / len(lb), 2)
        out["batch16_mlp"] = eb
        del lb, xb, yb
        torch.cuda.empty_cache()
    # dense BF16 reference: the same shapes, one copy per packed copy so the
    # weights stream from HBM too
    g = torch.Generator(device=dev)
    g.manual_seed(0)
    dense, dx, dy, dbytes = [], [], [], 0
    for _ in range(copies):
        for spec in work.mats:
            dense.append(torch.randn((spec.n, spec.k), generator=g, device=dev, dtype=torch.bfloat16) * 0.02)
            dx.append(torch.randn(spec.k, generator=g, device=dev, dtype=torch.bfloat16))
            dy.append(torch.empty(spec.n, device=dev, dtype=torch.bfloat16))
            dbytes += 2 * spec.n * spec.k + 2 * spec.k + 2 * spec.n
    ms = time_graph(torch, stream, lambda: [torch.mv(w, x, out=y) for w, x, y in zip(dense, dx, dy)], steps, warm)
    out["cublas_bf16"] = entry(ms, dbytes, copies, len(dense),
                               "dense BF16 weights of the same shapes, torch.mv (cuBLAS), layer-serial; "
                               "value counts the BF16 weight bytes it streams")
    del dense, dx, dy
    torch.cuda.empty_cache()
    # the export step: vbq_quantize of the stack's largest non-head matrix,
    # whole calls (device validation, host read-back of its flags, then the
    # quantisation kernel), timed with events on the stream
    cands = [m for m in work.mats if not m.name.startswith("head")] or list(work.mats)
    big = max(cands, key=lambda m: m.n * m.k)
    w = torch.randn((big.n, big.k), generator=g, device=dev, dtype=torch.float32) * 0.02
    wd = torch.tensor([1, 2, 4, 8], dtype=torch.uint8, device=dev)[
        torch.multinomial(torch.tensor(synth.DIST_MAIN, device=dev), big.n * (big.k // 64), replacement=True,
                          generator=g)].reshape(big.n, big.k // 64)
    qc = torch.empty((big.n, big.k), dtype=torch.uint8, device=dev)
    qs = torch.empty((big.n, big.k // 64), dtype=torch.int16, device=dev)
    for _ in range(3):
        vbq.vbq_quantize(w, wd, qc, qs, stream=stream)
    reps = 10
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(reps):
        vbq.vbq_quantize(w, wd, qc, qs, stream=stream)
    e1.record(stream)
    torch.cuda.synchronize()
    qms = e0.elapsed_time(e1) / reps
    qbytes = big.n * big.k * 5 + (big.n * big.k // 64) * 3      # fp32 in, codes out; width in, scale out
    out["quantize"] = {"ms_per_call": round(qms, 4), "value": round(qbytes / (qms * 1e-3) / 1e9, 1), "unit": "GB/s",
                       "weights_per_s": round(big.n * big.k / (qms * 1e-3), 1), "shape": [big.n, big.k],
                       "note": "vbq_quantize (Eq. 1 / 1-bit absmean per group) of an FP32 matrix at the main width "
                               "mix, whole calls: device validation pass and its flag read-back, then the "
                               "quantisation kernel; value counts 4 B in and 1 B out per weight"}
    del w, wd, qc, qs
    torch.cuda.empty_cache()
    try:
        out["soft_quant"] = soft_quant_mode(torch, vbq, big, dev)
    except Exception as e:                      # a companion never takes the headline down
        out["soft_quant"] = {"error": f"{type(e).__name__}: {e}"}
    return out


def soft_quant_mode(torch, vbq, spec, dev):
    """The training-time soft forward (vbq_soft_quant, §3.2 / Alg. 1) on the
    workload's largest non-head matrix: median of 10 calls, each after an L2
    flush, timed with events."""
    from synth import gen
    n, k = spec.n, spec.k
    w, lg, gb = gen.draw_soft_inputs(n, k, gen.rng_for((72, n, k)))
    W, L, E = (torch.from_numpy(a).to(dev) for a in (w, lg, gb))
    ws = torch.empty_like(W)
    eb = torch.empty((n, k // 64), dtype=torch.float32, device=dev)
    hw = torch.empty((n, k // 64), dtype=torch.uint8, device=dev)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    for _ in range(3):
        vbq.vbq_soft_quant(W, L, 0.5, gumbel=E, w_soft=ws, exp_bits=eb, hard_widths=hw)
    times = []
    for _ in range(10):
        flush.zero_()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        vbq.vbq_soft_quant(W, L, 0.5, gumbel=E, w_soft=ws, exp_bits=eb, hard_widths=hw)
        e1.record()
        torch.cuda.synchronize()
        times.append(e0.elapsed_time(e1))
    ms = statistics.median(times)
    groups = n * k // 64
    nbytes = n * k * 8 + groups * (16 + 16 + 4 + 1)
    del W, L, E, ws, eb, hw, flush
    torch.cuda.empty_cache()
    return {"ms_per_call": round(ms, 4), "value": round(nbytes / (ms * 1e-3) / 1e9, 1), "unit": "GB/s",
            "weights_per_s": round(n * k / (ms * 1e-3), 1), "shape": [n, k],
            "note": "vbq_soft_quant (training-time soft forward: pi = softmax((l + e) / tau), the convex "
                    "combination of the 1/2/4/8-bit reconstructions, expected and hardened widths) at tau 0.5 "
                    "with Gumbel noise; value counts 4 B in and 4 B out per weight, 32 B in and 5 B out per group"}


def run_ours(args, rank, world, local_rank):
    import torch
    import paper_2607_02893_gb300 as vbq
    import synth

    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    vbq.load()
    work = synth.workload(args.workload, args.batch)
    B = args.batch
    l2 = int(getattr(torch.cuda.get_device_properties(dev), "L2_cache_size", 0)) or (129 << 20)
    layouts, xs, ys, nbytes, host_x, copies = setup_stack(work, B, dev, min_bytes=3 * l2)
    step_bytes = sum(nbytes)
    stream = torch.cuda.Stream(device=dev)

    def launch_all(events=None):
        for i, lay in enumerate(layouts):
            if events is not None:
                events[i][0].record(stream)
            if B == 1:
                vbq.vbq_gemv(lay, xs[i][0], ys[i][0], stream=stream)
            else:
                vbq.vbq_gemm_small(lay, xs[i], ys[i], B, stream=stream)
            if events is not None:
                events[i][1].record(stream)

    # warm the kernels (sets function attributes outside capture)
    with torch.cuda.stream(stream):
        launch_all()
    torch.cuda.synchronize()

    # the step captured once as a CUDA graph
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        launch_all()
    torch.cuda.synchronize()

    def barrier():
        if world > 1:
            import torch.distributed as dist
            dist.barrier()

    with torch.cuda.stream(stream):
        for i in range(args.warmup):
            graph.replay()
    torch.cuda.synchronize()

    # --- timed region: device-resident inputs --------------------------------
    clocks = ClockSampler(int(os.environ.get("CUDA_VISIBLE_DEVICES", "0").split(",")[0])
                          if "CUDA_VISIBLE_DEVICES" in os.environ else local_rank)
    clocks.start()
    time.sleep(0.3)
    barrier()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    with torch.cuda.stream(stream):
        for i in range(args.steps):
            graph.replay()
    e1.record(stream)
    torch.cuda.synchronize()
    barrier()
    clk = clocks.stop()
    ms = e0.elapsed_time(e1) / args.steps

    # --- isolated launch durations: one step launched eagerly with an event
    # pair around every GEMV, queued behind a device-side sleep so that the
    # host has enqueued the whole step before the first launch runs (host
    # launch latency then never shows in the events). The events between
    # launches also remove the programmatic-dependent-launch overlap of the
    # graph, so these are the kernels' stand-alone durations.
    ring = max(1, args.event_ring)
    events = [[(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in layouts] for _ in range(ring)]
    sleep_cycles = 40_000_000
    queued_ahead = True
    for r in range(ring):
        for attempt in range(4):
            torch.cuda.synchronize()
            with torch.cuda.stream(stream):
                torch.cuda._sleep(sleep_cycles)
                launch_all(events[r])
            ahead = not stream.query()      # still busy: the host got ahead of the GPU
            torch.cuda.synchronize()
            if ahead:
                break
            sleep_cycles *= 2
        queued_ahead = queued_ahead and ahead
    durs = [ev[i][0].elapsed_time(ev[i][1]) for ev in events for i in range(len(layouts))]
    isolated_ms_per_step = sum(durs) / ring

    # --- e2e: host activations in, head logits out ------------------------------
    pinned_x = torch.from_numpy(np.concatenate([h.reshape(-1) for h in host_x])).pin_memory()
    dev_x_flat = torch.empty_like(pinned_x, device=dev)
    head_out = torch.empty(ys[-1].shape, dtype=torch.float32).pin_memory()
    offs = np.cumsum([0] + [h.size for h in host_x])
    xs_views = [dev_x_flat[offs[i]:offs[i + 1]].view(xs[i].shape) for i in range(len(xs))]
    g_e2e = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g_e2e, stream=stream):
        for i, lay in enumerate(layouts):
            if B == 1:
                vbq.vbq_gemv(lay, xs_views[i][0], ys[i][0], stream=stream)
            else:
                vbq.vbq_gemm_small(lay, xs_views[i], ys[i], B, stream=stream)
    h2d = pinned_x.numel() * 2
    d2h = head_out.numel() * 4
    e2e_steps = max(3, args.steps // 4)
    for i in range(3):
        with torch.cuda.stream(stream):
            dev_x_flat.copy_(pinned_x, non_blocking=True)
            g_e2e.replay()
            head_out.copy_(ys[-1], non_blocking=True)
    torch.cuda.synchronize()
    barrier()
    t0 = time.perf_counter()
    for i in range(e2e_steps):
        with torch.cuda.stream(stream):
            dev_x_flat.copy_(pinned_x, non_blocking=True)
            g_e2e.replay()
            head_out.copy_(ys[-1], non_blocking=True)
        stream.synchronize()
        _ = float(head_out[0, 0])          # the result is read on the host every step
    e2e_ms = (time.perf_counter() - t0) * 1e3 / e2e_steps
    barrier()

    ms_max, e2e_max = max_over_ranks([ms, e2e_ms], device=dev)
    gbs, tok_s = job_throughput(step_bytes, copies, B, world, ms_max)
    peak, peak_kind = measured_peak()
    # Every launch of the timed region is the GEMV kernel, so its average launch
    # duration is the timed region's device time over its launches (launches
    # overlap by their prologues under programmatic dependent launch).
    kernel_ms_per_step = ms
    kernel_gbs = step_bytes / (kernel_ms_per_step * 1e-3) / 1e9
    launches = len(layouts)
    traffic = profiled_traffic(work.mats * copies, nbytes, B)
    result = {
        "metric": METRIC,
        "value": round(gbs, 1),
        "unit": "GB/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(ms_max, 4),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "f32",
        "data": "synthetic",
        "config": {
            "workload": args.workload,
            "batch": B,
            "gemvs_per_step": launches,
            "copies": copies,
            "weights": work.weights * copies,
            "algorithmic_bytes_per_step": step_bytes,
            "tokens_per_s": round(tok_s, 1),
            "pct_of_nominal_8TBs": round(100 * gbs / world / NOMINAL_HBM_GBS, 2),
            "l2": (f"inputs larger than L2 ({l2 >> 20} MiB): each step streams every packed weight once"
                   + (f"; the workload is packed {copies} times to get there" if copies > 1 else "")),
            "activations": "BF16 N(0,1), one resident vector per GEMV",
        },
        "roofline": {
            "bound": "hbm",
            "kernel": "gemv1_kernel (vbq_gemv)" if B == 1 else "vbq_gemm_small (gemmb_kernel, or gemv1_kernel<2> for B = 2..4 by layout)",
            "achieved": round(kernel_gbs, 1),
            "peak": peak,
            "peak_kind": peak_kind,
            "unit": "GB/s",
            "frac": round(kernel_gbs / peak, 4),
            "traffic": None if traffic is None else round(traffic),
            "traffic_source": ("ncu dram__bytes_read.sum + dram__bytes_write.sum of one launch per matrix shape "
                               "(profiles/gemv1_dram_traffic_by_shape.md), as a ratio to that launch's "
                               "algorithmic bytes, applied to every launch of the step and averaged; null "
                               "when absent or the kernel changed since"),
            "launches_timed": launches * args.steps,
            "avg_launch_us": round(kernel_ms_per_step * 1e3 / launches, 3),
            "duration_source": "CUDA events around the timed region on the launching stream, "
                               "divided by its launches (all of them this kernel)",
            "isolated_avg_launch_us": round(isolated_ms_per_step * 1e3 / launches, 3),
            "isolated_note": (f"eager pass of {ring} step(s), an event pair per launch, queued behind a "
                              "device sleep" + ("" if queued_ahead else " that did not cover the host's queueing")
                              + "; no PDL overlap between launches"),
        },
        "e2e": {
            "value": round(job_throughput(step_bytes, copies, B, world, e2e_max)[0], 1),
            "unit": "GB/s",
            "h2d_bytes_per_step": int(h2d),
            "d2h_bytes_per_step": int(d2h),
            "tokens_per_s": round(job_throughput(step_bytes, copies, B, world, e2e_max)[1], 1),
        },
        "gpu_launches": launches * args.steps,
        "clocks": clk,
    }
    if B == 1 and not args.no_modes and world == 1:
        result["modes"] = companion_modes(args, work, layouts, xs, ys, step_bytes, copies, stream, dev, l2)
    return result, work


def run_sweep(args):
    """Every point of the roofline sweep: per (N, distribution) as many packed
    copies as it takes to exceed 3x L2, then per batch a CUDA graph of launches
    cycling through the copies; device time per launch, algorithmic GB/s and
    the fraction of the measured copy bandwidth."""
    import torch
    import paper_2607_02893_gb300 as vbq
    import synth
    from synth import gen
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    vbq.load()
    l2 = int(getattr(torch.cuda.get_device_properties(dev), "L2_cache_size", 0)) or (129 << 20)
    peak, peak_kind = measured_peak()
    stream = torch.cuda.Stream(device=dev)
    points = []
    for n in (4096, 8192, 16384):
        for dist in synth.SWEEP_DISTS:
            spec = synth.workload(f"sweep:{n}:{dist}", 16).mats[0]
            inp = gen.matrix_inputs(spec, 16)
            wd = torch.from_numpy(inp["widths"]).to(dev)
            sc = torch.from_numpy(inp["scales"].view(np.uint16).astype(np.int16)).to(dev)
            one = algorithmic_bytes(inp["widths"], n, n, 1)
            copies = max(1, -(-3 * l2 // one))
            codes = gen.codes_torch(wd, inp["key"], n, device=dev)
            lays = [vbq.vbq_pack(codes, wd, sc) for _ in range(copies)]
            del codes
            X = torch.from_numpy(inp["x_bits"].astype(np.uint16).view(np.int16).copy()).to(dev)
            for b in (1, 2, 4, 8, 16):
                Y = torch.empty((b, n), dtype=torch.float32, device=dev)
                reps = 4 * copies
                if b == 1:
                    fn = lambda: [vbq.vbq_gemv(lays[i % copies], X[0], Y[0], stream=stream) for i in range(reps)]
                else:
                    fn = lambda: [vbq.vbq_gemm_small(lays[i % copies], X[:b], Y, b, stream=stream)
                                  for i in range(reps)]
                ms = time_graph(torch, stream, fn, steps=5, warmup=3) / reps
                nb = algorithmic_bytes(inp["widths"], n, n, b)
                gbs = nb / (ms * 1e-3) / 1e9
                points.append({"n": n, "dist": dist, "batch": b, "us": round(ms * 1e3, 2),
                               "GBs": round(gbs, 1), "frac": round(gbs / peak, 4),
                               "tokens_per_s": round(b / (ms * 1e-3), 1)})
            del lays
            torch.cuda.empty_cache()
    return {"sweep": points, "peak": peak, "peak_kind": peak_kind, "unit": "GB/s",
            "note": "algorithmic bytes (payload + FP16 scales + BF16 x + FP32 y) per launch over its device time, "
                    "inputs larger than L2 (copies cycled)"}


def run_reference(args):
    """The CPU oracle as the reference arm, on every host core: each step is
    one round of row blocks, one per host process (spawned processes started
    together at a barrier), the blocks cycling through the workload's
    matrices. ms_per_step is a round's measured wall time (so steps x
    ms_per_step is the time the run spent in the oracle) and value is the
    algorithmic GB/s over the timed rounds. The time a whole token would take
    at that rate is reported separately, as an extrapolation."""
    import synth
    work = synth.workload(args.workload, args.batch)
    cores = host_cores()
    block_s = min(1.0, 100.0 / max(1, args.steps + args.warmup))
    rounds = oracle_parallel(work, args.workload, args.batch, cores, rounds=args.warmup + args.steps,
                             block_s=block_s, seed=1000)[args.warmup:]
    t = sum(r[0] for r in rounds)
    nbytes = sum(r[1] for r in rounds)
    rows_seen = sum(r[2] for r in rounds)
    gbs = nbytes / t / 1e9
    ms_per_step = t / args.steps * 1e3
    token_bytes = sum(algorithmic_bytes_est(mm, args.batch) for mm in work.mats)
    ms_per_token = token_bytes / (gbs * 1e9) * 1e3
    sample = (f"per step one random contiguous row block per host process ({cores} processes, about "
              f"{block_s:.2f} s of work each), cycling through the {len(work.mats)} matrices; {rows_seen} rows "
              f"timed; inputs prepared before the timed rounds")
    return {
        "impl": "reference",
        "metric": METRIC,
        "value": round(gbs, 4),
        "unit": "GB/s",
        "n_gpus": 1,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(ms_per_step, 3),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "f64",
        "data": "synthetic",
        "config": {"workload": args.workload, "batch": args.batch,
                   "step": "a bounded sample of the workload (see cpu_baseline.sample), not a whole token",
                   "ms_per_token_extrapolated": round(ms_per_token, 3),
                   "tokens_per_s_extrapolated": round(args.batch / (ms_per_token * 1e-3), 6)},
        "cpu_baseline": {"value": round(gbs, 4), "unit": "GB/s", "cores": cores, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": round(gbs, 4), "unit": "GB/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }


def algorithmic_bytes_est(spec, batch: int) -> int:
    """Algorithmic bytes of one matrix from its drawn widths."""
    from synth import gen
    rng = gen.rng_for(spec.seed_path)
    widths = gen.spec_widths(spec, rng)
    return algorithmic_bytes(widths, spec.n, spec.k, batch)


def main():
    args = parse()
    if args.warmup < 3:
        args.warmup = 3
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.gpus > 1 and "WORLD_SIZE" not in os.environ:
        # no launcher: start one replica per GPU the same way the driver does
        import socket
        with socket.socket() as sk:
            sk.bind(("127.0.0.1", 0))
            port = sk.getsockname()[1]
        cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", f"--nproc-per-node={args.gpus}",
               "--master-addr", "127.0.0.1", "--master-port", str(port), os.path.abspath(__file__), *sys.argv[1:]]
        sys.exit(subprocess.call(cmd))
    if world != args.gpus:
        sys.exit(f"bench.py: --gpus {args.gpus} but WORLD_SIZE is {world}")

    if args.sweep:
        if rank == 0:
            print(json.dumps(run_sweep(args)), flush=True)
        return

    if args.impl == "reference":
        if rank == 0:
            print(json.dumps(run_reference(args)), flush=True)
        return

    if world > 1:
        import torch
        import torch.distributed as dist
        torch.cuda.set_device(local_rank)
        dist.init_process_group("nccl")
    result, work = run_ours(args, rank, world, local_rank)
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        t, nb, frac = oracle_leg(work, args.batch, budget_s=8.0)
        cores = host_cores()
        rounds = oracle_parallel(work, args.workload, args.batch, cores, rounds=9, block_s=1.0, seed=5000)[1:]
        wall = sum(r[0] for r in rounds)
        nbp = sum(r[1] for r in rounds)
        result["cpu_baseline"] = {
            "value": round(nbp / wall / 1e9, 4), "unit": "GB/s", "cores": cores, "kind": "oracle",
            "sample": f"8 rounds (after one untimed) of one random contiguous row block per host process (about 1 s of work each; "
                      f"{sum(r[2] for r in rounds)} rows) cycling through the {len(work.mats)} matrices, "
                      f"{wall:.1f} s of wall time on {cores} processes at once (numpy fp64; inputs prepared "
                      f"before the timed rounds)",
            "single_core": {"value": round(nb / t / 1e9, 4), "unit": "GB/s", "cores": 1,
                            "sample": f"random contiguous row blocks, at least one of each matrix "
                                      f"({frac * 100:.3f}% of all rows), {t:.1f} s on one host core"},
        }
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
        dist.destroy_process_group()
    if rank == 0:
        print(json.dumps(result), flush=True)


if __name__ == "__main__":
    main()
