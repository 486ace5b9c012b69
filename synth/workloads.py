"""Workload descriptions: matrix shapes and per-group bit-width distributions.

Shapes follow the decoder families of the paper's inference study (§6,
Table 2: a ~131M TinyStories decoder, ~1B and ~9B models) as plain linear
stacks: per layer Q, K, V, O, gate, up, down, then the LM head. W is stored
N x K (output features x input features); groups of 64 run along K.

The "-fused" stacks hold the same projections with the ones that read the
same input stacked into one matrix, as a decode step issues them: Q, K and V
as one QKV matrix, gate and up as one matrix (4 products per layer instead of
7). Their weights are drawn per fused matrix (same shapes, same
distributions, their own seeds); O and down keep the per-projection seeds.

Bit-width distributions are probabilities over widths (1, 2, 4, 8):
  * main:  the adaptive-search allocation of §5.1 (most groups at 1 bit),
           p = (0.69, 0.15, 0.11, 0.05), mean 1.83 bits;
  * mlp0:  the first block's MLP, which keeps more precision (§5.1, §3.4),
           p = (0.40, 0.30, 0.22, 0.08), mean 2.50 bits;
  * head:  the LM head, mostly 1 bit (§5.1), p = (0.96, 0.025, 0.01, 0.005),
           mean 1.09 bits.
"""

from __future__ import annotations

from dataclasses import dataclass, field
from typing import Optional, List, Tuple

WIDTHS = (1, 2, 4, 8)

DIST_MAIN = (0.69, 0.15, 0.11, 0.05)
DIST_MLP0 = (0.40, 0.30, 0.22, 0.08)
DIST_HEAD = (0.96, 0.025, 0.01, 0.005)
DIST_ALL1 = (1.0, 0.0, 0.0, 0.0)
DIST_ALL2 = (0.0, 1.0, 0.0, 0.0)
DIST_ALL4 = (0.0, 0.0, 1.0, 0.0)
DIST_ALL8 = (0.0, 0.0, 0.0, 1.0)

SWEEP_DISTS = {
    "all1": DIST_ALL1, "all2": DIST_ALL2, "all4": DIST_ALL4, "all8": DIST_ALL8,
    "mixed": DIST_MAIN,
}


@dataclass(frozen=True)
class MatrixSpec:
    """One weight matrix of a workload: W is n x k, groups of 64 along k.

    Widths are drawn i.i.d. per group from dist, unless tiers is set: then
    every group of a row takes its row's tier width, tiers given as
    (cumulative fraction of rows, width) in row order (the recipe's
    frequency-tiered head, rows sorted by token frequency)."""
    name: str
    n: int
    k: int
    dist: Tuple[float, float, float, float]
    seed_path: Tuple[int, ...]   # (config_id, layer, proj_id) for the seed sequence
    tiers: Optional[Tuple[Tuple[float, int], ...]] = None


@dataclass
class Workload:
    name: str
    config_id: int
    batch: int
    mats: List[MatrixSpec] = field(default_factory=list)

    @property
    def weights(self) -> int:
        return sum(m.n * m.k for m in self.mats)


# The fixed VBQ recipe (§3.4): the first block's MLP at 4 bits, every other
# projection at 2 bits, the LM head tiered per row by token-frequency rank:
# top 0.5% of rows at 8 bits, next 1.5% at 4, next 10% at 2, the last 88% at 1.
RECIPE_HEAD_TIERS = ((0.005, 8), (0.02, 4), (0.12, 2), (1.0, 1))


def _stack(config_id: int, d_model: int, n_layers: int, d_q: int, d_kv: int,
           d_ff: int, vocab: int, fused: bool = False, recipe: bool = False) -> List[MatrixSpec]:
    mats: List[MatrixSpec] = []
    if recipe:
        config_id += 100            # its own seeds
    main = DIST_ALL2 if recipe else DIST_MAIN
    for layer in range(n_layers):
        mlp = (DIST_ALL4 if recipe else DIST_MLP0) if layer == 0 else main
        # (name, n, k, dist, proj_id)
        if fused:
            projs = [
                ("qkv", d_q + 2 * d_kv, d_model, main, 7),
                ("o", d_model, d_q, main, 3),
                ("gate_up", 2 * d_ff, d_model, mlp, 8),
                ("down", d_model, d_ff, mlp, 6),
            ]
        else:
            projs = [
                ("q", d_q, d_model, main, 0),
                ("k", d_kv, d_model, main, 1),
                ("v", d_kv, d_model, main, 2),
                ("o", d_model, d_q, main, 3),
                ("gate", d_ff, d_model, mlp, 4),
                ("up", d_ff, d_model, mlp, 5),
                ("down", d_model, d_ff, mlp, 6),
            ]
        for pname, n, k, dist, pid in projs:
            mats.append(MatrixSpec(f"l{layer}.{pname}", n, k, dist, (config_id, layer, pid)))
    if recipe:
        mats.append(MatrixSpec("head", vocab, d_model, DIST_HEAD, (config_id, n_layers, 0), RECIPE_HEAD_TIERS))
    else:
        mats.append(MatrixSpec("head", vocab, d_model, DIST_HEAD, (config_id, n_layers, 0)))
    return mats


# name -> (config_id, (d_model, n_layers, d_q, d_kv, d_ff, vocab))
_STACKS = {
    "stack131m": (1, (768, 12, 768, 768, 2048, 32000)),
    "stack1b": (2, (2048, 22, 2048, 256, 5632, 32000)),
    "stack9b": (3, (4096, 32, 4096, 1024, 14336, 128256)),
}


def workload(name: str, batch: int = 1) -> Workload:
    """Named workloads.

    single768   one 768 x 768 GEMV, main distribution.
    stack131m   d_model 768, 12 layers, MLP 2048, head 32000 (85 GEMVs).
    stack1b     d_model 2048, 22 layers, Q/O 2048, K/V 256, MLP 5632, head 32000 (155 GEMVs).
    stack9b     d_model 4096, 32 layers, Q/O 4096, K/V 1024, MLP 14336, head 128256 (225 GEMVs).
    <stack>-fused   the same stack with QKV and gate-up fused (131m: 49, 1b: 89, 9b: 129 GEMVs).
    <stack>-recipe  the same shapes with the fixed recipe's widths (§3.4): layer-0 MLP all
                    4-bit, other projections all 2-bit, head tiered per row (mean 1.18 bits).
    sweep:<n>:<dist>  one n x n GEMV, dist in all1/all2/all4/all8/mixed.
    matrix:<n>:<k>:<dist>  one n x k GEMV (for profiling single shapes).
    """
    if name.endswith("-fused") and name[:-6] in _STACKS:
        cid, dims = _STACKS[name[:-6]]
        return Workload(name, cid, batch, _stack(cid, *dims, fused=True))
    if name.endswith("-recipe") and name[:-7] in _STACKS:
        cid, dims = _STACKS[name[:-7]]
        return Workload(name, cid, batch, _stack(cid, *dims, recipe=True))
    if name in _STACKS:
        cid, dims = _STACKS[name]
        return Workload(name, cid, batch, _stack(cid, *dims))
    if name == "single768":
        return Workload(name, 0, batch, [MatrixSpec("w", 768, 768, DIST_MAIN, (0, 0, 0))])
    if name.startswith("matrix:"):
        # matrix:N:K:dist, dist in main / mlp0 / head / all1 / all2 / all4 / all8
        _, n, k, dist = name.split(":")
        dists = {"main": DIST_MAIN, "mlp0": DIST_MLP0, "head": DIST_HEAD, **{
            d: SWEEP_DISTS[d] for d in ("all1", "all2", "all4", "all8")}}
        n, k = int(n), int(k)
        return Workload(name, 5, batch, [MatrixSpec(f"m{n}x{k}.{dist}", n, k, dists[dist],
                                                    (5, n, k, list(dists).index(dist)))])
    if name.startswith("sweep:"):
        _, n, dist = name.split(":")
        n = int(n)
        didx = list(SWEEP_DISTS).index(dist)
        return Workload(name, 4, batch,
                        [MatrixSpec(f"sweep{n}.{dist}", n, n, SWEEP_DISTS[dist], (4, n, didx))])
    raise KeyError(name)


def workload_names() -> List[str]:
    return ["single768", "stack131m", "stack1b", "stack9b"]


def sweep_points() -> List[Tuple[int, int, str]]:
    """(n, batch, dist) of the roofline sweep: 3 sizes x 5 batches x 5 distributions."""
    return [(n, b, d) for n in (4096, 8192, 16384) for b in (1, 2, 4, 8, 16)
            for d in SWEEP_DISTS]
