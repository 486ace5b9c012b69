"""Seeded generators for VBQ inputs.

Draw order per matrix, from one PCG64 stream seeded by
SeedSequence([0, config_id, layer, proj_id]):
  1. widths  rng.choice([1,2,4,8], size=(N, G), p=dist)           (uint8)
             (a tiered matrix, the recipe's head, draws nothing here: its
             widths are fixed per row by tier)
  2. scales  |rng.normal(0, 0.02, (N, G))| + 1e-4 -> float16 (RNE)  (float16)
  3. x       rng.normal(0, 1, (B, K)) float32 -> bfloat16 (RNE)     (uint16 bits)

Codes are drawn by a counter-based generator so that any subset of rows can
be produced on any device (CPU for the oracle, the GPU for full-size runs)
with identical values: code[n, k] = h(n*K + k) & (2^b - 1), where b is the
width of the group holding column k and h is the low byte of MurmurHash3's
32-bit finaliser ("fmix32", A. Appleby) applied to a Weyl sequence
idx * 0x9E3779B9 + key (mod 2^32). The key comes from
SeedSequence([0, config_id, layer, proj_id, 1]). Codes are therefore
uniform over the 2^b codes of their group.
"""

from __future__ import annotations

from typing import Optional, Sequence

import numpy as np

WIDTH_VALUES = np.array([1, 2, 4, 8], dtype=np.uint8)
_M32 = 0xFFFFFFFF
_WEYL = 0x9E3779B9
_C1 = 0x85EBCA6B
_C2 = 0xC2B2AE35


def rng_for(seed_path: Sequence[int]) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([0, *seed_path])))


def draw_widths(n: int, g: int, dist, rng: np.random.Generator) -> np.ndarray:
    p = np.asarray(dist, dtype=np.float64)
    p = p / p.sum()
    return rng.choice(WIDTH_VALUES, size=(n, g), p=p).astype(np.uint8)


def draw_scales(n: int, g: int, rng: np.random.Generator) -> np.ndarray:
    return (np.abs(rng.normal(0.0, 0.02, size=(n, g))) + 1e-4).astype(np.float16)


def draw_dense_weights(n: int, k: int, rng: np.random.Generator) -> np.ndarray:
    """Dense float32 weights for the quantiser: N(0, 0.02) scaled per 64-column
    group by exp(N(0, 0.5)) (groups of different magnitude), with 1% of the
    weights eight times larger (outliers)."""
    g = k // 64
    w = rng.normal(0.0, 0.02, size=(n, k))
    w *= np.repeat(np.exp(rng.normal(0.0, 0.5, size=(n, g))), 64, axis=1)
    w *= np.where(rng.random((n, k)) < 0.01, 8.0, 1.0)
    return w.astype(np.float32)


def f32_to_bf16_bits(a: np.ndarray) -> np.ndarray:
    """Round float32 values to bfloat16 (round to nearest even); return the bit patterns."""
    bits = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32).astype(np.uint64)
    rounded = (bits + 0x7FFF + ((bits >> 16) & 1)) >> 16
    return rounded.astype(np.uint16)


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def draw_x_bf16(batch: int, k: int, rng: np.random.Generator) -> np.ndarray:
    return f32_to_bf16_bits(rng.normal(0.0, 1.0, size=(batch, k)).astype(np.float32))


def draw_gate_up(k: int, rng: np.random.Generator) -> np.ndarray:
    """A gate-up product's output as the down projection reads it: 2k float32,
    gate and up of feature i at 2i and 2i + 1, both N(0, 1.5) (about the
    spread of the synthetic gate-up products), with one feature in eight
    zero-padded (gate and up exactly 0)."""
    gu = rng.normal(0.0, 1.5, size=(k, 2))
    gu[rng.random(k) < 0.125] = 0.0
    return gu.astype(np.float32).reshape(2 * k)


def draw_soft_inputs(n: int, k: int, rng: np.random.Generator):
    """Inputs of the training-time soft forward: weights as draw_dense_weights
    draws them, per-group logits over the 4 candidates N(0, 2), and standard
    Gumbel noise of the same shape (the draws the selection makes, passed in
    as data). Returns (w N x K, logits N x K/64 x 4, gumbel N x K/64 x 4),
    all float32."""
    w = draw_dense_weights(n, k, rng)
    logits = rng.normal(0.0, 2.0, size=(n, k // 64, 4)).astype(np.float32)
    gumbel = rng.gumbel(size=(n, k // 64, 4)).astype(np.float32)
    return w, logits, gumbel


def code_key(seed_path: Sequence[int]) -> int:
    return int(np.random.SeedSequence([0, *seed_path, 1]).generate_state(1, dtype=np.uint32)[0])


def fmix32_py(h: int) -> int:
    """MurmurHash3 32-bit finaliser, on Python ints (reference for the tensor version)."""
    h &= _M32
    h ^= h >> 16
    h = (h * _C1) & _M32
    h ^= h >> 13
    h = (h * _C2) & _M32
    h ^= h >> 16
    return h


def _mul32(a, c: int):
    """(a * c) mod 2^32 for an int64 tensor a in [0, 2^32), without int64 overflow."""
    lo, hi = c & 0xFFFF, c >> 16
    return (a * lo + (((a * hi) & 0xFFFF) << 16)) & _M32


def _fmix32_t(h):
    h = h ^ (h >> 16)
    h = _mul32(h, _C1)
    h = h ^ (h >> 13)
    h = _mul32(h, _C2)
    return h ^ (h >> 16)


def codes_torch(widths, key: int, k: int, row0: int = 0, nrows: Optional[int] = None,
                device=None, chunk_elems: int = 1 << 26):
    """Codes for rows [row0, row0+nrows) of an N x K matrix as a torch uint8 tensor.

    `widths` is the full (N, G) uint8 array (numpy or torch); the result lives on
    `device` (default: the device of `widths` if it is a tensor, else CPU).
    """
    import torch

    if isinstance(widths, np.ndarray):
        wt = torch.from_numpy(widths)
    else:
        wt = widths
    if device is None:
        device = wt.device
    n_total, g = wt.shape
    assert g * 64 == k
    if nrows is None:
        nrows = n_total - row0
    out = torch.empty((nrows, k), dtype=torch.uint8, device=device)
    rows_per_chunk = max(1, chunk_elems // k)
    col = torch.arange(k, dtype=torch.int64, device=device)
    for r in range(0, nrows, rows_per_chunk):
        rr = min(rows_per_chunk, nrows - r)
        rows = torch.arange(row0 + r, row0 + r + rr, dtype=torch.int64, device=device)
        idx = (rows[:, None] * k + col[None, :]) & _M32
        h = _fmix32_t((_mul32(idx, _WEYL) + key) & _M32)
        wb = wt[row0 + r: row0 + r + rr].to(device=device, dtype=torch.int64)
        mask = (torch.ones_like(wb) << wb) - 1                 # 2^b - 1 per group
        mask = mask.repeat_interleave(64, dim=1)
        out[r:r + rr] = ((h & 0xFF) & mask).to(torch.uint8)
    return out


def tiered_widths(n: int, g: int, tiers) -> np.ndarray:
    """Per-row widths from (cumulative fraction of rows, width) tiers in row
    order, every group of a row at its row's width. Tier boundaries are
    round(fraction * n)."""
    w = np.empty(n, dtype=np.uint8)
    start = 0
    for frac, b in tiers:
        end = n if frac >= 1.0 else min(n, int(round(frac * n)))
        w[start:end] = b
        start = max(start, end)
    return np.repeat(w[:, None], g, axis=1)


def spec_widths(spec, rng: np.random.Generator) -> np.ndarray:
    """A matrix's widths: per-row tiers when the spec has them (no random
    draw), else drawn i.i.d. per group from its distribution."""
    g = spec.k // 64
    tiers = getattr(spec, "tiers", None)
    if tiers:
        return tiered_widths(spec.n, g, tiers)
    return draw_widths(spec.n, g, spec.dist, rng)


def matrix_inputs(spec, batch: int):
    """Widths, scales and x of one matrix (numpy), plus its code key."""
    rng = rng_for(spec.seed_path)
    g = spec.k // 64
    widths = spec_widths(spec, rng)
    scales = draw_scales(spec.n, g, rng)
    x_bits = draw_x_bf16(batch, spec.k, rng)
    return {"widths": widths, "scales": scales, "x_bits": x_bits,
            "key": code_key(spec.seed_path)}
