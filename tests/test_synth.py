"""Seeded input generators: determinism, ranges, and the paper's printed
distribution figures. CPU only."""

import os

import numpy as np
import pytest
import torch

import synth
from synth import gen, workloads

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _paper_numbers():
    out = {}
    with open(os.path.join(GOLDEN, "paper_numbers.txt")) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            name, val, _ = [p.strip() for p in line.split("|")]
            out[name] = val
    return out


def _mean_bits(dist):
    return sum(p * b for p, b in zip(dist, (1, 2, 4, 8)))


def test_distribution_means_match_paper():
    pn = _paper_numbers()
    assert abs(_mean_bits(synth.DIST_HEAD) - float(pn["head_mean_bits"])) < 0.005
    assert abs(_mean_bits(synth.DIST_MLP0) - float(pn["mlp0_mean_bits"])) < 0.05
    assert abs(synth.DIST_MAIN[0] - float(pn["one_bit_fraction"])) < 1e-9
    tiers = [t.split(":") for t in pn["recipe_head_tiers"].split()]
    recipe_mean = sum(float(f) * int(b) for f, b in tiers)
    assert abs(recipe_mean - float(pn["recipe_head_mean_bits"])) < 1e-9
    for d in (synth.DIST_MAIN, synth.DIST_MLP0, synth.DIST_HEAD):
        assert abs(sum(d) - 1.0) < 1e-12


def test_stack_shapes():
    w = synth.workload("stack9b")
    assert len(w.mats) == 32 * 7 + 1
    assert abs(w.weights / 7.5e9 - 1) < 0.01
    w1 = synth.workload("stack131m")
    assert len(w1.mats) == 85 and abs(w1.weights / 1.10e8 - 1) < 0.01
    w2 = synth.workload("stack1b")
    assert len(w2.mats) == 155 and abs(w2.weights / 1.03e9 - 1) < 0.01
    assert len(synth.sweep_points()) == 75
    for m in w.mats + w1.mats + w2.mats:
        assert m.k % 64 == 0


@pytest.mark.parametrize("name,layers", [("stack131m", 12), ("stack1b", 22), ("stack9b", 32)])
def test_fused_stack_shapes(name, layers):
    # same weights as the per-projection stack, 4 products per layer + the head
    a, b = synth.workload(name), synth.workload(name + "-fused")
    assert len(b.mats) == 4 * layers + 1 and b.weights == a.weights
    per = {m.name: m for m in a.mats}
    for m in b.mats:
        layer, _, proj = m.name.rpartition(".")
        if proj == "qkv":
            parts = [per[f"{layer}.{p}"] for p in ("q", "k", "v")]
        elif proj == "gate_up":
            parts = [per[f"{layer}.{p}"] for p in ("gate", "up")]
        else:
            parts = [per[m.name]]
            assert m.seed_path == parts[0].seed_path
        assert m.n == sum(p.n for p in parts) and all(p.k == m.k and p.dist == m.dist for p in parts)


def test_fmix32_tensor_matches_reference():
    # the int64-tensor formulation must equal the plain 32-bit definition
    key = gen.code_key((9, 9, 9))
    idx = np.array([0, 1, 2, 12345, 2**31 - 1, 2**32 - 1], dtype=np.int64)
    t = torch.from_numpy(idx)
    h = gen._fmix32_t((gen._mul32(t, gen._WEYL) + key) & gen._M32)
    ref = [gen.fmix32_py((int(i) * gen._WEYL + key) & gen._M32) for i in idx]
    assert h.tolist() == ref
    # published fmix32 fixed point: fmix32(0) == 0
    assert gen.fmix32_py(0) == 0


def test_codes_in_range_and_uniform():
    spec = synth.workload("single768").mats[0]
    inp = gen.matrix_inputs(spec, 1)
    codes = gen.codes_torch(inp["widths"], inp["key"], spec.k).numpy()
    wide = np.repeat(inp["widths"].astype(np.int64), 64, axis=1)
    assert (codes.astype(np.int64) < (1 << wide)).all()
    one = codes[wide == 1]
    assert abs(one.mean() - 0.5) < 0.01
    eight = codes[wide == 8]
    assert abs(eight.mean() - 127.5) < 3
    # a row subset reproduces the same rows
    sub = gen.codes_torch(inp["widths"], inp["key"], spec.k, row0=100, nrows=7).numpy()
    assert np.array_equal(sub, codes[100:107])


def test_recipe_stacks():
    """The fixed recipe (§3.4): layer-0 MLP all 4-bit, every other projection
    all 2-bit, the head tiered per row 8/4/2/1 bits over the top 0.5% / next
    1.5% / next 10% / last 88% of rows (mean 1.18 bits)."""
    for name, vocab in (("stack9b-recipe", 128256), ("stack131m-recipe", 32000)):
        work = synth.workload(name)
        plain = synth.workload(name[:-7])
        assert [(m.n, m.k) for m in work.mats] == [(m.n, m.k) for m in plain.mats]
        for spec in work.mats[:-1]:
            w = gen.matrix_inputs(spec, 1)["widths"]
            mlp0 = spec.name.split(".")[0] == "l0" and spec.name.split(".")[1] in ("gate", "up", "down")
            assert (w == (4 if mlp0 else 2)).all(), spec.name
        head = work.mats[-1]
        w = gen.matrix_inputs(head, 1)["widths"]
        assert head.n == vocab and (w == w[:, :1]).all()          # one width per row
        rows = w[:, 0]
        b8, b4, b2 = round(0.005 * vocab), round(0.02 * vocab), round(0.12 * vocab)
        assert (rows[:b8] == 8).all() and (rows[b8:b4] == 4).all() and (rows[b4:b2] == 2).all()
        assert (rows[b2:] == 1).all()
        assert abs(rows.astype(float).mean() - 1.18) < 0.005
    assert gen.tiered_widths(3, 2, ((0.5, 8), (1.0, 1))).tolist() == [[8, 8], [8, 8], [1, 1]]


def test_generators_deterministic():
    spec = synth.workload("stack131m").mats[3]
    a = gen.matrix_inputs(spec, 2)
    b = gen.matrix_inputs(spec, 2)
    for k in ("widths", "scales", "x_bits"):
        assert np.array_equal(a[k], b[k])
    assert a["key"] == b["key"]
    c = gen.matrix_inputs(spec, 1)
    assert np.array_equal(c["x_bits"][0], a["x_bits"][0])


def test_bf16_rounding_matches_torch():
    rng = np.random.default_rng(0)
    v = rng.normal(0, 1, size=10000).astype(np.float32)
    v[:4] = [1.0 + 2**-8, 1.0 + 3 * 2**-8, -0.0, 3.0e38]      # ties and edges
    bits = gen.f32_to_bf16_bits(v)
    ref = torch.from_numpy(v).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(bits, ref)
    assert np.array_equal(gen.bf16_bits_to_f32(bits), torch.from_numpy(v).to(torch.bfloat16).float().numpy())


def test_scales_fp16_positive():
    rng = gen.rng_for((0, 0, 0))
    s = gen.draw_scales(100, 10, rng)
    assert s.dtype == np.float16 and (s > 0).all()


def test_gate_up_vector():
    # the down projection's synthetic input: 2k float32, pairs (gate, up), one
    # feature in eight zero-padded (both exactly 0), the rest N(0, 1.5)
    a = gen.draw_gate_up(8192, gen.rng_for((89, 8192, 0)))
    b = gen.draw_gate_up(8192, gen.rng_for((89, 8192, 0)))
    assert a.dtype == np.float32 and a.shape == (16384,) and np.array_equal(a, b)
    pairs = a.reshape(-1, 2)
    padded = (pairs == 0).all(axis=1)
    assert abs(padded.mean() - 0.125) < 0.02
    live = pairs[~padded]
    assert abs(live.std() - 1.5) < 0.05 and abs(live.mean()) < 0.05


def test_soft_inputs():
    # weights, logits N(0, 2) and standard Gumbel noise (mean = the
    # Euler-Mascheroni constant, variance pi^2 / 6), all float32, seeded
    w, lg, gb = gen.draw_soft_inputs(64, 4096, gen.rng_for((70, 64, 4096)))
    w2, lg2, gb2 = gen.draw_soft_inputs(64, 4096, gen.rng_for((70, 64, 4096)))
    assert np.array_equal(w, w2) and np.array_equal(lg, lg2) and np.array_equal(gb, gb2)
    assert w.shape == (64, 4096) and lg.shape == gb.shape == (64, 64, 4)
    assert w.dtype == lg.dtype == gb.dtype == np.float32
    assert abs(lg.std() - 2.0) < 0.05
    assert abs(gb.mean() - 0.5772156649) < 0.02 and abs(gb.var() - np.pi ** 2 / 6) < 0.06
