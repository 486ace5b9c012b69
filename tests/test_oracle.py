"""The CPU oracle against its pins, and the pins against planted mistakes.

Runs on CPU only (no GPU marker)."""

import importlib.util
import os
import types

import numpy as np
import pytest

import oracle
from oracle import vbq_oracle
import oracle_pins as P

ORACLE_SRC = vbq_oracle.__file__


@pytest.mark.parametrize("pin", P.ALL_PINS, ids=lambda f: f.__name__)
def test_oracle_pin(pin):
    pin(vbq_oracle)


def _mutant(old: str, new: str) -> types.ModuleType:
    """A copy of the oracle module with one source fragment replaced."""
    src = open(ORACLE_SRC).read()
    assert src.count(old) == 1, f"mutation anchor not unique/absent: {old!r}"
    src = src.replace(old, new)
    mod = types.ModuleType("vbq_oracle_mutant")
    mod.__file__ = ORACLE_SRC
    exec(compile(src, "vbq_oracle_mutant", "exec"), mod.__dict__)
    return mod


MUTATIONS = {
    "zero_point_sign": ("return u - (1 << (b - 1))", "return (1 << (b - 1)) - u"),
    "zero_point_off_by_one": ("return u - (1 << (b - 1))", "return u - (1 << (b - 1)) + 1"),
    "zero_point_symmetric": ("return u - (1 << (b - 1))", "return u - ((1 << (b - 1)) - 1)"),
    "one_bit_polarity": ("return 2 * u - 1", "return 1 - 2 * u"),
    "one_bit_zero_one": ("return 2 * u - 1", "return u"),
    "dropped_scale": ("w[:, cols] = s[:, None] * lv.astype(np.float64)",
                      "w[:, cols] = lv.astype(np.float64)"),
    "wrong_group_scale": ("s = scales[:, g].astype(np.float64)",
                          "s = scales[:, (g + 1) % scales.shape[1]].astype(np.float64)"),
    "reversed_x": ("prod = w * x[bi][None, :]", "prod = w * x[bi][::-1][None, :]"),
    "bound_not_abs": ("a[bi] = np.abs(prod).sum(axis=1)", "a[bi] = prod.sum(axis=1)"),
    "round_half_away": ("q = np.clip(np.round(w / sf), -qmax, qmax)",
                        "q = np.clip(np.floor(w / sf + 0.5), -qmax, qmax)"),
    "unrounded_scale_for_codes": ("sf = float(s_used)", "sf = float(s)"),
    "qmax_too_large": ("qmax = (1 << (b - 1)) - 1\n    z = 1 << (b - 1)\n    m =",
                       "qmax = (1 << (b - 1))\n    z = 1 << (b - 1)\n    m ="),
    "one_bit_max_scale": ("s = pairwise_sum(np.abs(w)) / w.size", "s = float(np.max(np.abs(w))) / 1.0"),
    "one_bit_sequential_sum": ("s = pairwise_sum(np.abs(w)) / w.size",
                               "s = float(np.cumsum(np.abs(w))[-1]) / w.size"),
    "sign_zero_negative": ("codes = (w >= 0).astype(np.uint8)", "codes = (w > 0).astype(np.uint8)"),
    "pack_msb_first": ("acc |= int(codes[r, g * GROUP + i]) << (i * b)",
                       "acc |= int(codes[r, g * GROUP + i]) << ((GROUP - 1 - i) * b)"),
    "swiglu_swapped": ("return silu(y[:, 0::2]) * y[:, 1::2]", "return silu(y[:, 1::2]) * y[:, 0::2]"),
    "silu_sign": ("return z / (1.0 + np.exp(-z))", "return z / (1.0 + np.exp(z))"),
    "scale_bytes_one": ("return 2 * int(np.asarray(widths).size)",
                        "return int(np.asarray(widths).size)"),
    "soft_tau_ignored": ("    z = z / tau\n    z = z - z.max(axis=-1, keepdims=True)",
                         "    z = z - z.max(axis=-1, keepdims=True)"),
    "soft_noise_subtracted": ("        z = z + np.asarray(gumbel, dtype=np.float64)\n    z = z / tau\n    z = z - z.max(",
                              "        z = z - np.asarray(gumbel, dtype=np.float64)\n    z = z / tau\n    z = z - z.max("),
    "soft_candidates_reversed": ("CANDIDATES = (1, 2, 4, 8)", "CANDIDATES = (8, 4, 2, 1)"),
    "soft_not_normalised": ("    return p / p.sum(axis=-1, keepdims=True)", "    return p"),
    "soft_round_half_away": ("q = np.clip(np.rint(t), -qmax, qmax)", "q = np.clip(np.floor(t + 0.5), -qmax, qmax)"),
    "soft_one_bit_max": ("        mean = pairwise_sum(np.abs(w32.astype(np.float64))) / w32.size",
                         "        mean = float(np.max(np.abs(w32)))"),
    "soft_qmax_too_large": ("    qmax = np.float32((1 << (b - 1)) - 1)", "    qmax = np.float32(1 << (b - 1))"),
    "soft_hard_last_max": ("[np.argmax(logits, axis=-1)]",
                           "[3 - np.argmax(logits[..., ::-1], axis=-1)]"),
    "soft_bound_eps_loosened": ("    eps = 2.0 ** -20 * (1.0 + np.abs(z).max(axis=-1)) + 2.0 ** -20",
                                "    eps = 100.0 * (2.0 ** -20 * (1.0 + np.abs(z).max(axis=-1)) + 2.0 ** -20)"),
    "soft_bound_no_noise": ("        z = z + np.asarray(gumbel, dtype=np.float64)\n    z = z / tau\n    eps =",
                            "        z = z\n    z = z / tau\n    eps ="),
    "soft_expected_bits_unweighted": ("    exp_bits = (pi * cand).sum(axis=-1)", "    exp_bits = pi.sum(axis=-1) * cand.mean()"),
}


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_pins_catch_planted_mistake(name):
    old, new = MUTATIONS[name]
    mod = _mutant(old, new)
    failures = []
    for pin in P.ALL_PINS:
        try:
            pin(mod)
        except (P.PinFailed, AssertionError, ValueError, IndexError, OverflowError):
            failures.append(pin.__name__)
    assert failures, f"no pin caught the planted mistake {name!r}"


def test_oracle_rejects_bad_inputs():
    codes = np.zeros((2, 64), np.uint8)
    widths = np.ones((2, 1), np.uint8)
    scales = np.ones((2, 1), np.float16)
    with pytest.raises(ValueError):
        oracle.dequant(np.zeros((2, 65), np.uint8), widths, scales)
    with pytest.raises(ValueError):
        oracle.dequant(codes, np.full((2, 1), 3, np.uint8), scales)
    bad = codes.copy()
    bad[0, 5] = 2          # code 2 at 1 bit
    with pytest.raises(ValueError):
        oracle.dequant(bad, widths, scales)


def test_within_bound():
    y_ref = np.array([1.0, 0.0])
    a_ref = np.array([10.0, 0.0])
    assert oracle.within_bound(np.array([1.0 + 0.019, 9e-6]), y_ref, a_ref).all()
    assert not oracle.within_bound(np.array([1.0 + 0.0201, 0.0]), y_ref, a_ref)[0]
    assert not oracle.within_bound(np.array([1.0, 1.1e-5]), y_ref, a_ref)[1]
