"""Shared helpers for the GPU tests: seeded matrices on the device and the
oracle's view of the same inputs."""

from __future__ import annotations

import numpy as np
import torch

import synth
from synth import gen


def scales_to_i16(scales_f16: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(scales_f16).view(np.uint16).astype(np.int16))


def bits_to_i16(bits_u16: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(bits_u16).astype(np.uint16).view(np.int16))


class Matrix:
    """One seeded VBQ matrix: numpy widths/scales, codes (torch), x bits (numpy)."""

    def __init__(self, n, k, dist=synth.DIST_MAIN, seed_path=(99, 0, 0), batch=1,
                 codes_device="cpu"):
        self.n, self.k = n, k
        spec = synth.MatrixSpec("t", n, k, dist, tuple(seed_path))
        inp = gen.matrix_inputs(spec, batch)
        self.widths = inp["widths"]
        self.scales = inp["scales"]
        self.x_bits = inp["x_bits"]
        self.key = inp["key"]
        self.codes = gen.codes_torch(self.widths, self.key, k, device=codes_device)

    @classmethod
    def from_spec(cls, spec, batch=1, codes_device="cuda"):
        m = cls.__new__(cls)
        m.n, m.k = spec.n, spec.k
        inp = gen.matrix_inputs(spec, batch)
        m.widths, m.scales, m.x_bits, m.key = inp["widths"], inp["scales"], inp["x_bits"], inp["key"]
        m.codes = gen.codes_torch(torch.from_numpy(m.widths).to(codes_device), m.key, spec.k,
                                  device=codes_device)
        return m

    def rows_codes_cpu(self, rows):
        out = np.empty((len(rows), self.k), dtype=np.uint8)
        for i, r in enumerate(rows):
            out[i] = gen.codes_torch(self.widths, self.key, self.k, row0=int(r), nrows=1,
                                     device="cpu").numpy()[0]
        return out

    def x(self) -> np.ndarray:
        return gen.bf16_bits_to_f32(self.x_bits)

    def device_args(self, dev="cuda"):
        return (self.codes.to(dev), torch.from_numpy(self.widths).to(dev),
                scales_to_i16(self.scales).to(dev))
