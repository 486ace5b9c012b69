"""Seeded synthetic inputs for VBQ packed GEMV workloads.

This package draws the inputs that both the CUDA path and the CPU oracle
consume: per-group bit-widths, integer codes, FP16 scales and BF16
activations. It holds none of the method's arithmetic (no level map, no
dequantisation, no dot products); it only describes workloads and draws
random numbers for them.
"""

from .workloads import (  # noqa: F401
    DIST_MAIN, DIST_MLP0, DIST_HEAD, DIST_ALL1, DIST_ALL2, DIST_ALL4, DIST_ALL8,
    SWEEP_DISTS, MatrixSpec, Workload, workload, workload_names, sweep_points,
)
from .gen import (  # noqa: F401
    draw_widths, draw_scales, draw_x_bf16, bf16_bits_to_f32, f32_to_bf16_bits,
    code_key, codes_torch, matrix_inputs, fmix32_py, tiered_widths, spec_widths,
)
