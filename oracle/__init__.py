"""CPU oracle for VBQ (test infrastructure only).

Only tests/, __graft_entry__.smoke() and bench.py's CPU baseline leg may
import this package. The CUDA library and its Python binding never do.
"""

from .vbq_oracle import (  # noqa: F401
    GROUP, WIDTHS, level, check_inputs, dequant, gemv, within_bound,
    silu, swiglu, swiglu_error_bound, swiglu_within_bound, SILU_SLOPE_MAX,
    quantize_group, quantize, payload_bytes, scale_bytes, pack_lsb, unpack_lsb,
    CANDIDATES, reconstruct_fp32, soft_select, soft_quant_forward, soft_quant_within_bound,
)
