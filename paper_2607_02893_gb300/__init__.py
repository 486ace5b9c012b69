"""VBQ packed variable-bit-width GEMV for GB300 (sm_103a).

The compute lives in libvbq.so (CUDA kernels behind the C ABI of
include/vbq.h); this package is its thin Python binding.
"""

from .vbq import (  # noqa: F401
    Layout, VbqError, load, vbq_quantize, vbq_soft_quant, vbq_pack, vbq_packed_bytes, vbq_layout_shape, vbq_dequant,
    vbq_gemv, vbq_gemv_static, vbq_gemv_swiglu, vbq_gemv_swiglu_in, vbq_gemv_group, vbq_gemm_small, vbq_device_status, vbq_selftest_timeout, vbq_free,
    vbq_status_string, SIGNATURES, LIB_PATH, Chain, vbq_chain_create, vbq_chain_run, vbq_chain_free,
)
