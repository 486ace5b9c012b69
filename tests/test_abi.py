"""The C-ABI library: it loads, exports every symbol the header declares, and
rejects bad arguments on the host before touching the GPU. CPU only."""

import ctypes
import os
import re

import pytest

import paper_2607_02893_gb300 as vbq
from paper_2607_02893_gb300 import vbq as binding

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "vbq.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2607_02893_gb300 import build
    build.build()
    return vbq.load()


def header_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(vbq_[a-z_]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = header_functions()
    for required in ("vbq_pack", "vbq_dequant", "vbq_gemv", "vbq_gemm_small", "vbq_free"):
        assert required in names


def test_library_exports_every_declared_symbol(lib):
    names = header_functions()
    missing = [n for n in names if not hasattr(lib, n)]
    assert not missing, f"missing exports: {missing}"
    assert set(names) == set(binding.SIGNATURES), "binding and header disagree"


def test_status_strings(lib):
    assert vbq.vbq_status_string(0) == "VBQ_OK"
    for code, name in binding.STATUS_NAMES.items():
        assert vbq.vbq_status_string(code) == name
    assert vbq.vbq_status_string(-1234) == "VBQ_ERR_UNKNOWN"


def _pack_raw(lib, codes, widths, scales, n, k, on_dev):
    out = ctypes.c_void_p(12345)
    st = lib.vbq_pack(codes, widths, scales, n, k, on_dev, None, ctypes.byref(out))
    return st, out.value


def test_pack_rejects_bad_arguments_on_host(lib):
    buf = ctypes.create_string_buffer(64)
    p = ctypes.addressof(buf)
    assert lib.vbq_pack(p, p, p, 1, 64, 0, None, None) == -1          # out NULL
    st, out = _pack_raw(lib, None, p, p, 1, 64, 0)
    assert st == -1 and out is None                                      # codes NULL, out cleared
    assert _pack_raw(lib, p, p, p, 1, 64, 2)[0] == -1                   # bad flag
    assert _pack_raw(lib, p, p, p, 0, 64, 0)[0] == -2                   # N < 1
    assert _pack_raw(lib, p, p, p, 4, 65, 0)[0] == -2                   # K % 64
    assert _pack_raw(lib, p, p, p, 4, 0, 0)[0] == -2
    assert _pack_raw(lib, p + 1, p, p, 4, 64, 1)[0] == -5               # misaligned device ptr
    assert b"16-byte" in lib.vbq_last_error()


def test_quantize_rejects_bad_arguments_on_host(lib):
    buf = ctypes.create_string_buffer(256)
    p = (ctypes.addressof(buf) + 15) // 16 * 16
    assert lib.vbq_quantize(None, p, 1, 64, p, p, None) == -1            # w NULL
    assert lib.vbq_quantize(p, p, 1, 64, p, None, None) == -1            # scales NULL
    assert lib.vbq_quantize(p, p, 0, 64, p, p, None) == -2               # N < 1
    assert lib.vbq_quantize(p, p, 2, 96, p, p, None) == -2               # K % 64
    assert lib.vbq_quantize(p, p, 1 << 30, 1 << 20, p, p, None) == -7    # over 2^40 weights
    assert lib.vbq_quantize(p + 4, p, 1, 64, p, p, None) == -5           # misaligned
    assert lib.vbq_quantize(p, p, 1, 64, p + 2, p, None) == -5
    assert b"16-byte" in lib.vbq_last_error()


def test_calls_reject_null_layout(lib):
    assert lib.vbq_gemv(None, None, None, None) == -1
    assert lib.vbq_gemm_small(None, None, None, 4, None) == -1
    assert lib.vbq_gemv_swiglu(None, None, None, None, None) == -1
    assert lib.vbq_gemv_swiglu_in(None, None, None, None) == -1
    assert lib.vbq_chain_run(None, None) == -1
    assert lib.vbq_chain_free(None) == 0


def test_soft_quant_rejects_bad_arguments_on_host(lib):
    buf = ctypes.create_string_buffer(256)
    p = (ctypes.addressof(buf) + 15) // 16 * 16
    assert lib.vbq_soft_quant(None, p, None, 1.0, 1, 64, p, None, None, None) == -1      # w NULL
    assert lib.vbq_soft_quant(p, p, None, 1.0, 1, 64, None, None, None, None) == -1      # w_soft NULL
    for tau in (0.0, -2.0, float("inf"), float("nan")):
        assert lib.vbq_soft_quant(p, p, None, tau, 1, 64, p, None, None, None) == -1
    assert b"tau" in lib.vbq_last_error()
    assert lib.vbq_soft_quant(p, p, None, 1.0, 1, 96, p, None, None, None) == -2         # K % 64
    assert lib.vbq_soft_quant(p, p, None, 1.0, 0, 64, p, None, None, None) == -2         # N < 1
    assert lib.vbq_soft_quant(p, p, p + 4, 1.0, 1, 64, p, None, None, None) == -5        # misaligned noise
    assert lib.vbq_soft_quant(p, p, None, 1.0, 1, 64, p, None, p + 1, None) == -5        # misaligned widths


def test_chain_rejects_bad_arguments_on_host(lib):
    P = ctypes.c_void_p
    arr = (P * 2)()
    out = P(7)
    assert lib.vbq_chain_create(arr, arr, arr, None, 2, None) == -1         # out NULL
    assert lib.vbq_chain_create(None, arr, arr, None, 2, ctypes.byref(out)) == -1
    assert out.value is None                                               # cleared on error
    assert lib.vbq_chain_create(arr, arr, arr, None, 0, ctypes.byref(out)) == -1   # empty chain
    assert lib.vbq_chain_create(arr, arr, arr, None, -3, ctypes.byref(out)) == -1
    assert b"count" in lib.vbq_last_error()
    assert lib.vbq_dequant(None, None, None, None, None, None) == -1
    assert lib.vbq_packed_bytes(None, None, None, None) == -1
    assert lib.vbq_layout_shape(None, None, None) == -1
    assert lib.vbq_free(None) == 0


def test_group_rejects_bad_arguments_on_host(lib):
    P = ctypes.c_void_p
    arr = (P * 2)()
    assert lib.vbq_gemv_group(None, None, None, 0, None) == 0           # empty group: nothing to do
    assert lib.vbq_gemv_group(arr, arr, arr, -1, None) == -1             # negative count
    assert lib.vbq_gemv_group(None, arr, arr, 2, None) == -1             # NULL arrays
    assert lib.vbq_gemv_group(arr, arr, arr, 2, None) == -1              # NULL layout entries
    assert b"layout 0 is NULL" in lib.vbq_last_error()
    with pytest.raises(ValueError):
        vbq.vbq_gemv_group([None], [], [])


def test_binding_raises_typed_errors(lib):
    with pytest.raises(vbq.VbqError) as ei:
        vbq.vbq_pack(0, 0, 0, N=4, K=64, src_on_device=0)
    assert ei.value.name == "VBQ_ERR_ARG"


def test_missing_library_fails_loudly(tmp_path):
    with pytest.raises(RuntimeError, match="not built"):
        binding.load(str(tmp_path / "libvbq.so"))


def test_selftest_timeout_rejects_bad_limits():
    import paper_2607_02893_gb300 as vbq
    vbq.load()
    for bad in (0, -5, 1000001):
        with pytest.raises(vbq.VbqError) as e:
            vbq.vbq_selftest_timeout(bad, stream=0)
        assert e.value.name == "VBQ_ERR_ARG"
