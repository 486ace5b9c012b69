"""Python binding of the VBQ C ABI (include/vbq.h).

Argument marshalling only: every step of packing, unpacking and the products
runs in libvbq.so. Functions take torch tensors (or raw integer addresses)
and keep the C names. PyTorch is used only to own device memory and streams.
"""

from __future__ import annotations

import ctypes
import os
from typing import Optional, Tuple

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libvbq.so")

VBQ_OK = 0
STATUS_NAMES = {
    0: "VBQ_OK", -1: "VBQ_ERR_ARG", -2: "VBQ_ERR_SHAPE", -3: "VBQ_ERR_WIDTH",
    -4: "VBQ_ERR_CODE_RANGE", -5: "VBQ_ERR_ALIGN", -6: "VBQ_ERR_CUDA",
    -7: "VBQ_ERR_UNSUPPORTED", -8: "VBQ_ERR_TIMEOUT", -9: "VBQ_ERR_NOMEM",
}

# Every symbol include/vbq.h declares, with (restype, argtypes).
_P = ctypes.c_void_p
_I64 = ctypes.c_int64
_I = ctypes.c_int
_SZP = ctypes.POINTER(ctypes.c_size_t)
_I64P = ctypes.POINTER(ctypes.c_int64)
SIGNATURES = {
    "vbq_quantize": (_I, [_P, _P, _I64, _I64, _P, _P, _P]),
    "vbq_soft_quant": (_I, [_P, _P, _P, ctypes.c_float, _I64, _I64, _P, _P, _P, _P]),
    "vbq_pack": (_I, [_P, _P, _P, _I64, _I64, _I, _P, ctypes.POINTER(_P)]),
    "vbq_packed_bytes": (_I, [_P, _SZP, _SZP, _SZP]),
    "vbq_layout_shape": (_I, [_P, _I64P, _I64P]),
    "vbq_dequant": (_I, [_P, _P, _P, _P, _P, _P]),
    "vbq_gemv": (_I, [_P, _P, _P, _P]),
    "vbq_gemm_small": (_I, [_P, _P, _P, _I, _P]),
    "vbq_gemv_static": (_I, [_P, _P, _P, _P]),
    "vbq_gemv_swiglu": (_I, [_P, _P, _P, _P, _P]),
    "vbq_gemv_swiglu_in": (_I, [_P, _P, _P, _P]),
    "vbq_chain_create": (_I, [ctypes.POINTER(_P), ctypes.POINTER(_P), ctypes.POINTER(_P),
                              ctypes.POINTER(_I), _I, ctypes.POINTER(_P)]),
    "vbq_chain_run": (_I, [_P, _P]),
    "vbq_chain_free": (_I, [_P]),
    "vbq_gemv_group": (_I, [ctypes.POINTER(_P), ctypes.POINTER(_P), ctypes.POINTER(_P), _I, _P]),
    "vbq_device_status": (_I, [_P]),
    "vbq_selftest_timeout": (_I, [_I, _P]),
    "vbq_free": (_I, [_P]),
    "vbq_status_string": (ctypes.c_char_p, [_I]),
    "vbq_last_error": (ctypes.c_char_p, []),
}

_lib = None


class VbqError(RuntimeError):
    def __init__(self, status: int, detail: str):
        self.status = status
        self.name = STATUS_NAMES.get(status, str(status))
        super().__init__(f"{self.name}: {detail}")


def load(path: Optional[str] = None) -> ctypes.CDLL:
    """Load libvbq.so (built by paper_2607_02893_gb300.build). Fails loudly if absent."""
    global _lib
    if _lib is not None and path is None:
        return _lib
    p = path or LIB_PATH
    if not os.path.exists(p):
        raise RuntimeError(f"VBQ CUDA library not built: {p} is missing "
                           "(run `python -c 'import __graft_entry__ as g; g.build()'`)")
    lib = ctypes.CDLL(p)
    for name, (res, args) in SIGNATURES.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    if path is None:
        _lib = lib
    return lib


def _check(st: int):
    if st != VBQ_OK:
        detail = load().vbq_last_error().decode(errors="replace")
        raise VbqError(st, detail)


def _ptr(t) -> Optional[int]:
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(stream, *tensors) -> Optional[int]:
    if stream is None:
        import torch
        if any(getattr(t, "is_cuda", False) for t in tensors if t is not None):
            return torch.cuda.current_stream().cuda_stream or None
        return None
    if isinstance(stream, int):
        return stream or None
    return stream.cuda_stream or None


class Layout:
    """Owns one packed matrix (a vbq_layout*)."""

    def __init__(self, handle: int, n: int, k: int):
        self.handle = handle
        self.N = n
        self.K = k

    def __del__(self):
        try:
            self.free()
        except Exception:
            pass

    def free(self):
        if self.handle:
            h, self.handle = self.handle, None
            _check(load().vbq_free(h))

    @property
    def _as_parameter_(self):
        if not self.handle:
            raise ValueError("layout already freed")
        return ctypes.c_void_p(self.handle)


def vbq_quantize(w, bitwidths, codes_out=None, scales_out=None, stream=None):
    """Quantise w (N x K float32, device) at per-group widths (N x K/64 uint8,
    device) into codes (N x K uint8) and FP16 scale bit patterns (N x K/64,
    int16 storage); returns (codes, scales). Outputs are allocated when not given."""
    import torch
    n, k = int(w.shape[0]), int(w.shape[1])
    if codes_out is None:
        codes_out = torch.empty((n, k), dtype=torch.uint8, device=w.device)
    if scales_out is None:
        scales_out = torch.empty((n, k // 64), dtype=torch.int16, device=w.device)
    _check(load().vbq_quantize(_ptr(w), _ptr(bitwidths), n, k, _ptr(codes_out), _ptr(scales_out),
                               _stream(stream, w)))
    return codes_out, scales_out


def vbq_soft_quant(w, logits, tau: float, gumbel=None, w_soft=None, exp_bits=None, hard_widths=None,
                   stream=None):
    """Soft-quantised forward of w (N x K float32, device) under per-group
    logits (N x K/64 x 4 float32) and optional Gumbel noise of the same shape;
    returns (w_soft, exp_bits, hard_widths), allocating those not given (pass
    exp_bits=False / hard_widths=False to skip one)."""
    import torch
    n, k = int(w.shape[0]), int(w.shape[1])
    if w_soft is None:
        w_soft = torch.empty((n, k), dtype=torch.float32, device=w.device)
    if exp_bits is None:
        exp_bits = torch.empty((n, k // 64), dtype=torch.float32, device=w.device)
    if hard_widths is None:
        hard_widths = torch.empty((n, k // 64), dtype=torch.uint8, device=w.device)
    eb = None if exp_bits is False else exp_bits
    hw = None if hard_widths is False else hard_widths
    _check(load().vbq_soft_quant(_ptr(w), _ptr(logits), _ptr(gumbel), float(tau), n, k, _ptr(w_soft),
                                 _ptr(eb), _ptr(hw), _stream(stream, w)))
    return w_soft, eb, hw


def vbq_pack(codes, bitwidths, scales_fp16, N: Optional[int] = None, K: Optional[int] = None,
             src_on_device: Optional[int] = None, stream=None) -> Layout:
    """Pack codes (N x K uint8), bitwidths (N x K/64 uint8) and scales
    (N x K/64 float16 or int16/uint16 bit patterns) into a device layout."""
    if N is None:
        N, K = int(codes.shape[0]), int(codes.shape[1])
    if src_on_device is None:
        src_on_device = 1 if getattr(codes, "is_cuda", False) else 0
    out = ctypes.c_void_p()
    _check(load().vbq_pack(_ptr(codes), _ptr(bitwidths), _ptr(scales_fp16), int(N), int(K),
                           int(src_on_device), _stream(stream, codes), ctypes.byref(out)))
    return Layout(out.value, int(N), int(K))


def vbq_packed_bytes(layout: Layout) -> Tuple[int, int, int]:
    p, s, m = ctypes.c_size_t(), ctypes.c_size_t(), ctypes.c_size_t()
    _check(load().vbq_packed_bytes(layout, ctypes.byref(p), ctypes.byref(s), ctypes.byref(m)))
    return p.value, s.value, m.value


def vbq_layout_shape(layout: Layout) -> Tuple[int, int]:
    n, k = ctypes.c_int64(), ctypes.c_int64()
    _check(load().vbq_layout_shape(layout, ctypes.byref(n), ctypes.byref(k)))
    return n.value, k.value


def vbq_dequant(layout: Layout, codes_out=None, bitwidths_out=None, scales_out=None, w_out=None,
                stream=None) -> None:
    _check(load().vbq_dequant(layout, _ptr(codes_out), _ptr(bitwidths_out), _ptr(scales_out),
                              _ptr(w_out), _stream(stream, codes_out, w_out, bitwidths_out, scales_out)))


def vbq_gemv(layout: Layout, x, y, stream=None) -> None:
    _check(load().vbq_gemv(layout, _ptr(x), _ptr(y), _stream(stream, x, y)))


def vbq_gemv_swiglu(layout: Layout, x, y, h, stream=None) -> None:
    """Gate-up product with the SwiGLU epilogue: y = W x (N floats, rows
    alternating gate / up) and h = silu(y[0::2]) * y[1::2] as N/2 BF16 bit
    patterns (int16 or bfloat16 storage)."""
    _check(load().vbq_gemv_swiglu(layout, _ptr(x), _ptr(y), _ptr(h), _stream(stream, x, y, h)))


def vbq_gemv_swiglu_in(layout: Layout, gu, y, stream=None) -> None:
    """Down projection of a SwiGLU MLP: y = W h with h_k = silu(gu[2k]) *
    gu[2k + 1] computed in the kernel (gu: 2K float32, the y of a gate-up
    product with alternating rows)."""
    _check(load().vbq_gemv_swiglu_in(layout, _ptr(gu), _ptr(y), _stream(stream, gu, y)))


def vbq_gemv_static(layout: Layout, x, y, stream=None) -> None:
    """vbq_gemv that allocates nothing: its split-K control words live in a
    fixed array inside the library (see include/vbq.h)."""
    _check(load().vbq_gemv_static(layout, _ptr(x), _ptr(y), _stream(stream, x, y)))


def vbq_gemv_group(layouts, xs, ys, stream=None) -> None:
    """Independent batch-1 products y_i = W_i x_i whose launches overlap
    (distinct layouts and outputs; no x_i written inside the group)."""
    n = len(layouts)
    if len(xs) != n or len(ys) != n:
        raise ValueError("layouts, xs and ys must have the same length")
    arr = _P * max(n, 1)
    la = arr(*[lay._as_parameter_ for lay in layouts])
    xa = arr(*[_ptr(x) for x in xs])
    ya = arr(*[_ptr(y) for y in ys])
    _check(load().vbq_gemv_group(la, xa, ya, int(n), _stream(stream, *(list(xs) + list(ys)))))


class Chain:
    """Owns one vbq_chain*: products run in order by one persistent launch.
    Keeps references to its layouts and buffers so they outlive it."""

    def __init__(self, layouts, xs, ys, waits=None):
        n = len(layouts)
        if len(xs) != n or len(ys) != n or (waits is not None and len(waits) != n):
            raise ValueError("layouts, xs, ys (and waits) must have the same length")
        arr = _P * max(n, 1)
        la = arr(*[lay._as_parameter_ for lay in layouts])
        xa = arr(*[_ptr(x) for x in xs])
        ya = arr(*[_ptr(y) for y in ys])
        wa = None if waits is None else (_I * n)(*[int(w) for w in waits])
        out = ctypes.c_void_p()
        self.handle = None
        _check(load().vbq_chain_create(la, xa, ya, wa, int(n), ctypes.byref(out)))
        self.handle = out.value
        self._keep = (list(layouts), list(xs), list(ys))

    def run(self, stream=None) -> None:
        if not self.handle:
            raise ValueError("chain already freed")
        _check(load().vbq_chain_run(self.handle, _stream(stream, *self._keep[2])))

    def free(self) -> None:
        if self.handle:
            h, self.handle = self.handle, None
            _check(load().vbq_chain_free(h))

    def __del__(self):
        try:
            self.free()
        except Exception:
            pass


def vbq_chain_create(layouts, xs, ys, waits=None) -> Chain:
    return Chain(layouts, xs, ys, waits)


def vbq_chain_run(chain: Chain, stream=None) -> None:
    chain.run(stream)


def vbq_chain_free(chain: Chain) -> None:
    chain.free()


def vbq_gemm_small(layout: Layout, X, Y, B: Optional[int] = None, stream=None) -> None:
    if B is None:
        B = int(X.shape[0])
    _check(load().vbq_gemm_small(layout, _ptr(X), _ptr(Y), int(B), _stream(stream, X, Y)))


def vbq_device_status(stream=None) -> None:
    """Synchronise the stream; raise VbqError(VBQ_ERR_TIMEOUT) if a bounded
    device wait gave up since the last call (the record is cleared)."""
    _check(load().vbq_device_status(_stream(stream)))


def vbq_selftest_timeout(limit_us: int, stream=None) -> None:
    """Launch the one-block kernel whose wait runs out after limit_us."""
    _check(load().vbq_selftest_timeout(int(limit_us), _stream(stream)))


def vbq_free(layout: Layout) -> None:
    layout.free()


def vbq_status_string(status: int) -> str:
    return load().vbq_status_string(int(status)).decode()
