"""vbq_gemv_static: the batch-1 product for callers that cannot allocate
device memory when they run a product (a serving loop inside a fixed memory
budget, or a host framework whose allocator must own every device byte). Its
split-K control words live in a fixed array inside the library instead of in
the layout. Every call goes through the C ABI and is checked against the CPU
oracle with the library's accuracy bound: two calls in a row per shape, and a
sequence over two layouts whose row blocks overlap, so that the flags one
layout leaves in the shared array sit at the row blocks the other one uses.

This file is collected last on purpose: a run that stops at the first failure
has then already run every other test."""

import numpy as np
import pytest
import torch

import oracle
import paper_2607_02893_gb300 as vbq
from vbq_cases import Matrix, bits_to_i16

pytestmark = pytest.mark.gpu

DEV = "cuda"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2607_02893_gb300 import build
    build.build()
    vbq.load()
    torch.cuda.init()


def _reference(m: Matrix):
    y_ref, a_ref = oracle.gemv(m.codes.cpu().numpy(), m.widths, m.scales, m.x()[:1])
    return y_ref[0], a_ref[0]


def _static(layout, m: Matrix):
    x = bits_to_i16(m.x_bits[:1]).to(DEV)
    y = torch.full((m.n,), float("nan"), dtype=torch.float32, device=DEV)
    vbq.vbq_gemv_static(layout, x[0], y)
    torch.cuda.synchronize()
    return y.cpu().numpy()


def _assert_bound(y, ref, what):
    ok = oracle.within_bound(y, *ref)
    assert ok.all(), f"{what}: {int((~ok).sum())} of {ok.size} outputs outside the bound"


@pytest.mark.parametrize("shape", [(4096, 4096), (1000, 768), (300, 64 * 70), (129, 64)],
                         ids=lambda s: f"{s[0]}x{s[1]}")
def test_static_scratch_matches_oracle(shape):
    n, k = shape
    m = Matrix(n, k, seed_path=(88, n, k))
    layout = vbq.vbq_pack(*m.device_args(DEV))
    ref = _reference(m)
    for call in range(2):                    # two calls in a row share the fixed array
        _assert_bound(_static(layout, m), ref, f"{n}x{k} call {call}")
    layout.free()


def test_static_scratch_across_layouts():
    # A has more row blocks than B; both split K over several slabs, so every
    # call zeroes its rows and publishes flags in the shared array at the row
    # blocks B and A have in common. A, B, A, then the allocating product on
    # B, then B again.
    a = Matrix(2048, 64 * 70, seed_path=(89, 1, 0))
    b = Matrix(700, 64 * 40, seed_path=(89, 2, 0))
    la = vbq.vbq_pack(*a.device_args(DEV))
    lb = vbq.vbq_pack(*b.device_args(DEV))
    ra, rb = _reference(a), _reference(b)
    _assert_bound(_static(la, a), ra, "A first")
    _assert_bound(_static(lb, b), rb, "B after A")
    _assert_bound(_static(la, a), ra, "A after B")
    xb = bits_to_i16(b.x_bits[:1]).to(DEV)
    yb = torch.full((b.n,), float("nan"), dtype=torch.float32, device=DEV)
    vbq.vbq_gemv(lb, xb[0], yb)
    torch.cuda.synchronize()
    _assert_bound(yb.cpu().numpy(), rb, "B by vbq_gemv")
    _assert_bound(_static(lb, b), rb, "B after its allocating product")
    la.free()
    lb.free()


def test_static_scratch_rejects_layouts_over_the_limit():
    n, k = 8192 * 128 + 1, 64                # one row block more than the array covers
    codes = torch.zeros((n, k), dtype=torch.uint8, device=DEV)
    widths = torch.ones((n, 1), dtype=torch.uint8, device=DEV)
    scales = torch.zeros((n, 1), dtype=torch.int16, device=DEV)
    layout = vbq.vbq_pack(codes, widths, scales)
    x = torch.zeros(k, dtype=torch.int16, device=DEV)
    y = torch.zeros(n, dtype=torch.float32, device=DEV)
    with pytest.raises(vbq.VbqError) as e:
        vbq.vbq_gemv_static(layout, x, y)
    assert e.value.name == "VBQ_ERR_UNSUPPORTED"
    vbq.vbq_gemv(layout, x, y)               # the allocating path still takes it
    torch.cuda.synchronize()
    assert float(y.abs().max()) == 0.0
    layout.free()
