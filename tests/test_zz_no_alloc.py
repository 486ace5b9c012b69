"""vbq_gemv_static: the batch-1 product for callers that must not allocate
device memory (its split-K control words live in a fixed array inside the
library). Checked through the C ABI against vbq_gemv, two calls in a row.

This file is collected last on purpose: a run that stops at the first failure
has then already run every other test."""

import numpy as np
import pytest
import torch

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


@pytest.mark.parametrize("shape", [(4096, 4096), (1000, 768), (300, 64 * 70), (129, 64)],
                         ids=lambda s: f"{s[0]}x{s[1]}")
def test_static_scratch_matches_gemv(shape):
    n, k = shape
    m = Matrix(n, k, seed_path=(88, n, k))
    layout = vbq.vbq_pack(*m.device_args(DEV))
    x = bits_to_i16(m.x_bits[:1]).to(DEV)
    y_ref = torch.full((n,), float("nan"), dtype=torch.float32, device=DEV)
    vbq.vbq_gemv(layout, x[0], y_ref)
    torch.cuda.synchronize()
    ref = y_ref.cpu().numpy()
    for _ in range(2):                       # two calls in a row share the fixed array
        y = torch.full((n,), float("nan"), dtype=torch.float32, device=DEV)
        vbq.vbq_gemv_static(layout, x[0], y)
        torch.cuda.synchronize()
        assert np.allclose(y.cpu().numpy(), ref, rtol=1e-5, atol=1e-5)


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
