"""Failure detection on the device: a bounded wait that runs out is recorded
and reported through vbq_device_status, the block returns, and the CUDA
context stays usable (no fault, no hang). The wait is made to run out by the
library's self-test kernel, which waits on a barrier that nothing completes."""

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


def test_timeout_is_reported_once_and_the_context_survives():
    vbq.vbq_device_status()                      # start from a clear record
    vbq.vbq_selftest_timeout(20000)              # one wait, bounded to 20 ms
    with pytest.raises(vbq.VbqError) as e:
        vbq.vbq_device_status()
    assert e.value.name == "VBQ_ERR_TIMEOUT"
    vbq.vbq_device_status()                      # reading cleared it

    m = Matrix(1000, 768, seed_path=(91, 1000, 768))
    layout = vbq.vbq_pack(*m.device_args(DEV))
    x = bits_to_i16(m.x_bits[:1]).to(DEV)
    y = torch.full((1000,), float("nan"), dtype=torch.float32, device=DEV)
    vbq.vbq_gemv(layout, x[0], y)
    vbq.vbq_device_status()                      # a normal product records nothing
    y_ref, a_ref = oracle.gemv(m.codes.numpy(), m.widths, m.scales, m.x()[:1])
    assert oracle.within_bound(y.cpu().numpy()[None, :], y_ref, a_ref).all()
