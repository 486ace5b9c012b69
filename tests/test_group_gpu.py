"""vbq_gemv_group: independent batch-1 products whose launches overlap. Each
product is checked against the CPU oracle through the C ABI; the group is
repeated (split-K epochs advance per layout), followed by a dependent product
that reads one of its outputs (stream order at the group's end), and its
argument checks are exercised on real layouts."""

import numpy as np
import pytest
import torch

import oracle
import paper_2607_02893_gb300 as vbq
from vbq_cases import Matrix, bits_to_i16

pytestmark = pytest.mark.gpu

DEV = "cuda"
SHAPES = [(4096, 4096), (1000, 768), (300, 64 * 70), (129, 64), (2048, 5632), (640, 1024)]


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2607_02893_gb300 import build
    build.build()
    vbq.load()
    torch.cuda.init()


def _mats():
    return [Matrix(n, k, seed_path=(87, n, k)) for n, k in SHAPES]


def _check(m, y, x_bits):
    w = oracle.dequant(m.codes.numpy(), m.widths, m.scales)
    x = (np.asarray(x_bits, np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    y_ref = w @ x
    a_ref = np.abs(w) @ np.abs(x)
    got = y.cpu().numpy().astype(np.float64)
    bad = ~(np.abs(got - y_ref) <= 2e-3 * a_ref + 1e-5)
    assert not bad.any(), f"{int(bad.sum())} outputs outside the bound"


def test_group_matches_oracle_repeated():
    mats = _mats()
    lays = [vbq.vbq_pack(*m.device_args(DEV)) for m in mats]
    xs = [bits_to_i16(m.x_bits[:1]).to(DEV)[0] for m in mats]
    # one input per product here; a shared input is covered in the next test
    for rep in range(3):
        ys = [torch.full((m.n,), float("nan"), dtype=torch.float32, device=DEV) for m in mats]
        vbq.vbq_gemv_group(lays, xs, ys)
        torch.cuda.synchronize()
        for m, x, y in zip(mats, xs, ys):
            _check(m, y, x.cpu().numpy().view(np.uint16))


def test_group_output_feeds_a_later_product():
    mats = [Matrix(768, 768, seed_path=(86, 0, i)) for i in range(3)]
    lays = [vbq.vbq_pack(*m.device_args(DEV)) for m in mats]
    x = bits_to_i16(mats[0].x_bits[:1]).to(DEV)[0]
    ys = [torch.empty(768, dtype=torch.float32, device=DEV) for _ in mats]
    nxt = Matrix(512, 768, seed_path=(86, 1, 0))
    lay_n = vbq.vbq_pack(*nxt.device_args(DEV))
    y_n = torch.empty(512, dtype=torch.float32, device=DEV)
    for _ in range(3):
        vbq.vbq_gemv_group(lays, [x, x, x], ys)          # one input read by all three
        # the next product's input is the last group output, rounded to BF16 on
        # the same stream (round to nearest even on the bit pattern)
        b = ys[-1].view(torch.int32)
        x_n = ((b + 0x7FFF + ((b >> 16) & 1)) >> 16).to(torch.int16)
        vbq.vbq_gemv(lay_n, x_n, y_n)
        torch.cuda.synchronize()
        for m, y in zip(mats, ys):
            _check(m, y, x.cpu().numpy().view(np.uint16))
        _check(nxt, y_n, x_n.cpu().numpy().view(np.uint16))


def test_group_rejects_repeats():
    m = Matrix(256, 1024, seed_path=(85, 0, 0))
    lay = vbq.vbq_pack(*m.device_args(DEV))
    lay2 = vbq.vbq_pack(*m.device_args(DEV))
    x = bits_to_i16(m.x_bits[:1]).to(DEV)[0]
    y, y2 = torch.empty(256, device=DEV), torch.empty(256, device=DEV)
    for args in (([lay, lay], [x, x], [y, y2]), ([lay, lay2], [x, x], [y, y])):
        with pytest.raises(vbq.VbqError) as e:
            vbq.vbq_gemv_group(*args)
        assert e.value.name == "VBQ_ERR_ARG"
    vbq.vbq_gemv_group([lay, lay2], [x, x], [y, y2])
    torch.cuda.synchronize()
    assert torch.equal(torch.isfinite(y), torch.ones_like(y, dtype=torch.bool))
    _check(m, y, x.cpu().numpy().view(np.uint16))
    _check(m, y2, x.cpu().numpy().view(np.uint16))
