"""Boundary quantizers on the GPU against the oracle: float (f32 / f16 / bf16)
to int8 / int16 codes, codes back to f32, and fixed-point requantization
between int8 and int16 codes, bit for bit, over ties, infinities, NaN,
subnormals, every code, vector tails and unaligned (scalar-path) buffers."""
import numpy as np
import pytest

import oracle
from gpu_helpers import torch_cuda

pytestmark = pytest.mark.gpu


def mq():
    from paper_2408_13933_gb300 import mq as m
    return m


def _np_of(bits):
    return np.int8 if bits == 8 else np.int16


def _float_values(n, alpha, seed):
    """Values spread over the code range, near-ties, specials and subnormals."""
    rng = np.random.default_rng(seed)
    x = (rng.standard_normal(n) * alpha * 60).astype(np.float32)
    k = rng.integers(-300, 300, size=n // 4)
    x[: n // 4] = ((k + 0.5) * alpha).astype(np.float32)
    special = np.array([np.inf, -np.inf, np.nan, 0.0, -0.0, 1e-42, -1e-42, 3e38, -3e38],
                       np.float32)
    x[-special.size:] = special
    return x


@pytest.mark.parametrize("in_dtype", ["f32", "f16", "bf16"])
@pytest.mark.parametrize("bits", [8, 16])
@pytest.mark.parametrize("n", [1, 15, 16, 17, 4099, 1 << 20])
def test_quantize(in_dtype, bits, n):
    torch = torch_cuda()
    alpha, z = (0.05, 3) if bits == 8 else (2e-4, -1234)
    xf = _float_values(max(n, 9), alpha, n + bits)[:n]
    tdt = {"f32": torch.float32, "f16": torch.float16, "bf16": torch.bfloat16}[in_dtype]
    xt = torch.from_numpy(xf).to(tdt)
    # the oracle sees the same values, widened exactly to f32
    xo = xt.float().numpy()
    want = oracle.quantize(xo, alpha, z, bits)
    qd = torch.zeros(n, dtype=torch.int8 if bits == 8 else torch.int16, device="cuda")
    assert mq().quantize(xt.cuda(), alpha, z, qd) == 0
    torch.cuda.synchronize()
    assert np.array_equal(qd.cpu().numpy(), want)


@pytest.mark.parametrize("bits", [8, 16])
def test_quantize_unaligned_scalar_path(bits):
    torch = torch_cuda()
    n = 1000
    xf = _float_values(n + 3, 0.02, 7)
    xd = torch.from_numpy(xf).cuda()
    qd = torch.zeros(n + 3, dtype=torch.int8 if bits == 8 else torch.int16, device="cuda")
    # views starting one element in: 4 (or 1 / 2) bytes off the 16-byte grid
    assert mq().quantize(xd[1:n + 1], 0.02, -5, qd[3:n + 3]) == 0
    torch.cuda.synchronize()
    want = oracle.quantize(xf[1:n + 1], 0.02, -5, bits)
    got = qd.cpu().numpy()
    assert np.array_equal(got[3:], want)
    assert np.all(got[:3] == 0)


@pytest.mark.parametrize("bits", [8, 16])
def test_dequantize_every_code(bits):
    torch = torch_cuda()
    lo, hi = (-128, 127) if bits == 8 else (-32768, 32767)
    q = np.arange(lo, hi + 1, dtype=np.int64).astype(_np_of(bits))
    for alpha, z in ((0.0371, 5), (1.0 / 3.0, lo), (2.5e-4, hi)):
        f = torch.zeros(q.size, dtype=torch.float32, device="cuda")
        assert mq().dequantize(torch.from_numpy(q).cuda(), alpha, z, f) == 0
        torch.cuda.synchronize()
        want = oracle.dequantize(q, alpha, z)
        assert np.array_equal(f.cpu().numpy().view(np.uint32), want.view(np.uint32))


@pytest.mark.parametrize("in_bits", [8, 16])
@pytest.mark.parametrize("out_bits", [8, 16])
def test_requantize_every_code(in_bits, out_bits):
    torch = torch_cuda()
    ilo, ihi = (-128, 127) if in_bits == 8 else (-32768, 32767)
    lo, hi = (-128, 127) if out_bits == 8 else (-32768, 32767)
    q = np.arange(ilo, ihi + 1, dtype=np.int64).astype(_np_of(in_bits))
    rng = np.random.default_rng(in_bits * 3 + out_bits)
    params = [(0, 1 << 30, 31, 0), (ilo, (1 << 31) - 1, 1, hi), (ihi, 1 << 30, 62, lo)]
    for _ in range(5):
        params.append((int(rng.integers(ilo, ihi + 1)), int(rng.integers(1 << 30, 1 << 31)),
                       int(rng.integers(1, 63)), int(rng.integers(lo, hi + 1))))
    params.append((3, 0, 20, 7))  # M0 = 0: every output is zy
    qd = torch.from_numpy(q).cuda()
    for zx, m0, sh, zy in params:
        y = torch.zeros(q.size, dtype=torch.int8 if out_bits == 8 else torch.int16, device="cuda")
        assert mq().requantize(qd, zx, m0, sh, zy, y) == 0
        torch.cuda.synchronize()
        want = oracle.requantize(q, zx, m0, sh, zy, out_bits)
        assert np.array_equal(y.cpu().numpy(), want), (zx, m0, sh, zy)


def test_requantize_large_ragged():
    torch = torch_cuda()
    rng = np.random.default_rng(11)
    n = (1 << 22) + 13
    q = rng.integers(-32768, 32768, size=n).astype(np.int16)
    m0, sh = mq().requant_params(np.array([3.1e-4], np.float32), 1.0, 0.011)
    y = torch.zeros(n, dtype=torch.int8, device="cuda")
    assert mq().requantize(torch.from_numpy(q).cuda(), -40, int(m0[0]), int(sh[0]), 9, y) == 0
    torch.cuda.synchronize()
    assert np.array_equal(y.cpu().numpy(), oracle.requantize(q, -40, int(m0[0]), int(sh[0]), 9, 8))
