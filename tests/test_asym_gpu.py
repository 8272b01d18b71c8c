"""Asymmetric weights (a per-channel weight zero point zw) on the GPU against
the oracle's oracle_linear_asym: prefill and decode, int8 and int4, zero
points at the ends of the code range, split decode units, the int8 K limit,
the residual epilogue and a batch that mixes kernels and symmetric problems
(workspace layout)."""
import numpy as np
import pytest

import oracle
from gpu_helpers import assert_equal_int8, torch_cuda, upload
from paper_2408_13933_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True, params=[1, 2], ids=["tile256", "tile128"])
def prefill_kernel(request):
    """Every test runs on both prefill kernels: the 256-token one wherever the
    workspace allows (1), and the 128-token one (2)."""
    from paper_2408_13933_gb300 import mq
    assert mq.test_prefill_kernel(request.param) == 0
    yield request.param
    assert mq.test_prefill_kernel(0) == 0


def mq():
    from paper_2408_13933_gb300 import mq as m
    return m


def zero_points(seed, n, bits, ends=True):
    lo, hi = (-128, 127) if bits == 8 else (-8, 7)
    rng = np.random.default_rng(1000 + seed)
    zw = rng.integers(lo, hi + 1, size=n).astype(np.int32)
    if ends and n >= 2:
        zw[0], zw[-1] = lo, hi
    return zw


class AsymCase:
    """Device operands of one asymmetric problem and its oracle result."""

    def __init__(self, seed, m, k, n, bits, extreme=None, residual=False, zw=None, share=None):
        lib = mq()
        torch = torch_cuda()
        self.c = c = synth.random_case(seed, m, k, n, bits, extreme)
        if share is not None:  # read the input of another case (same device buffer)
            c.x, c.zx = share.c.x, share.c.zx
        self.zw = zero_points(seed, n, bits) if zw is None else zw
        packed, colsum = lib.pack_weights(c.w, bits)
        m0, sh = lib.requant_params(c.sw, c.sx, c.sy)
        self.dev = [upload(a) for a in (c.x, packed, colsum, m0, sh, self.zw)]
        if share is not None:
            self.dev[0] = share.dev[0]
        self.res = synth.residual_codes(seed, 0, m, n) if residual else None
        self.dres = upload(self.res) if residual else None
        self.y = torch.full((m, n), 77, dtype=torch.int8, device="cuda")

    def desc(self):
        c = self.c
        x, packed, colsum, m0, sh, zw = self.dev
        return mq().make_desc(x, c.zx, packed, colsum, c.N, m0, sh, c.zy, self.y, c.bits,
                              residual=self.dres, zw=zw)

    def want(self):
        c = self.c
        packed, _ = oracle.pack(c.w, c.bits)
        m0, sh = oracle.requant_params(c.sx, c.sw, c.sy)
        y = oracle.linear(c.x, c.zx, packed, c.bits, c.N, m0, sh, c.zy, zw=self.zw)
        if self.res is not None:
            y = oracle.residual_add(y, self.res)
        return y


def run(cases):
    torch = torch_cuda()
    lib = mq()
    descs = [c.desc() for c in cases]
    need = lib.workspace_size_batch(descs)
    ws = torch.zeros(max(need, 16), dtype=torch.uint8, device="cuda")
    rc = lib.linear_batch(descs, workspace=ws, ws_bytes=need)
    assert rc == 0, lib.status_string(rc)
    torch.cuda.synchronize()
    assert lib.check_device_status() == 0
    return [c.y.cpu().numpy() for c in cases]


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("shape", [(128, 256, 2048), (300, 200, 320), (17, 384, 512),
                                   (200, 64, 4096)], ids=lambda s: "x".join(map(str, s)))
def test_prefill_asym(shape, bits):
    m, n, k = shape
    c = AsymCase(m + n, m, k, n, bits)
    assert_equal_int8(run([c])[0], c.want(), f"prefill asym {shape} bits={bits}")


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("shape", [(1, 256, 8192), (5, 100, 4096), (16, 320, 2048),
                                   (3, 64, 64)], ids=lambda s: "x".join(map(str, s)))
def test_decode_asym(shape, bits):
    m, n, k = shape
    c = AsymCase(2 * m + n, m, k, n, bits)
    assert_equal_int8(run([c])[0], c.want(), f"decode asym {shape} bits={bits}")


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("extreme", ["min", "max", "mixed"])
@pytest.mark.parametrize("m", [1, 16, 150])
def test_asym_extreme_codes(m, extreme, bits):
    lo, hi = (-128, 127) if bits == 8 else (-8, 7)
    n = 96
    zw = np.where(np.arange(n) % 2 == 0, lo, hi).astype(np.int32)
    c = AsymCase(7 + m, m, 1024, n, bits, extreme, zw=zw)
    assert_equal_int8(run([c])[0], c.want(), f"asym extreme m={m} {extreme} bits={bits}")


@pytest.mark.parametrize("extreme", ["min", "max", "mixed"])
def test_asym_int4_extreme_codes_across_chunks(extreme):
    # int4 weights with zero points at the range ends, codes at the ends, K =
    # 20480: the tensor-core kernel's exact-f32 chunks of x (w - zw) (8192 k,
    # |x (w - zw)| <= 128 * 15) are full twice and ragged once
    n = 72
    zw = np.where(np.arange(n) % 2 == 0, -8, 7).astype(np.int32)
    c = AsymCase(19, 130, 20480, n, 4, extreme, zw=zw)
    assert_equal_int8(run([c])[0], c.want(), f"asym int4 long K {extreme}")


def test_asym_int8_at_k_limit():
    # K = MQ_MAX_K_ASYM8 with int8 weights: |acc| up to 255 * 255 * K < 2^31
    k = mq().MQ_MAX_K_ASYM8
    for m in (2, 40):
        c = AsymCase(31 + m, m, k, 48, 8, "mixed")
        assert_equal_int8(run([c])[0], c.want(), f"asym K limit m={m}")


@pytest.mark.parametrize("m", [4, 260])
def test_asym_residual(m):
    c = AsymCase(41 + m, m, 768, 160, 8, residual=True)
    assert_equal_int8(run([c])[0], c.want(), f"asym residual m={m}")


def test_asym_batch_mixes_kernels_and_symmetric(prefill_kernel):
    # decode and prefill, asymmetric and symmetric problems in one call: the
    # 128-token kernel needs the decode region only (the tensor-core kernel
    # folds the weight zero point into the widened weights); the 256-token one
    # adds its widened inputs after it
    a = AsymCase(51, 130, 512, 200, 8)
    b = AsymCase(52, 4, 1024, 96, 4)
    c = AsymCase(53, 70, 256, 64, 4)
    d = AsymCase(54, 2, 512, 80, 8, zw=np.zeros(80, np.int32))
    cases = [a, b, c, d]
    lib = mq()
    descs = [x.desc() for x in cases]
    descs[3].zw = None  # symmetric problem in the same batch
    need = lib.workspace_size_batch(descs)
    dec = lib.workspace_size(4, 96, 1024, 4)
    assert need == dec if prefill_kernel == 2 else need > dec
    torch = torch_cuda()
    ws = torch.zeros(need, dtype=torch.uint8, device="cuda")
    assert lib.linear_batch(descs, workspace=ws, ws_bytes=need) == 0
    torch.cuda.synchronize()
    assert lib.check_device_status() == 0
    for x in cases:
        assert_equal_int8(x.y.cpu().numpy(), x.want(), f"batch {x.c.name}")


def test_asym_shared_input(prefill_kernel):
    # q/k/v/gate/up-like problems reading one input (one asymmetric with zero
    # points, one symmetric), next to another input: no workspace for the
    # 128-token kernel; the 256-token one widens each distinct input once
    a = AsymCase(61, 96, 512, 128, 8)
    b = AsymCase(62, 96, 512, 64, 4, share=a)
    c = AsymCase(63, 96, 512, 200, 8, share=a)
    d = AsymCase(64, 96, 512, 48, 8, share=a, zw=np.zeros(48, np.int32))
    e = AsymCase(65, 80, 256, 72, 4)
    cases = [a, b, c, d, e]
    lib = mq()
    descs = [x.desc() for x in cases]
    descs[3].zw = None
    need = lib.workspace_size_batch(descs)
    region = lib.workspace_size(1, 1, 0, 4)
    if prefill_kernel == 2:
        assert need == 0
    else:  # two distinct inputs: f16 copies and row sums, each to 1024 bytes
        assert need == region + (2 * 96 * 512 + 1024) + (2 * 80 * 256 + 1024) + 1024
    torch = torch_cuda()
    ws = torch.zeros(max(need, 16), dtype=torch.uint8, device="cuda")
    assert lib.linear_batch(descs, workspace=ws, ws_bytes=need) == 0
    torch.cuda.synchronize()
    assert lib.check_device_status() == 0
    for x in cases:
        assert_equal_int8(x.y.cpu().numpy(), x.want(), f"shared input {x.c.name}")
