"""16-bit activations (W8A16 / W4A16) on the GPU against the oracle's
oracle_linear_a16: tensor-core and decode shapes, int8 and int4 weights,
codes at the ends of the int16 range, every requantization shift, the K
limit, split decode units, and batches that mix activation widths, kernels
and shared inputs (workspace planning)."""
import numpy as np
import pytest

import oracle
from gpu_helpers import torch_cuda, upload
from paper_2408_13933_gb300 import synth

pytestmark = pytest.mark.gpu


def mq():
    from paper_2408_13933_gb300 import mq as m
    return m


def assert_equal_int16(got: np.ndarray, want: np.ndarray, what: str):
    if not np.array_equal(got, want):
        bad = np.argwhere(got != want)
        i = tuple(bad[0])
        raise AssertionError(f"{what}: {len(bad)} of {want.size} outputs differ; first at {i}: "
                             f"got {int(got[i])}, want {int(want[i])}")


class A16Case:
    """Device operands of one 16-bit-activation problem and its oracle result."""

    def __init__(self, case, m0=None, shift=None, share=None, zw=None):
        lib = mq()
        torch = torch_cuda()
        self.c = c = case
        self.zw = None if zw is None else np.asarray(zw, np.int32)
        if share is not None:  # read the input of another case (same device buffer)
            c.x, c.zx = share.c.x, share.c.zx
        packed, colsum = lib.pack_weights(c.w, c.bits)
        if m0 is None:
            m0, shift = lib.requant_params(c.sw, c.sx, c.sy)
        self.m0, self.shift = np.asarray(m0, np.int32), np.asarray(shift, np.int32)
        self.dev = [upload(a) for a in (c.x, packed, colsum, self.m0, self.shift)]
        self.zw_dev = upload(self.zw) if self.zw is not None else None
        if share is not None:
            self.dev[0] = share.dev[0]
        self.y = torch.full((c.M, max(c.N, 1)), 12345, dtype=torch.int16, device="cuda")

    def desc(self):
        c = self.c
        x, packed, colsum, m0, sh = self.dev
        return mq().make_desc(x, c.zx, packed, colsum, c.N, m0, sh, c.zy, self.y, c.bits,
                              abits=16, zw=self.zw_dev)

    def run_single(self):
        c = self.c
        lib = mq()
        torch = torch_cuda()
        need = lib.workspace_size_a16(c.M, c.N, c.K, c.bits)
        ws = torch.zeros(max(need, 16), dtype=torch.uint8, device="cuda")
        x, packed, colsum, m0, sh = self.dev
        rc = lib.linear_a16(x, c.zx, packed, colsum, c.N, m0, sh, c.zy, self.y, c.bits,
                            workspace=ws, ws_bytes=need)
        assert rc == 0, lib.status_string(rc)
        torch.cuda.synchronize()
        assert lib.check_device_status() == 0
        return self.y.cpu().numpy()[:, :c.N], ws

    def want(self):
        c = self.c
        packed, _ = oracle.pack(c.w, c.bits)
        return oracle.linear_a16(c.x, c.zx, packed, c.bits, c.N, self.m0, self.shift, c.zy,
                                 zw=self.zw)


def run_batch(cases):
    torch = torch_cuda()
    lib = mq()
    descs = [c.desc() for c in cases]
    need = lib.workspace_size_batch(descs)
    ws = torch.zeros(max(need, 16), dtype=torch.uint8, device="cuda")
    rc = lib.linear_batch(descs, workspace=ws, ws_bytes=need)
    assert rc == 0, lib.status_string(rc)
    torch.cuda.synchronize()
    assert lib.check_device_status() == 0
    return [c.y.cpu().numpy()[:, :c.c.N] for c in cases]


SHAPES_PRE = [(128, 256, 2048), (300, 200, 320), (17, 384, 512), (9, 64, 4096), (200, 64, 4096)]
SHAPES_DEC = [(1, 256, 8192), (3, 100, 4096), (8, 320, 2048), (4, 64, 64), (5, 96, 1024)]


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("shape", SHAPES_PRE + SHAPES_DEC, ids=lambda s: "x".join(map(str, s)))
def test_a16_parity(shape, bits):
    m, n, k = shape
    c = A16Case(synth.random_case_a16(m + 3 * n + k, m, k, n, bits))
    got, _ = c.run_single()
    assert_equal_int16(got, c.want(), f"a16 {shape} bits={bits}")


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("extreme", ["min", "max", "mixed"])
@pytest.mark.parametrize("m", [1, 8, 150])
def test_a16_extreme_codes(m, extreme, bits):
    c = A16Case(synth.random_case_a16(90 + m, m, 1024, 96, bits, extreme))
    got, _ = c.run_single()
    assert_equal_int16(got, c.want(), f"a16 extreme m={m} {extreme} bits={bits}")


@pytest.mark.parametrize("m", [2, 40])
def test_a16_every_shift(m):
    # per-channel (M0, shift) over every shift 1..62 (multipliers from 2^31
    # down to 2^-32): both requantization branches of the 16-bit epilogue,
    # saturation at both ends, and the M0 = 0 case
    rng = np.random.default_rng(7 + m)
    n = 128
    base = synth.random_case_a16(70 + m, m, 512, n, 8, "mixed" if m == 2 else None)
    sh = np.array([1 + (i % 62) for i in range(n)], np.int32)
    m0 = rng.integers(1 << 30, 1 << 31, size=n).astype(np.int64)
    m0[::17] = 0
    c = A16Case(base, m0=m0.astype(np.int32), shift=sh)
    got, _ = c.run_single()
    assert_equal_int16(got, c.want(), f"a16 shifts m={m}")


@pytest.mark.parametrize("m", [2, 24])
def test_a16_k_limit(m):
    # K = 65536 with codes at the range ends: |acc| near 65535 * 127 * 65536
    for bits in (8, 4):
        c = A16Case(synth.random_case_a16(80 + m + bits, m, 65536, 40, bits, "max"))
        got, _ = c.run_single()
        assert_equal_int16(got, c.want(), f"a16 K=65536 m={m} bits={bits}")


def test_a16_empty_and_k0():
    lib = mq()
    torch = torch_cuda()
    # K = 0: every output is requant(0 - 0) = zy
    base = synth.random_case_a16(5, 6, 0, 20, 8)
    c = A16Case(base)
    got, _ = c.run_single()
    assert np.all(got == c.c.zy)
    # M = 0 and N = 0 return without work
    x = torch.zeros((0, 64), dtype=torch.int16, device="cuda")
    y = torch.zeros((0, 8), dtype=torch.int16, device="cuda")
    assert lib.linear_a16(x, 0, x, x, 8, x, x, 0, y, 8, k=64, ldx=64, ldy=8) == 0


def test_a16_decode_leaves_workspace_zero():
    torch = torch_cuda()
    for seed, (m, k, n, bits) in enumerate([(1, 5632, 2048, 4), (8, 16384, 300, 8),
                                            (3, 2080, 70, 4)]):
        c = A16Case(synth.random_case_a16(600 + seed, m, k, n, bits))
        got, ws = c.run_single()
        assert_equal_int16(got, c.want(), f"a16 ws m={m} k={k}")
        dec = mq().workspace_size(1, 1, 0, 4)
        assert int(torch.count_nonzero(ws[:dec])) == 0


def test_a16_batch_mixed_widths_kernels_and_shared_inputs():
    # 16-bit problems (prefill and decode, two sharing one input) next to
    # int8 problems (one asymmetric) in one call
    from gpu_helpers import GpuLinear, oracle_y, assert_equal_int8
    a = A16Case(synth.random_case_a16(201, 96, 512, 128, 8))
    b = A16Case(synth.random_case_a16(202, 96, 512, 64, 4), share=a)
    d = A16Case(synth.random_case_a16(203, 3, 1024, 200, 4))
    e = A16Case(synth.random_case_a16(204, 8, 256, 72, 8))
    g8 = GpuLinear(synth.random_case(205, 70, 512, 96, 8))
    g4 = GpuLinear(synth.random_case(206, 4, 1024, 80, 4))
    lib = mq()
    torch = torch_cuda()
    descs = [a.desc(), g8.desc(), b.desc(), d.desc(), g4.desc(), e.desc()]
    need = lib.workspace_size_batch(descs)
    dec = lib.workspace_size(1, 1, 0, 4)
    # planes only for the tensor-core inputs (a and b share one); decode reads int16 itself
    assert need == dec + 2 * 96 * 512
    ws = torch.zeros(need, dtype=torch.uint8, device="cuda")
    assert lib.linear_batch(descs, workspace=ws, ws_bytes=need) == 0
    torch.cuda.synchronize()
    assert lib.check_device_status() == 0
    for c in (a, b, d, e):
        assert_equal_int16(c.y.cpu().numpy()[:, :c.c.N], c.want(), f"batch {c.c.name}")
    for g in (g8, g4):
        assert_equal_int8(g.y.cpu().numpy(), oracle_y(g.case), f"batch {g.case.name}")
    assert int(torch.count_nonzero(ws[:dec])) == 0


def run_desc(c):
    # one 16-bit problem through the batch call (weight zero points are a
    # descriptor field)
    torch = torch_cuda()
    lib = mq()
    d = c.desc()
    need = lib.workspace_size_batch([d])
    ws = torch.zeros(max(need, 16), dtype=torch.uint8, device="cuda")
    assert lib.linear_batch([d], workspace=ws, ws_bytes=need) == 0
    torch.cuda.synchronize()
    assert lib.check_device_status() == 0
    return c.y.cpu().numpy()[:, :c.c.N], ws


def ends(n, bits):
    lo, hi = (-128, 127) if bits == 8 else (-8, 7)
    return np.where(np.arange(n) % 3 == 0, lo, np.where(np.arange(n) % 3 == 1, hi, 0)).astype(np.int32)


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("shape", SHAPES_PRE[:3] + SHAPES_DEC[:3], ids=lambda s: "x".join(map(str, s)))
def test_a16_weight_zero_points(shape, bits):
    # 16-bit activations against weights with per-channel zero points (the
    # attention matmul of the W8A16 setting, keys or V as the 8-bit operand)
    m, n, k = shape
    rng = np.random.default_rng(m * 7 + n)
    lo, hi = (-128, 127) if bits == 8 else (-8, 7)
    c = A16Case(synth.random_case_a16(5 * m + n + k, m, k, n, bits),
                zw=rng.integers(lo, hi + 1, size=n))
    got, _ = run_desc(c)
    assert_equal_int16(got, c.want(), f"a16 zw {shape} bits={bits}")


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("extreme", ["min", "max", "mixed"])
@pytest.mark.parametrize("m", [1, 8, 150])
def test_a16_weight_zero_points_extreme(m, extreme, bits):
    # codes and zero points at the range ends: |plane (w - zw)| up to 128 * 255
    c = A16Case(synth.random_case_a16(190 + m, m, 1024, 96, bits, extreme), zw=ends(96, bits))
    got, _ = run_desc(c)
    assert_equal_int16(got, c.want(), f"a16 zw extreme m={m} {extreme} bits={bits}")


@pytest.mark.parametrize("m", [2, 24])
def test_a16_weight_zero_points_k_limit(m):
    # K = 65536 with codes and zero points at the range ends: the decode
    # kernel's int32 plane sums reach 128 * 255 * 65536 < 2^31, the tensor-core
    # kernel's 512-k chunks run 128 times
    for bits in (8, 4):
        c = A16Case(synth.random_case_a16(280 + m + bits, m, 65536, 40, bits, "max"),
                    zw=ends(40, bits))
        got, ws = run_desc(c)
        assert_equal_int16(got, c.want(), f"a16 zw K=65536 m={m} bits={bits}")
        if 2 * m <= 16:
            dec = mq().workspace_size(1, 1, 0, 4)
            assert int(torch_cuda().count_nonzero(ws[:dec])) == 0


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("k", [0, 16, 64, 144, 1040, 2080])
@pytest.mark.parametrize("m", [1, 3, 8, 20])
def test_a16_weight_zero_points_ragged_k(m, k, bits):
    # K not a multiple of the decode stage (128 k int8, 256 k int4): the
    # zero-filled codes past K meet the zero point; K = 0: every output is
    # requant(0) = zy.  m = 20 runs the tensor-core kernel.
    if bits == 4 and k % 32:
        pytest.skip("int4 K is a multiple of 32")
    c = A16Case(synth.random_case_a16(700 + m + k + bits, m, k, 56, bits, "mixed"),
                zw=ends(56, bits))
    got, _ = run_desc(c)
    assert_equal_int16(got, c.want(), f"a16 zw ragged K={k} m={m} bits={bits}")
