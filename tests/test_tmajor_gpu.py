"""The token-major tensor-core kernel (tokens as the MMA's M: the attention
matmuls' short K and few channels) against the oracle, forced onto every
shape by its test hook: wide tiles (one exact run, 256 channels) and narrow
ones (64 channels, several runs with and without a weight zero point), int8
output with and without the residual, int16 output, ragged tokens, channels
and K, extreme codes at the exact-run bound, rows that take the scalar store
path, a batch over more problems than one launch holds, the automatic
choice (K <= 128 or N <= 64) against the other kernels' bytes, and weights
stored transposed ([K][N] inside wider rows, as attention's V)."""
import numpy as np
import pytest

import oracle
from gpu_helpers import torch_cuda, upload
from paper_2408_13933_gb300 import synth

pytestmark = pytest.mark.gpu


def mq():
    from paper_2408_13933_gb300 import mq as m
    return m


@pytest.fixture(autouse=True)
def force_tmajor():
    lib = mq()
    assert lib.test_tmajor_kernel(1) == 0
    yield
    assert lib.test_tmajor_kernel(0) == 0


def assert_equal(got, want, what):
    if not np.array_equal(got, want):
        bad = np.argwhere(got != want)
        i = tuple(bad[0])
        raise AssertionError(f"{what}: {len(bad)} of {want.size} differ; first at {i}: "
                             f"got {int(got[i])}, want {int(want[i])}")


class Case:
    """Device operands of one problem (int8 weights) and the oracle's result."""

    def __init__(self, seed, m, k, n, zw=False, residual=False, o16=False, extreme=None,
                 pad_y=0):
        torch = torch_cuda()
        lib = mq()
        self.c = c = synth.random_case(seed, m, k, n, 8, extreme)
        rng = np.random.default_rng(7000 + seed)
        self.zw = rng.integers(-128, 128, size=n).astype(np.int32) if zw else None
        if zw and n >= 2:
            self.zw[0], self.zw[-1] = -128, 127
        self.o16 = o16
        if o16:  # shifts on both sides of the multiply-high form's 33
            self.m0 = rng.integers(1 << 30, 1 << 31, size=n).astype(np.int32)
            self.sh = rng.integers(28, 47, size=n).astype(np.int32)
            self.zy = int(rng.integers(-20000, 20000))
        else:
            self.m0, self.sh = lib.requant_params(c.sw, c.sx, c.sy)
            self.zy = c.zy
        packed, colsum = lib.pack_weights(c.w, 8)
        self.keep = [upload(a) for a in (c.x, packed, colsum, self.m0, self.sh)]
        self.dzw = upload(self.zw) if zw else None
        self.res = synth.residual_codes(seed, 0, m, n + pad_y) if residual else None
        self.dres = upload(self.res) if residual else None
        ldy = n + pad_y
        self.y = torch.full((m, ldy), 77, dtype=torch.int16 if o16 else torch.int8, device="cuda")
        self.n = n

    def desc(self):
        c = self.c
        x, packed, colsum, m0, sh = self.keep
        return mq().make_desc(x, c.zx, packed, colsum, c.N, m0, sh, self.zy, self.y, 8,
                              residual=self.dres, zw=self.dzw)

    def want(self):
        c = self.c
        packed, _ = oracle.pack(c.w, 8)
        if self.o16:
            return oracle.linear_o16(c.x, c.zx, packed, 8, c.N, self.m0, self.sh, self.zy,
                                     zw=self.zw)
        y = oracle.linear(c.x, c.zx, packed, 8, c.N, self.m0, self.sh, self.zy, zw=self.zw)
        if self.res is not None:
            y = oracle.residual_add(y, np.ascontiguousarray(self.res[:, :c.N]))
        return y

    def got(self):
        return self.y.cpu().numpy()[:, :self.n]


def run(cases):
    torch = torch_cuda()
    lib = mq()
    descs = [c.desc() for c in cases]
    need = lib.workspace_size_batch(descs)
    ws = torch.zeros(max(need, 16), dtype=torch.uint8, device="cuda")
    assert lib.linear_batch(descs, workspace=ws, ws_bytes=need) == 0
    torch.cuda.synchronize()
    assert lib.check_device_status() == 0


SHAPES = [(128, 256, 64),    # one wide tile, K = one stage
          (300, 100, 320),   # ragged tokens, N < 256 in a wide tile, five stages
          (257, 520, 192),   # ragged tokens and channels over several wide tiles
          (200, 64, 1024),   # narrow tile, one run at its bound
          (130, 96, 2048),   # narrow tiles, two runs, ragged channels
          (40, 48, 3024),    # narrow, several runs, a ragged last stage
          (96, 200, 80)]     # wide, a ragged second stage (k past K must add 0)


@pytest.mark.parametrize("zw", [False, True], ids=["sym", "zw"])
@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: "x".join(map(str, s)))
def test_tmajor_int8_output(shape, zw):
    m, n, k = shape
    c = Case(m + n + k, m, k, n, zw=zw)
    run([c])
    assert_equal(c.got(), c.want(), f"int8 {shape} zw={zw}")


@pytest.mark.parametrize("shape", [(256, 320, 64), (150, 64, 1104), (96, 1024, 128)],
                         ids=lambda s: "x".join(map(str, s)))
@pytest.mark.parametrize("zw", [False, True], ids=["sym", "zw"])
def test_tmajor_int16_output(shape, zw):
    m, n, k = shape
    c = Case(5 * m + n, m, k, n, zw=zw, o16=True)
    run([c])
    assert_equal(c.got(), c.want(), f"int16 {shape} zw={zw}")


@pytest.mark.parametrize("shape", [(300, 100, 320), (130, 96, 2048)],
                         ids=lambda s: "x".join(map(str, s)))
def test_tmajor_residual(shape):
    m, n, k = shape
    c = Case(11 + m, m, k, n, zw=True, residual=True)
    run([c])
    assert_equal(c.got(), c.want(), f"residual {shape}")


@pytest.mark.parametrize("o16", [False, True], ids=["int8", "int16"])
def test_tmajor_scalar_store_path(o16):
    # output rows whose pitch is not a multiple of 16 bytes: every group takes
    # the per-element stores; the pad bytes stay untouched
    m, n, k = 140, 200, 128
    c = Case(21, m, k, n, zw=True, o16=o16, residual=not o16, pad_y=3)
    run([c])
    assert_equal(c.got(), c.want(), f"scalar path o16={o16}")
    pad = c.y.cpu().numpy()[:, n:]
    assert (pad == 77).all(), "bytes past N written"


@pytest.mark.parametrize("o16", [False, True], ids=["int8", "int16"])
@pytest.mark.parametrize("n", [100, 50])
def test_tmajor_row_tail_untouched(n, o16):
    # N * size not a multiple of 16 with rows that are: the bytes between N
    # and the row pitch stay untouched (a TMA store would clip only in whole
    # 16-byte chunks, so such rows take the per-element tail)
    m, k = 140, 256
    pad = (-n) % 16 + 16
    c = Case(61 + n, m, k, n, zw=True, o16=o16, pad_y=pad)
    run([c])
    assert_equal(c.got(), c.want(), f"tail n={n} o16={o16}")
    assert (c.y.cpu().numpy()[:, n:] == 77).all(), "bytes past N written"


@pytest.mark.parametrize("extreme", ["min", "max", "mixed"])
@pytest.mark.parametrize("shape", [(130, 300, 1024), (70, 64, 2048)],
                         ids=lambda s: "x".join(map(str, s)))
def test_tmajor_extreme_codes(shape, extreme):
    # all products at +-2^14: one run of 1024 k reaches 2^24, the f32 bound
    m, n, k = shape
    c = Case(31 + m, m, k, n, extreme=extreme)
    run([c])
    assert_equal(c.got(), c.want(), f"extreme {shape} {extreme}")


def test_tmajor_batch_over_two_launches():
    # 36 problems (more than one launch's 32), wide and narrow, int8 outputs
    cases = [Case(100 + i, 64 + 7 * i, 64 * (1 + i % 5), (24, 80, 300)[i % 3], zw=i % 2 == 1,
                  residual=i % 4 == 0) for i in range(36)]
    run(cases)
    for i, c in enumerate(cases):
        assert_equal(c.got(), c.want(), f"batch problem {i}")


@pytest.mark.parametrize("shape", [(512, 1024, 64), (1024, 64, 1024), (300, 2048, 2048)],
                         ids=lambda s: "x".join(map(str, s)))
def test_tmajor_choice_matches_other_kernels(shape):
    # the automatic choice (the first two shapes take the token-major kernel,
    # the third not) gives the bytes the other kernels give
    lib = mq()
    m, n, k = shape
    outs = []
    for mode in (0, 2):
        assert lib.test_tmajor_kernel(mode) == 0
        c = Case(41 + m, m, k, n, zw=True)
        run([c])
        outs.append(c.got())
    assert_equal(outs[0], outs[1], f"auto vs never {shape}")
    assert_equal(outs[0], c.want(), f"oracle {shape}")


class WtCase(Case):
    """A Case whose weights are stored transposed: int8 [K][N] at column `col`
    of rows `ldw` bytes apart (attention's V_g read in place), the other
    columns holding codes the kernel must not read."""

    def __init__(self, seed, m, k, n, ldw=None, col=0, **kw):
        super().__init__(seed, m, k, n, **kw)
        self.ldw = ldw or n
        self.col = col
        wt = np.full((k, self.ldw), 55, np.int8)
        wt[:, col:col + n] = self.c.w.T
        self.wt_dev = upload(wt)

    def desc(self):
        c = self.c
        x, _, _, m0, sh = self.keep
        return mq().make_desc(x, c.zx, self.wt_dev[:, self.col:], None, c.N, m0, sh, self.zy,
                              self.y, 8, residual=self.dres, zw=self.dzw, ldw=self.ldw, wt=True)


WT_SHAPES = [(200, 64, 1024, 64, 0),     # one narrow tile column, one run at its bound
             (130, 96, 2048, 96, 0),     # ragged second channel tile, two runs
             (40, 48, 3024, 48, 0),      # a ragged last stage
             (300, 100, 320, 128, 0),    # ragged rows: N inside a 128-byte pitch
             (1024, 64, 1024, 256, 64)]  # attention: V_1 of four KV heads


@pytest.mark.parametrize("zw", [False, True], ids=["sym", "zw"])
@pytest.mark.parametrize("shape", WT_SHAPES, ids=lambda s: "x".join(map(str, s)))
def test_tmajor_transposed_weights(shape, zw):
    m, n, k, ldw, col = shape
    c = WtCase(3 * m + k, m, k, n, ldw=ldw, col=col, zw=zw)
    run([c])
    assert_equal(c.got(), c.want(), f"wt {shape} zw={zw}")


@pytest.mark.parametrize("o16", [False, True], ids=["int8-residual", "int16"])
def test_tmajor_transposed_weights_outputs(o16):
    m, n, k = 256, 80, 1104
    c = WtCase(17, m, k, n, ldw=96, zw=True, o16=o16, residual=not o16)
    run([c])
    assert_equal(c.got(), c.want(), f"wt outputs o16={o16}")


@pytest.mark.parametrize("extreme", ["min", "max", "mixed"])
def test_tmajor_transposed_weights_extreme(extreme):
    m, n, k = 70, 64, 2048
    c = WtCase(47, m, k, n, extreme=extreme)
    run([c])
    assert_equal(c.got(), c.want(), f"wt extreme {extreme}")


@pytest.mark.parametrize("mode", [0, 1])
def test_tmajor_transposed_weights_in_a_mixed_batch(mode):
    # transposed and row-major weights in one call (one narrow launch holds
    # both kinds, beside a wide one); with the automatic choice a transposed
    # problem of long K and many channels still takes the token-major kernel
    lib = mq()
    assert lib.test_tmajor_kernel(mode) == 0
    cases = [WtCase(71, 300, 512, 256, zw=True), Case(72, 200, 1024, 64, zw=True),
             WtCase(73, 140, 640, 64, ldw=128, col=64), Case(74, 260, 64, 300)]
    run(cases)
    for i, c in enumerate(cases):
        assert_equal(c.got(), c.want(), f"mixed batch problem {i} mode {mode}")
