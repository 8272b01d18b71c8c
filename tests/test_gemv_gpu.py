"""The row-tile decode kernel (one or two tokens, mq_gemv.cu) on the GPU
against the oracle, bit for bit.  The hook mq_test_decode_kernel(1) makes the
library take it for every launch it can serve, so that small and ragged
shapes reach it too: 8-row tiles cut short by N, rows shorter than one
1024-byte chunk and rows ending in a partial chunk, K at its limit, int8 and
int4 weights at the ends of their ranges, weight zero points, the int16
output, the residual, a weight row pitch, weights written on the device, and
batches mixing problems of one and two tokens and of different K.  The same
launches through the split-K kernel (hook value 2) must give the same bytes."""
import numpy as np
import pytest

import oracle
from gpu_helpers import assert_equal_int8, torch_cuda, upload
from paper_2408_13933_gb300 import synth

pytestmark = pytest.mark.gpu


def mq():
    from paper_2408_13933_gb300 import mq as m
    return m


@pytest.fixture
def row_tile_kernel():
    lib = mq()
    assert lib.test_decode_kernel(1) == 0
    yield lib
    assert lib.test_decode_kernel(0) == 0


class Case:
    """Device operands of one decode problem and the oracle's result."""

    def __init__(self, seed, m, k, n, bits, extreme=None, zw=False, residual=False, o16=False,
                 pitch=0):
        lib = mq()
        torch = torch_cuda()
        self.c = c = synth.random_case(seed, m, k, n, bits, extreme)
        rng = np.random.default_rng(5000 + seed)
        lo, hi = (-128, 127) if bits == 8 else (-8, 7)
        self.zw = None
        if zw:
            self.zw = rng.integers(lo, hi + 1, size=n).astype(np.int32)
            self.zw[0], self.zw[-1] = lo, hi
        packed, colsum = lib.pack_weights(c.w, bits)
        row = packed.shape[1] if n else 0
        self.ldw = 0
        if pitch:   # weight rows `pitch` bytes apart inside a wider buffer
            wide = np.zeros((n, pitch), np.uint8)
            wide[:, :row] = packed
            packed, self.ldw = wide, pitch
        self.o16 = o16
        if o16:   # int16 outputs: multipliers about 2^-5, so that some saturate
            self.m0 = rng.integers(1 << 30, 1 << 31, size=n).astype(np.int32)
            self.sh = rng.integers(33, 38, size=n).astype(np.int32)
            self.zy = int(rng.integers(-300, 300))
        else:
            self.m0, self.sh = lib.requant_params(c.sw, c.sx, c.sy)
            self.zy = c.zy
        self.dev = [upload(a) for a in (c.x, packed, colsum, self.m0, self.sh)]
        self.dzw = upload(self.zw) if zw else None
        self.res = synth.residual_codes(seed, 0, m, n) if residual else None
        self.dres = upload(self.res) if residual else None
        self.y = torch.full((m, n), 77, dtype=torch.int16 if o16 else torch.int8, device="cuda")

    def desc(self, wdynamic=False):
        c = self.c
        x, packed, colsum, m0, sh = self.dev
        return mq().make_desc(x, c.zx, packed, colsum, c.N, m0, sh, self.zy, self.y, c.bits,
                              residual=self.dres, zw=self.dzw, ldw=self.ldw, wdynamic=wdynamic)

    def want(self):
        c = self.c
        packed, _ = oracle.pack(c.w, c.bits)
        if self.o16:
            return oracle.linear_o16(c.x, c.zx, packed, c.bits, c.N, self.m0, self.sh, self.zy,
                                     zw=self.zw)
        m0, sh = oracle.requant_params(c.sx, c.sw, c.sy)
        y = oracle.linear(c.x, c.zx, packed, c.bits, c.N, m0, sh, self.zy, zw=self.zw)
        if self.res is not None:
            y = oracle.residual_add(y, self.res)
        return y


def run(cases, wdynamic=False):
    torch = torch_cuda()
    lib = mq()
    for c in cases:
        c.y.fill_(77)
    descs = [c.desc(wdynamic) for c in cases]
    need = lib.workspace_size_batch(descs)
    ws = torch.zeros(max(need, 16), dtype=torch.uint8, device="cuda")
    rc = lib.linear_batch(descs, workspace=ws, ws_bytes=need)
    assert rc == 0, lib.status_string(rc)
    torch.cuda.synchronize()
    assert lib.check_device_status() == 0
    return [c.y.cpu().numpy() for c in cases]


def check(cases, what, wdynamic=False):
    for c, got in zip(cases, run(cases, wdynamic)):
        want = c.want()
        assert got.dtype == want.dtype
        if not np.array_equal(got, want):
            bad = np.argwhere(got != want)
            i = tuple(bad[0])
            raise AssertionError(f"{what}: {len(bad)} of {want.size} differ; first at {i}: "
                                 f"got {int(got[i])}, want {int(want[i])}")


# (N, K): one 8-row tile cut short, ragged tiles, rows shorter than a chunk,
# a partial last chunk (K = 5632 int4: 2816 bytes = 2 chunks + 768), many
# chunks, and K at its limit (int8: 64 chunks of 1024 bytes)
SHAPES4 = [(1, 32), (5, 64), (9, 2048), (100, 5632), (67, 1024), (24, 16384), (13, 65536)]
SHAPES8 = [(1, 16), (7, 48), (9, 1024), (100, 5632), (33, 2048), (11, 65536)]


@pytest.mark.parametrize("m", [1, 2, 3, 4])
@pytest.mark.parametrize("bits,shape", [(4, s) for s in SHAPES4] + [(8, s) for s in SHAPES8],
                         ids=lambda v: "x".join(map(str, v)) if isinstance(v, tuple) else str(v))
def test_row_tile_kernel_matches_oracle(row_tile_kernel, bits, shape, m):
    n, k = shape
    check([Case(100 + n + k % 997 + m, m, k, n, bits)], f"bits={bits} m={m} n={n} k={k}")


@pytest.mark.parametrize("bits", [4, 8])
@pytest.mark.parametrize("extreme", ["min", "max", "mixed"])
@pytest.mark.parametrize("m", [1, 2, 4])
def test_row_tile_kernel_extremes(row_tile_kernel, bits, extreme, m):
    check([Case(200 + m, m, 4096, 40, bits, extreme=extreme)], f"{extreme} bits={bits} m={m}")


@pytest.mark.parametrize("bits,k", [(4, 5632), (8, 2048), (8, 32768), (4, 65536)])
@pytest.mark.parametrize("m", [1, 2, 4])
def test_row_tile_kernel_weight_zero_points(row_tile_kernel, bits, k, m):
    check([Case(300 + k % 991 + m, m, k, 37, bits, zw=True),
           Case(310 + m, m, k, 16, bits, extreme="mixed", zw=True)], f"zw bits={bits} k={k}")


@pytest.mark.parametrize("bits", [4, 8])
def test_row_tile_kernel_int16_output_and_residual(row_tile_kernel, bits):
    check([Case(400, 1, 2048, 45, bits, zw=True, o16=True),
           Case(401, 2, 64, 300, bits, o16=True)], f"o16 bits={bits}")
    check([Case(402, 2, 5632, 50, bits, residual=True),
           Case(403, 1, 2048, 21, bits, zw=True, residual=True)], f"residual bits={bits}")
    check([Case(404, 4, 2048, 45, bits, zw=True, o16=True),
           Case(405, 3, 5632, 50, bits, residual=True)], f"four tokens bits={bits}")


def test_row_tile_kernel_pitch_and_device_written_weights(row_tile_kernel):
    cases = [Case(500, 1, 2048, 30, 4, pitch=1024 + 48), Case(501, 2, 512, 19, 8, pitch=768)]
    check(cases, "weight pitch")
    check(cases, "weights written on the device", wdynamic=True)


def test_row_tile_kernel_mixed_batch(row_tile_kernel):
    # one and two tokens, different K and N, two problems reading one input:
    # one launch of the two-token variant
    a = Case(600, 2, 2048, 70, 4)
    b = Case(601, 1, 2048, 9, 4)
    b.c.x = a.c.x[:1]
    b.dev[0] = a.dev[0][:1]
    cases = [a, b, Case(602, 1, 5632, 44, 4, zw=True), Case(603, 2, 64, 8, 4)]
    check(cases, "mixed batch")
    # up to four tokens: one launch of the four-token variant
    c = Case(604, 4, 2048, 70, 4)
    d = Case(605, 3, 2048, 9, 4)
    d.c.x = c.c.x[:3]
    d.dev[0] = c.dev[0][:3]
    check([c, d, Case(606, 1, 5632, 44, 4, zw=True), Case(607, 2, 64, 8, 4)], "mixed batch, 4")


def test_both_decode_kernels_agree_on_the_block():
    # the TinyLlama block's seven W4A8 linears at one and two tokens through
    # each decode kernel
    lib = mq()
    try:
        for m in (1, 2, 4):
            cases = [Case(700 + j, m, k, n, 4) for j, (_, k, n) in
                     enumerate(synth.TINYLLAMA_LINEARS)]
            outs = {}
            for which in (1, 2):
                assert lib.test_decode_kernel(which) == 0
                outs[which] = run(cases)
            for c, g1, g2 in zip(cases, outs[1], outs[2]):
                assert np.array_equal(g1, g2)
            for c, g in zip(cases[:2], outs[1]):
                assert_equal_int8(g, c.want(), f"block m={m}")
    finally:
        assert lib.test_decode_kernel(0) == 0
