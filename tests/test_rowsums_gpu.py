"""Descriptors without colsum (int8 weights): the token-major kernel folds both
zero points and reads no row sums, every other kernel gets them computed by
the call into its workspace.  Both routes against the oracle (8- and 16-bit
activations, prefill and decode shapes, with and without weight zero points),
the workspace accounting, one row-sum job per distinct weight matrix, and the
argument checks (int4 weights, the single-linear calls)."""
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
def restore_hook():
    yield
    assert mq().test_tmajor_kernel(0) == 0


class Case:
    def __init__(self, seed, m, k, n, zw=False, a16=False, share=None):
        torch = torch_cuda()
        lib = mq()
        gen = synth.random_case_a16 if a16 else synth.random_case
        self.c = c = gen(seed, m, k, n, 8)
        self.a16 = a16
        if share is not None:  # the weights of another case (same device buffer)
            c.w, c.sw = share.c.w, share.c.sw
        rng = np.random.default_rng(300 + seed)
        self.zw = rng.integers(-128, 128, size=n).astype(np.int32) if zw else None
        packed, _ = lib.pack_weights(c.w, 8)
        m0, sh = lib.requant_params(c.sw, c.sx, c.sy)
        self.m0, self.sh = m0, sh
        self.dev = [upload(a) for a in (c.x, packed, m0, sh)]
        if share is not None:
            self.dev[1] = share.dev[1]
        self.dzw = upload(self.zw) if zw else None
        self.y = torch.full((m, n), 77, dtype=torch.int16 if a16 else torch.int8, device="cuda")

    def desc(self):
        c = self.c
        x, packed, m0, sh = self.dev
        return mq().make_desc(x, c.zx, packed, None, c.N, m0, sh, c.zy, self.y, 8, zw=self.dzw)

    def want(self):
        c = self.c
        packed, _ = oracle.pack(c.w, 8)
        if self.a16:
            return oracle.linear_a16(c.x, c.zx, packed, 8, c.N, self.m0, self.sh, c.zy, zw=self.zw)
        return oracle.linear(c.x, c.zx, packed, 8, c.N, self.m0, self.sh, c.zy, zw=self.zw)


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
    return need


@pytest.mark.parametrize("mode", [0, 2], ids=["auto", "no_tmajor"])
def test_row_sums_derived_by_the_call(mode):
    # short K (token-major in auto mode), few channels, a plain prefill shape,
    # decode shapes, 16-bit activations, with and without zero points
    assert mq().test_tmajor_kernel(mode) == 0
    cases = [Case(1, 300, 64, 200, zw=True), Case(2, 130, 1024, 64, zw=True),
             Case(3, 260, 512, 300), Case(4, 4, 2048, 96, zw=True), Case(5, 1, 512, 80),
             Case(6, 200, 256, 160, a16=True), Case(7, 3, 256, 64, zw=True, a16=True)]
    run(cases)
    for i, c in enumerate(cases):
        got = c.y.cpu().numpy()
        want = c.want()
        assert np.array_equal(got, want), f"case {i}: {int((got != want).sum())} differ"


def test_row_sum_workspace():
    # the token-major route needs no row sums; other kernels take 4 N bytes
    # (to 128) per distinct weight matrix, shared weights counted once
    lib = mq()
    a = Case(11, 300, 64, 200)
    b = Case(12, 300, 64, 200, share=a)
    assert lib.test_tmajor_kernel(0) == 0
    auto = lib.workspace_size_batch([a.desc(), b.desc()])
    assert lib.test_tmajor_kernel(2) == 0
    never = lib.workspace_size_batch([a.desc(), b.desc()])
    assert never - auto >= 4 * 200 and never - auto <= 4 * 200 + 256
    run([a, b])  # mode 2: one row-sum job for the shared weights
    for c in (a, b):
        assert np.array_equal(c.y.cpu().numpy(), c.want())


def test_colsum_required_where_it_cannot_be_derived():
    lib = mq()
    torch = torch_cuda()
    c = synth.random_case(21, 40, 256, 64, 4)
    packed, _ = lib.pack_weights(c.w, 4)
    m0, sh = lib.requant_params(c.sw, c.sx, c.sy)
    x, p, m0d, shd = (upload(a) for a in (c.x, packed, m0, sh))
    y = torch.zeros((40, 64), dtype=torch.int8, device="cuda")
    d = lib.make_desc(x, c.zx, p, None, 64, m0d, shd, c.zy, y, 4)  # int4 weights
    ws = torch.zeros(1 << 22, dtype=torch.uint8, device="cuda")
    assert lib.linear_batch([d], workspace=ws, ws_bytes=ws.numel()) == lib.MQ_ERR_INVALID_ARG
    c8 = synth.random_case(22, 40, 256, 64, 8)
    p8, _ = lib.pack_weights(c8.w, 8)
    rc = lib.lib.mq_linear_w8a8(upload(c8.x).data_ptr(), 40, 256, 256, c8.zx,
                                upload(p8).data_ptr(), None, 64, m0d.data_ptr(), shd.data_ptr(),
                                c8.zy, y.data_ptr(), 64, ws.data_ptr(), ws.numel(), None)
    assert rc == lib.MQ_ERR_INVALID_ARG
