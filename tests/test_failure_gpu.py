"""Failure detection on the GPU without a fault: a bounded device wait that
runs out, reported through the device status word, with the CUDA context
still usable afterwards.

The decode kernel combines a 64-row unit whose k range is split among CTAs
in the unit's first CTA, which waits (bounded) for the later CTAs' partial
sums.  The test hook mq_test_skip_partials makes one of those CTAs skip its
store -- a split-K partner that never delivers -- and mq_set_wait_limit_ns
shortens the wait to a few milliseconds.  The launch must then report
MQ_ERR_DEVICE_TIMEOUT, and the next launches, with the hook off, must be
bit-exact against the oracle again (also without clearing the workspace:
every launch tags its partial sums with its own number).
"""
import numpy as np
import pytest

from gpu_helpers import oracle_y, torch_cuda, upload
from paper_2408_13933_gb300 import synth

pytestmark = pytest.mark.gpu

SHORT_NS = 2_000_000  # 2 ms


def mq():
    from paper_2408_13933_gb300 import mq as m
    return m


def prepare(m, n, k, bits, seed):
    lib = mq()
    c = synth.random_case(seed, m, k, n, bits)
    packed, colsum = lib.pack_weights(c.w, bits)
    m0, sh = lib.requant_params(c.sw, c.sx, c.sy)
    return c, [upload(a) for a in (c.x, packed, colsum, m0, sh)]


@pytest.fixture
def hooks():
    # the split-K decode kernel (the one with a partner to wait for)
    lib = mq()
    assert lib.test_decode_kernel(2) == 0
    yield lib
    assert lib.test_skip_partials(-1) == 0
    assert lib.set_wait_limit_ns(0) == 0
    assert lib.test_decode_kernel(0) == 0


# One 64-row unit with 16 (int4) or 32 (int8) stages: the decode grid has one
# CTA per stage, CTA 0 finishes the unit and CTAs 1.. contribute.
@pytest.mark.parametrize("m,k,bits", [(1, 4096, 4), (16, 4096, 4), (3, 4096, 8)])
def test_missing_partner_times_out_and_next_launch_is_exact(hooks, m, k, bits):
    torch = torch_cuda()
    lib = hooks
    n = 64
    c, (x, packed, colsum, m0, sh) = prepare(m, n, k, bits, seed=900 + m + bits)
    ws = torch.zeros(lib.workspace_size(m, n, k, bits), dtype=torch.uint8, device="cuda")
    y = torch.full((m, n), 77, dtype=torch.int8, device="cuda")
    want = oracle_y(c)

    assert lib.check_device_status() == 0
    assert lib.set_wait_limit_ns(SHORT_NS) == 0
    assert lib.test_skip_partials(1) == 0
    assert lib.linear(x, c.zx, packed, colsum, n, m0, sh, c.zy, y, bits, workspace=ws) == 0
    torch.cuda.synchronize()
    assert lib.check_device_status() == lib.MQ_ERR_DEVICE_TIMEOUT
    assert lib.check_device_status() == 0   # reading the status clears it

    assert lib.test_skip_partials(-1) == 0
    assert lib.set_wait_limit_ns(0) == 0
    for _ in range(2):   # the workspace still holds the timed-out launch's entries
        y.fill_(77)
        assert lib.linear(x, c.zx, packed, colsum, n, m0, sh, c.zy, y, bits, workspace=ws) == 0
        torch.cuda.synchronize()
        assert lib.check_device_status() == 0
        got = y.cpu().numpy()
        assert np.array_equal(got, want), f"{int(np.sum(got != want))} outputs differ"


def test_noalloc_entry_recovers_after_a_timeout(hooks):
    torch = torch_cuda()
    lib = hooks
    m, n, k = 2, 64, 4096
    c, (x, packed, colsum, m0, sh) = prepare(m, n, k, 4, seed=931)
    y = torch.full((m, n), 77, dtype=torch.int8, device="cuda")
    assert lib.set_wait_limit_ns(SHORT_NS) == 0
    assert lib.test_skip_partials(3) == 0
    assert lib.linear_w4a8_noalloc(x, c.zx, packed, colsum, n, m0, sh, c.zy, y) == 0
    torch.cuda.synchronize()
    assert lib.check_device_status() == lib.MQ_ERR_DEVICE_TIMEOUT
    assert lib.test_skip_partials(-1) == 0
    assert lib.set_wait_limit_ns(0) == 0
    y.fill_(77)
    assert lib.linear_w4a8_noalloc(x, c.zx, packed, colsum, n, m0, sh, c.zy, y) == 0
    torch.cuda.synchronize()
    assert lib.check_device_status() == 0
    assert np.array_equal(y.cpu().numpy(), oracle_y(c))
