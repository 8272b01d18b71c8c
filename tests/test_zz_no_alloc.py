"""mq_linear_w4a8_noalloc on the GPU against mq_linear_w4a8 (the workspace
entry point) and against the oracle: two calls in a row through the
library's static scratch give the workspace path's output and the oracle's
byte for byte, and allocate no device memory (neither through PyTorch's
caching allocator nor behind it: the device's free memory is unchanged).
The file name sorts last, so in a full run these tests also run after every
other GPU test."""
import copy

import numpy as np
import pytest

from gpu_helpers import oracle_y, torch_cuda, upload, workspace
from paper_2408_13933_gb300 import synth

pytestmark = pytest.mark.gpu

# (M, N, K): split 64-row units (K spread over many CTAs), full decode batch,
# a ragged M and N, one stage per unit, K = 0 (outputs are zy)
CASES = [(1, 256, 5632), (16, 2048, 2048), (7, 320, 4096), (1, 200, 64), (3, 96, 0)]


def mq():
    from paper_2408_13933_gb300 import mq as m
    return m


def prepare(m, n, k, seed):
    lib = mq()
    c = synth.random_case(seed, m, max(k, 32), n, 4)
    x = upload(c.x[:, :k] if k else np.zeros((m, 16), np.int8))
    w = c.w[:, :k] if k else np.zeros((n, 0), np.int8)
    packed, colsum = lib.pack_weights(np.ascontiguousarray(w), 4)
    m0, sh = lib.requant_params(c.sw, c.sx, c.sy)
    return c, x, upload(packed), upload(colsum), upload(m0), upload(sh)


def oracle_of(c, k):
    """The oracle's output of the case cut to its first k input features."""
    o = copy.copy(c)
    o.x = np.ascontiguousarray(c.x[:, :k])
    o.w = np.ascontiguousarray(c.w[:, :k])
    return oracle_y(o)


@pytest.mark.parametrize("m,n,k", CASES)
def test_noalloc_matches_workspace_entry_on_two_calls(m, n, k):
    torch = torch_cuda()
    lib = mq()
    c, x, packed, colsum, m0, sh = prepare(m, n, k, seed=700 + m + n)
    ys = [torch.full((m, n), 77, dtype=torch.int8, device="cuda") for _ in range(3)]
    assert lib.linear(x, c.zx, packed, colsum, n, m0, sh, c.zy, ys[0], 4, k=k,
                      workspace=workspace()) == 0
    torch.cuda.synchronize()
    before = torch.cuda.memory_allocated()
    free_before = torch.cuda.mem_get_info()[0]
    for y in ys[1:]:   # back to back on one stream, no synchronisation between
        assert lib.linear_w4a8_noalloc(x, c.zx, packed, colsum, n, m0, sh, c.zy, y, k=k) == 0
    torch.cuda.synchronize()
    assert lib.check_device_status() == 0
    assert torch.cuda.memory_allocated() == before
    assert torch.cuda.mem_get_info()[0] == free_before
    want = ys[0].cpu().numpy()
    assert np.array_equal(want, oracle_of(c, k)), "workspace entry point differs from the oracle"
    for i, y in enumerate(ys[1:]):
        got = y.cpu().numpy()
        assert np.array_equal(got, want), f"call {i + 1}: {int(np.sum(got != want))} differ"


def test_noalloc_rejects_more_tokens_than_its_scratch_holds():
    torch = torch_cuda()
    lib = mq()
    c, x, packed, colsum, m0, sh = prepare(17, 64, 64, seed=717)
    y = torch.full((17, 64), 77, dtype=torch.int8, device="cuda")
    assert lib.linear_w4a8_noalloc(x, c.zx, packed, colsum, 64, m0, sh, c.zy,
                                   y) == lib.MQ_ERR_UNSUPPORTED_SHAPE
    torch.cuda.synchronize()
    assert bool((y == 77).all())   # nothing was launched
