"""Split K for prefill calls that would leave most SMs idle (one M = 128
linear makes 8 pair tiles): S slices of K on the token-major kernel, each
writing raw int32 sums into the workspace, then one combine launch that
requantizes.  Against the oracle: the config-0 shape, zero points, the
residual, an int16 output, ragged N and K, several problems in one call; the
workspace accounting; and that the call without that workspace (or with a
prefill kernel forced) runs unsplit, with the same bytes."""
import numpy as np
import pytest

from gpu_helpers import torch_cuda
from test_tmajor_gpu import Case, assert_equal

pytestmark = pytest.mark.gpu


def mq():
    from paper_2408_13933_gb300 import mq as m
    return m


@pytest.fixture(autouse=True)
def auto_choice():
    lib = mq()
    assert lib.test_tmajor_kernel(0) == 0 and lib.test_prefill_kernel(0) == 0
    yield
    assert lib.test_tmajor_kernel(0) == 0 and lib.test_prefill_kernel(0) == 0


def run(cases, ws_bytes=None):
    torch = torch_cuda()
    lib = mq()
    descs = [c.desc() for c in cases]
    need = lib.workspace_size_batch(descs) if ws_bytes is None else ws_bytes
    ws = torch.zeros(max(need, 16), dtype=torch.uint8, device="cuda")
    assert lib.linear_batch(descs, workspace=ws, ws_bytes=need) == 0
    torch.cuda.synchronize()
    assert lib.check_device_status() == 0


@pytest.mark.parametrize("spec", [
    (128, 2048, 2048, False, False, False),   # config 0's shape
    (200, 300, 1024, True, False, False),     # zero points, ragged tokens and channels
    (130, 100, 2048, True, True, False),      # residual
    (64, 512, 4096, True, False, True),       # int16 output
    (96, 200, 1088, False, False, False),     # K not a multiple of the slice
], ids=lambda s: "x".join(map(str, s[:3])) + ("-zw" if s[3] else "") + ("-res" if s[4] else "")
                 + ("-o16" if s[5] else ""))
def test_split_k_single(spec):
    m, n, k, zw, res, o16 = spec
    c = Case(m + n + k, m, k, n, zw=zw, residual=res, o16=o16)
    need = mq().workspace_size_batch([c.desc()])
    assert need > 4 * m * n * 2, "the split's partial sums are counted"
    run([c])
    assert_equal(c.got(), c.want(), f"split {spec}")


def test_split_k_batch_of_small_problems():
    cases = [Case(900 + i, 40 + 37 * i, 512 * (1 + i % 3), (256, 96, 320)[i % 3], zw=i % 2 == 0)
             for i in range(4)]
    run(cases)
    for i, c in enumerate(cases):
        assert_equal(c.got(), c.want(), f"batch problem {i}")


def test_unsplit_without_room_or_with_a_forced_kernel():
    lib = mq()
    a = Case(77, 128, 2048, 2048, zw=True)
    run([a], ws_bytes=0)  # no workspace: the 128-token kernel
    unsplit = a.got().copy()
    assert_equal(unsplit, a.want(), "unsplit")
    assert lib.test_prefill_kernel(2) == 0  # a forced prefill kernel: no split
    assert lib.workspace_size_batch([a.desc()]) == 0
    run([a])
    assert_equal(a.got(), unsplit, "forced 128-token kernel")
    assert lib.test_prefill_kernel(0) == 0
    run([a])
    assert_equal(a.got(), unsplit, "split")
