"""Shared helpers for the GPU parity tests: run one synthetic case through the
C-ABI (libmq) and through the oracle, each with its own packing and
requantization parameters."""
from __future__ import annotations

import numpy as np

import oracle


def torch_cuda():
    import torch
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    return torch


_WS = None
# room for the 256-token prefill kernel's widened inputs of every shape the
# tests run through this workspace (2 M K + 4 M bytes after the decode region)
WS_BYTES = 256 << 20


def workspace():
    """One zero-filled workspace shared by the tests: the decode region (left
    zero-filled by every call) and room for widened prefill inputs (scratch)."""
    global _WS
    if _WS is None:
        torch = torch_cuda()
        from paper_2408_13933_gb300 import mq
        _WS = torch.zeros(max(WS_BYTES, mq.workspace_size(1, 1, 0, 4)), dtype=torch.uint8,
                          device="cuda")
    return _WS


def decode_region():
    """The decode region of the shared workspace (zero-filled between calls)."""
    from paper_2408_13933_gb300 import mq
    return workspace()[:mq.workspace_size(1, 1, 0, 4)]


def upload(a: np.ndarray):
    torch = torch_cuda()
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


class GpuLinear:
    """Device-resident operands of one case, prepared through libmq."""

    def __init__(self, case, device_pack: bool = False, ldy: int | None = None):
        from paper_2408_13933_gb300 import mq
        torch = torch_cuda()
        self.mq = mq
        self.case = case
        self.x = upload(case.x)
        if device_pack:
            self.packed, self.colsum = mq.pack_weights(upload(case.w), case.bits)
        else:
            p, cs = mq.pack_weights(case.w, case.bits)
            self.packed, self.colsum = upload(p), upload(cs)
        m0, sh = mq.requant_params(case.sw, case.sx, case.sy)
        self.m0, self.shift = upload(m0), upload(sh)
        self.ldy = ldy if ldy is not None else max(case.N, 1)
        self.y = torch.full((case.M, self.ldy), 77, dtype=torch.int8, device="cuda")
        self.residual = upload(case.residual) if case.residual is not None else None

    def desc(self):
        c = self.case
        return self.mq.make_desc(self.x, c.zx, self.packed, self.colsum, c.N, self.m0, self.shift,
                                 c.zy, self.y, c.bits, residual=self.residual, ldy=self.ldy)

    def run(self) -> np.ndarray:
        c = self.case
        rc = self.mq.linear(self.x, c.zx, self.packed, self.colsum, c.N, self.m0, self.shift, c.zy,
                            self.y, c.bits, ldy=self.ldy, workspace=workspace())
        assert rc == 0, self.mq.status_string(rc)
        return self.result()

    def result(self) -> np.ndarray:
        torch = torch_cuda()
        torch.cuda.synchronize()
        assert self.mq.check_device_status() == 0
        return self.y.cpu().numpy()


def oracle_y(case) -> np.ndarray:
    packed, _ = oracle.pack(case.w, case.bits)
    m0, sh = oracle.requant_params(case.sx, case.sw, case.sy)
    y = oracle.linear(case.x, case.zx, packed, case.bits, case.N, m0, sh, case.zy)
    if case.residual is not None:
        y = oracle.residual_add(y, case.residual)
    return y


def oracle_y_mt(case) -> np.ndarray:
    """oracle_y computed on every host core (the oracle over row blocks)."""
    packed, _ = oracle.pack(case.w, case.bits)
    m0, sh = oracle.requant_params(case.sx, case.sw, case.sy)
    y = oracle.linear_mt(case.x, case.zx, packed, case.bits, case.N, m0, sh, case.zy)
    if case.residual is not None:
        y = oracle.residual_add(y, case.residual)
    return y


def oracle_points(case, pts: np.ndarray):
    packed, _ = oracle.pack(case.w, case.bits)
    m0, sh = oracle.requant_params(case.sx, case.sw, case.sy)
    y, _ = oracle.linear_points(case.x, case.zx, packed, case.bits, case.N, m0, sh, case.zy, pts)
    return y


def assert_equal_int8(got: np.ndarray, want: np.ndarray, what: str):
    if not np.array_equal(got, want):
        bad = np.argwhere(got != want)
        i = tuple(bad[0])
        raise AssertionError(f"{what}: {len(bad)} of {want.size} outputs differ; first at {i}: "
                             f"got {int(got[i])}, want {int(want[i])}")


def sample_points(m: int, n: int, rng: np.random.Generator, count: int = 2048,
                  full_rows=(0,), full_cols=(0,)) -> np.ndarray:
    pts = [(r, c) for r in full_rows if r < m for c in range(n)]
    pts += [(r, c) for c in full_cols if c < n for r in range(m)]
    pts += [(int(rng.integers(0, m)), int(rng.integers(0, n))) for _ in range(count)]
    pts += [(m - 1, n - 1), (m - 1, 0), (0, n - 1)]
    return np.array(pts, np.int64)
