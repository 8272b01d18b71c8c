"""The five workload configurations, end to end on the GPU against the oracle.

cfg0  one W8A8 linear, M=128, K=N=2048 (all outputs compared)
cfg1  the seven W8A8 linears of a TinyLlama-1.1B-shaped block at M=1024 in one
      batched launch (all outputs compared)
cfg2  the same block's linears as W4A8 decode at M = 1, 4, 16 (all outputs)
cfg3  the 22-layer chained W8A8 stack at M=2048 plus the 2048->32000 head:
      the oracle runs the same chain on 64 token rows spread over the 2048
      (rows are independent through the stack) from the seeded inputs, and
      every layer's seven outputs and the head are compared at those rows
cfg4  Gemma-2B-shaped W8A8 linears at M=4096 with the 2048->256000 head, and
      W4A8 decode at M=1 of the block and the head (all outputs); weights
      with 1% Student-t(3) rows
The large cases run the oracle over row blocks on every host core
(oracle.linear_mt: the same C function on disjoint row slices).
"""
import numpy as np
import pytest

import oracle
from gpu_helpers import (GpuLinear, assert_equal_int8, oracle_y, oracle_y_mt, torch_cuda, upload,
                         workspace)
from paper_2408_13933_gb300 import synth

pytestmark = pytest.mark.gpu


def mq():
    from paper_2408_13933_gb300 import mq as m
    return m


def run_batch(gls):
    assert mq().linear_batch([g.desc() for g in gls], workspace=workspace()) == 0
    return [g.result() for g in gls]


def test_config0_single_linear():
    c = synth.make_linear(0, 0, 0, "cfg0", 128, 2048, 2048, 8)
    assert_equal_int8(GpuLinear(c).run(), oracle_y(c), "cfg0")


def test_config1_tinyllama_block_prefill():
    cases = synth.block_linears(1, 1024, 8, shared_input=True)
    cases[-1].residual = synth.residual_codes(1, 0, 1024, cases[-1].N)
    outs = run_batch([GpuLinear(c) for c in cases])
    for c, got in zip(cases, outs):
        assert_equal_int8(got, oracle_y_mt(c), f"cfg1 {c.name}")


@pytest.mark.parametrize("m", [1, 4, 16])
def test_config2_tinyllama_block_decode_w4a8(m):
    cases = synth.block_linears(2, m, 4)
    outs = run_batch([GpuLinear(c) for c in cases])
    for c, got in zip(cases, outs):
        assert_equal_int8(got, oracle_y(c), f"cfg2 m={m} {c.name}")


def test_config3_chained_stack():
    torch = torch_cuda()
    m, n_layers = 2048, 22
    x0, sx0, zx0, layers, head = synth.chain_stack(3, m, n_layers)
    rows = np.unique(np.concatenate([np.linspace(0, m - 1, 62).round().astype(np.int64),
                                     [1337, 2047]]))
    lib = mq()

    def prep(c):
        packed, colsum = lib.pack_weights(c.w, 8)
        m0, sh = lib.requant_params(c.sw, c.sx, c.sy)
        return [upload(a) for a in (packed, colsum, m0, sh)]

    x = upload(x0)
    gpu_rows = []   # per layer: {name: y[rows]}
    for L in layers:
        dev = {c.name: prep(c) for c in L.cases}
        out = {c.name: torch.empty((m, c.N), dtype=torch.int8, device="cuda") for c in L.cases}
        res = upload(L.residual)

        def desc(c, xin, residual=None):
            p = dev[c.name]
            return lib.make_desc(xin, c.zx, p[0], p[1], c.N, p[2], p[3], c.zy, out[c.name], 8,
                                 residual=residual)
        first = [desc(c, x) for c in L.cases if c.name in ("q", "k", "v", "gate", "up")]
        assert lib.linear_batch(first, workspace=workspace()) == 0
        cs = {c.name: c for c in L.cases}
        second = [desc(cs["o"], out["q"]), desc(cs["down"], out["up"], residual=res)]
        assert lib.linear_batch(second, workspace=workspace()) == 0
        torch.cuda.synchronize()
        assert lib.check_device_status() == 0
        gpu_rows.append({k: v[rows].cpu().numpy() for k, v in out.items()})
        x = out["down"]
    hp = prep(head)
    hy = torch.empty((m, head.N), dtype=torch.int8, device="cuda")
    assert lib.linear_batch([lib.make_desc(x, head.zx, hp[0], hp[1], head.N, hp[2], hp[3],
                                           head.zy, hy, 8)]) == 0
    torch.cuda.synchronize()
    head_rows = hy[rows].cpu().numpy()

    # the oracle runs the same chain on the sampled rows from the seeded inputs
    def olin(c, xin):
        packed, _ = oracle.pack(c.w, 8)
        m0, sh = oracle.requant_params(c.sx, c.sw, c.sy)
        return oracle.linear_mt(xin, c.zx, packed, 8, c.N, m0, sh, c.zy)
    xr = np.ascontiguousarray(x0[rows])
    for li, L in enumerate(layers):
        cs = {c.name: c for c in L.cases}
        ys = {}
        for name in ("q", "k", "v", "gate", "up"):
            ys[name] = olin(cs[name], xr)
        ys["o"] = olin(cs["o"], ys["q"])
        ys["down"] = oracle.residual_add(olin(cs["down"], ys["up"]),
                                         np.ascontiguousarray(L.residual[rows]))
        for name, y in ys.items():
            assert_equal_int8(gpu_rows[li][name], y, f"cfg3 layer {li} {name}")
        xr = ys["down"]
    assert_equal_int8(head_rows, olin(head, xr), "cfg3 head")


def test_config4_gemma_prefill():
    cases = synth.block_linears(4, 4096, 8, shapes=synth.GEMMA_LINEARS, t_rows_frac=0.01,
                                shared_input=True)
    hk, hn = synth.GEMMA_HEAD[1], synth.GEMMA_HEAD[2]
    head = synth.make_linear(4, 0, 7, "head", 4096, hk, hn, 8, t_rows_frac=0.01)
    outs = run_batch([GpuLinear(c) for c in cases])
    for c, got in zip(cases, outs):
        assert_equal_int8(got, oracle_y_mt(c), f"cfg4 {c.name}")
    del outs
    got = GpuLinear(head).run()
    assert_equal_int8(got, oracle_y_mt(head), "cfg4 head")


def test_config4_gemma_decode_w4a8():
    cases = synth.block_linears(4, 1, 4, shapes=synth.GEMMA_LINEARS, layer=1, t_rows_frac=0.01)
    hk, hn = synth.GEMMA_HEAD[1], synth.GEMMA_HEAD[2]
    cases.append(synth.make_linear(4, 1, 7, "head", 1, hk, hn, 4, t_rows_frac=0.01))
    outs = run_batch([GpuLinear(c) for c in cases])
    for c, got in zip(cases, outs):
        assert_equal_int8(got, oracle_y(c), f"cfg4 decode {c.name}")
