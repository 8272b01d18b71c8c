#!/usr/bin/env python
"""Benchmark of the integer-only quantized linear layer (MobileQuant W8A8 / W4A8).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl mq|reference]

Headline workload (the largest single-GPU configuration): a 22-layer
TinyLlama-1.1B-shaped stack of W8A8 linears at prefill M = 2048 tokens plus
the 2048 -> 32000 head.  Per layer: q 2048->2048, k/v 2048->256, gate/up
2048->5632 read x_l; o 2048->2048 reads q's int8 output and down 5632->2048
reads up's; x_{l+1} = sat8(down + r_l) with a seeded int8 residual, fused
into down's epilogue.  One step = the whole stack = 45 batched libmq calls
(two per layer + the head), each one launch of the tcgen05 prefill kernel;
4.24 T int8 ops and 1.03 GB of int8 weights per step.  `e2e` repeats it with
x_0 uploaded from pinned host memory and the head's output downloaded every
step.

Reported beside it, measured in the same run: config 0 (one M = 128 linear),
config 1 (the TinyLlama block at M = 1024, one launch), config 2 (W4A8 decode
of that block at M = 1, 4, 16, weight GB/s over 12 rotated layers), config 4
(the Gemma-2B-shaped block and its 256000-wide head: W8A8 prefill at M = 4096
and W4A8 decode at M = 1); asymmetric weights in the paper's settings; the
16-bit-activation baselines W8A16 / W4A16; one layer's attention matmuls at
T = 1024 (also in the W8A16 setting); the boundary quantizers; and the
offline weight pipeline.  The oracle re-computes every leg's parity sample
in the cpu_baseline leg (rank 0, one GPU), where it is also timed on all
host cores on a sample of the headline stack.

Multi-GPU (torchrun, one rank per GPU): replicas only -- every rank runs the
same workload on its own GPU, no collective on the data path; value is the
total over ranks divided by the slowest rank's time.

--impl reference runs the CPU oracle (oracle/, plain C, row blocks on every
host core) on a bounded sample of the same workload: each step runs a few
token rows of the stack through all 22 layers and the head.
"""
from __future__ import annotations

import argparse
import ctypes
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2408_13933_gb300 import synth  # noqa: E402

METRIC = "W8A8 prefill int8 TOPS (% of tensor peak); W4A8 decode weight GB/s (% HBM)"
PREFILL_M = 1024
PREFILL_LAYERS = 3
DECODE_LAYERS = 12
DECODE_MS = (1, 4, 16)
STACK_M, STACK_LAYERS = 2048, 22
CONFIG_ID_PREFILL = 1
CONFIG_ID_DECODE = 2
CONFIG_ID_STACK = 3
CONFIG_ID_GEMMA = 4
WORKLOAD = "tinyllama-1.1b-shaped-22-layer-w8a8-stack-m2048-plus-head"
BLOCK_WORKLOAD = "tinyllama-1.1b-block-w8a8-prefill-m1024"


# DRAM traffic (dram__bytes_read.sum + dram__bytes_write.sum) of the 256-token prefill kernel,
# from one-pass ncu captures (`--profile block` / `--profile stack`, summaries under profiles/):
# per launch on the config-1 block, and summed over the 45 launches of one headline-stack step
# (whose writes include the f16 copies of the chained outputs that leave L2 during the step).
# ncu flushes the caches before every captured launch, so the f16 token copies that the pre-pass
# has just written are read back from DRAM there (in the pipelined run they come from L2).
# Valid only for the kernel sources they were taken on: reported as null once those change.
PREFILL_TRAFFIC_BYTES = 66_821_376 + 1_439_402
PREFILL_TRAFFIC_SOURCES = ("mq_prefill2.cu", "mq_ptx.cuh", "mq_internal.h")
PREFILL_TRAFFIC_SHA = "448729e90029a98d"


def prefill_traffic():
    return PREFILL_TRAFFIC_BYTES if sources_sha() == PREFILL_TRAFFIC_SHA else None


STACK_TRAFFIC_BYTES = 2_029_162_240 + 332_227_840
STACK_TRAFFIC_SHA = PREFILL_TRAFFIC_SHA


def sources_sha() -> str:
    import hashlib
    h = hashlib.sha256()
    for f in PREFILL_TRAFFIC_SOURCES:
        with open(os.path.join(ROOT, "paper_2408_13933_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def stack_traffic():
    return STACK_TRAFFIC_BYTES if STACK_TRAFFIC_SHA and sources_sha() == STACK_TRAFFIC_SHA else None


def block_ops(m: int) -> int:
    return sum(2 * m * k * n for _, k, n in synth.TINYLLAMA_LINEARS)


def block_weight_bytes(bits: int) -> int:
    return sum(k * n * bits // 8 for _, k, n in synth.TINYLLAMA_LINEARS)


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        return {"hbm_gbs": float(p["hbm_gbs"]), "bf16_tflops": float(p["bf16_tflops"]),
                "bf16_tflops_sustained": float(p.get("bf16_tflops_sustained", p["bf16_tflops"])),
                "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
            "source": "fallback"}


# --------------------------------------------------------------------------- dist
def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


class Dist:
    """One process per GPU, replicas only: a barrier and the maximum over
    ranks (for the slowest rank's time); no collective touches the data path.
    The backend is NCCL on GPUs, gloo otherwise (host-side tests)."""

    def __init__(self, world: int, rank: int, local: int, backend: str | None = None):
        self.world, self.rank, self.local = world, rank, local
        self.pg = None
        self.device = "cpu"
        if world > 1:
            import torch
            import torch.distributed as dist
            backend = backend or ("nccl" if torch.cuda.is_available() else "gloo")
            if backend == "nccl":
                torch.cuda.set_device(local)
                dist.init_process_group("nccl", device_id=torch.device("cuda", local))
                self.device = "cuda"
            else:
                dist.init_process_group("gloo", rank=rank, world_size=world)
            self.pg = dist

    def barrier(self):
        if self.pg is not None:
            self.pg.barrier()

    def max(self, v: float) -> float:
        if self.pg is None:
            return v
        import torch
        t = torch.tensor([v], dtype=torch.float64, device=self.device)
        self.pg.all_reduce(t, op=self.pg.ReduceOp.MAX)
        return float(t.item())

    def close(self):
        if self.pg is not None:
            self.pg.destroy_process_group()


def whole_job_rate(units_per_rank: float, world: int, max_ms: float) -> float:
    """Units per second of the whole job: every rank's units over the
    slowest rank's time (weak scaling: each rank runs the full workload)."""
    return units_per_rank * world / (max_ms * 1e-3)


# --------------------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi sampling (every 100 ms) while the timed region runs."""
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.proc = None
        self.t0 = self.t1 = None
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(gpu_index), f"--query-gpu=timestamp,{self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None

    def start(self):
        self.t0 = time.time()

    def stop(self):
        self.t1 = time.time()

    def result(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.25)
        self.proc.terminate()
        out, _ = self.proc.communicate(timeout=5)
        rows = []
        for line in out.strip().splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                ts = time.mktime(time.strptime(parts[0].split(".")[0], "%Y/%m/%d %H:%M:%S"))
                rows.append((ts, float(parts[1]), float(parts[2]), parts[3:]))
            except ValueError:
                continue
        inside = [r for r in rows if self.t0 - 1 <= r[0] <= self.t1 + 1]
        use = inside if inside else rows
        if not use:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in use for i, v in enumerate(r[3][2:6])
                          if v.strip().lower() == "active"})
        return {"sm_mhz": statistics.median(r[1] for r in use),
                "sm_max_mhz": max(r[2] for r in use), "reasons": reasons,
                "samples": len(use), "samples_in_region": len(inside)}


# --------------------------------------------------------------------------- workload
class PrefillBlock:
    """Device-resident operands of one layer's seven W8A8 linears at M tokens
    (with asym, asymmetric weights in the paper's W8A8 setting)."""

    def __init__(self, mq, torch, layer: int, m: int, asym: bool = False):
        self.cases = synth.block_linears(CONFIG_ID_PREFILL, m, 8, layer=layer, shared_input=True,
                                         asym=asym)
        down = self.cases[-1]
        down.residual = synth.residual_codes(CONFIG_ID_PREFILL, layer, m, down.N)
        dev = "cuda"
        # distinct inputs (the shared x of q/k/v/gate/up, o's input, down's
        # input) as views of one device buffer, mirrored by one pinned host
        # buffer, so that a step uploads them with one copy; the outputs alike
        xs = []
        for c in self.cases:
            if all(c.x is not a for a in xs):
                xs.append(c.x)
        self.x_all_host = torch.from_numpy(np.concatenate([a.reshape(-1) for a in xs])).pin_memory()
        self.x_all = self.x_all_host.to(dev)
        self.x_dev, off = {}, 0
        for a in xs:
            self.x_dev[id(a)] = self.x_all[off:off + a.size].view(a.shape)
            off += a.size
        self.y_all = torch.empty(sum(m * c.N for c in self.cases), dtype=torch.int8, device=dev)
        self.y_all_host = torch.empty(self.y_all.numel(), dtype=torch.int8).pin_memory()
        self.descs, self.y, self.keep = [], [], []
        yoff = 0
        for c in self.cases:
            packed, colsum = mq.pack_weights(c.w, 8)
            m0, sh = mq.requant_params(c.sw, c.sx, c.sy)
            t = [torch.from_numpy(a).to(dev) for a in (packed, colsum, m0, sh)]
            t.append(mq.weight_sq_sums(t[0], c.N, c.K, 8))
            y = self.y_all[yoff:yoff + m * c.N].view(m, c.N)
            yoff += m * c.N
            res = torch.from_numpy(c.residual).to(dev) if c.residual is not None else None
            zw = torch.from_numpy(c.zw).to(dev) if c.zw is not None else None
            self.keep += t + [a for a in (res, zw) if a is not None]
            self.y.append(y)
            self.descs.append(mq.make_desc(self.x_dev[id(c.x)], c.zx, t[0], t[1], c.N, t[2], t[3],
                                           c.zy, y, 8, residual=res, zw=zw, wsq=t[4]))
        self.arr = (mq.LinearDesc * len(self.descs))(*self.descs)
        # decode shapes need the decode region; prefill (asymmetric or not) nothing
        self.ws_bytes = mq.workspace_size_batch(self.descs)
        self.ws = torch.zeros(max(16, self.ws_bytes), dtype=torch.uint8, device=dev)
        self.wsp = self.ws.data_ptr() if self.ws_bytes else None
        self.h2d_bytes = self.x_all.numel()
        self.d2h_bytes = self.y_all.numel()


class DecodeLayer:
    """One layer's seven W4A8 linears, uploaded once; descriptors for each
    decode width M use the first M rows of a 16-row seeded input."""

    def __init__(self, mq, torch, layer: int, asym: bool = False, ms=DECODE_MS, a16: bool = False):
        if a16:  # 16-bit activations and outputs (W4A16)
            cases = synth.block_linears_a16(CONFIG_ID_DECODE, max(ms), 4, layer=layer)
        else:
            cases = synth.block_linears(CONFIG_ID_DECODE, max(ms), 4, layer=layer, asym=asym)
        self.arr, self.keep = {}, []
        dev = []
        for c in cases:
            packed, colsum = mq.pack_weights(c.w, 4)
            m0, sh = mq.requant_params(c.sw, c.sx, c.sy)
            t = [torch.from_numpy(a).cuda() for a in (c.x, packed, colsum, m0, sh)]
            t.append(torch.from_numpy(c.zw).cuda() if c.zw is not None else None)
            self.keep += [a for a in t if a is not None]
            dev.append((c, t))
        for m in ms:
            descs = []
            for c, t in dev:
                y = torch.empty((m, c.N), dtype=torch.int16 if a16 else torch.int8, device="cuda")
                self.keep.append(y)
                descs.append(mq.make_desc(t[0], c.zx, t[1], t[2], c.N, t[3], t[4], c.zy, y, 4,
                                          m=m, zw=t[5]))
            self.arr[m] = (mq.LinearDesc * len(descs))(*descs)
        self.count = len(cases)


def run_prefill(mq, torch, dist: Dist, steps: int, warmup: int):
    """Config 1: the TinyLlama-shaped block's seven W8A8 linears at M = 1024,
    one batched launch per step, rotating over three layers."""
    blocks = [PrefillBlock(mq, torch, layer, PREFILL_M) for layer in range(PREFILL_LAYERS)]
    stream = torch.cuda.current_stream()
    sp = stream.cuda_stream
    call = mq.lib.mq_linear_batch

    def step(i):
        b = blocks[i % len(blocks)]
        rc = call(b.arr, len(b.descs), b.wsp, b.ws_bytes, sp)
        if rc:
            raise RuntimeError(f"mq_linear_batch failed: {mq.status_string(rc)}")

    for i in range(warmup):
        step(i)
    torch.cuda.synchronize()
    if mq.check_device_status() != 0:
        raise RuntimeError("device status error after warm-up")
    # No events between the launches of the timed region: consecutive launches
    # overlap (programmatic dependent launch) and an event between them would
    # serialize them.  The per-launch time is the region's time / launches.
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for i in range(steps):
        step(i)
    e1.record(stream)
    torch.cuda.synchronize()
    status = mq.check_device_status()
    if status != 0:
        raise RuntimeError(f"device status {mq.status_string(status)} after the block run")
    step(0)   # layer 0 last, for the parity sample
    torch.cuda.synchronize()
    # with room for widened inputs the call is the token pre-pass + the 256-token kernel
    kernels = 2 if blocks[0].ws_bytes > 0 else 1
    return {"blocks": blocks, "total_ms": e0.elapsed_time(e1), "kernels": kernels}


def run_decode(mq, torch, steps_per_m: int = 240, asym: bool = False, ms=DECODE_MS,
               a16: bool = False):
    """Weight GB/s of the W4A8 block linears at M = 1, 4, 16 (one batched
    launch per layer, 12 layers in rotation), timed with CUDA events per launch
    (kernel) and over a captured CUDA graph of back-to-back launches (stream).
    With asym, the weights are asymmetric per channel (the paper's W4A8)."""
    out = {}
    wbytes = block_weight_bytes(4)
    stream = torch.cuda.current_stream()
    layers = [DecodeLayer(mq, torch, layer, asym, ms, a16) for layer in range(DECODE_LAYERS)]
    ws = mq.workspace()
    wsp, wsn = ws.data_ptr(), ws.numel()

    def call(arr, count, _ws, _n, strm):
        return mq.lib.mq_linear_batch(arr, count, wsp, wsn, strm)
    sp = stream.cuda_stream
    for m in ms:
        for L in layers * 2:
            assert call(L.arr[m], L.count, None, 0, sp) == 0
        torch.cuda.synchronize()
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(steps_per_m)]
        for i in range(steps_per_m):
            L = layers[i % len(layers)]
            ev[i][0].record(stream)
            call(L.arr[m], L.count, None, 0, sp)
            ev[i][1].record(stream)
        torch.cuda.synchronize()
        kms = statistics.median(a.elapsed_time(b) for a, b in ev)
        # back-to-back launches from a CUDA graph (no host launch gaps)
        g = torch.cuda.CUDAGraph()
        side = torch.cuda.Stream()
        side.wait_stream(stream)
        with torch.cuda.stream(side):
            with torch.cuda.graph(g, stream=side):
                for L in layers:
                    call(L.arr[m], L.count, None, 0, side.cuda_stream)
        stream.wait_stream(side)
        g.replay()
        torch.cuda.synchronize()
        reps = max(1, steps_per_m // len(layers))
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(reps):
            g.replay()
        e1.record(stream)
        torch.cuda.synchronize()
        gms = e0.elapsed_time(e1) / (reps * len(layers))
        assert mq.check_device_status() == 0
        out[f"m{m}"] = {"kernel_us": round(kms * 1e3, 2), "kernel_gbs": round(wbytes / kms / 1e6, 1),
                        "stream_us": round(gms * 1e3, 2), "stream_gbs": round(wbytes / gms / 1e6, 1)}
        del g
    return out


def run_asym_prefill(mq, torch, steps: int = 900, check_rows: int = 4):
    """The same block with asymmetric weights in the paper's W8A8 setting (per
    tensor, down per channel): int8 TOPS over `steps` back-to-back batched
    calls (one prefill launch each), rotating over three layers,
    and the first `check_rows` token rows of layer 0 handed to the oracle check."""
    blocks = [PrefillBlock(mq, torch, layer, PREFILL_M, asym=True)
              for layer in range(PREFILL_LAYERS)]
    stream = torch.cuda.current_stream()
    sp = stream.cuda_stream

    def step(i):
        b = blocks[i % len(blocks)]
        rc = mq.lib.mq_linear_batch(b.arr, len(b.descs), b.wsp, b.ws_bytes, sp)
        if rc:
            raise RuntimeError(f"mq_linear_batch failed: {mq.status_string(rc)}")

    for i in range(6):
        step(i)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for i in range(steps):
        step(i)
    e1.record(stream)
    torch.cuda.synchronize()
    if mq.check_device_status() != 0:
        raise RuntimeError("device status error in the asymmetric prefill run")
    ms = e0.elapsed_time(e1) / steps
    # parity sample: run layer 0 once more; its first rows are checked against
    # the oracle in the cpu_baseline leg
    step(0)
    torch.cuda.synchronize()
    checks = [ParityCheck("asym_prefill_w8a8", "linear", c, check_rows,
                          blocks[0].y[j][:check_rows].cpu().numpy())
              for j, c in enumerate(blocks[0].cases)]
    return {"us_per_block": round(ms * 1e3, 2),
            "tops": round(block_ops(PREFILL_M) / (ms * 1e-3) / 1e12, 1),
            "launches_per_step": 1, "steps": steps,
            "weights": "asymmetric: per tensor (q k v o gate up), per channel (down)"}, checks

class A16Block:
    """Device-resident operands of one layer's seven linears with 16-bit
    activations and outputs (int8 or int4 weights) at M tokens."""

    def __init__(self, mq, torch, layer: int, m: int, bits: int, config: int, shared: bool):
        self.cases = synth.block_linears_a16(config, m, bits, layer=layer, shared_input=shared)
        xdev = {}
        self.descs, self.y, self.keep = [], [], []
        for c in self.cases:
            if id(c.x) not in xdev:
                xdev[id(c.x)] = torch.from_numpy(c.x).cuda()
            packed, colsum = mq.pack_weights(c.w, bits)
            m0, sh = mq.requant_params(c.sw, c.sx, c.sy)
            t = [torch.from_numpy(a).cuda() for a in (packed, colsum, m0, sh)]
            y = torch.empty((m, c.N), dtype=torch.int16, device="cuda")
            self.keep += t
            self.y.append(y)
            self.descs.append(mq.make_desc(xdev[id(c.x)], c.zx, t[0], t[1], c.N, t[2], t[3], c.zy,
                                           y, bits, abits=16))
        self.keep += list(xdev.values())
        self.arr = (mq.LinearDesc * len(self.descs))(*self.descs)
        self.ws_bytes = mq.workspace_size_batch(self.descs)
        self.ws = torch.zeros(max(16, self.ws_bytes), dtype=torch.uint8, device="cuda")


def _time_blocks(mq, torch, blocks, steps: int):
    stream = torch.cuda.current_stream()
    sp = stream.cuda_stream

    def step(i):
        b = blocks[i % len(blocks)]
        rc = mq.lib.mq_linear_batch(b.arr, len(b.descs), b.ws.data_ptr(), b.ws_bytes, sp)
        if rc:
            raise RuntimeError(f"mq_linear_batch failed: {mq.status_string(rc)}")

    for i in range(2 * len(blocks)):
        step(i)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for i in range(steps):
        step(i)
    e1.record(stream)
    torch.cuda.synchronize()
    if mq.check_device_status() != 0:
        raise RuntimeError("device status error in a 16-bit activation run")
    step(0)  # layer 0 last, for the parity sample
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / steps


def run_a16(mq, torch, prefill_steps: int = 600, check_rows: int = 4):
    """W8A16 prefill of the block at M = 1024 (the paper's 16-bit-activation
    baseline, Sec. 5.6), back-to-back batched calls (split pre-pass + kernel)
    rotating over three layers, the first rows of layer 0 handed to the oracle
    check; and W4A16 decode at M = 1 and 8, timed like the W4A8 decode
    (one launch per layer, per launch and over a CUDA graph)."""
    out = {}
    blocks = [A16Block(mq, torch, layer, PREFILL_M, 8, CONFIG_ID_PREFILL, True)
              for layer in range(PREFILL_LAYERS)]
    ms = _time_blocks(mq, torch, blocks, prefill_steps)
    checks = [ParityCheck("a16.prefill_w8a16", "a16", c, check_rows,
                          blocks[0].y[j][:check_rows].cpu().numpy())
              for j, c in enumerate(blocks[0].cases)]
    out["prefill_w8a16"] = {"us_per_block": round(ms * 1e3, 2),
                            "tops": round(block_ops(PREFILL_M) / (ms * 1e-3) / 1e12, 1),
                            "launches_per_step": 2, "steps": prefill_steps}
    del blocks
    for m, v in run_decode(mq, torch, a16=True, ms=(1, 8)).items():
        out[f"decode_w4a16_{m}"] = v
    return out, checks


def run_glue(mq, torch, n: int = 1 << 26, reps: int = 20):
    """The boundary quantizers on 64M elements (inputs larger than L2): GB/s
    of algorithmic bytes (input + output) per launch, back to back."""
    out = {}
    stream = torch.cuda.current_stream()
    g = torch.Generator(device="cuda")
    g.manual_seed(5)
    xf = torch.randn(n, device="cuda", generator=g) * 3
    q16 = torch.randint(-32768, 32768, (n,), device="cuda", generator=g, dtype=torch.int32).to(
        torch.int16)
    q8 = torch.empty(n, dtype=torch.int8, device="cuda")
    m0, sh = mq.requant_params(np.array([3.1e-4], np.float32), 1.0, 0.011)
    cases = {
        "quantize_f32_i8": (lambda: mq.quantize(xf, 0.05, 3, q8), 4 + 1),
        "requantize_i16_i8": (lambda: mq.requantize(q16, -40, int(m0[0]), int(sh[0]), 9, q8), 2 + 1),
    }
    for name, (fn, bpe) in cases.items():
        for _ in range(3):
            assert fn() == 0
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(reps):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1) / reps
        out[name] = {"elements": n, "us": round(ms * 1e3, 1),
                     "gbs": round(n * bpe / (ms * 1e-3) / 1e9, 1)}
    del xf, q16, q8
    return out


def run_weight_pipeline(mq, torch, reps: int = 5):
    """The offline weight pipeline (fold of eq. 1, quantization, packing,
    colsum) over the TinyLlama block's seven f32 weight matrices (176 MB), in
    the paper's W8A8 setting (asymmetric per tensor, down per channel) and
    W4A8 (asymmetric per channel): microseconds per block and GB/s of f32
    weights (each read twice: statistics, then codes), as one batched call
    (three launches) and as seven per-linear calls.  Each call allocates its
    outputs on the host side, so the timed steps are enqueued behind a device
    sleep and the region measures the device, not the call rate."""
    g = torch.Generator(device="cuda")
    g.manual_seed(9)
    mats = [(torch.randn((n, k), device="cuda", generator=g) * 0.02,
             torch.rand(k, device="cuda", generator=g) + 0.5) for _, k, n in synth.TINYLLAMA_LINEARS]
    stream = torch.cuda.current_stream()
    out = {}
    fbytes = sum(w.numel() * 4 for w, _ in mats)
    for bits in (8, 4):
        schemes = [synth.paper_weight_scheme(name, bits) for name, _, _ in synth.TINYLLAMA_LINEARS]
        codes = [mq.MQ_WEIGHTS_ASYM_TENSOR if s_ == "asym_tensor" else mq.MQ_WEIGHTS_ASYM_CHANNEL
                 for s_ in schemes]

        def per_linear():
            for (w, s_in), sc in zip(mats, codes):
                mq.fold_quantize_pack(w, bits, sc, s_in)

        def batched():
            mq.fold_quantize_pack_batch([(w, bits, sc, s_in, None)
                                         for (w, s_in), sc in zip(mats, codes)])

        def timed(block):
            block()
            torch.cuda.synchronize()
            torch.cuda._sleep(100_000_000)  # about 50 ms: the host enqueues every step meanwhile
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            for _ in range(reps):
                block()
            e1.record(stream)
            torch.cuda.synchronize()
            return e0.elapsed_time(e1) / reps

        ms = timed(batched)
        ms_each = timed(per_linear)
        out[f"w{bits}a8_block"] = {"us": round(ms * 1e3, 1),
                                   "gbs_f32_weights": round(fbytes / (ms * 1e-3) / 1e9, 1),
                                   "per_linear_calls_us": round(ms_each * 1e3, 1)}
    del mats
    return out


ATT_T, ATT_SETS = 1024, 3


class ParityCheck:
    """Host copies of the first `rows` token rows of one device output and of
    the operands that made it; the cpu_baseline leg recomputes them with the
    oracle.  kind: "linear" (int8 out, optional asymmetric weights and
    residual), "a16" (16-bit activations), "o16" (int8 in, int16 out).  With
    m0/sh given they are the device's fixed-point parameters; otherwise the
    oracle derives them from the case's float scales."""

    def __init__(self, leg: str, kind: str, case, rows: int, got: np.ndarray, m0=None, sh=None,
                 threaded: bool = False):
        self.leg, self.kind, self.case, self.rows, self.got = leg, kind, case, rows, got
        self.m0, self.sh, self.threaded = m0, sh, threaded


class AttentionSet:
    """Device operands and batched descriptors of one layer's attention matmuls
    (TinyLlama: 32 query heads over 4 KV heads, head dim 64, T tokens):
    S_h = Q_h K_g^T (int8 in, int16 scores, keys as the weights read through a
    row pitch, asymmetric per tensor: zw = zk) and O_h = P_h V_g (int8, V_g read
    in place as transposed weights [T][64] through V's row pitch, zw = zv; in
    the 16-bit setting V^T, made by one transpose launch), O written into head
    h's columns of [T][32 * 64].
    Both read weights written on the device in the same stream (wdynamic), and
    leave the weights' row sums to the calls (colsum omitted: the token-major
    kernel needs none; the 16-bit setting's kernels get them computed inside
    the call)."""

    M0_S, SH_S = 1 << 30, 34     # scores: scale 2^-5 (int16 output)
    M0_O, SH_O = 1 << 30, 40     # outputs: scale 2^-11
    ZY_S, ZY_O = 0, -3
    # the W8A16 setting: 16-bit Q and P against 8-bit keys and V, int16 outputs
    SH_S16, SH_O16 = 41, 39

    def __init__(self, mq, torch, layer: int, t: int, bits16: bool = False):
        a = synth.attention_operands(CONFIG_ID_PREFILL, layer, t, bits16=bits16)
        self.bits16 = bits16
        if bits16:
            self.SH_S, self.SH_O = self.SH_S16, self.SH_O16
        self.ops_host = a
        H, G, D = a.heads, a.kv_heads, a.d
        dev = "cuda"
        up = lambda arr: torch.from_numpy(np.ascontiguousarray(arr)).to(dev)
        self.q, self.k, self.v, self.p = up(a.q), up(a.k), up(a.v), up(a.p)
        self.s = torch.empty((H, t, t), dtype=torch.int16, device=dev)
        self.o = torch.empty((t, H * D), dtype=torch.int16 if bits16 else torch.int8, device=dev)
        # 16-bit setting: V^T of all heads at once [G d][T] (head g is rows g d ..
        # g d + d - 1); with 8-bit P the token-major kernel reads V itself
        self.vt = torch.empty((G * D, t), dtype=torch.int8, device=dev) if bits16 else None
        i32 = lambda n, v: up(np.full(n, v, np.int32))
        self.keep = [i32(t, self.M0_S), i32(t, self.SH_S), i32(t, a.zk),
                     i32(D, self.M0_O), i32(D, self.SH_O), i32(D, a.zv)]
        m0s, shs, zwk, m0o, sho, zwv = self.keep
        rep = H // G
        ds = [mq.make_desc(self.q[:, h * D:(h + 1) * D], a.zq, self.k[:, (h // rep) * D:],
                           None, t, m0s, shs, self.ZY_S, self.s[h], 8, zw=zwk,
                           ldw=G * D, wdynamic=True) for h in range(H)]
        if bits16:
            vt_g = lambda g: self.vt[g * D:(g + 1) * D]
            do = [mq.make_desc(self.p[h], a.zp, vt_g(h // rep), None, D, m0o, sho,
                               self.ZY_O, self.o[:, h * D:(h + 1) * D], 8, zw=zwv,
                               wdynamic=True) for h in range(H)]
        else:
            do = [mq.make_desc(self.p[h], a.zp, self.v[:, (h // rep) * D:], None, D, m0o, sho,
                               self.ZY_O, self.o[:, h * D:(h + 1) * D], 8, zw=zwv,
                               ldw=G * D, wdynamic=True, wt=True) for h in range(H)]
        self.arr_s = (mq.LinearDesc * H)(*ds)
        self.arr_o = (mq.LinearDesc * H)(*do)
        self.ws_s_bytes = mq.workspace_size_batch(ds)
        self.ws_o_bytes = mq.workspace_size_batch(do)
        self.ws_s = torch.zeros(max(16, self.ws_s_bytes), dtype=torch.uint8, device=dev)
        self.ws_o = torch.zeros(max(16, self.ws_o_bytes), dtype=torch.uint8, device=dev)
        self.H, self.G, self.D, self.t = H, G, D, t
        self.bytes = (self.q.numel() * self.q.element_size() + self.k.numel() + self.v.numel()
                      + 2 * self.s.numel() + self.p.numel() * self.p.element_size()
                      + self.o.numel() * self.o.element_size())

    def enqueue(self, mq, sp, phase: str = "all"):
        lib, H, G, D, t = mq.lib, self.H, self.G, self.D, self.t
        rcs = []
        if phase in ("all", "scores"):
            rcs.append(lib.mq_linear_batch(self.arr_s, H, self.ws_s.data_ptr(), self.ws_s_bytes,
                                           sp))
        if phase in ("all", "pv"):
            if self.vt is not None:
                rcs.append(lib.mq_transpose_i8(self.v.data_ptr(), t, G * D, G * D,
                                               self.vt.data_ptr(), t, sp))
            rcs.append(lib.mq_linear_batch(self.arr_o, H, self.ws_o.data_ptr(), self.ws_o_bytes,
                                           sp))
        if any(rcs):
            raise RuntimeError(f"attention launch failed: {[mq.status_string(r) for r in rcs]}")
        return len(rcs)

    def checks(self, rows: int, heads=(0, 31)):
        """ParityChecks of the scores and outputs of `heads`, first `rows` rows."""
        a, D, rep = self.ops_host, self.D, self.H // self.G
        out = []
        for h in heads:
            g = h // rep
            kg = np.ascontiguousarray(a.k[:, g * D:(g + 1) * D])
            sc = synth.LinearCase(f"scores{h}", np.ascontiguousarray(a.q[:rows, h * D:(h + 1) * D]),
                                  a.zq, 0.0, kg, None, 8, 0.0, self.ZY_S)
            sc.zw = np.full(self.t, a.zk, np.int32)
            leg = "attention_w8a16_t1024" if self.bits16 else "attention_w8a8_t1024"
            out.append(ParityCheck(leg, "a16" if self.bits16 else "o16", sc, rows,
                                   self.s[h, :rows].cpu().numpy(),
                                   np.full(self.t, self.M0_S, np.int32),
                                   np.full(self.t, self.SH_S, np.int32)))
            vt = np.ascontiguousarray(a.v[:, g * D:(g + 1) * D].T)
            pc = synth.LinearCase(f"pv{h}", np.ascontiguousarray(a.p[h, :rows]), a.zp, 0.0, vt,
                                  None, 8, 0.0, self.ZY_O)
            pc.zw = np.full(D, a.zv, np.int32)
            out.append(ParityCheck(leg, "a16" if self.bits16 else "linear", pc, rows,
                                   self.o[:rows, h * D:(h + 1) * D].cpu().numpy(),
                                   np.full(D, self.M0_O, np.int32),
                                   np.full(D, self.SH_O, np.int32)))
        return out


def run_attention(mq, torch, reps: int = 60, check_rows: int = 4, bits16: bool = False):
    """Grouped-query attention's two integer matmuls of one TinyLlama layer at
    T = 1024 (the softmax between them is outside the integer layer): per step
    S = Q K^T for 32 heads (one batched call, one token-major kernel launch,
    int16 scores, the keys' zero point folded in: no row sums) and O = P V for
    32 heads (one batched call reading V in place; in the 16-bit setting V^T of
    all heads by one transpose first, and each call also computes its weights'
    row sums).  Steps rotate over three
    layers' operands (about 300 MB, more than L2).  The host enqueues the timed
    steps behind a device sleep, so the region measures the device, not the
    ctypes call rate; a second pass times the two phases alone."""
    sets = [AttentionSet(mq, torch, layer, ATT_T, bits16) for layer in range(ATT_SETS)]
    stream = torch.cuda.current_stream()
    sp = stream.cuda_stream
    launches = 0
    for i in range(2 * ATT_SETS):
        launches = sets[i % ATT_SETS].enqueue(mq, sp)
    torch.cuda.synchronize()
    if mq.check_device_status() != 0:
        raise RuntimeError("device status error in the attention warm-up")

    def timed(phase: str, n: int) -> float:
        torch.cuda.synchronize()
        torch.cuda._sleep(100_000_000)  # about 50 ms: the host enqueues every step meanwhile
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for i in range(n):
            sets[i % ATT_SETS].enqueue(mq, sp, phase)
        e1.record(stream)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / n

    ms = timed("all", reps)
    ms_s = timed("scores", reps)
    ms_o = timed("pv", reps)
    if mq.check_device_status() != 0:
        raise RuntimeError("device status error in the attention run")
    sets[0].enqueue(mq, sp)   # layer 0 last, for the parity sample
    torch.cuda.synchronize()
    b = sets[0]
    ops = 2 * 2 * b.t * b.t * b.D * b.H
    checks = b.checks(check_rows)
    res = {"what": ("S = Q K^T (int16 scores) and O = P V, 32 query heads over 4 KV heads, "
                    "head dim 64, T = 1024; full T x T scores (the causal mask is applied by "
                    "the softmax, not here)"
                    + ("; W8A16 setting: 16-bit Q and P against 8-bit keys and V (with their "
                       "zero points), int16 outputs" if bits16 else "")),
           "us_per_layer": round(ms * 1e3, 2), "tops": round(ops / (ms * 1e-3) / 1e12, 1),
           "algorithmic_bytes": b.bytes,
           "gbs": round(b.bytes / (ms * 1e-3) / 1e9, 1),
           "scores_us": round(ms_s * 1e3, 2), "pv_us": round(ms_o * 1e3, 2),
           "calls_per_step": launches, "steps": reps}
    del sets
    return res, checks


# --------------------------------------------------------------------------- config 3: the stack
def stack_ops(m: int = STACK_M, layers: int = STACK_LAYERS) -> int:
    _, hk, hn = synth.TINYLLAMA_HEAD
    return layers * block_ops(m) + 2 * m * hk * hn


def stack_row_ops(layers: int = STACK_LAYERS) -> int:
    return stack_ops(1, layers)


class Stack:
    """Device-resident config-3 model: 22 TinyLlama-shaped layers of seven
    W8A8 linears at M tokens, chained as the workload defines (q/k/v/gate/up
    read x_l; o reads q's output, down reads up's; x_{l+1} = sat8(down +
    r_l)), and the 2048 -> 32000 head on x_22.  One step = 2 batched calls per
    layer + the head = 45 prefill launches, plus the pre-pass that widens x_0
    (every later input comes widened from the call that wrote it: q, up and
    down also write an f16 copy and row sums of squares).  The step's input x_0 and its
    result (the head's int8 output) are double-buffered so that the
    end-to-end loop can upload step i + 1 and download step i - 1 while step i
    computes; the seeded residuals r_l are model constants, resident like the
    weights."""

    def __init__(self, mq, torch, m: int = STACK_M, layers: int = STACK_LAYERS):
        x0, _, _, self.layers, self.head = synth.chain_stack(CONFIG_ID_STACK, m, layers)
        self.m, self.x0_np = m, x0
        dev = "cuda"
        up = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev)
        self.keep = []
        self.x0 = [up(x0) for _ in range(2)]
        self.x0_host = torch.from_numpy(np.ascontiguousarray(x0)).pin_memory()
        _, hk, hn = synth.TINYLLAMA_HEAD
        self.hy = [torch.empty((m, hn), dtype=torch.int8, device=dev) for _ in range(2)]
        self.hy_host = torch.empty((m, hn), dtype=torch.int8).pin_memory()
        self.outs = []
        calls_a, calls_b = [], []   # per x_0 / head buffer set
        # chained layers: q, up and down also write their outputs as f16 with each
        # row's sum of squares, which o, down, the next layer and the head read
        # instead of widening their inputs again (the row sums are zeroed once a
        # step, below)
        self.ysq = torch.zeros((len(self.layers), 3, m), dtype=torch.int32, device=dev)
        self.y16 = []

        def dev_linear(c):
            packed, colsum = mq.pack_weights(c.w, 8)
            m0, sh = mq.requant_params(c.sw, c.sx, c.sy)
            t = [up(a) for a in (packed, colsum, m0, sh)]
            t.append(mq.weight_sq_sums(t[0], c.N, c.K, 8))
            self.keep += t
            return t

        def arr(descs):
            return ((mq.LinearDesc * len(descs))(*descs), len(descs))

        for li, L in enumerate(self.layers):
            out = {c.name: torch.empty((m, c.N), dtype=torch.int8, device=dev) for c in L.cases}
            self.outs.append(out)
            res = up(L.residual)
            self.keep.append(res)
            cs = {c.name: c for c in L.cases}
            w = {c.name: dev_linear(c) for c in L.cases}

            y16 = {nm: torch.empty((m, cs[nm].N), dtype=torch.float16, device=dev)
                   for nm in ("q", "up", "down")}
            ysq = {nm: self.ysq[li, j] for j, nm in enumerate(("q", "up", "down"))}
            self.y16.append(y16)

            def desc(name, xin, residual=None, src=None):
                c, t = cs[name], w[name]
                copy = {"y16": y16[name], "ysq": ysq[name]} if name in y16 else {}
                if src is not None:  # x's f16 copy and row sums from the call that wrote x
                    copy.update(x16=src[0], xsq=src[1])
                return mq.make_desc(xin, c.zx, t[0], t[1], c.N, t[2], t[3], c.zy, out[name], 8,
                                    residual=residual, wsq=t[4], **copy)
            xin = (self.x0[0], self.x0[1]) if li == 0 else (self.outs[li - 1]["down"],) * 2
            prev = None if li == 0 else (self.y16[li - 1]["down"], self.ysq[li - 1, 2])
            for j, calls in enumerate((calls_a, calls_b)):
                calls.append(arr([desc(nm, xin[j], src=prev)
                                  for nm in ("q", "k", "v", "gate", "up")]))
            second = arr([desc("o", out["q"], src=(y16["q"], ysq["q"])),
                          desc("down", out["up"], residual=res, src=(y16["up"], ysq["up"]))])
            calls_a.append(second)
            calls_b.append(second)
        ht = dev_linear(self.head)
        h = self.head
        for j, calls in enumerate((calls_a, calls_b)):
            calls.append(arr([mq.make_desc(self.outs[-1]["down"], h.zx, ht[0], ht[1], h.N, ht[2],
                                           ht[3], h.zy, self.hy[j], 8, wsq=ht[4],
                                           x16=self.y16[-1]["down"], xsq=self.ysq[-1, 2])]))
        self.calls = (calls_a, calls_b)
        self.launches = len(calls_a)
        self.h2d_bytes = x0.size
        self.d2h_bytes = m * hn
        # one workspace for every call (its widened inputs are scratch; the
        # calls run one after another on one stream)
        sizes = [mq.workspace_size_batch(list(a)) for a, _ in calls_a]
        self.ws_bytes = max(sizes + [mq.workspace_size_batch(list(a)) for a, _ in calls_b])
        self.ws = torch.zeros(max(16, self.ws_bytes), dtype=torch.uint8, device=dev)
        # kernel launches a step: a prefill-only call with workspace beyond the
        # decode region takes the 256-token kernel after its token pre-pass
        self.kernels = sum(2 if b > 0 else 1 for b in sizes)

    def enqueue(self, mq, sp: int, j: int = 0):
        wsp = self.ws.data_ptr() if self.ws_bytes else None
        self.ysq.zero_()  # the calls add the row sums of squares of their outputs
        for a, n in self.calls[j]:
            rc = mq.lib.mq_linear_batch(a, n, wsp, self.ws_bytes, sp)
            if rc:
                raise RuntimeError(f"mq_linear_batch failed: {mq.status_string(rc)}")


def run_stack(mq, torch, dist: Dist, steps: int, warmup: int):
    """The headline: config 3's 22-layer chained W8A8 stack + head at M = 2048,
    device-resident (value, roofline), then end to end with host buffers."""
    st = Stack(mq, torch)
    stream = torch.cuda.current_stream()
    sp = stream.cuda_stream
    for i in range(warmup):
        st.enqueue(mq, sp, i & 1)
    torch.cuda.synchronize()
    if mq.check_device_status() != 0:
        raise RuntimeError("device status error after warm-up")
    # No events between launches: consecutive launches overlap through
    # programmatic dependent launch, and an event would serialize them.
    clocks = ClockSampler(dist.local)
    time.sleep(0.3)
    dist.barrier()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clocks.start()
    e0.record(stream)
    for i in range(steps):
        st.enqueue(mq, sp, i & 1)
    e1.record(stream)
    torch.cuda.synchronize()
    clocks.stop()
    dist.barrier()
    total_ms = e0.elapsed_time(e1)
    if mq.check_device_status() != 0:
        raise RuntimeError("device status error after the timed region")
    max_total_ms = dist.max(total_ms)

    # end to end: every step uploads x_0 from pinned host memory and downloads
    # the head's output into pinned host memory, on their own streams, so that
    # the copies of neighbouring steps overlap this step's kernels; buffer set
    # j = i % 2 is reused two steps later, after its copies are done
    e2e_steps = max(3, min(steps, 100))
    torch.cuda.synchronize()
    dist.barrier()
    s_in, s_out = torch.cuda.Stream(), torch.cuda.Stream()
    in_done = [torch.cuda.Event() for _ in range(e2e_steps)]
    comp_done = [torch.cuda.Event() for _ in range(e2e_steps)]
    out_done = [torch.cuda.Event() for _ in range(e2e_steps)]
    a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a0.record(stream)
    s_in.wait_event(a0)
    s_out.wait_event(a0)
    for i in range(e2e_steps):
        j = i & 1
        with torch.cuda.stream(s_in):
            if i >= 2:
                s_in.wait_event(comp_done[i - 2])  # step i - 2 no longer reads x_0[j]
            st.x0[j].copy_(st.x0_host, non_blocking=True)
            in_done[i].record(s_in)
        stream.wait_event(in_done[i])
        if i >= 2:
            stream.wait_event(out_done[i - 2])  # step i - 2's result is copied out
        st.enqueue(mq, sp, j)
        comp_done[i].record(stream)
        with torch.cuda.stream(s_out):
            s_out.wait_event(comp_done[i])
            st.hy_host.copy_(st.hy[j], non_blocking=True)
            out_done[i].record(s_out)
    stream.wait_stream(s_out)
    a1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = dist.max(a0.elapsed_time(a1))
    if mq.check_device_status() != 0:
        raise RuntimeError("device status error in the end-to-end run")
    return {"stack": st, "total_ms": max_total_ms, "clocks": clocks.result(), "e2e_ms": e2e_ms,
            "e2e_steps": e2e_steps, "h2d": st.h2d_bytes, "d2h": st.d2h_bytes,
            "launches_per_step": st.launches, "kernels_per_step": st.kernels}


def stack_parity(st, rows):
    """The oracle runs the stack's chain on `rows` from the seeded x_0 on every
    host core (row blocks), and every layer's seven outputs and the head are
    compared with the device's at those rows (the device buffers hold the
    last step, which read the same x_0).  Returns the check and the oracle's
    rate."""
    import oracle
    rows = np.asarray(rows)

    def prep(c):
        packed, _ = oracle.pack(c.w, 8)
        m0, sh = oracle.requant_params(c.sx, c.sw, c.sy)
        return packed, m0, sh
    prepared = [{c.name: prep(c) for c in L.cases} for L in st.layers]
    hp = prep(st.head)

    def lin(c, p, xin):
        return oracle.linear_mt(xin, c.zx, p[0], 8, c.N, p[1], p[2], c.zy)
    outputs = mism = 0
    xr = np.ascontiguousarray(st.x0_np[rows])
    t0 = time.perf_counter()
    want = []
    for L, P in zip(st.layers, prepared):
        cs = {c.name: c for c in L.cases}
        ys = {nm: lin(cs[nm], P[nm], xr) for nm in ("q", "k", "v", "gate", "up")}
        ys["o"] = lin(cs["o"], P["o"], ys["q"])
        ys["down"] = oracle.residual_add(lin(cs["down"], P["down"], ys["up"]),
                                         np.ascontiguousarray(L.residual[rows]))
        want.append(ys)
        xr = ys["down"]
    hwant = lin(st.head, hp, xr)
    secs = time.perf_counter() - t0
    import torch
    idx = torch.from_numpy(rows).cuda()
    for out, ys in zip(st.outs, want):
        for nm, y in ys.items():
            got = out[nm].index_select(0, idx).cpu().numpy()
            outputs += y.size
            mism += int(np.count_nonzero(got != y))
    got = st.hy[0].index_select(0, idx).cpu().numpy()
    outputs += hwant.size
    mism += int(np.count_nonzero(got != hwant))
    ops = len(rows) * stack_row_ops()
    return {"rows": len(rows), "outputs": outputs, "mismatches": mism}, ops, secs


# --------------------------------------------------------------------------- config 0
def run_single_linear(mq, torch, copies: int = 40, reps: int = 2000):
    """Config 0: one W8A8 linear, M = 128, K = N = 2048 (1.07 G int8 ops; with
    the workspace mq_workspace_size_batch asks for, split over K on the
    token-major kernel plus one combine launch), rotating over `copies`
    independent operand sets (180 MB > L2): back to back, and with CUDA events
    around every call."""
    c = synth.make_linear(0, 0, 0, "cfg0", 128, 2048, 2048, 8)
    packed, colsum = mq.pack_weights(c.w, 8)
    m0, sh = mq.requant_params(c.sw, c.sx, c.sy)
    up = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
    sets, keep, ys = [], [], []
    for _ in range(copies):
        t = [up(a) for a in (c.x, packed, colsum, m0, sh)]
        y = torch.empty((128, 2048), dtype=torch.int8, device="cuda")
        keep += t
        ys.append(y)
        sets.append((mq.LinearDesc * 1)(mq.make_desc(t[0], c.zx, t[1], t[2], 2048, t[3], t[4],
                                                     c.zy, y, 8)))
    stream = torch.cuda.current_stream()
    sp = stream.cuda_stream
    wsn = mq.workspace_size_batch([sets[0][0]])
    ws = torch.zeros(max(16, wsn), dtype=torch.uint8, device="cuda")
    wsp = ws.data_ptr() if wsn else None
    lib_call = mq.lib.mq_linear_batch
    call = lambda a, n, _w, _b, s: lib_call(a, n, wsp, wsn, s)
    for i in range(2 * copies):
        assert call(sets[i % copies], 1, None, 0, sp) == 0
    torch.cuda.synchronize()
    torch.cuda._sleep(50_000_000)  # the host enqueues the region meanwhile
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for i in range(reps):
        call(sets[i % copies], 1, None, 0, sp)
    e1.record(stream)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / reps
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(200)]
    for i, (a, b) in enumerate(ev):
        a.record(stream)
        call(sets[i % copies], 1, None, 0, sp)
        b.record(stream)
    torch.cuda.synchronize()
    kms = statistics.median(a.elapsed_time(b) for a, b in ev)
    if mq.check_device_status() != 0:
        raise RuntimeError("device status error in the config-0 run")
    ops = 2 * 128 * 2048 * 2048
    check = ParityCheck("config0_single_linear_m128", "linear", c, 128, ys[0].cpu().numpy(),
                        threaded=True)
    return {"what": "one W8A8 linear, M = 128, K = N = 2048", "int8_ops": ops,
            "workspace_bytes": wsn,
            "us_back_to_back": round(ms * 1e3, 2),
            "tops_back_to_back": round(ops / (ms * 1e-3) / 1e12, 1),
            "us_per_launch_events": round(kms * 1e3, 2),
            "tops_per_launch_events": round(ops / (kms * 1e-3) / 1e12, 1),
            "l2": f"{copies} operand sets rotated"}, [check]


# --------------------------------------------------------------------------- config 4
def gemma_block(m: int, bits: int, layer: int = 0):
    return synth.block_linears(CONFIG_ID_GEMMA, m, bits, shapes=synth.GEMMA_LINEARS, layer=layer,
                               t_rows_frac=0.01, shared_input=m > 16)


def gemma_head(m: int, bits: int):
    _, hk, hn = synth.GEMMA_HEAD
    return synth.make_linear(CONFIG_ID_GEMMA, 0, 7, "head", m, hk, hn, bits, t_rows_frac=0.01)


class DeviceCalls:
    """Device operands and one batched call per group of cases (outputs
    allocated on the device; the cases' inputs uploaded once per distinct x)."""

    def __init__(self, mq, torch, groups, bits: int):
        up = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
        xdev, self.keep, self.calls, self.y = {}, [], [], {}
        for cases in groups:
            descs = []
            for c in cases:
                if id(c.x) not in xdev:
                    xdev[id(c.x)] = up(c.x)
                packed, colsum = mq.pack_weights(c.w, bits)
                m0, sh = mq.requant_params(c.sw, c.sx, c.sy)
                t = [up(a) for a in (packed, colsum, m0, sh)]
                t.append(mq.weight_sq_sums(t[0], c.N, c.K, bits))
                y = torch.empty((c.M, c.N), dtype=torch.int8, device="cuda")
                self.keep += t + [y]
                self.y[c.name] = y
                descs.append(mq.make_desc(xdev[id(c.x)], c.zx, t[0], t[1], c.N, t[2], t[3],
                                          c.zy, y, bits, wsq=t[4]))
            self.calls.append(((mq.LinearDesc * len(descs))(*descs), len(descs)))
        self.keep += list(xdev.values())
        self.ws_bytes = max(mq.workspace_size_batch(list(a)) for a, _ in self.calls)
        self.ws = torch.zeros(max(16, self.ws_bytes), dtype=torch.uint8, device="cuda")

    def enqueue(self, mq, sp, ws=None, ws_bytes=0, which=None):
        """One batched call per group; without `ws`, the calls' own workspace."""
        if ws is None and self.ws_bytes:
            ws, ws_bytes = self.ws.data_ptr(), self.ws_bytes
        for i, (a, n) in enumerate(self.calls):
            if which is None or i in which:
                rc = mq.lib.mq_linear_batch(a, n, ws, ws_bytes, sp)
                if rc:
                    raise RuntimeError(f"mq_linear_batch failed: {mq.status_string(rc)}")


def run_gemma_prefill(mq, torch, steps: int = 30, check_rows: int = 64):
    """Config 4, prefill: the Gemma-2B-shaped block's seven W8A8 linears at
    M = 4096 (one batched launch) and the 2048 -> 256000 head (one launch);
    one step is both (0.90 + 4.29 T int8 ops; 630 MB of weights and a 1 GB
    head output per step, far beyond L2)."""
    cases, head = gemma_block(4096, 8), gemma_head(4096, 8)
    dc = DeviceCalls(mq, torch, [cases, [head]], 8)
    stream = torch.cuda.current_stream()
    sp = stream.cuda_stream
    for _ in range(2):
        dc.enqueue(mq, sp)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    times = {}
    for name, which in (("step", None), ("block", (0,)), ("head", (1,))):
        torch.cuda.synchronize()
        e0.record(stream)
        for _ in range(steps):
            dc.enqueue(mq, sp, which=which)
        e1.record(stream)
        torch.cuda.synchronize()
        times[name] = e0.elapsed_time(e1) / steps
    if mq.check_device_status() != 0:
        raise RuntimeError("device status error in the config-4 prefill run")
    bops = sum(2 * c.M * c.K * c.N for c in cases)
    hops = 2 * head.M * head.K * head.N
    checks = [ParityCheck("config4_gemma.prefill_m4096", "linear", c, check_rows,
                          dc.y[c.name][:check_rows].cpu().numpy(), threaded=True)
              for c in cases + [head]]
    out = {"what": "Gemma-2B-shaped block (7 W8A8 linears, one launch) + 2048->256000 head "
                   "(one launch) at M = 4096", "int8_ops_per_step": bops + hops,
           "us_per_step": round(times["step"] * 1e3, 1),
           "tops": round((bops + hops) / (times["step"] * 1e-3) / 1e12, 1),
           "block_us": round(times["block"] * 1e3, 1),
           "block_tops": round(bops / (times["block"] * 1e-3) / 1e12, 1),
           "head_us": round(times["head"] * 1e3, 1),
           "head_tops": round(hops / (times["head"] * 1e-3) / 1e12, 1), "steps": steps}
    del dc
    return out, checks


def run_gemma_decode(mq, torch, reps: int = 20, block_layers: int = 4):
    """Config 4, decode: the Gemma-2B-shaped block's seven W4A8 linears at
    M = 1 (55.1 MB of int4 weights, one launch) and the 2048 -> 256000 head
    (262 MB, one launch), timed back to back from CUDA graphs: the step
    (block + head), the head alone, and the block alone rotating over
    `block_layers` layers' weights (more than L2)."""
    ws = mq.workspace()
    wsp, wsn = ws.data_ptr(), ws.numel()
    head = gemma_head(1, 4)
    layers = []
    for layer in range(block_layers):
        cases = gemma_block(1, 4, layer=layer)
        layers.append((cases, DeviceCalls(mq, torch, [cases] + ([[head]] if layer == 0 else []),
                                          4)))
    cases0, dc0 = layers[0]
    bw = sum(c.K * c.N // 2 for c in cases0)
    hw = head.K * head.N // 2
    stream = torch.cuda.current_stream()

    def graph_time(fn, n_inner):
        side = torch.cuda.Stream()
        side.wait_stream(stream)
        fn(side.cuda_stream)   # warm-up outside the capture
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.stream(side):
            with torch.cuda.graph(g, stream=side):
                fn(side.cuda_stream)
        stream.wait_stream(side)
        g.replay()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(reps):
            g.replay()
        b.record(stream)
        torch.cuda.synchronize()
        del g
        return a.elapsed_time(b) / (reps * n_inner)

    inner = 8
    step_ms = graph_time(lambda s: [dc0.enqueue(mq, s, wsp, wsn) for _ in range(inner)], inner)
    head_ms = graph_time(lambda s: [dc0.enqueue(mq, s, wsp, wsn, which=(1,))
                                    for _ in range(inner)], inner)
    block_ms = graph_time(lambda s: [dc.enqueue(mq, s, wsp, wsn, which=(0,))
                                     for _ in range(2) for _, dc in layers], 2 * block_layers)
    if mq.check_device_status() != 0:
        raise RuntimeError("device status error in the config-4 decode run")
    checks = [ParityCheck("config4_gemma.decode_w4a8_m1", "linear", c, 1,
                          dc0.y[c.name].cpu().numpy()) for c in cases0 + [head]]
    gbs = lambda b, ms: round(b / (ms * 1e-3) / 1e9, 1)
    out = {"what": "Gemma-2B-shaped block (7 W4A8 linears, one launch) + 2048->256000 head "
                   "(one launch) at M = 1, back to back from CUDA graphs",
           "weight_bytes_per_step": bw + hw, "step_us": round(step_ms * 1e3, 2),
           "step_gbs": gbs(bw + hw, step_ms), "head_weight_bytes": hw,
           "head_us": round(head_ms * 1e3, 2), "head_gbs": gbs(hw, head_ms),
           "block_weight_bytes": bw, "block_us": round(block_ms * 1e3, 2),
           "block_gbs": gbs(bw, block_ms), "block_layers_rotated": block_layers}
    del layers, dc0
    return out, checks


# --------------------------------------------------------------------------- CPU oracle
def oracle_sample(blocks_cases, rows: range, col_frac: float = 1.0):
    """Run the oracle on `rows` of every linear of one block; returns
    (int8 ops done, seconds, {linear index: y})."""
    import oracle
    ops = 0
    outs = {}
    t0 = time.perf_counter()
    for j, c in enumerate(blocks_cases):
        n = max(1, int(round(c.N * col_frac)))
        packed, _ = oracle.pack(c.w[:n], c.bits)
        m0, sh = oracle.requant_params(c.sx, c.sw[:n], c.sy)
        x = np.ascontiguousarray(c.x[rows.start:rows.stop])
        y = oracle.linear(x, c.zx, packed, c.bits, n, m0, sh, c.zy)
        if c.residual is not None:
            y = oracle.residual_add(y, np.ascontiguousarray(c.residual[rows.start:rows.stop, :n]))
        outs[j] = y
        ops += 2 * x.shape[0] * c.K * n
    return ops, time.perf_counter() - t0, outs


def run_checks(checks) -> dict:
    """Recompute every ParityCheck with the oracle: {leg: {rows, outputs,
    mismatches}}."""
    import oracle
    out = {}
    for ck in checks:
        c = ck.case
        x = np.ascontiguousarray(c.x[:ck.rows])
        packed, _ = oracle.pack(c.w, c.bits)
        if ck.m0 is not None:
            m0, sh = ck.m0, ck.sh
        else:
            m0, sh = oracle.requant_params(c.sx, c.sw, c.sy)
        if ck.kind == "a16":
            y = oracle.linear_a16(x, c.zx, packed, c.bits, c.N, m0, sh, c.zy, zw=c.zw)
        elif ck.kind == "o16":
            y = oracle.linear_o16(x, c.zx, packed, c.bits, c.N, m0, sh, c.zy, zw=c.zw)
        else:
            fn = oracle.linear_mt if ck.threaded else oracle.linear
            y = fn(x, c.zx, packed, c.bits, c.N, m0, sh, c.zy, zw=c.zw)
            if c.residual is not None:
                y = oracle.residual_add(y, np.ascontiguousarray(c.residual[:ck.rows]))
        r = out.setdefault(ck.leg, {"rows": ck.rows, "outputs": 0, "mismatches": 0})
        r["outputs"] += int(y.size)
        r["mismatches"] += int(np.count_nonzero(ck.got != y))
    return out


def cpu_baseline(st, rows: int = 128, checks=()):
    """The oracle timed on every host core (row blocks) on `rows` token rows of
    the headline stack, spread over its 2048, through all 22 layers and the
    head; its outputs are compared with the device's at every layer.  Then
    the other legs' parity samples."""
    import oracle
    oracle.build()
    sel = np.linspace(0, st.m - 1, rows).round().astype(np.int64)
    par, ops, secs = stack_parity(st, sel)
    base = {"value": round(ops / secs / 1e12, 6), "unit": "TOPS", "cores": oracle.threads(),
            "kind": "oracle",
            "sample": f"{rows} token rows spread over the {st.m} through all {len(st.layers)} "
                      f"layers' 7 linears (+ residual) and the head: {ops / 1e9:.0f} G of the "
                      f"{stack_ops() / 1e12:.2f} T int8 ops of a step, row blocks on every core",
            "seconds": round(secs, 2), "parity_sample": par}
    return base, run_checks(checks)


def reference_stack_sample(st_cases, rows: np.ndarray, prepared, nthreads: int):
    """One reference step: the oracle's chain on `rows` of the stack."""
    import oracle
    x0, layers, head = st_cases
    xr = np.ascontiguousarray(x0[rows])

    def lin(c, p, xin):
        return oracle.linear_mt(xin, c.zx, p[0], 8, c.N, p[1], p[2], c.zy, nthreads=nthreads)
    for L, P in zip(layers, prepared[0]):
        cs = {c.name: c for c in L.cases}
        ys = {nm: lin(cs[nm], P[nm], xr) for nm in ("q", "up")}
        for nm in ("k", "v", "gate"):
            lin(cs[nm], P[nm], xr)
        lin(cs["o"], P["o"], ys["q"])
        xr = oracle.residual_add(lin(cs["down"], P["down"], ys["up"]),
                                 np.ascontiguousarray(L.residual[rows]))
    lin(head, prepared[1], xr)
    return len(rows) * stack_row_ops()


def run_reference(args, dist: Dist):
    """Reference arm: the CPU oracle timed on this host's cores on a bounded
    sample of the headline workload: each step runs a few token rows of the
    stack through all 22 layers and the head (row blocks on every core)."""
    if dist.rank != 0:
        return
    import oracle
    oracle.build()
    x0, _, _, layers, head = synth.chain_stack(CONFIG_ID_STACK, STACK_M, STACK_LAYERS)

    def prep(c):
        packed, _ = oracle.pack(c.w, 8)
        m0, sh = oracle.requant_params(c.sx, c.sw, c.sy)
        return packed, m0, sh
    prepared = ([{c.name: prep(c) for c in L.cases} for L in layers], prep(head))
    cores = oracle.threads()
    cases = (x0, layers, head)
    # size the per-step sample so that warm-up + steps take about 90 s at most
    t0 = time.perf_counter()
    reference_stack_sample(cases, np.arange(cores), prepared, cores)
    t_step = time.perf_counter() - t0
    budget = 90.0
    rows = cores if (args.steps + args.warmup) * t_step <= budget else max(
        1, int(cores * budget / ((args.steps + args.warmup) * t_step)))
    pick = lambda i: (np.arange(rows) * 131 + 17 * i) % STACK_M
    for i in range(args.warmup):
        reference_stack_sample(cases, pick(i), prepared, cores)
    ops = 0
    t0 = time.perf_counter()
    for i in range(args.steps):
        ops += reference_stack_sample(cases, pick(args.warmup + i), prepared, cores)
    secs = time.perf_counter() - t0
    value = ops / secs / 1e12
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "TOPS", "n_gpus": dist.world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": secs * 1e3 / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "int64",
        "data": "synthetic",
        "config": {"workload": WORKLOAD, "tokens": STACK_M, "layers": STACK_LAYERS,
                   "sample_per_step": f"{rows} token rows through all {STACK_LAYERS} layers' "
                                      "7 linears and the head"},
        "cpu_baseline": {"value": value, "unit": "TOPS", "cores": cores, "kind": "oracle",
                         "sample": f"{rows} token rows of the stack per step, row blocks on "
                                   f"{cores} threads"},
        "e2e": {"value": value, "unit": "TOPS", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# --------------------------------------------------------------------------- main
def run_profile_leg(mq, torch, dist, args):
    """One leg's timed loop alone, for a profiler (`--profile LEG`): the
    headline stack, the config-1 block, the config-2 decode block at M = 1,
    config 4's prefill step, config 4's decode step at M = 1 (block, then
    head), or one TinyLlama layer's attention matmuls at T = 1024.  Prints the
    leg's time per step."""
    t0 = time.time()
    if args.profile == "stack":
        r = run_stack(mq, torch, dist, args.steps, args.warmup)
        per = r["total_ms"] / args.steps
    elif args.profile == "block":
        r = run_prefill(mq, torch, dist, args.steps, args.warmup)
        per = r["total_ms"] / args.steps
    elif args.profile == "decode":
        r = run_decode(mq, torch, steps_per_m=args.steps, ms=(1,))
        per = r["m1"]["stream_us"] * 1e-3
    elif args.profile == "attention":
        r, _ = run_attention(mq, torch, reps=args.steps, check_rows=1)
        per = r["us_per_layer"] * 1e-3
    elif args.profile == "gemma_decode":
        r, _ = run_gemma_decode(mq, torch, reps=args.steps, block_layers=1)
        per = r["step_us"] * 1e-3
    else:
        r, _ = run_gemma_prefill(mq, torch, steps=args.steps, check_rows=1)
        per = r["us_per_step"] * 1e-3
    print(f"profile leg {args.profile}: {per:.4f} ms per step ({time.time() - t0:.1f} s)",
          flush=True)
    scalars = {k: v for k, v in r.items() if isinstance(v, (int, float, str))}
    print(json.dumps(scalars), flush=True)


def main():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawTextHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["mq", "reference"], default="mq")
    ap.add_argument("--profile", choices=["stack", "block", "decode", "gemma", "gemma_decode", "attention"], default=None,
                    help="run only this leg's timed loop (for a profiler; no JSON line)")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be at least 3")
    world, rank, local = dist_env()
    if args.impl == "reference":
        run_reference(args, Dist(1, rank, local))
        return

    import torch
    torch.cuda.set_device(local)
    dist = Dist(world, rank, local)
    from paper_2408_13933_gb300 import build
    build.build()
    from paper_2408_13933_gb300 import mq

    if args.profile:
        run_profile_leg(mq, torch, dist, args)
        return
    stack = run_stack(mq, torch, dist, args.steps, args.warmup)
    checks = []
    cfg0, more = run_single_linear(mq, torch)
    checks += more
    pre = run_prefill(mq, torch, dist, 2000, 5)
    checks += [ParityCheck("config1_tinyllama_block_m1024", "linear", c, 64,
                           pre["blocks"][0].y[j][:64].cpu().numpy(), threaded=True)
               for j, c in enumerate(pre["blocks"][0].cases)]
    del pre["blocks"]
    decode = run_decode(mq, torch)
    g_pre, more = run_gemma_prefill(mq, torch)
    checks += more
    g_dec, more = run_gemma_decode(mq, torch)
    checks += more
    asym_pre, more = run_asym_prefill(mq, torch)
    checks += more
    asym_dec = run_decode(mq, torch, asym=True, ms=(1, 16))
    a16, more = run_a16(mq, torch)
    checks += more
    attention, more = run_attention(mq, torch)
    checks += more
    attention16, more = run_attention(mq, torch, bits16=True)
    checks += more
    glue = run_glue(mq, torch)
    wpipe = run_weight_pipeline(mq, torch)
    peaks = measured_peaks()

    st = stack["stack"]
    ops = stack_ops()
    ms_per_step = stack["total_ms"] / args.steps
    value = whole_job_rate(ops * args.steps, world, stack["total_ms"]) / 1e12
    kern_tflops = ops / (ms_per_step * 1e-3) / 1e12
    e2e_value = whole_job_rate(ops * stack["e2e_steps"], world, stack["e2e_ms"]) / 1e12
    hbm = peaks["hbm_gbs"]
    for v in list(decode.values()) + list(asym_dec.values()):
        v["frac_hbm"] = round(v["stream_gbs"] / hbm, 3)
    for v in glue.values():
        v["frac_hbm"] = round(v["gbs"] / hbm, 3)
    for k, v in a16.items():
        if k.startswith("decode_"):
            v["frac_hbm"] = round(v["stream_gbs"] / hbm, 3)
    for k in ("step", "head", "block"):
        g_dec[f"{k}_frac_hbm"] = round(g_dec[f"{k}_gbs"] / hbm, 3)
    tc = peaks["bf16_tflops"]
    g_pre["frac_tensor"] = round(g_pre["tops"] / tc, 3)
    cfg0["frac_tensor_back_to_back"] = round(cfg0["tops_back_to_back"] / tc, 3)
    blk_ops = block_ops(PREFILL_M)
    blk_us = pre["total_ms"] / 2000 * 1e3
    blk_tops = blk_ops / (blk_us * 1e-6) / 1e12

    line = {
        "metric": METRIC, "value": round(value, 2), "unit": "TOPS", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_per_step, 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "int8",
        "data": "synthetic",
        "config": {"workload": WORKLOAD, "tokens": STACK_M, "layers": STACK_LAYERS,
                   "linears_per_layer": [f"{n} {k}->{nn}" for n, k, nn in synth.TINYLLAMA_LINEARS],
                   "head": "{} {}->{}".format(*synth.TINYLLAMA_HEAD),
                   "chain": "q/k/v/gate/up read x_l; o reads q, down reads up; "
                            "x_l+1 = sat8(down + r_l)",
                   "int8_ops_per_step": ops, "calls_per_step": stack["launches_per_step"],
                   "kernel_launches_per_step": stack["kernels_per_step"],
                   "l2": "each step streams 1.03 GB of int8 weights (more than the 129 MB L2); "
                         "activations pass between layers through L2 as in a model",
                   "parallelism": f"replicas x{world}"},
        "roofline": {"bound": "tensor", "achieved": round(kern_tflops, 1), "peak": tc,
                     "unit": "TFLOP/s", "frac": round(kern_tflops / tc, 3),
                     "traffic": stack_traffic(),
                     "traffic_unit": "DRAM bytes per step (45 prefill2_kernel launches; ncu "
                                     "flushes caches per launch, so the f16 inputs are read "
                                     "from DRAM)",
                     "kernel": "mq::prefill2::prefill2_kernel (45 launches a step; the first "
                               "after the pre-pass widen16_kernel that widens x_0, the rest "
                               "read the f16 copies the previous launches wrote)",
                     "peak_note": f"dense f16 tensor peak = bf16 burst ({peaks['source']}), "
                                  "int8 ops run as exact f16 MMAs; achieved = the step's int8 "
                                  "ops / its device time (CUDA events around the timed steps, "
                                  "the pre-pass launches included)"},
        "clocks": stack["clocks"],
        "e2e": {"value": round(e2e_value, 2), "unit": "TOPS", "h2d_bytes_per_step": stack["h2d"],
                "d2h_bytes_per_step": stack["d2h"]},
        "gpu_launches": args.steps * stack["kernels_per_step"],
        "config0_single_linear_m128": cfg0,
        "config1_tinyllama_block_m1024": {
            "workload": BLOCK_WORKLOAD, "us_per_block": round(blk_us, 2),
            "tops": round(blk_tops, 1), "frac_tensor": round(blk_tops / tc, 3),
            "launches_per_step": pre["kernels"], "steps": 2000,
            "l2": f"{PREFILL_LAYERS} layers rotated ({PREFILL_LAYERS * 72} MB > 129 MB L2)",
            "traffic": prefill_traffic(), "traffic_unit": "bytes per launch"},
        "decode_w4a8": {"unit": "GB/s of int4 weights", "weight_bytes_per_block":
                        block_weight_bytes(4), "layers_rotated": DECODE_LAYERS,
                        "hbm_peak_gbs": hbm, **decode},
        "config4_gemma": {"prefill_m4096": g_pre, "decode_w4a8_m1": g_dec},
        "asym_prefill_w8a8": {**asym_pre, "symmetric_us_per_block": round(blk_us, 2)},
        "asym_decode_w4a8": {"unit": "GB/s of int4 weights",
                             "weights": "asymmetric per channel", **asym_dec},
        "a16": {"activations": "int16 in and out", "ops": "2 M K N per block", **a16,
                "w8a8_us_per_block": round(blk_us, 2),
                "w4a8_m1_stream_us": decode["m1"]["stream_us"]},
        "attention_w8a8_t1024": {**attention,
                                 "frac_hbm": round(attention["gbs"] / hbm, 3)},
        "attention_w8a16_t1024": {**attention16,
                                  "frac_hbm": round(attention16["gbs"] / hbm, 3)},
        "boundary_quantizers": {"unit": "GB/s of input + output bytes", **glue},
        "weight_pipeline": {"what": "fold of eq. 1 + quantize + pack + colsum, 7 linears, "
                                    "176 MB of f32 weights, one batched call (3 launches); "
                                    "per_linear_calls_us: seven calls (14-20 launches)", **wpipe},
    }
    if rank == 0 and world == 1:
        line["cpu_baseline"], parity = cpu_baseline(st, checks=checks)
        for leg, r in parity.items():
            node = line
            for key in leg.split("."):
                node = node[key]
            node["parity_sample"] = r
    if rank == 0:
        print(json.dumps(line), flush=True)
    dist.close()


if __name__ == "__main__":
    main()
