"""Seeded synthetic inputs shaped like the paper's workloads.

This module is shared by the CUDA path's tests/benchmark and by the oracle's
tests.  It holds none of the integer layer's arithmetic: it draws float data,
quantizes it to int8/int4 codes (the data-synthesis step the workloads are
defined by) and picks static output ranges from the *float* layer, the way a
calibration set would (Sec. 3.1, "static quantization statistics ... computed
on a holdout calibration set").  It never computes an integer accumulator,
a zero-point correction or a fixed-point requantization.

Value recipe (the paper trains on data this code does not have; these are
synthetic stand-ins with the same structure):
  * activations: N(0, 1) floats, 4 seeded input channels scaled x20 (outliers),
    quantized per tensor, asymmetric: sx = (max - min) / 255,
    zx = clamp(rint(-128 - min / sx), -128, 127), x = clamp(rint(x / sx) + zx).
  * weights: N(0, 0.02) (optionally 1% of output rows drawn as 0.02 * t(3)),
    symmetric per output channel: int8 sw = max|w_n| / 127, w in [-127, 127];
    int4 sw = max|w_n| / 7, w in [-8, 7].
  * output range: min/max of the float layer (dequantized activations times
    float weights) over calibration rows -> sy = (max - min) / 255 and
    zy = clamp(rint(-128 - min / sy), -128, 127).
Seeds: numpy PCG64 seeded with SeedSequence([1234, config, layer, linear, role]).
"""
from __future__ import annotations

import os
from dataclasses import dataclass, field

import numpy as np

BASE_SEED = 1234
ROLE_X, ROLE_W, ROLE_OUTLIER, ROLE_TROWS, ROLE_RES = 0, 1, 2, 3, 4

# Decoder-block linear shapes (name, K, N), TinyLlama-1.1B (hidden 2048,
# 32 heads, 4 KV heads x 64, FFN 5632) and Gemma-2B (hidden 2048, 8 heads x 256,
# 1 KV head, FFN 16384).
TINYLLAMA_LINEARS = [
    ("q", 2048, 2048), ("k", 2048, 256), ("v", 2048, 256), ("o", 2048, 2048),
    ("gate", 2048, 5632), ("up", 2048, 5632), ("down", 5632, 2048),
]
TINYLLAMA_HEAD = ("head", 2048, 32000)
GEMMA_LINEARS = [
    ("q", 2048, 2048), ("k", 2048, 256), ("v", 2048, 256), ("o", 2048, 2048),
    ("gate", 2048, 16384), ("up", 2048, 16384), ("down", 16384, 2048),
]
GEMMA_HEAD = ("head", 2048, 256000)


def rng_for(config: int, layer: int, linear: int, role: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(
        np.random.SeedSequence([BASE_SEED, config, layer, linear, role])))


def rint_clip(v: np.ndarray, lo: int, hi: int) -> np.ndarray:
    return np.clip(np.rint(v), lo, hi)


def float_activations(rng: np.random.Generator, m: int, k: int, n_outliers: int = 4,
                      outlier_scale: float = 20.0, orng: np.random.Generator | None = None):
    xf = rng.standard_normal((m, k), dtype=np.float32)
    orng = orng if orng is not None else rng
    if n_outliers and k:
        ch = orng.choice(k, size=min(n_outliers, k), replace=False)
        xf[:, ch] *= outlier_scale
    return xf


def quantize_per_tensor(xf: np.ndarray, bits: int = 8):
    """Asymmetric per-tensor codes (eqs. 2-4, shifted to the signed range):
    int8, or int16 with bits=16 (the 16-bit activations of Sec. 4.1 / 5.6)."""
    qmin, qmax = (-128, 127) if bits == 8 else (-32768, 32767)
    lo = float(min(xf.min(), 0.0)) if xf.size else -1.0
    hi = float(max(xf.max(), 0.0)) if xf.size else 1.0
    if hi - lo <= 0:
        hi = lo + 1.0
    s = np.float32((hi - lo) / float(qmax - qmin))
    z = int(rint_clip(np.array(qmin - lo / float(s)), qmin, qmax))
    t = xf / s
    t += np.float32(z)
    np.rint(t, out=t)
    np.clip(t, qmin, qmax, out=t)
    return t.astype(np.int8 if bits == 8 else np.int16), float(s), z


_POOL = None
ROW_BLOCK = 256


def _pool():
    global _POOL
    if _POOL is None:
        from concurrent.futures import ThreadPoolExecutor
        _POOL = ThreadPoolExecutor(max_workers=max(1, min(16, os.cpu_count() or 1)))
    return _POOL


def float_weights(rng: np.random.Generator, n: int, k: int, std: float = 0.02,
                  t_rows_frac: float = 0.0, trng: np.random.Generator | None = None):
    """N(0, std) weights; rows are drawn in blocks of ROW_BLOCK, block b from a
    generator seeded by (rng's first draw, b), in parallel threads."""
    wf = np.empty((n, k), np.float32)
    base = int(rng.integers(0, 2**63 - 1))

    def fill(b):
        r = np.random.Generator(np.random.PCG64(np.random.SeedSequence([base, b])))
        lo, hi = b * ROW_BLOCK, min(n, (b + 1) * ROW_BLOCK)
        r.standard_normal((hi - lo, k), dtype=np.float32, out=wf[lo:hi])
        wf[lo:hi] *= np.float32(std)

    list(_pool().map(fill, range((n + ROW_BLOCK - 1) // ROW_BLOCK)))
    if t_rows_frac > 0 and n:
        trng = trng if trng is not None else rng
        nrows = max(1, int(round(n * t_rows_frac)))
        rows = trng.choice(n, size=nrows, replace=False)
        wf[rows] = (trng.standard_t(3.0, size=(nrows, k)) * std).astype(np.float32)
    return wf


def quantize_per_channel_symmetric(wf: np.ndarray, bits: int, inplace: bool = False):
    """Symmetric per-output-channel codes; with inplace=True wf is overwritten."""
    qmax = 127 if bits == 8 else 7
    qmin = -127 if bits == 8 else -8
    if wf.size:
        amax = np.maximum(wf.max(axis=1), -wf.min(axis=1))
    else:
        amax = np.zeros(wf.shape[0], np.float32)
    amax = np.where(amax > 0, amax, np.float32(1e-8)).astype(np.float32)
    sw = (amax / np.float32(qmax)).astype(np.float32)
    t = wf if inplace else wf.copy()
    np.divide(t, sw[:, None], out=t)
    np.rint(t, out=t)
    np.clip(t, qmin, qmax, out=t)
    return t.astype(np.int8), sw


def quantize_asymmetric(wf: np.ndarray, bits: int, per_channel: bool, inplace: bool = False):
    """Asymmetric weight codes, the min-max quantizer of Sec. 4.2 applied to
    weights as in the paper's main W8A8 / W4A8 settings: s = (max - min) /
    (2^bits - 1), z = clamp(rint(qmin - min / s), qmin, qmax),
    w = clamp(rint(w / s) + z, qmin, qmax), with min/max over the whole tensor
    or over each output channel.  Returns (codes int8 [N,K], sw float32 [N],
    zw int32 [N]); per tensor, sw and zw repeat one value."""
    qmin, qmax = (-128, 127) if bits == 8 else (-8, 7)
    n = wf.shape[0]
    if per_channel:
        lo = wf.min(axis=1) if wf.size else np.zeros(n, np.float32)
        hi = wf.max(axis=1) if wf.size else np.zeros(n, np.float32)
    else:
        lo = np.full(n, wf.min() if wf.size else 0.0, np.float32)
        hi = np.full(n, wf.max() if wf.size else 0.0, np.float32)
    lo, hi = np.minimum(lo, 0).astype(np.float32), np.maximum(hi, 0).astype(np.float32)
    span = np.where(hi - lo > 0, hi - lo, np.float32(1e-8)).astype(np.float32)
    sw = (span / np.float32(qmax - qmin)).astype(np.float32)
    zw = rint_clip(np.float32(qmin) - lo / sw, qmin, qmax).astype(np.int32)
    t = wf if inplace else wf.copy()
    np.divide(t, sw[:, None], out=t)
    np.rint(t, out=t)
    t += zw[:, None].astype(np.float32)
    np.clip(t, qmin, qmax, out=t)
    return t.astype(np.int8), sw, zw


def output_range(yf: np.ndarray, bits: int = 8):
    """Static output (sy, zy) from the float layer's min/max (calibration)."""
    return quantize_params_from_range(float(yf.min()) if yf.size else -1.0,
                                      float(yf.max()) if yf.size else 1.0, bits)


def quantize_params_from_range(lo: float, hi: float, bits: int = 8):
    qmin, qmax = (-128, 127) if bits == 8 else (-32768, 32767)
    lo, hi = min(lo, 0.0), max(hi, 0.0)
    if hi - lo <= 0:
        hi = lo + 1.0
    s = np.float32((hi - lo) / float(qmax - qmin))
    z = int(rint_clip(np.array(qmin - lo / float(s)), qmin, qmax))
    return float(s), z


@dataclass
class LinearCase:
    """One quantized linear problem: int8 (or int16) x [M,K], int weights
    [N,K], scales; the output has the activations' width."""
    name: str
    x: np.ndarray          # int8 [M, K], or int16 for 16-bit activations
    zx: int
    sx: float
    w: np.ndarray          # int8 values [N, K] (int4 range if bits == 4)
    sw: np.ndarray         # float32 [N]
    bits: int
    sy: float
    zy: int
    residual: np.ndarray | None = None   # optional int8 [M, N]
    zw: np.ndarray | None = None         # int32 [N] weight zero point, None = symmetric
    meta: dict = field(default_factory=dict)

    @property
    def M(self): return self.x.shape[0]

    @property
    def K(self): return self.x.shape[1]

    @property
    def N(self): return self.w.shape[0]

    @property
    def abits(self): return 16 if self.x.dtype == np.int16 else 8


def make_linear(config: int, layer: int, linear: int, name: str, m: int, k: int, n: int,
                bits: int, t_rows_frac: float = 0.0, calib_rows: int = 64,
                x: tuple | None = None, weights: str = "symmetric") -> LinearCase:
    """A seeded linear problem.  `x` may pass (x_int8, sx, zx) to reuse inputs.
    `weights`: "symmetric" (per channel), "asym_tensor" or "asym_channel"."""
    if x is None:
        xf = float_activations(rng_for(config, layer, linear, ROLE_X), m, k,
                               orng=rng_for(config, layer, linear, ROLE_OUTLIER))
        xq, sx, zx = quantize_per_tensor(xf)
    else:
        xq, sx, zx = x
    wf = float_weights(rng_for(config, layer, linear, ROLE_W), n, k, t_rows_frac=t_rows_frac,
                       trng=rng_for(config, layer, linear, ROLE_TROWS))
    rows = min(m, calib_rows)
    # Float layer on the calibration rows: dequantized activations times the
    # float weights (the unquantized model's output), for static output ranges.
    xdq = (xq[:rows].astype(np.float32) - np.float32(zx)) * np.float32(sx)
    yf = xdq @ wf.T if rows and n else np.zeros((0, n), np.float32)
    sy, zy = output_range(yf)
    if weights == "symmetric":
        wq, sw = quantize_per_channel_symmetric(wf, bits, inplace=True)
        return LinearCase(name, xq, zx, sx, wq, sw, bits, sy, zy)
    if weights not in ("asym_tensor", "asym_channel"):
        raise ValueError(f"unknown weight scheme {weights!r}")
    wq, sw, zw = quantize_asymmetric(wf, bits, weights == "asym_channel", inplace=True)
    return LinearCase(name, xq, zx, sx, wq, sw, bits, sy, zy, zw=zw)


def paper_weight_scheme(name: str, bits: int) -> str:
    """The paper's main asymmetric settings (Sec. 5.1): W8A8 per tensor except
    the MLP's last projection (down) per channel; W4A8 per channel."""
    if bits == 4 or name == "down":
        return "asym_channel"
    return "asym_tensor"


def block_linears(config: int, m: int, bits: int, shapes=TINYLLAMA_LINEARS, layer: int = 0,
                  t_rows_frac: float = 0.0, shared_input: bool = False, asym: bool = False):
    """All linears of one decoder block, each with its own seeded input
    (or, with shared_input, q/k/v/gate/up reading one x of width 2048);
    with asym, weights follow paper_weight_scheme."""
    out = []
    shared = None
    for j, (name, k, n) in enumerate(shapes):
        xin = None
        if shared_input and name in ("q", "k", "v", "gate", "up"):
            if shared is None:
                xf = float_activations(rng_for(config, layer, 99, ROLE_X), m, k,
                                       orng=rng_for(config, layer, 99, ROLE_OUTLIER))
                shared = quantize_per_tensor(xf)
            xin = shared
        out.append(make_linear(config, layer, j, name, m, k, n, bits,
                               t_rows_frac=t_rows_frac, x=xin,
                               weights=paper_weight_scheme(name, bits) if asym else "symmetric"))
    return out


def residual_codes(config: int, layer: int, m: int, n: int, scale: float = 8.0) -> np.ndarray:
    """Seeded fixed int8 residual r of the chained stack, whose layers end with
    x_{l+1} = sat8(y_down + r)."""
    r = rng_for(config, layer, 0, ROLE_RES).standard_normal((m, n), dtype=np.float32) * scale
    return rint_clip(r, -128, 127).astype(np.int8)


def make_linear_a16(config: int, layer: int, linear: int, name: str, m: int, k: int, n: int,
                    bits: int, calib_rows: int = 64, x: tuple | None = None) -> LinearCase:
    """A seeded linear problem with 16-bit activations and outputs (W8A16 /
    W4A16): the float data of make_linear, activations quantized per tensor
    to int16, the output range calibrated on the 16-bit grid, weights
    symmetric per channel.  `x` may pass (x_int16, sx, zx) to reuse inputs."""
    if x is None:
        xf = float_activations(rng_for(config, layer, linear, ROLE_X), m, k,
                               orng=rng_for(config, layer, linear, ROLE_OUTLIER))
        xq, sx, zx = quantize_per_tensor(xf, bits=16)
    else:
        xq, sx, zx = x
    wf = float_weights(rng_for(config, layer, linear, ROLE_W), n, k)
    rows = min(m, calib_rows)
    xdq = (xq[:rows].astype(np.float32) - np.float32(zx)) * np.float32(sx)
    yf = xdq @ wf.T if rows and n else np.zeros((0, n), np.float32)
    sy, zy = output_range(yf, bits=16)
    wq, sw = quantize_per_channel_symmetric(wf, bits, inplace=True)
    return LinearCase(name, xq, zx, sx, wq, sw, bits, sy, zy)


def block_linears_a16(config: int, m: int, bits: int, shapes=TINYLLAMA_LINEARS,
                      layer: int = 0, shared_input: bool = False):
    """All linears of one decoder block with 16-bit activations (see
    block_linears)."""
    out = []
    shared = None
    for j, (name, k, n) in enumerate(shapes):
        xin = None
        if shared_input and name in ("q", "k", "v", "gate", "up"):
            if shared is None:
                xf = float_activations(rng_for(config, layer, 99, ROLE_X), m, k,
                                       orng=rng_for(config, layer, 99, ROLE_OUTLIER))
                shared = quantize_per_tensor(xf, bits=16)
            xin = shared
        out.append(make_linear_a16(config, layer, j, name, m, k, n, bits, x=xin))
    return out


def random_case_a16(seed: int, m: int, k: int, n: int, bits: int,
                    extreme: str | None = None) -> LinearCase:
    """Small seeded problem with int16 activations for parity tests, optionally
    with extreme codes: 'min', 'max' or 'mixed' (as random_case)."""
    rng = np.random.Generator(np.random.PCG64(np.random.SeedSequence([BASE_SEED, 16, seed])))
    wlo, whi = (-128, 127) if bits == 8 else (-8, 7)
    x = rng.integers(-32768, 32768, size=(m, k), dtype=np.int32).astype(np.int16)
    w = rng.integers(wlo, whi + 1, size=(n, k), dtype=np.int16).astype(np.int8)
    zx = int(rng.integers(-32768, 32768))
    if extreme == "min":
        x[:] = -32768
        w[:] = wlo
        zx = 32767
    elif extreme == "max":
        x[:] = 32767
        w[:] = whi
        zx = -32768
    elif extreme == "mixed":
        x[:] = np.where(rng.random((m, k)) < 0.5, -32768, 32767).astype(np.int16)
        w[:] = np.where(rng.random((n, k)) < 0.5, wlo, whi).astype(np.int8)
    sx = float(np.float32(rng.uniform(2e-5, 2e-4)))
    sw = rng.uniform(1e-4, 3e-3, size=n).astype(np.float32)
    sy = float(np.float32(rng.uniform(5e-6, 5e-5) * (16 if bits == 8 else 1)))
    zy = int(rng.integers(-16384, 16384))
    return LinearCase(f"a16rand{seed}", x, zx, sx, w, sw, bits, sy, zy)


def random_case(seed: int, m: int, k: int, n: int, bits: int, extreme: str | None = None) -> LinearCase:
    """Small seeded problem for parity tests, optionally with extreme values:
    'min' (all codes at the most negative value), 'max', or 'mixed'."""
    rng = np.random.Generator(np.random.PCG64(np.random.SeedSequence([BASE_SEED, 7, seed])))
    wlo, whi = (-128, 127) if bits == 8 else (-8, 7)
    x = rng.integers(-128, 128, size=(m, k), dtype=np.int16).astype(np.int8)
    w = rng.integers(wlo, whi + 1, size=(n, k), dtype=np.int16).astype(np.int8)
    zx = int(rng.integers(-128, 128))
    if extreme == "min":
        x[:] = -128
        w[:] = wlo
        zx = 127
    elif extreme == "max":
        x[:] = 127
        w[:] = whi
        zx = -128
    elif extreme == "mixed":
        x[:] = np.where(rng.random((m, k)) < 0.5, -128, 127).astype(np.int8)
        w[:] = np.where(rng.random((n, k)) < 0.5, wlo, whi).astype(np.int8)
    sx = float(np.float32(rng.uniform(0.005, 0.05)))
    sw = rng.uniform(1e-4, 3e-3, size=n).astype(np.float32)
    sy = float(np.float32(rng.uniform(0.02, 0.2)))
    zy = int(rng.integers(-128, 128))
    return LinearCase(f"rand{seed}", x, zx, sx, w, sw, bits, sy, zy)


def _quantize_with(yf: np.ndarray, s: float, z: int) -> np.ndarray:
    t = yf / np.float32(s)
    t += np.float32(z)
    np.rint(t, out=t)
    np.clip(t, -128, 127, out=t)
    return t.astype(np.int8)


@dataclass
class ChainLayer:
    """One layer of the chained stack: seven linears (q, k, v, o, gate, up,
    down), the seeded residual r and the input/output scales of each linear."""
    cases: list          # LinearCase per linear, x left empty (filled by the chain)
    residual: np.ndarray  # int8 [M, hidden]


def chain_stack(config: int, m: int, layers: int, shapes=TINYLLAMA_LINEARS, head=TINYLLAMA_HEAD,
                calib_rows: int = 32, t_rows_frac: float = 0.0):
    """Seeded 22-layer-style W8A8 stack.

    Layer l: q/k/v/gate/up read x_l; o reads q's int8 output (stand-in for the
    attention output); down reads up's int8 output (stand-in for SiLU(gate) *
    up); x_{l+1} = sat8(y_down + r_l).  Static output ranges come from a float
    shadow of the chain on the first `calib_rows` rows (dequantized codes times
    float weights, quantized with the chosen ranges -- the calibration pass).
    Returns (x0, sx0, zx0, [ChainLayer], head LinearCase with empty x)."""
    hidden = shapes[0][1]
    xf = float_activations(rng_for(config, 0, 99, ROLE_X), m, hidden,
                           orng=rng_for(config, 0, 99, ROLE_OUTLIER))
    x0, sx0, zx0 = quantize_per_tensor(xf)
    c = min(m, calib_rows)
    cur_codes, cur_s, cur_z = x0[:c], sx0, zx0
    out_layers = []
    for layer in range(layers):
        cases = []
        produced = {}
        for j, (name, k, n) in enumerate(shapes):
            if name == "o":
                in_codes, in_s, in_z = produced["q"]
            elif name == "down":
                in_codes, in_s, in_z = produced["up"]
            else:
                in_codes, in_s, in_z = cur_codes, cur_s, cur_z
            wf = float_weights(rng_for(config, layer, j, ROLE_W), n, k, t_rows_frac=t_rows_frac,
                               trng=rng_for(config, layer, j, ROLE_TROWS))
            xin = (in_codes.astype(np.float32) - np.float32(in_z)) * np.float32(in_s)
            yf = xin @ wf.T
            sy, zy = output_range(yf)
            produced[name] = (_quantize_with(yf, sy, zy), sy, zy)
            wq, sw = quantize_per_channel_symmetric(wf, 8, inplace=True)
            cases.append(LinearCase(name, np.zeros((0, k), np.int8), in_z, in_s, wq, sw, 8, sy, zy))
        r = residual_codes(config, layer, m, hidden)
        dcodes, ds, dz = produced["down"]
        nxt = np.clip(dcodes.astype(np.int16) + r[:c], -128, 127).astype(np.int8)
        out_layers.append(ChainLayer(cases, r))
        cur_codes, cur_s, cur_z = nxt, ds, dz
    name, k, n = head
    wf = float_weights(rng_for(config, layers, 0, ROLE_W), n, k)
    xin = (cur_codes.astype(np.float32) - np.float32(cur_z)) * np.float32(cur_s)
    sy, zy = output_range(xin @ wf.T)
    wq, sw = quantize_per_channel_symmetric(wf, 8, inplace=True)
    head_case = LinearCase(name, np.zeros((0, k), np.int8), cur_z, cur_s, wq, sw, 8, sy, zy)
    return x0, sx0, zx0, out_layers, head_case


@dataclass
class AttentionOperands:
    """The int8 operands of one layer's grouped-query attention matmuls: Q
    [T][heads * d], K and V [T][kv_heads * d] (per-tensor asymmetric codes
    with zero points zq, zk, zv) and P [heads][T][T], the codes of a causal
    softmax output (scale 1/255, zero point -128)."""
    q: np.ndarray
    k: np.ndarray
    v: np.ndarray
    p: np.ndarray
    zq: int
    zk: int
    zv: int
    zp: int
    heads: int
    kv_heads: int
    d: int


ROLE_ATT_Q, ROLE_ATT_K, ROLE_ATT_V, ROLE_ATT_P = 10, 11, 12, 13


def attention_operands(config: int, layer: int, t: int, heads: int = 32, kv_heads: int = 4,
                       d: int = 64, logit_std: float = 2.0, bits16: bool = False) -> AttentionOperands:
    """Seeded stand-ins for the inputs of Q K^T and P V at T = t tokens.

    Q, K, V: N(0, 1) activations (4 outlier channels x20) quantized per tensor
    like every other activation here.  P: rows of softmax(N(0, logit_std)
    logits) over keys s <= query t (the causal mask; masked keys get
    probability 0), coded as clip(rint(255 p) - 128, -128, 127).  With bits16
    (the W8A16 setting), Q and P are 16-bit codes: Q quantized per tensor to
    int16, P coded as clip(rint(65535 p) - 32768, -32768, 32767), zero point
    -32768; K and V stay 8-bit."""
    codes = []
    for role, width in ((ROLE_ATT_Q, heads * d), (ROLE_ATT_K, kv_heads * d),
                        (ROLE_ATT_V, kv_heads * d)):
        xf = float_activations(rng_for(config, layer, role, ROLE_X), t, width,
                               orng=rng_for(config, layer, role, ROLE_OUTLIER))
        q, _, z = quantize_per_tensor(xf, 16 if (bits16 and role == ROLE_ATT_Q) else 8)
        codes.append((q, z))
    rng = rng_for(config, layer, ROLE_ATT_P, ROLE_X)
    p = np.empty((heads, t, t), np.int16 if bits16 else np.int8)
    future = np.triu(np.ones((t, t), bool), 1)
    for h in range(heads):
        logits = rng.standard_normal((t, t), dtype=np.float32) * np.float32(logit_std)
        logits[future] = -np.inf
        logits -= logits.max(axis=1, keepdims=True)
        e = np.exp(logits)
        e /= e.sum(axis=1, keepdims=True)
        if bits16:
            p[h] = rint_clip(e * np.float32(65535.0) - np.float32(32768.0), -32768,
                             32767).astype(np.int16)
        else:
            p[h] = rint_clip(e * np.float32(255.0) - np.float32(128.0), -128, 127).astype(np.int8)
    (q, zq), (k, zk), (v, zv) = codes
    return AttentionOperands(q, k, v, p, zq, zk, zv, -32768 if bits16 else -128, heads, kv_heads, d)
