"""Pins of the CPU oracle against facts that do not come from the oracle itself.

Each check ties the oracle to something independent of its code:
  * hand-derived worked examples (tests/golden/tiny_linear.json);
  * exhaustive brute force (K = 1 over every int8 x, w and zero point);
  * the zero-point identity sum((x - zx) w) = sum(x w) - zx colsum(w), with the
    right side from numpy's int64 matmul;
  * the exact dequantization invariant: with power-of-two scales the float64
    matmul of dequantized operands equals acc * sx * sw exactly;
  * closed-form requantization (multiplier 2^-t is a rounding right shift) and
    exact-rational rounding at ties (fractions.Fraction);
  * eq. 4's quantizer with the real multiplier, to within one step at near-ties;
  * the requant parameters' 2^-31 relative error bound.
A mutation test plants typical mistakes in a copy of the oracle and checks
that the battery above rejects every one of them.
"""
import json
import os
import random
from fractions import Fraction

import numpy as np
import pytest

import oracle
from oracle import Oracle
from paper_2408_13933_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "tiny_linear.json")


def load_golden():
    with open(GOLDEN) as f:
        return json.load(f)


# ----------------------------------------------------------------------------
# Pin battery: each returns None on success and raises AssertionError on a
# mismatch.  They take an Oracle so that the mutation test can reuse them.
# ----------------------------------------------------------------------------

def pin_golden(orc: Oracle):
    g = load_golden()
    for c in g["cases"]:
        w = np.array(c["w"], np.int8)
        packed, colsum = orc.pack(w, c["bits"])
        assert colsum.tolist() == c["colsum"], c["name"]
        if "packed" in c:
            assert packed.tolist() == c["packed"], c["name"]
        y, acc = orc.linear(np.array(c["x"], np.int8), c["zx"], packed, c["bits"], w.shape[0],
                            np.array(c["M0"], np.int32), np.array(c["shift"], np.int32),
                            c["zy"], want_acc=True)
        assert acc.tolist() == c["acc"], c["name"]
        assert y.tolist() == c["y"], c["name"]
    rq = g["requant_one"]
    for r in rq["rows"]:
        assert orc.requant_one(r["acc"], rq["M0"], rq["shift"], r["zy"]) == r["y"], r
    rp = g["requant_params"]
    m0, sh = orc.requant_params(rp["sx"], np.array(rp["sw"], np.float32), rp["sy"])
    assert m0.tolist() == rp["M0"] and sh.tolist() == rp["shift"]


def pin_k1_exhaustive(orc: Oracle, zxs=range(-128, 128)):
    xs = np.arange(-128, 128, dtype=np.int16).astype(np.int8).reshape(256, 1)
    ws = np.arange(-128, 128, dtype=np.int16).astype(np.int8).reshape(256, 1)
    packed, _ = orc.pack(ws, 8)
    m0 = np.full(256, 1 << 30, np.int32)
    sh = np.full(256, 31, np.int32)
    for zx in zxs:
        _, acc = orc.linear(xs, zx, packed, 8, 256, m0, sh, 0, want_acc=True)
        ref = np.outer(xs[:, 0].astype(np.int64) - zx, ws[:, 0].astype(np.int64))
        assert np.array_equal(acc.astype(np.int64), ref), zx


def pin_int4_exhaustive_pairs(orc: Oracle):
    # every pair of int4 weights against a spread of activations (K = 2)
    ws = np.array([[a, b] for a in range(-8, 8) for b in range(-8, 8)], np.int8)
    xs = np.array([[a, b] for a in (-128, -77, -1, 0, 1, 64, 127) for b in (-128, -3, 0, 5, 127)],
                  np.int8)
    packed, colsum = orc.pack(ws, 4)
    assert np.array_equal(colsum, ws.astype(np.int32).sum(1))
    m0 = np.full(ws.shape[0], 1 << 30, np.int32)
    sh = np.full(ws.shape[0], 31, np.int32)
    for zx in (-128, -5, 0, 3, 127):
        _, acc = orc.linear(xs, zx, packed, 4, ws.shape[0], m0, sh, 0, want_acc=True)
        ref = (xs.astype(np.int64) - zx) @ ws.astype(np.int64).T
        assert np.array_equal(acc.astype(np.int64), ref), zx


def pin_zero_point_identity(orc: Oracle, seeds=(1, 2, 3)):
    for seed in seeds:
        for bits in (8, 4):
            for extreme in (None, "min", "max", "mixed"):
                c = synth.random_case(seed, 7, 96, 13, bits, extreme)
                packed, colsum = orc.pack(c.w, bits)
                m0, sh = orc.requant_params(c.sx, c.sw, c.sy)
                _, acc = orc.linear(c.x, c.zx, packed, bits, c.N, m0, sh, c.zy, want_acc=True)
                xw = c.x.astype(np.int64) @ c.w.astype(np.int64).T
                ref = xw - c.zx * c.w.astype(np.int64).sum(1)[None, :]
                assert np.array_equal(acc.astype(np.int64), ref), (seed, bits, extreme)
                assert np.array_equal(colsum.astype(np.int64), c.w.astype(np.int64).sum(1))


def pin_exact_dequant(orc: Oracle):
    rng = np.random.default_rng(5)
    for bits in (8, 4):
        c = synth.random_case(11, 9, 160, 17, bits)
        a = 7
        b = rng.integers(3, 12, size=c.N)
        sx = 2.0 ** -a
        sw = (2.0 ** -b.astype(np.float64))
        packed, _ = orc.pack(c.w, bits)
        m0, sh = orc.requant_params(1.0, np.ones(c.N, np.float32), 1.0)
        _, acc = orc.linear(c.x, c.zx, packed, bits, c.N, m0, sh, 0, want_acc=True)
        xd = (c.x.astype(np.float64) - c.zx) * sx
        wd = c.w.astype(np.float64) * sw[:, None]
        yf = xd @ wd.T            # float64 BLAS; every partial sum is exact
        assert np.array_equal(yf, acc.astype(np.float64) * sx * sw[None, :])


def _round_half_up_frac(fr: Fraction) -> int:
    import math
    return math.floor(fr + Fraction(1, 2))


def pin_requant_closed_form(orc: Oracle):
    rng = random.Random(3)
    for t in (1, 2, 5, 8, 13, 20, 30):
        for _ in range(300):
            acc = rng.randint(-(1 << 31) + 1, (1 << 31) - 1) if rng.random() < 0.5 \
                else rng.randint(-4 << t, 4 << t)
            zy = rng.randint(-128, 127)
            q = (acc + (1 << (t - 1))) >> t      # Python >> floors: round half up
            want = max(-128, min(127, zy + q))
            assert orc.requant_one(acc, 1 << 30, 30 + t, zy) == want, (t, acc, zy)


def pin_requant_ties(orc: Oracle):
    rng = random.Random(4)
    for _ in range(400):
        s = rng.randint(1, 62)
        m0 = rng.randint(1 << 30, (1 << 31) - 1)
        # accumulators just around the tie points j + 1/2 of acc*m0/2^s
        j = rng.randint(-200, 200)
        centre = int(Fraction(2 * j + 1, 2) * Fraction(1 << s, m0))
        for acc in range(centre - 2, centre + 3):
            if not -(1 << 31) < acc < (1 << 31):
                continue
            q = _round_half_up_frac(Fraction(acc * m0, 1 << s))
            want = max(-128, min(127, q))
            assert orc.requant_one(acc, m0, s, 0) == want, (acc, m0, s)
    # exact ties for small shifts, both signs
    for s in range(1, 9):
        for acc in range(-300, 301):
            q = _round_half_up_frac(Fraction(acc * (1 << 30), 1 << s))
            assert orc.requant_one(acc, 1 << 30, s, 0) == max(-128, min(127, q)), (acc, s)


def pin_requant_vs_eq4(orc: Oracle):
    """Requantization with the fixed-point multiplier against eq. 4 applied to
    the real-valued layer output (float64): equal except at near-ties."""
    c = synth.make_linear(0, 0, 0, "q", 64, 256, 96, 8)
    packed, _ = orc.pack(c.w, 8)
    m0, sh = orc.requant_params(c.sx, c.sw, c.sy)
    y, acc = orc.linear(c.x, c.zx, packed, 8, c.N, m0, sh, c.zy, want_acc=True)
    yf = acc.astype(np.float64) * (c.sx * c.sw.astype(np.float64))[None, :]
    # eq. 4 with alpha = sy and beta = -(zy + 128), shifted to signed int8
    ref = np.clip(np.floor(yf / c.sy + 0.5) + c.zy, -128, 127)
    diff = np.abs(y.astype(np.int64) - ref)
    assert diff.max() <= 1
    assert (diff != 0).mean() < 1e-3
    # the calibration must leave most outputs unsaturated for the check to bite
    assert np.mean(np.abs(y.astype(np.int64)) < 127) > 0.9


def pin_requant_params_bound(orc: Oracle):
    rng = np.random.default_rng(9)
    for _ in range(20):
        sx = np.float32(rng.uniform(1e-3, 1.0))
        sy = np.float32(rng.uniform(1e-3, 1.0))
        sw = rng.uniform(1e-5, 1e-1, size=64).astype(np.float32)
        m0, sh = orc.requant_params(float(sx), sw, float(sy))
        for n in range(64):
            exact = Fraction(float(sx)) * Fraction(float(sw[n])) / Fraction(float(sy))
            got = Fraction(int(m0[n]), 1 << int(sh[n]))
            assert (1 << 30) <= int(m0[n]) < (1 << 31)
            assert 1 <= int(sh[n]) <= 62
            assert abs(got - exact) / exact <= Fraction(1, 1 << 31) + Fraction(1, 1 << 52)
    # powers of two are exact
    for t in range(0, 30):
        m0, sh = orc.requant_params(1.0, np.array([2.0 ** -t], np.float32), 1.0)
        # 2^-t = 0.5 * 2^(1-t): M0 = 0.5 * 2^31, shift = 31 - (1 - t)
        assert (int(m0[0]), int(sh[0])) == (1 << 30, 30 + t)


# ---- asymmetric weights (per-channel weight zero point zw) ----------------

def pin_asym_k1_exhaustive(orc: Oracle):
    # every int8 x against every int8 w (K = 1) for several zero-point pairs:
    # acc = (x - zx) (w - zw), checked against the product of Python integers
    xs = np.arange(-128, 128, dtype=np.int16).astype(np.int8).reshape(256, 1)
    ws = np.arange(-128, 128, dtype=np.int16).astype(np.int8).reshape(256, 1)
    packed, _ = orc.pack(ws, 8)
    m0 = np.full(256, 1 << 30, np.int32)
    sh = np.full(256, 31, np.int32)
    for zx, zw in ((-128, 127), (0, -128), (5, -3), (127, 0), (-1, 1)):
        _, acc = orc.linear(xs, zx, packed, 8, 256, m0, sh, 0, want_acc=True,
                            zw=np.full(256, zw, np.int32))
        ref = np.array([[(int(a) - zx) * (int(b) - zw) for b in ws[:, 0]] for a in xs[:, 0]])
        assert np.array_equal(acc.astype(np.int64), ref), (zx, zw)


def pin_asym_int4_pairs(orc: Oracle):
    # every pair of int4 weights (K = 2), every int4 weight zero point
    ws = np.array([[a, b] for a in range(-8, 8) for b in range(-8, 8)], np.int8)
    xs = np.array([[a, b] for a in (-128, -9, 0, 3, 127) for b in (-128, 0, 77, 127)], np.int8)
    packed, _ = orc.pack(ws, 4)
    m0 = np.full(ws.shape[0], 1 << 30, np.int32)
    sh = np.full(ws.shape[0], 31, np.int32)
    for zw in range(-8, 8):
        for zx in (-128, 0, 127):
            _, acc = orc.linear(xs, zx, packed, 4, ws.shape[0], m0, sh, 0, want_acc=True,
                                zw=np.full(ws.shape[0], zw, np.int32))
            ref = (xs.astype(np.int64) - zx) @ (ws.astype(np.int64) - zw).T
            assert np.array_equal(acc.astype(np.int64), ref), (zw, zx)


def pin_asym_identity(orc: Oracle, seeds=(4, 5)):
    # sum((x - zx)(w - zw)) = sum(x w) - zx colsum(w) - zw rowsum(x) + K zx zw,
    # with per-channel zw spanning the code range
    for seed in seeds:
        rng = np.random.default_rng(seed)
        for bits in (8, 4):
            lo, hi = (-128, 127) if bits == 8 else (-8, 7)
            for extreme in (None, "min", "max", "mixed"):
                c = synth.random_case(seed, 6, 96, 11, bits, extreme)
                zw = rng.integers(lo, hi + 1, size=c.N).astype(np.int32)
                zw[0], zw[-1] = lo, hi
                packed, colsum = orc.pack(c.w, bits)
                m0, sh = orc.requant_params(c.sx, c.sw, c.sy)
                _, acc = orc.linear(c.x, c.zx, packed, bits, c.N, m0, sh, c.zy, want_acc=True,
                                    zw=zw)
                x64, w64 = c.x.astype(np.int64), c.w.astype(np.int64)
                ref = (x64 @ w64.T - c.zx * w64.sum(1)[None, :]
                       - zw.astype(np.int64)[None, :] * x64.sum(1)[:, None]
                       + c.K * c.zx * zw.astype(np.int64)[None, :])
                assert np.array_equal(acc.astype(np.int64), ref), (seed, bits, extreme)


def pin_asym_reduces_to_symmetric(orc: Oracle):
    for bits in (8, 4):
        c = synth.random_case(6, 5, 64, 9, bits, "mixed")
        packed, _ = orc.pack(c.w, bits)
        m0, sh = orc.requant_params(c.sx, c.sw, c.sy)
        y0, a0 = orc.linear(c.x, c.zx, packed, bits, c.N, m0, sh, c.zy, want_acc=True)
        y1, a1 = orc.linear(c.x, c.zx, packed, bits, c.N, m0, sh, c.zy, want_acc=True,
                            zw=np.zeros(c.N, np.int32))
        assert np.array_equal(a0, a1) and np.array_equal(y0, y1)


def pin_asym_exact_dequant(orc: Oracle):
    # power-of-two scales: the float64 matmul of the dequantized operands
    # s_x (x - zx) and s_w (w - zw) is exact and equals acc s_x s_w
    rng = np.random.default_rng(8)
    for bits in (8, 4):
        lo, hi = (-128, 127) if bits == 8 else (-8, 7)
        c = synth.random_case(12, 9, 160, 17, bits)
        zw = rng.integers(lo, hi + 1, size=c.N).astype(np.int32)
        sx = 2.0 ** -6
        sw = 2.0 ** -rng.integers(3, 12, size=c.N).astype(np.float64)
        packed, _ = orc.pack(c.w, bits)
        m0, sh = orc.requant_params(1.0, np.ones(c.N, np.float32), 1.0)
        _, acc = orc.linear(c.x, c.zx, packed, bits, c.N, m0, sh, 0, want_acc=True, zw=zw)
        xd = (c.x.astype(np.float64) - c.zx) * sx
        wd = (c.w.astype(np.float64) - zw[:, None]) * sw[:, None]
        assert np.array_equal(xd @ wd.T, acc.astype(np.float64) * sx * sw[None, :])


# ---- 16-bit activations (W8A16 / W4A16) -------------------------------------

def _py_requant16(acc: int, m0: int, s: int, zy: int) -> int:
    # round half up of the exact rational acc m0 / 2^s, saturated to int16
    return max(-32768, min(32767, zy + _round_half_up_frac(Fraction(acc * m0, 1 << s))))


def pin_a16_k1_exhaustive(orc: Oracle):
    # every int16 code against int8 weights at the ends and middle of the
    # range (K = 1), several activation zero points: acc = (x - zx) w exactly
    xs = np.arange(-32768, 32768, dtype=np.int64).astype(np.int16).reshape(-1, 1)
    w = np.array([[-128], [-1], [0], [1], [127], [-77]], np.int8)
    packed, _ = orc.pack(w, 8)
    m0 = np.full(w.shape[0], 1 << 30, np.int32)
    sh = np.full(w.shape[0], 40, np.int32)
    for zx in (-32768, -1, 0, 12345, 32767):
        y, acc = orc.linear_a16(xs, zx, packed, 8, w.shape[0], m0, sh, 7, want_acc=True)
        ref = (xs.astype(np.int64) - zx) * w[:, 0].astype(np.int64)[None, :]
        assert np.array_equal(acc, ref), zx
        # requant of a sample of them against exact rationals (shift 40: acc / 2^10)
        for i in range(0, xs.shape[0], 4099):
            for j in range(w.shape[0]):
                assert int(y[i, j]) == _py_requant16(int(ref[i, j]), 1 << 30, 40, 7), (zx, i, j)


def pin_a16_int4_pairs(orc: Oracle):
    # K = 2, every pair of int4 weights, activation pairs at the range ends
    w = np.array([[a, b] for a in range(-8, 8) for b in range(-8, 8)], np.int8)
    packed, _ = orc.pack(w, 4)
    xs = np.array([[-32768, 32767], [32767, -32768], [-1, 1], [12345, -23456], [0, 0]],
                  np.int16)
    m0 = np.full(w.shape[0], 1 << 30, np.int32)
    sh = np.full(w.shape[0], 31, np.int32)
    for zx in (-32768, 0, 32767):
        _, acc = orc.linear_a16(xs, zx, packed, 4, w.shape[0], m0, sh, 0, want_acc=True)
        ref = (xs.astype(np.int64) - zx) @ w.astype(np.int64).T
        assert np.array_equal(acc, ref), zx


def pin_a16_matmul_and_brute_force(orc: Oracle):
    # acc against numpy's int64 matmul (exact) on random codes, and every
    # output of a small case against round half up of exact rationals
    for seed, bits in ((1, 8), (2, 4), (3, 8)):
        c = synth.random_case_a16(seed, 7, 96, 13, bits)
        packed, _ = orc.pack(c.w, bits)
        m0, sh = orc.requant_params(c.sx, c.sw, c.sy)
        y, acc = orc.linear_a16(c.x, c.zx, packed, bits, c.N, m0, sh, c.zy, want_acc=True)
        ref = (c.x.astype(np.int64) - c.zx) @ c.w.astype(np.int64).T
        assert np.array_equal(acc, ref), seed
        for m in range(c.M):
            for n in range(c.N):
                assert int(y[m, n]) == _py_requant16(int(ref[m, n]), int(m0[n]), int(sh[n]),
                                                     c.zy), (seed, m, n)


def pin_a16_large_accumulators(orc: Oracle):
    # extreme codes with |acc| up to 65535 * 128 * 1024 ~ 2^33 (int8 weights)
    # or 65535 * 8 * 8192 ~ 2^32 (int4), outside int32, against numpy's int64
    # matmul and exact rationals
    for extreme in ("min", "max", "mixed"):
        for bits, k in ((8, 1024), (4, 8192)):
            c = synth.random_case_a16(61, 3, k, 6, bits, extreme)
            packed, _ = orc.pack(c.w, bits)
            m0, sh = orc.requant_params(c.sx, c.sw, c.sy)
            y, acc = orc.linear_a16(c.x, c.zx, packed, bits, c.N, m0, sh, c.zy, want_acc=True)
            ref = (c.x.astype(np.int64) - c.zx) @ c.w.astype(np.int64).T
            assert np.array_equal(acc, ref), (extreme, bits)
            if extreme != "mixed":
                assert np.abs(ref).max() >= (1 << 31)
            for m in range(c.M):
                for n in range(c.N):
                    assert int(y[m, n]) == _py_requant16(int(ref[m, n]), int(m0[n]),
                                                         int(sh[n]), c.zy)


def pin_a16_reduces_to_int8(orc: Oracle):
    # activation codes and zero points inside the int8 range: the same
    # accumulator as the (separately pinned) int8 layer
    for bits in (8, 4):
        c = synth.random_case(21, 9, 128, 11, bits)
        packed, _ = orc.pack(c.w, bits)
        m0, sh = orc.requant_params(c.sx, c.sw, c.sy)
        _, a8 = orc.linear(c.x, c.zx, packed, bits, c.N, m0, sh, c.zy, want_acc=True)
        _, a16 = orc.linear_a16(c.x.astype(np.int16), c.zx, packed, bits, c.N, m0, sh, c.zy,
                                want_acc=True)
        assert np.array_equal(a16, a8.astype(np.int64))


def pin_a16_byte_planes(orc: Oracle):
    # x = 256 hi + (lo - 128) + 128 with hi the signed high byte and lo the
    # unsigned low byte: the int16 accumulator is 256 times the int8 layer on
    # the hi plane plus the int8 layer on the (lo - 128) plane plus
    # (128 - zx) colsum, each int8 layer with zero point 0
    for bits in (8, 4):
        c = synth.random_case_a16(31 + bits, 6, 160, 9, bits, "mixed" if bits == 4 else None)
        packed, colsum = orc.pack(c.w, bits)
        m0, sh = orc.requant_params(c.sx, c.sw, c.sy)
        _, acc = orc.linear_a16(c.x, c.zx, packed, bits, c.N, m0, sh, c.zy, want_acc=True)
        u = c.x.view(np.uint16).astype(np.int64)
        hi = ((u >> 8).astype(np.uint8)).view(np.int8)
        lo = ((u & 255) - 128).astype(np.int8)
        _, a_hi = orc.linear(hi, 0, packed, bits, c.N, m0, sh, 0, want_acc=True)
        _, a_lo = orc.linear(lo, 0, packed, bits, c.N, m0, sh, 0, want_acc=True)
        want = (256 * a_hi.astype(np.int64) + a_lo.astype(np.int64)
                + (128 - c.zx) * colsum.astype(np.int64)[None, :])
        assert np.array_equal(acc, want), bits


def pin_a16_exact_dequant(orc: Oracle):
    # power-of-two scales: the float64 matmul of sx (x - zx) and sw w is
    # exact (|partial sums| < 2^53) and equals acc sx sw
    rng = np.random.default_rng(15)
    for bits in (8, 4):
        c = synth.random_case_a16(41, 9, 160, 17, bits)
        sx = 2.0 ** -20
        sw = 2.0 ** -rng.integers(3, 12, size=c.N).astype(np.float64)
        packed, _ = orc.pack(c.w, bits)
        m0, sh = orc.requant_params(1.0, np.ones(c.N, np.float32), 1.0)
        _, acc = orc.linear_a16(c.x, c.zx, packed, bits, c.N, m0, sh, 0, want_acc=True)
        xd = (c.x.astype(np.float64) - c.zx) * sx
        wd = c.w.astype(np.float64) * sw[:, None]
        assert np.array_equal(xd @ wd.T, acc.astype(np.float64) * sx * sw[None, :])


def pin_a16_requant_closed_form_and_saturation(orc: Oracle):
    # multiplier 2^-t (M0 = 2^30, shift 30 + t) is a rounding right shift,
    # for accumulators up to the 2^40 bound; the output saturates at the
    # int16 ends, not the int8 ones
    rng = random.Random(16)
    for t in (1, 3, 9, 17, 25, 32):
        for _ in range(300):
            acc = rng.randint(-(1 << 40), 1 << 40) if rng.random() < 0.5 \
                else rng.randint(-(3 << t) * 40000, (3 << t) * 40000)
            zy = rng.randint(-32768, 32767)
            want = max(-32768, min(32767, zy + ((acc + (1 << (t - 1))) >> t)))
            assert orc.requant_one_a16(acc, 1 << 30, 30 + t, zy) == want, (t, acc, zy)
    # exact ties, both signs
    for s in range(1, 9):
        for acc in range(-300, 301):
            assert orc.requant_one_a16(acc, 1 << 30, s, 0) == _py_requant16(acc, 1 << 30, s, 0)
    assert orc.requant_one_a16(1 << 39, (1 << 31) - 1, 31, 0) == 32767
    assert orc.requant_one_a16(-(1 << 39), (1 << 31) - 1, 31, 0) == -32768
    assert orc.requant_one_a16(200, 1 << 30, 30, 32700) == 32767
    assert orc.requant_one_a16(-200, 1 << 30, 30, -32700) == -32768
    assert orc.requant_one_a16(200, 1 << 30, 30, -100) == 100


def pin_a16_requant_vs_eq4(orc: Oracle):
    """The 16-bit layer against eq. 4 on the 16-bit output grid applied to
    the real-valued layer output (float64): equal except at near-ties."""
    c = synth.make_linear_a16(0, 0, 0, "q", 64, 256, 96, 8)
    packed, _ = orc.pack(c.w, 8)
    m0, sh = orc.requant_params(c.sx, c.sw, c.sy)
    y, acc = orc.linear_a16(c.x, c.zx, packed, 8, c.N, m0, sh, c.zy, want_acc=True)
    yf = acc.astype(np.float64) * (c.sx * c.sw.astype(np.float64))[None, :]
    ref = np.clip(np.floor(yf / c.sy + 0.5) + c.zy, -32768, 32767)
    diff = np.abs(y.astype(np.int64) - ref)
    assert diff.max() <= 1
    assert (diff != 0).mean() < 1e-3
    assert np.mean(np.abs(y.astype(np.int64)) < 32767) > 0.9


# ---- boundary quantizers (float / int16 / int8 domains) ----------------------

def _f32_nearest(fr: Fraction) -> float:
    """The f32 value nearest to the rational fr, ties to even mantissa (IEEE
    round to nearest), found among the f32 neighbours of a first guess."""
    g = np.float32(float(fr))
    cands = {np.float32(g), np.nextafter(g, np.float32(np.inf)),
             np.nextafter(g, np.float32(-np.inf))}
    best = None
    for c in cands:
        if not np.isfinite(c):
            continue
        d = abs(Fraction(float(c)) - fr)
        key = (d, int(np.array(c, np.float32).view(np.int32)) & 1)  # ties: even mantissa first
        if best is None or key < best[0]:
            best = (key, c)
    return float(best[1])


def _quantize_ref(x: float, alpha: float, z: int, bits: int) -> int:
    lo, hi = (-128, 127) if bits == 8 else (-32768, 32767)
    if np.isnan(x):
        return z
    if np.isinf(x):
        return hi if x > 0 else lo
    qf = _f32_nearest(Fraction(float(np.float32(x))) / Fraction(float(np.float32(alpha))))
    return max(lo, min(hi, round(qf) + z))  # Python round: ties to even


def pin_quantize_exact(orc: Oracle):
    rng = np.random.default_rng(101)
    for bits in (8, 16):
        for alpha, z in ((np.float32(0.0371), -3), (np.float32(1.0 / 3.0), 17),
                         (np.float32(2.5e-4), -1000 if bits == 16 else -100)):
            scale = 140 if bits == 8 else 40000
            x = (rng.standard_normal(1500) * float(alpha) * scale / 3).astype(np.float32)
            # values whose quotient lies within an ulp of a .5 tie
            k = rng.integers(-scale, scale, size=300)
            near = ((k + 0.5) * float(alpha)).astype(np.float32)
            x = np.concatenate([x, near, np.nextafter(near, np.float32(np.inf)),
                                np.nextafter(near, np.float32(-np.inf)),
                                np.array([np.inf, -np.inf, np.nan, 0.0, -0.0], np.float32)])
            zz = z if bits == 16 else max(-128, min(127, z))
            got = orc.quantize(x, float(alpha), zz, bits)
            for i in range(x.size):
                assert int(got[i]) == _quantize_ref(float(x[i]), float(alpha), zz, bits), \
                    (bits, float(alpha), i, float(x[i]))


def pin_quantize_ties_and_invariants(orc: Oracle):
    # power-of-two scale: the quotient (k + 1/2) is exact, ties go to even
    k = np.arange(-100, 100)
    x = ((k + 0.5) / 8).astype(np.float32)
    got = orc.quantize(x, 0.125, 0, 8).astype(np.int64)
    want = np.where(k % 2 == 0, k, k + 1)
    assert np.array_equal(got, np.clip(want, -128, 127))
    # monotone, and within half a step of the value wherever not saturated
    rng = np.random.default_rng(102)
    xs = np.sort(rng.uniform(-6, 6, 5000).astype(np.float32))
    for bits, alpha, z in ((8, 0.03, 5), (16, 1e-4, -77)):
        q = orc.quantize(xs, alpha, z, bits).astype(np.int64)
        assert np.all(np.diff(q) >= 0)
        lo, hi = (-128, 127) if bits == 8 else (-32768, 32767)
        inside = (q > lo) & (q < hi)
        a64 = np.float64(np.float32(alpha))
        err = np.abs((q - z) * a64 - xs.astype(np.float64))
        # half a step, plus the f32 rounding of the quotient (half an ulp of |x / alpha|)
        bound = a64 * (0.5 + np.abs(xs.astype(np.float64) / a64) * 2.0 ** -24) * (1 + 1e-9)
        assert np.all(err[inside] <= bound[inside])
        assert inside.mean() > 0.5


def pin_dequantize_exact(orc: Oracle):
    for bits, alpha, z in ((8, np.float32(0.0371), -3), (16, np.float32(2.5e-4), 1234)):
        lo, hi = (-128, 127) if bits == 8 else (-32768, 32767)
        q = np.arange(lo, hi + 1, dtype=np.int64).astype(np.int8 if bits == 8 else np.int16)
        f = orc.dequantize(q, float(alpha), z)
        for i in range(0, q.size, 1 if bits == 8 else 97):
            want = _f32_nearest(Fraction(int(q[i]) - z) * Fraction(float(alpha)))
            assert float(f[i]) == want, (bits, int(q[i]))


def pin_requantize_exhaustive(orc: Oracle):
    # every int16 code to int8 and every int8 code to int16, for several
    # multipliers, against floor((q - zx) M0 / 2^s + 1/2) on Python integers
    rng = random.Random(103)
    all16 = np.arange(-32768, 32768, dtype=np.int64).astype(np.int16)
    all8 = np.arange(-128, 128, dtype=np.int64).astype(np.int8)
    for q, out_bits in ((all16, 8), (all8, 16), (all16, 16), (all8, 8)):
        in_lo, in_hi = (-128, 127) if q.dtype == np.int8 else (-32768, 32767)
        lo, hi = (-128, 127) if out_bits == 8 else (-32768, 32767)
        for _ in range(4):
            m0 = rng.randint(1 << 30, (1 << 31) - 1)
            s = rng.randint(20, 45)
            zx, zy = rng.randint(in_lo, in_hi), rng.randint(lo, hi)
            got = orc.requantize(q, zx, m0, s, zy, out_bits)
            for i in range(0, q.size, 1 if q.size <= 256 else 61):
                v = Fraction((int(q[i]) - zx) * m0, 1 << s)
                want = max(lo, min(hi, zy + _round_half_up_frac(v)))
                assert int(got[i]) == want, (out_bits, i, m0, s)
            # all codes at once with exact integer floor division
            v = (q.astype(np.int64) - zx) * m0 + (1 << (s - 1))
            want = np.clip(zy + np.floor_divide(v, 1 << s), lo, hi)
            assert np.array_equal(got.astype(np.int64), want)


def pin_requantize_vs_eq4(orc: Oracle):
    # int16 codes of one range requantized to int8 codes of another: within
    # one step of eq. 4 applied to the real value (float64)
    rng = np.random.default_rng(104)
    xf = rng.standard_normal(20000).astype(np.float32) * 3
    import paper_2408_13933_gb300.synth as sy
    q16, s16, z16 = sy.quantize_per_tensor(xf, bits=16)
    s8, z8 = sy.quantize_params_from_range(float(xf.min()), float(xf.max()))
    m0, sh = orc.requant_params(s16, np.ones(1, np.float32), s8)
    y = orc.requantize(q16, z16, int(m0[0]), int(sh[0]), z8, 8).astype(np.int64)
    real = (q16.astype(np.float64) - z16) * s16
    ref = np.clip(np.floor(real / s8 + 0.5) + z8, -128, 127)
    diff = np.abs(y - ref)
    assert diff.max() <= 1 and (diff != 0).mean() < 1e-3


# ---- offline fold of eq. 1 and weight quantization ------------------------------

def _fold_ref(w, s_in, s_out):
    n_, k_ = w.shape
    out = np.zeros((n_, k_), np.float64)
    for n in range(n_):
        for k in range(k_):
            v = float(w[n, k])
            if s_in is not None:
                v = _f32_nearest(Fraction(v) * Fraction(float(s_in[k])))
            if s_out is not None:
                v = _f32_nearest(Fraction(v) / Fraction(float(s_out[n])))
            out[n, k] = v
    return out


def _quantize_weights_ref(w, bits, scheme):
    """Every f32 operation of the definition rounded by hand from exact rationals."""
    qmin, qmax = (-128, 127) if bits == 8 else (-8, 7)
    n_, k_ = w.shape
    codes = np.zeros((n_, k_), np.int64)
    sw = np.zeros(n_)
    zw = np.zeros(n_, np.int64)
    tlo, thi = min(float(w.min()), 0.0), max(float(w.max()), 0.0)
    for n in range(n_):
        lo, hi = (tlo, thi) if scheme == 2 else (min(float(w[n].min()), 0.0),
                                                  max(float(w[n].max()), 0.0))
        if scheme == 0:
            amax = max(-lo, hi) or float(np.float32(1e-8))
            scale = _f32_nearest(Fraction(amax) / qmax)
            zero, cmin = 0, (-qmax if bits == 8 else qmin)
        else:
            span = _f32_nearest(Fraction(hi) - Fraction(lo))
            if not span > 0:
                span = float(np.float32(1e-8))
            scale = _f32_nearest(Fraction(span) / (qmax - qmin))
            zf = round(_f32_nearest(Fraction(qmin) - Fraction(_f32_nearest(Fraction(lo) /
                                                                             Fraction(scale)))))
            zero, cmin = max(qmin, min(qmax, zf)), qmin
        for k in range(k_):
            t = round(_f32_nearest(Fraction(float(w[n, k])) / Fraction(scale)))
            codes[n, k] = max(cmin, min(qmax, t + zero))
        sw[n], zw[n] = scale, zero
    return codes, sw, zw


def pin_fold_exact(orc: Oracle):
    rng = np.random.default_rng(201)
    w = (rng.standard_normal((5, 24)) * 0.02).astype(np.float32)
    s_in = rng.uniform(0.3, 3.0, 24).astype(np.float32)
    s_out = rng.uniform(0.3, 3.0, 5).astype(np.float32)
    for si, so in ((s_in, None), (None, s_out), (s_in, s_out)):
        got = orc.fold_weights(w, si, so).astype(np.float64)
        assert np.array_equal(got, _fold_ref(w, si, so))


def pin_quantize_weights_exact(orc: Oracle):
    rng = np.random.default_rng(202)
    w = (rng.standard_normal((6, 40)) * 0.02).astype(np.float32)
    w[2] += 0.01           # a channel biased positive
    w[3] = 0.0             # an all-zero channel
    w[4, :5] = [0.0625, -0.03125, 0.015625, 0.0, -0.0625]   # exact power-of-two values
    for bits in (8, 4):
        for scheme in (0, 1, 2):
            c, sw, zw = orc.quantize_weights(w, bits, scheme)
            rc, rsw, rzw = _quantize_weights_ref(w, bits, scheme)
            assert np.array_equal(c.astype(np.int64), rc), (bits, scheme)
            assert np.array_equal(sw.astype(np.float64), rsw), (bits, scheme)
            assert np.array_equal(zw.astype(np.int64), rzw), (bits, scheme)


def pin_fold_equivalence(orc: Oracle):
    """Eq. 1: X W = (X S^-1)(S W), before quantization, through one layer and
    through the norm + two linears of Figure 3 (S0 on the norm and W1's
    inputs, S1 between W1 and W2)."""
    rng = np.random.default_rng(203)
    x = rng.standard_normal((16, 64))
    w1 = (rng.standard_normal((48, 64)) * 0.05).astype(np.float32)
    w2 = (rng.standard_normal((32, 48)) * 0.05).astype(np.float32)
    s0 = rng.uniform(0.2, 5.0, 64).astype(np.float32)
    s1 = rng.uniform(0.2, 5.0, 48).astype(np.float32)
    gamma = rng.uniform(0.5, 1.5, 64).astype(np.float32)
    beta = rng.uniform(-0.2, 0.2, 64).astype(np.float32)
    ref1 = x @ w1.astype(np.float64).T
    f1 = orc.fold_weights(w1, s0, None).astype(np.float64)
    got1 = (x / s0.astype(np.float64)) @ f1.T
    assert np.allclose(got1, ref1, rtol=0, atol=1e-6 * np.abs(ref1).max())
    g1, b1 = orc.fold_norm(gamma, beta, s0)
    f1 = orc.fold_weights(w1, s0, s1).astype(np.float64)
    f2 = orc.fold_weights(w2, s1, None).astype(np.float64)
    h = x * gamma.astype(np.float64) + beta.astype(np.float64)
    ref2 = (h @ w1.astype(np.float64).T) @ w2.astype(np.float64).T
    hf = x * g1.astype(np.float64) + b1.astype(np.float64)
    got2 = (hf @ f1.T) @ f2.T
    assert np.allclose(got2, ref2, rtol=0, atol=2e-6 * np.abs(ref2).max())
    # with a wrong direction of either factor the equivalence breaks
    bad = orc.fold_weights(w1, 1 / s0, None).astype(np.float64)
    assert not np.allclose((x / s0) @ bad.T, ref1, atol=1e-3 * np.abs(ref1).max())


def pin_quantize_weights_properties(orc: Oracle):
    rng = np.random.default_rng(204)
    w = (rng.standard_normal((20, 300)) * 0.02).astype(np.float32)
    w[::3] -= 0.015
    for bits in (8, 4):
        qmin, qmax = (-128, 127) if bits == 8 else (-8, 7)
        c, sw, _ = orc.quantize_weights(w, bits, 0)
        c = c.astype(np.int64)
        # the largest magnitude of each row lands on +-qmax; half-step error
        assert np.all(np.abs(c).max(axis=1) == qmax)
        err = np.abs(c * sw[:, None].astype(np.float64) - w.astype(np.float64))
        assert np.all(err[np.abs(c) < qmax] <= 0.5 * sw[:, None].repeat(300, 1)[np.abs(c) < qmax]
                      * (1 + 1e-6))
        for scheme in (1, 2):
            c, sw, zw = orc.quantize_weights(w, bits, scheme)
            c = c.astype(np.int64)
            assert c.min() >= qmin and c.max() <= qmax
            # the real zero maps to the zero point exactly
            cz, _, zz = orc.quantize_weights(np.concatenate([w, np.zeros((20, 1), np.float32)], 1),
                                             bits, scheme)
            assert np.array_equal(cz[:, -1].astype(np.int64), zz.astype(np.int64))
            deq = (c - zw[:, None]) * sw[:, None].astype(np.float64)
            inside = (c > qmin) & (c < qmax)
            assert np.all(np.abs(deq - w)[inside] <= 0.5 * np.repeat(sw[:, None], 300, 1)[inside]
                          * (1 + 1e-5))
            if scheme == 2:
                assert len(set(sw.tolist())) == 1 and len(set(zw.tolist())) == 1
                assert c.min() == qmin or c.max() == qmax
            else:
                assert np.all((c.min(axis=1) == qmin) | (c.max(axis=1) == qmax))


# ---- 8-bit inputs, 16-bit outputs (scores ahead of a 16-bit non-linearity) ----

def pin_o16_k1_exhaustive(orc: Oracle):
    # every int8 x against every int8 w (K = 1), several zero points, outputs
    # against round half up of exact rationals saturated to int16
    xs = np.arange(-128, 128, dtype=np.int16).astype(np.int8).reshape(-1, 1)
    ws = np.arange(-128, 128, dtype=np.int16).astype(np.int8).reshape(-1, 1)
    packed, _ = orc.pack(ws, 8)
    n = ws.shape[0]
    for zx, zwv, m0, s in ((-128, 127, 1 << 30, 31), (5, -3, (1 << 31) - 1, 24), (0, 0, 1 << 30, 30)):
        y = orc.linear_o16(xs, zx, packed, 8, n, np.full(n, m0, np.int32),
                           np.full(n, s, np.int32), 7, zw=np.full(n, zwv, np.int32))
        for i in range(0, 256, 5):
            for j in range(0, 256, 3):
                acc = (int(xs[i, 0]) - zx) * (int(ws[j, 0]) - zwv)
                assert int(y[i, j]) == _py_requant16(acc, m0, s, 7), (zx, zwv, i, j)


def pin_o16_matches_asym_and_requant16(orc: Oracle):
    # the accumulator is oracle_linear_asym's and each output is
    # oracle_requant_one_a16 of it (both separately pinned)
    rng = np.random.default_rng(301)
    for bits in (8, 4):
        lo, hi = (-128, 127) if bits == 8 else (-8, 7)
        c = synth.random_case(71 + bits, 7, 96, 13, bits)
        zw = rng.integers(lo, hi + 1, size=c.N).astype(np.int32)
        packed, _ = orc.pack(c.w, bits)
        m0 = rng.integers(1 << 30, 1 << 31, size=c.N).astype(np.int32)
        sh = rng.integers(14, 40, size=c.N).astype(np.int32)
        _, acc = orc.linear(c.x, c.zx, packed, bits, c.N, m0, sh, 0, want_acc=True, zw=zw)
        zy = -1234
        y = orc.linear_o16(c.x, c.zx, packed, bits, c.N, m0, sh, zy, zw=zw)
        for m in range(c.M):
            for n in range(c.N):
                assert int(y[m, n]) == orc.requant_one_a16(int(acc[m, n]), int(m0[n]), int(sh[n]),
                                                           zy)
        assert (np.abs(y.astype(np.int64)) > 127).any()   # the 16-bit range is used


def pin_a16_asym_k1_exhaustive(orc: Oracle):
    # every int16 code x against int8 weight codes at the ends of the range and
    # spread over it (K = 1), weight zero points at the ends and middle of the
    # range: acc = (x - zx)(w - zw) exactly, and sampled outputs against round
    # half up of exact rationals
    xs = np.arange(-32768, 32768, dtype=np.int64).astype(np.int16).reshape(-1, 1)
    ws = np.array([-128, -127, -100, -64, -17, -2, -1, 0, 1, 2, 19, 63, 64, 101, 126, 127],
                  np.int8).reshape(-1, 1)
    packed, _ = orc.pack(ws, 8)
    n = ws.shape[0]
    for zx, zwv in ((-32768, 127), (0, -128), (12345, -3)):
        zw = np.full(n, zwv, np.int32)
        m0, s, zy = (1 << 30) + 12345, 44, -77
        y, acc = orc.linear_a16(xs, zx, packed, 8, n, np.full(n, m0, np.int32),
                                np.full(n, s, np.int32), zy, want_acc=True, zw=zw)
        ref = (xs.astype(np.int64) - zx) * (ws[:, 0].astype(np.int64) - zwv)[None, :]
        assert np.array_equal(acc, ref), (zx, zwv)
        for i in range(0, xs.shape[0], 3001):
            for j in range(n):
                assert int(y[i, j]) == _py_requant16(int(ref[i, j]), m0, s, zy), (zx, zwv, i, j)


def pin_a16_asym_identity_and_reduction(orc: Oracle):
    # numpy's int64 matmul of the shifted operands (int8 and int4 weights,
    # per-channel zero points), and oracle_linear_a16 when every zw is 0
    rng = np.random.default_rng(403)
    for seed, bits in ((11, 8), (12, 4)):
        c = synth.random_case_a16(seed, 6, 128, 17, bits, "mixed" if bits == 4 else None)
        lo, hi = (-128, 127) if bits == 8 else (-8, 7)
        zw = rng.integers(lo, hi + 1, size=c.N).astype(np.int32)
        packed, _ = orc.pack(c.w, bits)
        m0, sh = orc.requant_params(c.sx, c.sw, c.sy)
        _, acc = orc.linear_a16(c.x, c.zx, packed, bits, c.N, m0, sh, c.zy, want_acc=True, zw=zw)
        ref = (c.x.astype(np.int64) - c.zx) @ (c.w.astype(np.int64) - zw[:, None]).T
        assert np.array_equal(acc, ref), seed
        y0 = orc.linear_a16(c.x, c.zx, packed, bits, c.N, m0, sh, c.zy,
                            zw=np.zeros(c.N, np.int32))
        assert np.array_equal(y0, orc.linear_a16(c.x, c.zx, packed, bits, c.N, m0, sh, c.zy))


PIN_BATTERY = [pin_golden, pin_k1_exhaustive, pin_int4_exhaustive_pairs, pin_zero_point_identity,
               pin_exact_dequant, pin_requant_closed_form, pin_requant_ties, pin_requant_vs_eq4,
               pin_requant_params_bound, pin_asym_k1_exhaustive, pin_asym_int4_pairs,
               pin_asym_identity, pin_asym_reduces_to_symmetric, pin_asym_exact_dequant,
               pin_a16_k1_exhaustive, pin_a16_int4_pairs, pin_a16_matmul_and_brute_force,
               pin_a16_large_accumulators, pin_a16_reduces_to_int8, pin_a16_byte_planes, pin_a16_exact_dequant,
               pin_a16_requant_closed_form_and_saturation, pin_a16_requant_vs_eq4,
               pin_quantize_exact, pin_quantize_ties_and_invariants, pin_dequantize_exact,
               pin_requantize_exhaustive, pin_requantize_vs_eq4, pin_fold_exact,
               pin_quantize_weights_exact, pin_fold_equivalence, pin_quantize_weights_properties,
               pin_o16_k1_exhaustive, pin_o16_matches_asym_and_requant16,
               pin_a16_asym_k1_exhaustive, pin_a16_asym_identity_and_reduction]


# ----------------------------------------------------------------------------
# Tests
# ----------------------------------------------------------------------------

@pytest.fixture(scope="module")
def O():
    oracle.build()
    return oracle._default()


def test_golden_worked_examples(O):
    pin_golden(O)


def test_k1_exhaustive_all_zero_points(O):
    pin_k1_exhaustive(O)


def test_int4_pairs_exhaustive(O):
    pin_int4_exhaustive_pairs(O)


def test_zero_point_identity(O):
    pin_zero_point_identity(O)


def test_exact_dequantization_invariant(O):
    pin_exact_dequant(O)


def test_requant_closed_form_shift(O):
    pin_requant_closed_form(O)


def test_requant_exact_ties(O):
    pin_requant_ties(O)


def test_requant_matches_eq4_quantizer(O):
    pin_requant_vs_eq4(O)


def test_requant_params_error_bound(O):
    pin_requant_params_bound(O)


def test_bruteforce_small_k(O):
    rng = np.random.default_rng(1)
    for k in (1, 2, 3):
        for bits in (8, 4):
            lo, hi = (-128, 127) if bits == 8 else (-8, 7)
            if bits == 4 and k % 2:
                continue
            x = rng.integers(-128, 128, size=(5, k)).astype(np.int8)
            w = rng.integers(lo, hi + 1, size=(6, k)).astype(np.int8)
            zx = int(rng.integers(-128, 128))
            packed, _ = O.pack(w, bits)
            m0, sh = O.requant_params(0.02, np.full(6, 0.01, np.float32), 0.05)
            y, acc = O.linear(x, zx, packed, bits, 6, m0, sh, 3, want_acc=True)
            for m in range(5):
                for n in range(6):
                    a = sum((int(x[m, kk]) - zx) * int(w[n, kk]) for kk in range(k))
                    assert acc[m, n] == a
                    q = _round_half_up_frac(Fraction(a * int(m0[n]), 1 << int(sh[n])))
                    assert y[m, n] == max(-128, min(127, 3 + q))


def test_requant_params_special_cases(O):
    m0, sh = O.requant_params(2.0 ** -20, np.array([2.0 ** -20], np.float32), 1.0)
    assert (int(m0[0]), int(sh[0])) == (0, 1)          # below 2^-32: output is zy
    m0, sh = O.requant_params(2.0 ** 15, np.array([2.0 ** 14], np.float32), 1.0)
    assert (int(m0[0]), int(sh[0])) == (1 << 30, 1)    # 2^29: smallest legal shift
    with pytest.raises(oracle.OracleError):
        O.requant_params(2.0 ** 15, np.array([2.0 ** 15], np.float32), 1.0)  # 2^30
    for bad in (0.0, -1.0, float("nan"), float("inf")):
        with pytest.raises(oracle.OracleError):
            O.requant_params(bad, np.array([0.1], np.float32), 1.0)
        with pytest.raises(oracle.OracleError):
            O.requant_params(0.1, np.array([bad], np.float32), 1.0)


def test_pack_roundtrip_and_range(O):
    rng = np.random.default_rng(2)
    for bits, lo, hi in ((8, -128, 127), (4, -8, 7)):
        w = rng.integers(lo, hi + 1, size=(33, 64)).astype(np.int8)
        packed, colsum = O.pack(w, bits)
        assert np.array_equal(O.unpack(packed, 33, 64, bits), w)
        assert np.array_equal(colsum, w.astype(np.int64).sum(1))
    with pytest.raises(oracle.OracleError):
        O.pack(np.array([[8, 0]], np.int8), 4)
    with pytest.raises(oracle.OracleError):
        O.pack(np.array([[-9, 0]], np.int8), 4)


def test_accumulator_overflow_detected(O):
    k_ok, k_bad = 65536, 65794
    for k, ok in ((k_ok, True), (k_bad, False)):
        x = np.full((1, k), -128, np.int8)
        w = np.full((1, k), -128, np.int8)
        packed, _ = O.pack(w, 8)
        m0 = np.array([1 << 30], np.int32)
        sh = np.array([62], np.int32)
        if ok:
            _, acc = O.linear(x, 127, packed, 8, 1, m0, sh, 0, want_acc=True)
            assert int(acc[0, 0]) == 255 * 128 * k
        else:
            with pytest.raises(oracle.OracleError):
                O.linear(x, 127, packed, 8, 1, m0, sh, 0)


def test_asym_k1_exhaustive(O):
    pin_asym_k1_exhaustive(O)


def test_asym_int4_pairs(O):
    pin_asym_int4_pairs(O)


def test_asym_identity(O):
    pin_asym_identity(O)


def test_asym_reduces_to_symmetric(O):
    pin_asym_reduces_to_symmetric(O)


def test_asym_exact_dequant(O):
    pin_asym_exact_dequant(O)


def test_asym_rejects_zero_point_out_of_range(O):
    c = synth.random_case(3, 2, 32, 4, 4)
    packed, _ = O.pack(c.w, 4)
    m0, sh = O.requant_params(c.sx, c.sw, c.sy)
    with pytest.raises(oracle.OracleError):
        O.linear(c.x, c.zx, packed, 4, c.N, m0, sh, c.zy, zw=np.array([0, 8, 0, 0], np.int32))


def test_linear_points_agree_with_full(O):
    c = synth.random_case(21, 11, 64, 19, 4)
    packed, _ = O.pack(c.w, 4)
    m0, sh = O.requant_params(c.sx, c.sw, c.sy)
    y, acc = O.linear(c.x, c.zx, packed, 4, c.N, m0, sh, c.zy, want_acc=True)
    pts = np.array([(m, n) for m in range(11) for n in range(19)], np.int64)
    yp, ap = O.linear_points(c.x, c.zx, packed, 4, c.N, m0, sh, c.zy, pts)
    assert np.array_equal(yp, y.reshape(-1)) and np.array_equal(ap, acc.reshape(-1))


def test_residual_add_saturates(O):
    a = np.array([-128, -100, 0, 100, 127, 127, -1], np.int8)
    b = np.array([-1, -100, 5, 100, 1, -128, 1], np.int8)
    assert O.residual_add(a, b).tolist() == [-128, -128, 5, 127, 127, -1, 0]


def test_a16_k1_exhaustive(O):
    pin_a16_k1_exhaustive(O)


def test_a16_int4_pairs(O):
    pin_a16_int4_pairs(O)


def test_a16_matmul_and_brute_force(O):
    pin_a16_matmul_and_brute_force(O)


def test_a16_large_accumulators(O):
    pin_a16_large_accumulators(O)


def test_a16_reduces_to_int8(O):
    pin_a16_reduces_to_int8(O)


def test_a16_byte_planes(O):
    pin_a16_byte_planes(O)


def test_a16_exact_dequant(O):
    pin_a16_exact_dequant(O)


def test_a16_requant_closed_form_and_saturation(O):
    pin_a16_requant_closed_form_and_saturation(O)


def test_a16_requant_vs_eq4(O):
    pin_a16_requant_vs_eq4(O)


def test_a16_rejects_bad_arguments(O):
    w = np.zeros((2, 32), np.int8)
    packed, _ = O.pack(w, 8)
    m0 = np.full(2, 1 << 30, np.int32)
    sh = np.full(2, 31, np.int32)
    x = np.zeros((1, 32), np.int16)
    for zx, zy in ((32768, 0), (-32769, 0), (0, 32768), (0, -32769)):
        with pytest.raises(oracle.OracleError):
            O.linear_a16(x, zx, packed, 8, 2, m0, sh, zy)


def test_a16_points_agree_with_full(O):
    c = synth.random_case_a16(51, 11, 64, 23, 4)
    packed, _ = O.pack(c.w, 4)
    m0, sh = O.requant_params(c.sx, c.sw, c.sy)
    y, acc = O.linear_a16(c.x, c.zx, packed, 4, c.N, m0, sh, c.zy, want_acc=True)
    pts = np.array([[m, n] for m in range(0, 11, 3) for n in range(0, 23, 5)], np.int64)
    yp, ap = O.linear_points_a16(c.x, c.zx, packed, 4, c.N, m0, sh, c.zy, pts)
    assert np.array_equal(yp, y[pts[:, 0], pts[:, 1]])
    assert np.array_equal(ap, acc[pts[:, 0], pts[:, 1]])


def test_quantize_exact(O):
    pin_quantize_exact(O)


def test_quantize_ties_and_invariants(O):
    pin_quantize_ties_and_invariants(O)


def test_dequantize_exact(O):
    pin_dequantize_exact(O)


def test_requantize_exhaustive(O):
    pin_requantize_exhaustive(O)


def test_requantize_vs_eq4(O):
    pin_requantize_vs_eq4(O)


def test_boundary_quantizers_reject_bad_arguments(O):
    x = np.zeros(4, np.float32)
    for alpha, z, bits in ((0.0, 0, 8), (float("nan"), 0, 8), (1.0, 128, 8), (1.0, 0, 12),
                           (1.0, 40000, 16)):
        with pytest.raises(oracle.OracleError):
            O.quantize(x, alpha, z, bits)
    q = np.zeros(4, np.int8)
    with pytest.raises(oracle.OracleError):
        O.requantize(q, 0, 1 << 30, 0, 0, 8)      # shift 0
    with pytest.raises(oracle.OracleError):
        O.requantize(q, 200, 1 << 30, 31, 0, 8)   # zx outside int8


def test_fold_exact(O):
    pin_fold_exact(O)


def test_quantize_weights_exact(O):
    pin_quantize_weights_exact(O)


def test_fold_equivalence(O):
    pin_fold_equivalence(O)


def test_quantize_weights_properties(O):
    pin_quantize_weights_properties(O)


def test_o16_k1_exhaustive(O):
    pin_o16_k1_exhaustive(O)


def test_o16_matches_asym_and_requant16(O):
    pin_o16_matches_asym_and_requant16(O)


def test_a16_asym_k1_exhaustive(O):
    pin_a16_asym_k1_exhaustive(O)


def test_a16_asym_identity_and_reduction(O):
    pin_a16_asym_identity_and_reduction(O)


MUTATIONS = [
    ("zero point sign", "int64_t xv = (int64_t)x[(size_t)m * (size_t)ldx + (size_t)k] - zx;",
     "int64_t xv = (int64_t)x[(size_t)m * (size_t)ldx + (size_t)k] + zx;"),
    ("nibble order", "int nibble = (k % 2 == 0) ? (byte & 0x0F) : (byte >> 4);",
     "int nibble = (k % 2 == 0) ? (byte >> 4) : (byte & 0x0F);"),
    ("int4 sign extension", "return nibble >= 8 ? nibble - 16 : nibble;", "return nibble;"),
    ("round half down", "__int128 q = oracle_floor_div(2 * v + two_s, 2 * two_s);",
     "__int128 q = oracle_floor_div(2 * v + two_s - 1, 2 * two_s);"),
    ("truncating division", "if (r != 0 && a < 0) q -= 1;", "(void)r;"),
    ("dropped rounding term", "__int128 q = oracle_floor_div(2 * v + two_s, 2 * two_s);",
     "__int128 q = oracle_floor_div(2 * v, 2 * two_s);"),
    ("multiplier exponent off by one", "int s = 31 - e;", "int s = 30 - e;"),
    ("mantissa rounding", "long long m0 = llround(ldexp(f, 31));",
     "long long m0 = (long long)(ldexp(f, 31));"),
    ("missing zero point", "y[(size_t)m * (size_t)ldy + (size_t)n] =\n                    (int8_t)oracle_requant_one(acc, M0[n], shift[n], zy);",
     "y[(size_t)m * (size_t)ldy + (size_t)n] =\n                    (int8_t)oracle_requant_one(acc, M0[n], shift[n], 0);"),
    ("dropped last k", "for (int k = 0; k < K; ++k) {\n        int64_t xv",
     "for (int k = 0; k < K - 1; ++k) {\n        int64_t xv"),
    ("colsum of first row only", "if (colsum) colsum[n] = (int32_t)sum;",
     "if (colsum) colsum[n] = (int32_t)(n == 0 ? sum : 0);"),
    ("saturation bound", "if (out > 127) out = 127;", "if (out > 126) out = 126;"),
    ("weight zero point sign", "int64_t wv = oracle_weight_at(packed, bits, K, n, k) - zw;",
     "int64_t wv = oracle_weight_at(packed, bits, K, n, k) + zw;"),
    ("weight zero point ignored", "int64_t acc = oracle_dot_asym(x, K, ldx, zx, packed, bits, m, n, zw ? zw[n] : 0);",
     "int64_t acc = oracle_dot_asym(x, K, ldx, zx, packed, bits, m, n, 0);"),
    ("a16 zero point sign", "- (int64_t)zx;", "+ (int64_t)zx;"),
    ("a16 activation narrowed to int8",
     "int64_t x16 = (int64_t)x[(size_t)m * (size_t)ldx + (size_t)k]",
     "int64_t x16 = (int64_t)(int8_t)x[(size_t)m * (size_t)ldx + (size_t)k]"),
    ("a16 accumulator narrowed to int32", "acc16 += x16 * w16;",
     "acc16 = (int32_t)(acc16 + x16 * w16);"),
    ("a16 saturation at int8", "if (out > 32767) out = 32767;", "if (out > 127) out = 127;"),
    ("a16 round half down", "return oracle_floor_div(2 * v + two_s, 2 * two_s);",
     "return oracle_floor_div(2 * v + two_s - 1, 2 * two_s);"),
    ("quantize rounds half away from zero", "double t = (double)rintf(quotient) + (double)z;",
     "double t = (double)roundf(quotient) + (double)z;"),
    ("quantize by reciprocal multiply", "float quotient = x[i] / alpha;",
     "float quotient = x[i] * (1.0f / alpha);"),
    ("quantize zero point dropped", "double t = (double)rintf(quotient) + (double)z;",
     "double t = (double)rintf(quotient);"),
    ("dequantize zero point sign", "(double)(oracle_code_at(q, bits, i) - z)",
     "(double)(oracle_code_at(q, bits, i) + z)"),
    ("requantize input zero point dropped",
     "int64_t centered = (int64_t)oracle_code_at(q, in_bits, i) - zx;",
     "int64_t centered = (int64_t)oracle_code_at(q, in_bits, i);"),
    ("requantize wrong output range", "if (out > ohi) out = ohi;", "if (out > ihi) out = ihi;"),
    ("fold by reciprocal multiply", "if (s_out) v = v / s_out[n];",
     "if (s_out) v = v * (1.0f / s_out[n]);"),
    ("fold divides the input channel", "if (s_in) v = v * s_in[k];", "if (s_in) v = v / s_in[k];"),
    ("norm fold multiplies", "gamma_out[k] = gamma[k] / s[k];", "gamma_out[k] = gamma[k] * s[k];"),
    ("symmetric amax ignores negatives", "float amax = -lo > hi ? -lo : hi;", "float amax = hi;"),
    ("quantizer weight zero point sign", "float zf = rintf((float)qmin - lo / scale);",
     "float zf = rintf((float)qmin + lo / scale);"),
    ("per-tensor statistics per row", "        if (scheme == 2) {\n            lo = tlo;",
     "        if (scheme == 3) {\n            lo = tlo;"),
    ("asymmetric span from the row maximum only", "float span = hi - lo;", "float span = hi;"),
    ("o16 output narrowed to int8",
     "(int16_t)oracle_requant_one_a16(wide, M0[n], shift[n], zy);",
     "(int16_t)oracle_requant_one(wide, M0[n], shift[n], zy);"),
    ("a16 weight zero point ignored",
     "int64_t wv = oracle_weight_at(packed, bits, K, n, k) - zwn;",
     "int64_t wv = oracle_weight_at(packed, bits, K, n, k);"),
    ("a16 weight zero point sign",
     "int64_t wv = oracle_weight_at(packed, bits, K, n, k) - zwn;",
     "int64_t wv = oracle_weight_at(packed, bits, K, n, k) + zwn;"),
    ("o16 weight zero point ignored",
     "int64_t wide = oracle_dot_asym(x, K, ldx, zx, packed, bits, m, n, zw ? zw[n] : 0);",
     "int64_t wide = oracle_dot_asym(x, K, ldx, zx, packed, bits, m, n, 0);"),
    ("a16 output zero point dropped",
     "__int128 out = (__int128)zy + oracle_round_shift(acc, M0, shift);",
     "__int128 out = oracle_round_shift(acc, M0, shift);"),
]


@pytest.mark.parametrize("name,old,new", MUTATIONS, ids=[m[0] for m in MUTATIONS])
def test_pins_reject_planted_mistake(tmp_path, name, old, new):
    src = oracle.source()
    assert old in src, f"mutation anchor for '{name}' not found"
    lib = oracle.compile_variant(src.replace(old, new, 1), str(tmp_path / "libmut.so"))
    mutant = Oracle(lib)
    failures = 0
    for pin in PIN_BATTERY:
        try:
            if pin is pin_k1_exhaustive:
                pin(mutant, zxs=(-128, -1, 0, 1, 127))
            else:
                pin(mutant)
        except (AssertionError, oracle.OracleError):
            failures += 1
    assert failures > 0, f"no pin caught the planted mistake '{name}'"


def test_row_parallel_front_end_equals_the_single_threaded_oracle(orc):
    # linear_mt only cuts the token rows into blocks for a thread pool; rows
    # are independent, so every output equals the single-threaded call's,
    # including row counts that do not divide by the thread count
    from paper_2408_13933_gb300 import synth
    for m, k, n, bits, t in ((37, 256, 96, 8, 5), (3, 512, 64, 4, 8), (16, 64, 33, 8, 16)):
        c = synth.random_case(4000 + m, m, k, n, bits)
        packed, _ = orc.pack(c.w, bits)
        m0, sh = orc.requant_params(c.sx, c.sw, c.sy)
        want = orc.linear(c.x, c.zx, packed, bits, n, m0, sh, c.zy)
        got = orc.linear_mt(c.x, c.zx, packed, bits, n, m0, sh, c.zy, nthreads=t)
        assert got.shape == want.shape and np.array_equal(got, want)
