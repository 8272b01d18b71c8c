"""bench.py's host logic without a GPU: the parity accounting of the legs'
samples (ParityCheck / run_checks) recomputes each kind with the oracle and
counts mismatches; the reference-arm JSON line keeps the contract's keys."""
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
import oracle  # noqa: E402
from paper_2408_13933_gb300 import synth  # noqa: E402


def _requant(acc, m0, sh, zy, lo, hi):
    # round half up of acc * m0 / 2^sh, exact on Python integers
    q = (int(acc) * int(m0) + (1 << (int(sh) - 1))) >> int(sh)
    return max(lo, min(hi, q + zy))


def _direct(x, zx, w, zw, m0, sh, zy, lo, hi):
    acc = (x.astype(np.int64) - zx) @ (w.astype(np.int64) - zw[:, None]).T
    return np.array([[_requant(acc[i, j], m0[j], sh[j], zy, lo, hi) for j in range(acc.shape[1])]
                     for i in range(acc.shape[0])])


def test_run_checks_counts_each_kind():
    oracle.build()
    rng = np.random.default_rng(5)
    checks = []
    # int8 -> int8 with a weight zero point (the "linear" kind)
    c = synth.random_case(31, 3, 64, 12, 8)
    c.zw = rng.integers(-128, 128, size=12).astype(np.int32)
    m0 = np.full(12, 1 << 30, np.int32)
    sh = np.full(12, 38, np.int32)
    got = _direct(c.x, c.zx, c.w, c.zw, m0, sh, c.zy, -128, 127).astype(np.int8)
    checks.append(bench.ParityCheck("leg_a", "linear", c, 3, got, m0, sh))
    # int8 -> int16 (the "o16" kind), one planted wrong output
    c = synth.random_case(32, 2, 32, 8, 4)
    c.zw = rng.integers(-8, 8, size=8).astype(np.int32)
    m0 = np.full(8, (1 << 30) + 7, np.int32)
    sh = np.full(8, 30, np.int32)
    got = _direct(c.x, c.zx, c.w, c.zw, m0, sh, 5, -32768, 32767).astype(np.int16)
    got[1, 3] += 1
    c.zy = 5
    checks.append(bench.ParityCheck("leg_b", "o16", c, 2, got, m0, sh))
    # int16 -> int16 with a weight zero point (the "a16" kind)
    c = synth.random_case_a16(33, 2, 48, 6, 8)
    c.zw = rng.integers(-128, 128, size=6).astype(np.int32)
    m0 = np.full(6, 1 << 30, np.int32)
    sh = np.full(6, 44, np.int32)
    got = _direct(c.x, c.zx, c.w, c.zw, m0, sh, c.zy, -32768, 32767).astype(np.int16)
    checks.append(bench.ParityCheck("leg_c.sub", "a16", c, 2, got, m0, sh))
    res = bench.run_checks(checks)
    assert res["leg_a"] == {"rows": 3, "outputs": 36, "mismatches": 0}
    assert res["leg_b"] == {"rows": 2, "outputs": 16, "mismatches": 1}
    assert res["leg_c.sub"] == {"rows": 2, "outputs": 12, "mismatches": 0}


def test_reference_arm_line():
    # the reference arm (the oracle on this host) prints one JSON line with the
    # contract's keys, its own e2e and a cpu_baseline describing the run
    import io
    import json
    import types
    from contextlib import redirect_stdout
    buf = io.StringIO()
    with redirect_stdout(buf):
        bench.run_reference(types.SimpleNamespace(steps=1, warmup=3), bench.Dist(1, 0, 0))
    line = json.loads(buf.getvalue().strip().splitlines()[-1])
    for key in ("impl", "metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
                "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config",
                "cpu_baseline", "e2e"):
        assert key in line, key
    assert line["impl"] == "reference" and line["value"] > 0 and line["unit"] == "TOPS"
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["e2e"]["value"] == line["value"]
    assert line["cpu_baseline"]["kind"] == "oracle"
    assert line["cpu_baseline"]["cores"] == oracle.threads()
    assert line["config"]["workload"] == bench.WORKLOAD
