"""Host-side checks of libmq that need no GPU.

* the shared library loads and exports every function declared in include/mq.h;
* mq_requant_params agrees with the oracle's independent implementation;
* host-side mq_pack_weights agrees with the oracle's packing and colsum;
* argument validation rejects bad calls before anything is launched.
Every call made here either is host-only or fails validation, so nothing
touches a GPU.
"""
import ctypes
import os
import re

import numpy as np
import pytest

import oracle
from paper_2408_13933_gb300 import build, synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def mq():
    build.build()
    from paper_2408_13933_gb300 import mq as _mq
    return _mq


def declared_functions():
    text = open(os.path.join(ROOT, "include", "mq.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(mq_[a-z0-9_]+)\s*\(", text)))


def test_library_exports_every_declared_symbol(mq):
    names = declared_functions()
    assert len(names) >= 9
    for name in names:
        assert hasattr(mq.lib, name), name
    assert set(names) == set(mq.EXPORTED)


def test_status_strings(mq):
    for code in range(8):
        assert mq.status_string(code).startswith("MQ_")
    assert mq.status_string(99) == "MQ_ERR_UNKNOWN"


def test_requant_params_match_oracle(mq):
    rng = np.random.default_rng(1)
    for _ in range(50):
        sx = float(np.float32(rng.uniform(1e-4, 2.0)))
        sy = float(np.float32(rng.uniform(1e-4, 2.0)))
        sw = np.exp(rng.uniform(-14, 2, size=257)).astype(np.float32)
        try:
            ref = oracle.requant_params(sx, sw, sy)
        except oracle.OracleError:
            with pytest.raises(mq.MQError):
                mq.requant_params(sw, sx, sy)
            continue
        got = mq.requant_params(sw, sx, sy)
        assert np.array_equal(got[0], ref[0]) and np.array_equal(got[1], ref[1])


def test_requant_params_edge_cases(mq):
    cases = [(0.5, [0.25, 0.75, 1.0], 2.0), (2.0 ** -20, [2.0 ** -20], 1.0),
             (2.0 ** 15, [2.0 ** 14], 1.0), (1.0, [1.0 - 2.0 ** -24], 1.0),
             (3.0, [1.0 / 3.0], 1.0), (1e-30, [1e-30], 1.0)]
    for sx, sw, sy in cases:
        sw = np.array(sw, np.float32)
        ref = oracle.requant_params(sx, sw, sy)
        got = mq.requant_params(sw, sx, sy)
        assert got[0].tolist() == ref[0].tolist() and got[1].tolist() == ref[1].tolist()
    for sx, sw, sy in [(2.0 ** 15, [2.0 ** 15], 1.0), (0.0, [1.0], 1.0), (1.0, [-1.0], 1.0),
                       (1.0, [float("nan")], 1.0), (1.0, [1.0], float("inf"))]:
        with pytest.raises(mq.MQError) as e:
            mq.requant_params(np.array(sw, np.float32), sx, sy)
        assert e.value.code == mq.MQ_ERR_INVALID_ARG


def test_host_pack_matches_oracle(mq):
    for bits in (8, 4):
        for (n, k) in ((1, 2), (7, 64), (33, 130), (0, 16)):
            c = synth.random_case(3, 1, k, max(n, 1), bits)
            w = c.w[:n]
            packed, colsum = mq.pack_weights(w, bits)
            rp, rc = oracle.pack(w, bits)
            assert np.array_equal(packed.reshape(-1), rp.reshape(-1))
            assert np.array_equal(colsum, rc)


def test_host_pack_rejects_int4_out_of_range(mq):
    with pytest.raises(mq.MQError):
        mq.pack_weights(np.array([[0, 8]], np.int8), 4)
    with pytest.raises(mq.MQError):
        mq.pack_weights(np.array([[0, 1, 2]], np.int8), 4)  # odd K


def test_packed_and_workspace_sizes(mq):
    assert mq.packed_size(3, 64, 8) == 192
    assert mq.packed_size(3, 64, 4) == 96
    dec = mq.workspace_size(16, 2048, 2048, 4)
    assert dec > 0                                          # decode path: fixed size
    assert mq.workspace_size(1, 7, 64, 8) == dec
    assert mq.workspace_size(255, 2048, 2048, 8) == 0       # 128-token tensor-core kernel: none
    # from 256 tokens on: room for the 256-token kernel's widened input after
    # the decode region (f16 copy and row sums, each to 1024 bytes, + 1024)
    assert mq.workspace_size(1024, 2048, 2048, 8) == dec + 2 * 1024 * 2048 + 4096 + 1024
    assert mq.workspace_size(300, 256, 48, 4) == dec + 29696 + 2048 + 1024
    assert mq.workspace_size(300, 255, 48, 4) == 0          # N < 256: the 128-token kernel
    assert mq.workspace_size(300, 256, 0, 4) == 0           # K = 0: nothing to widen
    with pytest.raises(mq.MQError):
        mq.packed_size(3, 63, 4)
    with pytest.raises(mq.MQError):
        mq.packed_size(-1, 64, 8)


FAKE = 1 << 20  # a non-null, 16-byte aligned address; never dereferenced here


def _call(mq, bits=8, x=FAKE, M=32, K=64, ldx=64, zx=0, packed=FAKE, colsum=FAKE, N=32,
          m0=FAKE, shift=FAKE, zy=0, y=FAKE, ldy=32):
    fn = mq.lib.mq_linear_w8a8 if bits == 8 else mq.lib.mq_linear_w4a8
    return fn(x, M, K, ldx, zx, packed, colsum, N, m0, shift, zy, y, ldy, None, 0, None)


@pytest.mark.parametrize("kw,code", [
    (dict(x=None), 1), (dict(packed=None), 1), (dict(colsum=None), 1), (dict(m0=None), 1),
    (dict(shift=None), 1), (dict(y=None), 1), (dict(M=-1), 1), (dict(N=-1), 1),
    (dict(K=-16), 1), (dict(zx=128), 1), (dict(zx=-129), 1), (dict(zy=200), 1),
    (dict(ldx=32), 1), (dict(ldy=16), 1), (dict(K=65552, ldx=65552), 3),
    (dict(K=24, ldx=32), 4), (dict(ldx=72), 4), (dict(x=FAKE + 8), 4),
    (dict(packed=FAKE + 4), 4), (dict(bits=4, K=48, ldx=48), 4),
])
def test_linear_validation_rejects_before_launch(mq, kw, code):
    assert _call(mq, **kw) == code


def test_linear_bad_bits_and_batch_args(mq):
    d = mq.LinearDesc()
    d.bits = 3
    assert mq.lib.mq_linear_batch((mq.LinearDesc * 1)(d), 1, None, 0, None) == 1
    assert mq.lib.mq_linear_batch(None, 1, None, 0, None) == 1
    assert mq.lib.mq_linear_batch((mq.LinearDesc * 1)(), 0, None, 0, None) == 1
    assert mq.lib.mq_linear_batch((mq.LinearDesc * 1)(), mq.MQ_MAX_BATCH + 1, None, 0, None) == 1


def test_decode_requires_workspace(mq):
    # M <= 16 runs the decode kernel, which needs the caller's workspace; the
    # check happens before anything is launched
    fn = mq.lib.mq_linear_w4a8
    assert fn(FAKE, 8, 64, 64, 0, FAKE, FAKE, 32, FAKE, FAKE, 0, FAKE, 32, None, 0, None) == 7
    need = mq.workspace_size(8, 32, 64, 4)
    assert fn(FAKE, 8, 64, 64, 0, FAKE, FAKE, 32, FAKE, FAKE, 0, FAKE, 32, FAKE, need - 1,
              None) == 7
    assert fn(FAKE, 8, 64, 64, 0, FAKE, FAKE, 32, FAKE, FAKE, 0, FAKE, 32, FAKE + 4, need,
              None) == 7   # misaligned


def test_empty_problems_launch_nothing(mq):
    # M == 0 or N == 0 is valid and returns without touching the device
    assert _call(mq, M=0) == 0
    assert _call(mq, N=0) == 0


def _desc(mq, M, K, N, bits, zw):
    d = mq.LinearDesc()
    d.x = d.packed = d.colsum = d.M0 = d.shift = d.y = FAKE
    d.zw = FAKE if zw else None
    d.M, d.K, d.N, d.ldx, d.ldy, d.bits = M, K, N, K, N, bits
    return d


def test_asym_int8_k_limit_and_workspace(mq):
    # int8 weights with a weight zero point: K <= MQ_MAX_K_ASYM8, checked
    # before anything is launched; int4 keeps MQ_MAX_K
    k = mq.MQ_MAX_K_ASYM8 + 16
    bad = (mq.LinearDesc * 1)(_desc(mq, 64, k, 32, 8, True))
    assert mq.lib.mq_linear_batch(bad, 1, None, 0, None) == mq.MQ_ERR_K_OVERFLOW
    ok4 = _desc(mq, 64, k, 32, 4, True)
    # the tensor-core kernel folds the weight zero point into the widened
    # weights: asymmetric prefill needs no workspace; decode shapes need the
    # decode region whatever their weights
    assert mq.workspace_size_batch([ok4]) == 0
    dec = mq.workspace_size(8, 32, 64, 4)
    assert mq.workspace_size_batch([_desc(mq, 100, 64, 32, 8, False)]) == 0
    assert mq.workspace_size_batch([_desc(mq, 100, 64, 32, 8, True)]) == 0
    assert mq.workspace_size_batch([_desc(mq, 101, 64, 32, 8, True),
                                    _desc(mq, 8, 64, 32, 4, True)]) == dec
    assert mq.workspace_size_batch([_desc(mq, 8, 64, 32, 4, False)]) == dec
    # a decode-shaped asymmetric batch without its workspace is rejected up front
    one = (mq.LinearDesc * 1)(_desc(mq, 8, 64, 32, 8, True))
    assert mq.lib.mq_linear_batch(one, 1, None, 0, None) == mq.MQ_ERR_WORKSPACE


def test_synth_asymmetric_weights():
    # the asymmetric weight generator: codes span the range, the zero point
    # maps 0.0 into the code range, and dequantization s (w - z) is within half
    # a step of the float weight wherever the code did not clip
    import numpy as np
    from paper_2408_13933_gb300 import synth
    rng = np.random.default_rng(5)
    wf = (rng.standard_normal((40, 256)) * 0.02).astype(np.float32)
    wf[3] += 0.01  # a channel biased positive
    for bits in (8, 4):
        lo, hi = (-128, 127) if bits == 8 else (-8, 7)
        for per_channel in (False, True):
            q, s, z = synth.quantize_asymmetric(wf, bits, per_channel)
            assert q.dtype == np.int8 and q.min() >= lo and q.max() <= hi
            assert (z >= lo).all() and (z <= hi).all()
            if not per_channel:
                assert len(set(s.tolist())) == 1 and len(set(z.tolist())) == 1
            deq = s[:, None].astype(np.float64) * (q.astype(np.float64) - z[:, None])
            inside = (q > lo) & (q < hi)
            assert np.all(np.abs(deq - wf)[inside] <= 0.5 * s[:, None].repeat(256, 1)[inside] * 1.001)
            # the range ends are reached (per channel: in every channel)
            if per_channel:
                assert ((q == lo) | (q == hi)).any(axis=1).all()
    # the paper's settings: W8A8 per tensor except down per channel; W4A8 per channel
    assert synth.paper_weight_scheme("q", 8) == "asym_tensor"
    assert synth.paper_weight_scheme("down", 8) == "asym_channel"
    assert synth.paper_weight_scheme("q", 4) == "asym_channel"


def _desc16(mq, M, K, N, bits, **kw):
    d = _desc(mq, M, K, N, bits, False)
    d.abits = 16
    for k, v in kw.items():
        setattr(d, k, v)
    return d


def test_a16_validation_and_workspace(mq):
    # 16-bit activations: zero points over the int16 range, no residual,
    # 16-byte rows (ldx % 8), abits 8 or 16 only; every
    # rejection happens before anything is launched
    def rc(d):
        return mq.lib.mq_linear_batch((mq.LinearDesc * 1)(d), 1, FAKE, 1 << 30, None)
    assert rc(_desc16(mq, 4, 64, 32, 8, abits=12)) == mq.MQ_ERR_INVALID_ARG
    assert rc(_desc16(mq, 4, 64, 32, 8, zx=32768)) == mq.MQ_ERR_INVALID_ARG
    assert rc(_desc16(mq, 4, 64, 32, 8, zy=-32769)) == mq.MQ_ERR_INVALID_ARG
    assert rc(_desc16(mq, 4, 64, 32, 8, residual=FAKE)) == mq.MQ_ERR_INVALID_ARG
    # weight zero points are allowed with 16-bit activations (int64 accumulators);
    # with a residual the descriptor is still rejected before any launch
    assert rc(_desc16(mq, 4, 64, 32, 8, zw=FAKE, residual=FAKE)) == mq.MQ_ERR_INVALID_ARG
    assert rc(_desc16(mq, 4, 64, 32, 8, ldx=68)) == mq.MQ_ERR_ALIGNMENT
    assert rc(_desc16(mq, 4, 48, 32, 4, ldx=48)) == mq.MQ_ERR_ALIGNMENT   # int4: K % 32
    assert rc(_desc16(mq, 4, 65552, 32, 8, ldx=65552)) == mq.MQ_ERR_K_OVERFLOW
    # int8 zero points outside [-128, 127] stay invalid for 8-bit activations
    d8 = _desc(mq, 4, 64, 32, 8, False)
    d8.zx = 200
    assert rc(d8) == mq.MQ_ERR_INVALID_ARG
    # an A16 call without its workspace is rejected
    one = (mq.LinearDesc * 1)(_desc16(mq, 100, 64, 32, 8))
    assert mq.lib.mq_linear_batch(one, 1, None, 0, None) == mq.MQ_ERR_WORKSPACE
    # workspace: decode region when 2M <= 16, then the planes (2 M K, to 128)
    dec = mq.workspace_size(1, 1, 0, 4)
    assert mq.workspace_size_a16(100, 32, 64, 8) == 12800
    assert mq.workspace_size_a16(9, 32, 64, 8) == 1152            # 2M = 18: tensor cores
    assert mq.workspace_size_a16(8, 32, 64, 4) == dec             # 2M = 16: decode, no planes
    assert mq.workspace_size_a16(1, 32, 48, 8) == dec
    assert mq.workspace_size_a16(0, 32, 64, 8) == 0
    assert mq.workspace_size_a16(5, 32, 0, 8) == dec              # K = 0: no planes
    # batch: shared int16 input planned once; asymmetric int8 prefill next to
    # it adds nothing; after the decode region the planes start on a
    # 128-byte boundary
    a = _desc16(mq, 100, 64, 32, 8)
    b = _desc16(mq, 100, 64, 48, 4)
    assert mq.workspace_size_batch([a, b]) == 12800
    r = _desc(mq, 20, 64, 32, 8, True)
    r.x = FAKE + 8192
    assert mq.workspace_size_batch([r, a]) == 12800
    assert mq.workspace_size_batch([r]) == 0
    assert mq.workspace_size_batch([_desc(mq, 3, 64, 32, 4, True), a]) == dec + 12800


def test_a16_single_call_symbols(mq):
    for name in ("mq_linear_w8a16", "mq_linear_w4a16", "mq_workspace_size_a16"):
        assert hasattr(mq.lib, name)
    # the single calls validate like the batch (int16 zero point out of range)
    f = mq.lib.mq_linear_w8a16
    assert f(FAKE, 4, 64, 64, 40000, FAKE, FAKE, 32, FAKE, FAKE, 0, FAKE, 32, FAKE, 1 << 30,
             None) == mq.MQ_ERR_INVALID_ARG


def test_boundary_quantizer_validation(mq):
    # every rejection happens on the host, before a launch
    T = mq
    q = mq.lib.mq_quantize
    assert q(FAKE, T.MQ_TYPE_F32, 16, 0.0, 0, FAKE, T.MQ_TYPE_I8, None) == mq.MQ_ERR_INVALID_ARG
    assert q(FAKE, T.MQ_TYPE_F32, 16, float("inf"), 0, FAKE, T.MQ_TYPE_I8, None) == mq.MQ_ERR_INVALID_ARG
    assert q(FAKE, T.MQ_TYPE_F32, 16, 1.0, 128, FAKE, T.MQ_TYPE_I8, None) == mq.MQ_ERR_INVALID_ARG
    assert q(FAKE, T.MQ_TYPE_I8, 16, 1.0, 0, FAKE, T.MQ_TYPE_I8, None) == mq.MQ_ERR_INVALID_ARG
    assert q(FAKE, T.MQ_TYPE_F32, 16, 1.0, 0, FAKE, T.MQ_TYPE_F32, None) == mq.MQ_ERR_INVALID_ARG
    assert q(FAKE, T.MQ_TYPE_F32, -1, 1.0, 0, FAKE, T.MQ_TYPE_I8, None) == mq.MQ_ERR_INVALID_ARG
    assert q(None, T.MQ_TYPE_F32, 0, 1.0, 0, None, T.MQ_TYPE_I8, None) == 0   # nothing to do
    assert q(None, T.MQ_TYPE_F32, 4, 1.0, 0, FAKE, T.MQ_TYPE_I8, None) == mq.MQ_ERR_INVALID_ARG
    assert q(FAKE + 2, T.MQ_TYPE_F32, 4, 1.0, 0, FAKE, T.MQ_TYPE_I8, None) == mq.MQ_ERR_ALIGNMENT
    assert q(FAKE, T.MQ_TYPE_F16, 4, 1.0, 0, FAKE + 1, T.MQ_TYPE_I16, None) == mq.MQ_ERR_ALIGNMENT
    d = mq.lib.mq_dequantize
    assert d(FAKE, T.MQ_TYPE_I16, 4, 1.0, 40000, FAKE, None) == mq.MQ_ERR_INVALID_ARG
    assert d(FAKE, T.MQ_TYPE_F32, 4, 1.0, 0, FAKE, None) == mq.MQ_ERR_INVALID_ARG
    assert d(FAKE, T.MQ_TYPE_I8, 4, 1.0, 0, FAKE + 2, None) == mq.MQ_ERR_ALIGNMENT
    r = mq.lib.mq_requantize
    assert r(FAKE, T.MQ_TYPE_I16, 4, 0, 1 << 30, 0, 0, FAKE, T.MQ_TYPE_I8, None) == mq.MQ_ERR_INVALID_ARG
    assert r(FAKE, T.MQ_TYPE_I16, 4, 0, 1 << 30, 63, 0, FAKE, T.MQ_TYPE_I8, None) == mq.MQ_ERR_INVALID_ARG
    assert r(FAKE, T.MQ_TYPE_I16, 4, 0, -1, 31, 0, FAKE, T.MQ_TYPE_I8, None) == mq.MQ_ERR_INVALID_ARG
    assert r(FAKE, T.MQ_TYPE_I8, 4, 200, 1 << 30, 31, 0, FAKE, T.MQ_TYPE_I8, None) == mq.MQ_ERR_INVALID_ARG
    assert r(FAKE, T.MQ_TYPE_I8, 4, 0, 1 << 30, 31, 200, FAKE, T.MQ_TYPE_I8, None) == mq.MQ_ERR_INVALID_ARG
    assert r(FAKE + 1, T.MQ_TYPE_I16, 4, 0, 1 << 30, 31, 0, FAKE, T.MQ_TYPE_I8, None) == mq.MQ_ERR_ALIGNMENT


def test_fold_validation_and_norm(mq):
    import numpy as np
    f = mq.lib.mq_fold_quantize_pack
    # rejections before any launch
    assert f(FAKE, 4, 64, None, None, 6, 0, FAKE, FAKE, FAKE, None, FAKE, None) == mq.MQ_ERR_INVALID_ARG
    assert f(FAKE, 4, 63, None, None, 4, 0, FAKE, FAKE, FAKE, None, FAKE, None) == mq.MQ_ERR_INVALID_ARG
    assert f(FAKE, 4, 64, None, None, 8, 3, FAKE, FAKE, FAKE, FAKE, FAKE, None) == mq.MQ_ERR_INVALID_ARG
    assert f(FAKE, 4, 64, None, None, 8, 1, FAKE, FAKE, FAKE, None, FAKE, None) == mq.MQ_ERR_INVALID_ARG
    assert f(FAKE, 4, 64, None, None, 8, 0, FAKE, FAKE, FAKE, None, None, None) == mq.MQ_ERR_INVALID_ARG
    assert f(FAKE + 2, 4, 64, None, None, 8, 0, FAKE, FAKE, FAKE, None, FAKE, None) == mq.MQ_ERR_ALIGNMENT
    assert f(None, 0, 64, None, None, 8, 0, None, None, None, None, None, None) == 0
    # the norm fold on the host: gamma / s, beta / s in f32
    g = np.array([1.0, 2.0, -3.0, 0.5], np.float32)
    b = np.array([0.1, -0.2, 0.3, 0.0], np.float32)
    s = np.array([2.0, 0.5, 3.0, 1.0], np.float32)
    g2, b2 = mq.fold_norm(g, b, s)
    assert np.array_equal(g2, g / s) and np.array_equal(b2, b / s)
    g3, b3 = mq.fold_norm(g, None, s)
    assert b3 is None and np.array_equal(g3, g / s)
    with pytest.raises(mq.MQError):
        mq.fold_norm(g, b, np.array([1.0, 0.0, 1.0, 1.0], np.float32))


def test_o16_ldw_rowsums_transpose_validation(mq):
    # every rejection happens before a launch
    def rc(d):
        return mq.lib.mq_linear_batch((mq.LinearDesc * 1)(d), 1, FAKE, 1 << 30, None)
    d = _desc(mq, 40, 64, 32, 8, False)
    d.obits = 16
    d.zy = 40000
    assert rc(d) == mq.MQ_ERR_INVALID_ARG           # zy outside int16
    d.zy = 0
    d.residual = FAKE
    assert rc(d) == mq.MQ_ERR_INVALID_ARG           # no residual with a 16-bit output
    d = _desc(mq, 40, 64, 32, 8, False)
    d.abits, d.obits = 16, 8
    assert rc(d) == mq.MQ_ERR_INVALID_ARG           # 16-bit inputs need 16-bit outputs
    d = _desc(mq, 40, 64, 32, 8, False)
    d.obits = 12
    assert rc(d) == mq.MQ_ERR_INVALID_ARG
    d = _desc(mq, 40, 64, 32, 8, False)
    d.ldw = 48
    assert rc(d) == mq.MQ_ERR_INVALID_ARG           # pitch below the packed row (64 bytes)
    d.ldw = 72
    assert rc(d) == mq.MQ_ERR_ALIGNMENT             # not a multiple of 16
    d4 = _desc(mq, 40, 64, 32, 4, False)
    d4.ldw = 16
    assert rc(d4) == mq.MQ_ERR_INVALID_ARG          # int4 rows of K = 64 take 32 bytes
    r = mq.lib.mq_row_sums
    assert r(FAKE, 4, 40, 48, FAKE, None) == mq.MQ_ERR_ALIGNMENT
    assert r(FAKE, 4, 64, 32, FAKE, None) == mq.MQ_ERR_INVALID_ARG
    assert r(None, 0, 64, 64, None, None) == 0
    hr = mq.lib.mq_head_row_sums
    assert hr(FAKE, 4, 4, 64, 192, FAKE, None) == mq.MQ_ERR_INVALID_ARG   # ldx < heads d
    assert hr(FAKE, 4, 4, 40, 160, FAKE, None) == mq.MQ_ERR_ALIGNMENT     # d % 16
    assert hr(FAKE, 4, 4, 64, 264, FAKE, None) == mq.MQ_ERR_ALIGNMENT     # ldx % 16
    assert hr(FAKE + 8, 4, 4, 64, 256, FAKE, None) == mq.MQ_ERR_ALIGNMENT
    assert hr(FAKE, 4, 4, 64, 256, None, None) == mq.MQ_ERR_INVALID_ARG
    assert hr(None, 0, 4, 64, 256, None, None) == 0
    assert hr(None, 4, 0, 64, 256, None, None) == 0
    t = mq.lib.mq_transpose_i8
    assert t(FAKE, 4, 8, 4, FAKE, 4, None) == mq.MQ_ERR_INVALID_ARG   # lds < cols
    assert t(FAKE, 4, 8, 8, FAKE, 2, None) == mq.MQ_ERR_INVALID_ARG   # ldd < rows
    assert t(None, 0, 8, 8, None, 8, None) == 0


@pytest.mark.parametrize("struct", ["LinearDesc", "FoldDesc"])
def test_descriptor_layout_matches_the_header(mq, tmp_path, struct):
    # the binding's ctypes structs against the C compiler's layouts of
    # mq_linear_desc and mq_fold_desc
    cls = getattr(mq, struct)
    cname = {"LinearDesc": "mq_linear_desc", "FoldDesc": "mq_fold_desc"}[struct]
    fields = [f[0] for f in cls._fields_]
    src = tmp_path / "layout.c"
    body = "".join(f'    printf("{f} %zu\\n", offsetof({cname}, {f}));\n' for f in fields)
    src.write_text('#include <stddef.h>\n#include <stdio.h>\n#include "mq.h"\nint main(void) {\n'
                   + body + f'    printf("sizeof %zu\\n", sizeof({cname}));\n    return 0;\n}}\n')
    exe = tmp_path / "layout"
    import subprocess
    subprocess.run(["gcc", "-std=c11", "-I", os.path.join(ROOT, "include"), str(src), "-o",
                    str(exe)], check=True)
    out = dict(line.split() for line in subprocess.run([str(exe)], check=True, capture_output=True,
                                                       text=True).stdout.splitlines())
    for f in fields:
        assert int(out[f]) == getattr(cls, f).offset, f
    assert int(out["sizeof"]) == ctypes.sizeof(cls)


def test_colsum_optional_with_int8_weights(mq):
    # colsum may be omitted with int8 weights: no workspace where the
    # token-major kernel serves (it folds both zero points), the weights' row
    # sums (4 N bytes, to 128, once per distinct weight matrix) elsewhere;
    # int4 weights and the single-linear calls still require it
    def no_colsum(d):
        d.colsum = None
        return d
    short_k = no_colsum(_desc(mq, 300, 64, 200, 8, True))    # token-major: K <= 128
    long_k = no_colsum(_desc(mq, 300, 512, 200, 8, True))    # 128-token kernel
    assert mq.workspace_size_batch([short_k]) == 0
    assert mq.workspace_size_batch([long_k]) == 4 * 200 + (-4 * 200) % 128
    shared = no_colsum(_desc(mq, 100, 512, 200, 8, False))   # the same weights (FAKE)
    assert mq.workspace_size_batch([long_k, shared]) == 4 * 200 + (-4 * 200) % 128
    dec = mq.workspace_size(1, 1, 0, 4)
    decode = no_colsum(_desc(mq, 4, 512, 200, 8, False))
    assert mq.workspace_size_batch([decode]) == dec + 896
    assert mq.test_tmajor_kernel(2) == 0                     # forbidden: row sums needed
    try:
        assert mq.workspace_size_batch([short_k]) == 896
    finally:
        assert mq.test_tmajor_kernel(0) == 0
    # int4 weights without colsum: rejected before anything is launched
    bad = (mq.LinearDesc * 1)(no_colsum(_desc(mq, 300, 512, 200, 4, False)))
    assert mq.lib.mq_linear_batch(bad, 1, FAKE, 1 << 30, None) == mq.MQ_ERR_INVALID_ARG
    # the single-linear calls: colsum required
    assert mq.lib.mq_linear_w8a8(FAKE, 64, 512, 512, 0, FAKE, None, 32, FAKE, FAKE, 0, FAKE, 32,
                                 FAKE, 1 << 30, None) == mq.MQ_ERR_INVALID_ARG


def test_transposed_weights_checks_on_host(mq):
    # weights stored [K][N] (wt): int8 weights with 8-bit activations, k-rows
    # of at least N bytes (16-byte multiples), prefill shapes the token-major
    # kernel serves; every rejection happens before anything is launched, and
    # such descriptors need neither row sums nor a widened input
    def rc(d):
        return mq.lib.mq_linear_batch((mq.LinearDesc * 1)(d), 1, FAKE, 1 << 30, None)

    def wt(M=300, K=512, N=64, bits=8, **kw):
        d = _desc(mq, M, K, N, bits, True)
        d.colsum = None
        d.wt = 1
        for k, v in kw.items():
            setattr(d, k, v)
        return d
    assert rc(wt(bits=4)) == mq.MQ_ERR_INVALID_ARG
    assert rc(wt(abits=16)) == mq.MQ_ERR_INVALID_ARG
    assert rc(wt(N=64, ldw=48)) == mq.MQ_ERR_INVALID_ARG          # ldw < N
    assert rc(wt(ldw=72)) == mq.MQ_ERR_ALIGNMENT
    assert rc(wt(M=4)) == mq.MQ_ERR_UNSUPPORTED_SHAPE             # decode shape
    assert rc(wt(N=40)) == mq.MQ_ERR_UNSUPPORTED_SHAPE            # k-rows of 40 bytes
    assert rc(wt(packed=FAKE + 8, ldw=64)) == mq.MQ_ERR_ALIGNMENT
    assert mq.test_tmajor_kernel(2) == 0                          # kernel forbidden
    try:
        assert rc(wt()) == mq.MQ_ERR_UNSUPPORTED_SHAPE
    finally:
        assert mq.test_tmajor_kernel(0) == 0
    assert mq.workspace_size_batch([wt(M=2048, K=2048, N=2048)]) == 0
    assert mq.workspace_size_batch([wt(N=40, ldw=48)]) == 0


def test_fold_batch_argument_checks_on_host(mq):
    # count limits and an empty batch, before anything is launched
    many = (mq.FoldDesc * (mq.MQ_FOLD_MAX_JOBS + 1))()
    assert mq.lib.mq_fold_quantize_pack_batch(many, mq.MQ_FOLD_MAX_JOBS + 1, None) == \
        mq.MQ_ERR_INVALID_ARG
    assert mq.lib.mq_fold_quantize_pack_batch(None, 0, None) == 0
    assert mq.lib.mq_fold_quantize_pack_batch(None, 1, None) == mq.MQ_ERR_INVALID_ARG
    bad = mq.FoldDesc(FAKE, 16, 63, None, None, 4, 0, FAKE, FAKE, FAKE, None, FAKE)  # int4, odd K
    assert mq.lib.mq_fold_quantize_pack_batch((mq.FoldDesc * 1)(bad), 1, None) == \
        mq.MQ_ERR_INVALID_ARG
