"""The offline weight pipeline on the GPU (fold of eq. 1, weight quantization,
packing, colsum) against the oracle's fold_weights -> quantize_weights ->
pack, bit for bit, for every scheme and weight width; and the folded,
quantized weights driving the integer layer end to end."""
import numpy as np
import pytest

import oracle
from gpu_helpers import assert_equal_int8, torch_cuda, upload
from paper_2408_13933_gb300 import synth

pytestmark = pytest.mark.gpu


def mq():
    from paper_2408_13933_gb300 import mq as m
    return m


def _weights(seed, n, k):
    rng = np.random.default_rng(seed)
    w = (rng.standard_normal((n, k)) * 0.02).astype(np.float32)
    if n > 3:
        w[1] += 0.012          # biased channel
        w[2] = 0.0             # all-zero channel
        w[3, ::7] *= 15.0      # outliers
    s_in = rng.uniform(0.25, 4.0, k).astype(np.float32)
    s_out = rng.uniform(0.25, 4.0, n).astype(np.float32)
    return w, s_in, s_out


def _run(w, s_in, s_out, bits, scheme):
    lib = mq()
    wd = upload(w)
    si = upload(s_in) if s_in is not None else None
    so = upload(s_out) if s_out is not None else None
    packed, colsum, sw, zw = lib.fold_quantize_pack(wd, bits, scheme, si, so)
    torch_cuda().cuda.synchronize()
    return (packed.cpu().numpy(), colsum.cpu().numpy(), sw.cpu().numpy(),
            zw.cpu().numpy() if zw is not None else None)


def _want(w, s_in, s_out, bits, scheme):
    f = oracle.fold_weights(w, s_in, s_out)
    codes, sw, zw = oracle.quantize_weights(f, bits, scheme)
    packed, colsum = oracle.pack(codes, bits)
    return packed, colsum, sw, zw, codes


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("scheme", [0, 1, 2])
@pytest.mark.parametrize("factors", ["none", "in", "out", "both"])
@pytest.mark.parametrize("shape", [(37, 200), (256, 2048), (5, 5632), (19, 202)],
                         ids=lambda s: "x".join(map(str, s)))
def test_fold_quantize_pack(shape, factors, scheme, bits):
    n, k = shape
    w, s_in, s_out = _weights(n + k + scheme, n, k)
    si = s_in if factors in ("in", "both") else None
    so = s_out if factors in ("out", "both") else None
    got = _run(w, si, so, bits, scheme)
    want = _want(w, si, so, bits, scheme)
    assert np.array_equal(got[2].view(np.uint32), want[2].view(np.uint32)), "scales"
    assert np.array_equal(got[0].reshape(want[0].shape), want[0]), "packed codes"
    assert np.array_equal(got[1], want[1]), "colsum"
    if scheme != 0:
        assert np.array_equal(got[3], want[3]), "zero points"


@pytest.mark.parametrize("bits", [8, 4])
def test_fold_unaligned_rows(bits):
    # weights and input scales one float past a 16-byte boundary: the kernels
    # take their one-weight-per-load path even though K is a multiple of 4
    torch = torch_cuda()
    n, k = 24, 1024
    w, s_in, s_out = _weights(31 + bits, n, k)
    wbuf = torch.zeros(n * k + 1, dtype=torch.float32, device="cuda")
    wbuf[1:] = torch.from_numpy(w.reshape(-1)).cuda()
    sbuf = torch.zeros(k + 1, dtype=torch.float32, device="cuda")
    sbuf[1:] = torch.from_numpy(s_in).cuda()
    wd, sd = wbuf[1:].view(n, k), sbuf[1:]
    assert wd.data_ptr() % 16 == 4 and sd.data_ptr() % 16 == 4
    for scheme in (0, 1, 2):
        packed, colsum, sw, zw = mq().fold_quantize_pack(wd, bits, scheme, sd, upload(s_out))
        torch.cuda.synchronize()
        want = _want(w, s_in, s_out, bits, scheme)
        assert np.array_equal(packed.cpu().numpy().reshape(want[0].shape), want[0])
        assert np.array_equal(colsum.cpu().numpy(), want[1])
        assert np.array_equal(sw.cpu().numpy().view(np.uint32), want[2].view(np.uint32))
        if scheme != 0:
            assert np.array_equal(zw.cpu().numpy(), want[3])


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("scheme", [0, 1, 2])
def test_fold_ties(bits, scheme):
    # every row spans [-qmax, qmax] (symmetric) or [-qmax - 1, qmax] (the
    # asymmetric schemes) times a power of two, so the scale is that power of
    # two and the zero point 0; the other weights put v / scale exactly on a
    # half-integer or one f32 step to either side, where the code turns on
    # the tie rule of rint and on the quotient's last bit
    qmax = 127 if bits == 8 else 7
    step = np.float32(2.0 ** -7 if bits == 8 else 2.0 ** -3)
    lo_k = -qmax if scheme == 0 else -qmax - 1
    ties = (np.arange(lo_k, qmax, dtype=np.float32) + np.float32(0.5)) * step
    vals = np.concatenate([ties, np.nextafter(ties, np.float32(np.inf)),
                           np.nextafter(ties, np.float32(-np.inf))]).astype(np.float32)
    rng = np.random.default_rng(50 + bits + scheme)
    n, k = 16, 1024
    w = rng.choice(vals, (n, k)).astype(np.float32)
    w[:, 0] = np.float32(lo_k) * step
    w[:, 1] = np.float32(qmax) * step
    got = _run(w, None, None, bits, scheme)
    want = _want(w, None, None, bits, scheme)
    assert np.all(want[2] == step)
    assert np.array_equal(got[2].view(np.uint32), want[2].view(np.uint32)), "scales"
    assert np.array_equal(got[0].reshape(want[0].shape), want[0]), "packed codes"
    assert np.array_equal(got[1], want[1]), "colsum"
    if scheme != 0:
        assert np.array_equal(got[3], want[3]) and not np.any(want[3]), "zero points"


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("scheme", [0, 1, 2])
def test_fold_ties_general_scales(bits, scheme):
    # scales that are not powers of two, so 1 / scale is inexact and the
    # kernel's reciprocal product can land on the other side of a tie than the
    # correctly rounded quotient: each row fixes its range with two end
    # weights (scale and zero point follow from them), and every other weight
    # is the f32 nearest to a half-integer multiple of the row's scale (the
    # tensor's, per tensor), or up to three f32 steps to either side
    qmax = 127 if bits == 8 else 7
    qmin = -qmax if scheme == 0 else -qmax - 1
    n, k = 24, 1024
    rng = np.random.default_rng(70 + bits + scheme)
    unit = (0.003 * (1.0 + rng.random(n) * 3.0)).astype(np.float32)   # about the scale
    w = np.zeros((n, k), np.float32)
    w[:, 0] = unit * np.float32(qmin)
    w[:, 1] = unit * np.float32(qmax)
    if scheme == 2:   # one range for the whole tensor
        w[:, 0], w[:, 1] = w[:, 0].min(), w[:, 1].max()
    sw = _want(w, None, None, bits, scheme)[2]   # the scales these ranges give
    j = rng.integers(qmin, qmax, size=(n, k - 2)).astype(np.float64) + 0.5
    mid = (j * sw[:, None].astype(np.float64)).astype(np.float32)     # nearest f32 to the tie
    for _ in range(3):
        step = rng.integers(-1, 2, size=mid.shape)
        mid = np.where(step > 0, np.nextafter(mid, np.float32(np.inf)),
                       np.where(step < 0, np.nextafter(mid, np.float32(-np.inf)), mid))
    w[:, 2:] = np.clip(mid, w[:, :1], w[:, 1:2])
    got = _run(w, None, None, bits, scheme)
    want = _want(w, None, None, bits, scheme)
    assert np.array_equal(want[2], sw), "the end weights fix the scales"
    assert np.array_equal(got[2].view(np.uint32), want[2].view(np.uint32)), "scales"
    assert np.array_equal(got[0].reshape(want[0].shape), want[0]), "packed codes"
    assert np.array_equal(got[1], want[1]), "colsum"
    if scheme != 0:
        assert np.array_equal(got[3], want[3]), "zero points"


def test_fold_edge_shapes():
    for n, k in ((1, 2), (3, 0), (1, 64)):
        w, _, _ = _weights(9, n, k)
        for scheme in (0, 2):
            got = _run(w, None, None, 4 if k % 2 == 0 else 8, scheme)
            want = _want(w, None, None, 4 if k % 2 == 0 else 8, scheme)
            assert np.array_equal(got[1], want[1]) and np.array_equal(got[2], want[2])


@pytest.mark.parametrize("bits,scheme", [(8, 2), (8, 1), (4, 1), (4, 0)])
def test_folded_weights_drive_the_layer(bits, scheme):
    # fold -> quantize -> pack on the device, then the integer layer with the
    # resulting (asymmetric) weights, against the oracle's chain
    torch = torch_cuda()
    lib = mq()
    m, n, k = 40, 96, 512
    w, s_in, _ = _weights(77 + bits + scheme, n, k)
    packed, colsum, sw, zw = lib.fold_quantize_pack(upload(w), bits, scheme, upload(s_in))
    x = synth.random_case(78, m, k, n, bits).x
    zx, sx, sy, zy = 5, 0.02, 0.05, -7
    m0, sh = lib.requant_params(sw.cpu().numpy(), sx, sy)
    y = torch.full((m, n), 99, dtype=torch.int8, device="cuda")
    # the descriptor holds raw addresses: keep every operand alive until the call is done
    keep = [upload(a) for a in (x, m0, sh)]
    d = lib.make_desc(keep[0], zx, packed, colsum, n, keep[1], keep[2], zy, y, bits, zw=zw)
    need = lib.workspace_size_batch([d])
    ws = torch.zeros(max(need, 16), dtype=torch.uint8, device="cuda")
    assert lib.linear_batch([d], workspace=ws, ws_bytes=need) == 0
    torch.cuda.synchronize()
    assert lib.check_device_status() == 0
    _, _, osw, ozw, codes = _want(w, s_in, None, bits, scheme)
    opk, _ = oracle.pack(codes, bits)
    om0, osh = oracle.requant_params(sx, osw, sy)
    want = oracle.linear(x, zx, opk, bits, n, om0, osh, zy,
                         zw=ozw if scheme != 0 else None)
    assert_equal_int8(y.cpu().numpy(), want, f"folded layer bits={bits} scheme={scheme}")


def test_fold_batch_mixed():
    # one batched call over linears of every scheme, width and factor
    # combination, with K not a multiple of 4, rows off the 16-byte boundary,
    # N not a multiple of the eight rows of a CTA, an empty linear and the
    # block's largest shape: every linear's bytes equal the oracle's (and so
    # the per-linear entry point's)
    torch = torch_cuda()
    lib = mq()
    specs = [  # (n, k, bits, scheme, factors)
        (256, 2048, 8, 2, "both"), (37, 200, 4, 1, "in"), (5632, 2048, 8, 1, "out"),
        (19, 202, 8, 0, "none"), (0, 64, 8, 2, "none"), (300, 5632, 4, 2, "both"),
        (64, 1024, 4, 0, "in"), (129, 96, 8, 2, "out")]
    jobs, wants, keep = [], [], []
    for i, (n, k, bits, scheme, factors) in enumerate(specs):
        w, s_in, s_out = _weights(500 + i, n, k)
        si = s_in if factors in ("in", "both") else None
        so = s_out if factors in ("out", "both") else None
        if i == 3:  # off the 16-byte boundary
            wbuf = torch.zeros(n * k + 1, dtype=torch.float32, device="cuda")
            wbuf[1:] = torch.from_numpy(w.reshape(-1)).cuda()
            wd = wbuf[1:].view(n, k)
            keep.append(wbuf)
        else:
            wd = upload(w)
        jobs.append((wd, bits, scheme, upload(si) if si is not None else None,
                     upload(so) if so is not None else None))
        wants.append(_want(w, si, so, bits, scheme) if n else None)
    outs = lib.fold_quantize_pack_batch(jobs)
    torch.cuda.synchronize()
    for (n, k, bits, scheme, _), (packed, colsum, sw, zw), want in zip(specs, outs, wants):
        if n == 0:
            assert colsum.numel() == 0
            continue
        tag = f"batch job {n}x{k} bits={bits} scheme={scheme}"
        assert np.array_equal(sw.cpu().numpy().view(np.uint32), want[2].view(np.uint32)), tag
        assert np.array_equal(packed.cpu().numpy().reshape(want[0].shape), want[0]), tag
        assert np.array_equal(colsum.cpu().numpy(), want[1]), tag
        if scheme != 0:
            assert np.array_equal(zw.cpu().numpy(), want[3]), tag


def test_fold_batch_checks_every_descriptor_first():
    # a bad descriptor anywhere fails the call before anything is launched
    torch = torch_cuda()
    lib = mq()
    w = upload(_weights(7, 16, 64)[0])
    colsum = torch.full((16,), -5, dtype=torch.int32, device="cuda")
    sw = torch.zeros(16, dtype=torch.float32, device="cuda")
    stats = torch.zeros(32, dtype=torch.float32, device="cuda")
    packed = torch.zeros(16 * 64, dtype=torch.uint8, device="cuda")
    ok = lib.FoldDesc(w.data_ptr(), 16, 64, None, None, 8, 0, packed.data_ptr(),
                      colsum.data_ptr(), sw.data_ptr(), None, stats.data_ptr())
    bad = lib.FoldDesc(w.data_ptr(), 16, 63, None, None, 4, 0, packed.data_ptr(),
                       colsum.data_ptr(), sw.data_ptr(), None, stats.data_ptr())  # odd K, int4
    arr = (lib.FoldDesc * 2)(ok, bad)
    assert lib.lib.mq_fold_quantize_pack_batch(arr, 2, None) == lib.MQ_ERR_INVALID_ARG
    torch.cuda.synchronize()
    assert (colsum == -5).all(), "the good descriptor ran"
    too_many = (lib.FoldDesc * (lib.MQ_FOLD_MAX_JOBS + 1))()
    assert lib.lib.mq_fold_quantize_pack_batch(too_many, lib.MQ_FOLD_MAX_JOBS + 1, None) == \
        lib.MQ_ERR_INVALID_ARG
    assert lib.lib.mq_fold_quantize_pack_batch(None, 0, None) == 0
