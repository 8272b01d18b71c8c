"""GPU parity of the 256-token prefill kernel (mq_prefill2.cu) and its token
pre-pass against the oracle, bit for bit, with the cases that decide its
accumulation plan:

* activations drawn like the paper's (per-tensor int8 of N(0, 1) with outlier
  channels): the row sums of squares allow one exact f32 chunk for the whole K;
* uniform codes of moderate size at long K: a data-dependent chunk between
  the fixed one and K, so several chunks whose int32 sums add up;
* codes at the range ends: the fixed 1024-k chunk (int8) of the 128-token kernel;
* weight zero points, int4 weights, a residual, tails in M, N and K.

It also checks that both prefill kernels give the same bytes, that a
workspace without room for the widened inputs falls back to the 128-token
kernel, and that the widened inputs never touch the decode region."""
import numpy as np
import pytest

from gpu_helpers import GpuLinear, assert_equal_int8, oracle_y, torch_cuda, upload
from paper_2408_13933_gb300 import synth

pytestmark = pytest.mark.gpu


def mq():
    from paper_2408_13933_gb300 import mq as m
    return m


@pytest.fixture(autouse=True)
def wide_kernel():
    assert mq().test_prefill_kernel(1) == 0
    yield
    assert mq().test_prefill_kernel(0) == 0


def run_batch(gs, ws_bytes=None, ws=None):
    torch = torch_cuda()
    lib = mq()
    descs = [g.desc() for g in gs]
    need = lib.workspace_size_batch(descs)
    if ws is None:
        ws = torch.zeros(max(need, 16), dtype=torch.uint8, device="cuda")
    assert lib.linear_batch(descs, workspace=ws, ws_bytes=need if ws_bytes is None else ws_bytes) == 0
    torch.cuda.synchronize()
    assert lib.check_device_status() == 0
    return ws


def moderate_case(seed, m, k, n, bits, amp):
    """Uniform codes in [-amp, amp]: row sums of squares ~ k amp^2 / 3."""
    rng = np.random.default_rng(seed)
    wlo, whi = (-128, 127) if bits == 8 else (-8, 7)
    x = rng.integers(-amp, amp + 1, size=(m, k)).astype(np.int8)
    w = rng.integers(wlo, whi + 1, size=(n, k)).astype(np.int8)
    sw = rng.uniform(1e-5, 1e-4, size=n).astype(np.float32)
    return synth.LinearCase(f"moderate{seed}", x, int(rng.integers(-128, 128)), 0.01, w, sw,
                            bits, 0.05, int(rng.integers(-128, 128)))


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("shape", [(512, 2048, 512), (300, 5632, 264), (257, 1056, 300)],
                         ids=lambda s: "x".join(map(str, s)))
def test_model_like_activations_one_chunk(shape, bits):
    m, k, n = shape
    case = synth.make_linear(0, 1, bits, "wide", m, k, n, bits)
    g = GpuLinear(case)
    run_batch([g])
    assert_equal_int8(g.result(), oracle_y(case), f"model-like {shape} bits={bits}")


@pytest.mark.parametrize("bits,amp,k", [(8, 30, 8192), (8, 60, 4096), (4, 60, 65536),
                                         (4, 127, 65536)])
def test_data_dependent_chunks(bits, amp, k):
    # row sums of squares ~ k amp^2 / 3 make the exact run (X2 wmax^2 L <=
    # 2^48) shorter than K but longer than the fixed chunk: int8 |x| <= 30 at
    # K = 8192 gives two chunks (51 stages of 128 k and the rest), |x| <= 60 at
    # K = 4096 two (25 stages and the rest), int4 |x| <= 60 at K = 65536 two
    # (425 stages and the rest); at |x| <= 127 the bound falls below the fixed
    # 16384 k, which the tile takes instead (four chunks)
    case = moderate_case(11 + amp, 260, k, 300, bits, amp)
    g = GpuLinear(case)
    run_batch([g])
    assert_equal_int8(g.result(), oracle_y(case), f"chunks bits={bits} amp={amp} k={k}")


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("extreme", ["min", "max", "mixed"])
def test_extreme_codes_fixed_chunks(extreme, bits):
    case = synth.random_case(800 + len(extreme), 300, 4096, 264, bits, extreme)
    case.sw = np.full(case.N, 1e-8, np.float32)
    g = GpuLinear(case)
    run_batch([g])
    assert_equal_int8(g.result(), oracle_y(case), f"extreme {extreme} bits={bits}")


def test_residual_zero_points_and_tails():
    import oracle
    cases = [synth.random_case(820, 333, 1040, 300, 8), synth.random_case(821, 290, 2080, 72, 4)]
    rng = np.random.default_rng(3)
    cases[0].residual = rng.integers(-128, 128, size=(333, 300)).astype(np.int8)
    cases[1].zw = rng.integers(-8, 8, size=72).astype(np.int32)
    gs = [GpuLinear(c) for c in cases]
    zw = upload(cases[1].zw)
    descs = [gs[0].desc()]
    g = gs[1]
    c = cases[1]
    descs.append(mq().make_desc(g.x, c.zx, g.packed, g.colsum, c.N, g.m0, g.shift, c.zy, g.y,
                                c.bits, zw=zw))
    torch = torch_cuda()
    lib = mq()
    need = lib.workspace_size_batch(descs)
    ws = torch.zeros(need, dtype=torch.uint8, device="cuda")
    assert lib.linear_batch(descs, workspace=ws, ws_bytes=need) == 0
    assert_equal_int8(gs[0].result(), oracle_y(cases[0]), "residual")
    packed, _ = oracle.pack(c.w, c.bits)
    m0, sh = oracle.requant_params(c.sx, c.sw, c.sy)
    want = oracle.linear(c.x, c.zx, packed, c.bits, c.N, m0, sh, c.zy, zw=c.zw)
    assert_equal_int8(gs[1].result(), want, "weight zero points")


def test_both_kernels_same_bytes():
    lib = mq()
    cases = [synth.make_linear(0, 2, j, "both", m, k, n, b)
             for j, (m, k, n, b) in enumerate([(1024, 2048, 2048, 8), (700, 5632, 520, 8),
                                               (512, 2048, 264, 4)])]
    outs = []
    for which in (1, 2):
        assert lib.test_prefill_kernel(which) == 0
        gs = [GpuLinear(c) for c in cases]
        run_batch(gs)
        outs.append([g.result() for g in gs])
    for a, b, c in zip(outs[0], outs[1], cases):
        assert np.array_equal(a, b), f"kernels differ on {c.M}x{c.K}x{c.N}"


def test_small_workspace_falls_back_and_decode_region_stays_zero():
    torch = torch_cuda()
    lib = mq()
    pre = synth.make_linear(0, 3, 0, "fallback", 512, 2048, 512, 8)
    dec = synth.random_case(830, 4, 2048, 300, 4)
    gp, gd = GpuLinear(pre), GpuLinear(dec)
    descs = [gp.desc(), gd.desc()]
    need = lib.workspace_size_batch(descs)
    region = lib.workspace_size(1, 1, 0, 4)
    assert need > region + 2 * 512 * 2048
    ws = torch.zeros(need + 4096, dtype=torch.uint8, device="cuda")
    # only the required part (the decode region): the 128-token kernel, nothing
    # written past it
    assert lib.linear_batch(descs, workspace=ws, ws_bytes=region) == 0
    torch.cuda.synchronize()
    assert lib.check_device_status() == 0
    assert_equal_int8(gp.result(), oracle_y(pre), "fallback prefill")
    assert_equal_int8(gd.result(), oracle_y(dec), "fallback decode")
    assert int(torch.count_nonzero(ws)) == 0
    # the full size: the widened inputs go after the decode region, which the
    # call leaves zero-filled
    gp.y.fill_(77)
    assert lib.linear_batch(descs, workspace=ws, ws_bytes=need) == 0
    torch.cuda.synchronize()
    assert lib.check_device_status() == 0
    assert_equal_int8(gp.result(), oracle_y(pre), "wide prefill")
    assert int(torch.count_nonzero(ws[:region])) == 0
    assert int(torch.count_nonzero(ws[region:need])) > 0
    assert int(torch.count_nonzero(ws[need:])) == 0


def test_widened_copy_and_row_sums():
    # the pre-pass's output in the workspace: the f16 copy of x and the row
    # sums of squares, at the documented place
    torch = torch_cuda()
    lib = mq()
    case = synth.random_case(840, 300, 1040, 40, 8)
    g = GpuLinear(case)
    ws = run_batch([g])
    region = lib.workspace_size(1, 1, 0, 4)
    base = ws.data_ptr() + region
    off = ((base + 1023) & ~1023) - ws.data_ptr()
    n16 = 300 * 1040
    x16 = ws[off:off + 2 * n16].view(torch.float16).cpu().numpy().reshape(300, 1040)
    assert np.array_equal(x16, case.x.astype(np.float16))
    roff = off + ((2 * n16 + 1023) & ~1023)
    rowsq = ws[roff:roff + 4 * 300].view(torch.int32).cpu().numpy()
    assert np.array_equal(rowsq, (case.x.astype(np.int64) ** 2).sum(axis=1))


@pytest.mark.parametrize("bits", [8, 4])
def test_weight_sq_sums(bits):
    case = synth.random_case(850 + bits, 1, 2080 if bits == 8 else 2112, 301, bits, "mixed")
    packed, _ = mq().pack_weights(case.w, bits)
    got = mq().weight_sq_sums(upload(packed), case.N, case.K, bits).cpu().numpy()
    assert np.array_equal(got, (case.w.astype(np.int64) ** 2).sum(axis=1))


def test_weight_norms_allow_one_chunk():
    # full-range activations at K = 5632 (the down projection's input): the
    # |w| <= 128 bound splits K into runs of ~12 stages; with the weights'
    # sums of squares the whole K is one run.  Both plans are exact.
    lib = mq()
    case = synth.make_linear(0, 4, 0, "wsq", 512, 5632, 512, 8)
    rng = np.random.default_rng(9)
    case.x = rng.integers(-100, 101, size=(512, 5632)).astype(np.int8)
    want = oracle_y(case)
    for with_wsq in (False, True):
        g = GpuLinear(case)
        wsq = lib.weight_sq_sums(g.packed, case.N, case.K, 8) if with_wsq else None
        d = lib.make_desc(g.x, case.zx, g.packed, g.colsum, case.N, g.m0, g.shift, case.zy, g.y,
                          8, wsq=wsq)
        torch = torch_cuda()
        need = lib.workspace_size_batch([d])
        ws = torch.zeros(need, dtype=torch.uint8, device="cuda")
        assert lib.linear_batch([d], workspace=ws, ws_bytes=need) == 0
        assert_equal_int8(g.result(), want, f"wsq={with_wsq}")


def _chain_pair(seed, m, k, n1, n2, residual):
    """Two linears chained as layers are: A reads x, B reads A's output."""
    a = synth.make_linear(0, 5, seed, "chainA", m, k, n1, 8)
    if residual:
        a.residual = np.random.default_rng(seed).integers(-128, 128, size=(m, n1)).astype(np.int8)
    b = synth.make_linear(0, 6, seed, "chainB", m, n1, n2, 8)
    return a, b


@pytest.mark.parametrize("which", [0, 1, 2])   # default choice, 256-token forced, 128-token forced
@pytest.mark.parametrize("residual", [False, True])
def test_chained_f16_copies(which, residual):
    # A writes y16 / ysq (fused in the 256-token epilogue, or by the pre-pass
    # on y after the 128-token kernel); B reads them as x16 / xsq.  y16 is f16(y)
    # and ysq the row sums of squares of y exactly, and B equals the oracle on y.
    torch = torch_cuda()
    lib = mq()
    assert lib.test_prefill_kernel(which) == 0
    a, b = _chain_pair(30 + which, 512, 2048, 1024, 768, residual)
    ga = GpuLinear(a)
    y16 = torch.full((a.M, a.N), 7.0, dtype=torch.float16, device="cuda")
    ysq = torch.zeros(a.M, dtype=torch.int32, device="cuda")
    da = lib.make_desc(ga.x, a.zx, ga.packed, ga.colsum, a.N, ga.m0, ga.shift, a.zy, ga.y, 8,
                       residual=ga.residual, y16=y16, ysq=ysq)
    need = lib.workspace_size_batch([da])
    ws = torch.zeros(max(need, 16), dtype=torch.uint8, device="cuda")
    assert lib.linear_batch([da], workspace=ws, ws_bytes=need) == 0
    ya = ga.result()
    assert_equal_int8(ya, oracle_y(a), "A")
    assert np.array_equal(y16.cpu().numpy(), ya.astype(np.float16))
    assert np.array_equal(ysq.cpu().numpy(), (ya.astype(np.int64) ** 2).sum(axis=1))
    b.x = ya
    gb = GpuLinear(b)
    db = lib.make_desc(ga.y, b.zx, gb.packed, gb.colsum, b.N, gb.m0, gb.shift, b.zy, gb.y, 8,
                       x16=y16, xsq=ysq)
    need = lib.workspace_size_batch([db])
    assert need == 0   # its only input comes widened: no pre-pass, no workspace
    assert lib.linear_batch([db], workspace=None, ws_bytes=0) == 0
    assert_equal_int8(gb.result(), oracle_y(b), "B")


def test_chained_copy_of_a_small_output():
    # an output below the 256-token kernel's limits (N = 128): its f16 copy comes
    # from the pre-pass on y after the 128-token kernel
    torch = torch_cuda()
    lib = mq()
    assert lib.test_prefill_kernel(0) == 0
    a = synth.make_linear(0, 7, 0, "small", 300, 1024, 128, 8)
    ga = GpuLinear(a)
    y16 = torch.zeros((a.M, a.N), dtype=torch.float16, device="cuda")
    ysq = torch.zeros(a.M, dtype=torch.int32, device="cuda")
    da = lib.make_desc(ga.x, a.zx, ga.packed, ga.colsum, a.N, ga.m0, ga.shift, a.zy, ga.y, 8,
                       y16=y16, ysq=ysq)
    assert lib.linear_batch([da], workspace=None, ws_bytes=0) == 0
    ya = ga.result()
    assert np.array_equal(y16.cpu().numpy(), ya.astype(np.float16))
    assert np.array_equal(ysq.cpu().numpy(), (ya.astype(np.int64) ** 2).sum(axis=1))


def test_chained_fields_validated():
    lib = mq()
    torch = torch_cuda()
    a = synth.make_linear(0, 8, 0, "val", 300, 1024, 264, 8)
    ga = GpuLinear(a)
    y16 = torch.zeros((a.M, a.N), dtype=torch.float16, device="cuda")
    d = lib.make_desc(ga.x, a.zx, ga.packed, ga.colsum, a.N, ga.m0, ga.shift, a.zy, ga.y, 8,
                      y16=y16)   # no ysq
    assert lib.linear_batch([d]) == lib.MQ_ERR_INVALID_ARG
    ysq = torch.zeros(a.M, dtype=torch.int32, device="cuda")
    d = lib.make_desc(ga.x, a.zx, ga.packed, ga.colsum, a.N, ga.m0, ga.shift, a.zy, ga.y, 8,
                      y16=y16, ysq=ysq)   # N = 264: not a multiple of 16
    assert lib.linear_batch([d]) == lib.MQ_ERR_ALIGNMENT
