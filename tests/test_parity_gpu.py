"""GPU parity: libmq's kernels against the CPU oracle, bit for bit.

Every test runs on both prefill kernels (128- and 256-token tiles).
Shapes span several 128 x 256 tensor-core tiles with ragged M, N and K tails,
the 1024-deep f32 accumulation chunks of the int8 path, every decode width
M in [1, 16], both weight widths, and the degenerate cases (K = 0, one row,
one column, extreme codes).  The whole path is integer, so the bar is
equality of every int8 output.
"""
import numpy as np
import pytest

from gpu_helpers import (GpuLinear, assert_equal_int8, decode_region, oracle_y, torch_cuda, upload,
                         workspace)
from paper_2408_13933_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True, params=[1, 2], ids=["tile256", "tile128"])
def prefill_kernel(request):
    """Every test runs on both prefill kernels: the 256-token one wherever the
    workspace allows (1), and the 128-token one (2)."""
    from paper_2408_13933_gb300 import mq
    assert mq.test_prefill_kernel(request.param) == 0
    yield request.param
    assert mq.test_prefill_kernel(0) == 0


PREFILL_SHAPES = [
    # (M, K, N): tiles of 128 x 256, K blocks of 64, int8 chunks of 1024
    (300, 1040, 520),    # 3 x 3 tiles, ragged M/N, two chunks with a 16-deep tail
    (128, 2048, 256),    # exact tiles, two full chunks
    (17, 64, 1),         # smallest prefill M, single output column
    (129, 16, 257),      # one-element tails in M and N, K = one 16-chunk
    (256, 3072, 512),    # three chunks
    (200, 4160, 300),    # five chunks, last one 64 deep
]

DECODE_SHAPES = [(m, k, n) for m in (1, 2, 3, 4, 7, 8, 9, 15, 16)
                 for (k, n) in ((2080, 300), (64, 33))]


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("shape", PREFILL_SHAPES, ids=lambda s: "x".join(map(str, s)))
def test_prefill_random(shape, bits):
    m, k, n = shape
    if bits == 4 and k % 32:
        k += 16
    case = synth.random_case(100 + m + k + n, m, k, n, bits)
    got = GpuLinear(case).run()
    assert_equal_int8(got, oracle_y(case), f"prefill {shape} bits={bits}")


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("shape", DECODE_SHAPES, ids=lambda s: "x".join(map(str, s)))
def test_decode_random(shape, bits):
    m, k, n = shape
    case = synth.random_case(200 + m + k + n, m, k, n, bits)
    got = GpuLinear(case).run()
    assert_equal_int8(got, oracle_y(case), f"decode {shape} bits={bits}")


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("extreme", ["min", "max", "mixed"])
@pytest.mark.parametrize("m", [1, 16, 200])
def test_extreme_codes(m, extreme, bits):
    # all codes at -128 / 127 (int4: -8 / 7) with zx at the opposite end: the
    # largest accumulators the validation admits (|acc| = 255*128*K)
    case = synth.random_case(300 + m, m, 2048, 272, bits, extreme)
    # a multiplier that keeps the huge accumulators inside the output range
    case.sw = np.full(case.N, 1e-7, np.float32)
    got = GpuLinear(case).run()
    assert_equal_int8(got, oracle_y(case), f"extreme {extreme} m={m} bits={bits}")


def cancellation_case(m: int, k: int, n: int, bits: int, seed: int):
    """Accumulators whose partial sums climb to ~2^23 (constant-sign weights
    against x = 127) and then cancel (the second half repeats the weights
    against x = -127), leaving a small exact result that the unit multiplier
    (M0 = 2^30, shift 30) shows in y."""
    rng = np.random.default_rng(seed)
    lo, hi = (-128, 127) if bits == 8 else (-8, 7)
    half = k // 2
    w = np.where((np.arange(n) % 2 == 0)[:, None], hi, lo).repeat(k, axis=1).astype(np.int8)
    x = np.empty((m, k), np.int8)
    x[:, :half] = 127
    x[:, half:] = -127
    for j in range(4):      # perturbations in the middle, where partials peak
        kk = half - 1 - 7 * j
        w[:, kk] = rng.integers(-3, 4, size=n)
        w[:, kk + half] = w[:, kk]
        x[:, kk] = 127 - rng.integers(0, 3, size=m)
    return synth.LinearCase("cancel", x, 0, 1.0, w, np.ones(n, np.float32), bits, 1.0, 0)


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("m", [1, 9, 16, 160])
def test_large_partial_sums_stay_exact(m, bits):
    k = 1024 if bits == 8 else 16384
    case = cancellation_case(m, k, 264, bits, seed=m + bits)
    want = oracle_y(case)
    assert np.all(np.abs(want.astype(int)) <= 24)   # exact small results, never clamped
    got = GpuLinear(case).run()
    assert_equal_int8(got, want, f"cancellation m={m} bits={bits}")


@pytest.mark.parametrize("m", [1, 5, 130])
def test_k_zero_gives_zero_point(m):
    case = synth.random_case(7, m, 0, 40, 8)
    got = GpuLinear(case).run()
    assert_equal_int8(got, oracle_y(case), "K = 0")
    assert np.all(got == case.zy)


@pytest.mark.parametrize("m", [3, 140])
def test_row_stride_and_padding_untouched(m):
    case = synth.random_case(8, m, 256, 50, 8)
    g = GpuLinear(case, ldy=80)
    got = g.run()
    assert_equal_int8(got[:, :50], oracle_y(case), "strided y")
    assert np.all(got[:, 50:] == 77)          # columns past N are not written


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("m", [4, 300])
def test_residual_epilogue(m, bits):
    case = synth.random_case(9 + m, m, 512, 264, bits)
    case.residual = synth.rint_clip(np.random.default_rng(m).normal(0, 60, (m, 264)), -128,
                                    127).astype(np.int8)
    g = GpuLinear(case)
    from paper_2408_13933_gb300 import mq
    assert mq.linear_batch([g.desc()], workspace=workspace()) == 0
    assert_equal_int8(g.result(), oracle_y(case), f"residual m={m} bits={bits}")


def test_batch_mixes_kernels_and_widths():
    cases = [synth.random_case(40 + i, m, k, n, b) for i, (m, k, n, b) in enumerate(
        [(1, 256, 100, 4), (16, 512, 300, 8), (200, 1024, 260, 8), (130, 512, 64, 4),
         (8, 2048, 256, 4), (333, 64, 17, 8)])]
    gs = [GpuLinear(c) for c in cases]
    from paper_2408_13933_gb300 import mq
    assert mq.linear_batch([g.desc() for g in gs], workspace=workspace()) == 0
    for g, c in zip(gs, cases):
        assert_equal_int8(g.result(), oracle_y(c), f"batch {c.M}x{c.K}x{c.N} bits={c.bits}")


@pytest.mark.parametrize("bits", [8, 4])
def test_device_pack_matches_host_pack(bits):
    import oracle
    case = synth.random_case(12, 1, 2080, 301, bits)
    from paper_2408_13933_gb300 import mq
    packed, colsum = mq.pack_weights(upload(case.w), bits)
    rp, rc = oracle.pack(case.w, bits)
    assert np.array_equal(packed.cpu().numpy().reshape(-1), rp.reshape(-1))
    assert np.array_equal(colsum.cpu().numpy(), rc)


def test_device_pack_rejects_int4_range():
    from paper_2408_13933_gb300 import mq
    w = np.zeros((4, 64), np.int8)
    w[2, 5] = 9
    with pytest.raises(mq.MQError):
        mq.pack_weights(upload(w), 4)


def test_repeated_calls_are_deterministic():
    case = synth.random_case(13, 256, 2048, 512, 8)
    g = GpuLinear(case)
    a = g.run().copy()
    for _ in range(3):
        assert np.array_equal(g.run(), a)


@pytest.mark.parametrize("bits,extreme", [(4, None), (4, "mixed"), (8, "mixed"), (8, "min")])
def test_decode_unit_split_across_many_ctas(bits, extreme):
    # one 64-row unit of K = 65536: its 256 (int4) or 512 (int8) stages are
    # spread over up to 320 CTAs, which combine their partial sums in the
    # workspace; "min" drives the int32 accumulator to its largest magnitude
    case = synth.random_case(500 + bits, 5, 65536, 64, bits, extreme)
    case.sw = np.full(case.N, 2e-9, np.float32)
    assert_equal_int8(GpuLinear(case).run(), oracle_y(case), f"split K=65536 bits={bits}")


def test_decode_workspace_left_zero():
    torch = torch_cuda()
    for seed, (m, k, n, bits) in enumerate([(1, 5632, 2048, 4), (16, 16384, 300, 8),
                                            (7, 2080, 70, 4)]):
        c = synth.random_case(600 + seed, m, k, n, bits)
        assert_equal_int8(GpuLinear(c).run(), oracle_y(c), f"ws m={m} k={k}")
    torch.cuda.synchronize()
    assert int(torch.count_nonzero(decode_region())) == 0
