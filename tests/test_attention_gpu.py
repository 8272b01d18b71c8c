"""The attention matmul glue on the GPU against the oracle: 8-bit inputs with a
16-bit output (scores ahead of the 16-bit softmax), weights read through a
row pitch (a head's slice of a projection output), row sums of activation
matrices used as colsum, the int8 transpose, and grouped-query attention's
Q K^T (int16 scores) and P V (int8) through the batch call, P V also with V
read in place as transposed weights."""
import numpy as np
import pytest

import oracle
from gpu_helpers import assert_equal_int8, torch_cuda, upload
from paper_2408_13933_gb300 import synth

pytestmark = pytest.mark.gpu


def mq():
    from paper_2408_13933_gb300 import mq as m
    return m


def assert_equal(got, want, what):
    if not np.array_equal(got, want):
        bad = np.argwhere(got != want)
        i = tuple(bad[0])
        raise AssertionError(f"{what}: {len(bad)} of {want.size} differ; first at {i}: "
                             f"got {int(got[i])}, want {int(want[i])}")


def _run(descs, keep):
    torch = torch_cuda()
    lib = mq()
    need = lib.workspace_size_batch(descs)
    ws = torch.zeros(max(need, 16), dtype=torch.uint8, device="cuda")
    keep.append(ws)
    assert lib.linear_batch(descs, workspace=ws, ws_bytes=need) == 0
    torch.cuda.synchronize()
    assert lib.check_device_status() == 0


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("asym", [False, True])
@pytest.mark.parametrize("shape", [(128, 256, 512), (300, 100, 320), (1, 256, 2048), (9, 70, 1024)],
                         ids=lambda s: "x".join(map(str, s)))
def test_o16_parity(shape, asym, bits):
    torch = torch_cuda()
    lib = mq()
    m, n, k = shape
    c = synth.random_case(400 + m + n, m, k, n, bits)
    rng = np.random.default_rng(m * n)
    lo, hi = (-128, 127) if bits == 8 else (-8, 7)
    zw = rng.integers(lo, hi + 1, size=n).astype(np.int32) if asym else None
    m0 = rng.integers(1 << 30, 1 << 31, size=n).astype(np.int32)
    sh = rng.integers(28, 47, size=n).astype(np.int32)
    zy = int(rng.integers(-20000, 20000))
    packed, colsum = lib.pack_weights(c.w, bits)
    keep = [upload(a) for a in (c.x, packed, colsum, m0, sh)]
    zwd = upload(zw) if zw is not None else None
    y = torch.full((m, n), 7, dtype=torch.int16, device="cuda")
    keep += [zwd, y]
    d = lib.make_desc(keep[0], c.zx, keep[1], keep[2], n, keep[3], keep[4], zy, y, bits, zw=zwd)
    assert d.obits == 16 and d.abits == 8
    _run([d], keep)
    opk, _ = oracle.pack(c.w, bits)
    want = oracle.linear_o16(c.x, c.zx, opk, bits, n, m0, sh, zy, zw=zw)
    assert_equal(y.cpu().numpy(), want, f"o16 {shape} asym={asym} bits={bits}")


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("m", [2, 80])
def test_weights_through_a_row_pitch(m, bits):
    # the weights are columns [64, 64 + K) of a wider matrix: ldw = its row bytes
    torch = torch_cuda()
    lib = mq()
    n, k, kfull, off = 96, 128, 320, 64
    big = synth.random_case(500 + m + bits, m, kfull, n, bits)
    w = np.ascontiguousarray(big.w[:, off:off + k])
    x = np.ascontiguousarray(big.x[:, :k])
    packed_full, _ = lib.pack_weights(big.w, bits)
    _, colsum = lib.pack_weights(w, bits)
    m0, sh = lib.requant_params(big.sw, big.sx, big.sy)
    row = kfull if bits == 8 else kfull // 2
    first = off if bits == 8 else off // 2
    pk = upload(packed_full)
    keep = [upload(a) for a in (x, colsum, m0, sh)] + [pk]
    y = torch.full((m, n), 5, dtype=torch.int8, device="cuda")
    keep.append(y)
    d = lib.make_desc(keep[0], big.zx, pk[:, first:], keep[1], n, keep[2], keep[3], big.zy, y, bits,
                      ldw=row)
    _run([d], keep)
    opk, _ = oracle.pack(w, bits)
    om0, osh = oracle.requant_params(big.sx, big.sw, big.sy)
    want = oracle.linear(x, big.zx, opk, bits, n, om0, osh, big.zy)
    assert_equal_int8(y.cpu().numpy(), want, f"ldw m={m} bits={bits}")


def test_row_sums_and_transpose():
    torch = torch_cuda()
    lib = mq()
    rng = np.random.default_rng(3)
    for rows, cols in ((1, 16), (100, 64), (1024, 4096), (33, 2048)):
        a = rng.integers(-128, 128, size=(rows, cols), dtype=np.int16).astype(np.int8)
        ad = upload(a)
        got = lib.row_sums(ad).cpu().numpy()
        assert np.array_equal(got, a.astype(np.int64).sum(1))
    # a strided view: columns 64..127 of a [200, 256] matrix
    a = rng.integers(-128, 128, size=(200, 256), dtype=np.int16).astype(np.int8)
    ad = upload(a)
    assert np.array_equal(lib.row_sums(ad[:, 64:128]).cpu().numpy(),
                          a[:, 64:128].astype(np.int64).sum(1))
    for rows, cols in ((1, 1), (33, 70), (1024, 64), (64, 1000), (257, 129)):
        a = rng.integers(-128, 128, size=(rows, cols), dtype=np.int16).astype(np.int8)
        ad = upload(a)
        t = lib.transpose_i8(ad)
        torch.cuda.synchronize()
        assert np.array_equal(t.cpu().numpy(), a.T)
    a = rng.integers(-128, 128, size=(96, 256), dtype=np.int16).astype(np.int8)
    ad = upload(a)
    t = lib.transpose_i8(ad[:, 128:192])   # a head's slice
    torch.cuda.synchronize()
    assert np.array_equal(t.cpu().numpy(), a[:, 128:192].T)
    # every head slice at once: [M, heads * d] -> [heads, M], incl. more heads than one launch takes
    for m, heads, d, pad in ((1024, 4, 64, 0), (33, 3, 16, 32), (7, 70, 16, 0)):
        a = rng.integers(-128, 128, size=(m, heads * d + pad), dtype=np.int16).astype(np.int8)
        ad = upload(a)
        got = lib.head_row_sums(ad[:, :heads * d], heads).cpu().numpy()
        want = a[:, :heads * d].astype(np.int64).reshape(m, heads, d).sum(2).T
        assert np.array_equal(got, want), (m, heads, d)


@pytest.mark.parametrize("t_q", [96, 1])
def test_grouped_query_attention_matmuls(t_q):
    # 4 query heads over 2 KV heads, head dim 64, T = 96 keys; t_q query tokens
    # (96: prefill kernel, 1: decode kernel).  Three rounds of new K and V
    # rewrite the same V^T and row-sum buffers, all enqueued back to back on
    # one stream (programmatic dependent launches from the producers into the
    # batched calls, weights marked as written on the device), checked after.
    torch = torch_cuda()
    lib = mq()
    rng = np.random.default_rng(11 + t_q)
    T, H, G, D, R = 96, 4, 2, 64, 3
    rep = H // G
    i8 = lambda *s: rng.integers(-128, 128, size=s, dtype=np.int16).astype(np.int8)
    q = i8(t_q, H * D)
    ks, vs, ps = [i8(T, G * D) for _ in range(R)], [i8(T, G * D) for _ in range(R)], \
        [i8(H, t_q, T) for _ in range(R)]
    zq, zk, zv, zp = -5, 12, -20, 7
    qd = upload(q)
    kds, vds, pds = [upload(a) for a in ks], [upload(a) for a in vs], [upload(a) for a in ps]
    keep = [qd] + kds + vds + pds
    m0s, shs, zys = np.full(T, 1 << 30, np.int32), np.full(T, 33, np.int32), 100  # scale 1/8
    m0o, sho, zyo = np.full(D, 1 << 30, np.int32), np.full(D, 40, np.int32), -3   # 2^-10
    dev = [upload(a) for a in (m0s, shs, np.full(T, zk, np.int32), m0o, sho,
                               np.full(D, zv, np.int32))]
    keep += dev
    m0sd, shsd, zwk, m0od, shod, zwv = dev
    colk = torch.empty((G, T), dtype=torch.int32, device="cuda")       # rewritten each round
    vt = torch.empty((G, D, T), dtype=torch.int8, device="cuda")
    colv = torch.empty((G, D), dtype=torch.int32, device="cuda")
    scores = [torch.full((H, t_q, T), 3, dtype=torch.int16, device="cuda") for _ in range(R)]
    outs = [torch.full((t_q, H * D), 9, dtype=torch.int8, device="cuda") for _ in range(R)]
    keep += [colk, vt, colv] + scores + outs
    arr_s, arr_o = [], []
    for r in range(R):
        ds = [lib.make_desc(qd[:, h * D:(h + 1) * D], zq, kds[r][:, (h // rep) * D:],
                            colk[h // rep], T, m0sd, shsd, zys, scores[r][h], 8, zw=zwk, k=D,
                            ldw=G * D, wdynamic=True) for h in range(H)]
        do = [lib.make_desc(pds[r][h], zp, vt[h // rep], colv[h // rep], D, m0od, shod, zyo,
                            outs[r][:, h * D:(h + 1) * D], 8, zw=zwv, wdynamic=True)
              for h in range(H)]
        arr_s.append((lib.LinearDesc * H)(*ds))
        arr_o.append((lib.LinearDesc * H)(*do))
    need = max(lib.workspace_size_batch(list(a)) for a in arr_s + arr_o)
    ws = torch.zeros(max(need, 16), dtype=torch.uint8, device="cuda")
    keep.append(ws)
    torch.cuda.synchronize()
    sp = torch.cuda.current_stream().cuda_stream
    for r in range(R):
        if r == 0:  # per head
            for g in range(G):
                assert lib.lib.mq_row_sums(kds[r][:, g * D:].data_ptr(), T, D, G * D,
                                           colk[g].data_ptr(), sp) == 0
        else:       # all heads in one launch
            assert lib.lib.mq_head_row_sums(kds[r].data_ptr(), T, G, D, G * D,
                                            colk.data_ptr(), sp) == 0
        assert lib.lib.mq_linear_batch(arr_s[r], H, ws.data_ptr(), need, sp) == 0
        if r == 0:  # per head
            for g in range(G):
                assert lib.lib.mq_transpose_i8(vds[r][:, g * D:].data_ptr(), T, D, G * D,
                                               vt[g].data_ptr(), T, sp) == 0
                assert lib.lib.mq_row_sums(vt[g].data_ptr(), D, T, T, colv[g].data_ptr(),
                                           sp) == 0
        else:       # V^T of all heads [G d][T] at once (vt is [G][d][T] contiguous)
            assert lib.lib.mq_transpose_i8(vds[r].data_ptr(), T, G * D, G * D, vt.data_ptr(),
                                           T, sp) == 0
            assert lib.lib.mq_row_sums(vt.data_ptr(), G * D, T, T, colv.data_ptr(), sp) == 0
        assert lib.lib.mq_linear_batch(arr_o[r], H, ws.data_ptr(), need, sp) == 0
    torch.cuda.synchronize()
    assert lib.check_device_status() == 0
    for r in range(R):
        for h in range(H):
            g = h // rep
            kg = np.ascontiguousarray(ks[r][:, g * D:(g + 1) * D])
            opk, _ = oracle.pack(kg, 8)
            want = oracle.linear_o16(np.ascontiguousarray(q[:, h * D:(h + 1) * D]), zq, opk, 8, T,
                                     m0s, shs, zys, zw=np.full(T, zk, np.int32))
            assert_equal(scores[r][h].cpu().numpy(), want, f"round {r} scores head {h}")
            vtg = np.ascontiguousarray(vs[r][:, g * D:(g + 1) * D].T)
            opk, _ = oracle.pack(vtg, 8)
            want = oracle.linear(np.ascontiguousarray(ps[r][h]), zp, opk, 8, D, m0o, sho, zyo,
                                 zw=np.full(D, zv, np.int32))
            assert_equal_int8(outs[r][:, h * D:(h + 1) * D].cpu().numpy(), want,
                              f"round {r} P V head {h}")


@pytest.mark.parametrize("t_q", [200, 1024])
def test_pv_reads_v_in_place(t_q):
    # O_h = P_h V_g with V_g read where it lies ([T][G d], head g at columns
    # g d, transposed weights through V's row pitch): no transpose, no row
    # sums.  Three rounds rewrite the same V buffer on the stream just before
    # each call (weights written on the device), all enqueued back to back.
    torch = torch_cuda()
    lib = mq()
    rng = np.random.default_rng(23 + t_q)
    T, H, G, D, R = 320, 8, 2, 64, 3
    rep = H // G
    i8 = lambda *s: rng.integers(-128, 128, size=s, dtype=np.int16).astype(np.int8)
    vs, ps = [i8(T, G * D) for _ in range(R)], [i8(H, t_q, T) for _ in range(R)]
    zp, zv = 9, -17
    vds, pds = [upload(a) for a in vs], [upload(a) for a in ps]
    m0o, sho, zyo = np.full(D, 1 << 30, np.int32), np.full(D, 40, np.int32), -3
    dev = [upload(a) for a in (m0o, sho, np.full(D, zv, np.int32))]
    m0od, shod, zwv = dev
    vbuf = torch.empty((T, G * D), dtype=torch.int8, device="cuda")
    outs = [torch.full((t_q, H * D), 9, dtype=torch.int8, device="cuda") for _ in range(R)]
    keep = vds + pds + dev + [vbuf] + outs
    arrs = []
    for r in range(R):
        do = [lib.make_desc(pds[r][h], zp, vbuf[:, (h // rep) * D:], None, D, m0od, shod, zyo,
                            outs[r][:, h * D:(h + 1) * D], 8, zw=zwv, ldw=G * D,
                            wdynamic=True, wt=True) for h in range(H)]
        arrs.append((lib.LinearDesc * H)(*do))
    need = lib.workspace_size_batch(list(arrs[0]))
    assert need == 0
    torch.cuda.synchronize()
    sp = torch.cuda.current_stream().cuda_stream
    for r in range(R):
        vbuf.copy_(vds[r])
        assert lib.lib.mq_linear_batch(arrs[r], H, None, 0, sp) == 0
    torch.cuda.synchronize()
    assert lib.check_device_status() == 0
    for r in range(R):
        for h in range(H):
            g = h // rep
            vtg = np.ascontiguousarray(vs[r][:, g * D:(g + 1) * D].T)
            opk, _ = oracle.pack(vtg, 8)
            want = oracle.linear(np.ascontiguousarray(ps[r][h]), zp, opk, 8, D, m0o, sho, zyo,
                                 zw=np.full(D, zv, np.int32))
            assert_equal_int8(outs[r][:, h * D:(h + 1) * D].cpu().numpy(), want,
                              f"round {r} P V head {h}")
    del keep


@pytest.mark.parametrize("m", [3, 140])
def test_o16_int4_zero_points_across_chunks(m):
    # int16 outputs, int4 weights with zero points at the range ends, K = 20480:
    # the tensor-core kernel's 8192-k chunks of x (w - zw) full twice and
    # ragged once (m = 140), the decode kernel's stages (m = 3)
    torch = torch_cuda()
    lib = mq()
    n, k = 72, 20480
    c = synth.random_case(900 + m, m, k, n, 4, "mixed")
    zw = np.where(np.arange(n) % 2 == 0, -8, 7).astype(np.int32)
    rng = np.random.default_rng(m)
    m0 = rng.integers(1 << 30, 1 << 31, size=n).astype(np.int32)
    sh = rng.integers(36, 48, size=n).astype(np.int32)
    packed, colsum = lib.pack_weights(c.w, 4)
    keep = [upload(a) for a in (c.x, packed, colsum, m0, sh, zw)]
    y = torch.full((m, n), 1, dtype=torch.int16, device="cuda")
    keep.append(y)
    d = lib.make_desc(keep[0], c.zx, keep[1], keep[2], n, keep[3], keep[4], -1000, y, 4,
                      zw=keep[5])
    _run([d], keep)
    opk, _ = oracle.pack(c.w, 4)
    want = oracle.linear_o16(c.x, c.zx, opk, 4, n, m0, sh, -1000, zw=zw)
    assert_equal(y.cpu().numpy(), want, f"o16 int4 zw K=20480 m={m}")


def test_batch_mixes_output_widths_and_kernels():
    # one call: int16-output problems (prefill and decode), 8-bit problems (one
    # asymmetric, one decode) and 16-bit-activation problems: every (kernel,
    # width) family is launched, results as if each ran alone
    torch = torch_cuda()
    lib = mq()
    keep, descs, wants, outs = [], [], [], []

    def add(seed, m, k, n, bits, obits=8, abits=8, asym=False):
        case = (synth.random_case_a16(seed, m, k, n, bits) if abits == 16
                else synth.random_case(seed, m, k, n, bits))
        rng = np.random.default_rng(seed)
        if obits == 16 and abits == 8:
            m0 = rng.integers(1 << 30, 1 << 31, size=n).astype(np.int32)
            sh = rng.integers(36, 46, size=n).astype(np.int32)
        else:
            m0, sh = lib.requant_params(case.sw, case.sx, case.sy)
        lo, hi = (-128, 127) if bits == 8 else (-8, 7)
        zw = rng.integers(lo, hi + 1, size=n).astype(np.int32) if asym else None
        packed, colsum = lib.pack_weights(case.w, bits)
        dev = [upload(a) for a in (case.x, packed, colsum, m0, sh)]
        zwd = upload(zw) if asym else None
        y = torch.full((m, n), 3, dtype=torch.int16 if 16 in (obits, abits) else torch.int8,
                       device="cuda")
        keep.extend(dev + [zwd, y])
        descs.append(lib.make_desc(dev[0], case.zx, dev[1], dev[2], n, dev[3], dev[4], case.zy
                                   if obits == 8 or abits == 16 else 77, y, bits, zw=zwd,
                                   abits=abits))
        opk, _ = oracle.pack(case.w, bits)
        if abits == 16:
            om0, osh = oracle.requant_params(case.sx, case.sw, case.sy)
            wants.append(oracle.linear_a16(case.x, case.zx, opk, bits, n, om0, osh, case.zy))
        elif obits == 16:
            wants.append(oracle.linear_o16(case.x, case.zx, opk, bits, n, m0, sh, 77, zw=zw))
        else:
            om0, osh = oracle.requant_params(case.sx, case.sw, case.sy)
            wants.append(oracle.linear(case.x, case.zx, opk, bits, n, om0, osh, case.zy, zw=zw))
        outs.append(y)

    add(1001, 96, 512, 100, 8, obits=16, asym=True)    # prefill, int16 out
    add(1002, 4, 1024, 80, 4, obits=16)                # decode, int16 out
    add(1003, 130, 768, 64, 8, asym=True)              # prefill, int8, asymmetric
    add(1004, 2, 512, 96, 4)                           # decode, int8
    add(1005, 40, 256, 72, 8, abits=16)                # prefill, 16-bit activations
    add(1006, 3, 256, 48, 4, abits=16)                 # decode, 16-bit activations
    _run(descs, keep)
    for i, (y, want) in enumerate(zip(outs, wants)):
        assert_equal(y.cpu().numpy(), want, f"mixed batch problem {i}")


def test_transpose_into_a_padded_destination():
    torch = torch_cuda()
    lib = mq()
    rng = np.random.default_rng(21)
    a = rng.integers(-128, 128, size=(70, 200), dtype=np.int16).astype(np.int8)
    ad = upload(a)
    dst = torch.full((200, 96), 5, dtype=torch.int8, device="cuda")   # ldd 96 > rows 70
    lib.transpose_i8(ad[:, 8:200], dst=dst[:192])
    torch.cuda.synchronize()
    got = dst.cpu().numpy()
    assert np.array_equal(got[:192, :70], a[:, 8:200].T)
    assert np.all(got[:192, 70:] == 5) and np.all(got[192:] == 5)   # padding untouched


@pytest.mark.parametrize("t_q", [96, 2])
def test_w8a16_setting_attention_matmuls(t_q):
    # the W8A16 setting's attention: 16-bit Q against 8-bit keys (a head's
    # slice through the row pitch, key zero point as zw), 16-bit P against 8-bit
    # V^T (value zero point), int16 outputs; t_q = 96: tensor-core kernel (plane
    # pre-pass), t_q = 2: decode kernel
    torch = torch_cuda()
    lib = mq()
    rng = np.random.default_rng(77 + t_q)
    T, H, G, D = 96, 4, 2, 64
    rep = H // G
    q = rng.integers(-32768, 32768, size=(t_q, H * D)).astype(np.int16)
    kk = rng.integers(-128, 128, size=(T, G * D)).astype(np.int8)
    v = rng.integers(-128, 128, size=(T, G * D)).astype(np.int8)
    p = rng.integers(-32768, 32768, size=(H, t_q, T)).astype(np.int16)
    zq, zk, zv, zp = 1234, -7, 100, -32768
    qd, kd, vd, pd = upload(q), upload(kk), upload(v), upload(p)
    keep = [qd, kd, vd, pd]
    colk = lib.head_row_sums(kd, G)
    vt = lib.transpose_i8(vd)                 # [G d][T]
    colv = lib.row_sums(vt)
    m0s, shs = np.full(T, 1 << 30, np.int32), np.full(T, 40, np.int32)
    m0o, sho = np.full(D, 1 << 30, np.int32), np.full(D, 44, np.int32)
    dev = [upload(a) for a in (m0s, shs, np.full(T, zk, np.int32), m0o, sho,
                               np.full(D, zv, np.int32))]
    keep += [colk, vt, colv] + dev
    m0sd, shsd, zwk, m0od, shod, zwv = dev
    s = torch.full((H, t_q, T), 3, dtype=torch.int16, device="cuda")
    o = torch.full((t_q, H * D), 3, dtype=torch.int16, device="cuda")
    keep += [s, o]
    descs = [lib.make_desc(qd[:, h * D:(h + 1) * D], zq, kd[:, (h // rep) * D:], colk[h // rep],
                           T, m0sd, shsd, 11, s[h], 8, zw=zwk, ldw=G * D, wdynamic=True)
             for h in range(H)]
    descs += [lib.make_desc(pd[h], zp, vt[(h // rep) * D:(h // rep + 1) * D],
                            colv[(h // rep) * D:(h // rep + 1) * D], D, m0od, shod, -9,
                            o[:, h * D:(h + 1) * D], 8, zw=zwv, wdynamic=True)
              for h in range(H)]
    assert all(d.abits == 16 and d.obits == 16 for d in descs)
    _run(descs[:H], keep)
    _run(descs[H:], keep)
    for h in range(H):
        g = h // rep
        opk, _ = oracle.pack(np.ascontiguousarray(kk[:, g * D:(g + 1) * D]), 8)
        want = oracle.linear_a16(np.ascontiguousarray(q[:, h * D:(h + 1) * D]), zq, opk, 8, T,
                                 m0s, shs, 11, zw=np.full(T, zk, np.int32))
        assert_equal(s[h].cpu().numpy(), want, f"w8a16 scores head {h}")
        opk, _ = oracle.pack(np.ascontiguousarray(v[:, g * D:(g + 1) * D].T), 8)
        want = oracle.linear_a16(np.ascontiguousarray(p[h]), zp, opk, 8, D, m0o, sho, -9,
                                 zw=np.full(D, zv, np.int32))
        assert_equal(o[:, h * D:(h + 1) * D].cpu().numpy(), want, f"w8a16 P V head {h}")
