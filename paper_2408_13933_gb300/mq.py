"""Thin ctypes binding of libmq (include/mq.h): argument marshalling only.

Every computation runs in libmq's CUDA kernels (or, for the host-side calls
mq_requant_params / mq_pack_weights(on_device=0), in its C++ host code).
Importing this module loads libmq.so and raises ImportError if it has not
been built -- there is no fallback.

Tensors are torch tensors (device memory and streams come from PyTorch);
numpy arrays are accepted where the C call takes host memory.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

from . import build as _build

_LIB_PATH = _build.LIB
if not os.path.exists(_LIB_PATH):
    raise ImportError(
        f"libmq.so not found at {_LIB_PATH}: build it first "
        "(python -m paper_2408_13933_gb300.build, or __graft_entry__.build())")
lib = ctypes.CDLL(_LIB_PATH)

MQ_OK = 0
MQ_ERR_INVALID_ARG = 1
MQ_ERR_UNSUPPORTED_SHAPE = 2
MQ_ERR_K_OVERFLOW = 3
MQ_ERR_ALIGNMENT = 4
MQ_ERR_CUDA = 5
MQ_ERR_DEVICE_TIMEOUT = 6
MQ_ERR_WORKSPACE = 7
MQ_MAX_K = 65536
MQ_MAX_K_ASYM8 = 32768
MQ_MAX_BATCH = 256
MQ_FOLD_MAX_JOBS = 32

EXPORTED = ["mq_status_string", "mq_requant_params", "mq_packed_size", "mq_pack_weights",
            "mq_workspace_size", "mq_linear_w8a8", "mq_linear_w4a8", "mq_linear_batch",
            "mq_check_device_status", "mq_linear_w4a8_noalloc", "mq_workspace_size_batch",
            "mq_linear_w8a16", "mq_linear_w4a16", "mq_workspace_size_a16", "mq_quantize",
            "mq_dequantize", "mq_requantize", "mq_fold_quantize_pack", "mq_fold_norm",
            "mq_row_sums", "mq_head_row_sums", "mq_transpose_i8", "mq_set_wait_limit_ns",
            "mq_test_skip_partials", "mq_test_decode_kernel", "mq_test_prefill_kernel",
            "mq_weight_sq_sums", "mq_fold_quantize_pack_batch", "mq_test_tmajor_kernel"]
MQ_WEIGHTS_SYM_CHANNEL, MQ_WEIGHTS_ASYM_CHANNEL, MQ_WEIGHTS_ASYM_TENSOR = 0, 1, 2
MQ_TYPE_F32, MQ_TYPE_F16, MQ_TYPE_BF16, MQ_TYPE_I8, MQ_TYPE_I16 = 0, 1, 2, 3, 4

_vp, _i32, _int, _sz = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int, ctypes.c_size_t


class LinearDesc(ctypes.Structure):
    """Mirror of mq_linear_desc."""
    _fields_ = [("x", _vp), ("packed", _vp), ("colsum", _vp), ("M0", _vp), ("shift", _vp),
                ("residual", _vp), ("zw", _vp), ("y", _vp), ("M", _i32), ("N", _i32), ("K", _i32),
                ("ldx", _i32), ("ldy", _i32), ("zx", _i32), ("zy", _i32), ("bits", _i32),
                ("abits", _i32), ("obits", _i32), ("ldw", _i32),
                ("wdynamic", _i32), ("wsq", _vp), ("y16", _vp), ("ysq", _vp), ("x16", _vp),
                ("xsq", _vp), ("wt", _i32)]


class FoldDesc(ctypes.Structure):
    """Mirror of mq_fold_desc."""
    _fields_ = [("w", _vp), ("N", _i32), ("K", _i32), ("s_in", _vp), ("s_out", _vp),
                ("bits", _i32), ("scheme", _i32), ("packed", _vp), ("colsum", _vp), ("sw", _vp),
                ("zw", _vp), ("stats", _vp)]


lib.mq_status_string.argtypes = [_int]
lib.mq_status_string.restype = ctypes.c_char_p
lib.mq_requant_params.argtypes = [_vp, _int, ctypes.c_float, ctypes.c_float, _vp, _vp]
lib.mq_packed_size.argtypes = [_int, _int, _int, ctypes.POINTER(_sz)]
lib.mq_pack_weights.argtypes = [_vp, _int, _int, _int, _vp, _vp, _int, _vp]
lib.mq_workspace_size.argtypes = [_int, _int, _int, _int, ctypes.POINTER(_sz)]
_linear_args = [_vp, _int, _int, _int, _i32, _vp, _vp, _int, _vp, _vp, _i32, _vp, _int, _vp,
                _sz, _vp]
lib.mq_linear_w8a8.argtypes = _linear_args
lib.mq_linear_w4a8.argtypes = _linear_args
lib.mq_linear_w8a16.argtypes = _linear_args
lib.mq_linear_w4a16.argtypes = _linear_args
lib.mq_workspace_size_a16.argtypes = [_int, _int, _int, _int, ctypes.POINTER(_sz)]
lib.mq_linear_w4a8_noalloc.argtypes = [_vp, _int, _int, _int, _i32, _vp, _vp, _int, _vp, _vp, _i32,
                                       _vp, _int, _vp]
lib.mq_linear_batch.argtypes = [ctypes.POINTER(LinearDesc), _int, _vp, _sz, _vp]
lib.mq_workspace_size_batch.argtypes = [ctypes.POINTER(LinearDesc), _int, ctypes.POINTER(_sz)]
lib.mq_check_device_status.argtypes = [_vp]
_i64, _f32 = ctypes.c_int64, ctypes.c_float
lib.mq_quantize.argtypes = [_vp, _int, _i64, _f32, _i32, _vp, _int, _vp]
lib.mq_dequantize.argtypes = [_vp, _int, _i64, _f32, _i32, _vp, _vp]
lib.mq_requantize.argtypes = [_vp, _int, _i64, _i32, _i32, _i32, _i32, _vp, _int, _vp]
lib.mq_fold_quantize_pack.argtypes = [_vp, _int, _int, _vp, _vp, _int, _int, _vp, _vp, _vp, _vp,
                                      _vp, _vp]
lib.mq_fold_quantize_pack_batch.argtypes = [ctypes.POINTER(FoldDesc), _int, _vp]
lib.mq_fold_norm.argtypes = [_vp, _vp, _vp, _int, _vp, _vp]
lib.mq_row_sums.argtypes = [_vp, _int, _int, _int, _vp, _vp]
lib.mq_head_row_sums.argtypes = [_vp, _int, _int, _int, _int, _vp, _vp]
lib.mq_transpose_i8.argtypes = [_vp, _int, _int, _int, _vp, _int, _vp]
lib.mq_set_wait_limit_ns.argtypes = [ctypes.c_uint64]
lib.mq_test_skip_partials.argtypes = [_int]
lib.mq_test_decode_kernel.argtypes = [_int]
lib.mq_test_prefill_kernel.argtypes = [_int]
lib.mq_test_tmajor_kernel.argtypes = [_int]
lib.mq_weight_sq_sums.argtypes = [_vp, _int, _int, _int, _int, _vp, _vp]
for _f in EXPORTED:
    if _f != "mq_status_string":
        getattr(lib, _f).restype = _int


class MQError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = code
        super().__init__(f"{where}: {status_string(code)} ({code})")


def status_string(code: int) -> str:
    return lib.mq_status_string(int(code)).decode()


def _check(code: int, where: str):
    if code != MQ_OK:
        raise MQError(code, where)


def _ptr(t) -> int | None:
    """Address of a torch tensor's or numpy array's data (None for None)."""
    if t is None:
        return None
    if isinstance(t, np.ndarray):
        assert t.flags["C_CONTIGUOUS"]
        return t.ctypes.data
    return t.data_ptr()


def _stream(stream) -> int | None:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    return stream if isinstance(stream, int) else stream.cuda_stream


def requant_params(sw: np.ndarray, sx: float, sy: float):
    """mq_requant_params on host arrays: returns (M0, shift) int32 [N]."""
    sw = np.ascontiguousarray(sw, dtype=np.float32)
    n = sw.shape[0]
    m0 = np.zeros(n, np.int32)
    sh = np.zeros(n, np.int32)
    _check(lib.mq_requant_params(_ptr(sw), n, float(sx), float(sy), _ptr(m0), _ptr(sh)),
           "mq_requant_params")
    return m0, sh


def packed_size(n: int, k: int, bits: int) -> int:
    out = _sz(0)
    _check(lib.mq_packed_size(n, k, bits, ctypes.byref(out)), "mq_packed_size")
    return out.value


def workspace_size(m: int, n: int, k: int, bits: int) -> int:
    out = _sz(0)
    _check(lib.mq_workspace_size(m, n, k, bits, ctypes.byref(out)), "mq_workspace_size")
    return out.value


def workspace_size_a16(m: int, n: int, k: int, bits: int) -> int:
    out = _sz(0)
    _check(lib.mq_workspace_size_a16(m, n, k, bits, ctypes.byref(out)), "mq_workspace_size_a16")
    return out.value


def workspace(device=None):
    """A zero-filled device workspace large enough for any mq_linear_* or
    mq_linear_batch call (see mq_workspace_size); torch allocates it."""
    import torch
    n = workspace_size(1, 1, 0, 4)
    return torch.zeros(n, dtype=torch.uint8, device=device or "cuda")


def pack_weights(w, bits: int, stream=None):
    """mq_pack_weights.  `w` int8 [N, K]: a numpy array (host path) or a CUDA
    torch tensor (device path).  Returns (packed, colsum) on the same side."""
    n, k = w.shape
    size = packed_size(n, k, bits)
    if isinstance(w, np.ndarray):
        w = np.ascontiguousarray(w, dtype=np.int8)
        packed = np.zeros(size, np.uint8)
        colsum = np.zeros(n, np.int32)
        _check(lib.mq_pack_weights(_ptr(w), n, k, bits, _ptr(packed), _ptr(colsum), 0, None),
               "mq_pack_weights(host)")
        return packed.reshape(n, -1) if n else packed, colsum
    import torch
    assert w.is_cuda and w.dtype == torch.int8 and w.is_contiguous()
    packed = torch.empty(size, dtype=torch.uint8, device=w.device)
    colsum = torch.empty(n, dtype=torch.int32, device=w.device)
    _check(lib.mq_pack_weights(_ptr(w), n, k, bits, _ptr(packed), _ptr(colsum), 1,
                               _stream(stream)), "mq_pack_weights(device)")
    return packed.view(n, -1) if n else packed, colsum


def linear(x, zx: int, packed, colsum, n: int, m0, shift, zy: int, y, bits: int,
           ldx: int | None = None, ldy: int | None = None, m: int | None = None,
           k: int | None = None, stream=None, workspace=None, ws_bytes: int | None = None) -> int:
    """mq_linear_w8a8 / mq_linear_w4a8 on CUDA tensors; returns the status code."""
    if ws_bytes is None:
        ws_bytes = workspace.numel() * workspace.element_size() if workspace is not None else 0
    m = x.shape[0] if m is None else m
    k = x.shape[1] if k is None else k
    ldx = x.stride(0) if ldx is None else ldx
    ldy = y.stride(0) if ldy is None else ldy
    fn = lib.mq_linear_w8a8 if bits == 8 else lib.mq_linear_w4a8
    return fn(_ptr(x), m, k, ldx, int(zx), _ptr(packed), _ptr(colsum), n, _ptr(m0), _ptr(shift),
              int(zy), _ptr(y), ldy, _ptr(workspace), ws_bytes, _stream(stream))


def linear_a16(x, zx: int, packed, colsum, n: int, m0, shift, zy: int, y, bits: int,
               ldx: int | None = None, ldy: int | None = None, m: int | None = None,
               k: int | None = None, stream=None, workspace=None,
               ws_bytes: int | None = None) -> int:
    """mq_linear_w8a16 / mq_linear_w4a16 on CUDA tensors (int16 x and y);
    returns the status code."""
    if ws_bytes is None:
        ws_bytes = workspace.numel() * workspace.element_size() if workspace is not None else 0
    m = x.shape[0] if m is None else m
    k = x.shape[1] if k is None else k
    ldx = x.stride(0) if ldx is None else ldx
    ldy = y.stride(0) if ldy is None else ldy
    fn = lib.mq_linear_w8a16 if bits == 8 else lib.mq_linear_w4a16
    return fn(_ptr(x), m, k, ldx, int(zx), _ptr(packed), _ptr(colsum), n, _ptr(m0), _ptr(shift),
              int(zy), _ptr(y), ldy, _ptr(workspace), ws_bytes, _stream(stream))


def _type_of(t) -> int:
    import torch
    return {torch.float32: MQ_TYPE_F32, torch.float16: MQ_TYPE_F16, torch.bfloat16: MQ_TYPE_BF16,
            torch.int8: MQ_TYPE_I8, torch.int16: MQ_TYPE_I16}[t.dtype]


def quantize(x, alpha: float, z: int, q, stream=None) -> int:
    """mq_quantize on CUDA tensors (float x -> int8 / int16 q); returns the status."""
    return lib.mq_quantize(_ptr(x), _type_of(x), x.numel(), float(alpha), int(z), _ptr(q),
                           _type_of(q), _stream(stream))


def dequantize(q, alpha: float, z: int, f, stream=None) -> int:
    """mq_dequantize on CUDA tensors (int8 / int16 q -> f32 f); returns the status."""
    return lib.mq_dequantize(_ptr(q), _type_of(q), q.numel(), float(alpha), int(z), _ptr(f),
                             _stream(stream))


def requantize(q, zx: int, m0: int, shift: int, zy: int, y, stream=None) -> int:
    """mq_requantize on CUDA tensors (int8 / int16 codes -> int8 / int16 codes)."""
    return lib.mq_requantize(_ptr(q), _type_of(q), q.numel(), int(zx), int(m0), int(shift),
                             int(zy), _ptr(y), _type_of(y), _stream(stream))


def fold_quantize_pack(w, bits: int, scheme: int, s_in=None, s_out=None, stream=None):
    """mq_fold_quantize_pack on a CUDA f32 tensor [N, K]: returns (packed, colsum,
    sw, zw) on the device (zw None for the symmetric scheme)."""
    import torch
    n, k = w.shape
    dev = w.device
    packed = torch.empty(packed_size(n, k, bits), dtype=torch.uint8, device=dev)
    colsum = torch.empty(n, dtype=torch.int32, device=dev)
    sw = torch.empty(n, dtype=torch.float32, device=dev)
    zw = torch.empty(n, dtype=torch.int32, device=dev) if scheme != MQ_WEIGHTS_SYM_CHANNEL else None
    stats = torch.empty(2 * max(n, 1), dtype=torch.float32, device=dev)
    _check(lib.mq_fold_quantize_pack(_ptr(w), n, k, _ptr(s_in), _ptr(s_out), bits, scheme,
                                     _ptr(packed), _ptr(colsum), _ptr(sw), _ptr(zw), _ptr(stats),
                                     _stream(stream)), "mq_fold_quantize_pack")
    return (packed.view(n, packed.numel() // n) if n else packed), colsum, sw, zw


def fold_quantize_pack_batch(jobs, stream=None):
    """mq_fold_quantize_pack_batch: `jobs` is a list of (w, bits, scheme, s_in,
    s_out) with w a CUDA f32 tensor [N, K]; returns one (packed, colsum, sw, zw)
    per job, as fold_quantize_pack."""
    import torch
    outs, descs, keep = [], [], []
    for w, bits, scheme, s_in, s_out in jobs:
        n, k = w.shape
        dev = w.device
        packed = torch.empty(packed_size(n, k, bits), dtype=torch.uint8, device=dev)
        colsum = torch.empty(n, dtype=torch.int32, device=dev)
        sw = torch.empty(n, dtype=torch.float32, device=dev)
        zw = (torch.empty(n, dtype=torch.int32, device=dev)
              if scheme != MQ_WEIGHTS_SYM_CHANNEL else None)
        stats = torch.empty(2 * max(n, 1), dtype=torch.float32, device=dev)
        keep.append(stats)
        descs.append(FoldDesc(_ptr(w), n, k, _ptr(s_in), _ptr(s_out), bits, scheme, _ptr(packed),
                              _ptr(colsum), _ptr(sw), _ptr(zw), _ptr(stats)))
        outs.append(((packed.view(n, packed.numel() // n) if n else packed), colsum, sw, zw))
    arr = (FoldDesc * max(len(descs), 1))(*descs)
    _check(lib.mq_fold_quantize_pack_batch(arr, len(descs), _stream(stream)),
           "mq_fold_quantize_pack_batch")
    return outs


def fold_norm(gamma: np.ndarray, beta, s: np.ndarray):
    """mq_fold_norm on host f32 arrays: returns (gamma', beta')."""
    gamma = np.ascontiguousarray(gamma, dtype=np.float32)
    s = np.ascontiguousarray(s, dtype=np.float32)
    g = np.zeros_like(gamma)
    b = np.zeros_like(gamma) if beta is not None else None
    if beta is not None:
        beta = np.ascontiguousarray(beta, dtype=np.float32)
    _check(lib.mq_fold_norm(_ptr(gamma), _ptr(beta), _ptr(s), gamma.size, _ptr(g), _ptr(b)),
           "mq_fold_norm")
    return g, b


def weight_sq_sums(packed, n: int, k: int, bits: int, ldw: int = 0, out=None, stream=None):
    """mq_weight_sq_sums on packed CUDA weights: int32 [N], sum_k w[n][k]^2."""
    import torch
    if out is None:
        out = torch.empty(n, dtype=torch.int32, device=packed.device)
    _check(lib.mq_weight_sq_sums(_ptr(packed), n, k, bits, ldw, _ptr(out), _stream(stream)),
           "mq_weight_sq_sums")
    return out


def row_sums(x, out=None, m=None, k=None, ldx=None, stream=None):
    """mq_row_sums on an int8 CUDA tensor [M, K] (or a strided view): int32 [M]."""
    import torch
    m = x.shape[0] if m is None else m
    k = x.shape[1] if k is None else k
    ldx = x.stride(0) if ldx is None else ldx
    if out is None:
        out = torch.empty(m, dtype=torch.int32, device=x.device)
    _check(lib.mq_row_sums(_ptr(x), m, k, ldx, _ptr(out), _stream(stream)), "mq_row_sums")
    return out


def head_row_sums(x, heads: int, out=None, stream=None):
    """mq_head_row_sums on an int8 CUDA tensor [M, heads * d] (or a row-strided
    view): int32 [heads, M], the row sums of every d-wide head slice."""
    import torch
    m, width = x.shape
    assert width % heads == 0
    d = width // heads
    if out is None:
        out = torch.empty((heads, m), dtype=torch.int32, device=x.device)
    _check(lib.mq_head_row_sums(_ptr(x), m, heads, d, x.stride(0), _ptr(out), _stream(stream)),
           "mq_head_row_sums")
    return out


def transpose_i8(src, dst=None, stream=None):
    """mq_transpose_i8 on an int8 CUDA tensor [R, C] (or a row-strided view)."""
    import torch
    rows, cols = src.shape
    if dst is None:
        dst = torch.empty((cols, rows), dtype=torch.int8, device=src.device)
    _check(lib.mq_transpose_i8(_ptr(src), rows, cols, src.stride(0), _ptr(dst), dst.stride(0),
                               _stream(stream)), "mq_transpose_i8")
    return dst


def linear_w4a8_noalloc(x, zx: int, packed, colsum, n: int, m0, shift, zy: int, y,
                        ldx: int | None = None, ldy: int | None = None, m: int | None = None,
                        k: int | None = None, stream=None) -> int:
    """mq_linear_w4a8_noalloc on CUDA tensors (decode shapes, no workspace);
    returns the status code."""
    m = x.shape[0] if m is None else m
    k = x.shape[1] if k is None else k
    ldx = x.stride(0) if ldx is None else ldx
    ldy = y.stride(0) if ldy is None else ldy
    return lib.mq_linear_w4a8_noalloc(_ptr(x), m, k, ldx, int(zx), _ptr(packed), _ptr(colsum), n,
                                      _ptr(m0), _ptr(shift), int(zy), _ptr(y), ldy,
                                      _stream(stream))


def make_desc(x, zx, packed, colsum, n, m0, shift, zy, y, bits, residual=None,
              ldx=None, ldy=None, m=None, k=None, zw=None, abits=None, obits=None,
              ldw: int = 0, wdynamic: bool = False, wsq=None, y16=None, ysq=None, x16=None,
              xsq=None, wt: bool = False) -> LinearDesc:
    """One mq_linear_desc; `zw` (device int32 [N]) gives asymmetric weights;
    abits 16 (default: 16 for an int16 x) gives int16 activations and outputs;
    obits 16 with int8 x (default: 16 for an int16 y) an int16 output; `ldw`
    the bytes between weight rows (0: packed); `wdynamic` marks weights written
    by earlier work on the stream (read only after it completes); `wsq`
    (device int32 [N], weight_sq_sums) the weights' sums of squares; `y16` /
    `ysq` (device f16 [M, N] / zero-filled int32 [M]) receive y as f16 and its
    row sums of squares, `x16` / `xsq` pass those of an earlier call as this
    call's x (chained layers, see mq.h); `wt` says `packed` holds the weights
    transposed, int8 [K][N] with `ldw` bytes between k-rows (see mq.h)."""
    d = LinearDesc()
    if abits is None:
        abits = 16 if getattr(x, "element_size", lambda: 1)() == 2 else 8
    if obits is None:
        obits = 16 if getattr(y, "element_size", lambda: 1)() == 2 else 8
    d.abits = int(abits)
    d.obits = int(obits)
    d.ldw = int(ldw)
    d.wdynamic = int(bool(wdynamic))
    d.wt = int(bool(wt))
    d.x, d.packed, d.colsum = _ptr(x), _ptr(packed), _ptr(colsum)
    d.M0, d.shift, d.residual, d.y = _ptr(m0), _ptr(shift), _ptr(residual), _ptr(y)
    d.zw = _ptr(zw)
    d.wsq = _ptr(wsq)
    d.y16, d.ysq, d.x16, d.xsq = _ptr(y16), _ptr(ysq), _ptr(x16), _ptr(xsq)
    d.M = x.shape[0] if m is None else m
    d.K = x.shape[1] if k is None else k
    d.N = n
    d.ldx = x.stride(0) if ldx is None else ldx
    d.ldy = y.stride(0) if ldy is None else ldy
    d.zx, d.zy, d.bits = int(zx), int(zy), int(bits)
    return d


def workspace_size_batch(descs) -> int:
    """mq_workspace_size_batch over a list of LinearDesc."""
    arr = (LinearDesc * len(descs))(*descs)
    out = _sz(0)
    _check(lib.mq_workspace_size_batch(arr, len(descs), ctypes.byref(out)),
           "mq_workspace_size_batch")
    return out.value


def linear_batch(descs, stream=None, workspace=None, ws_bytes: int | None = None) -> int:
    """mq_linear_batch over a list of LinearDesc; returns the status code."""
    if ws_bytes is None:
        ws_bytes = workspace.numel() * workspace.element_size() if workspace is not None else 0
    arr = (LinearDesc * len(descs))(*descs)
    return lib.mq_linear_batch(arr, len(descs), _ptr(workspace), ws_bytes, _stream(stream))


def check_device_status(stream=None) -> int:
    return lib.mq_check_device_status(_stream(stream))


def set_wait_limit_ns(ns: int) -> int:
    """mq_set_wait_limit_ns: the limit of every device-side wait of later
    launches (0 restores the 1-second default)."""
    return lib.mq_set_wait_limit_ns(int(ns))


def test_skip_partials(cta: int) -> int:
    """mq_test_skip_partials (failure-detection test hook; -1 turns it off)."""
    return lib.mq_test_skip_partials(int(cta))


def test_decode_kernel(which: int) -> int:
    """mq_test_decode_kernel (test hook): 0 by shape, 1 the row-tile kernel
    whenever it can serve the launch, 2 never."""
    return lib.mq_test_decode_kernel(int(which))


def test_prefill_kernel(which: int) -> int:
    """mq_test_prefill_kernel (test hook): 0 by shape and workspace, 1 the
    256-token kernel whenever the workspace allows, 2 never."""
    return lib.mq_test_prefill_kernel(int(which))


def test_tmajor_kernel(which: int) -> int:
    """mq_test_tmajor_kernel (test hook): 0 the token-major kernel for K <= 128
    or N <= 64, 1 whenever it can serve a problem, 2 never."""
    return lib.mq_test_tmajor_kernel(int(which))
