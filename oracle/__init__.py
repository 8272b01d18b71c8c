"""CPU oracle for the integer-only quantized linear layer (MobileQuant, arXiv 2408.13933).

TEST INFRASTRUCTURE ONLY: the test suite, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline leg are the only callers.  The product path (the CUDA
library and its Python binding) never imports this package.

The arithmetic lives in plain C (``mq_oracle.c``); this module compiles it
with gcc and marshals numpy arrays through ctypes.  Function-by-function
citations of the paper are in ``mq_oracle.h``.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "mq_oracle.c")
_HDR = os.path.join(_HERE, "mq_oracle.h")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

OK, EINVAL, EOVERFLOW = 0, 1, 2


def build(force: bool = False) -> str:
    """Compile liboracle.so with gcc (-O2, no vectorisation flags, one thread)."""
    newest = max(os.path.getmtime(_SRC), os.path.getmtime(_HDR))
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < newest:
        tmp = _LIB + ".tmp.%d" % os.getpid()
        subprocess.check_call(
            ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fPIC", "-shared", "-Wall",
             "-Wextra", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


def _bind(lib):
    p = ctypes.c_void_p
    i32, i64, f32, ci = ctypes.c_int32, ctypes.c_int64, ctypes.c_float, ctypes.c_int
    lib.oracle_requant_params.argtypes = [f32, p, ci, f32, p, p]
    lib.oracle_pack.argtypes = [p, ci, ci, ci, p, p]
    lib.oracle_unpack.argtypes = [p, ci, ci, ci, p]
    lib.oracle_linear.argtypes = [p, ci, ci, ci, i32, p, ci, ci, p, p, i32, p, ci, p]
    lib.oracle_linear_points.argtypes = [p, ci, ci, ci, i32, p, ci, ci, p, p, i32, p, ci, p, p]
    lib.oracle_linear_asym.argtypes = [p, ci, ci, ci, i32, p, ci, ci, p, p, p, i32, p, ci, p]
    lib.oracle_linear_points_asym.argtypes = [p, ci, ci, ci, i32, p, ci, ci, p, p, p, i32, p,
                                              ci, p, p]
    lib.oracle_requant_one.argtypes = [i64, i32, i32, i32]
    lib.oracle_requant_one.restype = i32
    lib.oracle_linear_a16.argtypes = [p, ci, ci, ci, i32, p, ci, ci, p, p, i32, p, ci, p]
    lib.oracle_linear_a16_asym.argtypes = [p, ci, ci, ci, i32, p, ci, ci, p, p, p, i32, p, ci, p]
    lib.oracle_linear_points_a16.argtypes = [p, ci, ci, ci, i32, p, ci, ci, p, p, i32, p, ci,
                                             p, p]
    lib.oracle_requant_one_a16.argtypes = [i64, i32, i32, i32]
    lib.oracle_requant_one_a16.restype = i32
    lib.oracle_quantize_f32.argtypes = [p, i64, f32, i32, ci, p]
    lib.oracle_dequantize.argtypes = [p, ci, i64, f32, i32, p]
    lib.oracle_requantize.argtypes = [p, ci, i64, i32, i32, i32, i32, p, ci]
    lib.oracle_fold_weights.argtypes = [p, ci, ci, p, p, p]
    lib.oracle_linear_o16.argtypes = [p, ci, ci, ci, i32, p, ci, ci, p, p, p, i32, p, ci]
    lib.oracle_quantize_weights.argtypes = [p, ci, ci, ci, ci, p, p, p]
    lib.oracle_fold_norm.argtypes = [p, p, p, ci, p, p]
    lib.oracle_residual_add.argtypes = [p, p, i64, p]
    lib.oracle_residual_add.restype = None
    return lib


def _ptr(a: np.ndarray):
    assert a.flags["C_CONTIGUOUS"], "oracle arrays must be C-contiguous"
    return a.ctypes.data_as(ctypes.c_void_p)


class OracleError(RuntimeError):
    pass


def _check(rc: int, what: str):
    if rc != OK:
        raise OracleError(f"{what} failed with oracle code {rc}")


class Oracle:
    """numpy front end over one compiled copy of the C oracle."""

    def __init__(self, lib_path: str):
        self.lib = _bind(ctypes.CDLL(lib_path))

    def requant_params(self, sx: float, sw: np.ndarray, sy: float):
        """Per-channel (M0, shift) with M0 * 2^-shift ~= sx*sw[n]/sy (see header)."""
        sw = np.ascontiguousarray(sw, dtype=np.float32)
        n = sw.shape[0]
        m0 = np.zeros(n, np.int32)
        sh = np.zeros(n, np.int32)
        _check(self.lib.oracle_requant_params(float(sx), _ptr(sw), n, float(sy), _ptr(m0),
                                              _ptr(sh)), "oracle_requant_params")
        return m0, sh

    def pack(self, w: np.ndarray, bits: int):
        """Pack int8 values [N, K] -> (packed uint8, colsum int32)."""
        w = np.ascontiguousarray(w, dtype=np.int8)
        n, k = w.shape
        packed = np.zeros((n, k if bits == 8 else k // 2), np.uint8)
        colsum = np.zeros(n, np.int32)
        _check(self.lib.oracle_pack(_ptr(w), n, k, bits, _ptr(packed), _ptr(colsum)),
               "oracle_pack")
        return packed, colsum

    def unpack(self, packed: np.ndarray, n: int, k: int, bits: int) -> np.ndarray:
        packed = np.ascontiguousarray(packed, dtype=np.uint8)
        w = np.zeros((n, k), np.int8)
        _check(self.lib.oracle_unpack(_ptr(packed), n, k, bits, _ptr(w)), "oracle_unpack")
        return w

    def linear(self, x: np.ndarray, zx: int, packed: np.ndarray, bits: int, n: int,
               m0: np.ndarray, shift: np.ndarray, zy: int, want_acc: bool = False,
               zw: np.ndarray | None = None):
        """Full integer linear layer: returns y int8 [M, N] (and acc int32 [M, N]).
        `zw` (int32 [N]) gives asymmetric weights (oracle_linear_asym)."""
        x = np.ascontiguousarray(x, dtype=np.int8)
        m, k = x.shape
        packed = np.ascontiguousarray(packed, dtype=np.uint8)
        m0 = np.ascontiguousarray(m0, dtype=np.int32)
        shift = np.ascontiguousarray(shift, dtype=np.int32)
        y = np.zeros((m, n), np.int8)
        acc = np.zeros((m, n), np.int32) if want_acc else None
        accp = _ptr(acc) if acc is not None else None
        if zw is None:
            _check(self.lib.oracle_linear(_ptr(x), m, k, k, int(zx), _ptr(packed), bits, n,
                                          _ptr(m0), _ptr(shift), int(zy), _ptr(y), n, accp),
                   "oracle_linear")
        else:
            zw = np.ascontiguousarray(zw, dtype=np.int32)
            _check(self.lib.oracle_linear_asym(_ptr(x), m, k, k, int(zx), _ptr(packed), bits, n,
                                               _ptr(zw), _ptr(m0), _ptr(shift), int(zy),
                                               _ptr(y), n, accp),
                   "oracle_linear_asym")
        return (y, acc) if want_acc else y

    def linear_points(self, x: np.ndarray, zx: int, packed: np.ndarray, bits: int, n: int,
                      m0: np.ndarray, shift: np.ndarray, zy: int, pts: np.ndarray,
                      zw: np.ndarray | None = None):
        """The layer at listed (m, n) coordinates only: returns (y[i], acc[i])."""
        x = np.ascontiguousarray(x, dtype=np.int8)
        m, k = x.shape
        pts = np.ascontiguousarray(pts, dtype=np.int64).reshape(-1, 2)
        cnt = pts.shape[0]
        y = np.zeros(cnt, np.int8)
        acc = np.zeros(cnt, np.int32)
        packed = np.ascontiguousarray(packed, dtype=np.uint8)
        m0 = np.ascontiguousarray(m0, dtype=np.int32)
        shift = np.ascontiguousarray(shift, dtype=np.int32)
        if zw is None:
            _check(self.lib.oracle_linear_points(_ptr(x), m, k, k, int(zx), _ptr(packed), bits,
                                                 n, _ptr(m0), _ptr(shift), int(zy), _ptr(pts),
                                                 cnt, _ptr(y), _ptr(acc)),
                   "oracle_linear_points")
        else:
            zw = np.ascontiguousarray(zw, dtype=np.int32)
            _check(self.lib.oracle_linear_points_asym(_ptr(x), m, k, k, int(zx), _ptr(packed),
                                                      bits, n, _ptr(zw), _ptr(m0), _ptr(shift),
                                                      int(zy), _ptr(pts), cnt, _ptr(y),
                                                      _ptr(acc)),
                   "oracle_linear_points_asym")
        return y, acc

    def requant_one(self, acc: int, m0: int, shift: int, zy: int) -> int:
        return int(self.lib.oracle_requant_one(int(acc), int(m0), int(shift), int(zy)))

    def linear_a16(self, x: np.ndarray, zx: int, packed: np.ndarray, bits: int, n: int,
                   m0: np.ndarray, shift: np.ndarray, zy: int, want_acc: bool = False,
                   zw=None):
        """The layer with int16 activations (oracle_linear_a16; with a weight
        zero point zw [N], oracle_linear_a16_asym): returns y int16 [M, N] (and
        acc int64 [M, N])."""
        x = np.ascontiguousarray(x, dtype=np.int16)
        m, k = x.shape
        packed = np.ascontiguousarray(packed, dtype=np.uint8)
        m0 = np.ascontiguousarray(m0, dtype=np.int32)
        shift = np.ascontiguousarray(shift, dtype=np.int32)
        y = np.zeros((m, n), np.int16)
        acc = np.zeros((m, n), np.int64) if want_acc else None
        if zw is not None:
            zw = np.ascontiguousarray(zw, dtype=np.int32)
            _check(self.lib.oracle_linear_a16_asym(_ptr(x), m, k, k, int(zx), _ptr(packed), bits,
                                                   n, _ptr(zw), _ptr(m0), _ptr(shift), int(zy),
                                                   _ptr(y), n, _ptr(acc) if acc is not None
                                                   else None), "oracle_linear_a16_asym")
        else:
            _check(self.lib.oracle_linear_a16(_ptr(x), m, k, k, int(zx), _ptr(packed), bits, n,
                                              _ptr(m0), _ptr(shift), int(zy), _ptr(y), n,
                                              _ptr(acc) if acc is not None else None),
                   "oracle_linear_a16")
        return (y, acc) if want_acc else y

    def linear_points_a16(self, x: np.ndarray, zx: int, packed: np.ndarray, bits: int, n: int,
                          m0: np.ndarray, shift: np.ndarray, zy: int, pts: np.ndarray):
        """oracle_linear_a16 at listed (m, n) coordinates: returns (y[i], acc[i])."""
        x = np.ascontiguousarray(x, dtype=np.int16)
        m, k = x.shape
        pts = np.ascontiguousarray(pts, dtype=np.int64).reshape(-1, 2)
        cnt = pts.shape[0]
        y = np.zeros(cnt, np.int16)
        acc = np.zeros(cnt, np.int64)
        packed = np.ascontiguousarray(packed, dtype=np.uint8)
        m0 = np.ascontiguousarray(m0, dtype=np.int32)
        shift = np.ascontiguousarray(shift, dtype=np.int32)
        _check(self.lib.oracle_linear_points_a16(_ptr(x), m, k, k, int(zx), _ptr(packed), bits,
                                                 n, _ptr(m0), _ptr(shift), int(zy), _ptr(pts),
                                                 cnt, _ptr(y), _ptr(acc)),
               "oracle_linear_points_a16")
        return y, acc

    def requant_one_a16(self, acc: int, m0: int, shift: int, zy: int) -> int:
        return int(self.lib.oracle_requant_one_a16(int(acc), int(m0), int(shift), int(zy)))

    def linear_o16(self, x: np.ndarray, zx: int, packed: np.ndarray, bits: int, n: int,
                   m0: np.ndarray, shift: np.ndarray, zy: int, zw: np.ndarray | None = None):
        """oracle_linear_o16: int8 x, 16-bit output y int16 [M, N]."""
        x = np.ascontiguousarray(x, dtype=np.int8)
        m, k = x.shape
        packed = np.ascontiguousarray(packed, dtype=np.uint8)
        m0 = np.ascontiguousarray(m0, dtype=np.int32)
        shift = np.ascontiguousarray(shift, dtype=np.int32)
        zwa = np.ascontiguousarray(zw, dtype=np.int32) if zw is not None else None
        y = np.zeros((m, n), np.int16)
        _check(self.lib.oracle_linear_o16(_ptr(x), m, k, k, int(zx), _ptr(packed), bits, n,
                                          _ptr(zwa) if zwa is not None else None, _ptr(m0),
                                          _ptr(shift), int(zy), _ptr(y), n), "oracle_linear_o16")
        return y

    def fold_weights(self, w: np.ndarray, s_in, s_out) -> np.ndarray:
        """oracle_fold_weights: f32 [N, K] -> folded f32 [N, K]."""
        w = np.ascontiguousarray(w, dtype=np.float32)
        n, k = w.shape
        si = np.ascontiguousarray(s_in, dtype=np.float32) if s_in is not None else None
        so = np.ascontiguousarray(s_out, dtype=np.float32) if s_out is not None else None
        out = np.zeros((n, k), np.float32)
        _check(self.lib.oracle_fold_weights(_ptr(w), n, k, _ptr(si) if si is not None else None,
                                            _ptr(so) if so is not None else None, _ptr(out)),
               "oracle_fold_weights")
        return out

    def quantize_weights(self, w: np.ndarray, bits: int, scheme: int):
        """oracle_quantize_weights: f32 [N, K] -> (codes int8 [N, K], sw f32 [N], zw int32 [N])."""
        w = np.ascontiguousarray(w, dtype=np.float32)
        n, k = w.shape
        codes = np.zeros((n, k), np.int8)
        sw = np.zeros(n, np.float32)
        zw = np.zeros(n, np.int32)
        _check(self.lib.oracle_quantize_weights(_ptr(w), n, k, bits, scheme, _ptr(codes), _ptr(sw),
                                                _ptr(zw)), "oracle_quantize_weights")
        return codes, sw, zw

    def fold_norm(self, gamma: np.ndarray, beta, s: np.ndarray):
        gamma = np.ascontiguousarray(gamma, dtype=np.float32)
        s = np.ascontiguousarray(s, dtype=np.float32)
        k = gamma.size
        g = np.zeros(k, np.float32)
        b = np.zeros(k, np.float32) if beta is not None else None
        beta = np.ascontiguousarray(beta, dtype=np.float32) if beta is not None else None
        _check(self.lib.oracle_fold_norm(_ptr(gamma), _ptr(beta) if beta is not None else None,
                                         _ptr(s), k, _ptr(g), _ptr(b) if b is not None else None),
               "oracle_fold_norm")
        return g, b

    def quantize(self, x: np.ndarray, alpha: float, z: int, bits: int) -> np.ndarray:
        """oracle_quantize_f32: f32 values -> int8 / int16 codes."""
        x = np.ascontiguousarray(x, dtype=np.float32)
        q = np.zeros(x.shape, np.int8 if bits == 8 else np.int16)
        _check(self.lib.oracle_quantize_f32(_ptr(x), x.size, float(alpha), int(z), bits, _ptr(q)),
               "oracle_quantize_f32")
        return q

    def dequantize(self, q: np.ndarray, alpha: float, z: int) -> np.ndarray:
        bits = 8 if q.dtype == np.int8 else 16
        q = np.ascontiguousarray(q)
        f = np.zeros(q.shape, np.float32)
        _check(self.lib.oracle_dequantize(_ptr(q), bits, q.size, float(alpha), int(z), _ptr(f)),
               "oracle_dequantize")
        return f

    def requantize(self, q: np.ndarray, zx: int, m0: int, shift: int, zy: int,
                   out_bits: int) -> np.ndarray:
        in_bits = 8 if q.dtype == np.int8 else 16
        q = np.ascontiguousarray(q)
        y = np.zeros(q.shape, np.int8 if out_bits == 8 else np.int16)
        _check(self.lib.oracle_requantize(_ptr(q), in_bits, q.size, int(zx), int(m0), int(shift),
                                          int(zy), _ptr(y), out_bits), "oracle_requantize")
        return y

    def residual_add(self, a: np.ndarray, b: np.ndarray) -> np.ndarray:
        a = np.ascontiguousarray(a, dtype=np.int8)
        b = np.ascontiguousarray(b, dtype=np.int8)
        assert a.shape == b.shape
        out = np.zeros_like(a)
        self.lib.oracle_residual_add(_ptr(a), _ptr(b), a.size, _ptr(out))
        return out


def _default() -> Oracle:
    global _lib
    with _lock:
        if _lib is None:
            build()
            _lib = Oracle(_LIB)
    return _lib


def requant_params(sx, sw, sy):
    return _default().requant_params(sx, sw, sy)


def pack(w, bits):
    return _default().pack(w, bits)


def unpack(packed, n, k, bits):
    return _default().unpack(packed, n, k, bits)


def linear(x, zx, packed, bits, n, m0, shift, zy, want_acc=False, zw=None):
    return _default().linear(x, zx, packed, bits, n, m0, shift, zy, want_acc, zw)


def threads() -> int:
    """Host threads the row-parallel front end uses (every core)."""
    return max(1, os.cpu_count() or 1)


def linear_mt(x, zx, packed, bits, n, m0, shift, zy, zw=None, nthreads=None):
    """oracle.linear over row blocks on every host core: the same C function,
    called on disjoint slices of the token rows from a thread pool (ctypes
    releases the GIL during the call).  Rows are independent in the layer, so
    the result is the single-threaded one.  Returns y int8 [M, N]."""
    from concurrent.futures import ThreadPoolExecutor
    x = np.ascontiguousarray(x, dtype=np.int8)
    m = x.shape[0]
    t = min(nthreads or threads(), max(1, m))
    if t <= 1:
        return linear(x, zx, packed, bits, n, m0, shift, zy, zw=zw)
    bounds = [m * i // t for i in range(t + 1)]
    o = _default()
    with ThreadPoolExecutor(max_workers=t) as ex:
        parts = list(ex.map(
            lambda i: o.linear(x[bounds[i]:bounds[i + 1]], zx, packed, bits, n, m0, shift, zy,
                               zw=zw), range(t)))
    return np.concatenate(parts, axis=0) if parts else np.zeros((0, n), np.int8)


def linear_points(x, zx, packed, bits, n, m0, shift, zy, pts, zw=None):
    return _default().linear_points(x, zx, packed, bits, n, m0, shift, zy, pts, zw)


def requant_one(acc, m0, shift, zy):
    return _default().requant_one(acc, m0, shift, zy)


def linear_a16(x, zx, packed, bits, n, m0, shift, zy, want_acc=False, zw=None):
    return _default().linear_a16(x, zx, packed, bits, n, m0, shift, zy, want_acc, zw)


def linear_points_a16(x, zx, packed, bits, n, m0, shift, zy, pts):
    return _default().linear_points_a16(x, zx, packed, bits, n, m0, shift, zy, pts)


def requant_one_a16(acc, m0, shift, zy):
    return _default().requant_one_a16(acc, m0, shift, zy)


def fold_weights(w, s_in, s_out):
    return _default().fold_weights(w, s_in, s_out)


def linear_o16(x, zx, packed, bits, n, m0, shift, zy, zw=None):
    return _default().linear_o16(x, zx, packed, bits, n, m0, shift, zy, zw)


def quantize_weights(w, bits, scheme):
    return _default().quantize_weights(w, bits, scheme)


def fold_norm(gamma, beta, s):
    return _default().fold_norm(gamma, beta, s)


def quantize(x, alpha, z, bits):
    return _default().quantize(x, alpha, z, bits)


def dequantize(q, alpha, z):
    return _default().dequantize(q, alpha, z)


def requantize(q, zx, m0, shift, zy, out_bits):
    return _default().requantize(q, zx, m0, shift, zy, out_bits)


def residual_add(a, b):
    return _default().residual_add(a, b)


def compile_variant(src_text: str, out_path: str) -> str:
    """Compile a (test-modified) copy of the oracle source to out_path."""
    d = os.path.dirname(out_path)
    c_path = os.path.join(d, "mq_oracle_variant.c")
    with open(c_path, "w") as f:
        f.write(src_text)
    import shutil
    shutil.copy(_HDR, os.path.join(d, "mq_oracle.h"))
    subprocess.check_call(["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fPIC", "-shared",
                           "-o", out_path, c_path, "-lm"])
    return out_path


def source() -> str:
    with open(_SRC) as f:
        return f.read()


def raw():
    """The ctypes handle (for tests that probe argument validation)."""
    return _default().lib
