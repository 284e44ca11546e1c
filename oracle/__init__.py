"""fp64 CPU oracle of the Subspace Networks stage-boundary codec.

TEST INFRASTRUCTURE ONLY.  Only the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this package.  It shares no code
with the CUDA library and the product path never reaches it.

Arrays are numpy: bf16 tensors travel as ``np.uint16`` bit patterns, fp32 as
``np.float32`` and fp64 as ``np.float64``.  Each call returns the rounded
output, the unrounded fp64 output and the oracle's status code.

Definitions (each evaluated in fp64 and rounded once, nearest-even):
  compress_fwd    C  = (X - T_fixed[ids] - P[pos]) U      Sec. 4.3.1, Eq. (subtract)
  decompress_fwd  X  = C U^T + P[pos] + T_fixed[ids]        Sec. 4.3.1
  compress_bwd    Cg = G U                                  Sec. 4.4, Eq. (grad_compress)
  decompress_bwd  G  = Cg U^T                               Sec. 4.4
  project_weight  W' = U (U^T W)                            Sec. 4.3, Sec. 5, App. A
"""
import ctypes

import numpy as np

from . import build as _build

BF16, F32, F64 = 0, 1, 2
OK, ERR_INVALID_ARG, ERR_BAD_ID = 0, 1, 4

_NP = {BF16: np.uint16, F32: np.float32, F64: np.float64}
_P = ctypes.c_void_p
_I64 = ctypes.c_int64
_I32 = ctypes.c_int32
_INT = ctypes.c_int


def dtype_code(arr):
    """Oracle dtype code of a numpy array (uint16 means bf16 bits)."""
    if arr.dtype == np.uint16:
        return BF16
    if arr.dtype == np.float32:
        return F32
    if arr.dtype == np.float64:
        return F64
    raise TypeError("unsupported dtype %s" % arr.dtype)


def _ptr(a):
    return None if a is None else a.ctypes.data_as(_P)


def _c(a, dt=None):
    if a is None:
        return None
    a = np.ascontiguousarray(a)
    if dt is not None and a.dtype != dt:
        raise TypeError("expected %s, got %s" % (dt, a.dtype))
    return a


class Oracle:
    """ctypes view of one build of the oracle library."""

    def __init__(self, lib_path=None):
        if lib_path is None:
            lib_path = _build.build()
        self.path = lib_path
        lib = ctypes.CDLL(lib_path)
        lib.sno_compress_fwd.argtypes = [_INT, _P, _P, _P, _I64, _I32, _P, _I64, _P, _INT, _P,
                                         _I32, _I32, _P, _P]
        lib.sno_decompress_fwd.argtypes = lib.sno_compress_fwd.argtypes
        lib.sno_compress_bwd.argtypes = [_INT, _P, _I64, _INT, _P, _I32, _I32, _P, _P]
        lib.sno_decompress_bwd.argtypes = lib.sno_compress_bwd.argtypes
        lib.sno_project_weight.argtypes = [_INT, _P, _I64, _I64, _I64, _INT, _P, _I32, _I32, _P,
                                           _P]
        lib.sno_wire_bytes.argtypes = [_INT, _I64, _I32]
        lib.sno_wire_bytes.restype = _I64
        lib.sno_round_bf16.argtypes = [_P, _P, _I64]
        for f in ("sno_compress_fwd", "sno_decompress_fwd", "sno_compress_bwd",
                  "sno_decompress_bwd", "sno_project_weight"):
            getattr(lib, f).restype = _INT
        self.lib = lib

    # -- helpers ------------------------------------------------------------
    @staticmethod
    def _u(U):
        U = np.ascontiguousarray(U)
        if U.dtype not in (np.float32, np.float64):
            raise TypeError("U must be float32 or float64")
        return U, (F32 if U.dtype == np.float32 else F64)

    def round_bf16(self, x):
        x = np.ascontiguousarray(x, dtype=np.float64)
        out = np.empty(x.shape, np.uint16)
        self.lib.sno_round_bf16(_ptr(x), _ptr(out), x.size)
        return out

    def wire_bytes(self, dtype, T, k):
        return int(self.lib.sno_wire_bytes(dtype, T, k))

    # -- the five operations -------------------------------------------------
    def compress_fwd(self, X, ids, tok_emb, U, seq_len, pos_emb=None, pos=None):
        X = _c(X)
        dt = dtype_code(X)
        T, d = X.shape
        U, udt = self._u(U)
        k = U.shape[1]
        ids = _c(ids, np.int32)
        pos = _c(pos, np.int32)
        tok_emb = _c(tok_emb, X.dtype)
        pos_emb = _c(pos_emb, X.dtype)
        C = np.empty((T, k), _NP[dt])
        C64 = np.empty((T, k), np.float64)
        st = self.lib.sno_compress_fwd(dt, _ptr(X), _ptr(ids), _ptr(pos), T, seq_len,
                                       _ptr(tok_emb), tok_emb.shape[0], _ptr(pos_emb), udt,
                                       _ptr(U), d, k, _ptr(C), _ptr(C64))
        return C, C64, st

    def decompress_fwd(self, C, ids, tok_emb, U, seq_len, pos_emb=None, pos=None):
        C = _c(C)
        dt = dtype_code(C)
        T, k = C.shape
        U, udt = self._u(U)
        d = U.shape[0]
        ids = _c(ids, np.int32)
        pos = _c(pos, np.int32)
        tok_emb = _c(tok_emb, C.dtype)
        pos_emb = _c(pos_emb, C.dtype)
        X = np.empty((T, d), _NP[dt])
        X64 = np.empty((T, d), np.float64)
        st = self.lib.sno_decompress_fwd(dt, _ptr(C), _ptr(ids), _ptr(pos), T, seq_len,
                                         _ptr(tok_emb), tok_emb.shape[0], _ptr(pos_emb), udt,
                                         _ptr(U), d, k, _ptr(X), _ptr(X64))
        return X, X64, st

    def compress_bwd(self, G, U):
        G = _c(G)
        dt = dtype_code(G)
        T, d = G.shape
        U, udt = self._u(U)
        k = U.shape[1]
        C = np.empty((T, k), _NP[dt])
        C64 = np.empty((T, k), np.float64)
        st = self.lib.sno_compress_bwd(dt, _ptr(G), T, udt, _ptr(U), d, k, _ptr(C), _ptr(C64))
        return C, C64, st

    def decompress_bwd(self, C, U):
        C = _c(C)
        dt = dtype_code(C)
        T, k = C.shape
        U, udt = self._u(U)
        d = U.shape[0]
        G = np.empty((T, d), _NP[dt])
        G64 = np.empty((T, d), np.float64)
        st = self.lib.sno_decompress_bwd(dt, _ptr(C), T, udt, _ptr(U), d, k, _ptr(G),
                                         _ptr(G64))
        return G, G64, st

    def project_weight(self, W, U):
        W = _c(W)
        dt = dtype_code(W)
        rows, cols = W.shape
        U, udt = self._u(U)
        d, k = U.shape
        Wo = np.empty_like(W)
        W64 = np.empty((rows, cols), np.float64)
        st = self.lib.sno_project_weight(dt, _ptr(W), rows, cols, cols, udt, _ptr(U), d, k,
                                         _ptr(Wo), _ptr(W64))
        return Wo, W64, st


_DEFAULT = None


def default():
    """The oracle built from oracle/sn_oracle.c (built on first use)."""
    global _DEFAULT
    if _DEFAULT is None:
        _DEFAULT = Oracle()
    return _DEFAULT


def bf16_to_f64(bits):
    """Widen bf16 bit patterns (uint16) to fp64 exactly."""
    bits = np.ascontiguousarray(bits, dtype=np.uint16)
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


__all__ = ["Oracle", "default", "bf16_to_f64", "BF16", "F32", "F64", "OK", "ERR_BAD_ID",
           "ERR_INVALID_ARG"]
