"""Thin Python binding of libsn.so (C ABI in include/sn.h).

Argument marshalling only: each function checks tensor shapes and dtypes,
passes raw pointers, sizes and the current CUDA stream to the C entry point of
the same name, and raises SNError on a non-OK status.  Every step of the
boundary runs in the library's kernels; torch supplies device memory, pinned
host memory and streams.  There is no fallback: importing this module fails
loudly when the library has not been built.
"""
import ctypes
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libsn.so")

SN_OK, SN_ERR_INVALID_ARG, SN_ERR_ALIGNMENT, SN_ERR_UNSUPPORTED = 0, 1, 2, 3
SN_ERR_BAD_ID, SN_ERR_TIMEOUT, SN_ERR_CUDA, SN_ERR_NUMERIC = 4, 5, 6, 7
SN_BF16, SN_F32 = 0, 1

if not os.path.exists(LIB_PATH):
    raise ImportError("libsn.so is not built: run `python -c \"import __graft_entry__ as g; "
                      "g.build()\"` (needs nvcc)")

_lib = ctypes.CDLL(LIB_PATH)
_P = ctypes.c_void_p
_I32, _I64, _SZ = ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t
_ST = ctypes.c_int


def _sig(name, args, res=_ST):
    f = getattr(_lib, name)
    f.argtypes = args
    f.restype = res
    return f


_sig("sn_basis_create", [_P, _I32, _I32, ctypes.POINTER(_P), _P])
_sig("sn_basis_destroy", [_P])
_sig("sn_basis_shape", [_P, ctypes.POINTER(_I32), ctypes.POINTER(_I32)])
_sig("sn_compress_fwd", [_P, _ST, _P, _P, _P, _I64, _I32, _P, _I64, _P, _P, _P])
_sig("sn_decompress_fwd", [_P, _ST, _P, _P, _P, _I64, _I32, _P, _I64, _P, _P, _P])
_sig("sn_compress_bwd", [_P, _ST, _P, _I64, _P, _P])
_sig("sn_decompress_bwd", [_P, _ST, _P, _I64, _P, _P])
_sig("sn_project_weight_workspace", [_P, _ST, _I64, ctypes.POINTER(_SZ)])
_sig("sn_project_weight", [_P, _ST, _P, _I64, _I64, _I64, _P, _P, _SZ, _P])
_sig("sn_project_weight_noalloc", [_P, _ST, _P, _I64, _I64, _I64, _P, _P])
_sig("sn_project_tables", [_P, _ST, _P, _I64, _P, _I32, _P, _P, _P])
_sig("sn_compress_fwd_projected", [_P, _ST, _P, _P, _P, _I64, _I32, _P, _I64, _P, _P, _P])
_sig("sn_build_ts", [_P, _ST, _P, _I64, _P, _P, _SZ, _P])
_sig("sn_grassmann_workspace", [_P, _I64, ctypes.POINTER(_SZ), ctypes.POINTER(_SZ)])
_sig("sn_grassmann_accumulate", [_P, _ST, _P, _P, _I64, _P, _P, _SZ, _P])
_sig("sn_grassmann_residual", [_P, _ST, _P, _P, _I64, _P, _P])
_sig("sn_grassmann_step", [_P, _P, _I32, ctypes.c_float, _P, _P, _SZ, _P])
_sig("sn_adamw_rowconst", [_ST, _P, _P, _P, _P, _I64, _I64, _I64, ctypes.c_float, ctypes.c_float,
                           ctypes.c_float, ctypes.c_float, ctypes.c_float, _P, _SZ, _P])
_sig("sn_topk_compress", [_P, _I64, _I32, _I32, _P, _P, _P])
_sig("sn_topk_restore", [_P, _P, _I64, _I32, _I32, _P, _P])
_sig("sn_sign_compress", [_P, _I64, _I32, _P, _P, _P])
_sig("sn_sign_restore", [_P, _P, _I64, _I32, _P, _P])
_sig("sn_quant_compress", [_P, _I64, _I32, _I32, _P, _P, _P])
_sig("sn_quant_restore", [_P, _P, _I64, _I32, _I32, _P, _P])
_sig("sn_wire_bytes", [_P, _ST, _I64, ctypes.POINTER(_SZ)])
_sig("sn_wire_send", [_P, _P, _SZ, _P])
_sig("sn_wire_recv", [_P, _P, _SZ, _P])
_sig("sn_check_errors", [_P, _P])
_sig("sn_selftest_wait_timeout", [_P, _P])
_sig("sn_launch_count", [], ctypes.c_uint64)
_sig("sn_status_string", [_ST], ctypes.c_char_p)

#: every function the C header declares (checked against include/sn.h by tests)
EXPORTS = ["sn_basis_create", "sn_basis_destroy", "sn_basis_shape", "sn_compress_fwd",
           "sn_decompress_fwd", "sn_compress_bwd", "sn_decompress_bwd",
           "sn_project_weight_workspace", "sn_project_weight", "sn_project_weight_noalloc",
           "sn_project_tables", "sn_compress_fwd_projected", "sn_build_ts",
           "sn_grassmann_workspace", "sn_grassmann_accumulate", "sn_grassmann_residual",
           "sn_grassmann_step", "sn_adamw_rowconst", "sn_topk_compress", "sn_topk_restore",
           "sn_sign_compress", "sn_sign_restore", "sn_quant_compress", "sn_quant_restore",
           "sn_wire_bytes", "sn_wire_send",
           "sn_wire_recv", "sn_check_errors", "sn_selftest_wait_timeout", "sn_launch_count",
           "sn_status_string"]


class SNError(RuntimeError):
    def __init__(self, status, where):
        self.status = status
        name = _lib.sn_status_string(status).decode()
        super().__init__("%s returned %s" % (where, name))


def _check(status, where):
    if status != SN_OK:
        raise SNError(status, where)


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream if hasattr(stream, "cuda_stream") else stream)


def _dtype(t):
    if t.dtype == torch.bfloat16:
        return SN_BF16
    if t.dtype == torch.float32:
        return SN_F32
    raise TypeError("unsupported dtype %s (bf16 or fp32)" % t.dtype)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _check_rows(T, seq_len, d, pos_emb, pos, width=None):
    """pos has T entries and the positional table seq_len rows of `width`
    (d, or k for a projected table): the kernels index them without bounds
    information, so a short table is refused here."""
    if pos is not None and pos.shape != (T,):
        raise ValueError("pos must have shape [T]")
    if pos_emb is not None and (pos_emb.dim() != 2 or pos_emb.shape[0] < seq_len or
                                pos_emb.shape[1] != (d if width is None else width)):
        raise ValueError("the positional table must have seq_len rows of the right width")


def _check_out(out, shape):
    if tuple(out.shape) != tuple(shape):
        raise ValueError("out must have shape %s" % (tuple(shape),))


def _need(t, name, dtype=None, contiguous=True):
    if not isinstance(t, torch.Tensor):
        raise TypeError("%s must be a torch.Tensor" % name)
    if not t.is_cuda:
        raise ValueError("%s must be a CUDA tensor" % name)
    if dtype is not None and t.dtype != dtype:
        raise TypeError("%s must be %s, got %s" % (name, dtype, t.dtype))
    if contiguous and not t.is_contiguous():
        raise ValueError("%s must be contiguous" % name)


class Basis:
    """A basis handle: U [d, k] fp32 with orthonormal columns (Sec. 4.3)."""

    def __init__(self, U, stream=None):
        _need(U, "U", torch.float32)
        if U.dim() != 2 or not U.is_cuda:
            raise ValueError("U must be a 2-D CUDA tensor [d, k]")
        h = _P()
        _check(_lib.sn_basis_create(_ptr(U), U.shape[0], U.shape[1], ctypes.byref(h),
                                    _stream(stream)), "sn_basis_create")
        self._h = h
        self.d, self.k = int(U.shape[0]), int(U.shape[1])
        self.device = U.device

    @property
    def handle(self):
        if self._h is None:
            raise RuntimeError("basis destroyed")
        return self._h

    def destroy(self):
        if getattr(self, "_h", None) is not None:
            _check(_lib.sn_basis_destroy(self._h), "sn_basis_destroy")
            self._h = None

    def __del__(self):
        try:
            self.destroy()
        except Exception:
            pass


def sn_basis_create(U, stream=None):
    return Basis(U, stream)


def sn_basis_destroy(basis):
    basis.destroy()


def sn_basis_shape(basis):
    d, k = _I32(), _I32()
    _check(_lib.sn_basis_shape(basis.handle, ctypes.byref(d), ctypes.byref(k)), "sn_basis_shape")
    return int(d.value), int(k.value)


def sn_compress_fwd(basis, X, ids, tok_emb, seq_len, pos_emb=None, pos=None, out=None,
                    stream=None):
    """C = (X - tok_emb[ids] - pos_emb[p]) U  (Sec. 4.3.1, Eq. subtract)."""
    _need(X, "X")
    _need(ids, "ids", torch.int32)
    _need(tok_emb, "tok_emb", X.dtype)
    if pos_emb is not None:
        _need(pos_emb, "pos_emb", X.dtype)
    if pos is not None:
        _need(pos, "pos", torch.int32)
    T = X.shape[0]
    if X.shape != (T, basis.d) or ids.shape != (T,) or tok_emb.shape[1] != basis.d:
        raise ValueError("shape mismatch")
    _check_rows(T, seq_len, basis.d, pos_emb, pos)
    if out is None:
        out = torch.empty(T, basis.k, dtype=X.dtype, device=X.device)
    _need(out, "out", X.dtype)
    _check_out(out, (T, basis.k))
    _check(_lib.sn_compress_fwd(basis.handle, _dtype(X), _ptr(X), _ptr(ids), _ptr(pos), T,
                                seq_len, _ptr(tok_emb), tok_emb.shape[0], _ptr(pos_emb),
                                _ptr(out), _stream(stream)), "sn_compress_fwd")
    return out


def sn_project_tables(basis, tok_emb, pos_emb=None, TU=None, PU=None, stream=None):
    """TU = tok_emb U and PU = pos_emb U in fp32 (projected tables); returns (TU, PU)."""
    _need(tok_emb, "tok_emb")
    V = tok_emb.shape[0]
    if tok_emb.shape != (V, basis.d):
        raise ValueError("shape mismatch")
    if TU is None:
        TU = torch.empty(V, basis.k, dtype=torch.float32, device=tok_emb.device)
    _need(TU, "TU", torch.float32)
    _check_out(TU, (V, basis.k))
    n = 0
    if pos_emb is not None:
        _need(pos_emb, "pos_emb", tok_emb.dtype)
        n = pos_emb.shape[0]
        if pos_emb.shape != (n, basis.d):
            raise ValueError("shape mismatch")
        if PU is None:
            PU = torch.empty(n, basis.k, dtype=torch.float32, device=tok_emb.device)
        _need(PU, "PU", torch.float32)
        _check_out(PU, (n, basis.k))
    else:
        PU = None
    _check(_lib.sn_project_tables(basis.handle, _dtype(tok_emb), _ptr(tok_emb), V, _ptr(pos_emb),
                                  n, _ptr(TU), _ptr(PU), _stream(stream)), "sn_project_tables")
    return TU, PU


def sn_compress_fwd_projected(basis, X, ids, TU, seq_len, PU=None, pos=None, out=None,
                              stream=None):
    """C = X U - TU[ids] - PU[p]  (Eq. subtract with projected tables)."""
    _need(X, "X")
    _need(ids, "ids", torch.int32)
    _need(TU, "TU", torch.float32)
    if PU is not None:
        _need(PU, "PU", torch.float32)
    if pos is not None:
        _need(pos, "pos", torch.int32)
    T = X.shape[0]
    if X.shape != (T, basis.d) or ids.shape != (T,) or TU.dim() != 2 or TU.shape[1] != basis.k:
        raise ValueError("shape mismatch")
    _check_rows(T, seq_len, basis.d, PU, pos, width=basis.k)
    if out is None:
        out = torch.empty(T, basis.k, dtype=X.dtype, device=X.device)
    _need(out, "out", X.dtype)
    _check_out(out, (T, basis.k))
    _check(_lib.sn_compress_fwd_projected(basis.handle, _dtype(X), _ptr(X), _ptr(ids), _ptr(pos),
                                          T, seq_len, _ptr(TU), TU.shape[0], _ptr(PU), _ptr(out),
                                          _stream(stream)), "sn_compress_fwd_projected")
    return out


def sn_build_ts(basis, tok_emb, out=None, workspace=None, stream=None):
    """T_S = tok_emb U U^T (the low-rank token-embedding table, Sec. 4.3.1)."""
    _need(tok_emb, "tok_emb")
    V = tok_emb.shape[0]
    if tok_emb.shape != (V, basis.d):
        raise ValueError("shape mismatch")
    if out is None:
        out = torch.empty_like(tok_emb)
    _need(out, "out", tok_emb.dtype)
    _check_out(out, (V, basis.d))
    nbytes = sn_wire_bytes(basis, tok_emb.dtype, V)
    if workspace is None:
        workspace = torch.empty(max(16, nbytes), dtype=torch.uint8, device=tok_emb.device)
    _need(workspace, "workspace")
    _check(_lib.sn_build_ts(basis.handle, _dtype(tok_emb), _ptr(tok_emb), V, _ptr(out),
                            _ptr(workspace), workspace.numel() * workspace.element_size(),
                            _stream(stream)), "sn_build_ts")
    return out


def sn_grassmann_workspace(basis, T):
    """(accumulate bytes for T tokens, step bytes)."""
    a, b = _SZ(), _SZ()
    _check(_lib.sn_grassmann_workspace(basis.handle, T, ctypes.byref(a), ctypes.byref(b)),
           "sn_grassmann_workspace")
    return int(a.value), int(b.value)


def sn_grassmann_accumulate(basis, G, Cg, M, workspace=None, stream=None):
    """M += G^T Cg (Cg = G U from sn_compress_bwd); M fp32 [d, k] (Sec. 4.5, Sec. 6)."""
    _need(G, "G", torch.bfloat16)
    _need(Cg, "Cg", torch.bfloat16)
    _need(M, "M", torch.float32)
    T = G.shape[0]
    if G.shape != (T, basis.d) or Cg.shape != (T, basis.k) or M.shape != (basis.d, basis.k):
        raise ValueError("shape mismatch")
    if workspace is None:
        workspace = torch.empty(max(256, sn_grassmann_workspace(basis, T)[0]), dtype=torch.uint8,
                                device=G.device)
    _need(workspace, "workspace")
    _check(_lib.sn_grassmann_accumulate(basis.handle, SN_BF16, _ptr(G), _ptr(Cg), T, _ptr(M),
                                        _ptr(workspace),
                                        workspace.numel() * workspace.element_size(),
                                        _stream(stream)),
           "sn_grassmann_accumulate")
    return M


def sn_grassmann_residual(basis, G, Cg, acc, stream=None):
    """acc (device fp64 scalar) += ||G (I - U U^T)||_F^2 = ||G||^2 - ||Cg||^2."""
    _need(G, "G", torch.bfloat16)
    _need(Cg, "Cg", torch.bfloat16)
    _need(acc, "acc", torch.float64)
    T = G.shape[0]
    if G.shape != (T, basis.d) or Cg.shape != (T, basis.k) or acc.numel() < 1:
        raise ValueError("shape mismatch")
    _check(_lib.sn_grassmann_residual(basis.handle, SN_BF16, _ptr(G), _ptr(Cg), T, _ptr(acc),
                                      _stream(stream)), "sn_grassmann_residual")
    return acc


def sn_grassmann_step(basis, M, K, eta, out=None, workspace=None, stream=None):
    """U_new = QR-retraction of U - eta * tangent(-2 M / K) (Sec. 4.5); fp32 [d, k]."""
    _need(M, "M", torch.float32)
    if M.shape != (basis.d, basis.k):
        raise ValueError("shape mismatch")
    if out is None:
        out = torch.empty_like(M)
    _need(out, "out", torch.float32)
    _check_out(out, (basis.d, basis.k))
    if workspace is None:
        workspace = torch.empty(max(256, sn_grassmann_workspace(basis, 1)[1]), dtype=torch.uint8,
                                device=M.device)
    _need(workspace, "workspace")
    _check(_lib.sn_grassmann_step(basis.handle, _ptr(M), int(K), float(eta), _ptr(out),
                                  _ptr(workspace), workspace.numel() * workspace.element_size(),
                                  _stream(stream)),
           "sn_grassmann_step")
    return out


def sn_adamw_rowconst(W, grad, M, V, step, lr, beta1=0.9, beta2=0.999, eps=1e-8, lam=0.0,
                      workspace=None, stream=None):
    """One row-constant AdamW step on W [d, cols] (one adaptive rate per column; Sec. 5).
    W, M, V fp32, updated in place; grad bf16 or fp32."""
    for t_, nm in ((W, "W"), (M, "M"), (V, "V")):
        _need(t_, nm, torch.float32)
    _need(grad, "grad")
    if W.dim() != 2 or grad.shape != W.shape or M.shape != W.shape or V.shape != W.shape:
        raise ValueError("shape mismatch")
    rows, cols = W.shape
    if workspace is None:
        workspace = torch.empty(cols, dtype=torch.float32, device=W.device)
    _need(workspace, "workspace")
    _check(_lib.sn_adamw_rowconst(_dtype(grad), _ptr(W), _ptr(grad), _ptr(M), _ptr(V), rows, cols,
                                  int(step), float(lr), float(beta1), float(beta2), float(eps),
                                  float(lam), _ptr(workspace),
                                  workspace.numel() * workspace.element_size(), _stream(stream)),
           "sn_adamw_rowconst")
    return W


def sn_topk_compress(X, kk, values=None, cols=None, stream=None):
    """Per-row top-kk by magnitude of a bf16 batch: (values bf16 [T, kk], cols uint16-as-int16 [T, kk])."""
    _need(X, "X", torch.bfloat16)
    T, d = X.shape
    vals = values if values is not None else torch.empty(T, kk, dtype=torch.bfloat16,
                                                         device=X.device)
    if cols is None:
        cols = torch.empty(T, kk, dtype=torch.int16, device=X.device)
    _need(vals, "values", torch.bfloat16)
    _need(cols, "cols", torch.int16)
    if vals.shape != (T, kk) or cols.shape != (T, kk):
        raise ValueError("values and cols must be [T, kk]")
    _check(_lib.sn_topk_compress(_ptr(X), T, d, kk, _ptr(vals), _ptr(cols), _stream(stream)),
           "sn_topk_compress")
    return vals, cols


def sn_topk_restore(vals, cols, d, out=None, stream=None):
    _need(vals, "values", torch.bfloat16)
    _need(cols, "cols", torch.int16)
    T, kk = vals.shape
    if cols.shape != vals.shape:
        raise ValueError("values and cols must have the same shape [T, kk]")
    if out is None:
        out = torch.empty(T, d, dtype=torch.bfloat16, device=vals.device)
    _need(out, "out", torch.bfloat16)
    _check_out(out, (T, d))
    _check(_lib.sn_topk_restore(_ptr(vals), _ptr(cols), T, d, kk, _ptr(out), _stream(stream)),
           "sn_topk_restore")
    return out


def sn_sign_compress(X, bits=None, scale=None, stream=None):
    """1-bit signs (int32 words [T, ceil(d/32)]) and fp32 mean-magnitude row scales [T]."""
    _need(X, "X", torch.bfloat16)
    T, d = X.shape
    if bits is None:
        bits = torch.empty(T, (d + 31) // 32, dtype=torch.int32, device=X.device)
    if scale is None:
        scale = torch.empty(T, dtype=torch.float32, device=X.device)
    _need(bits, "bits", torch.int32)
    _need(scale, "scale", torch.float32)
    if bits.shape != (T, (d + 31) // 32) or scale.shape != (T,):
        raise ValueError("bits must be [T, ceil(d/32)] and scale [T]")
    _check(_lib.sn_sign_compress(_ptr(X), T, d, _ptr(bits), _ptr(scale), _stream(stream)),
           "sn_sign_compress")
    return bits, scale


def sn_sign_restore(bits, scale, d, out=None, stream=None):
    _need(bits, "bits", torch.int32)
    _need(scale, "scale", torch.float32)
    T = scale.shape[0]
    if scale.dim() != 1 or bits.shape != (T, (d + 31) // 32):
        raise ValueError("bits must be [T, ceil(d/32)] and scale [T]")
    if out is None:
        out = torch.empty(T, d, dtype=torch.bfloat16, device=scale.device)
    _need(out, "out", torch.bfloat16)
    _check_out(out, (T, d))
    _check(_lib.sn_sign_restore(_ptr(bits), _ptr(scale), T, d, _ptr(out), _stream(stream)),
           "sn_sign_restore")
    return out


#: 8-bit formats of sn_quant_compress
QUANT_FORMATS = {"int8": 0, "e4m3": 1}


def sn_quant_compress(X, fmt, codes=None, scale=None, stream=None):
    """Row-scaled 8-bit codes (uint8 [T, d]) and fp32 row scales max|x| / qmax [T];
    fmt "int8" (qmax 127) or "e4m3" (fp8, qmax 448)."""
    _need(X, "X", torch.bfloat16)
    T, d = X.shape
    if codes is None:
        codes = torch.empty(T, d, dtype=torch.uint8, device=X.device)
    if scale is None:
        scale = torch.empty(T, dtype=torch.float32, device=X.device)
    _need(codes, "codes", torch.uint8)
    _need(scale, "scale", torch.float32)
    if codes.shape != (T, d) or scale.shape != (T,):
        raise ValueError("codes must be [T, d] and scale [T]")
    _check(_lib.sn_quant_compress(_ptr(X), T, d, QUANT_FORMATS[fmt], _ptr(codes), _ptr(scale),
                                  _stream(stream)), "sn_quant_compress")
    return codes, scale


def sn_quant_restore(codes, scale, fmt, out=None, stream=None):
    _need(codes, "codes", torch.uint8)
    _need(scale, "scale", torch.float32)
    T, d = codes.shape
    if scale.shape != (T,):
        raise ValueError("scale must be [T]")
    if out is None:
        out = torch.empty(T, d, dtype=torch.bfloat16, device=codes.device)
    _need(out, "out", torch.bfloat16)
    _check_out(out, (T, d))
    _check(_lib.sn_quant_restore(_ptr(codes), _ptr(scale), T, d, QUANT_FORMATS[fmt], _ptr(out),
                                 _stream(stream)), "sn_quant_restore")
    return out


def sn_decompress_fwd(basis, C, ids, tok_emb, seq_len, pos_emb=None, pos=None, out=None,
                      stream=None):
    """X = C U^T + pos_emb[p] + tok_emb[ids]  (Sec. 4.3.1)."""
    _need(C, "C")
    _need(ids, "ids", torch.int32)
    _need(tok_emb, "tok_emb", C.dtype)
    if pos_emb is not None:
        _need(pos_emb, "pos_emb", C.dtype)
    if pos is not None:
        _need(pos, "pos", torch.int32)
    T = C.shape[0]
    if C.shape != (T, basis.k) or ids.shape != (T,) or tok_emb.shape[1] != basis.d:
        raise ValueError("shape mismatch")
    _check_rows(T, seq_len, basis.d, pos_emb, pos)
    if out is None:
        out = torch.empty(T, basis.d, dtype=C.dtype, device=C.device)
    _need(out, "out", C.dtype)
    _check_out(out, (T, basis.d))
    _check(_lib.sn_decompress_fwd(basis.handle, _dtype(C), _ptr(C), _ptr(ids), _ptr(pos), T,
                                  seq_len, _ptr(tok_emb), tok_emb.shape[0], _ptr(pos_emb),
                                  _ptr(out), _stream(stream)), "sn_decompress_fwd")
    return out


def sn_compress_bwd(basis, G, out=None, stream=None):
    """C_g = G U  (Sec. 4.4, Eq. grad_compress)."""
    _need(G, "G")
    T = G.shape[0]
    if G.shape != (T, basis.d):
        raise ValueError("shape mismatch")
    if out is None:
        out = torch.empty(T, basis.k, dtype=G.dtype, device=G.device)
    _need(out, "out", G.dtype)
    _check_out(out, (T, basis.k))
    _check(_lib.sn_compress_bwd(basis.handle, _dtype(G), _ptr(G), T, _ptr(out), _stream(stream)),
           "sn_compress_bwd")
    return out


def sn_decompress_bwd(basis, C, out=None, stream=None):
    """G = C_g U^T  (Sec. 4.4)."""
    _need(C, "C")
    T = C.shape[0]
    if C.shape != (T, basis.k):
        raise ValueError("shape mismatch")
    if out is None:
        out = torch.empty(T, basis.d, dtype=C.dtype, device=C.device)
    _need(out, "out", C.dtype)
    _check_out(out, (T, basis.d))
    _check(_lib.sn_decompress_bwd(basis.handle, _dtype(C), _ptr(C), T, _ptr(out),
                                  _stream(stream)), "sn_decompress_bwd")
    return out


def sn_project_weight_workspace(basis, dtype, cols):
    n = _SZ()
    code = SN_BF16 if dtype == torch.bfloat16 else SN_F32
    _check(_lib.sn_project_weight_workspace(basis.handle, code, cols, ctypes.byref(n)),
           "sn_project_weight_workspace")
    return int(n.value)


def sn_project_weight(basis, W, out=None, workspace=None, stream=None):
    """W' = U (U^T W) for torch-layout W [d, cols] (Sec. 4.3, Sec. 5, App. A).
    `out` may be W itself (in place).  W may be a row-strided view."""
    _need(W, "W", contiguous=False)
    if W.dim() != 2 or W.shape[0] != basis.d or W.stride(1) != 1:
        raise ValueError("W must be [d, cols] with unit column stride")
    rows, cols = W.shape
    ld = W.stride(0)
    if out is None:
        out = torch.empty_like(W)
    _need(out, "out", W.dtype, contiguous=False)
    if out.stride() != W.stride() or out.shape != W.shape:
        raise ValueError("out must have W's shape and strides")
    need = sn_project_weight_workspace(basis, W.dtype, cols)
    if workspace is None:
        workspace = torch.empty(max(need, 16), dtype=torch.uint8, device=W.device)
    _need(workspace, "workspace")
    _check(_lib.sn_project_weight(basis.handle, _dtype(W), _ptr(W), rows, cols, ld, _ptr(out),
                                  _ptr(workspace), workspace.numel() * workspace.element_size(),
                                  _stream(stream)), "sn_project_weight")
    return out


def sn_project_weight_noalloc(basis, W, out, stream=None):
    """W' = U (U^T W) like sn_project_weight, for callers that cannot allocate
    device memory: the library's fixed 32 MiB device scratch array is used
    instead of a workspace, and the caller provides `out` (may be W).  bf16
    only.  Calls that overlap on the GPU share the scratch and race."""
    _need(W, "W", torch.bfloat16, contiguous=False)
    _need(out, "out", torch.bfloat16, contiguous=False)
    if W.dim() != 2 or W.shape[0] != basis.d or W.stride(1) != 1:
        raise ValueError("W must be [d, cols] with unit column stride")
    if out.stride() != W.stride() or out.shape != W.shape or out.dtype != W.dtype:
        raise ValueError("out must have W's shape, strides and dtype")
    rows, cols = W.shape
    _check(_lib.sn_project_weight_noalloc(basis.handle, SN_BF16, _ptr(W), rows, cols,
                                          W.stride(0), _ptr(out), _stream(stream)),
           "sn_project_weight_noalloc")
    return out


def sn_wire_bytes(basis, dtype, T):
    n = _SZ()
    code = SN_BF16 if dtype == torch.bfloat16 else SN_F32
    _check(_lib.sn_wire_bytes(basis.handle, code, T, ctypes.byref(n)), "sn_wire_bytes")
    return int(n.value)


def sn_wire_send(src_device, dst_host, stream=None):
    """Device tensor -> (pinned) host tensor of the same byte size."""
    n = src_device.numel() * src_device.element_size()
    if not src_device.is_cuda:
        raise ValueError("source must be a CUDA tensor")
    if dst_host.numel() * dst_host.element_size() < n or dst_host.is_cuda:
        raise ValueError("destination must be host memory of at least %d bytes" % n)
    _check(_lib.sn_wire_send(_ptr(src_device), _ptr(dst_host), n, _stream(stream)),
           "sn_wire_send")
    return dst_host


def sn_wire_recv(src_host, dst_device, stream=None):
    """(Pinned) host tensor -> device tensor of the same byte size."""
    n = src_host.numel() * src_host.element_size()
    if src_host.is_cuda:
        raise ValueError("source must be host memory")
    if dst_device.numel() * dst_device.element_size() < n or not dst_device.is_cuda:
        raise ValueError("destination must be device memory of at least %d bytes" % n)
    _check(_lib.sn_wire_recv(_ptr(src_host), _ptr(dst_device), n, _stream(stream)),
           "sn_wire_recv")
    return dst_device


def sn_check_errors(basis, stream=None):
    """Synchronise the stream; raise SNError if a bad id or a timeout was recorded."""
    _check(_lib.sn_check_errors(basis.handle, _stream(stream)), "sn_check_errors")


def sn_selftest_wait_timeout(basis, stream=None):
    """Launch the bounded-wait self-test: one CTA waits on a barrier nothing
    completes, gives up after the library's wait limit (2 s) and records
    SN_ERR_TIMEOUT for the next sn_check_errors."""
    _check(_lib.sn_selftest_wait_timeout(basis.handle, _stream(stream)),
           "sn_selftest_wait_timeout")


def sn_launch_count():
    return int(_lib.sn_launch_count())


def sn_status_string(status):
    return _lib.sn_status_string(status).decode()
