"""Round trips of the lossy comparators (Sec. 8, comparison against lossy
compressions) through the library, for measuring their reconstruction error
against the subspace codec at about the same wire size.

Each function takes a bf16 batch X [T, d] on the GPU and returns the restored
batch and the bytes the method would send.  Top-k and sign quantization are
kernels of the library; the low-rank comparator is a randomized rank-r
factorisation X ~ Q B of the whole batch (sketch X Om with a Gaussian Om,
power iterations, orthonormal Q of the sketch, B^T = X^T Q), composed of the
library's contraction, accumulation and expansion calls.  The [T, r] sketch is
orthonormalised by the library too: the Grassmann step's retraction is
CholeskyQR2 of U - eta * (step), so with eta = 0 it returns the orthonormal
factor Q of its input (diag(R) > 0); it sends Q and B, (T + d) r values.
"""
import math

import torch

from . import sn


def topk_roundtrip(X, kk):
    vals, cols = sn.sn_topk_compress(X, kk)
    return sn.sn_topk_restore(vals, cols, X.shape[1]), X.shape[0] * kk * 4


def sign_roundtrip(X):
    bits, scale = sn.sn_sign_compress(X)
    T, d = X.shape
    return sn.sn_sign_restore(bits, scale, d), T * ((d + 7) // 8) + 4 * T


def quant_roundtrip(X, fmt):
    """Row-scaled 8-bit round trip ("int8" or "e4m3"): T * d code bytes and one
    fp32 scale per row."""
    codes, scale = sn.sn_quant_compress(X, fmt)
    T, d = X.shape
    return sn.sn_quant_restore(codes, scale, fmt), T * d + 4 * T


def lowrank_roundtrip(X, r, power_iters=1, seed=0):
    T, d = X.shape
    gen = torch.Generator(device=X.device).manual_seed(seed)
    om = (torch.randn(d, r, generator=gen, device=X.device) / math.sqrt(d)).contiguous()
    b_om = sn.Basis(om)

    def orth(Y):
        # the Grassmann step's CholeskyQR2 retraction of Y itself (no step: eta = 0)
        Yf = Y.float().contiguous()
        b_y = sn.Basis(Yf)
        Q = sn.sn_grassmann_step(b_y, torch.zeros_like(Yf), 1, 0.0)
        b_y.destroy()
        return Q.to(torch.bfloat16).contiguous()

    def xt_times(Q):                                   # X^T Q, fp32 [d, r]
        M = torch.zeros(d, r, dtype=torch.float32, device=X.device)
        sn.sn_grassmann_accumulate(b_om, X, Q, M)
        return M

    Y = sn.sn_compress_bwd(b_om, X)                    # X Om
    for _ in range(power_iters):
        b_m = sn.Basis(xt_times(orth(Y)))
        Y = sn.sn_compress_bwd(b_m, X)                 # X X^T Q
        b_m.destroy()
    Q = orth(Y)
    b_b = sn.Basis(xt_times(Q))                        # B^T = X^T Q
    Xh = sn.sn_decompress_bwd(b_b, Q)                  # Q B
    b_b.destroy()
    b_om.destroy()
    return Xh, 2 * (T + d) * r
