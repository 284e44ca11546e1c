"""Helpers shared by the GPU parity tests: host <-> device transfers of exact
bytes, guard-banded output buffers and the error metrics of the parity bar."""
import os

import numpy as np
import torch

from paper_2506_01260_gb300 import workloads as W

#: max relative Frobenius error against the oracle's fp64 value
TOL = {"bf16": 1e-2, "f32": 1e-5}
#: max relative error of any one row (a token's vector, or a row of a weight)
#: against the oracle: one RNE rounding of every element (2^-9 relative in
#: bf16) plus the bf16 copy of U (at most 2^-9 relative per element of U, so
#: at most 2^-9 sqrt(k) relative on a row whose vector lies in the subspace,
#: 2.2e-2 at k = 128); fp32 rows carry only the fp32 accumulation error
ROW_TOL = {"bf16": 3e-2, "f32": 1e-4}

GUARD = 4096          # guard elements on each side of an output buffer
GUARD_BITS = 0x7FBF   # a NaN pattern no kernel writes


def dev(a, device="cuda"):
    """numpy (uint16 bf16 bits, float32, int32) -> device tensor with the same bytes."""
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint16:
        return torch.from_numpy(a.view(np.int16)).to(device).view(torch.bfloat16)
    return torch.from_numpy(a).to(device)


def host(t):
    """device tensor -> numpy with the same bytes (bf16 as uint16 bits)."""
    t = t.detach().contiguous().cpu()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view(np.uint16)
    return t.numpy()


def widen(a):
    a = np.asarray(a)
    if a.dtype == np.uint16:
        return W.bf16_bits_to_f32(a).astype(np.float64)
    return a.astype(np.float64)


def rel_fro(got, ref64):
    got64 = widen(got)
    den = float(np.linalg.norm(ref64))
    return float(np.linalg.norm(got64 - ref64)) / (den if den > 0 else 1.0)


def row_rel_max(got, ref64):
    """Largest ||got_r - ref_r|| / max(||ref_r||, ||ref||_rms / 4) over the rows
    r (the last axis is the row; ||ref||_rms is the root mean square row norm).
    The floor keeps a row that cancels to almost nothing (k = 1 outputs of
    inputs outside the subspace) from being judged against its own tiny norm;
    every row of ordinary size is judged against its own norm.  A row whose
    reference is exactly zero must come out exactly zero (it then counts 0,
    otherwise infinity)."""
    got64 = widen(got)
    ref64 = np.asarray(ref64, dtype=np.float64)
    if ref64.ndim == 1:
        got64, ref64 = got64.reshape(1, -1), ref64.reshape(1, -1)
    got64 = got64.reshape(-1, ref64.shape[-1])
    ref64 = ref64.reshape(-1, ref64.shape[-1])
    num = np.linalg.norm(got64 - ref64, axis=1)
    den = np.linalg.norm(ref64, axis=1)
    zero = den == 0
    if np.any(num[zero] > 0):
        return float("inf")
    if np.all(zero):
        return 0.0
    floor = 0.25 * float(np.sqrt(np.mean(den * den)))
    return float(np.max(num[~zero] / np.maximum(den[~zero], floor)))


def assert_parity(got, ref64, dtype, scale=1.0):
    """The parity bar: relative Frobenius error over the whole output within
    TOL and the relative error of every row within ROW_TOL (both scaled by
    `scale` where a comparison carries two roundings)."""
    fro = rel_fro(got, ref64)
    row = row_rel_max(got, ref64)
    log = os.environ.get("SN_PARITY_LOG")
    if log:                       # a record of the measured errors, one line per check
        with open(log, "a") as f:
            f.write("%s %s rel_fro %.3e row %.3e\n" % (
                os.environ.get("PYTEST_CURRENT_TEST", "?").split(" ")[0], dtype, fro, row))
    assert fro <= scale * TOL[dtype] and row <= scale * ROW_TOL[dtype], (
        "rel_fro %.3e (bar %.1e), worst row %.3e (bar %.1e)"
        % (fro, scale * TOL[dtype], row, scale * ROW_TOL[dtype]))
    return fro, row


def guarded(shape, dtype, device="cuda"):
    """An output tensor with GUARD sentinel elements before and after it."""
    n = int(np.prod(shape))
    full = torch.empty(n + 2 * GUARD, dtype=dtype, device=device)
    if dtype == torch.bfloat16:
        full.view(torch.int16).fill_(GUARD_BITS)
    else:
        full.view(torch.int32).fill_(0x7FBFFFFF)
    view = full[GUARD:GUARD + n].view(*shape)
    return full, view


def guards_intact(full):
    g = torch.cat([full[:GUARD], full[-GUARD:]])
    if g.dtype == torch.bfloat16:
        return bool((g.view(torch.int16) == GUARD_BITS).all())
    return bool((g.view(torch.int32) == 0x7FBFFFFF).all())


def dtname(t):
    return "bf16" if t.dtype == torch.bfloat16 else "f32"
