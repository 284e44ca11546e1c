"""Helpers shared by the GPU parity tests: host <-> device transfers of exact
bytes, guard-banded output buffers and the error metrics of the parity bar."""
import numpy as np
import torch

from paper_2506_01260_gb300 import workloads as W

#: max relative Frobenius error against the oracle's fp64 value
TOL = {"bf16": 1e-2, "f32": 1e-5}

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
