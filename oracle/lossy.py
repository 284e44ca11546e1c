"""fp64 oracle of the lossy comparators of Sec. 8 ("Comparison against lossy
compressions": Top-k, quantization and low-rank projection, at the wire size
of the subspace codec).

TEST INFRASTRUCTURE ONLY.  Only the tests may import this module; it shares no
code with the CUDA library.  Plain numpy; the exact SVD of numpy serves as the
low-rank comparator's ideal.

Definitions (rows are tokens, X is [T, d]):
  top-k      keep, in every row, the kk entries of largest magnitude (ties
             broken towards the lower column index), zero the rest; wire =
             kk values + kk column indices per row
  sign       one bit per entry (1 for a negative value) and one fp32 scale per
             row, the mean magnitude of the row; restore = scale * (+-1)
  low rank   the best rank-r approximation of the whole batch (truncated SVD);
             wire = (T + d) * r values
Selections are made on bf16 magnitudes (the bits the GPU sees), so the kept
columns are defined exactly.
"""
import numpy as np


def bf16_magnitude_bits(bits):
    """|x| as the 15 low bits of the bf16 pattern (monotone in |x| for finite x)."""
    return np.asarray(bits, np.uint16) & np.uint16(0x7FFF)


def topk_columns(bits, kk):
    """Column indices kept in each row, ascending: the kk largest |x|, ties
    towards the lower index."""
    mag = bf16_magnitude_bits(bits).astype(np.int64)
    T, d = mag.shape
    out = np.empty((T, kk), np.int64)
    for t in range(T):
        order = sorted(range(d), key=lambda c: (-mag[t, c], c))   # largest first, then lower index
        out[t] = sorted(order[:kk])
    return out


def topk_restore(values, cols, d):
    """Zero rows with the kept values scattered back to their columns."""
    T = values.shape[0]
    X = np.zeros((T, d))
    for t in range(T):
        X[t, cols[t]] = values[t]
    return X


def sign_compress(X):
    """(bits, scale): bits[t, c] = 1 where X[t, c] < 0; scale[t] = mean |X[t, :]|."""
    X = np.asarray(X, np.float64)
    return (X < 0).astype(np.uint8), np.abs(X).mean(axis=1)


def sign_restore(bits, scale):
    return np.where(np.asarray(bits) == 1, -1.0, 1.0) * np.asarray(scale, np.float64)[:, None]


def lowrank(X, r):
    """Best rank-r approximation of X (truncated SVD)."""
    Uu, s, Vt = np.linalg.svd(np.asarray(X, np.float64), full_matrices=False)
    return (Uu[:, :r] * s[:r]) @ Vt[:r]


def wire_bytes(kind, T, d, k=None, kk=None, r=None):
    """Bytes each method sends for a [T, d] bf16 batch."""
    if kind == "subspace":
        return 2 * T * k
    if kind == "topk":
        return T * kk * (2 + 2)                  # bf16 value + 16-bit column index
    if kind == "sign":
        return T * ((d + 7) // 8) + 4 * T
    if kind == "lowrank":
        return 2 * (T + d) * r
    raise ValueError(kind)
