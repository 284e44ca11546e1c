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
  8-bit      one 8-bit code per entry and one fp32 scale per row: a = max |x|,
             scale = a / qmax, code = Q(x * r) with r = qmax / a (0 for a zero
             row), Q = round half to even and clamp to +-127 (int8, qmax =
             127) or round to the nearest e4m3 value, ties to even, saturating
             at +-448 (fp8 e4m3, qmax = 448); restore = decode(code) * scale.
             The code is an integer decided by floating point, so it is taken
             in fp32 like the kernel: r, x * r and scale are fp32 operations
             and restore rounds the fp32 product once to bf16.
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


QMAX = {"int8": 127.0, "e4m3": 448.0}


def bf16_bits_to_f32(bits):
    """bf16 bit patterns -> float32 (exact)."""
    return (np.asarray(bits, np.uint16).astype(np.uint32) << 16).view(np.float32)


def f32_to_bf16_bits(x):
    """float32 -> bf16 bit patterns, round to nearest even (finite inputs)."""
    u = np.ascontiguousarray(x, np.float32).view(np.uint32).astype(np.uint64)
    return ((u + 0x7FFF + ((u >> 16) & 1)) >> 16).astype(np.uint16)


def e4m3_decode(codes):
    """fp8 e4m3 codes -> float64: sign, 4 exponent bits (bias 7), 3 mantissa
    bits; exponent field 0 holds the subnormals m * 2^-9; S.1111.111 is NaN and
    there are no infinities (largest finite value 448 = 1.75 * 2^8)."""
    c = np.asarray(codes, np.uint8).astype(np.int64)
    E, M = (c >> 3) & 15, c & 7
    mag = np.where(E == 0, M * 2.0 ** -9, (8 + M) * np.exp2(E - 10.0))
    mag = np.where((E == 15) & (M == 7), np.nan, mag)
    return np.where(c & 0x80, -mag, mag)


def e4m3_encode(p):
    """float32 values -> e4m3 codes: the nearest e4m3 value, ties to the even
    mantissa, magnitudes at or past 448 saturated to 448; the sign bit is kept
    (a negative value that rounds to zero gives -0)."""
    p = np.asarray(p, np.float32).astype(np.float64)
    neg = np.signbit(p)
    v = np.abs(p)
    e = np.frexp(np.where(v > 0, v, 1.0))[1] - 1           # floor(log2 v) for v > 0
    e = np.maximum(e, -6)                                   # below 2^-6: the subnormal grid
    n = np.rint(v / np.exp2(e - 3.0))                       # multiples of the exponent's quantum
    carry = n == 16
    e, n = np.where(carry, e + 1, e), np.where(carry, 8, n)
    sub = n < 8                                             # only when e == -6
    code = np.where(sub, n, (e + 7) * 8 + (n - 8))
    code = np.where(v >= 448.0, 0x7E, code)
    code = np.where(v == 0, 0, code)
    return (code.astype(np.int64) | np.where(neg, 0x80, 0)).astype(np.uint8)


def quant_compress(bits, fmt):
    """(codes uint8 [T, d], scale float32 [T]) of bf16 bit patterns [T, d]."""
    x = bf16_bits_to_f32(bits)
    qmax = np.float32(QMAX[fmt])
    a = np.abs(x).max(axis=1)
    scale = (a / qmax).astype(np.float32)
    r = np.where(a > 0, qmax / np.where(a > 0, a, np.float32(1)), np.float32(0)).astype(np.float32)
    p = (x * r[:, None]).astype(np.float32)
    if fmt == "int8":
        codes = np.clip(np.rint(p), -127, 127).astype(np.int8).view(np.uint8)
    else:
        codes = e4m3_encode(p)
    return codes, scale


def quant_decode(codes, fmt):
    if fmt == "int8":
        return np.asarray(codes, np.uint8).view(np.int8).astype(np.float64)
    return e4m3_decode(codes)


def quant_restore(codes, scale, fmt):
    """bf16 bit patterns of decode(code) * scale, the product taken in fp32."""
    q = quant_decode(codes, fmt).astype(np.float32)
    return f32_to_bf16_bits(q * np.asarray(scale, np.float32)[:, None])


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
    if kind in QMAX:
        return T * d + 4 * T
    raise ValueError(kind)
