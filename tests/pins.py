"""Pins of the fp64 oracle to facts fixed outside it.

Each pin takes an `oracle.Oracle` and raises AssertionError when the oracle
disagrees with something the paper or plain mathematics fixes:
  * the hand-worked example in tests/golden/worked_d4.txt,
  * closed forms (X = E + Z U^T + N with N orthogonal to U gives C = Z and a
    reconstruction error of exactly -N; Sec. 4.3, Sec. 4.3.1),
  * bases that reduce the contraction to a library routine (columns of the
    identity: slicing; Walsh-Hadamard columns: a butterfly transform),
  * pure gathers (C = 0 reconstructs T_fixed[ids] and P[pos] bit-exactly),
  * U^T U = I consequences (idempotence, P^2 = P, P U = U; App. A),
  * the gradient identity of App. A: (G P) W' = G W' when W' = P W,
  * numpy.matmul at tiny sizes, and torch's fp32 -> bf16 rounding.
The same list is run against deliberately broken builds of the oracle
(tests/test_oracle_mutants.py) to show each plausible mistake is caught.
"""
import os

import numpy as np

from paper_2506_01260_gb300 import workloads as wlmod

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")

BF16, F32, F64 = 0, 1, 2


def bf(x64):
    return wlmod.to_bf16(x64)


def widen(bits):
    return wlmod.bf16_bits_to_f32(bits).astype(np.float64)


def read_golden(name):
    vals = {}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            key, rest = line.split(":", 1)
            vals[key.strip()] = np.array([float(v) for v in rest.split()])
    return vals


def _small_planted(rng, T=37, d=16, k=3, vocab=11, n=5, noise=True):
    """fp64 inputs with X = E + Z U^T (+ N, N orthogonal to U)."""
    U = wlmod.orthonormal_basis(d, k, rng)
    tok = 0.02 * rng.standard_normal((vocab, d))
    pe = 0.02 * rng.standard_normal((n, d))
    ids = rng.integers(0, vocab, T).astype(np.int32)
    pos = (np.arange(T) % n)
    Z = rng.standard_normal((T, k))
    N = np.zeros((T, d))
    if noise:
        N0 = rng.standard_normal((T, d))
        N = 0.3 * (N0 - (N0 @ U) @ U.T)
    X = tok[ids] + pe[pos] + Z @ U.T + N
    return dict(U=U, tok=tok, pe=pe, ids=ids, Z=Z, N=N, X=X, n=n)


# ---- rounding ----------------------------------------------------------------

def pin_round_bf16_vs_torch(orc):
    """fp32-representable values round exactly as torch's fp32 -> bf16 (RNE)."""
    import torch
    rng = np.random.default_rng(1)
    f = np.concatenate([
        rng.standard_normal(20000).astype(np.float32) * np.float32(3.0),
        (rng.standard_normal(2000) * 1e-38).astype(np.float32),
        # exact ties: 8 significant bits + one half-ulp bit
        np.array([1 + 2**-8, 1 + 3 * 2**-8, -(1 + 2**-8), 2**-126 * (1 + 2**-8),
                  65504.0, 3.0e38, -0.0, 0.0], np.float32),
    ])
    ref = torch.from_numpy(f).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    got = orc.round_bf16(f.astype(np.float64))
    assert np.array_equal(got, ref), "bf16 rounding differs from torch RNE"
    # Direct rounding from fp64: 1 + 2^-8 + 2^-40 is above the tie, so it rounds
    # up (a detour through fp32 would create a tie and round down to 1.0).
    assert orc.round_bf16(np.array([1 + 2**-8 + 2**-40]))[0] == 0x3F81
    assert orc.round_bf16(np.array([3.5e38]))[0] == 0x7F80     # overflow -> inf


# ---- hand-worked example -----------------------------------------------------

def pin_worked_example(orc):
    """tests/golden/worked_d4.txt: exact in every dtype."""
    g = read_golden("worked_d4.txt")
    d, k = 4, 2
    U = g["U"].reshape(d, k)
    seq = int(g["seq_len"][0])
    ids = g["ids"].astype(np.int32)
    for dt, conv, back in ((F64, lambda a: a, lambda a: a),
                           (F32, lambda a: a.astype(np.float32), lambda a: a.astype(np.float64)),
                           (BF16, bf, widen)):
        tok = conv(g["tok_emb"].reshape(3, d))
        pe = conv(g["pos_emb"].reshape(seq, d))
        X = conv(g["X"].reshape(3, d))
        for Uin in (U, U.astype(np.float32)):
            C, _, st = orc.compress_fwd(X, ids, tok, Uin, seq, pos_emb=pe)
            assert st == 0 and np.array_equal(back(C), g["C"].reshape(3, k)), (dt, back(C))
            Xr, _, st = orc.decompress_fwd(conv(g["C"].reshape(3, k)), ids, tok, Uin, seq,
                                           pos_emb=pe)
            assert st == 0 and np.array_equal(back(Xr), g["X_rec"].reshape(3, d)), back(Xr)
            Cg, _, _ = orc.compress_bwd(conv(g["G"].reshape(1, d)), Uin)
            assert np.array_equal(back(Cg), g["Cg"].reshape(1, k))
            Gr, _, _ = orc.decompress_bwd(conv(g["Cg"].reshape(1, k)), Uin)
            assert np.array_equal(back(Gr), g["G_rec"].reshape(1, d))
            Wp, _, _ = orc.project_weight(conv(g["W"].reshape(d, 2)), Uin)
            assert np.array_equal(back(Wp), g["W_proj"].reshape(d, 2)), back(Wp)


# ---- closed forms ------------------------------------------------------------

def pin_closed_form_fwd(orc):
    """X = E + Z U^T + N, N orthogonal to U: C = Z and X_rec = X - N (fp64)."""
    rng = np.random.default_rng(2)
    p = _small_planted(rng)
    C, C64, st = orc.compress_fwd(p["X"], p["ids"], p["tok"], p["U"], p["n"], pos_emb=p["pe"])
    assert st == 0
    assert np.max(np.abs(C64 - p["Z"])) < 1e-12
    Xr, _, st = orc.decompress_fwd(p["Z"], p["ids"], p["tok"], p["U"], p["n"],
                                   pos_emb=p["pe"])
    assert st == 0
    assert np.max(np.abs((p["X"] - Xr) - p["N"])) < 1e-12


def pin_closed_form_explicit_positions(orc):
    """An explicit position array equal to t mod n gives the same result; a
    permuted one matches inputs built with the permuted positions."""
    rng = np.random.default_rng(3)
    p = _small_planted(rng, noise=False)
    T = p["X"].shape[0]
    pos = (np.arange(T) % p["n"]).astype(np.int32)
    C1, _, _ = orc.compress_fwd(p["X"], p["ids"], p["tok"], p["U"], p["n"], pos_emb=p["pe"])
    C2, _, _ = orc.compress_fwd(p["X"], p["ids"], p["tok"], p["U"], p["n"], pos_emb=p["pe"],
                                pos=pos)
    assert np.array_equal(C1, C2)
    pos2 = rng.integers(0, p["n"], T).astype(np.int32)
    X2 = p["tok"][p["ids"]] + p["pe"][pos2] + p["Z"] @ p["U"].T
    _, C64, st = orc.compress_fwd(X2, p["ids"], p["tok"], p["U"], p["n"], pos_emb=p["pe"],
                                  pos=pos2)
    assert st == 0 and np.max(np.abs(C64 - p["Z"])) < 1e-12


def pin_closed_form_bwd(orc):
    """G = Z U^T + N: C_g = Z and the recovered gradient is G - N (Sec. 4.4)."""
    rng = np.random.default_rng(4)
    p = _small_planted(rng)
    G = p["Z"] @ p["U"].T + p["N"]
    _, C64, _ = orc.compress_bwd(G, p["U"])
    assert np.max(np.abs(C64 - p["Z"])) < 1e-12
    _, G64, _ = orc.decompress_bwd(p["Z"], p["U"])
    assert np.max(np.abs(G64 - (G - p["N"]))) < 1e-12


def pin_no_positional_table(orc):
    """With no positional table nothing positional is subtracted or added."""
    rng = np.random.default_rng(5)
    p = _small_planted(rng, noise=False)
    X = p["tok"][p["ids"]] + p["Z"] @ p["U"].T
    _, C64, st = orc.compress_fwd(X, p["ids"], p["tok"], p["U"], p["n"])
    assert st == 0 and np.max(np.abs(C64 - p["Z"])) < 1e-12
    _, X64, _ = orc.decompress_fwd(p["Z"], p["ids"], p["tok"], p["U"], p["n"])
    assert np.max(np.abs(X64 - X)) < 1e-12


# ---- bases that reduce to library routines ----------------------------------

def pin_identity_columns(orc):
    """U = columns `cols` of I_d: C = (X - E)[:, cols] (planted, slicing), and the
    reconstruction scatters C into those columns (bf16 in/out, bit-exact)."""
    rng = np.random.default_rng(6)
    T, d, vocab, n = 40, 24, 9, 7
    cols = np.array([17, 3, 11, 0, 23])
    U = np.eye(d)[:, cols]
    tok = bf(0.02 * rng.standard_normal((vocab, d)))
    pe = bf(0.02 * rng.standard_normal((n, d)))
    ids = rng.integers(0, vocab, T).astype(np.int32)
    pos = np.arange(T) % n
    # planted residual S with few significant bits so E + S is exact in bf16
    S = np.round(rng.standard_normal((T, d)) * 8) / 8 + 0.0   # no negative zeros
    tok0 = np.zeros_like(tok)
    pe0 = np.zeros_like(pe)
    X = bf(S)
    C, _, _ = orc.compress_fwd(X, ids, tok0, U.astype(np.float32), n, pos_emb=pe0)
    assert np.array_equal(C, bf(S[:, cols]))
    # nonzero tables on a coarse grid (multiples of 1/32, |E| <= 1/4) and S on
    # multiples of 1/4 with |S| <= 1.75: E + S is exact in bf16, so is C
    tokc = bf(np.clip(np.round(rng.standard_normal((vocab, d)) * 2), -4, 4) / 32 + 0.0)
    pec = bf(np.clip(np.round(rng.standard_normal((n, d)) * 2), -4, 4) / 32 + 0.0)
    Sc = np.clip(np.round(rng.standard_normal((T, d)) * 2), -7, 7) / 4 + 0.0
    X2 = bf(widen(tokc)[ids] + widen(pec)[pos] + Sc)
    C2, _, _ = orc.compress_fwd(X2, ids, tokc, U.astype(np.float32), n, pos_emb=pec)
    assert np.array_equal(C2, bf(Sc[:, cols]))
    # reconstruction with zero tables is a scatter into `cols`
    Cin = bf(rng.standard_normal((T, len(cols))))
    Xr, _, _ = orc.decompress_fwd(Cin, ids, tok0, U.astype(np.float32), n, pos_emb=pe0)
    expect = np.zeros((T, d), np.uint16)
    expect[:, cols] = Cin
    assert np.array_equal(Xr, expect)


def _fwht(a):
    """Unnormalised fast Walsh-Hadamard transform along the last axis."""
    a = a.copy()
    h = 1
    n = a.shape[-1]
    while h < n:
        a = a.reshape(a.shape[:-1] + (n // (2 * h), 2, h))
        x, y = a[..., 0, :].copy(), a[..., 1, :].copy()
        a[..., 0, :], a[..., 1, :] = x + y, x - y
        a = a.reshape(a.shape[:-3] + (n,))
        h *= 2
    return a


def pin_hadamard_basis(orc):
    """U = columns of H_d / sqrt(d) (Sylvester order): C = FWHT(X - E)[:, cols]/sqrt(d)."""
    rng = np.random.default_rng(7)
    d, T, vocab, n = 64, 50, 13, 8
    cols = np.array([0, 5, 63, 32, 17, 9])
    H = np.array([[1.0]])
    while H.shape[0] < d:
        H = np.block([[H, H], [H, -H]])
    U = H[:, cols] / np.sqrt(d)
    tok = 0.02 * rng.standard_normal((vocab, d))
    pe = 0.02 * rng.standard_normal((n, d))
    ids = rng.integers(0, vocab, T).astype(np.int32)
    S = rng.standard_normal((T, d))
    X = tok[ids] + pe[np.arange(T) % n] + S
    _, C64, _ = orc.compress_fwd(X, ids, tok, U, n, pos_emb=pe)
    expect = _fwht(S)[:, cols] / np.sqrt(d)
    assert np.max(np.abs(C64 - expect)) < 1e-11
    # backward path with the same basis
    _, Cg, _ = orc.compress_bwd(S, U)
    assert np.max(np.abs(Cg - expect)) < 1e-11


def pin_gather_exact(orc):
    """C = 0 reconstructs the gathered embeddings: T_fixed[ids] alone, P[pos]
    alone (zero token table), bit-exact in bf16."""
    rng = np.random.default_rng(8)
    T, d, k, vocab, n = 45, 32, 4, 17, 6
    U = wlmod.orthonormal_basis(d, k, rng).astype(np.float32)
    tok = bf(0.02 * rng.standard_normal((vocab, d)))
    pe = bf(0.02 * rng.standard_normal((n, d)))
    ids = rng.integers(0, vocab, T).astype(np.int32)
    C0 = np.zeros((T, k), np.uint16)
    Xr, _, _ = orc.decompress_fwd(C0, ids, tok, U, n)
    assert np.array_equal(Xr, tok[ids])
    Xr, _, _ = orc.decompress_fwd(C0, ids, np.zeros_like(tok), U, n, pos_emb=pe)
    assert np.array_equal(Xr, np.tile(pe, (T // n + 1, 1))[:T])
    pos = rng.integers(0, n, T).astype(np.int32)
    Xr, _, _ = orc.decompress_fwd(C0, ids, np.zeros_like(tok), U, n, pos_emb=pe, pos=pos)
    assert np.array_equal(Xr, pe[pos])


# ---- orthonormality consequences --------------------------------------------

def pin_idempotence(orc):
    """U^T U = I: compress(decompress(C)) = C; decompress∘compress is idempotent."""
    rng = np.random.default_rng(9)
    p = _small_planted(rng)
    C = rng.standard_normal(p["Z"].shape)
    _, X64, _ = orc.decompress_fwd(C, p["ids"], p["tok"], p["U"], p["n"], pos_emb=p["pe"])
    _, C64, _ = orc.compress_fwd(X64, p["ids"], p["tok"], p["U"], p["n"], pos_emb=p["pe"])
    assert np.max(np.abs(C64 - C)) < 1e-12
    X = p["X"] + rng.standard_normal(p["X"].shape)
    _, C1, _ = orc.compress_fwd(X, p["ids"], p["tok"], p["U"], p["n"], pos_emb=p["pe"])
    _, X1, _ = orc.decompress_fwd(C1, p["ids"], p["tok"], p["U"], p["n"], pos_emb=p["pe"])
    _, C2, _ = orc.compress_fwd(X1, p["ids"], p["tok"], p["U"], p["n"], pos_emb=p["pe"])
    _, X2, _ = orc.decompress_fwd(C2, p["ids"], p["tok"], p["U"], p["n"], pos_emb=p["pe"])
    assert np.max(np.abs(X2 - X1)) < 1e-12


def pin_projection_properties(orc):
    """W' = U(U^T W): P^2 = P, P U = U, P N = 0 for N orthogonal to U, and
    (G P) W' = G W' (App. A: projecting the incoming gradient is lossless)."""
    rng = np.random.default_rng(10)
    d, k, m = 24, 5, 19
    U = wlmod.orthonormal_basis(d, k, rng)
    W = rng.standard_normal((d, m))
    _, W1, _ = orc.project_weight(W, U)
    _, W2, _ = orc.project_weight(W1, U)
    assert np.max(np.abs(W2 - W1)) < 1e-12
    B = rng.standard_normal((k, m))
    _, Win, _ = orc.project_weight(U @ B, U)
    assert np.max(np.abs(Win - U @ B)) < 1e-12
    N0 = rng.standard_normal((d, m))
    N = N0 - U @ (U.T @ N0)
    _, Wn, _ = orc.project_weight(N, U)
    assert np.max(np.abs(Wn)) < 1e-12
    # ||W||^2 = ||W'||^2 + ||W - W'||^2 (orthogonal projection)
    assert abs(np.sum(W * W) - np.sum(W1 * W1) - np.sum((W - W1) ** 2)) < 1e-9
    G = rng.standard_normal((7, d))
    _, Cg, _ = orc.compress_bwd(G, U)
    _, Gp, _ = orc.decompress_bwd(Cg, U)
    assert np.max(np.abs(Gp @ W1 - G @ W1)) < 1e-11
    # leading dimension: a sub-block of a wider matrix projects the same way
    Wwide = rng.standard_normal((d, m + 6))
    sub = np.ascontiguousarray(Wwide[:, :m])
    _, Ws, _ = orc.project_weight(sub, U)
    out = np.empty((d, m + 6))
    st = orc.lib.sno_project_weight(F64, Wwide.ctypes.data, d, m, m + 6, F64, U.ctypes.data,
                                    d, k, out.ctypes.data, None)
    assert st == 0 and np.max(np.abs(out[:, :m] - Ws)) < 1e-12


# ---- numpy brute force at tiny sizes -----------------------------------------

def pin_numpy_matmul_tiny(orc):
    """d <= 16, k <= 4: every output equals numpy's fp64 matmul of the same
    definition (Sec. 4.3.1 / Sec. 4.4 / Sec. 5)."""
    rng = np.random.default_rng(11)
    for (T, d, k, vocab, n) in ((1, 1, 1, 1, 1), (9, 8, 3, 5, 4), (13, 16, 4, 7, 3)):
        U = rng.standard_normal((d, k))          # any matrix works for the GEMM identity
        X = rng.standard_normal((T, d))
        tok = rng.standard_normal((vocab, d))
        pe = rng.standard_normal((n, d))
        ids = rng.integers(0, vocab, T).astype(np.int32)
        pos = rng.integers(0, n, T).astype(np.int32)
        _, C, _ = orc.compress_fwd(X, ids, tok, U, n, pos_emb=pe, pos=pos)
        assert np.allclose(C, np.matmul(X - tok[ids] - pe[pos], U), rtol=0, atol=1e-12)
        Cin = rng.standard_normal((T, k))
        _, Xr, _ = orc.decompress_fwd(Cin, ids, tok, U, n, pos_emb=pe, pos=pos)
        assert np.allclose(Xr, np.matmul(Cin, U.T) + tok[ids] + pe[pos], rtol=0, atol=1e-12)
        _, Cg, _ = orc.compress_bwd(X, U)
        assert np.allclose(Cg, np.matmul(X, U), rtol=0, atol=1e-12)
        _, Gr, _ = orc.decompress_bwd(Cin, U)
        assert np.allclose(Gr, np.matmul(Cin, U.T), rtol=0, atol=1e-12)
        W = rng.standard_normal((d, 3))
        _, Wp, _ = orc.project_weight(W, U)
        assert np.allclose(Wp, np.matmul(U, np.matmul(U.T, W)), rtol=0, atol=1e-11)


# ---- invalid ids and wire size -----------------------------------------------

def pin_bad_ids(orc):
    """An id outside [0, vocab) or a position outside [0, n) zeroes that row and
    reports BAD_ID; every other row is computed."""
    rng = np.random.default_rng(12)
    p = _small_planted(rng, T=10, noise=False)
    vocab = p["tok"].shape[0]
    ids = p["ids"].copy()
    ids[3] = vocab
    ids[7] = -1
    C, C64, st = orc.compress_fwd(p["X"], ids, p["tok"], p["U"], p["n"], pos_emb=p["pe"])
    assert st == 4
    assert np.all(C64[[3, 7]] == 0)
    good = [i for i in range(10) if i not in (3, 7)]
    assert np.max(np.abs(C64[good] - p["Z"][good])) < 1e-12
    _, X64, st = orc.decompress_fwd(p["Z"], ids, p["tok"], p["U"], p["n"], pos_emb=p["pe"])
    assert st == 4 and np.all(X64[[3, 7]] == 0)
    pos = (np.arange(10) % p["n"]).astype(np.int32)
    pos[5] = p["n"]
    _, C64, st = orc.compress_fwd(p["X"], p["ids"], p["tok"], p["U"], p["n"],
                                  pos_emb=p["pe"], pos=pos)
    assert st == 4 and np.all(C64[5] == 0)
    # without a positional table positions are not consulted
    _, _, st = orc.compress_fwd(p["X"], p["ids"], p["tok"], p["U"], p["n"], pos=pos)
    assert st == 0


def pin_wire_bytes(orc):
    """The wire carries T*k elements: k/d of the uncompressed activation (Sec. 4.3)."""
    for dt, s in ((BF16, 2), (F32, 4), (F64, 8)):
        for (T, d, k) in ((256, 256, 8), (8192, 2048, 20), (65536, 8192, 82)):
            wb = orc.wire_bytes(dt, T, k)
            assert wb == T * k * s
            assert wb * d == T * d * s * k     # = (k/d) |X|
    assert orc.wire_bytes(BF16, 4096, 40) * 100 < 4096 * 4096 * 2 * 1.03  # k=40, d=4096: ~100x


PINS = [pin_round_bf16_vs_torch, pin_worked_example, pin_closed_form_fwd,
        pin_closed_form_explicit_positions, pin_closed_form_bwd, pin_no_positional_table,
        pin_identity_columns, pin_hadamard_basis, pin_gather_exact, pin_idempotence,
        pin_projection_properties, pin_numpy_matmul_tiny, pin_bad_ids, pin_wire_bytes]
