"""Seeded synthetic workloads for the stage-boundary codec.

This module only synthesises inputs.  It holds none of the codec's arithmetic
(no compression, reconstruction or projection); the CUDA library and the CPU
oracle both consume the exact bytes produced here.

The paper trains Llama-style decoders on C4 / WikiText / OpenWebText /
BookCorpus (Sec. 8.1).  Those corpora and trained weights are not available, so
these seeded inputs stand in for them with the paper's shapes: d = 2048..8192,
context 1024..4096, k about 1% of d (k = 40 at d = 4096 gives the 100x wire
ratio of Sec. 8.1), token ids uniform or Zipf-distributed.

Recipe (fp64 draws, one rounding to fp32 and one round-to-nearest-even to bf16):
  U       = Q of QR(N(0,1)[d, k]) with diag(R) > 0, stored fp32  (Sec. 8.1: Gaussian init,
            Sec. 4.3: orthonormal columns)
  T_fixed, P (positional table) ~ N(0, 0.02^2)
  Z ~ N(0, 1) [T, k];  G ~ N(0, 1) [T, d];  W ~ N(0, 0.02^2)
  X = T_fixed[ids] + P[t mod n] + Z U^T + N, where N = s (I - U U^T) N0 is planted
      off-subspace noise (absolute scale s, or scaled to a fraction of ||X - E||^2).
"""
from dataclasses import dataclass, replace

import numpy as np

SEED_BASE = 20250601


@dataclass(frozen=True)
class Workload:
    name: str
    batch: int
    seq_len: int
    d: int
    k: int
    vocab: int
    seed: int
    ids: str = "uniform"        # "uniform" or "zipf1.1"
    off_scale: float = 0.0      # N = off_scale * (I - P) N0
    off_energy: float = 0.0     # or: ||N||^2 = off_energy * ||Z U^T + N||^2
    grad: bool = False          # also draw an activation gradient G

    @property
    def T(self):
        return self.batch * self.seq_len

    def with_tokens(self, batch, seq_len):
        return replace(self, batch=batch, seq_len=seq_len)


WORKLOADS = {
    # T = 2 x 128, d = 256, k = 8, vocab 1024; X exactly in E + span(U)
    "tiny": Workload("tiny", 2, 128, 256, 8, 1024, SEED_BASE + 0),
    # 1B-class: T = 8 x 1024, d = 2048, k = 20, vocab 32000, 1e-3 off-subspace noise
    "1b": Workload("1b", 8, 1024, 2048, 20, 32000, SEED_BASE + 1, off_scale=1e-3),
    # 8B-class: T = 4 x 4096, d = 4096, k = 41, vocab 128256, plus G ~ N(0, 1)
    "8b": Workload("8b", 4, 4096, 4096, 41, 128256, SEED_BASE + 2, off_scale=1e-3, grad=True),
    # large stream: T = 16 x 4096, d = 8192, k = 82, Zipf(1.1) ids, 5% off-subspace energy
    "large": Workload("large", 16, 4096, 8192, 82, 128256, SEED_BASE + 4, ids="zipf1.1",
                      off_energy=0.05, grad=True),
}

# weight projection: W_o [4096, 4096] and W_down [4096, 14336], U [4096, 41]
WEIGHT_SEED = SEED_BASE + 3
WEIGHT_SHAPES = {"W_o": (4096, 4096), "W_down": (4096, 14336)}
WEIGHT_D, WEIGHT_K = 4096, 41


# ---- encodings -------------------------------------------------------------

def f32_to_bf16_bits(a):
    """fp32 -> bf16 bit patterns, round-to-nearest-even (finite inputs)."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    bits = a.view(np.uint32).astype(np.uint64)
    bias = 0x7FFF + ((bits >> 16) & 1)
    return ((bits + bias) >> 16).astype(np.uint16)


def bf16_bits_to_f32(bits):
    bits = np.ascontiguousarray(bits, dtype=np.uint16)
    return (bits.astype(np.uint32) << 16).view(np.float32)


def to_bf16(a64):
    """fp64 draw -> fp32 -> bf16 bits (the input encoding used everywhere)."""
    return f32_to_bf16_bits(np.asarray(a64, dtype=np.float64).astype(np.float32))


# ---- draws -----------------------------------------------------------------

def orthonormal_basis(d, k, rng):
    """U = Q of QR(N(0,1)[d, k]) with diag(R) > 0 (unique), fp64."""
    A = rng.standard_normal((d, k))
    Q, R = np.linalg.qr(A)
    s = np.sign(np.diag(R))
    s[s == 0] = 1.0
    return Q * s


def zipf_ids(T, vocab, rng, a=1.1):
    """Truncated Zipf(a) over ranks 0..vocab-1 (P ~ (r+1)^-a), ranks mapped
    through a seeded permutation of the vocabulary."""
    p = (np.arange(vocab, dtype=np.float64) + 1.0) ** (-a)
    p /= p.sum()
    ranks = rng.choice(vocab, size=T, p=p)
    perm = rng.permutation(vocab)
    return perm[ranks].astype(np.int32)


def token_ids(wl, rng, T=None):
    T = wl.T if T is None else T
    if wl.ids == "uniform":
        return rng.integers(0, wl.vocab, size=T, dtype=np.int64).astype(np.int32)
    if wl.ids == "zipf1.1":
        return zipf_ids(T, wl.vocab, rng)
    raise ValueError(wl.ids)


def generate(wl, seed=None, T=None, dtype="bf16"):
    """All inputs of a workload as numpy arrays (host, exact bytes).

    Returns a dict: U64 (fp64 basis), U (fp32 basis as passed to the library),
    tok_emb / pos_emb / X (bf16 bits, or fp32 values when dtype == "f32"),
    ids (int32), Z (fp64 coefficients planted in X), and G when the workload
    has a gradient.  `T` overrides the token count (positions stay t mod n).
    Intended for sizes that fit comfortably in host memory.
    """
    rng = np.random.default_rng(wl.seed if seed is None else seed)
    T = wl.T if T is None else T
    d, k, n = wl.d, wl.k, wl.seq_len
    enc = to_bf16 if dtype == "bf16" else (lambda a: np.asarray(a).astype(np.float32))
    dec = bf16_bits_to_f32 if dtype == "bf16" else (lambda a: a)
    U64 = orthonormal_basis(d, k, rng)
    U32 = U64.astype(np.float32)
    tok = enc(0.02 * rng.standard_normal((wl.vocab, d)))
    pe = enc(0.02 * rng.standard_normal((n, d)))
    ids = token_ids(wl, rng, T)
    Z = rng.standard_normal((T, k))
    S = Z @ U64.T
    if wl.off_scale > 0 or wl.off_energy > 0:
        N0 = rng.standard_normal((T, d))
        N = N0 - (N0 @ U64) @ U64.T
        if wl.off_energy > 0:
            e = wl.off_energy
            N *= np.sqrt(e * np.sum(S * S) / ((1.0 - e) * np.sum(N * N)))
        else:
            N *= wl.off_scale
        S = S + N
    E = dec(tok)[ids].astype(np.float64) + dec(pe)[np.arange(T) % n].astype(np.float64)
    out = dict(U64=U64, U=U32, tok_emb=tok, pos_emb=pe, ids=ids, Z=Z, X=enc(E + S))
    if wl.grad:
        out["G"] = enc(rng.standard_normal((T, d)))
    return out


def weight_inputs(cols=None, seed=WEIGHT_SEED, d=WEIGHT_D, k=WEIGHT_K):
    """U [d, k] and the two residual-writing weights ~ N(0, 0.02^2), bf16 bits.
    `cols` optionally overrides the column counts (same draws, truncated)."""
    rng = np.random.default_rng(seed)
    U64 = orthonormal_basis(d, k, rng)
    out = dict(U64=U64, U=U64.astype(np.float32))
    for name, (rows, c) in WEIGHT_SHAPES.items():
        c = c if cols is None else min(c, cols)
        out[name] = to_bf16(0.02 * rng.standard_normal((rows, WEIGHT_SHAPES[name][1]))[:, :c])
    return out


# ---- device-side synthesis for full-size workloads -------------------------

def generate_on_device(wl, device, seed=None, dtype="bf16", grad=None):
    """Full-size inputs synthesised on the GPU with a seeded torch generator.

    Same recipe as `generate`, drawn with torch's device RNG so that gigabyte
    tables never pass through host memory.  U comes from the host fp64 QR.
    Returns torch tensors on `device`; bf16 tensors unless dtype == "f32".
    `grad` forces (or suppresses) the gradient G regardless of the workload.
    """
    import torch

    seed = wl.seed if seed is None else seed
    rng = np.random.default_rng(seed)
    T, d, k, n = wl.T, wl.d, wl.k, wl.seq_len
    U64 = orthonormal_basis(d, k, rng)
    ids_np = token_ids(wl, rng)
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    U = torch.from_numpy(U64.astype(np.float32)).to(device)
    ids = torch.from_numpy(ids_np).to(device)
    tok = (0.02 * torch.randn(wl.vocab, d, generator=g, device=device)).to(tdt)
    pe = (0.02 * torch.randn(n, d, generator=g, device=device)).to(tdt)
    X = torch.empty(T, d, dtype=tdt, device=device)
    chunk = 4096
    # planted subspace part and off-subspace noise, chunk by chunk
    z_sq = 0.0
    n_sq = 0.0
    parts = []
    for t0 in range(0, T, chunk):
        t1 = min(T, t0 + chunk)
        Z = torch.randn(t1 - t0, k, generator=g, device=device)
        S = Z @ U.T
        z_sq += float((S * S).sum())
        if wl.off_scale > 0 or wl.off_energy > 0:
            N0 = torch.randn(t1 - t0, d, generator=g, device=device)
            N = N0 - (N0 @ U) @ U.T
            n_sq += float((N * N).sum())
            parts.append((t0, t1, S, N))
        else:
            parts.append((t0, t1, S, None))
    if wl.off_energy > 0:
        e = wl.off_energy
        scale = (e * z_sq / ((1.0 - e) * n_sq)) ** 0.5
    else:
        scale = wl.off_scale
    pos = torch.arange(T, device=device) % n
    for t0, t1, S, N in parts:
        E = tok[ids[t0:t1]].float() + pe[pos[t0:t1]].float()
        Y = E + S if N is None else E + S + scale * N
        X[t0:t1] = Y.to(tdt)
    del parts
    out = dict(U=U, tok_emb=tok, pos_emb=pe, ids=ids, X=X, ids_host=ids_np)
    if wl.grad if grad is None else grad:
        out["G"] = torch.randn(T, d, generator=g, device=device).to(tdt)
    return out


def unique_ids(ids):
    return int(np.unique(np.asarray(ids)).size)
