"""GPU parity of the paired reconstruction (Sec. 4.3.1): when a batch holds an
even number of whole sequences whose length is a multiple of 128 and the model
has a positional table, sn_decompress_fwd processes the tiles of sequences 2i
and 2i + 1 at one position block together (they add the same positional tile).

Checked against the fp64 oracle: k from 1 to 128 (odd and even k, one to four
16-word chunks of A per tile), widths of one to eight 128-column blocks, more
work items than SMs (several items per CTA, so the next item's operands are
prepared during the current one, or written at the item's start when the items
are short), invalid ids, and C = 0, where the output is
round(T_fixed[id] + P[pos]) bit for bit.  The same batch with the positions
given explicitly runs the single-tile kernel; both kernels compute the same
fp32 sums and must agree bit for bit.
"""
import numpy as np
import pytest
import torch

from gpu_util import assert_parity, dev, guarded, guards_intact, host, widen
from paper_2506_01260_gb300 import workloads as W

pytestmark = pytest.mark.gpu

# (name, sequences, seq_len, d, k, vocab)
PAIR_CASES = [
    ("pairs_d512_k41", 4, 256, 512, 41, 3000),
    ("pairs_d1024_k82", 2, 512, 1024, 82, 2000),
    ("pairs_d256_k128", 6, 128, 256, 128, 700),
    ("pairs_d128_k1", 2, 128, 128, 1, 50),
    ("pairs_d384_k33", 8, 128, 384, 33, 900),
]


def inputs(name, nseq, n, d, k, vocab, seed=0):
    wl = W.Workload(name, 1, n, d, k, vocab, 2000 + seed + d + k, off_scale=1e-2, grad=False)
    return W.generate(wl, T=nseq * n, dtype="bf16")


@pytest.mark.parametrize("case", PAIR_CASES, ids=[c[0] for c in PAIR_CASES])
def test_paired_reconstruction_matches_oracle(sn, oracle, case):
    name, nseq, n, d, k, vocab = case
    T = nseq * n
    inp = inputs(name, nseq, n, d, k, vocab)
    basis = sn.Basis(dev(inp["U"]))
    C = sn.sn_compress_fwd(basis, dev(inp["X"]), dev(inp["ids"]), dev(inp["tok_emb"]), n,
                           pos_emb=dev(inp["pos_emb"]))
    fullX, Xr = guarded((T, d), torch.bfloat16)
    sn.sn_decompress_fwd(basis, C, dev(inp["ids"]), dev(inp["tok_emb"]), n,
                         pos_emb=dev(inp["pos_emb"]), out=Xr)
    sn.sn_check_errors(basis)
    assert guards_intact(fullX)
    _, X64, st = oracle.decompress_fwd(host(C), inp["ids"], inp["tok_emb"], inp["U"], n,
                                       pos_emb=inp["pos_emb"])
    assert st == 0
    assert_parity(host(Xr), X64, "bf16")
    basis.destroy()


def test_paired_more_items_than_sms(sn, oracle):
    """More tile pairs than SMs and 16 half blocks per item: CTAs take several
    items, each loading the next item's ids and A operand during the current."""
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    nseq, n, d, k, vocab = 2 * (sms + 8), 128, 1024, 24, 600
    T = nseq * n
    inp = inputs("pairs_many", nseq, n, d, k, vocab, seed=3)
    basis = sn.Basis(dev(inp["U"]))
    C = sn.sn_compress_fwd(basis, dev(inp["X"]), dev(inp["ids"]), dev(inp["tok_emb"]), n,
                           pos_emb=dev(inp["pos_emb"]))
    fullX, Xr = guarded((T, d), torch.bfloat16)
    sn.sn_decompress_fwd(basis, C, dev(inp["ids"]), dev(inp["tok_emb"]), n,
                         pos_emb=dev(inp["pos_emb"]), out=Xr)
    sn.sn_check_errors(basis)
    assert guards_intact(fullX)
    _, X64, st = oracle.decompress_fwd(host(C), inp["ids"], inp["tok_emb"], inp["U"], n,
                                       pos_emb=inp["pos_emb"])
    assert st == 0
    assert_parity(host(Xr), X64, "bf16")
    basis.destroy()


def test_paired_short_items_write_a_at_item_start(sn, oracle):
    """k = 128 (four chunks of A per tile) and items of two blocks: an item is
    too short to load the next item's eight chunks during it, so every later
    item's A is written by the gather warps at the item's start."""
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    nseq, n, d, k, vocab = 2 * (sms + 8), 128, 256, 128, 900
    T = nseq * n
    inp = inputs("pairs_short", nseq, n, d, k, vocab, seed=7)
    basis = sn.Basis(dev(inp["U"]))
    C = np.asarray(W.to_bf16(np.random.default_rng(7).standard_normal((T, k))))
    fullX, Xr = guarded((T, d), torch.bfloat16)
    sn.sn_decompress_fwd(basis, dev(C), dev(inp["ids"]), dev(inp["tok_emb"]), n,
                         pos_emb=dev(inp["pos_emb"]), out=Xr)
    sn.sn_check_errors(basis)
    assert guards_intact(fullX)
    _, X64, st = oracle.decompress_fwd(C, inp["ids"], inp["tok_emb"], inp["U"], n,
                                       pos_emb=inp["pos_emb"])
    assert st == 0
    assert_parity(host(Xr), X64, "bf16")
    basis.destroy()


def test_paired_bad_ids_zero_rows_and_report(sn, oracle):
    nseq, n, d, k, vocab = 4, 256, 512, 20, 500
    T = nseq * n
    inp = inputs("pairs_bad", nseq, n, d, k, vocab, seed=5)
    ids = inp["ids"].copy()
    bad = [3, 256 + 17, 2 * 256 + 255, T - 1]      # rows in both tiles of both pairs
    ids[bad] = [vocab, -1, 2**31 - 1, -2**31]
    basis = sn.Basis(dev(inp["U"]))
    C = np.asarray(W.to_bf16(np.random.default_rng(5).standard_normal((T, k))))
    Xr = sn.sn_decompress_fwd(basis, dev(C), dev(ids), dev(inp["tok_emb"]), n,
                              pos_emb=dev(inp["pos_emb"]))
    with pytest.raises(sn.SNError) as e:
        sn.sn_check_errors(basis)
    assert e.value.status == sn.SN_ERR_BAD_ID
    Xh = host(Xr)
    assert np.all(widen(Xh[bad]) == 0)
    _, X64, st = oracle.decompress_fwd(C, ids, inp["tok_emb"], inp["U"], n,
                                       pos_emb=inp["pos_emb"])
    assert st == 4
    assert_parity(Xh, X64, "bf16")
    basis.destroy()


def test_paired_gather_bit_exact(sn, oracle):
    """C = 0: every output is round(T_fixed[id] + P[pos]), bit for bit."""
    nseq, n, d, k, vocab = 6, 256, 1024, 33, 4000
    T = nseq * n
    inp = inputs("pairs_gather", nseq, n, d, k, vocab, seed=9)
    basis = sn.Basis(dev(inp["U"]))
    C0 = np.zeros((T, k), np.uint16)
    Xr = sn.sn_decompress_fwd(basis, dev(C0), dev(inp["ids"]), dev(inp["tok_emb"]), n,
                              pos_emb=dev(inp["pos_emb"]))
    sn.sn_check_errors(basis)
    Xo, _, _ = oracle.decompress_fwd(C0, inp["ids"], inp["tok_emb"], inp["U"], n,
                                     pos_emb=inp["pos_emb"])
    assert np.array_equal(host(Xr), Xo)
    basis.destroy()


@pytest.mark.parametrize("k", [41, 82, 128])
def test_paired_equals_single_tile_kernel(sn, k):
    """Explicit positions (t mod seq_len) give the same sums through the
    single-tile kernel: the two outputs must be identical."""
    nseq, n, d, vocab = 4, 256, 1024, 3000
    T = nseq * n
    inp = inputs("pairs_vs_single", nseq, n, d, k, vocab, seed=13)
    basis = sn.Basis(dev(inp["U"]))
    C = np.asarray(W.to_bf16(np.random.default_rng(13).standard_normal((T, k))))
    args = (basis, dev(C), dev(inp["ids"]), dev(inp["tok_emb"]), n)
    Xp = sn.sn_decompress_fwd(*args, pos_emb=dev(inp["pos_emb"]))
    pos = (np.arange(T) % n).astype(np.int32)
    Xs = sn.sn_decompress_fwd(*args, pos_emb=dev(inp["pos_emb"]), pos=dev(pos))
    sn.sn_check_errors(basis)
    assert np.array_equal(host(Xp), host(Xs))
    basis.destroy()


def _sweep_cases():
    """Seeded small shapes on both sides of the pairing conditions."""
    rng = np.random.default_rng(2024)
    cases = []
    for i in range(16):
        nseq = int(rng.integers(1, 7))                 # odd counts run the single-tile kernel
        n = int(rng.choice([128, 256, 384, 200]))      # 200: not a whole number of tiles
        d = int(rng.choice([128, 256, 384, 520]))      # 520: not a whole number of blocks
        k = int(rng.choice([1, 7, 16, 41, 64, 96, 128]))
        k = min(k, d)
        explicit = bool(rng.integers(0, 4) == 0)       # explicit positions: single-tile kernel
        cases.append((i, nseq, n, d, k, explicit))
    return cases


@pytest.mark.parametrize("case", _sweep_cases(), ids=lambda c: "s%d_b%d_n%d_d%d_k%d%s" % (
    c[0], c[1], c[2], c[3], c[4], "_pos" if c[5] else ""))
def test_reconstruction_shape_sweep(sn, oracle, case):
    """Paired and single-tile reconstructions against the oracle over seeded
    shapes (even and odd sequence counts, lengths and widths on and off the
    tile and block sizes, explicit positions)."""
    i, nseq, n, d, k, explicit = case
    T = nseq * n
    inp = inputs("sweep%d" % i, nseq, n, d, k, 700, seed=100 + i)
    basis = sn.Basis(dev(inp["U"]))
    C = np.asarray(W.to_bf16(np.random.default_rng(i).standard_normal((T, k))))
    pos = (np.arange(T) % n).astype(np.int32) if explicit else None
    fullX, Xr = guarded((T, d), torch.bfloat16)
    sn.sn_decompress_fwd(basis, dev(C), dev(inp["ids"]), dev(inp["tok_emb"]), n,
                         pos_emb=dev(inp["pos_emb"]), pos=None if pos is None else dev(pos),
                         out=Xr)
    sn.sn_check_errors(basis)
    assert guards_intact(fullX)
    _, X64, st = oracle.decompress_fwd(C, inp["ids"], inp["tok_emb"], inp["U"], n,
                                       pos_emb=inp["pos_emb"], pos=pos)
    assert st == 0
    assert_parity(host(Xr), X64, "bf16")
    basis.destroy()
