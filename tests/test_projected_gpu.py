"""GPU parity of the projected-table variant of the forward compress (bf16).

Because the compress of Sec. 4.3.1, Eq. (subtract), is linear, the library
can project T_fixed and P onto U once (sn_project_tables) and compress with
k-wide rows (sn_compress_fwd_projected).  Its result is checked against the
oracle's plain definition of the forward compress, the tables against the
oracle's fp64 products, and T_S = T_fixed U U^T against the oracle's exact
projection.  Bar: 1e-2 relative Frobenius error (bf16), as for every bf16 call.
"""
import numpy as np
import pytest
import torch

from gpu_util import assert_parity, dev, host, widen
from paper_2506_01260_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def inputs(T, n, d, k, vocab, seed):
    wl = W.Workload("proj", 1, n, d, k, vocab, 3000 + seed, off_scale=1e-2, grad=False)
    return W.generate(wl, T=T, dtype="bf16")


@pytest.mark.parametrize("T,n,d,k,vocab", [(1000, 300, 512, 20, 3000), (4173, 1024, 1024, 41, 5000),
                                           (260, 4096, 8192, 82, 700), (1, 7, 64, 1, 5)])
def test_tables_and_projected_compress(sn, oracle, T, n, d, k, vocab):
    inp = inputs(T, n, d, k, vocab, seed=d + k)
    basis = sn.Basis(dev(inp["U"]))
    tok, pe, X, ids = dev(inp["tok_emb"]), dev(inp["pos_emb"]), dev(inp["X"]), dev(inp["ids"])
    TU, PU = sn.sn_project_tables(basis, tok, pos_emb=pe)
    # the tables: fp32 products of the bf16 tables with U (U rounded once to bf16)
    _, TU64, _ = oracle.compress_bwd(inp["tok_emb"], inp["U"])
    _, PU64, _ = oracle.compress_bwd(inp["pos_emb"], inp["U"])
    assert_parity(TU.cpu().numpy(), TU64, "bf16")
    assert_parity(PU.cpu().numpy(), PU64, "bf16")
    # the compress: the same C as the definition
    C = sn.sn_compress_fwd_projected(basis, X, ids, TU, n, PU=PU)
    sn.sn_check_errors(basis)
    _, C64, st = oracle.compress_fwd(inp["X"], inp["ids"], inp["tok_emb"], inp["U"], n,
                                     pos_emb=inp["pos_emb"])
    assert st == 0
    assert_parity(host(C), C64, "bf16")
    # and the same C as the d-wide kernel, within the bf16 bar
    Cd = sn.sn_compress_fwd(basis, X, ids, tok, n, pos_emb=pe)
    assert_parity(host(C), widen(host(Cd)), "bf16")
    basis.destroy()


def test_projected_without_positions_and_with_explicit_positions(sn, oracle):
    T, n, d, k, vocab = 700, 50, 512, 24, 900
    inp = inputs(T, n, d, k, vocab, seed=7)
    rng = np.random.default_rng(4)
    pos = rng.integers(0, n, T).astype(np.int32)
    basis = sn.Basis(dev(inp["U"]))
    tok, pe, X, ids = dev(inp["tok_emb"]), dev(inp["pos_emb"]), dev(inp["X"]), dev(inp["ids"])
    TU, PU = sn.sn_project_tables(basis, tok, pos_emb=pe)
    TU_only, none = sn.sn_project_tables(basis, tok)
    assert none is None
    C1 = sn.sn_compress_fwd_projected(basis, X, ids, TU, n, PU=PU, pos=dev(pos))
    C2 = sn.sn_compress_fwd_projected(basis, X, ids, TU_only, n)
    sn.sn_check_errors(basis)
    _, C64, _ = oracle.compress_fwd(inp["X"], inp["ids"], inp["tok_emb"], inp["U"], n,
                                    pos_emb=inp["pos_emb"], pos=pos)
    assert_parity(host(C1), C64, "bf16")
    _, C64, _ = oracle.compress_fwd(inp["X"], inp["ids"], inp["tok_emb"], inp["U"], n)
    assert_parity(host(C2), C64, "bf16")
    basis.destroy()


def test_projected_bad_ids_zero_rows(sn, oracle):
    T, n, d, k, vocab = 300, 128, 256, 16, 400
    inp = inputs(T, n, d, k, vocab, seed=9)
    ids = inp["ids"].copy()
    ids[5], ids[250] = -1, vocab
    basis = sn.Basis(dev(inp["U"]))
    TU, PU = sn.sn_project_tables(basis, dev(inp["tok_emb"]), pos_emb=dev(inp["pos_emb"]))
    C = sn.sn_compress_fwd_projected(basis, dev(inp["X"]), dev(ids), TU, n, PU=PU)
    with pytest.raises(sn.SNError) as e:
        sn.sn_check_errors(basis)
    assert e.value.status == sn.SN_ERR_BAD_ID
    c = host(C)
    assert not c[5].any() and not c[250].any()
    _, C64, _ = oracle.compress_fwd(inp["X"], ids, inp["tok_emb"], inp["U"], n,
                                    pos_emb=inp["pos_emb"])
    keep = np.ones(T, bool)
    keep[[5, 250]] = False
    assert_parity(c[keep], C64[keep], "bf16")
    basis.destroy()


@pytest.mark.parametrize("vocab,d,k", [(3000, 512, 20), (777, 2048, 128), (5, 64, 1)])
def test_build_ts(sn, oracle, vocab, d, k):
    inp = inputs(8, 8, d, k, vocab, seed=vocab)
    basis = sn.Basis(dev(inp["U"]))
    TS = sn.sn_build_ts(basis, dev(inp["tok_emb"]))
    sn.sn_check_errors(basis)
    _, TU64, _ = oracle.compress_bwd(inp["tok_emb"], inp["U"])
    _, TS64, _ = oracle.decompress_bwd(TU64, inp["U"])     # T_fixed U U^T in fp64
    assert_parity(host(TS), TS64, "bf16")
    basis.destroy()


def test_projected_argument_errors(sn):
    d, k, vocab = 256, 8, 64
    U = torch.linalg.qr(torch.randn(d, k, dtype=torch.float64))[0].float().contiguous().cuda()
    basis = sn.Basis(U)
    tok = torch.zeros(vocab, d, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(sn.SNError) as e:                  # fp32 is not offered
        sn.sn_project_tables(basis, tok.float())
    assert e.value.status == sn.SN_ERR_UNSUPPORTED
    TU, _ = sn.sn_project_tables(basis, tok)
    X = torch.zeros(4, d, dtype=torch.bfloat16, device="cuda")
    ids = torch.zeros(4, dtype=torch.int32, device="cuda")
    with pytest.raises(sn.SNError) as e:                  # output overlapping the input
        sn.sn_compress_fwd_projected(basis, X, ids, TU, 4, out=X.view(-1)[: 4 * k].view(4, k))
    assert e.value.status == sn.SN_ERR_INVALID_ARG
    with pytest.raises(sn.SNError) as e:                  # workspace too small
        sn.sn_build_ts(basis, tok, workspace=torch.empty(16, dtype=torch.uint8, device="cuda"))
    assert e.value.status == sn.SN_ERR_INVALID_ARG
    basis.destroy()
