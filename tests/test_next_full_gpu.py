"""GPU parity of the method's other parts at the large stream's full sizes, in the
calls the benchmark times, on samples the fp64 oracles compute one by one:
- the projected-table compress (Eq. subtract with T_fixed U, P U): sampled
  tokens against the plain compress of the oracle;
- the Grassmann accumulation M = G^T (G U) over all 65536 tokens (Sec. 6):
  sampled rows of M against the Grassmann oracle's sum, fed a chunk of tokens
  at a time;
- the row-constant AdamW step on W_o [8192, 8192] (Sec. 5): sampled columns
  (each column's rate depends only on that column);
- the top-k, sign and 8-bit comparators on X (Sec. 8): sampled rows.
Bars as everywhere: 1e-2 relative Frobenius error and 3e-2 on the worst row for
bf16 results (the Grassmann accumulation takes the bf16 bar: it reads the bf16
G and the tensor cores' bf16 products), 1e-5 for fp32 ones, exact for selected
columns, sign bits and 8-bit codes."""
import importlib.util
import os

import numpy as np
import pytest
import torch

from gpu_util import assert_parity, host, widen
from paper_2506_01260_gb300 import workloads as W

pytestmark = pytest.mark.gpu
HERE = os.path.dirname(os.path.abspath(__file__))


def _load(name):
    spec = importlib.util.spec_from_file_location("oracle_" + name,
                                                  os.path.join(HERE, "..", "oracle", name + ".py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


@pytest.fixture(scope="module")
def large():
    wl = W.WORKLOADS["large"]
    inp = W.generate_on_device(wl, "cuda", grad=True)
    yield wl, inp
    del inp
    torch.cuda.empty_cache()


def _rows(T, seed, n=96):
    rng = np.random.default_rng(seed)
    picks = set(rng.choice(T, size=n, replace=False).tolist()) | {0, 127, 128, T - 1}
    return np.array(sorted(picks))


def test_projected_compress_full_size(sn, oracle, large):
    wl, inp = large
    basis = sn.Basis(inp["U"])
    n = wl.seq_len
    TU, PU = sn.sn_project_tables(basis, inp["tok_emb"], pos_emb=inp["pos_emb"])
    C = sn.sn_compress_fwd_projected(basis, inp["X"], inp["ids"], TU, n, PU=PU)
    sn.sn_check_errors(basis)
    rows = _rows(wl.T, 21)
    rt = torch.from_numpy(rows).cuda()
    ids = inp["ids"][rt].cpu().numpy()
    uniq, inv = np.unique(ids, return_inverse=True)
    tok = host(inp["tok_emb"][torch.from_numpy(uniq).cuda()])
    pe = host(inp["pos_emb"][torch.from_numpy(rows % n).cuda()])
    _, C64, st = oracle.compress_fwd(host(inp["X"][rt]), inv.astype(np.int32), tok,
                                     inp["U"].cpu().numpy(), len(rows), pos_emb=pe,
                                     pos=np.arange(len(rows), dtype=np.int32))
    assert st == 0
    assert_parity(host(C[rt]), C64, "bf16")
    basis.destroy()


def test_grassmann_accumulate_full_size(sn, large):
    g = _load("grassmann")
    wl, inp = large
    basis = sn.Basis(inp["U"])
    G = inp["G"]
    Cg = sn.sn_compress_bwd(basis, G)
    M = torch.zeros(wl.d, wl.k, dtype=torch.float32, device="cuda")
    sn.sn_grassmann_accumulate(basis, G, Cg, M)
    sn.sn_check_errors(basis)
    U64 = inp["U"].double().cpu().numpy()
    rows = _rows(wl.d, 22, n=24)
    ref = np.zeros((len(rows), wl.k))
    for t0 in range(0, wl.T, 4096):       # the oracle's sum, a chunk of tokens at a time
        ref = g.accumulate_rows(ref, widen(host(G[t0:t0 + 4096])), U64, rows)
    got = M[torch.from_numpy(rows).cuda()].cpu().numpy()
    assert_parity(got, ref, "bf16")
    basis.destroy()


def test_adamw_rowconst_full_size(sn):
    a = _load("adamw")
    rows, cols = 8192, 8192
    g = torch.Generator(device="cuda").manual_seed(5)
    Wt = 0.02 * torch.randn(rows, cols, generator=g, device="cuda")
    Mt = torch.zeros_like(Wt)
    Vt = torch.zeros_like(Wt)
    J = torch.from_numpy(_rows(cols, 23, n=32)).cuda()
    W64 = Wt[:, J].double().cpu().numpy()
    M64 = np.zeros_like(W64)
    V64 = np.zeros_like(W64)
    hp = dict(lr=1e-3, beta1=0.9, beta2=0.95, eps=1e-8, lam=1e-4)
    for t in (1, 2):
        gr = (0.01 * torch.randn(rows, cols, generator=g, device="cuda")).to(torch.bfloat16)
        sn.sn_adamw_rowconst(Wt, gr, Mt, Vt, t, hp["lr"], hp["beta1"], hp["beta2"], hp["eps"],
                             hp["lam"])
        W64, M64, V64 = a.step(W64, widen(host(gr[:, J])), M64, V64, t, hp["lr"], hp["beta1"],
                               hp["beta2"], hp["eps"], hp["lam"])
    torch.cuda.synchronize()
    for got, ref in ((Wt, W64), (Mt, M64), (Vt, V64)):
        got64 = got[:, J].double().cpu().numpy()
        assert np.linalg.norm(got64 - ref) / np.linalg.norm(ref) <= 1e-5


def test_lossy_comparators_full_size(sn, large):
    o = _load("lossy")
    wl, inp = large
    X = inp["X"]
    kk = wl.k // 2
    vals, colsel = sn.sn_topk_compress(X, kk)
    bits, scale = sn.sn_sign_compress(X)
    rows = _rows(wl.T, 24, n=48)
    rt = torch.from_numpy(rows).cuda()
    xb = host(X[rt])
    ref_cols = o.topk_columns(xb, kk)
    assert np.array_equal(host(colsel[rt]).view(np.uint16).astype(np.int64), ref_cols)
    assert np.array_equal(host(vals[rt]), np.take_along_axis(xb, ref_cols, axis=1))
    rb, rs = o.sign_compress(widen(xb))
    words = host(bits[rt]).view(np.uint32)
    got = ((words[:, :, None] >> np.arange(32)[None, None, :]) & 1).reshape(len(rows), -1)
    assert np.array_equal(got[:, :wl.d].astype(np.uint8), rb)
    assert np.max(np.abs(host(scale[rt]).astype(np.float64) - rs) / rs) <= 1e-6
    for fmt in ("int8", "e4m3"):
        codes, qs = sn.sn_quant_compress(X, fmt)
        rc, rq = o.quant_compress(xb, fmt)
        assert np.array_equal(host(codes[rt]), rc), fmt
        assert np.array_equal(host(qs[rt]).view(np.uint32), rq.view(np.uint32)), fmt
