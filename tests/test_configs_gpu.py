"""GPU parity on the five workload configurations at full size.

tiny and 1B-class run the oracle on every token.  The 8B-class, weight and
large-stream configurations run the GPU over the full tensors, in the same
calls the benchmark times, and check sampled tokens (or weight columns)
against the oracle, which computes each one independently: every sampled row
depends only on its own inputs, so the sample is checked exactly as the full
tensor would be.
"""
import numpy as np
import pytest
import torch

from gpu_util import TOL, assert_parity, dev, host
from paper_2506_01260_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def _sample_rows(T, rng, n=192):
    """Random tokens plus the first tile, the tile seams and the last tokens."""
    picks = set(rng.choice(T, size=min(n, T), replace=False).tolist())
    picks |= set(range(0, min(T, 8))) | set(range(max(0, T - 40), T))
    picks |= {t for t in (127, 128, 129, 255, 256) if t < T}
    return np.array(sorted(picks))


def _compact(inp_dev, rows, seq_len):
    """Oracle inputs for the sampled tokens: their X/G rows, and token/positional
    tables reduced to the rows they use (ids and positions remapped)."""
    ids = inp_dev["ids"][rows].cpu().numpy()
    uniq, inv = np.unique(ids, return_inverse=True)
    tok = host(inp_dev["tok_emb"][torch.from_numpy(uniq).cuda()])
    p = rows % seq_len
    pe = host(inp_dev["pos_emb"][torch.from_numpy(p).cuda()])
    return tok, inv.astype(np.int32), pe, np.arange(len(rows), dtype=np.int32)


@pytest.mark.parametrize("name", ["tiny", "1b"])
def test_full_oracle_configs(sn, oracle, name):
    wl = W.WORKLOADS[name]
    inp = W.generate(wl)
    basis = sn.Basis(dev(inp["U"]))
    X, tok, pe, ids = dev(inp["X"]), dev(inp["tok_emb"]), dev(inp["pos_emb"]), dev(inp["ids"])
    C = sn.sn_compress_fwd(basis, X, ids, tok, wl.seq_len, pos_emb=pe)
    Xr = sn.sn_decompress_fwd(basis, C, ids, tok, wl.seq_len, pos_emb=pe)
    sn.sn_check_errors(basis)
    _, C64, _ = oracle.compress_fwd(inp["X"], inp["ids"], inp["tok_emb"], inp["U"], wl.seq_len,
                                    pos_emb=inp["pos_emb"])
    assert_parity(host(C), C64, "bf16")
    # closed form: C recovers the planted coefficients Z up to the planted noise
    assert_parity(host(C), inp["Z"], "bf16")
    _, X64, _ = oracle.decompress_fwd(host(C), inp["ids"], inp["tok_emb"], inp["U"], wl.seq_len,
                                      pos_emb=inp["pos_emb"])
    assert_parity(host(Xr), X64, "bf16")
    basis.destroy()


@pytest.mark.parametrize("name", ["8b", "large"])
def test_sampled_full_size_configs(sn, oracle, name):
    wl = W.WORKLOADS[name]
    inp = W.generate_on_device(wl, "cuda")
    basis = sn.Basis(inp["U"])
    U = inp["U"].cpu().numpy()
    n = wl.seq_len
    C = sn.sn_compress_fwd(basis, inp["X"], inp["ids"], inp["tok_emb"], n,
                           pos_emb=inp["pos_emb"])
    # through the emulated wire, as the benchmark does
    wire = torch.empty(C.numel() * 2, dtype=torch.uint8, pin_memory=True)
    sn.sn_wire_send(C, wire)
    C_rx = torch.empty_like(C)
    sn.sn_wire_recv(wire, C_rx)
    Xr = sn.sn_decompress_fwd(basis, C_rx, inp["ids"], inp["tok_emb"], n, pos_emb=inp["pos_emb"])
    Cg = sn.sn_compress_bwd(basis, inp["G"])
    Gr = sn.sn_decompress_bwd(basis, Cg)
    sn.sn_check_errors(basis)
    assert torch.equal(C_rx, C)
    rows = _sample_rows(wl.T, np.random.default_rng(wl.seed))
    rt = torch.from_numpy(rows).cuda()
    tok, ids, pe, pos = _compact(inp, rows, n)
    Xs = host(inp["X"][rt])
    _, C64, st = oracle.compress_fwd(Xs, ids, tok, U, len(rows), pos_emb=pe, pos=pos)
    assert st == 0
    assert_parity(host(C[rt]), C64, "bf16")
    _, X64, _ = oracle.decompress_fwd(host(C[rt]), ids, tok, U, len(rows), pos_emb=pe, pos=pos)
    assert_parity(host(Xr[rt]), X64, "bf16")
    _, Cg64, _ = oracle.compress_bwd(host(inp["G"][rt]), U)
    assert_parity(host(Cg[rt]), Cg64, "bf16")
    _, Gr64, _ = oracle.decompress_bwd(host(Cg[rt]), U)
    assert_parity(host(Gr[rt]), Gr64, "bf16")
    # every token: reconstruction error equals the planted off-subspace part
    # (5% of the residual energy at the large config, 1e-3 noise at 8B)
    E = inp["tok_emb"][inp["ids"]].float()
    E += inp["pos_emb"][torch.arange(wl.T, device="cuda") % n].float()
    R = inp["X"].float() - E
    off = float(((Xr.float() - inp["X"].float()).norm() / R.norm()) ** 2)
    expect = wl.off_energy if wl.off_energy else 0.0
    assert abs(off - expect) < 0.01, off
    basis.destroy()


@pytest.mark.parametrize("wname", ["W_o", "W_down"])
def test_weight_projection_config(sn, oracle, wname):
    win = W.weight_inputs()
    basis = sn.Basis(dev(win["U"]))
    Wd = dev(win[wname])
    Wp = sn.sn_project_weight(basis, Wd)
    sn.sn_check_errors(basis)
    cols = np.random.default_rng(3).choice(Wd.shape[1], size=48, replace=False)
    cols = np.unique(np.concatenate([cols, [0, Wd.shape[1] - 1]]))
    Wc = np.ascontiguousarray(win[wname][:, cols])
    _, W64, _ = oracle.project_weight(Wc, win["U"])
    assert_parity(host(Wp)[:, cols], W64, "bf16")
    # P^2 = P on the full output
    Wpp = sn.sn_project_weight(basis, Wp)
    err = float((Wpp.float() - Wp.float()).norm() / Wp.float().norm())
    assert err <= TOL["bf16"], err
    basis.destroy()
