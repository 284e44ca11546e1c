"""GPU parity of the row-constant AdamW step (Sec. 5) against the fp64 oracle in
oracle/adamw.py.  Bar: 1e-5 relative Frobenius error on W, M and V after three
steps (fp32 arithmetic; bf16 gradients are handed to the oracle as the exact
values the GPU saw), and a weight in S stays in S to 1e-5 relative."""
import importlib.util
import os

import numpy as np
import pytest
import torch

from gpu_util import widen
from paper_2506_01260_gb300 import workloads as W_

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))
HP = dict(lr=3e-3, beta1=0.9, beta2=0.95, eps=1e-8, lam=1e-4)


def adamw_oracle():
    spec = importlib.util.spec_from_file_location("oracle_adamw",
                                                  os.path.join(HERE, "..", "oracle", "adamw.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def rel(a, b):
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


@pytest.mark.parametrize("gdt", ["f32", "bf16"])
@pytest.mark.parametrize("rows,cols", [(512, 1000), (4096, 300), (7, 3), (130, 1002)])
def test_three_steps_match_oracle(sn, gdt, rows, cols):
    a = adamw_oracle()
    rng = np.random.default_rng(rows + cols)
    W0 = rng.standard_normal((rows, cols)).astype(np.float32)
    W = torch.tensor(W0, device="cuda")
    M = torch.zeros_like(W)
    V = torch.zeros_like(W)
    W64, M64, V64 = W0.astype(np.float64), np.zeros((rows, cols)), np.zeros((rows, cols))
    for t in (1, 2, 3):
        g64 = rng.standard_normal((rows, cols)) * rng.uniform(0.1, 3.0, (1, cols))
        if gdt == "bf16":
            gb = W_.to_bf16(g64)
            g = torch.from_numpy(gb.view(np.int16)).view(torch.bfloat16).cuda()
            gx = widen(gb)
        else:
            g = torch.tensor(g64.astype(np.float32), device="cuda")
            gx = g64.astype(np.float32).astype(np.float64)
        sn.sn_adamw_rowconst(W, g, M, V, t, HP["lr"], HP["beta1"], HP["beta2"], HP["eps"],
                             HP["lam"])
        W64, M64, V64 = a.step(W64, gx, M64, V64, t, HP["lr"], HP["beta1"], HP["beta2"],
                               HP["eps"], HP["lam"])
    torch.cuda.synchronize()
    assert rel(W.cpu().numpy().astype(np.float64), W64) <= 1e-5
    assert rel(M.cpu().numpy().astype(np.float64), M64) <= 1e-5
    assert rel(V.cpu().numpy().astype(np.float64), V64) <= 1e-5


def test_weight_in_subspace_stays_there(sn):
    rng = np.random.default_rng(11)
    d, k, n = 1024, 20, 700
    U = W_.orthonormal_basis(d, k, rng)
    W = torch.tensor((U @ rng.standard_normal((k, n))).astype(np.float32), device="cuda")
    M = torch.zeros_like(W)
    V = torch.zeros_like(W)
    Ut = torch.tensor(U, device="cuda")
    for t in range(1, 6):
        g = torch.tensor((U @ rng.standard_normal((k, n))).astype(np.float32), device="cuda")
        sn.sn_adamw_rowconst(W, g, M, V, t, 1e-2, 0.9, 0.99, 1e-8, 1e-3)
    Wd = W.double()
    out = Wd - Ut @ (Ut.t() @ Wd)
    assert float(out.norm() / Wd.norm()) <= 1e-5


def test_adamw_argument_errors(sn):
    W = torch.zeros(64, 32, device="cuda")
    M = torch.zeros_like(W)
    V = torch.zeros_like(W)
    g = torch.zeros_like(W)
    with pytest.raises(sn.SNError) as e:
        sn.sn_adamw_rowconst(W, g, M, V, 0, 1e-3)             # steps count from 1
    assert e.value.status == sn.SN_ERR_INVALID_ARG
    with pytest.raises(sn.SNError) as e:
        sn.sn_adamw_rowconst(W, g, M, M, 1, 1e-3)             # V overlapping M
    assert e.value.status == sn.SN_ERR_INVALID_ARG
    with pytest.raises(sn.SNError) as e:
        sn.sn_adamw_rowconst(W, g, M, V, 1, 1e-3, workspace=torch.empty(4, device="cuda"))
    assert e.value.status == sn.SN_ERR_INVALID_ARG
