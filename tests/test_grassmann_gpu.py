"""GPU parity of the Grassmann subspace update (Sec. 4.5, Sec. 6) against the
fp64 oracle in oracle/grassmann.py.

Bars: the accumulation M = sum_t G_t^T (G_t U) within 1e-2 relative Frobenius
error (bf16 G and Cg); the residual within 1e-3 relative; the step (fp32,
CholeskyQR2) within 1e-4 relative Frobenius error of the oracle's step from the
same M, with U_new^T U_new = I to 1e-5.
"""
import os
import importlib.util

import numpy as np
import pytest
import torch

from gpu_util import dev, host, widen
from paper_2506_01260_gb300 import workloads as W

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))


def grassmann_oracle():
    spec = importlib.util.spec_from_file_location(
        "oracle_grassmann", os.path.join(HERE, "..", "oracle", "grassmann.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def basis_and_grads(sn, d, k, T, n_iter, seed):
    rng = np.random.default_rng(seed)
    U = W.orthonormal_basis(d, k, rng)                # fp64, diag(R) > 0
    U32 = U.astype(np.float32)
    Gs = [W.to_bf16(rng.standard_normal((T, d))) for _ in range(n_iter)]
    return U32, Gs


def rel(a, b):
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


@pytest.mark.parametrize("d,k,T", [(512, 20, 3000), (1024, 41, 777), (256, 128, 300), (64, 1, 5)])
def test_accumulate_and_residual(sn, d, k, T):
    g = grassmann_oracle()
    U32, Gs = basis_and_grads(sn, d, k, T, 2, seed=d + k)
    basis = sn.Basis(dev(U32))
    M = torch.zeros(d, k, dtype=torch.float32, device="cuda")
    acc = torch.zeros(1, dtype=torch.float64, device="cuda")
    M64 = np.zeros((d, k))
    res64 = 0.0
    for Gb in Gs:
        G = dev(Gb)
        Cg = sn.sn_compress_bwd(basis, G)
        sn.sn_grassmann_accumulate(basis, G, Cg, M)
        sn.sn_grassmann_residual(basis, G, Cg, acc)
        G64 = widen(Gb)
        M64 = g.accumulate(M64, G64, U32.astype(np.float64))
        res64 += g.residual(G64, U32.astype(np.float64))
    sn.sn_check_errors(basis)
    assert rel(M.cpu().numpy().astype(np.float64), M64) <= 1e-2
    assert abs(acc.item() - res64) <= 1e-3 * res64
    basis.destroy()


@pytest.mark.parametrize("d,k", [(512, 20), (2048, 82), (256, 128)])
def test_step_matches_oracle(sn, d, k):
    g = grassmann_oracle()
    U32, Gs = basis_and_grads(sn, d, k, 400, 3, seed=7 * d + k)
    U64 = U32.astype(np.float64)
    M64 = np.zeros((d, k))
    for Gb in Gs:
        M64 = g.accumulate(M64, widen(Gb), U64)
    K = len(Gs)
    M32 = M64.astype(np.float32)
    eta = 0.1 / (2.0 * np.linalg.norm(M64, 2) / K)       # a step of ~0.1 in the tangent direction
    basis = sn.Basis(dev(U32))
    Unew = sn.sn_grassmann_step(basis, dev(M32), K, eta)
    sn.sn_check_errors(basis)
    U1 = Unew.cpu().numpy().astype(np.float64)
    ref = g.step(U64, M32.astype(np.float64), K, eta)
    assert rel(U1, ref) <= 1e-4
    assert np.max(np.abs(U1.T @ U1 - np.eye(k))) <= 1e-5
    # and the step lowers the Grassmann loss of the gradients it was taken on
    G64 = [widen(Gb) for Gb in Gs]
    assert g.loss(G64, U1) < g.loss(G64, U64)
    basis.destroy()


def test_step_reports_a_failed_factorisation(sn):
    d, k = 256, 8
    U32, _ = basis_and_grads(sn, d, k, 4, 0, seed=1)
    basis = sn.Basis(dev(U32))
    M = torch.full((d, k), float("nan"), dtype=torch.float32, device="cuda")
    sn.sn_grassmann_step(basis, M, 1, 0.1)
    with pytest.raises(sn.SNError) as e:
        sn.sn_check_errors(basis)
    assert e.value.status == sn.SN_ERR_NUMERIC
    sn.sn_check_errors(basis)                       # cleared
    basis.destroy()


def test_grassmann_argument_errors(sn):
    d, k = 256, 8
    U32, _ = basis_and_grads(sn, d, k, 4, 0, seed=2)
    basis = sn.Basis(dev(U32))
    M = torch.zeros(d, k, dtype=torch.float32, device="cuda")
    with pytest.raises(sn.SNError) as e:
        sn.sn_grassmann_step(basis, M, 0, 0.1)       # K >= 1
    assert e.value.status == sn.SN_ERR_INVALID_ARG
    with pytest.raises(sn.SNError) as e:
        sn.sn_grassmann_step(basis, M, 1, 0.1, out=M)   # output overlapping M
    assert e.value.status == sn.SN_ERR_INVALID_ARG
    G = torch.zeros(4, d, dtype=torch.bfloat16, device="cuda")
    Cg = torch.zeros(4, k, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(sn.SNError) as e:
        sn.sn_grassmann_accumulate(basis, G, Cg, M,
                                   workspace=torch.empty(256, dtype=torch.uint8, device="cuda"))
    assert e.value.status == sn.SN_ERR_INVALID_ARG
    basis.destroy()
