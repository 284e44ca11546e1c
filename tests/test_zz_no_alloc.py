"""sn_project_weight_noalloc: the projection for callers that cannot allocate.

Some callers cannot call cudaMalloc or provide scratch where they project a
weight; this entry point uses the library's fixed 32 MiB device scratch array
instead of a workspace.  Its results must match sn_project_weight (which takes
a caller workspace) within the bf16 parity bar, and the fp64 oracle on sampled
columns, on consecutive calls that reuse the same scratch: out of place into a
strided output whose padding columns must stay untouched, in place, and after
a call with another column count has left other partial sums in the array.
Collected last so that a stop-at-first-failure run has already run every other
test.
"""
import numpy as np
import pytest
import torch

from gpu_util import assert_parity, dev, host, widen
from paper_2506_01260_gb300 import workloads as W

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("d,k,cols,ld", [(4096, 41, 4096, 4096), (1024, 20, 777, 784),
                                         (8192, 82, 2048, 2048)])
def test_noalloc_matches_workspace_entry_point(sn, oracle, d, k, cols, ld):
    rng = np.random.default_rng(d + cols)
    U = W.orthonormal_basis(d, k, rng).astype(np.float32)
    basis = sn.Basis(dev(U))
    Wh = W.to_bf16(0.02 * rng.standard_normal((d, ld)))
    Wd = dev(Wh)[:, :cols]
    ref = torch.zeros(d, ld, dtype=torch.bfloat16, device="cuda")[:, :cols]
    sn.sn_project_weight(basis, Wd, out=ref)
    sample = np.unique(np.concatenate([rng.choice(cols, size=24, replace=False), [0, cols - 1]]))
    _, W64, _ = oracle.project_weight(np.ascontiguousarray(Wh[:, sample]), U)
    for call in range(2):         # two calls in a row share the scratch array
        if call == 1:
            # a call with another column count (another split of d) first
            oc = 8 * ((3 * cols // 2 + 7) // 8) + 8
            other = dev(W.to_bf16(0.02 * rng.standard_normal((d, oc))))
            sn.sn_project_weight_noalloc(basis, other, other)
        full = torch.full((d, ld), 3.0, dtype=torch.bfloat16, device="cuda")
        out = full[:, :cols]
        sn.sn_project_weight_noalloc(basis, Wd, out)
        sn.sn_check_errors(basis)
        assert_parity(host(out), widen(host(ref)), "bf16")
        assert_parity(host(out)[:, sample], W64, "bf16")
        if ld > cols:             # the padding columns of the strided output are untouched
            assert bool((full[:, cols:] == 3.0).all())
    # in place: W_out is W
    Wfull = dev(Wh)
    Win = Wfull[:, :cols]
    sn.sn_project_weight_noalloc(basis, Win, Win)
    sn.sn_check_errors(basis)
    assert_parity(host(Win), widen(host(ref)), "bf16")
    basis.destroy()


def test_noalloc_rejects_what_it_cannot_hold(sn):
    rng = np.random.default_rng(1)
    d, k = 128, 128
    basis = sn.Basis(dev(W.orthonormal_basis(d, k, rng).astype(np.float32)))
    cols = 65536                  # needs more than 32 MiB of scratch
    assert sn.sn_project_weight_workspace(basis, torch.bfloat16, cols) > 32 << 20
    Wbig = torch.zeros(d, cols, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(sn.SNError) as e:
        sn.sn_project_weight_noalloc(basis, Wbig, Wbig)
    assert e.value.status == sn.SN_ERR_UNSUPPORTED
    W32 = torch.zeros(d, 64, dtype=torch.float32, device="cuda")
    with pytest.raises((sn.SNError, TypeError)):
        sn.sn_project_weight_noalloc(basis, W32, W32)
    basis.destroy()
