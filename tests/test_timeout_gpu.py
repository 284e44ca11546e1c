"""Failure detection on the GPU without a fault: a bounded in-kernel wait that
runs out (a barrier phase nothing completes) ends its kernel after the wait
limit with SN_ERR_TIMEOUT in the error word, which sn_check_errors reports once
and clears; the tensor memory the CTA held is freed and the context stays
usable: a boundary round trip right after (its CTAs allocate all of an SM's
tensor memory) matches the oracle."""
import pytest
import torch

from gpu_util import assert_parity, dev, host
from paper_2506_01260_gb300 import workloads as W

pytestmark = pytest.mark.gpu

LIMIT_S = 2.0       # the library's wait limit


def test_expired_wait_reports_timeout_and_context_survives(sn, oracle):
    inp = W.generate(W.WORKLOADS["1b"])
    basis = sn.Basis(torch.from_numpy(inp["U"]).cuda())
    s = torch.cuda.current_stream()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(s)
    sn.sn_selftest_wait_timeout(basis)
    b.record(s)
    with pytest.raises(sn.SNError) as e:
        sn.sn_check_errors(basis)
    assert e.value.status == sn.SN_ERR_TIMEOUT
    elapsed = a.elapsed_time(b) / 1e3
    assert LIMIT_S * 0.95 <= elapsed <= LIMIT_S * 2.0, elapsed
    sn.sn_check_errors(basis)                 # reported once, then cleared

    # a reconstruction CTA allocates all of its SM's tensor memory: columns
    # left allocated by the expired CTA would stall it
    X, ids, tok, pe = dev(inp["X"]), dev(inp["ids"]), dev(inp["tok_emb"]), dev(inp["pos_emb"])
    n = W.WORKLOADS["1b"].seq_len
    C = sn.sn_compress_fwd(basis, X, ids, tok, n, pos_emb=pe)
    Xr = sn.sn_decompress_fwd(basis, C, ids, tok, n, pos_emb=pe)
    sn.sn_check_errors(basis)
    _, C64, st = oracle.compress_fwd(inp["X"], inp["ids"], inp["tok_emb"], inp["U"], n,
                                     pos_emb=inp["pos_emb"])
    assert st == 0
    assert_parity(host(C), C64, "bf16")
    X64, st = oracle.decompress_fwd(host(C), inp["ids"], inp["tok_emb"], inp["U"], n,
                                    pos_emb=inp["pos_emb"])[1:]
    assert st == 0
    assert_parity(host(Xr), X64, "bf16")
    basis.destroy()


def test_selftest_rejects_bad_arguments(sn):
    class Null:
        handle = None
    with pytest.raises(sn.SNError) as e:
        sn.sn_selftest_wait_timeout(Null())
    assert e.value.status == sn.SN_ERR_INVALID_ARG
