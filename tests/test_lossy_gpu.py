"""GPU parity of the lossy comparators against the fp64 oracle in
oracle/lossy.py: top-k columns, values and restores bit-exact (selection on bf16
magnitudes, ties towards the lower column); sign bits exact and the row scale
within 1e-6 relative; int8 and fp8 e4m3 codes, scales and restores bit-exact; the randomized low-rank round trip within 1.5 times the
error of the exact truncated SVD (plus 1e-3) on a noisy low-rank batch."""
import importlib.util
import os

import numpy as np
import pytest
import torch

from gpu_util import dev, host, widen
from paper_2506_01260_gb300 import comparators
from paper_2506_01260_gb300 import workloads as W

pytestmark = pytest.mark.gpu
HERE = os.path.dirname(os.path.abspath(__file__))


def lossy_oracle():
    spec = importlib.util.spec_from_file_location("oracle_lossy",
                                                  os.path.join(HERE, "..", "oracle", "lossy.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def batch(T, d, seed, ties=False, const=False):
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((T, d))
    if ties:                                           # many equal magnitudes
        x = np.round(x * 2) / 2
    if const:                                          # one magnitude per row, random signs
        x = np.sign(x) * rng.uniform(0.5, 2.0, (T, 1))
    return W.to_bf16(x)


# Most cases take the candidate path (few entries reach the bound, M = 1..4
# chunk maxima vouched for per lane); kk > 96, rows of one magnitude and
# heavy ties on wide rows take the exact whole-row path.
@pytest.mark.parametrize("T,d,kk,ties,const", [
    (300, 512, 41, False, False), (20, 8192, 41, False, False), (64, 256, 30, True, False),
    (9, 64, 64, True, False), (5, 128, 1, False, False), (40, 2048, 256, True, False),
    (4, 8192, 300, False, False), (3, 4096, 41, False, True), (6, 256, 17, False, True),
    (2, 65536, 4096, False, False), (50, 4096, 70, False, False), (50, 4096, 90, False, False),
    (33, 8200, 41, False, False)])
def test_topk_bit_exact(sn, T, d, kk, ties, const):
    o = lossy_oracle()
    xb = batch(T, d, seed=T + d, ties=ties, const=const)
    vals, cols = sn.sn_topk_compress(dev(xb), kk)
    c = host(cols).view(np.uint16).astype(np.int64)
    ref_cols = o.topk_columns(xb, kk)
    assert np.array_equal(c, ref_cols)
    assert np.array_equal(host(vals), np.take_along_axis(xb, ref_cols, axis=1))
    Xh = sn.sn_topk_restore(vals, cols, d)
    ref = o.topk_restore(widen(np.take_along_axis(xb, ref_cols, axis=1)), ref_cols, d)
    assert np.array_equal(widen(host(Xh)), ref)


@pytest.mark.parametrize("T,d", [(300, 512), (7, 8200), (3, 40)])
def test_sign_quantization(sn, T, d):
    o = lossy_oracle()
    xb = batch(T, d, seed=d)
    xb[0, :5] = np.array([0x8000, 0x0000, 0x8001, 0x0001, 0xBF80], np.uint16)   # -0, +0, tiny, -1
    bits, scale = sn.sn_sign_compress(dev(xb))
    rb, rs = o.sign_compress(widen(xb))
    words = host(bits).view(np.uint32)
    got = ((words[:, :, None] >> np.arange(32)[None, None, :]) & 1).reshape(T, -1)[:, :d]
    assert np.array_equal(got.astype(np.uint8), rb)
    s = host(scale).astype(np.float64)
    assert np.max(np.abs(s - rs) / rs) <= 1e-6
    Xh = widen(host(sn.sn_sign_restore(bits, scale, d)))
    want = widen(W.to_bf16(np.where(rb == 1, -1.0, 1.0) * s[:, None].astype(np.float32)))
    assert np.array_equal(Xh, want)


def test_lowrank_roundtrip_close_to_svd(sn):
    o = lossy_oracle()
    rng = np.random.default_rng(4)
    T, d, r0, r = 3000, 512, 20, 24
    x = rng.standard_normal((T, r0)) @ rng.standard_normal((r0, d)) / np.sqrt(r0)
    x += 1e-2 * rng.standard_normal((T, d))
    xb = W.to_bf16(x)
    Xh, wire = comparators.lowrank_roundtrip(dev(xb), r)
    x64 = widen(xb)
    err = np.linalg.norm(widen(host(Xh)) - x64) / np.linalg.norm(x64)
    best = np.linalg.norm(o.lowrank(x64, r) - x64) / np.linalg.norm(x64)
    assert err <= 1.5 * best + 1e-3
    assert wire == o.wire_bytes("lowrank", T, d, r=r)


def test_lossy_argument_errors(sn):
    X = torch.zeros(4, 64, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(sn.SNError) as e:
        sn.sn_topk_compress(X, 65)                      # kk > d
    assert e.value.status == sn.SN_ERR_INVALID_ARG
    with pytest.raises(sn.SNError) as e:
        sn.sn_sign_compress(torch.zeros(4, 60, dtype=torch.bfloat16, device="cuda"))   # d % 8
    assert e.value.status == sn.SN_ERR_INVALID_ARG


# Row-scaled 8-bit quantization: codes, scales and restores bit for bit against
# the oracle's fp32 decisions.  Rows of mixed magnitudes (2^-8 .. 2^8), a zero
# row, a row with one nonzero entry, signed zeros and entries small enough to
# round to (signed) zero in e4m3.
@pytest.mark.parametrize("fmt", ["int8", "e4m3"])
@pytest.mark.parametrize("T,d", [(1, 8), (37, 264), (300, 4096), (4, 65536), (9, 8200)])
def test_quant_bit_exact(sn, fmt, T, d):
    o = lossy_oracle()
    rng = np.random.default_rng(3 * T + d)
    x = rng.standard_normal((T, d)) * np.exp2(rng.uniform(-8, 8, (T, 1)))
    x[0, :4] = [-0.0, 0.0, 1e-7 * np.abs(x[0]).max(), -1e-7 * np.abs(x[0]).max()]
    if T >= 3:
        x[1] = 0.0
        x[2] = 0.0
        x[2, d // 2] = -3.0
    xb = W.to_bf16(x)
    codes, scale = sn.sn_quant_compress(dev(xb), fmt)
    rc, rs = o.quant_compress(xb, fmt)
    assert np.array_equal(host(codes), rc)
    assert np.array_equal(host(scale).view(np.uint32), rs.view(np.uint32))
    back = sn.sn_quant_restore(codes, scale, fmt)
    assert np.array_equal(host(back), o.quant_restore(rc, rs, fmt))


def test_quant_argument_errors(sn):
    X = torch.zeros(4, 64, dtype=torch.bfloat16, device="cuda")
    codes = torch.empty(4, 64, dtype=torch.uint8, device="cuda")
    scale = torch.empty(4, dtype=torch.float32, device="cuda")
    lib = sn._lib
    st = lib.sn_quant_compress(X.data_ptr(), 4, 64, 2, codes.data_ptr(), scale.data_ptr(), None)
    assert st == sn.SN_ERR_INVALID_ARG                  # unknown format
    st = lib.sn_quant_compress(X.data_ptr(), 4, 64, 0, codes.data_ptr() + 4, scale.data_ptr(),
                               None)
    assert st == sn.SN_ERR_ALIGNMENT                    # codes not 8-byte aligned
    st = lib.sn_quant_restore(codes.data_ptr(), scale.data_ptr(), 4, 60, 1, X.data_ptr(), None)
    assert st == sn.SN_ERR_INVALID_ARG                  # d % 8
    st = lib.sn_quant_compress(X.data_ptr(), 4, 64, 1, X.data_ptr(), scale.data_ptr(), None)
    assert st == sn.SN_ERR_INVALID_ARG                  # codes overlap X
