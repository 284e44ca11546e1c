"""The GPU tests' parity bar (gpu_util.assert_parity) on planted mistakes, on the
CPU: a result that differs from the reference only by one bf16 rounding per
element passes; a zeroed row, a wrong 128-column block inside one d = 8192 row,
two swapped rows, or a nonzero row where the reference row is zero fail, in
shapes where the whole-tensor relative Frobenius error alone stays under its
bar.
"""
import numpy as np
import pytest

from gpu_util import ROW_TOL, TOL, assert_parity, rel_fro, row_rel_max
from paper_2506_01260_gb300 import workloads as W


def reference(rows, cols, seed):
    return np.random.default_rng(seed).standard_normal((rows, cols))


def bf16(x):
    """Rounded once to bf16: what a correct kernel returns."""
    return W.to_bf16(x)


def test_one_rounding_passes():
    ref = reference(512, 8192, 0)
    fro, row = assert_parity(bf16(ref), ref, "bf16")
    assert fro < 3e-3 and row < 4e-3


def test_zeroed_row_fails():
    ref = reference(16384, 256, 1)
    got = bf16(ref)
    got[17] = 0
    assert rel_fro(got, ref) <= TOL["bf16"]          # the tensor norm alone would pass
    with pytest.raises(AssertionError):
        assert_parity(got, ref, "bf16")


def test_wrong_column_block_inside_one_row_fails():
    ref = reference(512, 8192, 2)
    got = bf16(ref)
    got[201, 4096:4224] = 0                         # one 128-column block of one token
    assert rel_fro(got, ref) <= TOL["bf16"]
    assert row_rel_max(got, ref) > ROW_TOL["bf16"]
    with pytest.raises(AssertionError):
        assert_parity(got, ref, "bf16")


def test_swapped_rows_fail():
    ref = reference(65536, 64, 3)
    got = bf16(ref)
    got[[5, 6]] = got[[6, 5]]
    assert rel_fro(got, ref) <= TOL["bf16"]
    with pytest.raises(AssertionError):
        assert_parity(got, ref, "bf16")


def test_row_that_must_be_zero():
    ref = reference(256, 512, 4)
    ref[9] = 0                                      # e.g. a token with an invalid id
    got = bf16(ref)
    assert_parity(got, ref, "bf16")
    got[9, 0] = W.f32_to_bf16_bits(np.array([1e-3], np.float32))[0]
    assert row_rel_max(got, ref) == float("inf")
    with pytest.raises(AssertionError):
        assert_parity(got, ref, "bf16")


def test_fp32_bar():
    ref = reference(64, 1024, 5)
    got = ref.astype(np.float32)
    assert_parity(got, ref, "f32")
    got[3, :8] += 0.05
    with pytest.raises(AssertionError):
        assert_parity(got, ref, "f32")
