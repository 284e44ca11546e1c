"""Pins of the lossy-comparator oracle against cases whose answer is known
without it: a row with planted large entries (top-k), ties, a row of +-c (sign
quantization is then exact), an exactly low-rank batch (the truncated SVD
recovers it) and the Eckart-Young error of the truncated SVD (the sum of the
discarded squared singular values, from numpy's eigvalsh of X^T X)."""
import importlib.util
import os

import numpy as np
import pytest

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "..", "oracle", "lossy.py")


def load(text=None):
    spec = importlib.util.spec_from_loader("lossy_under_test", loader=None)
    mod = importlib.util.module_from_spec(spec)
    exec(compile(text if text is not None else open(SRC).read(), SRC, "exec"), mod.__dict__)
    return mod


def bf16(x):
    x = np.asarray(x, np.float32)
    u = x.view(np.uint32)
    return ((u + 0x7FFF + ((u >> 16) & 1)) >> 16).astype(np.uint16)


def pin_topk_planted(o):
    rng = np.random.default_rng(0)
    x = rng.uniform(-1, 1, (3, 40))
    planted = [[3, 17, 29], [0, 1, 39], [5, 6, 7]]
    for t, cs in enumerate(planted):
        for j, c in enumerate(cs):
            x[t, c] = (10 + j) * (-1) ** j
    cols = o.topk_columns(bf16(x), 3)
    return all(list(cols[t]) == sorted(planted[t]) for t in range(3))


def pin_topk_ties_lower_index(o):
    x = np.array([[1.0, -2.0, 2.0, 0.5, -2.0, 2.0]])
    return list(o.topk_columns(bf16(x), 2)[0]) == [1, 2]


def pin_topk_restore(o):
    vals = np.array([[5.0, -7.0]])
    X = o.topk_restore(vals, np.array([[1, 3]]), 5)
    return np.array_equal(X, np.array([[0, 5.0, 0, -7.0, 0]]))


def pin_sign_exact_on_pm_c(o):
    rng = np.random.default_rng(1)
    c = rng.uniform(0.5, 2, (4, 1))
    X = c * rng.choice([-1.0, 1.0], (4, 33))
    bits, scale = o.sign_compress(X)
    return np.allclose(o.sign_restore(bits, scale), X, rtol=0, atol=1e-15) and bits.dtype == np.uint8


def pin_sign_scale_is_mean_magnitude(o):
    bits, scale = o.sign_compress(np.array([[1.0, -3.0, 0.0, 4.0]]))
    return list(bits[0]) == [0, 1, 0, 0] and abs(scale[0] - 2.0) <= 1e-15


def pin_lowrank_recovers_rank_r(o):
    rng = np.random.default_rng(2)
    X = rng.standard_normal((50, 4)) @ rng.standard_normal((4, 30))
    return np.allclose(o.lowrank(X, 4), X, atol=1e-10)


def pin_lowrank_eckart_young(o):
    rng = np.random.default_rng(3)
    X = rng.standard_normal((40, 25))
    ev = np.sort(np.linalg.eigvalsh(X.T @ X))          # squared singular values, ascending
    err2 = np.sum((X - o.lowrank(X, 6)) ** 2)
    return abs(err2 - ev[:-6].sum()) <= 1e-8 * ev.sum()


def pin_wire_sizes(o):
    return (o.wire_bytes("subspace", 10, 8192, k=82) == 1640
            and o.wire_bytes("topk", 10, 8192, kk=41) == 1640
            and o.wire_bytes("sign", 10, 8192) == 10 * 1024 + 40
            and o.wire_bytes("lowrank", 10, 8192, r=2) == 4 * 8202)


PINS = [pin_topk_planted, pin_topk_ties_lower_index, pin_topk_restore, pin_sign_exact_on_pm_c,
        pin_sign_scale_is_mean_magnitude, pin_lowrank_recovers_rank_r, pin_lowrank_eckart_young, pin_wire_sizes]


@pytest.mark.parametrize("pin", PINS, ids=[p.__name__ for p in PINS])
def test_lossy_oracle_pins(pin):
    assert pin(load())


MUTANTS = {
    "ties_higher_index": ("key=lambda c: (-mag[t, c], c)", "key=lambda c: (-mag[t, c], -c)"),
    "smallest_magnitudes": ("key=lambda c: (-mag[t, c], c)", "key=lambda c: (mag[t, c], c)"),
    "sign_of_positive": ("(X < 0).astype(np.uint8)", "(X > 0).astype(np.uint8)"),
    "scale_rms": ("np.abs(X).mean(axis=1)", "np.sqrt((X * X).mean(axis=1))"),
    "lowrank_off_by_one": ("(Uu[:, :r] * s[:r]) @ Vt[:r]", "(Uu[:, :r - 1] * s[:r - 1]) @ Vt[:r - 1]"),
    "index_bytes": ("return T * kk * (2 + 2)", "return T * kk * (2 + 4)"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_lossy_mutants_are_caught(name):
    a, b = MUTANTS[name]
    text = open(SRC).read()
    assert a in text
    mod = load(text.replace(a, b))
    failed = []
    for pin in PINS:
        try:
            ok = pin(mod)
        except Exception:
            ok = False
        if not ok:
            failed.append(pin.__name__)
    assert failed, "mutant %s passed every pin" % name
