"""Pins of the Grassmann-update oracle (Sec. 4.5, Sec. 6) against mathematics
that does not come from the oracle itself: finite differences, a brute-force
accumulation matrix, the trace identity of the loss, the tangent space, the QR
factorisation, descent, the fixed point of an in-subspace gradient, and the
minimiser of the loss (the dominant eigen-subspace of S, from numpy's eigh).
Each plausible mistake in the oracle (a sign, a factor, a transpose, a missing
projection or sign fix) fails at least one of them (see the mutants below)."""
import importlib.util
import os

import numpy as np
import pytest

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "..", "oracle", "grassmann.py")


def load(text=None):
    spec = importlib.util.spec_from_loader("grassmann_under_test", loader=None)
    mod = importlib.util.module_from_spec(spec)
    exec(compile(text if text is not None else open(SRC).read(), SRC, "exec"), mod.__dict__)
    return mod


def orth(rng, d, k):
    Q, R = np.linalg.qr(rng.standard_normal((d, k)))
    return Q * np.sign(np.diag(R))


def problem(seed=0, d=24, k=3, K=4, T=10):
    rng = np.random.default_rng(seed)
    Gs = [rng.standard_normal((T, d)) for _ in range(K)]
    return rng, Gs, orth(rng, d, k)


def pin_finite_difference(g):
    rng, Gs, U = problem(1)
    A = rng.standard_normal(U.shape)                 # any U, not only orthonormal ones
    M = np.zeros_like(A)
    for G in Gs:
        M = g.accumulate(M, G, A)
    grad = g.euclidean_grad(M, len(Gs))
    S = sum(G.T @ G for G in Gs) / len(Gs)
    f = lambda X: -np.trace(X.T @ S @ X)             # loss up to a constant in U
    h, num = 1e-6, np.zeros_like(A)
    for i in range(A.shape[0]):
        for j in range(A.shape[1]):
            E = np.zeros_like(A)
            E[i, j] = h
            num[i, j] = (f(A + E) - f(A - E)) / (2 * h)
    return np.max(np.abs(grad - num)) <= 1e-5 * max(1.0, np.max(np.abs(num)))


def pin_accumulation(g):
    _, Gs, U = problem(2)
    M = np.zeros_like(U)
    for G in Gs:
        M = g.accumulate(M, G, U)
    S = sum(G.T @ G for G in Gs) / len(Gs)           # brute force, written out here
    return (np.allclose(M / len(Gs), S @ U, rtol=1e-12, atol=1e-12)
            and np.allclose(g.accumulation_matrix(Gs), S, rtol=1e-12, atol=1e-12))


def pin_accumulation_rows(g):
    rng, Gs, U = problem(9)
    rows = np.array([0, 5, 6, 23])
    M0 = rng.standard_normal((len(rows), U.shape[1]))
    Mr = M0.copy()
    for G in Gs:
        Mr = g.accumulate_rows(Mr, G, U, rows)
    S = sum(G.T @ G for G in Gs)                     # brute force, written out here
    return np.allclose(Mr, M0 + (S @ U)[rows], rtol=1e-12, atol=1e-12)


def pin_loss_trace(g):
    _, Gs, U = problem(3)
    S = sum(G.T @ G for G in Gs) / len(Gs)
    const = sum(np.sum(G * G) for G in Gs) / len(Gs)
    return abs(g.loss(Gs, U) - (const - np.trace(U.T @ S @ U))) <= 1e-9 * const


def pin_tangent(g):
    rng, Gs, U = problem(4)
    X = rng.standard_normal(U.shape)
    t = g.tangent(X, U)
    return np.max(np.abs(U.T @ t)) <= 1e-12 and np.allclose(g.tangent(t, U), t, atol=1e-12)


def pin_retraction(g):
    rng = np.random.default_rng(5)
    A = rng.standard_normal((20, 4))
    Q = g.retract(A)
    R = Q.T @ A
    return (np.allclose(Q.T @ Q, np.eye(4), atol=1e-12)
            and np.allclose(np.tril(R, -1), 0, atol=1e-12)
            and np.all(np.diag(R) > 0)
            and np.allclose(Q @ R, A, atol=1e-12))


def pin_descent(g):
    _, Gs, U = problem(6)
    M = np.zeros_like(U)
    for G in Gs:
        M = g.accumulate(M, G, U)
    U1 = g.step(U, M, len(Gs), 1e-3)
    return g.loss(Gs, U1) < g.loss(Gs, U) and np.allclose(U1.T @ U1, np.eye(U.shape[1]), atol=1e-12)


def pin_in_subspace_fixed_point(g):
    rng, _, U = problem(7)
    Gs = [rng.standard_normal((10, U.shape[1])) @ U.T for _ in range(3)]   # rows in Col(U)
    M = np.zeros_like(U)
    for G in Gs:
        M = g.accumulate(M, G, U)
    ok_res = all(g.residual(G, U) <= 1e-20 * max(1.0, np.sum(G * G)) for G in Gs)
    U1 = g.step(U, M, len(Gs), 0.5)
    return ok_res and np.allclose(U1, U, atol=1e-10)


def pin_converges_to_top_eigenspace(g):
    rng, Gs, U = problem(8, d=16, k=2, K=3, T=40)
    S = sum(G.T @ G for G in Gs) / len(Gs)
    w, V = np.linalg.eigh(S)
    P_top = V[:, -2:] @ V[:, -2:].T
    eta = 0.25 / w[-1]
    for _ in range(400):
        M = np.zeros_like(U)
        for G in Gs:
            M = g.accumulate(M, G, U)
        U = g.step(U, M, len(Gs), eta)
    return np.max(np.abs(U @ U.T - P_top)) <= 1e-6


PINS = [pin_finite_difference, pin_accumulation, pin_accumulation_rows, pin_loss_trace, pin_tangent, pin_retraction,
        pin_descent, pin_in_subspace_fixed_point, pin_converges_to_top_eigenspace]


@pytest.mark.parametrize("pin", PINS, ids=[p.__name__ for p in PINS])
def test_grassmann_oracle_pins(pin):
    assert pin(load())


MUTANTS = {
    "gradient_sign": ("return -2.0 * np.asarray(M, np.float64) / K",
                      "return 2.0 * np.asarray(M, np.float64) / K"),
    "gradient_factor": ("return -2.0 * np.asarray(M, np.float64) / K",
                        "return -1.0 * np.asarray(M, np.float64) / K"),
    "accumulate_forgets_sum": ("return np.asarray(M, np.float64) + G.T @ (G @ np.asarray(U, np.float64))",
                               "return G.T @ (G @ np.asarray(U, np.float64))"),
    "accumulate_gram_of_rows": ("return np.asarray(M, np.float64) + G.T @ (G @ np.asarray(U, np.float64))",
                                "return np.asarray(M, np.float64) + (G.T @ G).T @ np.asarray(U, np.float64) * (G.shape[0] / G.shape[1])"),
    "rows_forget_sum": ("return np.asarray(M_rows, np.float64) + G[:, rows].T @ (G @ np.asarray(U, np.float64))",
                        "return G[:, rows].T @ (G @ np.asarray(U, np.float64))"),
    "rows_transposed": ("return np.asarray(M_rows, np.float64) + G[:, rows].T @ (G @ np.asarray(U, np.float64))",
                        "return np.asarray(M_rows, np.float64) + (G.T @ (G @ np.asarray(U, np.float64)))[rows[::-1]]"),
    "tangent_missing": ("return g - U @ (U.T @ g)", "return g"),
    "tangent_sign": ("return g - U @ (U.T @ g)", "return g + U @ (U.T @ g)"),
    "retract_no_sign_fix": ("return Q * s", "return Q"),
    "leftover_sign": ("return G - (G @ U) @ U.T", "return G + (G @ U) @ U.T"),
    "step_sign": ("return retract(U - eta * tangent(euclidean_grad(M, K), U))",
                  "return retract(U + eta * tangent(euclidean_grad(M, K), U))"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_grassmann_mutants_are_caught(name):
    a, b = MUTANTS[name]
    text = open(SRC).read()
    assert a in text
    g = load(text.replace(a, b))
    failed = []
    for pin in PINS:
        try:
            ok = pin(g)
        except Exception:
            ok = False
        if not ok:
            failed.append(pin.__name__)
    assert failed, "mutant %s passed every pin" % name
