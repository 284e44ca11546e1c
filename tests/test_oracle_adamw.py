"""Pins of the row-constant AdamW oracle (Sec. 5) against mathematics that does
not come from the oracle itself: torch's own AdamW (a library routine) in the
case where the row-constant rule changes nothing, the closure of the update in
the subspace S, and the first step written out by hand.  Each plausible mistake
(the garbled bias correction, the mean over the wrong axis, the square root,
weight decay scaled by the learning rate, a stale moment) fails at least one
of them (see the mutants below)."""
import importlib.util
import os

import numpy as np
import pytest
import torch

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "..", "oracle", "adamw.py")
HP = dict(lr=0.01, beta1=0.9, beta2=0.99, eps=1e-6, lam=1e-3)


def load(text=None):
    spec = importlib.util.spec_from_loader("adamw_under_test", loader=None)
    mod = importlib.util.module_from_spec(spec)
    exec(compile(text if text is not None else open(SRC).read(), SRC, "exec"), mod.__dict__)
    return mod


def run(a, W, grads):
    M = np.zeros_like(W)
    V = np.zeros_like(W)
    for t, g in enumerate(grads, 1):
        W, M, V = a.step(W, g, M, V, t, HP["lr"], HP["beta1"], HP["beta2"], HP["eps"], HP["lam"])
    return W


def pin_matches_torch_adamw_when_columns_are_constant(a):
    # |g| constant down each column at every step: V^ is already constant per
    # column, the row-constant rule is the identity and the step is AdamW's
    rng = np.random.default_rng(0)
    d, n = 16, 6
    W0 = rng.standard_normal((d, n))
    grads = [rng.choice([-1.0, 1.0], (d, n)) * rng.uniform(0.5, 2.0, (1, n)) for _ in range(4)]
    Wt = torch.tensor(W0, dtype=torch.float64, requires_grad=True)
    opt = torch.optim.AdamW([Wt], lr=HP["lr"], betas=(HP["beta1"], HP["beta2"]), eps=HP["eps"],
                            weight_decay=HP["lam"] / HP["lr"])
    for g in grads:
        Wt.grad = torch.tensor(g, dtype=torch.float64)
        opt.step()
    return np.allclose(run(a, W0, grads), Wt.detach().numpy(), rtol=1e-12, atol=1e-12)


def pin_update_stays_in_subspace(a):
    rng = np.random.default_rng(1)
    d, k, n = 32, 4, 10
    Q, R = np.linalg.qr(rng.standard_normal((d, k)))
    U = Q * np.sign(np.diag(R))
    W0 = U @ rng.standard_normal((k, n))                      # columns in S
    grads = [U @ rng.standard_normal((k, n)) for _ in range(5)]
    W = run(a, W0, grads)
    out = W - U @ (U.T @ W)
    return np.linalg.norm(out) <= 1e-12 * np.linalg.norm(W)


def pin_first_step_by_hand(a):
    rng = np.random.default_rng(2)
    d, n = 5, 3
    W0 = rng.standard_normal((d, n))
    g = rng.standard_normal((d, n))
    W1, M1, V1 = a.step(W0, g, np.zeros_like(W0), np.zeros_like(W0), 1, HP["lr"], HP["beta1"],
                        HP["beta2"], HP["eps"], HP["lam"])
    expect = np.empty_like(W0)
    for c in range(n):
        mean_g2 = sum(g[r, c] ** 2 for r in range(d)) / d     # V^ = g^2 after one step
        for r in range(d):
            expect[r, c] = (W0[r, c] - HP["lr"] * g[r, c] / (np.sqrt(mean_g2) + HP["eps"])
                            - HP["lam"] * W0[r, c])
    return (np.allclose(W1, expect, rtol=1e-13, atol=1e-13)
            and np.allclose(M1, (1 - HP["beta1"]) * g) and np.allclose(V1, (1 - HP["beta2"]) * g * g))


PINS = [pin_matches_torch_adamw_when_columns_are_constant, pin_update_stays_in_subspace,
        pin_first_step_by_hand]


@pytest.mark.parametrize("pin", PINS, ids=[p.__name__ for p in PINS])
def test_adamw_oracle_pins(pin):
    assert pin(load())


def test_plain_adamw_leaves_the_subspace():
    """Why the rule exists: torch's element-wise AdamW moves W out of S."""
    rng = np.random.default_rng(1)
    d, k, n = 32, 4, 10
    Q, _ = np.linalg.qr(rng.standard_normal((d, k)))
    W0 = Q @ rng.standard_normal((k, n))
    Wt = torch.tensor(W0, requires_grad=True)
    opt = torch.optim.AdamW([Wt], lr=HP["lr"], betas=(HP["beta1"], HP["beta2"]), eps=HP["eps"])
    for _ in range(5):
        Wt.grad = torch.tensor(Q @ rng.standard_normal((k, n)))
        opt.step()
    W = Wt.detach().numpy()
    assert np.linalg.norm(W - Q @ (Q.T @ W)) > 1e-4 * np.linalg.norm(W)


MUTANTS = {
    "garbled_bias_correction": ("Vhat = V / (1.0 - beta2 ** t)", "Vhat = V / (beta2 + eps)"),
    "mean_over_rows": ("mu = Vhat.mean(axis=0)", "mu = Vhat.mean(axis=1)[:, None]"),
    "no_square_root": ("alpha = 1.0 / (np.sqrt(mu) + eps)", "alpha = 1.0 / (mu + eps)"),
    "decay_times_lr": ("- lam * W", "- lr * lam * W"),
    "first_moment_bias": ("Mhat = M / (1.0 - beta1 ** t)", "Mhat = M"),
    "stale_second_moment": ("V = beta2 * np.asarray(V, np.float64) + (1.0 - beta2) * g * g",
                            "V = beta2 * np.asarray(V, np.float64) + (1.0 - beta2) * np.asarray(M, np.float64) ** 2"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_adamw_mutants_are_caught(name):
    a_, b_ = MUTANTS[name]
    text = open(SRC).read()
    assert a_ in text
    mod = load(text.replace(a_, b_))
    failed = []
    for pin in PINS:
        try:
            ok = pin(mod)
        except Exception:
            ok = False
        if not ok:
            failed.append(pin.__name__)
    assert failed, "mutant %s passed every pin" % name
