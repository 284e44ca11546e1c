"""fp64 oracle of the row-constant AdamW step for W_p2 (Sec. 5).

TEST INFRASTRUCTURE ONLY.  Only the tests may import this module; it shares no
code with the CUDA library.  Plain numpy in fp64.

Layout: the torch weight W is [d, n] (d = model width, n = d_ff); its columns
are the rows of the paper's W_p2 in R^{n x d}, i.e. the d-vectors that must stay
in S.  The paper's row-wise mean (over the m = d entries of a row of W_p2) is
therefore a mean over the d entries of each torch column.

One step, in the paper's order, with t >= 1 the step number:
  M_t  = beta1 M_{t-1} + (1 - beta1) g                          Sec. 5
  V_t  = beta2 V_{t-1} + (1 - beta2) g^2                        Sec. 5
  M^   = M_t / (1 - beta1^t),  V^ = V_t / (1 - beta2^t)         bias correction (reading)
  mu   = mean of V^ over each column (the paper's row mean)     Sec. 5
  alpha= 1 / (sqrt(mu) + eps), one value per column             Sec. 5
  W    = W - eta alpha M^ - lambda W                            Sec. 5, eq. (weight_update)
Reading: the paper prints the bias correction as V_t / (beta2 + eps) (and the
same for M); that garbles the standard AdamW correction 1 - beta^t, which is
used here.  Weight decay is the paper's -lambda W (torch's AdamW has
-lr * weight_decay * W, i.e. lambda = lr * weight_decay).
"""
import numpy as np


def step(W, g, M, V, t, lr, beta1, beta2, eps, lam):
    """One row-constant AdamW step; returns (W, M, V) as new fp64 arrays."""
    W = np.asarray(W, np.float64)
    g = np.asarray(g, np.float64)
    M = beta1 * np.asarray(M, np.float64) + (1.0 - beta1) * g
    V = beta2 * np.asarray(V, np.float64) + (1.0 - beta2) * g * g
    Mhat = M / (1.0 - beta1 ** t)
    Vhat = V / (1.0 - beta2 ** t)
    mu = Vhat.mean(axis=0)                       # one value per column of W
    alpha = 1.0 / (np.sqrt(mu) + eps)
    W = W - lr * Mhat * alpha[None, :] - lam * W
    return W, M, V
