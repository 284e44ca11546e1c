"""fp64 oracle of the subspace update on the Grassmann manifold (Sec. 4.5, Sec. 6).

TEST INFRASTRUCTURE ONLY.  Only the tests may import this module; it shares no
code with the CUDA library.  Plain numpy in fp64; a library QR serves as the
retraction step.

Definitions, in the paper's order:
  leftover gradient   G (I - U U^T)                               Sec. 4.5
  Grassmann loss      L(U) = (1/K) sum_t ||G_t (I - U U^T)||_F^2     Sec. 4.5
  accumulation        S = (1/K) sum_t G_t^T G_t                     Sec. 6
  Euclidean gradient  -2 S U                                       Sec. 6
  Riemannian grad.    g - U (U^T g)                                Sec. 4.5
  step                U - eta * tangent                            Sec. 4.5
  retraction          Q of the QR decomposition (diag(R) > 0)      Sec. 4.5
Because U only changes at a step, S U is accumulated as M = sum_t G_t^T (G_t U)
(G_t U is the compressed gradient of Eq. (grad_compress)), so the [d, d]
matrix S is never formed: S U = M / K.
"""
import numpy as np


def leftover(G, U):
    """G (I - U U^T): the part of the gradient outside the subspace."""
    G = np.asarray(G, np.float64)
    U = np.asarray(U, np.float64)
    return G - (G @ U) @ U.T


def residual(G, U):
    """||G (I - U U^T)||_F^2 of one gradient."""
    R = leftover(G, U)
    return float(np.sum(R * R))


def loss(Gs, U):
    """L(U) = (1/K) sum_t ||G_t (I - U U^T)||_F^2 over the K gradients Gs."""
    return sum(residual(G, U) for G in Gs) / len(Gs)


def accumulation_matrix(Gs):
    """S = (1/K) sum_t G_t^T G_t (the symmetric [d, d] matrix of Sec. 6)."""
    S = sum(np.asarray(G, np.float64).T @ np.asarray(G, np.float64) for G in Gs)
    return S / len(Gs)


def accumulate(M, G, U):
    """M + G^T (G U): one iteration's contribution to K * S U."""
    G = np.asarray(G, np.float64)
    return np.asarray(M, np.float64) + G.T @ (G @ np.asarray(U, np.float64))


def accumulate_rows(M_rows, G, U, rows):
    """Rows `rows` of M + G^T (G U) alone: M_rows + G[:, rows]^T (G U).  The
    same sum as `accumulate`, for checking a large accumulation on sampled
    rows (G U still needs every column of G)."""
    G = np.asarray(G, np.float64)
    return np.asarray(M_rows, np.float64) + G[:, rows].T @ (G @ np.asarray(U, np.float64))


def euclidean_grad(M, K):
    """-2 S U with S U = M / K."""
    return -2.0 * np.asarray(M, np.float64) / K


def tangent(g, U):
    """Projection of a Euclidean gradient onto the tangent space at U."""
    U = np.asarray(U, np.float64)
    return g - U @ (U.T @ g)


def retract(A):
    """Orthonormal basis of Col(A): Q of A = QR with the diagonal of R positive."""
    Q, R = np.linalg.qr(np.asarray(A, np.float64))
    s = np.sign(np.diag(R))
    s[s == 0] = 1.0
    return Q * s


def step(U, M, K, eta):
    """One Grassmann step: U - eta * tangent(-2 M / K), retracted."""
    U = np.asarray(U, np.float64)
    return retract(U - eta * tangent(euclidean_grad(M, K), U))
