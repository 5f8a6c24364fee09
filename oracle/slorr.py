"""SLORR regularizer value and gradient, fp64 numpy (oracle; test infrastructure only).

Follows, in order and in the paper's notation:

* Sec. 3 problem statement: L_hoyer = sum_i ||W_i||_*^2 / ||W_i||_F^2,
  L_nuc = sum_i ||W_i||_*;
* Eq. 1: grad L_hoyer = 2 (n/f) (U V^T / f - n W / f^3), grad L_nuc = U V^T;
* Sec. 3 "Computing the polar factor": P_hat = Polar Express applied to
  W / (||W||_F + eps);
* Sec. 3 "Computing the nuclear and Frobenius norms": n_hat = sum(W * P_hat);
* Listing 1 (forward/backward with eps substituted separately):
  frob = ||W||_F + eps, reg = n_hat / frob, value reg^2,
  G = P_hat / frob - n_hat / frob^3 W, gradient 2 reg G (times the incoming
  gradient, here lambda);
* Alg. 2 (memory-efficient loop): W.grad <- W.grad + lambda * G_hat(W);
* Sec. 3 "Computational cost": per step 4 P^2 Q + 2 P^3 FLOPs with
  P = min(M, N), Q = max(M, N), which fixes the Gram-side form of the
  iteration: X is P x Q (X = W^T when M > N), A = X X^T,
  B = b A + c A^2, X <- a X + B X.

Readings where the paper is silent: eps = 1e-7 and the same eps is used in the
normalisation and in frob; for M > N the iteration runs on W^T and the result
is transposed back; SLORR-Nuc uses value n_hat and gradient P_hat; lambda
scales both the loss and the gradient, grad_scale scales the gradient only.
"""

from __future__ import annotations

import numpy as np


def frobenius(W) -> float:
    """||W||_F = sqrt(sum_ij W_ij^2) in fp64."""
    W = np.asarray(W, dtype=np.float64)
    return float(np.sqrt(np.sum(W * W)))


def polar_express_steps(W, coeffs, eps: float = 1e-7):
    """Polar Express on the Gram (min) side, returning every iterate.

    Returns (list of X_t in the P x Q orientation for t = 0..T, transposed flag).
    X_0 = W / (||W||_F + eps) (transposed first when M > N)."""
    W = np.asarray(W, dtype=np.float64)
    m, n = W.shape
    transposed = m > n
    X = (W.T if transposed else W) / (frobenius(W) + eps)
    out = [X.copy()]
    for a, b, c in np.asarray(coeffs, dtype=np.float64):
        A = X @ X.T
        B = b * A + c * (A @ A)
        X = a * X + B @ X
        out.append(X.copy())
    return out, transposed


def polar_express(W, coeffs, eps: float = 1e-7):
    """P_hat, the Polar Express approximation of U V^T, in W's orientation."""
    steps, transposed = polar_express_steps(W, coeffs, eps)
    X = steps[-1]
    return X.T.copy() if transposed else X


def reg_single(W, variant: str, coeffs, eps: float = 1e-7):
    """One matrix: returns (L_i, G_hat_i, n_hat, frob).

    L_i is the unweighted value (reg^2 for Hoyer, n_hat for Nuc) and G_hat_i
    its approximate gradient (Listing 1 backward with grad_output = 1)."""
    W = np.asarray(W, dtype=np.float64)
    P_hat = polar_express(W, coeffs, eps)
    n_hat = float(np.sum(W * P_hat))
    frob = frobenius(W) + eps
    if variant == "hoyer":
        reg = n_hat / frob
        G = P_hat / frob - (n_hat / frob ** 3) * W
        return reg * reg, 2.0 * reg * G, n_hat, frob
    if variant == "nuclear":
        return n_hat, P_hat, n_hat, frob
    raise ValueError("variant must be 'hoyer' or 'nuclear'")


def reg_forward_backward(weights, variant: str, coeffs, lam: float,
                         eps: float = 1e-7, grad_scale: float = 1.0):
    """Whole weight set (Alg. 2 semantics).

    Returns (loss, per_matrix, grad_increments) where
      loss            = lam * sum_i L_i,
      per_matrix[i]   = L_i (unweighted),
      grad_increments = [lam * grad_scale * G_hat_i], to be added to W_i.grad."""
    per = []
    incs = []
    for W in weights:
        L, G, _, _ = reg_single(W, variant, coeffs, eps)
        per.append(L)
        incs.append((lam * grad_scale) * G)
    per = np.array(per, dtype=np.float64)
    return float(lam * per.sum()), per, incs


def exact_values(W, rel_tol: float = 1e-12):
    """Exact (n, f, hoyer, P = U V^T) by numpy's SVD (Sec. 3 problem statement).

    U V^T is restricted to singular values above rel_tol * sigma_max (thin SVD
    over the nonzero singular values, Sec. 3 footnote on the generalized polar
    factor)."""
    W = np.asarray(W, dtype=np.float64)
    U, s, Vt = np.linalg.svd(W, full_matrices=False)
    keep = s > rel_tol * (s[0] if s.size and s[0] > 0 else 1.0)
    n = float(s.sum())
    f = float(np.sqrt((s * s).sum()))
    P = (U[:, keep] * 1.0) @ Vt[keep, :]
    hoyer = n * n / (f * f) if f > 0 else 0.0
    return n, f, hoyer, P


def exact_grad(W, variant: str, rel_tol: float = 1e-12):
    """Eq. 1 with the exact polar factor (no eps)."""
    n, f, _, P = exact_values(W, rel_tol)
    W = np.asarray(W, dtype=np.float64)
    if variant == "nuclear":
        return P
    if variant == "hoyer":
        return 2.0 * (n / f) * (P / f - (n / f ** 3) * W)
    raise ValueError("variant must be 'hoyer' or 'nuclear'")


def pe_flops(m: int, n: int, T: int = 6) -> int:
    """T * (4 P^2 Q + 2 P^3) with P = min(m, n), Q = max(m, n) (Sec. 3)."""
    P, Q = min(m, n), max(m, n)
    return int(T) * (4 * P * P * Q + 2 * P ** 3)


def weight_set_flops(shapes, T: int = 6) -> int:
    """Sum of pe_flops over a weight set."""
    return sum(pe_flops(m, n, T) for m, n in shapes)
