"""Regularizer-only descent and the spectral-energy metric, fp64 numpy (oracle;
test infrastructure only).

Follows, in the paper's notation:

* Alg. 1 (App. C.2, decoupled SLORR), last line: W <- W - eta lambda G_pre,
  with G_pre the SLORR gradient at the weights before the step.  With no task
  update in between this is the "regularizer-only gradient step" that Props. 2
  and 3 (Sec. 3.1) reason about.  Here G_pre is the Polar Express gradient of
  ``oracle.slorr.reg_single`` (Listing 1 backward), scaled by grad_scale as in
  Alg. 2.
* Prop. 2: the threshold tau = ||W||_F^2 / ||W||_*; under a small enough
  regularizer-only SLORR-Hoyer step, singular values above tau grow and those
  below shrink.
* App. D.4, energy truncation: E(P) = sum_{i<=P} sigma_i^2 / sum_{i<=R} sigma_i^2
  (R = min(M, N), sigma sorted descending) and P* = min{P : E(P) >= rho}.
  Prop. 3 states that the relative tail error 1 - E(k) falls under the step
  for every k with sigma_k > tau.
"""

from __future__ import annotations

import numpy as np

from .slorr import reg_single


def descent_step(W, eta: float, variant: str, coeffs, lam: float = 1.0, grad_scale: float = 1.0,
                 eps: float = 1e-7):
    """One regularizer-only step: returns (W_plus, L) with
    W_plus = W - eta * lam * grad_scale * G_hat(W) and L the unweighted value at W."""
    W = np.asarray(W, dtype=np.float64)
    L, G, _, _ = reg_single(W, variant, coeffs, eps)
    return W - (eta * lam * grad_scale) * G, L


def descent_trajectory(W, eta: float, steps: int, variant: str, coeffs, lam: float = 1.0,
                       grad_scale: float = 1.0, eps: float = 1e-7):
    """`steps` successive descent steps from W: returns ([W_0, ..., W_steps], [L(W_0), ..., L(W_{steps-1})])."""
    Ws = [np.asarray(W, dtype=np.float64).copy()]
    Ls = []
    for _ in range(int(steps)):
        Wn, L = descent_step(Ws[-1], eta, variant, coeffs, lam, grad_scale, eps)
        Ws.append(Wn)
        Ls.append(L)
    return Ws, Ls


def singular_values(W) -> np.ndarray:
    """sigma_1 >= ... >= sigma_R of W (numpy's SVD, fp64)."""
    return np.linalg.svd(np.asarray(W, dtype=np.float64), compute_uv=False)


def hoyer_tau(W) -> float:
    """tau = ||W||_F^2 / ||W||_* (Prop. 2)."""
    s = singular_values(W)
    return float(np.sum(s * s) / np.sum(s))


def energy(W, P: int) -> float:
    """Retained energy E(P) of the rank-P truncation (App. D.4)."""
    s = singular_values(W)
    P = int(min(max(P, 0), s.size))
    tot = float(np.sum(s * s))
    return float(np.sum(s[:P] ** 2) / tot) if tot > 0 else 1.0


def energy_rank(W, rho: float) -> int:
    """P* = min{P : E(P) >= rho} (App. D.4); R when no smaller P qualifies."""
    s = singular_values(W)
    tot = float(np.sum(s * s))
    if tot == 0.0:
        return 0
    for P in range(1, s.size + 1):
        if float(np.sum(s[:P] ** 2)) / tot >= rho:
            return P
    return int(s.size)
