"""Pins for the oracle's regularizer-only descent step and energy metric
(Alg. 1 last line, Props. 2 and 3 of Sec. 3.1, App. D.4).

Each pin reaches the function through a route other than its own code: an
independent Jacobi SVD, the closed form of Prop. 2's proof, the per-singular-
value form of the Polar Express gradient (the scalar map, pinned on its own in
the schedule tests), and brute force.  A plausible slip -- sigma instead of
sigma^2 in E(P), a wrong sign or a dropped lambda / grad_scale in the step, the
wrong threshold -- fails at least one of them."""

import numpy as np
import pytest

import oracle
from oracle import svd_jacobi

CO = oracle.pe_coefficients(T=6)
EPS = 1e-7


def _with_spectrum(m, n, sigma, seed):
    """U diag(sigma) V^T with random orthonormal U (m x r), V (n x r)."""
    rng = np.random.default_rng(seed)
    r = len(sigma)
    U, _ = np.linalg.qr(rng.normal(size=(m, r)))
    V, _ = np.linalg.qr(rng.normal(size=(n, r)))
    return (U * np.asarray(sigma, dtype=np.float64)) @ V.T


# ---- App. D.4: E(P) and P* ----------------------------------------------------

@pytest.mark.parametrize("shape", [(5, 3), (4, 6), (7, 7)])
def test_energy_equals_truncation_error_identity(shape):
    """E(P) = 1 - ||W - W_P||_F^2 / ||W||_F^2, with W_P the rank-P truncation
    rebuilt from an independent (Jacobi) SVD."""
    W = np.random.default_rng(sum(shape)).normal(size=shape)
    U, s, Vt = svd_jacobi.jacobi_svd(W) if shape[0] >= shape[1] else svd_jacobi.jacobi_svd(W)
    R = min(shape)
    f2 = float(np.sum(W * W))
    for P in range(0, R + 1):
        WP = (U[:, :P] * s[:P]) @ Vt[:P, :]
        want = 1.0 - float(np.sum((W - WP) ** 2)) / f2
        assert oracle.energy(W, P) == pytest.approx(want, abs=1e-12)
    assert oracle.energy(W, R) == pytest.approx(1.0, abs=1e-15)
    assert oracle.energy(W, 0) == 0.0


def test_energy_and_rank_on_diagonal_closed_form():
    d = np.array([0.5, -3.0, 0.0, 2.0, -1.0])
    W = np.diag(d)
    sq = np.sort(d * d)[::-1]                      # 9, 4, 1, 0.25, 0
    cum = np.cumsum(sq) / sq.sum()
    for P in range(1, 6):
        assert oracle.energy(W, P) == pytest.approx(cum[P - 1], abs=1e-15)
    # brute force over rho: the smallest P whose E(P) reaches rho
    for rho in [0.1, 9 / 14.25, 0.7, 13 / 14.25, 0.95, 14 / 14.25, 0.99, 1.0]:
        want = next(P for P in range(1, 6) if cum[P - 1] >= rho - 1e-15)
        assert oracle.energy_rank(W, rho) == want
    assert oracle.energy_rank(np.zeros((3, 4)), 0.9) == 0


def test_hoyer_tau_closed_form():
    W = _with_spectrum(9, 6, [4.0, 2.0, 1.0], seed=3)
    assert oracle.hoyer_tau(W) == pytest.approx((16 + 4 + 1) / 7.0, rel=1e-13)


# ---- Prop. 2, exact gradient: sigma+ = sigma + e (sigma - tau) ----------------

@pytest.mark.parametrize("shape,sigma", [((12, 8), [3.0, 2.5, 1.0, 0.6, 0.2]),
                                         ((8, 12), [1.0, 0.9, 0.1]),
                                         ((6, 6), [2.0, 1.5, 1.2, 0.4, 0.3, 0.05])])
def test_prop2_closed_form_exact_gradient(shape, sigma):
    """In W's SVD basis the exact Hoyer gradient (Eq. 1) is diagonal, so one step
    maps each sigma_i to sigma_i + e (sigma_i - tau) with tau = f^2 / n and
    e = 2 eta n^2 / f^4 (the identity behind Prop. 2)."""
    W = _with_spectrum(*shape, sigma, seed=len(sigma))
    s = np.array(sigma)
    n, f2 = s.sum(), (s * s).sum()
    tau = f2 / n
    eta = 1e-3 * f2
    e = 2.0 * eta * n * n / (f2 * f2)
    Wp = W - eta * oracle.exact_grad(W, "hoyer")
    got = oracle.singular_values(Wp)[: len(s)]
    assert np.allclose(got, s + e * (s - tau), rtol=0, atol=1e-12 * s.max())
    assert oracle.hoyer_tau(W) == pytest.approx(tau, rel=1e-13)
    # the sign law of Prop. 2
    assert np.all(np.sign(got - s) == np.sign(s - tau))


# ---- the oracle's Polar Express descent step, per singular value --------------

@pytest.mark.parametrize("variant", ["hoyer", "nuclear"])
def test_descent_step_matches_scalar_map_form(variant):
    """W+ = W - eta lam s G_hat(W).  With W = U diag(sigma) V^T every Polar
    Express iterate shares U and V, and P_hat = U diag(g(sigma / frob)) V^T with
    g the composed scalar map; so W+ = U diag(sigma+) V^T with
      Hoyer: sigma+ = sigma - eta lam s 2 (n/frob) (g / frob - n sigma / frob^3),
             n = sum sigma g;
      Nuc:   sigma+ = sigma - eta lam s g."""
    sigma = np.array([2.0, 1.4, 0.9, 0.5, 0.3, 0.12])
    W = _with_spectrum(14, 10, sigma, seed=11)
    frob = np.sqrt((sigma * sigma).sum()) + EPS
    g = oracle.pe_scalar_map(sigma / frob, CO)
    lam, gs, eta = 0.7, 1.3, 0.05
    if variant == "hoyer":
        n = float(np.sum(sigma * g))
        want = sigma - eta * lam * gs * 2.0 * (n / frob) * (g / frob - n * sigma / frob ** 3)
    else:
        want = sigma - eta * lam * gs * g
    Wp, L = oracle.descent_step(W, eta, variant, CO, lam=lam, grad_scale=gs, eps=EPS)
    got = oracle.singular_values(Wp)[: sigma.size]
    assert np.allclose(np.sort(got), np.sort(want), rtol=0, atol=1e-12)
    # the value returned is the one at the old weights
    if variant == "hoyer":
        assert L == pytest.approx((n / frob) ** 2, rel=1e-12)
    else:
        assert L == pytest.approx(float(np.sum(sigma * g)), rel=1e-12)


def test_prop2_sign_law_with_polar_express_gradient():
    """Prop. 2 with the approximate gradient: away from tau (farther than the
    Polar Express error moves the threshold), singular values above tau grow
    and those below shrink."""
    W = np.random.default_rng(7).normal(size=(40, 24))
    s = oracle.singular_values(W)
    tau = oracle.hoyer_tau(W)
    Wp, _ = oracle.descent_step(W, 1e-3 * float(np.sum(s * s)), "hoyer", CO)
    sp = oracle.singular_values(Wp)
    far = np.abs(s - tau) > 0.05 * tau
    assert far.sum() >= 20
    assert np.all(np.sign(sp - s)[far] == np.sign(s - tau)[far])


def test_hoyer_step_never_shrinks_frobenius_norm():
    """<W, grad L_hoyer> = 0 (Sec. 3.1), so ||W+||_F^2 = ||W||_F^2 + eta^2 ||G||^2
    >= ||W||_F^2; with the approximate gradient <W, G_hat> vanishes up to eps."""
    W = np.random.default_rng(8).normal(size=(20, 30))
    eta = 0.3
    _, G, _, _ = oracle.reg_single(W, "hoyer", CO, EPS)
    Wp, _ = oracle.descent_step(W, eta, "hoyer", CO)
    lhs = float(np.sum(Wp * Wp))
    assert lhs >= float(np.sum(W * W))
    assert lhs == pytest.approx(float(np.sum(W * W)) + eta * eta * float(np.sum(G * G)), rel=1e-9)


# ---- Prop. 3: energy concentration -------------------------------------------

@pytest.mark.parametrize("grad", ["exact", "polar_express"])
def test_prop3_tail_error_falls_for_every_k_above_tau(grad):
    rng = np.random.default_rng(21)
    W = rng.normal(size=(32, 20)) + 2.0 * np.outer(rng.normal(size=32), rng.normal(size=20)) / 6.0
    s = oracle.singular_values(W)
    tau = oracle.hoyer_tau(W)
    eta = 1e-3 * float(np.sum(s * s))
    if grad == "exact":
        Wp = W - eta * oracle.exact_grad(W, "hoyer")
    else:
        Wp, _ = oracle.descent_step(W, eta, "hoyer", CO)
    ks = [k for k in range(1, s.size) if s[k - 1] > tau]
    assert len(ks) >= 3
    for k in ks:
        assert 1.0 - oracle.energy(Wp, k) < 1.0 - oracle.energy(W, k)


def test_descent_trajectory_concentrates_energy():
    """Repeated regularizer-only steps on a spiked matrix: the Hoyer value falls
    at every step and the energy held by the spike's rank rises.  (With a fixed
    step the small singular values eventually overshoot zero and oscillate at
    about e tau, so "sufficiently small" in Props. 2 and 3 bounds the run to
    the first dozen steps at this eta.)"""
    W = np.random.default_rng(5).normal(0, 0.02, size=(48, 32))
    W += _with_spectrum(48, 32, [0.3, 0.25, 0.2, 0.15], seed=6)
    eta = 0.005 * float(np.sum(W * W))
    Ws, Ls = oracle.descent_trajectory(W, eta, 12, "hoyer", CO)
    assert all(b < a for a, b in zip(Ls, Ls[1:]))
    E = [oracle.energy(X, 4) for X in Ws]
    assert all(b > a for a, b in zip(E, E[1:]))
    assert oracle.energy_rank(Ws[-1], 0.95) < oracle.energy_rank(Ws[0], 0.95)
