"""Pins for the oracle's SLORR value and gradient (Sec. 3, Eq. 1, Listing 1,
Prop. 1, App. A/B), each chosen so a plausible slip in the oracle fails one:
closed forms, invariants, the scalar-map (SVD) form of the matrix iteration,
finite differences, brute-force SVD and hand-derived golden values."""

import os

import numpy as np
import pytest

import oracle
from oracle import svd_jacobi

GOLD = os.path.join(os.path.dirname(__file__), "golden")
CO = oracle.pe_coefficients(T=6)
EPS = 1e-7


def _read_golden(name):
    out = {}
    with open(os.path.join(GOLD, name)) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            k, *v = line.split()
            out[k] = np.array([float(x) for x in v])
    return out


def _rand(shape, seed, std=1.0):
    return np.random.default_rng(seed).normal(0.0, std, size=shape)


# ---- the matrix iteration equals the scalar map on the singular values -------

@pytest.mark.parametrize("shape", [(1, 1), (1, 5), (5, 1), (3, 7), (7, 3), (16, 16),
                                   (33, 64), (64, 17)])
def test_iteration_equals_scalar_map_on_svd(shape):
    W = _rand(shape, seed=sum(shape))
    U, s, Vt = np.linalg.svd(W, full_matrices=False)
    f = oracle.frobenius(W)
    g = oracle.pe_scalar_map(s / (f + EPS), CO)
    expect = (U * g) @ Vt
    got = oracle.polar_express(W, CO, EPS)
    assert got.shape == W.shape
    assert np.allclose(got, expect, rtol=0, atol=1e-12)


def test_gram_side_orientation():
    """P x Q iterates: X_0 is W^T when M > N, and the Gram matrix is P x P."""
    W = _rand((9, 4), 3)
    steps, tr = oracle.polar_express_steps(W, CO, EPS)
    assert tr and steps[0].shape == (4, 9)
    assert np.allclose(steps[0], W.T / (oracle.frobenius(W) + EPS))
    W2 = _rand((4, 9), 3)
    steps2, tr2 = oracle.polar_express_steps(W2, CO, EPS)
    assert not tr2 and steps2[0].shape == (4, 9)


def test_nuclear_estimate_identity():
    """n_hat = sum_i sigma_i g(sigma_i / (f + eps)) exactly (trace identity, Sec. 3)."""
    W = _rand((12, 20), 11)
    s = np.linalg.svd(W, compute_uv=False)
    f = oracle.frobenius(W)
    L, G, n_hat, frob = oracle.reg_single(W, "nuclear", CO, EPS)
    assert n_hat == pytest.approx(np.sum(s * oracle.pe_scalar_map(s / (f + EPS), CO)), rel=1e-12)
    assert frob == pytest.approx(f + EPS, rel=1e-15)


# ---- closed forms -----------------------------------------------------------

@pytest.mark.parametrize("m,n", [(6, 6), (5, 8), (8, 5)])
def test_orthogonal_closed_form(m, n):
    Q, _ = np.linalg.qr(_rand((max(m, n), min(m, n)), 7))
    Q = Q if m >= n else Q.T
    P = min(m, n)
    nn, f, hoyer, UV = oracle.exact_values(Q)
    assert nn == pytest.approx(P) and hoyer == pytest.approx(P)
    assert np.allclose(oracle.exact_grad(Q, "hoyer"), 0.0, atol=1e-12)
    assert np.allclose(oracle.exact_grad(Q, "nuclear"), Q, atol=1e-12)
    # PE: all normalised singular values equal 1/(sqrt(P)+eps) -> P_hat = g * Q
    g = oracle.pe_scalar_map(np.array([1.0 / (np.sqrt(P) + EPS)]), CO)[0]
    L, G, n_hat, frob = oracle.reg_single(Q, "hoyer", CO, EPS)
    assert n_hat == pytest.approx(P * g, rel=1e-12)
    assert L == pytest.approx((P * g / (np.sqrt(P) + EPS)) ** 2, rel=1e-12)
    Ln, Gn, _, _ = oracle.reg_single(Q, "nuclear", CO, EPS)
    assert Ln == pytest.approx(P * g, rel=1e-12)
    assert np.allclose(Gn, g * Q, atol=1e-12)


def test_rank1_closed_form():
    u = _rand((7, 1), 1)
    v = _rand((4, 1), 2)
    u /= np.linalg.norm(u)
    v /= np.linalg.norm(v)
    s = 3.5
    W = s * (u @ v.T)
    nn, f, hoyer, _ = oracle.exact_values(W)
    assert hoyer == pytest.approx(1.0)            # unsquared ratio 1, squared 1
    assert np.allclose(oracle.exact_grad(W, "hoyer"), 0.0, atol=1e-12)
    g = oracle.pe_scalar_map(np.array([s / (s + EPS)]), CO)[0]
    L, G, n_hat, frob = oracle.reg_single(W, "hoyer", CO, EPS)
    assert L == pytest.approx((s * g / (s + EPS)) ** 2, rel=1e-12)
    assert np.allclose(G, 2 * (s * g / (s + EPS)) * g * (u @ v.T) * (1 / (s + EPS) - s * s / (s + EPS) ** 3),
                       atol=1e-12)


def test_scaled_identity_closed_form():
    n = 9
    W = 2.5 * np.eye(n)
    nn, f, hoyer, _ = oracle.exact_values(W)
    assert np.sqrt(hoyer) == pytest.approx(np.sqrt(n))   # unsquared ratio sqrt(n)
    assert hoyer == pytest.approx(n)
    assert np.allclose(oracle.exact_grad(W, "hoyer"), 0.0, atol=1e-12)


def test_diagonal_signs_zeros_closed_form():
    d = np.array([3.0, -1.5, 0.0, 0.7, -2.2])
    W = np.diag(d)
    n = np.abs(d).sum()
    f = np.sqrt((d * d).sum())
    expect = np.diag(2 * n / f ** 2 * np.sign(d) - 2 * n ** 2 / f ** 4 * d)
    assert np.allclose(oracle.exact_grad(W, "hoyer"), expect, atol=1e-12)
    # PE version in the SVD basis: P_hat = diag(sign(d_i) g(|d_i|/(f+eps)))
    Ph = np.diag(np.sign(d) * oracle.pe_scalar_map(np.abs(d) / (f + EPS), CO))
    assert np.allclose(oracle.polar_express(W, CO, EPS), Ph, atol=1e-12)
    L, G, n_hat, frob = oracle.reg_single(W, "hoyer", CO, EPS)
    reg = n_hat / frob
    assert np.allclose(G, 2 * reg * (Ph / frob - n_hat / frob ** 3 * W), atol=1e-14)


def test_golden_diag_3_4():
    g = _read_golden("hoyer_diag_3_4.txt")
    W = g["W"].reshape(2, 2)
    nn, f, hoyer, _ = oracle.exact_values(W)
    assert hoyer == pytest.approx(g["hoyer_value"][0], rel=1e-14)
    assert np.allclose(oracle.exact_grad(W, "hoyer").ravel(), g["hoyer_grad"], atol=1e-14)
    assert nn == pytest.approx(g["nuc_value"][0], rel=1e-14)
    assert np.allclose(oracle.exact_grad(W, "nuclear").ravel(), g["nuc_grad"], atol=1e-14)


@pytest.mark.parametrize("case", ["case1", "case2", "case3"])
def test_golden_diag_signs(case):
    g = _read_golden("hoyer_diag_signs.txt")
    raw = g[case + "_W"]
    m, n = int(raw[0]), int(raw[1])
    W = raw[2:].reshape(m, n)
    _, _, hoyer, _ = oracle.exact_values(W)
    assert hoyer == pytest.approx(g[case + "_value"][0], rel=1e-13)
    assert np.allclose(oracle.exact_grad(W, "hoyer").ravel(), g[case + "_grad"], atol=1e-13)


def test_zero_matrix_gives_zero():
    W = np.zeros((4, 6))
    loss, per, incs = oracle.reg_forward_backward([W], "hoyer", CO, lam=0.5, eps=EPS)
    assert loss == 0.0 and np.all(incs[0] == 0.0)
    loss, per, incs = oracle.reg_forward_backward([W], "nuclear", CO, lam=0.5, eps=EPS)
    assert loss == 0.0 and np.all(incs[0] == 0.0)


# ---- invariants ---------------------------------------------------------------

def test_gradient_orthogonal_to_W():
    """<W, G_hat> = n_hat/frob (1 - f^2/frob^2): zero but for the eps terms (Sec. 3.1)."""
    W = _rand((10, 15), 5)
    L, G, n_hat, frob = oracle.reg_single(W, "hoyer", CO, EPS)
    f = frob - EPS
    inner = np.sum(W * G)
    reg = n_hat / frob
    assert inner == pytest.approx(2 * reg * n_hat / frob * (1 - f * f / frob ** 2), rel=1e-6, abs=1e-14)
    assert abs(inner) < 1e-6 * np.linalg.norm(G) * np.linalg.norm(W)
    # and exactly orthogonal for the exact gradient
    assert abs(np.sum(W * oracle.exact_grad(W, "hoyer"))) < 1e-12


def test_scale_invariance():
    W = _rand((8, 12), 9)
    L1 = oracle.reg_single(W, "hoyer", CO, EPS)[0]
    L2 = oracle.reg_single(7.0 * W, "hoyer", CO, EPS)[0]
    assert L1 == pytest.approx(L2, rel=1e-7)
    assert oracle.exact_values(W)[2] == pytest.approx(oracle.exact_values(7.0 * W)[2], rel=1e-13)


def test_null_space_preserved():
    """p(0) = 0: P_hat annihilates the right null space of a rank-deficient W (App. B)."""
    A = _rand((9, 3), 4)
    B = _rand((3, 7), 6)
    W = A @ B                                  # rank 3, 9 x 7
    _, s, Vt = np.linalg.svd(W)
    null = Vt[3:].T
    Ph = oracle.polar_express(W, CO, EPS)
    assert np.abs(Ph @ null).max() < 1e-10
    assert np.abs(null.T @ Ph.T @ Ph @ null).max() < 1e-10


def test_lambda_and_grad_scale_placement():
    Ws = [_rand((5, 8), 1), _rand((8, 5), 2)]
    loss1, per1, inc1 = oracle.reg_forward_backward(Ws, "hoyer", CO, lam=1.0, eps=EPS)
    loss2, per2, inc2 = oracle.reg_forward_backward(Ws, "hoyer", CO, lam=0.25, eps=EPS, grad_scale=4.0)
    assert loss2 == pytest.approx(0.25 * loss1)
    assert np.allclose(per1, per2)
    for a, b in zip(inc1, inc2):
        assert np.allclose(a, b)


# ---- Prop. 1, sharpened -------------------------------------------------------

def _with_singular_values(s, m, n, seed):
    U, _ = np.linalg.qr(_rand((m, len(s)), seed))
    V, _ = np.linalg.qr(_rand((n, len(s)), seed + 1))
    return (U * s) @ V.T


@pytest.mark.parametrize("T", [4, 6, 8])
def test_prop1_sharpened_bounds(T):
    co = oracle.pe_coefficients(T=T)
    E_T = oracle.achieved_error(co)
    delta = oracle.paper_delta(1e-3, T, 5)
    rng = np.random.default_rng(T)
    sig = np.exp(rng.uniform(np.log(0.05), 0.0, size=6))
    W = _with_singular_values(sig, 10, 8, seed=T)
    f = oracle.frobenius(W)
    assert (sig / f).min() >= 1e-3 and (sig / f).max() <= 1.0
    nn, _, hoyer, UV = oracle.exact_values(W)
    L, G, n_hat, frob = oracle.reg_single(W, "hoyer", co, eps=0.0)
    fp = 1e-12   # fp64 rounding allowance once E_T reaches machine precision
    assert abs(n_hat - nn) / nn <= E_T * (1 + 1e-9) + fp
    assert abs(n_hat - nn) / nn <= delta
    assert abs(L - hoyer) / hoyer <= E_T * (2 + E_T) * (1 + 1e-9) + fp
    Ph = oracle.polar_express(W, co, eps=0.0)
    assert np.linalg.norm(Ph - UV, 2) <= E_T * (1 + 1e-9) + fp
    R = oracle.exact_grad(W, "hoyer")
    bound = 2 * E_T * (2 + E_T) * (nn / f ** 2 + nn ** 2 / f ** 4 * np.linalg.norm(W, 2))
    assert np.linalg.norm(R - G, 2) <= bound * (1 + 1e-9) + fp * np.linalg.norm(R, 2) + fp


# ---- finite differences and brute force ---------------------------------------

@pytest.mark.parametrize("shape", [(3, 2), (4, 4), (5, 3)])
@pytest.mark.parametrize("variant", ["hoyer", "nuclear"])
def test_exact_gradient_finite_differences(shape, variant):
    """Central differences of the exact losses vs Eq. 1 (well-separated sigma)."""
    m, n = shape
    P = min(m, n)
    W = _with_singular_values(np.linspace(2.0, 1.0, P) ** 2, m, n, seed=m * 10 + n)

    def loss(X):
        nn, f, hoyer, _ = oracle.exact_values(X)
        return hoyer if variant == "hoyer" else nn

    G = oracle.exact_grad(W, variant)
    h = 1e-6
    num = np.zeros_like(W)
    for i in range(m):
        for j in range(n):
            E = np.zeros_like(W)
            E[i, j] = h
            num[i, j] = (loss(W + E) - loss(W - E)) / (2 * h)
    assert np.allclose(num, G, rtol=1e-6, atol=1e-7)


@pytest.mark.parametrize("shape", [(2, 2), (3, 5), (6, 4), (8, 8)])
def test_brute_force_jacobi_svd(shape):
    W = _rand(shape, 100 + shape[0])
    U, s, Vt = svd_jacobi.jacobi_svd(W)
    assert np.allclose((U * s) @ Vt, W, atol=1e-12)
    assert np.allclose(s, np.linalg.svd(W, compute_uv=False), rtol=1e-12)
    # exact values and polar factor from the Jacobi SVD agree with the oracle's
    nn, f, hoyer, UV = oracle.exact_values(W)
    assert nn == pytest.approx(s.sum(), rel=1e-12)
    assert np.allclose(U @ Vt, UV, atol=1e-10)
    g = oracle.pe_scalar_map(s / (np.sqrt((s * s).sum()) + EPS), CO)
    assert np.allclose((U * g) @ Vt, oracle.polar_express(W, CO, EPS), atol=1e-11)


def test_flop_model():
    """4 P^2 Q + 2 P^3 per step with P = min, Q = max (Sec. 3 'Computational cost')."""
    assert oracle.pe_flops(256, 256, T=1) == 6 * 256 ** 3
    assert oracle.pe_flops(1024, 4096, T=1) == oracle.pe_flops(4096, 1024, T=1)
    assert oracle.pe_flops(320, 1280, T=1) == 4 * 320 ** 2 * 1280 + 2 * 320 ** 3
    assert oracle.weight_set_flops([(256, 256)] * 8, T=6) == 8 * 6 * 6 * 256 ** 3
