"""GPU parity on the method's closed-form and degenerate inputs (Sec. 3, Eq. 1,
App. B "Remark about zero singular values", Prop. 1), through the C ABI,
against the fp64 oracle, in fp16-operand (tensor cores), bf16 hi/lo
(bf16_split) and fp32 modes, at sizes that take several 256 x 256
tensor-core tiles.

Inputs and what pins them besides the oracle:
* orthogonal Q (square, wide, tall): every singular value 1, so
  L_hoyer = P g(1/sqrt(P))^2 and P_hat = g(1/sqrt(P)) Q, within Prop. 1's
  achieved error E_T of the exact values P and Q;
* alpha I_n: the unsquared Hoyer ratio is sqrt(n), L = n (within E_T);
* rank one s u v^T: L = g(1)^2, within E_T of 1; the exact Hoyer gradient is 0;
* signed diagonals with zero entries: the zero rows and columns of W stay
  exactly zero in every iterate, so the gradient there is exactly 0 (App. B);
* rank-deficient W = A B (rank 32 and 256);
* a tiny-norm and a large-norm matrix (the fused norm pass re-casts both).

Zero singular values under rounding.  In exact arithmetic P_hat v = 0 for
every v in W's right null space (App. B).  With rounded iterates it is not:
each rounding of X leaves a perturbation in the null space whose singular
values are about sigma_e = u ||X_t||_F (1/sqrt(P) + 1/sqrt(Q)) (u the unit
roundoff of the stored iterate), and the remaining steps amplify values that
small by the slope of their polynomials at zero, G_t = prod_{s>t} a_s
(G_0 = 1846 for the T = 6 schedule, since every sigma below ell is still in
the linear regime).  So a rank-deficient W gets P_hat v of order
sum_t G_t sigma_e,t, not 0: 0.04 to 0.1 in spectral norm with fp16 iterates
(2 to 39% of ||P_hat||_F, depending on how many null directions there are),
about 1e-4 in fp32.  The tests therefore hold the part of P_hat and of the
gradient on W's row space to the parity tolerance, and the null-space part
to that estimate: 3 x the estimate in fp16 and bf16_split; in fp32 the worst case
u (G_0 + 1.1 sqrt(r) sum_{t>=1} G_t) (every rounding aligned with the null
space).
"""

import numpy as np
import pytest

import oracle
import workloads

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

EPS = 1e-7
TOL = {"fp32": 1e-5, "fp16": 2e-2, "bf16_split": 2e-2}
# bf16_split: the iterates are bf16 hi/lo pairs (about 2^-17) until X_T, which
# is stored in fp16: its leak bound is taken as fp16's, a looser one
UNIT_ROUNDOFF = {"fp32": 2.0 ** -24, "fp16": 2.0 ** -11, "bf16_split": 2.0 ** -11}
CO = oracle.pe_coefficients(6)
E_T = oracle.achieved_error(CO)


@pytest.fixture(scope="module", autouse=True)
def _need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2607_08754_gb300 import slorr
    slorr.load_library()   # raises if the extension is missing: no fallback


def run(Ws, variant, compute, lam=1.0):
    """One forward + backward of the set; returns (loss, per-matrix values,
    gradients, P_hat in W's orientation) as fp64 numpy."""
    from paper_2607_08754_gb300.slorr import Regularizer
    reg = Regularizer([W.shape for W in Ws], variant=variant, compute=compute, lam=lam)
    w = [torch.from_numpy(np.ascontiguousarray(W, dtype=np.float32)).cuda() for W in Ws]
    g = [torch.zeros_like(x) for x in w]
    per = torch.full((len(Ws),), float("nan"), device="cuda")
    loss = reg(w, g, per_matrix=per).item()
    torch.cuda.synchronize()
    assert reg.status() == 0
    p_hat = []
    for i, W in enumerate(Ws):
        x = reg.iterate(i, 6).double().cpu().numpy()    # P x Q
        p_hat.append(x.T if W.shape[0] > W.shape[1] else x)
    return loss, per.double().cpu().numpy(), [x.double().cpu().numpy() for x in g], p_hat


def rel(a, b):
    return np.linalg.norm(a - b) / np.linalg.norm(b)


def first_term_norm(W, lam=1.0):
    """||2 reg P_hat / frob||_F of the oracle: the scale of a Hoyer gradient
    whose two terms cancel (rank one, equal singular values)."""
    L, _, n_hat, frob = oracle.reg_single(W, "hoyer", CO, EPS)
    return abs(lam) * 2.0 * (n_hat / frob) / frob * np.linalg.norm(oracle.polar_express(W, CO, EPS))


def check_full(W, got_L, got_G, got_P, variant, compute):
    """Element-wise parity of one matrix's value, gradient and P_hat."""
    tol = TOL[compute]
    W64 = W.astype(np.float64)
    L, G, _, _ = oracle.reg_single(W64, variant, CO, EPS)
    P = oracle.polar_express(W64, CO, EPS)
    assert abs(got_L - L) <= tol * abs(L) + 1e-30, (got_L, L)
    assert rel(got_P, P) <= tol, rel(got_P, P)
    nG = np.linalg.norm(G)
    scale = nG
    if variant == "hoyer":
        t = first_term_norm(W64)
        if nG < 0.05 * t:        # the exact gradient is (close to) zero: the terms cancel
            scale = t
    assert np.linalg.norm(got_G - G) <= tol * scale, (np.linalg.norm(got_G - G) / scale)
    return L, G, P


def leak_bound(compute, P, Q, r):
    """Bound on ||P_hat V_null||_2 for a rank-r P x Q input (module docstring)."""
    u = UNIT_ROUNDOFF[compute]
    a = [c[0] for c in CO]
    G = [float(np.prod(a[t:])) for t in range(len(a))] + [1.0]   # G[t] = prod_{s>t} a_s, s = 1..T
    amp = G[0] + 1.1 * np.sqrt(r) * sum(G[1:])
    if compute != "fp32":
        return min(1.0 + E_T, 3.0 * u * (1.0 / np.sqrt(P) + 1.0 / np.sqrt(Q)) * amp)
    return u * amp


def check_rank_deficient(W, r, got_L, got_G, got_P, variant, compute):
    """Row-space parity at the tolerance, null-space leak within its bound."""
    tol = TOL[compute]
    W64 = W.astype(np.float64)
    L, G, _, _ = oracle.reg_single(W64, variant, CO, EPS)
    P = oracle.polar_express(W64, CO, EPS)
    _, s, Vt = np.linalg.svd(W64, full_matrices=True)
    assert s[r - 1] > 1e-8 * s[0] and (r == min(W.shape) or s[r] < 1e-12 * s[0])
    Vr, Vn = Vt[:r].T, Vt[r:].T
    assert abs(got_L - L) <= tol * abs(L), (got_L, L)      # n_hat = <W, P_hat> sees the row space only
    assert np.linalg.norm((got_P - P) @ Vr) <= tol * np.linalg.norm(P), \
        np.linalg.norm((got_P - P) @ Vr) / np.linalg.norm(P)
    scale = np.linalg.norm(G @ Vr)
    if variant == "hoyer":
        t = first_term_norm(W64)
        if scale < 0.05 * t:
            scale = t
    assert np.linalg.norm((got_G - G) @ Vr) <= tol * scale
    leak = np.linalg.norm(got_P @ Vn, 2) if Vn.shape[1] else 0.0
    bound = leak_bound(compute, min(W.shape), max(W.shape), r)
    assert leak <= bound, (leak, bound)
    assert np.linalg.norm(got_P, 2) <= 1.0 + E_T + 8 * UNIT_ROUNDOFF[compute] * np.sqrt(min(W.shape))
    return leak


def orthonormal(m, n, seed):
    q, _ = np.linalg.qr(np.random.default_rng(seed).normal(size=(max(m, n), min(m, n))))
    return q if m >= n else q.T


# ---- orthogonal matrices and the scaled identity ------------------------------------

@pytest.mark.parametrize("compute", ["fp16", "fp32", "bf16_split"])
@pytest.mark.parametrize("variant", ["hoyer", "nuclear"])
def test_orthogonal_matrices(compute, variant):
    shapes = [(256, 256), (256, 640), (640, 256), (384, 1000)]
    Ws = [orthonormal(m, n, 70 + i).astype(np.float32) for i, (m, n) in enumerate(shapes)]
    loss, per, grads, p_hat = run(Ws, variant, compute)
    tol = TOL[compute]
    for i, W in enumerate(Ws):
        Pdim = min(W.shape)
        L, G, P = check_full(W, per[i], grads[i], p_hat[i], variant, compute)
        # closed forms: ||Q||_* = P, Hoyer L = P, P_hat = Q, each within Prop. 1's E_T
        exact = float(Pdim)
        assert abs(per[i] - exact) <= exact * (E_T * (2 + E_T) + tol)
        assert np.linalg.norm(p_hat[i] - W) <= (E_T + tol) * np.linalg.norm(W)
        if variant == "nuclear":
            assert rel(grads[i], W.astype(np.float64)) <= E_T + tol


@pytest.mark.parametrize("compute", ["fp16", "fp32", "bf16_split"])
def test_scaled_identity(compute):
    Ws = [0.37 * np.eye(384, dtype=np.float32), 3.0 * np.eye(256, dtype=np.float32)]
    loss, per, grads, p_hat = run(Ws, "hoyer", compute)
    for i, W in enumerate(Ws):
        check_full(W, per[i], grads[i], p_hat[i], "hoyer", compute)
        n = W.shape[0]
        # unsquared ratio sqrt(n), squared n (within E_T); the exact gradient is 0
        assert abs(np.sqrt(per[i]) - np.sqrt(n)) <= np.sqrt(n) * (E_T + TOL[compute])


# ---- rank one and rank-deficient inputs ---------------------------------------------

def low_rank(m, n, r, seed):
    """Exactly rank r in fp32 and fp16: W = A B 2^-10 with integer A, B in
    [-2, 2], so every entry is an integer of magnitude <= 4 r <= 1024 (exact in
    both types) times a power of two."""
    rng = np.random.default_rng(seed)
    while True:
        A = rng.integers(-2, 3, size=(m, r)).astype(np.float64)
        B = rng.integers(-2, 3, size=(r, n)).astype(np.float64)
        W = A @ B
        if np.linalg.matrix_rank(W) == r:
            return (W * 2.0 ** -10).astype(np.float32)


@pytest.mark.parametrize("compute", ["fp16", "fp32", "bf16_split"])
@pytest.mark.parametrize("variant", ["hoyer", "nuclear"])
def test_rank_one(compute, variant):
    shapes = [(256, 700), (700, 256), (300, 520)]
    Ws = [low_rank(m, n, 1, 90 + i) for i, (m, n) in enumerate(shapes)]
    loss, per, grads, p_hat = run(Ws, variant, compute)
    for i, W in enumerate(Ws):
        check_rank_deficient(W, 1, per[i], grads[i], p_hat[i], variant, compute)
        if variant == "hoyer":
            # unsquared ratio 1 (Sec. 3): L = g(1)^2 within Prop. 1's E_T of 1
            assert abs(per[i] - 1.0) <= E_T * (2 + E_T) + TOL[compute]


@pytest.mark.parametrize("compute", ["fp16", "fp32", "bf16_split"])
def test_rank_deficient(compute):
    specs = [(512, 768, 32), (768, 512, 32), (512, 768, 256), (640, 256, 8)]
    Ws = [low_rank(m, n, r, 110 + i) for i, (m, n, r) in enumerate(specs)]
    for variant in ("hoyer", "nuclear"):
        loss, per, grads, p_hat = run(Ws, variant, compute)
        for i, (m, n, r) in enumerate(specs):
            check_rank_deficient(Ws[i], r, per[i], grads[i], p_hat[i], variant, compute)


@pytest.mark.parametrize("compute", ["fp16", "fp32", "bf16_split"])
@pytest.mark.parametrize("variant", ["hoyer", "nuclear"])
def test_signed_diagonal_with_zeros(compute, variant):
    """W = [diag(d) 0] (and its transpose) with signed d and zero entries: the
    zero rows and columns stay exactly zero through every product, so the
    gradient there is exactly 0 (App. B); the rest matches the oracle and, for
    Hoyer, the closed form 2 n/f^2 sign(d_i) g_i - 2 n^2/f^4 d_i (App. A in
    the singular basis, with g_i = g(|d_i| / (f + eps)))."""
    rng = np.random.default_rng(131)
    Ws = []
    for m, n in [(300, 520), (520, 300), (256, 256)]:
        k = min(m, n)
        d = rng.uniform(0.2, 1.0, size=k) * rng.choice([-1.0, 1.0], size=k)
        d[rng.choice(k, size=k // 5, replace=False)] = 0.0
        W = np.zeros((m, n), np.float32)
        W[np.arange(k), np.arange(k)] = d
        Ws.append(W)
    loss, per, grads, p_hat = run(Ws, variant, compute)
    for i, W in enumerate(Ws):
        check_full(W, per[i], grads[i], p_hat[i], variant, compute)
        zero_rows = ~np.any(W != 0, axis=1)
        zero_cols = ~np.any(W != 0, axis=0)
        assert np.all(grads[i][zero_rows, :] == 0.0) and np.all(grads[i][:, zero_cols] == 0.0)
        assert np.all(p_hat[i][zero_rows, :] == 0.0) and np.all(p_hat[i][:, zero_cols] == 0.0)
        if variant == "hoyer":
            W64 = W.astype(np.float64)
            f = np.linalg.norm(W64) + EPS
            dd = np.diag(W64)[: min(W.shape)]
            gvals = oracle.pe_scalar_map(np.abs(dd) / f, CO)
            n_hat = float(np.sum(np.abs(dd) * gvals))
            closed = np.zeros_like(W64)
            k = min(W.shape)
            closed[np.arange(k), np.arange(k)] = 2 * n_hat / f ** 2 * np.sign(dd) * gvals - 2 * n_hat ** 2 / f ** 4 * dd
            assert np.linalg.norm(grads[i] - closed) <= TOL[compute] * np.linalg.norm(closed) + 1e-6


# ---- norms far from 1 ----------------------------------------------------------------

@pytest.mark.parametrize("compute", ["fp16", "fp32", "bf16_split"])
@pytest.mark.parametrize("variant", ["hoyer", "nuclear"])
def test_tiny_and_large_norms(compute, variant):
    """||W||_F = 1e-5 (fp16 would hold W itself only as subnormals) and
    ||W||_F = 1e6 with entries above 2^15 (beyond fp16's exponent range
    unscaled): the fused norm pass re-casts both as W / (||W||_F + eps)."""
    base = [workloads.random_matrix((320, 700), 141, 1.0), workloads.random_matrix((700, 320), 142, 1.0)]
    tiny = (base[0] * (1e-5 / np.linalg.norm(base[0]))).astype(np.float32)
    large = (base[1] * (1e6 / np.linalg.norm(base[1]))).astype(np.float32)
    large[3, 7] = 6.0e4
    Ws = [tiny, large]
    loss, per, grads, p_hat = run(Ws, variant, compute)
    for i, W in enumerate(Ws):
        check_full(W, per[i], grads[i], p_hat[i], variant, compute)
