"""GPU parity of the in-place regularizer-only descent step
(slorr_reg_descent_step: W <- W - eta lambda grad_scale G_hat(W), the last line
of Alg. 1 with no task update; the step of Props. 2 and 3) against the oracle's
``descent_step`` / ``descent_trajectory`` on the same seeded inputs.

Tolerances.  One step: the update dW = W+ - W must match the oracle's within
the parity tolerance of the gradient (1e-5 fp32 mode, 2e-2 fp16 mode) times
||dW||, plus the rounding of storing W+ in fp32 (at most 2^-24 |w+| per
element, so 2^-24 ||W+||_F).  K steps (fp32 mode): each step adds at most that
bound; over a short run with steps this small the gradient's Lipschitz growth
is well under 2x, so K steps are held to 2 K times the one-step bound.
"""

import numpy as np
import pytest

import oracle
import workloads

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

TOL = {"fp32": 1e-5, "fp16": 2e-2, "bf16_split": 2e-2}
EPS = 1e-7
U24 = 2.0 ** -24


@pytest.fixture(scope="module", autouse=True)
def _need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2607_08754_gb300 import slorr
    slorr.load_library()   # raises if the extension is missing: no fallback


def _spiked(m, n, seed):
    """Small Gaussian noise plus a rank-4 spike (energy to concentrate)."""
    rng = np.random.default_rng(seed)
    U, _ = np.linalg.qr(rng.normal(size=(m, 4)))
    V, _ = np.linalg.qr(rng.normal(size=(n, 4)))
    W = rng.normal(0, 0.02, size=(m, n)) + (U * np.array([0.3, 0.25, 0.2, 0.15])) @ V.T
    return np.ascontiguousarray(W.astype(np.float32))


def _set():
    return [_spiked(48, 32, 1), _spiked(200, 130, 2), workloads.random_matrix((96, 256), 3, 0.05),
            workloads.random_matrix((333, 77), 4, 0.1), workloads.random_matrix((256, 256), 5, 1.0 / 16)]


def _eta(Ws, lam, target=0.05, variant="hoyer"):
    """A step moving every matrix by about `target` of its norm or less (an
    input chosen from W_0 and the oracle alone)."""
    co = oracle.pe_coefficients(6)
    r = [np.linalg.norm(W) / (lam * np.linalg.norm(oracle.reg_single(W.astype(np.float64), variant, co, EPS)[1]))
         for W in Ws]
    return float(target * min(r))


def _gpu_steps(Ws, eta, steps, compute="fp32", variant="hoyer", lam=1.0, grad_scale=1.0):
    from paper_2607_08754_gb300.slorr import Regularizer
    reg = Regularizer([W.shape for W in Ws], variant=variant, compute=compute, lam=lam, grad_scale=grad_scale)
    w = [torch.from_numpy(W).cuda() for W in Ws]
    traj = [[W.astype(np.float64) for W in Ws]]
    pers = []
    for _ in range(steps):
        per = torch.full((len(Ws),), float("nan"), device="cuda")
        reg.descent_step(w, eta, per_matrix=per)
        torch.cuda.synchronize()
        assert reg.status() == 0
        traj.append([x.double().cpu().numpy() for x in w])
        pers.append(per.double().cpu().numpy())
    return traj, pers


@pytest.mark.parametrize("compute", ["fp32", "fp16", "bf16_split"])
@pytest.mark.parametrize("variant", ["hoyer", "nuclear"])
def test_one_descent_step_matches_oracle(compute, variant):
    Ws = _set()
    lam, gs = 0.5, 1.5
    eta = _eta(Ws, lam * gs, variant=variant)
    traj, pers = _gpu_steps(Ws, eta, 1, compute, variant, lam, gs)
    co = oracle.pe_coefficients(6)
    for i, W in enumerate(Ws):
        W0 = W.astype(np.float64)
        ref, L = oracle.descent_step(W0, eta, variant, co, lam=lam, grad_scale=gs, eps=EPS)
        dW_ref = ref - W0
        dW = traj[1][i] - W0
        bound = TOL[compute] * np.linalg.norm(dW_ref) + U24 * np.linalg.norm(traj[1][i])
        assert np.linalg.norm(dW - dW_ref) <= bound, (i, np.linalg.norm(dW - dW_ref), bound)
        assert abs(pers[0][i] - L) <= TOL[compute] * abs(L) + 1e-6, (i, pers[0][i], L)


def test_descent_trajectory_matches_oracle_and_concentrates_energy():
    """Ten fp32-mode steps: the GPU trajectory stays within the accumulated
    bound of the oracle's, and shows what Props. 2 and 3 predict -- the Hoyer
    value falls at every step and the energy of the spike's rank rises."""
    Ws = _set()[:2]
    K = 10
    eta = _eta(Ws, 1.0, target=0.02)
    traj, pers = _gpu_steps(Ws, eta, K)
    ref_traj, ref_L = zip(*[oracle.descent_trajectory(W.astype(np.float64), eta, K, "hoyer",
                                                       oracle.pe_coefficients(6)) for W in Ws])
    for i in range(len(Ws)):
        step = max(np.linalg.norm(ref_traj[i][k + 1] - ref_traj[i][k]) for k in range(K))
        wmax = max(np.linalg.norm(X) for X in ref_traj[i])
        bound = 2 * K * (TOL["fp32"] * step + U24 * wmax)
        err = np.linalg.norm(traj[K][i] - ref_traj[i][K])
        assert err <= bound, (i, err, bound)
        L = [p[i] for p in pers]
        assert all(b < a for a, b in zip(L, L[1:])), L
        assert np.allclose(L, ref_L[i], rtol=TOL["fp32"])
        E = [oracle.energy(traj[k][i], 4) for k in range(K + 1)]
        assert all(b > a for a, b in zip(E, E[1:])), E


def test_zero_step_leaves_weights_bit_identical_and_matches_forward_loss():
    from paper_2607_08754_gb300.slorr import Regularizer
    Ws = _set()
    reg = Regularizer([W.shape for W in Ws], compute="fp16")
    w = [torch.from_numpy(W).cuda() for W in Ws]
    loss_d = reg.descent_step(w, 0.0).item()
    g = [torch.zeros_like(x) for x in w]
    loss_f = reg(w, g).item()
    torch.cuda.synchronize()
    assert reg.status() == 0
    for x, W in zip(w, Ws):
        assert torch.equal(x.cpu(), torch.from_numpy(W))
    assert loss_d == loss_f           # the same kernels in the same order


def test_descent_leaves_nonfinite_matrix_untouched():
    from paper_2607_08754_gb300.slorr import Regularizer
    W = workloads.random_matrix((64, 64), 11, 0.1)
    W[3, 5] = np.inf
    V = workloads.random_matrix((32, 48), 12, 0.1)
    reg = Regularizer([W.shape, V.shape])
    w = [torch.from_numpy(W).cuda(), torch.from_numpy(V).cuda()]
    reg.descent_step(w, 0.01)
    torch.cuda.synchronize()
    assert reg.status() == 6            # SLORR_ERR_NONFINITE
    assert torch.equal(w[0].cpu(), torch.from_numpy(W))
    assert not torch.equal(w[1].cpu(), torch.from_numpy(V))   # the finite matrix still steps
