"""Polar Express coefficient schedule, fp64 (oracle; test infrastructure only).

What the paper fixes (Sec. 3 "Computing the polar factor"; App. C.1 "On our
use of Polar Express"; Prop. 1 and App. B):

* the polar factor U V^T is approximated by T steps of an odd polynomial
  iteration of degree d = 5 (q = 2) applied to W / (||W||_F + eps);
* the lower bound on the normalised nonzero singular values is ell = 1e-3;
* T = 6 steps by default;
* each step's polynomial is the one chosen by Polar Express (greedy minimax
  optimal odd polynomial for the current singular-value interval), with the
  cited authors' recommended numerical stabilisations.

The coefficient values themselves are not printed in the paper.  They are
generated here from the definition of the greedy minimax schedule:

    for t = 1..T:   p_t = argmin over odd quintics p of max_{x in [l_t, u_t]} |1 - p(x)|
                    l_{t+1} = p_t(l_t),  u_{t+1} = 2 - l_{t+1}       (l_1 = ell, u_1 = 1)

and two stabilisations whose exact form is a reading (the paper names them
without defining them):

* cushion: the polynomial of step t is designed on [max(l_t, kappa*u_t), u_t]
  and then rescaled so that p(l_t) + p(u_t) = 2 (so the recurrence above still
  holds).  kappa is the lower-bound ratio at which the minimax quintic on
  [kappa, 1] has error exactly 9/11, i.e. maps its interval onto one whose
  bound ratio is 1:10; it is found by bisection, not stored.
* safety factor s = 1.01: the polynomials of steps 1..T-1 are replaced by
  x -> p_t(x / s) after the schedule has been designed; the last step is left
  unchanged.

Once the design interval is narrower than 1e-4 the minimax quintic coincides
(to below fp64 resolution of the schedule) with the maximal-contact polynomial
(15 x - 10 x^3 + 3 x^5) / 8, which is used there instead of a Remez solve.
"""

from __future__ import annotations

import numpy as np

# Width below which the Remez solve is replaced by the maximal-contact quintic.
NARROW_WIDTH = 1e-4
# Error level that defines the cushion ratio kappa (image bound ratio 1:10).
CUSHION_ERROR = 9.0 / 11.0


def _eval_odd(a: float, b: float, c: float, x):
    """p(x) = a x + b x^3 + c x^5."""
    x2 = x * x
    return x * (a + x2 * (b + x2 * c))


def minimax_odd_quintic(lo: float, hi: float, iters: int = 60):
    """Best uniform approximation of 1 on [lo, hi] by p(x) = a x + b x^3 + c x^5.

    Remez exchange on the Chebyshev system {x, x^3, x^5} (0 < lo < hi): the
    optimum equioscillates at four points lo < x1 < x2 < hi with
    1 - p = +E, -E, +E, -E, and x1, x2 are the roots of p'(x) = 0.  The linear
    system is written in a local quadratic basis in z = x^2 so that it stays
    well conditioned for narrow intervals.

    Returns (a, b, c, E, x1, x2).
    """
    lo = float(lo)
    hi = float(hi)
    if not (0.0 < lo < hi):
        raise ValueError("need 0 < lo < hi")
    z0 = 0.5 * (lo * lo + hi * hi)
    s = 0.5 * (hi * hi - lo * lo)
    w = hi - lo
    x1, x2 = lo + 0.3 * w, lo + 0.8 * w
    signs = np.array([1.0, -1.0, 1.0, -1.0])
    for _ in range(iters):
        pts = np.array([lo, x1, x2, hi])
        d = (pts * pts - z0) / s
        M = np.stack([pts, pts * d, pts * d * d, signs], axis=1)
        al, be, ga, E = np.linalg.solve(M, np.ones(4))
        # p(x) = x (al + be d + ga d^2);  p'(x) = 0  <=>
        # 5 ga d^2 + (3 be + 4 ga z0/s) d + (al + 2 be z0/s) = 0
        qa = 5.0 * ga
        qb = 3.0 * be + 4.0 * ga * z0 / s
        qc = al + 2.0 * be * z0 / s
        disc = qb * qb - 4.0 * qa * qc
        if disc < 0.0 or qa == 0.0:
            raise ArithmeticError("Remez exchange lost the two interior extrema")
        root = np.sqrt(disc)
        qq = -0.5 * (qb + np.copysign(root, qb))
        r = sorted([qq / qa, qc / qq])
        nx1 = np.sqrt(z0 + s * r[0])
        nx2 = np.sqrt(z0 + s * r[1])
        nx1 = min(max(nx1, lo), hi)
        nx2 = min(max(nx2, lo), hi)
        if nx1 == x1 and nx2 == x2:
            break
        x1, x2 = nx1, nx2
    c = ga / (s * s)
    b = be / s - 2.0 * ga * z0 / (s * s)
    a = al - be * z0 / s + ga * z0 * z0 / (s * s)
    return float(a), float(b), float(c), float(E), float(x1), float(x2)


def cushion_ratio() -> float:
    """kappa with minimax error E(kappa) = 9/11 on [kappa, 1] (bisection).

    E(l) decreases monotonically in l on (0, 1)."""
    lo, hi = 1e-6, 0.5
    for _ in range(200):
        mid = 0.5 * (lo + hi)
        if mid == lo or mid == hi:
            break
        if minimax_odd_quintic(mid, 1.0)[3] > CUSHION_ERROR:
            lo = mid
        else:
            hi = mid
    return 0.5 * (lo + hi)


def pe_schedule(T: int = 6, ell: float = 1e-3, cushion: float | None = None,
                safety: float = 1.01):
    """Greedy minimax Polar Express schedule.

    cushion: None -> the derived kappa; 0 -> no cushion; else the ratio used.
    safety:  factor s (1 disables it).

    Returns a dict with
      'coeffs'  (T, 3) array of (a_t, b_t, c_t) as used by the iteration,
      'design'  list of (l_t, u_t, E_t) of the designed polynomials,
      'kappa', 'ell', 'safety'.
    """
    if T < 1:
        raise ValueError("T must be >= 1")
    if not (0.0 < ell < 1.0):
        raise ValueError("ell must lie in (0, 1)")
    kappa = cushion_ratio() if cushion is None else float(cushion)
    lo, hi = float(ell), 1.0
    coeffs = []
    design = []
    for _ in range(T):
        lo_d = max(lo, kappa * hi)
        if hi - lo_d < NARROW_WIDTH:
            a, b, c, E = 15.0 / 8.0, -10.0 / 8.0, 3.0 / 8.0, float("nan")
        else:
            a, b, c, E = minimax_odd_quintic(lo_d, hi)[:4]
        # Re-centre on [lo, hi]:  p(lo) + p(hi) = 2.
        r = 2.0 / (_eval_odd(a, b, c, lo) + _eval_odd(a, b, c, hi))
        a, b, c = a * r, b * r, c * r
        design.append((lo, hi, E))
        coeffs.append([a, b, c])
        lo = _eval_odd(a, b, c, lo)
        hi = 2.0 - lo
    coeffs = np.array(coeffs, dtype=np.float64)
    s = float(safety)
    if s != 1.0:
        for t in range(T - 1):
            coeffs[t, 0] /= s
            coeffs[t, 1] /= s ** 3
            coeffs[t, 2] /= s ** 5
    return {"coeffs": coeffs, "design": design, "kappa": kappa, "ell": ell,
            "safety": s}


def pe_coefficients(T: int = 6, ell: float = 1e-3, cushion: float | None = None,
                    safety: float = 1.01) -> np.ndarray:
    """The (T, 3) coefficient table (a_t, b_t, c_t) of ``pe_schedule``."""
    return pe_schedule(T, ell, cushion, safety)["coeffs"]


def pe_scalar_map(x, coeffs):
    """g(x) = p_T(...p_1(x)): the map the iteration applies to each singular value.

    The matrix step X <- a X + (b A + c A^2) X with A = X X^T acts on the SVD
    X = U diag(x) V^T as x -> a x + b x^3 + c x^5 (App. B, "zero singular values
    stay zero": p(0) = 0)."""
    y = np.asarray(x, dtype=np.float64).copy()
    for a, b, c in np.asarray(coeffs, dtype=np.float64):
        y = _eval_odd(a, b, c, y)
    return y


def paper_delta(ell: float = 1e-3, T: int = 6, d: int = 5) -> float:
    """delta = |1 - ell^2|^((q+1)^T) with d = 2q + 1 (Prop. 1)."""
    q = (d - 1) // 2
    return abs(1.0 - ell * ell) ** ((q + 1) ** T)


def achieved_error(coeffs, ell: float = 1e-3, hi: float = 1.0, n: int = 200001) -> float:
    """E_T = max_{x in [ell, hi]} |1 - g(x)| of the composed scalar map.

    Dense logarithmic + linear grid, refined by golden-section around the
    worst grid point; used as the sharpened form of Prop. 1's delta."""
    xs = np.unique(np.concatenate([np.geomspace(ell, hi, n), np.linspace(ell, hi, n)]))
    err = np.abs(1.0 - pe_scalar_map(xs, coeffs))
    i = int(np.argmax(err))
    best = float(err[i])
    lo = xs[max(i - 1, 0)]
    up = xs[min(i + 1, len(xs) - 1)]
    f = lambda t: -abs(1.0 - float(pe_scalar_map(np.array([t]), coeffs)[0]))
    gr = (np.sqrt(5.0) - 1.0) / 2.0
    a, b = lo, up
    for _ in range(100):
        c1 = b - gr * (b - a)
        c2 = a + gr * (b - a)
        if f(c1) < f(c2):
            b = c2
        else:
            a = c1
    return max(best, -f(0.5 * (a + b)))
