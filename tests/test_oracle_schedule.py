"""Pins for the oracle's Polar Express schedule (Sec. 3, App. C.1, Prop. 1).

The schedule is not printed in the paper, so it is pinned to its definition:
minimax optimality (equioscillation, and agreement with an independent
linear-programming minimax solve), the interval recurrence, the cushion and
safety-factor readings, the maximal-contact limit and Prop. 1's delta.
"""

import numpy as np
import pytest

from oracle import schedule as pe


def _p(abc, x):
    a, b, c = abc
    return a * x + b * x ** 3 + c * x ** 5


@pytest.mark.parametrize("lo,hi", [(1e-3, 1.0), (0.02, 1.0), (0.1, 1.9), (0.5, 1.5), (0.9, 1.1)])
def test_remez_equioscillates(lo, hi):
    a, b, c, E, x1, x2 = pe.minimax_odd_quintic(lo, hi)
    pts = [lo, x1, x2, hi]
    errs = [1.0 - _p((a, b, c), x) for x in pts]
    # alternating signs +E, -E, +E, -E at the four extremal points
    assert np.allclose(errs, [E, -E, E, -E], rtol=1e-10, atol=1e-13)
    xs = np.linspace(lo, hi, 400001)
    emax = np.max(np.abs(1.0 - _p((a, b, c), xs)))
    assert emax == pytest.approx(E, rel=1e-9)
    assert lo < x1 < x2 < hi


@pytest.mark.parametrize("lo,hi", [(1e-2, 1.0), (0.2, 1.8)])
def test_remez_matches_linear_programming_minimax(lo, hi):
    """An independent minimax solve: minimise t s.t. |1 - p(x_k)| <= t on a grid."""
    scipy_opt = pytest.importorskip("scipy.optimize")
    xs = np.concatenate([np.geomspace(lo, hi, 3000), np.linspace(lo, hi, 3000)])
    V = np.stack([xs, xs ** 3, xs ** 5], axis=1)
    # variables (a, b, c, t); rows:  V p - t <= 1 ... i.e. p - 1 <= t and 1 - p <= t
    A_ub = np.vstack([np.hstack([V, -np.ones((len(xs), 1))]),
                      np.hstack([-V, -np.ones((len(xs), 1))])])
    b_ub = np.concatenate([np.ones(len(xs)), -np.ones(len(xs))])
    res = scipy_opt.linprog(c=[0, 0, 0, 1], A_ub=A_ub, b_ub=b_ub,
                            bounds=[(None, None)] * 4, method="highs")
    assert res.success
    a, b, c, E = pe.minimax_odd_quintic(lo, hi)[:4]
    assert res.x[3] == pytest.approx(E, rel=1e-4)
    got = np.array([a, b, c])
    assert np.allclose(res.x[:3], got, rtol=2e-3, atol=2e-3 * np.abs(got).max())


def test_cushion_ratio_definition():
    k = pe.cushion_ratio()
    a, b, c, E = pe.minimax_odd_quintic(k, 1.0)[:4]
    assert E == pytest.approx(9.0 / 11.0, rel=1e-12)
    # image interval [1 - E, 1 + E] has bound ratio 1 : 10
    assert (1.0 - E) / (1.0 + E) == pytest.approx(0.1, rel=1e-11)
    assert 0.02 < k < 0.03


def test_schedule_without_stabilisations_is_plain_greedy_minimax():
    sch = pe.pe_schedule(T=6, ell=1e-3, cushion=0.0, safety=1.0)
    lo, hi = 1e-3, 1.0
    for t in range(6):
        a, b, c, E = pe.minimax_odd_quintic(lo, hi)[:4]
        got = sch["coeffs"][t]
        assert np.allclose(got, [a, b, c], rtol=1e-12, atol=1e-12)
        # optimal polynomials are already centred: p(lo) = 1 - E, p(hi) = 1 + E
        assert _p(got, lo) == pytest.approx(1.0 - E, rel=1e-10)
        assert _p(got, hi) == pytest.approx(1.0 + E, rel=1e-10)
        lo = _p(got, lo)
        hi = 2.0 - lo


def test_schedule_recurrence_and_centering_with_cushion():
    sch = pe.pe_schedule(T=6, ell=1e-3, cushion=None, safety=1.0)
    k = sch["kappa"]
    lo, hi = 1e-3, 1.0
    for t, (dlo, dhi, E) in enumerate(sch["design"]):
        assert dlo == pytest.approx(lo, rel=1e-13) and dhi == pytest.approx(hi, rel=1e-13)
        abc = sch["coeffs"][t]
        assert _p(abc, lo) + _p(abc, hi) == pytest.approx(2.0, rel=1e-13)
        # the design polynomial is the minimax one on [max(lo, k hi), hi], rescaled
        ref = np.array(pe.minimax_odd_quintic(max(lo, k * hi), hi)[:3])
        ratio = abc / ref
        assert np.allclose(ratio, ratio[0], rtol=1e-10)
        # p(lo) is the minimum and p(hi) the maximum of p over [lo, hi]
        xs = np.linspace(lo, hi, 200001)
        v = _p(abc, xs)
        assert v.min() >= _p(abc, lo) * (1 - 1e-12)
        assert v.max() <= _p(abc, hi) * (1 + 1e-12)
        lo = _p(abc, lo)
        hi = 2.0 - lo
    # the cushion only changes the early, badly-conditioned steps
    plain = pe.pe_schedule(T=6, ell=1e-3, cushion=0.0, safety=1.0)["coeffs"]
    assert not np.allclose(plain[0], sch["coeffs"][0])


def test_safety_factor_reading():
    base = pe.pe_schedule(T=6, safety=1.0)["coeffs"]
    safe = pe.pe_schedule(T=6, safety=1.01)["coeffs"]
    s = 1.01
    for t in range(5):
        assert np.allclose(safe[t], base[t] / np.array([s, s ** 3, s ** 5]), rtol=1e-14)
        x = np.linspace(0, 1.2, 101)
        assert np.allclose(_p(safe[t], x), _p(base[t], x / s), rtol=1e-12, atol=1e-14)
    assert np.array_equal(safe[5], base[5])


def test_narrow_interval_limit_polynomial():
    a, b, c = 15 / 8, -10 / 8, 3 / 8
    # maximal contact at 1: p(1) = 1, p'(1) = 0, p''(1) = 0
    assert a + b + c == pytest.approx(1.0)
    assert a + 3 * b + 5 * c == pytest.approx(0.0, abs=1e-15)
    assert 6 * b + 20 * c == pytest.approx(0.0, abs=1e-15)
    # the minimax quintic on [1 - w/2, 1 + w/2] tends to it as O(w^2)
    d = []
    for w in [1e-1, 1e-2]:
        got = pe.minimax_odd_quintic(1 - w / 2, 1 + w / 2)[0]
        d.append(got - a)
    assert d[0] / d[1] == pytest.approx(100.0, rel=0.05)
    # long schedules reach the narrow regime and stay finite and convergent
    sch = pe.pe_schedule(T=10)
    assert np.all(np.isfinite(sch["coeffs"]))
    assert np.allclose(sch["coeffs"][-1], [a, b, c], rtol=1e-6)


def test_design_errors_decrease_and_T1():
    sch = pe.pe_schedule(T=6)
    lows = [d[0] for d in sch["design"]]
    assert all(l2 > l1 for l1, l2 in zip(lows, lows[1:]))
    # T = 1: a single, unscaled (last-step) polynomial
    one = pe.pe_schedule(T=1)
    assert np.array_equal(one["coeffs"][0], pe.pe_schedule(T=1, safety=1.0)["coeffs"][0])


def test_prop1_delta_and_achieved_error():
    d = pe.paper_delta(1e-3, 6, 5)
    assert d == pytest.approx((1 - 1e-6) ** 729, rel=1e-14)
    assert 0.999 < d < 0.9993            # vacuous at the paper's settings
    co = pe.pe_coefficients(T=6)
    E_T = pe.achieved_error(co)
    assert 0.0 < E_T < d                 # sharpened bound is within Prop. 1's
    # error shrinks with more steps (NEXT-style T sweep)
    Es = [pe.achieved_error(pe.pe_coefficients(T=t)) for t in (4, 6, 8)]
    assert Es[0] > Es[1] > Es[2]


def test_scalar_map_zero_and_odd():
    co = pe.pe_coefficients()
    assert pe.pe_scalar_map(np.array([0.0]), co)[0] == 0.0
    x = np.linspace(-1, 1, 11)
    assert np.allclose(pe.pe_scalar_map(-x, co), -pe.pe_scalar_map(x, co))
