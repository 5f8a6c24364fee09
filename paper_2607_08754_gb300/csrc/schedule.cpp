// Polar Express coefficient schedule for libslorr (host code, double precision).
//
// Sec. 3 "Computing the polar factor" and App. C.1: the polar factor is
// approximated by T odd quintic steps p_t(x) = a_t x + b_t x^3 + c_t x^5 chosen
// greedily: p_t is the best uniform approximation of 1 on the current interval
// [l_t, u_t] of normalised singular values, and the interval then becomes
// [p_t(l_t), 2 - p_t(l_t)] (l_1 = ell, u_1 = 1).  The paper does not print the
// coefficients and names, without defining them, the cited authors'
// stabilisations; this library reads them as
//   * a cushion: the step-t polynomial is designed on [max(l_t, kappa u_t), u_t]
//     and rescaled so that p(l_t) + p(u_t) = 2, where kappa is the interval
//     ratio whose minimax error is 9/11 (the image interval then has bound
//     ratio 1:10), found here by bisection;
//   * a safety factor s: steps 1..T-1 use x -> p_t(x / s); the last step does not.
// For design intervals narrower than 1e-4 the minimax quintic is replaced by
// its limit, the maximal-contact quintic (15 x - 10 x^3 + 3 x^5) / 8.
#include <cmath>

#include "internal.h"

namespace slorr {
namespace host {
namespace {

// Solve the 4x4 system M y = r in place by Gaussian elimination with partial
// pivoting.  Returns false when a pivot vanishes.
bool solve4(double M[4][4], double r[4]) {
    for (int col = 0; col < 4; ++col) {
        int piv = col;
        for (int row = col + 1; row < 4; ++row)
            if (std::fabs(M[row][col]) > std::fabs(M[piv][col])) piv = row;
        if (M[piv][col] == 0.0) return false;
        if (piv != col) {
            for (int k = 0; k < 4; ++k) {
                double t = M[col][k];
                M[col][k] = M[piv][k];
                M[piv][k] = t;
            }
            double t = r[col];
            r[col] = r[piv];
            r[piv] = t;
        }
        for (int row = col + 1; row < 4; ++row) {
            double f = M[row][col] / M[col][col];
            for (int k = col; k < 4; ++k) M[row][k] -= f * M[col][k];
            r[row] -= f * r[col];
        }
    }
    for (int row = 3; row >= 0; --row) {
        double acc = r[row];
        for (int k = row + 1; k < 4; ++k) acc -= M[row][k] * r[k];
        r[row] = acc / M[row][row];
    }
    return true;
}

double odd5(double a, double b, double c, double x) {
    double x2 = x * x;
    return x * (a + x2 * (b + x2 * c));
}

}  // namespace

// Remez exchange for min over (a, b, c) of max_{x in [lo, hi]} |1 - p(x)|.
// The unknown polynomial is written as p(x) = x (al + be zeta + ga T2(zeta)) with
// zeta = (x^2 - z0) / s mapping [lo^2, hi^2] onto [-1, 1] and T2 the Chebyshev
// polynomial 2 zeta^2 - 1, which keeps the reference system well conditioned.
// The optimum alternates 1 - p = +E, -E, +E, -E at lo < x1 < x2 < hi where
// x1, x2 are the zeros of p'.  out = {a, b, c, E}.
bool minimax_quintic(double lo, double hi, double out[4]) {
    if (!(lo > 0.0) || !(hi > lo)) return false;
    const double z0 = 0.5 * (hi * hi + lo * lo);
    const double s = 0.5 * (hi * hi - lo * lo);
    double x1 = lo + 0.3 * (hi - lo);
    double x2 = lo + 0.8 * (hi - lo);
    double al = 0, be = 0, ga = 0, E = 0;
    for (int it = 0; it < 60; ++it) {
        const double pts[4] = {lo, x1, x2, hi};
        const double sg[4] = {1.0, -1.0, 1.0, -1.0};
        double M[4][4], r[4];
        for (int k = 0; k < 4; ++k) {
            double zeta = (pts[k] * pts[k] - z0) / s;
            M[k][0] = pts[k];
            M[k][1] = pts[k] * zeta;
            M[k][2] = pts[k] * (2.0 * zeta * zeta - 1.0);
            M[k][3] = sg[k];
            r[k] = 1.0;
        }
        if (!solve4(M, r)) return false;
        al = r[0];
        be = r[1];
        ga = r[2];
        E = r[3];
        // Monomial coefficients in z = x^2 of q(z) = p(x)/x.
        const double q2 = 2.0 * ga / (s * s);
        const double q1 = be / s - 4.0 * ga * z0 / (s * s);
        const double q0 = al - ga - be * z0 / s + 2.0 * ga * z0 * z0 / (s * s);
        // p'(x) = q0 + 3 q1 z + 5 q2 z^2 = 0, solved in zeta = (z - z0)/s:
        //   5 q2 s^2 zeta^2 + (3 q1 s + 10 q2 z0 s) zeta + (q0 + 3 q1 z0 + 5 q2 z0^2) = 0
        const double A2 = 5.0 * q2 * s * s;
        const double A1 = 3.0 * q1 * s + 10.0 * q2 * z0 * s;
        const double A0 = q0 + 3.0 * q1 * z0 + 5.0 * q2 * z0 * z0;
        const double disc = A1 * A1 - 4.0 * A2 * A0;
        if (!(disc >= 0.0) || A2 == 0.0) return false;
        const double root = std::sqrt(disc);
        const double qq = -0.5 * (A1 + (A1 >= 0.0 ? root : -root));
        double r1 = qq / A2, r2 = A0 / qq;
        if (r1 > r2) {
            double t = r1;
            r1 = r2;
            r2 = t;
        }
        double n1 = std::sqrt(z0 + s * r1), n2 = std::sqrt(z0 + s * r2);
        n1 = std::fmin(std::fmax(n1, lo), hi);
        n2 = std::fmin(std::fmax(n2, lo), hi);
        const bool done = (n1 == x1 && n2 == x2);
        x1 = n1;
        x2 = n2;
        if (done) break;
    }
    const double q2 = 2.0 * ga / (s * s);
    const double q1 = be / s - 4.0 * ga * z0 / (s * s);
    const double q0 = al - ga - be * z0 / s + 2.0 * ga * z0 * z0 / (s * s);
    out[0] = q0;
    out[1] = q1;
    out[2] = q2;
    out[3] = E;
    return std::isfinite(q0) && std::isfinite(q1) && std::isfinite(q2) && std::isfinite(E);
}

double cushion_ratio() {
    double lo = 1e-6, hi = 0.5;
    double out[4];
    for (int it = 0; it < 200; ++it) {
        double mid = 0.5 * (lo + hi);
        if (mid == lo || mid == hi) break;
        if (!minimax_quintic(mid, 1.0, out)) return NAN;
        if (out[3] > 9.0 / 11.0)
            lo = mid;
        else
            hi = mid;
    }
    return 0.5 * (lo + hi);
}

bool pe_schedule(int T, double ell, double cushion, double safety, double* abc) {
    if (T < 1 || !(ell > 0.0 && ell < 1.0) || !(safety >= 1.0)) return false;
    const double kappa = cushion < 0.0 ? cushion_ratio() : cushion;
    if (!std::isfinite(kappa)) return false;
    double lo = ell, hi = 1.0;
    for (int t = 0; t < T; ++t) {
        const double dlo = std::fmax(lo, kappa * hi);
        double a, b, c;
        if (hi - dlo < 1e-4) {
            a = 15.0 / 8.0;
            b = -10.0 / 8.0;
            c = 3.0 / 8.0;
        } else {
            double out[4];
            if (!minimax_quintic(dlo, hi, out)) return false;
            a = out[0];
            b = out[1];
            c = out[2];
        }
        const double rescale = 2.0 / (odd5(a, b, c, lo) + odd5(a, b, c, hi));
        a *= rescale;
        b *= rescale;
        c *= rescale;
        abc[3 * t + 0] = a;
        abc[3 * t + 1] = b;
        abc[3 * t + 2] = c;
        lo = odd5(a, b, c, lo);
        hi = 2.0 - lo;
    }
    if (safety != 1.0) {
        for (int t = 0; t < T - 1; ++t) {
            abc[3 * t + 0] /= safety;
            abc[3 * t + 1] /= safety * safety * safety;
            abc[3 * t + 2] /= safety * safety * safety * safety * safety;
        }
    }
    return true;
}

}  // namespace host
}  // namespace slorr
