// esb_alpha.cpp -- host solver for the DDA scale alpha*(b,k) (Sec. III-D).
//
// D(alpha) (Eq. objective_function_expansion) is the mean squared error of
// nearest-element projection of N(0,1) data on the non-negative half, each
// set element alpha*q owning the interval between the midpoints to its
// neighbours (the last one up to infinity).  Over one interval [l, h],
//   int (t-q)^2 phi = M2 - 2 q M1 + q^2 M0,
// with the truncated moments M0 = Phi(h)-Phi(l), M1 = phi(l)-phi(h),
// M2 = M0 + l phi(l) - h phi(h).  alpha* is the first local minimum of D
// from small alpha (Eq. optimal_alpha_seeking; D is not convex for large
// N, and the first minimum is the value Table 1 prints), located on a
// geometric grid and refined as the zero of dD/dalpha.  For power-of-two
// like sets with very large N, D has a ladder of minima at ever smaller
// alpha; the search range [1e-4, 4] (the paper searches (0, 3]) fixes which
// one is meant.  Every format of Table 1 has its first minimum inside it.
#include <cmath>
#include <vector>

#include "esb_internal.h"

namespace esb {

namespace {

void nonneg_elements(int b, int k, std::vector<double>& s)
{
    const int N = (1 << (b - k - 1)) - 1;
    s.clear();
    for (int f = 0; f < (1 << k); f++) s.push_back(std::ldexp((double)f, -k));
    for (int i = 1; i <= N; i++)
        for (int f = 0; f < (1 << k); f++) s.push_back(std::ldexp((double)((1 << k) + f), i - k - 1));
}

inline double pdf(double t) { return std::exp(-0.5 * t * t) * 0.39894228040143267794; }

// Upper-tail mass Q(t) = 1 - Phi(t) (accurate for large t).
inline double upper(double t) { return 0.5 * std::erfc(t * 0.70710678118654752440); }

double objective(double alpha, const std::vector<double>& s)
{
    const size_t n = s.size();
    double total = 0.0;
    for (size_t j = 0; j < n; j++) {
        const double q = alpha * s[j];
        const double l = (j == 0) ? 0.0 : 0.5 * alpha * (s[j - 1] + s[j]);
        const bool last = (j + 1 == n);
        const double h = last ? 0.0 : 0.5 * alpha * (s[j] + s[j + 1]);
        const double M0 = upper(l) - (last ? 0.0 : upper(h));
        const double M1 = pdf(l) - (last ? 0.0 : pdf(h));
        const double M2 = M0 + l * pdf(l) - (last ? 0.0 : h * pdf(h));
        total += M2 - 2.0 * q * M1 + q * q * M0;
    }
    return total;
}

// dD/dalpha: the boundary terms cancel because each boundary is the
// midpoint of its two elements, so D' = -2 sum_j q_j (M1_j - alpha q_j M0_j).
double slope(double alpha, const std::vector<double>& s)
{
    const size_t n = s.size();
    double g = 0.0;
    for (size_t j = 0; j < n; j++) {
        const double l = (j == 0) ? 0.0 : 0.5 * alpha * (s[j - 1] + s[j]);
        const bool last = (j + 1 == n);
        const double h = last ? 0.0 : 0.5 * alpha * (s[j] + s[j + 1]);
        const double M0 = upper(l) - (last ? 0.0 : upper(h));
        const double M1 = pdf(l) - (last ? 0.0 : pdf(h));
        g -= 2.0 * s[j] * (M1 - alpha * s[j] * M0);
    }
    return g;
}

}  // namespace

double alpha_star_solve(int b, int k, double* dda)
{
    std::vector<double> s;
    nonneg_elements(b, k, s);
    // Bracket the first local minimum on a geometric grid ...
    const double a_lo = 1e-4, a_hi = 4.0;   // search range of alpha*; see the reading above
    const int G = 30000;
    const double ratio = std::pow(a_hi / a_lo, 1.0 / (G - 1));
    double prev2 = objective(a_lo, s), prev = objective(a_lo * ratio, s);
    double lo = a_lo, hi = a_hi;
    double a = a_lo * ratio;
    for (int i = 2; i < G; i++) {
        const double an = a * ratio;
        const double cur = objective(an, s);
        if (prev < prev2 && prev <= cur) { lo = a / ratio; hi = an; break; }
        prev2 = prev; prev = cur; a = an;
    }
    // ... then regula falsi (Illinois variant) on the zero of D'.
    double flo = slope(lo, s), fhi = slope(hi, s);
    int side = 0;
    for (int it = 0; it < 300 && flo < 0.0 && fhi > 0.0; it++) {
        const double x = (lo * fhi - hi * flo) / (fhi - flo);
        if (!(x > lo && x < hi)) break;
        const double fx = slope(x, s);
        if (fx == 0.0) { lo = hi = x; break; }
        if (fx < 0.0) { lo = x; flo = fx; if (side == -1) fhi *= 0.5; side = -1; }
        else { hi = x; fhi = fx; if (side == 1) flo *= 0.5; side = 1; }
        if (hi - lo <= 4e-16 * hi) break;
    }
    const double best = 0.5 * (lo + hi);
    if (dda) *dda = 2.0 * objective(best, s);
    return best;
}

}  // namespace esb
