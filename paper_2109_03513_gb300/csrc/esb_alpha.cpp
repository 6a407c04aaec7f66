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
// The paper assumes N(0,1) data; the same search runs for two other data
// densities: Laplace with unit variance (heavy tails) and the empirical
// density of a histogram of the normalised data.
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

// Truncated moments of the data density over one interval [l, h] of the
// non-negative half (h = +inf for the last element's interval):
// m_r = int_l^h t^r p(t) dt.
struct Moments { double m0, m1, m2; };

// N(0,1): m0 = Q(l) - Q(h), m1 = phi(l) - phi(h), m2 = m0 + l phi(l) - h phi(h).
struct Gaussian {
    Moments between(double l, double h, bool last) const
    {
        Moments m;
        m.m0 = upper(l) - (last ? 0.0 : upper(h));
        m.m1 = pdf(l) - (last ? 0.0 : pdf(h));
        m.m2 = m.m0 + l * pdf(l) - (last ? 0.0 : h * pdf(h));
        return m;
    }
};

// Laplace with unit variance, p(t) = (lambda / 2) exp(-lambda |t|), lambda =
// sqrt 2: the upper tails int_x^inf t^r p are exp(-lambda x) / 2 times 1,
// x + 1/lambda and x^2 + 2x/lambda + 2/lambda^2.
struct Laplace {
    static constexpr double lam = 1.41421356237309504880;
    static void tails(double x, double& g0, double& g1, double& g2)
    {
        const double e = 0.5 * std::exp(-lam * x);
        g0 = e;
        g1 = (x + 1.0 / lam) * e;
        g2 = (x * x + 2.0 * x / lam + 2.0 / (lam * lam)) * e;
    }
    Moments between(double l, double h, bool last) const
    {
        double a0, a1, a2, b0 = 0.0, b1 = 0.0, b2 = 0.0;
        tails(l, a0, a1, a2);
        if (!last) tails(h, b0, b1, b2);
        return Moments{a0 - b0, a1 - b1, a2 - b2};
    }
};

// Piecewise-constant density of a histogram of |t| (bins of width w over
// [0, t_max), bin i holding counts[i] of the n values): mass counts[i] / (2n)
// spread evenly over the bin, so that the half-line holds 1/2 as for the
// symmetric densities above.  Suffix sums give the upper tails exactly.
struct Histogram {
    int nb = 0;
    double w = 0.0;
    std::vector<double> p, s0, s1, s2;   // density per bin; tails from each bin edge
    Histogram(const unsigned long long* counts, int nbins, double t_max) : nb(nbins), w(t_max / nbins)
    {
        double n = 0.0;
        for (int i = 0; i < nb; i++) n += (double)counts[i];
        p.assign(nb, 0.0);
        s0.assign(nb + 1, 0.0); s1.assign(nb + 1, 0.0); s2.assign(nb + 1, 0.0);
        for (int i = 0; i < nb; i++) p[i] = n > 0.0 ? (double)counts[i] / (2.0 * n * w) : 0.0;
        for (int i = nb - 1; i >= 0; i--) {
            const double e0 = i * w, e1 = (i + 1) * w;
            s0[i] = s0[i + 1] + p[i] * (e1 - e0);
            s1[i] = s1[i + 1] + p[i] * (e1 * e1 - e0 * e0) / 2.0;
            s2[i] = s2[i + 1] + p[i] * (e1 * e1 * e1 - e0 * e0 * e0) / 3.0;
        }
    }
    void tails(double x, double& g0, double& g1, double& g2) const
    {
        if (x <= 0.0) { g0 = s0[0]; g1 = s1[0]; g2 = s2[0]; return; }
        const int i = (int)std::floor(x / w);
        if (i >= nb) { g0 = g1 = g2 = 0.0; return; }
        const double e1 = (i + 1) * w;
        g0 = s0[i + 1] + p[i] * (e1 - x);
        g1 = s1[i + 1] + p[i] * (e1 * e1 - x * x) / 2.0;
        g2 = s2[i + 1] + p[i] * (e1 * e1 * e1 - x * x * x) / 3.0;
    }
    Moments between(double l, double h, bool last) const
    {
        double a0, a1, a2, b0 = 0.0, b1 = 0.0, b2 = 0.0;
        tails(l, a0, a1, a2);
        if (!last) tails(h, b0, b1, b2);
        return Moments{a0 - b0, a1 - b1, a2 - b2};
    }
};

// Over the interval of element q: int (t - q)^2 p = m2 - 2 q m1 + q^2 m0.
template <class Dens>
double objective(double alpha, const std::vector<double>& s, const Dens& d)
{
    const size_t n = s.size();
    double total = 0.0;
    for (size_t j = 0; j < n; j++) {
        const double q = alpha * s[j];
        const double l = (j == 0) ? 0.0 : 0.5 * alpha * (s[j - 1] + s[j]);
        const bool last = (j + 1 == n);
        const double h = last ? 0.0 : 0.5 * alpha * (s[j] + s[j + 1]);
        const Moments m = d.between(l, h, last);
        total += m.m2 - 2.0 * q * m.m1 + q * q * m.m0;
    }
    return total;
}

// dD/dalpha: the boundary terms cancel because each boundary is the
// midpoint of its two elements (and the density is bounded), so
// D' = -2 sum_j q_j (m1_j - alpha q_j m0_j).
template <class Dens>
double slope(double alpha, const std::vector<double>& s, const Dens& d)
{
    const size_t n = s.size();
    double g = 0.0;
    for (size_t j = 0; j < n; j++) {
        const double l = (j == 0) ? 0.0 : 0.5 * alpha * (s[j - 1] + s[j]);
        const bool last = (j + 1 == n);
        const double h = last ? 0.0 : 0.5 * alpha * (s[j] + s[j + 1]);
        const Moments m = d.between(l, h, last);
        g -= 2.0 * s[j] * (m.m1 - alpha * s[j] * m.m0);
    }
    return g;
}

template <class Dens>
double first_minimum(int b, int k, const Dens& d, double* dda)
{
    std::vector<double> s;
    nonneg_elements(b, k, s);
    // Bracket the first local minimum on a geometric grid ...
    const double a_lo = 1e-4, a_hi = 4.0;   // search range of alpha*; see the reading above
    const int G = 30000;
    const double ratio = std::pow(a_hi / a_lo, 1.0 / (G - 1));
    double prev2 = objective(a_lo, s, d), prev = objective(a_lo * ratio, s, d);
    double lo = a_lo, hi = a_hi;
    double a = a_lo * ratio;
    for (int i = 2; i < G; i++) {
        const double an = a * ratio;
        const double cur = objective(an, s, d);
        if (prev < prev2 && prev <= cur) { lo = a / ratio; hi = an; break; }
        prev2 = prev; prev = cur; a = an;
    }
    // ... then regula falsi (Illinois variant) on the zero of D'.
    double flo = slope(lo, s, d), fhi = slope(hi, s, d);
    int side = 0;
    for (int it = 0; it < 300 && flo < 0.0 && fhi > 0.0; it++) {
        const double x = (lo * fhi - hi * flo) / (fhi - flo);
        if (!(x > lo && x < hi)) break;
        const double fx = slope(x, s, d);
        if (fx == 0.0) { lo = hi = x; break; }
        if (fx < 0.0) { lo = x; flo = fx; if (side == -1) fhi *= 0.5; side = -1; }
        else { hi = x; fhi = fx; if (side == 1) flo *= 0.5; side = 1; }
        if (hi - lo <= 4e-16 * hi) break;
    }
    const double best = 0.5 * (lo + hi);
    if (dda) *dda = 2.0 * objective(best, s, d);
    return best;
}

}  // namespace

double alpha_star_solve(int b, int k, double* dda) { return first_minimum(b, k, Gaussian{}, dda); }

double alpha_star_solve_laplace(int b, int k, double* dda) { return first_minimum(b, k, Laplace{}, dda); }

double alpha_star_solve_hist(const unsigned long long* counts, int nbins, double t_max, int b, int k, double* dda)
{
    return first_minimum(b, k, Histogram(counts, nbins, t_max), dda);
}

}  // namespace esb
