// Daubechies filter banks by spectral factorisation (host code).
//
// The WSM uses db4 and the WTA Haar (Section 4.1; Fig. "wavelet ablation"
// names the bases).  The filter of order p is the minimum-phase square root
// of |m0(w)|^2 = cos^{2p}(w/2) P(sin^2(w/2)), P(y) = sum_{k<p} C(p-1+k,k) y^k
// (Daubechies 1988).  Roots of P are found with the Durand-Kerner iteration
// and polished by Newton steps in long double; every root y maps to the root
// z of z^2 + (4y-2) z + 1 = 0 inside the unit circle; the filter is the
// coefficient list of (z+1)^p prod (z - z_i), normalised to sum sqrt(2).
#include <cmath>
#include <complex>
#include <vector>

#include "wz_internal.cuh"

namespace wz {

namespace {

using cld = std::complex<long double>;

long double binom(int n, int k) {
    long double r = 1.0L;
    for (int i = 1; i <= k; ++i) r = r * (n - k + i) / i;
    return r;
}

// Evaluate sum c[k] x^k (ascending coefficients) and its derivative.
void horner(const std::vector<long double> &c, cld x, cld &v, cld &dv) {
    v = 0.0L;
    dv = 0.0L;
    for (int k = (int)c.size() - 1; k >= 0; --k) {
        dv = dv * x + v;
        v = v * x + c[k];
    }
}

std::vector<cld> poly_roots(const std::vector<long double> &c) {
    const int deg = (int)c.size() - 1;
    std::vector<cld> r(deg);
    if (deg <= 0) return r;
    const long double lead = c[deg];
    const cld seed(0.4L, 0.9L);
    cld s = 1.0L;
    for (int i = 0; i < deg; ++i) {
        r[i] = s;
        s *= seed;
    }
    for (int it = 0; it < 2000; ++it) {
        long double moved = 0.0L;
        for (int i = 0; i < deg; ++i) {
            cld v, dv;
            horner(c, r[i], v, dv);
            cld den = lead;
            for (int j = 0; j < deg; ++j)
                if (j != i) den *= (r[i] - r[j]);
            cld step = v / den;
            r[i] -= step;
            moved = std::max(moved, std::abs(step));
        }
        if (moved < 1e-18L) break;
    }
    for (int i = 0; i < deg; ++i) {
        for (int it = 0; it < 5; ++it) {
            cld v, dv;
            horner(c, r[i], v, dv);
            if (std::abs(dv) == 0.0L) break;
            r[i] -= v / dv;
        }
    }
    return r;
}

}  // namespace

bool daubechies(int p, double *dec_lo, double *dec_hi, double *rec_lo, double *rec_hi) {
    if (p < 1 || 2 * p > kMaxTaps) return false;
    std::vector<long double> P(p);
    for (int k = 0; k < p; ++k) P[k] = binom(p - 1 + k, k);
    std::vector<cld> zs;
    for (const cld &y : poly_roots(P)) {
        const cld b = 4.0L * y - 2.0L;                 // z^2 + b z + 1 = 0
        const cld d = std::sqrt(b * b - 4.0L);
        const cld z1 = (-b + d) / 2.0L, z2 = (-b - d) / 2.0L;
        zs.push_back(std::abs(z1) < 1.0L ? z1 : z2);
    }
    for (int i = 0; i < p; ++i) zs.push_back(cld(-1.0L, 0.0L));
    // Coefficients of prod (z - z_i), highest power first.
    std::vector<cld> poly(1, cld(1.0L, 0.0L));
    for (const cld &z : zs) {
        std::vector<cld> next(poly.size() + 1, cld(0.0L, 0.0L));
        for (size_t k = 0; k < poly.size(); ++k) {
            next[k] += poly[k];
            next[k + 1] -= poly[k] * z;
        }
        poly.swap(next);
    }
    const int F = 2 * p;
    long double sum = 0.0L;
    for (int k = 0; k < F; ++k) sum += poly[k].real();
    const long double scale = std::sqrt(2.0L) / sum;
    long double h[kMaxTaps];
    for (int k = 0; k < F; ++k) h[k] = poly[k].real() * scale;
    for (int k = 0; k < F; ++k) {
        const long double g = ((k & 1) ? -1.0L : 1.0L) * h[F - 1 - k];   // rec_hi
        if (rec_lo) rec_lo[k] = (double)h[k];
        if (rec_hi) rec_hi[k] = (double)g;
        if (dec_lo) dec_lo[F - 1 - k] = (double)h[k];
        if (dec_hi) dec_hi[F - 1 - k] = (double)g;
    }
    return true;
}

}  // namespace wz
