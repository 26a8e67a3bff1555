// Wavelet filter banks by spectral factorisation (host code): Daubechies
// db1-db10 and the biorthogonal bior4.4.
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
#include <mutex>
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

// bior4.4 (CDF 9/7): the product filter of db4, cos^8(w/2) P(sin^2(w/2)) with
// P(y) = 1 + 4y + 10y^2 + 20y^3, split into two zero-phase factors
// cos^4 q(sin^2) (7 taps, q from the real root of P) and cos^4 q~(sin^2)
// (9 taps, q~ from the complex pair), each normalised to sum sqrt(2); in z,
// cos^2(w/2) = (z + 2 + 1/z) / 4 and sin^2(w/2) = (-z + 2 - 1/z) / 4.
// 10-tap layout: analysis lowpass in dec_lo[1..9], synthesis lowpass in
// rec_lo[1..7]; each high-pass is the alternating flip of the other side's
// lowpass.
bool bior44(double *dec_lo, double *dec_hi, double *rec_lo, double *rec_hi) {
    const std::vector<long double> P = {1.0L, 4.0L, 10.0L, 20.0L};
    const std::vector<cld> roots = poly_roots(P);
    cld yr = roots[0], yc = roots[0];
    for (const cld &y : roots) {
        if (std::fabs(y.imag()) < std::fabs(yr.imag())) yr = y;
        if (y.imag() > yc.imag()) yc = y;
    }
    auto conv = [](const std::vector<long double> &a, const std::vector<long double> &b) {
        std::vector<long double> r(a.size() + b.size() - 1, 0.0L);
        for (size_t i = 0; i < a.size(); ++i)
            for (size_t j = 0; j < b.size(); ++j) r[i + j] += a[i] * b[j];
        return r;
    };
    const std::vector<long double> cos4 = {1.0L / 16, 4.0L / 16, 6.0L / 16, 4.0L / 16, 1.0L / 16};
    const std::vector<long double> s2 = {-0.25L, 0.5L, -0.25L};           // sin^2(w/2)
    const long double inv_r = 1.0L / yr.real();
    const std::vector<long double> q = {-s2[0] * inv_r, 1.0L - s2[1] * inv_r, -s2[2] * inv_r};
    const cld inv_c = 1.0L / yc;
    const long double alpha = 2.0L * inv_c.real();                      // 1/y + 1/conj(y)
    const long double beta = std::norm(inv_c);                            // 1/|y|^2
    const std::vector<long double> ss = conv(s2, s2);
    std::vector<long double> qt(5, 0.0L);
    qt[2] = 1.0L;
    for (int k = 0; k < 3; ++k) qt[k + 1] -= alpha * s2[k];
    for (int k = 0; k < 5; ++k) qt[k] += beta * ss[k];
    std::vector<long double> h = conv(cos4, q), ht = conv(cos4, qt);   // 7 and 9 taps
    long double sh = 0.0L, sht = 0.0L;
    for (long double v : h) sh += v;
    for (long double v : ht) sht += v;
    const int F = 10;
    long double rl[F] = {}, htp[F] = {};
    for (int k = 0; k < 7; ++k) rl[1 + k] = h[k] * std::sqrt(2.0L) / sh;
    for (int k = 0; k < 9; ++k) htp[k] = ht[k] * std::sqrt(2.0L) / sht;
    for (int k = 0; k < F; ++k) {
        const long double sg = (k & 1) ? -1.0L : 1.0L;
        if (rec_lo) rec_lo[k] = (double)rl[k];
        if (dec_lo) dec_lo[k] = (double)htp[F - 1 - k];
        if (rec_hi) rec_hi[k] = (double)(sg * htp[F - 1 - k]);
        if (dec_hi) dec_hi[F - 1 - k] = (double)(sg * rl[F - 1 - k]);
    }
    return true;
}

int wavelet_taps(int wavelet) {
    if (wavelet >= 1 && 2 * wavelet <= kMaxTaps) return 2 * wavelet;
    if (wavelet == WZ_WAVELET_BIOR44) return 10;
    return 0;
}

// Each bank is derived once and kept: the derivation runs in long double,
// which hosts with a 128-bit long double emulate in software, and every
// condensation call sets up two banks.
bool wavelet_bank(int wavelet, double *dec_lo, double *dec_hi, double *rec_lo, double *rec_hi) {
    struct Bank {
        bool done = false, ok = false;
        double f[4][kMaxTaps] = {};
    };
    static std::mutex mu;
    static Bank banks[WZ_WAVELET_BIOR44 + 1];
    if (wavelet < 1 || wavelet > WZ_WAVELET_BIOR44) return false;
    Bank &b = banks[wavelet];
    {
        std::lock_guard<std::mutex> lock(mu);
        if (!b.done) {
            b.ok = wavelet == WZ_WAVELET_BIOR44 ? bior44(b.f[0], b.f[1], b.f[2], b.f[3])
                                                : daubechies(wavelet, b.f[0], b.f[1], b.f[2], b.f[3]);
            b.done = true;
        }
    }
    if (!b.ok) return false;
    double *out[4] = {dec_lo, dec_hi, rec_lo, rec_hi};
    const int F = wavelet_taps(wavelet);
    for (int j = 0; j < 4; ++j)
        if (out[j])
            for (int k = 0; k < F; ++k) out[j][k] = b.f[j][k];
    return true;
}

}  // namespace wz
