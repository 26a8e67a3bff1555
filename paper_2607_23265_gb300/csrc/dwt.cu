// Standalone single-level DWT / IDWT (Eq. 8, 10, 11, 14).
//
//   dwt1d   cA[i] = sum_j dec_lo[j] x^[2i+1-j], cD with dec_hi (x^ extended)
//   idwt1d  x[k]  = sum_i cA[i] rec_lo[k+F-2-2i] + cD[i] rec_hi[k+F-2-2i]
//   dwt2d   height axis then width axis per frame and channel; bands LL, LH,
//           HL, HH with the height filter first
//   idwt2d  width inverse then height inverse
//
// The 2D kernels stage a frame's map for a chunk of CT channels in shared
// memory and run both separable passes there.
#include <algorithm>

#include "wz_internal.cuh"

namespace wz {

struct Taps {
    float lo[kMaxTaps], hi[kMaxTaps];
};

__global__ void dwt1d_kernel(const float *x, int rows, int L, int F, int mode, Taps t,
                             float *cA, float *cD) {
    const int Lo = (L + F - 1) / 2;
    const int64_t id = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (id >= (int64_t)rows * Lo) return;
    const int64_t r = id / Lo;
    const int i = (int)(id % Lo);
    const float *xr = x + r * L;
    float a = 0.f, d = 0.f;
    for (int j = 0; j < F; ++j) {
        const int s = ext_index(2 * i + 1 - j, L, mode);
        if (s < 0) continue;
        const float v = xr[s];
        a = fmaf(t.lo[j], v, a);
        d = fmaf(t.hi[j], v, d);
    }
    cA[id] = a;
    cD[id] = d;
}

__global__ void idwt1d_kernel(const float *cA, const float *cD, int rows, int L, int F, Taps t,
                              float *x) {
    const int Lo = (L + F - 1) / 2;
    const int64_t id = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (id >= (int64_t)rows * L) return;
    const int64_t r = id / L;
    const int k = (int)(id % L);
    float s = 0.f;
    const int ilo = max(0, (k - 1 + 1) / 2), ihi = min(Lo - 1, (k + F - 2) / 2);
    for (int i = ilo; i <= ihi; ++i) {
        const int tt = k + F - 2 - 2 * i;
        if (tt < 0 || tt >= F) continue;
        s = fmaf(t.lo[tt], cA[r * Lo + i], s);
        s = fmaf(t.hi[tt], cD[r * Lo + i], s);
    }
    x[id] = s;
}

template <typename Tin>
__global__ void __launch_bounds__(256) dwt2d_kernel(const Tin *X, int H, int W, int D, int CT, int F,
                                                    int mode, Taps t, float *LL, float *LH, float *HL,
                                                    float *HH) {
    extern __shared__ float sm[];
    const int hp = (H + F - 1) / 2, wp = (W + F - 1) / 2;
    const int64_t fr = blockIdx.y;
    const int c0 = blockIdx.x * CT;
    float *sx = sm;                        // [H][W][CT]
    float *sr = sm + (size_t)H * W * CT;   // [H][2][wp][CT] width pass (lo, hi)
    const Tin *Xf = X + (size_t)fr * H * W * D;
    for (int k = threadIdx.x; k < H * W * CT; k += blockDim.x) {
        const int cc = k % CT, p = k / CT;
        sx[k] = c0 + cc < D ? load_scalar<Tin>(Xf + (size_t)p * D + c0 + cc) : 0.f;
    }
    __syncthreads();
    for (int k = threadIdx.x; k < H * wp * CT; k += blockDim.x) {
        const int cc = k % CT, b = (k / CT) % wp, i = k / (CT * wp);
        float lo = 0.f, hi = 0.f;
        for (int j = 0; j < F; ++j) {
            const int s = ext_index(2 * b + 1 - j, W, mode);
            if (s < 0) continue;
            const float v = sx[(i * W + s) * CT + cc];
            lo = fmaf(t.lo[j], v, lo);
            hi = fmaf(t.hi[j], v, hi);
        }
        sr[((i * 2 + 0) * wp + b) * CT + cc] = lo;
        sr[((i * 2 + 1) * wp + b) * CT + cc] = hi;
    }
    __syncthreads();
    for (int k = threadIdx.x; k < hp * wp * CT; k += blockDim.x) {
        const int cc = k % CT, b = (k / CT) % wp, a = k / (CT * wp);
        float ll = 0.f, lh = 0.f, hl = 0.f, hh = 0.f;
        for (int j = 0; j < F; ++j) {
            const int s = ext_index(2 * a + 1 - j, H, mode);
            if (s < 0) continue;
            const float vl = sr[((s * 2 + 0) * wp + b) * CT + cc];
            const float vh = sr[((s * 2 + 1) * wp + b) * CT + cc];
            ll = fmaf(t.lo[j], vl, ll);
            lh = fmaf(t.lo[j], vh, lh);
            hl = fmaf(t.hi[j], vl, hl);
            hh = fmaf(t.hi[j], vh, hh);
        }
        if (c0 + cc < D) {
            const size_t o = (((size_t)fr * hp + a) * wp + b) * D + c0 + cc;
            LL[o] = ll;
            LH[o] = lh;
            HL[o] = hl;
            HH[o] = hh;
        }
    }
}

__global__ void __launch_bounds__(256) idwt2d_kernel(const float *LL, const float *LH, const float *HL,
                                                     const float *HH, int H, int W, int D, int CT,
                                                     int F, Taps t, float *out) {
    extern __shared__ float sm[];
    const int hp = (H + F - 1) / 2, wp = (W + F - 1) / 2;
    const int64_t fr = blockIdx.y;
    const int c0 = blockIdx.x * CT;
    float *sb = sm;                                 // [4][hp][wp][CT]
    float *sr = sm + (size_t)4 * hp * wp * CT;      // [H][2][wp][CT]
    const float *bands[4] = {LL, LH, HL, HH};
    for (int k = threadIdx.x; k < 4 * hp * wp * CT; k += blockDim.x) {
        const int cc = k % CT, p = (k / CT) % (hp * wp), bnd = k / (CT * hp * wp);
        sb[k] = c0 + cc < D ? bands[bnd][((size_t)fr * hp * wp + p) * D + c0 + cc] : 0.f;
    }
    __syncthreads();
    // height inverse: rows y of the width-low and width-high planes
    for (int k = threadIdx.x; k < H * wp * CT; k += blockDim.x) {
        const int cc = k % CT, b = (k / CT) % wp, y = k / (CT * wp);
        float lo = 0.f, hi = 0.f;
        for (int a = 0; a < hp; ++a) {
            const int tt = y + F - 2 - 2 * a;
            if (tt < 0 || tt >= F) continue;
            const size_t o = ((size_t)a * wp + b) * CT + cc;
            lo = fmaf(t.lo[tt], sb[0 * hp * wp * CT + o], lo);   // LL
            lo = fmaf(t.hi[tt], sb[2 * hp * wp * CT + o], lo);   // HL
            hi = fmaf(t.lo[tt], sb[1 * hp * wp * CT + o], hi);   // LH
            hi = fmaf(t.hi[tt], sb[3 * hp * wp * CT + o], hi);   // HH
        }
        sr[((y * 2 + 0) * wp + b) * CT + cc] = lo;
        sr[((y * 2 + 1) * wp + b) * CT + cc] = hi;
    }
    __syncthreads();
    for (int k = threadIdx.x; k < H * W * CT; k += blockDim.x) {
        const int cc = k % CT, x = (k / CT) % W, y = k / (CT * W);
        float s = 0.f;
        for (int b = 0; b < wp; ++b) {
            const int tt = x + F - 2 - 2 * b;
            if (tt < 0 || tt >= F) continue;
            s = fmaf(t.lo[tt], sr[((y * 2 + 0) * wp + b) * CT + cc], s);
            s = fmaf(t.hi[tt], sr[((y * 2 + 1) * wp + b) * CT + cc], s);
        }
        if (c0 + cc < D) out[(((size_t)fr * H + y) * W + x) * D + c0 + cc] = s;
    }
}

namespace {

Taps make_taps(const float *lo, const float *hi, int F) {
    Taps t{};
    for (int k = 0; k < F; ++k) {
        t.lo[k] = lo[k];
        t.hi[k] = hi[k];
    }
    return t;
}

// Channels per CTA so that the staged planes fit in shared memory.
int pick_ct(size_t floats_per_channel) {
    int ct = 16;
    while (ct > 1 && floats_per_channel * ct * sizeof(float) > 200 * 1024) ct >>= 1;
    return ct;
}

}  // namespace

cudaError_t launch_dwt1d(const float *x, int rows, int L, int F, int mode, const float *dlo,
                         const float *dhi, float *cA, float *cD, cudaStream_t s) {
    const int64_t n = (int64_t)rows * ((L + F - 1) / 2);
    if (n == 0) return cudaSuccess;
    dwt1d_kernel<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(x, rows, L, F, mode, make_taps(dlo, dhi, F), cA, cD);
    return cudaGetLastError();
}

cudaError_t launch_idwt1d(const float *cA, const float *cD, int rows, int L, int F,
                          const float *rlo, const float *rhi, float *x, cudaStream_t s) {
    const int64_t n = (int64_t)rows * L;
    if (n == 0) return cudaSuccess;
    idwt1d_kernel<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(cA, cD, rows, L, F, make_taps(rlo, rhi, F), x);
    return cudaGetLastError();
}

cudaError_t launch_dwt2d(const void *X, int dtype, int T, int H, int W, int D, int F, int mode,
                         const float *dlo, const float *dhi, float *LL, float *LH, float *HL,
                         float *HH, cudaStream_t s) {
    const int wp = (W + F - 1) / 2;
    const int ct = pick_ct((size_t)H * W + (size_t)H * 2 * wp);
    const size_t smem = ((size_t)H * W + (size_t)H * 2 * wp) * ct * sizeof(float);
    const dim3 grid((unsigned)((D + ct - 1) / ct), (unsigned)T);
    const Taps t = make_taps(dlo, dhi, F);
    cudaError_t e;
    if (dtype == WZ_DTYPE_BF16) {
        e = cudaFuncSetAttribute(dwt2d_kernel<__nv_bfloat16>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        dwt2d_kernel<__nv_bfloat16><<<grid, 256, smem, s>>>(static_cast<const __nv_bfloat16 *>(X), H, W, D, ct, F,
                                                          mode, t, LL, LH, HL, HH);
    } else {
        e = cudaFuncSetAttribute(dwt2d_kernel<float>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        dwt2d_kernel<float><<<grid, 256, smem, s>>>(static_cast<const float *>(X), H, W, D, ct, F, mode, t, LL,
                                                   LH, HL, HH);
    }
    return cudaGetLastError();
}

cudaError_t launch_idwt2d(const float *LL, const float *LH, const float *HL, const float *HH,
                          int T, int H, int W, int D, int F, const float *rlo, const float *rhi,
                          float *out, cudaStream_t s) {
    const int hp = (H + F - 1) / 2, wp = (W + F - 1) / 2;
    const int ct = pick_ct((size_t)4 * hp * wp + (size_t)H * 2 * wp);
    const size_t smem = ((size_t)4 * hp * wp + (size_t)H * 2 * wp) * ct * sizeof(float);
    cudaError_t e = cudaFuncSetAttribute(idwt2d_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const dim3 grid((unsigned)((D + ct - 1) / ct), (unsigned)T);
    idwt2d_kernel<<<grid, 256, smem, s>>>(LL, LH, HL, HH, H, W, D, ct, F, make_taps(rlo, rhi, F), out);
    return cudaGetLastError();
}

}  // namespace wz
