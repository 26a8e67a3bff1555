// Spatial operator of the condensation pass (Eq. 6, 11-14, 16).
//
// For a retained frame m the WSM (Eq. 11-14) and the bilinear condensation
// Psi (Eq. 16) are linear in the feature map and act identically on every
// channel: the gate G_m (Eq. 12) depends on position only.  The condensed
// tokens are therefore Z_m = W_m X_m with one matrix W_m (n_m x H*W) per
// frame, X_m the frame's [H*W][D] token matrix.  With A_u / A'_v the db
// analysis matrices along height / width (symmetric extension folded in),
// S_u / S'_v the synthesis matrices, g_LL = 1 and g_LH = g_HL = g_HH = G_m,
// and P_u = R_y S_u, Q_v = R_x S'_v the bilinear rows pushed through the
// synthesis:
//
//   W_m[(p,q),(i,j)] = sum_v sum_b Q_v[q,b] A'_v[b,j] Y_v[b,i],
//   Y_v[b,i]         = sum_u sum_a P_u[p,a] A_u[a,i] g_uv[a,b].
//
// One CTA per (frame, grid row p) builds the w_m rows of W_m for that grid
// row in fp32 from tables in shared memory (each thread owns one output
// token q and input column j and sums only over the few b where A'_v[b, j]
// is nonzero), writes them as bf16 hi/lo pairs
// (tensor-core path) or fp32 (CUDA-core path), writes the index map rows,
// and trailing CTAs fill rows that cannot be produced with -1 / zeros.
#include <cmath>

#include "wz_internal.cuh"

namespace wz {

constexpr int kSpatialThreads = 256;
constexpr int kTailBlocks = 64;

struct SpatialSmem {
    int N, hp, wp, H, W, HP4;
    // float offsets
    int M, G, AHl, AHh, AWl, AWh, PAl, PAh, Yl, Yh, Ql, Qh, red, blo, bhi, total;
    // Every table starts on a 16-byte boundary (float4 reads of Y).
    __host__ __device__ void init(int H_, int W_, int hp_, int wp_) {
        H = H_; W = W_; hp = hp_; wp = wp_; N = H * W;
        HP4 = (H + 3) & ~3;
        int o = 0;
        auto take = [&](int n) {
            const int at = o;
            o = (o + n + 3) & ~3;
            return at;
        };
        M = take(N);
        G = take(hp * wp);
        AHl = take(hp * H);
        AHh = take(hp * H);
        AWl = take(wp * W);
        AWh = take(wp * W);
        PAl = take(hp * H);
        PAh = take(hp * H);
        Yl = take(wp * HP4);
        Yh = take(wp * HP4);
        Ql = take(W * wp);
        Qh = take(W * wp);
        red = take(64);
        blo = take(W);
        bhi = take(W);
        total = o;
    }
};

__device__ __forceinline__ float synth(const float *rec, int F, int y, int a) {
    const int k = y + F - 2 - 2 * a;
    return (k >= 0 && k < F) ? rec[k] : 0.f;
}

// Half-pixel bilinear source (align_corners = false): rows y0, y1, weight of y1.
__device__ __forceinline__ void bilinear_src(int i, int in, int out, int &y0, int &y1, float &l) {
    double s = (i + 0.5) * ((double)in / (double)out) - 0.5;
    if (s < 0.0) s = 0.0;
    int f = (int)floor(s);
    if (f > in - 1) f = in - 1;
    y0 = f;
    y1 = f + 1 < in ? f + 1 : in - 1;
    l = (float)(s - f);
}

template <int HMAX>
__global__ void __launch_bounds__(kSpatialThreads) spatial_kernel(Ctx c) {
    extern __shared__ float sm[];
    const int tid = threadIdx.x;
    const int64_t nblk_frames = (int64_t)c.V * c.T * c.H;
    if ((int64_t)blockIdx.x >= nblk_frames) {
        // rows past the produced count: index -1, zero tokens
        const int tb = (int)(blockIdx.x - nblk_frames);
        const size_t esz = c.dtype == WZ_DTYPE_BF16 ? 2 : 4;
        const int nvec = (int)((size_t)c.D * esz / 16);
        for (int v = 0; v < c.V; ++v) {
            const int r0 = c.vpar[v].row0 + c.prod[v];
            const int r1 = c.vpar[v].row0 + c.vpar[v].B;
            for (int r = r0 + tb; r < r1; r += kTailBlocks) {
                uint4 *o = reinterpret_cast<uint4 *>(static_cast<char *>(c.out) + (size_t)r * c.D * esz);
                for (int k = tid; k < nvec; k += blockDim.x) o[k] = make_uint4(0u, 0u, 0u, 0u);
                if (tid < 3) c.out_index[(size_t)r * 3 + tid] = -1;
            }
        }
        return;
    }
    const int64_t f = blockIdx.x / c.H;
    const int pi = (int)(blockIdx.x % c.H);
    const int n = c.n[f];
    if (n <= 0) return;
    const int h = c.hw[2 * f], w = c.hw[2 * f + 1];
    if (pi >= h) return;
    const int H = c.H, W = c.W, N = c.N, hp = c.hp, wp = c.wp, F = c.F;
    SpatialSmem L;
    L.init(H, W, hp, wp);
    float *M = sm + L.M, *G = sm + L.G;
    float *AHl = sm + L.AHl, *AHh = sm + L.AHh, *AWl = sm + L.AWl, *AWh = sm + L.AWh;
    float *PAl = sm + L.PAl, *PAh = sm + L.PAh, *Yl = sm + L.Yl, *Yh = sm + L.Yh;
    float *Ql = sm + L.Ql, *Qh = sm + L.Qh, *red = sm + L.red;
    int *blo = reinterpret_cast<int *>(sm + L.blo), *bhi = reinterpret_cast<int *>(sm + L.bhi);
    const int HP4 = L.HP4;

    // saliency map M (Eq. 6): per-frame min-max of a_{t,n}
    const float *a = c.a + f * N;
    float lo = INFINITY, hi = -INFINITY;
    for (int k = tid; k < N; k += blockDim.x) {
        const float x = a[k];
        M[k] = x;
        lo = fminf(lo, x);
        hi = fmaxf(hi, x);
    }
    for (int o = 16; o > 0; o >>= 1) {
        lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, o));
        hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, o));
    }
    if ((tid & 31) == 0) {
        red[tid >> 5] = lo;
        red[32 + (tid >> 5)] = hi;
    }
    // analysis matrices (zero first)
    for (int k = tid; k < hp * H; k += blockDim.x) AHl[k] = AHh[k] = 0.f;
    for (int k = tid; k < wp * W; k += blockDim.x) AWl[k] = AWh[k] = 0.f;
    __syncthreads();
    lo = INFINITY;
    hi = -INFINITY;
    for (int k = 0; k < (int)(blockDim.x >> 5); ++k) {
        lo = fminf(lo, red[k]);
        hi = fmaxf(hi, red[32 + k]);
    }
    const float rng = hi - lo;
    for (int k = tid; k < N; k += blockDim.x) M[k] = rng > 0.f ? (M[k] - lo) / rng : 0.f;
    // A[a][i] = sum_j dec[j] [ext(2a+1-j) == i]; one thread per row a
    if (tid < hp) {
        for (int j = 0; j < F; ++j) {
            const int i = ext_index(2 * tid + 1 - j, H, c.mode);
            if (i >= 0) {
                AHl[tid * H + i] += c.dec_lo[j];
                AHh[tid * H + i] += c.dec_hi[j];
            }
        }
    } else if (tid >= 128 && tid < 128 + wp) {
        const int b = tid - 128;
        for (int j = 0; j < F; ++j) {
            const int i = ext_index(2 * b + 1 - j, W, c.mode);
            if (i >= 0) {
                AWl[b * W + i] += c.dec_lo[j];
                AWh[b * W + i] += c.dec_hi[j];
            }
        }
    }
    __syncthreads();
    // gate G = lambda * adaptive-average-pool(M) to hp x wp (Eq. 12)
    for (int k = tid; k < hp * wp; k += blockDim.x) {
        const int ai = k / wp, bj = k % wp;
        const int r0 = (ai * H) / hp, r1 = ((ai + 1) * H + hp - 1) / hp;
        const int c0 = (bj * W) / wp, c1 = ((bj + 1) * W + wp - 1) / wp;
        float s = 0.f;
        for (int y = r0; y < r1; ++y)
            for (int x = c0; x < c1; ++x) s += M[y * W + x];
        G[k] = c.lambda * (s / (float)((r1 - r0) * (c1 - c0)));
    }
    // bilinear rows through the synthesis: P_u[a] for this grid row, Q_v[q][b]
    int y0, y1;
    float ly;
    bilinear_src(pi, H, h, y0, y1, ly);
    for (int k = tid; k < hp * H; k += blockDim.x) {
        const int ai = k / H;
        const float pl = (1.f - ly) * synth(c.rec_lo, F, y0, ai) + ly * synth(c.rec_lo, F, y1, ai);
        const float ph = (1.f - ly) * synth(c.rec_hi, F, y0, ai) + ly * synth(c.rec_hi, F, y1, ai);
        PAl[k] = pl * AHl[k];
        PAh[k] = ph * AHh[k];
    }
    for (int k = tid; k < w * wp; k += blockDim.x) {
        const int q = k / wp, b = k % wp;
        int x0, x1;
        float lx;
        bilinear_src(q, W, w, x0, x1, lx);
        Ql[k] = (1.f - lx) * synth(c.rec_lo, F, x0, b) + lx * synth(c.rec_lo, F, x1, b);
        Qh[k] = (1.f - lx) * synth(c.rec_hi, F, x0, b) + lx * synth(c.rec_hi, F, x1, b);
    }
    // support of the width analysis: rows b of A' that reach column j
    for (int j = tid; j < W; j += blockDim.x) {
        int lo_b = wp, hi_b = -1;
        for (int b = 0; b < wp; ++b)
            if (AWl[b * W + j] != 0.f || AWh[b * W + j] != 0.f) {
                lo_b = min(lo_b, b);
                hi_b = max(hi_b, b);
            }
        blo[j] = lo_b;
        bhi[j] = hi_b;
    }
    __syncthreads();
    // Y_v[b][i], rows padded to a multiple of 4 with zeros
    for (int k = tid; k < wp * HP4; k += blockDim.x) {
        const int b = k / HP4, i = k % HP4;
        float yl = 0.f, yh = 0.f;
        if (i < H) {
            for (int ai = 0; ai < hp; ++ai) {
                const float g = G[ai * wp + b];
                const float pl = PAl[ai * H + i], ph = PAh[ai * H + i];
                yl += pl + ph * g;
                yh += (pl + ph) * g;
            }
        }
        Yl[k] = yl;
        Yh[k] = yh;
    }
    __syncthreads();
    // operator rows of this grid row: p = pi*w + q, q < w, p < n
    const int nq = min(w, n - pi * w);
    const int64_t row0 = (int64_t)c.off[f] + (int64_t)pi * w;      // output row
    const bool bf = c.path == WZ_PATH_TENSOR;
    const int64_t wrow0 = bf ? (int64_t)c.woff[f] + (int64_t)pi * w : row0;   // operator row
    __nv_bfloat16 *Whi = static_cast<__nv_bfloat16 *>(c.Wop);
    __nv_bfloat16 *Wlo = Whi + (size_t)c.w_rows * c.K_pad;
    float *W32 = static_cast<float *>(c.Wop);
    // one thread per (output q, input column j): all H rows i in registers,
    // summed over the support of column j only
    for (int item = tid; item < nq * W; item += blockDim.x) {
        const int q = item / W, j = item % W;
        float acc[HMAX];
#pragma unroll
        for (int i = 0; i < HMAX; ++i) acc[i] = 0.f;
        for (int b = blo[j]; b <= bhi[j]; ++b) {
            const float ql = Ql[q * wp + b] * AWl[b * W + j];
            const float qh = Qh[q * wp + b] * AWh[b * W + j];
            const float4 *yl = reinterpret_cast<const float4 *>(Yl + b * HP4);
            const float4 *yh = reinterpret_cast<const float4 *>(Yh + b * HP4);
#pragma unroll
            for (int i4 = 0; i4 < HMAX / 4; ++i4) {
                if (4 * i4 < H) {
                    const float4 a = yl[i4], d = yh[i4];
                    acc[4 * i4 + 0] = fmaf(a.x, ql, fmaf(d.x, qh, acc[4 * i4 + 0]));
                    acc[4 * i4 + 1] = fmaf(a.y, ql, fmaf(d.y, qh, acc[4 * i4 + 1]));
                    acc[4 * i4 + 2] = fmaf(a.z, ql, fmaf(d.z, qh, acc[4 * i4 + 2]));
                    acc[4 * i4 + 3] = fmaf(a.w, ql, fmaf(d.w, qh, acc[4 * i4 + 3]));
                }
            }
        }
        const size_t rbase = (size_t)(row0 + q) * c.K_pad;
#pragma unroll
        for (int i = 0; i < HMAX; ++i) {
            if (i < H) {
                const float s = acc[i];
                if (bf) {
                    const size_t k = tile_index(wrow0 + q, i * W + j, c.w_rows);
                    const __nv_bfloat16 hb = __float2bfloat16_rn(s);
                    Whi[k] = hb;
                    Wlo[k] = __float2bfloat16_rn(s - __bfloat162float(hb));
                } else {
                    W32[rbase + (size_t)i * W + j] = s;
                }
            }
        }
    }
    // zero the K padding of these rows, and the index map rows
    const int padw = c.K_pad - N;
    for (int k = tid; k < nq * padw; k += blockDim.x) {
        if (bf) {
            const size_t idx = tile_index(wrow0 + k / padw, N + (k % padw), c.w_rows);
            Whi[idx] = __float2bfloat16_rn(0.f);
            Wlo[idx] = __float2bfloat16_rn(0.f);
        } else {
            W32[(size_t)(row0 + k / padw) * c.K_pad + N + (k % padw)] = 0.f;
        }
    }
    const int t = (int)(f % c.T);
    for (int q = tid; q < nq; q += blockDim.x) {
        int *o = c.out_index + (size_t)(row0 + q) * 3;
        o[0] = t;
        o[1] = pi;
        o[2] = q;
    }
}

size_t spatial_smem_bytes(const Ctx &c) {
    SpatialSmem L;
    L.init(c.H, c.W, c.hp, c.wp);
    return (size_t)L.total * sizeof(float);
}

cudaError_t launch_spatial(const Ctx &c, cudaStream_t s) {
    SpatialSmem L;
    L.init(c.H, c.W, c.hp, c.wp);
    if ((L.Yl & 3) != 0 || (L.Yh & 3) != 0) return cudaErrorMisalignedAddress;
    const size_t smem = spatial_smem_bytes(c);
    const unsigned blocks = (unsigned)((int64_t)c.V * c.T * c.H + kTailBlocks);
    const void *fn;
    if (c.H <= 16) fn = (const void *)spatial_kernel<16>;
    else if (c.H <= 32) fn = (const void *)spatial_kernel<32>;
    else if (c.H <= 64) fn = (const void *)spatial_kernel<64>;
    else return cudaErrorInvalidValue;
    cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    void *args[] = {const_cast<Ctx *>(&c)};
    return cudaLaunchKernel(fn, dim3(blocks), dim3(kSpatialThreads), args, smem, s);
}

}  // namespace wz
