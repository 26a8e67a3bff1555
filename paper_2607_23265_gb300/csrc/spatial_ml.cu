// Spatial operator of the condensation pass with a multi-level WSM (Eq. 11-14
// cascaded on LL, then Psi of Eq. 16).  The operator of every level has the
// single-level form with the level's folded analysis rows and synthesis
// columns (tables built once per pass, see MLTables):
//
//   W_m[(p,q),(i,j)] = sum_l sum_v sum_b Q_v^l[q,b] AW_v^l[b,j] Y_v^l[b,i],
//   Y_v^l[b,i]       = sum_u sum_a P_u^l[p,a] AH_u^l[a,i] g_uv^l[a,b],
//
// with g_LL = 1 only at the deepest level.  S CTAs per frame take the grid
// rows p = s0, s0 + S, ...; per row every level's Y goes to shared memory,
// then each thread owns one (output token q, input column j) and sums all
// levels into the H rows it keeps in registers (HMAX >= H), over the b where
// both Q^l and AW^l are nonzero.
#include <cmath>

#include "wz_spatial.cuh"

namespace wz {

template <int HMAX>
__global__ void __launch_bounds__(kSpatialThreads) spatial_ml_kernel(Ctx c, int S) {
    pdl_wait();
    pdl_trigger();
    extern __shared__ float sm[];
    const int tid = threadIdx.x;
    const int64_t nblk_frames = (int64_t)c.V * c.T * S;
    if ((int64_t)blockIdx.x >= nblk_frames) {
        tail_rows(c, (int)(blockIdx.x - nblk_frames));
        return;
    }
    const int64_t f = blockIdx.x / S;
    const int s0 = (int)(blockIdx.x % S);
    const int n = c.n[f];
    if (n <= 0) return;
    const int h = c.hw[2 * f], w = c.hw[2 * f + 1];
    if (s0 >= h || s0 * w >= n) return;
    if (s0 == 0 && c.path == WZ_PATH_TENSOR) unit_records(c, f, n);

    const int H = c.H, W = c.W, N = c.N, J = c.wsm_levels;
    MLTables T;
    T.init(H, W, c.F, J);
    MLSmem L;
    L.init(T);
    const float *gt = c.stab;                                   // global tables
    const int *gi = reinterpret_cast<const int *>(c.stab);
    int *si = reinterpret_cast<int *>(sm);
    float *G = sm + L.G, *PAl = sm + L.PAl, *PAh = sm + L.PAh, *red = sm + L.red, *stg = sm + L.stage;
    int *irange = reinterpret_cast<int *>(red + 48);
    const int HP4 = L.HP4;
    // per-level offsets for the inner loop, read as shared-memory broadcasts
    enum { kWl, kQl, kQh, kAWl, kAWh, kYl, kYh, kBlo, kBhi, kQlo, kQhi, kMeta };
    __shared__ int meta[kMaxLevels][kMeta];
    if (tid < J) {
        int *m = meta[tid];
        m[kWl] = T.w[tid + 1];
        m[kQl] = L.Ql[tid]; m[kQh] = L.Qh[tid];
        m[kAWl] = T.AWl[tid]; m[kAWh] = T.AWh[tid];
        m[kYl] = L.Yl[tid]; m[kYh] = L.Yh[tid];
        m[kBlo] = T.blo[tid]; m[kBhi] = T.bhi[tid];
        m[kQlo] = L.qlo[tid]; m[kQhi] = L.qhi[tid];
    }

    // ---- per-frame tables ------------------------------------------------
    {   // 16-byte copies, two in flight per thread (T.copy is a multiple of 4 words)
        const int n4 = T.copy >> 2;
        const int4 *src = reinterpret_cast<const int4 *>(gi);
        int4 *dst = reinterpret_cast<int4 *>(si);
        const int bd = (int)blockDim.x;
        for (int k = tid; k < n4; k += 2 * bd) {
            const int4 x0 = src[k];
            const bool two = k + bd < n4;
            const int4 x1 = two ? src[k + bd] : x0;
            dst[k] = x0;
            if (two) dst[k + bd] = x1;
        }
    }
    const float *Gf = c.gate + f * (int64_t)c.gate_stride;
    for (int k = tid; k < c.gate_stride; k += blockDim.x) G[k] = Gf[k];
    // bilinear columns through each level's synthesis, and their supports
    for (int l = 0; l < J; ++l) {
        const int wl = T.w[l + 1];
        float *Ql = sm + L.Ql[l], *Qh = sm + L.Qh[l];
        int *qlo = si + L.qlo[l], *qhi = si + L.qhi[l];
        for (int k = tid; k < w * wl; k += blockDim.x) {
            const int q = k / wl, b = k % wl;
            int x0, x1;
            float lx;
            bilinear_src(q, W, w, x0, x1, lx);
            Ql[k] = (1.f - lx) * gt[T.SWl[l] + x0 * wl + b] + lx * gt[T.SWl[l] + x1 * wl + b];
            Qh[k] = (1.f - lx) * gt[T.SWh[l] + x0 * wl + b] + lx * gt[T.SWh[l] + x1 * wl + b];
            if (b == 0) {
                qlo[q] = min(gi[T.xlo[l] + x0], gi[T.xlo[l] + x1]);
                qhi[q] = max(gi[T.xhi[l] + x0], gi[T.xhi[l] + x1]);
            }
        }
    }

    const bool bf = c.path == WZ_PATH_TENSOR;
    __nv_bfloat16 *Whi = static_cast<__nv_bfloat16 *>(c.Wop);
    __nv_bfloat16 *Wlo = Whi + (size_t)c.w_rows * c.K_pad;
    float *W32 = static_cast<float *>(c.Wop);
    const int K_pad = c.K_pad;
    const int wsh = W <= 32 ? 5 : 6;
    const size_t kstride = (size_t)(c.w_rows >> 3) * 256;
    const int t = (int)(f % c.T);

    for (int pi = s0; pi < h && pi * w < n; pi += S) {
        const int nq = min(w, n - pi * w);
        int y0, y1;
        float ly;
        bilinear_src(pi, H, h, y0, y1, ly);
        __syncthreads();   // previous row's Y / stage reads, the frame tables
        if (tid == 0) {
            irange[0] = HMAX;
            irange[1] = -1;
        }
        int my_lo = HMAX, my_hi = -1;
        for (int l = 0; l < J; ++l) {
            const int hl = T.h[l + 1], wl = T.w[l + 1];
            const int alo = min(gi[T.slo[l] + y0], gi[T.slo[l] + y1]);
            const int ahi = max(gi[T.shi[l] + y0], gi[T.shi[l] + y1]);
            const int na = ahi - alo + 1;
            const float *AHl = sm + T.AHl[l], *AHh = sm + T.AHh[l];
            for (int k = tid; k < na * H; k += blockDim.x) {
                const int ai = alo + k / H, i = k % H;
                const float pl = (1.f - ly) * gt[T.SHl[l] + y0 * hl + ai] + ly * gt[T.SHl[l] + y1 * hl + ai];
                const float ph = (1.f - ly) * gt[T.SHh[l] + y0 * hl + ai] + ly * gt[T.SHh[l] + y1 * hl + ai];
                PAl[k] = pl * AHl[ai * H + i];
                PAh[k] = ph * AHh[ai * H + i];
            }
            __syncthreads();
            const float gll = l == J - 1 ? 1.f : 0.f;   // LL is decomposed further above the deepest level
            const float *Gl = G + c.goff[l];
            float *Yl = sm + L.Yl[l], *Yh = sm + L.Yh[l];
            for (int k = tid; k < wl * HP4; k += blockDim.x) {
                const int b = k / HP4, i = k % HP4;
                float yl = 0.f, yh = 0.f;
                if (i < H) {
                    for (int u = 0; u < na; ++u) {
                        const float g = Gl[(alo + u) * wl + b];
                        const float pl = PAl[u * H + i], ph = PAh[u * H + i];
                        yl += pl * gll + ph * g;
                        yh += (pl + ph) * g;
                    }
                    if (yl != 0.f || yh != 0.f) {
                        my_lo = min(my_lo, i);
                        my_hi = max(my_hi, i);
                    }
                }
                Yl[k] = yl;
                Yh[k] = yh;
            }
            __syncthreads();   // PA is reused by the next level
        }
        for (int o = 16; o > 0; o >>= 1) {
            my_lo = min(my_lo, __shfl_xor_sync(0xffffffffu, my_lo, o));
            my_hi = max(my_hi, __shfl_xor_sync(0xffffffffu, my_hi, o));
        }
        if ((tid & 31) == 0 && my_hi >= 0) {
            atomicMin(&irange[0], my_lo);
            atomicMax(&irange[1], my_hi);
        }
        __syncthreads();
        const int i4lo = irange[0] >> 2, i4hi = irange[1] >> 2;
        const int64_t row0 = (int64_t)c.off[f] + (int64_t)pi * w;
        const int64_t wrow0 = bf ? (int64_t)c.woff[f] + (int64_t)pi * w : row0;
        for (int q0 = 0; q0 < nq; q0 += L.QB) {
            const int qn = min(L.QB, nq - q0);
            for (int item = tid; item < (qn << wsh); item += blockDim.x) {
                const int ql_ = item >> wsh, j = item & ((1 << wsh) - 1);
                if (j >= W) continue;
                const int q = q0 + ql_;
                float acc[HMAX];
#pragma unroll
                for (int i = 0; i < HMAX; ++i) acc[i] = 0.f;
#pragma unroll 1
                for (int l = 0; l < J; ++l) {
                    const int *m = meta[l];
                    const int wl = m[kWl];
                    const float *Ql = sm + m[kQl], *Qh = sm + m[kQh];
                    const float *AWl = sm + m[kAWl], *AWh = sm + m[kAWh];
                    const float *Yl = sm + m[kYl], *Yh = sm + m[kYh];
                    const int b1 = min(si[m[kBhi] + j], si[m[kQhi] + q]);
                    for (int b = max(si[m[kBlo] + j], si[m[kQlo] + q]); b <= b1; ++b) {
                        const float ql = Ql[q * wl + b] * AWl[b * W + j];
                        const float qh = Qh[q * wl + b] * AWh[b * W + j];
                        const float4 *yl = reinterpret_cast<const float4 *>(Yl + b * HP4);
                        const float4 *yh = reinterpret_cast<const float4 *>(Yh + b * HP4);
#pragma unroll
                        for (int i4 = 0; i4 < HMAX / 4; ++i4) {
                            if (i4 >= i4lo && i4 <= i4hi) {
                                const float4 a4 = yl[i4], d4 = yh[i4];
                                acc[4 * i4 + 0] = fmaf(a4.x, ql, fmaf(d4.x, qh, acc[4 * i4 + 0]));
                                acc[4 * i4 + 1] = fmaf(a4.y, ql, fmaf(d4.y, qh, acc[4 * i4 + 1]));
                                acc[4 * i4 + 2] = fmaf(a4.z, ql, fmaf(d4.z, qh, acc[4 * i4 + 2]));
                                acc[4 * i4 + 3] = fmaf(a4.w, ql, fmaf(d4.w, qh, acc[4 * i4 + 3]));
                            }
                        }
                    }
                }
                float *srow = stg + ql_ * L.KS;
#pragma unroll
                for (int i = 0; i < HMAX; ++i)
                    if (i < H) srow[i * W + j] = acc[i];
            }
            for (int k = tid; k < qn * (K_pad - N); k += blockDim.x)
                stg[(k / (K_pad - N)) * L.KS + N + k % (K_pad - N)] = 0.f;
            __syncthreads();
            write_rows(c, stg, L.KS, qn, K_pad, (bf ? wrow0 : row0) + q0, bf, Whi, Wlo, W32, kstride, 0, K_pad);
            if (q0 + L.QB < nq) __syncthreads();
        }
        for (int q = tid; q < nq; q += blockDim.x) {
            if (!wz_in_range(c.status, row0 + q < c.rows_total)) break;
            int *o = c.out_index + (size_t)(row0 + q) * 3;
            o[0] = t;
            o[1] = pi;
            o[2] = q;
        }
    }
}

size_t spatial_ml_smem_bytes(int H, int W, int F, int J) {
    MLTables T;
    T.init(H, W, F, J);
    MLSmem L;
    L.init(T);
    const size_t bytes = (size_t)L.total * sizeof(float);
    return bytes <= 200 * 1024 && L.QB >= 1 ? bytes : 0;
}

int spatial_split(const Ctx &c, int resident);

cudaError_t launch_spatial_ml(const Ctx &c, cudaStream_t s) {
    const size_t smem = spatial_ml_smem_bytes(c.H, c.W, c.F, c.wsm_levels);
    if (smem == 0) return cudaErrorInvalidValue;
    const void *fn;
    if (c.H <= 16) fn = (const void *)spatial_ml_kernel<16>;
    else if (c.H <= 32) fn = (const void *)spatial_ml_kernel<32>;
    else if (c.H <= 64) fn = (const void *)spatial_ml_kernel<64>;
    else return cudaErrorInvalidValue;
    cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    int dev = 0, sms = 0, per_sm = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
    if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, kSpatialThreads, smem)) != cudaSuccess)
        return e;
    int S = spatial_split(c, sms * (per_sm > 0 ? per_sm : 1));
    const unsigned blocks = (unsigned)((int64_t)c.V * c.T * S + kTailBlocks);
    void *args[] = {const_cast<Ctx *>(&c), &S};
    return launch_kernel(fn, dim3(blocks), dim3(kSpatialThreads), smem, s, args, c.pdl != 0);
}

}  // namespace wz
