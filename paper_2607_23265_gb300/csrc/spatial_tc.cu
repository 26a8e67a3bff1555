// Spatial operator rows of the tensor-core condensation, sixteen operator
// rows at a time (single-level WSM, Eq. 11-14, with the bilinear
// condensation of Eq. 16).  The operator is the one spatial_wsm_kernel forms
// (see spatial.cu):
//
//   W_m[(p,q),(i,j)] = sum_v sum_b Q_v[q,b] A'_v[b,j] Y_v[b,i],
//   Y_v[b,i]         = sum_u sum_a P_u[p,a] A_u[a,i] g_uv[a,b],
//
// with g_LL = 1 and g_LH = g_HL = g_HH = G_m, here organised for the
// tensor-core layout.  Every frame's operator rows start on a 16-row boundary
// (budgets padded to 16), so a work item is one 16-row group of one frame and
// owns its rows outright: the CTA forms the group in shared memory directly
// in the tiled bf16 hi / lo layout of tile_index() (one 1 KB block per
// 32-column chunk and half) and sends the whole group, zeros included, to
// global memory with one 4D tensor store (256 elements x 2 row groups x
// chunks x halves).  Thread (t, s) of the 256 takes operator row t
// of the group (token j = 16 g + t, grid cell (p, q)) and the map rows
// i = zlo + s, zlo + s + 16, ... that the row reaches: it forms the
// coefficients c_v[b] = Q_v[q,b] Y_v[b,i] for the few b of the column's
// support in registers, straight from P_u A_u and the gate, and then the
// row's columns j four at a time from 16-byte reads of A'_v.  The CTAs are
// persistent and pull groups from a global counter over the prefix of the
// frames' group counts; the frame-independent tables are formed before the
// wait for the temporal kernel.  Tensor path, at most kCompactFrames frames
// and maps whose 16-row group fits in shared memory; spatial_wsm_kernel
// serves the rest.
#include <algorithm>

#include "wz_ptx.cuh"
#include "wz_spatial.cuh"

namespace wz {

namespace {

constexpr int kTcRows = 16;                       // operator rows per work item
constexpr int kGateRegs = 4;                      // gate entries per thread held in registers
constexpr int kTcChunkBytes = kTcRows * 32 * 2;   // 16 rows x 32 columns of one bf16 half: 1 KB

// Float offsets of the CTA's shared memory after the frame-independent tables.
struct TcSmem {
    int gpre;    // [VT + 1] int: 16-row groups of the frames before f
    int fdat;    // [VT][3] int: n | h << 13 | w << 20, off, woff of frame f
    int G;       // [hp][wp]: the item's frame gate
    int P;       // [16][2][BMAX]: P_L, P_H of row t's grid row at a = a0(t) + k
    int Q;       // [16][2][BMAX]: Q_L, Q_H of row t's grid column at b = b0(t) + k
    int tok;     // [16][8] int: per row t (see kTok*)
    int stage;   // [2][KC][512] bf16: the group's hi chunks, then its lo chunks
    int total;
    __host__ __device__ void init(const SpatialSmem &L, int VT, int bmax) {
        int o = L.tables;
        auto take = [&](int n, int align) {
            o = (o + align - 1) / align * align;
            const int at = o;
            o += n;
            return at;
        };
        gpre = take(VT + 1, 4);
        fdat = take(3 * VT, 4);
        G = take(L.hp * L.wp, 4);
        P = take(kTcRows * 2 * bmax, 4);
        Q = take(kTcRows * 2 * bmax, 4);
        tok = take(kTcRows * 8, 4);
        stage = take((L.K_pad >> 5) * kTcChunkBytes * 2 / 4, 32);   // 128-byte aligned
        total = o;
    }
};

// Per-row ints of TcSmem::tok.
enum { kTokA0 = 0, kTokNA, kTokB0, kTokNB, kTokZlo, kTokSpan, kTokJ4 };

// Operator entries (row t of the group, columns k ...) as bf16 hi and lo
// halves in the staged tiled layout: chunk k / 32, then the 8-row group, then
// the 8-column quarter, then row and column within the 8 x 8 core matrix.
__device__ __forceinline__ int stage_elem(int t, int k) {
    return (k >> 5) * 512 + (t >> 3) * 256 + ((k >> 3) & 3) * 64 + (t & 7) * 8 + (k & 7);
}
__device__ __forceinline__ void stage_put1(__nv_bfloat16 *hi, int lo_off, int t, int k, float x) {
    const int e = stage_elem(t, k);
    const __nv_bfloat16 h = __float2bfloat16_rn(x);
    hi[e] = h;
    hi[lo_off + e] = __float2bfloat16_rn(x - __bfloat162float(h));
}
// Columns k, k + 1 with k even: one quarter, one 32-bit store per half.
__device__ __forceinline__ void stage_put2(__nv_bfloat16 *hi, int lo_off, int t, int k, float x, float y) {
    const int e = stage_elem(t, k);
    const __nv_bfloat162 h = __floats2bfloat162_rn(x, y);
    const float2 hf = __bfloat1622float2(h);
    *reinterpret_cast<__nv_bfloat162 *>(hi + e) = h;
    *reinterpret_cast<__nv_bfloat162 *>(hi + lo_off + e) = __floats2bfloat162_rn(x - hf.x, y - hf.y);
}
// Columns k .. k + n - 1 (1 <= n <= 4) from v.x ...
__device__ __forceinline__ void stage_put4(__nv_bfloat16 *hi, int lo_off, int t, int k, float4 v, int n) {
    if ((k & 1) == 0) {
        if (n >= 2) stage_put2(hi, lo_off, t, k, v.x, v.y);
        else stage_put1(hi, lo_off, t, k, v.x);
        if (n == 4) stage_put2(hi, lo_off, t, k + 2, v.z, v.w);
        else if (n == 3) stage_put1(hi, lo_off, t, k + 2, v.z);
    } else {
        stage_put1(hi, lo_off, t, k, v.x);
        if (n >= 3) stage_put2(hi, lo_off, t, k + 1, v.y, v.z);
        else if (n == 2) stage_put1(hi, lo_off, t, k + 1, v.y);
        if (n == 4) stage_put1(hi, lo_off, t, k + 3, v.w);
    }
}

}  // namespace

template <int BMAX>
__global__ void __launch_bounds__(kSpatialThreads, BMAX <= 6 ? 3 : 2)
    spatial_wsm_tc_kernel(const __grid_constant__ CUtensorMap wmap, Ctx c) {
    pdl_trigger();
    extern __shared__ __align__(128) float sm[];
    __shared__ int s_item, s_f, s_wsum[kSpatialThreads / 32];
    const int tid = threadIdx.x;
    if (tid == 0) ptx::prefetch_tmap(&wmap);
    const int H = c.H, W = c.W, hp = c.hp, wp = c.wp, F = c.F, VT = c.V * c.T;
    SpatialSmem L;
    L.init(H, W, hp, wp);
    TcSmem S;
    S.init(L, VT, BMAX);
    // the frame-independent tables come from the kernel parameters alone:
    // formed while the temporal kernel runs
    build_spatial_tables_smem(c, L, sm);
    pdl_wait();
    // thread 0 claims the next group while the current one is formed
    int claimed = tid == 0 ? atomicAdd(c.spatial_next, 1) : 0;
    if ((int)blockIdx.x < kTailBlocks) tail_rows(c, (int)blockIdx.x);
    int *gpre = reinterpret_cast<int *>(sm + S.gpre), *fdat = reinterpret_cast<int *>(sm + S.fdat);
    // the prefix of the frames' group counts; the frames' budgets, grids and
    // row offsets stay in shared memory (n <= 4096, h, w <= 64)
    frame_prefix(VT, gpre, s_wsum, [&](int f) {
        const int n = max(c.n[f], 0);
        fdat[3 * f] = n | (c.hw[2 * f] << 13) | (c.hw[2 * f + 1] << 20);
        fdat[3 * f + 1] = c.off[f];
        fdat[3 * f + 2] = c.woff[f];
        return (n + kTcRows - 1) / kTcRows;
    });
    __syncthreads();
    const int items = gpre[VT];

    const float *AHl = sm + L.AHl, *AHh = sm + L.AHh, *AWl = sm + L.AWl, *AWh = sm + L.AWh;
    const int *jlo = reinterpret_cast<const int *>(sm + L.jlo), *jhi = reinterpret_cast<const int *>(sm + L.jhi);
    const int *ilo = reinterpret_cast<const int *>(sm + L.ilo), *ihi = reinterpret_cast<const int *>(sm + L.ihi);
    float *G = sm + S.G, *Pt = sm + S.P, *Qt = sm + S.Q;
    int *tok = reinterpret_cast<int *>(sm + S.tok);
    unsigned char *stg = reinterpret_cast<unsigned char *>(sm + S.stage);
    __nv_bfloat16 *shi = reinterpret_cast<__nv_bfloat16 *>(stg);
    const int KC = L.K_pad >> 5, WP4 = L.WP4;
    const int lo_off = KC * 512;                           // elements from a hi entry to its lo entry
    const int stage_words = KC * kTcChunkBytes * 2 / 16;   // uint4 words of the stage
    const int t = tid >> 4, s = tid & 15;   // operator row of the group, slot of the row's work

    // the frames' tensor-core unit records, frame f by CTA f mod gridDim.x
    // (before the groups: the counter balances the CTAs afterwards)
    for (int f = blockIdx.x; f < VT; f += gridDim.x) {
        const int nhw = fdat[3 * f], n = nhw & 8191;
        if (n > 0) unit_records(c, f, n, (nhw >> 13) & 127, nhw >> 20, ilo, ihi);
    }

    for (;;) {
        __syncthreads();   // the previous group's reads of shared memory
        if (tid == 0) {
            const int it = claimed;
            if (it < items) claimed = atomicAdd(c.spatial_next, 1);
            int fi = 0;
            if (it < items) {
                // the last frame whose first group is <= it (frames without
                // groups share their successor's prefix)
                int lo = 0, hi = VT - 1;
                while (lo < hi) {
                    const int mid = (lo + hi + 1) >> 1;
                    if (gpre[mid] <= it) lo = mid;
                    else hi = mid - 1;
                }
                fi = lo;
            }
            s_item = it;
            s_f = fi;
        }
        __syncthreads();
        const int item = s_item;
        if (item >= items) break;
        const int f = s_f, g = item - gpre[f];
        const int nhw = fdat[3 * f], n = nhw & 8191, h = (nhw >> 13) & 127, w = nhw >> 20;
        // gate G of the frame (Eq. 6, Eq. 12), pooled by frame_stats: loaded
        // into registers here, stored to shared memory after the row setup
        const float *Gf = c.gate + (int64_t)f * c.gate_stride;
        const int ng = hp * wp;
        float gr[kGateRegs];
#pragma unroll
        for (int r = 0; r < kGateRegs; ++r) {
            const int k = tid + r * kSpatialThreads;
            gr[r] = k < ng ? Gf[k] : 0.f;
        }
        {
            // row t: token j of the frame, grid cell (p, q); the bilinear row
            // and column through the synthesis (P_u[p, a], Q_v[q, b]) and the
            // map rows and columns the row reaches
            const int j = kTcRows * g + t;
            const bool valid = j < n;
            const int p = valid ? j / w : 0, q = valid ? j - p * w : 0;
            int y0, y1, x0, x1, a0, a1, b0, b1;
            float ly, lx;
            bilinear_src(p, H, h, y0, y1, ly);
            bilinear_src(q, W, w, x0, x1, lx);
            synth_support(y0, y1, F, hp, a0, a1);
            synth_support(x0, x1, F, wp, b0, b1);
            if (s < BMAX) {
                const int a = a0 + s, b = b0 + s;
                float *P = Pt + t * 2 * BMAX, *Q = Qt + t * 2 * BMAX;
                P[s] = a <= a1 ? (1.f - ly) * synth(c.rec_lo, F, y0, a) + ly * synth(c.rec_lo, F, y1, a) : 0.f;
                P[BMAX + s] = a <= a1 ? (1.f - ly) * synth(c.rec_hi, F, y0, a) + ly * synth(c.rec_hi, F, y1, a) : 0.f;
                Q[s] = b <= b1 ? (1.f - lx) * synth(c.rec_lo, F, x0, b) + lx * synth(c.rec_lo, F, x1, b) : 0.f;
                Q[BMAX + s] = b <= b1 ? (1.f - lx) * synth(c.rec_hi, F, x0, b) + lx * synth(c.rec_hi, F, x1, b) : 0.f;
            }
            if (s == 0) {
                const int na = min(a1 - a0 + 1, BMAX), nb = min(b1 - b0 + 1, BMAX);
                int zlo = H, zhi = -1, jl = WP4, jh = -1;
                for (int u = 0; u < na; ++u) {
                    zlo = min(zlo, ilo[a0 + u]);
                    zhi = max(zhi, ihi[a0 + u]);
                }
                for (int bb = 0; bb < nb; ++bb) {
                    jl = min(jl, jlo[b0 + bb]);
                    jh = max(jh, jhi[b0 + bb]);
                }
                int *T = tok + 8 * t;
                T[kTokA0] = a0;
                T[kTokNA] = na;
                T[kTokB0] = b0;
                T[kTokNB] = nb;
                T[kTokZlo] = zlo;
                T[kTokSpan] = valid && jh >= 0 ? max(0, zhi - zlo + 1) : 0;
                T[kTokJ4] = jh >= 0 ? (jl >> 2) | ((jh >> 2) << 16) : 0;
                const int64_t row = (int64_t)fdat[3 * f + 1] + j;
                if (valid && wz_in_range(c.status, row < c.rows_total)) {
                    int *o = c.out_index + (size_t)row * 3;
                    o[0] = f % c.T;
                    o[1] = p;
                    o[2] = q;
                }
            }
        }
#pragma unroll
        for (int r = 0; r < kGateRegs; ++r) {
            const int k = tid + r * kSpatialThreads;
            if (k < ng) G[k] = gr[r];
        }
        for (int k = tid + kGateRegs * kSpatialThreads; k < ng; k += kSpatialThreads) G[k] = Gf[k];
        // thread 0 issued the previous group's store: its reads of the stage
        // have finished (waited for here, after the loads above) before the
        // stage is cleared
        if (tid == 0) ptx::bulk_wait_read();
        __syncthreads();
        {
            uint4 *z = reinterpret_cast<uint4 *>(stg);
            for (int k = tid; k < stage_words; k += blockDim.x) z[k] = make_uint4(0u, 0u, 0u, 0u);
        }
        __syncthreads();   // the stage is clear; G, P, Q and the row data are in place
        {
            const int *T = tok + 8 * t;
            const int span = T[kTokSpan];
            const int a0 = T[kTokA0], na = T[kTokNA], b0 = T[kTokB0], nb = T[kTokNB], zlo = T[kTokZlo];
            const int j4lo = T[kTokJ4] & 0xffff, j4hi = T[kTokJ4] >> 16;
            const float *P = Pt + t * 2 * BMAX, *Q = Qt + t * 2 * BMAX;
            for (int ri = s; ri < span; ri += 16) {
                const int i = zlo + ri;
                // P_u[p, a] A_u[a, i] for the row's coefficients a
                float pal[BMAX], pah[BMAX];
#pragma unroll
                for (int u = 0; u < BMAX; ++u) {
                    pal[u] = u < na ? P[u] * AHl[(a0 + u) * H + i] : 0.f;
                    pah[u] = u < na ? P[BMAX + u] * AHh[(a0 + u) * H + i] : 0.f;
                }
                // c_v[b] = Q_v[q, b] Y_v[b, i]
                float cl[BMAX], ch[BMAX];
#pragma unroll
                for (int bb = 0; bb < BMAX; ++bb) {
                    float yl = 0.f, yh = 0.f;
                    if (bb < nb) {
#pragma unroll
                        for (int u = 0; u < BMAX; ++u) {
                            if (u < na) {
                                const float gg = G[(a0 + u) * wp + b0 + bb];
                                yl += pal[u] + pah[u] * gg;
                                yh += (pal[u] + pah[u]) * gg;
                            }
                        }
                    }
                    cl[bb] = bb < nb ? Q[bb] * yl : 0.f;
                    ch[bb] = bb < nb ? Q[BMAX + bb] * yh : 0.f;
                }
                // row i of the operator row: columns 4 j4 .. 4 j4 + 3
                for (int j4 = j4lo; j4 <= j4hi; ++j4) {
                    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
                    for (int bb = 0; bb < BMAX; ++bb) {
                        if (bb < nb) {
                            const float4 a4 = reinterpret_cast<const float4 *>(AWl + (b0 + bb) * WP4)[j4];
                            const float4 d4 = reinterpret_cast<const float4 *>(AWh + (b0 + bb) * WP4)[j4];
                            acc.x = fmaf(cl[bb], a4.x, fmaf(ch[bb], d4.x, acc.x));
                            acc.y = fmaf(cl[bb], a4.y, fmaf(ch[bb], d4.y, acc.y));
                            acc.z = fmaf(cl[bb], a4.z, fmaf(ch[bb], d4.z, acc.z));
                            acc.w = fmaf(cl[bb], a4.w, fmaf(ch[bb], d4.w, acc.w));
                        }
                    }
                    stage_put4(shi, lo_off, t, i * W + 4 * j4, acc, min(4, W - 4 * j4));
                }
            }
        }
        // the stage goes out as one tensor store: row groups r0 / 8 and
        // r0 / 8 + 1 of every chunk, hi and lo
        ptx::fence_proxy_async_smem();
        __syncthreads();
        if (tid == 0) {
            const int64_t r0 = (int64_t)fdat[3 * f + 2] + kTcRows * g;
            if (wz_in_range(c.status, r0 + kTcRows <= c.w_rows)) ptx::tma_store_4d(&wmap, stg, 0, (int)(r0 >> 3), 0, 0);
            ptx::bulk_commit();
        }
    }
    // the operator rows are in global memory before the CTA ends
    if (tid == 0) ptx::bulk_wait();
}

// Dynamic shared memory of spatial_wsm_tc_kernel (bytes).
size_t spatial_tc_smem_bytes(const Ctx &c, int bmax) {
    SpatialSmem L;
    L.init(c.H, c.W, c.hp, c.wp);
    TcSmem S;
    S.init(L, c.V * c.T, bmax);
    return (size_t)S.total * sizeof(float);
}

// The 16-row kernel when it applies (tensor path, single-level WSM, at most
// kCompactFrames frames, two CTAs per SM): *launched = true and its launch
// status; else *launched = false.
cudaError_t launch_spatial_tc(const Ctx &c, cudaStream_t s, bool *launched) {
    *launched = false;
    if (c.path != WZ_PATH_TENSOR || c.spatial_mode != WZ_SPATIAL_WSM || c.wsm_levels > 1) return cudaSuccess;
    if ((int64_t)c.V * c.T > kCompactFrames) return cudaSuccess;
    const int bmax = (c.F - 1) / 2 + 2;
    const void *fn;
    int bm;
    if (bmax <= 6) {
        fn = (const void *)spatial_wsm_tc_kernel<6>;
        bm = 6;
    } else if (bmax <= 12) {
        fn = (const void *)spatial_wsm_tc_kernel<12>;
        bm = 12;
    } else {
        return cudaSuccess;
    }
    const size_t smem = spatial_tc_smem_bytes(c, bm);
    const int KC = (c.H * c.W + 31) / 32;
    auto enc = tmap_encode_fn();
    if (smem > (size_t)100 * 1024 || KC > 256 || !enc) return cudaSuccess;
    // the tiled operator as [half][chunk][8-row group][256 elements]
    CUtensorMap wmap;
    {
        const cuuint64_t groups = (cuuint64_t)(c.w_rows >> 3);
        cuuint64_t dims[4] = {256, groups, (cuuint64_t)KC, 2};
        cuuint64_t strides[3] = {512, groups * 512, (cuuint64_t)c.w_rows * (cuuint64_t)(32 * KC) * 2};
        cuuint32_t box[4] = {256, 2, (cuuint32_t)KC, 2};
        cuuint32_t es[4] = {1, 1, 1, 1};
        if (enc(&wmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, c.Wop, dims, strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
                CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_NONE,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return cudaSuccess;
    }
    cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    int dev = 0, sms = 0, per_sm = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
    if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, kSpatialThreads, smem)) != cudaSuccess)
        return e;
    if (per_sm < 1) return cudaSuccess;
    // persistent: every resident CTA pulls groups; at least kTailBlocks CTAs
    // so that the tail rows are covered
    const unsigned blocks = (unsigned)std::max(sms * per_sm, kTailBlocks);
    void *args[] = {&wmap, const_cast<Ctx *>(&c)};
    *launched = true;
    return launch_kernel(fn, dim3(blocks), dim3(kSpatialThreads), smem, s, args, c.pdl != 0);
}

}  // namespace wz
