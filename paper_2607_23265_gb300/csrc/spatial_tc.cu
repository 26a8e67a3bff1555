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
// 32-column chunk and half) and sends each block to global memory with one
// bulk copy, zeros included.  Thread (t, s) of the 256 takes operator row t
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
constexpr int kTcChunkBytes = kTcRows * 32 * 2;   // 16 rows x 32 columns of one bf16 half: 1 KB

// Float offsets of the CTA's shared memory after the frame-independent tables.
struct TcSmem {
    int gpre;    // [VT + 1] int: 16-row groups of the frames before f
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

// Operator entry (row t of the group, column k) as bf16 hi and lo halves in
// the staged tiled layout: chunk k / 32, then the 8-row group, then the
// 8-column quarter, then row and column within the 8 x 8 core matrix.
__device__ __forceinline__ void stage_put(__nv_bfloat16 *hi, int lo_off, int t, int k, float x) {
    const int e = (k >> 5) * 512 + (t >> 3) * 256 + ((k >> 3) & 3) * 64 + (t & 7) * 8 + (k & 7);
    const __nv_bfloat16 h = __float2bfloat16_rn(x);
    hi[e] = h;
    hi[lo_off + e] = __float2bfloat16_rn(x - __bfloat162float(h));
}

}  // namespace

template <int BMAX>
__global__ void __launch_bounds__(kSpatialThreads, BMAX <= 6 ? 3 : 2) spatial_wsm_tc_kernel(Ctx c) {
    pdl_trigger();
    extern __shared__ __align__(16) float sm[];
    __shared__ int s_item, s_f, s_wsum[kSpatialThreads / 32];
    const int tid = threadIdx.x, lane = tid & 31;
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
    int *gpre = reinterpret_cast<int *>(sm + S.gpre);
    frame_prefix(VT, gpre, s_wsum, [&](int f) { return (max(c.n[f], 0) + kTcRows - 1) / kTcRows; });
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
    __nv_bfloat16 *Whi = static_cast<__nv_bfloat16 *>(c.Wop);
    __nv_bfloat16 *Wlo = Whi + (size_t)c.w_rows * L.K_pad;
    const int t = tid >> 4, s = tid & 15;   // operator row of the group, slot of the row's work

    for (;;) {
        __syncthreads();   // the previous group's reads of shared memory
        // warp 0 issued the previous group's bulk stores: their reads of the
        // stage have finished before the stage is cleared
        if (tid < 32) ptx::bulk_wait_read();
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
        const int n = c.n[f], h = c.hw[2 * f], w = c.hw[2 * f + 1];
        if (g == 0) unit_records(c, f, n, h, w, ilo, ihi);
        {
            uint4 *z = reinterpret_cast<uint4 *>(stg);
            for (int k = tid; k < stage_words; k += blockDim.x) z[k] = make_uint4(0u, 0u, 0u, 0u);
        }
        {
            // gate G of the frame (Eq. 6, Eq. 12), pooled by frame_stats
            const float *Gf = c.gate + (int64_t)f * c.gate_stride;
            for (int k = tid; k < hp * wp; k += blockDim.x) G[k] = Gf[k];
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
                const int64_t row = (int64_t)c.off[f] + j;
                if (valid && wz_in_range(c.status, row < c.rows_total)) {
                    int *o = c.out_index + (size_t)row * 3;
                    o[0] = f % c.T;
                    o[1] = p;
                    o[2] = q;
                }
            }
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
                    const int k = i * W + 4 * j4;
                    stage_put(shi, lo_off, t, k, acc.x);
                    if (4 * j4 + 1 < W) stage_put(shi, lo_off, t, k + 1, acc.y);
                    if (4 * j4 + 2 < W) stage_put(shi, lo_off, t, k + 2, acc.z);
                    if (4 * j4 + 3 < W) stage_put(shi, lo_off, t, k + 3, acc.w);
                }
            }
        }
        // the stage goes out as 2 * KC bulk copies of 1 KB (hi chunks, then lo)
        ptx::fence_proxy_async_smem();
        __syncthreads();
        if (tid < 32) {
            const int64_t r0 = (int64_t)c.woff[f] + kTcRows * g;
            if (wz_in_range(c.status, r0 + kTcRows <= c.w_rows))
                for (int k = lane; k < 2 * KC; k += 32) {
                    const int kc = k < KC ? k : k - KC;
                    __nv_bfloat16 *dst = (k < KC ? Whi : Wlo) + tile_index(r0, 32 * kc, c.w_rows);
                    ptx::bulk_store(dst, stg + (size_t)k * kTcChunkBytes, kTcChunkBytes);
                }
            ptx::bulk_commit();
        }
    }
    // the operator rows are in global memory before the CTA ends
    if (tid < 32) ptx::bulk_wait();
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
    if (smem > (size_t)100 * 1024) return cudaSuccess;
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
    void *args[] = {const_cast<Ctx *>(&c)};
    *launched = true;
    return launch_kernel(fn, dim3(blocks), dim3(kSpatialThreads), smem, s, args, c.pdl != 0);
}

}  // namespace wz
