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
// spatial_wsm_kernel is persistent: each CTA forms the frame-independent
// tables (analysis matrices with their row and column supports) once, before
// it waits for the temporal kernel, and then pulls grid rows from a global
// counter; a new frame reloads its gate and the width rows Q_v.  Per grid
// row: P_u A_u, then Y_v over the map rows the row's operator rows reach,
// then the tokens with lane = input row i (two tokens per warp when at most
// 16 rows are reached), each lane keeping c_v[b] = Q_v[q,b] Y_v[b,i] for the
// few b of the column's support in registers and forming row i of the
// token's operator row four columns at a time from 16-byte reads of A'_v.
// Rows are staged in shared memory and
// leave as 512-byte coalesced warp stores of bf16 hi/lo halves in the tiled
// operator layout (tensor-core path) or as fp32 rows (CUDA-core path), with
// the index map rows.  The ablation modes without the WSM use
// spatial_plain_kernel (S CTAs per frame).  CTAs with a low index also fill
// the rows that cannot be produced (tau > 0) with -1 / zeros.
#include <algorithm>
#include <cmath>

#include "wz_spatial.cuh"

namespace wz {

// Operator rows of the ablation modes without the WSM (spatial "saliency" and
// "none"): W[(p,q),(y,x)] = Ry[p][y] Rx[q][x] s(y, x), the bilinear weights of
// Eq. 16 times s = lambda * M_t (Eq. 6 map) or 1.  Same staging, layout and
// index rows as the WSM operator.
__device__ void plain_operator_rows(const Ctx &c, const SpatialSmem &L, float *sm, int64_t f, int s0, int S, int n,
                                    int h, int w) {
    const int tid = threadIdx.x, H = c.H, W = c.W, N = c.N, K_pad = c.K_pad;
    float *stg = sm + L.stage, *M = sm + L.M, *red = sm + L.red;
    const bool sal = c.spatial_mode == WZ_SPATIAL_SALIENCY;
    if (sal) {
        const float *a = (c.ext_a ? c.ext_a : c.a) + f * N;
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
            red[16 + (tid >> 5)] = hi;
        }
        __syncthreads();
        lo = INFINITY;
        hi = -INFINITY;
        for (int k = 0; k < (int)(blockDim.x >> 5); ++k) {
            lo = fminf(lo, red[k]);
            hi = fmaxf(hi, red[16 + k]);
        }
        const float rng = hi - lo;
        for (int k = tid; k < N; k += blockDim.x) M[k] = c.lambda * (rng > 0.f ? (M[k] - lo) / rng : 0.f);
    }
    const bool bf = c.path == WZ_PATH_TENSOR;
    __nv_bfloat16 *Whi = static_cast<__nv_bfloat16 *>(c.Wop);
    __nv_bfloat16 *Wlo = Whi + (size_t)c.w_rows * K_pad;
    float *W32 = static_cast<float *>(c.Wop);
    const size_t kstride = (size_t)(c.w_rows >> 3) * 256;
    const int t = (int)(f % c.T);
    for (int pi = s0; pi < h && pi * w < n; pi += S) {
        const int nq = min(w, n - pi * w);
        int y0, y1;
        float ly;
        bilinear_src(pi, H, h, y0, y1, ly);
        const int64_t row0 = (int64_t)c.off[f] + (int64_t)pi * w;
        const int64_t wrow0 = bf ? (int64_t)c.woff[f] + (int64_t)pi * w : row0;
        for (int q0 = 0; q0 < nq; q0 += L.QB) {
            const int qn = min(L.QB, nq - q0);
            __syncthreads();   // M, and the previous batch's reads of the stage
            for (int k = tid; k < qn * L.KS; k += blockDim.x) stg[k] = 0.f;
            __syncthreads();
            for (int ql_ = tid; ql_ < qn; ql_ += blockDim.x) {
                int x0, x1;
                float lx;
                bilinear_src(q0 + ql_, W, w, x0, x1, lx);
                float *row = stg + ql_ * L.KS;
                const int ys[2] = {y0, y1}, xs[2] = {x0, x1};
                const float wy[2] = {1.f - ly, ly}, wx[2] = {1.f - lx, lx};
#pragma unroll
                for (int u = 0; u < 2; ++u)
#pragma unroll
                    for (int v = 0; v < 2; ++v) {
                        const int k = ys[u] * W + xs[v];
                        row[k] += wy[u] * wx[v] * (sal ? M[k] : 1.f);
                    }
            }
            __syncthreads();
            write_rows(c, stg, L.KS, qn, K_pad, (bf ? wrow0 : row0) + q0, bf, Whi, Wlo, W32, kstride, 0, K_pad);
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

// Ablation modes without the WSM: S CTAs per frame, grid rows p = s0, s0 + S, ...
__global__ void __launch_bounds__(kSpatialThreads) spatial_plain_kernel(Ctx c, int S) {
    pdl_wait();
    pdl_trigger();
    extern __shared__ float sm[];
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
    SpatialSmem L;
    L.init(c.H, c.W, c.hp, c.wp);
    plain_operator_rows(c, L, sm, f, s0, S, n, h, w);
}

// Grid rows of frame f that hold output tokens: p < h and p * w < n.
__device__ __forceinline__ int frame_rows(const Ctx &c, int f) {
    const int n = c.n[f];
    if (n <= 0) return 0;
    const int h = c.hw[2 * f], w = c.hw[2 * f + 1];
    return min(h, (n + w - 1) / w);
}

// The WSM operator rows (single level), persistent: every CTA copies the
// frame-independent tables once, then takes grid rows (frame f, row p) from
// a global counter until none is left; a row whose frame changes reloads
// the frame's gate and width rows.  Rows of frames with a small budget cost
// as much as others, so the dynamic order keeps the SMs evenly loaded.  With
// compact != 0 (at most kCompactFrames frames) every CTA first forms the
// prefix of the frames' grid rows in shared memory and the counter runs over
// the rows that exist; otherwise it runs over all V*T*H (frame, row) pairs.
template <int BMAX>
__global__ void __launch_bounds__(kSpatialThreads, 4) spatial_wsm_kernel(Ctx c, int compact) {
    pdl_trigger();
    extern __shared__ float sm[];
    __shared__ int s_item, s_f, s_wsum[kSpatialThreads / 32];
    const int tid = threadIdx.x;
    const int H = c.H, W = c.W, N = c.N, hp = c.hp, wp = c.wp, F = c.F;
    SpatialSmem L;
    L.init(H, W, hp, wp);
    // the frame-independent tables (analysis matrices, supports) come from the
    // kernel parameters alone: formed before the wait for the temporal kernel,
    // while it runs
    build_spatial_tables_smem(c, L, sm);
    pdl_wait();
    // thread 0 claims the next row while the current one is formed, so the
    // counter's round trip overlaps the work
    int claimed = tid == 0 ? atomicAdd(c.spatial_next, 1) : 0;
    if ((int)blockIdx.x < kTailBlocks) tail_rows(c, (int)blockIdx.x);
    float *G = sm + L.G;
    float *AHl = sm + L.AHl, *AHh = sm + L.AHh, *AWl = sm + L.AWl, *AWh = sm + L.AWh;
    float *PAl = sm + L.PAl, *PAh = sm + L.PAh, *Yl = sm + L.Yl, *Yh = sm + L.Yh;
    float *Ql = sm + L.Ql, *Qh = sm + L.Qh, *red = sm + L.red;
    const int *jlo = reinterpret_cast<const int *>(sm + L.jlo), *jhi = reinterpret_cast<const int *>(sm + L.jhi);
    const int *ilo = reinterpret_cast<const int *>(sm + L.ilo), *ihi = reinterpret_cast<const int *>(sm + L.ihi);
    int *rowpre = reinterpret_cast<int *>(sm + L.total);   // compact: [V*T + 1]
    int *qlo = reinterpret_cast<int *>(sm + L.qlo), *qhi = reinterpret_cast<int *>(sm + L.qhi);
    float *stg = sm + L.stage;
    const int HP4 = L.HP4, WP4 = L.WP4;
    (void)red;

    const bool bf = c.path == WZ_PATH_TENSOR;
    __nv_bfloat16 *Whi = static_cast<__nv_bfloat16 *>(c.Wop);
    __nv_bfloat16 *Wlo = Whi + (size_t)c.w_rows * c.K_pad;
    float *W32 = static_cast<float *>(c.Wop);
    const int K_pad = c.K_pad;
    const size_t kstride = (size_t)(c.w_rows >> 3) * 256;   // tile_index step of 32 columns
    const int lane = tid & 31, warp = tid >> 5, nwarp = (int)(blockDim.x >> 5);
    const int IH = (H + 31) >> 5;                            // 32-row slices of the map

    // candidates (frame, grid row): f * H + p < V * T * H < 2^31, 32-bit
    // index arithmetic throughout (no 64-bit divisions in the loop)
    const int VT = c.V * c.T;
    if (compact) {
        frame_prefix(VT, rowpre, s_wsum, [&](int fr) { return frame_rows(c, fr); });
        __syncthreads();
    }
    const int items = compact ? rowpre[VT] : VT * H;
    int cur_f = -1;
    for (;;) {
        __syncthreads();   // the previous row's reads of shared memory
        if (tid == 0) {
            const int it = claimed;
            if (it < items) claimed = atomicAdd(c.spatial_next, 1);
            int fi = 0;
            if (compact && it < items) {
                // the last frame whose first row is <= it (frames without
                // rows share their successor's prefix)
                int lo = 0, hi = VT - 1;
                while (lo < hi) {
                    const int mid = (lo + hi + 1) >> 1;
                    if (rowpre[mid] <= it) lo = mid;
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
        const int f = compact ? s_f : item / H;
        const int pi = compact ? item - rowpre[f] : item - f * H;
        const int n = c.n[f];
        if (n <= 0) continue;
        const int h = c.hw[2 * f], w = c.hw[2 * f + 1];
        if (pi >= h || pi * w >= n) continue;
        if (pi == 0 && c.path == WZ_PATH_TENSOR) unit_records(c, f, n, h, w, ilo, ihi);
        const int t = f % c.T;
        if (f != cur_f) {
            // gate G of this frame (Eq. 6, Eq. 12), pooled by frame_stats
            const float *Gf = c.gate + (int64_t)f * c.gate_stride;
            for (int k = tid; k < hp * wp; k += 2 * blockDim.x) {
                const float g0 = Gf[k];
                const bool two = k + (int)blockDim.x < hp * wp;
                const float g1 = two ? Gf[k + blockDim.x] : 0.f;
                G[k] = g0;
                if (two) G[k + blockDim.x] = g1;
            }
            // bilinear columns through the synthesis: Q_v[q][b] and its support
            for (int q = warp; q < w; q += nwarp) {   // warp per column q, lanes over b
                int x0, x1;
                float lx;
                bilinear_src(q, W, w, x0, x1, lx);
                for (int b = lane; b < wp; b += 32) {
                    Ql[q * wp + b] = (1.f - lx) * synth(c.rec_lo, F, x0, b) + lx * synth(c.rec_lo, F, x1, b);
                    Qh[q * wp + b] = (1.f - lx) * synth(c.rec_hi, F, x0, b) + lx * synth(c.rec_hi, F, x1, b);
                }
                if (lane == 0) {
                    int l_, h_;
                    synth_support(x0, x1, F, wp, l_, h_);
                    qlo[q] = l_;
                    qhi[q] = h_;
                }
            }
            cur_f = f;
        }
        const int nq = min(w, n - pi * w);
        // bilinear row through the synthesis: P_u[a] is nonzero for a in [alo, ahi]
        int y0, y1;
        float ly;
        bilinear_src(pi, H, h, y0, y1, ly);
        int alo, ahi;
        synth_support(y0, y1, F, hp, alo, ahi);
        const int na = ahi - alo + 1;
        int zlo = H, zhi = -1;   // map rows the operator rows of this grid row reach
        for (int a = alo; a <= ahi; ++a) {
            zlo = min(zlo, ilo[a]);
            zhi = max(zhi, ihi[a]);
        }
        __syncthreads();   // previous row's Y / stage reads, the frame tables
        for (int u = warp; u < na; u += nwarp) {   // warp per coefficient row, lanes over i
            const int ai = alo + u;
            const float pl = (1.f - ly) * synth(c.rec_lo, F, y0, ai) + ly * synth(c.rec_lo, F, y1, ai);
            const float ph = (1.f - ly) * synth(c.rec_hi, F, y0, ai) + ly * synth(c.rec_hi, F, y1, ai);
            for (int i = lane; i < H; i += 32) {
                PAl[u * H + i] = pl * AHl[ai * H + i];
                PAh[u * H + i] = ph * AHh[ai * H + i];
            }
        }
        __syncthreads();
        // Y_v[b][i], rows padded to a multiple of 4 with zeros; with at most
        // 16 map rows reached (paired, below) only those rows, two columns b
        // per warp
        const int span = zhi - zlo + 1;
        const bool paired = span <= 16 && H <= 32;
        if (paired) {
            const int r = lane & 15;
            for (int b = 2 * warp + (lane >> 4); b < wp; b += 2 * nwarp) {
                if (r < span) {
                    const int i = zlo + r;
                    float yl = 0.f, yh = 0.f;
                    for (int u = 0; u < na; ++u) {
                        const float g = G[(alo + u) * wp + b];
                        const float pl = PAl[u * H + i], ph = PAh[u * H + i];
                        yl += pl + ph * g;
                        yh += (pl + ph) * g;
                    }
                    Yl[b * HP4 + i] = yl;
                    Yh[b * HP4 + i] = yh;
                }
            }
        } else {
            for (int b = warp; b < wp; b += nwarp)   // warp per subband column b, lanes over i
            for (int i = lane; i < HP4; i += 32) {
                const int k = b * HP4 + i;
                float yl = 0.f, yh = 0.f;
                if (i < H) {
                    for (int u = 0; u < na; ++u) {
                        const float g = G[(alo + u) * wp + b];
                        const float pl = PAl[u * H + i], ph = PAh[u * H + i];
                        yl += pl + ph * g;
                        yh += (pl + ph) * g;
                    }
                }
                Yl[k] = yl;
                Yh[k] = yh;
            }
        }
        __syncthreads();
        const int64_t row0 = (int64_t)c.off[f] + (int64_t)pi * w;                 // output row
        const int64_t wrow0 = bf ? (int64_t)c.woff[f] + (int64_t)pi * w : row0;   // operator row
        // Rows are produced QB at a time.  The operator rows of this grid row
        // reach the map rows [zlo, zhi] only (columns [zc_lo, zc_hi]); write_rows
        // reads the staged columns [rc_lo, rc_hi) (the 32-column groups that
        // meet them) and writes zeros elsewhere.  Lane = input row i: the
        // lane's coefficients c_v[b] = Q_v[q,b] Y_v[b,i] over the support of
        // Q_v[q,.] (at most BMAX values) stay in registers; each 4-column
        // group j of row i of the staged token q is then
        // sum_b c_L[b] A'_L[b,j] + c_H[b] A'_H[b,j], with the analysis rows read
        // as 16-byte words and only the groups the support reaches computed.
        // With at most 16 such rows a warp forms two tokens (a half-warp each,
        // lanes over rows zlo + r), zeroing the read columns of their staged
        // rows first; otherwise one warp per (token, 32-row slice of the map).
        const int zc_lo = zlo * W, zc_hi = (zhi + 1) * W - 1;
        const int rc_lo = span > 0 ? (zc_lo >> 5) << 5 : 0;
        const int rc_hi = span > 0 ? min(K_pad, ((zc_hi >> 5) + 1) << 5) : 0;
        for (int q0 = 0; q0 < nq; q0 += L.QB) {
            const int qn = min(L.QB, nq - q0);
            if (paired) {
                const int half = lane >> 4, r = lane & 15;
                for (int pr = warp; 2 * pr < qn; pr += nwarp) {
                    const int ql_ = 2 * pr + half;
                    const bool tok = ql_ < qn;
                    if (tok) {
                        float4 *z = reinterpret_cast<float4 *>(stg + ql_ * L.KS + rc_lo);
                        for (int k = r; k < ((rc_hi - rc_lo) >> 2); k += 16) z[k] = make_float4(0.f, 0.f, 0.f, 0.f);
                    }
                    __syncwarp();
                    const int q = q0 + (tok ? ql_ : 0);
                    const bool live = tok && r < span;
                    const int i = zlo + (live ? r : 0);
                    const int b0 = qlo[q], nb = min(qhi[q] - b0 + 1, BMAX);
                    float cl[BMAX], ch[BMAX];
                    int jl = WP4, jh = -1;
#pragma unroll
                    for (int bb = 0; bb < BMAX; ++bb) {
                        const int b = b0 + bb;
                        const bool on = bb < nb;
                        cl[bb] = on && live ? Ql[q * wp + b] * Yl[b * HP4 + i] : 0.f;
                        ch[bb] = on && live ? Qh[q * wp + b] * Yh[b * HP4 + i] : 0.f;
                        if (on) {
                            jl = min(jl, jlo[b]);
                            jh = max(jh, jhi[b]);
                        }
                    }
                    float *srow = stg + ql_ * L.KS + i * W;
                    const int j4lo = jl >> 2, j4hi = jh >> 2;   // empty when jh < 0
                    for (int j4 = 0; 4 * j4 < W; ++j4) {
                        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
                        if (j4 >= j4lo && j4 <= j4hi) {
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
                        }
                        if (live) {
                            const int j = 4 * j4;
                            srow[j] = acc.x;
                            if (j + 1 < W) srow[j + 1] = acc.y;
                            if (j + 2 < W) srow[j + 2] = acc.z;
                            if (j + 3 < W) srow[j + 3] = acc.w;
                        }
                    }
                }
            } else {
                for (int item = warp; item < qn * IH; item += nwarp) {
                    const int ql_ = IH == 1 ? item : item / IH, i = (item - ql_ * IH) * 32 + lane;
                    const int q = q0 + ql_;
                    const bool live = i < H;
                    const int b0 = qlo[q], nb = min(qhi[q] - b0 + 1, BMAX);
                    float cl[BMAX], ch[BMAX];
                    int jl = WP4, jh = -1;
#pragma unroll
                    for (int bb = 0; bb < BMAX; ++bb) {
                        const int b = b0 + bb;
                        const bool on = bb < nb;
                        cl[bb] = on && live ? Ql[q * wp + b] * Yl[b * HP4 + i] : 0.f;
                        ch[bb] = on && live ? Qh[q * wp + b] * Yh[b * HP4 + i] : 0.f;
                        if (on) {
                            jl = min(jl, jlo[b]);
                            jh = max(jh, jhi[b]);
                        }
                    }
                    float *srow = stg + ql_ * L.KS + i * W;
                    const int j4lo = jl >> 2, j4hi = jh >> 2;   // empty when jh < 0
                    for (int j4 = 0; 4 * j4 < W; ++j4) {
                        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
                        if (j4 >= j4lo && j4 <= j4hi) {
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
                        }
                        if (live) {
                            const int j = 4 * j4;
                            srow[j] = acc.x;
                            if (j + 1 < W) srow[j + 1] = acc.y;
                            if (j + 2 < W) srow[j + 2] = acc.z;
                            if (j + 3 < W) srow[j + 3] = acc.w;
                        }
                    }
                }
                for (int ql_ = warp; ql_ < qn; ql_ += nwarp)   // padding columns [N, K_pad)
                    for (int j = N + lane; j < K_pad; j += 32) stg[ql_ * L.KS + j] = 0.f;
            }
            __syncthreads();
            write_rows(c, stg, L.KS, qn, K_pad, (bf ? wrow0 : row0) + q0, bf, Whi, Wlo, W32, kstride, rc_lo, rc_hi - 1);
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

size_t spatial_smem_bytes(const Ctx &c) {
    SpatialSmem L;
    L.init(c.H, c.W, c.hp, c.wp);
    return (size_t)L.total * sizeof(float);
}

// The WSM kernel's shared memory with the grid-row prefix of V*T frames.
static size_t spatial_compact_smem_bytes(const Ctx &c) {
    return (spatial_smem_bytes(c) + ((size_t)c.V * c.T + 1) * sizeof(int) + 15) & ~(size_t)15;
}

// CTAs per frame: about four waves over the SMs, at most one per grid row.
int spatial_split(const Ctx &c, int resident) {
    const int64_t frames = (int64_t)c.V * c.T;
    int64_t S = (4 * (int64_t)resident + frames - 1) / frames;
    if (S < 1) S = 1;
    if (S > c.H) S = c.H;
    return (int)S;
}

cudaError_t launch_spatial(const Ctx &c, cudaStream_t s) {
    if (c.spatial_mode == WZ_SPATIAL_WSM && c.wsm_levels > 1) return launch_spatial_ml(c, s);
    // tensor path: the 16-row kernel where it applies
    bool launched = false;
    const cudaError_t et = launch_spatial_tc(c, s, &launched);
    if (launched || et != cudaSuccess) return et;
    SpatialSmem L;
    L.init(c.H, c.W, c.hp, c.wp);
    if ((L.AWl & 3) != 0 || (L.AWh & 3) != 0 || (L.stage & 3) != 0 || L.QB < 1) return cudaErrorMisalignedAddress;
    const size_t smem = spatial_smem_bytes(c);
    const bool plain = c.spatial_mode != WZ_SPATIAL_WSM;
    const void *fn;
    if (plain) fn = (const void *)spatial_plain_kernel;
    // BMAX bounds the support of a bilinear column through the synthesis:
    // at most (F - 1) / 2 + 2 coefficients
    else if ((c.F - 1) / 2 + 2 <= 6) fn = (const void *)spatial_wsm_kernel<6>;
    else if ((c.F - 1) / 2 + 2 <= 12) fn = (const void *)spatial_wsm_kernel<12>;
    else return cudaErrorInvalidValue;
    // the compact row list when its prefix fits without costing a resident CTA
    const size_t smem_c = spatial_compact_smem_bytes(c);
    const size_t smem_max = plain || (int64_t)c.V * c.T > kCompactFrames ? smem : smem_c;
    cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_max);
    if (e != cudaSuccess) return e;
    int dev = 0, sms = 0, per_sm = 0, per_sm_c = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
    if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, kSpatialThreads, smem)) != cudaSuccess)
        return e;
    if (smem_max > smem &&
        (e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm_c, fn, kSpatialThreads, smem_c)) != cudaSuccess)
        return e;
    int compact = smem_max > smem && per_sm_c >= per_sm ? 1 : 0;
    const int resident = sms * (per_sm > 0 ? per_sm : 1);
    if (plain) {
        int S = spatial_split(c, resident);
        const unsigned blocks = (unsigned)((int64_t)c.V * c.T * S + kTailBlocks);
        void *args[] = {const_cast<Ctx *>(&c), &S};
        return launch_kernel(fn, dim3(blocks), dim3(kSpatialThreads), smem, s, args, c.pdl != 0);
    }
    // persistent: every resident CTA pulls grid rows; at least kTailBlocks
    // CTAs so that the tail rows are covered
    const unsigned blocks = (unsigned)std::max(resident, kTailBlocks);
    void *args[] = {const_cast<Ctx *>(&c), &compact};
    return launch_kernel(fn, dim3(blocks), dim3(kSpatialThreads), compact ? smem_c : smem, s, args, c.pdl != 0);
}

}  // namespace wz
