// Shared-memory layout of the spatial-operator CTA and the frame-independent
// tables it starts from (Eq. 11-14): the db analysis matrices along height
// and width with the boundary extension folded in, and the first and last
// nonzero entry of every analysis row.  The tables depend only on (H, W,
// filter, extension), so each spatial CTA forms them from its kernel
// parameters at the head of its shared-memory block.
#pragma once

#include "wz_internal.cuh"

namespace wz {

constexpr int kStageFloats = 8 * 1024;   // staged operator rows (32 KB)

struct SpatialSmem {
    int N, hp, wp, H, W, HP4, WP4, K_pad, KS, QB;
    // float offsets; [0, tables) is the frame-independent part.  The width
    // analysis rows A'_v[b][.] are padded to WP4 columns (16-byte rows);
    // jlo / jhi[b] are the first / last column where A'_L or A'_H is nonzero,
    // ilo / ihi[a] the first / last row where A_L or A_H is nonzero.
    int AHl, AHh, AWl, AWh, jlo, jhi, ilo, ihi, tables;
    int G, PAl, PAh, Yl, Yh, Ql, Qh, red, qlo, qhi, M, stage, total;
    // Every table starts on a 16-byte boundary (float4 reads of Y, staged rows).
    __host__ __device__ void init(int H_, int W_, int hp_, int wp_) {
        H = H_; W = W_; hp = hp_; wp = wp_; N = H * W;
        K_pad = (N + 31) & ~31;
        KS = K_pad + 4;                            // staged row stride (see write_rows)
        QB = kStageFloats / KS;                    // rows staged at a time (>= 1 for N <= 4096)
        HP4 = (H + 3) & ~3;
        WP4 = (W + 3) & ~3;
        int o = 0;
        auto take = [&](int n) {
            const int at = o;
            o = (o + n + 3) & ~3;
            return at;
        };
        AHl = take(hp * H);
        AHh = take(hp * H);
        AWl = take(wp * WP4);
        AWh = take(wp * WP4);
        jlo = take(wp);
        jhi = take(wp);
        ilo = take(hp);
        ihi = take(hp);
        tables = o;
        G = take(hp * wp);
        PAl = take(hp * H);
        PAh = take(hp * H);
        Yl = take(wp * HP4);
        Yh = take(wp * HP4);
        Ql = take(W * wp);
        Qh = take(W * wp);
        red = take(64);
        qlo = take(W);
        qhi = take(W);
        M = take(N);                               // saliency map (ablation mode "saliency")
        stage = take(QB * KS);
        total = o;
    }
};

// Synthesis weight of coefficient a at sample y (upsample, filter, keep the
// samples from offset F - 2).
__device__ __forceinline__ float synth(const float *rec, int F, int y, int a) {
    const int k = y + F - 2 - 2 * a;
    return (k >= 0 && k < F) ? rec[k] : 0.f;
}

// Half-pixel bilinear source (align_corners = false): rows y0, y1, weight of
// y1.  The source coordinate s = (i + 1/2) in / out - 1/2, clamped at 0, is
// the rational ((2i + 1) in - out) / (2 out): its floor and remainder are
// exact in integers, and the weight is the remainder divided in fp32.
__device__ __forceinline__ void bilinear_src(int i, int in, int out, int &y0, int &y1, float &l) {
    const int num = (2 * i + 1) * in - out, den = 2 * out;
    int f = 0, rem = 0;
    if (num > 0) {
        f = num / den;
        rem = num - f * den;
    }
    if (f > in - 1) {
        f = in - 1;
        rem = 0;
    }
    y0 = f;
    y1 = f + 1 < in ? f + 1 : in - 1;
    l = (float)rem / (float)den;
}

// Coefficients a with synth(y, a) != 0 for y in {y0, y1}: y + F - 2 - 2a in [0, F).
__device__ __forceinline__ void synth_support(int y0, int y1, int F, int na, int &lo, int &hi) {
    lo = y0 >> 1;
    hi = min(na - 1, (y1 + F - 2) >> 1);
}

// Staged rows [0, qn) of a grid row (row stride ks floats) go out in
// 8-column groups: bf16 hi and lo halves at tile_index(r, 8 g, w_rows)
// (tensor path; r = r_first + row) or fp32 rows (CUDA-core path).  On the
// tensor path a warp writes one 8-row group x 32-column chunk: lane = (column
// quarter, row within the group), so its 32 16-byte stores fill one
// contiguous 512-byte block of the tiled layout.  A stride ks = K_pad + 4
// keeps the eight rows' shared-memory reads on distinct banks.  Columns
// outside [zc_lo, zc_hi] are zero in every staged row: a column group that
// holds only such columns is written as zeros without reading the stage.
__device__ __forceinline__ void write_rows(const Ctx &c, const float *stg, int ks, int qn, int K_pad, int64_t r_first,
                                           bool bf, __nv_bfloat16 *Whi, __nv_bfloat16 *Wlo, float *W32, size_t kstride,
                                           int zc_lo, int zc_hi) {
    // operator rows that exist: w_rows (tensor path), rows_total (fp32 rows)
    if (!wz_in_range(c.status, r_first + qn <= (bf ? c.w_rows : c.rows_total))) return;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarp = (int)(blockDim.x >> 5);
    if (bf) {
        const int rr = lane & 7, qq = lane >> 3;
        const int64_t rg0 = r_first >> 3, rg1 = (r_first + qn - 1) >> 3;
        const int nrg = (int)(rg1 - rg0 + 1), nk = K_pad >> 5;
        for (int it = warp; it < nrg * nk; it += nwarp) {
            const int rgi = it / nk, g4 = it - rgi * nk;
            const int64_t r = (rg0 + rgi) * 8 + rr;
            const int ql_ = (int)(r - r_first);
            if (ql_ < 0 || ql_ >= qn) continue;
            uint32_t hw[4] = {0u, 0u, 0u, 0u}, lw[4] = {0u, 0u, 0u, 0u};
            if (32 * g4 + 31 >= zc_lo && 32 * g4 <= zc_hi) {
                const float *src = stg + ql_ * ks + 32 * g4 + 8 * qq;
                const float4 v0 = *reinterpret_cast<const float4 *>(src);
                const float4 v1 = *reinterpret_cast<const float4 *>(src + 4);
                const float v[8] = {v0.x, v0.y, v0.z, v0.w, v1.x, v1.y, v1.z, v1.w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const __nv_bfloat162 hh = __floats2bfloat162_rn(v[2 * e], v[2 * e + 1]);
                    const __nv_bfloat162 ll =
                        __floats2bfloat162_rn(v[2 * e] - __low2float(hh), v[2 * e + 1] - __high2float(hh));
                    hw[e] = *reinterpret_cast<const uint32_t *>(&hh);
                    lw[e] = *reinterpret_cast<const uint32_t *>(&ll);
                }
            }
            const size_t ti = (size_t)g4 * kstride + (size_t)(r >> 3) * 256 + (size_t)rr * 8 + (size_t)qq * 64;
            *reinterpret_cast<uint4 *>(Whi + ti) = make_uint4(hw[0], hw[1], hw[2], hw[3]);
            *reinterpret_cast<uint4 *>(Wlo + ti) = make_uint4(lw[0], lw[1], lw[2], lw[3]);
        }
    } else {
        const int G8 = K_pad / 8;
        for (int it = threadIdx.x; it < qn * G8; it += blockDim.x) {
            const int ql_ = it / G8, g = it - ql_ * G8;
            float *dst = W32 + (size_t)(r_first + ql_) * K_pad + 8 * g;
            float4 v0 = make_float4(0.f, 0.f, 0.f, 0.f), v1 = v0;
            if (8 * g + 7 >= zc_lo && 8 * g <= zc_hi) {
                const float *src = stg + ql_ * ks + 8 * g;
                v0 = *reinterpret_cast<const float4 *>(src);
                v1 = *reinterpret_cast<const float4 *>(src + 4);
            }
            *reinterpret_cast<float4 *>(dst) = v0;
            *reinterpret_cast<float4 *>(dst + 4) = v1;
        }
    }
}

constexpr int kSpatialThreads = 256;
constexpr int kTailBlocks = 64;
constexpr int kCompactFrames = 2048;   // frames whose work prefix a spatial CTA keeps in shared memory

// pre[f] = sum of count(f') over the frames f' < f, pre[F] = the total
// (F <= kCompactFrames; a block-wide scan, every thread a contiguous range of
// frames).  The caller synchronises the block before reading pre.
template <class Count>
__device__ void frame_prefix(int F, int *pre, int *wsum, Count count) {
    constexpr int kPer = kCompactFrames / kSpatialThreads;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int per = (F + kSpatialThreads - 1) / kSpatialThreads;
    const int f0 = tid * per;
    int cnt[kPer];
    int sum = 0;
#pragma unroll
    for (int k = 0; k < kPer; ++k) {
        cnt[k] = (k < per && f0 + k < F) ? count(f0 + k) : 0;
        sum += cnt[k];
    }
    int incl = sum;
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
    }
    if (lane == 31) wsum[warp] = incl;
    __syncthreads();
    int run = incl - sum;
    for (int w = 0; w < warp; ++w) run += wsum[w];
#pragma unroll
    for (int k = 0; k < kPer; ++k) {
        if (k < per && f0 + k < F) pre[f0 + k] = run;
        run += cnt[k];
    }
    if (tid == 0) {
        int tot = 0;
        for (int w = 0; w < kSpatialThreads / 32; ++w) tot += wsum[w];
        pre[F] = tot;
    }
}

// Rows past the produced count (tau > 0): index -1, zero tokens.  Tail CTA
// tb of kTailBlocks.
__device__ inline void tail_rows(const Ctx &c, int tb) {
    const size_t esz = c.dtype == WZ_DTYPE_BF16 ? 2 : 4;
    const int nvec = (int)((size_t)c.D * esz / 16);
    for (int v = 0; v < c.V; ++v) {
        const int r0 = c.vpar[v].row0 + c.prod[v];
        const int r1 = c.vpar[v].row0 + c.vpar[v].B;
        for (int r = r0 + tb; r < r1; r += kTailBlocks) {
            uint4 *o = reinterpret_cast<uint4 *>(static_cast<char *>(c.out) + (size_t)r * c.D * esz);
            for (int k = threadIdx.x; k < nvec; k += blockDim.x) o[k] = make_uint4(0u, 0u, 0u, 0u);
            if (threadIdx.x < 3) c.out_index[(size_t)r * 3 + threadIdx.x] = -1;
        }
    }
}

// The tensor-core work units of frame f (the temporal kernel placed them: the
// first block's units at ustart[f], the later blocks' at ustartB[f]):
// column blocks of <= 256 tokens, each in groups of unit_tiles(round16(nc))
// 128-channel tiles, as even as n_ct allows.  A record is (f, j0, first tile,
// nc | tiles << 9 | kc_lo << 12 | kc_hi << 20 | ranged): the unit's operator
// rows are zero outside the 32-column chunks [kc_lo, kc_hi] (K_pad <= 4096,
// so chunks fit 8 bits).  With the row supports ilo / ihi of the height
// analysis (single-level WSM; h x w the frame's grid) that range is the
// chunks of the map rows the block's grid rows reach, else every chunk; and
// for blocks of more than 64 tokens (two MMAs per step, see unit_fused) each
// chunk also gets the rows of the block whose grid rows reach it (Ctx::krange,
// flag kUnitRanged): the others are zero there, so the condensation neither
// loads nor multiplies them.
__device__ inline void unit_records(const Ctx &c, int64_t f, int n, int h = 0, int w = 0, const int *ilo = nullptr,
                                    const int *ihi = nullptr) {
    const int v = (int)(f / c.T);
    int4 *units = c.units + (size_t)v * c.max_units_v;
    int u0 = c.ustart[f];
    const int KC = c.K_pad >> 5;
    for (int j0 = 0; j0 < n; j0 += kColBlock) {
        if (j0 == kColBlock) u0 = c.ustartB[f];   // later blocks: the second part of the list
        const int nc = min(kColBlock, n - j0);
        const int cg = unit_tiles((nc + 15) / 16 * 16);
        const int cnt = (c.n_ct + cg - 1) / cg;
        int klo = 0, khi = KC - 1;
        if (ilo != nullptr && w > 0) {
            // the analysis rows of grid rows p0..p1 lie in [alo(p0), ahi(p1)]
            // (both ends grow with p): the union of their row supports
            const int p0 = j0 / w, p1 = min(h - 1, (j0 + nc - 1) / w);
            int y0, y1, alo, ahi, a0, a1;
            float ly;
            bilinear_src(p0, c.H, h, y0, y1, ly);
            synth_support(y0, y1, c.F, c.hp, a0, ahi);
            bilinear_src(p1, c.H, h, y0, y1, ly);
            synth_support(y0, y1, c.F, c.hp, alo, a1);
            int zlo = c.H, zhi = -1;
            for (int a = a0; a <= a1; ++a) {
                zlo = min(zlo, ilo[a]);
                zhi = max(zhi, ihi[a]);
            }
            if (zhi >= zlo) {
                klo = min(KC - 1, (zlo * c.W) >> 5);
                khi = min(KC - 1, ((zhi + 1) * c.W - 1) >> 5);
            } else {
                klo = khi = 0;   // an all-zero block: one chunk of zeros
            }
        }
        const int ncp = (nc + 15) & ~15;
        int ranged = 0;
        if (ilo != nullptr && w > 0 && c.krange != nullptr && !unit_fused(ncp) && (j0 >> 8) < c.krange_nblk) {
            // per chunk: the grid rows p of the block whose map rows [zl(p),
            // zh(p)] meet the chunk's map rows, as 16-row operator ranges
            ranged = kUnitRanged;
            uint16_t *kr = c.krange + ((size_t)f * c.krange_nblk + (j0 >> 8)) * KC;
            const int p0 = j0 / w, p1 = min(h - 1, (j0 + nc - 1) / w);
            // a warp per chunk, a lane per grid row (p1 - p0 < 64): the rows
            // that reach the chunk by ballot
            const int lane = threadIdx.x & 31, nwarp = (int)(blockDim.x >> 5);
            int zl[2], zh[2];
#pragma unroll
            for (int r = 0; r < 2; ++r) {
                const int p = p0 + lane + 32 * r;
                zl[r] = c.H;
                zh[r] = -1;
                if (p <= p1) {
                    int y0, y1, a0, a1;
                    float ly;
                    bilinear_src(p, c.H, h, y0, y1, ly);
                    synth_support(y0, y1, c.F, c.hp, a0, a1);
                    for (int a = a0; a <= a1; ++a) {
                        zl[r] = min(zl[r], ilo[a]);
                        zh[r] = max(zh[r], ihi[a]);
                    }
                }
            }
            for (int kc = klo + (int)(threadIdx.x >> 5); kc <= khi; kc += nwarp) {
                const int z0 = (kc * 32) / c.W, z1 = min(c.H - 1, (kc * 32 + 31) / c.W);
                const unsigned m0 = __ballot_sync(0xffffffffu, zh[0] >= z0 && zl[0] <= z1);
                const unsigned m1 = __ballot_sync(0xffffffffu, zh[1] >= z0 && zl[1] <= z1);
                int pf = h, pl = -1;
                if (m0 | m1) {
                    pf = p0 + (m0 ? __ffs(m0) - 1 : 32 + __ffs(m1) - 1);
                    pl = p0 + (m1 ? 63 - __clz(m1) : 31 - __clz(m0));
                }
                int ja = 0, jb = 16;   // a chunk no row reaches: one group of zero rows
                if (pl >= pf) {
                    const int t0 = max(pf * w, j0) - j0, t1 = min((pl + 1) * w, j0 + nc) - j0;
                    ja = (t0 >> 4) << 4;
                    jb = min(ncp, (t1 + 15) & ~15);
                    if (jb <= ja) {
                        ja = 0;
                        jb = 16;
                    }
                }
                if (lane == 0) kr[kc] = (uint16_t)((ja >> 4) | ((jb >> 4) << 8));
            }
        }
        for (int li = threadIdx.x; li < cnt; li += blockDim.x) {
            // tiles of group li: [li * n_ct / cnt, (li + 1) * n_ct / cnt), sizes differing by at most one
            const int ct = li * c.n_ct / cnt, ct1 = (li + 1) * c.n_ct / cnt;
            if (u0 + li < c.max_units_v)
                units[u0 + li] = make_int4((int)f, j0, ct, nc | ((ct1 - ct) << 9) | (klo << 12) | (khi << 20) | ranged);
        }
        u0 += cnt;
    }
}

// The frame-independent tables, built by each spatial CTA into the head of
// its own shared memory (tb) from the filter taps in the kernel parameters:
//   A[a][i] = sum_j dec[j] [ext(2a + 1 - j) == i]   (analysis along a side)
//   jlo/jhi[b] = first / last column j with A'[b][j] != 0, ilo/ihi[a] the
//                same for the rows of A
// Called by the whole block (hp + wp <= blockDim.x).
__device__ inline void build_spatial_tables_smem(const Ctx &c, const SpatialSmem &L, float *tb) {
    int *ti = reinterpret_cast<int *>(tb);
    const int H = c.H, W = c.W, hp = c.hp, wp = c.wp, F = c.F;
    // one thread per analysis row: zero it, add tap j at ext(2a + 1 - j) for
    // j = 0, 1, ... (each entry sums its taps in ascending order), then scan
    // the row for its first and last nonzero column
    const int r = threadIdx.x;
    if (r < hp + wp) {
        const bool hgt = r < hp;
        const int a = hgt ? r : r - hp, n = hgt ? H : W, len = hgt ? H : L.WP4;
        float *lo = tb + (hgt ? L.AHl + a * H : L.AWl + a * L.WP4);
        float *hi = tb + (hgt ? L.AHh + a * H : L.AWh + a * L.WP4);
        for (int i = 0; i < len; ++i) {
            lo[i] = 0.f;
            hi[i] = 0.f;
        }
        for (int j = 0; j < F; ++j) {
            const int i = ext_index(2 * a + 1 - j, n, c.mode);   // -1: outside (zero extension)
            if (i >= 0 && i < n) {
                lo[i] += c.dec_lo[j];
                hi[i] += c.dec_hi[j];
            }
        }
        int first = hgt ? H : L.WP4, last = -1;
        for (int i = 0; i < n; ++i)
            if (lo[i] != 0.f || hi[i] != 0.f) {
                first = min(first, i);
                last = i;
            }
        ti[(hgt ? L.ilo : L.jlo) + a] = first;
        ti[(hgt ? L.ihi : L.jhi) + a] = last;
    }
    __syncthreads();
}

// Bytes of the frame-independent tables for an image of H x W and F taps.
inline size_t spatial_table_bytes(int H, int W, int F) {
    SpatialSmem L;
    L.init(H, W, (H + F - 1) / 2, (W + F - 1) / 2);
    return (size_t)L.tables * 4;
}


}  // namespace wz

namespace wz {

// ---- multi-level WSM --------------------------------------------------------
// With J levels the DWT2 cascades on LL (level l of an h_{l-1} x w_{l-1} band
// gives h_l x w_l subbands).  Folded into matrices along one side, level l's
// analysis rows are AH_u^l = A_u^l AH_L^{l-1} (h_l x H, AH_L^0 = I, A_u^l the
// single-level analysis of length h_{l-1}, extension folded in) and its
// synthesis columns SH_u^l = SH_L^{l-1} S_u^l (H x h_l).  The operator is
//
//   W_m[(p,q),(i,j)] = sum_l sum_v sum_b Q_v^l[q,b] AW_v^l[b,j] Y_v^l[b,i],
//   Y_v^l[b,i]       = sum_u sum_a P_u^l[p,a] AH_u^l[a,i] g_uv^l[a,b],
//
// P_u^l = R_y SH_u^l, Q_v^l = R_x SW_v^l, g_LH = g_HL = g_HH = G_l (the gate
// of level l), g_LL = 1 at level J and 0 above it (that band is decomposed
// further).  One level gives the single-level operator.
struct MLTables {
    int J, H, W;
    int h[kMaxLevels + 1], w[kMaxLevels + 1];
    // copied into shared memory: [0, copy)
    int AHl[kMaxLevels], AHh[kMaxLevels];   // [h_l][H]
    int AWl[kMaxLevels], AWh[kMaxLevels];   // [w_l][W]
    int blo[kMaxLevels], bhi[kMaxLevels];   // [W] int: rows b of AW^l nonzero at column j
    int copy;
    // read from global memory
    int SHl[kMaxLevels], SHh[kMaxLevels];   // [H][h_l]
    int SWl[kMaxLevels], SWh[kMaxLevels];   // [W][w_l]
    int slo[kMaxLevels], shi[kMaxLevels];   // [H] int: columns a of SH^l nonzero at row y
    int xlo[kMaxLevels], xhi[kMaxLevels];   // [W] int: columns b of SW^l nonzero at row x
    int total;
    __host__ __device__ void init(int H_, int W_, int F, int J_) {
        J = J_; H = H_; W = W_;
        for (int l = 0; l <= kMaxLevels; ++l) {
            h[l] = level_size(H, F, l);
            w[l] = level_size(W, F, l);
        }
        int o = 0;
        auto take = [&](int n) {
            const int at = o;
            o = (o + n + 3) & ~3;
            return at;
        };
        for (int l = 0; l < J; ++l) {
            AHl[l] = take(h[l + 1] * H);
            AHh[l] = take(h[l + 1] * H);
            AWl[l] = take(w[l + 1] * W);
            AWh[l] = take(w[l + 1] * W);
            blo[l] = take(W);
            bhi[l] = take(W);
        }
        copy = o;
        for (int l = 0; l < J; ++l) {
            SHl[l] = take(H * h[l + 1]);
            SHh[l] = take(H * h[l + 1]);
            SWl[l] = take(W * w[l + 1]);
            SWh[l] = take(W * w[l + 1]);
            slo[l] = take(H);
            shi[l] = take(H);
            xlo[l] = take(W);
            xhi[l] = take(W);
        }
        total = o;
    }
};

inline size_t ml_table_bytes(int H, int W, int F, int J) {
    MLTables T;
    T.init(H, W, F, J);
    return (size_t)T.total * 4;
}

// Shared memory of one multi-level spatial CTA.
struct MLSmem {
    int HP4, K_pad, KS, QB;
    int G;                                  // the frame's gates, levels 1..J (c.goff layout)
    int Ql[kMaxLevels], Qh[kMaxLevels];     // [w][w_l] (w <= W)
    int qlo[kMaxLevels], qhi[kMaxLevels];   // [W] int
    int PAl, PAh;                           // [h_1][H], one level at a time
    int Yl[kMaxLevels], Yh[kMaxLevels];     // [w_l][HP4]
    int red, stage, total;
    __host__ __device__ void init(const MLTables &T) {
        const int H = T.H, W = T.W, N = H * W;
        K_pad = (N + 31) & ~31;
        KS = K_pad + 4;                            // staged row stride (see write_rows)
        QB = kStageFloats / KS;
        HP4 = (H + 3) & ~3;
        int o = T.copy;
        auto take = [&](int n) {
            const int at = o;
            o = (o + n + 3) & ~3;
            return at;
        };
        int gs = 0;
        for (int l = 1; l <= T.J; ++l) gs += T.h[l] * T.w[l];
        G = take(gs);
        for (int l = 0; l < T.J; ++l) {
            Ql[l] = take(W * T.w[l + 1]);
            Qh[l] = take(W * T.w[l + 1]);
            qlo[l] = take(W);
            qhi[l] = take(W);
            Yl[l] = take(T.w[l + 1] * HP4);
            Yh[l] = take(T.w[l + 1] * HP4);
        }
        int hmax = 0;
        for (int l = 1; l <= T.J; ++l) hmax = T.h[l] > hmax ? T.h[l] : hmax;
        PAl = take(hmax * H);
        PAh = take(hmax * H);
        red = take(64);
        stage = take(QB * KS);
        total = o;
    }
};

// Build the multi-level tables into c.stab (one CTA).  Level l's matrices
// are formed from level l-1's in global memory; a block barrier separates
// the levels (global writes of the block are visible to it after the barrier).
static __device__ __noinline__ void build_ml_tables(const Ctx &c) {
    MLTables T;
    T.init(c.H, c.W, c.F, c.wsm_levels);
    float *tb = c.stab;
    int *ti = reinterpret_cast<int *>(c.stab);
    const int F = c.F, H = c.H, W = c.W;
    // supports, gathered with shared-memory atomics while the tables are formed
    __shared__ int sup[6][kMaxLevels][WZ_MAX_HW];   // blo, bhi (AW rows), slo, shi (SH), xlo, xhi (SW)
    for (int k = threadIdx.x; k < kMaxLevels * WZ_MAX_HW; k += blockDim.x) {
        const int l = k / WZ_MAX_HW, x = k % WZ_MAX_HW;
        sup[0][l][x] = sup[2][l][x] = sup[4][l][x] = 1 << 30;
        sup[1][l][x] = sup[3][l][x] = sup[5][l][x] = -1;
    }
    __syncthreads();
    for (int l = 0; l < T.J; ++l) {
        // analysis rows: AX_u^{l+1}[a][i] = sum_j dec_u[j] AX_L^l[ext(2a + 1 - j)][i]
        for (int side = 0; side < 2; ++side) {
            const int n = side ? W : H, nin = side ? T.w[l] : T.h[l], nout = side ? T.w[l + 1] : T.h[l + 1];
            float *lo = tb + (side ? T.AWl[l] : T.AHl[l]), *hi = tb + (side ? T.AWh[l] : T.AHh[l]);
            const float *prev = l ? tb + (side ? T.AWl[l - 1] : T.AHl[l - 1]) : nullptr;
            for (int k = threadIdx.x; k < nout * n; k += blockDim.x) {
                const int a = k / n, i = k % n;
                float sl = 0.f, sh = 0.f;
#pragma unroll 4
                for (int j = 0; j < F; ++j) {
                    const int e = ext_index(2 * a + 1 - j, nin, c.mode);
                    if (e < 0) continue;
                    const float x = prev ? prev[e * n + i] : (e == i ? 1.f : 0.f);
                    sl += c.dec_lo[j] * x;
                    sh += c.dec_hi[j] * x;
                }
                lo[k] = sl;
                hi[k] = sh;
                if (side && (sl != 0.f || sh != 0.f)) {
                    atomicMin(&sup[0][l][i], a);
                    atomicMax(&sup[1][l][i], a);
                }
            }
            // synthesis columns: SX_u^{l+1}[y][a] = sum_k SX_L^l[y][k] rec_u[k + F - 2 - 2a]
            float *slo_ = tb + (side ? T.SWl[l] : T.SHl[l]), *shi_ = tb + (side ? T.SWh[l] : T.SHh[l]);
            const float *sprev = l ? tb + (side ? T.SWl[l - 1] : T.SHl[l - 1]) : nullptr;
            for (int k = threadIdx.x; k < n * nout; k += blockDim.x) {
                const int y = k / nout, a = k % nout;
                float sl = 0.f, sh = 0.f;
                const int k0 = max(0, 2 * a - F + 2), k1 = min(nin - 1, 2 * a + 1);
#pragma unroll 4
                for (int kk = k0; kk <= k1; ++kk) {
                    const float x = sprev ? sprev[y * nin + kk] : (y == kk ? 1.f : 0.f);
                    sl += x * c.rec_lo[kk + F - 2 - 2 * a];
                    sh += x * c.rec_hi[kk + F - 2 - 2 * a];
                }
                slo_[k] = sl;
                shi_[k] = sh;
                if (sl != 0.f || sh != 0.f) {
                    atomicMin(&sup[side ? 4 : 2][l][y], a);
                    atomicMax(&sup[side ? 5 : 3][l][y], a);
                }
            }
        }
        __syncthreads();
    }
    // supports (empty: lo = the band length, hi = -1)
    for (int l = 0; l < T.J; ++l) {
        for (int x = threadIdx.x; x < W; x += blockDim.x) {
            ti[T.blo[l] + x] = min(sup[0][l][x], T.w[l + 1]);
            ti[T.bhi[l] + x] = sup[1][l][x];
            ti[T.xlo[l] + x] = min(sup[4][l][x], T.w[l + 1]);
            ti[T.xhi[l] + x] = sup[5][l][x];
        }
        for (int y = threadIdx.x; y < H; y += blockDim.x) {
            ti[T.slo[l] + y] = min(sup[2][l][y], T.h[l + 1]);
            ti[T.shi[l] + y] = sup[3][l][y];
        }
    }
}

}  // namespace wz
