// Temporal tail of the condensation pass, one CTA per video, in fp64, with
// the per-video arrays in shared memory:
//
//   gamma_t   min-max of delta over the video         Section 3.2.2
//             (r_t and delta_t, Eq. 7, come from frame_stats)
//   M         {1} u {t : delta_t >= tau}              Section 3.2.2 (frame filter)
//   r~        Haar DWT of r_M, detail * pair-mean of gamma, inverse DWT   Eq. 8-10
//   n_m       largest-remainder apportionment of B over max(r~, 0),
//             capped at N with re-apportionment       Eq. 5, Eq. 15
//   offsets   exclusive prefix of n over frames       Eq. 18 (temporal order)
//   (h, w)    condensation grid of each frame         Eq. 16
//   units     the tensor-core work list of the frame  (this library)
//
// Every reduction runs in a fixed order for a fixed block size, so results
// do not depend on scheduling.
#include <cmath>

#include "wz_spatial.cuh"

namespace wz {

constexpr int kTemporalThreads = 512;

// Exclusive scan of one int per thread over the block; returns the prefix and
// writes the block total to *total.
__device__ int block_excl_scan(int x, int *ws, int *total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int nw = blockDim.x >> 5;
    int incl = x;
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
    }
    __syncthreads();
    if (lane == 31) ws[warp] = incl;
    __syncthreads();
    if (warp == 0) {
        int w = lane < nw ? ws[lane] : 0;
        int wi = w;
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, wi, o);
            if (lane >= o) wi += y;
        }
        if (lane < nw) ws[32 + lane] = wi - w;
        if (lane == nw - 1) ws[64] = wi;
    }
    __syncthreads();
    const int r = ws[32 + warp] + incl - x;
    *total = ws[64];
    __syncthreads();
    return r;
}

// Three exclusive block scans at once (same barriers as one); ws holds
// >= 3 * 33 ints.  Returns the exclusive prefixes and the totals.
template <int K>
__device__ void block_excl_scan(const int (&x)[K], int *ws, int (&excl)[K], int (&total)[K]) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int nw = blockDim.x >> 5;
    int incl[K];
#pragma unroll
    for (int k = 0; k < K; ++k) incl[k] = x[k];
    for (int o = 1; o < 32; o <<= 1) {
#pragma unroll
        for (int k = 0; k < K; ++k) {
            const int y = __shfl_up_sync(0xffffffffu, incl[k], o);
            if (lane >= o) incl[k] += y;
        }
    }
    __syncthreads();
    if (lane == 31) {
#pragma unroll
        for (int k = 0; k < K; ++k) ws[33 * k + warp] = incl[k];
    }
    __syncthreads();
    if (warp == 0) {
#pragma unroll
        for (int k = 0; k < K; ++k) {
            const int w = lane < nw ? ws[33 * k + lane] : 0;
            int wi = w;
            for (int o = 1; o < 32; o <<= 1) {
                const int y = __shfl_up_sync(0xffffffffu, wi, o);
                if (lane >= o) wi += y;
            }
            __syncwarp();
            if (lane < nw) ws[33 * k + lane] = wi - w;
            if (lane == nw - 1) ws[33 * k + 32] = wi;
        }
    }
    __syncthreads();
#pragma unroll
    for (int k = 0; k < K; ++k) {
        excl[k] = ws[33 * k + warp] + incl[k] - x[k];
        total[k] = ws[33 * k + 32];
    }
    __syncthreads();
}


// h = min(H, ceil(sqrt(n H / W))): a float estimate corrected to the exact
// smallest h >= 1 with h^2 W >= n H in integers.
__device__ __forceinline__ int grid_h(int n, int H, int W) {
    if (n <= 0) return 0;
    long long h = (long long)ceilf(sqrtf((float)n * (float)H / (float)W));
    if (h < 1) h = 1;
    while (h * h * W < (long long)n * H) ++h;
    while (h > 1 && (h - 1) * (h - 1) * W >= (long long)n * H) --h;
    return (int)(h < H ? h : H);
}

// Shared-memory arrays of one video, indexed by retained frame m (wgt,
// keys, lst, nb) or by frame t (nf).
// keys start on a 16-byte boundary (the rank reads them two at a time)
__host__ __device__ inline size_t temporal_smem_keys(int T) { return ((size_t)T * 8 + 15) & ~(size_t)15; }
// the quotas of the current round (double, indexed by m) follow nf
__host__ __device__ inline size_t temporal_smem_quota(int T) {
    return (temporal_smem_keys(T) + (size_t)T * (8 + 4 + 4 + 4) + 7) & ~(size_t)7;
}
__host__ __device__ inline size_t temporal_smem_offset_coef(int T) { return temporal_smem_quota(T) + (size_t)T * 8; }
// WTA coefficient arrays: the longest subband of any level (any filter).
__host__ __device__ inline int temporal_coef_len(int T, int J) {
    const int k = (T + kMaxTaps - 1) / 2;
    return J > 1 && k < kMaxTaps ? kMaxTaps : k;
}
// Detail coefficients of all J levels, back to back (lengths halve, plus at
// most F/2 per level).
__host__ __device__ inline int temporal_detail_len(int T, int J) {
    const int k = temporal_coef_len(T, J);
    return J > 1 ? 2 * k + J * kMaxTaps : k;
}
// The coefficient part: approximation A0 | details | (J > 1) A1 | G0 | G1.
__host__ __device__ inline size_t temporal_smem_bytes(int T, int J) {
    const size_t k = (size_t)temporal_coef_len(T, J);
    const size_t coef = k + (size_t)temporal_detail_len(T, J) + (J > 1 ? 3 * k : 0);
    return temporal_smem_offset_coef(T) + sizeof(double) * coef;
}

// Threads of the CTA: one frame per thread up to 512 frames, at most
// WZ_MAX_T / kTemporalThreads frames per thread beyond (fp64 work scales with
// the warps).
inline int temporal_threads(int T) { return T <= 512 ? (T < 32 ? 32 : (T + 31) / 32 * 32) : 512; }

// WTA levels 2..J (J > 1): level 1 left its approximation in A0, its gate in
// G0 and its gated details in dall[0, K1).  Each further level analyses the
// previous approximation (gate: the pairwise mean of the previous gate) and
// appends its gated details to dall; the inverse then cascades back to level
// 1's approximation, whose buffer is returned.  Called by the whole block.
__device__ __noinline__ const double *wta_deeper_levels(const Ctx &c, double *A0, double *A1, double *G0, double *G1,
                                                         double *dall, int K1, int J) {
    const int FT = c.wta_F;
    int lens[kMaxLevels + 1], doff[kMaxLevels];
    lens[1] = K1;
    doff[0] = 0;
    for (int j = 2, o = K1; j <= J; ++j) {
        lens[j] = (lens[j - 1] + FT - 1) / 2;
        doff[j - 1] = o;
        o += lens[j];
    }
    double *ain = A0, *gin = G0, *aout = A1, *gout = G1;
    for (int j = 2; j <= J; ++j) {
        const int n = lens[j - 1], K = lens[j];
        for (int k = threadIdx.x; k < K; k += blockDim.x) {
            double ca = 0.0, cd = 0.0;
            for (int i = 0; i < FT; ++i) {
                const double x = ain[ext_index(2 * k + 1 - i, n, WZ_MODE_SYMMETRIC)];
                ca += c.wta_dec_lo[i] * x;
                cd += c.wta_dec_hi[i] * x;
            }
            const double g = 0.5 * (gin[ext_index(2 * k, n, WZ_MODE_SYMMETRIC)] +
                                    gin[ext_index(2 * k + 1, n, WZ_MODE_SYMMETRIC)]);
            aout[k] = ca;
            if (j < J) gout[k] = g;
            dall[doff[j - 1] + k] = g * cd;
        }
        __syncthreads();
        double *t_ = ain;
        ain = aout;
        aout = t_;
        t_ = gin;
        gin = gout;
        gout = t_;
    }
    for (int j = J; j >= 2; --j) {   // inverse of levels J .. 2
        const int n = lens[j - 1], K = lens[j];
        const double *dj = dall + doff[j - 1];
        for (int m = threadIdx.x; m < n; m += blockDim.x) {
            double x = 0.0;
            const int alo = m >> 1, ahi = min(K - 1, (m + FT - 2) >> 1);
            for (int ai = alo; ai <= ahi; ++ai) {
                const int kk = m + FT - 2 - 2 * ai;
                x += c.wta_rec_lo[kk] * ain[ai] + c.wta_rec_hi[kk] * dj[ai];
            }
            aout[m] = x;
        }
        __syncthreads();
        double *t_ = ain;
        ain = aout;
        aout = t_;
    }
    return ain;
}

__global__ void __launch_bounds__(kTemporalThreads) temporal_kernel(Ctx c) {
    pdl_wait();
    pdl_trigger();
    if ((int)blockIdx.x == c.V) {
        // the extra CTA: the spatial kernel's row counter, the condensation's
        // unit counter and, with several WSM levels, the multi-level tables
        // of the spatial operator (the single-level kernel forms its tables
        // itself)
        if (threadIdx.x == 0 && c.spatial_next) {
            c.spatial_next[0] = 0;
            c.spatial_next[1] = 0;
        }
        if (c.wsm_levels > 1) build_ml_tables(c);
        return;
    }
    extern __shared__ __align__(16) unsigned char tsm[];
    __shared__ double dscr[64];
    __shared__ long long lscr[66];
    __shared__ int iscr[4 * 33];
    const int v = blockIdx.x;
    const int T = c.T;
    const int64_t base = (int64_t)v * T;
    const VideoPar vp = c.vpar[v];
    double *fr = c.fr + base * 4;          // r, delta, gamma, r~
    double *wgt = reinterpret_cast<double *>(tsm);                        // weight of retained frame m
    unsigned long long *keys = reinterpret_cast<unsigned long long *>(tsm + temporal_smem_keys(T));   // remainder key
    int *lst = reinterpret_cast<int *>(keys + T);                         // retained frames
    int *nb = lst + T;                     // budget of retained frame m; -1 while active
    int *nf = nb + T;                      // budget of frame t
    double *qv = reinterpret_cast<double *>(tsm + temporal_smem_quota(T));   // quota of retained frame m
    const int J = c.wta_levels;
    const int KH = temporal_coef_len(T, J);
    double *A0 = reinterpret_cast<double *>(tsm + temporal_smem_offset_coef(T));   // WTA approximation
    double *dall = A0 + KH;                                                         // gated details, all levels
    double *A1 = dall + temporal_detail_len(T, J);                                  // (J > 1) ping-pong
    double *G0 = A1 + KH, *G1 = G0 + KH;                                            // (J > 1) gates of a level

    // r_t and delta_t come from frame_stats, which also kept the range of
    // delta over the video (Eq. 7)
    const double lo = __longlong_as_double((long long)c.drange[2 * v]);
    const double hi = __longlong_as_double((long long)c.drange[2 * v + 1]);
    // gamma_t and the retained set (frame 1 always kept)
    const double tau = (double)c.tau;
    // each thread owns `per` consecutive frames t0 .. t1 - 1;
    // nf[t] holds the frame's keep flag until the retained list is written
    const int per = (T + (int)blockDim.x - 1) / (int)blockDim.x;
    const int t0 = threadIdx.x * per, t1 = min(T, t0 + per);
    int cnt = 0;
    for (int t = t0; t < t1; ++t) {
        const double d = fr[4 * t + 1];
        const double gm = hi > lo ? (d - lo) / (hi - lo) : 0.0;
        fr[4 * t + 2] = gm;
        fr[4 * t + 3] = NAN;
        if (c.out_rel) {   // r~ follows with the WTA (NaN: filtered)
            float *orl = c.out_rel + (base + t) * 4;
            orl[0] = (float)fr[4 * t];
            orl[1] = (float)d;
            orl[2] = (float)gm;
            orl[3] = NAN;
        }
        const int kp = (t == 0 || d >= tau) ? 1 : 0;
        nf[t] = kp;
        cnt += kp;
    }
    int L = 0;
    int pos = block_excl_scan(cnt, iscr, &L);
    for (int t = t0; t < t1; ++t) {
        if (nf[t]) lst[pos++] = t;
        nf[t] = 0;
    }
    __syncthreads();

    // WTA (Eq. 8-10): DWT of r over the retained sequence with the WTA
    // wavelet (Daubechies p, 2p taps; half-sample symmetric extension, as the
    // WSM's), each detail coefficient k gated by the mean of the extended gate
    // samples 2k and 2k+1, inverse DWT.  For Haar an odd last sample pairs
    // with its mirror image, so its detail is 0 and it passes through.  With
    // J > 1 levels the DWT cascades on the approximation and level j's gate is
    // the same pairwise mean of level j-1's gate; the inverse cascades back.
    // Budget weights are max(r~, 0) (Eq. 5); the ablation modes use max(r, 0)
    // ("raw") or 1 ("uniform") instead.
    const int FT = c.wta_F;
    const int K = (L + FT - 1) / 2;
    for (int k = threadIdx.x; k < K; k += blockDim.x) {
        double ca = 0.0, cd = 0.0;
        for (int j = 0; j < FT; ++j) {
            const double x = fr[4 * lst[ext_index(2 * k + 1 - j, L, WZ_MODE_SYMMETRIC)]];
            ca += c.wta_dec_lo[j] * x;
            cd += c.wta_dec_hi[j] * x;
        }
        const int m0 = ext_index(2 * k, L, WZ_MODE_SYMMETRIC), m1 = ext_index(2 * k + 1, L, WZ_MODE_SYMMETRIC);
        const double g = 0.5 * (fr[4 * lst[m0] + 2] + fr[4 * lst[m1] + 2]);
        A0[k] = ca;
        dall[k] = g * cd;
        if (J > 1) G0[k] = g;
    }
    __syncthreads();
    const double *ain = J > 1 ? wta_deeper_levels(c, A0, A1, G0, G1, dall, K, J) : A0;
    int anypos = 0;
    for (int m = threadIdx.x; m < L; m += blockDim.x) {
        double rt = 0.0;
        const int alo = m >> 1, ahi = min(K - 1, (m + FT - 2) >> 1);
        for (int ai = alo; ai <= ahi; ++ai) {
            const int kk = m + FT - 2 - 2 * ai;       // synthesis tap, 0 <= kk < FT
            rt += c.wta_rec_lo[kk] * ain[ai] + c.wta_rec_hi[kk] * dall[ai];
        }
        const int t = lst[m];
        fr[4 * t + 3] = rt;
        if (c.out_rel) c.out_rel[(base + t) * 4 + 3] = (float)rt;
        const double wv = c.temporal_mode == WZ_TEMPORAL_WTA ? rt
                          : c.temporal_mode == WZ_TEMPORAL_RAW ? fr[4 * t] : 1.0;
        wgt[m] = fmax(wv, 0.0);
        anypos |= (wv > 0.0);
    }
    // uniform weights if none is positive
    anypos = __syncthreads_or(anypos);
    for (int m = threadIdx.x; m < L; m += blockDim.x) {
        nb[m] = -1;
        if (!anypos) wgt[m] = 1.0;
    }
    __syncthreads();

    // Budgets (Eq. 5, Eq. 15): largest-remainder apportionment of B over the
    // weights, frames whose quota exceeds N capped at N and the rest
    // re-apportioned.
    const int N = c.N;
    const int B = vp.B;
    if ((long long)L * N <= (long long)B) {
        for (int m = threadIdx.x; m < L; m += blockDim.x) nb[m] = N;
    } else {
        long long remaining = B;
        for (int round = 0; round <= L; ++round) {
            // candidates: active frames with positive weight, else all active
            double sp = 0.0;
            int npos = 0;
            for (int m = threadIdx.x; m < L; m += blockDim.x)
                if (nb[m] < 0 && wgt[m] > 0.0) {
                    sp += wgt[m];
                    npos = 1;
                }
            npos = __syncthreads_or(npos);
            const bool uniform = (npos == 0);
            double S = 0.0;
            if (uniform) {
                int na = 0;
                for (int m = threadIdx.x; m < L; m += blockDim.x) na += (nb[m] < 0);
                S = (double)block_sum_ll(na, lscr);
            } else {
                S = block_sum(sp, dscr);
            }
            // quota q_m = remaining * w_m / S of every candidate; in the same
            // pass the caps that bind and, for the largest remainder, the
            // floors and the fractional parts (non-negative doubles order like
            // their bit patterns; a candidate's key is its pattern + 1, others
            // 0, so non-candidates rank below every candidate)
            long long ncap = 0, fsum = 0;
            for (int m = threadIdx.x; m < L; m += blockDim.x) {
                const double w = uniform ? 1.0 : wgt[m];
                unsigned long long key = 0ull;
                if (nb[m] < 0 && (uniform || w > 0.0)) {
                    const double q = (double)remaining * w / S;
                    const double fl = floor(q);
                    ncap += (q > (double)N);
                    fsum += (long long)fl;
                    key = (unsigned long long)__double_as_longlong(q - fl) + 1ull;
                    qv[m] = q;
                }
                keys[m] = key;
            }
            block_sum2_ll(ncap, fsum, lscr);
            if (ncap > 0) {
                for (int m = threadIdx.x; m < L; m += blockDim.x)
                    if (keys[m] != 0ull && qv[m] > (double)N) nb[m] = N;
                remaining -= (long long)N * ncap;
                __syncthreads();
                continue;
            }
            const long long R = remaining - fsum;
            const ulonglong2 *k2 = reinterpret_cast<const ulonglong2 *>(keys);
            // rank = #{k : key_k > key_m, or key_k == key_m and k < m}, counted
            // by gs lanes per frame (the largest power of two <= 32 with
            // gs * L <= threads), each over every gs-th pair of keys with
            // broadcast 16-byte reads, summed by shuffles; the floor and the
            // remainder unit together
            int gs = 1;
            while (gs < 32 && 2 * gs * L <= (int)blockDim.x) gs <<= 1;
            const int sl = threadIdx.x & (gs - 1);
            for (int b0 = 0; b0 < L * gs; b0 += blockDim.x) {
                const int m = (b0 + (int)threadIdx.x) / gs;
                const bool on = m < L;
                const unsigned long long km = on ? keys[m] : 0ull;
                int r0 = 0, r1 = 0;
                if (on) {
#pragma unroll 4
                    for (int i = sl; i < (L >> 1); i += gs) {
                        const ulonglong2 p = k2[i];
                        r0 += (p.x > km) | ((p.x == km) & (2 * i < m));
                        r1 += (p.y > km) | ((p.y == km) & (2 * i + 1 < m));
                    }
                    if ((L & 1) && sl == 0) {
                        const unsigned long long p = keys[L - 1];
                        r0 += (p > km) | ((p == km) & (L - 1 < m));
                    }
                }
                int r = r0 + r1;
                for (int o = 1; o < gs; o <<= 1) r += __shfl_xor_sync(0xffffffffu, r, o);
                if (on && sl == 0 && km != 0ull) nb[m] = (int)floor(qv[m]) + (r < R ? 1 : 0);
            }
            __syncthreads();
            break;
        }
        for (int m = threadIdx.x; m < L; m += blockDim.x)
            if (nb[m] < 0) nb[m] = 0;
    }
    __syncthreads();
    // scatter to frames, offsets, grids
    for (int m = threadIdx.x; m < L; m += blockDim.x) nf[lst[m]] = nb[m];
    __syncthreads();
    // per frame: output rows, tensor-core operator rows (budgets padded to
    // 16) and tensor-core units (column blocks of <= 256 tokens, each in
    // groups of unit_tiles(round16(nc)) 128-channel tiles; the spatial kernel
    // writes the unit records); one block scan gives all the offsets.  The
    // units of every frame's first block come first in the video's list, the
    // units of later blocks (frames over 256 tokens; their operator rows
    // reach only part of the map, so they are the short ones) after them:
    // the condensation claims units in list order, and short units last keep
    // its tail short.
    const bool tc = c.path == WZ_PATH_TENSOR;
    // units of frame t's first block (ua) and of its later blocks (ub)
    auto frame_units = [&](int n, int &ua, int &ub) {
        ua = ub = 0;
        if (tc)
            for (int j0 = 0; j0 < n; j0 += kColBlock) {
                const int nc = min(kColBlock, n - j0);
                const int cg = unit_tiles((nc + 15) / 16 * 16), add = (c.n_ct + cg - 1) / cg;
                if (j0 == 0) ua += add;
                else ub += add;
            }
    };
    // this thread's frames t0 .. t1 - 1 (their budgets re-read from shared
    // memory: no per-thread arrays)
    int part[4] = {0, 0, 0, 0};
    for (int t = t0; t < t1; ++t) {
        const int n = nf[t];
        int ua, ub;
        frame_units(n, ua, ub);
        part[0] += n;
        part[1] += (n + 15) & ~15;
        part[2] += ua;
        part[3] += ub;
    }
    int pre[4], tot[4];
    block_excl_scan<4>(part, iscr, pre, tot);
    int o = pre[0], wo = pre[1], u = pre[2], uB = tot[2] + pre[3];
    for (int t = t0; t < t1; ++t) {
        const int n = nf[t];
        int ua, ub;
        frame_units(n, ua, ub);
        c.n[base + t] = n;
        c.off[base + t] = vp.row0 + o;
        c.woff[base + t] = vp.w_row0 + wo;
        if (tc) {
            c.ustart[base + t] = u;
            c.ustartB[base + t] = uB;
        }
        const int h = grid_h(n, c.H, c.W);
        c.hw[2 * (base + t)] = h;
        c.hw[2 * (base + t) + 1] = h > 0 ? (n + h - 1) / h : 0;
        if (c.out_budgets) c.out_budgets[base + t] = n;
        o += n;
        wo += (n + 15) & ~15;
        u += ua;
        uB += ub;
    }
    if (threadIdx.x == 0) {
        c.prod[v] = tot[0];
        if (c.out_count) c.out_count[v] = tot[0];
        if (tc) {
            c.ucount[v] = min(tot[2] + tot[3], c.max_units_v);
            if (tot[2] + tot[3] > c.max_units_v) atomicOr(c.status, 2);
        }
    }
}

cudaError_t launch_temporal(const Ctx &c, cudaStream_t s) {
    const size_t smem = temporal_smem_bytes(c.T, c.wta_levels);
    cudaError_t e = cudaFuncSetAttribute(temporal_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    void *args[] = {const_cast<Ctx *>(&c)};
    return launch_kernel((const void *)temporal_kernel, dim3(c.V + 1), dim3(temporal_threads(c.T)), smem, s, args,
                         c.pdl != 0);
}

}  // namespace wz
