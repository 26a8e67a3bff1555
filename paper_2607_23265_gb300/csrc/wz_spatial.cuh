// Shared-memory layout of the spatial-operator CTA and the frame-independent
// tables it starts from (Eq. 11-14): the db analysis matrices along height
// and width with the boundary extension folded in, and the rows of the width
// analysis that reach each column.  The tables depend only on (H, W, filter, extension); one CTA builds
// them per pass into global memory with the same layout as the head of the
// shared-memory block, so each spatial CTA copies them in one loop.
#pragma once

#include "wz_internal.cuh"

namespace wz {

constexpr int kStageFloats = 8 * 1024;   // staged operator rows (32 KB)

struct SpatialSmem {
    int N, hp, wp, H, W, HP4, K_pad, QB;
    // float offsets; [0, tables) is the frame-independent part
    int AHl, AHh, AWl, AWh, blo, bhi, tables;
    int G, PAl, PAh, Yl, Yh, Ql, Qh, red, qlo, qhi, M, stage, total;
    // Every table starts on a 16-byte boundary (float4 reads of Y, staged rows).
    __host__ __device__ void init(int H_, int W_, int hp_, int wp_) {
        H = H_; W = W_; hp = hp_; wp = wp_; N = H * W;
        K_pad = (N + 31) & ~31;
        QB = kStageFloats / K_pad;                 // rows staged at a time (>= 2 for N <= 4096)
        HP4 = (H + 3) & ~3;
        int o = 0;
        auto take = [&](int n) {
            const int at = o;
            o = (o + n + 3) & ~3;
            return at;
        };
        AHl = take(hp * H);
        AHh = take(hp * H);
        AWl = take(wp * W);
        AWh = take(wp * W);
        blo = take(W);
        bhi = take(W);
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
        stage = take(QB * K_pad);
        total = o;
    }
};

// Bytes of the frame-independent tables for an image of H x W and F taps.
inline size_t spatial_table_bytes(int H, int W, int F) {
    SpatialSmem L;
    L.init(H, W, (H + F - 1) / 2, (W + F - 1) / 2);
    return (size_t)L.tables * 4;
}

// Build the tables into c.stab (one CTA, any size).
//   A[a][i] = sum_j dec[j] [ext(2a + 1 - j) == i]   (analysis along a side)
//   blo/bhi[j] = first / last row b of A' with A'[b][j] != 0 (shared-memory
//                atomics while A' is formed)
__device__ inline void build_spatial_tables(const Ctx &c) {
    SpatialSmem L;
    L.init(c.H, c.W, c.hp, c.wp);
    float *tb = c.stab;
    int *ti = reinterpret_cast<int *>(c.stab);
    const int H = c.H, W = c.W, hp = c.hp, wp = c.wp, F = c.F;
    for (int k = threadIdx.x; k < hp * H; k += blockDim.x) {
        const int a = k / H, i = k % H;
        float sl = 0.f, sh = 0.f;
        for (int j = 0; j < F; ++j)
            if (ext_index(2 * a + 1 - j, H, c.mode) == i) {
                sl += c.dec_lo[j];
                sh += c.dec_hi[j];
            }
        tb[L.AHl + k] = sl;
        tb[L.AHh + k] = sh;
    }
    __shared__ int s_blo[WZ_MAX_HW], s_bhi[WZ_MAX_HW];
    for (int j = threadIdx.x; j < W; j += blockDim.x) {
        s_blo[j] = wp;
        s_bhi[j] = -1;
    }
    __syncthreads();
    for (int k = threadIdx.x; k < wp * W; k += blockDim.x) {
        const int b = k / W, i = k % W;
        float sl = 0.f, sh = 0.f;
        for (int j = 0; j < F; ++j)
            if (ext_index(2 * b + 1 - j, W, c.mode) == i) {
                sl += c.dec_lo[j];
                sh += c.dec_hi[j];
            }
        tb[L.AWl + k] = sl;
        tb[L.AWh + k] = sh;
        if (sl != 0.f || sh != 0.f) {
            atomicMin(&s_blo[i], b);
            atomicMax(&s_bhi[i], b);
        }
    }
    __syncthreads();
    for (int j = threadIdx.x; j < W; j += blockDim.x) {
        ti[L.blo + j] = s_blo[j];
        ti[L.bhi + j] = s_bhi[j];
    }
}

}  // namespace wz
