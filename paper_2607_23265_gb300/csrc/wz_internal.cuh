// Internal declarations of the WaveZip CUDA library (not part of the C ABI).
#pragma once

#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include "../../include/wavezip.h"

namespace wz {

constexpr int kMaxTaps = 20;          // Daubechies order <= 10
constexpr int kMaxLevels = WZ_MAX_LEVELS;   // decomposition levels of the WTA / WSM
constexpr int kG1Max = 2048;          // relevance-pass CTAs (upper bound)
constexpr int kColBlock = 256;        // output tokens per tensor-core unit
constexpr int kUnitRanged = 1 << 28;  // unit record flag: per-chunk operator row ranges in Ctx::krange
constexpr int kTileC = 128;           // channels per tensor-core M tile
constexpr int kTmemCols = 512;        // tensor-memory columns of one condensation CTA

// Per-video parameters written to the workspace by the query-pool kernel.
struct VideoPar {
    int q_row0;    // first query row of the video
    int Lq;        // query rows
    int B;         // global budget of the video
    int row0;      // first output row of the video
    int w_row0;    // first tensor-core operator row of the video (multiple of 16)
};

// Everything a kernel of one call needs: sizes, inputs, workspace views,
// outputs and scalar parameters.  Passed by value.
struct Ctx {
    int V, T, H, W, D, N;
    int dtype;            // WZ_DTYPE_*
    int hp, wp;           // WSM subband sizes
    int K_pad;            // N rounded up to 32 (row length of the operator)
    int G1;               // relevance CTAs actually launched
    int n_ct;             // 128-channel tiles
    int max_units_v;      // unit-list capacity per video
    int F;                // WSM filter taps
    int64_t L1;           // tokens per relevance CTA
    int64_t rows_total;   // sum of budgets over videos (output rows)
    int64_t w_rows;       // operator rows of the tensor-core layout (frames padded to 16)

    const void *X;
    const void *Q;

    float *qbar32;        // [V][D]
    double *qbar64;       // [V][D]
    VideoPar *vpar;       // [V]
    float *a;             // [V*T][N] token saliency
    float *part;          // [G1 + V*T][D] column-sum partials
    double *fr;           // [V*T][4] (r, delta, gamma, r~); r, delta from frame_stats
    int *list;            // [V][2T] retained frames and their budgets
    int *n;               // [V*T] budgets
    int *off;             // [V*T] global output row of the frame's first token
    int *woff;            // [V*T] first tensor-core operator row of the frame
    int *hw;              // [V*T][2] condensation grid
    int *prod;            // [V] produced rows
    int4 *units;          // [V][max_units_v] tensor-core work units
    int *ucount;          // [V]
    int *ustart;          // [V*T] first unit of each frame's first block in its video's list
    int *ustartB;         // [V*T] first unit of the frame's later blocks (after every first block)
    float *stab;          // frame-independent tables of the spatial operator
    unsigned long long *drange;   // [V][2] min / max of delta_t as bit patterns (delta >= +0)
    float *gate;          // [V*T][hp*wp] gate G of each frame (Eq. 12)
    void *Wop;            // operator: tensor path bf16 hi then lo in the tiled
                          // layout of tile_index(), CUDA-core path f32 [rows][K_pad]
    uint16_t *krange;     // [V*T][krange_nblk][K_pad/32] operator rows of a 256-token block that
                          // reach a 32-token chunk: [16*(r & 0xff), 16*(r >> 8)) (tensor path)
    int krange_nblk;      // blocks of 256 tokens per frame: ceil(H*W / 256)
    int *status;          // device status word (bounded waits)
    int *spatial_next;    // [0]: next (frame, grid row) of the spatial operator kernel, [1]: next
                          // tensor-core unit of the condensation; both zeroed by temporal

    void *out;            // [rows][D] dtype
    int *out_index;       // [rows][3]
    int *out_budgets;     // [V*T] or null
    int *out_count;       // [V] or null
    float *out_rel;       // [V*T][4] or null
    float *frame_mean;    // [V*T][D] or null (relevance entry point)
    float *frame_scores;  // [V*T] or null (relevance entry point)

    float lambda, tau;
    int mode;             // WZ_MODE_*
    int path;             // resolved WZ_PATH_TENSOR or WZ_PATH_SIMT
    int temporal_mode;    // WZ_TEMPORAL_*
    int spatial_mode;     // WZ_SPATIAL_*
    const float *ext_a;   // [V*T][N] external token scores, or null
    const float *ext_r;   // [V*T] external frame scores, or null
    int relevance_mode;   // WZ_RELEVANCE_*
    float *qnorm;         // [V][WZ_MAX_LQ_MAXSIM] query row norms (max-over-query scorer)
    __nv_bfloat16 *qhl;   // [2 WZ_MAX_LQ_MAXSIM][D] normalised rows, bf16 hi then lo (one video at a time)
    int wta_levels;       // WTA decomposition levels (1 = the paper's single level)
    int wsm_levels;       // WSM decomposition levels
    int gate_stride;      // floats of c.gate per frame: sum over levels of lvl_h * lvl_w
    int lvl_h[kMaxLevels + 1], lvl_w[kMaxLevels + 1];   // WSM subband grid of level l (l = 0: H x W)
    int goff[kMaxLevels]; // offset of level l+1's gate within a frame's gate
    int pdl;              // host: launch with programmatic stream serialization
    float dec_lo[kMaxTaps], dec_hi[kMaxTaps], rec_lo[kMaxTaps], rec_hi[kMaxTaps];
    int wta_F;            // WTA filter taps (temporal DWT, fp64)
    double wta_dec_lo[kMaxTaps], wta_dec_hi[kMaxTaps], wta_rec_lo[kMaxTaps], wta_rec_hi[kMaxTaps];
};

// ---- device helpers -------------------------------------------------------

// Index checks of the bounds-checked build (WZ_CHECKED): a write whose index
// is out of range records WZ_STATUS_BOUNDS in the status word and is skipped.
// In the normal build the check is a constant true and costs nothing.
__device__ __forceinline__ bool wz_in_range(const int *status, bool ok) {
#ifdef WZ_CHECKED
    if (!ok) atomicOr(const_cast<int *>(status), WZ_STATUS_BOUNDS);
    return ok;
#else
    (void)status;
    (void)ok;
    return true;
#endif
}

// ---- programmatic dependent launch ---------------------------------------
// Each kernel of the pass waits for the grid before it in the stream before it
// touches global memory and then lets the next grid be scheduled, so launch
// latency and prologues overlap the previous kernel's tail.  Launched without
// the attribute, both instructions return at once.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

inline cudaError_t launch_kernel(const void *fn, dim3 grid, dim3 block, size_t smem, cudaStream_t s, void **args,
                                 bool pdl) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelExC(&cfg, fn, args);
}

__device__ __forceinline__ int ext_index(int i, int n, int mode) {
    if (i >= 0 && i < n) return i;
    if (mode == WZ_MODE_ZERO) return -1;
    if (mode == WZ_MODE_PERIODIC) {
        int k = i % n;
        return k < 0 ? k + n : k;
    }
    int p = 2 * n;
    int k = i % p;
    if (k < 0) k += p;
    return k < n ? k : p - 1 - k;
}

__device__ __forceinline__ float bf16_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t v) { return __uint_as_float(v & 0xffff0000u); }

template <typename T> struct VecOf;
template <> struct VecOf<__nv_bfloat16> { static constexpr int kElems = 8; };
template <> struct VecOf<float> { static constexpr int kElems = 4; };

// Unpack a 16-byte vector into floats.
__device__ __forceinline__ void unpack(const uint4 &v, float (&f)[8], __nv_bfloat16 *) {
    f[0] = bf16_lo(v.x); f[1] = bf16_hi(v.x);
    f[2] = bf16_lo(v.y); f[3] = bf16_hi(v.y);
    f[4] = bf16_lo(v.z); f[5] = bf16_hi(v.z);
    f[6] = bf16_lo(v.w); f[7] = bf16_hi(v.w);
}
__device__ __forceinline__ void unpack(const uint4 &v, float (&f)[4], float *) {
    f[0] = __uint_as_float(v.x); f[1] = __uint_as_float(v.y);
    f[2] = __uint_as_float(v.z); f[3] = __uint_as_float(v.w);
}

__device__ __forceinline__ uint4 ldg_stream(const uint4 *p) {
    uint4 r;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w) : "l"(p));
    return r;
}

template <typename T>
__device__ __forceinline__ float load_scalar(const T *p);
template <> __device__ __forceinline__ float load_scalar<float>(const float *p) { return *p; }
template <> __device__ __forceinline__ float load_scalar<__nv_bfloat16>(const __nv_bfloat16 *p) {
    return __bfloat162float(*p);
}

template <typename T>
__device__ __forceinline__ T from_float(float v);
template <> __device__ __forceinline__ float from_float<float>(float v) { return v; }
template <> __device__ __forceinline__ __nv_bfloat16 from_float<__nv_bfloat16>(float v) {
    return __float2bfloat16_rn(v);
}

// Block-wide sum of a double in a fixed order (deterministic for a fixed
// block size): warp trees, then one warp reduces the warp totals.
// `scratch` holds >= 33 doubles; all threads receive the sum.
__device__ __forceinline__ double block_sum(double v, double *scratch) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int nw = (blockDim.x + 31) >> 5;
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    __syncthreads();
    if (lane == 0) scratch[warp] = v;
    __syncthreads();
    if (warp == 0) {
        double s = lane < nw ? scratch[lane] : 0.0;
        for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
        if (lane == 0) scratch[32] = s;
    }
    __syncthreads();
    return scratch[32];
}

__device__ __forceinline__ long long block_sum_ll(long long v, long long *scratch) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int nw = (blockDim.x + 31) >> 5;
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    __syncthreads();
    if (lane == 0) scratch[warp] = v;
    __syncthreads();
    if (warp == 0) {
        long long s = lane < nw ? scratch[lane] : 0;
        for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
        if (lane == 0) scratch[32] = s;
    }
    __syncthreads();
    return scratch[32];
}

// Two block-wide sums of long longs at once; `scratch` holds >= 66 values;
// all threads receive both sums in place.
__device__ __forceinline__ void block_sum2_ll(long long &a, long long &b, long long *scratch) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int nw = (blockDim.x + 31) >> 5;
    for (int o = 16; o > 0; o >>= 1) {
        a += __shfl_xor_sync(0xffffffffu, a, o);
        b += __shfl_xor_sync(0xffffffffu, b, o);
    }
    __syncthreads();
    if (lane == 0) {
        scratch[warp] = a;
        scratch[33 + warp] = b;
    }
    __syncthreads();
    if (warp == 0) {
        long long s = lane < nw ? scratch[lane] : 0, t = lane < nw ? scratch[33 + lane] : 0;
        for (int o = 16; o > 0; o >>= 1) {
            s += __shfl_xor_sync(0xffffffffu, s, o);
            t += __shfl_xor_sync(0xffffffffu, t, o);
        }
        if (lane == 0) {
            scratch[32] = s;
            scratch[65] = t;
        }
    }
    __syncthreads();
    a = scratch[32];
    b = scratch[65];
}

// ---- packed fp32 pairs (f32x2 instructions of sm_100-class GPUs) ----------

typedef unsigned long long f2_t;

__device__ __forceinline__ f2_t pack2(float lo, float hi) {
    f2_t r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
    return r;
}

__device__ __forceinline__ float2 unpack2(f2_t v) {
    float2 r;
    asm("mov.b64 {%0, %1}, %2;" : "=f"(r.x), "=f"(r.y) : "l"(v));
    return r;
}

__device__ __forceinline__ f2_t fma2(f2_t a, f2_t b, f2_t c) {
    f2_t d;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
    return d;
}

__device__ __forceinline__ f2_t add2(f2_t a, f2_t b) {
    f2_t d;
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
    return d;
}

// A 16-byte vector as VEC/2 packed pairs of consecutive elements.
__device__ __forceinline__ void unpack_pairs(const uint4 &v, f2_t (&p)[4], __nv_bfloat16 *) {
    p[0] = pack2(bf16_lo(v.x), bf16_hi(v.x));
    p[1] = pack2(bf16_lo(v.y), bf16_hi(v.y));
    p[2] = pack2(bf16_lo(v.z), bf16_hi(v.z));
    p[3] = pack2(bf16_lo(v.w), bf16_hi(v.w));
}
__device__ __forceinline__ void unpack_pairs(const uint4 &v, f2_t (&p)[2], float *) {
    p[0] = pack2(__uint_as_float(v.x), __uint_as_float(v.y));
    p[1] = pack2(__uint_as_float(v.z), __uint_as_float(v.w));
}

// Error-free sum of two floats (Knuth's TwoSum): a + b = s + e exactly.
__device__ __forceinline__ void two_sum(float a, float b, float &s, float &e) {
    s = a + b;
    const float bb = s - a;
    e = (a - (s - bb)) + (b - bb);
}

// Element index of operator entry (row r, column k) in the tensor-core
// layout: 8 x 8 core matrices (8 rows of 8 bf16 = 16 bytes), ordered by
// 32-column K chunk, then 8-row group, then the four 8-column quarters of the
// chunk.  The rows [r0, r0 + n) of one K chunk (r0, n multiples of 8) are
// therefore one contiguous block that a single bulk copy moves into shared
// memory, where it is the canonical no-swizzle K-major operand of tcgen05.mma.
__host__ __device__ __forceinline__ size_t tile_index(int64_t r, int k, int64_t w_rows) {
    return ((((size_t)(k >> 5) * (size_t)(w_rows >> 3) + (size_t)(r >> 3)) * 4 + ((k >> 3) & 3)) * 64) +
           (size_t)(r & 7) * 8 + (size_t)(k & 7);
}

// Channel tiles per tensor-core work unit for a column block of ncp (padded)
// output tokens.  Up to 128 tokens, hi and lo are one MMA of N = 2*ncp and
// take 2*ncp accumulator columns per tile; above, they accumulate into the
// same ncp columns.  Either way a unit fits one 256-column buffer.
// Subband length after l cascaded levels of an F-tap DWT: n_l = (n_{l-1} + F - 1) / 2.
__host__ __device__ __forceinline__ int level_size(int n, int F, int l) {
    for (int k = 0; k < l; ++k) n = (n + F - 1) / 2;
    return n;
}

// Floats of one frame's WSM gates over J levels (level l: h_l x w_l).
__host__ __device__ __forceinline__ int gate_floats(int H, int W, int F, int J) {
    int s = 0;
    for (int l = 1; l <= J; ++l) s += level_size(H, F, l) * level_size(W, F, l);
    return s;
}

// Tensor-core unit shape for a block of ncp (a multiple of 16, <= 256)
// output tokens: the hi and lo operator halves form one MMA of N = 2 ncp for
// ncp <= 64, else two MMAs of N = ncp; a unit spans as many 128-channel tiles
// (at most 4) as the 512 accumulator columns of tensor memory hold, so each
// operator tile in shared memory serves 2-4 channel tiles.
__host__ __device__ __forceinline__ bool unit_fused(int ncp) { return ncp <= 64; }

__host__ __device__ __forceinline__ int unit_tiles(int ncp) {
    const int cols = unit_fused(ncp) ? 2 * ncp : ncp;
    const int cg = 512 / cols;
    return cg < 1 ? 1 : (cg > 4 ? 4 : cg);
}

// ---- launchers (one per kernel family) -------------------------------------

cudaError_t launch_query_pool(const Ctx &c, const VideoPar *hpar, cudaStream_t s);
cudaError_t launch_relevance_pass(const Ctx &c, cudaStream_t s);
cudaError_t launch_frame_stats(const Ctx &c, cudaStream_t s);
cudaError_t launch_temporal(const Ctx &c, cudaStream_t s);
cudaError_t launch_spatial(const Ctx &c, cudaStream_t s);
cudaError_t launch_spatial_tc(const Ctx &c, cudaStream_t s, bool *launched);
// cuTensorMapEncodeTiled from the driver (resolved once; null when missing).
PFN_cuTensorMapEncodeTiled_v12000 tmap_encode_fn();
cudaError_t launch_spatial_ml(const Ctx &c, cudaStream_t s);
size_t spatial_ml_smem_bytes(int H, int W, int F, int J);   // 0 if the layout does not fit
cudaError_t launch_project_gemm(const void *A, int M, int K, const void *B, int N, const float *bias, void *out,
                                bool gelu, int *status, bool pdl, cudaStream_t s);
// Max-over-query relevance of one video in one pass over the features
// (maxsim.cu): token norms, channel-sum partials and a_{t,n}, in place of the
// relevance pass and the max-over-query GEMM.
bool maxsim_pass_supported(const Ctx &c, int Lqp);
cudaError_t launch_maxsim_pass(const Ctx &c, int Lq, int Lqp, cudaStream_t s);
cudaError_t launch_maxsim_gemm(const void *X, int M, int K, const void *QHL, int Lq, int Lqp, float *a, int *status,
                               bool pdl, cudaStream_t s);
cudaError_t launch_query_rows(const Ctx &c, int v, int q_row0, int Lq, int Lqp, cudaStream_t s);
cudaError_t launch_condense_simt(const Ctx &c, cudaStream_t s);
cudaError_t launch_condense_tc(const Ctx &c, cudaStream_t s);
int relevance_grid(const Ctx &c);   // CTAs for the relevance pass on this device

cudaError_t launch_dwt1d(const float *x, int rows, int L, int F, int mode, const float *dlo,
                         const float *dhi, float *cA, float *cD, cudaStream_t s);
cudaError_t launch_idwt1d(const float *cA, const float *cD, int rows, int L, int F,
                          const float *rlo, const float *rhi, float *x, cudaStream_t s);
cudaError_t launch_dwt2d(const void *X, int dtype, int T, int H, int W, int D, int F, int mode,
                         const float *dlo, const float *dhi, float *LL, float *LH, float *HL,
                         float *HH, cudaStream_t s);
cudaError_t launch_idwt2d(const float *LL, const float *LH, const float *HL, const float *HH,
                          int T, int H, int W, int D, int F, const float *rlo, const float *rhi,
                          float *out, cudaStream_t s);

// Host: Daubechies filter bank of order p (2p taps); false if p is out of range.
bool daubechies(int p, double *dec_lo, double *dec_hi, double *rec_lo, double *rec_hi);
bool bior44(double *dec_lo, double *dec_hi, double *rec_lo, double *rec_hi);
int wavelet_taps(int wavelet);   // 2p for db<p>, 10 for bior4.4, 0 if unsupported
bool wavelet_bank(int wavelet, double *dec_lo, double *dec_hi, double *rec_lo, double *rec_hi);

}  // namespace wz
