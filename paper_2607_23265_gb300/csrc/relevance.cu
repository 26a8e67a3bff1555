// Cross-Modal Scorer, similarity branch (Section 3.2.1), on the GPU.
//
//   query_pool      u_q = mean of the query rows (fp64) and ||u_q||.
//   relevance_pass  one streaming read of the features: per token
//                   a_{t,n} = <u, u_q> / (||u|| ||u_q||) (the input of Eq. 6)
//                   and per-CTA column sums of every frame it touches (the
//                   average pool of Section 3.2.1 / Eq. 7), in fp32.
//   frame_stats     sums the column partials of a frame in fp64 in a fixed
//                   order and reduces <v_t,u_q>, <v_t,v_t>, <v_t,v_{t-1}> per
//                   256-channel chunk, which give r_t and delta_t (Eq. 7).
//
// The relevance pass is HBM bound: it reads T*H*W*D elements once with
// 16-byte non-allocating loads; each CTA owns one contiguous range of the
// flattened token index so the grid is exactly balanced.
#include <algorithm>
#include <cstring>

#include "wz_internal.cuh"

namespace wz {

struct VideoParBlock {
    VideoPar v[WZ_MAX_VIDEOS];
};

template <typename T>
__global__ void __launch_bounds__(1024) query_pool_kernel(Ctx c, VideoParBlock par) {
    __shared__ double scratch[32];
    const int v = blockIdx.x;
    const VideoPar vp = par.v[v];
    if (threadIdx.x == 0) c.vpar[v] = vp;
    const T *Q = static_cast<const T *>(c.Q) + (size_t)vp.q_row0 * c.D;
    double ss = 0.0;
    for (int d = threadIdx.x; d < c.D; d += blockDim.x) {
        double s = 0.0;
        for (int j = 0; j < vp.Lq; ++j) s += (double)load_scalar<T>(Q + (size_t)j * c.D + d);
        s /= (double)vp.Lq;
        c.qbar64[(size_t)v * c.D + d] = s;
        c.qbar32[(size_t)v * c.D + d] = (float)s;
        ss += s * s;
    }
    const double tot = block_sum(ss, scratch);
    if (threadIdx.x == 0) c.qnorm[v] = sqrt(tot);
}

// Reduce the NV values held by every lane across the warp (NV a power of
// two <= 32).  Each of the first log2(NV) steps halves the values a lane
// keeps; the remaining steps are plain butterflies.  On return lane l holds
// the warp total of value l >> (5 - log2(NV)).
template <int NV>
__device__ __forceinline__ float transpose_reduce(float (&v)[NV]) {
    const int lane = threadIdx.x & 31;
    int half = NV / 2;
    int o = 16;
#pragma unroll
    for (; half >= 1; half >>= 1, o >>= 1) {
        const bool upper = (lane & o) != 0;
#pragma unroll
        for (int i = 0; i < half; ++i) {
            const float keep = upper ? v[i + half] : v[i];
            const float send = upper ? v[i] : v[i + half];
            v[i] = keep + __shfl_xor_sync(0xffffffffu, send, o);
        }
    }
    float r = v[0];
#pragma unroll
    for (; o >= 1; o >>= 1) r += __shfl_xor_sync(0xffffffffu, r, o);
    return r;
}

// One CTA streams tokens [blockIdx.x*L1, +L1) of the flattened [V*T*N] index.
template <typename T, int VPT>
__global__ void __launch_bounds__(256) relevance_pass_kernel(Ctx c) {
    constexpr int VEC = VecOf<T>::kElems;
    constexpr int GROUP = VPT >= 8 ? 1 : 8 / VPT;   // tokens per reduction step
    constexpr int NV = 2 * GROUP;                   // GROUP dots + GROUP norms
    constexpr int SHIFT = NV == 16 ? 1 : NV == 8 ? 2 : NV == 4 ? 3 : 4;
    __shared__ float red[2][8][NV];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int nw = blockDim.x >> 5;
    const int n_vec = c.D / VEC;
    const int64_t total = (int64_t)c.V * c.T * c.N;
    const int64_t start = (int64_t)blockIdx.x * c.L1;
    const int64_t end = min(start + c.L1, total);
    const uint4 *X = static_cast<const uint4 *>(c.X);
    int cur_v = -1;
    float q[VPT][VEC];
    float qn = 0.f;
    int gi = 0;
    for (int64_t tok = start; tok < end;) {
        const int64_t f = tok / c.N;
        const int64_t seg_end = min(end, (f + 1) * (int64_t)c.N);
        const int v = (int)(f / c.T);
        if (v != cur_v) {
            cur_v = v;
            qn = (float)c.qnorm[v];
#pragma unroll
            for (int vi = 0; vi < VPT; ++vi) {
                const int vidx = threadIdx.x + vi * blockDim.x;
#pragma unroll
                for (int e = 0; e < VEC; ++e)
                    q[vi][e] = vidx < n_vec ? c.qbar32[(size_t)v * c.D + vidx * VEC + e] : 0.f;
            }
        }
        float cs[VPT][VEC];
#pragma unroll
        for (int vi = 0; vi < VPT; ++vi)
#pragma unroll
            for (int e = 0; e < VEC; ++e) cs[vi][e] = 0.f;

        for (int64_t g0 = tok; g0 < seg_end; g0 += GROUP, ++gi) {
            uint4 raw[GROUP][VPT];
#pragma unroll
            for (int k = 0; k < GROUP; ++k)
#pragma unroll
                for (int vi = 0; vi < VPT; ++vi) {
                    const int vidx = threadIdx.x + vi * blockDim.x;
                    if (g0 + k < seg_end && vidx < n_vec)
                        raw[k][vi] = ldg_stream(X + (size_t)(g0 + k) * n_vec + vidx);
                    else
                        raw[k][vi] = make_uint4(0u, 0u, 0u, 0u);
                }
            float acc[NV];
#pragma unroll
            for (int k = 0; k < NV; ++k) acc[k] = 0.f;
#pragma unroll
            for (int k = 0; k < GROUP; ++k)
#pragma unroll
                for (int vi = 0; vi < VPT; ++vi) {
                    float x[VEC];
                    unpack(raw[k][vi], x, (T *)nullptr);
#pragma unroll
                    for (int e = 0; e < VEC; ++e) {
                        cs[vi][e] += x[e];
                        acc[k] = fmaf(x[e], q[vi][e], acc[k]);
                        acc[k + GROUP] = fmaf(x[e], x[e], acc[k + GROUP]);
                    }
                }
            const float tot = transpose_reduce<NV>(acc);
            const int b = gi & 1;
            if ((lane & ((1 << SHIFT) - 1)) == 0) red[b][warp][lane >> SHIFT] = tot;
            __syncthreads();
            if (threadIdx.x < 32) {
                float s = 0.f;
                if (lane < NV)
                    for (int w = 0; w < nw; ++w) s += red[b][w][lane];
                const float nrm = __shfl_down_sync(0xffffffffu, s, GROUP);
                if (lane < GROUP && g0 + lane < seg_end) {
                    const float a = (nrm > 0.f && qn > 0.f) ? s / (sqrtf(nrm) * qn) : 0.f;
                    c.a[g0 + lane] = a;
                }
            }
        }
        // column partial of frame f from this CTA: slot blockIdx.x + f
        float *dst = c.part + ((size_t)blockIdx.x + (size_t)f) * c.D;
#pragma unroll
        for (int vi = 0; vi < VPT; ++vi) {
            const int vidx = threadIdx.x + vi * blockDim.x;
            if (vidx < n_vec) {
#pragma unroll
                for (int e = 0; e < VEC; e += 4)
                    *reinterpret_cast<float4 *>(dst + vidx * VEC + e) =
                        make_float4(cs[vi][e], cs[vi][e + 1], cs[vi][e + 2], cs[vi][e + 3]);
            }
        }
        tok = seg_end;
    }
}

// Per (256-channel chunk, frame): fp64 frame sums from the fixed list of CTA
// partials, and their products with u_q and with the previous frame.
__global__ void __launch_bounds__(kStatsChunk) frame_stats_kernel(Ctx c) {
    __shared__ double scratch[32];
    const int64_t f = blockIdx.y;
    const int t = (int)(f % c.T);
    const int v = (int)(f / c.T);
    const int d = blockIdx.x * kStatsChunk + threadIdx.x;
    double sf = 0.0, sp = 0.0, q = 0.0;
    if (d < c.D) {
        const int64_t lo = f * c.N / c.L1;
        const int64_t hi = min((int64_t)c.G1 - 1, ((f + 1) * c.N - 1) / c.L1);
        for (int64_t cc = lo; cc <= hi; ++cc) sf += (double)c.part[(size_t)(cc + f) * c.D + d];
        if (t > 0) {
            const int64_t g = f - 1;
            const int64_t lo2 = g * c.N / c.L1;
            const int64_t hi2 = min((int64_t)c.G1 - 1, ((g + 1) * c.N - 1) / c.L1);
            for (int64_t cc = lo2; cc <= hi2; ++cc) sp += (double)c.part[(size_t)(cc + g) * c.D + d];
        }
        q = c.qbar64[(size_t)v * c.D + d];
        if (c.frame_mean) c.frame_mean[(size_t)f * c.D + d] = (float)(sf / c.N);
    }
    const double s0 = block_sum(sf * q, scratch);
    const double s1 = block_sum(sf * sf, scratch);
    const double s2 = block_sum(sf * sp, scratch);
    if (threadIdx.x == 0) {
        double *o = c.trip + ((size_t)f * c.DC + blockIdx.x) * 3;
        o[0] = s0;
        o[1] = s1;
        o[2] = s2;
    }
}

// r_t only (the relevance entry point); the condensation pass does this in
// the temporal kernel.
__global__ void relevance_finalize_kernel(Ctx c) {
    const int64_t f = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (f >= (int64_t)c.V * c.T) return;
    const int v = (int)(f / c.T);
    double dq = 0.0, ff = 0.0;
    for (int k = 0; k < c.DC; ++k) {
        dq += c.trip[((size_t)f * c.DC + k) * 3 + 0];
        ff += c.trip[((size_t)f * c.DC + k) * 3 + 1];
    }
    const double qn = c.qnorm[v];
    c.frame_scores[f] = (ff > 0.0 && qn > 0.0) ? (float)(dq / (sqrt(ff) * qn)) : 0.f;
}

cudaError_t launch_query_pool(const Ctx &c, const VideoPar *hpar, cudaStream_t s) {
    VideoParBlock blk;   // copied into the launch parameters
    memset(&blk, 0, sizeof(blk));
    for (int v = 0; v < c.V; ++v) blk.v[v] = hpar[v];
    if (c.dtype == WZ_DTYPE_BF16)
        query_pool_kernel<__nv_bfloat16><<<c.V, 1024, 0, s>>>(c, blk);
    else
        query_pool_kernel<float><<<c.V, 1024, 0, s>>>(c, blk);
    return cudaGetLastError();
}

namespace {

template <typename T, int VPT>
void relevance_config(const Ctx &c, const void *&fn, int &threads) {
    fn = (const void *)relevance_pass_kernel<T, VPT>;
    constexpr int VEC = VecOf<T>::kElems;
    const int n_vec = c.D / VEC;
    threads = ((n_vec + VPT - 1) / VPT + 31) / 32 * 32;
    if (threads < 32) threads = 32;
}

template <typename T>
bool pick(const Ctx &c, const void *&fn, int &threads) {
    constexpr int VEC = VecOf<T>::kElems;
    const int n_vec = c.D / VEC;
    if (n_vec <= 256) relevance_config<T, 1>(c, fn, threads);
    else if (n_vec <= 512) relevance_config<T, 2>(c, fn, threads);
    else if (n_vec <= 1024) relevance_config<T, 4>(c, fn, threads);
    else if (n_vec <= 2048) relevance_config<T, 8>(c, fn, threads);
    else return false;
    return true;
}

bool pick_any(const Ctx &c, const void *&fn, int &threads) {
    return c.dtype == WZ_DTYPE_BF16 ? pick<__nv_bfloat16>(c, fn, threads) : pick<float>(c, fn, threads);
}

}  // namespace

int relevance_grid(const Ctx &c) {
    const void *fn = nullptr;
    int threads = 0;
    if (!pick_any(c, fn, threads)) return 0;
    int dev = 0, sms = 0, per_sm = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, threads, 0) != cudaSuccess) return 0;
    if (per_sm < 1) per_sm = 1;
    const int64_t total = (int64_t)c.V * c.T * c.N;
    int64_t g = (int64_t)sms * per_sm;
    const int64_t min_tokens = 16;
    g = std::min<int64_t>(g, (total + min_tokens - 1) / min_tokens);
    g = std::min<int64_t>(g, kG1Max);
    return (int)std::max<int64_t>(g, 1);
}

cudaError_t launch_relevance_pass(const Ctx &c, cudaStream_t s) {
    const void *fn = nullptr;
    int threads = 0;
    if (!pick_any(c, fn, threads)) return cudaErrorInvalidValue;
    void *args[] = {const_cast<Ctx *>(&c)};
    return cudaLaunchKernel(fn, dim3(c.G1), dim3(threads), args, 0, s);
}

cudaError_t launch_frame_stats(const Ctx &c, cudaStream_t s) {
    frame_stats_kernel<<<dim3(c.DC, c.V * c.T), kStatsChunk, 0, s>>>(c);
    return cudaGetLastError();
}

cudaError_t launch_relevance_finalize(const Ctx &c, cudaStream_t s) {
    const int n = c.V * c.T;
    relevance_finalize_kernel<<<(n + 255) / 256, 256, 0, s>>>(c);
    return cudaGetLastError();
}

}  // namespace wz
