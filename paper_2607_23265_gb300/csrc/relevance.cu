// Cross-Modal Scorer, similarity branch (Section 3.2.1), on the GPU.
//
//   query_pool      u_q = mean of the query rows (compensated fp32 -> fp64).
//   relevance_pass  one streaming read of the features: per token
//                   a_{t,n} = <u, u_q> / (||u|| ||u_q||) (the input of Eq. 6)
//                   and per-CTA column sums of every frame it touches (the
//                   average pool of Section 3.2.1 / Eq. 7), in fp32.
//   frame_stats     sums the column partials of a frame in fp64 in a fixed
//                   order and reduces <v_t,u_q>, <v_t,v_t>, <v_t,v_{t-1}> and
//                   <u_q,u_q> per 2048-channel chunk, which give r_t and
//                   delta_t (Eq. 7).
//
// The relevance pass is HBM bound: it reads T*H*W*D elements once, streamed
// by TMA bulk copies through a shared-memory ring; each CTA owns one
// contiguous range of the flattened token index so the grid is balanced.
#include <algorithm>
#include <cstring>

#include "wz_internal.cuh"
#include "wz_ptx.cuh"

namespace wz {

struct VideoParBlock {
    VideoPar v[WZ_MAX_VIDEOS];
};

// u_q = mean of the query rows: a block covers 32 channels with 8 row
// slices; compensated fp32 sums (TwoSum) per slice, combined in a fixed
// order, stored as fp64 and fp32.
template <typename T>
__global__ void __launch_bounds__(256) query_pool_kernel(Ctx c, VideoParBlock par) {
    __shared__ float ps[8][32], pe[8][32];
    const int v = blockIdx.y;
    const VideoPar vp = par.v[v];
    if (blockIdx.x == 0 && threadIdx.x == 0) c.vpar[v] = vp;
    const int cl = threadIdx.x & 31, slice = threadIdx.x >> 5;
    const int d = blockIdx.x * 32 + cl;
    float s = 0.f, e = 0.f;
    if (d < c.D) {
        const T *Q = static_cast<const T *>(c.Q) + (size_t)vp.q_row0 * c.D + d;
        for (int j = slice; j < vp.Lq; j += 8) {
            float t, err;
            two_sum(s, load_scalar<T>(Q + (size_t)j * c.D), t, err);
            s = t;
            e += err;
        }
    }
    ps[slice][cl] = s;
    pe[slice][cl] = e;
    __syncthreads();
    if (slice == 0 && d < c.D) {
        float S = 0.f, E = 0.f;
        for (int k = 0; k < 8; ++k) {
            float t, err;
            two_sum(S, ps[k][cl], t, err);
            S = t;
            E += err + pe[k][cl];
        }
        const double m = ((double)S + (double)E) / (double)vp.Lq;
        c.qbar64[(size_t)v * c.D + d] = m;
        c.qbar32[(size_t)v * c.D + d] = (float)m;
    }
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

// Tokens per TMA chunk: never crosses a frame boundary.
__device__ __forceinline__ int64_t chunk_len(int64_t tok, int64_t end, int N, int CH) {
    const int64_t f_end = (tok / N + 1) * (int64_t)N;
    return min((int64_t)CH, min(end, f_end) - tok);
}

constexpr int kRelStages = 3;
constexpr int kRelMaxConsumers = 512;
constexpr uint64_t kRelTimeoutNs = 2000000000ull;

// One CTA streams tokens [blockIdx.x*L1, +L1) of the flattened [V*T*N] index.
// The last warp copies chunks of CH consecutive tokens (contiguous in HBM)
// into a 3-stage shared-memory ring with cp.async.bulk; the other warps
// (NC threads, VPT 16-byte vectors each) read them from shared memory.
template <typename T, int VPT>
__global__ void __launch_bounds__(kRelMaxConsumers + 32, 1) relevance_pass_kernel(Ctx c, int CH) {
    constexpr int VEC = VecOf<T>::kElems;
    constexpr int GROUP = 8;                 // tokens per cross-warp reduction
    constexpr int NV = 2 * GROUP;            // GROUP dots + GROUP squared norms
    extern __shared__ __align__(128) uint8_t rsm[];
    __shared__ float red[2][kRelMaxConsumers / 32][NV];
    __shared__ float qsum[kRelMaxConsumers / 32];
    __shared__ uint64_t full[kRelStages], empty[kRelStages];
    __shared__ int ok_flag;
    const int NC = blockDim.x - 32;          // consumer threads
    const int nw = NC >> 5;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int n_vec = c.D / VEC;
    const size_t rowb = (size_t)c.D * sizeof(T);
    const size_t stage_bytes = (size_t)CH * rowb;
    const int64_t total = (int64_t)c.V * c.T * c.N;
    const int64_t start = (int64_t)blockIdx.x * c.L1;
    const int64_t end = min(start + c.L1, total);
    if (threadIdx.x == 0) {
        for (int s = 0; s < kRelStages; ++s) {
            ptx::mbar_init(&full[s], 1);
            ptx::mbar_init(&empty[s], 1);
        }
        ok_flag = 1;
        ptx::fence_barrier_init();
        ptx::fence_proxy_async_smem();
    }
    __syncthreads();
    if (start >= end) return;

    if (warp == nw) {
        // ---------------- producer ----------------
        if (lane == 0) {
            const uint64_t pol = ptx::policy_evict_first();
            const char *X = static_cast<const char *>(c.X);
            int s = 0;
            uint32_t ph = 0;
            int issued[kRelStages] = {-1, -1, -1};
            for (int64_t tok = start; tok < end;) {
                const int64_t n = chunk_len(tok, end, c.N, CH);
                if (!ptx::mbar_wait(&empty[s], ph ^ 1u, kRelTimeoutNs)) {
                    atomicOr(c.status, 16);
                    break;
                }
                ptx::mbar_arrive_expect_tx(&full[s], (uint32_t)(n * rowb));
                ptx::bulk_load(rsm + s * stage_bytes, X + (size_t)tok * rowb, (uint32_t)(n * rowb), &full[s], pol);
                issued[s] = (int)ph;
                tok += n;
                if (++s == kRelStages) {
                    s = 0;
                    ph ^= 1u;
                }
            }
            for (int k = 0; k < kRelStages; ++k)
                if (issued[k] >= 0) ptx::mbar_wait(&full[k], (uint32_t)issued[k], kRelTimeoutNs);
        }
        return;
    }

    // ---------------- consumers ----------------
    auto consumer_sync = [&]() { asm volatile("bar.sync 1, %0;" ::"r"(NC) : "memory"); };
    constexpr int NP = VEC / 2;                  // packed pairs per 16-byte vector
    int cur_v = -1;
    f2_t q[VPT][NP];
    float qn = 0.f;
    f2_t cs[VPT][NP];
    int gi = 0;
    int s = 0;
    uint32_t ph = 0;
    int64_t cur_f = -1;
    for (int64_t tok = start; tok < end;) {
        const int64_t f = tok / c.N;
        const int64_t n = chunk_len(tok, end, c.N, CH);
        if (f != cur_f) {
            cur_f = f;
            const int v = (int)(f / c.T);
            if (v != cur_v) {
                cur_v = v;
                float qq = 0.f;
#pragma unroll
                for (int vi = 0; vi < VPT; ++vi) {
                    const int vidx = threadIdx.x + vi * NC;
#pragma unroll
                    for (int e = 0; e < NP; ++e) {
                        const float q0 = vidx < n_vec ? c.qbar32[(size_t)v * c.D + vidx * VEC + 2 * e] : 0.f;
                        const float q1 = vidx < n_vec ? c.qbar32[(size_t)v * c.D + vidx * VEC + 2 * e + 1] : 0.f;
                        q[vi][e] = pack2(q0, q1);
                        qq = fmaf(q0, q0, fmaf(q1, q1, qq));
                    }
                }
                for (int o = 16; o > 0; o >>= 1) qq += __shfl_xor_sync(0xffffffffu, qq, o);
                consumer_sync();
                if (lane == 0) qsum[warp] = qq;
                consumer_sync();
                qq = 0.f;
                for (int w = 0; w < nw; ++w) qq += qsum[w];
                qn = sqrtf(qq);
            }
#pragma unroll
            for (int vi = 0; vi < VPT; ++vi)
#pragma unroll
                for (int e = 0; e < NP; ++e) cs[vi][e] = 0ull;
        }
        // wait for the chunk (one bounded waiter decides for all consumers)
        if (threadIdx.x == 0) ok_flag = ptx::mbar_wait(&full[s], ph, kRelTimeoutNs) ? 1 : 0;
        consumer_sync();
        if (!ok_flag) {
            if (threadIdx.x == 0) atomicOr(c.status, 32);
            break;
        }
        ptx::mbar_wait(&full[s], ph, kRelTimeoutNs);   // completed: acquire for this thread
        const uint32_t st32 = ptx::smem_u32(rsm) + (uint32_t)(s * stage_bytes);
        const uint32_t rowb32 = (uint32_t)rowb;
        const int nt = (int)n;
        for (int g0 = 0; g0 < nt; g0 += GROUP, ++gi) {
            float acc[NV];
            const bool full_group = nt - g0 >= GROUP;
#pragma unroll
            for (int k = 0; k < GROUP; ++k) {
                f2_t dd = 0ull, nn = 0ull;
                if (full_group || g0 + k < nt) {
                    const uint32_t row = st32 + (uint32_t)(g0 + k) * rowb32;
#pragma unroll
                    for (int vi = 0; vi < VPT; ++vi) {
                        const int vidx = threadIdx.x + vi * NC;
                        if (vidx < n_vec) {
                            const uint4 raw = ptx::lds128(row + (uint32_t)vidx * 16u);
                            f2_t x[NP];
                            unpack_pairs(raw, x, (T *)nullptr);
#pragma unroll
                            for (int e = 0; e < NP; ++e) {
                                cs[vi][e] = add2(cs[vi][e], x[e]);
                                dd = fma2(x[e], q[vi][e], dd);
                                nn = fma2(x[e], x[e], nn);
                            }
                        }
                    }
                }
                const float2 d2 = unpack2(dd), n2 = unpack2(nn);
                acc[k] = d2.x + d2.y;
                acc[k + GROUP] = n2.x + n2.y;
            }
            const float tot = transpose_reduce<NV>(acc);
            const int b = gi & 1;
            if ((lane & 1) == 0) red[b][warp][lane >> 1] = tot;
            consumer_sync();
            if (threadIdx.x < 32) {
                float sm = 0.f;
                if (lane < NV)
                    for (int w = 0; w < nw; ++w) sm += red[b][w][lane];
                const float nrm = __shfl_down_sync(0xffffffffu, sm, GROUP);
                if (lane < GROUP && g0 + lane < nt) {
                    const float a = (nrm > 0.f && qn > 0.f) ? sm / (sqrtf(nrm) * qn) : 0.f;
                    c.a[tok + g0 + lane] = a;
                }
            }
        }
        // every consumer has passed its last read of the stage (the group
        // barrier above), so the stage goes back to the producer
        if (threadIdx.x == 0) ptx::mbar_arrive(&empty[s]);
        if (++s == kRelStages) {
            s = 0;
            ph ^= 1u;
        }
        tok += n;
        const bool frame_done = (tok % c.N == 0) || tok >= end;
        if (frame_done) {
            // column partial of frame f from this CTA: slot blockIdx.x + f
            float *dst = c.part + ((size_t)blockIdx.x + (size_t)f) * c.D;
#pragma unroll
            for (int vi = 0; vi < VPT; ++vi) {
                const int vidx = threadIdx.x + vi * NC;
                if (vidx < n_vec) {
#pragma unroll
                    for (int e = 0; e < NP; e += 2) {
                        const float2 a = unpack2(cs[vi][e]), b = unpack2(cs[vi][e + 1]);
                        *reinterpret_cast<float4 *>(dst + vidx * VEC + 2 * e) = make_float4(a.x, a.y, b.x, b.y);
                    }
                }
            }
        }
    }
}

// Per (2048-channel chunk, frame): fp64 frame sums from the fixed list of CTA
// partials (8 channels per thread), and their products with u_q, with the
// previous frame and of u_q with itself.
__global__ void __launch_bounds__(256) frame_stats_kernel(Ctx c) {
    __shared__ double scratch[40];
    const int64_t f = blockIdx.y;
    const int t = (int)(f % c.T);
    const int v = (int)(f / c.T);
    const int64_t lo = f * c.N / c.L1;
    const int64_t hi = min((int64_t)c.G1 - 1, ((f + 1) * c.N - 1) / c.L1);
    const int64_t g = f - 1;
    const int64_t lo2 = t > 0 ? g * c.N / c.L1 : 0;
    const int64_t hi2 = t > 0 ? min((int64_t)c.G1 - 1, ((g + 1) * c.N - 1) / c.L1) : -1;
    // fp32 products summed over this thread's 8 channels, fp64 across threads
    float p0 = 0.f, p1 = 0.f, p2 = 0.f, p3 = 0.f;
    for (int k = 0; k < kStatsChunk / 256; ++k) {
        const int d = blockIdx.x * kStatsChunk + k * 256 + threadIdx.x;
        if (d >= c.D) break;
        float sf = 0.f, sp = 0.f;
        for (int64_t cc = lo; cc <= hi; ++cc) sf += c.part[(size_t)(cc + f) * c.D + d];
        for (int64_t cc = lo2; cc <= hi2; ++cc) sp += c.part[(size_t)(cc + g) * c.D + d];
        const float q = c.qbar32[(size_t)v * c.D + d];
        if (c.frame_mean) c.frame_mean[(size_t)f * c.D + d] = sf / (float)c.N;
        p0 = fmaf(sf, q, p0);
        p1 = fmaf(sf, sf, p1);
        p2 = fmaf(sf, sp, p2);
        p3 = fmaf(q, q, p3);
    }
    double s0 = p0, s1 = p1, s2 = p2, s3 = p3;
    s0 = block_sum(s0, scratch);
    s1 = block_sum(s1, scratch);
    s2 = block_sum(s2, scratch);
    s3 = block_sum(s3, scratch);
    if (threadIdx.x == 0) {
        double *o = c.trip + ((size_t)f * c.DC + blockIdx.x) * 4;
        o[0] = s0;
        o[1] = s1;
        o[2] = s2;
        o[3] = s3;
    }
}

// r_t only (the relevance entry point); the condensation pass does this in
// the temporal kernel.
__global__ void relevance_finalize_kernel(Ctx c) {
    const int64_t f = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (f >= (int64_t)c.V * c.T) return;
    double dq = 0.0, ff = 0.0, qq = 0.0;
    for (int k = 0; k < c.DC; ++k) {
        dq += c.trip[((size_t)f * c.DC + k) * 4 + 0];
        ff += c.trip[((size_t)f * c.DC + k) * 4 + 1];
        qq += c.trip[((size_t)f * c.DC + k) * 4 + 3];
    }
    const double qn = sqrt(qq);
    c.frame_scores[f] = (ff > 0.0 && qn > 0.0) ? (float)(dq / (sqrt(ff) * qn)) : 0.f;
}

cudaError_t launch_query_pool(const Ctx &c, const VideoPar *hpar, cudaStream_t s) {
    VideoParBlock blk;   // copied into the launch parameters
    memset(&blk, 0, sizeof(blk));
    for (int v = 0; v < c.V; ++v) blk.v[v] = hpar[v];
    const dim3 grid((unsigned)((c.D + 31) / 32), (unsigned)c.V);
    if (c.dtype == WZ_DTYPE_BF16)
        query_pool_kernel<__nv_bfloat16><<<grid, 256, 0, s>>>(c, blk);
    else
        query_pool_kernel<float><<<grid, 256, 0, s>>>(c, blk);
    return cudaGetLastError();
}

namespace {

struct RelCfg {
    const void *fn = nullptr;
    int threads = 0;     // consumers + one producer warp
    int CH = 0;          // tokens per chunk
    size_t smem = 0;
};

template <typename T, int VPT>
void relevance_config(const Ctx &c, RelCfg &r) {
    r.fn = (const void *)relevance_pass_kernel<T, VPT>;
    constexpr int VEC = VecOf<T>::kElems;
    const int n_vec = c.D / VEC;
    const int nc = std::max(32, ((n_vec + VPT - 1) / VPT + 31) / 32 * 32);
    r.threads = nc + 32;
    const size_t rowb = (size_t)c.D * sizeof(T);
    int ch = (int)std::max<size_t>(1, (56 * 1024) / rowb);
    ch = std::min(ch, 32);
    if (ch >= 8) ch = ch / 8 * 8;
    r.CH = ch;
    r.smem = (size_t)kRelStages * ch * rowb;
}

template <typename T>
bool pick(const Ctx &c, RelCfg &r) {
    constexpr int VEC = VecOf<T>::kElems;
    const int n_vec = c.D / VEC;
    if (n_vec <= 512) relevance_config<T, 1>(c, r);
    else if (n_vec <= 1024) relevance_config<T, 2>(c, r);
    else if (n_vec <= 2048) relevance_config<T, 4>(c, r);
    else if (n_vec <= 4096) relevance_config<T, 8>(c, r);
    else return false;
    return true;
}

bool pick_any(const Ctx &c, RelCfg &r) {
    return c.dtype == WZ_DTYPE_BF16 ? pick<__nv_bfloat16>(c, r) : pick<float>(c, r);
}

}  // namespace

int relevance_grid(const Ctx &c) {
    RelCfg r;
    if (!pick_any(c, r)) return 0;
    int dev = 0, sms = 0, per_sm = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    if (cudaFuncSetAttribute(r.fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)r.smem) != cudaSuccess) return 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, r.fn, r.threads, r.smem) != cudaSuccess) return 0;
    if (per_sm < 1) per_sm = 1;
    const int64_t total = (int64_t)c.V * c.T * c.N;
    int64_t g = (int64_t)sms * per_sm;
    const int64_t min_tokens = 16;
    g = std::min<int64_t>(g, (total + min_tokens - 1) / min_tokens);
    g = std::min<int64_t>(g, kG1Max);
    return (int)std::max<int64_t>(g, 1);
}

cudaError_t launch_relevance_pass(const Ctx &c, cudaStream_t s) {
    RelCfg r;
    if (!pick_any(c, r)) return cudaErrorInvalidValue;
    cudaError_t e = cudaFuncSetAttribute(r.fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)r.smem);
    if (e != cudaSuccess) return e;
    int CH = r.CH;
    void *args[] = {const_cast<Ctx *>(&c), &CH};
    return cudaLaunchKernel(r.fn, dim3(c.G1), dim3(r.threads), args, r.smem, s);
}

cudaError_t launch_frame_stats(const Ctx &c, cudaStream_t s) {
    frame_stats_kernel<<<dim3(c.DC, c.V * c.T), 256, 0, s>>>(c);
    return cudaGetLastError();
}

cudaError_t launch_relevance_finalize(const Ctx &c, cudaStream_t s) {
    const int n = c.V * c.T;
    relevance_finalize_kernel<<<(n + 255) / 256, 256, 0, s>>>(c);
    return cudaGetLastError();
}

}  // namespace wz
