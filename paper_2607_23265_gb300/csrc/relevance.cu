// Cross-Modal Scorer, similarity branch (Section 3.2.1), on the GPU.
//
//   query_pool      u_q = mean of the query rows (compensated fp32 -> fp64).
//   relevance_pass  one streaming read of the features: per token
//                   a_{t,n} = <u, u_q> / (||u|| ||u_q||) (the input of Eq. 6)
//                   and per-CTA column sums of every frame it touches (the
//                   average pool of Section 3.2.1 / Eq. 7), in fp32.
//   frame_stats     one block per frame sums the column partials of the frame
//                   in a fixed order and forms r_t and delta_t (Eq. 7) from
//                   <v_t,u_q>, <v_t,v_t>, <v_t,v_{t-1}>, <v_{t-1},v_{t-1}>
//                   and <u_q,u_q>, reduced in fp64.
//   query_rows      (max-over-query scorer) the norms of the query rows and
//                   the rows scaled to unit length, split into bf16 hi + lo
//                   halves: the B operand of the token x row cosine GEMM.
//
// With the max-over-query scorer the relevance pass stores ||u|| in place of
// a_{t,n}; the tensor-core GEMM that follows divides max_j <u, q_j/||q_j||>
// by it, and frame_stats takes r_t = max_j cos(v_bar_t, q_j) from the raw
// rows and their norms.
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
    pdl_wait();
    pdl_trigger();
    const int v = blockIdx.y;
    const VideoPar vp = par.v[v];
    if (blockIdx.x == 0 && threadIdx.x == 0) {
        c.vpar[v] = vp;
        if (c.drange) {   // empty range of delta_t, filled by frame_stats
            c.drange[2 * v] = 0x7ff0000000000000ull;   // +inf
            c.drange[2 * v + 1] = 0ull;                // +0
        }
    }
    const int cl = threadIdx.x & 31, slice = threadIdx.x >> 5;
    const int d = blockIdx.x * 32 + cl;
    float s = 0.f, e = 0.f;
    if (d < c.D) {
        const T *Q = static_cast<const T *>(c.Q) + (size_t)vp.q_row0 * c.D + d;
        // rows slice, slice + 8, ...: loaded 8 at a time, then summed in order
        for (int j0 = slice; j0 < vp.Lq; j0 += 64) {
            float x[8];
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                const int j = j0 + 8 * k;
                x[k] = j < vp.Lq ? load_scalar<T>(Q + (size_t)j * c.D) : 0.f;
            }
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                if (j0 + 8 * k < vp.Lq) {
                    float t, err;
                    two_sum(s, x[k], t, err);
                    s = t;
                    e += err;
                }
            }
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

// Query rows of video v for the max-over-query scorer: block j < Lq writes
// ||q_j|| (fp64 sum of fp32 squares) to qnorm and q_j / ||q_j|| as bf16 hi
// (row j of qhl) and lo = bf16(x - hi) (row Lqp + j); blocks Lq <= j < Lqp
// write zero rows, so the GEMM's padding columns are zero.  bf16 rows.
__global__ void __launch_bounds__(256) query_rows_kernel(Ctx c, int v, int q_row0, int Lq, int Lqp) {
    __shared__ double red[33];
    pdl_wait();
    pdl_trigger();
    const int j = blockIdx.x;
    const int D = c.D;
    __nv_bfloat16 *hi = c.qhl + (size_t)j * D;
    __nv_bfloat16 *lo = c.qhl + (size_t)(Lqp + j) * D;
    const __nv_bfloat16 zero = __float2bfloat16_rn(0.f);
    if (j >= Lq) {
        for (int d = threadIdx.x; d < D; d += blockDim.x) {
            hi[d] = zero;
            lo[d] = zero;
        }
        return;
    }
    const __nv_bfloat16 *q = static_cast<const __nv_bfloat16 *>(c.Q) + (size_t)(q_row0 + j) * D;
    float ss = 0.f;
    for (int d = threadIdx.x; d < D; d += blockDim.x) {
        const float x = __bfloat162float(q[d]);
        ss = fmaf(x, x, ss);
    }
    const double qn = sqrt(block_sum((double)ss, red));
    if (threadIdx.x == 0) c.qnorm[(size_t)v * WZ_MAX_LQ_MAXSIM + j] = (float)qn;
    const float inv = qn > 0.0 ? (float)(1.0 / qn) : 0.f;
    for (int d = threadIdx.x; d < D; d += blockDim.x) {
        const float x = __bfloat162float(q[d]) * inv;
        const __nv_bfloat16 h = __float2bfloat16_rn(x);
        hi[d] = h;
        lo[d] = __float2bfloat16_rn(x - __bfloat162float(h));
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

// Tokens per TMA chunk starting at token `tok`, index `pos` within its
// frame: never crosses a frame boundary or the end of the range.
__device__ __forceinline__ int chunk_len(int pos, int64_t tok, int64_t end, int N, int CH) {
    return (int)min((int64_t)min(CH, N - pos), end - tok);
}

constexpr int kRelStages = 3;
constexpr int kRelMaxConsumers = 512;
constexpr uint64_t kRelTimeoutNs = 2000000000ull;

// One CTA streams tokens [blockIdx.x*L1, +L1) of the flattened [V*T*N] index.
// The last warp copies chunks of CH consecutive tokens (contiguous in HBM)
// into a 3-stage shared-memory ring with cp.async.bulk; the other warps
// (NC threads, VPT 16-byte vectors each) read them from shared memory.  Each
// consumer warp waits for a chunk itself and hands it back itself; per-token
// partial dots and norms go to a shared window that all consumers reduce
// together once per <= 64 tokens, so block barriers are rare.
template <typename T, int VPT>
__global__ void __launch_bounds__(kRelMaxConsumers + 32, 1) relevance_pass_kernel(Ctx c, int CH) {
    // The producer streams only the features, which the kernels before this
    // one do not write, so it starts before the wait for the previous grid
    // (the query pooling) and fills the ring meanwhile; the consumers wait
    // for it before they read u_q or write anything.
    pdl_trigger();
    constexpr int VEC = VecOf<T>::kElems;
    constexpr int GROUP = 8;                 // tokens per warp transpose-reduction
    constexpr int NV = 2 * GROUP;            // GROUP dots + GROUP squared norms
    constexpr int WIN = 128;                 // tokens per cross-warp reduction
    constexpr int NWMAX = kRelMaxConsumers / 32;
    extern __shared__ __align__(128) uint8_t rsm[];
    __shared__ float wpart[2][NWMAX][2][WIN];
    __shared__ float qsum[NWMAX];
    __shared__ uint64_t full[kRelStages], empty[kRelStages];
    __shared__ volatile int abort_flag;
    const int NC = blockDim.x - 32;          // consumer threads
    const int nw = NC >> 5;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int n_vec = c.D / VEC;
    const bool maxsim = c.relevance_mode == WZ_RELEVANCE_MAXSIM;
    const size_t rowb = (size_t)c.D * sizeof(T);
    const size_t stage_bytes = (size_t)CH * rowb;
    const int64_t total = (int64_t)c.V * c.T * c.N;
    const int64_t start = (int64_t)blockIdx.x * c.L1;
    const int64_t end = min(start + c.L1, total);
    if (threadIdx.x == 0) {
        for (int s = 0; s < kRelStages; ++s) {
            ptx::mbar_init(&full[s], 1);
            ptx::mbar_init(&empty[s], (uint32_t)nw);
        }
        abort_flag = 0;
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
            int pos = (int)(start % c.N);   // token index within its frame
            for (int64_t tok = start; tok < end && !abort_flag;) {
                const int n = chunk_len(pos, tok, end, c.N, CH);
                if (!ptx::mbar_wait(&empty[s], ph ^ 1u, kRelTimeoutNs)) {
                    atomicOr(c.status, 16);
                    abort_flag = 1;
                    break;
                }
                ptx::mbar_arrive_expect_tx(&full[s], (uint32_t)(n * rowb));
                ptx::bulk_load(rsm + s * stage_bytes, X + (size_t)tok * rowb, (uint32_t)(n * rowb), &full[s], pol);
                issued[s] = (int)ph;
                tok += n;
                pos += n;
                if (pos == c.N) pos = 0;
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
    pdl_wait();
    auto consumer_sync = [&]() { asm volatile("bar.sync 1, %0;" ::"r"(NC) : "memory"); };
    constexpr int NP = VEC / 2;                  // packed pairs per 16-byte vector
    constexpr int SHIFT = 1;                     // lane l holds reduced value l >> 1
    int cur_v = -1;
    f2_t q[VPT][NP];
    float qn = 0.f;
    // column sums, split by token parity when registers allow (two shorter
    // dependent chains per group)
    constexpr int CSP = VPT == 1 ? 2 : 1;
    f2_t cs[CSP][VPT][NP];
    int s = 0;
    uint32_t ph = 0;
    bool dead = false;
    int buf = 0, wcount = 0;
    int64_t wbase = start;
    // frame f, its position t in the video v, and the token index within the
    // frame are carried along: no 64-bit divisions inside the loop
    int64_t f = start / c.N;
    int pos = (int)(start - f * c.N);
    int tf = (int)(f % c.T), v = (int)(f / c.T);
    bool frame_new = true;
    for (int64_t tok = start; tok < end;) {
        const int n = chunk_len(pos, tok, end, c.N, CH);
        if (frame_new) {
            frame_new = false;
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
                for (int e = 0; e < NP; ++e) cs[0][vi][e] = cs[CSP - 1][vi][e] = 0ull;
        }
        // this warp waits for the chunk itself (bounded)
        int ok = 1;
        if (lane == 0 && !dead) ok = ptx::mbar_wait(&full[s], ph, kRelTimeoutNs) ? 1 : 0;
        ok = __shfl_sync(0xffffffffu, ok, 0);
        if (!ok && !dead) {
            dead = true;
            if (lane == 0) {
                abort_flag = 1;
                atomicOr(c.status, 32);
            }
        }
        const int nt = (int)n;
        if (!dead) {
            ptx::mbar_wait(&full[s], ph, kRelTimeoutNs);   // completed: acquire for this thread
            const uint32_t st32 = ptx::smem_u32(rsm) + (uint32_t)(s * stage_bytes);
            const uint32_t rowb32 = (uint32_t)rowb;
            for (int g0 = 0; g0 < nt; g0 += GROUP) {
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
                                    cs[k & (CSP - 1)][vi][e] = add2(cs[k & (CSP - 1)][vi][e], x[e]);
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
                const int idx = lane >> SHIFT;              // value held by this lane
                const int kk = idx & (GROUP - 1);
                if ((lane & 1) == 0 && g0 + kk < nt)
                    wpart[buf][warp][idx >> 3][wcount + g0 + kk] = tot;
            }
        }
        // hand the stage back once this warp's reads are done
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(&empty[s]);
        if (++s == kRelStages) {
            s = 0;
            ph ^= 1u;
        }
        tok += n;
        pos += n;
        wcount += nt;
        const bool frame_done = pos == c.N || tok >= end;
        if (frame_done && !dead &&
            wz_in_range(c.status, (int64_t)blockIdx.x + (int64_t)f < (int64_t)c.G1 + (int64_t)c.V * c.T)) {
            // column partial of frame f from this CTA: slot blockIdx.x + f
            float *dst = c.part + ((size_t)blockIdx.x + (size_t)f) * c.D;
#pragma unroll
            for (int vi = 0; vi < VPT; ++vi) {
                const int vidx = threadIdx.x + vi * NC;
                if (vidx < n_vec) {
#pragma unroll
                    for (int e = 0; e < NP; e += 2) {
                        f2_t s0 = cs[0][vi][e], s1 = cs[0][vi][e + 1];
                        if (CSP == 2) {
                            s0 = add2(s0, cs[CSP - 1][vi][e]);
                            s1 = add2(s1, cs[CSP - 1][vi][e + 1]);
                        }
                        const float2 a = unpack2(s0), b = unpack2(s1);
                        *reinterpret_cast<float4 *>(dst + vidx * VEC + 2 * e) = make_float4(a.x, a.y, b.x, b.y);
                    }
                }
            }
        }
        if (pos == c.N) {
            pos = 0;
            ++f;
            frame_new = true;
            if (++tf == c.T) {
                tf = 0;
                ++v;
            }
        }
        // reduce the window across warps: when it is full, at the end of the
        // range, and before a new video changes u_q
        const bool new_video = tok < end && v != cur_v;
        if (tok >= end || wcount + CH > WIN || new_video) {
            consumer_sync();
            if (abort_flag) break;
            if (!wz_in_range(c.status, wbase + wcount <= total)) wcount = 0;
            for (int t = threadIdx.x; t < wcount; t += NC) {
                float dot = 0.f, nrm = 0.f;
                for (int w = 0; w < nw; ++w) {
                    dot += wpart[buf][w][0][t];
                    nrm += wpart[buf][w][1][t];
                }
                c.a[wbase + t] = maxsim ? sqrtf(nrm)   // ||u||, divided out by the row-max GEMM
                                        : (nrm > 0.f && qn > 0.f) ? dot / (sqrtf(nrm) * qn) : 0.f;
            }
            buf ^= 1;
            wbase = tok;
            wcount = 0;
        }
    }
}

// Gate of the WSM for frame f (Eq. 6, Eq. 12): the saliency map M = min-max
// normalised a_{t,n} over the frame, average-pooled to the subband grid of
// each DWT level (hp x wp for the first) and scaled by lambda.  `red` is >= 32
// floats of shared scratch.
constexpr int kGatePerThread = WZ_MAX_HW * WZ_MAX_HW / 512;   // a_{t,n} per thread of a 512-thread block

// The frame's a_{t,n} (an external scorer's if given), this thread's share
// k = threadIdx.x + 512 r, loaded into registers early so that the loads
// overlap the frame statistics.
__device__ __forceinline__ void gate_prefetch(const Ctx &c, int64_t f, float (&av)[kGatePerThread]) {
    const float *a = (c.ext_a ? c.ext_a : c.a) + f * c.N;
#pragma unroll
    for (int r = 0; r < kGatePerThread; ++r) {
        const int k = (int)threadIdx.x + 512 * r;
        av[r] = k < c.N ? a[k] : 0.f;
    }
}

__device__ void frame_gate(const Ctx &c, int64_t f, float *red, const float (&av)[kGatePerThread], float *M) {
    const int N = c.N, H = c.H, W = c.W;
    float lo = INFINITY, hi = -INFINITY;
#pragma unroll
    for (int r = 0; r < kGatePerThread; ++r) {
        const int k = (int)threadIdx.x + 512 * r;
        if (k < N) {
            M[k] = av[r];
            lo = fminf(lo, av[r]);
            hi = fmaxf(hi, av[r]);
        }
    }
    for (int o = 16; o > 0; o >>= 1) {
        lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, o));
        hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, o));
    }
    __syncthreads();   // red is free (the caller's reads are done)
    if ((threadIdx.x & 31) == 0) {
        red[threadIdx.x >> 5] = lo;
        red[16 + (threadIdx.x >> 5)] = hi;
    }
    __syncthreads();
    lo = INFINITY;
    hi = -INFINITY;
    for (int k = 0; k < (int)(blockDim.x >> 5); ++k) {
        lo = fminf(lo, red[k]);
        hi = fmaxf(hi, red[16 + k]);
    }
    const float rng = hi - lo;
    for (int k = threadIdx.x; k < N; k += blockDim.x) M[k] = rng > 0.f ? (M[k] - lo) / rng : 0.f;
    __syncthreads();
    for (int l = 1; l <= c.wsm_levels; ++l) {
        const int hp = c.lvl_h[l], wp = c.lvl_w[l];
        if (!wz_in_range(c.status, c.goff[l - 1] + hp * wp <= c.gate_stride)) break;
        float *G = c.gate + f * (int64_t)c.gate_stride + c.goff[l - 1];
        for (int k = threadIdx.x; k < hp * wp; k += blockDim.x) {
            const int ai = k / wp, bj = k % wp;
            const int r0 = (ai * H) / hp, r1 = ((ai + 1) * H + hp - 1) / hp;
            const int c0 = (bj * W) / wp, c1 = ((bj + 1) * W + wp - 1) / wp;
            float s = 0.f;
            for (int y = r0; y < r1; ++y)
                for (int x = c0; x < c1; ++x) s += M[y * W + x];
            G[k] = c.lambda * (s / (float)((r1 - r0) * (c1 - c0)));
        }
    }
}

// The gate of frame f (as frame_gate) formed by the upper half of
// frame_stats_kernel's threads (t0 = threadIdx.x - nth, named barrier 2 over
// nth threads) while the lower half forms the frame statistics: the two
// chains overlap.
__device__ void gate_half(const Ctx &c, int64_t f, int t0, int nth, float *M2) {
    __shared__ float red2[32];
    auto sync = [nth] { asm volatile("bar.sync 2, %0;" ::"r"(nth) : "memory"); };
    const int N = c.N, H = c.H, W = c.W, lane = t0 & 31, w = t0 >> 5, nw = nth >> 5;
    const float *a = (c.ext_a ? c.ext_a : c.a) + f * N;
    float lo = INFINITY, hi = -INFINITY;
    for (int k = t0; k < N; k += nth) {
        const float x = a[k];
        M2[k] = x;
        lo = fminf(lo, x);
        hi = fmaxf(hi, x);
    }
    for (int o = 16; o > 0; o >>= 1) {
        lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, o));
        hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, o));
    }
    if (lane == 0) {
        red2[w] = lo;
        red2[16 + w] = hi;
    }
    sync();
    lo = INFINITY;
    hi = -INFINITY;
    for (int k = 0; k < nw; ++k) {
        lo = fminf(lo, red2[k]);
        hi = fmaxf(hi, red2[16 + k]);
    }
    const float rng = hi - lo;
    for (int k = t0; k < N; k += nth) M2[k] = rng > 0.f ? (M2[k] - lo) / rng : 0.f;
    sync();
    for (int l = 1; l <= c.wsm_levels; ++l) {
        const int hp = c.lvl_h[l], wp = c.lvl_w[l];
        if (!wz_in_range(c.status, c.goff[l - 1] + hp * wp <= c.gate_stride)) break;
        float *G = c.gate + f * (int64_t)c.gate_stride + c.goff[l - 1];
        for (int k = t0; k < hp * wp; k += nth) {
            const int ai = k / wp, bj = k % wp;
            const int r0 = (ai * H) / hp, r1 = ((ai + 1) * H + hp - 1) / hp;
            const int c0 = (bj * W) / wp, c1 = ((bj + 1) * W + wp - 1) / wp;
            float s = 0.f;
            for (int y = r0; y < r1; ++y)
                for (int x = c0; x < c1; ++x) s += M2[y * W + x];
            G[k] = c.lambda * (s / (float)((r1 - r0) * (c1 - c0)));
        }
    }
}

// One block per frame: the frame sums (fixed list of CTA partials) for all
// channels, read as 16-byte vectors; fp32 products summed over each thread's
// channels and across each warp, the warp totals in fp64; then
// r_t = cos(v_bar_t, u_q) and delta_t = 1 - cos(v_bar_t, v_bar_{t-1})
// clamped to [0, 2] (Eq. 7) in fp64.
//
// With the max-over-query scorer the frame sums are kept in shared memory
// (D floats of dynamic shared memory) and every warp takes query rows j:
// <v_t, q_j> in fp32 (as the per-warp partials of the mean scorer), divided
// by ||q_j|| in fp64; r_t = max_j of that / ||v_t||.
__global__ void __launch_bounds__(512) frame_stats_kernel(Ctx c) {
    pdl_wait();
    pdl_trigger();
    __shared__ float wsum[16][5];
    __shared__ double wmax[16];
    __shared__ float gate_map[WZ_MAX_HW * WZ_MAX_HW];   // the frame's saliency map (either gate form)
    extern __shared__ float4 sfs[];   // [D/4] frame sums (max-over-query scorer only)
    const bool maxsim = c.relevance_mode == WZ_RELEVANCE_MAXSIM;
    const bool do_gate = c.gate && c.spatial_mode == WZ_SPATIAL_WSM;
    const int64_t f = blockIdx.x;
    // with the mean scorer, the upper half of the threads forms the gate
    // while the lower half forms the statistics; the max-over-query scorer
    // takes every warp for its query rows and forms the gate after them
    const bool split = !maxsim && do_gate;
    const int half = (int)blockDim.x / 2;
    if (split && (int)threadIdx.x >= half) {
        gate_half(c, f, (int)threadIdx.x - half, half, gate_map);
        return;
    }
    const int nst = split ? half : (int)blockDim.x;   // threads forming the statistics
    float av[kGatePerThread];
    if (do_gate && !split) gate_prefetch(c, f, av);
    const int t = (int)(f % c.T);
    const int v = (int)(f / c.T);
    const int64_t lo = f * c.N / c.L1;
    const int64_t hi = min((int64_t)c.G1 - 1, ((f + 1) * c.N - 1) / c.L1);
    const int64_t g = f - 1;
    const int64_t lo2 = t > 0 ? g * c.N / c.L1 : 0;
    const int64_t hi2 = t > 0 ? min((int64_t)c.G1 - 1, ((g + 1) * c.N - 1) / c.L1) : -1;
    const int nv = c.D / 4;
    const float4 *P = reinterpret_cast<const float4 *>(c.part);
    const float4 *Qv = reinterpret_cast<const float4 *>(c.qbar32 + (size_t)v * c.D);
    float p0 = 0.f, p1 = 0.f, p2 = 0.f, p3 = 0.f, p4 = 0.f;
    for (int i = threadIdx.x; i < nv; i += nst) {
        float4 sf = make_float4(0.f, 0.f, 0.f, 0.f), sp = sf;
        for (int64_t cc = lo; cc <= hi; cc += 2) {   // two partial rows in flight, summed in order
            const float4 x = P[(size_t)(cc + f) * nv + i];
            const float4 y = cc + 1 <= hi ? P[(size_t)(cc + 1 + f) * nv + i] : make_float4(0.f, 0.f, 0.f, 0.f);
            sf.x += x.x; sf.y += x.y; sf.z += x.z; sf.w += x.w;
            if (cc + 1 <= hi) { sf.x += y.x; sf.y += y.y; sf.z += y.z; sf.w += y.w; }
        }
        for (int64_t cc = lo2; cc <= hi2; cc += 2) {
            const float4 x = P[(size_t)(cc + g) * nv + i];
            const float4 y = cc + 1 <= hi2 ? P[(size_t)(cc + 1 + g) * nv + i] : make_float4(0.f, 0.f, 0.f, 0.f);
            sp.x += x.x; sp.y += x.y; sp.z += x.z; sp.w += x.w;
            if (cc + 1 <= hi2) { sp.x += y.x; sp.y += y.y; sp.z += y.z; sp.w += y.w; }
        }
        const float4 q = Qv[i];
        if (maxsim) sfs[i] = sf;
        if (c.frame_mean) {   // caller's buffer: 4-byte alignment only
            float *fm = c.frame_mean + (size_t)f * c.D + 4 * i;
            fm[0] = sf.x / (float)c.N;
            fm[1] = sf.y / (float)c.N;
            fm[2] = sf.z / (float)c.N;
            fm[3] = sf.w / (float)c.N;
        }
        p0 = fmaf(sf.x, q.x, fmaf(sf.y, q.y, fmaf(sf.z, q.z, fmaf(sf.w, q.w, p0))));
        p1 = fmaf(sf.x, sf.x, fmaf(sf.y, sf.y, fmaf(sf.z, sf.z, fmaf(sf.w, sf.w, p1))));
        p2 = fmaf(sf.x, sp.x, fmaf(sf.y, sp.y, fmaf(sf.z, sp.z, fmaf(sf.w, sp.w, p2))));
        p3 = fmaf(q.x, q.x, fmaf(q.y, q.y, fmaf(q.z, q.z, fmaf(q.w, q.w, p3))));
        p4 = fmaf(sp.x, sp.x, fmaf(sp.y, sp.y, fmaf(sp.z, sp.z, fmaf(sp.w, sp.w, p4))));
    }
    for (int o = 16; o > 0; o >>= 1) {
        p0 += __shfl_xor_sync(0xffffffffu, p0, o);
        p1 += __shfl_xor_sync(0xffffffffu, p1, o);
        p2 += __shfl_xor_sync(0xffffffffu, p2, o);
        p3 += __shfl_xor_sync(0xffffffffu, p3, o);
        p4 += __shfl_xor_sync(0xffffffffu, p4, o);
    }
    const int warp = threadIdx.x >> 5, nw = nst >> 5;
    if (maxsim) {
        __syncthreads();   // sfs complete
        const int lane = threadIdx.x & 31;
        const VideoPar vp = c.vpar[v];
        const int n8 = c.D / 8;
        double best = -INFINITY;
        const int rot = (int)(f % vp.Lq);   // frames start on different rows: no hot L2 lines
        for (int jr = warp; jr < vp.Lq; jr += nw) {
            const int j = jr + rot < vp.Lq ? jr + rot : jr + rot - vp.Lq;
            const uint4 *qr = reinterpret_cast<const uint4 *>(static_cast<const __nv_bfloat16 *>(c.Q) +
                                                              (size_t)(vp.q_row0 + j) * c.D);
            float acc = 0.f;
            for (int i0 = lane; i0 < n8; i0 += 32 * 8) {   // 8 loads in flight per lane (L2 latency)
                uint4 qv[8];
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    const int i = i0 + 32 * u;
                    qv[u] = i < n8 ? __ldg(qr + i) : make_uint4(0u, 0u, 0u, 0u);
                }
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    const int i = i0 + 32 * u;
                    if (i < n8) {
                        float qf[8];
                        unpack(qv[u], qf, (__nv_bfloat16 *)nullptr);
                        const float4 s0 = sfs[2 * i], s1 = sfs[2 * i + 1];
                        acc = fmaf(s0.x, qf[0], fmaf(s0.y, qf[1], fmaf(s0.z, qf[2], fmaf(s0.w, qf[3],
                              fmaf(s1.x, qf[4], fmaf(s1.y, qf[5], fmaf(s1.z, qf[6], fmaf(s1.w, qf[7], acc))))))));
                    }
                }
            }
            for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
            const double qn = (double)c.qnorm[(size_t)v * WZ_MAX_LQ_MAXSIM + j];
            best = fmax(best, qn > 0.0 ? (double)acc / qn : 0.0);
        }
        if (lane == 0) wmax[warp] = best;
    }
    if ((threadIdx.x & 31) == 0) {
        wsum[warp][0] = p0;
        wsum[warp][1] = p1;
        wsum[warp][2] = p2;
        wsum[warp][3] = p3;
        wsum[warp][4] = p4;
    }
    if (split) asm volatile("bar.sync 1, %0;" ::"r"(half) : "memory");   // the statistics' warps only
    else __syncthreads();
    if (warp == 0) {
        // lane k < 5 sums quantity k over the warps in order (one fp64 warp
        // instruction per warp partial instead of five)
        const int lane = threadIdx.x & 31;
        double acc = 0.0;
        if (lane < 5)
            for (int w = 0; w < nw; ++w) acc += (double)wsum[w][lane];
        const double vq = __shfl_sync(0xffffffffu, acc, 0), vv = __shfl_sync(0xffffffffu, acc, 1);
        const double vp = __shfl_sync(0xffffffffu, acc, 2), qq = __shfl_sync(0xffffffffu, acc, 3);
        const double pp = __shfl_sync(0xffffffffu, acc, 4);
        if (lane == 0) {
            const double qn = sqrt(qq);
            double r = (vv > 0.0 && qn > 0.0) ? vq / (sqrt(vv) * qn) : 0.0;
            if (maxsim) {
                double best = -INFINITY;
                for (int w = 0; w < nw; ++w) best = fmax(best, wmax[w]);
                r = vv > 0.0 ? best / sqrt(vv) : 0.0;
            }
            if (c.ext_r) r = (double)c.ext_r[f];   // an external scorer's r_t
            double d = 0.0;
            if (t > 0) {
                const double den = sqrt(vv * pp);
                const double cs = den > 0.0 ? vp / den : 0.0;
                d = fmin(2.0, fmax(0.0, 1.0 - cs)) + 0.0;   // + 0.0: never -0
            }
            c.fr[4 * f + 0] = r;
            c.fr[4 * f + 1] = d;
            if (c.drange) {   // non-negative doubles order like their bit patterns
                const unsigned long long bits = (unsigned long long)__double_as_longlong(d);
                atomicMin(&c.drange[2 * v], bits);
                atomicMax(&c.drange[2 * v + 1], bits);
            }
            if (c.frame_scores) c.frame_scores[f] = (float)r;
        }
    }
    if (do_gate && !split) frame_gate(c, f, wsum[0], av, gate_map);
}

cudaError_t launch_query_pool(const Ctx &c, const VideoPar *hpar, cudaStream_t s) {
    VideoParBlock blk;   // copied into the launch parameters
    memset(&blk, 0, sizeof(blk));
    for (int v = 0; v < c.V; ++v) blk.v[v] = hpar[v];
    const dim3 grid((unsigned)((c.D + 31) / 32), (unsigned)c.V);
    void *args[] = {const_cast<Ctx *>(&c), &blk};
    const void *fn = c.dtype == WZ_DTYPE_BF16 ? (const void *)query_pool_kernel<__nv_bfloat16>
                                              : (const void *)query_pool_kernel<float>;
    return launch_kernel(fn, grid, dim3(256), 0, s, args, c.pdl != 0);
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
    return launch_kernel(r.fn, dim3(c.G1), dim3(r.threads), r.smem, s, args, c.pdl != 0);
}

cudaError_t launch_frame_stats(const Ctx &c, cudaStream_t s) {
    void *args[] = {const_cast<Ctx *>(&c)};
    const size_t smem = c.relevance_mode == WZ_RELEVANCE_MAXSIM ? (size_t)c.D * 4 : 0;
    if (smem > 0) {
        const cudaError_t e =
            cudaFuncSetAttribute((const void *)frame_stats_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
    }
    // 512 threads a frame (4 CTAs per SM); with the mean scorer's split form
    // and more frames than one wave of those, 256 (twice the CTAs in flight)
    const bool split = c.relevance_mode != WZ_RELEVANCE_MAXSIM && c.gate && c.spatial_mode == WZ_SPATIAL_WSM;
    int dev = 0, sms = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    const int threads = split && (int64_t)c.V * c.T > 4 * (int64_t)sms ? 256 : 512;
    return launch_kernel((const void *)frame_stats_kernel, dim3(c.V * c.T), dim3(threads), smem, s, args,
                         c.pdl != 0);
}

cudaError_t launch_query_rows(const Ctx &c, int v, int q_row0, int Lq, int Lqp, cudaStream_t s) {
    void *args[] = {const_cast<Ctx *>(&c), &v, &q_row0, &Lq, &Lqp};
    return launch_kernel((const void *)query_rows_kernel, dim3((unsigned)Lqp), dim3(256), 0, s, args, c.pdl != 0);
}

}  // namespace wz
