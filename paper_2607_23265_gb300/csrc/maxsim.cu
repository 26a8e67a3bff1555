// Max-over-query relevance in one pass over the features (the scorer of
// reading R22 for a single video): the token x query-row cosines on the
// 5th-generation tensor cores, and, from the same shared-memory tiles, each
// token's norm and the per-frame channel sums that the frame statistics
// (r_t, delta_t; Section 3.2.1, Eq. 7) need.
//
//   a_{t,n} = max_{j < Lq} <u_{t,n}, q_j / ||q_j||> / ||u_{t,n}||
//
// Token tiles of 128 rows (M) x K steps of 64 channels: A = the features,
// K-major with 128-byte swizzle; B = the unit query rows as bf16 hi rows then
// lo rows (query_rows_kernel), N = 2 Lqp <= 256.  A stage holds G
// consecutive K steps, loaded by one 3D TMA box ({64, 128, G} for the
// features, {64, 2 Lqp, G} for the query rows): a token row arrives as G * 128
// contiguous bytes per load, not 128, which keeps HBM reads efficient.  The
// features and the query rows have rings of their own, so the query rows
// (read from L2 for every tile) take two stages and the rest of shared memory
// keeps feature reads in flight.  fp32 accumulators in tensor memory, two
// buffers, so the epilogue of a tile overlaps the main loop of the next.
// CTA c covers the tokens [c L1, (c+1) L1), exactly as the relevance pass
// does, and writes its channel sums of every frame it touches into partial
// slot c + t, so frame_stats_kernel reads them unchanged.
//   warp 0       TMA producer of the features (one thread)
//   warp 1       TMEM allocation and the MMA issuer (one thread)
//   warps 2-9    channel sums and token norms: 4 channel pairs per warp, a
//                lane per channel pair and class of the tile's rows mod 8
//                (two warps per SM sub-partition; every element is read from
//                shared memory once); the classes combined by shuffles; the
//                squares of a row's channels kept per lane over the tile's K
//                steps and combined at the end of the tile; the sums of the
//                frame open at the start of a tile and of the frame that
//                starts inside it (frames have >= 128 tokens, so at most one
//                starts inside a tile) accumulate in shared memory and are
//                written to the frame's slot when the frame ends or the
//                CTA's range does.  After each tile warps 2-5 also form
//                a_{t,n} for the rows of their tensor-memory lane quadrant:
//                tcgen05.ld -> max over the query rows of hi + lo -> / ||u||
//   warp 10      TMA producer of the query rows (one thread)
// Every mbarrier wait is bounded; on a timeout the kernel records a status
// bit, drains what it issued, frees tensor memory and exits.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <cstring>

#include "wz_internal.cuh"
#include "wz_ptx.cuh"

namespace wz {

namespace {

constexpr int kXM = 128, kXK = 64;
constexpr int kXABytes = kXM * kXK * 2;             // 16 KB
constexpr int kXMaxStages = 8;
constexpr int kXGroups = 4;                         // K steps per ring stage (at most)
constexpr int kXMinStages = 2;
constexpr int kXThreads = 11 * 32;
constexpr int kXBStages = 2;                        // query-row stages (their own ring)
constexpr int kXAccCols = 256;
constexpr uint64_t kXTimeoutNs = 2000000000ull;
constexpr int kXReaders = 8;                        // channel-sum warps reading each stage

struct XShared {
    uint64_t full[kXMaxStages];    // feature ring
    uint64_t empty[kXMaxStages];
    uint64_t bfull[kXBStages];     // query-row ring
    uint64_t bempty[kXBStages];
    uint64_t tfull[2], tempty[2];
    uint64_t csync[2];
    uint64_t drain;
    uint32_t tmem_base;
    int abort;
    float npart[2][kXReaders][kXM];   // per channel-sum warp: squares of its channels, per row
};

struct XMaps {
    CUtensorMap a, b;
};

struct XArgs {
    int stages, stage_stride;   // feature ring: stages and bytes per stage (G A tiles)
    int b_off, b_stride;        // query-row ring (kXBStages stages of G B tiles): byte offset, bytes per stage
    int Lq, Lqp;
    int acc_off;                // byte offset of the two channel-sum buffers (2 x D floats)
    int shared_off;             // byte offset of XShared
};

__device__ __forceinline__ void xfail(const Ctx &c, volatile int *abort_flag, int code) {
    *abort_flag = 1;
    atomicOr(c.status, code);
}

// Token tile `it` of this CTA: first token and valid rows.
__device__ __forceinline__ void xtile(const Ctx &c, int it, int64_t &base, int &nr) {
    const int64_t total = (int64_t)c.T * c.N;
    const int64_t beg = (int64_t)blockIdx.x * c.L1;
    const int64_t end = min(total, beg + c.L1);
    base = beg + (int64_t)it * kXM;
    nr = (int)min((int64_t)kXM, end - base);
}

__device__ __forceinline__ int xtiles(const Ctx &c) {
    const int64_t total = (int64_t)c.T * c.N;
    const int64_t beg = (int64_t)blockIdx.x * c.L1;
    const int64_t end = min(total, beg + c.L1);
    return beg < end ? (int)((end - beg + kXM - 1) / kXM) : 0;
}

// The channel sums of this warp's 8 channels of every K step (acc), to the
// partial slot of frame f, then acc cleared: lane group lane / 8 takes every
// fourth K step.
__device__ __forceinline__ void xflush(const Ctx &c, float *acc, int64_t f, int ch_lo, int lane) {
    float *dst = c.part + ((size_t)blockIdx.x + (size_t)f) * c.D;
    for (int k0 = (lane >> 3) * kXK; k0 < c.D; k0 += 4 * kXK) {
        const int ch = k0 + ch_lo + (lane & 7);
        if (wz_in_range(c.status, (int64_t)blockIdx.x + f < (int64_t)c.G1 + c.T)) dst[ch] = acc[ch];
        acc[ch] = 0.f;
    }
}

}  // namespace

template <int G>   // K steps per ring stage
__global__ void __launch_bounds__(kXThreads, 1) maxsim_pass_kernel(const __grid_constant__ XMaps maps, Ctx c, XArgs p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *ring = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const size_t ring_off = (size_t)(ring - smem_raw);
    float *acc_buf = reinterpret_cast<float *>(ring + p.acc_off);
    XShared *S = reinterpret_cast<XShared *>(ring + p.shared_off);
    volatile int *abort_flag = &S->abort;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < p.stages; ++s) {
            ptx::mbar_init(&S->full[s], 1);
            ptx::mbar_init(&S->empty[s], 1 + kXReaders);
        }
        for (int s = 0; s < kXBStages; ++s) {
            ptx::mbar_init(&S->bfull[s], 1);
            ptx::mbar_init(&S->bempty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            ptx::mbar_init(&S->tfull[b], 1);
            ptx::mbar_init(&S->tempty[b], 4);
            ptx::mbar_init(&S->csync[b], kXReaders);
        }
        ptx::mbar_init(&S->drain, 1);
        S->abort = 0;
        ptx::fence_barrier_init();
        ptx::fence_proxy_async_smem();
    }
    if (warp == 1) {
        ptx::tmem_alloc(&S->tmem_base, 2 * kXAccCols);
        ptx::tmem_relinquish();
    }
    if (warp == 0 && lane == 0) {
        ptx::prefetch_tmap(&maps.a);
        ptx::prefetch_tmap(&maps.b);
    }
    // channel sums start at zero (shared memory only: before the wait)
    for (int k = threadIdx.x; k < 2 * c.D; k += blockDim.x) acc_buf[k] = 0.f;
    pdl_wait();   // the query rows come from the previous grid
    pdl_trigger();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem = S->tmem_base;
    const int ntile = xtiles(c);
    const int KS = c.D / kXK;

    if (warp == 0 && lane == 0) {
        // ---------------- TMA producer: features ----------------
        const uint64_t pol_a = ptx::policy_evict_first();
        const uint32_t stage_bytes = (uint32_t)G * (uint32_t)kXABytes;
        int stage = 0;
        uint32_t phase = 0;
        int issued_parity[kXMaxStages];
        for (int s = 0; s < kXMaxStages; ++s) issued_parity[s] = -1;
        for (int it = 0; it < ntile && !*abort_flag; ++it) {
            int64_t base;
            int nr;
            xtile(c, it, base, nr);
            bool ok = true;
            for (int ks = 0; ks < KS; ks += G) {
                if (!ptx::mbar_wait(&S->empty[stage], phase ^ 1u, kXTimeoutNs)) {
                    xfail(c, abort_flag, 16);
                    ok = false;
                    break;
                }
                uint8_t *st = ring + (size_t)stage * p.stage_stride;
                ptx::mbar_arrive_expect_tx(&S->full[stage], stage_bytes);
                ptx::tma_load_3d(st, &maps.a, &S->full[stage], 0, (int)base, ks, pol_a);
                issued_parity[stage] = (int)phase;
                if (++stage == p.stages) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
            if (!ok) break;
        }
        for (int s = 0; s < p.stages; ++s)
            if (issued_parity[s] >= 0) ptx::mbar_wait(&S->full[s], (uint32_t)issued_parity[s], kXTimeoutNs);
    } else if (warp == 10 && lane == 0) {
        // ---------------- TMA producer: query rows (from L2), K step by K step ----------------
        const uint64_t pol_b = ptx::policy_evict_last();
        const uint32_t stage_bytes = (uint32_t)G * 2u * (uint32_t)p.Lqp * kXK * 2u;
        int stage = 0;
        uint32_t phase = 0;
        int issued_parity[kXBStages];
        for (int s = 0; s < kXBStages; ++s) issued_parity[s] = -1;
        for (int it = 0; it < ntile && !*abort_flag; ++it) {
            bool ok = true;
            for (int ks = 0; ks < KS; ks += G) {
                if (!ptx::mbar_wait(&S->bempty[stage], phase ^ 1u, kXTimeoutNs)) {
                    xfail(c, abort_flag, 16);
                    ok = false;
                    break;
                }
                ptx::mbar_arrive_expect_tx(&S->bfull[stage], stage_bytes);
                ptx::tma_load_3d(ring + p.b_off + (size_t)stage * p.b_stride, &maps.b, &S->bfull[stage], 0, 0, ks,
                                 pol_b);
                issued_parity[stage] = (int)phase;
                if (++stage == kXBStages) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
            if (!ok) break;
        }
        for (int s = 0; s < kXBStages; ++s)
            if (issued_parity[s] >= 0) ptx::mbar_wait(&S->bfull[s], (uint32_t)issued_parity[s], kXTimeoutNs);
    } else if (warp == 1 && lane == 0) {
        // ---------------- MMA issuer ----------------
        const uint32_t idesc = ptx::idesc_bf16(kXM, 2 * p.Lqp, false, false);   // both K-major
        const uint32_t ring32 = ptx::smem_u32(ring);
        const uint64_t a_base = ptx::smem_desc(ring32, 16, 1024, 2);              // 128-B swizzle
        const uint64_t b_base = ptx::smem_desc(ring32 + (uint32_t)p.b_off, 16, 1024, 2);
        const uint64_t b_sub = (uint64_t)((2 * p.Lqp * kXK * 2) >> 4);   // one K step of B
        const uint64_t stage_desc = (uint64_t)(p.stage_stride >> 4), bstage_desc = (uint64_t)(p.b_stride >> 4);
        int stage = 0, bstage = 0;
        uint32_t phase = 0, bphase = 0;
        for (int it = 0; it < ntile && !*abort_flag; ++it) {
            const int b = it & 1;
            const uint32_t use = (uint32_t)(it >> 1);
            if (!ptx::mbar_wait(&S->tempty[b], (use & 1u) ^ 1u, kXTimeoutNs)) {
                xfail(c, abort_flag, 16);
                break;
            }
            ptx::tc_fence_after();
            const uint32_t d = tmem + (uint32_t)(b * kXAccCols);
            bool ok = true;
            for (int ks = 0; ks < KS; ks += G) {
                if (!ptx::mbar_wait(&S->full[stage], phase, kXTimeoutNs) ||
                    !ptx::mbar_wait(&S->bfull[bstage], bphase, kXTimeoutNs)) {
                    xfail(c, abort_flag, 16);
                    ok = false;
                    break;
                }
                ptx::tc_fence_after();
                const uint64_t so = (uint64_t)stage * stage_desc, sbo = (uint64_t)bstage * bstage_desc;
#pragma unroll
                for (int g = 0; g < G; ++g) {
                    const uint64_t ao = so + (uint64_t)g * (kXABytes >> 4), bo = sbo + (uint64_t)g * b_sub;
#pragma unroll
                    for (int k = 0; k < kXK / 16; ++k)   // K = 16 per MMA: 32 bytes along the swizzled row
                        ptx::mma_bf16(d, a_base + ao + (uint64_t)(2 * k), b_base + bo + (uint64_t)(2 * k), idesc,
                                      (ks | g | k) ? 1u : 0u);
                }
                ptx::mma_commit(&S->empty[stage]);
                ptx::mma_commit(&S->bempty[bstage]);
                if (++stage == p.stages) {
                    stage = 0;
                    phase ^= 1u;
                }
                if (++bstage == kXBStages) {
                    bstage = 0;
                    bphase ^= 1u;
                }
            }
            if (!ok) break;
            ptx::mma_commit(&S->tfull[b]);
        }
        ptx::mma_commit(&S->drain);
        ptx::mbar_wait(&S->drain, 0, kXTimeoutNs);
    } else if (warp >= 2 && warp < 10) {
        // ---------------- channel sums and token norms (warps 2-9), a_{t,n} (warps 2-5) ----------------
        // lane: channel pair p4 of this warp's 8 channels of a K step, and the
        // rows r = 8 i + re (i < 16) of the tile it sums.  With the 128-byte
        // swizzle (16-byte chunk k of row r at r * 128 + ((k ^ (r & 7)) << 4))
        // every one of those rows has r & 7 = re, so the lane's words sit at
        // lane_off + 1024 i (the eight values of re put the 32 lanes on 32
        // banks).  Warps 2-5 then take the tile's a_{t,n} for the rows of
        // their tensor-memory lane quadrant.
        const int wsel = warp - 2;
        const bool epi = warp < 6;
        const int p4 = lane & 3, re = lane >> 2;
        const int cw = wsel * 8 + 2 * p4;               // channels cw, cw + 1 of the K step
        const uint32_t lane_off = (uint32_t)(re * 128) + ((uint32_t)(wsel ^ re) << 4) + (uint32_t)(4 * p4);
        float *acc_open = acc_buf, *acc_next = acc_buf + c.D;
        int64_t open_f = ntile > 0 ? ((int64_t)blockIdx.x * c.L1) / c.N : 0;
        bool open_has = false;
        int stage = 0;
        uint32_t phase = 0;
        for (int it = 0; it < ntile && !*abort_flag; ++it) {
            int64_t base;
            int nr;
            xtile(c, it, base, nr);
            // a frame starts inside the tile at row rb (frames have >= 128 tokens)
            const int to_end = (int)((int64_t)c.N - base % c.N);
            const int rb = to_end < nr ? to_end : nr;
            const bool whole = rb == kXM;   // every row of the tile in the open frame
            float sq[16];                   // squares of this lane's two channels, row 8 i + re
#pragma unroll
            for (int i = 0; i < 16; ++i) sq[i] = 0.f;
            bool ok = true;
            for (int ks = 0; ks < KS; ks += G) {
                if (!ptx::mbar_wait(&S->full[stage], phase, kXTimeoutNs)) {
                    xfail(c, abort_flag, 32);
                    ok = false;
                    break;
                }
                // (indexed from the shared array itself: shared-memory loads)
                const uint8_t *st0 = smem_raw + ring_off + (size_t)stage * p.stage_stride;
#pragma unroll
                for (int g = 0; g < G; ++g) {
                    const uint8_t *lb = st0 + g * kXABytes + lane_off;
                    float s0x = 0.f, s0y = 0.f, s1x = 0.f, s1y = 0.f;
                    if (whole) {
                        // even and odd rows in two sums each (shorter dependent chains)
#pragma unroll
                        for (int i = 0; i < 16; ++i) {
                            const uint32_t wv = *reinterpret_cast<const uint32_t *>(lb + 1024 * i);
                            const float x = __uint_as_float(wv << 16), y = __uint_as_float(wv & 0xffff0000u);
                            sq[i] = fmaf(x, x, fmaf(y, y, sq[i]));
                            if (i & 1) {
                                s1x += x;
                                s1y += y;
                            } else {
                                s0x += x;
                                s0y += y;
                            }
                        }
                        s0x += s1x;
                        s0y += s1y;
                        s1x = s1y = 0.f;
                    } else {
#pragma unroll
                        for (int i = 0; i < 16; ++i) {
                            const int r = 8 * i + re;
                            const uint32_t wv = *reinterpret_cast<const uint32_t *>(lb + 1024 * i);
                            const float x = __uint_as_float(wv << 16), y = __uint_as_float(wv & 0xffff0000u);
                            sq[i] = fmaf(x, x, fmaf(y, y, sq[i]));
                            if (r < rb) {
                                s0x += x;
                                s0y += y;
                            } else if (r < nr) {
                                s1x += x;
                                s1y += y;
                            }
                        }
                    }
                    if (g == G - 1) {   // the stage's last K step is in registers: hand the stage back
                        __syncwarp();
                        if (lane == 0) ptx::mbar_arrive(&S->empty[stage]);
                    }
#pragma unroll
                    for (int o = 4; o < 32; o <<= 1) {   // the eight row classes, in a fixed order
                        s0x += __shfl_xor_sync(0xffffffffu, s0x, o);
                        s0y += __shfl_xor_sync(0xffffffffu, s0y, o);
                        s1x += __shfl_xor_sync(0xffffffffu, s1x, o);
                        s1y += __shfl_xor_sync(0xffffffffu, s1y, o);
                    }
                    if (re == 0) {
                        const int ch = (ks + g) * kXK + cw;
                        acc_open[ch] += s0x;
                        acc_open[ch + 1] += s0y;
                        if (rb < nr) {
                            acc_next[ch] += s1x;
                            acc_next[ch + 1] += s1y;
                        }
                    }
                }
                if (++stage == p.stages) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
            if (!ok) break;
            // token norms: this warp's squares summed over its 4 channel pairs,
            // one partial per warp and row
            const int b = it & 1;
            const uint32_t use = (uint32_t)(it >> 1);
#pragma unroll
            for (int i = 0; i < 16; ++i) {
                float v = sq[i];
                v += __shfl_xor_sync(0xffffffffu, v, 1);
                v += __shfl_xor_sync(0xffffffffu, v, 2);
                if (p4 == 0) S->npart[b][wsel][8 * i + re] = v;
            }
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&S->csync[b]);
            open_has = true;
            if (rb < nr) {   // the open frame ended inside the tile
                xflush(c, acc_open, open_f, wsel * 8, lane);
                float *t = acc_open;
                acc_open = acc_next;
                acc_next = t;
                ++open_f;
            }
            if ((base + nr) % c.N == 0) {   // and the frame open now ends with the tile
                __syncwarp();
                xflush(c, acc_open, open_f, wsel * 8, lane);
                ++open_f;
                open_has = false;
            }
            __syncwarp();
            if (epi) {
                // a_{t,n} of the rows of this warp's lane quadrant: the eight
                // warps' partial squares in a fixed order, then the max over
                // the query rows of hi + lo from tensor memory
                if (!ptx::mbar_wait(&S->csync[b], use & 1u, kXTimeoutNs) ||
                    !ptx::mbar_wait(&S->tfull[b], use & 1u, kXTimeoutNs)) {
                    xfail(c, abort_flag, 32);
                    break;
                }
                ptx::tc_fence_after();
                const int q = warp & 3;                  // TMEM lane quadrant: rows q*32 .. q*32+31
                const int row = q * 32 + lane;
                float t2 = 0.f;
#pragma unroll
                for (int w = 0; w < kXReaders; ++w) t2 += S->npart[b][w][row];
                const float nrm = sqrtf(t2);
                const uint32_t tbase = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(b * kXAccCols);
                float best = -INFINITY;
                for (int c0 = 0; c0 < p.Lqp; c0 += 16) {
                    uint32_t hi[16], lo[16];
                    ptx::tmem_ld_32x32b_x16(tbase + (uint32_t)c0, hi);
                    ptx::tmem_ld_32x32b_x16(tbase + (uint32_t)(p.Lqp + c0), lo);
                    ptx::tmem_ld_wait();
                    ptx::reg_fence16(hi);
                    ptx::reg_fence16(lo);
#pragma unroll
                    for (int j = 0; j < 16; ++j)
                        if (c0 + j < p.Lq) best = fmaxf(best, __uint_as_float(hi[j]) + __uint_as_float(lo[j]));
                }
                if (row < nr && wz_in_range(c.status, base + row < (int64_t)c.T * c.N))
                    c.a[base + row] = nrm > 0.f ? best / nrm : 0.f;
                ptx::tc_fence_before();
                __syncwarp();
                if (lane == 0) ptx::mbar_arrive(&S->tempty[b]);
            }
        }
        if (open_has && !*abort_flag) xflush(c, acc_open, open_f, wsel * 8, lane);   // the CTA's share of it
    }
    __syncthreads();
    if (warp == 1) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem, 2 * kXAccCols);
    }
}

namespace {

// [rows][cols] bf16 as {64 channels, rows, cols / 64 K steps}: box {64,
// box_rows, G}, i.e. G consecutive K-step tiles of box_rows rows.
bool xencode(PFN_cuTensorMapEncodeTiled_v12000 enc, CUtensorMap *m, const void *base, int64_t rows, int cols,
             int box_rows, int G) {
    cuuint64_t dims[3] = {(cuuint64_t)kXK, (cuuint64_t)rows, (cuuint64_t)(cols / kXK)};
    cuuint64_t strides[2] = {(cuuint64_t)cols * 2, (cuuint64_t)kXK * 2};
    cuuint32_t box[3] = {(cuuint32_t)kXK, (cuuint32_t)box_rows, (cuuint32_t)G};
    cuuint32_t es[3] = {1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(base), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

struct XLayout {
    int stages, stride, G, b_off, b_stride, acc_off, shared_off;
    size_t smem;
};

// K steps per stage: the most of kXGroups (dividing the D / 64 K steps)
// that leaves kXMinStages feature stages beside the kXBStages query-row
// stages.
XLayout xlayout(int D, int Lqp) {
    XLayout L{};
    const size_t fixed = 1024 + (size_t)2 * D * 4 + (sizeof(XShared) + 127) / 128 * 128;
    const size_t cap = 227 * 1024;
    for (int G = kXGroups; G >= 1; G >>= 1) {
        if ((D / kXK) % G != 0) continue;
        L.G = G;
        L.stride = G * kXABytes;
        L.b_stride = G * 2 * Lqp * kXK * 2;   // multiples of 1 KB (2 Lqp % 16 == 0)
        const size_t used = fixed + (size_t)kXBStages * L.b_stride;
        L.stages = used < cap ? (int)((cap - used) / (size_t)L.stride) : 0;
        if (L.stages >= kXMinStages) break;
    }
    if (L.stages > kXMaxStages) L.stages = kXMaxStages;
    L.b_off = L.stages * L.stride;
    L.acc_off = L.b_off + kXBStages * L.b_stride;
    L.shared_off = L.acc_off + 2 * D * 4;
    L.smem = 1024 + (size_t)L.shared_off + sizeof(XShared);
    return L;
}

}  // namespace

// The fused pass applies to one video with frames of at least 128 tokens,
// D a multiple of 64 up to 4096 and at most 128 query rows (Lqp <= 128).
bool maxsim_pass_supported(const Ctx &c, int Lqp) {
    if (c.V != 1 || c.N < kXM || c.D % kXK != 0 || c.D > 4096 || c.dtype != WZ_DTYPE_BF16) return false;
    if (Lqp < 16 || Lqp > 128 || Lqp % 16 != 0) return false;
    return xlayout(c.D, Lqp).stages >= 2;
}

cudaError_t launch_maxsim_pass(const Ctx &c, int Lq, int Lqp, cudaStream_t s) {
    if (!maxsim_pass_supported(c, Lqp) || Lq < 1 || Lq > Lqp) return cudaErrorInvalidValue;
    auto enc = tmap_encode_fn();
    if (!enc) return cudaErrorNotSupported;
    XMaps maps;
    memset(&maps, 0, sizeof(maps));
    const XLayout L = xlayout(c.D, Lqp);
    if (!xencode(enc, &maps.a, c.X, (int64_t)c.T * c.N, c.D, kXM, L.G) ||
        !xencode(enc, &maps.b, c.qhl, 2 * Lqp, c.D, 2 * Lqp, L.G))
        return cudaErrorInvalidValue;
    XArgs p{};
    p.stages = L.stages;
    p.stage_stride = L.stride;
    p.b_off = L.b_off;
    p.b_stride = L.b_stride;
    p.Lq = Lq;
    p.Lqp = Lqp;
    p.acc_off = L.acc_off;
    p.shared_off = L.shared_off;
    const void *fn = L.G == 4 ? (const void *)maxsim_pass_kernel<4>
                     : L.G == 2 ? (const void *)maxsim_pass_kernel<2>
                                : (const void *)maxsim_pass_kernel<1>;
    cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)L.smem);
    if (e != cudaSuccess) return e;
    void *args[] = {&maps, const_cast<Ctx *>(&c), &p};
    return launch_kernel(fn, dim3(c.G1), dim3(kXThreads), L.smem, s, args, c.pdl != 0);
}

}  // namespace wz
