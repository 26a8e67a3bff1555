// Condensed tokens Z_m = W_m X_m on the 5th-generation tensor cores
// (tcgen05.mma, TMA, tensor memory) -- the fused WSM + bilinear + pack step
// (Eq. 11-14, 16, 18) as one streaming pass over the features.
//
// Orientation: the MMA computes D[c][j] = sum_k X_m[k][c] * W_m[j][k] with
//   A = X tile, M = 128 channels, K = 16 tokens, MN-major (channels
//       contiguous, exactly as the features lie in HBM), loaded by TMA with
//       128-byte swizzle, box 64 channels x 32 tokens x 1 frame;
//   B = W tile, N = n (the frame's condensed tokens, <= 256 per unit, padded
//       to 16), K-major 8x8 core matrices without swizzle, stored in HBM in
//       exactly that order (tile_index) so one bulk copy moves a stage;
//   D = fp32 accumulators in tensor memory, 128 lanes x N columns per
//       128-channel tile.
// W_m is fp32 split into bf16 hi + lo (two MMAs into one accumulator), so the
// product keeps ~16 bits of W while X (exact in bf16) streams once.
//
// A unit of work is (frame, <= 256 output tokens, CG <= 4 channel tiles) over
// the 32-token chunks [kclo, kchi] its operator rows reach (every chunk unless
// a frame of more than 256 tokens is condensed in blocks); the rest of its
// operator rows are zero and are neither loaded nor multiplied.
// The cost of an MMA instruction hardly depends on N, so for N <= 128 the hi
// and lo operator halves (adjacent in shared memory) form one MMA of N = 2N
// whose accumulator holds the hi and lo products side by side; for larger N
// hi and lo are two MMAs into the same accumulator.  Every unit fits one of
// two 256-column accumulator buffers, so the epilogue of a unit overlaps the
// main loop of the next.  The epilogue transposes each warp's 32 channels x
// 32 tokens through shared memory and writes 16-byte rows.  One CTA per SM,
// persistent over the unit list:
//   warp 0     TMA producer (one thread), 5-stage shared-memory ring
//   warp 1     TMEM allocation and the MMA issuer (one thread)
//   warps 2-5  epilogue: tcgen05.ld -> bf16 -> packed output rows
// Every mbarrier wait is bounded; on a timeout the kernel records a status
// bit, drains what it issued, frees tensor memory and exits.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <cstring>

#include "wz_internal.cuh"
#include "wz_ptx.cuh"

namespace wz {

namespace {

constexpr int kKC = 32;                    // tokens per K chunk (two K=16 MMA steps)
constexpr int kStages = 5;
constexpr int kStageBytes = 40 * 1024;     // >= CG*8 KB (X) + 2*N*64 B (W hi, lo)
constexpr int kThreads = 192;
constexpr int kAccCols = 256;             // one of the two accumulator buffers
constexpr int kBufs = 2;
constexpr uint64_t kTimeoutNs = 2000000000ull;

struct TcShared {
    uint64_t full[kStages];
    uint64_t empty[kStages];
    uint64_t tfull[2];
    uint64_t tempty[2];
    uint64_t drain;
    uint32_t tmem_base;
    int abort;
    int vprefix[WZ_MAX_VIDEOS + 1];
};

constexpr int kEpiWarps = 4;
constexpr int kEpiBytes = 32 * 32 * 2;     // one warp's 32 channels x 32 tokens, bf16
constexpr size_t kSharedBytes = (sizeof(TcShared) + 127) / 128 * 128;   // epilogue tiles start 128-B aligned
constexpr size_t kSmemBytes = 1024 + (size_t)kStages * kStageBytes + kSharedBytes + kEpiWarps * kEpiBytes;
static_assert(kSmemBytes <= 227 * 1024, "shared memory of the condensation CTA");

// Feature tensor maps: a 4D view [frames][D/64][N][64] whose box covers all
// 2*CG 64-channel blocks of a stage in one copy (one map per CG), and the 3D
// view [frames][N][D] for D not a multiple of 64 (two copies per tile).
struct TcMaps {
    CUtensorMap x3;
    CUtensorMap x4[4];
    int use4;
};

struct Unit {
    int f, j0, ct0, nc, cg, kclo, kchi;   // operator chunks [kclo, kchi] (the rest are zero)
};

__device__ __forceinline__ Unit decode_unit(const Ctx &c, const int *vprefix, int u) {
    int lo = 0, hi = c.V - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (vprefix[mid] <= u) lo = mid;
        else hi = mid - 1;
    }
    const int4 q = c.units[(size_t)lo * c.max_units_v + (u - vprefix[lo])];
    Unit r;
    r.f = q.x;
    r.j0 = q.y;
    r.ct0 = q.z;
    r.nc = q.w & 0x1ff;
    r.cg = (q.w >> 9) & 7;
    r.kclo = (q.w >> 12) & 0xff;
    r.kchi = (q.w >> 20) & 0xff;
    return r;
}

__device__ __forceinline__ void fail(const Ctx &c, volatile int *abort_flag, int code) {
    *abort_flag = 1;
    atomicOr(c.status, code);
}

// The MMAs of one unit: stages kclo..kchi of kKC tokens, each two K = 16 steps over
// CG channel tiles (hi|lo fused into one MMA, or hi and lo as two).  The
// pattern is fixed at compile time and the stage descriptors are advanced by
// a constant, so the issuing thread spends a few instructions per MMA.
template <int CG, bool FUSED>
__device__ __forceinline__ bool mma_unit(TcShared *S, uint8_t *ring, const Ctx &c, volatile int *abort_flag, int kclo,
                                         int kchi,
                                         int &stage, uint32_t &phase, uint32_t dbase, int tcols, uint32_t idesc,
                                         int ncp) {
    const uint32_t ring32 = ptx::smem_u32(ring);
    // stage 0 descriptors; the 14-bit start-address field of stage s is
    // (ring + s * kStageBytes) >> 4, reached by adding to the descriptor
    const uint64_t a_base = ptx::smem_desc(ring32, 4096, 1024, 2);              // X: MN-major, 128-B swizzle
    const uint64_t b_base = ptx::smem_desc(ring32 + CG * 8192u, 128, 512, 0);  // W: K-major, no swizzle
    const uint64_t lo_off = (uint64_t)((ncp * 64) >> 4);
    constexpr uint64_t kStageDesc = (uint64_t)(kStageBytes >> 4);
    uint32_t d[CG];
#pragma unroll
    for (int ct = 0; ct < CG; ++ct) d[ct] = dbase + (uint32_t)(ct * tcols);
    for (int kc = kclo; kc <= kchi; ++kc) {
        if (!ptx::mbar_wait(&S->full[stage], phase, kTimeoutNs)) {
            fail(c, abort_flag, 4);
            return false;
        }
        ptx::tc_fence_after();
        const uint64_t so = (uint64_t)stage * kStageDesc;
        const uint64_t a0 = a_base + so, b0 = b_base + so;
        const uint32_t acc = kc > kclo ? 1u : 0u;
#pragma unroll
        for (int s = 0; s < 2; ++s) {
#pragma unroll
            for (int ct = 0; ct < CG; ++ct) {
                const uint64_t a = a0 + (uint64_t)((ct * 8192 + s * 2048) >> 4);
                ptx::mma_bf16(d[ct], a, b0 + (uint64_t)(s * 16), idesc, acc | (uint32_t)s);
                if (!FUSED) ptx::mma_bf16(d[ct], a, b0 + lo_off + (uint64_t)(s * 16), idesc, 1u);
            }
        }
        ptx::mma_commit(&S->empty[stage]);
        if (++stage == kStages) {
            stage = 0;
            phase ^= 1u;
        }
    }
    return true;
}

}  // namespace

__global__ void __launch_bounds__(kThreads, 1)
condense_tc_kernel(const __grid_constant__ TcMaps maps, Ctx c) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *ring = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    TcShared *S = reinterpret_cast<TcShared *>(ring + (size_t)kStages * kStageBytes);
    volatile int *abort_flag = &S->abort;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            ptx::mbar_init(&S->full[s], 1);
            ptx::mbar_init(&S->empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            ptx::mbar_init(&S->tfull[b], 1);
            ptx::mbar_init(&S->tempty[b], 4);
        }
        ptx::mbar_init(&S->drain, 1);
        S->abort = 0;
        ptx::fence_barrier_init();
        ptx::fence_proxy_async_smem();
    }
    if (warp == 1) {
        ptx::tmem_alloc(&S->tmem_base, kAccCols * kBufs);
        ptx::tmem_relinquish();
    }
    if (warp == 0 && lane == 0) {
        if (maps.use4)
            for (int g = 0; g < 4; ++g) ptx::prefetch_tmap(&maps.x4[g]);
        else
            ptx::prefetch_tmap(&maps.x3);
    }
    // global memory from here on: the previous grid has completed
    pdl_wait();
    pdl_trigger();
    if (threadIdx.x == 0) {
        int acc = 0;
        for (int v = 0; v < c.V; ++v) {
            S->vprefix[v] = acc;
            acc += c.ucount[v];
        }
        S->vprefix[c.V] = acc;
    }
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem = S->tmem_base;
    const int n_units = S->vprefix[c.V];
    const int KC = c.K_pad / kKC;

    if (warp == 0 && lane == 0) {
        // ---------------- TMA producer ----------------
        const uint64_t pol_x = ptx::policy_evict_first();
        const uint64_t pol_w = ptx::policy_evict_last();
        const char *whi = static_cast<const char *>(c.Wop);
        const char *wlo = whi + (size_t)c.w_rows * c.K_pad * 2;
        const size_t groups = (size_t)(c.w_rows >> 3);
        int stage = 0;
        uint32_t phase = 0;
        int issued_parity[kStages];
        for (int s = 0; s < kStages; ++s) issued_parity[s] = -1;
        for (int u = blockIdx.x; u < n_units && !*abort_flag; u += gridDim.x) {
            const Unit un = decode_unit(c, S->vprefix, u);
            const int ncp = (un.nc + 15) & ~15;
            const int64_t wrow0 = (int64_t)c.woff[un.f] + un.j0;     // multiple of 16
            const uint32_t bytes = (uint32_t)un.cg * 8192u + 2u * (uint32_t)ncp * 64u;
            if (un.kclo > un.kchi || un.kchi >= KC) {   // not a record the spatial kernel writes
                fail(c, abort_flag, 4);
                break;
            }
            bool ok = true;
            for (int kc = un.kclo; kc <= un.kchi; ++kc) {
                if (!ptx::mbar_wait(&S->empty[stage], phase ^ 1u, kTimeoutNs)) {
                    fail(c, abort_flag, 1);
                    ok = false;
                    break;
                }
                uint8_t *st = ring + (size_t)stage * kStageBytes;
                ptx::mbar_arrive_expect_tx(&S->full[stage], bytes);
                if (maps.use4) {
                    ptx::tma_load_4d(st, &maps.x4[un.cg - 1], &S->full[stage], 0, kc * kKC, 2 * un.ct0, un.f, pol_x);
                } else {
                    for (int ct = 0; ct < un.cg; ++ct)
                        for (int h = 0; h < 2; ++h)
                            ptx::tma_load_3d(st + ct * 8192 + h * 4096, &maps.x3, &S->full[stage],
                                             (un.ct0 + ct) * kTileC + h * 64, kc * kKC, un.f, pol_x);
                }
                uint8_t *wh = st + un.cg * 8192;
                const size_t toff = ((size_t)kc * groups + (size_t)(wrow0 >> 3)) * 512;
                ptx::bulk_load(wh, whi + toff, (uint32_t)ncp * 64u, &S->full[stage], pol_w);
                ptx::bulk_load(wh + ncp * 64, wlo + toff, (uint32_t)ncp * 64u, &S->full[stage], pol_w);
                issued_parity[stage] = (int)phase;
                if (++stage == kStages) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
            if (!ok) break;
        }
        // let every copy this thread issued land before the CTA can exit
        for (int s = 0; s < kStages; ++s)
            if (issued_parity[s] >= 0) ptx::mbar_wait(&S->full[s], (uint32_t)issued_parity[s], kTimeoutNs);
    } else if (warp == 1 && lane == 0) {
        // ---------------- MMA issuer ----------------
        int stage = 0;
        uint32_t phase = 0;
        int it = 0;
        for (int u = blockIdx.x; u < n_units && !*abort_flag; u += gridDim.x, ++it) {
            const Unit un = decode_unit(c, S->vprefix, u);
            const int ncp = (un.nc + 15) & ~15;
            const bool fused = ncp <= 128;             // hi|lo as one MMA of N = 2*ncp
            const int tcols = fused ? 2 * ncp : ncp;   // accumulator columns per tile
            const int b = it % kBufs;
            const uint32_t use = (uint32_t)(it / kBufs);
            if (!ptx::mbar_wait(&S->tempty[b], (use & 1u) ^ 1u, kTimeoutNs)) {
                fail(c, abort_flag, 2);
                break;
            }
            ptx::tc_fence_after();
            if (un.kclo > un.kchi || un.kchi >= KC) {
                fail(c, abort_flag, 4);
                break;
            }
            const uint32_t idesc = ptx::idesc_bf16(128, fused ? 2 * ncp : ncp, true, false);
            const uint32_t dbase = tmem + (uint32_t)(b * kAccCols);
            bool ok = false;
            if (fused) {
                switch (un.cg) {
                    case 1: ok = mma_unit<1, true>(S, ring, c, abort_flag, un.kclo, un.kchi, stage, phase, dbase, tcols, idesc, ncp); break;
                    case 2: ok = mma_unit<2, true>(S, ring, c, abort_flag, un.kclo, un.kchi, stage, phase, dbase, tcols, idesc, ncp); break;
                    case 3: ok = mma_unit<3, true>(S, ring, c, abort_flag, un.kclo, un.kchi, stage, phase, dbase, tcols, idesc, ncp); break;
                    case 4: ok = mma_unit<4, true>(S, ring, c, abort_flag, un.kclo, un.kchi, stage, phase, dbase, tcols, idesc, ncp); break;
                    default: fail(c, abort_flag, 4); break;
                }
            } else if (un.cg == 1) {
                ok = mma_unit<1, false>(S, ring, c, abort_flag, un.kclo, un.kchi, stage, phase, dbase, tcols, idesc, ncp);
            } else {
                fail(c, abort_flag, 4);
            }
            if (!ok) break;
            ptx::mma_commit(&S->tfull[b]);
        }
        // every MMA issued by this thread completes before tensor memory is freed
        ptx::mma_commit(&S->drain);
        ptx::mbar_wait(&S->drain, 0, kTimeoutNs);
    } else if (warp >= 2) {
        // ---------------- epilogue ----------------
        const int q = warp & 3;                          // TMEM lane quadrant of this warp
        uint8_t *tr = reinterpret_cast<uint8_t *>(S) + kSharedBytes + (size_t)(warp - 2) * kEpiBytes;
        const uint32_t tr32 = ptx::smem_u32(tr);
        char *out = static_cast<char *>(c.out);
        const size_t rowb = (size_t)c.D * 2;
        int it = 0;
        for (int u = blockIdx.x; u < n_units && !*abort_flag; u += gridDim.x, ++it) {
            const Unit un = decode_unit(c, S->vprefix, u);
            const int ncp = (un.nc + 15) & ~15;
            const bool fused = ncp <= 128;
            const int tcols = fused ? 2 * ncp : ncp;
            const int b = it % kBufs;
            const uint32_t use = (uint32_t)(it / kBufs);
            if (!ptx::mbar_wait(&S->tfull[b], use & 1u, kTimeoutNs)) {
                fail(c, abort_flag, 8);
                break;
            }
            ptx::tc_fence_after();
            const size_t row0 = (size_t)c.off[un.f] + un.j0;
            const uint32_t tbase = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(b * kAccCols);
            for (int ct = 0; ct < un.cg; ++ct) {
                const int ch0 = (un.ct0 + ct) * kTileC + q * 32;          // this warp's 32 channels
                for (int j0 = 0; j0 < ncp; j0 += 32) {
                    // lane = channel ch0 + lane, registers = tokens j0 .. j0+31
                    uint32_t v[32];
                    {
                        uint32_t h0[16], h1[16];
                        const uint32_t col = (uint32_t)(ct * tcols + j0);
                        ptx::tmem_ld_32x32b_x16(tbase + col, h0);
                        if (j0 + 16 < ncp) ptx::tmem_ld_32x32b_x16(tbase + col + 16, h1);
                        if (fused) {
                            uint32_t l0[16], l1[16];
                            ptx::tmem_ld_32x32b_x16(tbase + col + (uint32_t)ncp, l0);
                            if (j0 + 16 < ncp) ptx::tmem_ld_32x32b_x16(tbase + col + (uint32_t)ncp + 16, l1);
                            ptx::tmem_ld_wait();
#pragma unroll
                            for (int j = 0; j < 16; ++j) {
                                v[j] = __float_as_uint(__uint_as_float(h0[j]) + __uint_as_float(l0[j]));
                                v[16 + j] = (j0 + 16 < ncp) ? __float_as_uint(__uint_as_float(h1[j]) + __uint_as_float(l1[j])) : 0u;
                            }
                        } else {
                            ptx::tmem_ld_wait();
#pragma unroll
                            for (int j = 0; j < 16; ++j) {
                                v[j] = h0[j];
                                v[16 + j] = (j0 + 16 < ncp) ? h1[j] : 0u;
                            }
                        }
                    }
                    // transpose: row t of the tile = 32 channels of token j0 + t
                    __syncwarp();
#pragma unroll
                    for (int j = 0; j < 32; ++j) {
                        const __nv_bfloat16 bv = __float2bfloat16_rn(__uint_as_float(v[j]));
                        asm volatile("st.shared.b16 [%0], %1;" ::"r"(tr32 + (uint32_t)(j * 64 + lane * 2)),
                                     "h"(*reinterpret_cast<const unsigned short *>(&bv)));
                    }
                    __syncwarp();
                    // 16-byte pieces: 4 per token row, 8 tokens per warp instruction
#pragma unroll
                    for (int r = 0; r < 4; ++r) {
                        const int t = r * 8 + (lane >> 2);
                        const int cc = (lane & 3) * 8;
                        if (j0 + t < un.nc && ch0 + cc < c.D &&
                            wz_in_range(c.status, (int64_t)(row0 + j0 + t) < c.rows_total)) {
                            const uint4 val = ptx::lds128(tr32 + (uint32_t)(t * 64 + cc * 2));
                            *reinterpret_cast<uint4 *>(out + (row0 + j0 + t) * rowb + (size_t)(ch0 + cc) * 2) = val;
                        }
                    }
                }
            }
            ptx::tc_fence_before();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&S->tempty[b]);
        }
    }
    __syncthreads();
    if (warp == 1) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem, kAccCols * kBufs);
    }
}

namespace {

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    if (!fn) {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    }
    return fn;
}

}  // namespace

bool tensor_path_available() { return true; }

cudaError_t launch_condense_tc(const Ctx &c, cudaStream_t s) {
    auto enc = encode_fn();
    if (!enc) return cudaErrorNotSupported;
    if (c.dtype != WZ_DTYPE_BF16 || c.rows_total < 1) return cudaErrorInvalidValue;
    TcMaps maps;
    memset(&maps, 0, sizeof(maps));
    void *X = const_cast<void *>(c.X);
    const cuuint64_t frames = (cuuint64_t)c.V * c.T;
    {
        cuuint64_t dims[3] = {(cuuint64_t)c.D, (cuuint64_t)c.N, frames};
        cuuint64_t strides[2] = {(cuuint64_t)c.D * 2, (cuuint64_t)c.N * c.D * 2};
        cuuint32_t box[3] = {64, (cuuint32_t)kKC, 1};
        cuuint32_t es[3] = {1, 1, 1};
        if (enc(&maps.x3, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, X, dims, strides, box, es,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return cudaErrorInvalidValue;
    }
    maps.use4 = 0;
    if (c.D % 64 == 0) {
        cuuint64_t dims[4] = {64, (cuuint64_t)c.N, (cuuint64_t)(c.D / 64), frames};
        cuuint64_t strides[3] = {(cuuint64_t)c.D * 2, 128, (cuuint64_t)c.N * c.D * 2};
        cuuint32_t es[4] = {1, 1, 1, 1};
        bool ok = true;
        for (int g = 0; g < 4 && ok; ++g) {
            cuuint32_t box[4] = {64, (cuuint32_t)kKC, (cuuint32_t)(2 * (g + 1)), 1};
            ok = enc(&maps.x4[g], CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, X, dims, strides, box, es,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
        }
        maps.use4 = ok ? 1 : 0;
    }
    int dev = 0, sms = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(condense_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes);
    if (e != cudaSuccess) return e;
    void *args[] = {&maps, const_cast<Ctx *>(&c)};
    return launch_kernel((const void *)condense_tc_kernel, dim3(sms), dim3(kThreads), kSmemBytes, s, args,
                         c.pdl != 0);
}

}  // namespace wz
