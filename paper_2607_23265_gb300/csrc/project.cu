// Projector P of Eq. 17 on the condensed tokens: P(Z) = GELU(Z W1^T + b1) W2^T + b2,
// two bf16 GEMMs with fp32 accumulation on the 5th-generation tensor cores,
// each with a fused bias + activation epilogue:
//
//   Out[m][n] = act(sum_k A[m][k] B[n][k] + bias[n]),   A [M][K], B [N][K] bf16
//
// (B is a torch.nn.Linear weight, out x in).  Tiles of 128 x 256 (M x N) with
// K steps of 64: both operands K-major with 128-byte swizzle, one 2D TMA box
// per operand per step ({64, 128} and {64, 256}), a 4-stage ring of 48 KB;
// fp32 accumulators in TMEM (two buffers of 256 columns) so the epilogue of a
// tile overlaps the main loop of the next.  Persistent CTAs walk the tiles
// m-major, so CTAs that run at the same time share the A rows in L2 and the
// weights stay L2-resident.
//   warp 0     TMA producer (one thread)
//   warp 1     TMEM allocation and the MMA issuer (one thread)
//   warps 2-5  epilogue: tcgen05.ld (TMEM lane = row m, columns = n) -> + bias
//              -> activation -> bf16 -> 16-byte stores of contiguous row pieces
// The same kernel with a row-max epilogue computes the max-over-query
// relevance: the token x query-row cosines (B = the normalised query rows as
// bf16 hi and lo halves, N = 2 Lqp), maximum over the rows per token.
// Every mbarrier wait is bounded; on a timeout the kernel records a status
// bit, drains what it issued, frees tensor memory and exits.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <cstring>

#include "wz_internal.cuh"
#include "wz_ptx.cuh"

namespace wz {

namespace {

constexpr int kPM = 128, kPN = 256, kPK = 64;
constexpr int kPStages = 4;                          // projector ring (48 KB stages)
constexpr int kPMaxStages = 8;                       // smaller stages of the row-max GEMM
constexpr int kPABytes = kPM * kPK * 2;             // 16 KB
constexpr int kPBBytes = kPN * kPK * 2;             // 32 KB
constexpr int kPStageBytes = kPABytes + kPBBytes;
constexpr int kPThreads = 192;
constexpr int kPAccCols = 256;
constexpr uint64_t kPTimeoutNs = 2000000000ull;

struct PShared {
    uint64_t full[kPMaxStages];
    uint64_t empty[kPMaxStages];
    uint64_t tfull[2];
    uint64_t tempty[2];
    uint64_t drain;
    uint32_t tmem_base;
    int abort;
};

constexpr size_t kPSmemBytes = 1024 + (size_t)kPStages * kPStageBytes + sizeof(PShared);
static_assert(kPSmemBytes <= 227 * 1024, "shared memory of the projector CTA");

struct PMaps {
    CUtensorMap a, b;
};

struct PArgs {
    int M, N, K;
    int tileN;           // MMA N of a tile (<= 256, multiple of 32); the B box height
    int stages;          // ring stages (<= kPMaxStages, stages * stage_stride <= the ring)
    int stage_stride;    // bytes per stage: (kPM + tileN) * kPK * 2 rounded to 1 KB
    // epilogue 0 (projector): out = act(acc + bias)
    const float *bias;   // [N] or null
    __nv_bfloat16 *out;  // [M][N]
    int gelu;            // 1: exact GELU after the bias
    // epilogue 1 (max-over-query relevance): columns [0, Lqp) and [Lqp, 2 Lqp)
    // hold the hi and lo parts of the dots with the normalised query rows;
    // a[m] = max_{j < Lq} (hi_j + lo_j) / a[m] (a[m] holds ||u_m|| on entry)
    float *a;
    int Lq, Lqp;
    int *status;
};

__device__ __forceinline__ void pfail(const PArgs &p, volatile int *abort_flag, int code) {
    *abort_flag = 1;
    if (p.status) atomicOr(p.status, code);
}

}  // namespace

template <int EPI>
__global__ void __launch_bounds__(kPThreads, 1)
project_gemm_kernel(const __grid_constant__ PMaps maps, PArgs p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *ring = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    PShared *S = reinterpret_cast<PShared *>(ring + (size_t)kPStages * kPStageBytes);
    volatile int *abort_flag = &S->abort;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < p.stages; ++s) {
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
        ptx::tmem_alloc(&S->tmem_base, 2 * kPAccCols);
        ptx::tmem_relinquish();
    }
    if (warp == 0 && lane == 0) {
        ptx::prefetch_tmap(&maps.a);
        ptx::prefetch_tmap(&maps.b);
    }
    pdl_wait();   // A may be the previous grid's output
    pdl_trigger();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem = S->tmem_base;
    const int mt = (p.M + kPM - 1) / kPM, nt = (p.N + p.tileN - 1) / p.tileN;
    const int tiles = mt * nt;
    const int KS = p.K / kPK;

    if (warp == 0 && lane == 0) {
        // ---------------- TMA producer ----------------
        const uint64_t pol_a = ptx::policy_evict_first();
        const uint64_t pol_b = ptx::policy_evict_last();
        int stage = 0;
        uint32_t phase = 0;
        int issued_parity[kPMaxStages];
        for (int s = 0; s < kPMaxStages; ++s) issued_parity[s] = -1;
        for (int t = blockIdx.x; t < tiles && !*abort_flag; t += gridDim.x) {
            const int m0 = (t / nt) * kPM, n0 = (t % nt) * p.tileN;
            const uint32_t stage_bytes = (uint32_t)(kPM + p.tileN) * kPK * 2;
            bool ok = true;
            for (int ks = 0; ks < KS; ++ks) {
                if (!ptx::mbar_wait(&S->empty[stage], phase ^ 1u, kPTimeoutNs)) {
                    pfail(p, abort_flag, 1);
                    ok = false;
                    break;
                }
                uint8_t *st = ring + (size_t)stage * p.stage_stride;
                ptx::mbar_arrive_expect_tx(&S->full[stage], stage_bytes);
                ptx::tma_load_2d(st, &maps.a, &S->full[stage], ks * kPK, m0, pol_a);
                ptx::tma_load_2d(st + kPABytes, &maps.b, &S->full[stage], ks * kPK, n0, pol_b);
                issued_parity[stage] = (int)phase;
                if (++stage == p.stages) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
            if (!ok) break;
        }
        for (int s = 0; s < p.stages; ++s)
            if (issued_parity[s] >= 0) ptx::mbar_wait(&S->full[s], (uint32_t)issued_parity[s], kPTimeoutNs);
    } else if (warp == 1 && lane == 0) {
        // ---------------- MMA issuer ----------------
        const uint32_t idesc = ptx::idesc_bf16(kPM, p.tileN, false, false);   // both K-major
        const uint32_t ring32 = ptx::smem_u32(ring);
        const uint64_t a_base = ptx::smem_desc(ring32, 16, 1024, 2);              // 128-B swizzle
        const uint64_t b_base = ptx::smem_desc(ring32 + kPABytes, 16, 1024, 2);
        const uint64_t stage_desc = (uint64_t)(p.stage_stride >> 4);
        int stage = 0;
        uint32_t phase = 0;
        int it = 0;
        for (int t = blockIdx.x; t < tiles && !*abort_flag; t += gridDim.x, ++it) {
            const int b = it & 1;
            const uint32_t use = (uint32_t)(it >> 1);
            if (!ptx::mbar_wait(&S->tempty[b], (use & 1u) ^ 1u, kPTimeoutNs)) {
                pfail(p, abort_flag, 2);
                break;
            }
            ptx::tc_fence_after();
            const uint32_t d = tmem + (uint32_t)(b * kPAccCols);
            bool ok = true;
            for (int ks = 0; ks < KS; ++ks) {
                if (!ptx::mbar_wait(&S->full[stage], phase, kPTimeoutNs)) {
                    pfail(p, abort_flag, 4);
                    ok = false;
                    break;
                }
                ptx::tc_fence_after();
                const uint64_t so = (uint64_t)stage * stage_desc;
#pragma unroll
                for (int k = 0; k < kPK / 16; ++k)   // K = 16 per MMA: 32 bytes along the swizzled row
                    ptx::mma_bf16(d, a_base + so + (uint64_t)(2 * k), b_base + so + (uint64_t)(2 * k), idesc,
                                  (ks | k) ? 1u : 0u);
                ptx::mma_commit(&S->empty[stage]);
                if (++stage == p.stages) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
            if (!ok) break;
            ptx::mma_commit(&S->tfull[b]);
        }
        ptx::mma_commit(&S->drain);
        ptx::mbar_wait(&S->drain, 0, kPTimeoutNs);
    } else if (warp >= 2) {
        // ---------------- epilogue ----------------
        const int q = warp & 3;                      // TMEM lane quadrant: rows q*32 .. q*32+31
        int it = 0;
        for (int t = blockIdx.x; t < tiles && !*abort_flag; t += gridDim.x, ++it) {
            const int b = it & 1;
            const uint32_t use = (uint32_t)(it >> 1);
            if (!ptx::mbar_wait(&S->tfull[b], use & 1u, kPTimeoutNs)) {
                pfail(p, abort_flag, 8);
                break;
            }
            ptx::tc_fence_after();
            const int m0 = (t / nt) * kPM, n0 = (t % nt) * p.tileN;
            const int row = m0 + q * 32 + lane;
            const uint32_t tbase = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(b * kPAccCols);
            if constexpr (EPI == 1) {
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
                if (row < p.M) {
                    const float nrm = p.a[row];
                    p.a[row] = nrm > 0.f ? best / nrm : 0.f;
                }
            } else
            for (int c0 = 0; c0 < kPN && n0 + c0 < p.N; c0 += 32) {
                uint32_t v0[16], v1[16];
                ptx::tmem_ld_32x32b_x16(tbase + (uint32_t)c0, v0);
                ptx::tmem_ld_32x32b_x16(tbase + (uint32_t)c0 + 16, v1);
                ptx::tmem_ld_wait();
                ptx::reg_fence16(v0);
                ptx::reg_fence16(v1);
                float x[32];
#pragma unroll
                for (int j = 0; j < 16; ++j) {
                    x[j] = __uint_as_float(v0[j]);
                    x[16 + j] = __uint_as_float(v1[j]);
                }
                if (p.bias) {
                    const float4 *bb = reinterpret_cast<const float4 *>(p.bias + n0 + c0);
#pragma unroll
                    for (int j = 0; j < 8; ++j) {
                        const float4 v = __ldg(bb + j);
                        x[4 * j] += v.x;
                        x[4 * j + 1] += v.y;
                        x[4 * j + 2] += v.z;
                        x[4 * j + 3] += v.w;
                    }
                }
                if (p.gelu) {
#pragma unroll
                    for (int j = 0; j < 32; ++j) x[j] = 0.5f * x[j] * (1.f + erff(x[j] * 0.70710678118654752f));
                }
                uint32_t w[16];
#pragma unroll
                for (int j = 0; j < 16; ++j) {
                    const __nv_bfloat162 h2 = __floats2bfloat162_rn(x[2 * j], x[2 * j + 1]);
                    w[j] = *reinterpret_cast<const uint32_t *>(&h2);
                }
                if (row < p.M) {
                    uint4 *dst = reinterpret_cast<uint4 *>(p.out + (size_t)row * p.N + n0 + c0);
#pragma unroll
                    for (int j = 0; j < 4; ++j) dst[j] = make_uint4(w[4 * j], w[4 * j + 1], w[4 * j + 2], w[4 * j + 3]);
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
        ptx::tmem_dealloc(tmem, 2 * kPAccCols);
    }
}

namespace {

bool encode_2d(PFN_cuTensorMapEncodeTiled_v12000 enc, CUtensorMap *m, const void *base, int rows, int cols,
               int box_rows) {
    cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
    cuuint32_t box[2] = {(cuuint32_t)kPK, (cuuint32_t)box_rows};
    cuuint32_t es[2] = {1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

// Out[M][N] = act(A[M][K] B[N][K]^T + bias): K and N multiples of 64, 16-byte
// aligned rows; launched with programmatic stream serialization when pdl.
cudaError_t launch_project_gemm(const void *A, int M, int K, const void *B, int N, const float *bias, void *out,
                                bool gelu, int *status, bool pdl, cudaStream_t s) {
    if (M < 1) return cudaSuccess;
    auto enc = tmap_encode_fn();
    if (!enc) return cudaErrorNotSupported;
    PMaps maps;
    memset(&maps, 0, sizeof(maps));
    if (!encode_2d(enc, &maps.a, A, M, K, kPM) || !encode_2d(enc, &maps.b, B, N, K, kPN))
        return cudaErrorInvalidValue;
    PArgs p{};
    p.M = M; p.N = N; p.K = K; p.tileN = kPN;
    p.stages = kPStages;
    p.stage_stride = kPStageBytes;
    p.bias = bias; p.out = static_cast<__nv_bfloat16 *>(out); p.gelu = gelu ? 1 : 0; p.status = status;
    int dev = 0, sms = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(project_gemm_kernel<0>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kPSmemBytes);
    if (e != cudaSuccess) return e;
    const int tiles = ((M + kPM - 1) / kPM) * ((N + kPN - 1) / kPN);
    const int grid = tiles < sms ? tiles : sms;
    void *args[] = {&maps, &p};
    return launch_kernel((const void *)project_gemm_kernel<0>, dim3(grid), dim3(kPThreads), kPSmemBytes, s, args,
                         pdl);
}

// Max-over-query relevance of M tokens X [M][K] against the hi/lo rows
// QHL [2 Lqp][K] of the normalised queries: a[m] = max_j <x_m, q^_j> / a[m].
cudaError_t launch_maxsim_gemm(const void *X, int M, int K, const void *QHL, int Lq, int Lqp, float *a, int *status,
                               bool pdl, cudaStream_t s) {
    if (M < 1) return cudaSuccess;
    if (Lq < 1 || Lqp % 16 != 0 || Lq > Lqp || 2 * Lqp > kPN || K % kPK != 0) return cudaErrorInvalidValue;
    auto enc = tmap_encode_fn();
    if (!enc) return cudaErrorNotSupported;
    PMaps maps;
    memset(&maps, 0, sizeof(maps));
    if (!encode_2d(enc, &maps.a, X, M, K, kPM) || !encode_2d(enc, &maps.b, QHL, 2 * Lqp, K, 2 * Lqp))
        return cudaErrorInvalidValue;
    PArgs p{};
    p.M = M; p.N = 2 * Lqp; p.K = K; p.tileN = 2 * Lqp;
    // a narrower B tile: more, smaller stages in the same ring keep more of the
    // feature stream in flight (the GEMM is HBM bound at N <= 256)
    p.stage_stride = (kPM + p.tileN) * kPK * 2;   // multiple of 4 KB (tileN % 32 == 0)
    p.stages = (kPStages * kPStageBytes) / p.stage_stride;
    if (p.stages > kPMaxStages) p.stages = kPMaxStages;
    p.a = a; p.Lq = Lq; p.Lqp = Lqp; p.status = status;
    int dev = 0, sms = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(project_gemm_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kPSmemBytes);
    if (e != cudaSuccess) return e;
    const int tiles = (M + kPM - 1) / kPM;
    const int grid = tiles < sms ? tiles : sms;
    void *args[] = {&maps, &p};
    return launch_kernel((const void *)project_gemm_kernel<1>, dim3(grid), dim3(kPThreads), kPSmemBytes, s, args,
                         pdl);
}

}  // namespace wz
