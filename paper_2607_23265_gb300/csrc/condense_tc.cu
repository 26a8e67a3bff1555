// Condensed tokens Z_m = W_m X_m on the 5th-generation tensor cores
// (tcgen05.mma, TMA, tensor memory) -- the fused WSM + bilinear + pack step
// (Eq. 11-14, 16, 18) as one streaming pass over the features.
//
// Orientation: the MMA computes D[c][j] = sum_k X_m[k][c] * W_m[j][k] with
//   A = X tile, M = 128 channels, K = 16 tokens, MN-major (channels
//       contiguous, exactly as the features lie in HBM), loaded by TMA with
//       128-byte swizzle, box 64 channels x 32 tokens x 2 CG blocks;
//   B = W tile, N = the block's condensed tokens (<= 256, padded to 16),
//       K-major 8x8 core matrices without swizzle, stored in HBM in exactly
//       that order (tile_index) so one bulk copy moves a stage;
//   D = fp32 accumulators in tensor memory, 128 lanes x N columns per
//       128-channel tile.
// W_m is fp32 split into bf16 hi + lo (two MMAs into one accumulator, or one
// MMA of N = 2n with hi and lo side by side for n <= 64), so the product keeps
// ~16 bits of W while X (exact in bf16) streams once.
//
// A unit of work is (frame, <= 256 output tokens, CG <= 4 channel tiles) over
// the 32-token chunks [kclo, kchi] its operator rows reach.  CG is as large as
// the 512 accumulator columns allow (unit_tiles), so each operator stage in
// shared memory serves CG channel tiles; a unit that needs more than half of
// the columns takes both accumulator buffers, else one, and the epilogue of
// one unit overlaps the main loop of the next whenever two fit.  Per chunk,
// only the operator rows whose grid rows reach that chunk's map rows are
// loaded and multiplied (Ctx::krange; the first chunk covers every row, so
// each accumulator column is initialised).  Units are claimed from a global
// counter, so SMs that drew small units take more of them.  One CTA per SM:
//   warp 0      unit claims and the TMA producer (one thread), 4-stage ring
//   warp 1      TMEM allocation and the MMA issuer (one thread)
//   warps 2-13  epilogue, three warps per TMEM lane quadrant: 16x256b
//               tcgen05.ld -> bf16 pairs -> stmatrix.trans into a 2 KB tile
//               -> 16-byte rows of the output
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
constexpr int kStages = 4;
constexpr int kStageBytes = 48 * 1024;     // >= CG*8 KB (X) + 2*ncp*64 B (W hi, lo) of every unit shape
constexpr int kParts = 3;                  // epilogue warps per TMEM lane quadrant
constexpr int kEpiWarps = 4 * kParts;
constexpr int kThreads = (2 + kEpiWarps) * 32;
constexpr int kAccCols = 256;              // one of the two accumulator buffers
constexpr int kBufs = 2;
constexpr int kQueue = 8;                  // claimed units between the producer and the consumers
constexpr uint64_t kTimeoutNs = 2000000000ull;

struct TcShared {
    uint64_t full[kStages];
    uint64_t empty[kStages];
    uint64_t tfull[kBufs];
    uint64_t tempty[kBufs];
    uint64_t qfull[kQueue];
    uint64_t qempty[kQueue];
    uint64_t drain;
    uint32_t tmem_base;
    int abort;
    int uq[kQueue];
    uint32_t srange[kStages];              // operator rows [ja, jb) of each stage's chunk: ja | jb << 16
    uint16_t krow[128];                    // the producer's copy of its unit's chunk ranges
    int vprefix[WZ_MAX_VIDEOS + 1];
};

constexpr int kEpiBytes = 32 * 32 * 2;     // one warp's transpose tile: 32 tokens x 32 channels, bf16
constexpr size_t kSharedBytes = (sizeof(TcShared) + 127) / 128 * 128;   // epilogue tiles start 128-B aligned
constexpr size_t kSmemBytes = 1024 + (size_t)kStages * kStageBytes + kSharedBytes + kEpiWarps * kEpiBytes;
static_assert(kSmemBytes <= 227 * 1024, "shared memory of the condensation CTA");
static_assert(4 * 8192 + 2 * 128 * 64 <= kStageBytes && 3 * 8192 + 2 * 160 * 64 <= kStageBytes &&
                  2 * 8192 + 2 * 256 * 64 <= kStageBytes && 4 * 8192 + 2 * 64 * 64 <= kStageBytes,
              "a stage holds the features and operator halves of every unit shape");

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
    bool ranged;                          // per-chunk operator rows in c.krange
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
    r.ranged = (q.w & kUnitRanged) != 0;
    return r;
}

// Accumulator shape of a unit: hi|lo fused into one MMA of N = 2*ncp for
// small budgets, else two MMAs of N = ncp into one accumulator; a unit
// whose tiles need more than one buffer's columns takes both buffers.
struct UnitShape {
    int ncp, tcols;
    bool fused, wide, valid;
};

__device__ __forceinline__ UnitShape unit_shape(const Unit &un, int KC) {
    UnitShape sh;
    sh.ncp = (un.nc + 15) & ~15;
    sh.fused = unit_fused(sh.ncp);
    sh.tcols = sh.fused ? 2 * sh.ncp : sh.ncp;
    sh.wide = un.cg * sh.tcols > kAccCols;
    sh.valid = un.nc >= 1 && un.nc <= kColBlock && un.cg >= 1 && un.cg <= 4 &&
               un.cg * sh.tcols <= kBufs * kAccCols && un.kclo <= un.kchi && un.kchi < KC && KC <= 128 &&
               un.cg * 8192 + 2 * sh.ncp * 64 <= kStageBytes && (!un.ranged || !sh.fused);
    return sh;
}

__device__ __forceinline__ void fail(const Ctx &c, volatile int *abort_flag, int code) {
    *abort_flag = 1;
    atomicOr(c.status, code);
}

// The MMAs of one unit: stages kclo..kchi of kKC tokens, each two K = 16 steps over
// CG channel tiles (hi|lo fused into one MMA, or hi and lo as two).  The
// pattern is fixed at compile time and the stage descriptors are advanced by
// a constant, so the issuing thread spends a few instructions per MMA.
// Unfused units take the operator rows [ja, jb) of each stage from
// S->srange (the rows that reach the chunk; the first chunk of a unit always
// covers every row, so each accumulator column is written before it is
// accumulated into): the MMAs run over N = jb - ja columns from column ja.
template <int CG, bool FUSED>
__device__ __forceinline__ bool mma_unit(TcShared *S, uint8_t *ring, const Ctx &c, volatile int *abort_flag, int kclo,
                                         int kchi,
                                         int &stage, uint32_t &phase, uint32_t dbase, int tcols, uint32_t idesc,
                                         int ncp) {
    const volatile uint32_t *srange = S->srange;
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
        const uint64_t a0 = a_base + so;
        uint64_t b0 = b_base + so;
        uint32_t id = idesc, col = 0;
        if (!FUSED) {
            const uint32_t r = srange[stage];
            const uint32_t ja = r & 0xffffu, jb = r >> 16;
            b0 += (uint64_t)((ja * 64u) >> 4);
            id = ptx::idesc_bf16(128, (int)(jb - ja), true, false);
            col = ja;
        }
        const uint32_t acc = kc > kclo ? 1u : 0u;
#pragma unroll
        for (int s = 0; s < 2; ++s) {
#pragma unroll
            for (int ct = 0; ct < CG; ++ct) {
                const uint64_t a = a0 + (uint64_t)((ct * 8192 + s * 2048) >> 4);
                ptx::mma_bf16(d[ct] + col, a, b0 + (uint64_t)(s * 16), id, acc | (uint32_t)s);
                if (!FUSED) ptx::mma_bf16(d[ct] + col, a, b0 + lo_off + (uint64_t)(s * 16), id, 1u);
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

template <bool FUSED>
__device__ __forceinline__ bool mma_unit_cg(int cg, TcShared *S, uint8_t *ring, const Ctx &c,
                                            volatile int *abort_flag, int kclo, int kchi, int &stage,
                                            uint32_t &phase, uint32_t dbase, int tcols, uint32_t idesc, int ncp) {
    switch (cg) {
        case 1: return mma_unit<1, FUSED>(S, ring, c, abort_flag, kclo, kchi, stage, phase, dbase, tcols, idesc, ncp);
        case 2: return mma_unit<2, FUSED>(S, ring, c, abort_flag, kclo, kchi, stage, phase, dbase, tcols, idesc, ncp);
        case 3: return mma_unit<3, FUSED>(S, ring, c, abort_flag, kclo, kchi, stage, phase, dbase, tcols, idesc, ncp);
        case 4: return mma_unit<4, FUSED>(S, ring, c, abort_flag, kclo, kchi, stage, phase, dbase, tcols, idesc, ncp);
        default: fail(c, abort_flag, 4); return false;
    }
}

__device__ __forceinline__ uint32_t pack_bf16x2(uint32_t lo, uint32_t hi) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(__uint_as_float(lo), __uint_as_float(hi));
    return *reinterpret_cast<const uint32_t *>(&h);
}

// One epilogue block: a warp's 32 channels (its tensor-memory lane quadrant,
// from channel ch0) x 32 tokens (accumulator columns colb .. colb+31 = tokens
// j0 .. j0+31 of the unit) -> bf16 rows of the output.  The 16x256b loads
// give each thread channel pairs of token pairs (the mma fragment layout);
// stmatrix.trans writes them as token rows of 8 channels into the warp's
// 2 KB tile (16-byte chunk o of row r at chunk o ^ ((r >> 1) & 3), free of
// bank conflicts), and 16-byte pieces leave for global memory, 8 token rows
// per store instruction.  For fused units the lo half sits ncp columns
// further and is added first.
__device__ __forceinline__ void block_load(uint32_t colb, bool full, uint32_t (&v)[2][16]) {
#pragma unroll
    for (int hh = 0; hh < 2; ++hh) {
        const uint32_t ta = colb + ((uint32_t)(16 * hh) << 16);
        if (full) ptx::tmem_ld_16x256b_x4(ta, v[hh]);
        else ptx::tmem_ld_16x256b_x2(ta, *reinterpret_cast<uint32_t(*)[8]>(v[hh]));
    }
}

__device__ __forceinline__ void block_loaded(uint32_t (&v)[2][16]) {
    ptx::reg_fence16(v[0]);
    ptx::reg_fence16(v[1]);
}

__device__ __forceinline__ void block_epilogue(uint32_t colb, bool fused, int ncp, int j0, uint32_t tr32, int lane,
                                               char *out, size_t rowb, size_t row0, int nc, int ch0, const Ctx &c) {
    const bool full = j0 + 16 < ncp;          // 32 valid columns, else 16
    uint32_t v[2][16];
    block_load(colb, full, v);
    if (fused) {
        uint32_t w[2][16];
        block_load(colb + (uint32_t)ncp, full, w);
        ptx::tmem_ld_wait();
        block_loaded(v);
        block_loaded(w);
#pragma unroll
        for (int hh = 0; hh < 2; ++hh)
#pragma unroll
            for (int k = 0; k < 16; ++k)
                v[hh][k] = __float_as_uint(__uint_as_float(v[hh][k]) + __uint_as_float(w[hh][k]));
    } else {
        ptx::tmem_ld_wait();
        block_loaded(v);
    }
    uint32_t p[2][4][2];
#pragma unroll
    for (int hh = 0; hh < 2; ++hh)
#pragma unroll
        for (int g = 0; g < 4; ++g)
#pragma unroll
            for (int k = 0; k < 2; ++k)
                p[hh][g][k] = (g < 2 || full) ? pack_bf16x2(v[hh][4 * g + 2 * k], v[hh][4 * g + 2 * k + 1]) : 0u;
    __syncwarp();   // the previous block's reads of the tile
    const int m = lane >> 3, i = lane & 7;
#pragma unroll
    for (int hh = 0; hh < 2; ++hh)
#pragma unroll
        for (int ga = 0; ga < 4; ga += 2) {
            if (ga == 0 || full) {
                const int g = ga + (m >> 1), o = 2 * hh + (m & 1), row = 8 * g + i;
                const uint32_t addr = tr32 + (uint32_t)(row * 64 + ((o ^ ((row >> 1) & 3)) << 4));
                ptx::stmatrix_x4_trans(addr, p[hh][ga][0], p[hh][ga][1], p[hh][ga + 1][0], p[hh][ga + 1][1]);
            }
        }
    __syncwarp();
#pragma unroll
    for (int r = 0; r < 4; ++r) {
        const int t = r * 8 + (lane >> 2);
        const int cc = lane & 3;                  // 8-channel chunk
        if (j0 + t < nc && ch0 + cc * 8 < c.D && wz_in_range(c.status, (int64_t)(row0 + j0 + t) < c.rows_total)) {
            const uint4 val = ptx::lds128(tr32 + (uint32_t)(t * 64 + ((cc ^ ((t >> 1) & 3)) << 4)));
            *reinterpret_cast<uint4 *>(out + (row0 + j0 + t) * rowb + (size_t)(ch0 + cc * 8) * 2) = val;
        }
    }
}

}  // namespace

// Units are claimed dynamically: the producer thread takes the next unit of
// the whole call from a global counter (zeroed by the temporal kernel) and
// hands its index to the MMA thread and the epilogue warps through a small
// queue in shared memory, so CTAs that drew small units take more of them.
// Accumulator buffers: a unit uses one of the two 256-column buffers when its
// tiles fit, else both; the MMA thread and the epilogue walk the same unit
// sequence and keep the same per-buffer use counts, which give the barrier
// parities.
__global__ void __launch_bounds__(kThreads, 1)
condense_tc_kernel(const __grid_constant__ TcMaps maps, Ctx c) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *ring = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    TcShared *S = reinterpret_cast<TcShared *>(ring + (size_t)kStages * kStageBytes);
    volatile int *abort_flag = &S->abort;
    volatile int *uq = S->uq;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            ptx::mbar_init(&S->full[s], 1);
            ptx::mbar_init(&S->empty[s], 1);
        }
        for (int b = 0; b < kBufs; ++b) {
            ptx::mbar_init(&S->tfull[b], 1);
            ptx::mbar_init(&S->tempty[b], kEpiWarps);
        }
        for (int q = 0; q < kQueue; ++q) {
            ptx::mbar_init(&S->qfull[q], 1);
            ptx::mbar_init(&S->qempty[q], 1 + kEpiWarps);   // the MMA thread and every epilogue warp
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
        // ---------------- unit claims and TMA producer ----------------
        const uint64_t pol_x = ptx::policy_evict_first();
        const uint64_t pol_w = ptx::policy_evict_last();
        const char *whi = static_cast<const char *>(c.Wop);
        const char *wlo = whi + (size_t)c.w_rows * c.K_pad * 2;
        const size_t groups = (size_t)(c.w_rows >> 3);
        int stage = 0;
        uint32_t phase = 0;
        int issued_parity[kStages];
        for (int s = 0; s < kStages; ++s) issued_parity[s] = -1;
        for (int k = 0;; ++k) {
            const int slot = k & (kQueue - 1);
            if (!ptx::mbar_wait(&S->qempty[slot], ((uint32_t)(k / kQueue) & 1u) ^ 1u, kTimeoutNs)) {
                fail(c, abort_flag, 1);
                break;
            }
            int u = *abort_flag ? -1 : atomicAdd(c.spatial_next + 1, 1);
            if (u >= n_units) u = -1;
            uq[slot] = u;
            ptx::mbar_arrive(&S->qfull[slot]);
            if (u < 0) break;
            const Unit un = decode_unit(c, S->vprefix, u);
            const UnitShape sh = unit_shape(un, KC);
            if (!sh.valid) {   // not a record the spatial kernel writes
                fail(c, abort_flag, 4);
                break;
            }
            const int64_t wrow0 = (int64_t)c.woff[un.f] + un.j0;     // multiple of 16
            if (un.ranged) {   // the unit's chunk ranges, loaded together
                const uint16_t *kr = c.krange + ((size_t)un.f * c.krange_nblk + (un.j0 >> 8)) * KC;
                for (int kc = un.kclo + 1; kc <= un.kchi; ++kc) S->krow[kc] = kr[kc];
            }
            bool ok = true;
            for (int kc = un.kclo; kc <= un.kchi; ++kc) {
                uint32_t ja = 0, jb = (uint32_t)sh.ncp;
                if (un.ranged && kc > un.kclo) {
                    const uint32_t r = S->krow[kc];
                    ja = (r & 0xffu) << 4;
                    jb = (r >> 8) << 4;
                    if (jb <= ja || jb > (uint32_t)sh.ncp) {   // not a range the spatial kernel writes
                        fail(c, abort_flag, 4);
                        ok = false;
                        break;
                    }
                }
                const uint32_t bytes = (uint32_t)un.cg * 8192u + 2u * (jb - ja) * 64u;
                if (!ptx::mbar_wait(&S->empty[stage], phase ^ 1u, kTimeoutNs)) {
                    fail(c, abort_flag, 1);
                    ok = false;
                    break;
                }
                uint8_t *st = ring + (size_t)stage * kStageBytes;
                S->srange[stage] = ja | (jb << 16);
                ptx::mbar_arrive_expect_tx(&S->full[stage], bytes);
                if (maps.use4) {
                    ptx::tma_load_4d(st, &maps.x4[un.cg - 1], &S->full[stage], 0, kc * kKC, 2 * un.ct0, un.f, pol_x);
                } else {
                    for (int ct = 0; ct < un.cg; ++ct)
                        for (int h = 0; h < 2; ++h)
                            ptx::tma_load_3d(st + ct * 8192 + h * 4096, &maps.x3, &S->full[stage],
                                             (un.ct0 + ct) * kTileC + h * 64, kc * kKC, un.f, pol_x);
                }
                uint8_t *wh = st + un.cg * 8192 + ja * 64u;
                const size_t toff = ((size_t)kc * groups + (size_t)(wrow0 >> 3)) * 512 + (size_t)ja * 64u;
                ptx::bulk_load(wh, whi + toff, (jb - ja) * 64u, &S->full[stage], pol_w);
                ptx::bulk_load(wh + sh.ncp * 64, wlo + toff, (jb - ja) * 64u, &S->full[stage], pol_w);
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
        uint32_t uses[kBufs] = {0u, 0u};
        int nb = 0;
        for (int k = 0; !*abort_flag; ++k) {
            const int slot = k & (kQueue - 1);
            if (!ptx::mbar_wait(&S->qfull[slot], (uint32_t)(k / kQueue) & 1u, kTimeoutNs)) {
                fail(c, abort_flag, 2);
                break;
            }
            const int u = uq[slot];
            ptx::mbar_arrive(&S->qempty[slot]);
            if (u < 0) break;
            const Unit un = decode_unit(c, S->vprefix, u);
            const UnitShape sh = unit_shape(un, KC);
            if (!sh.valid) {
                fail(c, abort_flag, 4);
                break;
            }
            const int b = nb;
            bool ok = ptx::mbar_wait(&S->tempty[b], (uses[b] & 1u) ^ 1u, kTimeoutNs);
            if (ok && sh.wide) ok = ptx::mbar_wait(&S->tempty[b ^ 1], (uses[b ^ 1] & 1u) ^ 1u, kTimeoutNs);
            if (!ok) {
                fail(c, abort_flag, 2);
                break;
            }
            ptx::tc_fence_after();
            const uint32_t idesc = ptx::idesc_bf16(128, sh.tcols, true, false);
            const uint32_t dbase = tmem + (sh.wide ? 0u : (uint32_t)(b * kAccCols));
            ok = sh.fused ? mma_unit_cg<true>(un.cg, S, ring, c, abort_flag, un.kclo, un.kchi, stage, phase, dbase,
                                              sh.tcols, idesc, sh.ncp)
                          : mma_unit_cg<false>(un.cg, S, ring, c, abort_flag, un.kclo, un.kchi, stage, phase, dbase,
                                               sh.tcols, idesc, sh.ncp);
            if (!ok) break;
            ptx::mma_commit(&S->tfull[b]);
            ++uses[b];
            if (sh.wide) {
                ptx::mma_commit(&S->tfull[b ^ 1]);
                ++uses[b ^ 1];
            } else {
                nb ^= 1;
            }
        }
        // every MMA issued by this thread completes before tensor memory is freed
        ptx::mma_commit(&S->drain);
        ptx::mbar_wait(&S->drain, 0, kTimeoutNs);
    } else if (warp >= 2) {
        // ---------------- epilogue ----------------
        const int ew = warp - 2;                         // 0 .. kEpiWarps-1
        const int q = warp & 3;                          // TMEM lane quadrant of this warp
        const int part = ew >> 2;                        // this warp's share of the quadrant's blocks
        const uint32_t tr32 = ptx::smem_u32(reinterpret_cast<uint8_t *>(S) + kSharedBytes + (size_t)ew * kEpiBytes);
        char *out = static_cast<char *>(c.out);
        const size_t rowb = (size_t)c.D * 2;
        uint32_t uses[kBufs] = {0u, 0u};
        int nb = 0;
        for (int k = 0; !*abort_flag; ++k) {
            const int slot = k & (kQueue - 1);
            if (!ptx::mbar_wait(&S->qfull[slot], (uint32_t)(k / kQueue) & 1u, kTimeoutNs)) {
                fail(c, abort_flag, 8);
                break;
            }
            const int u = uq[slot];
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&S->qempty[slot]);
            if (u < 0) break;
            const Unit un = decode_unit(c, S->vprefix, u);
            const UnitShape sh = unit_shape(un, KC);
            if (!sh.valid) {
                fail(c, abort_flag, 4);
                break;
            }
            const int ncp = sh.ncp;
            const int b = nb;
            bool ok = ptx::mbar_wait(&S->tfull[b], uses[b] & 1u, kTimeoutNs);
            if (ok && sh.wide) ok = ptx::mbar_wait(&S->tfull[b ^ 1], uses[b ^ 1] & 1u, kTimeoutNs);
            if (!ok) {
                fail(c, abort_flag, 8);
                break;
            }
            ptx::tc_fence_after();
            const size_t row0 = (size_t)c.off[un.f] + un.j0;
            const uint32_t tbase = tmem + ((uint32_t)(q * 32) << 16) + (sh.wide ? 0u : (uint32_t)(b * kAccCols));
            // the unit's 32-token blocks of this warp's quadrant (tile ct,
            // tokens j0), dealt round-robin over the quadrant's kParts warps
            const int nbj = (ncp + 31) / 32;
            const int nblocks = un.cg * nbj;
            for (int bi = part; bi < nblocks; bi += kParts) {
                const int ct = bi / nbj, j0 = (bi - ct * nbj) * 32;
                block_epilogue(tbase + (uint32_t)(ct * sh.tcols + j0), sh.fused, ncp, j0, tr32, lane, out, rowb,
                               row0, un.nc, (un.ct0 + ct) * kTileC + q * 32, c);
            }
            ptx::tc_fence_before();
            __syncwarp();
            if (lane == 0) {
                ptx::mbar_arrive(&S->tempty[b]);
                if (sh.wide) ptx::mbar_arrive(&S->tempty[b ^ 1]);
            }
            ++uses[b];
            if (sh.wide) ++uses[b ^ 1];
            else nb ^= 1;
        }
    }
    __syncthreads();
    if (warp == 1) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem, kAccCols * kBufs);
    }
}

// cuTensorMapEncodeTiled from the driver (resolved once; null when missing).
PFN_cuTensorMapEncodeTiled_v12000 tmap_encode_fn() {
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

bool tensor_path_available() { return true; }

cudaError_t launch_condense_tc(const Ctx &c, cudaStream_t s) {
    auto enc = tmap_encode_fn();
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
