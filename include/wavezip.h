/*
 * wavezip.h -- C ABI of the GB300 (sm_103a) WaveZip condensation library.
 *
 * WaveZip (arXiv 2607.23265, Section 3) condenses the visual tokens of a video
 * before they reach the LLM: query relevance per token and per frame
 * (Section 3.2.1), a visual-change prior over adjacent frames (Section 3.2.2,
 * Eq. 7), a single-level Haar DWT of the frame-relevance sequence whose detail
 * coefficients are gated by that prior (Eq. 8-10), integer per-frame token
 * budgets (Eq. 5, Eq. 15), a single-level db4 2D DWT of each frame whose
 * detail bands are modulated by the query saliency (Eq. 11-14), and
 * budget-guided bilinear condensation and packing (Eq. 16, Eq. 18).
 *
 * Conventions shared by every entry point
 *   - Every array argument is a DEVICE pointer unless its comment says host.
 *     The caller allocates and owns all buffers; the library keeps no
 *     reference after the call returns.
 *   - Features are channels-last: [T][H][W][D] (token n = i*W + j of frame t
 *     at offset ((t*H + i)*W + j)*D), D contiguous; queries are [Lq][D].
 *   - dtype WZ_DTYPE_BF16 (bfloat16) or WZ_DTYPE_F32; features, queries and
 *     condensed tokens share it.  D must be a multiple of 8 and feature /
 *     query / token pointers 16-byte aligned.
 *   - Calls are asynchronous on `stream` (NULL = legacy default stream).
 *     Argument errors are detected on the host and returned before anything
 *     is enqueued; CUDA launch errors return WZ_ERR_CUDA.  No C++ exception
 *     crosses this interface.  Results are valid once the stream completes.
 *   - A workspace pointer may be NULL: the call then takes its scratch memory
 *     with cudaMallocAsync on `stream` and frees it with cudaFreeAsync after
 *     the last kernel.
 *   - Paper defaults: lambda = 1.5, Haar for WTA, db4 for WSM, one level
 *     (Section 4.1); tau = 0 (the frame filter keeps every frame).
 *
 * Readings of points the paper leaves open (they fix the results below):
 *   u_q is the mean of the query rows; per-frame min-max saliency; Haar and
 *   db4 with half-sample symmetric extension (DWT length floor((n+F-1)/2));
 *   B = round-half-away(ratio*T*H*W); budgets by largest remainder with ties
 *   to the earlier frame, capped at H*W with the excess re-apportioned and a
 *   uniform split when no frame has positive relevance; the n_m tokens of a
 *   frame are the first n_m points, in raster order, of an h x w grid with
 *   h = min(H, ceil(sqrt(n_m*H/W))), w = ceil(n_m/h), sampled bilinearly with
 *   half-pixel centres.
 */
#ifndef WAVEZIP_H
#define WAVEZIP_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#if defined(__GNUC__)
#define WZ_API __attribute__((visibility("default")))
#else
#define WZ_API
#endif

/* Same type as cudaStream_t / CUstream. */
typedef struct CUstream_st *wz_stream_t;

/* Status codes. */
#define WZ_OK               0
#define WZ_ERR_INVALID_ARG  (-1) /* null pointer, bad size, bad enum          */
#define WZ_ERR_UNSUPPORTED  (-2) /* valid but outside the library's limits   */
#define WZ_ERR_CUDA         (-3) /* a CUDA runtime/driver call failed         */
#define WZ_ERR_NO_MEMORY    (-4) /* cudaMallocAsync of the workspace failed   */
#define WZ_ERR_WORKSPACE    (-5) /* caller's workspace smaller than required  */

#define WZ_DTYPE_BF16 0
#define WZ_DTYPE_F32  1

/* Signal extension at the borders for the DWT entry points. */
#define WZ_MODE_SYMMETRIC 0 /* half-sample symmetric: x[-1-k] = x[k]        */
#define WZ_MODE_ZERO      1 /* zeros outside the signal                     */
#define WZ_MODE_PERIODIC  2 /* x[n+k] = x[k]                                */

/* Which kernel computes the fused WSM + bilinear + pack step. */
#define WZ_PATH_AUTO   0 /* tensor cores for bf16, CUDA cores for f32        */
#define WZ_PATH_TENSOR 1 /* tcgen05.mma (bf16 only)                          */
#define WZ_PATH_SIMT   2 /* fp32 CUDA-core GEMM                              */

/* Kernels of one condensation call, in launch order (for kernel_events). */
#define WZ_KERNEL_QUERY_POOL     0 /* u_q                                      */
#define WZ_KERNEL_RELEVANCE      1 /* streaming pass: a_{t,n}, column sums     */
#define WZ_KERNEL_FRAME_STATS    2 /* fp64 frame sums and dot products          */
#define WZ_KERNEL_TEMPORAL       3 /* r, delta, gamma, WTA, budgets, offsets    */
#define WZ_KERNEL_SPATIAL        4 /* operator rows W_m, index map, tail rows   */
#define WZ_KERNEL_CONDENSE       5 /* Z_m = W_m X_m, packed                     */
#define WZ_NUM_KERNELS           6

/* Ablation modes (Section 4 "Ablation Study", Appendix B).  The defaults
 * (0, 0) are the method itself. */
#define WZ_TEMPORAL_WTA      0 /* budgets from the WTA-rectified relevance r~      */
#define WZ_TEMPORAL_RAW      1 /* "Raw Top-k": budgets from the raw relevance r_t   */
#define WZ_TEMPORAL_UNIFORM  2 /* equal budgets over the retained frames          */
#define WZ_SPATIAL_WSM       0 /* wavelet spatial modulator (Eq. 11-14)            */
#define WZ_SPATIAL_SALIENCY  1 /* "Saliency-Only": lambda * M_t * X_t, no wavelets */
#define WZ_SPATIAL_NONE      2 /* no modulation: Psi of the features itself       */

/* Relevance scorer.  MEAN: the similarity branch with the mean query row
 * u_q (Section 3.2.1); MAXSIM: no pooling of the query, the maximum cosine
 * over its rows for both a_{t,n} and r_t (bf16 features, D % 64 == 0,
 * Lq <= WZ_MAX_LQ_MAXSIM; the token x row cosines run on the tensor cores). */
#define WZ_RELEVANCE_MEAN    0
#define WZ_RELEVANCE_MAXSIM  1
#define WZ_MAX_LQ_MAXSIM     128

/* Decomposition levels of the WTA and the WSM (the paper's modules use one;
 * with J > 1 the DWT cascades on the approximation band, level j's details
 * gated by the pairwise mean of level j-1's gate (WTA) or by the saliency
 * map pooled to level j's subband grid (WSM)). */
#define WZ_MAX_LEVELS 4

/* Wavelets: Daubechies filters named by their vanishing moments p (2p
 * taps), 1 = Haar, 4 = db4, 1 <= p <= 10; and the biorthogonal bior4.4
 * (CDF 9/7, 10-tap arrays), the third basis of the paper's "Wavelet Basis"
 * ablation (Section 4). */
#define WZ_WAVELET_HAAR   1
#define WZ_WAVELET_DB4    4
#define WZ_WAVELET_BIOR44 44

/* Limits of the library (WZ_ERR_UNSUPPORTED beyond them). */
#define WZ_MAX_HW      64    /* H, W <= 64                                  */
#define WZ_MAX_T       4096  /* frames per video                            */
#define WZ_MAX_VIDEOS  1024  /* videos per batch call                       */
#define WZ_MAX_D       32768 /* channels (bf16; half of it for f32)         */

/* ------------------------------------------------------------------------ */
/* Condensation C_WaveZip(X, Q) (Section 3.2, Eq. 18)                        */
/* ------------------------------------------------------------------------ */

/*
 * Global budget B = round-half-away(ratio * T * H * W) (Section 4.1: B = rho
 * N_v with N_v counted before compression).  Host only; returns -1 for
 * invalid sizes or ratio outside (0, 1].
 */
WZ_API int64_t wz_budget_size(int T, int H, int W, float ratio);

/*
 * Condense one bf16 video with the paper's defaults.
 *   features   [T][H][W][D] bf16          query [Lq][D] bf16
 *   ratio      keep ratio rho in (0, 1]
 *   out_tokens [B][D] bf16, B = wz_budget_size(T, H, W, ratio)
 *   out_index  [B][3] int32: (t, i, j) = frame and position of each token in
 *              that frame's h x w condensation grid; rows are grouped by
 *              frame in temporal order.  Rows past the produced count (only
 *              possible with tau > 0) hold -1 and zero tokens.
 * Equivalent to wz_condense_ex with defaults and a NULL workspace.
 */
WZ_API int wz_condense(const void *features, int T, int H, int W, int D,
                const void *query, int Lq, float ratio,
                void *out_tokens, int32_t *out_index, wz_stream_t stream);

typedef struct {
    const void *features;    /* [T][H][W][D], dtype                          */
    int T, H, W, D;
    int dtype;               /* WZ_DTYPE_*                                   */
    const void *query;       /* [Lq][D], dtype                               */
    int Lq;
    float ratio;             /* rho in (0, 1]                                */
    float lambda;            /* WSM gate strength (Eq. 12), default 1.5      */
    float tau;               /* frame-filter threshold on delta, default 0   */
    int wta_wavelet;         /* WTA wavelet: 1..10 or WZ_WAVELET_BIOR44,     */
                             /* default 1 (Haar, Eq. 8-10)                   */
    int wsm_wavelet;         /* WSM wavelet: 1..10 or WZ_WAVELET_BIOR44,     */
                             /* default 4 (db4)                              */
    int mode;                /* WZ_MODE_* extension for the WSM DWT          */
    int path;                /* WZ_PATH_*                                    */
    int temporal_mode;       /* WZ_TEMPORAL_*, default WTA                   */
    int spatial_mode;        /* WZ_SPATIAL_*, default WSM                    */
    const float *token_scores; /* [T][N] f32 device, an external scorer's    */
                             /* a_{t,n} (Section 3.2.1) replacing the        */
                             /* similarity branch's; nullable                */
    const float *frame_scores; /* [T] f32 device, external r_t; nullable     */
    int relevance_mode;      /* WZ_RELEVANCE_*, default MEAN                 */
    int wta_levels;          /* 1..WZ_MAX_LEVELS, default 1                  */
    int wsm_levels;          /* 1..WZ_MAX_LEVELS, default 1                  */
    void *out_tokens;        /* [B][D], dtype                                */
    int32_t *out_index;      /* [B][3]                                       */
    int32_t *out_budgets;    /* [T] n_t (0 for filtered frames); nullable    */
    int32_t *out_count;      /* [1] tokens produced (= B unless tau > 0);    */
                             /* nullable                                     */
    float *out_relevance;    /* [T][4] (r_t, delta_t, gamma_t, r~_t; r~ is   */
                             /* NaN for filtered frames); nullable           */
    void *workspace;         /* >= wz_condense_workspace_size() bytes, 256-B */
    size_t workspace_bytes;  /* aligned; NULL = cudaMallocAsync on stream    */
    int32_t *device_status;  /* [1] set nonzero by a kernel whose bounded    */
                             /* wait timed out; nullable                     */
    void *const *kernel_events; /* [2*WZ_NUM_KERNELS] cudaEvent_t, nullable: */
                             /* events[2k] / [2k+1] are recorded on `stream` */
                             /* right before / after kernel k (profiling)    */
    wz_stream_t stream;
} wz_condense_args;

/* Fill `a` with the paper's defaults and zero pointers/sizes. */
WZ_API void wz_condense_args_init(wz_condense_args *a);

/* Workspace bytes that wz_condense_ex needs for these sizes. */
WZ_API size_t wz_condense_workspace_size(int T, int H, int W, int D, int dtype, float ratio);

/*
 * Condense one video (arguments above).  Returns a WZ_* status.
 * Replay cache: when `workspace` is given, `kernel_events` is NULL and
 * `stream` is not being captured, an argument set (every pointer, size and
 * option, on the current device) seen for the second time has its launch
 * sequence captured into a CUDA graph (on a private stream; that call pays
 * the capture and instantiation on the host), and that call and every later
 * one with identical arguments launch the graph into `stream`; the first call
 * with an argument set launches the kernels one by one.  The inputs are read when
 * the graph runs, so new contents in the same buffers are condensed anew.
 * Otherwise the kernels are launched one by one.  See wz_graph_cache.
 */
WZ_API int wz_condense_ex(const wz_condense_args *a);

/*
 * wz_condense_ex with the features, the query and the outputs in HOST memory
 * (pinned for asynchronous copies; pageable works, with the copies staged by
 * the driver): the call allocates device staging on `stream`
 * (cudaMallocAsync), copies the inputs in, runs the pass, copies out_tokens,
 * out_index and whichever of out_budgets / out_count / out_relevance are
 * non-NULL back, and frees the staging, all ordered on `stream`.  The host
 * buffers must stay valid until the stream reaches the end of the call.
 * token_scores, frame_scores and kernel_events must be NULL (they are device
 * inputs); workspace and device_status are ignored.  Returns WZ_ERR_NO_MEMORY
 * when the staging cannot be allocated.
 */
WZ_API int wz_condense_host(const wz_condense_args *a);

/*
 * Serving batch: V independent videos of equal T, H, W, D in one launch
 * sequence (the paper processes one video per request; a batch is V such
 * requests).  Per-video query lengths and keep ratios.
 *   features    [V][T][H][W][D]
 *   queries     [sum_v Lq[v]][D], video v's rows follow video v-1's
 *   Lq, ratio   HOST arrays [V]
 *   out_tokens  [R][D], R = sum_v B_v, video v's B_v rows start at
 *               row_offsets[v]; out_index [R][3] as for wz_condense
 *   row_offsets HOST array [V+1] filled by the call (nullable)
 *   out_budgets [V][T], out_count [V], out_relevance [V][T][4] (nullable)
 */
typedef struct {
    int V;
    const void *features;
    int T, H, W, D;
    int dtype;
    const void *queries;
    const int32_t *Lq;       /* host */
    const float *ratio;      /* host */
    float lambda, tau;
    int wta_wavelet, wsm_wavelet, mode, path;
    int temporal_mode, spatial_mode;   /* WZ_TEMPORAL_*, WZ_SPATIAL_* */
    const float *token_scores;         /* [V][T][N] device, nullable   */
    const float *frame_scores;         /* [V][T] device, nullable      */
    int relevance_mode;                /* WZ_RELEVANCE_*               */
    int wta_levels, wsm_levels;        /* 1..WZ_MAX_LEVELS             */
    void *out_tokens;
    int32_t *out_index;
    int64_t *row_offsets;    /* host, [V+1], nullable */
    int32_t *out_budgets;
    int32_t *out_count;
    float *out_relevance;
    void *workspace;
    size_t workspace_bytes;
    int32_t *device_status;
    void *const *kernel_events;
    wz_stream_t stream;
} wz_batch_args;

WZ_API void wz_batch_args_init(wz_batch_args *a);

/* Total output rows R = sum_v B_v; fills host row_offsets[V+1] if non-NULL.
 * Returns -1 on invalid arguments. */
WZ_API int64_t wz_batch_rows(int V, int T, int H, int W, const float *ratio, int64_t *row_offsets);

WZ_API size_t wz_batch_workspace_size(int V, int T, int H, int W, int D, int dtype, const float *ratio);

/* The serving batch (arguments above; same replay cache as wz_condense_ex). */
WZ_API int wz_condense_batch(const wz_batch_args *a);

/*
 * Replay cache of wz_condense_ex / wz_condense_batch: the number of argument
 * sets whose executable graphs are kept (least recently used dropped first;
 * default 8).  capacity >= 0 sets it (0 disables the cache and frees every
 * kept graph; a graph still running is freed when it completes); a negative
 * capacity only queries.  stats: HOST int64[3], nullable, filled after the
 * change with {graphs kept, replays, captures} (the last two count since the
 * library was loaded).  Returns the capacity in force before the call.
 * Thread-safe; host only.
 */
WZ_API int wz_graph_cache(int capacity, int64_t *stats);

/* ------------------------------------------------------------------------ */
/* Cross-Modal Scorer, similarity branch (Section 3.2.1)                     */
/* ------------------------------------------------------------------------ */

/*
 * token_scores [T][H*W] f32: a_{t,n} = cos(u_{t,n}, u_q), u_q = mean of the
 *              query rows (0 where a norm is 0).
 * frame_scores [T] f32: r_t = cos(mean_n u_{t,n}, u_q).
 * frame_mean   [T][D] f32: the pooled feature v_bar_t (nullable).
 * workspace    >= wz_relevance_workspace_size() bytes, or NULL.
 * device_status [1] int32, nullable: a bounded wait of the relevance pass
 *              that gives up ORs a nonzero code into it (the caller zeroes
 *              it; the bounds-checked build adds WZ_STATUS_BOUNDS); without
 *              it the workspace's own word, zeroed on `stream`, takes the
 *              code and the failure is not reported.
 */
WZ_API int wz_relevance(const void *features, int T, int H, int W, int D, int dtype,
                 const void *query, int Lq, float *token_scores, float *frame_scores,
                 float *frame_mean, void *workspace, size_t workspace_bytes,
                 int32_t *device_status, wz_stream_t stream);

WZ_API size_t wz_relevance_workspace_size(int T, int H, int W, int D);

/*
 * The scores of wz_relevance for callers that must not allocate device
 * memory.  The paper has no counterpart: this is a deployment convenience of
 * this library.  Callers that need it include code running while a stream is
 * captured into a CUDA graph that may hold no allocation nodes, serving loops
 * that fix their memory budget at start-up so a request can never fail on an
 * out-of-memory or wait on an allocator, and hosts whose device memory is
 * managed by another framework's caching allocator.  Inputs and outputs are
 * the caller's, as for wz_relevance; the intermediate sums go to one fixed
 * array of WZ_STATIC_SCRATCH_BYTES compiled into the library, which every GPU
 * that loads the library keeps until the process exits.
 *   - No cudaMalloc, cudaFree or other allocating call is made.
 *   - The array used is the one of the current device: `stream` must belong
 *     to the current device, and so must every pointer.
 *   - The first call on a device looks the array's device address up
 *     (cudaGetSymbolAddress) with that device current; make that first call
 *     before any stream capture.
 *   - Sizes whose sums do not fit the array return WZ_ERR_WORKSPACE before
 *     anything is enqueued.  The sums take, each rounded up to 256 bytes,
 *     12*D + 32 (query mean in f32 and f64, per-call parameters), (G1 + T)*D*4
 *     (column partials), 32*T (per-frame statistics) and 16 (status word),
 *     where G1 = min(2048, ceil(T*H*W/16), SMs x resident relevance CTAs per
 *     SM) is the relevance grid (152 on a GB300 at D = 3584: about T <= 1000
 *     frames fit at that width).
 *   - device_status [1] int32, nullable: as for wz_relevance.  Without it the
 *     array's own status word is zeroed on `stream` (cudaMemsetAsync) and
 *     takes the bits, so a timed-out wait is not reported.
 *   - Every call shares the one array; apart from that status word nothing
 *     in it must start at zero and no state passes from one call to the next,
 *     but calls that overlap on the GPU (other streams, other host threads)
 *     race on it: serialise them.
 */
#define WZ_STATIC_SCRATCH_BYTES (16u << 20)
WZ_API int wz_relevance_static(const void *features, int T, int H, int W, int D, int dtype,
                               const void *query, int Lq, float *token_scores, float *frame_scores,
                               float *frame_mean, int32_t *device_status, wz_stream_t stream);

/* ------------------------------------------------------------------------ */
/* Projector P (Eq. 17): the condensed tokens through the model's MLP         */
/* ------------------------------------------------------------------------ */

/*
 * out = GELU(tokens W1^T + b1) W2^T + b2, the two-layer projector of
 * LLaVA-style models that Eq. 17 applies after the condensation Psi, with
 * the exact (erf) GELU.  bf16 operands, fp32 accumulation on the tensor
 * cores (tcgen05), bf16 results; the hidden layer [B][C] is stored in bf16
 * in the workspace (as a bf16 model stores it).
 *   tokens [B][D], w1 [C][D], w2 [E][C] bf16 (torch.nn.Linear weights,
 *   out x in); b1 [C], b2 [E] f32, nullable; out [B][E] bf16.
 *   D, C, E: multiples of 64, at most 65536; every pointer 16-byte aligned.
 * Errors: WZ_ERR_INVALID_ARG (null, misaligned, bad size), WZ_ERR_WORKSPACE,
 * WZ_ERR_NO_MEMORY, WZ_ERR_CUDA; nothing is launched on an argument error.
 */
typedef struct {
    const void *tokens;      /* [B][D] bf16                                  */
    int64_t B;
    int D;
    const void *w1;          /* [C][D] bf16                                  */
    const float *b1;         /* [C] or NULL                                  */
    int C;
    const void *w2;          /* [E][C] bf16                                  */
    const float *b2;         /* [E] or NULL                                  */
    int E;
    void *out;               /* [B][E] bf16                                  */
    void *workspace;         /* >= wz_project_workspace_size(B, C), 256-B    */
    size_t workspace_bytes;  /* aligned; NULL = cudaMallocAsync on stream    */
    int32_t *device_status;  /* [1] set nonzero on a bounded-wait timeout;   */
                             /* nullable                                     */
    wz_stream_t stream;
} wz_project_args;

WZ_API size_t wz_project_workspace_size(int64_t B, int C);
WZ_API int wz_project(const wz_project_args *a);

/* ------------------------------------------------------------------------ */
/* Single-level DWT (Eq. 8, 10, 11, 14)                                      */
/* ------------------------------------------------------------------------ */

/* Coefficients per band for a length-n signal: floor((n + F - 1) / 2), F the
 * wavelet's taps (2p, or 10 for bior4.4).  Returns -1 for n < 1 or an
 * unsupported wavelet. */
WZ_API int wz_dwt_len(int n, int wavelet);

/*
 * Filter bank of the wavelet as derived by this library (HOST arrays of F
 * doubles each; any may be NULL).  db<p>: rec_lo is minimum phase with sum
 * sqrt(2); dec_lo is its reverse; rec_hi[k] = (-1)^k rec_lo[2p-1-k]; dec_hi
 * reverses rec_hi.  bior4.4: the 9-tap analysis lowpass in dec_lo[1..9], the
 * 7-tap synthesis lowpass in rec_lo[1..7], both with sum sqrt(2); each
 * high-pass filter is the alternating flip of the other side's lowpass.
 */
WZ_API int wz_wavelet_filters(int wavelet, double *dec_lo, double *dec_hi,
                       double *rec_lo, double *rec_hi);

/*
 * Batched 1D DWT along the last axis: x [rows][L] f32 -> cA, cD
 * [rows][wz_dwt_len(L)] f32, cA[i] = sum_j dec_lo[j] x^[2i+1-j] with x^ the
 * extended signal (mode), cD likewise with dec_hi.
 */
WZ_API int wz_dwt1d(const float *x, int rows, int L, int wavelet, int mode,
             float *cA, float *cD, wz_stream_t stream);

/* Inverse: x[k] = sum_i cA[i] rec_lo[k+F-2-2i] + cD[i] rec_hi[k+F-2-2i],
 * k < L, F = 2p.  Exact inverse of wz_dwt1d in every mode. */
WZ_API int wz_idwt1d(const float *cA, const float *cD, int rows, int L, int wavelet,
              float *x, wz_stream_t stream);

/*
 * Separable 2D DWT of every frame and channel: features [T][H][W][D] (dtype)
 * -> LL, LH, HL, HH [T][h'][w'][D] f32, h' = wz_dwt_len(H), w' likewise.
 * The first band letter is the height filter, the second the width filter.
 */
WZ_API int wz_dwt2d(const void *features, int T, int H, int W, int D, int dtype,
             int wavelet, int mode, float *LL, float *LH, float *HL, float *HH,
             wz_stream_t stream);

/* Inverse of wz_dwt2d: four bands -> out [T][H][W][D] f32. */
WZ_API int wz_idwt2d(const float *LL, const float *LH, const float *HL, const float *HH,
              int T, int H, int W, int D, int wavelet, float *out, wz_stream_t stream);

/* ------------------------------------------------------------------------ */
/* Misc                                                                      */
/* ------------------------------------------------------------------------ */

/* Static English text for a WZ_* status. */
WZ_API const char *wz_status_string(int status);

/* Library version, 10000*major + 100*minor + patch. */
WZ_API int wz_version(void);

/*
 * Self-test of the bounded waits that every pipelined kernel uses (TMA and
 * tensor-core handoffs through shared-memory barriers): one block waits on a
 * barrier that nothing completes, gives up after `timeout_ns` (globaltimer
 * nanoseconds), records WZ_STATUS_WAIT_TIMEOUT in device_status[0] and
 * exits, so the context stays usable.  device_status: [1] int32 device
 * buffer, caller-owned, OR-ed into (not cleared).  Returns WZ_ERR_INVALID_ARG
 * for a null status or a timeout of 0 or over one second, WZ_ERR_CUDA on a
 * launch error, else WZ_OK (asynchronous on `stream`).
 */
#define WZ_STATUS_WAIT_TIMEOUT 0x100
/* Set only by the bounds-checked build of the library (libwavezip_checked.so,
 * compiled with WZ_CHECKED): a kernel computed an out-of-range index for a
 * global write and skipped the write. */
#define WZ_STATUS_BOUNDS 0x200
WZ_API int wz_selftest_bounded_wait(uint64_t timeout_ns, int32_t *device_status, wz_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* WAVEZIP_H */
