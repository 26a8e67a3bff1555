// wz_relevance_static: the relevance scores of wz_relevance, computed with
// no device-memory allocation at all.
//
// Some callers cannot allocate device memory when they need the scores: code
// running while a stream is being captured into a CUDA graph where the
// capture must not contain allocation nodes, serving loops that freeze their
// memory budget after start-up so that a request can never fail on an
// out-of-memory or stall on the allocator, and hosts whose device memory is
// owned by another framework's caching allocator that a foreign cudaMalloc
// would bypass.  Such callers still pass their own inputs and outputs; the
// intermediate sums live in one fixed array compiled into this library.
//
// The array `g_relevance_scratch` (WZ_STATIC_SCRATCH_BYTES) exists on every
// GPU that loads the library, from load until the process exits.  Its name
// is only a host-side stand-in in host code, so the device address is looked
// up once per device with cudaGetSymbolAddress (with that device current) on
// the first call made on that device, and passed to the kernels.  A 16-byte
// slot of the array is the status word of the bounded waits when the caller
// passes none; it is zeroed on the stream at every call.
#include <mutex>

#include "wz_internal.cuh"

namespace wz {

namespace {

static __device__ __align__(256) unsigned char g_relevance_scratch[WZ_STATIC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mu;
void *g_scratch_addr[kMaxDevices];

// Device address of the fixed array on the current device (looked up once).
int static_scratch(void **out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        cudaGetLastError();
        return WZ_ERR_CUDA;
    }
    if (dev < 0 || dev >= kMaxDevices) return WZ_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lock(g_scratch_mu);
    if (!g_scratch_addr[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_relevance_scratch) != cudaSuccess || p == nullptr) {
            cudaGetLastError();
            return WZ_ERR_CUDA;
        }
        g_scratch_addr[dev] = p;
    }
    *out = g_scratch_addr[dev];
    return WZ_OK;
}

size_t up256(size_t x) { return (x + 255) / 256 * 256; }

// Byte offsets of the sub-buffers carved from the fixed array for T frames
// of D channels and a relevance grid of G1 CTAs.
struct ScratchLayout {
    size_t q32, q64, vpar, part, fr, status, total;
};

ScratchLayout scratch_layout(int T, int D, int G1) {
    ScratchLayout L{};
    size_t o = 0;
    L.q32 = o;
    o = up256(o + (size_t)D * 4);
    L.q64 = o;
    o = up256(o + (size_t)D * 8);
    L.vpar = o;
    o = up256(o + sizeof(VideoPar));
    L.part = o;
    o = up256(o + ((size_t)G1 + T) * D * 4);
    L.fr = o;
    o = up256(o + (size_t)T * 4 * 8);
    L.status = o;
    o = up256(o + 16);
    L.total = o;
    return L;
}

size_t scratch_bytes(int T, int D, int G1) { return scratch_layout(T, D, G1).total; }

bool is_aligned(const void *p, size_t a) { return ((uintptr_t)p % a) == 0; }

}  // namespace

}  // namespace wz

using namespace wz;

extern "C" int wz_relevance_static(const void *features, int T, int H, int W, int D, int dtype,
                                   const void *query, int Lq, float *token_scores, float *frame_scores,
                                   float *frame_mean, int32_t *device_status, wz_stream_t stream) {
    if (T < 1 || H < 1 || W < 1 || D < 1 || Lq < 1) return WZ_ERR_INVALID_ARG;
    if (dtype != WZ_DTYPE_BF16 && dtype != WZ_DTYPE_F32) return WZ_ERR_INVALID_ARG;
    if (D % 8 != 0) return WZ_ERR_UNSUPPORTED;
    if (T > WZ_MAX_T || H > WZ_MAX_HW || W > WZ_MAX_HW || D > WZ_MAX_D) return WZ_ERR_UNSUPPORTED;
    if (dtype == WZ_DTYPE_F32 && D > WZ_MAX_D / 2) return WZ_ERR_UNSUPPORTED;
    if (!features || !query || !token_scores || !frame_scores) return WZ_ERR_INVALID_ARG;
    if (!is_aligned(features, 16) || !is_aligned(query, 16) || !is_aligned(token_scores, 4) ||
        !is_aligned(frame_scores, 4) || (frame_mean && !is_aligned(frame_mean, 4)) ||
        !is_aligned(device_status, 4))
        return WZ_ERR_INVALID_ARG;
    // Sizes that cannot fit even with a one-CTA relevance grid are refused
    // before the CUDA runtime is touched.
    if (scratch_bytes(T, D, 1) > (size_t)WZ_STATIC_SCRATCH_BYTES) return WZ_ERR_WORKSPACE;

    Ctx c{};
    c.V = 1;
    c.T = T;
    c.H = H;
    c.W = W;
    c.D = D;
    c.N = H * W;
    c.dtype = dtype;
    c.G1 = relevance_grid(c);
    if (c.G1 < 1) {
        cudaGetLastError();
        return WZ_ERR_CUDA;
    }
    c.L1 = ((int64_t)T * c.N + c.G1 - 1) / c.G1;

    // Carve the fixed array.  Every byte the kernels read is written earlier
    // in the same call, except the status word, which is cleared below when
    // the caller passes none.
    const ScratchLayout o = scratch_layout(T, D, c.G1);
    if (o.total > (size_t)WZ_STATIC_SCRATCH_BYTES) return WZ_ERR_WORKSPACE;

    void *base = nullptr;
    const int st = static_scratch(&base);
    if (st != WZ_OK) return st;
    char *b = static_cast<char *>(base);
    c.qbar32 = reinterpret_cast<float *>(b + o.q32);
    c.qbar64 = reinterpret_cast<double *>(b + o.q64);
    c.vpar = reinterpret_cast<VideoPar *>(b + o.vpar);
    c.part = reinterpret_cast<float *>(b + o.part);
    c.fr = reinterpret_cast<double *>(b + o.fr);
    // The bounded waits of the relevance pass (and the index checks of the
    // checked build) record failures in a status word: the caller's, else
    // the array's own slot, zeroed on the stream (cudaMemsetAsync allocates
    // nothing).
    c.status = device_status ? device_status : reinterpret_cast<int *>(b + o.status);
    c.X = features;
    c.Q = query;
    c.a = token_scores;
    c.frame_scores = frame_scores;
    c.frame_mean = frame_mean;

    const VideoPar par{0, Lq, 0, 0, 0};
    const cudaStream_t s = (cudaStream_t)stream;
    if ((!device_status && cudaMemsetAsync(c.status, 0, sizeof(int), s) != cudaSuccess) ||
        launch_query_pool(c, &par, s) != cudaSuccess || launch_relevance_pass(c, s) != cudaSuccess ||
        launch_frame_stats(c, s) != cudaSuccess) {
        cudaGetLastError();
        return WZ_ERR_CUDA;
    }
    return WZ_OK;
}
