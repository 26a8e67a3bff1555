// Condensed tokens Z_m = W_m X_m on CUDA cores in fp32 (Eq. 16, 18).
//
// Used for fp32 features (the tensor cores would need a split of X as well)
// and as an independent second path for bf16.  Tiles of 64 output rows x 64
// channels, K in steps of 16 tokens, 4 x 4 outputs per thread.
#include "wz_internal.cuh"

namespace wz {

template <typename Tin>
__global__ void __launch_bounds__(256) condense_simt_kernel(Ctx c) {
    pdl_wait();
    pdl_trigger();
    __shared__ float Ws[16][68];
    __shared__ float Xs[16][68];
    const int64_t f = blockIdx.x;
    const int n = c.n[f];
    const int r0 = blockIdx.y * 64;
    if (r0 >= n) return;
    const int c0 = blockIdx.z * 64;
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    const int N = c.N, D = c.D;
    const int64_t orow = c.off[f];
    const float *Wr = static_cast<const float *>(c.Wop) + (size_t)(orow + r0) * c.K_pad;
    const Tin *Xf = static_cast<const Tin *>(c.X) + (size_t)f * N * D;
    float acc[4][4] = {};
    for (int k0 = 0; k0 < N; k0 += 16) {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const int idx = tid + e * 256;
            const int r = idx >> 4, kk = idx & 15;
            Ws[kk][r] = (r0 + r < n && k0 + kk < c.K_pad) ? Wr[(size_t)r * c.K_pad + k0 + kk] : 0.f;
            const int xk = idx >> 6, ch = idx & 63;
            Xs[xk][ch] = (k0 + xk < N && c0 + ch < D)
                             ? load_scalar<Tin>(Xf + (size_t)(k0 + xk) * D + c0 + ch) : 0.f;
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < 16; ++kk) {
            float av[4], bv[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                av[i] = Ws[kk][ty * 4 + i];
                bv[i] = Xs[kk][tx * 4 + i];
            }
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(av[i], bv[j], acc[i][j]);
        }
        __syncthreads();
    }
    Tin *out = static_cast<Tin *>(c.out);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int r = r0 + ty * 4 + i;
        if (r >= n || !wz_in_range(c.status, (int64_t)orow + r < c.rows_total)) continue;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int ch = c0 + tx * 4 + j;
            if (ch < D) out[(size_t)(orow + r) * D + ch] = from_float<Tin>(acc[i][j]);
        }
    }
}

cudaError_t launch_condense_simt(const Ctx &c, cudaStream_t s) {
    const dim3 grid((unsigned)((int64_t)c.V * c.T), (unsigned)((c.N + 63) / 64), (unsigned)((c.D + 63) / 64));
    void *args[] = {const_cast<Ctx *>(&c)};
    const void *fn = c.dtype == WZ_DTYPE_BF16 ? (const void *)condense_simt_kernel<__nv_bfloat16>
                                              : (const void *)condense_simt_kernel<float>;
    return launch_kernel(fn, grid, dim3(256), 0, s, args, c.pdl != 0);
}

}  // namespace wz
