// sn_adamw.cu — the row-constant AdamW step that keeps W_p2 inside the
// subspace (Sec. 5), memory-bound, on the CUDA cores.
//
// W is the torch weight [rows = d, cols = n]; its columns are the paper's rows
// of W_p2 (the d-vectors that live in S).  One step t >= 1:
//   M = b1 M + (1 - b1) g,  V = b2 V + (1 - b2) g^2          (in place, fp32)
//   mu[c] = mean over the column of V / (1 - b2^t)             (the paper's row mean)
//   W = W - lr (M / (1 - b1^t)) / (sqrt(mu[c]) + eps) - lambda W
// Pass 1 updates the moments and adds each block's column sums of V^ to a
// zeroed [cols] fp32 workspace with one atomic per column and block; pass 2
// updates W.  Each thread owns one column of a block of rows, so every access
// is coalesced along the columns.
#include "sn_internal.cuh"

namespace sn {
namespace {

constexpr int kCols = 256;   // columns per block (one per thread)
constexpr int kRows = 64;    // rows per block

template <typename GT>
__device__ __forceinline__ float load_grad(const GT *g, int64_t e);
template <>
__device__ __forceinline__ float load_grad<float>(const float *g, int64_t e)
{
    return __ldg(g + e);
}
template <>
__device__ __forceinline__ float load_grad<__nv_bfloat16>(const __nv_bfloat16 *g, int64_t e)
{
    return __bfloat162float(g[e]);
}

template <typename GT>
__global__ void __launch_bounds__(kCols) k_adamw_moments(const GT *__restrict__ g,
                                                          float *__restrict__ M,
                                                          float *__restrict__ V, int64_t rows,
                                                          int64_t cols, float b1, float b2,
                                                          float vcorr, float *__restrict__ colsum)
{
    const int64_t c = (int64_t)blockIdx.x * kCols + threadIdx.x;
    const int64_t r0 = (int64_t)blockIdx.y * kRows;
    if (c >= cols)
        return;
    const int64_t r1 = r0 + kRows < rows ? r0 + kRows : rows;
    float s = 0.f;
    for (int64_t r = r0; r < r1; ++r) {
        const int64_t e = r * cols + c;
        const float gv = load_grad(g, e);
        const float m = b1 * M[e] + (1.f - b1) * gv;
        const float v = b2 * V[e] + (1.f - b2) * gv * gv;
        M[e] = m;
        V[e] = v;
        s += v * vcorr;
    }
    atomicAdd(colsum + c, s);
}

__global__ void __launch_bounds__(kCols) k_adamw_apply(float *__restrict__ W,
                                                        const float *__restrict__ M, int64_t rows,
                                                        int64_t cols, float lr, float mcorr,
                                                        float eps, float lam, float inv_rows,
                                                        const float *__restrict__ colsum)
{
    const int64_t c = (int64_t)blockIdx.x * kCols + threadIdx.x;
    const int64_t r0 = (int64_t)blockIdx.y * kRows;
    if (c >= cols)
        return;
    const float alpha = 1.f / (sqrtf(colsum[c] * inv_rows) + eps);
    const float step = lr * mcorr * alpha;
    const int64_t r1 = r0 + kRows < rows ? r0 + kRows : rows;
    for (int64_t r = r0; r < r1; ++r) {
        const int64_t e = r * cols + c;
        const float w = W[e];
        W[e] = w - step * M[e] - lam * w;
    }
}

}  // namespace

cudaError_t adamw_rowconst(bool grad_bf16, float *W, const void *g, float *M, float *V,
                           int64_t rows, int64_t cols, int64_t t, float lr, float b1, float b2,
                           float eps, float lam, float *colsum, cudaStream_t s)
{
    cudaError_t e = cudaMemsetAsync(colsum, 0, sizeof(float) * (size_t)cols, s);
    if (e != cudaSuccess)
        return e;
    // bias corrections of step t, in double before rounding to fp32
    const float vcorr = (float)(1.0 / (1.0 - pow((double)b2, (double)t)));
    const float mcorr = (float)(1.0 / (1.0 - pow((double)b1, (double)t)));
    const dim3 grid((unsigned)((cols + kCols - 1) / kCols), (unsigned)((rows + kRows - 1) / kRows));
    if (grad_bf16)
        k_adamw_moments<__nv_bfloat16><<<grid, kCols, 0, s>>>(
            (const __nv_bfloat16 *)g, M, V, rows, cols, b1, b2, vcorr, colsum);
    else
        k_adamw_moments<float><<<grid, kCols, 0, s>>>((const float *)g, M, V, rows, cols, b1, b2,
                                                     vcorr, colsum);
    k_adamw_apply<<<grid, kCols, 0, s>>>(W, M, rows, cols, lr, mcorr, eps, lam,
                                         (float)(1.0 / (double)rows), colsum);
    count_launch(2);
    return cudaGetLastError();
}

}  // namespace sn
