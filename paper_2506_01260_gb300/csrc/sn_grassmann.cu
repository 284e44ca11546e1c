// sn_grassmann.cu — the subspace update on the Grassmann manifold (Sec. 4.5,
// closed-form gradient of Sec. 6), on the CUDA cores.
//
// With S = (1/K) sum_t G_t^T G_t accumulated as M = sum_t G_t^T (G_t U) = K S U
// (the tensor-core accumulation lives with the contraction kernels), one step is
//   grad    = -2 S U = -(2/K) M                         Euclidean gradient
//   tangent = grad - U (U^T grad)                        Riemannian gradient
//   A       = U - eta * tangent
//   U_new   = Q of A = Q R with diag(R) > 0               retraction
// The retraction is CholeskyQR2: R1 = chol(A^T A), Q1 = A R1^-1, then the
// same once more on Q1 (the Cholesky factor has a positive diagonal, so Q is
// the unique QR factor with diag(R) > 0).  Gram matrices are accumulated in
// fp64.  Everything here is O(d k^2) and runs once every K iterations.
#include "sn_internal.cuh"

namespace sn {
namespace {

constexpr int kRows = 64;    // rows of A, B per block in the Gram kernel

// out[a, b] += sum_i A[i, a] B[i, b] (k x k, fp64), A, B fp32 [d, k] row-major.
// Each block adds the products of its chunks of kRows rows with fp64 atomics.
__global__ void k_gram(const float *__restrict__ A, const float *__restrict__ B, int d, int k,
                       double *__restrict__ out)
{
    extern __shared__ float sm[];               // [kRows][k] of A, then of B
    float *sa = sm, *sb = sm + kRows * k;
    const int npair = k * k;
    for (int r0 = blockIdx.x * kRows; r0 < d; r0 += gridDim.x * kRows) {
        const int nr = min(kRows, d - r0);
        __syncthreads();
        for (int e = threadIdx.x; e < kRows * k; e += blockDim.x) {
            const int r = e / k;
            sa[e] = r < nr ? A[(size_t)(r0 + r) * k + e % k] : 0.f;
            sb[e] = r < nr ? B[(size_t)(r0 + r) * k + e % k] : 0.f;
        }
        __syncthreads();
        for (int pr = threadIdx.x; pr < npair; pr += blockDim.x) {
            const int a = pr / k, bb = pr - a * k;
            double s = 0.0;
            for (int r = 0; r < nr; ++r)
                s += (double)sa[r * k + a] * (double)sb[r * k + bb];
            atomicAdd(out + pr, s);
        }
    }
}

// out[i, :] = A[i, :] + s1 * B[i, :] + s2 * (A[i, :] W)   (W k x k fp64)
__global__ void k_rowmix(const float *__restrict__ A, const float *__restrict__ B,
                         const double *__restrict__ W, int d, int k, double s1, double s2,
                         float *__restrict__ out)
{
    extern __shared__ double sw[];
    for (int e = threadIdx.x; e < k * k; e += blockDim.x)
        sw[e] = W[e];
    __syncthreads();
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < (int64_t)d * k;
         e += (int64_t)gridDim.x * blockDim.x) {
        const int64_t i = e / k;
        const int j = (int)(e - i * k);
        double s = 0.0;
        for (int l = 0; l < k; ++l)
            s += (double)A[i * k + l] * sw[l * k + j];
        out[e] = (float)((double)A[e] + s1 * (double)B[e] + s2 * s);
    }
}

// In place: the upper Cholesky factor R of the symmetric positive-definite
// G (k x k, fp64), G = R^T R; the strictly lower part is zeroed.  One block.
// Sets *bad when a pivot is not positive.
__global__ void k_cholesky(double *G, int k, unsigned int *bad)
{
    for (int j = 0; j < k; ++j) {
        // R[j, j] = sqrt(G[j, j] - sum_{l<j} R[l, j]^2)
        __syncthreads();
        if (threadIdx.x == 0) {
            double s = G[j * k + j];
            for (int l = 0; l < j; ++l)
                s -= G[l * k + j] * G[l * k + j];
            if (!(s > 0.0)) {
                atomicOr(bad, SN_EBIT_NUMERIC);
                s = 1.0;
            }
            G[j * k + j] = sqrt(s);
        }
        __syncthreads();
        // R[j, c] = (G[j, c] - sum_{l<j} R[l, j] R[l, c]) / R[j, j], c > j
        const double rjj = G[j * k + j];
        for (int c = j + 1 + threadIdx.x; c < k; c += blockDim.x) {
            double s = G[j * k + c];
            for (int l = 0; l < j; ++l)
                s -= G[l * k + j] * G[l * k + c];
            G[j * k + c] = s / rjj;
        }
    }
    __syncthreads();
    for (int e = threadIdx.x; e < k * k; e += blockDim.x)
        if (e / k > e % k)
            G[e] = 0.0;
}

// out[i, :] = A[i, :] R^-1 (R upper triangular k x k fp64): solve x R = a per row.
__global__ void k_solve_rows(const float *__restrict__ A, const double *__restrict__ R, int d,
                             int k, float *__restrict__ out)
{
    extern __shared__ double sr[];
    for (int e = threadIdx.x; e < k * k; e += blockDim.x)
        sr[e] = R[e];
    __syncthreads();
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < d;
         i += (int64_t)gridDim.x * blockDim.x) {
        double x[128];
        for (int j = 0; j < k; ++j) {
            double s = (double)A[i * k + j];
            for (int l = 0; l < j; ++l)
                s -= x[l] * sr[l * k + j];
            x[j] = s / sr[j * k + j];
            out[i * k + j] = (float)x[j];
        }
    }
}

// acc += sum(G^2) - sum(Cg^2) over bf16 G [T, d] and Cg [T, k]
__global__ void k_residual(const __nv_bfloat16 *__restrict__ G, int64_t ng,
                           const __nv_bfloat16 *__restrict__ Cg, int64_t nc, double *acc)
{
    double s = 0.0;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    const int64_t t0 = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    for (int64_t e = t0; e < ng / 8; e += stride) {
        const uint4 w = __ldg((const uint4 *)G + e);
        const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const float lo = __uint_as_float(ws[q] << 16), hi = __uint_as_float(ws[q] & 0xFFFF0000u);
            s += (double)lo * lo + (double)hi * hi;
        }
    }
    for (int64_t e = (ng / 8) * 8 + t0; e < ng; e += stride) {
        const float v = __bfloat162float(G[e]);
        s += (double)v * v;
    }
    for (int64_t e = t0; e < nc; e += stride) {
        const float v = __bfloat162float(Cg[e]);
        s -= (double)v * v;
    }
    for (int o = 16; o > 0; o >>= 1)
        s += __shfl_xor_sync(0xffffffffu, s, o);
    __shared__ double red[32];
    if ((threadIdx.x & 31) == 0)
        red[threadIdx.x >> 5] = s;
    __syncthreads();
    if (threadIdx.x == 0) {
        double t = 0.0;
        for (int w = 0; w < (int)(blockDim.x >> 5); ++w)
            t += red[w];
        atomicAdd(acc, t);
    }
}

int grid_of(int64_t n, int block)
{
    int dev = 0, sms = 148;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t want = (n + block - 1) / block;
    return (int)(want < 4 * sms ? (want > 0 ? want : 1) : 4 * sms);
}

size_t align256(size_t v) { return (v + 255) & ~(size_t)255; }

}  // namespace

cudaError_t grassmann_residual(const sn_basis &b, const __nv_bfloat16 *G,
                               const __nv_bfloat16 *Cg, int64_t T, double *acc, cudaStream_t s)
{
    k_residual<<<grid_of(T * b.d / 8, 256), 256, 0, s>>>(G, T * b.d, Cg, T * b.k, acc);
    count_launch();
    return cudaGetLastError();
}

// workspace: Y, R1, R2 (k x k fp64 each) | A, Q1 (d x k fp32 each)
size_t grassmann_step_workspace(const sn_basis &b)
{
    const size_t kk = align256(sizeof(double) * (size_t)b.k * b.k);
    const size_t dk = align256(sizeof(float) * (size_t)b.d * b.k);
    return 3 * kk + 2 * dk;
}

cudaError_t grassmann_step(const sn_basis &b, const float *M, int K, float eta, float *U_new,
                           void *workspace, cudaStream_t s)
{
    const int d = b.d, k = b.k;
    const size_t kk = align256(sizeof(double) * (size_t)k * k);
    const size_t dk = align256(sizeof(float) * (size_t)d * k);
    char *w = (char *)workspace;
    double *Y = (double *)w, *R1 = (double *)(w + kk), *R2 = (double *)(w + 2 * kk);
    float *A = (float *)(w + 3 * kk), *Q1 = (float *)(w + 3 * kk + dk);
    const size_t gram_smem = sizeof(float) * 2 * kRows * k;
    const size_t kk_smem = sizeof(double) * (size_t)k * k;
    const int gblocks = (d + kRows - 1) / kRows;
    cudaError_t e;
    if ((e = cudaFuncSetAttribute(k_gram, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)gram_smem)) != cudaSuccess ||
        (e = cudaFuncSetAttribute(k_rowmix, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)kk_smem)) != cudaSuccess ||
        (e = cudaFuncSetAttribute(k_solve_rows, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)kk_smem)) != cudaSuccess)
        return e;
    // Y = U^T M;  A = U - eta * (c M - U (c Y)) with c = -2 / K
    const double c = -2.0 / K;
    if ((e = cudaMemsetAsync(w, 0, 3 * kk, s)) != cudaSuccess)
        return e;
    k_gram<<<gblocks, 256, gram_smem, s>>>(b.u32, M, d, k, Y);
    k_rowmix<<<grid_of((int64_t)d * k, 256), 256, kk_smem, s>>>(b.u32, M, Y, d, k, -eta * c,
                                                                   eta * c, A);
    // CholeskyQR2
    k_gram<<<gblocks, 256, gram_smem, s>>>(A, A, d, k, R1);
    k_cholesky<<<1, 128, 0, s>>>(R1, k, b.err);
    k_solve_rows<<<grid_of(d, 128), 128, kk_smem, s>>>(A, R1, d, k, Q1);
    k_gram<<<gblocks, 256, gram_smem, s>>>(Q1, Q1, d, k, R2);
    k_cholesky<<<1, 128, 0, s>>>(R2, k, b.err);
    k_solve_rows<<<grid_of(d, 128), 128, kk_smem, s>>>(Q1, R2, d, k, U_new);
    count_launch(8);
    return cudaGetLastError();
}

}  // namespace sn
