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
// the unique QR factor with diag(R) > 0).  The O(d k^2) products run in fp32
// on the CUDA cores (Gram matrices as per-64-row partial products summed in
// fp64 without atomics; A R^-1 as a row-by-matrix product), the O(k^3)
// Cholesky factor and its triangular inverse in fp32 in one block (this GPU's
// fp64 rate is a small fraction of its fp32 rate).  A is within a small step
// of orthonormal, so its Gram matrix is near the identity and the second pass
// removes what the first leaves; it all runs once every K iterations.
#include "sn_internal.cuh"

namespace sn {
namespace {

constexpr int kRows = 64;    // rows of A, B per block in the Gram kernel
constexpr int kMixRows = 4;  // rows per pass of the row-mix kernel

// part[blk, a, b] = sum over the block's kRows rows i of A[i, a] B[i, b] (fp32
// products and sums over 64 rows); A, B fp32 [d, k] row-major.  Each thread
// owns 4 x 4 tiles of (a, b) pairs: per row 8 shared loads feed 16 FMAs.
__global__ void __launch_bounds__(256) k_gram_part(const float *__restrict__ A,
                                                   const float *__restrict__ B, int d, int k,
                                                   float *__restrict__ part)
{
    extern __shared__ float sm[];               // [kRows][k4] of A, then of B (k4 = k padded to 4)
    const int k4 = (k + 3) & ~3;
    float *sa = sm, *sb = sm + kRows * k4;
    const int r0 = blockIdx.x * kRows;
    const int nr = min(kRows, d - r0);
    for (int e = threadIdx.x; e < kRows * k4; e += blockDim.x) {
        const int r = e / k4, c = e - r * k4;
        const bool in = r < nr && c < k;
        sa[e] = in ? A[(size_t)(r0 + r) * k + c] : 0.f;
        sb[e] = in ? B[(size_t)(r0 + r) * k + c] : 0.f;
    }
    __syncthreads();
    float *dst = part + (size_t)blockIdx.x * k * k;
    const int nt = k4 / 4;
    for (int tl = threadIdx.x; tl < nt * nt; tl += blockDim.x) {
        const int ta = 4 * (tl / nt), tb = 4 * (tl % nt);
        float acc[4][4] = {};
        for (int r = 0; r < nr; ++r) {
            const float4 x = *(const float4 *)(sa + r * k4 + ta);
            const float4 y = *(const float4 *)(sb + r * k4 + tb);
            const float xa[4] = {x.x, x.y, x.z, x.w}, yb[4] = {y.x, y.y, y.z, y.w};
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j)
                    acc[i][j] = fmaf(xa[i], yb[j], acc[i][j]);
        }
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int j = 0; j < 4; ++j)
                if (ta + i < k && tb + j < k)
                    dst[(ta + i) * k + tb + j] = acc[i][j];
    }
}

// out[e] = sum over the nblk blocks of part[blk, e], summed in fp64 and stored
// in fp32 (e < k*k): four lanes per element, each summing every fourth block,
// then a shuffle.
__global__ void __launch_bounds__(256) k_gram_sum(const float *__restrict__ part, int nblk, int kk,
                                                  float *__restrict__ out)
{
    const int e = (blockIdx.x * blockDim.x + threadIdx.x) >> 2, q = threadIdx.x & 3;
    double s = 0.0;
    if (e < kk)
        for (int b = q; b < nblk; b += 4)
            s += (double)part[(size_t)b * kk + e];
    s += __shfl_xor_sync(0xffffffffu, s, 1);
    s += __shfl_xor_sync(0xffffffffu, s, 2);
    if (e < kk && q == 0)
        out[e] = (float)s;
}

// out[i, :] = alpha A[i, :] + beta B[i, :] + gamma (A[i, :] W)  (W k x k fp32).
// One thread per column (k <= 128); kMixRows rows of A staged per pass give
// each thread kMixRows independent accumulations.
__global__ void __launch_bounds__(128) k_rowmix(const float *__restrict__ A,
                                                const float *__restrict__ B,
                                                const float *__restrict__ W, int d, int k,
                                                float alpha, float beta, float gamma,
                                                float *__restrict__ out)
{
    extern __shared__ float sw[];               // W (k x k), then kMixRows rows of A
    float *srow = sw + k * k;
    for (int e = threadIdx.x; e < k * k; e += blockDim.x)
        sw[e] = W[e];
    const int j = threadIdx.x;
    for (int i0 = kMixRows * blockIdx.x; i0 < d; i0 += kMixRows * gridDim.x) {
        __syncthreads();
        for (int e = threadIdx.x; e < kMixRows * k; e += blockDim.x) {
            const int r = e / k;
            srow[e] = i0 + r < d ? A[(size_t)i0 * k + e] : 0.f;
        }
        __syncthreads();
        if (j < k) {
            float acc[kMixRows] = {};
            for (int l = 0; l < k; ++l) {
                const float w = sw[l * k + j];
#pragma unroll
                for (int r = 0; r < kMixRows; ++r)
                    acc[r] = fmaf(srow[r * k + l], w, acc[r]);
            }
#pragma unroll
            for (int r = 0; r < kMixRows; ++r)
                if (i0 + r < d) {
                    const size_t o = (size_t)(i0 + r) * k + j;
                    out[o] = alpha * srow[r * k + j] + beta * B[o] + gamma * acc[r];
                }
        }
    }
}

// Rinv = R^-1 for R the upper Cholesky factor of the symmetric positive-definite
// G (k x k), G = R^T R, in fp32 (G is the Gram matrix of a nearly orthonormal
// A, within a small step of the identity).  One block of 128 threads, all in
// shared memory: R in the upper triangle of s, R^-1 transposed in its strictly
// lower triangle, the diagonal of R^-1 apart.  Sets *bad when a pivot is not
// positive.
__global__ void __launch_bounds__(128) k_cholesky_inv(const float *__restrict__ G, int k,
                                                      float *__restrict__ Rinv, unsigned int *bad)
{
    extern __shared__ float sc[];                // k x k, then k (diagonal of R^-1)
    float *dinv = sc + k * k;
    for (int e = threadIdx.x; e < k * k; e += blockDim.x)
        sc[e] = G[e];
    __syncthreads();
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int j = 0; j < k; ++j) {
        // R[j, j] = sqrt(G[j, j] - sum_{l<j} R[l, j]^2), one warp
        if (warp == 0) {
            float t = 0.f;
            for (int l = lane; l < j; l += 32)
                t = fmaf(sc[l * k + j], sc[l * k + j], t);
            for (int o = 16; o > 0; o >>= 1)
                t += __shfl_xor_sync(0xffffffffu, t, o);
            if (lane == 0) {
                float v = sc[j * k + j] - t;
                if (!(v > 0.f)) {
                    atomicOr(bad, SN_EBIT_NUMERIC);
                    v = 1.f;
                }
                sc[j * k + j] = sqrtf(v);
            }
        }
        __syncthreads();
        // R[j, c] = (G[j, c] - sum_{l<j} R[l, j] R[l, c]) / R[j, j], c > j
        const float rjj = sc[j * k + j];
        for (int c = j + 1 + threadIdx.x; c < k; c += blockDim.x) {
            float t = sc[j * k + c];
            for (int l = 0; l < j; ++l)
                t = fmaf(-sc[l * k + j], sc[l * k + c], t);
            sc[j * k + c] = t / rjj;
        }
        __syncthreads();
    }
    // column c of R^-1 (R x = e_c, x_i = 0 for i > c), kept transposed at
    // sc[c * k + i] for i < c
    for (int c = threadIdx.x; c < k; c += blockDim.x) {
        dinv[c] = 1.f / sc[c * k + c];
        for (int i = c - 1; i >= 0; --i) {
            float t = sc[i * k + c] * dinv[c];
            for (int l = i + 1; l < c; ++l)
                t = fmaf(sc[i * k + l], sc[c * k + l], t);
            sc[c * k + i] = -t / sc[i * k + i];
        }
    }
    __syncthreads();
    for (int e = threadIdx.x; e < k * k; e += blockDim.x) {
        const int i = e / k, c = e - i * k;
        Rinv[e] = i < c ? sc[c * k + i] : (i == c ? dinv[c] : 0.f);
    }
}

// acc += sum(G^2) - sum(Cg^2) over bf16 G [T, d] and Cg [T, k]
__global__ void k_residual(const __nv_bfloat16 *__restrict__ G, int64_t ng,
                           const __nv_bfloat16 *__restrict__ Cg, int64_t nc, double *acc)
{
    // squares summed in fp32 over 16 chunks of 8 (128 positive terms) at a
    // time, then into fp64: this GPU's fp64 rate could not keep up with one
    // fp64 operation per element
    double s = 0.0;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    const int64_t t0 = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t n8 = ng / 8;
    for (int64_t e0 = t0; e0 < n8; e0 += 16 * stride) {
        float f = 0.f;
        for (int64_t e1 = e0; e1 < e0 + 16 * stride && e1 < n8; e1 += 4 * stride) {
            uint4 w[4];
#pragma unroll
            for (int u = 0; u < 4; ++u)     // four 16-byte loads in flight
                w[u] = e1 + u * stride < n8 ? __ldg((const uint4 *)G + e1 + u * stride)
                                            : make_uint4(0, 0, 0, 0);
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const uint32_t ws[4] = {w[u].x, w[u].y, w[u].z, w[u].w};
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const float lo = __uint_as_float(ws[q] << 16);
                    const float hi = __uint_as_float(ws[q] & 0xFFFF0000u);
                    f = fmaf(lo, lo, fmaf(hi, hi, f));
                }
            }
        }
        s += (double)f;
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

// workspace: Y, G1, G2, R1^-1, R2^-1 (k x k fp32 each) | A, Q1 (d x k fp32
// each) | Gram partials (one k x k fp32 block per kRows rows)
size_t grassmann_step_workspace(const sn_basis &b)
{
    const size_t kk = align256(sizeof(float) * (size_t)b.k * b.k);
    const size_t dk = align256(sizeof(float) * (size_t)b.d * b.k);
    const size_t parts = align256(sizeof(float) * (size_t)((b.d + kRows - 1) / kRows) * b.k * b.k);
    return 5 * kk + 2 * dk + parts;
}

cudaError_t grassmann_step(const sn_basis &b, const float *M, int K, float eta, float *U_new,
                           void *workspace, cudaStream_t s)
{
    const int d = b.d, k = b.k;
    const size_t kk = align256(sizeof(float) * (size_t)k * k);
    const size_t dk = align256(sizeof(float) * (size_t)d * k);
    char *w = (char *)workspace;
    float *Y = (float *)w, *G1 = (float *)(w + kk), *G2 = (float *)(w + 2 * kk);
    float *R1i = (float *)(w + 3 * kk), *R2i = (float *)(w + 4 * kk);
    float *A = (float *)(w + 5 * kk), *Q1 = (float *)(w + 5 * kk + dk);
    float *part = (float *)(w + 5 * kk + 2 * dk);
    const int nblk = (d + kRows - 1) / kRows;
    const size_t gram_smem = sizeof(float) * 2 * kRows * ((k + 3) & ~3);
    const size_t mix_smem = sizeof(float) * ((size_t)k * k + (size_t)kMixRows * k);
    const size_t chol_smem = sizeof(float) * ((size_t)k * k + k);
    cudaError_t e;
    if ((e = cudaFuncSetAttribute(k_gram_part, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)gram_smem)) != cudaSuccess ||
        (e = cudaFuncSetAttribute(k_rowmix, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)mix_smem)) != cudaSuccess ||
        (e = cudaFuncSetAttribute(k_cholesky_inv, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)chol_smem)) != cudaSuccess)
        return e;
    const int mix_grid = grid_of((int64_t)(d + kMixRows - 1) / kMixRows * 128, 128);
    const int sum_grid = (4 * k * k + 255) / 256;
    auto gram = [&](const float *X, const float *Z, float *out) {
        k_gram_part<<<nblk, 256, gram_smem, s>>>(X, Z, d, k, part);
        k_gram_sum<<<sum_grid, 256, 0, s>>>(part, nblk, k * k, out);
    };
    // Y = U^T M;  A = U - eta * (c M - U (c Y)) with c = -2 / K
    const double c = -2.0 / K;
    gram(b.u32, M, Y);
    k_rowmix<<<mix_grid, 128, mix_smem, s>>>(b.u32, M, Y, d, k, 1.f, (float)(-eta * c),
                                             (float)(eta * c), A);
    // CholeskyQR2: Q = A R^-1 with R = chol(A^T A), twice
    gram(A, A, G1);
    k_cholesky_inv<<<1, 128, chol_smem, s>>>(G1, k, R1i, b.err);
    k_rowmix<<<mix_grid, 128, mix_smem, s>>>(A, A, R1i, d, k, 0.f, 0.f, 1.f, Q1);
    gram(Q1, Q1, G2);
    k_cholesky_inv<<<1, 128, chol_smem, s>>>(G2, k, R2i, b.err);
    k_rowmix<<<mix_grid, 128, mix_smem, s>>>(Q1, Q1, R2i, d, k, 0.f, 0.f, 1.f, U_new);
    count_launch(12);
    return cudaGetLastError();
}

}  // namespace sn
