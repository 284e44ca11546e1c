// sn_simt.cu — CUDA-core kernels: the fp32 path of every boundary operation
// and the one-off preparation of a basis handle's padded copies of U.
//
// fp32 inputs must match the fp64 definition to ~1e-5 relative, which rules
// out TF32/bf16 tensor-core inputs; these kernels use fp32 FMA with fp32
// accumulation in ascending-d order per output.
#include <algorithm>

#include "sn_internal.cuh"

namespace sn {
namespace {

__device__ __forceinline__ float to_f(float v) { return v; }
__device__ __forceinline__ float to_f(__nv_bfloat16 v) { return __bfloat162float(v); }
template <typename E> __device__ __forceinline__ E from_f(float v);
template <> __device__ __forceinline__ float from_f<float>(float v) { return v; }
template <> __device__ __forceinline__ __nv_bfloat16 from_f<__nv_bfloat16>(float v)
{
    return __float2bfloat16_rn(v);
}

constexpr int KMAX = 128;   // largest k a handle accepts

// Row state of a token inside a block: skip (t >= T), compute, or zero (bad id).
enum : int { ROW_SKIP = 0, ROW_OK = 1, ROW_BAD = 2 };

// Validate token t's id and position; returns the row state and the element
// offsets of its token-table and positional-table rows.
__device__ __forceinline__ int token_rows(int64_t t, int64_t T, bool gather,
                                          const int32_t *ids, const int32_t *pos,
                                          int seq_len, int64_t vocab, bool has_pe, int d,
                                          int64_t *tok_off, int64_t *pe_off,
                                          unsigned int *err)
{
    *tok_off = 0;
    *pe_off = 0;
    if (t >= T)
        return ROW_SKIP;
    if (!gather)
        return ROW_OK;
    int64_t id = ids[t];
    int64_t p = 0;
    bool bad = id < 0 || id >= vocab;
    if (has_pe) {
        p = pos ? (int64_t)pos[t] : t % seq_len;
        bad = bad || p < 0 || p >= seq_len;
    }
    if (bad) {
        atomicOr(err, SN_EBIT_BAD_ID);
        return ROW_BAD;
    }
    *tok_off = id * d;
    *pe_off = p * d;
    return ROW_OK;
}

// ---- C[t, :] = (X[t, :] - tok[id] - pe[p]) U  (or G U when !GATHER) -----------
constexpr int CT = 32;          // tokens per block
constexpr int CDC = 64;         // d-chunk staged in shared memory
constexpr int CTHREADS = 256;
constexpr int CQ = CT * KMAX / CTHREADS;

template <typename E, bool GATHER>
__global__ void __launch_bounds__(CTHREADS)
k_simt_compress(const float *__restrict__ U32, int d, int k, const E *__restrict__ X,
                const int32_t *__restrict__ ids, const int32_t *__restrict__ pos, int64_t T,
                int seq_len, const E *__restrict__ tok, int64_t vocab,
                const E *__restrict__ pe, E *__restrict__ C, unsigned int *err)
{
    __shared__ float Rs[CT][CDC + 1];
    __shared__ float Us[CDC * KMAX];
    __shared__ int64_t rtok[CT], rpe[CT];
    __shared__ int rstate[CT];
    const int tid = threadIdx.x;
    const int64_t t0 = (int64_t)blockIdx.x * CT;
    if (tid < CT)
        rstate[tid] = token_rows(t0 + tid, T, GATHER, ids, pos, seq_len, vocab, pe != nullptr,
                                 d, &rtok[tid], &rpe[tid], err);
    float acc[CQ];
#pragma unroll
    for (int q = 0; q < CQ; ++q)
        acc[q] = 0.f;
    const int nout = CT * k;
    for (int i0 = 0; i0 < d; i0 += CDC) {
        const int dc = min(CDC, d - i0);
        __syncthreads();
        for (int e = tid; e < CT * CDC; e += CTHREADS) {
            const int tl = e / CDC, ii = e % CDC;
            float r = 0.f;
            if (ii < dc && rstate[tl] == ROW_OK) {
                r = to_f(X[(t0 + tl) * d + i0 + ii]);
                if (GATHER) {
                    r -= to_f(tok[rtok[tl] + i0 + ii]);
                    if (pe)
                        r -= to_f(pe[rpe[tl] + i0 + ii]);
                }
            }
            Rs[tl][ii] = r;
        }
        for (int e = tid; e < dc * k; e += CTHREADS)
            Us[e] = U32[(int64_t)i0 * k + e];
        __syncthreads();
#pragma unroll
        for (int q = 0; q < CQ; ++q) {
            const int o = tid + q * CTHREADS;
            if (o < nout) {
                const int tl = o / k, j = o % k;
                float s = acc[q];
                for (int ii = 0; ii < dc; ++ii)
                    s = fmaf(Rs[tl][ii], Us[ii * k + j], s);
                acc[q] = s;
            }
        }
    }
#pragma unroll
    for (int q = 0; q < CQ; ++q) {
        const int o = tid + q * CTHREADS;
        if (o < nout) {
            const int tl = o / k, j = o % k;
            if (rstate[tl] == ROW_OK)
                C[(t0 + tl) * k + j] = from_f<E>(acc[q]);
            else if (rstate[tl] == ROW_BAD)
                C[(t0 + tl) * k + j] = from_f<E>(0.f);
        }
    }
}

// ---- X[t, i] = sum_j C[t, j] U[i, j] (+ pe[p, i] + tok[id, i]) -----------------
constexpr int DT = 8;           // tokens per block
constexpr int DTHREADS = 256;   // columns per block

template <typename E, bool GATHER>
__global__ void __launch_bounds__(DTHREADS)
k_simt_decompress(const float *__restrict__ U32T, int d, int k, const E *__restrict__ C,
                  const int32_t *__restrict__ ids, const int32_t *__restrict__ pos, int64_t T,
                  int seq_len, const E *__restrict__ tok, int64_t vocab,
                  const E *__restrict__ pe, E *__restrict__ X, unsigned int *err)
{
    __shared__ float Cs[DT][KMAX];
    __shared__ int64_t rtok[DT], rpe[DT];
    __shared__ int rstate[DT];
    const int tid = threadIdx.x;
    const int i = blockIdx.x * DTHREADS + tid;
    for (int64_t t0 = (int64_t)blockIdx.y * DT; t0 < T; t0 += (int64_t)gridDim.y * DT) {
        __syncthreads();
        if (tid < DT)
            rstate[tid] = token_rows(t0 + tid, T, GATHER, ids, pos, seq_len, vocab,
                                     pe != nullptr, d, &rtok[tid], &rpe[tid], err);
        for (int e = tid; e < DT * k; e += DTHREADS) {
            const int tl = e / k, j = e % k;
            const int64_t t = t0 + tl;
            Cs[tl][j] = t < T ? to_f(C[t * k + j]) : 0.f;
        }
        __syncthreads();
        if (i >= d)
            continue;
        float acc[DT];
#pragma unroll
        for (int tl = 0; tl < DT; ++tl)
            acc[tl] = 0.f;
        for (int j = 0; j < k; ++j) {
            const float u = U32T[(int64_t)j * d + i];
#pragma unroll
            for (int tl = 0; tl < DT; ++tl)
                acc[tl] = fmaf(Cs[tl][j], u, acc[tl]);
        }
#pragma unroll
        for (int tl = 0; tl < DT; ++tl) {
            const int64_t t = t0 + tl;
            if (rstate[tl] == ROW_OK) {
                float v = acc[tl];
                if (GATHER) {
                    if (pe)
                        v += to_f(pe[rpe[tl] + i]);
                    v += to_f(tok[rtok[tl] + i]);
                }
                X[t * d + i] = from_f<E>(v);
            } else if (rstate[tl] == ROW_BAD) {
                X[t * d + i] = from_f<E>(0.f);
            }
        }
    }
}

// ---- W' = U (U^T W): A = U^T W (fp32 [k, cols]) then W' = U A ----------------
constexpr int PJ = 16;          // U columns per thread in the first pass

template <typename E>
__global__ void __launch_bounds__(256)
k_simt_project_a(const float *__restrict__ U32, int d, int k, const E *__restrict__ W,
                 int64_t cols, int64_t ld, float *__restrict__ A)
{
    const int64_t c = (int64_t)blockIdx.x * 256 + threadIdx.x;
    const int j0 = blockIdx.y * PJ;
    if (c >= cols)
        return;
    float acc[PJ];
#pragma unroll
    for (int jj = 0; jj < PJ; ++jj)
        acc[jj] = 0.f;
    for (int i = 0; i < d; ++i) {
        const float w = to_f(W[(int64_t)i * ld + c]);
        const float *u = U32 + (int64_t)i * k + j0;
#pragma unroll
        for (int jj = 0; jj < PJ; ++jj)
            if (j0 + jj < k)
                acc[jj] = fmaf(u[jj], w, acc[jj]);
    }
#pragma unroll
    for (int jj = 0; jj < PJ; ++jj)
        if (j0 + jj < k)
            A[(int64_t)(j0 + jj) * cols + c] = acc[jj];
}

template <typename E>
__global__ void __launch_bounds__(256)
k_simt_project_b(const float *__restrict__ U32, int d, int k, const float *__restrict__ A,
                 int64_t cols, int64_t ld, E *__restrict__ W_out)
{
    const int64_t c = (int64_t)blockIdx.x * 256 + threadIdx.x;
    const int i = blockIdx.y;
    if (c >= cols || i >= d)
        return;
    float s = 0.f;
    for (int j = 0; j < k; ++j)
        s = fmaf(U32[(int64_t)i * k + j], A[(int64_t)j * cols + c], s);
    W_out[(int64_t)i * ld + c] = from_f<E>(s);
}

// ---- padded copies of U ---------------------------------------------------------
__global__ void k_prepare_basis(const float *__restrict__ U, int d, int k, int n_pad, int k64,
                                float *__restrict__ u32t, __nv_bfloat16 *__restrict__ ut16,
                                __nv_bfloat16 *__restrict__ up16)
{
    const int64_t n_t = (int64_t)k * d, n_ut = (int64_t)n_pad * d, n_up = (int64_t)d * k64;
    const int64_t n = max(n_t, max(n_ut, n_up));
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < n;
         e += (int64_t)gridDim.x * blockDim.x) {
        if (e < n_t) {            // u32t[j, i] = U[i, j]
            const int64_t j = e / d, i = e % d;
            u32t[e] = U[i * k + j];
        }
        if (e < n_ut) {           // ut16[j, i] = U[i, j], zero rows j >= k
            const int64_t j = e / d, i = e % d;
            ut16[e] = __float2bfloat16_rn(j < k ? U[i * k + j] : 0.f);
        }
        if (e < n_up) {           // up16[i, j] = U[i, j], zero columns j >= k
            const int64_t i = e / k64, j = e % k64;
            up16[e] = __float2bfloat16_rn(j < k ? U[i * k + j] : 0.f);
        }
    }
}

}  // namespace

template <typename E>
cudaError_t simt_compress(const sn_basis &b, const E *X, const int32_t *ids, const int32_t *pos,
                          int64_t T, int seq_len, const E *tok, int64_t vocab, const E *pe,
                          E *C, bool gather, cudaStream_t s)
{
    const int64_t blocks = (T + CT - 1) / CT;
    if (gather)
        k_simt_compress<E, true><<<(unsigned)blocks, CTHREADS, 0, s>>>(
            b.u32, b.d, b.k, X, ids, pos, T, seq_len, tok, vocab, pe, C, b.err);
    else
        k_simt_compress<E, false><<<(unsigned)blocks, CTHREADS, 0, s>>>(
            b.u32, b.d, b.k, X, nullptr, nullptr, T, 1, nullptr, 1, nullptr, C, b.err);
    count_launch();
    return cudaGetLastError();
}

template <typename E>
cudaError_t simt_decompress(const sn_basis &b, const E *C, const int32_t *ids,
                            const int32_t *pos, int64_t T, int seq_len, const E *tok,
                            int64_t vocab, const E *pe, E *X, bool gather, cudaStream_t s)
{
    const int64_t tiles = (T + DT - 1) / DT;
    dim3 grid((b.d + DTHREADS - 1) / DTHREADS, (unsigned)std::min<int64_t>(tiles, 65535));
    if (gather)
        k_simt_decompress<E, true><<<grid, DTHREADS, 0, s>>>(
            b.u32t, b.d, b.k, C, ids, pos, T, seq_len, tok, vocab, pe, X, b.err);
    else
        k_simt_decompress<E, false><<<grid, DTHREADS, 0, s>>>(
            b.u32t, b.d, b.k, C, nullptr, nullptr, T, 1, nullptr, 1, nullptr, X, b.err);
    count_launch();
    return cudaGetLastError();
}

template <typename E>
cudaError_t simt_project(const sn_basis &b, const E *W, int64_t cols, int64_t ld, E *W_out,
                         float *A, cudaStream_t s)
{
    dim3 ga((unsigned)((cols + 255) / 256), (b.k + PJ - 1) / PJ);
    k_simt_project_a<E><<<ga, 256, 0, s>>>(b.u32, b.d, b.k, W, cols, ld, A);
    dim3 gb((unsigned)((cols + 255) / 256), b.d);
    k_simt_project_b<E><<<gb, 256, 0, s>>>(b.u32, b.d, b.k, A, cols, ld, W_out);
    count_launch(2);
    return cudaGetLastError();
}

cudaError_t prepare_basis(sn_basis &b, const float *U, cudaStream_t s)
{
    cudaError_t e = cudaMemcpyAsync(b.u32, U, sizeof(float) * (size_t)b.d * b.k,
                                    cudaMemcpyDeviceToDevice, s);
    if (e != cudaSuccess)
        return e;
    k_prepare_basis<<<304, 256, 0, s>>>(U, b.d, b.k, b.n_pad, b.k64, b.u32t, b.ut16, b.up16);
    count_launch();
    return cudaGetLastError();
}

template cudaError_t simt_compress<float>(const sn_basis &, const float *, const int32_t *,
                                          const int32_t *, int64_t, int, const float *, int64_t,
                                          const float *, float *, bool, cudaStream_t);
template cudaError_t simt_compress<__nv_bfloat16>(const sn_basis &, const __nv_bfloat16 *,
                                                  const int32_t *, const int32_t *, int64_t, int,
                                                  const __nv_bfloat16 *, int64_t,
                                                  const __nv_bfloat16 *, __nv_bfloat16 *, bool,
                                                  cudaStream_t);
template cudaError_t simt_decompress<float>(const sn_basis &, const float *, const int32_t *,
                                            const int32_t *, int64_t, int, const float *,
                                            int64_t, const float *, float *, bool, cudaStream_t);
template cudaError_t simt_decompress<__nv_bfloat16>(const sn_basis &, const __nv_bfloat16 *,
                                                    const int32_t *, const int32_t *, int64_t,
                                                    int, const __nv_bfloat16 *, int64_t,
                                                    const __nv_bfloat16 *, __nv_bfloat16 *, bool,
                                                    cudaStream_t);
template cudaError_t simt_project<float>(const sn_basis &, const float *, int64_t, int64_t,
                                         float *, float *, cudaStream_t);
template cudaError_t simt_project<__nv_bfloat16>(const sn_basis &, const __nv_bfloat16 *, int64_t,
                                                 int64_t, __nv_bfloat16 *, float *, cudaStream_t);

}  // namespace sn
