// sn_internal.cuh — types shared by the library's translation units.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "sn.h"

// Bits of the per-basis device error word.
enum : unsigned int {
    SN_EBIT_BAD_ID = 1u,    // an id or position was out of range (row zeroed)
    SN_EBIT_TIMEOUT = 2u,   // a bounded wait expired; the kernel gave up
    SN_EBIT_NUMERIC = 4u,   // a factorisation met a non-positive pivot
};

// Padded copies of U kept by a basis handle.
//   u32  [d, k]      fp32, as given (CUDA-core paths, row i = U[i, :])
//   u32t [k, d]      fp32 transpose (CUDA-core reconstruction, coalesced in d)
//   ut16 [n_pad, d]  bf16 U^T, rows >= k zero: B operand of the d -> k contraction
//   up16 [d, k64]    bf16 U, columns >= k zero: operand of the k -> d expansion
struct sn_basis {
    int device;
    int d, k;
    int n_pad;   // k rounded up to 16 (MMA N of the compress contraction)
    int k64;     // k rounded up to 64 (whole 128-byte swizzle atoms)
    float *u32;
    float *u32t;
    __nv_bfloat16 *ut16;
    __nv_bfloat16 *up16;
    unsigned int *err;
    // fp32 partial rows of the compress contractions' split last-round tiles:
    // [0] forward (X and projected-table modes), [1] backward; tail_cap row
    // tiles of 128 x n_pad each (one per SM of the device)
    float *tail[2];
    int tail_cap;
};

namespace sn {

// Counts every kernel the library launches (reported by sn_launch_count).
void count_launch(int n = 1);

// ---- CUDA-core kernels (fp32 path) -------------------------------------------
template <typename E>
cudaError_t simt_compress(const sn_basis &b, const E *X, const int32_t *ids, const int32_t *pos,
                          int64_t T, int seq_len, const E *tok, int64_t vocab, const E *pe,
                          E *C, bool gather, cudaStream_t s);
template <typename E>
cudaError_t simt_decompress(const sn_basis &b, const E *C, const int32_t *ids,
                            const int32_t *pos, int64_t T, int seq_len, const E *tok,
                            int64_t vocab, const E *pe, E *X, bool gather, cudaStream_t s);
template <typename E>
cudaError_t simt_project(const sn_basis &b, const E *W, int64_t cols, int64_t ld, E *W_out,
                         float *A, cudaStream_t s);

cudaError_t prepare_basis(sn_basis &b, const float *U, cudaStream_t s);

// ---- tensor-core kernels (bf16 path, tcgen05 + TMA) -----------------------------
struct TcArgs {
    const __nv_bfloat16 *X;     // compress: X or G [T, d]; decompress: output X or G
    const int32_t *ids;
    const int32_t *pos;
    const __nv_bfloat16 *tok;
    const __nv_bfloat16 *pe;
    __nv_bfloat16 *C;           // compress: output [T, k]; decompress: input
    int64_t T;
    int64_t vocab;
    int seq_len;
    bool gather;                // subtract / add the embeddings
};
cudaError_t tc_compress(const sn_basis &b, const TcArgs &a, cudaStream_t s);
cudaError_t tc_decompress(const sn_basis &b, const TcArgs &a, __nv_bfloat16 *X_out,
                          cudaStream_t s);
cudaError_t tc_project(const sn_basis &b, const __nv_bfloat16 *W, int64_t cols, int64_t ld,
                       __nv_bfloat16 *W_out, void *workspace, cudaStream_t s);
size_t tc_project_workspace(const sn_basis &b, int64_t cols);
// out[r, :] = A[r, :] U in fp32 (projected tables: T_fixed U, P U)
cudaError_t tc_contract_f32(const sn_basis &b, const __nv_bfloat16 *A, int64_t rows, float *out,
                            cudaStream_t s);
// Grassmann accumulation M += G^T Cg (M fp32 [d, k]); workspace bytes for T tokens
size_t tc_grassmann_workspace(const sn_basis &b, int64_t T);
cudaError_t tc_grassmann_accumulate(const sn_basis &b, const __nv_bfloat16 *G,
                                    const __nv_bfloat16 *Cg, int64_t T, float *M, void *workspace,
                                    cudaStream_t s);
// ||G||^2 - ||Cg||^2 added to *acc (fp64); the Grassmann step (CUDA cores)
cudaError_t grassmann_residual(const sn_basis &b, const __nv_bfloat16 *G,
                               const __nv_bfloat16 *Cg, int64_t T, double *acc, cudaStream_t s);
size_t grassmann_step_workspace(const sn_basis &b);
cudaError_t grassmann_step(const sn_basis &b, const float *M, int K, float eta, float *U_new,
                           void *workspace, cudaStream_t s);
// Row-constant AdamW step (fp32 W, M, V; grad bf16 or fp32); colsum: [cols] fp32 scratch
cudaError_t adamw_rowconst(bool grad_bf16, float *W, const void *g, float *M, float *V,
                           int64_t rows, int64_t cols, int64_t t, float lr, float b1, float b2,
                           float eps, float lam, float *colsum, cudaStream_t s);
// Lossy comparators (bf16 batches [T, d])
cudaError_t lossy_topk(const void *X, int64_t T, int d, int kk, void *vals, uint16_t *cols,
                       cudaStream_t s);
cudaError_t lossy_topk_restore(const void *vals, const uint16_t *cols, int64_t T, int d, int kk,
                               void *out, cudaStream_t s);
cudaError_t lossy_sign(const void *X, int64_t T, int d, uint32_t *bits, float *scale,
                       cudaStream_t s);
cudaError_t lossy_sign_restore(const uint32_t *bits, const float *scale, int64_t T, int d,
                               void *out, cudaStream_t s);
cudaError_t lossy_quant(const void *X, int64_t T, int d, int format, uint8_t *codes, float *scale,
                        cudaStream_t s);
cudaError_t lossy_quant_restore(const uint8_t *codes, const float *scale, int64_t T, int d,
                                int format, void *out, cudaStream_t s);
// C = X U - TU[ids] - PU[pos] (PU may be null)
cudaError_t tc_compress_projected(const sn_basis &b, const __nv_bfloat16 *X, const int32_t *ids,
                                  const int32_t *pos, int64_t T, int seq_len, const float *TU,
                                  int64_t vocab, const float *PU, __nv_bfloat16 *C,
                                  cudaStream_t s);

}  // namespace sn
