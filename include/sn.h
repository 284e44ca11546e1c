/*
 * sn.h — C ABI of the GB300 (sm_103a) stage-boundary codec of Subspace Networks
 * (arXiv 2506.01260).
 *
 * At a pipeline boundary the residual-stream activation X^{l+1} minus the
 * locally recomputable embeddings lies in S = Col(U) once the projection
 * weights' rows are confined to S (Sec. 4.2, Eq. recursive2; Sec. 4.3), so only
 * its k coefficients on the orthonormal basis U cross the wire (Sec. 4.3.1,
 * Eq. subtract), and the activation gradient is compressed the same way
 * (Sec. 4.4, Eq. grad_compress).  The residual-writing weights are kept inside
 * S by projecting them with P = U U^T (Sec. 4.3, Sec. 5, App. A).
 *
 * Conventions shared by every call
 *   - Tensor pointers are device pointers (memory of the current CUDA device,
 *     or managed memory) unless stated otherwise, owned by the caller,
 *     contiguous row-major, and 16-byte aligned (SN_ERR_ALIGNMENT otherwise).
 *     Host memory, pageable or pinned, is refused with SN_ERR_INVALID_ARG
 *     (checked with cudaPointerGetAttributes) rather than handed to a kernel.
 *   - Calls are stream-ordered and asynchronous: they validate their
 *     arguments, enqueue kernels on `stream` and return.  An argument error
 *     returns synchronously and enqueues nothing.
 *   - `dtype` applies to X, C, G, the embedding tables and W alike.  SN_BF16 runs
 *     on the tensor cores (fp32 accumulation, one round-to-nearest-even to
 *     bf16 at the end); SN_F32 runs in fp32 on the CUDA cores.  U is fp32 at
 *     the ABI in both cases.
 *   - Token t's position is pos[t] when `pos` is non-NULL, else t mod seq_len
 *     (the batch is the row-major flattening of [b, seq_len]).  The positional
 *     table has seq_len rows; when it is NULL nothing positional is subtracted
 *     or added and `pos` is ignored.
 *   - An id outside [0, vocab) (or a position outside [0, seq_len)) is never
 *     clamped: that token's output row is written as zeros and the basis'
 *     device error word records SN_ERR_BAD_ID, reported by sn_check_errors.
 *   - Only sn_basis_create allocates (and sn_basis_destroy frees); no other
 *     call allocates memory or falls back to the CPU.  A basis holds two
 *     scratch areas of (SM count) x 128 x (k rounded up to 16) floats that the
 *     bf16 contractions use for the partial sums of their last-round row
 *     tiles: one for the forward calls (sn_compress_fwd,
 *     sn_compress_fwd_projected, sn_project_tables), one for sn_compress_bwd.
 *     Forward calls on one basis must therefore not overlap each other in time
 *     (other streams, other host threads), nor backward calls each other; a
 *     forward and a backward call may.
 *   - Every wait inside a kernel is bounded; a wait that expires records
 *     SN_ERR_TIMEOUT in the error word and the kernel returns.
 */
#ifndef SN_H
#define SN_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    SN_OK = 0,
    SN_ERR_INVALID_ARG = 1,   /* bad size, NULL pointer, k > d, overlap, ... */
    SN_ERR_ALIGNMENT = 2,     /* a pointer or leading dimension breaks the 16-byte rule */
    SN_ERR_UNSUPPORTED = 3,   /* valid request the library does not implement */
    SN_ERR_BAD_ID = 4,        /* asynchronous: an id or position was out of range */
    SN_ERR_TIMEOUT = 5,       /* asynchronous: a bounded in-kernel wait expired */
    SN_ERR_CUDA = 6,          /* a CUDA runtime call failed */
    SN_ERR_NUMERIC = 7        /* asynchronous: a factorisation met a non-positive pivot */
} sn_status;

typedef enum { SN_BF16 = 0, SN_F32 = 1 } sn_dtype;

/* Opaque basis handle: padded bf16/fp32 copies of U and the device error word. */
typedef struct sn_basis *sn_basis_t;

/* Same type as cudaStream_t (NULL = the legacy default stream). */
typedef struct CUstream_st *sn_stream_t;

/* Create a basis handle from U, a device fp32 [d, k] row-major matrix with
 * orthonormal columns (Sec. 4.3: U_k, Col(U_k) = S; shared by every node and
 * never sent per step).  U is copied; the caller keeps ownership of its
 * buffer.  Requires 16 <= d, d % 8 == 0, 1 <= k <= min(d, 128).  Allocates the
 * handle's device buffers, enqueues their initialisation on `stream` and
 * synchronises `stream` before returning.  *out is set only on SN_OK. */
sn_status sn_basis_create(const float *U, int32_t d, int32_t k, sn_basis_t *out,
                          sn_stream_t stream);

/* Free a handle (synchronises the device).  NULL is a no-op. */
sn_status sn_basis_destroy(sn_basis_t basis);

/* d and k of a handle (either pointer may be NULL). */
sn_status sn_basis_shape(sn_basis_t basis, int32_t *d, int32_t *k);

/* Forward compress, Sec. 4.3.1 Eq. (subtract):
 *   C[t, :] = (X[t, :] - tok_emb[ids[t], :] - pos_emb[p(t), :]) U
 * X: [T, d]; ids: int32 [T]; pos: int32 [T] or NULL; tok_emb: [vocab, d]
 * (T_fixed, the fixed high-rank table); pos_emb: [seq_len, d] or NULL;
 * C: [T, k], contiguous, no padding (the wire tensor, k/d of X). */
sn_status sn_compress_fwd(sn_basis_t basis, sn_dtype dtype, const void *X, const int32_t *ids,
                          const int32_t *pos, int64_t T, int32_t seq_len, const void *tok_emb,
                          int64_t vocab, const void *pos_emb, void *C, sn_stream_t stream);

/* Forward reconstruct, Sec. 4.3.1 (recovery at the next node):
 *   X[t, :] = C[t, :] U^T + pos_emb[p(t), :] + tok_emb[ids[t], :]
 * Arguments as in sn_compress_fwd with C an input [T, k] and X the output [T, d]. */
sn_status sn_decompress_fwd(sn_basis_t basis, sn_dtype dtype, const void *C, const int32_t *ids,
                            const int32_t *pos, int64_t T, int32_t seq_len, const void *tok_emb,
                            int64_t vocab, const void *pos_emb, void *X, sn_stream_t stream);

/* Gradient compress, Sec. 4.4 Eq. (grad_compress): C[t, :] = G[t, :] U.
 * G: [T, d] activation gradient; C: [T, k]. */
sn_status sn_compress_bwd(sn_basis_t basis, sn_dtype dtype, const void *G, int64_t T, void *C,
                          sn_stream_t stream);

/* Gradient recover, Sec. 4.4: G[t, :] = C[t, :] U^T.  C: [T, k]; G: [T, d]. */
sn_status sn_decompress_bwd(sn_basis_t basis, sn_dtype dtype, const void *C, int64_t T, void *G,
                            sn_stream_t stream);

/* Bytes of device workspace sn_project_weight needs for `cols` columns. */
sn_status sn_project_weight_workspace(sn_basis_t basis, sn_dtype dtype, int64_t cols,
                                      size_t *bytes);

/* Weight projection onto S, Sec. 4.3 (Row(W_p1), Row(W_p2) in S), Sec. 5
 * (W_p1 every iteration, W_p2 at initialisation), App. A.  In the paper's
 * layout W_p in R^{m x d} and W_p <- W_p U U^T; torch stores the transpose, so
 * for W [rows = d, cols] with leading dimension ld (elements):
 *   W_out = U (U^T W)     (A = U^T W is accumulated in fp32)
 * W_out may equal W (in place); any other overlap is SN_ERR_INVALID_ARG.
 * ld * element size must be a multiple of 16.  `workspace` is device memory of
 * at least sn_project_weight_workspace bytes, used only during the call. */
sn_status sn_project_weight(sn_basis_t basis, sn_dtype dtype, const void *W, int64_t rows,
                            int64_t cols, int64_t ld, void *W_out, void *workspace,
                            size_t workspace_bytes, sn_stream_t stream);

/* sn_project_weight for callers that cannot allocate device memory: no
 * workspace argument, no allocation.  The paper has no counterpart; this is a
 * convenience of the library.  Some callers cannot call cudaMalloc or hand out
 * scratch at the point where they project a weight (for example a training
 * runtime whose caching allocator already owns the device memory, or code that
 * must not enter the CUDA allocator between its own synchronisation points).
 * The scratch lives in a fixed file-scope device array of 32 MiB (33554432
 * bytes) that every GPU loading this library holds until the process exits.
 * Arguments, layout and results are those of sn_project_weight; bf16 only.
 * Returns SN_ERR_UNSUPPORTED for SN_F32 and when sn_project_weight_workspace
 * for `cols` exceeds 32 MiB.  The first call on a device (with that device
 * current) looks up the array's device address in the current CUDA context;
 * a call made under another context of the device (after cudaDeviceReset, or
 * under a caller's own context) looks it up again.  Make the first call in
 * each context before any stream capture.  All calls share the one array: calls whose executions
 * overlap on the GPU (other streams, other host threads) race and corrupt each
 * other's results, so order them on one stream.  Each call writes every
 * scratch element it reads before reading it; nothing is kept between calls. */
sn_status sn_project_weight_noalloc(sn_basis_t basis, sn_dtype dtype, const void *W,
                                    int64_t rows, int64_t cols, int64_t ld, void *W_out,
                                    sn_stream_t stream);

/* ---- Projected embedding tables (a variant of the forward compress) ----------
 * Because the compress of Sec. 4.3.1, Eq. (subtract), is linear,
 *   (X - T_fixed[ids] - P[p]) U = X U - (T_fixed U)[ids] - (P U)[p],
 * and T_fixed is fixed for the whole run (Sec. 4.3.1: sent to every node once),
 * the embedding rows can be projected once per U and the per-step compress then
 * reads k-wide rows instead of d-wide ones.  bf16 only (SN_ERR_UNSUPPORTED for
 * SN_F32). */

/* TU = T_fixed U (fp32 [vocab, k], row-major) and, when pos_emb is non-NULL,
 * PU = P U (fp32 [seq_len, k]).  tok_emb [vocab, d], pos_emb [seq_len, d];
 * pos_emb and PU are both NULL or both non-NULL.  Accumulated in fp32 from the
 * bf16 tables and the bf16 copy of U, never rounded. */
sn_status sn_project_tables(sn_basis_t basis, sn_dtype dtype, const void *tok_emb, int64_t vocab,
                            const void *pos_emb, int32_t seq_len, float *TU, float *PU,
                            sn_stream_t stream);

/* C[t, :] = X[t, :] U - TU[ids[t], :] - PU[p(t), :], one rounding to bf16 (the
 * same C as sn_compress_fwd with the tables TU, PU were projected from).
 * Arguments as in sn_compress_fwd with TU [vocab, k] and PU [seq_len, k] (or
 * NULL: nothing positional is subtracted and `pos` is ignored) in place of the
 * d-wide tables.  Invalid ids and positions behave as in sn_compress_fwd. */
sn_status sn_compress_fwd_projected(sn_basis_t basis, sn_dtype dtype, const void *X,
                                    const int32_t *ids, const int32_t *pos, int64_t T,
                                    int32_t seq_len, const float *TU, int64_t vocab,
                                    const float *PU, void *C, sn_stream_t stream);

/* The low-rank part of the token embeddings, Sec. 4.3.1: T_S = T_fixed U U^T
 * (bf16 [vocab, d]; computed as (T_fixed U) U^T with T_fixed U rounded once to
 * bf16 in between, like the weight projection).  `workspace` is device memory of
 * at least sn_wire_bytes(basis, dtype, vocab) bytes, used only during the call.
 * T_S may not overlap tok_emb or the workspace. */
sn_status sn_build_ts(sn_basis_t basis, sn_dtype dtype, const void *tok_emb, int64_t vocab,
                      void *T_S, void *workspace, size_t workspace_bytes, sn_stream_t stream);

/* ---- Subspace update on the Grassmann manifold (Sec. 4.5; gradient of Sec. 6)
 * The Grassmann loss (1/K) sum_t ||G_t (I - U U^T)||_F^2 over the activation
 * gradients G_t of the last compressed layer has the Euclidean gradient -2 S U
 * with S = (1/K) sum_t G_t^T G_t.  U changes only at a step, so S U is
 * accumulated directly as M = sum_t G_t^T (G_t U) = K S U: G_t U is the
 * compressed gradient Cg of Eq. (grad_compress) (sn_compress_bwd), and the
 * [d, d] matrix S is never formed.  Every K iterations the step takes the
 * tangent component of -2 M / K, moves U by -eta times it and retracts onto the
 * manifold with a QR factorisation (diag(R) > 0); a new basis handle is then
 * created from the result. */

/* Workspace bytes of sn_grassmann_accumulate for T tokens and of
 * sn_grassmann_step (either pointer may be NULL). */
sn_status sn_grassmann_workspace(sn_basis_t basis, int64_t T, size_t *accumulate_bytes,
                                 size_t *step_bytes);

/* M += G^T Cg.  G: bf16 [T, d]; Cg: bf16 [T, k] = G U from sn_compress_bwd with
 * this basis; M: fp32 [d, k] row-major, caller-owned (zero it at the start of a
 * window of K iterations).  Accumulated on the tensor cores in fp32.  bf16 only. */
sn_status sn_grassmann_accumulate(sn_basis_t basis, sn_dtype dtype, const void *G, const void *Cg,
                                  int64_t T, float *M, void *workspace, size_t workspace_bytes,
                                  sn_stream_t stream);

/* *acc += ||G (I - U U^T)||_F^2, evaluated as ||G||_F^2 - ||Cg||_F^2 in fp64 from
 * the bf16 tensors (so its error is ~2^-8 ||G||_F^2: a monitoring metric for
 * gradients that are not almost entirely inside the subspace).  acc: device
 * fp64 scalar.  bf16 only. */
sn_status sn_grassmann_residual(sn_basis_t basis, sn_dtype dtype, const void *G, const void *Cg,
                                int64_t T, double *acc, sn_stream_t stream);

/* U_new = Q of U - eta * tangent(-2 M / K), the QR factor with diag(R) > 0
 * (CholeskyQR2 in fp32, Gram matrices summed over row blocks in fp64; U_new^T
 * U_new = I to about 1e-7 for a step within reach of the identity).  M: fp32 [d, k] from
 * sn_grassmann_accumulate over K >= 1 iterations; U_new: fp32 [d, k], may not
 * overlap M.  A non-positive pivot records SN_ERR_NUMERIC for sn_check_errors. */
sn_status sn_grassmann_step(sn_basis_t basis, const float *M, int32_t K, float eta, float *U_new,
                            void *workspace, size_t workspace_bytes, sn_stream_t stream);

/* ---- Row-constant AdamW for W_p2 (Sec. 5) ---------------------------------------
 * Element-wise AdamW rescales each coordinate of an update by its own rate,
 * which turns rows of the update out of S.  The paper keeps one adaptive rate
 * per row of W_p2 (the mean of the bias-corrected second moment over the row),
 * so a weight whose rows lie in S stays there under in-S gradients without
 * further projection.  In the torch layout W is [rows = d, cols = d_ff] and the
 * paper's rows are its columns: one rate per column.  One step t >= 1:
 *   M = beta1 M + (1 - beta1) g,  V = beta2 V + (1 - beta2) g^2
 *   W = W - lr (M / (1 - beta1^t)) / (sqrt(mean_col(V) / (1 - beta2^t)) + eps) - lambda W
 * (the bias correction is AdamW's 1 - beta^t; the paper's printed V/(beta2 + eps)
 * is read as that; lambda is applied as printed, i.e. torch's lr * weight_decay).
 * W, M, V: fp32 [rows, cols], updated in place (zero M and V before step 1);
 * grad: [rows, cols] in `grad_dtype` (SN_BF16 or SN_F32); workspace: device
 * memory of at least cols * 4 bytes, used only during the call.  No basis is
 * involved.  Buffers may not overlap. */
sn_status sn_adamw_rowconst(sn_dtype grad_dtype, float *W, const void *grad, float *M, float *V,
                            int64_t rows, int64_t cols, int64_t step, float lr, float beta1,
                            float beta2, float eps, float lambda, void *workspace,
                            size_t workspace_bytes, sn_stream_t stream);

/* ---- Lossy comparators (Sec. 8, comparison against lossy compressions) --------
 * What a stage boundary could send instead of C at (about) the same number of
 * bytes, for measuring their reconstruction error on the same batches.  X is a
 * bf16 batch [T, d] with d % 8 == 0; everything is device memory.  bf16 only. */

/* Per row, the kk entries of largest magnitude (ties towards the lower column)
 * in ascending column order: values bf16 [T, kk], cols uint16 [T, kk].
 * 1 <= kk <= min(d, 4096), d <= 65536.  At 4 bytes per kept entry, kk = k / 2
 * matches the subspace codec's 2 k bytes per token. */
sn_status sn_topk_compress(const void *X, int64_t T, int32_t d, int32_t kk, void *values,
                           uint16_t *cols, sn_stream_t stream);

/* X_out [T, d] bf16: zero except values[t, j] at column cols[t, j]. */
sn_status sn_topk_restore(const void *values, const uint16_t *cols, int64_t T, int32_t d,
                          int32_t kk, void *X_out, sn_stream_t stream);

/* One bit per entry, 1 where X < 0 (bit c % 32 of word c / 32 of the row's
 * ceil(d / 32) words of `bits`), and scale[t] = mean |X[t, :]| (fp32): 16 times
 * smaller than bf16, the best rate of a quantizer. */
sn_status sn_sign_compress(const void *X, int64_t T, int32_t d, uint32_t *bits, float *scale,
                           sn_stream_t stream);

/* X_out[t, c] = -scale[t] where the bit is set, else scale[t] (bf16). */
sn_status sn_sign_restore(const uint32_t *bits, const float *scale, int64_t T, int32_t d,
                          void *X_out, sn_stream_t stream);

/* Row-scaled 8-bit quantization (int8 or fp8 e4m3): rate points of the
 * comparison's quantizer beside the 1-bit one.  X finite; a row whose largest
 * magnitude lies in (0, 2^-119) is outside the domain.  Per row t:
 * a = max |X[t, :]|, scale[t] = a / qmax (fp32), codes[t, c] = Q(X[t, c] * r)
 * with r = qmax / a (0 for a zero row), both fp32 operations.
 *   SN_Q_INT8  qmax = 127, Q = round half to even, clamp to [-127, 127],
 *              codes are int8 two's complement;
 *   SN_Q_E4M3  qmax = 448, Q = nearest fp8 e4m3 value (1-4-3, bias 7), ties to
 *              even, magnitudes past 448 saturate to 448, sign kept.
 * codes: uint8 [T, d] row-major (8-byte aligned), scale: fp32 [T]; T * d + 4 T
 * bytes on the wire, half of bf16.  Errors: SN_ERR_INVALID_ARG (format, sizes,
 * null or overlapping buffers), SN_ERR_ALIGNMENT. */
typedef enum { SN_Q_INT8 = 0, SN_Q_E4M3 = 1 } sn_qformat;
sn_status sn_quant_compress(const void *X, int64_t T, int32_t d, int32_t format, uint8_t *codes,
                            float *scale, sn_stream_t stream);

/* X_out[t, c] = decode(codes[t, c]) * scale[t], the product in fp32 rounded
 * once to bf16. */
sn_status sn_quant_restore(const uint8_t *codes, const float *scale, int64_t T, int32_t d,
                           int32_t format, void *X_out, sn_stream_t stream);

/* Bytes on the wire for T tokens: T * k * element size (Sec. 4.3: k/d of X). */
sn_status sn_wire_bytes(sn_basis_t basis, sn_dtype dtype, int64_t T, size_t *bytes);

/* The emulated pipeline link (Sec. 8.1 sends the compressed tensor between
 * stages; here the boundary is a pinned host buffer in one process).
 * sn_wire_send copies `bytes` from device memory to host memory (pinned for
 * asynchrony); sn_wire_recv copies host memory to device memory.  Both are
 * stream-ordered cudaMemcpyAsync calls. */
sn_status sn_wire_send(const void *src_device, void *dst_host, size_t bytes, sn_stream_t stream);
sn_status sn_wire_recv(const void *src_host, void *dst_device, size_t bytes, sn_stream_t stream);

/* Synchronise `stream`, then return and clear the basis' asynchronous error
 * (SN_ERR_BAD_ID or SN_ERR_TIMEOUT; SN_OK if none was recorded). */
sn_status sn_check_errors(sn_basis_t basis, sn_stream_t stream);

/* Failure-detection self-test of the bounded-wait rule: every in-kernel wait
 * (mbarrier phases, copies, MMA commits) gives up after a fixed limit of 2 s
 * instead of hanging.  Launches on `stream` one CTA of two warps that sets up
 * like the pipeline kernels (an mbarrier, an abort flag, 32 columns of tensor
 * memory) and waits for a barrier phase that nothing ever completes, with the
 * same bounded wait.  The first warp past the limit records SN_ERR_TIMEOUT in
 * the basis' error word and raises the abort flag, the other stops on the flag,
 * and the CTA frees its tensor memory and returns.  Asynchronous: the next
 * sn_check_errors on the basis returns SN_ERR_TIMEOUT; the basis and the CUDA
 * context stay usable.  Errors: SN_ERR_INVALID_ARG (null basis, basis of
 * another device), SN_ERR_CUDA (launch failure). */
sn_status sn_selftest_wait_timeout(sn_basis_t basis, sn_stream_t stream);

/* Number of kernels this library has launched in this process. */
uint64_t sn_launch_count(void);

/* Static, human-readable name of a status code. */
const char *sn_status_string(sn_status status);

#ifdef __cplusplus
}
#endif
#endif /* SN_H */
