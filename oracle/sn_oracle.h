/*
 * sn_oracle.h — fp64 CPU oracle of the Subspace Networks stage-boundary codec.
 *
 * TEST INFRASTRUCTURE ONLY.  This is the plain, slow, obviously-correct
 * statement of what the boundary computes, used to check the CUDA library.
 * Only the tests, the package smoke check and the benchmark's CPU-baseline
 * leg may load it.  It shares no code, header, table or helper with the CUDA
 * path and must never be reached from the product path.
 *
 * Every operation evaluates the paper's definition in fp64 and rounds once,
 * round-to-nearest-even, to the output dtype:
 *   compress_fwd    c = (x - T_fixed[id] - P[pos]) U            Sec. 4.3.1, Eq. (subtract)
 *   decompress_fwd  x = c U^T + P[pos] + T_fixed[id]              Sec. 4.3.1 (reconstruction)
 *   compress_bwd    c_g = g U                                     Sec. 4.4, Eq. (grad_compress)
 *   decompress_bwd  g = c_g U^T                                   Sec. 4.4 (recovery)
 *   project_weight  W' = U (U^T W)  (torch layout [d, m])          Sec. 4.3 (Row(W_p) in S), Sec. 5, App. A
 *
 * Layouts: all matrices row-major and contiguous.  X, G: [T, d].  C: [T, k].
 * U: [d, k], orthonormal columns.  tok_emb: [vocab, d].  pos_emb: [seq_len, d].
 * W: [d, m] with leading dimension ld (elements).
 *
 * Position of token t: pos[t] when pos != NULL, else t mod seq_len (row-major
 * [b, n] flattening of the batch).  When pos_emb is NULL no positional term is
 * subtracted or added and positions are not checked.
 *
 * An id outside [0, vocab) or a position outside [0, seq_len) zeroes that
 * token's output row; the call returns SNO_ERR_BAD_ID after finishing every
 * other row.
 */
#ifndef SN_ORACLE_H
#define SN_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum { SNO_BF16 = 0, SNO_F32 = 1, SNO_F64 = 2 };
enum { SNO_OK = 0, SNO_ERR_INVALID_ARG = 1, SNO_ERR_BAD_ID = 4 };

/* Optional *_f64 outputs receive the unrounded fp64 result (NULL to skip). */

int sno_compress_fwd(int dtype, const void *X, const int32_t *ids, const int32_t *pos,
                     int64_t T, int32_t seq_len, const void *tok_emb, int64_t vocab,
                     const void *pos_emb, int u_dtype, const void *U, int32_t d, int32_t k,
                     void *C, double *C_f64);

int sno_decompress_fwd(int dtype, const void *C, const int32_t *ids, const int32_t *pos,
                       int64_t T, int32_t seq_len, const void *tok_emb, int64_t vocab,
                       const void *pos_emb, int u_dtype, const void *U, int32_t d, int32_t k,
                       void *X, double *X_f64);

int sno_compress_bwd(int dtype, const void *G, int64_t T, int u_dtype, const void *U,
                     int32_t d, int32_t k, void *C, double *C_f64);

int sno_decompress_bwd(int dtype, const void *C, int64_t T, int u_dtype, const void *U,
                       int32_t d, int32_t k, void *G, double *G_f64);

int sno_project_weight(int dtype, const void *W, int64_t rows, int64_t cols, int64_t ld,
                       int u_dtype, const void *U, int32_t d, int32_t k, void *W_out,
                       double *W_f64);

/* Wire bytes of one compressed tensor: T * k * sizeof(dtype).  Returns -1 on bad args. */
int64_t sno_wire_bytes(int dtype, int64_t T, int32_t k);

/* fp64 -> bf16 bit pattern, round-to-nearest-even (exposed so tests can pin it). */
void sno_round_bf16(const double *in, uint16_t *out, int64_t n);

#ifdef __cplusplus
}
#endif
#endif
