/*
 * sn_oracle.c — fp64 CPU oracle of the Subspace Networks stage-boundary codec.
 *
 * TEST INFRASTRUCTURE ONLY (see sn_oracle.h): loaded by tests, the smoke
 * check and the benchmark's CPU-baseline leg, never by the product path.
 *
 * Every function is the paper's definition written out with plain loops:
 * inputs are widened exactly to fp64 (bf16 and fp32 embed exactly), each
 * contraction is summed in ascending index order, and the result is rounded
 * once, round-to-nearest-even, to the output dtype.  No blocking, fusion or
 * reordering.  Single-threaded.
 *
 * Build: gcc -O2 -ffp-contract=off -fPIC -shared (no fused multiply-add, so
 * the same bits come out on x86-64 and aarch64).
 */
#include "sn_oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>

/* ---- scalar conversions ------------------------------------------------- */

static double bf16_bits_to_f64(uint16_t h)
{
    /* A bf16 value is the upper half of an fp32 bit pattern. */
    uint32_t bits = (uint32_t)h << 16;
    float f;
    memcpy(&f, &bits, sizeof f);
    return (double)f;
}

/* Round an fp64 value to bf16 (8 significant bits, fp32 exponent range),
 * round-to-nearest-even, directly from fp64 (no intermediate fp32 rounding). */
static uint16_t f64_to_bf16_rne(double v)
{
    if (isnan(v))
        return 0x7fc0;
    uint16_t sign = signbit(v) ? 0x8000 : 0;
    double a = fabs(v);
    if (a == 0.0)
        return sign;
    if (isinf(a))
        return sign | 0x7f80;
    int e;
    frexp(a, &e);            /* a = m * 2^e with m in [0.5, 1) */
    int lead = e - 1;        /* a in [2^lead, 2^(lead+1)) */
    if (lead < -126)
        lead = -126;         /* subnormal bf16: fixed spacing 2^-133 */
    double ulp = ldexp(1.0, lead - 7);
    double q = nearbyint(a / ulp);   /* exact power-of-two scaling; ties to even */
    double r = q * ulp;
    if (r >= 0x1p128)
        return sign | 0x7f80;        /* overflow to infinity */
    float f = (float)r;              /* exact: <= 8 significant bits */
    uint32_t bits;
    memcpy(&bits, &f, sizeof bits);
    return sign | (uint16_t)(bits >> 16);
}

void sno_round_bf16(const double *in, uint16_t *out, int64_t n)
{
    for (int64_t i = 0; i < n; ++i)
        out[i] = f64_to_bf16_rne(in[i]);
}

static double load(const void *p, int dtype, int64_t i)
{
    switch (dtype) {
    case SNO_BF16: return bf16_bits_to_f64(((const uint16_t *)p)[i]);
    case SNO_F32:  return (double)((const float *)p)[i];
    default:       return ((const double *)p)[i];
    }
}

static void store(void *p, int dtype, int64_t i, double v)
{
    switch (dtype) {
    case SNO_BF16: ((uint16_t *)p)[i] = f64_to_bf16_rne(v); break;
    case SNO_F32:  ((float *)p)[i] = (float)v; break;   /* C conversion: nearest-even */
    default:       ((double *)p)[i] = v; break;
    }
}

static int dtype_ok(int dt) { return dt == SNO_BF16 || dt == SNO_F32 || dt == SNO_F64; }
static int u_dtype_ok(int dt) { return dt == SNO_F32 || dt == SNO_F64; }

int64_t sno_wire_bytes(int dtype, int64_t T, int32_t k)
{
    static const int64_t size[3] = {2, 4, 8};
    if (!dtype_ok(dtype) || T < 0 || k <= 0)
        return -1;
    return T * (int64_t)k * size[dtype];
}

/* Token t's position: explicit pos[t], else t mod seq_len (row-major [b, n]). */
static int64_t position_of(const int32_t *pos, int64_t t, int32_t seq_len)
{
    return pos ? (int64_t)pos[t] : t % seq_len;
}

/* Returns 1 if token t's embedding indices are valid, writing them out. */
static int token_indices(const int32_t *ids, const int32_t *pos, int64_t t, int32_t seq_len,
                         int64_t vocab, int has_pe, int64_t *id_out, int64_t *p_out)
{
    int64_t id = ids[t];
    int64_t p = has_pe ? position_of(pos, t, seq_len) : 0;
    *id_out = id;
    *p_out = p;
    if (id < 0 || id >= vocab)
        return 0;
    if (has_pe && (p < 0 || p >= seq_len))
        return 0;
    return 1;
}

/* ---- Sec. 4.3.1, Eq. (subtract): C = (X - PE - T_fixed[ids]) U ---------- */

int sno_compress_fwd(int dtype, const void *X, const int32_t *ids, const int32_t *pos,
                     int64_t T, int32_t seq_len, const void *tok_emb, int64_t vocab,
                     const void *pos_emb, int u_dtype, const void *U, int32_t d, int32_t k,
                     void *C, double *C_f64)
{
    if (!dtype_ok(dtype) || !u_dtype_ok(u_dtype) || T < 0 || d <= 0 || k <= 0 || k > d ||
        seq_len <= 0 || vocab <= 0 || (T > 0 && (!X || !ids || !tok_emb || !U || !C)))
        return SNO_ERR_INVALID_ARG;
    double *r = malloc(sizeof(double) * (size_t)d);
    double *c = malloc(sizeof(double) * (size_t)k);
    if (!r || !c) { free(r); free(c); return SNO_ERR_INVALID_ARG; }
    int status = SNO_OK;
    for (int64_t t = 0; t < T; ++t) {
        int64_t id, p;
        if (!token_indices(ids, pos, t, seq_len, vocab, pos_emb != NULL, &id, &p)) {
            for (int32_t j = 0; j < k; ++j) {
                store(C, dtype, t * k + j, 0.0);
                if (C_f64) C_f64[t * k + j] = 0.0;
            }
            status = SNO_ERR_BAD_ID;
            continue;
        }
        /* residual with the locally recomputable embeddings removed */
        for (int32_t i = 0; i < d; ++i) {
            double x = load(X, dtype, t * d + i);
            double te = load(tok_emb, dtype, id * d + i);
            double pe = pos_emb ? load(pos_emb, dtype, p * d + i) : 0.0;
            r[i] = x - te - pe;
        }
        /* coefficients on the orthonormal basis: c_j = sum_i r_i U[i, j] */
        for (int32_t j = 0; j < k; ++j)
            c[j] = 0.0;
        for (int32_t i = 0; i < d; ++i)
            for (int32_t j = 0; j < k; ++j)
                c[j] += r[i] * load(U, u_dtype, (int64_t)i * k + j);
        for (int32_t j = 0; j < k; ++j) {
            store(C, dtype, t * k + j, c[j]);
            if (C_f64) C_f64[t * k + j] = c[j];
        }
    }
    free(r);
    free(c);
    return status;
}

/* ---- Sec. 4.3.1: X_recovered = C U^T + PE + T_fixed[ids] --------------- */

int sno_decompress_fwd(int dtype, const void *C, const int32_t *ids, const int32_t *pos,
                       int64_t T, int32_t seq_len, const void *tok_emb, int64_t vocab,
                       const void *pos_emb, int u_dtype, const void *U, int32_t d, int32_t k,
                       void *X, double *X_f64)
{
    if (!dtype_ok(dtype) || !u_dtype_ok(u_dtype) || T < 0 || d <= 0 || k <= 0 || k > d ||
        seq_len <= 0 || vocab <= 0 || (T > 0 && (!C || !ids || !tok_emb || !U || !X)))
        return SNO_ERR_INVALID_ARG;
    int status = SNO_OK;
    for (int64_t t = 0; t < T; ++t) {
        int64_t id, p;
        if (!token_indices(ids, pos, t, seq_len, vocab, pos_emb != NULL, &id, &p)) {
            for (int32_t i = 0; i < d; ++i) {
                store(X, dtype, t * d + i, 0.0);
                if (X_f64) X_f64[t * d + i] = 0.0;
            }
            status = SNO_ERR_BAD_ID;
            continue;
        }
        for (int32_t i = 0; i < d; ++i) {
            double s = 0.0;
            for (int32_t j = 0; j < k; ++j)
                s += load(C, dtype, t * k + j) * load(U, u_dtype, (int64_t)i * k + j);
            double te = load(tok_emb, dtype, id * d + i);
            double pe = pos_emb ? load(pos_emb, dtype, p * d + i) : 0.0;
            double x = s + pe + te;
            store(X, dtype, t * d + i, x);
            if (X_f64) X_f64[t * d + i] = x;
        }
    }
    return status;
}

/* ---- Sec. 4.4, Eq. (grad_compress): C_g = G U --------------------------- */

int sno_compress_bwd(int dtype, const void *G, int64_t T, int u_dtype, const void *U,
                     int32_t d, int32_t k, void *C, double *C_f64)
{
    if (!dtype_ok(dtype) || !u_dtype_ok(u_dtype) || T < 0 || d <= 0 || k <= 0 || k > d ||
        (T > 0 && (!G || !U || !C)))
        return SNO_ERR_INVALID_ARG;
    double *c = malloc(sizeof(double) * (size_t)k);
    if (!c) return SNO_ERR_INVALID_ARG;
    for (int64_t t = 0; t < T; ++t) {
        for (int32_t j = 0; j < k; ++j)
            c[j] = 0.0;
        for (int32_t i = 0; i < d; ++i) {
            double g = load(G, dtype, t * d + i);
            for (int32_t j = 0; j < k; ++j)
                c[j] += g * load(U, u_dtype, (int64_t)i * k + j);
        }
        for (int32_t j = 0; j < k; ++j) {
            store(C, dtype, t * k + j, c[j]);
            if (C_f64) C_f64[t * k + j] = c[j];
        }
    }
    free(c);
    return SNO_OK;
}

/* ---- Sec. 4.4: grad_recovered = C_g U^T --------------------------------- */

int sno_decompress_bwd(int dtype, const void *C, int64_t T, int u_dtype, const void *U,
                       int32_t d, int32_t k, void *G, double *G_f64)
{
    if (!dtype_ok(dtype) || !u_dtype_ok(u_dtype) || T < 0 || d <= 0 || k <= 0 || k > d ||
        (T > 0 && (!C || !U || !G)))
        return SNO_ERR_INVALID_ARG;
    for (int64_t t = 0; t < T; ++t) {
        for (int32_t i = 0; i < d; ++i) {
            double s = 0.0;
            for (int32_t j = 0; j < k; ++j)
                s += load(C, dtype, t * k + j) * load(U, u_dtype, (int64_t)i * k + j);
            store(G, dtype, t * d + i, s);
            if (G_f64) G_f64[t * d + i] = s;
        }
    }
    return SNO_OK;
}

/* ---- Sec. 4.3 / Sec. 5 / App. A: keep Row(W_p) inside S = Col(U) -------
 * Math layout W_p in R^{m x d} with W_p <- W_p U U^T; the torch weight is its
 * transpose W in R^{d x m}, so the update is W <- U (U^T W).  A = U^T W is a
 * [k, m] fp64 intermediate, then W'[i, c] = sum_j U[i, j] A[j, c].  W_out may
 * alias W: A is complete before any output is written. */

int sno_project_weight(int dtype, const void *W, int64_t rows, int64_t cols, int64_t ld,
                       int u_dtype, const void *U, int32_t d, int32_t k, void *W_out,
                       double *W_f64)
{
    if (!dtype_ok(dtype) || !u_dtype_ok(u_dtype) || d <= 0 || k <= 0 || k > d ||
        rows != d || cols < 0 || ld < cols || (cols > 0 && (!W || !U || !W_out)))
        return SNO_ERR_INVALID_ARG;
    if (cols == 0)
        return SNO_OK;
    double *A = malloc(sizeof(double) * (size_t)k * (size_t)cols);
    if (!A) return SNO_ERR_INVALID_ARG;
    for (int32_t j = 0; j < k; ++j)
        for (int64_t c = 0; c < cols; ++c) {
            double s = 0.0;
            for (int64_t i = 0; i < rows; ++i)
                s += load(U, u_dtype, i * k + j) * load(W, dtype, i * ld + c);
            A[(int64_t)j * cols + c] = s;
        }
    for (int64_t i = 0; i < rows; ++i)
        for (int64_t c = 0; c < cols; ++c) {
            double s = 0.0;
            for (int32_t j = 0; j < k; ++j)
                s += load(U, u_dtype, i * k + j) * A[(int64_t)j * cols + c];
            store(W_out, dtype, i * ld + c, s);
            if (W_f64) W_f64[i * cols + c] = s;
        }
    free(A);
    return SNO_OK;
}
