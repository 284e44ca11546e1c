// sn_api.cu — the C ABI (include/sn.h): argument validation, basis handles,
// the launch of each call's kernels (bf16: tcgen05 tensor-core kernels; fp32:
// CUDA-core kernels), the wire copies and the asynchronous error word.
#include <atomic>
#include <cstdlib>
#include <initializer_list>
#include <new>

#include "sn_internal.cuh"

namespace sn {
static std::atomic<uint64_t> g_launches{0};
void count_launch(int n) { g_launches.fetch_add((uint64_t)n, std::memory_order_relaxed); }
}  // namespace sn

namespace {

constexpr int kMaxK = 128;
constexpr int64_t kMaxRows = (int64_t)1 << 31;   // TMA coordinates are 32-bit

bool aligned(const void *p, uintptr_t a) { return ((uintptr_t)p % a) == 0; }

bool overlap(const void *a, size_t na, const void *b, size_t nb)
{
    const uintptr_t pa = (uintptr_t)a, pb = (uintptr_t)b;
    return pa < pb + nb && pb < pa + na;
}

size_t esize(sn_dtype dt) { return dt == SN_BF16 ? 2 : 4; }

sn_status cuda_status(cudaError_t e) { return e == cudaSuccess ? SN_OK : SN_ERR_CUDA; }

// Kernels dereference every tensor pointer, so each must be device memory of
// the current device or managed memory; host memory (pageable or pinned) is
// refused here instead of faulting in a kernel.  Null pointers are left to the
// callers' own checks.
bool on_device(std::initializer_list<const void *> ptrs)
{
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess)
        return false;
    for (const void *p : ptrs) {
        if (!p)
            continue;
        cudaPointerAttributes a;
        if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
            (void)cudaGetLastError();
            return false;
        }
        if (a.type == cudaMemoryTypeManaged)
            continue;
        if (a.type != cudaMemoryTypeDevice || a.device != dev)
            return false;
    }
    return true;
}

// Common checks of a basis handle and dtype; the handle must live on the
// current device.
sn_status check_basis(sn_basis_t b, sn_dtype dt)
{
    if (!b || (dt != SN_BF16 && dt != SN_F32))
        return SN_ERR_INVALID_ARG;
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess)
        return SN_ERR_CUDA;
    return dev == b->device ? SN_OK : SN_ERR_INVALID_ARG;
}

// Checks shared by the forward (embedding) calls.
sn_status check_fwd(sn_basis_t b, sn_dtype dt, const void *in, const int32_t *ids,
                    const int32_t *pos, int64_t T, int32_t seq_len, const void *tok,
                    int64_t vocab, const void *pe, const void *out, size_t in_row,
                    size_t out_row)
{
    sn_status st = check_basis(b, dt);
    if (st != SN_OK)
        return st;
    if (T < 0 || T >= kMaxRows || seq_len <= 0 || vocab <= 0 || vocab >= kMaxRows)
        return SN_ERR_INVALID_ARG;
    if (T == 0)
        return SN_OK;
    if (!in || !ids || !tok || !out)
        return SN_ERR_INVALID_ARG;
    if (!aligned(in, 16) || !aligned(tok, 16) || !aligned(out, 16) || (pe && !aligned(pe, 16)) ||
        !aligned(ids, 4) || (pos && !aligned(pos, 4)))
        return SN_ERR_ALIGNMENT;
    const size_t es = esize(dt);
    if (overlap(in, (size_t)T * in_row * es, out, (size_t)T * out_row * es))
        return SN_ERR_INVALID_ARG;
    return on_device({in, ids, pos, tok, pe, out}) ? SN_OK : SN_ERR_INVALID_ARG;
}

}  // namespace

extern "C" {

const char *sn_status_string(sn_status s)
{
    switch (s) {
    case SN_OK: return "SN_OK";
    case SN_ERR_INVALID_ARG: return "SN_ERR_INVALID_ARG";
    case SN_ERR_ALIGNMENT: return "SN_ERR_ALIGNMENT";
    case SN_ERR_UNSUPPORTED: return "SN_ERR_UNSUPPORTED";
    case SN_ERR_BAD_ID: return "SN_ERR_BAD_ID";
    case SN_ERR_TIMEOUT: return "SN_ERR_TIMEOUT";
    case SN_ERR_CUDA: return "SN_ERR_CUDA";
    case SN_ERR_NUMERIC: return "SN_ERR_NUMERIC";
    }
    return "SN_ERR_UNKNOWN";
}

uint64_t sn_launch_count(void) { return sn::g_launches.load(std::memory_order_relaxed); }

sn_status sn_basis_create(const float *U, int32_t d, int32_t k, sn_basis_t *out,
                          sn_stream_t stream)
{
    if (!U || !out || d < 16 || d % 8 != 0 || k < 1 || k > d || k > kMaxK)
        return SN_ERR_INVALID_ARG;
    if (!aligned(U, 16))
        return SN_ERR_ALIGNMENT;
    if (!on_device({U}))
        return SN_ERR_INVALID_ARG;
    sn_basis *b = new (std::nothrow) sn_basis();
    if (!b)
        return SN_ERR_CUDA;
    if (cudaGetDevice(&b->device) != cudaSuccess) {
        delete b;
        return SN_ERR_CUDA;
    }
    b->d = d;
    b->k = k;
    b->n_pad = (k + 15) / 16 * 16;
    b->k64 = (k + 63) / 64 * 64;
    cudaError_t e = cudaSuccess;
    if (e == cudaSuccess) e = cudaMalloc(&b->u32, sizeof(float) * (size_t)d * k);
    if (e == cudaSuccess) e = cudaMalloc(&b->u32t, sizeof(float) * (size_t)d * k);
    if (e == cudaSuccess) e = cudaMalloc(&b->ut16, sizeof(__nv_bfloat16) * (size_t)b->n_pad * d);
    if (e == cudaSuccess) e = cudaMalloc(&b->up16, sizeof(__nv_bfloat16) * (size_t)d * b->k64);
    if (e == cudaSuccess) e = cudaMalloc(&b->err, sizeof(unsigned int));
    if (e == cudaSuccess)
        e = cudaDeviceGetAttribute(&b->tail_cap, cudaDevAttrMultiProcessorCount, b->device);
    for (int i = 0; i < 2 && e == cudaSuccess; ++i)
        e = cudaMalloc(&b->tail[i], sizeof(float) * (size_t)b->tail_cap * 128 * b->n_pad);
    if (e == cudaSuccess) e = cudaMemsetAsync(b->err, 0, sizeof(unsigned int), stream);
    if (e == cudaSuccess) e = sn::prepare_basis(*b, U, stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(stream);
    if (e != cudaSuccess) {
        sn_basis_destroy(b);
        return SN_ERR_CUDA;
    }
    *out = b;
    return SN_OK;
}

sn_status sn_basis_destroy(sn_basis_t b)
{
    if (!b)
        return SN_OK;
    cudaError_t e = cudaSuccess, e2;
    if ((e2 = cudaFree(b->u32)) != cudaSuccess) e = e2;
    if ((e2 = cudaFree(b->u32t)) != cudaSuccess) e = e2;
    if ((e2 = cudaFree(b->ut16)) != cudaSuccess) e = e2;
    if ((e2 = cudaFree(b->up16)) != cudaSuccess) e = e2;
    if ((e2 = cudaFree(b->err)) != cudaSuccess) e = e2;
    for (int i = 0; i < 2; ++i)
        if ((e2 = cudaFree(b->tail[i])) != cudaSuccess) e = e2;
    delete b;
    return cuda_status(e);
}

sn_status sn_basis_shape(sn_basis_t b, int32_t *d, int32_t *k)
{
    if (!b)
        return SN_ERR_INVALID_ARG;
    if (d) *d = b->d;
    if (k) *k = b->k;
    return SN_OK;
}

sn_status sn_compress_fwd(sn_basis_t b, sn_dtype dt, const void *X, const int32_t *ids,
                          const int32_t *pos, int64_t T, int32_t seq_len, const void *tok,
                          int64_t vocab, const void *pe, void *C, sn_stream_t stream)
{
    sn_status st = check_fwd(b, dt, X, ids, pos, T, seq_len, tok, vocab, pe, C, b ? b->d : 0,
                             b ? b->k : 0);
    if (st != SN_OK || T == 0)
        return st;
    cudaStream_t s = (cudaStream_t)stream;
    if (dt == SN_F32)
        return cuda_status(sn::simt_compress<float>(*b, (const float *)X, ids, pos, T, seq_len,
                                                    (const float *)tok, vocab, (const float *)pe,
                                                    (float *)C, true, s));
    sn::TcArgs a{(const __nv_bfloat16 *)X, ids, pos, (const __nv_bfloat16 *)tok,
                 (const __nv_bfloat16 *)pe, (__nv_bfloat16 *)C, T, vocab, seq_len, true};
    return cuda_status(sn::tc_compress(*b, a, s));
}

sn_status sn_decompress_fwd(sn_basis_t b, sn_dtype dt, const void *C, const int32_t *ids,
                            const int32_t *pos, int64_t T, int32_t seq_len, const void *tok,
                            int64_t vocab, const void *pe, void *X, sn_stream_t stream)
{
    sn_status st = check_fwd(b, dt, C, ids, pos, T, seq_len, tok, vocab, pe, X, b ? b->k : 0,
                             b ? b->d : 0);
    if (st != SN_OK || T == 0)
        return st;
    cudaStream_t s = (cudaStream_t)stream;
    if (dt == SN_F32)
        return cuda_status(sn::simt_decompress<float>(*b, (const float *)C, ids, pos, T, seq_len,
                                                      (const float *)tok, vocab,
                                                      (const float *)pe, (float *)X, true, s));
    sn::TcArgs a{nullptr, ids, pos, (const __nv_bfloat16 *)tok, (const __nv_bfloat16 *)pe,
                 (__nv_bfloat16 *)C, T, vocab, seq_len, true};
    return cuda_status(sn::tc_decompress(*b, a, (__nv_bfloat16 *)X, s));
}

sn_status sn_compress_bwd(sn_basis_t b, sn_dtype dt, const void *G, int64_t T, void *C,
                          sn_stream_t stream)
{
    sn_status st = check_basis(b, dt);
    if (st != SN_OK)
        return st;
    if (T < 0 || T >= kMaxRows)
        return SN_ERR_INVALID_ARG;
    if (T == 0)
        return SN_OK;
    if (!G || !C)
        return SN_ERR_INVALID_ARG;
    if (!aligned(G, 16) || !aligned(C, 16))
        return SN_ERR_ALIGNMENT;
    const size_t es = esize(dt);
    if (overlap(G, (size_t)T * b->d * es, C, (size_t)T * b->k * es) || !on_device({G, C}))
        return SN_ERR_INVALID_ARG;
    cudaStream_t s = (cudaStream_t)stream;
    if (dt == SN_F32)
        return cuda_status(sn::simt_compress<float>(*b, (const float *)G, nullptr, nullptr, T, 1,
                                                    nullptr, 1, nullptr, (float *)C, false, s));
    sn::TcArgs a{(const __nv_bfloat16 *)G, nullptr, nullptr, nullptr, nullptr,
                 (__nv_bfloat16 *)C, T, 1, 1, false};
    return cuda_status(sn::tc_compress(*b, a, s));
}

sn_status sn_decompress_bwd(sn_basis_t b, sn_dtype dt, const void *C, int64_t T, void *G,
                            sn_stream_t stream)
{
    sn_status st = check_basis(b, dt);
    if (st != SN_OK)
        return st;
    if (T < 0 || T >= kMaxRows)
        return SN_ERR_INVALID_ARG;
    if (T == 0)
        return SN_OK;
    if (!G || !C)
        return SN_ERR_INVALID_ARG;
    if (!aligned(G, 16) || !aligned(C, 16))
        return SN_ERR_ALIGNMENT;
    const size_t es = esize(dt);
    if (overlap(G, (size_t)T * b->d * es, C, (size_t)T * b->k * es) || !on_device({G, C}))
        return SN_ERR_INVALID_ARG;
    cudaStream_t s = (cudaStream_t)stream;
    if (dt == SN_F32)
        return cuda_status(sn::simt_decompress<float>(*b, (const float *)C, nullptr, nullptr, T,
                                                      1, nullptr, 1, nullptr, (float *)G, false,
                                                      s));
    sn::TcArgs a{nullptr, nullptr, nullptr, nullptr, nullptr, (__nv_bfloat16 *)C, T, 1, 1,
                 false};
    return cuda_status(sn::tc_decompress(*b, a, (__nv_bfloat16 *)G, s));
}

sn_status sn_project_weight_workspace(sn_basis_t b, sn_dtype dt, int64_t cols, size_t *bytes)
{
    if (!b || !bytes || cols < 0 || (dt != SN_BF16 && dt != SN_F32))
        return SN_ERR_INVALID_ARG;
    if (dt == SN_F32) {
        *bytes = sizeof(float) * (size_t)b->k * (size_t)cols;
        return SN_OK;
    }
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess || dev != b->device)
        return SN_ERR_INVALID_ARG;
    *bytes = sn::tc_project_workspace(*b, cols);
    return SN_OK;
}

sn_status sn_project_weight(sn_basis_t b, sn_dtype dt, const void *W, int64_t rows,
                            int64_t cols, int64_t ld, void *W_out, void *ws, size_t ws_bytes,
                            sn_stream_t stream)
{
    sn_status st = check_basis(b, dt);
    if (st != SN_OK)
        return st;
    if (rows != b->d || cols < 0 || ld < cols || cols >= kMaxRows || ld >= kMaxRows)
        return SN_ERR_INVALID_ARG;
    if (cols == 0)
        return SN_OK;
    if (!W || !W_out || !ws)
        return SN_ERR_INVALID_ARG;
    const size_t es = esize(dt);
    if (!aligned(W, 16) || !aligned(W_out, 16) || !aligned(ws, 16) || (ld * es) % 16 != 0)
        return SN_ERR_ALIGNMENT;
    size_t need = 0;
    sn_project_weight_workspace(b, dt, cols, &need);
    if (ws_bytes < need)
        return SN_ERR_INVALID_ARG;
    const size_t wbytes = ((size_t)(rows - 1) * ld + cols) * es;
    if (W != W_out && overlap(W, wbytes, W_out, wbytes))
        return SN_ERR_INVALID_ARG;
    if (overlap(ws, need, W, wbytes) || overlap(ws, need, W_out, wbytes) ||
        !on_device({W, W_out, ws}))
        return SN_ERR_INVALID_ARG;
    cudaStream_t s = (cudaStream_t)stream;
    if (dt == SN_F32)
        return cuda_status(sn::simt_project<float>(*b, (const float *)W, cols, ld, (float *)W_out,
                                                   (float *)ws, s));
    return cuda_status(sn::tc_project(*b, (const __nv_bfloat16 *)W, cols, ld,
                                      (__nv_bfloat16 *)W_out, ws, s));
}

sn_status sn_project_tables(sn_basis_t b, sn_dtype dt, const void *tok, int64_t vocab,
                            const void *pe, int32_t seq_len, float *TU, float *PU,
                            sn_stream_t stream)
{
    sn_status st = check_basis(b, dt);
    if (st != SN_OK)
        return st;
    if (dt != SN_BF16)
        return SN_ERR_UNSUPPORTED;
    if (vocab <= 0 || vocab >= kMaxRows || !tok || !TU || (pe == nullptr) != (PU == nullptr) ||
        (pe && (seq_len <= 0 || seq_len >= kMaxRows)))
        return SN_ERR_INVALID_ARG;
    if (!aligned(tok, 16) || !aligned(TU, 16) || (pe && (!aligned(pe, 16) || !aligned(PU, 16))))
        return SN_ERR_ALIGNMENT;
    if (overlap(tok, (size_t)vocab * b->d * 2, TU, (size_t)vocab * b->k * 4) ||
        (pe && (overlap(pe, (size_t)seq_len * b->d * 2, PU, (size_t)seq_len * b->k * 4) ||
                overlap(TU, (size_t)vocab * b->k * 4, PU, (size_t)seq_len * b->k * 4))) ||
        !on_device({tok, pe, TU, PU}))
        return SN_ERR_INVALID_ARG;
    cudaStream_t s = (cudaStream_t)stream;
    cudaError_t e = sn::tc_contract_f32(*b, (const __nv_bfloat16 *)tok, vocab, TU, s);
    if (e == cudaSuccess && pe)
        e = sn::tc_contract_f32(*b, (const __nv_bfloat16 *)pe, seq_len, PU, s);
    return cuda_status(e);
}

sn_status sn_compress_fwd_projected(sn_basis_t b, sn_dtype dt, const void *X, const int32_t *ids,
                                    const int32_t *pos, int64_t T, int32_t seq_len,
                                    const float *TU, int64_t vocab, const float *PU, void *C,
                                    sn_stream_t stream)
{
    sn_status st = check_fwd(b, dt, X, ids, pos, T, seq_len, TU, vocab, PU, C, b ? b->d : 0,
                             b ? b->k : 0);
    if (st != SN_OK || T == 0)
        return st;
    if (dt != SN_BF16)
        return SN_ERR_UNSUPPORTED;
    return cuda_status(sn::tc_compress_projected(*b, (const __nv_bfloat16 *)X, ids, pos, T,
                                                 seq_len, TU, vocab, PU, (__nv_bfloat16 *)C,
                                                 (cudaStream_t)stream));
}

sn_status sn_build_ts(sn_basis_t b, sn_dtype dt, const void *tok, int64_t vocab, void *T_S,
                      void *ws, size_t ws_bytes, sn_stream_t stream)
{
    sn_status st = check_basis(b, dt);
    if (st != SN_OK)
        return st;
    if (dt != SN_BF16)
        return SN_ERR_UNSUPPORTED;
    if (vocab <= 0 || vocab >= kMaxRows || !tok || !T_S || !ws)
        return SN_ERR_INVALID_ARG;
    const size_t table = (size_t)vocab * b->d * 2, coeff = (size_t)vocab * b->k * 2;
    if (ws_bytes < coeff)
        return SN_ERR_INVALID_ARG;
    if (!aligned(tok, 16) || !aligned(T_S, 16) || !aligned(ws, 16))
        return SN_ERR_ALIGNMENT;
    if (overlap(tok, table, T_S, table) || overlap(tok, table, ws, coeff) ||
        overlap(T_S, table, ws, coeff) || !on_device({tok, T_S, ws}))
        return SN_ERR_INVALID_ARG;
    cudaStream_t s = (cudaStream_t)stream;
    sn::TcArgs a{(const __nv_bfloat16 *)tok, nullptr, nullptr, nullptr, nullptr,
                 (__nv_bfloat16 *)ws, vocab, 1, 1, false};
    cudaError_t e = sn::tc_compress(*b, a, s);
    if (e == cudaSuccess)
        e = sn::tc_decompress(*b, a, (__nv_bfloat16 *)T_S, s);
    return cuda_status(e);
}

sn_status sn_grassmann_workspace(sn_basis_t b, int64_t T, size_t *acc_bytes, size_t *step_bytes)
{
    sn_status st = check_basis(b, SN_BF16);
    if (st != SN_OK)
        return st;
    if (T < 0 || T >= kMaxRows)
        return SN_ERR_INVALID_ARG;
    if (acc_bytes)
        *acc_bytes = sn::tc_grassmann_workspace(*b, T > 0 ? T : 1);
    if (step_bytes)
        *step_bytes = sn::grassmann_step_workspace(*b);
    return SN_OK;
}

sn_status sn_grassmann_accumulate(sn_basis_t b, sn_dtype dt, const void *G, const void *Cg,
                                  int64_t T, float *M, void *ws, size_t ws_bytes,
                                  sn_stream_t stream)
{
    sn_status st = check_basis(b, dt);
    if (st != SN_OK)
        return st;
    if (dt != SN_BF16)
        return SN_ERR_UNSUPPORTED;
    if (T < 0 || T >= kMaxRows)
        return SN_ERR_INVALID_ARG;
    if (T == 0)
        return SN_OK;
    if (!G || !Cg || !M || !ws || ws_bytes < sn::tc_grassmann_workspace(*b, T))
        return SN_ERR_INVALID_ARG;
    if (!aligned(G, 16) || !aligned(Cg, 16) || !aligned(M, 16) || !aligned(ws, 256))
        return SN_ERR_ALIGNMENT;
    const size_t mb = (size_t)b->d * b->k * 4;
    if (overlap(M, mb, G, (size_t)T * b->d * 2) || overlap(M, mb, Cg, (size_t)T * b->k * 2) ||
        overlap(ws, ws_bytes, M, mb) || overlap(ws, ws_bytes, G, (size_t)T * b->d * 2) ||
        overlap(ws, ws_bytes, Cg, (size_t)T * b->k * 2) || !on_device({G, Cg, M, ws}))
        return SN_ERR_INVALID_ARG;
    return cuda_status(sn::tc_grassmann_accumulate(*b, (const __nv_bfloat16 *)G,
                                                   (const __nv_bfloat16 *)Cg, T, M, ws,
                                                   (cudaStream_t)stream));
}

sn_status sn_grassmann_residual(sn_basis_t b, sn_dtype dt, const void *G, const void *Cg,
                                int64_t T, double *acc, sn_stream_t stream)
{
    sn_status st = check_basis(b, dt);
    if (st != SN_OK)
        return st;
    if (dt != SN_BF16)
        return SN_ERR_UNSUPPORTED;
    if (T < 0 || T >= kMaxRows || !acc)
        return SN_ERR_INVALID_ARG;
    if (T == 0)
        return SN_OK;
    if (!G || !Cg)
        return SN_ERR_INVALID_ARG;
    if (!aligned(G, 16) || !aligned(Cg, 2) || !aligned(acc, 8))
        return SN_ERR_ALIGNMENT;
    if (!on_device({G, Cg, acc}))
        return SN_ERR_INVALID_ARG;
    return cuda_status(sn::grassmann_residual(*b, (const __nv_bfloat16 *)G,
                                              (const __nv_bfloat16 *)Cg, T, acc,
                                              (cudaStream_t)stream));
}

sn_status sn_grassmann_step(sn_basis_t b, const float *M, int32_t K, float eta, float *U_new,
                            void *ws, size_t ws_bytes, sn_stream_t stream)
{
    sn_status st = check_basis(b, SN_F32);
    if (st != SN_OK)
        return st;
    if (!M || !U_new || !ws || K < 1 || !(eta >= 0.f) ||
        ws_bytes < sn::grassmann_step_workspace(*b))
        return SN_ERR_INVALID_ARG;
    if (!aligned(M, 16) || !aligned(U_new, 16) || !aligned(ws, 256))
        return SN_ERR_ALIGNMENT;
    const size_t mb = (size_t)b->d * b->k * 4;
    if (overlap(M, mb, U_new, mb) || overlap(ws, ws_bytes, M, mb) ||
        overlap(ws, ws_bytes, U_new, mb) || !on_device({M, U_new, ws}))
        return SN_ERR_INVALID_ARG;
    return cuda_status(sn::grassmann_step(*b, M, K, eta, U_new, ws, (cudaStream_t)stream));
}

sn_status sn_adamw_rowconst(sn_dtype gdt, float *W, const void *g, float *M, float *V,
                            int64_t rows, int64_t cols, int64_t t, float lr, float b1, float b2,
                            float eps, float lam, void *ws, size_t ws_bytes, sn_stream_t stream)
{
    if (gdt != SN_BF16 && gdt != SN_F32)
        return SN_ERR_INVALID_ARG;
    if (rows <= 0 || cols <= 0 || rows >= kMaxRows || cols >= kMaxRows || t < 1 ||
        !(b1 >= 0.f && b1 < 1.f) || !(b2 >= 0.f && b2 < 1.f) || !(eps >= 0.f) || !(lr >= 0.f) ||
        !(lam >= 0.f) || !W || !g || !M || !V || !ws || ws_bytes < (size_t)cols * 4)
        return SN_ERR_INVALID_ARG;
    if (!aligned(W, 16) || !aligned(g, 16) || !aligned(M, 16) || !aligned(V, 16) ||
        !aligned(ws, 16))
        return SN_ERR_ALIGNMENT;
    const size_t n4 = (size_t)rows * cols * 4, ng = (size_t)rows * cols * esize(gdt);
    const void *bufs[5] = {W, g, M, V, ws};
    const size_t lens[5] = {n4, ng, n4, n4, (size_t)cols * 4};
    for (int i = 0; i < 5; ++i)
        for (int j = i + 1; j < 5; ++j)
            if (overlap(bufs[i], lens[i], bufs[j], lens[j]))
                return SN_ERR_INVALID_ARG;
    if (!on_device({W, g, M, V, ws}))
        return SN_ERR_INVALID_ARG;
    return cuda_status(sn::adamw_rowconst(gdt == SN_BF16, W, g, M, V, rows, cols, t, lr, b1, b2,
                                          eps, lam, (float *)ws, (cudaStream_t)stream));
}

namespace {
sn_status check_batch(const void *X, int64_t T, int32_t d)
{
    if (T < 0 || T >= kMaxRows || d <= 0 || d % 8 != 0 || !X)
        return SN_ERR_INVALID_ARG;
    return aligned(X, 16) ? SN_OK : SN_ERR_ALIGNMENT;
}
}  // namespace

sn_status sn_topk_compress(const void *X, int64_t T, int32_t d, int32_t kk, void *vals,
                           uint16_t *cols, sn_stream_t stream)
{
    sn_status st = check_batch(X, T, d);
    if (st != SN_OK)
        return st;
    if (d > 65536 || kk < 1 || kk > d || kk > 4096 || !vals || !cols)
        return SN_ERR_INVALID_ARG;
    if (!aligned(vals, 2) || !aligned(cols, 2))
        return SN_ERR_ALIGNMENT;
    if (T == 0)
        return SN_OK;
    const size_t nx = (size_t)T * d * 2, nk = (size_t)T * kk * 2;
    if (overlap(X, nx, vals, nk) || overlap(X, nx, cols, nk) || overlap(vals, nk, cols, nk) ||
        !on_device({X, vals, cols}))
        return SN_ERR_INVALID_ARG;
    return cuda_status(sn::lossy_topk(X, T, d, kk, vals, cols, (cudaStream_t)stream));
}

sn_status sn_topk_restore(const void *vals, const uint16_t *cols, int64_t T, int32_t d,
                          int32_t kk, void *X_out, sn_stream_t stream)
{
    sn_status st = check_batch(X_out, T, d);
    if (st != SN_OK)
        return st;
    if (d > 65536 || kk < 1 || kk > d || !vals || !cols)
        return SN_ERR_INVALID_ARG;
    if (!aligned(vals, 2) || !aligned(cols, 2))
        return SN_ERR_ALIGNMENT;
    if (T == 0)
        return SN_OK;
    const size_t nx = (size_t)T * d * 2, nk = (size_t)T * kk * 2;
    if (overlap(X_out, nx, vals, nk) || overlap(X_out, nx, cols, nk) ||
        !on_device({vals, cols, X_out}))
        return SN_ERR_INVALID_ARG;
    return cuda_status(sn::lossy_topk_restore(vals, cols, T, d, kk, X_out, (cudaStream_t)stream));
}

sn_status sn_sign_compress(const void *X, int64_t T, int32_t d, uint32_t *bits, float *scale,
                           sn_stream_t stream)
{
    sn_status st = check_batch(X, T, d);
    if (st != SN_OK)
        return st;
    if (!bits || !scale)
        return SN_ERR_INVALID_ARG;
    if (!aligned(bits, 4) || !aligned(scale, 4))
        return SN_ERR_ALIGNMENT;
    if (T == 0)
        return SN_OK;
    const size_t nx = (size_t)T * d * 2, nb = (size_t)T * ((d + 31) / 32) * 4, ns = (size_t)T * 4;
    if (overlap(X, nx, bits, nb) || overlap(X, nx, scale, ns) || overlap(bits, nb, scale, ns) ||
        !on_device({X, bits, scale}))
        return SN_ERR_INVALID_ARG;
    return cuda_status(sn::lossy_sign(X, T, d, bits, scale, (cudaStream_t)stream));
}

sn_status sn_sign_restore(const uint32_t *bits, const float *scale, int64_t T, int32_t d,
                          void *X_out, sn_stream_t stream)
{
    sn_status st = check_batch(X_out, T, d);
    if (st != SN_OK)
        return st;
    if (!bits || !scale)
        return SN_ERR_INVALID_ARG;
    if (!aligned(bits, 4) || !aligned(scale, 4))
        return SN_ERR_ALIGNMENT;
    if (T == 0)
        return SN_OK;
    const size_t nx = (size_t)T * d * 2;
    if (overlap(X_out, nx, bits, (size_t)T * ((d + 31) / 32) * 4) ||
        overlap(X_out, nx, scale, (size_t)T * 4) || !on_device({bits, scale, X_out}))
        return SN_ERR_INVALID_ARG;
    return cuda_status(sn::lossy_sign_restore(bits, scale, T, d, X_out, (cudaStream_t)stream));
}

sn_status sn_quant_compress(const void *X, int64_t T, int32_t d, int32_t format, uint8_t *codes,
                            float *scale, sn_stream_t stream)
{
    sn_status st = check_batch(X, T, d);
    if (st != SN_OK)
        return st;
    if ((format != SN_Q_INT8 && format != SN_Q_E4M3) || !codes || !scale)
        return SN_ERR_INVALID_ARG;
    if (!aligned(codes, 8) || !aligned(scale, 4))
        return SN_ERR_ALIGNMENT;
    if (T == 0)
        return SN_OK;
    const size_t nx = (size_t)T * d * 2, nc = (size_t)T * d, ns = (size_t)T * 4;
    if (overlap(X, nx, codes, nc) || overlap(X, nx, scale, ns) || overlap(codes, nc, scale, ns) ||
        !on_device({X, codes, scale}))
        return SN_ERR_INVALID_ARG;
    return cuda_status(sn::lossy_quant(X, T, d, format, codes, scale, (cudaStream_t)stream));
}

sn_status sn_quant_restore(const uint8_t *codes, const float *scale, int64_t T, int32_t d,
                           int32_t format, void *X_out, sn_stream_t stream)
{
    sn_status st = check_batch(X_out, T, d);
    if (st != SN_OK)
        return st;
    if ((format != SN_Q_INT8 && format != SN_Q_E4M3) || !codes || !scale)
        return SN_ERR_INVALID_ARG;
    if (!aligned(codes, 8) || !aligned(scale, 4))
        return SN_ERR_ALIGNMENT;
    if (T == 0)
        return SN_OK;
    const size_t nx = (size_t)T * d * 2;
    if (overlap(X_out, nx, codes, (size_t)T * d) || overlap(X_out, nx, scale, (size_t)T * 4) ||
        !on_device({codes, scale, X_out}))
        return SN_ERR_INVALID_ARG;
    return cuda_status(sn::lossy_quant_restore(codes, scale, T, d, format, X_out,
                                               (cudaStream_t)stream));
}

sn_status sn_wire_bytes(sn_basis_t b, sn_dtype dt, int64_t T, size_t *bytes)
{
    if (!b || !bytes || T < 0 || (dt != SN_BF16 && dt != SN_F32))
        return SN_ERR_INVALID_ARG;
    *bytes = (size_t)T * (size_t)b->k * esize(dt);
    return SN_OK;
}

sn_status sn_wire_send(const void *src_device, void *dst_host, size_t bytes, sn_stream_t stream)
{
    if (bytes == 0)
        return SN_OK;
    if (!src_device || !dst_host || !on_device({src_device}))
        return SN_ERR_INVALID_ARG;
    return cuda_status(cudaMemcpyAsync(dst_host, src_device, bytes, cudaMemcpyDeviceToHost,
                                       (cudaStream_t)stream));
}

sn_status sn_wire_recv(const void *src_host, void *dst_device, size_t bytes, sn_stream_t stream)
{
    if (bytes == 0)
        return SN_OK;
    if (!src_host || !dst_device || !on_device({dst_device}))
        return SN_ERR_INVALID_ARG;
    return cuda_status(cudaMemcpyAsync(dst_device, src_host, bytes, cudaMemcpyHostToDevice,
                                       (cudaStream_t)stream));
}

sn_status sn_check_errors(sn_basis_t b, sn_stream_t stream)
{
    if (!b)
        return SN_ERR_INVALID_ARG;
    unsigned int word = 0;
    cudaError_t e = cudaStreamSynchronize((cudaStream_t)stream);
    if (e == cudaSuccess)
        e = cudaMemcpy(&word, b->err, sizeof word, cudaMemcpyDeviceToHost);
    if (e == cudaSuccess && word)
        e = cudaMemset(b->err, 0, sizeof word);
    if (e != cudaSuccess)
        return SN_ERR_CUDA;
    if (word & SN_EBIT_TIMEOUT)
        return SN_ERR_TIMEOUT;
    if (word & SN_EBIT_BAD_ID)
        return SN_ERR_BAD_ID;
    if (word & SN_EBIT_NUMERIC)
        return SN_ERR_NUMERIC;
    return SN_OK;
}

}  // extern "C"
