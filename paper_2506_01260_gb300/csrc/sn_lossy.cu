// sn_lossy.cu — the lossy comparators of the paper's comparison at equal wire
// size (Sec. 8, "Comparison against lossy compressions"): per-row top-k and
// 1-bit sign quantization of a bf16 batch, with their restores.  One CTA per
// row (grid-stride over rows), 256 threads.
//
// Top-k keeps the kk entries of largest magnitude of each row, ties towards the
// lower column, and writes them in ascending column order.  The threshold
// magnitude is found exactly by a two-pass radix select on the 15-bit bf16
// magnitude (high 8 bits, then low 7); a third pass scans the row in column
// order (warp ballots) to place the kept entries and to take, among entries
// equal to the threshold, the lowest columns first.
#include "sn_internal.cuh"

namespace sn {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;

// Exclusive prefix of `flag` over the block in thread order and the block
// total; all threads must call it.  `ws` holds kWarps ints of shared memory.
__device__ __forceinline__ int block_scan(bool flag, int *ws, int &total)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const unsigned m = __ballot_sync(0xffffffffu, flag);
    __syncthreads();                          // ws free from the previous scan
    if (lane == 0)
        ws[warp] = __popc(m);
    __syncthreads();
    int before = 0;
    total = 0;
    for (int w = 0; w < kWarps; ++w) {
        before += w < warp ? ws[w] : 0;
        total += ws[w];
    }
    return before + __popc(m & ((1u << lane) - 1u));
}

__global__ void __launch_bounds__(kThreads) k_topk(const uint16_t *__restrict__ X, int64_t T,
                                                    int d, int kk, uint16_t *__restrict__ vals,
                                                    uint16_t *__restrict__ cols)
{
    extern __shared__ uint16_t row[];         // d bf16 patterns
    __shared__ int hist[256];
    __shared__ int ws[kWarps];
    __shared__ int sel[4];                    // bin, threshold, above, need
    for (int64_t t = blockIdx.x; t < T; t += gridDim.x) {
        const uint16_t *src = X + t * (int64_t)d;
        __syncthreads();
        for (int c = threadIdx.x; c < d / 8; c += kThreads)
            ((uint4 *)row)[c] = __ldg((const uint4 *)src + c);
        for (int c = threadIdx.x; c < 256; c += kThreads)
            hist[c] = 0;
        __syncthreads();
        // pass 1: high 8 bits of the magnitude
        for (int c = threadIdx.x; c < d; c += kThreads)
            atomicAdd(&hist[(row[c] & 0x7FFF) >> 7], 1);
        __syncthreads();
        if (threadIdx.x == 0) {
            int above = 0, b = 255;
            while (above + hist[b] < kk)
                above += hist[b--];
            sel[0] = b;
            sel[2] = above;
        }
        __syncthreads();
        const int B = sel[0];
        for (int c = threadIdx.x; c < 128; c += kThreads)
            hist[c] = 0;
        __syncthreads();
        // pass 2: low 7 bits of the entries in bin B
        for (int c = threadIdx.x; c < d; c += kThreads) {
            const int m = row[c] & 0x7FFF;
            if ((m >> 7) == B)
                atomicAdd(&hist[m & 127], 1);
        }
        __syncthreads();
        if (threadIdx.x == 0) {
            int above = sel[2], l = 127;
            while (above + hist[l] < kk)
                above += hist[l--];
            sel[1] = (B << 7) | l;
            sel[2] = above;
            sel[3] = kk - above;
        }
        __syncthreads();
        const int thr = sel[1], need = sel[3];
        // pass 3: place the kept entries in column order
        int kept = 0, eqs = 0;
        for (int c0 = 0; c0 < d; c0 += kThreads) {
            const int c = c0 + threadIdx.x;
            const int m = c < d ? (row[c] & 0x7FFF) : -1;
            int eq_total, keep_total;
            const int eq_rank = eqs + block_scan(m == thr, ws, eq_total);
            const bool keep = m > thr || (m == thr && eq_rank < need);
            const int slot = kept + block_scan(keep, ws, keep_total);
            if (keep) {
                vals[t * kk + slot] = row[c];
                cols[t * kk + slot] = (uint16_t)c;
            }
            kept += keep_total;
            eqs += eq_total;
        }
    }
}

__global__ void __launch_bounds__(kThreads) k_topk_restore(const uint16_t *__restrict__ vals,
                                                            const uint16_t *__restrict__ cols,
                                                            int64_t T, int d, int kk,
                                                            uint16_t *__restrict__ out)
{
    for (int64_t t = blockIdx.x; t < T; t += gridDim.x) {
        uint16_t *dst = out + t * (int64_t)d;
        __syncthreads();
        for (int c = threadIdx.x; c < d / 8; c += kThreads)
            ((uint4 *)dst)[c] = make_uint4(0, 0, 0, 0);
        __syncthreads();
        for (int j = threadIdx.x; j < kk; j += kThreads)
            dst[cols[t * kk + j]] = vals[t * kk + j];
    }
}

__global__ void __launch_bounds__(kThreads) k_sign(const uint16_t *__restrict__ X, int64_t T, int d,
                                                    uint32_t *__restrict__ bits,
                                                    float *__restrict__ scale)
{
    __shared__ float red[kWarps];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int words = (d + 31) / 32;
    for (int64_t t = blockIdx.x; t < T; t += gridDim.x) {
        const uint16_t *src = X + t * (int64_t)d;
        float s = 0.f;
        for (int w = warp; w < words; w += kWarps) {
            const int c = 32 * w + lane;
            const uint16_t b = c < d ? src[c] : (uint16_t)0;
            s += __uint_as_float((uint32_t)(b & 0x7FFF) << 16);
            const unsigned m = __ballot_sync(0xffffffffu, (b & 0x8000) && (b & 0x7FFF));
            if (lane == 0)
                bits[t * words + w] = m;
        }
        for (int o = 16; o > 0; o >>= 1)
            s += __shfl_xor_sync(0xffffffffu, s, o);
        __syncthreads();
        if (lane == 0)
            red[warp] = s;
        __syncthreads();
        if (threadIdx.x == 0) {
            float tot = 0.f;
            for (int w = 0; w < kWarps; ++w)
                tot += red[w];
            scale[t] = tot / (float)d;
        }
    }
}

__global__ void k_sign_restore(const uint32_t *__restrict__ bits, const float *__restrict__ scale,
                               int64_t T, int d, __nv_bfloat16 *__restrict__ out)
{
    const int words = (d + 31) / 32;
    const int64_t n = T * (int64_t)d;
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < n;
         e += (int64_t)gridDim.x * blockDim.x) {
        const int64_t t = e / d;
        const int c = (int)(e - t * d);
        const bool neg = (bits[t * words + c / 32] >> (c & 31)) & 1u;
        out[e] = __float2bfloat16_rn(neg ? -scale[t] : scale[t]);
    }
}

int row_grid(int64_t T)
{
    int dev = 0, sms = 148;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    return (int)(T < 8 * (int64_t)sms ? T : 8 * (int64_t)sms);
}

}  // namespace

cudaError_t lossy_topk(const void *X, int64_t T, int d, int kk, void *vals, uint16_t *cols,
                       cudaStream_t s)
{
    const size_t smem = sizeof(uint16_t) * (size_t)d;
    cudaError_t e = cudaFuncSetAttribute(k_topk, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess)
        return e;
    k_topk<<<row_grid(T), kThreads, smem, s>>>((const uint16_t *)X, T, d, kk, (uint16_t *)vals,
                                                cols);
    count_launch();
    return cudaGetLastError();
}

cudaError_t lossy_topk_restore(const void *vals, const uint16_t *cols, int64_t T, int d, int kk,
                               void *out, cudaStream_t s)
{
    k_topk_restore<<<row_grid(T), kThreads, 0, s>>>((const uint16_t *)vals, cols, T, d, kk,
                                                     (uint16_t *)out);
    count_launch();
    return cudaGetLastError();
}

cudaError_t lossy_sign(const void *X, int64_t T, int d, uint32_t *bits, float *scale,
                       cudaStream_t s)
{
    k_sign<<<row_grid(T), kThreads, 0, s>>>((const uint16_t *)X, T, d, bits, scale);
    count_launch();
    return cudaGetLastError();
}

cudaError_t lossy_sign_restore(const uint32_t *bits, const float *scale, int64_t T, int d,
                               void *out, cudaStream_t s)
{
    k_sign_restore<<<4 * row_grid(T), 256, 0, s>>>(bits, scale, T, d, (__nv_bfloat16 *)out);
    count_launch();
    return cudaGetLastError();
}

}  // namespace sn
