// sn_tc_host.cu — host side of the tensor-core (bf16) path: TMA tensor maps,
// shared-memory stage planning, work splitting, and the launch sequences of
// the boundary calls.
#include <algorithm>
#include <climits>
#include <cstring>
#include <mutex>

#include "sn_tc.cuh"
#include "sn_tc_kernels.cuh"

namespace sn {
namespace tc {
namespace {

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                  const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                  const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn()
{
    static EncodeTiledFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *f = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = (EncodeTiledFn)f;
    });
    return fn;
}

// A 2-D bf16 tensor of `outer` rows x `inner` elements, `row_bytes` apart.
bool map2d(CUtensorMap *m, const void *ptr, uint64_t inner, uint64_t outer, uint64_t row_bytes,
           uint32_t box_inner, uint32_t box_outer, bool sw128)
{
    EncodeTiledFn fn = encode_fn();
    if (!fn)
        return false;
    const cuuint64_t dims[2] = {inner, outer};
    const cuuint64_t strides[1] = {row_bytes};
    const cuuint32_t box[2] = {box_inner, box_outer};
    const cuuint32_t estr[2] = {1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(ptr), dims, strides, box,
              estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
              sw128 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int sm_count(int device)
{
    static int cache[64] = {0};
    if (device < 0 || device >= 64)
        return 148;
    if (cache[device] == 0) {
        int n = 0;
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, device) != cudaSuccess ||
            n <= 0)
            n = 148;
        cache[device] = n;
    }
    return cache[device];
}

int pow2_at_least(int v, int lo)
{
    int p = lo;
    while (p < v)
        p *= 2;
    return p;
}

int contract_stages(int mode, int n_pad, int k, int has_pe)
{
    int s = 8;
    while (s > 2 && contract_plan(mode, n_pad, k, has_pe, s).total > kSmemLimit)
        --s;
    return s;
}

int expand_stages(int katoms)
{
    int s = 8;
    while (s > 2 && expand_plan(katoms, s).total > kSmemLimit)
        --s;
    return s;
}

// Two B stages; as many embedding stages as fit (at most 12).
void recon_stages(int katoms, int has_pe, int *sb, int *se)
{
    *sb = 2;
    int s = 12;
    while (s > 2 && recon_plan(katoms, has_pe, *sb, s).total > kSmemLimit)
        --s;
    *se = s;
}

// Paired reconstruction: two B stages of 64 U rows, as many 48 KB embedding
// stages as fit (at most 12).
void pair_stages(int katoms, int *sb, int *se)
{
    *sb = 2;
    int s = 12;
    while (s > 2 && pair_plan(katoms, *sb, s).total > kSmemLimit)
        --s;
    *se = s;
}

// Tiles ordered position-block-major when every sequence of the batch shares
// the same positional rows in whole 128-row blocks.
void tile_order(int64_t T, int seq_len, bool has_pe, bool has_pos, int *reorder, int *batches)
{
    *reorder = 0;
    *batches = 1;
    if (has_pe && !has_pos && seq_len % BM == 0 && T % seq_len == 0 && T / seq_len > 1) {
        *reorder = 1;
        *batches = (int)(T / seq_len);
    }
}

// Split `nblk` column blocks of `ntiles` row tiles into work items of `bpi`
// blocks for a persistent grid of `sms` CTAs: the longest CTA's time, counted
// in blocks, is (rounds of the grid) x (bpi + 1), an item's start-up (its A
// operand, the pipeline refill) costing about one block (measured on the
// projection's third pass at W [8192, 8192]: 7 blocks per item 0.086 ms, 32
// blocks on 128 CTAs 0.080 ms).  Among equal costs, the fewest items.
void split_blocks(int ntiles, int nblk, int sms, int *bpi, int *chunks)
{
    int64_t best = -1;
    for (int b = nblk; b >= 1; --b) {
        const int ch = (nblk + b - 1) / b;
        if ((nblk + ch - 1) / ch != b)
            continue;                         // same chunk count as a larger b
        const int64_t rounds = ((int64_t)ntiles * ch + sms - 1) / sms;
        const int64_t cost = rounds * (b + 1);
        if (best < 0 || cost < best) {
            best = cost;
            *bpi = b;
            *chunks = ch;
        }
    }
}

// d-range splits of the projection's first pass: the chunk count per item that
// minimises the longest CTA's time, counted in chunks: (rounds of the
// persistent grid) x (chunks per item + 2 for the item's partial-sum write),
// plus 4 per split for the partials the second pass reads back (measured on
// W [8192, 8192]: 16 splits 0.097 ms, 4 splits 0.089 ms, 2 splits 0.086 ms),
// with at least 8 chunks per item and, among equal costs, the fewest splits.
void project_splits(int d, int64_t m, int sms, int *splits, int *kc_per)
{
    const int nkc = (d + BK - 1) / BK;
    const int64_t ntiles = (m + BM - 1) / BM;
    int64_t best = -1;
    for (int kp = nkc; kp >= 1; --kp) {
        if (kp < 8 && kp < nkc)
            break;
        const int sp = (nkc + kp - 1) / kp;
        if ((nkc + sp - 1) / sp != kp)
            continue;                         // same split count as a larger kp
        const int64_t rounds = (ntiles * sp + sms - 1) / sms;
        const int64_t cost = rounds * (kp + 2) + 4 * sp;
        if (best < 0 || cost < best) {
            best = cost;
            *kc_per = kp;
            *splits = sp;
        }
    }
}

size_t align256(size_t v) { return (v + 255) & ~(size_t)255; }

// Launch `kernel` so that it may start while the previous kernel of the
// stream finishes; the kernel waits for it in griddep_wait.
template <typename... KArgs, typename... Args>
cudaError_t launch_dependent(void (*kernel)(KArgs...), dim3 grid, dim3 block, cudaStream_t s,
                             Args... args)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, args...);
}

// A^T[c, j] = sum over splits of P[split, c, j], rounded once to bf16 and
// zero-padded to k64 columns.  One thread per four adjacent outputs (16-byte
// partial loads: n_pad is a multiple of 16; an 8-byte store); k64 is 64 or 128.
__global__ void k_sum_partials(const float *__restrict__ P, int splits, int64_t m, int n_pad,
                               int k, int k64_log2, __nv_bfloat16 *__restrict__ At)
{
    griddep_wait();                   // the first pass's partials are visible
    griddep_launch_dependents();
    const int64_t n = m << (k64_log2 - 2);
    const int64_t split_stride = m * n_pad;
    const int q_log2 = k64_log2 - 2;
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < n;
         e += (int64_t)gridDim.x * blockDim.x) {
        const int64_t c = e >> q_log2;
        const int j = 4 * (int)(e & ((1 << q_log2) - 1));
        float4 s = make_float4(0.f, 0.f, 0.f, 0.f);
        if (j < k) {
            const float *src = P + c * n_pad + j;
            for (int sp = 0; sp < splits; ++sp, src += split_stride) {
                const float4 v = __ldg((const float4 *)src);
                s.x += v.x;
                s.y += v.y;
                s.z += v.z;
                s.w += v.w;
            }
        }
        __nv_bfloat162 lo = __floats2bfloat162_rn(j < k ? s.x : 0.f, j + 1 < k ? s.y : 0.f);
        __nv_bfloat162 hi = __floats2bfloat162_rn(j + 2 < k ? s.z : 0.f, j + 3 < k ? s.w : 0.f);
        uint2 out;
        out.x = *(const uint32_t *)&lo;
        out.y = *(const uint32_t *)&hi;
        *(uint2 *)(At + (c << k64_log2) + j) = out;
    }
}

int current_device()
{
    int d = 0;
    cudaGetDevice(&d);
    return d;
}

}  // namespace
}  // namespace tc

// Last-round split of the compress contractions and of the fp32 table
// projection.  With one CTA per SM a grid
// whose last round holds rem < sms / 2 row tiles leaves most SMs idle for a
// whole tile; those tiles instead run as s = min(4, sms / rem) items over
// d-ranges of at least 8 chunks, writing fp32 partials to the basis' scratch,
// and k_sum_tail adds them up (large stream: 512 tiles = 3 x 152 + 56, the
// last round halves).  Without scratch every item is a whole tile.
void plan_tail(tc::ContractParams &p, int sms, float *scratch, int cap)
{
    p.tail_tiles = 0;
    p.tail_splits = 1;
    p.tail_kc = p.nkc;
    p.Ptail = nullptr;
    const int rem = p.ntiles % sms;
    if (!scratch || rem == 0 || p.splits != 1)
        return;
    const int s = std::min(std::min(4, sms / rem), p.nkc / 8);
    if (s < 2 || rem * s > cap)
        return;
    const int kc = (p.nkc + s - 1) / s;
    p.tail_tiles = rem;
    p.tail_splits = (p.nkc + kc - 1) / kc;
    p.tail_kc = kc;
    p.Ptail = scratch;
}

// C rows of the split tiles: the sum of their d-range partials (minus the
// projected embedding rows in XP mode), rounded once to bf16; a row with an
// invalid id or position is written as zeros and flagged (X and XP modes).
// The fp32 table projection (GF mode) keeps the sum in fp32.
// Grid (tail tiles, 128 / 8): one warp per row, the lanes across its k columns.
__global__ void __launch_bounds__(256) k_sum_tail(const __grid_constant__ tc::ContractParams p,
                                                  int mode)
{
    using namespace tc;
    griddep_wait();                   // the contraction's partials are visible
    const int tt = blockIdx.x;
    const int r = 8 * blockIdx.y + (threadIdx.x >> 5), lane = threadIdx.x & 31;
    const int64_t row = tile_row0(p.ntiles - p.tail_tiles + tt, p.reorder, p.batches, p.seq_len) + r;
    if (row >= p.rows)
        return;
    bool bad = false;
    int id = 0, ps = 0;
    if (mode != CMODE_G && mode != CMODE_GF) {
        id = p.ids[row];
        bad = id < 0 || id >= p.vocab;
        if (p.has_pe) {
            ps = p.has_pos ? p.pos[row] : (int)(row % p.seq_len);
            bad = bad || ps < 0 || ps >= p.seq_len;
        }
        if (bad && lane == 0)
            atomicOr(p.err, SN_EBIT_BAD_ID);
    }
    const float *src = p.Ptail + ((int64_t)tt * p.tail_splits * BM + r) * p.n_pad;
    const int64_t split_stride = (int64_t)BM * p.n_pad;
    for (int j = lane; j < p.k; j += 32) {
        float v = 0.f;
        for (int sp = 0; sp < p.tail_splits; ++sp)
            v += src[sp * split_stride + j];
        if (!bad && mode == CMODE_XP) {
            v -= p.TU[(int64_t)id * p.k + j];
            if (p.has_pe)
                v -= p.PU[(int64_t)ps * p.k + j];
        }
        if (mode == CMODE_GF)
            p.Cf[row * p.k + j] = v;            // projected table rows stay fp32
        else
            p.C[row * p.k + j] = __float2bfloat16_rn(bad ? 0.f : v);
    }
}

// The contraction over a persistent grid, then the sum of any split tiles.
cudaError_t launch_compress(int mode, const tc::ContractParams &p, int sms, cudaStream_t s)
{
    using namespace tc;
    cudaError_t e = launch_contract(mode, p, std::min(contract_items(p), sms), s);
    if (e != cudaSuccess || p.tail_tiles == 0)
        return e;
    e = launch_dependent(k_sum_tail, dim3(p.tail_tiles, BM / 8), dim3(256), s, p, mode);
    count_launch();
    return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t tc_compress(const sn_basis &b, const TcArgs &a, cudaStream_t s)
{
    using namespace tc;
    ContractParams p;
    std::memset(&p, 0, sizeof p);
    const bool has_pe = a.gather && a.pe != nullptr;
    bool ok = map2d(&p.mapA, a.X, b.d, a.T, (uint64_t)b.d * 2, BK, BM, true) &&
              map2d(&p.mapU, b.ut16, b.d, b.n_pad, (uint64_t)b.d * 2, BK, b.n_pad, true);
    if (ok && has_pe)
        ok = map2d(&p.mapPE, a.pe, b.d, a.seq_len, (uint64_t)b.d * 2, BK, BM, true);
    else
        p.mapPE = p.mapA;
    if (!ok)
        return cudaErrorInvalidValue;
    const int mode = a.gather ? CMODE_X : CMODE_G;
    p.tok = a.tok;
    p.pe = has_pe ? a.pe : nullptr;
    p.ids = a.ids;
    p.pos = a.pos;
    p.C = a.C;
    p.err = b.err;
    p.rows = a.T;
    p.vocab = a.vocab;
    p.seq_len = a.seq_len;
    p.has_pe = has_pe;
    p.has_pos = a.gather && a.pos != nullptr;
    p.d = b.d;
    p.k = b.k;
    p.n_pad = b.n_pad;
    p.acc_stride = pow2_at_least(b.n_pad, 32);
    p.nkc = (b.d + BK - 1) / BK;
    p.kc_per_item = p.nkc;
    p.splits = 1;
    p.ntiles = (int)((a.T + BM - 1) / BM);
    tile_order(a.T, a.seq_len, has_pe, p.has_pos, &p.reorder, &p.batches);
    p.stages = contract_stages(mode, b.n_pad, b.k, has_pe);
    const int sms = sm_count(current_device());
    plan_tail(p, sms, b.tail[mode == CMODE_X ? 0 : 1], b.tail_cap);
    return launch_compress(mode, p, sms, s);
}

namespace {

// Contraction parameters shared by the projected-table calls: A [rows, d]
// K-major through TMA, U^T chunks, no embedding tiles.
bool contract_plain(tc::ContractParams &p, const sn_basis &b, const __nv_bfloat16 *A,
                    int64_t rows)
{
    using namespace tc;
    std::memset(&p, 0, sizeof p);
    if (!map2d(&p.mapA, A, b.d, rows, (uint64_t)b.d * 2, BK, BM, true) ||
        !map2d(&p.mapU, b.ut16, b.d, b.n_pad, (uint64_t)b.d * 2, BK, b.n_pad, true))
        return false;
    p.mapPE = p.mapA;
    p.err = b.err;
    p.rows = rows;
    p.vocab = 1;
    p.seq_len = 1;
    p.d = b.d;
    p.k = b.k;
    p.n_pad = b.n_pad;
    p.acc_stride = pow2_at_least(b.n_pad, 32);
    p.nkc = (b.d + BK - 1) / BK;
    p.kc_per_item = p.nkc;
    p.splits = 1;
    p.ntiles = (int)((rows + BM - 1) / BM);
    return true;
}

}  // namespace

cudaError_t tc_contract_f32(const sn_basis &b, const __nv_bfloat16 *A, int64_t rows, float *out,
                            cudaStream_t s)
{
    using namespace tc;
    ContractParams p;
    if (!contract_plain(p, b, A, rows))
        return cudaErrorInvalidValue;
    p.Cf = out;
    p.stages = contract_stages(CMODE_GF, b.n_pad, b.k, 0);
    // short tables (a positional table of a few thousand rows) split their
    // last round over d like the compress calls, on the forward scratch
    const int sms = sm_count(current_device());
    plan_tail(p, sms, b.tail[0], b.tail_cap);
    return launch_compress(CMODE_GF, p, sms, s);
}

cudaError_t tc_compress_projected(const sn_basis &b, const __nv_bfloat16 *X, const int32_t *ids,
                                  const int32_t *pos, int64_t T, int seq_len, const float *TU,
                                  int64_t vocab, const float *PU, __nv_bfloat16 *C,
                                  cudaStream_t s)
{
    using namespace tc;
    ContractParams p;
    if (!contract_plain(p, b, X, T))
        return cudaErrorInvalidValue;
    p.C = C;
    p.ids = ids;
    p.pos = PU ? pos : nullptr;
    p.TU = TU;
    p.PU = PU;
    p.vocab = vocab;
    p.seq_len = seq_len;
    p.has_pe = PU != nullptr;
    p.has_pos = PU != nullptr && pos != nullptr;
    p.stages = contract_stages(CMODE_XP, b.n_pad, b.k, 0);
    const int sms = sm_count(current_device());
    plan_tail(p, sms, b.tail[0], b.tail_cap);
    return launch_compress(CMODE_XP, p, sms, s);
}

cudaError_t tc_decompress(const sn_basis &b, const TcArgs &a, __nv_bfloat16 *X_out,
                          cudaStream_t s)
{
    using namespace tc;
    ExpandParams p;
    std::memset(&p, 0, sizeof p);
    const bool has_pe = a.gather && a.pe != nullptr;
    const int nb = BN_WIDE;
    bool ok = map2d(&p.mapB, b.up16, b.k64, b.d, (uint64_t)b.k64 * 2, 64, nb, true) &&
              map2d(&p.mapOut, X_out, b.d / 8 * 8, a.T, (uint64_t)b.d * 2, 64, 32, true);
    p.mapA = p.mapB;
    if (ok && has_pe)
        ok = map2d(&p.mapPE, a.pe, b.d, a.seq_len, (uint64_t)b.d * 2, 64, BM, true);
    else
        p.mapPE = p.mapB;
    if (!ok)
        return cudaErrorInvalidValue;
    const int sms = sm_count(current_device());
    p.tok = a.tok;
    p.pe = has_pe ? a.pe : nullptr;
    p.C = a.C;
    p.ids = a.ids;
    p.pos = a.pos;
    p.err = b.err;
    p.rows = a.T;
    p.vocab = a.vocab;
    p.seq_len = a.seq_len;
    p.has_pe = has_pe;
    p.has_pos = a.gather && a.pos != nullptr;
    p.k = b.k;
    p.katoms = b.k64 / 64;
    p.kmma = b.n_pad / 16;
    p.out = X_out;
    p.out_ld = b.d;
    p.ncols = b.d;
    p.ncols8 = b.d / 8 * 8;
    p.nblk = (b.d + nb - 1) / nb;
    p.ntiles = (int)((a.T + BM - 1) / BM);
    split_blocks(p.ntiles, p.nblk, sms, &p.bpi, &p.chunks);
    tile_order(a.T, a.seq_len, has_pe, p.has_pos, &p.reorder, &p.batches);
    if (a.gather && has_pe && p.reorder && p.batches % 2 == 0 && b.d % nb == 0 && b.n_pad <= 128) {
        // sequences 2i and 2i + 1 add the same positional tiles: one work item
        // covers both tiles of a pair (p.ntiles counts pairs), U in 64-row boxes
        if (!map2d(&p.mapA, b.up16, b.k64, b.d, (uint64_t)b.k64 * 2, 64, 64, true))
            return cudaErrorInvalidValue;
        p.ntiles /= 2;
        split_blocks(p.ntiles, p.nblk, sms, &p.bpi, &p.chunks);
        pair_stages(p.katoms, &p.stages, &p.estages);
        return launch_reconstruct_pair(p, std::min(p.ntiles * p.chunks, sms), s);
    }
    const int grid = std::min(p.ntiles * p.chunks, sms);
    if (a.gather) {
        recon_stages(p.katoms, has_pe, &p.stages, &p.estages);
        return launch_reconstruct(p, grid, s);
    }
    p.stages = expand_stages(p.katoms);
    return launch_expand(AMODE_REPACK, p, grid, s);
}

size_t tc_project_workspace(const sn_basis &b, int64_t cols)
{
    using namespace tc;
    int splits, kc_per;
    project_splits(b.d, cols, sm_count(current_device()), &splits, &kc_per);
    return align256(sizeof(float) * (size_t)splits * cols * b.n_pad) +
           align256(sizeof(__nv_bfloat16) * (size_t)cols * b.k64);
}

namespace tc {
namespace {

// CgT[j, t] = Cg[t, j] for j < k, t < T; zero for k <= j < n_pad and T <= t < Tp.
__global__ void __launch_bounds__(256) k_transpose_pad(const __nv_bfloat16 *__restrict__ Cg, int64_t T,
                                                      int k, int n_pad, int64_t Tp,
                                                      __nv_bfloat16 *__restrict__ CgT)
{
    // 64 tokens per block through shared memory: their k-wide rows are one
    // contiguous run of Cg (coalesced reads), each output row j gets 64
    // consecutive tokens (128-byte writes); the row pitch of 130 elements keeps
    // the column reads on distinct banks.  k <= 128.
    __shared__ __nv_bfloat16 tile[64][130];
    const int64_t t0 = (int64_t)blockIdx.x * 64;
    const int nt = (int)(T - t0 < 64 ? (T - t0 > 0 ? T - t0 : 0) : 64);
    for (int f = threadIdx.x; f < 64 * k; f += blockDim.x) {
        const int tl = f / k, j = f - tl * k;
        tile[tl][j] = tl < nt ? Cg[t0 * k + f] : __float2bfloat16_rn(0.f);
    }
    __syncthreads();
    for (int f = threadIdx.x; f < n_pad * 64; f += blockDim.x) {
        const int j = f >> 6, t = f & 63;
        CgT[(int64_t)j * Tp + t0 + t] = j < k ? tile[t][j] : __float2bfloat16_rn(0.f);
    }
}

// M[i, j] += sum over splits of P[split, i, j], j < k (M row-major [d, k]).
__global__ void __launch_bounds__(256) k_accumulate_partials(const float *__restrict__ P, int splits,
                                                            int64_t d, int n_pad, int k,
                                                            float *__restrict__ M)
{
    griddep_wait();                   // the contraction's partials are visible
    // two rows of M per block, one thread per column (k <= 128)
    const int64_t i = 2 * (int64_t)blockIdx.x + (threadIdx.x >> 7);
    const int j = threadIdx.x & 127;
    if (i >= d || j >= k)
        return;
    float s = 0.f;
    for (int sp = 0; sp < splits; ++sp)
        s += __ldg(P + ((int64_t)sp * d + i) * n_pad + j);
    M[i * k + j] += s;
}

}  // namespace
}  // namespace tc

size_t tc_grassmann_workspace(const sn_basis &b, int64_t T)
{
    using namespace tc;
    int splits, kc_per;
    project_splits((int)std::min<int64_t>(T, INT32_MAX), b.d, sm_count(current_device()), &splits,
                   &kc_per);
    const int64_t Tp = (T + 63) / 64 * 64;
    return align256(sizeof(__nv_bfloat16) * (size_t)b.n_pad * Tp) +
           align256(sizeof(float) * (size_t)splits * b.d * b.n_pad);
}

cudaError_t tc_grassmann_accumulate(const sn_basis &b, const __nv_bfloat16 *G,
                                    const __nv_bfloat16 *Cg, int64_t T, float *M, void *workspace,
                                    cudaStream_t s)
{
    using namespace tc;
    const int sms = sm_count(current_device());
    int splits, kc_per;
    project_splits((int)T, b.d, sms, &splits, &kc_per);
    const int64_t Tp = (T + 63) / 64 * 64;
    __nv_bfloat16 *CgT = (__nv_bfloat16 *)workspace;
    float *P = (float *)((char *)workspace +
                         align256(sizeof(__nv_bfloat16) * (size_t)b.n_pad * Tp));
    // Cg^T, K-major over the tokens: the B operand of M = G^T Cg
    k_transpose_pad<<<(unsigned)(Tp / 64), 256, 0, s>>>(Cg, T, b.k, b.n_pad, Tp, CgT);
    count_launch();
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess)
        return e;
    // fp32 partials of G^T Cg over token ranges: the projection's first pass with G
    // in the role of W (read MN-major) and Cg^T in the role of U^T
    ContractParams p;
    std::memset(&p, 0, sizeof p);
    bool ok = map2d(&p.mapA, G, b.d, T, (uint64_t)b.d * 2, 64, BK, true) &&
              map2d(&p.mapU, CgT, Tp, b.n_pad, (uint64_t)Tp * 2, BK, b.n_pad, true);
    p.mapPE = p.mapA;
    if (!ok)
        return cudaErrorInvalidValue;
    p.P = P;
    p.err = b.err;
    p.rows = b.d;
    p.vocab = 1;
    p.seq_len = 1;
    p.d = (int)T;
    p.k = b.k;
    p.n_pad = b.n_pad;
    p.acc_stride = pow2_at_least(b.n_pad, 32);
    p.nkc = (int)((T + BK - 1) / BK);
    p.kc_per_item = kc_per;
    p.splits = splits;
    p.ntiles = (b.d + BM - 1) / BM;
    p.stages = contract_stages(CMODE_W, b.n_pad, b.k, 0);
    e = launch_contract(CMODE_W, p, std::min(p.ntiles * splits, sms), s, true);
    if (e != cudaSuccess)
        return e;
    e = launch_dependent(k_accumulate_partials, dim3((unsigned)((b.d + 1) / 2)), dim3(256), s,
                         (const float *)P, splits, (int64_t)b.d, b.n_pad, b.k, M);
    count_launch();
    return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t tc_project(const sn_basis &b, const __nv_bfloat16 *W, int64_t cols, int64_t ld,
                       __nv_bfloat16 *W_out, void *workspace, cudaStream_t s)
{
    using namespace tc;
    const int sms = sm_count(current_device());
    int splits, kc_per;
    project_splits(b.d, cols, sms, &splits, &kc_per);
    float *P = (float *)workspace;
    __nv_bfloat16 *At = (__nv_bfloat16 *)((char *)workspace +
                                          align256(sizeof(float) * (size_t)splits * cols * b.n_pad));
    // pass 1: fp32 partials of A^T = (U^T W)^T over d-ranges
    ContractParams p;
    std::memset(&p, 0, sizeof p);
    bool ok = map2d(&p.mapA, W, cols, b.d, (uint64_t)ld * 2, 64, BK, true) &&
              map2d(&p.mapU, b.ut16, b.d, b.n_pad, (uint64_t)b.d * 2, BK, b.n_pad, true);
    p.mapPE = p.mapA;
    if (!ok)
        return cudaErrorInvalidValue;
    p.P = P;
    p.err = b.err;
    p.rows = cols;
    p.vocab = 1;
    p.seq_len = 1;
    p.d = b.d;
    p.k = b.k;
    p.n_pad = b.n_pad;
    p.acc_stride = pow2_at_least(b.n_pad, 32);
    p.nkc = (b.d + BK - 1) / BK;
    p.kc_per_item = kc_per;
    p.splits = splits;
    p.ntiles = (int)((cols + BM - 1) / BM);
    p.stages = contract_stages(CMODE_W, b.n_pad, b.k, 0);
    cudaError_t e = launch_contract(CMODE_W, p, std::min(p.ntiles * splits, sms), s);
    if (e != cudaSuccess)
        return e;
    // pass 2: sum the partials, round A^T to bf16 [cols, k64] (zero-padded)
    {
        // launched to start while the first pass finishes (it waits for it)
        const int64_t n4 = cols * (b.k64 / 4);
        e = launch_dependent(k_sum_partials, dim3((unsigned)std::min<int64_t>((n4 + 255) / 256, 4 * sms)),
                             dim3(256), s, (const float *)P, splits, cols, b.n_pad, b.k,
                             b.k64 == 64 ? 6 : 7, At);
        if (e != cudaSuccess)
            return e;
    }
    count_launch();
    if ((e = cudaGetLastError()) != cudaSuccess)
        return e;
    // pass 3: W' = U A, written through the W' tensor map
    ExpandParams q;
    std::memset(&q, 0, sizeof q);
    ok = map2d(&q.mapA, b.up16, b.k64, b.d, (uint64_t)b.k64 * 2, 64, BM, true) &&
         map2d(&q.mapB, At, b.k64, cols, (uint64_t)b.k64 * 2, 64, BN_WIDE, true) &&
         map2d(&q.mapOut, W_out, std::max<int64_t>(8, cols / 8 * 8), b.d, (uint64_t)ld * 2, 64,
               32, true);
    q.mapPE = q.mapB;
    if (!ok)
        return cudaErrorInvalidValue;
    q.err = b.err;
    q.rows = b.d;
    q.vocab = 1;
    q.seq_len = 1;
    q.k = b.k;
    q.katoms = b.k64 / 64;
    q.kmma = b.n_pad / 16;
    q.out = W_out;
    q.out_ld = ld;
    q.ncols = (int)cols;
    q.ncols8 = (int)(cols / 8 * 8);
    q.nblk = (int)((cols + BN_WIDE - 1) / BN_WIDE);
    q.ntiles = (b.d + BM - 1) / BM;
    split_blocks(q.ntiles, q.nblk, sms, &q.bpi, &q.chunks);
    q.stages = expand_stages(q.katoms);
    return launch_expand(AMODE_TMA, q, std::min(q.ntiles * q.chunks, sms), s, true);
}

}  // namespace sn
