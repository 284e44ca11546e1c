// sn_tc_contract.cu — the d -> k contraction on the tcgen05 tensor cores.
//
//   CMODE_X  C[t, :] = (X[t, :] - T_fixed[id_t, :] - P[p_t, :]) U     Sec. 4.3.1, Eq. (subtract)
//   CMODE_G  C[t, :] = G[t, :] U                                       Sec. 4.4, Eq. (grad_compress)
//   CMODE_W  A^T[c, :] = W[:, c]^T U  (fp32 partials over a d-range)    first pass of W' = U (U^T W)
//   CMODE_GF C[r, :] = A[r, :] U, fp32 out                            projected tables T_fixed U, P U
//   CMODE_XP C[t, :] = X[t, :] U - TU[id_t, :] - PU[p_t, :]             Eq. (subtract), projected tables
//
// Persistent CTAs walk 128-row tiles in 64-column chunks of d through a ring
// of shared-memory stages (all operand tiles 128-byte swizzled, K-major):
//   warp 0     TMA producer: the X/G tile (or the W tile, which the MMA reads
//              MN-major, as two 64-column swizzled boxes), the U^T chunk and,
//              when a tile's positions are contiguous, the positional tile;
//   warp 1     allocates TMEM and issues tcgen05.mma (M = 128, N = k padded
//              to 16, K = 16) into a double-buffered fp32 accumulator.  CMODE_X
//              accumulates X U - T_fixed[ids] U - P[pos] U: three MMAs per
//              K-step, the embedding terms with the descriptor's negate-A bit,
//              so the residual is never rounded;
//   warps 2-5  drain the accumulator (tcgen05.ld), round once to bf16 and
//              store each warp's 32 rows of C as one contiguous slab (CMODE_W:
//              fp32 partial rows);
//   warps 6-9  CMODE_X: gather the T_fixed rows (and non-contiguous positional
//              rows) with 16-byte cp.async copies straight into their swizzled
//              positions; each thread hands its copies to the stage's barrier
//              (cp.async.mbarrier.arrive), so the gather warps never wait for
//              their own copies, and the MMA thread fences toward the async
//              proxy after the barrier completes.  The next item's ids are
//              loaded and turned into row indices during the current item,
//              and the gather warps' waits for free stages are relaxed, so an
//              item's first copies wait for no load.
// Each CTA walks an item's chunks starting at its own offset, so the CTAs' U^T
// reads are spread over the L2 instead of converging on one slice.
// Every wait is bounded; a wait that expires raises SN_EBIT_TIMEOUT and the
// CTA drains its in-flight copies and MMAs, frees TMEM and returns.
#include "sn_tc.cuh"
#include "sn_tc_kernels.cuh"

namespace sn {
namespace tc {
namespace {

// chunk of an item at which the gather warps prepare the next item's rows
// (their ids were loaded at chunk 1)
constexpr int kRowsPrep = 6;

// j-th chunk of an item: every CTA starts at a different chunk so that the
// CTAs do not all read the same U^T chunk from one L2 slice at once.
__device__ __forceinline__ int chunk_at(int kc0, int kc1, int j)
{
    return kc0 + (int)((j + blockIdx.x) % (kc1 - kc0));
}

template <int MODE>
__global__ void __launch_bounds__(contract_threads(MODE), 1)
    k_contract(const __grid_constant__ ContractParams p)
{
    extern __shared__ uint8_t smem_raw[];
    uint32_t base = smem_u32(smem_raw);
    const uint32_t pad = (1024u - (base & 1023u)) & 1023u;
    base += pad;
    uint8_t *smem = smem_raw + pad;

    const int S = p.stages;
    const ContractPlan pl = contract_plan(MODE, p.n_pad, p.k, p.has_pe, S);
    const uint32_t bar = base + pl.bar_off;
    const uint32_t full_b = bar, empty_b = bar + 8 * S;
    const uint32_t accf_b = bar + 16 * S, acce_b = accf_b + 16, drain_b = acce_b + 16;
    uint32_t *tmem_slot = (uint32_t *)(smem + pl.bar_off + 8 * (2 * S + 5));
    volatile int *abort_flag = (volatile int *)(tmem_slot + 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t tmem_cols = 2 * p.acc_stride;

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(full_b + 8 * s, MODE == CMODE_X ? 1 + 128 : 1);   // TMA + gather threads
            mbar_init(empty_b + 8 * s, 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(accf_b + 8 * b, 1);
            mbar_init(acce_b + 8 * b, 4);
        }
        mbar_init(drain_b, 1);
        *abort_flag = 0;
        mbar_fence_init();
    }
    if (warp == 1)
        tmem_alloc(smem_u32(tmem_slot), tmem_cols);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    griddep_launch_dependents();   // a dependent launch may be scheduled now
    griddep_wait();                // launched as a dependent: the previous kernel's writes

    const int nitems = contract_items(p);

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            tma_prefetch(&p.mapA);
            tma_prefetch(&p.mapU);
            if (MODE == CMODE_X && p.has_pe)
                tma_prefetch(&p.mapPE);
        }
        uint32_t g = 0;
        bool ok = true;
        for (int item = blockIdx.x; item < nitems && ok; item += gridDim.x) {
            const ItemSpan sp = item_span(p, item);
            const int tile = sp.tile, kc0 = sp.kc0, kc1 = sp.kc1;
            const int64_t r0 = MODE == CMODE_W ? (int64_t)tile * BM
                                               : tile_row0(tile, p.reorder, p.batches, p.seq_len);
            const bool pe_tile = MODE == CMODE_X && p.has_pe && !p.has_pos &&
                                 (r0 % p.seq_len) + BM <= p.seq_len;
            const uint32_t tx = pl.a_bytes + pl.u_bytes + (pe_tile ? kTile : 0);
            for (int j = 0; j < kc1 - kc0; ++j, ++g) {
                const int kc = chunk_at(kc0, kc1, j);
                const int s = g % S;
                const uint32_t n = g / S;
                if (!warp_wait(empty_b + 8 * s, (n & 1) ^ 1, abort_flag, p.err)) {
                    ok = false;
                    break;
                }
                const uint32_t st = base + s * pl.stage_bytes;
                const uint32_t fb = full_b + 8 * s;
                if (lane == 0) {
                    mbar_arrive_tx(fb, tx);
                    if (MODE == CMODE_W) {   // W[kc*64 .. +64, r0 .. r0+128): d rows x c
                        tma_load_2d(st, &p.mapA, (int)r0, kc * BK, fb);
                        tma_load_2d(st + kTile / 2, &p.mapA, (int)r0 + 64, kc * BK, fb);
                    } else {
                        tma_load_2d(st, &p.mapA, kc * BK, (int)r0, fb);
                    }
                    tma_load_2d(st + pl.a_bytes, &p.mapU, kc * BK, 0, fb);
                    if (pe_tile)
                        tma_load_2d(st + pl.a_bytes + pl.u_bytes + pl.raw_bytes, &p.mapPE,
                                    kc * BK, (int)(r0 % p.seq_len), fb);
                }
                __syncwarp();
            }
        }
        if (!ok && lane == 0) {   // let copies already issued land before the CTA exits
            for (uint32_t i = g > (uint32_t)S ? g - S : 0; i < g; ++i)
                drain_wait(full_b + 8 * (i % S), (i / S) & 1);
        }
        __syncwarp();
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16(BM, p.n_pad, false, MODE == CMODE_W);
            const uint32_t idesc_neg = idesc_bf16(BM, p.n_pad, true);
            uint32_t g = 0, it = 0;
            bool ok = true;
            for (int item = blockIdx.x; item < nitems && ok; item += gridDim.x, ++it) {
                const ItemSpan sp = item_span(p, item);
                const int kc0 = sp.kc0, kc1 = sp.kc1;
                const uint32_t b = it & 1, nb = it >> 1;
                if (!mbar_wait(acce_b + 8 * b, (nb & 1) ^ 1, abort_flag, p.err)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t d_tmem = tmem + b * p.acc_stride;
                for (int j = 0; j < kc1 - kc0; ++j, ++g) {
                    const int s = g % S;
                    const uint32_t n = g / S;
                    if (!mbar_wait(full_b + 8 * s, n & 1, abort_flag, p.err)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    if (MODE == CMODE_X)   // gathered rows (generic proxy) -> MMA reads
                        fence_async_smem();
                    const uint32_t st = base + s * pl.stage_bytes;
                    const uint32_t ub = st + pl.a_bytes;
#pragma unroll
                    for (int kk = 0; kk < BK / 16; ++kk) {
                        const uint64_t bd = sdesc_sw128(ub + kk * 32);
                        // A: K-major rows (X, G), or the W tile MN-major (16 d rows
                        // per step; the second 64 columns 8 KB on)
                        const uint64_t ad = MODE == CMODE_W
                                                ? sdesc_mn_sw128(st + kk * 2048, kTile / 2, 1024)
                                                : sdesc_sw128(st + kk * 32);
                        mma_bf16(d_tmem, ad, bd, idesc,
                                 (j > 0 || kk > 0) ? 1u : 0u);
                        if (MODE == CMODE_X) {   // - T_fixed[ids] U - P[pos] U
                            const uint32_t tb = ub + pl.u_bytes;
                            mma_bf16(d_tmem, sdesc_sw128(tb + kk * 32), bd, idesc_neg, 1u);
                            if (p.has_pe)
                                mma_bf16(d_tmem, sdesc_sw128(tb + pl.raw_bytes + kk * 32), bd,
                                         idesc_neg, 1u);
                        }
                    }
                    mma_commit(empty_b + 8 * s);
                }
                if (ok)
                    mma_commit(accf_b + 8 * b);
            }
            if (!ok) {   // wait for MMAs already issued before TMEM is freed
                mma_commit(drain_b);
                drain_wait(drain_b, 0);
            }
        }
        __syncwarp();
    } else if (warp < 6) {
        // ------------------------------------------------------------ epilogue warps
        const int q = warp & 3;              // TMEM lane quarter of this warp
        const int row = 32 * q + lane;
        uint32_t it = 0;
        bool ok = true;
        for (int item = blockIdx.x; item < nitems && ok; item += gridDim.x, ++it) {
            const ItemSpan sp = item_span(p, item);
            const int tile = sp.tile, split = sp.split;
            const int64_t r0 = MODE == CMODE_W ? (int64_t)tile * BM
                                               : tile_row0(tile, p.reorder, p.batches, p.seq_len);
            if (MODE == CMODE_XP && !sp.tail && r0 + row < p.rows) {
                // this row's TU and PU rows are read after the item's main loop:
                // start them towards L2 now (the epilogue warps are idle until then)
                const int64_t t = r0 + row;
                const int id = p.ids[t];
                if (id >= 0 && id < p.vocab)
                    prefetch_l2_range(p.TU + (int64_t)id * p.k, p.k * 4);
                if (p.has_pe) {
                    const int ps = p.has_pos ? p.pos[t] : (int)(t % p.seq_len);
                    if (ps >= 0 && ps < p.seq_len)
                        prefetch_l2_range(p.PU + (int64_t)ps * p.k, p.k * 4);
                }
            }
            // ---- accumulator -> output
            const uint32_t b = it & 1, nb = it >> 1;
            if (!warp_wait(accf_b + 8 * b, nb & 1, abort_flag, p.err)) {
                ok = false;
                break;
            }
            tc_fence_after();
            const uint32_t taddr = tmem + b * p.acc_stride + ((uint32_t)(32 * q) << 16);
            if (MODE != CMODE_W && sp.tail) {
                // a d-range of a tail tile: fp32 partial row, summed by k_sum_tail
                float *dst = p.Ptail +
                             (((int64_t)(tile - (p.ntiles - p.tail_tiles)) * p.tail_splits + split) *
                                  BM + row) * p.n_pad;
                for (int cc = 0; cc < p.n_pad / 16; ++cc) {
                    float v[16];
                    tmem_ld16(taddr + 16 * cc, v);
                    tmem_ld_wait();
#pragma unroll
                    for (int j = 0; j < 16; j += 4)
                        *(float4 *)(dst + 16 * cc + j) = make_float4(v[j], v[j + 1], v[j + 2], v[j + 3]);
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0)
                    mbar_arrive(acce_b + 8 * b);
            } else if (MODE == CMODE_W) {
                const int64_t c = r0 + row;
                float *dst = p.P + ((int64_t)split * p.rows + c) * p.n_pad;
                for (int cc = 0; cc < p.n_pad / 16; ++cc) {
                    float v[16];
                    tmem_ld16(taddr + 16 * cc, v);
                    tmem_ld_wait();
                    if (c < p.rows) {
#pragma unroll
                        for (int j = 0; j < 16; j += 4)
                            *(float4 *)(dst + 16 * cc + j) =
                                make_float4(v[j], v[j + 1], v[j + 2], v[j + 3]);
                    }
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0)
                    mbar_arrive(acce_b + 8 * b);
            } else {
                const int64_t t = r0 + row;
                bool bad = false;
                int64_t tu_off = 0, pu_off = -1;   // XP: this row's TU and PU rows
                if ((MODE == CMODE_X || MODE == CMODE_XP) && t < p.rows) {
                    const int id = p.ids[t];
                    bad = id < 0 || id >= p.vocab;
                    int ps = 0;
                    if (p.has_pe) {
                        ps = p.has_pos ? p.pos[t] : (int)(t % p.seq_len);
                        bad = bad || ps < 0 || ps >= p.seq_len;
                    }
                    if (bad)
                        atomicOr(p.err, SN_EBIT_BAD_ID);
                    else if (MODE == CMODE_XP) {
                        tu_off = (int64_t)id * p.k;
                        if (p.has_pe)
                            pu_off = (int64_t)ps * p.k;
                    }
                }
                // stage the rows (bf16, or fp32 in GF mode) for contiguous slab stores
                constexpr int es = MODE == CMODE_GF ? 4 : 2;
                uint8_t *cst = smem + (size_t)S * pl.stage_bytes;
                for (int cc = 0; cc < p.n_pad / 16; ++cc) {
                    float v[16];
                    tmem_ld16(taddr + 16 * cc, v);
                    tmem_ld_wait();
#pragma unroll
                    for (int j = 0; j < 16; ++j) {
                        const int col = 16 * cc + j;
                        if (col < p.k) {
                            if (MODE == CMODE_GF) {
                                ((float *)cst)[(size_t)row * p.k + col] = v[j];
                            } else {
                                float x = v[j];
                                if (MODE == CMODE_XP && !bad) {
                                    x -= __ldg(p.TU + tu_off + col);
                                    if (pu_off >= 0)
                                        x -= __ldg(p.PU + pu_off + col);
                                }
                                ((__nv_bfloat16 *)cst)[(size_t)row * p.k + col] =
                                    __float2bfloat16_rn(bad ? 0.f : x);
                            }
                        }
                    }
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0)
                    mbar_arrive(acce_b + 8 * b);
                // this warp's 32 rows are one contiguous slab of 32 * k elements of the output
                const int64_t wr0 = r0 + 32 * q;
                const int64_t nrows = p.rows - wr0 < 32 ? p.rows - wr0 : 32;
                if (nrows > 0) {
                    const uint32_t src = smem_u32(cst + (size_t)32 * q * p.k * es);
                    uint8_t *dst = MODE == CMODE_GF ? (uint8_t *)(p.Cf + wr0 * p.k)
                                                    : (uint8_t *)(p.C + wr0 * p.k);
                    const int nbytes = (int)nrows * p.k * es;
                    for (int v = lane; v < nbytes / 16; v += 32)
                        *(uint4 *)(dst + 16 * v) = lds128(src + 16 * v);
                    for (int e = (nbytes / 16) * 16 + 2 * lane; e < nbytes; e += 64)
                        *(unsigned short *)(dst + e) =
                            *(const unsigned short *)(cst + (size_t)32 * q * p.k * es + e);
                }
                __syncwarp();
            }
        }
    } else if (MODE == CMODE_X) {
        // ------------------------------------------------------------ gather warps
        const int tt = threadIdx.x - 192;    // 0..127
        uint32_t g = 0;
        bool ok = true;
        // The next item's gather rows (this thread's 8 rows of T_fixed and P)
        // are prepared during the current item, where the gather warps wait for
        // free stages anyway: its ids and positions are loaded after the
        // item's first chunk and turned into row indices a few chunks later,
        // so an item starts with its first copies.
        int nrow_t[8], nrow_p[8];
        bool npe_tile = false;
        int64_t nq0 = p.rows;
        auto load_rows = [&](int tile_) {
            nq0 = tile_ >= 0 ? tile_row0(tile_, p.reorder, p.batches, p.seq_len) : p.rows;
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int64_t t = nq0 + (tt >> 3) + 16 * u;
                nrow_t[u] = 0;
                nrow_p[u] = 0;
                if (t < p.rows) {
                    nrow_t[u] = ld_issue(p.ids + t);
                    if (p.has_pe && p.has_pos)
                        nrow_p[u] = ld_issue(p.pos + t);
                }
            }
        };
        // ids / positions -> row indices (invalid ones read row 0; the epilogue
        // zeroes those rows); positional rows only where they are gathered
        auto prep_rows = [&]() {
            const int base = p.has_pe && !p.has_pos ? (int)(nq0 % p.seq_len) : 0;
            npe_tile = p.has_pe && !p.has_pos && base + BM <= p.seq_len;
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int off = (tt >> 3) + 16 * u;
                const bool in = nq0 + off < p.rows;
                int id = nrow_t[u];
                if (!in || id < 0 || id >= p.vocab)
                    id = 0;
                nrow_t[u] = id;
                int ps = 0;
                if (p.has_pe && !npe_tile && in) {
                    ps = p.has_pos ? nrow_p[u] : (base + off) % p.seq_len;
                    if (ps < 0 || ps >= p.seq_len)
                        ps = 0;
                }
                nrow_p[u] = ps;
            }
        };
        load_rows((int)blockIdx.x < nitems ? item_span(p, blockIdx.x).tile : -1);
        prep_rows();
        for (int item = blockIdx.x; item < nitems && ok; item += gridDim.x) {
            const ItemSpan sp = item_span(p, item);
            const int kc0 = sp.kc0, kc1 = sp.kc1;
            const bool pe_tile = npe_tile;
            int trow[8], prow[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                trow[u] = nrow_t[u];
                prow[u] = nrow_p[u];
            }
            const int next_tile =
                item + (int)gridDim.x < nitems ? item_span(p, item + gridDim.x).tile : -1;
            const int nj = kc1 - kc0;
            for (int j = 0; j < nj; ++j, ++g) {
                if (j == 1)
                    load_rows(next_tile);
                else if (j == kRowsPrep)
                    prep_rows();
                const int kc = chunk_at(kc0, kc1, j);
                const int s = g % S;
                const uint32_t n = g / S;
                if (!warp_wait_relaxed(empty_b + 8 * s, (n & 1) ^ 1, abort_flag, p.err)) {
                    ok = false;
                    break;
                }
                const uint32_t tb = base + s * pl.stage_bytes + pl.a_bytes + pl.u_bytes;
                gather_rows_async(tb, p.tok, trow, (int64_t)kc * BK, p.d, tt);
                if (p.has_pe && !pe_tile)
                    gather_rows_async(tb + pl.raw_bytes, p.pe, prow, (int64_t)kc * BK, p.d, tt);
                cp_async_arrive(full_b + 8 * s);
            }
            // items too short to reach those chunks
            if (nj <= 1)
                load_rows(next_tile);
            if (nj <= kRowsPrep)
                prep_rows();
        }
        cp_async_wait0();
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, tmem_cols);
    }
}

}  // namespace

namespace {

template <int MODE>
cudaError_t launch_mode(const ContractParams &p, int grid, uint32_t smem, cudaStream_t s,
                        bool dependent)
{
    cudaError_t e =
        cudaFuncSetAttribute(k_contract<MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess)
        return e;
    if (!dependent) {
        k_contract<MODE><<<grid, contract_threads(MODE), smem, s>>>(p);
        return e;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(contract_threads(MODE));
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, k_contract<MODE>, p);
}

}  // namespace

cudaError_t launch_contract(int mode, const ContractParams &p, int grid, cudaStream_t s,
                            bool dependent)
{
    const ContractPlan pl = contract_plan(mode, p.n_pad, p.k, p.has_pe, p.stages);
    cudaError_t e;
    switch (mode) {
    case CMODE_X: e = launch_mode<CMODE_X>(p, grid, pl.total, s, dependent); break;
    case CMODE_G: e = launch_mode<CMODE_G>(p, grid, pl.total, s, dependent); break;
    case CMODE_W: e = launch_mode<CMODE_W>(p, grid, pl.total, s, dependent); break;
    case CMODE_GF: e = launch_mode<CMODE_GF>(p, grid, pl.total, s, dependent); break;
    default: e = launch_mode<CMODE_XP>(p, grid, pl.total, s, dependent); break;
    }
    if (e != cudaSuccess)
        return e;
    count_launch();
    return cudaGetLastError();
}

}  // namespace tc
}  // namespace sn
