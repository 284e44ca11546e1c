// sn_tc_expand.cu — the plain k -> d expansion on the tcgen05 tensor cores.
//
//   decompress_bwd  G[t, :] = C[t, :] U^T                                 Sec. 4.4
//   project (b)     W'[i, :] = U[i, :] A   with A = U^T W from the first pass
//
// (The forward reconstruction, which also adds the embeddings, has its own
// kernel.)  A work item is one 128-row tile and a run of 128-column output
// blocks.
//   warp 0     TMA producer: per block, the 128 rows of the B operand (U, or
//              A^T); per item, the A operand when it comes from a tensor map
//              (all 128-byte swizzled);
//   warp 1     TMEM allocation and tcgen05.mma into four fp32 accumulator
//              buffers (M = 128, N = 128): C U^T over K = k padded to 16;
//   warps 2-9  two epilogue groups taking alternate blocks: drain the
//              accumulator 64 columns at a time, round once to bf16 into the
//              group's swizzled staging tile and write each warp's 32 rows with
//              coalesced 16-byte stores (the TMA unit is left to the loads);
//              together the groups repack each item's C rows into the swizzled
//              K-major A operand (zero-padded).  Stages are released by the MMA
//              commit.
// Each CTA walks an item's blocks starting at its own offset, so the CTAs'
// B-operand reads are spread over the L2 instead of converging on one slice.
// Every wait is bounded (SN_EBIT_TIMEOUT); an aborting CTA drains its copies
// and MMAs and frees TMEM before it returns.
#include "sn_tc.cuh"
#include "sn_tc_kernels.cuh"

namespace sn {
namespace tc {
namespace {

// j-th block of an item: every CTA starts at a different block so that the
// CTAs do not all read the same rows of the B operand from one L2 slice at once.
__device__ __forceinline__ int block_at(int blk0, int blk1, int j)
{
    const int nb = blk1 - blk0;
    return blk0 + (int)((j + blockIdx.x) % nb);
}

template <int AMODE>
__global__ void __launch_bounds__(kExpandThreads, 1) k_expand(const __grid_constant__ ExpandParams p)
{
    extern __shared__ uint8_t smem_raw[];
    uint32_t base = smem_u32(smem_raw);
    const uint32_t pad = (1024u - (base & 1023u)) & 1023u;
    base += pad;
    uint8_t *smem = smem_raw + pad;

    const int S = p.stages;
    const ExpandPlan pl = expand_plan(p.katoms, S);
    const uint32_t a_s = base, out_s = base + pl.a_bytes;
    const uint32_t stage0 = out_s + pl.out_bytes;
    const uint32_t bar = base + pl.bar_off;
    const uint32_t full_b = bar, empty_b = bar + 8 * S;
    const uint32_t accf_b = bar + 16 * S, acce_b = accf_b + 8 * kExpandAcc;
    const uint32_t afull_b = acce_b + 8 * kExpandAcc, aempty_b = afull_b + 8;
    const uint32_t drain_b = aempty_b + 8;
    uint32_t *tmem_slot = (uint32_t *)(smem + pl.bar_off + 8 * (2 * S + 2 * kExpandAcc + 3));
    volatile int *abort_flag = (volatile int *)(tmem_slot + 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    constexpr int NB = BN_WIDE;
    constexpr uint32_t kTmemCols = kExpandAcc * NB;

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(full_b + 8 * s, 1);
            mbar_init(empty_b + 8 * s, 1);
        }
        for (int b = 0; b < kExpandAcc; ++b) {
            mbar_init(accf_b + 8 * b, 1);
            mbar_init(acce_b + 8 * b, 4);
        }
        mbar_init(afull_b, AMODE == AMODE_REPACK ? 8 : 1);
        mbar_init(aempty_b, 1);
        mbar_init(drain_b, 1);
        *abort_flag = 0;
        mbar_fence_init();
    }
    if (warp == 1)
        tmem_alloc(smem_u32(tmem_slot), kTmemCols);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    griddep_wait();   // the projection's third pass: the previous passes' writes are visible
    const int nitems = p.ntiles * p.chunks;

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            tma_prefetch(&p.mapB);
            if (AMODE == AMODE_TMA)
                tma_prefetch(&p.mapA);
        }
        uint32_t g = 0, it = 0;
        bool ok = true;
        for (int item = blockIdx.x; item < nitems && ok; item += gridDim.x, ++it) {
            const int tile = item / p.chunks, ch = item % p.chunks;
            const int blk0 = ch * p.bpi, blk1 = min(blk0 + p.bpi, p.nblk);
            const int64_t r0 = tile_row0(tile, p.reorder, p.batches, p.seq_len);
            if (AMODE == AMODE_TMA) {
                if (!warp_wait(aempty_b, (it & 1) ^ 1, abort_flag, p.err)) {
                    ok = false;
                    break;
                }
                if (lane == 0) {
                    mbar_arrive_tx(afull_b, pl.a_bytes);
                    for (int a = 0; a < p.katoms; ++a)
                        tma_load_2d(a_s + a * kTile, &p.mapA, a * 64, (int)r0, afull_b);
                }
                __syncwarp();
            }
            const uint32_t tx = pl.b_bytes;
            for (int j = 0; j < blk1 - blk0; ++j, ++g) {
                const int blk = block_at(blk0, blk1, j);
                const int s = g % S;
                const uint32_t n = g / S;
                if (!warp_wait(empty_b + 8 * s, (n & 1) ^ 1, abort_flag, p.err)) {
                    ok = false;
                    break;
                }
                const uint32_t st = stage0 + s * pl.stage_bytes;
                const uint32_t fb = full_b + 8 * s;
                if (lane == 0) {
                    mbar_arrive_tx(fb, tx);
                    for (int a = 0; a < p.katoms; ++a)
                        tma_load_2d(st + a * (NB * 128), &p.mapB, a * 64, blk * NB, fb);
                }
                __syncwarp();
            }
        }
        if (!ok && lane == 0) {
            for (uint32_t i = g > (uint32_t)S ? g - S : 0; i < g; ++i)
                drain_wait(full_b + 8 * (i % S), (i / S) & 1);
            if (AMODE == AMODE_TMA && it > 0)
                drain_wait(afull_b, (it - 1) & 1);
        }
        __syncwarp();
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16(BM, NB);
            uint32_t g = 0, it = 0;
            bool ok = true;
            for (int item = blockIdx.x; item < nitems && ok; item += gridDim.x, ++it) {
                const int ch = item % p.chunks;
                const int blk0 = ch * p.bpi, blk1 = min(blk0 + p.bpi, p.nblk);
                if (!mbar_wait(afull_b, it & 1, abort_flag, p.err)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                for (int j = 0; j < blk1 - blk0; ++j, ++g) {
                    const int s = g % S;
                    const uint32_t n = g / S, b = g % kExpandAcc, nb = g / kExpandAcc;
                    if (!mbar_wait(full_b + 8 * s, n & 1, abort_flag, p.err) ||
                        !mbar_wait(acce_b + 8 * b, (nb & 1) ^ 1, abort_flag, p.err)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t st = stage0 + s * pl.stage_bytes;
                    const uint32_t d_tmem = tmem + b * NB;
                    for (int kk = 0; kk < p.kmma; ++kk) {
                        const uint32_t a = kk >> 2, off = (kk & 3) * 32;
                        mma_bf16(d_tmem, sdesc_sw128(a_s + a * kTile + off),
                                 sdesc_sw128(st + a * (NB * 128) + off), idesc, kk > 0 ? 1u : 0u);
                    }
                    mma_commit(empty_b + 8 * s);     // stage free once these MMAs finish
                    mma_commit(accf_b + 8 * b);
                }
                if (ok)
                    mma_commit(aempty_b);
            }
            if (!ok) {
                mma_commit(drain_b);
                drain_wait(drain_b, 0);
            }
        }
        __syncwarp();
    } else if (warp < 10) {
        // ------------------------------------------------------------ epilogue groups
        const int q = warp & 3;
        const int grp = (warp - 2) >> 2;     // blocks g with g % 2 == grp
        const int tt = 32 * ((warp - 2) & 3) + lane;   // 0..127 within the group
        const int row = 32 * q + lane;
        uint32_t g = 0, it = 0;
        bool ok = true;
        for (int item = blockIdx.x; item < nitems && ok; item += gridDim.x, ++it) {
            const int tile = item / p.chunks, ch = item % p.chunks;
            const int blk0 = ch * p.bpi, blk1 = min(blk0 + p.bpi, p.nblk);
            const int64_t r0 = tile_row0(tile, p.reorder, p.batches, p.seq_len);
            if (AMODE == AMODE_REPACK) {
                // A operand: rows r0 .. r0+127 of C, zero-padded to katoms * 64
                // columns.  Both groups share it: thread (r, half) covers atom
                // `half` (two atoms) or chunks 4 half .. 4 half + 3 (one atom) of
                // row r, issuing all of its loads before the first use.
                if (!warp_wait(aempty_b, (it & 1) ^ 1, abort_flag, p.err)) {
                    ok = false;
                    break;
                }
                const int r = tt, half = grp;
                const int64_t t = r0 + r;
                const int a = p.katoms == 2 ? half : 0;
                const int cbeg = p.katoms == 2 ? 0 : 4 * half;
                const int jbeg = a * 64 + cbeg * 8;
                const unsigned short *crow = (const unsigned short *)p.C + t * p.k;
                uint32_t h[32];
#pragma unroll
                for (int e = 0; e < 32; ++e) {
                    const int j0 = jbeg + 2 * e;
                    // one atom covers 64 columns: with two atoms each thread takes
                    // 32 words, with one atom 16 words
                    const bool want = (p.katoms == 2 || e < 16) && t < p.rows;
                    const uint32_t lo = (want && j0 < p.k) ? __ldg(crow + j0) : 0u;
                    const uint32_t hi = (want && j0 + 1 < p.k) ? __ldg(crow + j0 + 1) : 0u;
                    h[e] = lo | (hi << 16);
                }
                const int nchunks = p.katoms == 2 ? 8 : 4;
#pragma unroll
                for (int c = 0; c < 8; ++c)
                    if (c < nchunks)
                        sts128(a_s + a * kTile + sw128(r, cbeg + c),
                               make_uint4(h[4 * c], h[4 * c + 1], h[4 * c + 2], h[4 * c + 3]));
                fence_async_smem();
                __syncwarp();
                if (lane == 0)
                    mbar_arrive(afull_b);
            }
            for (int j = 0; j < blk1 - blk0; ++j, ++g) {
                if ((int)(g & 1) != grp)
                    continue;
                const int blk = block_at(blk0, blk1, j);
                const uint32_t b = g % kExpandAcc, nb = g / kExpandAcc;
                if (!warp_wait(accf_b + 8 * b, nb & 1, abort_flag, p.err)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                // drain the accumulator 64 columns at a time and stage the rounded
                // values in this group's swizzled staging tile (one [128 x 64]
                // atom per 64 columns; the warp touches only its own 32 rows)
                const uint32_t slot = out_s + grp * (NB / 64) * kTile;
                const int c0 = blk * NB;
#pragma unroll
                for (int h = 0; h < NB / 64; ++h) {
                    float v[64];
                    const uint32_t taddr = tmem + b * NB + 64 * h + ((uint32_t)(32 * q) << 16);
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        tmem_ld16(taddr + 16 * i, *(float(*)[16])(v + 16 * i));
                    tmem_ld_wait();
                    if (h == NB / 64 - 1) {
                        tc_fence_before();
                        __syncwarp();
                        if (lane == 0)
                            mbar_arrive(acce_b + 8 * b);
                    }
#pragma unroll
                    for (int c = 0; c < 8; ++c) {
                        sts128(slot + h * kTile + sw128(row, c),
                               make_uint4(pack_bf16(v[8 * c + 0], v[8 * c + 1]),
                                          pack_bf16(v[8 * c + 2], v[8 * c + 3]),
                                          pack_bf16(v[8 * c + 4], v[8 * c + 5]),
                                          pack_bf16(v[8 * c + 6], v[8 * c + 7])));
                    }
                    // columns past the 8-aligned width are written element by element
                    const int ch0 = c0 + 64 * h;
                    if (ch0 + 64 > p.ncols8 && p.ncols > p.ncols8) {
                        const int64_t t = r0 + row;
                        if (t < p.rows) {
#pragma unroll
                            for (int e = 0; e < 64; ++e)
                                if (ch0 + e >= p.ncols8 && ch0 + e < p.ncols)
                                    p.out[t * p.out_ld + ch0 + e] = __float2bfloat16_rn(v[e]);
                        }
                    }
                }
                __syncwarp();
                // coalesced 16-byte stores: NB / 8 lanes per output row segment
                constexpr int kCpr = NB / 8, kRpi = 32 / kCpr;
                const int chunk = lane % kCpr;
                const bool col_ok = c0 + 8 * chunk + 8 <= p.ncols8;
                const uint32_t src = slot + (chunk >> 3) * kTile;
#pragma unroll
                for (int i = 0; i < 32 / kRpi; ++i) {
                    const int rr = 32 * q + kRpi * i + lane / kCpr;
                    const int64_t t = r0 + rr;
                    const uint4 o = lds128(src + sw128(rr, chunk & 7));
                    if (col_ok && t < p.rows)
                        *(uint4 *)(p.out + t * p.out_ld + c0 + 8 * chunk) = o;
                }
                __syncwarp();
            }
        }

    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

}  // namespace

cudaError_t launch_expand(int amode, const ExpandParams &p, int grid, cudaStream_t s,
                          bool dependent)
{
    const ExpandPlan pl = expand_plan(p.katoms, p.stages);
    cudaError_t e;
    if (amode == AMODE_REPACK) {
        e = cudaFuncSetAttribute(k_expand<AMODE_REPACK>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 pl.total);
        if (e == cudaSuccess)
            k_expand<AMODE_REPACK><<<grid, kExpandThreads, pl.total, s>>>(p);
    } else {
        e = cudaFuncSetAttribute(k_expand<AMODE_TMA>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 pl.total);
        if (e == cudaSuccess && dependent) {
            // may start while the previous kernel of the stream finishes (it
            // waits for it in griddep_wait before touching global memory)
            cudaLaunchConfig_t cfg = {};
            cfg.gridDim = dim3(grid);
            cfg.blockDim = dim3(kExpandThreads);
            cfg.dynamicSmemBytes = pl.total;
            cfg.stream = s;
            cudaLaunchAttribute attr[1];
            attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
            attr[0].val.programmaticStreamSerializationAllowed = 1;
            cfg.attrs = attr;
            cfg.numAttrs = 1;
            e = cudaLaunchKernelEx(&cfg, k_expand<AMODE_TMA>, p);
        } else if (e == cudaSuccess) {
            k_expand<AMODE_TMA><<<grid, kExpandThreads, pl.total, s>>>(p);
        }
    }
    if (e != cudaSuccess)
        return e;
    count_launch();
    return cudaGetLastError();
}

}  // namespace tc
}  // namespace sn
