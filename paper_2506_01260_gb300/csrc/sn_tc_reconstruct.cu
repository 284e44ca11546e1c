// sn_tc_reconstruct.cu — the forward reconstruction on the tcgen05 tensor cores,
//
//   X[t, :] = C[t, :] U^T + P[p_t, :] + T_fixed[id_t, :]          Sec. 4.3.1
//
// A work item is one 128-row tile and a run of 128-column output blocks.
//   warp 0     TMA producer: per block, the 128 rows of U (the B operand,
//              128-byte swizzled) into a ring of B stages;
//   warp 1     TMEM allocation and tcgen05.mma into three fp32 accumulator
//              buffers (M = 128, N = 128, K = k padded to 16) with the A
//              operand read from TMEM; each commit frees the B stage and
//              publishes the accumulator;
//   warps 2-9  two epilogue groups, one per 64-column half of every block.  A
//              thread drains its row of the group's half of the accumulator,
//              adds the row's positional and T_fixed entries in fp32, rounds
//              once to bf16 and writes the result over the T_fixed tile it just
//              read; the warp then stores its 32 rows with one TMA store and
//              frees the embedding stage once the store has read them;
//   warps 10-13 write each item's C rows into one of two TMEM A buffers (a
//              thread per row, zero-padded to a multiple of 16; 4-byte loads
//              when k is even), the next item's during the current item's
//              last half blocks (the first item's are written by the idle
//              epilogue warps), and fill the ring of embedding stages: per
//              half block, the T_fixed rows of the tile's ids (and the
//              positional rows when positions are not one contiguous run) with
//              16-byte cp.async copies into swizzled positions, or the
//              positional tile with one TMA load.  Each
//              thread hands its copies to the stage's barrier
//              (cp.async.mbarrier.arrive), which completes when all of them
//              have landed, so the gather warps never wait for their own copies
//              and every free stage can have copies in flight.
// The embeddings never pass through the tensor core, so the MMA issues only the
// k/16 instructions of C U^T per block; the B ring and the embedding ring are
// separate, so U rows are released as soon as the MMAs have read them; with A
// in TMEM, shared memory is left to the two rings.
// Each CTA walks an item's blocks starting at its own offset, so the CTAs'
// B-operand reads are spread over the L2 instead of converging on one slice.
// An item's start costs the gather warps, the pipeline's bottleneck, almost
// nothing: the next item's ids (and positions) are loaded and turned into
// row indices a few half blocks into the current item, and its A operand is
// loaded a chunk at a time over the current item's last half blocks; the
// gather warps' own waits and arrivals on the embedding ring are relaxed
// (they publish nothing and read nothing the epilogue wrote), so none of
// them holds a warp until those loads have returned.
// Every wait is bounded (SN_EBIT_TIMEOUT); an aborting CTA drains its copies
// and MMAs and frees TMEM before it returns.
#include "sn_tc.cuh"
#include "sn_tc_kernels.cuh"

namespace sn {
namespace tc {
namespace {

constexpr int NB = BN_WIDE;
// half blocks between the loads of one chunk of the next item's A and its
// write to TMEM (about the time a load spends behind the copies in flight)
constexpr int kAPreDist = 10;
// half block of an item at which the next item's gather rows are prepared
// (their ids were loaded at half block 1)
constexpr int kRowsPrep = 6;
constexpr uint32_t kTmemCols = 512;
static_assert(kReconAcc * NB <= (int)kReconACol && kReconACol + 2 * kReconAStride <= kTmemCols,
              "TMEM plan");
// paired form: two accumulator slots, then two A buffers of two tiles' C rows
// (at most 64 columns per tile, k <= 128)
static_assert(kPairAcc * NB <= (int)kPairACol && kPairACol + 2 * 2 * 64 <= kTmemCols,
              "TMEM plan (pairs)");

__device__ __forceinline__ int block_at(int blk0, int blk1, int j)
{
    const int nb = blk1 - blk0;
    return blk0 + (int)((j + blockIdx.x) % nb);
}

// acc + P + T_fixed for two adjacent columns, rounded once to bf16
__device__ __forceinline__ uint32_t add_emb(float a0, float a1, uint32_t pe, uint32_t te)
{
    return pack_bf16(add_bf16_lo(te, add_bf16_lo(pe, a0)), add_bf16_hi(te, add_bf16_hi(pe, a1)));
}

// 16 words (32 bf16) of C row t from word w0 on, zero past k and past the end;
// 4-byte loads when k is even (rows 4-byte aligned), 2-byte loads otherwise
__device__ __forceinline__ void load_c_words(const ExpandParams &p, int64_t t, int w0,
                                             uint32_t (&h)[16])
{
    const unsigned short *crow = (const unsigned short *)p.C + t * p.k;
    const uint32_t *crow32 = (const uint32_t *)(p.C + t * p.k);
    if ((p.k & 1) == 0) {
#pragma unroll
        for (int i = 0; i < 16; ++i)
            h[i] = (t < p.rows && 2 * (w0 + i) < p.k) ? __ldg(crow32 + w0 + i) : 0u;
    } else {
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            const int j0 = 2 * (w0 + i);
            const uint32_t lo = (t < p.rows && j0 < p.k) ? __ldg(crow + j0) : 0u;
            const uint32_t hi = (t < p.rows && j0 + 1 < p.k) ? __ldg(crow + j0 + 1) : 0u;
            h[i] = lo | (hi << 16);
        }
    }
}

__global__ void __launch_bounds__(kReconThreads, 1) k_reconstruct(const __grid_constant__ ExpandParams p)
{
    extern __shared__ uint8_t smem_raw[];
    uint32_t base = smem_u32(smem_raw);
    const uint32_t pad = (1024u - (base & 1023u)) & 1023u;
    base += pad;
    uint8_t *smem = smem_raw + pad;

    const int SB = p.stages, SE = p.estages;
    const ReconPlan pl = recon_plan(p.katoms, p.has_pe, SB, SE);
    const uint32_t b0 = base, e0 = b0 + SB * pl.b_bytes;
    const uint32_t bar = base + pl.bar_off;
    const uint32_t bfull_b = bar, bempty_b = bar + 8 * SB;
    const uint32_t efull_b = bar + 16 * SB, eempty_b = efull_b + 8 * SE;
    const uint32_t accf_b = eempty_b + 8 * SE, acce_b = accf_b + 8 * kReconAcc;
    const uint32_t afull_b = acce_b + 8 * kReconAcc, aempty_b = afull_b + 16;
    const uint32_t drain_b = aempty_b + 16;
    uint32_t *tmem_slot = (uint32_t *)(smem + pl.bar_off + 8 * (2 * SB + 2 * SE + 2 * kReconAcc + 5));
    volatile int *abort_flag = (volatile int *)(tmem_slot + 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < SB; ++s) {
            mbar_init(bfull_b + 8 * s, 1);
            mbar_init(bempty_b + 8 * s, 1);
        }
        for (int s = 0; s < SE; ++s) {
            // one copy-tracking arrival per gather thread + one for the
            // positional tile (a TMA load, or a plain arrival without one)
            mbar_init(efull_b + 8 * s, 128 + 1);
            mbar_init(eempty_b + 8 * s, 4);   // the four warps of one epilogue group
        }
        for (int b = 0; b < kReconAcc; ++b) {
            mbar_init(accf_b + 8 * b, 1);
            mbar_init(acce_b + 8 * b, 8);     // both epilogue groups
        }
        for (int b = 0; b < 2; ++b) {
            // the eight epilogue warps (the first item), or the four gather
            // warps arriving twice each (every later item)
            mbar_init(afull_b + 8 * b, 8);
            mbar_init(aempty_b + 8 * b, 1);
        }
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
    const int nitems = p.ntiles * p.chunks;

    if (warp == 0) {
        // ------------------------------------------------------------ B producer
        if (lane == 0)
            tma_prefetch(&p.mapB);
        uint32_t g = 0;
        bool ok = true;
        for (int item = blockIdx.x; item < nitems && ok; item += gridDim.x) {
            const int ch = item % p.chunks;
            const int blk0 = ch * p.bpi, blk1 = min(blk0 + p.bpi, p.nblk);
            for (int j = 0; j < blk1 - blk0; ++j, ++g) {
                const int blk = block_at(blk0, blk1, j);
                const int s = g % SB;
                if (!warp_wait(bempty_b + 8 * s, ((g / SB) & 1) ^ 1, abort_flag, p.err)) {
                    ok = false;
                    break;
                }
                if (lane == 0) {
                    const uint32_t fb = bfull_b + 8 * s, st = b0 + s * pl.b_bytes;
                    mbar_arrive_tx(fb, pl.b_bytes);
                    for (int a = 0; a < p.katoms; ++a)
                        tma_load_2d(st + a * (NB * 128), &p.mapB, a * 64, blk * NB, fb);
                }
                __syncwarp();
            }
        }
        if (!ok && lane == 0)
            for (uint32_t i = g > (uint32_t)SB ? g - SB : 0; i < g; ++i)
                drain_wait(bfull_b + 8 * (i % SB), (i / SB) & 1);
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
                const uint32_t ab = it & 1;
                if (!mbar_wait(afull_b + 8 * ab, (it >> 1) & 1, abort_flag, p.err)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t a_tmem = tmem + kReconACol + ab * kReconAStride;
                for (int j = 0; j < blk1 - blk0; ++j, ++g) {
                    const int s = g % SB;
                    const uint32_t b = g % kReconAcc;
                    if (!mbar_wait(bfull_b + 8 * s, (g / SB) & 1, abort_flag, p.err) ||
                        !mbar_wait(acce_b + 8 * b, ((g / kReconAcc) & 1) ^ 1, abort_flag, p.err)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t st = b0 + s * pl.b_bytes;
                    const uint32_t d_tmem = tmem + b * NB;
                    for (int kk = 0; kk < p.kmma; ++kk) {
                        const uint32_t a = kk >> 2, off = (kk & 3) * 32;
                        mma_bf16_ta(d_tmem, a_tmem + 8 * kk, sdesc_sw128(st + a * (NB * 128) + off),
                                    idesc, kk > 0 ? 1u : 0u);
                    }
                    mma_commit(bempty_b + 8 * s);    // U rows free once these MMAs finish
                    mma_commit(accf_b + 8 * b);
                }
                if (ok)
                    mma_commit(aempty_b + 8 * ab);   // A buffer free once this item's MMAs finish
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
        const int grp = (warp - 2) >> 2;     // the group's 64-column half of each block
        const int row = 32 * q + lane;
        uint32_t g = 0;
        bool ok = true;
        // the id (and position) of this thread's row, loaded an item ahead so
        // that an item's start does not wait for them
        int nid = 0, npos = 0;
        auto load_row = [&](int item_) {
            nid = 0;
            npos = 0;
            if (item_ < nitems) {
                const int64_t t = tile_row0(item_ / p.chunks, p.reorder, p.batches, p.seq_len) + row;
                if (t < p.rows) {
                    nid = p.ids[t];
                    if (p.has_pe && p.has_pos)
                        npos = p.pos[t];
                }
            }
        };
        load_row(blockIdx.x);
        if ((int)blockIdx.x < nitems) {
            // The first item's A operand: the epilogue warps are idle until the
            // first accumulator, so they write it (group g the 16-word chunks
            // m = g, g + 2) while the gather warps start their copies.
            const int nch = (8 * p.kmma + 15) / 16;
            const int64_t t = tile_row0((int)blockIdx.x / p.chunks, p.reorder, p.batches, p.seq_len) + row;
            uint32_t h[2][16];
#pragma unroll
            for (int i = 0; i < 2; ++i)
                if (grp + 2 * i < nch)
                    load_c_words(p, t, 16 * (grp + 2 * i), h[i]);
            const uint32_t a_lane = tmem + ((uint32_t)(32 * q) << 16) + kReconACol;
#pragma unroll
            for (int i = 0; i < 2; ++i)
                if (grp + 2 * i < nch)
                    tmem_st16(a_lane + 16 * (grp + 2 * i), h[i]);
            tmem_st_wait();
            tc_fence_before();
            __syncwarp();
            if (lane == 0)
                mbar_arrive(afull_b);              // A buffer 0
        }
        for (int item = blockIdx.x; item < nitems && ok; item += gridDim.x) {
            const int tile = item / p.chunks, ch = item % p.chunks;
            const int blk0 = ch * p.bpi, blk1 = min(blk0 + p.bpi, p.nblk);
            const int64_t r0 = tile_row0(tile, p.reorder, p.batches, p.seq_len);
            const int id = nid, ps = npos;
            load_row(item + gridDim.x);
            bool bad = false;
            if (r0 + row < p.rows) {
                bad = id < 0 || id >= p.vocab;
                if (p.has_pe && p.has_pos)
                    bad = bad || ps < 0 || ps >= p.seq_len;
                if (bad && ch == 0)
                    atomicOr(p.err, SN_EBIT_BAD_ID);
            }
            for (int j = 0; j < blk1 - blk0 && ok; ++j, ++g) {
                const int blk = block_at(blk0, blk1, j);
                const uint32_t b = g % kReconAcc;
                const uint32_t e = 2 * g + grp, es = e % SE, ph = (e / SE) & 1;
                if (!warp_wait(accf_b + 8 * b, (g / kReconAcc) & 1, abort_flag, p.err)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                float v[64];
                const uint32_t taddr = tmem + b * NB + 64 * grp + ((uint32_t)(32 * q) << 16);
#pragma unroll
                for (int i = 0; i < 4; ++i)
                    tmem_ld16(taddr + 16 * i, *(float(*)[16])(v + 16 * i));
                tmem_ld_wait();
                tc_fence_before();
                __syncwarp();
                if (lane == 0)
                    mbar_arrive(acce_b + 8 * b);
                if (!warp_wait(efull_b + 8 * es, ph, abort_flag, p.err)) {
                    ok = false;
                    break;
                }
                // the thread's own row of the T_fixed and positional tiles (a
                // quarter-warp's 8 rows fall in 8 different banks), summed in
                // fp32 and written back over the T_fixed tile
                const uint32_t tb = e0 + es * pl.e_bytes;
#pragma unroll
                for (int cb = 0; cb < 8; cb += 4) {
                    // all loads of four chunks first, then their sums
                    uint4 tv[4], pv[4];
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const uint32_t off = sw128(row, cb + i);
                        tv[i] = lds128(tb + off);
                        pv[i] = p.has_pe ? lds128(tb + pl.t_bytes + off) : make_uint4(0, 0, 0, 0);
                    }
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const float *a = v + 8 * (cb + i);
                        uint4 o = make_uint4(add_emb(a[0], a[1], pv[i].x, tv[i].x),
                                             add_emb(a[2], a[3], pv[i].y, tv[i].y),
                                             add_emb(a[4], a[5], pv[i].z, tv[i].z),
                                             add_emb(a[6], a[7], pv[i].w, tv[i].w));
                        if (bad)
                            o = make_uint4(0, 0, 0, 0);
                        sts128(tb + sw128(row, cb + i), o);
                    }
                }
                // the warp's 32 rows leave with one TMA store (clipped at the
                // tensor's edges); the stage is free once the store has read them
                fence_async_smem();
                __syncwarp();
                {
                    const int c0 = blk * NB + 64 * grp;
                    if (lane == 0 && r0 + 32 * q < p.rows && c0 < p.ncols8) {
                        tma_store_2d(&p.mapOut, tb + 32 * q * 128, c0, (int)(r0 + 32 * q));
                        bulk_commit();
                        bulk_wait_read0();
                    }
                }
                __syncwarp();
                if (lane == 0)
                    mbar_arrive(eempty_b + 8 * es);
            }
        }
        if (lane == 0)
            bulk_wait_all0();
    } else {
        // ------------------------------------------------------------ embedding gathers
        const int tt = threadIdx.x - 320;    // 0..127
        const int arow = 32 * (warp & 3) + lane;   // this thread's TMEM lane (A row)
        if (tt == 0 && p.has_pe)
            tma_prefetch(&p.mapPE);
        uint32_t g = 0, e = 0, it = 0;
        bool ok = true;
        // The next item's gather rows (this thread's 8 rows of T_fixed and P)
        // are prepared during the current item, where the gather warps wait for
        // free stages anyway: its ids and positions are loaded after the
        // item's first half block and turned into row indices a few half
        // blocks later, so an item starts with its first copies.
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
        const uint32_t a_lane = tmem + ((uint32_t)(32 * (warp & 3)) << 16) + kReconACol;
        const int nch = (8 * p.kmma + 15) / 16;    // 16-word chunks of a row of A
        load_rows((int)blockIdx.x < nitems ? (int)blockIdx.x / p.chunks : -1);
        prep_rows();
        // this item's A is written (the first item's by the epilogue warps,
        // later ones during the previous item)
        bool a_ready = true;
        for (int item = blockIdx.x; item < nitems && ok; item += gridDim.x, ++it) {
            const int ch = item % p.chunks;
            const int blk0 = ch * p.bpi, blk1 = min(blk0 + p.bpi, p.nblk);
            const int64_t r0 = nq0;
            const bool pe_tile = npe_tile;
            const int pe_row0 = pe_tile ? (int)(r0 % p.seq_len) : 0;
            int trow[8], prow[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                trow[u] = nrow_t[u];
                prow[u] = nrow_p[u];
            }
            if (!a_ready) {
                // A operand: row arow of the tile's C rows, two bf16 per TMEM
                // column, zero past k (and for rows past the end)
                const uint32_t ab = it & 1;
                if (!warp_wait(aempty_b + 8 * ab, ((it >> 1) & 1) ^ 1, abort_flag, p.err)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                for (int m = 0; m < nch; ++m) {
                    uint32_t h[16];
                    load_c_words(p, r0 + arow, 16 * m, h);
                    tmem_st16(a_lane + ab * kReconAStride + 16 * m, h);
                }
                tmem_st_wait();
                tc_fence_before();
                __syncwarp();
                if (lane == 0)
                    mbar_arrive_cnt(afull_b + 8 * ab, 2);
            }
            const bool has_next = item + (int)gridDim.x < nitems;
            const int next_tile = has_next ? (item + (int)gridDim.x) / p.chunks : -1;
            // The next item's A goes into the other A buffer while this item's
            // last nch * kAPreDist half blocks are issued: chunk m is loaded at
            // half block nh - (nch - m) kAPreDist and written to TMEM one
            // distance later, so its loads are in flight behind the copies
            // already queued instead of holding up the next item's start.
            const int nh = 2 * (blk1 - blk0);
            const bool pre = has_next && nh >= nch * kAPreDist;
            const uint32_t nab = (it + 1) & 1;
            const int64_t nt = (has_next ? tile_row0(next_tile, p.reorder, p.batches, p.seq_len) : 0) + arow;
            uint32_t ha[16];
            int mq = 0, hq = 0;
            for (int j = 0; j < blk1 - blk0 && ok; ++j, ++g) {
                const int blk = block_at(blk0, blk1, j);
                for (int hh = 0; hh < 2; ++hh, ++e, ++hq) {
                    if (hq == 1)
                        load_rows(next_tile);
                    else if (hq == kRowsPrep)
                        prep_rows();
                    if (pre && hq == nh - (nch - mq) * kAPreDist) {
                        if (mq == 0) {
                            if (!warp_wait_relaxed(aempty_b + 8 * nab, (((it + 1) >> 1) & 1) ^ 1,
                                                   abort_flag, p.err)) {
                                ok = false;
                                break;
                            }
                            tc_fence_after();
                        } else {
                            tmem_st16(a_lane + nab * kReconAStride + 16 * (mq - 1), ha);
                        }
                        load_c_words(p, nt, 16 * mq, ha);
                        ++mq;
                    }
                    const uint32_t es = e % SE;
                    if (!warp_wait_relaxed(eempty_b + 8 * es, ((e / SE) & 1) ^ 1, abort_flag, p.err)) {
                        ok = false;
                        break;
                    }
                    const uint32_t tb = e0 + es * pl.e_bytes;
                    const int col0 = blk * NB + 64 * hh;
                    if (tt == 0) {
                        const uint32_t pb = efull_b + 8 * es;
                        if (pe_tile) {
                            mbar_arrive_tx_relaxed(pb, kTile);
                            tma_load_2d(tb + pl.t_bytes, &p.mapPE, col0, pe_row0, pb);
                        } else {
                            mbar_arrive_relaxed(pb);
                        }
                    }
                    gather_rows_async(tb, p.tok, trow, col0, p.ncols, tt);
                    if (p.has_pe && !pe_tile)
                        gather_rows_async(tb + pl.t_bytes, p.pe, prow, col0, p.ncols, tt);
                    cp_async_arrive(efull_b + 8 * es);
                }
            }
            // items too short to reach those half blocks
            if (nh <= 1)
                load_rows(next_tile);
            if (nh <= kRowsPrep)
                prep_rows();
            if (pre) {
                if (mq > 0)
                    tmem_st16(a_lane + nab * kReconAStride + 16 * (mq - 1), ha);
                tmem_st_wait();
                if (ok) {
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0)
                        mbar_arrive_cnt_relaxed(afull_b + 8 * nab, 2);
                }
            }
            a_ready = pre && ok;
        }
        cp_async_wait0();
        // positional tiles still in flight after an abort
        if (!ok && tt == 0)
            for (uint32_t i = e > (uint32_t)SE ? e - SE : 0; i < e; ++i)
                drain_wait(efull_b + 8 * (i % SE), (i / SE) & 1);
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}


// ---------------------------------------------------------------------------------
// The paired form.  When every sequence of the batch covers the same positions in
// whole 128-row blocks, the tiles of sequences 2i and 2i + 1 at one position block
// add the same positional tile.  A work item is such a pair of tiles and a run of
// 128-column output blocks, walked in 64-column half blocks:
//   warp 0     TMA producer: per half block, its 64 rows of U (B operand);
//   warp 1     tcgen05.mma: per half block, one chain per tile (M = 128, N = 64,
//              K = k padded to 16) into the two halves of one of two 128-column
//              accumulator slots, A read from the tile's TMEM A buffer;
//   warps 2-5  the pair's first tile, warps 6-9 its second: a thread drains its
//              row of its tile's half of the slot, adds the shared positional
//              row and its T_fixed row in fp32, rounds once to bf16, writes over
//              its T_fixed tile and each warp stores its 32 rows with one TMA
//              store (both groups free the stage);
//   warps 10-13 both tiles' A operands for every item after the first (over
//              the previous item's last half blocks) and, per half block, both
//              tiles' T_fixed rows by 16-byte cp.async and the positional tile by
//              one TMA load.  The first item's A operands are written by the
//              epilogue warps, idle until the first accumulator, each thread a
//              whole C row in one round trip, so the first copies go out at once.
// One embedding stage holds two output half tiles in 48 KB instead of 64 KB and
// a B stage is 64 rows of U, so the ring holds 8 output half tiles where the
// single-tile form holds 5.  All rows of a batch of whole sequences are valid, so
// no row of a tile is clipped; invalid ids give zero rows as in the single-tile
// form.
__global__ void __launch_bounds__(kReconThreads, 1)
    k_reconstruct_pair(const __grid_constant__ ExpandParams p)
{
    extern __shared__ uint8_t smem_raw[];
    uint32_t base = smem_u32(smem_raw);
    const uint32_t pad = (1024u - (base & 1023u)) & 1023u;
    base += pad;
    uint8_t *smem = smem_raw + pad;

    const int SB = p.stages, SE = p.estages;
    const PairPlan pl = pair_plan(p.katoms, SB, SE);
    const uint32_t b0 = base, e0 = b0 + SB * pl.b_bytes;
    const uint32_t bar = base + pl.bar_off;
    const uint32_t bfull_b = bar, bempty_b = bar + 8 * SB;
    const uint32_t efull_b = bar + 16 * SB, eempty_b = efull_b + 8 * SE;
    const uint32_t accf_b = eempty_b + 8 * SE, acce_b = accf_b + 8 * kPairAcc;
    const uint32_t afull_b = acce_b + 8 * kPairAcc, aempty_b = afull_b + 16;
    const uint32_t drain_b = aempty_b + 16;
    uint32_t *tmem_slot = (uint32_t *)(smem + pl.bar_off + 8 * (2 * SB + 2 * SE + 2 * kPairAcc + 5));
    volatile int *abort_flag = (volatile int *)(tmem_slot + 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // TMEM columns of one tile's A operand (16-word chunks of a C row)
    const int nch = (8 * p.kmma + 15) / 16;
    const uint32_t aw = 16 * nch;

    if (threadIdx.x == 0) {
        for (int s = 0; s < SB; ++s) {
            mbar_init(bfull_b + 8 * s, 1);
            mbar_init(bempty_b + 8 * s, 1);
        }
        for (int s = 0; s < SE; ++s) {
            mbar_init(efull_b + 8 * s, 128 + 1);   // the gather threads + the positional tile
            mbar_init(eempty_b + 8 * s, 8);        // both epilogue groups
        }
        for (int b = 0; b < kPairAcc; ++b) {
            mbar_init(accf_b + 8 * b, 1);
            mbar_init(acce_b + 8 * b, 8);
        }
        for (int b = 0; b < 2; ++b) {
            // the eight epilogue warps (the first item), or the four gather
            // warps arriving twice each (every later item)
            mbar_init(afull_b + 8 * b, 8);
            mbar_init(aempty_b + 8 * b, 1);
        }
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
    const int nitems = p.ntiles * p.chunks;    // p.ntiles counts tile pairs here

    if (warp == 0) {
        // ------------------------------------------------------------ B producer
        if (lane == 0)
            tma_prefetch(&p.mapA);
        uint32_t g = 0;
        bool ok = true;
        for (int item = blockIdx.x; item < nitems && ok; item += gridDim.x) {
            const int ch = item % p.chunks;
            const int blk0 = ch * p.bpi, blk1 = min(blk0 + p.bpi, p.nblk);
            for (int j = 0; j < blk1 - blk0 && ok; ++j) {
                const int blk = block_at(blk0, blk1, j);
                for (int hh = 0; hh < 2; ++hh, ++g) {
                    const int s = g % SB;
                    if (!warp_wait(bempty_b + 8 * s, ((g / SB) & 1) ^ 1, abort_flag, p.err)) {
                        ok = false;
                        break;
                    }
                    if (lane == 0) {
                        const uint32_t fb = bfull_b + 8 * s, st = b0 + s * pl.b_bytes;
                        mbar_arrive_tx(fb, pl.b_bytes);
                        for (int a = 0; a < p.katoms; ++a)
                            tma_load_2d(st + a * (64 * 128), &p.mapA, a * 64, blk * NB + 64 * hh, fb);
                    }
                    __syncwarp();
                }
            }
        }
        if (!ok && lane == 0)
            for (uint32_t i = g > (uint32_t)SB ? g - SB : 0; i < g; ++i)
                drain_wait(bfull_b + 8 * (i % SB), (i / SB) & 1);
        __syncwarp();
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16(BM, 64);
            uint32_t g = 0, it = 0;
            bool ok = true;
            for (int item = blockIdx.x; item < nitems && ok; item += gridDim.x, ++it) {
                const int ch = item % p.chunks;
                const int blk0 = ch * p.bpi, blk1 = min(blk0 + p.bpi, p.nblk);
                const uint32_t ab = it & 1;
                if (!mbar_wait(afull_b + 8 * ab, (it >> 1) & 1, abort_flag, p.err)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t a_tmem = tmem + kPairACol + ab * 2 * aw;
                for (int j = 0; j < blk1 - blk0 && ok; ++j) {
                    for (int hh = 0; hh < 2; ++hh, ++g) {
                        const int s = g % SB;
                        const uint32_t b = g % kPairAcc;
                        if (!mbar_wait(bfull_b + 8 * s, (g / SB) & 1, abort_flag, p.err) ||
                            !mbar_wait(acce_b + 8 * b, ((g / kPairAcc) & 1) ^ 1, abort_flag, p.err)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        const uint32_t st = b0 + s * pl.b_bytes;
                        for (int t = 0; t < 2; ++t) {
                            const uint32_t d_tmem = tmem + b * NB + 64 * t;
                            for (int kk = 0; kk < p.kmma; ++kk) {
                                const uint32_t a = kk >> 2, off = (kk & 3) * 32;
                                mma_bf16_ta(d_tmem, a_tmem + t * aw + 8 * kk,
                                            sdesc_sw128(st + a * (64 * 128) + off), idesc,
                                            kk > 0 ? 1u : 0u);
                            }
                        }
                        mma_commit(bempty_b + 8 * s);    // U rows free once these MMAs finish
                        mma_commit(accf_b + 8 * b);
                    }
                }
                if (ok)
                    mma_commit(aempty_b + 8 * ab);       // the item's A buffer (both tiles) free
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
        const int grp = (warp - 2) >> 2;     // the group's tile of the pair
        const int row = 32 * q + lane;
        uint32_t g = 0;
        bool ok = true;
        // the id of this thread's row, loaded an item ahead
        int nid = 0;
        auto load_row = [&](int item_) {
            nid = 0;
            if (item_ < nitems) {
                const int64_t t = pair_row0(item_ / p.chunks, p.batches, p.seq_len) +
                                  (int64_t)grp * p.seq_len + row;
                if (t < p.rows)
                    nid = p.ids[t];
            }
        };
        load_row(blockIdx.x);
        if ((int)blockIdx.x < nitems) {
            // The first item's A operand, this group's tile: the epilogue warps
            // are idle until the first accumulator and can hold a whole C row,
            // so it arrives in one round trip while the gather warps start.
            const int64_t t = pair_row0((int)blockIdx.x / p.chunks, p.batches, p.seq_len) +
                              (int64_t)grp * p.seq_len + row;
            uint32_t h[4][16];
#pragma unroll
            for (int m = 0; m < 4; ++m)
                if (m < nch)
                    load_c_words(p, t, 16 * m, h[m]);
            const uint32_t a_lane = tmem + ((uint32_t)(32 * q) << 16) + kPairACol + grp * aw;
#pragma unroll
            for (int m = 0; m < 4; ++m)
                if (m < nch)
                    tmem_st16(a_lane + 16 * m, h[m]);
            tmem_st_wait();
            tc_fence_before();
            __syncwarp();
            if (lane == 0)
                mbar_arrive(afull_b);              // A buffer 0
        }
        for (int item = blockIdx.x; item < nitems && ok; item += gridDim.x) {
            const int pp = item / p.chunks, ch = item % p.chunks;
            const int blk0 = ch * p.bpi, blk1 = min(blk0 + p.bpi, p.nblk);
            const int64_t r0 = pair_row0(pp, p.batches, p.seq_len) + (int64_t)grp * p.seq_len;
            const int id = nid;
            load_row(item + gridDim.x);
            bool bad = false;
            if (r0 + row < p.rows) {
                bad = id < 0 || id >= p.vocab;
                if (bad && ch == 0)
                    atomicOr(p.err, SN_EBIT_BAD_ID);
            }
            for (int j = 0; j < blk1 - blk0 && ok; ++j) {
                const int blk = block_at(blk0, blk1, j);
                for (int hh = 0; hh < 2; ++hh, ++g) {
                    const uint32_t b = g % kPairAcc;
                    const uint32_t es = g % SE, ph = (g / SE) & 1;
                    if (!warp_wait(accf_b + 8 * b, (g / kPairAcc) & 1, abort_flag, p.err)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    float v[64];
                    const uint32_t taddr = tmem + b * NB + 64 * grp + ((uint32_t)(32 * q) << 16);
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        tmem_ld16(taddr + 16 * i, *(float(*)[16])(v + 16 * i));
                    tmem_ld_wait();
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0)
                        mbar_arrive(acce_b + 8 * b);
                    if (!warp_wait(efull_b + 8 * es, ph, abort_flag, p.err)) {
                        ok = false;
                        break;
                    }
                    const uint32_t tb = e0 + es * pl.e_bytes + grp * kTile;
                    const uint32_t pb = e0 + es * pl.e_bytes + 2 * kTile;
#pragma unroll
                    for (int cb = 0; cb < 8; cb += 4) {
                        uint4 tv[4], pv[4];
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            const uint32_t off = sw128(row, cb + i);
                            tv[i] = lds128(tb + off);
                            pv[i] = lds128(pb + off);
                        }
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            const float *a = v + 8 * (cb + i);
                            uint4 o = make_uint4(add_emb(a[0], a[1], pv[i].x, tv[i].x),
                                                 add_emb(a[2], a[3], pv[i].y, tv[i].y),
                                                 add_emb(a[4], a[5], pv[i].z, tv[i].z),
                                                 add_emb(a[6], a[7], pv[i].w, tv[i].w));
                            if (bad)
                                o = make_uint4(0, 0, 0, 0);
                            sts128(tb + sw128(row, cb + i), o);
                        }
                    }
                    fence_async_smem();
                    __syncwarp();
                    if (lane == 0 && r0 + 32 * q < p.rows) {
                        tma_store_2d(&p.mapOut, tb + 32 * q * 128, blk * NB + 64 * hh, (int)(r0 + 32 * q));
                        bulk_commit();
                        bulk_wait_read0();
                    }
                    __syncwarp();
                    if (lane == 0)
                        mbar_arrive(eempty_b + 8 * es);
                }
            }
        }
        if (lane == 0)
            bulk_wait_all0();
    } else {
        // ------------------------------------------------------------ gathers and A
        const int tt = threadIdx.x - 320;    // 0..127
        const int arow = 32 * (warp & 3) + lane;   // this thread's TMEM lane (A row)
        if (tt == 0)
            tma_prefetch(&p.mapPE);
        uint32_t e = 0, it = 0;
        bool ok = true;
        // T_fixed rows of this thread's 8 rows of each tile for the next item,
        // loaded one half block into the current item and checked a few later
        int nrow[2][8];
        int64_t nq0 = 0;
        auto load_rows = [&](int pp) {
            nq0 = pp >= 0 ? pair_row0(pp, p.batches, p.seq_len) : 0;
#pragma unroll
            for (int t = 0; t < 2; ++t)
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    const int64_t r = nq0 + (int64_t)t * p.seq_len + (tt >> 3) + 16 * u;
                    nrow[t][u] = pp >= 0 && r < p.rows ? ld_issue(p.ids + r) : 0;
                }
        };
        auto prep_rows = [&]() {   // invalid ids read row 0; the epilogue zeroes those rows
#pragma unroll
            for (int t = 0; t < 2; ++t)
#pragma unroll
                for (int u = 0; u < 8; ++u)
                    if (nrow[t][u] < 0 || nrow[t][u] >= p.vocab)
                        nrow[t][u] = 0;
        };
        const uint32_t a_lane = tmem + ((uint32_t)(32 * (warp & 3)) << 16) + kPairACol;
        const int nck = 2 * nch;               // chunks of one item's A (both tiles)
        load_rows((int)blockIdx.x < nitems ? (int)blockIdx.x / p.chunks : -1);
        prep_rows();
        // this item's A is written (the first item's by the epilogue warps,
        // later ones during the previous item)
        bool a_ready = true;
        for (int item = blockIdx.x; item < nitems && ok; item += gridDim.x, ++it) {
            const int ch = item % p.chunks;
            const int blk0 = ch * p.bpi, blk1 = min(blk0 + p.bpi, p.nblk);
            const int64_t r0 = nq0;
            const int pe_row0 = (int)(r0 % p.seq_len);
            int trow[2][8];
#pragma unroll
            for (int t = 0; t < 2; ++t)
#pragma unroll
                for (int u = 0; u < 8; ++u)
                    trow[t][u] = nrow[t][u];
            if (!a_ready) {
                const uint32_t ab = it & 1;
                if (!warp_wait(aempty_b + 8 * ab, ((it >> 1) & 1) ^ 1, abort_flag, p.err)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                for (int m = 0; m < nck; ++m) {
                    uint32_t h[16];
                    load_c_words(p, r0 + (int64_t)(m / nch) * p.seq_len + arow, 16 * (m % nch), h);
                    tmem_st16(a_lane + ab * 2 * aw + (m / nch) * aw + 16 * (m % nch), h);
                }
                tmem_st_wait();
                tc_fence_before();
                __syncwarp();
                if (lane == 0)
                    mbar_arrive_cnt(afull_b + 8 * ab, 2);
            }
            const bool has_next = item + (int)gridDim.x < nitems;
            const int next_pp = has_next ? (item + (int)gridDim.x) / p.chunks : -1;
            // The next item's A goes into the other A buffer while this item's
            // last half blocks are issued: chunk m is loaded at half block
            // nh - (nck - m) dist and written to TMEM one distance later.
            const int nh = 2 * (blk1 - blk0);
            const int dist = min(kAPreDist, nh / nck);
            const bool pre = has_next && dist >= 1;
            const uint32_t nab = (it + 1) & 1;
            const int64_t nr0 = has_next ? pair_row0(next_pp, p.batches, p.seq_len) : 0;
            uint32_t ha[16];
            int mq = 0, hq = 0;
            for (int j = 0; j < blk1 - blk0 && ok; ++j) {
                const int blk = block_at(blk0, blk1, j);
                for (int hh = 0; hh < 2; ++hh, ++e, ++hq) {
                    if (hq == 1)
                        load_rows(next_pp);
                    else if (hq == kRowsPrep)
                        prep_rows();
                    if (pre && hq == nh - (nck - mq) * dist) {
                        if (mq == 0) {
                            if (!warp_wait_relaxed(aempty_b + 8 * nab, (((it + 1) >> 1) & 1) ^ 1,
                                                   abort_flag, p.err)) {
                                ok = false;
                                break;
                            }
                            tc_fence_after();
                        } else {
                            const int m = mq - 1;
                            tmem_st16(a_lane + nab * 2 * aw + (m / nch) * aw + 16 * (m % nch), ha);
                        }
                        load_c_words(p, nr0 + (int64_t)(mq / nch) * p.seq_len + arow, 16 * (mq % nch), ha);
                        ++mq;
                    }
                    const uint32_t es = e % SE;
                    if (!warp_wait_relaxed(eempty_b + 8 * es, ((e / SE) & 1) ^ 1, abort_flag, p.err)) {
                        ok = false;
                        break;
                    }
                    const uint32_t sb = e0 + es * pl.e_bytes;
                    const int col0 = blk * NB + 64 * hh;
                    if (tt == 0) {
                        const uint32_t fb = efull_b + 8 * es;
                        mbar_arrive_tx_relaxed(fb, kTile);
                        tma_load_2d(sb + 2 * kTile, &p.mapPE, col0, pe_row0, fb);
                    }
                    gather_rows_async(sb, p.tok, trow[0], col0, p.ncols, tt);
                    gather_rows_async(sb + kTile, p.tok, trow[1], col0, p.ncols, tt);
                    cp_async_arrive(efull_b + 8 * es);
                }
            }
            // items too short to reach those half blocks
            if (nh <= 1)
                load_rows(next_pp);
            if (nh <= kRowsPrep)
                prep_rows();
            if (pre) {
                if (mq > 0) {
                    const int m = mq - 1;
                    tmem_st16(a_lane + nab * 2 * aw + (m / nch) * aw + 16 * (m % nch), ha);
                }
                tmem_st_wait();
                if (ok) {
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0)
                        mbar_arrive_cnt_relaxed(afull_b + 8 * nab, 2);
                }
            }
            a_ready = pre && ok;
        }
        cp_async_wait0();
        // positional tiles still in flight after an abort
        if (!ok && tt == 0)
            for (uint32_t i = e > (uint32_t)SE ? e - SE : 0; i < e; ++i)
                drain_wait(efull_b + 8 * (i % SE), (i / SE) & 1);
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}
}  // namespace

cudaError_t launch_reconstruct(const ExpandParams &p, int grid, cudaStream_t s)
{
    const ReconPlan pl = recon_plan(p.katoms, p.has_pe, p.stages, p.estages);
    cudaError_t e = cudaFuncSetAttribute(k_reconstruct, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         pl.total);
    if (e != cudaSuccess)
        return e;
    k_reconstruct<<<grid, kReconThreads, pl.total, s>>>(p);
    count_launch();
    return cudaGetLastError();
}

cudaError_t launch_reconstruct_pair(const ExpandParams &p, int grid, cudaStream_t s)
{
    const PairPlan pl = pair_plan(p.katoms, p.stages, p.estages);
    cudaError_t e = cudaFuncSetAttribute(k_reconstruct_pair, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         pl.total);
    if (e != cudaSuccess)
        return e;
    k_reconstruct_pair<<<grid, kReconThreads, pl.total, s>>>(p);
    count_launch();
    return cudaGetLastError();
}

}  // namespace tc
}  // namespace sn
