// sn_tc_kernels.cuh — parameter blocks and shared-memory plans of the
// tensor-core kernels (shared by the kernels and their host launchers).
#pragma once

#include <cuda.h>
#include <stdint.h>

#include "sn_internal.cuh"

namespace sn {
namespace tc {

constexpr int BM = 128;          // rows (tokens / W columns / d rows) per tile = MMA M
constexpr int BK = 64;           // contraction chunk: one 128-byte swizzle row of bf16
constexpr int BN_WIDE = 128;     // output columns per block of the expansions
constexpr uint32_t kSmemLimit = 232448;   // 227 KB per CTA
constexpr uint32_t kTile = BM * 128;      // one [128 x 64] bf16 swizzled tile

// ---- contraction: out[r, :] = A[r, :] . U   (A = X - E, G, or W^T) -----------
enum {
    CMODE_G = 0,    // C = G U (bf16 out)
    CMODE_X = 1,    // C = (X - T_fixed[ids] - P[pos]) U (bf16 out)
    CMODE_W = 2,    // fp32 partials of W^T U over d-ranges (projection pass 1)
    CMODE_GF = 3,   // C = A U, fp32 out (projected tables T_fixed U, P U)
    CMODE_XP = 4    // C = X U - TU[ids] - PU[pos] (bf16 out, projected tables)
};

struct ContractParams {
    CUtensorMap mapA;    // X or G [T, d] (SW128, box 64 x 128) | W [d, m] (SW128, box 64 x 64)
    CUtensorMap mapU;    // U^T padded [n_pad, d] (SW128, box 64 x n_pad)
    CUtensorMap mapPE;   // P [seq_len, d] (SW128, box 64 x 128), contiguous positions
    const __nv_bfloat16 *tok;   // T_fixed [vocab, d], rows gathered with cp.async
    const __nv_bfloat16 *pe;    // P [seq_len, d], gathered when positions are not contiguous
    const int32_t *ids;
    const int32_t *pos;
    __nv_bfloat16 *C;    // [T, k] output (G, X, XP modes)
    float *P;            // [splits, rows, n_pad] fp32 partial output (W mode)
    float *Cf;           // [rows, k] fp32 output (GF mode)
    const float *TU;     // [vocab, k] fp32 T_fixed U (XP mode)
    const float *PU;     // [seq_len, k] fp32 P U (XP mode) or null
    unsigned int *err;
    int64_t rows;        // T, or m (columns of W)
    int64_t vocab;
    int seq_len, has_pe, has_pos;
    int d, k, n_pad, acc_stride;
    int nkc;             // 64-wide chunks of d
    int kc_per_item;     // chunks per work item (all of them unless split)
    int splits;          // work items per row tile (W mode)
    int ntiles;          // row tiles
    int reorder, batches;
    int stages;
    // X, G, XP modes: the last tail_tiles row tiles run as tail_splits items of
    // tail_kc chunks each (the grid's last round would otherwise leave most SMs
    // idle); those items write fp32 partial rows to Ptail
    // [tail_tiles, tail_splits, 128, n_pad], summed afterwards by k_sum_tail
    int tail_tiles, tail_splits, tail_kc;
    float *Ptail;
};

// The row tile, split index and chunk range of work item `item`.
struct ItemSpan {
    int tile, split, kc0, kc1;
    bool tail;
};

__host__ __device__ inline int contract_items(const ContractParams &p)
{
    return (p.ntiles - p.tail_tiles) * p.splits + p.tail_tiles * p.tail_splits;
}

__host__ __device__ inline ItemSpan item_span(const ContractParams &p, int item)
{
    ItemSpan r;
    const int head = (p.ntiles - p.tail_tiles) * p.splits;
    if (item < head) {
        r.tile = item / p.splits;
        r.split = item % p.splits;
        r.kc0 = r.split * p.kc_per_item;
        r.kc1 = r.kc0 + p.kc_per_item < p.nkc ? r.kc0 + p.kc_per_item : p.nkc;
        r.tail = false;
    } else {
        const int j = item - head;
        r.tile = p.ntiles - p.tail_tiles + j / p.tail_splits;
        r.split = j % p.tail_splits;
        r.kc0 = r.split * p.tail_kc;
        r.kc1 = r.kc0 + p.tail_kc < p.nkc ? r.kc0 + p.tail_kc : p.nkc;
        r.tail = true;
    }
    return r;
}

__host__ __device__ constexpr int contract_threads(int mode) { return mode == CMODE_X ? 320 : 192; }

struct ContractPlan {
    uint32_t a_bytes, u_bytes, raw_bytes, pe_bytes, stage_bytes, cst_bytes, bar_off, total;
    uint32_t tx_bytes;
};

__host__ __device__ inline ContractPlan contract_plan(int mode, int n_pad, int k, int has_pe,
                                                      int stages)
{
    ContractPlan p;
    p.a_bytes = kTile;
    p.u_bytes = (uint32_t)n_pad * 128;
    p.raw_bytes = (mode == CMODE_X) ? kTile : 0;   // T_fixed rows
    p.pe_bytes = (mode == CMODE_X && has_pe) ? kTile : 0;
    p.stage_bytes = p.a_bytes + p.u_bytes + p.raw_bytes + p.pe_bytes;
    p.cst_bytes = (mode == CMODE_W)
                      ? 0
                      : (((uint32_t)BM * k * (mode == CMODE_GF ? 4 : 2) + 1023) & ~1023u);
    p.bar_off = (uint32_t)stages * p.stage_bytes + p.cst_bytes;
    p.total = p.bar_off + 8 * (2 * stages + 5) + 16 + 1024;   // + alignment slack
    p.tx_bytes = p.a_bytes + p.u_bytes + p.pe_bytes;
    return p;
}

// ---- expansion: out[r, n0:n0+128] = A[r, :] . B[n0:n0+128, :]^T ----------------------
enum { AMODE_REPACK = 0, AMODE_TMA = 1 };

// Shared by the plain expansion and the reconstruction.
struct ExpandParams {
    CUtensorMap mapA;    // A by TMA: U padded [d, k64] (SW128, box 64 x 128)
    CUtensorMap mapB;    // B rows: U padded [d, k64] | A^T [m, k64] (SW128, box 64 x 128)
    CUtensorMap mapOut;  // output [rows, ncols] (SW128, box 64 x 32)
    CUtensorMap mapPE;   // P (SW128, box 64 x 128), contiguous positions
    const __nv_bfloat16 *tok;   // T_fixed [vocab, ncols], rows gathered with cp.async
    const __nv_bfloat16 *pe;    // P [seq_len, ncols], gathered when positions are not contiguous
    const __nv_bfloat16 *C;   // A by repacking: [rows, k]
    __nv_bfloat16 *out;       // output base (ragged last columns are stored directly)
    int64_t out_ld;           // output leading dimension (elements)
    int ncols8;               // columns covered by mapOut: ncols rounded down to 8
    const int32_t *ids;
    const int32_t *pos;
    unsigned int *err;
    int64_t rows;        // T, or d
    int64_t vocab;
    int seq_len, has_pe, has_pos;
    int k, katoms, kmma;
    int ncols, nblk, bpi, chunks, ntiles;
    int reorder, batches;
    int stages;          // B-operand stages
    int estages;         // embedding stages (reconstruction)
};

// warp 0 producer, warp 1 MMA, warps 2-5 and 6-9 two epilogue groups
// (alternate blocks)
constexpr int kExpandThreads = 320;
constexpr int kExpandAcc = 4;     // TMEM accumulator buffers of 128 columns

struct ExpandPlan {
    uint32_t a_bytes, out_bytes, b_bytes, stage_bytes, bar_off, total;
};

// Shared memory of the plain expansion: A operand | two output staging tiles |
// stages of B rows | barriers.  A stage is released by the MMA commit; outputs
// have their own staging, so the stores never hold back the loads.
__host__ __device__ inline ExpandPlan expand_plan(int katoms, int stages)
{
    ExpandPlan p;
    p.a_bytes = (uint32_t)katoms * kTile;
    p.out_bytes = 2 * BM * BN_WIDE * 2;           // one staging tile per epilogue group
    p.b_bytes = (uint32_t)katoms * BN_WIDE * 128;
    p.stage_bytes = p.b_bytes;
    p.bar_off = p.a_bytes + p.out_bytes + (uint32_t)stages * p.stage_bytes;
    p.total = p.bar_off + 8 * (2 * stages + 2 * kExpandAcc + 3) + 16 + 1024;
    return p;
}

// ---- reconstruction: out[r, n0:n0+128] = C[r, :] . U[n0:n0+128, :]^T + P rows + T_fixed rows
// The A operand (the tile's C rows) lives in TMEM, double-buffered, next to three
// fp32 accumulators, so shared memory holds only `sb` B stages of 128 U rows and
// `se` embedding stages, each the [128 x 64] T_fixed tile and (with a positional
// table) the [128 x 64] positional tile of one half of an output block.  The
// epilogue writes each half's bf16 result over its T_fixed tile and stores it
// from there, so no separate staging tile is needed.
constexpr int kReconAcc = 3;              // accumulators of 128 columns
constexpr uint32_t kReconACol = 384;      // first TMEM column of the A buffers
constexpr uint32_t kReconAStride = 64;    // TMEM columns per A buffer (k <= 128)

struct ReconPlan {
    uint32_t b_bytes, t_bytes, e_bytes, bar_off, total;
};

__host__ __device__ inline ReconPlan recon_plan(int katoms, int has_pe, int sb, int se)
{
    ReconPlan p;
    p.b_bytes = (uint32_t)katoms * BN_WIDE * 128;
    p.t_bytes = kTile;
    p.e_bytes = has_pe ? 2 * kTile : kTile;
    p.bar_off = (uint32_t)sb * p.b_bytes + (uint32_t)se * p.e_bytes;
    p.total = p.bar_off + 8 * (2 * sb + 2 * se + 2 * kReconAcc + 5) + 16 + 1024;
    return p;
}

// warp 0 producer, warp 1 MMA, warps 2-5 and 6-9 two epilogue groups
// (one per half block), warps 10-13 A operand and row gathers
constexpr int kReconThreads = 448;

// The paired reconstruction (two row tiles that add the same positional tile):
// per 64-column half block, one B stage of 64 U rows and one embedding stage of
// both tiles' [128 x 64] T_fixed tiles and their one positional tile.  TMEM
// holds two accumulator slots of 128 columns (the half block of each tile side
// by side) and two A buffers of both tiles' C rows.
constexpr int kPairAcc = 2;               // accumulator slots of 2 x 64 columns
constexpr uint32_t kPairACol = 256;       // first TMEM column of the A buffers

struct PairPlan {
    uint32_t b_bytes, e_bytes, bar_off, total;
};

__host__ __device__ inline PairPlan pair_plan(int katoms, int sb, int se)
{
    PairPlan p;
    p.b_bytes = (uint32_t)katoms * 64 * 128;
    p.e_bytes = 3 * kTile;
    p.bar_off = (uint32_t)sb * p.b_bytes + (uint32_t)se * p.e_bytes;
    p.total = p.bar_off + 8 * (2 * sb + 2 * se + 2 * kPairAcc + 5) + 16 + 1024;
    return p;
}

// First row of the first tile of pair `pp`: pairs run position-block-major
// over sequences (0, 1), (2, 3), ... of a batch of `batches` (even) sequences of
// seq_len rows; the pair's second tile starts seq_len rows later.
__host__ __device__ inline int64_t pair_row0(int pp, int batches, int seq_len)
{
    const int half = batches >> 1;
    return (int64_t)(2 * (pp % half)) * seq_len + (int64_t)(pp / half) * BM;
}

// Row tile -> first row.  With `reorder`, tiles run position-block-major so the
// b sequences of a batch that share positional rows are processed together
// and the positional table is read from HBM once.
__host__ __device__ inline int64_t tile_row0(int tile, int reorder, int batches, int seq_len)
{
    if (reorder) {
        const int b = tile % batches, pt = tile / batches;
        return (int64_t)b * seq_len + (int64_t)pt * BM;
    }
    return (int64_t)tile * BM;
}

// ---- host side -----------------------------------------------------------------------
cudaError_t launch_contract(int mode, const ContractParams &p, int grid, cudaStream_t s,
                            bool dependent = false);
cudaError_t launch_expand(int amode, const ExpandParams &p, int grid, cudaStream_t s,
                          bool dependent = false);
cudaError_t launch_reconstruct(const ExpandParams &p, int grid, cudaStream_t s);
cudaError_t launch_reconstruct_pair(const ExpandParams &p, int grid, cudaStream_t s);

}  // namespace tc
}  // namespace sn
