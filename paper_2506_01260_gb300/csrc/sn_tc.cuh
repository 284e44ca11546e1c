// sn_tc.cuh — inline-PTX building blocks for the sm_103a tensor-core kernels:
// mbarriers with bounded waits, TMA tile loads and stores, cp.async row gathers,
// tcgen05 TMEM allocation, MMA (kind::f16, bf16 in, fp32 accumulate), commit
// and TMEM loads, and the shared-memory matrix descriptors for the 128-byte
// swizzled K-major operand layout.
#pragma once

#include <cuda.h>
#include <stdint.h>

#include "sn_internal.cuh"

namespace sn {
namespace tc {

// A wait that has not completed after this long gives up (SN_EBIT_TIMEOUT).
constexpr uint64_t kWaitLimitNs = 2000000000ull;

__device__ __forceinline__ uint32_t smem_u32(const void *p)
{
    return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ uint64_t global_ns()
{
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// ---- mbarrier ----------------------------------------------------------------
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_fence_init()
{
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar)
{
    asm volatile("mbarrier.arrive.release.cta.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void mbar_arrive_cnt(uint32_t bar, uint32_t count)
{
    asm volatile("mbarrier.arrive.release.cta.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(count)
                 : "memory");
}
__device__ __forceinline__ void mbar_arrive_tx(uint32_t bar, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.release.cta.shared::cta.b64 _, [%0], %1;" ::"r"(bar),
                 "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ bool mbar_test(uint32_t bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{ .reg .pred p; mbarrier.try_wait.parity.acquire.cta.shared::cta.b64 p, [%1], %2; "
        "selp.u32 %0, 1, 0, p; }"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

// Bounded wait for the phase of `bar` with parity `parity` to complete (the
// usual convention: a fresh barrier reports parity 1 as complete).  Gives up
// when another role raised `abort` or after kWaitLimitNs, in which case it
// raises `abort` and records SN_EBIT_TIMEOUT.  Returns true on completion.
// The loop polls try_wait without a suspend-time hint: with a 100 us hint the
// expansion kernels' pipeline hand-offs came out 1.5% slower.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int *abort,
                                          unsigned int *err)
{
    if (mbar_test(bar, parity))
        return true;
    const uint64_t t0 = global_ns();
    while (true) {
        if (mbar_test(bar, parity))
            return true;
        if (*abort)
            return false;
        if (global_ns() - t0 > kWaitLimitNs) {
            *abort = 1;
            atomicOr(err, SN_EBIT_TIMEOUT);
            return false;
        }
    }
}

// Warp-uniform bounded wait: lane 0 waits (and decides on abort/timeout), the
// decision is broadcast, and every lane then observes the completed phase
// with acquire semantics.  All 32 lanes must call it.
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, volatile int *abort,
                                          unsigned int *err)
{
    int ok = 1;
    if ((threadIdx.x & 31) == 0)
        ok = mbar_wait(bar, parity, abort, err);
    ok = __shfl_sync(0xffffffffu, ok, 0);
    if (ok && (threadIdx.x & 31))
        mbar_test(bar, parity);
    return ok != 0;
}

// Relaxed forms for a role that, after a wait, only issues copies into a buffer
// another role has released and reads nothing that role published: a relaxed
// wait or arrival does not hold the thread until its own earlier loads have
// returned, so loads issued ahead (the next work item's ids and C rows) stay
// in flight across it.
__device__ __forceinline__ void mbar_arrive_relaxed(uint32_t bar)
{
    asm volatile("mbarrier.arrive.relaxed.cta.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void mbar_arrive_cnt_relaxed(uint32_t bar, uint32_t count)
{
    asm volatile("mbarrier.arrive.relaxed.cta.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(count)
                 : "memory");
}
__device__ __forceinline__ void mbar_arrive_tx_relaxed(uint32_t bar, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.relaxed.cta.shared::cta.b64 _, [%0], %1;" ::"r"(bar),
                 "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ bool mbar_test_relaxed(uint32_t bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{ .reg .pred p; mbarrier.try_wait.parity.relaxed.cta.shared::cta.b64 p, [%1], %2; "
        "selp.u32 %0, 1, 0, p; }"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}
// warp_wait with a relaxed poll by lane 0 alone (the other lanes observe
// nothing themselves).  All 32 lanes must call it.
__device__ __forceinline__ bool warp_wait_relaxed(uint32_t bar, uint32_t parity,
                                                  volatile int *abort, unsigned int *err)
{
    int ok = 1;
    if ((threadIdx.x & 31) == 0 && !mbar_test_relaxed(bar, parity)) {
        const uint64_t t0 = global_ns();
        while (true) {
            if (mbar_test_relaxed(bar, parity))
                break;
            if (*abort) {
                ok = 0;
                break;
            }
            if (global_ns() - t0 > kWaitLimitNs) {
                *abort = 1;
                atomicOr(err, SN_EBIT_TIMEOUT);
                ok = 0;
                break;
            }
        }
    }
    return __shfl_sync(0xffffffffu, ok, 0) != 0;
}

// Short bounded wait used only while draining after an abort.
__device__ __forceinline__ void drain_wait(uint32_t bar, uint32_t parity)
{
    const uint64_t t0 = global_ns();
    while (!mbar_test(bar, parity) && global_ns() - t0 < 200000000ull) {
    }
}

// ---- TMA ---------------------------------------------------------------------------
__device__ __forceinline__ void tma_prefetch(const CUtensorMap *m)
{
    asm volatile("prefetch.tensormap [%0];" ::"l"(m) : "memory");
}
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap *m, int x, int y,
                                            uint32_t bar)
{
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes "
        "[%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
        "l"(m), "r"(x), "r"(y), "r"(bar)
        : "memory");
}
__device__ __forceinline__ void tma_store_2d(const CUtensorMap *m, uint32_t src, int x, int y)
{
    asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%2, %3}], [%1];" ::
                     "l"(m),
                 "r"(src), "r"(x), "r"(y)
                 : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read0()
{
    asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}
__device__ __forceinline__ void bulk_wait_all0()
{
    asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
}
// Order this thread's generic-proxy shared-memory writes before later
// async-proxy (TMA, tensor core) accesses.
__device__ __forceinline__ void fence_async_smem()
{
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// ---- tcgen05 -----------------------------------------------------------------------
__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t ncols)
{
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     dst_smem),
                 "r"(ncols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols)
{
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
                 : "memory");
}
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// D[tmem] (+)= A[smem] * B[smem]; one thread issues.
__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc,
                                         uint32_t idesc, uint32_t accumulate)
{
    asm volatile(
        "{ .reg .pred p; setp.ne.u32 p, %4, 0; "
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p; }" ::"r"(d_tmem),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}
// D[tmem] (+)= A[tmem] * B[smem]; one thread issues.  Row m of A is TMEM lane
// m, its K elements packed two bf16 per 32-bit column (even element in the low
// half), K = 16 per instruction (8 columns).
__device__ __forceinline__ void mma_bf16_ta(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc,
                                            uint32_t idesc, uint32_t accumulate)
{
    asm volatile(
        "{ .reg .pred p; setp.ne.u32 p, %4, 0; "
        "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p; }" ::"r"(d_tmem),
        "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}
// Arrive on `bar` once every MMA this thread issued so far has completed.
__device__ __forceinline__ void mma_commit(uint32_t bar)
{
    asm volatile(
        "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
        : "memory");
}

// 32 lanes x 16 consecutive fp32 columns: thread i of the warp gets lane
// (warp quarter base + i), columns col .. col+15.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float (&v)[16])
{
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
        "%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
          "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
#pragma unroll
    for (int i = 0; i < 16; ++i)
        v[i] = __uint_as_float(r[i]);
}
__device__ __forceinline__ void tmem_ld_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

// 32 lanes x 16 consecutive 32-bit columns from registers: thread i of the warp
// writes lane (warp quarter base + i), columns col .. col+15.
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&v)[16])
{
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,"
        "%13,%14,%15,%16};" ::"r"(taddr),
        "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]),
        "r"(v[8]), "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]),
        "r"(v[15])
        : "memory");
}
__device__ __forceinline__ void tmem_st_wait() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// Instruction descriptor, kind::f16: bf16 A and B (K-major unless
// `a_mn_major`), fp32 D, shape M x N; `negate_a` computes D (+)= (-A) B.
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N, bool negate_a = false,
                                                  bool a_mn_major = false)
{
    return (1u << 4)                     // D format: fp32
           | (1u << 7)                   // A format: bf16
           | (1u << 10)                  // B format: bf16
           | ((negate_a ? 1u : 0u) << 13)
           | ((a_mn_major ? 1u : 0u) << 15)   // A stored MN-major
           | ((uint32_t)(N >> 3) << 17)  // N / 8
           | ((uint32_t)(M >> 4) << 24); // M / 16
}

// Shared-memory matrix descriptor of a K-major operand in the 128-byte
// swizzle layout: rows of 128 bytes (64 bf16 along K), 8-row groups 1024
// bytes apart, tile base 1024-byte aligned.  Stepping K by 16 elements inside
// the 128-byte row advances the start address by 32 bytes.
__device__ __forceinline__ uint64_t sdesc_sw128(uint32_t saddr)
{
    uint64_t d = 0;
    d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);   // start address / 16
    d |= (uint64_t)(16 >> 4) << 16;             // leading byte offset (unused here)
    d |= (uint64_t)(1024 >> 4) << 32;           // stride byte offset: 8 rows x 128 B
    d |= (uint64_t)1 << 46;                     // descriptor version (sm_100 family)
    d |= (uint64_t)2 << 61;                     // swizzle: 128 B
    return d;
}

// Shared-memory matrix descriptor of an MN-major operand in the 128-byte
// swizzle layout: each K row holds 64 consecutive M (or N) elements in 128
// bytes, 8-row K groups are `k_group_bytes` apart (stride byte offset) and the
// next 64 M elements start `mn_block_bytes` later (leading byte offset).
// Stepping K by 16 rows advances the start address by 2 K groups.
__device__ __forceinline__ uint64_t sdesc_mn_sw128(uint32_t saddr, uint32_t mn_block_bytes,
                                                   uint32_t k_group_bytes)
{
    uint64_t d = 0;
    d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
    d |= (uint64_t)((mn_block_bytes >> 4) & 0x3FFFu) << 16;
    d |= (uint64_t)((k_group_bytes >> 4) & 0x3FFFu) << 32;
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)2 << 61;
    return d;
}

// Byte offset of 16-byte chunk c (0..7) of row r in a 128-byte-swizzled tile.
__device__ __forceinline__ uint32_t sw128(int r, int c)
{
    return (uint32_t)(r * 128 + ((c ^ (r & 7)) << 4));
}

// ---- shared-memory vectors and bf16 packing -------------------------------------
__device__ __forceinline__ uint4 lds128(uint32_t a)
{
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "r"(a));
    return v;
}
__device__ __forceinline__ void sts128(uint32_t a, uint4 v)
{
    asm volatile("st.shared.v4.u32 [%0], {%1,%2,%3,%4};" ::"r"(a), "r"(v.x), "r"(v.y), "r"(v.z),
                 "r"(v.w)
                 : "memory");
}
__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }
// Two fp32 values -> packed bf16x2 (round-to-nearest-even), `lo` in the low half.
// c + (bf16 in the low / high half of w), one fp32 rounding, no unpacking
__device__ __forceinline__ float add_bf16_lo(uint32_t w, float c)
{
    float r;
    asm("{ .reg .b16 l, h; mov.b32 {l, h}, %1; add.rn.f32.bf16 %0, l, %2; }"
        : "=f"(r)
        : "r"(w), "f"(c));
    return r;
}
__device__ __forceinline__ float add_bf16_hi(uint32_t w, float c)
{
    float r;
    asm("{ .reg .b16 l, h; mov.b32 {l, h}, %1; add.rn.f32.bf16 %0, h, %2; }"
        : "=f"(r)
        : "r"(w), "f"(c));
    return r;
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi)
{
    uint32_t r;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
    return r;
}

// Programmatic dependent launch: a kernel launched with programmatic stream
// serialization may start before the previous kernel of its stream ends;
// griddep_wait blocks until that kernel has completed and its writes are
// visible (a no-op for a kernel launched normally), griddep_launch_dependents
// lets the next such kernel start being scheduled.
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void griddep_launch_dependents()
{
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Prefetch the 128-byte lines of [p, p + bytes) into L2.
__device__ __forceinline__ void prefetch_l2_range(const void *p, int bytes)
{
    const uintptr_t a0 = (uintptr_t)p & ~(uintptr_t)127, a1 = (uintptr_t)p + bytes;
    for (uintptr_t a = a0; a < a1; a += 128)
        asm volatile("prefetch.global.L2 [%0];" ::"l"(a));
}

// ---- cp.async: 16-byte global -> shared copies issued per thread -------------
// Used for row gathers: each thread places its chunks directly at their
// swizzled positions and hands their completion to the stage's mbarrier with
// cp_async_arrive (cp.async.mbarrier.arrive.noinc); the consumer that waits on
// that barrier fences toward the async proxy before the tensor cores or a TMA
// store read the rows.
// Copies `src_bytes` (0 or 16) bytes and zero-fills the rest of the 16.
__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src, uint32_t src_bytes)
{
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src),
                 "r"(src_bytes)
                 : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait1() { asm volatile("cp.async.wait_group 1;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait0() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }
// Arrive on `bar` once every cp.async this thread has issued so far has
// landed (the arrival is one of the barrier's expected arrivals).
__device__ __forceinline__ void cp_async_arrive(uint32_t bar)
{
    asm volatile("cp.async.mbarrier.arrive.noinc.shared::cta.b64 [%0];" ::"r"(bar) : "memory");
}

// Row gather of one [128 x 64] bf16 tile: thread tt (0..127) copies chunk
// (tt & 7) of rows (tt >> 3) + 16 u, u = 0..7, from src_rows[u] (element
// offsets into `table`) + col0, into the swizzled tile at `dst`.  Columns at
// or past `row_len` (a ragged last chunk) are zero-filled without a read.
__device__ __forceinline__ void gather_tile_async(uint32_t dst, const __nv_bfloat16 *table,
                                                  const int64_t (&src_rows)[8], int64_t col0,
                                                  int64_t row_len, int tt)
{
    const int c = tt & 7;
    const int64_t col = col0 + 8 * c;
    const bool in = col + 8 <= row_len;       // row_len is a multiple of 8
#pragma unroll
    for (int u = 0; u < 8; ++u) {
        const int r = (tt >> 3) + 16 * u;
        cp_async16(dst + sw128(r, c), table + src_rows[u] + (in ? col : 0), in ? 16u : 0u);
    }
}


// A 4-byte load issued where it is written: an asm volatile statement keeps its
// place among the other volatile statements, so a load meant to be in flight
// ahead of its use is not moved down to the use.
__device__ __forceinline__ int ld_issue(const int *p)
{
    int v;
    asm volatile("ld.global.nc.b32 %0, [%1];" : "=r"(v) : "l"(p));
    return v;
}

// gather_tile_async with the 8 rows given as row indices of a table whose rows
// are row_len elements long
__device__ __forceinline__ void gather_rows_async(uint32_t dst, const __nv_bfloat16 *table,
                                                  const int (&rows)[8], int64_t col0,
                                                  int64_t row_len, int tt)
{
    const int c = tt & 7;
    const int64_t col = col0 + 8 * c;
    const bool in = col + 8 <= row_len;       // row_len is a multiple of 8
#pragma unroll
    for (int u = 0; u < 8; ++u) {
        const int r = (tt >> 3) + 16 * u;
        cp_async16(dst + sw128(r, c), table + (int64_t)rows[u] * row_len + (in ? col : 0),
                   in ? 16u : 0u);
    }
}

}  // namespace tc
}  // namespace sn
