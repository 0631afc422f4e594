// Helpers of the product-sums that run on CTA pairs (tcgen05 cta_group::2):
// cluster rank and barrier, peer shared-memory addresses and arrivals, TMA
// copies counted on the leader's barrier, the pair MMA and its commit, and
// the collective TMEM allocation.
#pragma once

#include "common.cuh"

namespace emu {

// ---- CTA pairs: a cluster of two CTAs on one TPC sharing each MMA
// (tcgen05 cta_group::2).  CTA rank 0 of the cluster (the leader) issues the
// MMAs; each CTA holds half of every operand tile and receives half of D.
__device__ __forceinline__ uint32_t cluster_rank()
{
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

// All threads of both CTAs: arrive with release, wait with acquire.
__device__ __forceinline__ void cluster_sync()
{
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// The shared::cluster address of the same shared-memory offset in CTA `rank`.
__device__ __forceinline__ uint32_t peer_addr(uint32_t local, uint32_t rank)
{
    uint32_t a;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(a) : "r"(local), "r"(rank));
    return a;
}

// Arrive on a barrier of the other CTA of the pair, given by its
// shared::cluster address.  Release at CTA scope, as for a local arrive: the
// barrier only orders TMEM reads (tcgen05 fences on both sides) and the
// arriving thread's own memory writes need not be visible to the waiter.  A
// cluster-scope release would make every arrive wait until the thread's
// outstanding global reductions are performed (measured: the pair kernel
// 27 % slower).
__device__ __forceinline__ void mbar_arrive_peer(uint32_t cl_addr)
{
    asm volatile("mbarrier.arrive.release.cta.shared::cluster.b64 _, [%0];" ::"r"(cl_addr) : "memory");
}

// TMA tile load into this CTA's shared memory whose bytes are counted on a
// barrier of either CTA of the pair (bar: a shared::cluster address).
__device__ __forceinline__ void tma_load_3d_pair(uint32_t dst, const CUtensorMap *map, uint32_t bar, int32_t c0,
                                                 int32_t c1, int32_t c2)
{
    asm volatile("cp.async.bulk.tensor.3d.cta_group::2.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
                 " [%0], [%1, {%3, %4, %5}], [%2];"
                 ::"r"(dst), "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(c0), "r"(c1), "r"(c2)
                 : "memory");
}

// D (+)= A x B^T over the pair, M = 256: A's rows 0-127 come from the leader's
// shared memory and rows 128-255 from the peer's (same offset), B's N rows
// half from each; D's rows 0-127 land in the leader's TMEM, 128-255 in the
// peer's (same address).
__device__ __forceinline__ void mma_bf16_pair(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                              uint32_t accumulate)
{
    asm volatile("{\n\t.reg .pred p;\n\t"
                 "setp.ne.b32 p, %4, 0;\n\t"
                 "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}"
                 ::"r"(d_tmem), "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
                 : "memory");
}

// One arrive on the barrier at this offset in both CTAs of the pair once the
// pair MMAs issued so far have completed.
__device__ __forceinline__ void mma_commit_pair(uint32_t bar)
{
    asm volatile("tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;"
                 ::"r"(bar), "h"((uint16_t)3) : "memory");
}

// TMEM of a pair: one warp in each CTA allocates and frees, collectively.
__device__ __forceinline__ void tmem_alloc_pair(uint32_t dst_smem, uint32_t ncols)
{
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem), "r"(ncols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols)
{
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}

}  // namespace emu
