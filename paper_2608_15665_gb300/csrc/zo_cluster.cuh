// Inline-PTX pieces of the SM-pair (2-CTA cluster) tensor-core kernels: the cluster rank
// and shared::cluster addresses, arrivals on the leader CTA's barriers, TMA loads whose
// bytes complete on the leader's barrier, the M = 256 tcgen05.mma of a pair and its
// commit to both CTAs.  Written against the public PTX ISA description of these
// instructions (cta_group::2 forms).
#pragma once

#include <cstdint>

#include "zo_sm100.cuh"

namespace zo {
namespace cta2 {

using sm100::smem_u32;

__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// shared::cluster address of `p` (a variable of this CTA's shared memory) in CTA `rank`
__device__ __forceinline__ uint32_t map_to(const void* p, uint32_t rank) {
  uint32_t a;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(a) : "r"(smem_u32(p)), "r"(rank));
  return a;
}
// arrive on the barrier at the same offset in the leader CTA
__device__ __forceinline__ void arrive_leader(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cluster.b64 _, [%0];" ::"r"(map_to(bar, 0)) : "memory");
}
// set the int at the same offset in the other CTA of the pair
__device__ __forceinline__ void store_peer(int* p, int v) {
  asm volatile("st.shared::cluster.u32 [%0], %1;" ::"r"(map_to(p, cluster_rank() ^ 1u)), "r"(v)
               : "memory");
}
// TMA load of a box into this CTA's shared memory whose bytes complete on the barrier at
// the same offset in the leader CTA
__device__ __forceinline__ void tma_load_2d_to_leader(void* smem_dst, const void* tmap, int32_t x,
                                                      int32_t y, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(smem_u32(smem_dst)),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(x), "r"(y), "r"(map_to(bar, 0))
      : "memory");
}
// every thread of both CTAs (non-aligned forms: the role branches of a kernel may leave a
// warp diverged; each warp reconverges first)
__device__ __forceinline__ void cluster_sync_all() {
  __syncwarp();
  asm volatile("barrier.cluster.arrive.release;" ::: "memory");
  asm volatile("barrier.cluster.wait.acquire;" ::: "memory");
}
__device__ __forceinline__ void tmem_alloc_pair(uint32_t* slot, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(slot)),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
// D (+)= A B^T over the pair: A (M = 256 rows, 128 in each CTA) from Tensor Memory, B (N
// rows, N / 2 in each CTA at the same shared-memory offset) from shared memory
__device__ __forceinline__ void mma_pair_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc,
                                            uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// the same with A from shared memory (128 rows in each CTA at the same offset)
__device__ __forceinline__ void mma_pair_ss(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                            uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// arrive once on the barrier at this offset in both CTAs when the pair's MMAs so far complete
__device__ __forceinline__ void commit_both(uint64_t* bar) {
  const uint16_t mask = 3;
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64"
      " [%0], %1;" ::"r"(smem_u32(bar)),
      "h"(mask)
      : "memory");
}

}  // namespace cta2
}  // namespace zo
