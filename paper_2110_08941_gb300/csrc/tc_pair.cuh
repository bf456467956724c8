// PTX wrappers for the SM-pair (cluster of two CTAs, tcgen05 cta_group::2) tensor-core kernels:
// cluster rank and barrier, shared-memory address mapping, pair TMA loads, the collective
// tensor-memory allocation, pair MMA issue and multicast commit.  Internal to libhs.
#pragma once

#include "tc_device.cuh"

namespace hs {
namespace tcpair {

__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// Address of the same shared-memory variable in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t map_to_rank(uint32_t addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
  return r;
}
__device__ __forceinline__ void tma_load_2d_pair(uint32_t dst, const CUtensorMap* tm, int c0, int c1,
                                                 uint32_t leader_bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];"
      ::"r"(dst), "l"(reinterpret_cast<uint64_t>(tm)), "r"(c0), "r"(c1), "r"(leader_bar)
      : "memory");
}
__device__ __forceinline__ void tma_load_4d_pair(uint32_t dst, const CUtensorMap* tm, const int (&c)[4],
                                                 uint32_t leader_bar) {
  asm volatile(
      "cp.async.bulk.tensor.4d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes "
      "[%0], [%1, {%2, %3, %4, %5}], [%6];"
      ::"r"(dst), "l"(reinterpret_cast<uint64_t>(tm)), "r"(c[0]), "r"(c[1]), "r"(c[2]), "r"(c[3]), "r"(leader_bar)
      : "memory");
}
__device__ __forceinline__ void tmem_alloc_pair(uint32_t dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish_pair() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void umma_bf16_pair(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                               uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}"
      ::"r"(d_tmem), "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// Arrive (once the issuing thread's MMAs complete) on the barrier at this offset in both CTAs.
__device__ __forceinline__ void umma_commit_pair(uint32_t bar) {
  const uint16_t mask = 3;
  asm volatile("tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;"
               ::"r"(bar), "h"(mask)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t cluster_addr) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr) : "memory");
}


// The pair MMAs of one k-block (64 rows of K, four 16-row steps) from the stage whose A and B
// descriptors are `ad` and `bd`: within a stage a K step advances the start address by 2 KB
// (MN-major tile) or 32 B (K-major tile), i.e. the descriptor's address field by 128 or 2.  The
// issuing thread is on the tensor core's critical path, so descriptors are formed by one add.
template <bool A_MN, bool B_MN>
__device__ __forceinline__ void mma_kblock_pair(uint32_t d_tmem, uint64_t ad, uint64_t bd, uint32_t idesc,
                                                uint32_t acc0) {
  constexpr uint64_t kA = A_MN ? (2048 >> 4) : (32 >> 4);
  constexpr uint64_t kB = B_MN ? (2048 >> 4) : (32 >> 4);
  umma_bf16_pair(d_tmem, ad, bd, idesc, acc0);
  umma_bf16_pair(d_tmem, ad + kA, bd + kB, idesc, 1u);
  umma_bf16_pair(d_tmem, ad + 2 * kA, bd + 2 * kB, idesc, 1u);
  umma_bf16_pair(d_tmem, ad + 3 * kA, bd + 3 * kB, idesc, 1u);
}
// The first `steps` (1..4) of them: a group's last k-block, whose later steps are zero fill.
template <bool A_MN, bool B_MN>
__device__ __forceinline__ void mma_ksteps_pair(uint32_t d_tmem, uint64_t ad, uint64_t bd, uint32_t idesc,
                                                uint32_t acc0, int steps) {
  constexpr uint64_t kA = A_MN ? (2048 >> 4) : (32 >> 4);
  constexpr uint64_t kB = B_MN ? (2048 >> 4) : (32 >> 4);
#pragma unroll 1
  for (int kk = 0; kk < steps; ++kk)
    umma_bf16_pair(d_tmem, ad + kk * kA, bd + kk * kB, idesc, kk ? 1u : acc0);
}

}  // namespace tcpair
}  // namespace hs
