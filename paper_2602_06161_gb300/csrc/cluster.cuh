// cluster.cuh - inline-PTX wrappers for thread-block clusters on sm_103a: the CTA's rank, the
// mapping of a shared-memory address into another CTA of the cluster, bulk copies into another
// CTA's shared memory, and the cluster barrier.
#pragma once

#include <stdint.h>

namespace cover {

__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}

// The address, in the shared memory of the cluster's CTA `rank`, of what sits at this CTA's
// shared-memory address saddr (every CTA of the kernel has the same layout).
__device__ __forceinline__ uint32_t cluster_map(uint32_t saddr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(saddr), "r"(rank));
  return r;
}

// Bulk copy of `bytes` (a multiple of 16, both addresses 16-byte aligned) from this CTA's shared
// memory into the shared memory of a CTA of the cluster, completing `bytes` transactions on
// that CTA's mbarrier (cluster addresses from cluster_map).
__device__ __forceinline__ void bulk_copy_cluster(uint32_t dst_cluster, uint32_t src, uint32_t bytes,
                                                  uint32_t bar_cluster) {
  asm volatile("cp.async.bulk.shared::cluster.shared::cta.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                   dst_cluster),
               "r"(src), "r"(bytes), "r"(bar_cluster)
               : "memory");
}

// The cluster barrier, for every thread of every CTA of the cluster (converged warps): writes
// before a thread's arrival are visible to the cluster's reads after its wait. cluster_arrive
// and cluster_wait are its two halves, for work between a thread's arrival and its wait.
__device__ __forceinline__ void cluster_arrive() {
  asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait() { asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory"); }
__device__ __forceinline__ void cluster_sync() {
  cluster_arrive();
  cluster_wait();
}

}  // namespace cover
