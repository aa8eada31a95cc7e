// Distributed shared memory access within a thread-block cluster through
// 32-bit shared::cluster addresses (mapa + ld/st.shared::cluster).
#pragma once
#include <stdint.h>

namespace rosetta {

__device__ __forceinline__ uint32_t smem_addr(const void *p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// Address of the same shared-memory location in CTA `rank` of the cluster
// (the windows are linear: mapa(a + off, r) = mapa(a, r) + off).
__device__ __forceinline__ uint32_t dsmem_map(uint32_t local, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(local), "r"(rank));
  return r;
}

// Cluster barrier that orders shared memory only: each thread's earlier
// writes to its own CTA's shared memory are visible to the reads that the
// cluster's CTAs make through distributed shared memory after the barrier.
// The plain cluster barrier (release and acquire at cluster scope) orders
// global memory as well, which the blind-rotation step loops never need
// across a barrier (their global accesses read keys and inputs only); a
// release fence restricted to shared::cta before a relaxed arrive, and an
// acquire fence restricted to shared::cluster after the wait, give the
// ordering they do need.  Valid only where every write before the barrier
// that a remote CTA reads after it went to the writer's own shared memory.
__device__ __forceinline__ void cluster_sync_shared() {
  asm volatile(
      "fence.release.sync_restrict::shared::cta.cluster;\n\t"
      "barrier.cluster.arrive.relaxed.aligned;\n\t"
      "barrier.cluster.wait.aligned;\n\t"
      "fence.acquire.sync_restrict::shared::cluster.cluster;" ::: "memory");
}

__device__ __forceinline__ uint64_t dsmem_ld_u64(uint32_t a) {
  uint64_t v;
  asm volatile("ld.shared::cluster.u64 %0, [%1];" : "=l"(v) : "r"(a) : "memory");
  return v;
}

__device__ __forceinline__ int32_t dsmem_ld_s32(uint32_t a) {
  int32_t v;
  asm volatile("ld.shared::cluster.s32 %0, [%1];" : "=r"(v) : "r"(a) : "memory");
  return v;
}

__device__ __forceinline__ uint32_t dsmem_ld_u32(uint32_t a) {
  uint32_t v;
  asm volatile("ld.shared::cluster.u32 %0, [%1];" : "=r"(v) : "r"(a) : "memory");
  return v;
}

__device__ __forceinline__ int32_t dsmem_ld_s16(uint32_t a) {
  int32_t v;
  asm volatile("ld.shared::cluster.s16 %0, [%1];" : "=r"(v) : "r"(a) : "memory");
  return v;
}

__device__ __forceinline__ uint4 dsmem_ld_v4_u32(uint32_t a) {
  uint4 v;
  asm volatile("ld.shared::cluster.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "r"(a)
               : "memory");
  return v;
}

__device__ __forceinline__ uint2 dsmem_ld_v2_u32(uint32_t a) {
  uint2 v;
  asm volatile("ld.shared::cluster.v2.u32 {%0, %1}, [%2];" : "=r"(v.x), "=r"(v.y) : "r"(a) : "memory");
  return v;
}

__device__ __forceinline__ void dsmem_st_v4_u32(uint32_t a, uint4 v) {
  asm volatile("st.shared::cluster.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(a), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
               : "memory");
}

__device__ __forceinline__ void dsmem_st_v2_u32(uint32_t a, uint2 v) {
  asm volatile("st.shared::cluster.v2.u32 [%0], {%1, %2};" ::"r"(a), "r"(v.x), "r"(v.y) : "memory");
}

__device__ __forceinline__ void dsmem_st_u32(uint32_t a, uint32_t v) {
  asm volatile("st.shared::cluster.u32 [%0], %1;" ::"r"(a), "r"(v) : "memory");
}

}  // namespace rosetta
