// Device helpers of the persistent tensor-core conditioning kernels: bounded
// waits on counters and mbarriers, the CTA-pair (cluster of two) primitives of
// tcgen05.mma.cta_group::2, and the broadcast-e gate-bias GEMV that idle warps
// of those kernels run.  Every wait is bounded (kWaitLimitNs) and reports
// expiry through the workspace status word instead of spinning forever.
#pragma once

#include "common.cuh"

namespace retrace {
namespace {

__device__ __forceinline__ void raise_abort(volatile int* s_abort, uint32_t* status) {
  *s_abort = 1;
  atomicOr(status, kFlagWaitTimeout);
}

// Lane 0 waits, the warp agrees on the outcome.  The __syncwarp orders the
// other lanes' later reads after lane 0's acquire: without it the compiler may
// schedule their loads of what the arrive published (a tile index, a row
// count) before lane 0 has seen the phase complete.
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, volatile int* abort) {
  int ok = 1;
  if ((threadIdx.x & 31) == 0) ok = mbar_wait_bounded(bar, parity, abort) ? 1 : 0;
  ok = __shfl_sync(0xFFFFFFFFu, ok, 0);
  __syncwarp();
  return ok != 0;
}

__device__ __forceinline__ uint32_t ld_acquire(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Waits until *counter >= target (written by other CTAs of this grid).
// Bounded like every other wait: false after kWaitLimitNs or on abort.
__device__ __forceinline__ bool wait_counter(const uint32_t* counter, uint32_t target,
                                             volatile int* abort) {
  if (ld_acquire(counter) >= target) return true;
  const unsigned long long t0 = global_ns();
  for (uint32_t it = 1;; ++it) {
    __nanosleep(64);
    if (ld_acquire(counter) >= target) return true;
    if ((it & 63u) == 0u) {
      if (*abort) return false;
      if (global_ns() - t0 > kWaitLimitNs) return false;
    }
  }
}

__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}

// Non-blocking: has the phase with this parity completed?
__device__ __forceinline__ bool mbar_test_parity(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// One warp: rows i of ge = W_g[:, :d] e (broadcast e), claimed from a global
// counter until all d rows are taken; each finished row is counted.  Eight
// 16-byte loads per lane are in flight (d a multiple of 8).  With a stop
// barrier (a shared::cta address, not 0) the warp takes no further row once
// that barrier's phase 0 has completed.
__device__ void gate_bias_rows(const __nv_bfloat16* e, const __nv_bfloat16* Wg, float* ge, int d, int lane,
                               uint32_t* next, uint32_t* done, uint32_t stop_bar = 0u) {
  const int vpr = d / 8;
  const uint4* ev = reinterpret_cast<const uint4*>(e);
  for (;;) {
    int i = 0;
    if (lane == 0) i = (stop_bar != 0u && mbar_test_parity(stop_bar, 0u)) ? d : (int)atomicAdd(next, 1u);
    i = __shfl_sync(0xFFFFFFFFu, i, 0);
    if (i >= d) break;
    const uint4* wr = reinterpret_cast<const uint4*>(Wg + (long long)i * 2 * d);
    float acc = 0.f;
    for (int v0 = 0; v0 < vpr; v0 += 8 * 32) {
      uint4 w[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int v = v0 + u * 32 + lane;
        w[u] = v < vpr ? __ldcs(wr + v) : make_uint4(0u, 0u, 0u, 0u);
      }
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int v = v0 + u * 32 + lane;
        if (v < vpr) {
          const uint4 x = __ldg(ev + v);
          const uint32_t ww[4] = {w[u].x, w[u].y, w[u].z, w[u].w}, xx[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            acc = fmaf(bf16_lo(ww[q]), bf16_lo(xx[q]), acc);
            acc = fmaf(bf16_hi(ww[q]), bf16_hi(xx[q]), acc);
          }
        }
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xFFFFFFFFu, acc, o);
    if (lane == 0) {
      ge[i] = acc;
      __threadfence();
      atomicAdd(done, 1u);
    }
  }
}

__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// The shared::cluster address of `addr` (this CTA's shared memory) in CTA `rank`.
__device__ __forceinline__ uint32_t map_rank(uint32_t addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
  return r;
}
__device__ __forceinline__ void mbar_arrive_remote(uint32_t cluster_addr) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr) : "memory");
}
__device__ __forceinline__ void st_remote_u32(uint32_t cluster_addr, uint32_t v) {
  asm volatile("st.shared::cluster.u32 [%0], %1;" ::"r"(cluster_addr), "r"(v) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait_acq_cluster(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
// mbar_wait_bounded for a barrier that the peer CTA arrives on.
__device__ __forceinline__ bool mbar_wait_cluster_bounded(uint32_t bar, uint32_t parity, volatile int* abort) {
  unsigned long long t0 = 0ull;
  for (uint32_t it = 1;; ++it) {
    if (mbar_try_wait_acq_cluster(bar, parity)) return true;
    if ((it & 255u) == 0u) {
      if (*abort) return false;
      const unsigned long long now = global_ns();
      if (t0 == 0ull)
        t0 = now;
      else if (now - t0 > kWaitLimitNs)
        return false;
    }
  }
}
__device__ __forceinline__ bool warp_wait_cluster(uint32_t bar, uint32_t parity, volatile int* abort) {
  int ok = 1;
  if ((threadIdx.x & 31) == 0) ok = mbar_wait_cluster_bounded(bar, parity, abort) ? 1 : 0;
  ok = __shfl_sync(0xFFFFFFFFu, ok, 0);
  __syncwarp();
  return ok != 0;
}
// The generic address of `p` (this CTA's shared memory) in cluster CTA `rank`:
// plain loads through it read that CTA's shared memory.
template <typename T>
__device__ __forceinline__ const T* map_rank_ptr(const T* p, uint32_t rank) {
  uint64_t r;
  asm volatile("mapa.u64 %0, %1, %2;" : "=l"(r) : "l"(reinterpret_cast<uint64_t>(p)), "r"(rank));
  return reinterpret_cast<const T*>(r);
}
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_alloc_pair(uint32_t slot_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(slot_smem), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish_pair() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tc_mma_pair(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                            uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// Arrive once on the barrier at `bar` in both CTAs of the pair when the MMAs
// issued so far complete.
__device__ __forceinline__ void tc_commit_pair(uint32_t bar) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(bar),
      "h"((uint16_t)0x3)
      : "memory");
}
// A 2D tile load into this CTA's shared memory that completes on a barrier
// of either CTA of the pair (`bar` a shared::cluster address).
__device__ __forceinline__ void tma_load_2d_pair(uint32_t dst, const CUtensorMap* map, int x, int y, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(map), "r"(x), "r"(y), "r"(bar)
      : "memory");
}

}  // namespace
}  // namespace retrace
