// Device helpers shared by the libretrace kernels (sm_103a).
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace retrace {

// ---------------------------------------------------------------------------
// Workspace status word (first 4 bytes of every workspace).
// ---------------------------------------------------------------------------
enum : uint32_t {
  kFlagWaitTimeout = 1u,  // a bounded mbarrier wait in a tensor-core kernel expired
};

// Wall-clock bound of every device-side wait, in nanoseconds.  Kernels finish
// in well under a millisecond; a wait this long means a broken pipeline.
constexpr unsigned long long kWaitLimitNs = 1000ull * 1000ull * 1000ull;

__device__ __forceinline__ unsigned long long global_ns() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// ---------------------------------------------------------------------------
// Scalar conversions
// ---------------------------------------------------------------------------
__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

template <typename T>
__device__ __forceinline__ float to_f32(T x);
template <>
__device__ __forceinline__ float to_f32<float>(float x) { return x; }
template <>
__device__ __forceinline__ float to_f32<__nv_bfloat16>(__nv_bfloat16 x) { return __bfloat162float(x); }

template <typename T>
__device__ __forceinline__ T from_f32(float x);
template <>
__device__ __forceinline__ float from_f32<float>(float x) { return x; }
template <>
__device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float x) { return __float2bfloat16_rn(x); }

// Two fp32 values rounded to nearest-even bf16 and packed low|high.
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// Logistic function from the fast exponential and division intrinsics: their
// relative error (a few fp32 ulp) is far below the bf16 rounding of the
// outputs it feeds.  The argument is clamped to [-80, 80], where the fp32
// logistic is already 0 or 1 to within its rounding.
__device__ __forceinline__ float fast_sigmoid(float x) {
  return __fdividef(1.f, 1.f + __expf(-fminf(fmaxf(x, -80.f), 80.f)));
}

// ---------------------------------------------------------------------------
// Argmax keys.  A 64-bit key orders (value, index) pairs by value, then by
// LOWER index: the high word maps the float to an unsigned integer with the
// same order (sign bit flipped for non-negatives, all bits flipped for
// negatives; -0 is first canonicalised to +0 so the two compare equal), the
// low word is ~index.  max() over keys is then argmax with lowest-index ties,
// and it is associative, so partial results can be combined in any order.
// Key 0 is below every key of a real (non-NaN) value.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t ordered_bits(float f) {
  uint32_t u = __float_as_uint(f);
  if (u == 0x80000000u) u = 0u;  // -0 -> +0
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ unsigned long long make_key(float v, uint32_t idx) {
  return ((unsigned long long)ordered_bits(v) << 32) | (unsigned long long)(0xFFFFFFFFu - idx);
}
__device__ __forceinline__ uint32_t key_index(unsigned long long key) {
  return 0xFFFFFFFFu - (uint32_t)(key & 0xFFFFFFFFull);
}
// The value of a key (the inverse of ordered_bits; -0 comes back as +0).
__device__ __forceinline__ float key_value(unsigned long long key) {
  const uint32_t o = (uint32_t)(key >> 32);
  return __uint_as_float((o & 0x80000000u) ? (o & 0x7FFFFFFFu) : ~o);
}
__device__ __forceinline__ unsigned long long umax64(unsigned long long a, unsigned long long b) {
  return a > b ? a : b;
}
__device__ __forceinline__ unsigned long long warp_max_key(unsigned long long k) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) k = umax64(k, __shfl_xor_sync(0xFFFFFFFFu, k, off));
  return k;
}

// ---------------------------------------------------------------------------
// Block-wide copy of n 16-byte vectors: element i = load(i) goes to store(i, .).
// Each thread keeps kInFlight independent loads in flight before it stores,
// so a copy of a few hundred KB per block is not a chain of memory latencies.
// ---------------------------------------------------------------------------
template <int kInFlight = 8, typename Load, typename Store>
__device__ __forceinline__ void copy_vectors(long long n, Load load, Store store) {
  const long long stride = blockDim.x;
  for (long long i0 = threadIdx.x; i0 < n; i0 += kInFlight * stride) {
    uint4 v[kInFlight];
#pragma unroll
    for (int q = 0; q < kInFlight; ++q) {
      const long long i = i0 + q * stride;
      if (i < n) v[q] = load(i);
    }
#pragma unroll
    for (int q = 0; q < kInFlight; ++q) {
      const long long i = i0 + q * stride;
      if (i < n) store(i, v[q]);
    }
  }
}

// ---------------------------------------------------------------------------
// Programmatic dependent launch: a kernel launched with the programmatic
// stream-serialisation attribute may start once every CTA of the previous
// kernel in the stream has called pdl_launch_dependents (or exited); it must
// call pdl_wait before it reads anything the previous kernel writes, and
// pdl_wait returns once that kernel has completed and its writes are visible.
// Both are no-ops for a kernel launched without the attribute.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void pdl_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// ---------------------------------------------------------------------------
// Shared-memory address helpers
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}

// ---------------------------------------------------------------------------
// Block-wide copy of n 16-byte vectors through shared memory: thread t copies
// vectors t, t + blockDim.x, ... .  kStage of them at a time go from global
// memory into the thread's own slots of `staging` (kStage * blockDim.x
// vectors) with cp.async, which holds no registers while in flight, then from
// the slots to their destination.  No block barrier: each thread reads back
// only the slots it filled.  src(i) and dst(i) give 16-byte aligned addresses.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void cp_async16(uint32_t smem_dst, const void* gsrc) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_dst), "l"(gsrc) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.commit_group;\n\tcp.async.wait_group 0;" ::: "memory");
}
template <int kStage, typename Src, typename Dst>
__device__ __forceinline__ void copy_vectors_staged(long long n, uint4* staging, Src src, Dst dst) {
  const long long stride = blockDim.x;
  for (long long i0 = threadIdx.x; i0 < n; i0 += kStage * stride) {
#pragma unroll
    for (int q = 0; q < kStage; ++q) {
      const long long i = i0 + q * stride;
      if (i < n) cp_async16(smem_u32(staging + q * stride + threadIdx.x), src(i));
    }
    cp_async_wait_all();
#pragma unroll
    for (int q = 0; q < kStage; ++q) {
      const long long i = i0 + q * stride;
      if (i < n) *dst(i) = staging[q * stride + threadIdx.x];
    }
  }
}

// ---------------------------------------------------------------------------
// mbarrier
// ---------------------------------------------------------------------------
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
// Waits for the phase with `parity` to complete.  Gives up (returns false)
// when *abort becomes non-zero or after kWaitLimitNs; never spins forever.
// The clock is read only every 256 polls, so a short wait costs no clock read.
__device__ __forceinline__ bool mbar_wait_bounded(uint32_t bar, uint32_t parity,
                                                  volatile int* abort) {
  unsigned long long t0 = 0ull;
  for (uint32_t it = 1;; ++it) {
    if (mbar_try_wait(bar, parity)) return true;
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

// Spins until ready() holds (true), or until *abort becomes non-zero or about
// kWaitLimitNs have passed (false), sleeping `sleep_ns` between polls; the
// clock is read every 64 polls only.
template <typename Ready>
__device__ __forceinline__ bool spin_until(Ready&& ready, volatile int* abort, unsigned sleep_ns) {
  unsigned long long t0 = 0ull;
  for (uint32_t it = 1;; ++it) {
    if (ready()) return true;
    if (sleep_ns) __nanosleep(sleep_ns);
    if ((it & 63u) == 0u) {
      if (*abort) return false;
      const unsigned long long now = global_ns();
      if (t0 == 0ull)
        t0 = now;
      else if (now - t0 > kWaitLimitNs)
        return false;
    }
  }
}

// ---------------------------------------------------------------------------
// TMA (cp.async.bulk.tensor)
// ---------------------------------------------------------------------------
__device__ __forceinline__ void tma_prefetch_desc(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(map) : "memory");
}
// 2D tiled load of one box at (x = inner coordinate, y = row) into shared memory.
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int x, int y,
                                            uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(map), "r"(x), "r"(y), "r"(bar)
      : "memory");
}
// Gathers four rows (r0..r3) of a 2D tensor, columns [x, x + box width), into
// four consecutive box rows at `dst` (the tensor map's box is one row high).
__device__ __forceinline__ void tma_gather4(uint32_t dst, const CUtensorMap* map, int x, int r0,
                                            int r1, int r2, int r3, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile::gather4.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4, %5, %6}], [%7];" ::"r"(dst),
      "l"(map), "r"(x), "r"(r0), "r"(r1), "r"(r2), "r"(r3), "r"(bar)
      : "memory");
}

// ---------------------------------------------------------------------------
// tcgen05 (5th-generation tensor cores, accumulators in tensor memory)
// ---------------------------------------------------------------------------
__device__ __forceinline__ void tmem_alloc(uint32_t slot_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(slot_smem),
               "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
// D[tmem] (+)= A[smem] * B[smem]^T, bf16 inputs, fp32 accumulation.
__device__ __forceinline__ void tc_mma_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                            uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// Arrive once on `bar` when every tcgen05 operation issued so far by this thread completes.
__device__ __forceinline__ void tc_commit(uint32_t bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
      : "memory");
}
// Each thread of the warp reads 32 consecutive fp32 columns of its TMEM lane.
__device__ __forceinline__ void tmem_ld_32cols(uint32_t taddr, float (&v)[32]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
        "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
        "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr)
      : "memory");
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// Shared-memory matrix descriptor for a K-major bf16 operand tile stored as
// rows of 64 elements (128 bytes) with the 128-byte swizzle, 8-row groups
// 1024 bytes apart (the layout a TMA load with CU_TENSOR_MAP_SWIZZLE_128B and
// a 64-element inner box writes).  Fields: start address >> 4 (bits 0-13),
// leading-dimension byte offset >> 4 (16-29; unused for this layout, set to
// 1), stride-dimension byte offset >> 4 (32-45) = 1024 B between 8-row groups,
// descriptor version 1 (46-47), swizzle mode 2 = 128-byte (61-63).
__device__ __forceinline__ uint64_t sw128_kmajor_desc(uint32_t saddr) {
  uint64_t desc = 0;
  desc |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  desc |= (uint64_t)1 << 16;
  desc |= (uint64_t)(1024u >> 4) << 32;
  desc |= (uint64_t)1 << 46;
  desc |= (uint64_t)2 << 61;
  return desc;
}

// Instruction descriptor of tcgen05.mma kind::f16: fp32 accumulator (bits
// 4-5 = 1), A and B bf16 (bits 7-9 = 1, 10-12 = 1), both K-major (bits 15,
// 16 = 0), N >> 3 in bits 17-22, M >> 4 in bits 24-28.
__host__ __device__ constexpr uint32_t idesc_bf16_f32(int M, int N) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) |
         ((uint32_t)(M >> 4) << 24);
}

}  // namespace retrace
