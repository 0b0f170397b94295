// Low-rank realisation of the conditioning path (Appendix "Concurrent-Serving
// Experiment": rank-64 rejected-suffix latents, a rank-32 target-aware
// correction, input-side latent residual fusion, one-round lifetime).  Per
// conditioned row, with m = hD[b, A+1+j] and u = hT[b, A+j] (Eq. 4-5):
//
//   z   = P m                                   latent           P  [64, d]
//   rho = z + beta A_c (B_c [z; u])             rank-32 correction B_c [32, 64+d], A_c [64, 32]
//   e~  = e + (W_v rho) * sigmoid(W_g [e; rho]) latent fusion    W_v [d, 64], W_g [d, d+64]
//
// z and rho are rounded to bf16 where they are stored (bf16 workloads); e is
// the broadcast mask embedding, so W_g[:, :d] e is one GEMV per call.
//
// Tensor-core path (bf16, d a multiple of 128), two launches after the GEMV:
//   lr_project_kernel  split-K over the packed [m; u] rows: the m half against
//                      P (N = 64), the u half against B_c's u columns (N = 32);
//                      fp32 partials per split, and the last CTA of each
//                      (row block, warp quarter) sums them in a fixed order and
//                      finishes z, t and rho for its 32 rows on CUDA cores;
//   lr_fuse_kernel     one (128-row, 128-feature) tile per CTA: rho [128, 64]
//                      against [W_v; W_g,rho] [256, 64] in four K16 MMAs, the
//                      gate and residual in the epilogue.
// FFMA path (fp32, other shapes): lr_simt_kernel, one CTA per conditioned row.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "common.cuh"
#include "internal.h"

namespace retrace {
namespace {

constexpr int L = kLowRankLatent, C = kLowRankCorrection;
constexpr int BM = 128, BK = 64;
constexpr int ST = 4;                         // operand stages of the projection
constexpr int A_BYTES = BM * BK * 2;          // 16 KB: 128 packed rows x 64
constexpr int BP_BYTES = L * BK * 2;          // 8 KB: P tile (the 4 KB B_c tile uses the same slot)
constexpr int STAGE_BYTES = A_BYTES + BP_BYTES;
constexpr int SMEM_PROJECT = ST * STAGE_BYTES + 1024;
// 48 KB of operands, padded so that at most two CTAs share an SM: each holds
// 256 TMEM columns, and a third would wait in tcgen05.alloc.
constexpr int SMEM_FUSE = 80 * 1024;
constexpr uint32_t IDESC_P = idesc_bf16_f32(128, L);
constexpr uint32_t IDESC_B = idesc_bf16_f32(128, C);
constexpr uint32_t IDESC_F = idesc_bf16_f32(128, 256);

struct LrParams {
  int d, H;  // H: splits per half of the [m; u] reduction
  const int32_t* R;
  float beta;
  const __nv_bfloat16* Bc;  // [32, 64 + d]
  const __nv_bfloat16* Ac;  // [64, 32]
  float* zpart;             // [H, R_max, 64]
  float* tpart;             // [H, R_max, 32]
  __nv_bfloat16* rho;       // [R_max, 64]
  uint32_t* tickets;        // [4 * row blocks]
  long long rmax;
  uint32_t* status;
};

struct LrFuseParams {
  int d;
  const int32_t* R;
  const int32_t* rowmap;
  const __nv_bfloat16* e;  // [d]
  const float* ge;         // [d]: W_g[:, :d] e
  __nv_bfloat16* e_out;
  uint32_t* status;
};

__device__ __forceinline__ void raise_abort(volatile int* abort, uint32_t* status) {
  *abort = 1;
  atomicOr(status, kFlagWaitTimeout);
}

__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, volatile int* abort) {
  int ok = 1;
  if ((threadIdx.x & 31) == 0) ok = mbar_wait_bounded(bar, parity, abort) ? 1 : 0;
  ok = __shfl_sync(0xFFFFFFFFu, ok, 0);
  __syncwarp();  // the other lanes after lane 0's acquire
  return ok != 0;
}

__device__ __forceinline__ float bf16_round(float x) { return __bfloat162float(__float2bfloat16_rn(x)); }

// z, t and rho of packed row g from the split partials (fixed summation order).
__device__ void finish_row(const LrParams& p, long long g) {
  const int d = p.d;
  float z[L], t[C];
#pragma unroll
  for (int i = 0; i < L; ++i) z[i] = 0.f;
#pragma unroll
  for (int c = 0; c < C; ++c) t[c] = 0.f;
  for (int s = 0; s < p.H; ++s) {
    const float4* zp = reinterpret_cast<const float4*>(p.zpart + ((long long)s * p.rmax + g) * L);
    const float4* tp = reinterpret_cast<const float4*>(p.tpart + ((long long)s * p.rmax + g) * C);
#pragma unroll
    for (int q = 0; q < L / 4; ++q) {
      const float4 v = __ldcg(zp + q);
      z[4 * q] += v.x;
      z[4 * q + 1] += v.y;
      z[4 * q + 2] += v.z;
      z[4 * q + 3] += v.w;
    }
#pragma unroll
    for (int q = 0; q < C / 4; ++q) {
      const float4 v = __ldcg(tp + q);
      t[4 * q] += v.x;
      t[4 * q + 1] += v.y;
      t[4 * q + 2] += v.z;
      t[4 * q + 3] += v.w;
    }
  }
#pragma unroll
  for (int i = 0; i < L; ++i) z[i] = bf16_round(z[i]);  // the stored latent
  // t += B_c[:, :64] z   (the u part is already in t)
#pragma unroll
  for (int c = 0; c < C; ++c) {
    const __nv_bfloat16* brow = p.Bc + (long long)c * (L + d);
    float s = t[c];
#pragma unroll
    for (int i = 0; i < L; ++i) s = fmaf(__bfloat162float(brow[i]), z[i], s);
    t[c] = s;
  }
  // rho = z + beta A_c t, rounded; 64 bf16 = 128 bytes
  uint4* out = reinterpret_cast<uint4*>(p.rho + g * L);
#pragma unroll
  for (int q = 0; q < L / 8; ++q) {
    uint32_t w[4];
#pragma unroll
    for (int h = 0; h < 4; ++h) {
      float r2[2];
#pragma unroll
      for (int k = 0; k < 2; ++k) {
        const int i = 8 * q + 2 * h + k;
        const __nv_bfloat16* arow = p.Ac + i * C;
        float s = 0.f;
#pragma unroll
        for (int c = 0; c < C; ++c) s = fmaf(__bfloat162float(arow[c]), t[c], s);
        r2[k] = z[i] + p.beta * s;
      }
      w[h] = pack_bf16x2(r2[0], r2[1]);
    }
    out[q] = make_uint4(w[0], w[1], w[2], w[3]);
  }
}

// grid (row blocks, 2H): blockIdx.y < H reduces over the m half against P,
// the rest over the u half against B_c[:, 64:].
__global__ void __launch_bounds__(256, 1)
    lr_project_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmP,
                      const __grid_constant__ CUtensorMap tmBc, const LrParams p) {
  extern __shared__ uint8_t dsmem[];
  __shared__ __align__(8) uint64_t bar_full[ST];
  __shared__ __align__(8) uint64_t bar_empty[ST];
  __shared__ __align__(8) uint64_t bar_acc;
  __shared__ uint32_t s_tmem;
  __shared__ volatile int s_abort;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int R = *(volatile const int32_t*)p.R;
  const int m0 = blockIdx.x * BM;
  if (m0 >= R) return;
  const int d = p.d;
  const int half = (int)blockIdx.y / p.H, part = (int)blockIdx.y % p.H;
  const int KB = d / BK;  // k-blocks per half
  const int kb0 = part * KB / p.H, kb1 = (part + 1) * KB / p.H;
  const int nkb = kb1 - kb0;
  const int N = half == 0 ? L : C;

  if (threadIdx.x == 0) {
    s_abort = 0;
    for (int s = 0; s < ST; ++s) {
      mbar_init(smem_u32(&bar_full[s]), 1);
      mbar_init(smem_u32(&bar_empty[s]), 1);
    }
    mbar_init(smem_u32(&bar_acc), 1);
    fence_mbar_init();
  }
  if (warp == 2) {
    tmem_alloc(smem_u32(&s_tmem), 64);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s_tmem;
  const uint32_t base = (smem_u32(dsmem) + 1023u) & ~1023u;

  if (warp == 0) {
    if (lane == 0) {
      bool ok = true;
      int i = 0;
      for (; i < nkb; ++i) {
        const uint32_t s = i % ST, ph = (i / ST) & 1u;
        if (!mbar_wait_bounded(smem_u32(&bar_empty[s]), ph ^ 1u, &s_abort)) {
          ok = false;
          break;
        }
        const uint32_t a_dst = base + s * STAGE_BYTES, b_dst = a_dst + A_BYTES;
        const int kb = kb0 + i;
        mbar_arrive_expect_tx(smem_u32(&bar_full[s]), A_BYTES + N * BK * 2);
        tma_load_2d(a_dst, &tmA, half * d + kb * BK, m0, smem_u32(&bar_full[s]));
        if (half == 0)
          tma_load_2d(b_dst, &tmP, kb * BK, 0, smem_u32(&bar_full[s]));
        else
          tma_load_2d(b_dst, &tmBc, L + kb * BK, 0, smem_u32(&bar_full[s]));
      }
      if (!ok) {
        raise_abort(&s_abort, p.status);
        volatile int never = 0;  // drain this CTA's own copies in flight
        for (int k = i > ST ? i - ST : 0; k < i; ++k)
          mbar_wait_bounded(smem_u32(&bar_full[k % ST]), (k / ST) & 1u, &never);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      bool ok = true;
      for (int i = 0; i < nkb; ++i) {
        const uint32_t s = i % ST, ph = (i / ST) & 1u;
        if (!mbar_wait_bounded(smem_u32(&bar_full[s]), ph, &s_abort)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t a_base = base + s * STAGE_BYTES, b_base = a_base + A_BYTES;
#pragma unroll
        for (int k = 0; k < BK / 16; ++k) {
          const uint64_t adesc = sw128_kmajor_desc(a_base + (uint32_t)k * 32u);
          const uint64_t bdesc = sw128_kmajor_desc(b_base + (uint32_t)k * 32u);
          tc_mma_bf16(tmem, adesc, bdesc, half == 0 ? IDESC_P : IDESC_B, (i > 0 || k > 0) ? 1u : 0u);
        }
        tc_commit(smem_u32(&bar_empty[s]));
      }
      tc_commit(smem_u32(&bar_acc));  // also when nothing was issued, or after a failure
      if (!ok) raise_abort(&s_abort, p.status);
    }
    __syncwarp();
  } else if (warp >= 4) {
    const int q = (warp - 4) * 32 + lane;
    const long long g = m0 + q;
    const uint32_t taddr = tmem + ((uint32_t)((warp & 3) * 32) << 16);
    bool ok = warp_wait(smem_u32(&bar_acc), 0, &s_abort);
    tc_fence_after();
    if (ok && !s_abort) {
      float* dst = half == 0 ? p.zpart + ((long long)part * p.rmax + g) * L : p.tpart + ((long long)part * p.rmax + g) * C;
      for (int cc = 0; cc < N / 32; ++cc) {
        float v[32];
        tmem_ld_32cols(taddr + (uint32_t)(cc * 32), v);
        if (g < R) {
          float4* o = reinterpret_cast<float4*>(dst + cc * 32);
#pragma unroll
          for (int x = 0; x < 8; ++x)
            o[x] = nkb > 0 ? make_float4(v[4 * x], v[4 * x + 1], v[4 * x + 2], v[4 * x + 3]) : make_float4(0.f, 0.f, 0.f, 0.f);
        }
      }
      // The last of the 2H split CTAs to finish this warp's 32 rows finishes them.
      __threadfence();
      __syncwarp();
      int last = 0;
      if (lane == 0) {
        uint32_t* tk = p.tickets + (long long)blockIdx.x * 4 + (warp - 4);
        last = atomicAdd(tk, 1u) == (uint32_t)(2 * p.H - 1) ? 1 : 0;
        if (last) *tk = 0u;  // ready for the next call
      }
      last = __shfl_sync(0xFFFFFFFFu, last, 0);
      if (last) {
        __threadfence();
        if (g < R) finish_row(p, g);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, 64);
  }
}

// grid (row blocks, d / 128): rows [m0, m0+128) x features [n0, n0+128).
__global__ void __launch_bounds__(256, 1)
    lr_fuse_kernel(const __grid_constant__ CUtensorMap tmRho, const __grid_constant__ CUtensorMap tmWv,
                   const __grid_constant__ CUtensorMap tmWg, const LrFuseParams p) {
  extern __shared__ uint8_t dsmem[];
  __shared__ __align__(8) uint64_t bar_full;
  __shared__ __align__(8) uint64_t bar_acc;
  __shared__ uint32_t s_tmem;
  __shared__ volatile int s_abort;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int R = *(volatile const int32_t*)p.R;
  const int m0 = blockIdx.x * BM, n0 = blockIdx.y * 128;
  if (m0 >= R) return;
  const int d = p.d;
  if (threadIdx.x == 0) {
    s_abort = 0;
    mbar_init(smem_u32(&bar_full), 1);
    mbar_init(smem_u32(&bar_acc), 1);
    fence_mbar_init();
  }
  if (warp == 2) {
    tmem_alloc(smem_u32(&s_tmem), 256);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s_tmem;
  const uint32_t a_base = (smem_u32(dsmem) + 1023u) & ~1023u;
  const uint32_t b_base = a_base + BM * BK * 2;

  if (warp == 0) {
    if (lane == 0) {
      // rho rows, then the B tile: 128 rows of W_v over the matching 128 rows
      // of W_g[:, d:d+64], so v and the gate pre-activation share a TMEM lane
      mbar_arrive_expect_tx(smem_u32(&bar_full), BM * BK * 2 + 256 * BK * 2);
      tma_load_2d(a_base, &tmRho, 0, m0, smem_u32(&bar_full));
      tma_load_2d(b_base, &tmWv, 0, n0, smem_u32(&bar_full));
      tma_load_2d(b_base + 128 * BK * 2, &tmWg, d, n0, smem_u32(&bar_full));
      const bool ok = mbar_wait_bounded(smem_u32(&bar_full), 0, &s_abort);
      if (ok) {
        tc_fence_after();
#pragma unroll
        for (int k = 0; k < BK / 16; ++k)
          tc_mma_bf16(tmem, sw128_kmajor_desc(a_base + (uint32_t)k * 32u),
                      sw128_kmajor_desc(b_base + (uint32_t)k * 32u), IDESC_F, k > 0 ? 1u : 0u);
      } else {
        raise_abort(&s_abort, p.status);
      }
      tc_commit(smem_u32(&bar_acc));
    }
    __syncwarp();
  } else if (warp >= 4) {
    const int q = (warp - 4) * 32 + lane;
    const int g = m0 + q;
    const uint32_t taddr = tmem + ((uint32_t)((warp & 3) * 32) << 16);
    const bool ok = warp_wait(smem_u32(&bar_acc), 0, &s_abort);
    tc_fence_after();
    if (ok && !s_abort) {
      const long long orow = g < R ? __ldg(p.rowmap + g) : 0;
      for (int cc = 0; cc < 4; ++cc) {
        float v[32], gt[32];
        tmem_ld_32cols(taddr + (uint32_t)(cc * 32), v);
        tmem_ld_32cols(taddr + 128u + (uint32_t)(cc * 32), gt);
        if (g < R) {
          const int n = n0 + cc * 32;
          const uint4* ev = reinterpret_cast<const uint4*>(p.e + n);
          uint4* ov = reinterpret_cast<uint4*>(p.e_out + orow * d + n);
#pragma unroll
          for (int x = 0; x < 4; ++x) {
            const uint4 ew = __ldg(ev + x);
            const uint32_t ewords[4] = {ew.x, ew.y, ew.z, ew.w};
            uint32_t o[4];
#pragma unroll
            for (int w = 0; w < 4; ++w) {
              const int c0 = x * 8 + 2 * w;
              const float g0 = gt[c0] + __ldg(p.ge + n + c0), g1 = gt[c0 + 1] + __ldg(p.ge + n + c0 + 1);
              const float s0 = 1.f / (1.f + expf(-g0)), s1 = 1.f / (1.f + expf(-g1));
              o[w] = pack_bf16x2(bf16_lo(ewords[w]) + v[c0] * s0, bf16_hi(ewords[w]) + v[c0 + 1] * s1);
            }
            ov[x] = make_uint4(o[0], o[1], o[2], o[3]);
          }
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, 256);
  }
}

// W_g[:, :d] e with W_g's rows `stride` elements apart: one warp per output.
template <typename T>
__global__ void __launch_bounds__(256) lr_gemv_kernel(const T* __restrict__ Wg, long long stride,
                                                      const T* __restrict__ e, int d, float* __restrict__ ge) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int i = blockIdx.x * 8 + warp;
  if (i >= d) return;
  const T* w = Wg + (long long)i * stride;
  float s = 0.f;
  constexpr int E = 16 / (int)sizeof(T);
  const bool vec = (d % E == 0) && ((uintptr_t)w % 16 == 0) && ((uintptr_t)e % 16 == 0);
  if (vec) {
    const uint4* wv = reinterpret_cast<const uint4*>(w);
    const uint4* evv = reinterpret_cast<const uint4*>(e);
    for (int k = lane; k < d / E; k += 32) {
      const uint4 a = __ldg(wv + k), b = __ldg(evv + k);
      const T* ta = reinterpret_cast<const T*>(&a);
      const T* tb = reinterpret_cast<const T*>(&b);
#pragma unroll
      for (int x = 0; x < E; ++x) s = fmaf(to_f32(ta[x]), to_f32(tb[x]), s);
    }
  } else {
    for (int k = lane; k < d; k += 32) s = fmaf(to_f32(w[k]), to_f32(e[k]), s);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xFFFFFFFFu, s, off);
  if (lane == 0) ge[i] = s;
}

// FFMA path: one CTA of 256 threads per position (b, j < K-1); rows j >= n_b
// return at once (verification already wrote e there).
template <typename T>
__global__ void __launch_bounds__(256) lr_simt_kernel(const LowRankArgs a) {
  __shared__ float s_z[L], s_t[C], s_rho[L];
  const int K = a.K, d = a.d;
  const int b = (int)(blockIdx.x / (unsigned)(K - 1)), j = (int)(blockIdx.x % (unsigned)(K - 1));
  int A = a.accept_len[b];
  A = A < 0 ? 0 : (A > K ? K : A);
  const int nb = K - 1 - A > 0 ? K - 1 - A : 0;
  if (j >= nb) return;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const bool rnd = sizeof(T) == 2;
  const T* m = reinterpret_cast<const T*>(a.hD) + ((long long)b * K + A + 1 + j) * d;
  const T* u = reinterpret_cast<const T*>(a.hT) + ((long long)b * K + A + j) * d;
  const T* P = reinterpret_cast<const T*>(a.P);
  const T* Bc = reinterpret_cast<const T*>(a.Bc);
  const T* Ac = reinterpret_cast<const T*>(a.Ac);
  const T* Wv = reinterpret_cast<const T*>(a.Wv);
  const T* Wg = reinterpret_cast<const T*>(a.Wg);
  const T* e = reinterpret_cast<const T*>(a.e);
  for (int i = warp; i < L; i += 8) {  // z = P m
    float s = 0.f;
    for (int k = lane; k < d; k += 32) s = fmaf(to_f32(P[(long long)i * d + k]), to_f32(m[k]), s);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xFFFFFFFFu, s, off);
    if (lane == 0) s_z[i] = rnd ? bf16_round(s) : s;
  }
  __syncthreads();
  for (int c = warp; c < C; c += 8) {  // t = B_c [z; u]
    const T* brow = Bc + (long long)c * (L + d);
    float s = 0.f;
    for (int k = lane; k < L + d; k += 32) s = fmaf(to_f32(brow[k]), k < L ? s_z[k] : to_f32(u[k - L]), s);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xFFFFFFFFu, s, off);
    if (lane == 0) s_t[c] = s;
  }
  __syncthreads();
  if (threadIdx.x < L) {  // rho = z + beta A_c t
    float s = 0.f;
    for (int c = 0; c < C; ++c) s = fmaf(to_f32(Ac[threadIdx.x * C + c]), s_t[c], s);
    const float r = s_z[threadIdx.x] + a.beta * s;
    s_rho[threadIdx.x] = rnd ? bf16_round(r) : r;
  }
  __syncthreads();
  T* out = reinterpret_cast<T*>(a.e_out) + ((long long)b * K + j) * d;
  for (int f = threadIdx.x; f < d; f += 256) {
    const T* vrow = Wv + (long long)f * L;
    const T* grow = Wg + (long long)f * (d + L) + d;
    float v = 0.f, gg = a.ge[f];
#pragma unroll 8
    for (int i = 0; i < L; ++i) {
      v = fmaf(to_f32(vrow[i]), s_rho[i], v);
      gg = fmaf(to_f32(grow[i]), s_rho[i], gg);
    }
    out[f] = from_f32<T>(to_f32(e[f]) + v * (1.f / (1.f + expf(-gg))));
  }
}

}  // namespace

bool lowrank_tc_supported(retrace_dtype dtype, int d) { return dtype == RETRACE_BF16 && d % 128 == 0; }

cudaError_t launch_lowrank(const LowRankArgs& a, bool tc, cudaStream_t stream) {
  const long long rmax = (long long)a.B * (a.K > 1 ? a.K - 1 : 0);
  if (rmax <= 0) return cudaSuccess;
  const unsigned gemv_grid = (unsigned)((a.d + 7) / 8);
  if (a.dtype == RETRACE_BF16)
    lr_gemv_kernel<__nv_bfloat16><<<gemv_grid, 256, 0, stream>>>(
        reinterpret_cast<const __nv_bfloat16*>(a.Wg), (long long)a.d + L,
        reinterpret_cast<const __nv_bfloat16*>(a.e), a.d, a.ge);
  else
    lr_gemv_kernel<float><<<gemv_grid, 256, 0, stream>>>(reinterpret_cast<const float*>(a.Wg), (long long)a.d + L,
                                                         reinterpret_cast<const float*>(a.e), a.d, a.ge);
  cudaError_t err = cudaGetLastError();
  if (err != cudaSuccess) return err;
  if (!tc) {
    if (a.dtype == RETRACE_BF16)
      lr_simt_kernel<__nv_bfloat16><<<(unsigned)rmax, 256, 0, stream>>>(a);
    else
      lr_simt_kernel<float><<<(unsigned)rmax, 256, 0, stream>>>(a);
    return cudaGetLastError();
  }
  static bool attr_done[64] = {false};
  int dev = 0;
  if ((err = cudaGetDevice(&dev)) != cudaSuccess) return err;
  if (!attr_done[dev & 63]) {
    if ((err = cudaFuncSetAttribute(lr_project_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_PROJECT)) !=
        cudaSuccess)
      return err;
    if ((err = cudaFuncSetAttribute(lr_fuse_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_FUSE)) !=
        cudaSuccess)
      return err;
    attr_done[dev & 63] = true;
  }
  const uint64_t d = (uint64_t)a.d;
  CUtensorMap mA, mP, mBc, mRho, mWv, mWg;
  if (encode_tensor_map_2d(&mA, a.apack, 2 * d, (uint64_t)rmax, 4 * d, BK, BM) != CUDA_SUCCESS ||
      encode_tensor_map_2d(&mP, a.P, d, L, 2 * d, BK, L) != CUDA_SUCCESS ||
      encode_tensor_map_2d(&mBc, a.Bc, L + d, C, 2 * (L + d), BK, C) != CUDA_SUCCESS ||
      encode_tensor_map_2d(&mRho, a.rho, L, (uint64_t)rmax, 2 * L, BK, BM) != CUDA_SUCCESS ||
      encode_tensor_map_2d(&mWv, a.Wv, L, d, 2 * L, BK, 128) != CUDA_SUCCESS ||
      encode_tensor_map_2d(&mWg, a.Wg, d + L, d, 2 * (d + L), BK, 128) != CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  const unsigned mt = (unsigned)((rmax + BM - 1) / BM);
  LrParams p{};
  p.d = a.d;
  p.H = kLowRankSplits;
  p.R = a.R;
  p.beta = a.beta;
  p.Bc = reinterpret_cast<const __nv_bfloat16*>(a.Bc);
  p.Ac = reinterpret_cast<const __nv_bfloat16*>(a.Ac);
  p.zpart = a.zpart;
  p.tpart = a.tpart;
  p.rho = reinterpret_cast<__nv_bfloat16*>(a.rho);
  p.tickets = a.tickets;
  p.rmax = rmax;
  p.status = a.status;
  lr_project_kernel<<<dim3(mt, 2 * kLowRankSplits), 256, SMEM_PROJECT, stream>>>(mA, mP, mBc, p);
  if ((err = cudaGetLastError()) != cudaSuccess) return err;
  LrFuseParams f{};
  f.d = a.d;
  f.R = a.R;
  f.rowmap = a.rowmap;
  f.e = reinterpret_cast<const __nv_bfloat16*>(a.e);
  f.ge = a.ge;
  f.e_out = reinterpret_cast<__nv_bfloat16*>(a.e_out);
  f.status = a.status;
  lr_fuse_kernel<<<dim3(mt, (unsigned)(a.d / 128)), 256, SMEM_FUSE, stream>>>(mRho, mWv, mWg, f);
  return cudaGetLastError();
}

}  // namespace retrace
