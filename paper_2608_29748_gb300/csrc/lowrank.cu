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
// Tensor-core path (bf16, d a multiple of 128), three launches:
//   lr_project_kernel  split-K over the packed [m; u] rows: the m half against
//                      P (N = 64), the u half against B_c's u columns (N = 32),
//                      fp32 partials per split;
//   lr_finish_kernel   one warp per row: sums the partials in a fixed order
//                      (bitwise repeatable), rounds z, adds B_c[:, :64] z and
//                      forms rho (lanes over the latent and correction ranks);
//                      then every warp takes rows of the GEMV W_g[:, :d] e from
//                      a counter (the grid has at least two CTAs per SM);
//   lr_fuse_kernel     persistent over (128-row, 64-feature) tiles, two CTAs
//                      per SM: rho [128, 64] against [W_v; W_g,rho] [128, 64]
//                      in four K16 MMAs into one of two TMEM accumulators, the
//                      gate and residual in an eight-warp epilogue (with K = 64
//                      the epilogue, not the MMA, is the long pole).
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
constexpr int kFuseThreads = 384;  // warps 0-3: TMA, MMA, TMEM; warps 4-11: epilogue
constexpr int kFuseFeat = 64;      // features per fusion tile
// Two stages of (rho tile 16 KB + B tile 16 KB), padded so that exactly two
// CTAs share an SM: each holds 256 TMEM columns (two 128-column accumulators),
// and a third CTA would only wait in tcgen05.alloc.
constexpr int SMEM_FUSE = 80 * 1024;
static_assert(SMEM_FUSE >= 2 * (BM * BK * 2 + 2 * kFuseFeat * BK * 2) + 1024, "fusion operands do not fit");
static_assert(3 * SMEM_FUSE > 228 * 1024, "a third fusion CTA must not fit on an SM");
constexpr uint32_t IDESC_P = idesc_bf16_f32(128, L);
constexpr uint32_t IDESC_B = idesc_bf16_f32(128, C);
constexpr uint32_t IDESC_F = idesc_bf16_f32(128, 128);

constexpr int H = kLowRankSplits;  // split-K parts per half of the [m; u] reduction

struct LrParams {
  int d;
  const int32_t* R;
  float beta;
  const __nv_bfloat16* Bc;  // [32, 64 + d]
  const __nv_bfloat16* Ac;  // [64, 32]
  float* zpart;             // [H, R_max, 64]
  float* tpart;             // [H, R_max, 32]
  __nv_bfloat16* rho;       // [R_max, 64]
  long long rmax;
  // W_g[:, :d] e in the projection's idle warps
  const __nv_bfloat16* Wg;  // [d, d + 64]
  const __nv_bfloat16* e;   // [d]
  float* ge;                // [d]
  uint32_t* gemv_next;      // row counter, zero before the launch
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
  pdl_launch_dependents();
  pdl_wait();  // the packed rows and R come from verification
  const int R = *(volatile const int32_t*)p.R;
  const int m0 = blockIdx.x * BM;
  if (m0 >= R) return;
  const int d = p.d;
  const int half = (int)blockIdx.y / H, part = (int)blockIdx.y % H;
  const int KB = d / BK;  // k-blocks per half
  const int kb0 = part * KB / H, kb1 = (part + 1) * KB / H;
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
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, 64);
  }
}

// One warp per packed row g: z = sum of the split partials (fixed order),
// rounded; t = the u partials + B_c[:, :64] z; rho = z + beta A_c t, rounded.
// B_c[:, :64] and A_c are staged as fp32, transposed so lanes read
// consecutive words.  Called by whole CTAs (it synchronises them).
__device__ __forceinline__ void finish_rows(const LrParams& p, long long g, int R, int d, int lane) {
  __shared__ float s_bct[L * C];  // B_c[c][i] at [i][c]
  __shared__ float s_act[C * L];  // A_c[i][c] at [c][i]
  for (int k = threadIdx.x; k < C * L; k += 256) {  // consecutive threads write consecutive words
    const int i = k / C, c = k % C;
    s_bct[k] = __bfloat162float(p.Bc[(long long)c * (L + d) + i]);
    const int c2 = k / L, i2 = k % L;
    s_act[k] = __bfloat162float(p.Ac[i2 * C + c2]);
  }
  __syncthreads();
  if (g >= R) return;
  float zs[H][2], ts[H];
#pragma unroll
  for (int s2 = 0; s2 < H; ++s2) {  // every load in flight at once
    const float* zp = p.zpart + ((long long)s2 * p.rmax + g) * L;
    zs[s2][0] = __ldcg(zp + lane);
    zs[s2][1] = __ldcg(zp + 32 + lane);
    ts[s2] = __ldcg(p.tpart + ((long long)s2 * p.rmax + g) * C + lane);
  }
  float z0 = 0.f, z1 = 0.f, t = 0.f;
#pragma unroll
  for (int s2 = 0; s2 < H; ++s2) {  // fixed order over the splits
    z0 += zs[s2][0];
    z1 += zs[s2][1];
    t += ts[s2];
  }
  z0 = bf16_round(z0);  // the stored latent
  z1 = bf16_round(z1);
  const unsigned FULL = 0xFFFFFFFFu;
#pragma unroll
  for (int i = 0; i < 32; ++i) t = fmaf(s_bct[i * C + lane], __shfl_sync(FULL, z0, i), t);
#pragma unroll
  for (int i = 0; i < 32; ++i) t = fmaf(s_bct[(32 + i) * C + lane], __shfl_sync(FULL, z1, i), t);
  float r0 = 0.f, r1 = 0.f;
#pragma unroll
  for (int c = 0; c < C; ++c) {
    const float tc = __shfl_sync(FULL, t, c);
    r0 = fmaf(s_act[c * L + lane], tc, r0);
    r1 = fmaf(s_act[c * L + 32 + lane], tc, r1);
  }
  p.rho[g * L + lane] = __float2bfloat16_rn(z0 + p.beta * r0);
  p.rho[g * L + 32 + lane] = __float2bfloat16_rn(z1 + p.beta * r1);
}

// W_g[:, :d] e, one row of W_g per claim from the counter; eight 16-byte loads
// in flight per lane (d a multiple of 8).
__device__ __forceinline__ void lr_gemv_rows(const LrParams& p, int d, int lane) {
  const uint4* ev = reinterpret_cast<const uint4*>(p.e);
  const int nv = d / 8;
  for (;;) {
    uint32_t i = 0;
    if (lane == 0) i = atomicAdd(p.gemv_next, 1u);
    i = __shfl_sync(0xFFFFFFFFu, i, 0);
    if (i >= (uint32_t)d) return;
    const uint4* wv = reinterpret_cast<const uint4*>(p.Wg + (long long)i * (d + L));
    float acc = 0.f;
    for (int k0 = 0; k0 < nv; k0 += 8 * 32) {
      uint4 a[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int k = k0 + u * 32 + lane;
        a[u] = k < nv ? __ldg(wv + k) : make_uint4(0u, 0u, 0u, 0u);
      }
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int k = k0 + u * 32 + lane;
        if (k < nv) {
          const uint4 b = __ldg(ev + k);
          const uint32_t aw[4] = {a[u].x, a[u].y, a[u].z, a[u].w}, bw[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
          for (int x = 0; x < 4; ++x) {
            acc = fmaf(bf16_lo(aw[x]), bf16_lo(bw[x]), acc);
            acc = fmaf(bf16_hi(aw[x]), bf16_hi(bw[x]), acc);
          }
        }
      }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) acc += __shfl_xor_sync(0xFFFFFFFFu, acc, off);
    if (lane == 0) p.ge[i] = acc;
  }
}

// grid >= ceil(R_max / 8) and >= two CTAs per SM.  The GEMV reads only the
// inputs, so it runs first, while the projection may still be running
// (programmatic dependent launch); the rows wait for the projection's partials.
__global__ void __launch_bounds__(256) lr_finish_kernel(const LrParams p) {
  pdl_launch_dependents();
  const long long g = (long long)blockIdx.x * 8 + (threadIdx.x >> 5);
  const int d = p.d, lane = threadIdx.x & 31;
  lr_gemv_rows(p, d, lane);
  pdl_wait();
  const int R = *(volatile const int32_t*)p.R;
  if ((long long)blockIdx.x * 8 < R) finish_rows(p, g, R, d, lane);  // uniform over the CTA
}

// Persistent: CTA c takes tiles c, c + G, ... of the (row block, 64-feature
// block) grid, feature blocks fastest.  Two operand stages (rho tile + B tile)
// and two TMEM accumulators, so a tile's loads and MMAs overlap the previous
// tile's epilogue; two CTAs per SM interleave their epilogues.
__global__ void __launch_bounds__(kFuseThreads, 2)
    lr_fuse_kernel(const __grid_constant__ CUtensorMap tmRho, const __grid_constant__ CUtensorMap tmWv,
                   const __grid_constant__ CUtensorMap tmWg, const LrFuseParams p) {
  extern __shared__ uint8_t dsmem[];
  __shared__ __align__(8) uint64_t bar_full[2];
  __shared__ __align__(8) uint64_t bar_empty[2];
  __shared__ __align__(8) uint64_t bar_acc[2];
  __shared__ __align__(8) uint64_t bar_free[2];
  __shared__ uint32_t s_tmem;
  __shared__ volatile int s_abort;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  pdl_launch_dependents();
  pdl_wait();  // rho and W_g[:, :d] e come from the finishing kernel
  const int R = *(volatile const int32_t*)p.R;
  const int d = p.d;
  const int nb = d / kFuseFeat;
  const int tiles = (R + BM - 1) / BM * nb;
  if ((int)blockIdx.x >= tiles) return;
  const int my_tiles = (tiles - (int)blockIdx.x + (int)gridDim.x - 1) / (int)gridDim.x;
  if (threadIdx.x == 0) {
    s_abort = 0;
    for (int b = 0; b < 2; ++b) {
      mbar_init(smem_u32(&bar_full[b]), 1);
      mbar_init(smem_u32(&bar_empty[b]), 1);
      mbar_init(smem_u32(&bar_acc[b]), 1);
      mbar_init(smem_u32(&bar_free[b]), 8);  // one arrival per epilogue warp
    }
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
  const uint32_t base = (smem_u32(dsmem) + 1023u) & ~1023u;
  constexpr uint32_t A_TILE = BM * BK * 2, B_TILE = 2 * kFuseFeat * BK * 2, STAGE = A_TILE + B_TILE;

  if (warp == 0) {
    // ---- TMA: the rho tile and the B tile of each of this CTA's tiles ----
    if (lane == 0) {
      bool ok = true;
      int k = 0;
      for (; k < my_tiles; ++k) {
        const int t = (int)blockIdx.x + k * (int)gridDim.x;
        const int m0 = t / nb * BM, n0 = t % nb * kFuseFeat;
        const uint32_t b = k & 1, ph = (k >> 1) & 1u;
        if (!mbar_wait_bounded(smem_u32(&bar_empty[b]), ph ^ 1u, &s_abort)) {
          ok = false;
          break;
        }
        const uint32_t a_dst = base + b * STAGE, b_dst = a_dst + A_TILE;
        // 64 rows of W_v over the matching 64 rows of W_g[:, d:d+64]: v and
        // the gate pre-activation of a feature share a TMEM lane
        mbar_arrive_expect_tx(smem_u32(&bar_full[b]), STAGE);
        tma_load_2d(a_dst, &tmRho, 0, m0, smem_u32(&bar_full[b]));
        tma_load_2d(b_dst, &tmWv, 0, n0, smem_u32(&bar_full[b]));
        tma_load_2d(b_dst + kFuseFeat * BK * 2, &tmWg, d, n0, smem_u32(&bar_full[b]));
      }
      if (!ok) {
        raise_abort(&s_abort, p.status);
        volatile int never = 0;  // drain this CTA's own copies in flight
        for (int j = k > 2 ? k - 2 : 0; j < k; ++j) mbar_wait_bounded(smem_u32(&bar_full[j & 1]), (j >> 1) & 1u, &never);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---- MMA: tile k into accumulator k % 2 ----
    if (lane == 0) {
      bool ok = true;
      for (int k = 0; k < my_tiles; ++k) {
        const uint32_t b = k & 1, ph = (k >> 1) & 1u;
        if (!mbar_wait_bounded(smem_u32(&bar_free[b]), ph ^ 1u, &s_abort) ||
            !mbar_wait_bounded(smem_u32(&bar_full[b]), ph, &s_abort)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t a_src = base + b * STAGE, b_src = a_src + A_TILE;
#pragma unroll
        for (int kk = 0; kk < BK / 16; ++kk)
          tc_mma_bf16(tmem + b * 128u, sw128_kmajor_desc(a_src + (uint32_t)kk * 32u),
                      sw128_kmajor_desc(b_src + (uint32_t)kk * 32u), IDESC_F, kk > 0 ? 1u : 0u);
        tc_commit(smem_u32(&bar_empty[b]));  // operand stage free once these MMAs complete
        tc_commit(smem_u32(&bar_acc[b]));
      }
      if (!ok) {
        raise_abort(&s_abort, p.status);
        for (int b = 0; b < 2; ++b) tc_commit(smem_u32(&bar_acc[b]));  // release a waiting epilogue
      }
    }
    __syncwarp();
  } else if (warp >= 4) {
    // ---- epilogue: e~ = e + v * sigmoid(ge + g); warp w: rows 32 (w % 4) + lane
    // (a warp reaches TMEM lanes 32 (w % 4) .. +31 only), features
    // 32 ((w - 4) / 4) .. +31 of the tile ----
    const int fh = (warp - 4) >> 2;
    for (int k = 0; k < my_tiles; ++k) {
      const int t = (int)blockIdx.x + k * (int)gridDim.x;
      const int m0 = t / nb * BM, n = t % nb * kFuseFeat + fh * 32;
      const int g = m0 + (warp & 3) * 32 + lane;
      const uint32_t b = k & 1, ph = (k >> 1) & 1u;
      const bool ok = warp_wait(smem_u32(&bar_acc[b]), ph, &s_abort);
      tc_fence_after();
      if (!ok || s_abort) {
        if (!ok && lane == 0) raise_abort(&s_abort, p.status);
        break;
      }
      const long long orow = g < R ? __ldg(p.rowmap + g) : 0;
      const uint32_t taddr = tmem + b * 128u + ((uint32_t)((warp & 3) * 32) << 16);
      float v[32], gt[32];
      tmem_ld_32cols(taddr + (uint32_t)(fh * 32), v);
      tmem_ld_32cols(taddr + (uint32_t)(kFuseFeat + fh * 32), gt);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&bar_free[b]));  // accumulator read: the next tile may use it
      if (g < R) {
        const uint4* ev = reinterpret_cast<const uint4*>(p.e + n);
        const float4* gv = reinterpret_cast<const float4*>(p.ge + n);
        uint4* ov = reinterpret_cast<uint4*>(p.e_out + orow * d + n);
#pragma unroll
        for (int x = 0; x < 4; ++x) {
          const uint4 ew = __ldg(ev + x);
          const float4 ga = __ldg(gv + 2 * x), gb = __ldg(gv + 2 * x + 1);
          const float gw[8] = {ga.x, ga.y, ga.z, ga.w, gb.x, gb.y, gb.z, gb.w};
          const uint32_t ewords[4] = {ew.x, ew.y, ew.z, ew.w};
          uint32_t o[4];
#pragma unroll
          for (int w = 0; w < 4; ++w) {
            const int c0 = x * 8 + 2 * w;
            const float s0 = fast_sigmoid(gt[c0] + gw[2 * w]), s1 = fast_sigmoid(gt[c0 + 1] + gw[2 * w + 1]);
            o[w] = pack_bf16x2(bf16_lo(ewords[w]) + v[c0] * s0, bf16_hi(ewords[w]) + v[c0 + 1] * s1);
          }
          ov[x] = make_uint4(o[0], o[1], o[2], o[3]);
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

bool lowrank_tc_supported(retrace_dtype dtype, int d) { return dtype == RETRACE_BF16 && d % kFuseFeat == 0; }

cudaError_t launch_lowrank(const LowRankArgs& a, bool tc, cudaStream_t stream) {
  const long long rmax = (long long)a.B * (a.K > 1 ? a.K - 1 : 0);
  if (rmax <= 0) return cudaSuccess;
  cudaError_t err;
  if (!tc) {
    const unsigned gemv_grid = (unsigned)((a.d + 7) / 8);
    if (a.dtype == RETRACE_BF16)
      lr_gemv_kernel<__nv_bfloat16><<<gemv_grid, 256, 0, stream>>>(
          reinterpret_cast<const __nv_bfloat16*>(a.Wg), (long long)a.d + L,
          reinterpret_cast<const __nv_bfloat16*>(a.e), a.d, a.ge);
    else
      lr_gemv_kernel<float><<<gemv_grid, 256, 0, stream>>>(reinterpret_cast<const float*>(a.Wg), (long long)a.d + L,
                                                           reinterpret_cast<const float*>(a.e), a.d, a.ge);
    if ((err = cudaGetLastError()) != cudaSuccess) return err;
    if (a.dtype == RETRACE_BF16)
      lr_simt_kernel<__nv_bfloat16><<<(unsigned)rmax, 256, 0, stream>>>(a);
    else
      lr_simt_kernel<float><<<(unsigned)rmax, 256, 0, stream>>>(a);
    return cudaGetLastError();
  }
  DeviceInfo info{0, 148};
  if ((err = device_info(&info)) != cudaSuccess) return err;
  static std::atomic<int> attr_done[64];
  if (!attr_done[info.device & 63].load(std::memory_order_acquire)) {
    if ((err = cudaFuncSetAttribute(lr_project_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_PROJECT)) !=
        cudaSuccess)
      return err;
    if ((err = cudaFuncSetAttribute(lr_fuse_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_FUSE)) !=
        cudaSuccess)
      return err;
    attr_done[info.device & 63].store(1, std::memory_order_release);
  }
  const uint64_t d = (uint64_t)a.d;
  CUtensorMap mA, mP, mBc, mRho, mWv, mWg;
  if (encode_tensor_map_2d(&mA, a.apack, 2 * d, (uint64_t)rmax, 4 * d, BK, BM) != CUDA_SUCCESS ||
      encode_tensor_map_2d(&mP, a.P, d, L, 2 * d, BK, L) != CUDA_SUCCESS ||
      encode_tensor_map_2d(&mBc, a.Bc, L + d, C, 2 * (L + d), BK, C) != CUDA_SUCCESS ||
      encode_tensor_map_2d(&mRho, a.rho, L, (uint64_t)rmax, 2 * L, BK, BM) != CUDA_SUCCESS ||
      encode_tensor_map_2d(&mWv, a.Wv, L, d, 2 * L, BK, kFuseFeat) != CUDA_SUCCESS ||
      encode_tensor_map_2d(&mWg, a.Wg, d + L, d, 2 * (d + L), BK, kFuseFeat) != CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  const unsigned mt = (unsigned)((rmax + BM - 1) / BM);
  LrParams p{};
  p.d = a.d;
  p.R = a.R;
  p.beta = a.beta;
  p.Bc = reinterpret_cast<const __nv_bfloat16*>(a.Bc);
  p.Ac = reinterpret_cast<const __nv_bfloat16*>(a.Ac);
  p.zpart = a.zpart;
  p.tpart = a.tpart;
  p.rho = reinterpret_cast<__nv_bfloat16*>(a.rho);
  p.rmax = rmax;
  p.Wg = reinterpret_cast<const __nv_bfloat16*>(a.Wg);
  p.e = reinterpret_cast<const __nv_bfloat16*>(a.e);
  p.ge = a.ge;
  p.gemv_next = a.gemv_next;
  p.status = a.status;
  // Each of the three kernels may start while the previous one finishes
  // (programmatic dependent launch), and waits for its outputs in the kernel.
  if ((err = launch_dependent(lr_project_kernel, dim3(mt, 2 * H), dim3(256), SMEM_PROJECT, stream, 1, mA, mP, mBc,
                              p)) != cudaSuccess)
    return err;
  const long long fgrid = (rmax + 7) / 8 > 2LL * info.sm_count ? (rmax + 7) / 8 : 2LL * info.sm_count;
  if ((err = launch_dependent(lr_finish_kernel, dim3((unsigned)fgrid), dim3(256), 0, stream, 1, p)) != cudaSuccess)
    return err;
  LrFuseParams f{};
  f.d = a.d;
  f.R = a.R;
  f.rowmap = a.rowmap;
  f.e = reinterpret_cast<const __nv_bfloat16*>(a.e);
  f.ge = a.ge;
  f.e_out = reinterpret_cast<__nv_bfloat16*>(a.e_out);
  f.status = a.status;
  const long long tiles_max = (long long)mt * (a.d / kFuseFeat);
  const long long slots = 2LL * info.sm_count;  // two CTAs per SM
  const unsigned grid = (unsigned)(tiles_max < slots ? tiles_max : slots);
  return launch_dependent(lr_fuse_kernel, dim3(grid), dim3(kFuseThreads), SMEM_FUSE, stream, 1, mRho, mWv, mWg, f);
}

}  // namespace retrace
