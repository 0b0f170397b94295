// Conditioning projections on the 5th-generation tensor cores (tcgen05).
//
//   MODE 0, correction (Eq. 6-7):  r = m + beta * W_c [m; u]
//       A = [m; u] rows gathered from hD / hT by the device row plan
//       (m_j = hD[b, A_b+1+j], u_j = hT[b, A_b+j]); B = W_c (K-major, [d, 2d]).
//       One CTA computes a 128 x 256 tile of c; the epilogue adds m and beta
//       and writes r in bf16.
//   MODE 1, gated fusion (Eq. 8):  e~ = e + (W_v r) .* sigmoid(W_g [e; r])
//       A = r rows; the B tile stacks 128 rows of W_v over the matching 128
//       rows of W_g[:, d:2d], so one N = 256 MMA yields v (TMEM columns
//       0..127) and the r half of the gate (columns 128..255) for the same
//       128 output features.  The e half of the gate is either a broadcast
//       vector precomputed once (W_g[:, :d] e, added in the epilogue) or, for
//       per-position e, extra K blocks accumulated into the gate columns.
//
// Warp roles (256 threads, one CTA per SM):
//   warp 0  TMA producer: 32 lanes each issue one gather4 (4 rows of 128 B)
//           per stage for A, lane 0 the tiled weight box(es) for B;
//   warp 1  MMA issuer: one thread issues 4 x (M128 N256 K16) per stage and
//           commits the stage back to the producer;
//   warp 2  TMEM allocation (256 fp32 columns = the 128 x 256 accumulator);
//   warps 4-7  epilogue: tcgen05.ld of their 32 TMEM lanes (= tile rows).
// Every mbarrier wait is bounded; on expiry the CTA raises the workspace
// status flag, drains its own copies in flight, frees TMEM and returns.
#include "common.cuh"
#include "internal.h"
#include "plan.cuh"

namespace retrace {
namespace {

constexpr int BM = 128;
constexpr int BK = 64;  // 64 bf16 = 128 bytes = one swizzle row
constexpr int STAGES = 4;
constexpr int THREADS = 256;
constexpr int A_BYTES = BM * BK * 2;   // 16 KB
constexpr int B_BYTES = 256 * BK * 2;  // 32 KB
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + 1024;  // + slack for 1024-B alignment
constexpr uint32_t TMEM_COLS = 256;
constexpr uint32_t IDESC_N256 = idesc_bf16_f32(128, 256);
constexpr uint32_t IDESC_N128 = idesc_bf16_f32(128, 128);

struct TcParams {
  int B, K, d;
  RowSource rows;
  const __nv_bfloat16* hD;  // MODE 0: re-read in the epilogue (m term)
  float beta;
  const __nv_bfloat16* e;  // MODE 1
  int e_dense;
  const float* ge;
  int r_compact;
  __nv_bfloat16* out;
  int compact_out;  // MODE 0: write r compact [R, d] (1) or [B, K, d] (0)
  uint32_t* status;
};

__device__ __forceinline__ void raise_abort(volatile int* s_abort, uint32_t* status) {
  *s_abort = 1;
  atomicOr(status, kFlagWaitTimeout);
}

// Lane 0 waits, the warp agrees on the outcome.
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, volatile int* abort) {
  const int lane = threadIdx.x & 31;
  int ok = 1;
  if (lane == 0) ok = mbar_wait_bounded(bar, parity, abort) ? 1 : 0;
  return __shfl_sync(0xFFFFFFFFu, ok, 0) != 0;
}

template <int MODE>
__global__ void __launch_bounds__(THREADS, 1)
    tc_cond_kernel(const __grid_constant__ CUtensorMap tmA0, const __grid_constant__ CUtensorMap tmA1,
                   const __grid_constant__ CUtensorMap tmB0, const __grid_constant__ CUtensorMap tmB1,
                   const TcParams p) {
  extern __shared__ uint8_t dsmem[];
  __shared__ __align__(8) uint64_t bar_full[STAGES];
  __shared__ __align__(8) uint64_t bar_empty[STAGES];
  __shared__ __align__(8) uint64_t bar_acc;
  __shared__ uint32_t s_tmem;
  __shared__ volatile int s_abort;
  __shared__ int s_b[BM], s_j[BM], s_nb[BM], s_scan[THREADS / 32 + 1];
  __shared__ int s_src0[BM], s_src1[BM];

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int K = p.K, d = p.d;
  const long long m0 = (long long)blockIdx.x * BM;
  const int n0 = blockIdx.y * (MODE == 0 ? 256 : 128);

  const int R = plan_tile<THREADS, BM>(p.rows, p.B, K, m0, s_b, s_j, s_nb, s_scan);
  if (m0 >= R) return;  // uniform: this tile has no conditioned rows

  for (int q = tid; q < BM; q += THREADS) {
    const int b = s_b[q];
    int src0 = 0, src1 = 0;  // padding rows read row 0 (valid) and are never stored
    if (b >= 0) {
      const int j = s_j[q];
      if (MODE == 0) {
        const int A = K - 1 - s_nb[q];
        src0 = b * K + A + 1 + j;  // m_j = hD[b, A_b + 1 + j]   (Eq. 4)
        src1 = b * K + A + j;      // u_j = hT[b, A_b + j]       (Eq. 5)
      } else {
        src0 = p.r_compact ? (int)(m0 + q) : b * K + j;
        src1 = b * K + j;
      }
    }
    s_src0[q] = src0;
    s_src1[q] = src1;
  }
  if (tid == 0) {
    s_abort = 0;
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(smem_u32(&bar_full[s]), 1);
      mbar_init(smem_u32(&bar_empty[s]), 1);
    }
    mbar_init(smem_u32(&bar_acc), 1);
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA0);
    tma_prefetch_desc(&tmB0);
    if (MODE == 1) tma_prefetch_desc(&tmB1);
  }
  if (warp == 2) {
    tmem_alloc(smem_u32(&s_tmem), TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s_tmem;
  const uint32_t base = (smem_u32(dsmem) + 1023u) & ~1023u;

  const int kb_half = d / BK;  // K blocks of one d-wide operand half
  const int nkb = (MODE == 0) ? 2 * kb_half : kb_half + (p.e_dense ? kb_half : 0);

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    int kb = 0;
    bool ok = true;
    for (; kb < nkb; ++kb) {
      const int s = kb % STAGES;
      const uint32_t ph = (uint32_t)(kb / STAGES) & 1u;
      if (!warp_wait(smem_u32(&bar_empty[s]), ph ^ 1u, &s_abort)) {
        ok = false;
        break;
      }
      const uint32_t a_dst = base + (uint32_t)(s * STAGE_BYTES);
      const uint32_t b_dst = a_dst + A_BYTES;
      const uint32_t full = smem_u32(&bar_full[s]);
      const bool second = kb >= kb_half;  // u rows (MODE 0) or e rows (MODE 1)
      const int acol = (second ? kb - kb_half : kb) * BK;
      uint32_t bytes;
      if (MODE == 0) bytes = A_BYTES + B_BYTES;
      else bytes = A_BYTES + (second ? B_BYTES / 2 : B_BYTES);
      if (lane == 0) mbar_arrive_expect_tx(full, bytes);
      __syncwarp();
      const CUtensorMap* amap = second ? &tmA1 : &tmA0;
      const int* src = second ? s_src1 : s_src0;
      tma_gather4(a_dst + (uint32_t)lane * 512u, amap, acol, src[4 * lane], src[4 * lane + 1],
                  src[4 * lane + 2], src[4 * lane + 3], full);
      if (lane == 0) {
        if (MODE == 0) {
          tma_load_2d(b_dst, &tmB0, kb * BK, n0, full);  // W_c[n0:n0+256, kb*64 : +64]
        } else if (!second) {
          tma_load_2d(b_dst, &tmB0, kb * BK, n0, full);                   // W_v rows n0..n0+127
          tma_load_2d(b_dst + B_BYTES / 2, &tmB1, d + kb * BK, n0, full);  // W_g[:, d + ...]
        } else {
          tma_load_2d(b_dst + B_BYTES / 2, &tmB1, (kb - kb_half) * BK, n0, full);  // W_g[:, :d]
        }
      }
    }
    if (!ok) {
      if (lane == 0) raise_abort(&s_abort, p.status);
      // Drain this CTA's own copies still in flight before the CTA may exit.
      volatile int never = 0;
      const int first = kb - STAGES > 0 ? kb - STAGES : 0;
      for (int k = first; k < kb; ++k)
        if (lane == 0) mbar_wait_bounded(smem_u32(&bar_full[k % STAGES]), (uint32_t)(k / STAGES) & 1u, &never);
      __syncwarp();
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      bool ok = true;
      for (int kb = 0; kb < nkb; ++kb) {
        const int s = kb % STAGES;
        const uint32_t ph = (uint32_t)(kb / STAGES) & 1u;
        if (!mbar_wait_bounded(smem_u32(&bar_full[s]), ph, &s_abort)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t a_base = base + (uint32_t)(s * STAGE_BYTES);
        const uint32_t b_base = a_base + A_BYTES;
        const bool e_part = (MODE == 1) && kb >= kb_half;
#pragma unroll
        for (int k = 0; k < BK / 16; ++k) {
          const uint64_t adesc = sw128_kmajor_desc(a_base + (uint32_t)k * 32u);
          if (!e_part) {
            const uint64_t bdesc = sw128_kmajor_desc(b_base + (uint32_t)k * 32u);
            tc_mma_bf16(tmem, adesc, bdesc, IDESC_N256, (kb > 0 || k > 0) ? 1u : 0u);
          } else {
            const uint64_t bdesc = sw128_kmajor_desc(b_base + B_BYTES / 2 + (uint32_t)k * 32u);
            tc_mma_bf16(tmem + 128u, adesc, bdesc, IDESC_N128, 1u);
          }
        }
        tc_commit(smem_u32(&bar_empty[s]));
      }
      tc_commit(smem_u32(&bar_acc));  // tracks every MMA issued above, even after a failure
      if (!ok) raise_abort(&s_abort, p.status);
    }
    __syncwarp();
  } else if (warp >= 4) {
    // ---------------- epilogue ----------------
    const bool ok = warp_wait(smem_u32(&bar_acc), 0u, &s_abort);
    tc_fence_after();
    if (ok && !s_abort) {
      const int q = (warp - 4) * 32 + lane;  // tile row = TMEM lane
      const uint32_t taddr = tmem + ((uint32_t)((warp & 3) * 32) << 16);
      const int b = s_b[q];
      const bool valid = b >= 0;
      if (MODE == 0) {
        const long long orow = p.compact_out ? (m0 + q) : ((long long)b * K + s_j[q]);
        const __nv_bfloat16* mrow = p.hD + (long long)s_src0[q] * d;
        for (int cc = 0; cc < 8; ++cc) {
          float acc[32];
          tmem_ld_32cols(taddr + (uint32_t)(cc * 32), acc);
          if (valid) {
            const int n = n0 + cc * 32;
            const uint4* mv = reinterpret_cast<const uint4*>(mrow + n);
            uint4* ov = reinterpret_cast<uint4*>(p.out + orow * d + n);
#pragma unroll
            for (int v = 0; v < 4; ++v) {
              const uint4 mw = __ldg(mv + v);
              const uint32_t mwords[4] = {mw.x, mw.y, mw.z, mw.w};
              uint32_t o[4];
#pragma unroll
              for (int t = 0; t < 4; ++t) {
                const float lo = bf16_lo(mwords[t]) + p.beta * acc[v * 8 + 2 * t];
                const float hi = bf16_hi(mwords[t]) + p.beta * acc[v * 8 + 2 * t + 1];
                o[t] = pack_bf16x2(lo, hi);
              }
              ov[v] = make_uint4(o[0], o[1], o[2], o[3]);
            }
          }
        }
      } else {
        const long long pos = valid ? ((long long)b * K + s_j[q]) : 0;
        const __nv_bfloat16* erow = p.e + (p.e_dense ? pos * d : 0);
        for (int cc = 0; cc < 4; ++cc) {
          float vacc[32], gacc[32];
          tmem_ld_32cols(taddr + (uint32_t)(cc * 32), vacc);
          tmem_ld_32cols(taddr + 128u + (uint32_t)(cc * 32), gacc);
          if (valid) {
            const int n = n0 + cc * 32;
            const uint4* ev = reinterpret_cast<const uint4*>(erow + n);
            uint4* ov = reinterpret_cast<uint4*>(p.out + pos * d + n);
#pragma unroll
            for (int v = 0; v < 4; ++v) {
              const uint4 ew = __ldg(ev + v);
              const uint32_t ewords[4] = {ew.x, ew.y, ew.z, ew.w};
              uint32_t o[4];
#pragma unroll
              for (int t = 0; t < 4; ++t) {
                const int c0 = v * 8 + 2 * t;
                float g0 = gacc[c0], g1 = gacc[c0 + 1];
                if (!p.e_dense) {
                  g0 += __ldg(p.ge + n + c0);
                  g1 += __ldg(p.ge + n + c0 + 1);
                }
                const float s0 = 1.f / (1.f + expf(-g0));
                const float s1 = 1.f / (1.f + expf(-g1));
                const float lo = bf16_lo(ewords[t]) + vacc[c0] * s0;
                const float hi = bf16_hi(ewords[t]) + vacc[c0 + 1] * s1;
                o[t] = pack_bf16x2(lo, hi);
              }
              ov[v] = make_uint4(o[0], o[1], o[2], o[3]);
            }
          }
        }
      }
    }
  }
  // ---------------- teardown ----------------
  tc_fence_before();
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

bool encode_row_gather_map(CUtensorMap* m, const void* base, int d, long long rows) {
  return encode_tensor_map_2d(m, base, (uint64_t)d, (uint64_t)rows, (uint64_t)d * 2, BK, 1) ==
         CUDA_SUCCESS;
}

template <int MODE>
cudaError_t ensure_smem_attr() {
  static int done[64] = {0};
  int dev = 0;
  cudaError_t err = cudaGetDevice(&dev);
  if (err != cudaSuccess) return err;
  if (!done[dev & 63]) {
    err = cudaFuncSetAttribute(tc_cond_kernel<MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               SMEM_BYTES);
    if (err != cudaSuccess) return err;
    done[dev & 63] = 1;
  }
  return cudaSuccess;
}

}  // namespace

bool tc_supported(retrace_dtype dtype, int d) {
  return dtype == RETRACE_BF16 && d >= 256 && d % 256 == 0;
}

cudaError_t launch_correct_tc(const CorrectArgs& a, uint32_t* status, cudaStream_t stream) {
  const long long rmax = (long long)a.B * (a.K - 1);
  if (rmax <= 0) return cudaSuccess;
  cudaError_t err = ensure_smem_attr<0>();
  if (err != cudaSuccess) return err;
  CUtensorMap mA0, mA1, mB0;
  const long long rows = (long long)a.B * a.K;
  if (!encode_row_gather_map(&mA0, a.hD, a.d, rows) || !encode_row_gather_map(&mA1, a.hT, a.d, rows) ||
      encode_tensor_map_2d(&mB0, a.Wc, (uint64_t)2 * a.d, (uint64_t)a.d, (uint64_t)a.d * 4, BK, 256) !=
          CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  TcParams p{};
  p.B = a.B;
  p.K = a.K;
  p.d = a.d;
  p.rows = a.rows;
  p.hD = reinterpret_cast<const __nv_bfloat16*>(a.hD);
  p.beta = a.beta;
  p.out = reinterpret_cast<__nv_bfloat16*>(a.r_out);
  p.compact_out = a.compact_out;
  p.status = status;
  dim3 grid((unsigned)((rmax + BM - 1) / BM), (unsigned)(a.d / 256));
  tc_cond_kernel<0><<<grid, THREADS, SMEM_BYTES, stream>>>(mA0, mA1, mB0, mB0, p);
  return cudaGetLastError();
}

cudaError_t launch_gate_tc(const GateArgs& a, uint32_t* status, cudaStream_t stream) {
  const long long rmax = (long long)a.B * (a.K - 1);
  if (rmax <= 0) return cudaSuccess;
  cudaError_t err = ensure_smem_attr<1>();
  if (err != cudaSuccess) return err;
  CUtensorMap mA0, mA1, mB0, mB1;
  const long long rows = (long long)a.B * a.K;
  if (!encode_row_gather_map(&mA0, a.r, a.d, a.r_rows) ||
      !encode_row_gather_map(&mA1, a.e_dense ? a.e : a.r, a.d, a.e_dense ? rows : a.r_rows) ||
      encode_tensor_map_2d(&mB0, a.Wv, (uint64_t)a.d, (uint64_t)a.d, (uint64_t)a.d * 2, BK, 128) !=
          CUDA_SUCCESS ||
      encode_tensor_map_2d(&mB1, a.Wg, (uint64_t)2 * a.d, (uint64_t)a.d, (uint64_t)a.d * 4, BK, 128) !=
          CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  TcParams p{};
  p.B = a.B;
  p.K = a.K;
  p.d = a.d;
  p.rows = a.rows;
  p.e = reinterpret_cast<const __nv_bfloat16*>(a.e);
  p.e_dense = a.e_dense;
  p.ge = a.ge;
  p.r_compact = a.r_compact;
  p.out = reinterpret_cast<__nv_bfloat16*>(a.e_out);
  p.status = status;
  dim3 grid((unsigned)((rmax + BM - 1) / BM), (unsigned)(a.d / 128));
  tc_cond_kernel<1><<<grid, THREADS, SMEM_BYTES, stream>>>(mA0, mA1, mB0, mB1, p);
  return cudaGetLastError();
}

}  // namespace retrace
