// Conditioning projections on the 5th-generation tensor cores (tcgen05).
//
// Two steps per projection family:
//
// 1. pack_rows_kernel lays the conditioned rows out contiguously, in sequence
//    order (R = sum_b n_b rows, n_b = max(0, K-1-A_b)):
//      correction operand  Apack[g] = [ hD[b, A_b+1+j] ; hT[b, A_b+j] ]  (Eq. 4-5),
//      or the corrected signal rows r[b, j] for a standalone gate call,
//      plus, for per-position e, Epack[g] = e[b, j];
//    with rowmap[g] = b*K + j and the row count R.  Contiguous rows let the
//    GEMMs stream their A operand with tiled TMA boxes (per-row gathers were
//    measured to starve the tensor pipe).
//
// 2. tc_gemm_kernel, persistent (one CTA per SM, static tile schedule):
//    MODE 0, correction (Eq. 6-7):  r = m + beta * W_c [m; u]
//        A = Apack [R, 2d]; B = W_c [d, 2d] (K-major); 128 x 256 tiles of c;
//        the epilogue adds m (the first d columns of Apack) and writes r bf16.
//    MODE 1, gated fusion (Eq. 8):  e~ = e + (W_v r) .* sigmoid(W_g [e; r])
//        A = r rows; the B tile stacks 128 rows of W_v over the matching 128
//        rows of W_g[:, d:2d], so one N = 256 MMA yields v (accumulator
//        columns 0..127) and the r half of the gate (128..255) for the same
//        output features.  The e half of the gate is a broadcast vector
//        precomputed once (added in the epilogue) or, for per-position e,
//        extra K blocks (Epack x W_g[:, :d]) accumulated into the gate columns.
//
// Warp roles of the GEMM (256 threads):
//   warp 0     TMA producer (one elected lane): A box + weight box(es) per stage;
//   warp 1     MMA issuer (one lane): 4 x tcgen05.mma M128 N256 K16 per stage;
//   warp 2     TMEM allocation: 2 accumulators x 256 fp32 columns = 512 columns;
//   warps 4-7  epilogue: tcgen05.ld of their 32 TMEM lanes (= tile rows).
// The two accumulators alternate between tiles, so a tile's epilogue overlaps
// the next tile's main loop.  Every mbarrier wait is bounded; on expiry the CTA
// raises the workspace status flag, drains its own copies in flight, frees
// TMEM and returns.
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
constexpr uint32_t ACC_COLS = 256;
constexpr uint32_t TMEM_COLS = 2 * ACC_COLS;
constexpr uint32_t IDESC_N256 = idesc_bf16_f32(128, 256);
constexpr uint32_t IDESC_N128 = idesc_bf16_f32(128, 128);

// ---------------------------------------------------------------------------
// Row packing
// ---------------------------------------------------------------------------
struct PackParams {
  int B, K, d;
  RowSource rows;
  int mode;  // 0: [m; u] from hD / hT; 1: r rows from r [B, K, d]
  const __nv_bfloat16* src0;
  const __nv_bfloat16* src1;
  const __nv_bfloat16* e;
  int e_dense;
  __nv_bfloat16* apack;
  __nv_bfloat16* epack;
  int32_t* rowmap;
  int32_t* R_out;
};

// One CTA per sequence.  Its first packed row is the number of rows of all
// earlier sequences (a block-wide sum), so the layout is the sequence order.
__global__ void __launch_bounds__(256) pack_rows_kernel(const PackParams p) {
  __shared__ int s_red[8];
  const int b = blockIdx.x, tid = threadIdx.x, K = p.K, d = p.d;
  int part = 0;
  for (int x = tid; x < b; x += 256) part += rows_of(p.rows, x, K);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(0xFFFFFFFFu, part, o);
  if ((tid & 31) == 0) s_red[tid >> 5] = part;
  __syncthreads();
  int off = 0;
#pragma unroll
  for (int w = 0; w < 8; ++w) off += s_red[w];
  const int nb = rows_of(p.rows, b, K);
  if (b == p.B - 1 && tid == 0) *p.R_out = off + nb;
  if (nb == 0) return;
  for (int j = tid; j < nb; j += 256) p.rowmap[off + j] = b * K + j;
  const int vpr = d / 8;  // 16-byte vectors per d-wide row
  const long long base = (long long)b * K;
  if (p.mode == 0) {
    const int A = K - 1 - nb;
    const uint4* hD = reinterpret_cast<const uint4*>(p.src0);
    const uint4* hT = reinterpret_cast<const uint4*>(p.src1);
    uint4* out = reinterpret_cast<uint4*>(p.apack);
    for (int i = tid; i < nb * 2 * vpr; i += 256) {
      const int j = i / (2 * vpr), c = i % (2 * vpr);
      const uint4 v = (c < vpr) ? __ldg(hD + (base + A + 1 + j) * vpr + c)   // m_j (Eq. 4)
                                : __ldg(hT + (base + A + j) * vpr + c - vpr);  // u_j (Eq. 5)
      out[(long long)(off + j) * 2 * vpr + c] = v;
    }
  } else {
    const uint4* r = reinterpret_cast<const uint4*>(p.src0);
    uint4* out = reinterpret_cast<uint4*>(p.apack);
    for (int i = tid; i < nb * vpr; i += 256) {
      const int j = i / vpr, c = i % vpr;
      out[(long long)(off + j) * vpr + c] = __ldg(r + (base + j) * vpr + c);
    }
  }
  if (p.e_dense) {
    const uint4* e = reinterpret_cast<const uint4*>(p.e);
    uint4* out = reinterpret_cast<uint4*>(p.epack);
    for (int i = tid; i < nb * vpr; i += 256) {
      const int j = i / vpr, c = i % vpr;
      out[(long long)(off + j) * vpr + c] = __ldg(e + (base + j) * vpr + c);
    }
  }
}

// ---------------------------------------------------------------------------
// Persistent GEMM
// ---------------------------------------------------------------------------
struct TcParams {
  int d;
  int tiles_n;       // N tiles (d/256 for MODE 0, d/128 for MODE 1)
  const int32_t* R;  // conditioned rows (written by the pack kernel)
  const int32_t* rowmap;
  const __nv_bfloat16* apack;  // MODE 0: [R, 2d], the m half is re-read by the epilogue
  float beta;
  const __nv_bfloat16* e;  // MODE 1: broadcast vector [d] or Epack [R, d]
  int e_dense;
  const float* ge;
  __nv_bfloat16* out;
  int compact_out;  // MODE 0: write row g (1) or row rowmap[g] (0)
  uint32_t* status;
  // MODE 0 only, optional: ge_out[i] = sum_k W_g[i, k] e[k] over the e half
  // (k < d) for a broadcast e, computed by the otherwise idle warps 2-3 while
  // the tensor cores run, so the gated-fusion kernel finds it ready.
  const __nv_bfloat16* Wg;
  const __nv_bfloat16* e_vec;
  float* ge_out;
};

__device__ __forceinline__ void raise_abort(volatile int* s_abort, uint32_t* status) {
  *s_abort = 1;
  atomicOr(status, kFlagWaitTimeout);
}

// Lane 0 waits, the warp agrees on the outcome.
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, volatile int* abort) {
  int ok = 1;
  if ((threadIdx.x & 31) == 0) ok = mbar_wait_bounded(bar, parity, abort) ? 1 : 0;
  return __shfl_sync(0xFFFFFFFFu, ok, 0) != 0;
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

template <int MODE>
__global__ void __launch_bounds__(THREADS, 1)
    tc_gemm_kernel(const __grid_constant__ CUtensorMap tmA0, const __grid_constant__ CUtensorMap tmA1,
                   const __grid_constant__ CUtensorMap tmB0, const __grid_constant__ CUtensorMap tmB1,
                   const TcParams p) {
  extern __shared__ uint8_t dsmem[];
  __shared__ __align__(8) uint64_t bar_full[STAGES];
  __shared__ __align__(8) uint64_t bar_empty[STAGES];
  __shared__ __align__(8) uint64_t bar_tfull[2];
  __shared__ __align__(8) uint64_t bar_tempty[2];
  __shared__ uint32_t s_tmem;
  __shared__ volatile int s_abort;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int d = p.d;
  const int R = *(volatile const int32_t*)p.R;
  const int tiles_m = (R + BM - 1) / BM;
  const int tiles = tiles_m * p.tiles_n;
  if ((int)blockIdx.x >= tiles) return;  // uniform: no tile for this CTA

  if (tid == 0) {
    s_abort = 0;
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(smem_u32(&bar_full[s]), 1);
      mbar_init(smem_u32(&bar_empty[s]), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(smem_u32(&bar_tfull[a]), 1);
      mbar_init(smem_u32(&bar_tempty[a]), 4);  // one arrival per epilogue warp
    }
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA0);
    tma_prefetch_desc(&tmB0);
    if (MODE == 1) {
      tma_prefetch_desc(&tmA1);
      tma_prefetch_desc(&tmB1);
    }
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
  const int n_width = (MODE == 0) ? 256 : 128;

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      uint32_t it = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x) {
        const int m0 = (t % tiles_m) * BM, n0 = (t / tiles_m) * n_width;
        for (int kb = 0; kb < nkb; ++kb, ++it) {
          const uint32_t s = it % STAGES, ph = (it / STAGES) & 1u;
          if (!mbar_wait_bounded(smem_u32(&bar_empty[s]), ph ^ 1u, &s_abort)) {
            ok = false;
            break;
          }
          const uint32_t a_dst = base + s * STAGE_BYTES, b_dst = a_dst + A_BYTES;
          const uint32_t full = smem_u32(&bar_full[s]);
          if (MODE == 0) {
            mbar_arrive_expect_tx(full, A_BYTES + B_BYTES);
            tma_load_2d(a_dst, &tmA0, kb * BK, m0, full);  // [m; u] rows, K block kb
            tma_load_2d(b_dst, &tmB0, kb * BK, n0, full);  // W_c rows n0..n0+255
          } else if (kb < kb_half) {
            mbar_arrive_expect_tx(full, A_BYTES + B_BYTES);
            tma_load_2d(a_dst, &tmA0, kb * BK, m0, full);                    // r rows
            tma_load_2d(b_dst, &tmB0, kb * BK, n0, full);                    // W_v rows
            tma_load_2d(b_dst + B_BYTES / 2, &tmB1, d + kb * BK, n0, full);  // W_g[:, d:2d] rows
          } else {
            mbar_arrive_expect_tx(full, A_BYTES + B_BYTES / 2);
            tma_load_2d(a_dst, &tmA1, (kb - kb_half) * BK, m0, full);                    // e rows
            tma_load_2d(b_dst + B_BYTES / 2, &tmB1, (kb - kb_half) * BK, n0, full);  // W_g[:, :d]
          }
        }
      }
      if (!ok) {
        raise_abort(&s_abort, p.status);
        // Drain this CTA's own copies still in flight before the CTA may exit.
        volatile int never = 0;
        const uint32_t first = it > STAGES ? it - STAGES : 0;
        for (uint32_t k = first; k < it; ++k)
          mbar_wait_bounded(smem_u32(&bar_full[k % STAGES]), (k / STAGES) & 1u, &never);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      uint32_t it = 0, lt = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x, ++lt) {
        const uint32_t acc = lt & 1u, aph = (lt >> 1) & 1u;
        if (!mbar_wait_bounded(smem_u32(&bar_tempty[acc]), aph ^ 1u, &s_abort)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem + acc * ACC_COLS;
        for (int kb = 0; kb < nkb; ++kb, ++it) {
          const uint32_t s = it % STAGES, ph = (it / STAGES) & 1u;
          if (!mbar_wait_bounded(smem_u32(&bar_full[s]), ph, &s_abort)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a_base = base + s * STAGE_BYTES, b_base = a_base + A_BYTES;
          const bool e_part = (MODE == 1) && kb >= kb_half;
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            const uint64_t adesc = sw128_kmajor_desc(a_base + (uint32_t)k * 32u);
            if (!e_part) {
              const uint64_t bdesc = sw128_kmajor_desc(b_base + (uint32_t)k * 32u);
              tc_mma_bf16(d_tmem, adesc, bdesc, IDESC_N256, (kb > 0 || k > 0) ? 1u : 0u);
            } else {
              const uint64_t bdesc = sw128_kmajor_desc(b_base + B_BYTES / 2 + (uint32_t)k * 32u);
              tc_mma_bf16(d_tmem + 128u, adesc, bdesc, IDESC_N128, 1u);
            }
          }
          tc_commit(smem_u32(&bar_empty[s]));  // stage reusable once these MMAs finish
        }
        tc_commit(smem_u32(&bar_tfull[acc]));  // accumulator ready (also after a failure)
      }
      if (!ok) raise_abort(&s_abort, p.status);
    }
    __syncwarp();
  } else if (MODE == 0 && (warp == 2 || warp == 3)) {
    // ---------------- gate bias W_g[:, :d] e (broadcast e) ----------------
    if (p.ge_out) {
      const int active = tiles < (int)gridDim.x ? tiles : (int)gridDim.x;
      const int vpr = d / 8;
      const uint4* ev = reinterpret_cast<const uint4*>(p.e_vec);
      for (int i = (int)blockIdx.x * 2 + (warp - 2); i < d; i += 2 * active) {
        const uint4* wr = reinterpret_cast<const uint4*>(p.Wg + (long long)i * 2 * d);
        float acc = 0.f;
        for (int v = lane; v < vpr; v += 32) {
          const uint4 w = __ldcs(wr + v), x = __ldg(ev + v);
          const uint32_t ww[4] = {w.x, w.y, w.z, w.w}, xx[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
          for (int t = 0; t < 4; ++t) {
            acc = fmaf(bf16_lo(ww[t]), bf16_lo(xx[t]), acc);
            acc = fmaf(bf16_hi(ww[t]), bf16_hi(xx[t]), acc);
          }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xFFFFFFFFu, acc, o);
        if (lane == 0) p.ge_out[i] = acc;
      }
    }
  } else if (warp >= 4) {
    // ---------------- epilogue ----------------
    const int q = (warp - 4) * 32 + lane;  // tile row = TMEM lane
    const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
    uint32_t lt = 0;
    for (int t = blockIdx.x; t < tiles; t += gridDim.x, ++lt) {
      const uint32_t acc = lt & 1u, aph = (lt >> 1) & 1u;
      const bool ok = warp_wait(smem_u32(&bar_tfull[acc]), aph, &s_abort);
      tc_fence_after();
      if (!ok) {
        if (lane == 0) raise_abort(&s_abort, p.status);
        break;
      }
      if (s_abort) break;
      const int m0 = (t % tiles_m) * BM, n0 = (t / tiles_m) * n_width;
      const int g = m0 + q;
      const bool valid = g < R;
      const uint32_t taddr = tmem + acc * ACC_COLS + lane_base;
      if (MODE == 0) {
        const __nv_bfloat16* mrow = p.apack + (long long)g * 2 * d;  // m = first d columns
        const long long orow = valid ? (p.compact_out ? g : p.rowmap[g]) : 0;
        for (int cc = 0; cc < 8; ++cc) {
          float c[32];
          tmem_ld_32cols(taddr + (uint32_t)(cc * 32), c);
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
              for (int w = 0; w < 4; ++w) {
                const float lo = bf16_lo(mwords[w]) + p.beta * c[v * 8 + 2 * w];
                const float hi = bf16_hi(mwords[w]) + p.beta * c[v * 8 + 2 * w + 1];
                o[w] = pack_bf16x2(lo, hi);
              }
              ov[v] = make_uint4(o[0], o[1], o[2], o[3]);
            }
          }
        }
      } else {
        const long long orow = valid ? p.rowmap[g] : 0;
        const __nv_bfloat16* erow = p.e + (p.e_dense ? (long long)g * d : 0);
        for (int cc = 0; cc < 4; ++cc) {
          float v[32], gt[32];
          tmem_ld_32cols(taddr + (uint32_t)(cc * 32), v);
          tmem_ld_32cols(taddr + 128u + (uint32_t)(cc * 32), gt);
          if (valid) {
            const int n = n0 + cc * 32;
            const uint4* ev = reinterpret_cast<const uint4*>(erow + n);
            uint4* ov = reinterpret_cast<uint4*>(p.out + orow * d + n);
#pragma unroll
            for (int x = 0; x < 4; ++x) {
              const uint4 ew = __ldg(ev + x);
              const uint32_t ewords[4] = {ew.x, ew.y, ew.z, ew.w};
              uint32_t o[4];
#pragma unroll
              for (int w = 0; w < 4; ++w) {
                const int c0 = x * 8 + 2 * w;
                float g0 = gt[c0], g1 = gt[c0 + 1];
                if (!p.e_dense) {
                  g0 += __ldg(p.ge + n + c0);
                  g1 += __ldg(p.ge + n + c0 + 1);
                }
                const float s0 = 1.f / (1.f + expf(-g0));
                const float s1 = 1.f / (1.f + expf(-g1));
                o[w] = pack_bf16x2(bf16_lo(ewords[w]) + v[c0] * s0, bf16_hi(ewords[w]) + v[c0 + 1] * s1);
              }
              ov[x] = make_uint4(o[0], o[1], o[2], o[3]);
            }
          }
        }
      }
      // hand the accumulator back to the MMA warp
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&bar_tempty[acc]));
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

template <int MODE>
cudaError_t ensure_smem_attr() {
  static int done[64] = {0};
  int dev = 0;
  cudaError_t err = cudaGetDevice(&dev);
  if (err != cudaSuccess) return err;
  if (!done[dev & 63]) {
    err = cudaFuncSetAttribute(tc_gemm_kernel<MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               SMEM_BYTES);
    if (err != cudaSuccess) return err;
    done[dev & 63] = 1;
  }
  return cudaSuccess;
}

unsigned persistent_grid(long long tiles_max) {
  DeviceInfo info{0, 148};
  device_info(&info);
  long long g = info.sm_count;
  if (tiles_max < g) g = tiles_max;
  return (unsigned)(g > 0 ? g : 1);
}

}  // namespace

bool tc_supported(retrace_dtype dtype, int d) {
  return dtype == RETRACE_BF16 && d >= 256 && d % 256 == 0;
}

cudaError_t launch_pack(const PackArgs& a, cudaStream_t stream) {
  if (a.B <= 0) return cudaSuccess;
  PackParams p;
  p.B = a.B;
  p.K = a.K;
  p.d = a.d;
  p.rows = a.rows;
  p.mode = a.mode;
  p.src0 = reinterpret_cast<const __nv_bfloat16*>(a.src0);
  p.src1 = reinterpret_cast<const __nv_bfloat16*>(a.src1);
  p.e = reinterpret_cast<const __nv_bfloat16*>(a.e);
  p.e_dense = a.e_dense;
  p.apack = reinterpret_cast<__nv_bfloat16*>(a.apack);
  p.epack = reinterpret_cast<__nv_bfloat16*>(a.epack);
  p.rowmap = a.rowmap;
  p.R_out = a.R;
  pack_rows_kernel<<<(unsigned)a.B, 256, 0, stream>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_correct_tc(const TcCorrectArgs& a, cudaStream_t stream) {
  const long long rmax = (long long)a.B * (a.K - 1);
  if (rmax <= 0) return cudaSuccess;
  cudaError_t err = ensure_smem_attr<0>();
  if (err != cudaSuccess) return err;
  CUtensorMap mA, mB;
  if (encode_tensor_map_2d(&mA, a.apack, (uint64_t)2 * a.d, (uint64_t)rmax, (uint64_t)a.d * 4, BK, BM) !=
          CUDA_SUCCESS ||
      encode_tensor_map_2d(&mB, a.Wc, (uint64_t)2 * a.d, (uint64_t)a.d, (uint64_t)a.d * 4, BK, 256) != CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  TcParams p{};
  p.d = a.d;
  p.tiles_n = a.d / 256;
  p.R = a.R;
  p.rowmap = a.rowmap;
  p.apack = reinterpret_cast<const __nv_bfloat16*>(a.apack);
  p.beta = a.beta;
  p.out = reinterpret_cast<__nv_bfloat16*>(a.r_out);
  p.compact_out = a.compact_out;
  p.status = a.status;
  p.Wg = reinterpret_cast<const __nv_bfloat16*>(a.Wg);
  p.e_vec = reinterpret_cast<const __nv_bfloat16*>(a.e_vec);
  p.ge_out = a.ge_out;
  const long long tiles_max = (rmax + BM - 1) / BM * p.tiles_n;
  tc_gemm_kernel<0><<<persistent_grid(tiles_max), THREADS, SMEM_BYTES, stream>>>(mA, mA, mB, mB, p);
  return cudaGetLastError();
}

cudaError_t launch_gate_tc(const TcGateArgs& a, cudaStream_t stream) {
  const long long rmax = (long long)a.B * (a.K - 1);
  if (rmax <= 0) return cudaSuccess;
  cudaError_t err = ensure_smem_attr<1>();
  if (err != cudaSuccess) return err;
  CUtensorMap mA0, mA1, mB0, mB1;
  const void* e_rows = a.e_dense ? a.epack : a.rpack;
  if (encode_tensor_map_2d(&mA0, a.rpack, (uint64_t)a.d, (uint64_t)rmax, (uint64_t)a.d * 2, BK, BM) !=
          CUDA_SUCCESS ||
      encode_tensor_map_2d(&mA1, e_rows, (uint64_t)a.d, (uint64_t)rmax, (uint64_t)a.d * 2, BK, BM) !=
          CUDA_SUCCESS ||
      encode_tensor_map_2d(&mB0, a.Wv, (uint64_t)a.d, (uint64_t)a.d, (uint64_t)a.d * 2, BK, 128) != CUDA_SUCCESS ||
      encode_tensor_map_2d(&mB1, a.Wg, (uint64_t)2 * a.d, (uint64_t)a.d, (uint64_t)a.d * 4, BK, 128) !=
          CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  TcParams p{};
  p.d = a.d;
  p.tiles_n = a.d / 128;
  p.R = a.R;
  p.rowmap = a.rowmap;
  p.e = reinterpret_cast<const __nv_bfloat16*>(a.e_dense ? a.epack : a.e);
  p.e_dense = a.e_dense;
  p.ge = a.ge;
  p.out = reinterpret_cast<__nv_bfloat16*>(a.e_out);
  p.status = a.status;
  const long long tiles_max = (rmax + BM - 1) / BM * p.tiles_n;
  tc_gemm_kernel<1><<<persistent_grid(tiles_max), THREADS, SMEM_BYTES, stream>>>(mA0, mA1, mB0, mB1, p);
  return cudaGetLastError();
}

}  // namespace retrace
