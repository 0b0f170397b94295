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
// 2. one persistent launch runs both projections from a dynamic tile queue
//    (every correction tile, then every gate tile; a gate tile of a row block
//    waits until the correction epilogues of that block have written r):
//    correction (Eq. 6-7):  r = m + beta * W_c [m; u]
//        A = Apack [R, 2d]; B = W_c [d, 2d] (K-major); N = 256 tiles of c;
//        the epilogue adds m (the first d columns of Apack) and writes r bf16.
//    gated fusion (Eq. 8):  e~ = e + (W_v r) .* sigmoid(W_g [e; r])
//        A = r rows; the B tile stacks 128 rows of W_v over the matching 128
//        rows of W_g[:, d:2d], so one N = 256 MMA yields v (accumulator
//        columns 0..127) and the r half of the gate (128..255) for the same
//        output features.  The e half of the gate is a broadcast vector
//        computed once by idle warps (W_g[:, :d] e, added in the epilogue)
//        or, for per-position e, extra K blocks (Epack x W_g[:, :d])
//        accumulated into the gate columns.
//    Two kernels implement it:
//    cond_pair_kernel   (broadcast e) clusters of two CTAs, 256-row tiles,
//                       tcgen05.mma.cta_group::2 M256 N256 K16; each CTA
//                       stages its own 128 rows and half of the weight tile
//                       (described at the kernel);
//    cond_kernel<false> (per-position e) one CTA per SM, 128-row tiles,
//                       tcgen05.mma.cta_group::1 M128 N256 K16;
//    cond_kernel<true>  the overlapped round: the same plus verification
//                       streamed through shared memory (verify_stream.cuh).
//
// Warp roles of cond_kernel<false> (256 threads; the pair kernel's are alike):
//   warp 0     tile scheduler + TMA producer (one elected lane);
//   warp 1     MMA issuer (one lane): 4 x tcgen05.mma per 64-deep stage;
//   warp 2     TMEM allocation: 2 accumulators x 256 fp32 columns = 512 columns;
//   warps 2-3  the broadcast-e GEMV W_g[:, :d] e, rows claimed from a counter;
//   warps 4-7  epilogue: tcgen05.ld of their 32 TMEM lanes (= tile rows).
// The two accumulators alternate between tiles, so a tile's epilogue overlaps
// the next tile's main loop.  Every mbarrier wait is bounded; on expiry the CTA
// raises the workspace status flag, drains its own copies in flight, frees
// TMEM and returns.
#include "common.cuh"
#include "internal.h"
#include "plan.cuh"
#include "tc_pair.cuh"
#include "verify_stream.cuh"

namespace retrace {
namespace {

constexpr int BM = 128;
constexpr int BK = 64;  // 64 bf16 = 128 bytes = one swizzle row
constexpr int STAGES = 4;
constexpr int THREADS = 256;
constexpr int THREADS_FUSED = 2 * THREADS + 32;  // + consumer warps 8-15 and the bookkeeper warp 16
constexpr int A_BYTES = BM * BK * 2;   // 16 KB
constexpr int B_BYTES = 256 * BK * 2;  // 32 KB
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + 1024;  // + slack for 1024-B alignment
// The fused round kernel keeps three operand stages and gives the rest of the
// shared memory to the ring that streams the logits.
constexpr int STAGES_FUSED = 3;
constexpr int SMEM_BYTES_FUSED = STAGES_FUSED * STAGE_BYTES + kRingBufs * kChunkBytes + kStageBytes + 1024;
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
// Persistent, dynamically scheduled projections
// ---------------------------------------------------------------------------
struct CondParams {
  int d;
  int do_correct, do_gate;
  const int32_t* R;
  const int32_t* rowmap;
  // correction
  const __nv_bfloat16* apack;  // [R, 2d]; the m half is re-read by the epilogue
  float beta;
  __nv_bfloat16* r_out;
  int compact_out;
  // gate
  const __nv_bfloat16* e;  // broadcast vector [d], or packed e rows [R, d] (e_dense)
  int e_dense;
  const __nv_bfloat16* Wg;
  float* ge;  // [d] = W_g[:, :d] e, computed here for a broadcast e
  __nv_bfloat16* e_out;
  uint32_t* sync;
  uint32_t* block_done;   // per 128-row block: correction epilogue warps finished
  uint32_t* block_ready;  // per 128-row block: packed rows published (FUSED)
  int max_blocks;         // 128-row blocks of the largest possible R
  // CTA-pair kernel: the gate tiles of a last wave of at most split_max
  // tiles run as two K halves on two pairs.  Each half writes its fp32
  // accumulator to split_part and counts on split_ticket; the half that
  // counts second adds the other's accumulator to its own and runs the
  // epilogue.
  float* split_part;
  uint32_t* split_ticket;
  int split_max;
  uint32_t* status;
};

constexpr int TILE_SLOTS = 2;

// gate_bias_rows (tc_pair.cuh) over this kernel's broadcast e, W_g and ge.
__device__ __forceinline__ void gate_bias_rows(const CondParams& p, int d, int lane, uint32_t* next, uint32_t* done) {
  gate_bias_rows(p.e, p.Wg, p.ge, d, lane, next, done);
}

// Correction epilogue of one tile row (Eq. 7): r = m + beta * c for the 256
// accumulator columns n0.., m = the first d columns of the packed row g.
__device__ __forceinline__ void epilogue_correction(const CondParams& p, uint32_t taddr, int g, bool valid, int n0,
                                                    int d) {
  const __nv_bfloat16* mrow = p.apack + (long long)g * 2 * d;
  const long long orow = valid ? (p.compact_out ? g : __ldcg(p.rowmap + g)) : 0;
  for (int cc = 0; cc < 8; ++cc) {
    float c[32];
    tmem_ld_32cols(taddr + (uint32_t)(cc * 32), c);
    if (valid) {
      const int n = n0 + cc * 32;
      const uint4* mv = reinterpret_cast<const uint4*>(mrow + n);
      uint4* ov = reinterpret_cast<uint4*>(p.r_out + orow * d + n);
#pragma unroll
      for (int v = 0; v < 4; ++v) {
        const uint4 mw = __ldcg(mv + v);
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
}

// Gated-fusion epilogue of one tile row (Eq. 8): e~ = e + v * sigmoid(g) for
// the 128 features n0.., v in accumulator columns 0..127, the r half of the
// gate in 128..255 (plus W_g[:, :d] e from ge for a broadcast e, the same
// 32 values for every lane: one 16-byte broadcast load per four features).
// With `other` (a split tile), the other K half's accumulator of this row is
// added first: column c at other[128 c].
__device__ __forceinline__ void epilogue_gate(const CondParams& p, uint32_t taddr, int g, bool valid, int n0, int d,
                                              const float* other = nullptr) {
  const long long orow = valid ? __ldcg(p.rowmap + g) : 0;
  const __nv_bfloat16* erow = p.e + (p.e_dense ? (long long)g * d : 0);
  for (int cc = 0; cc < 4; ++cc) {
    float v[32], gt[32];
    tmem_ld_32cols(taddr + (uint32_t)(cc * 32), v);
    tmem_ld_32cols(taddr + 128u + (uint32_t)(cc * 32), gt);
    if (valid) {
      const int n = n0 + cc * 32;
      if (other) {
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          v[i] += __ldcg(other + (cc * 32 + i) * 128);
          gt[i] += __ldcg(other + (128 + cc * 32 + i) * 128);
        }
      }
      if (!p.e_dense) {
        const float4* gb = reinterpret_cast<const float4*>(p.ge + n);
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const float4 b = __ldcg(gb + j);
          gt[4 * j] += b.x;
          gt[4 * j + 1] += b.y;
          gt[4 * j + 2] += b.z;
          gt[4 * j + 3] += b.w;
        }
      }
      const uint4* ev = reinterpret_cast<const uint4*>(erow + n);
      uint4* ov = reinterpret_cast<uint4*>(p.e_out + orow * d + n);
#pragma unroll
      for (int x = 0; x < 4; ++x) {
        const uint4 ew = __ldcg(ev + x);
        const uint32_t ewords[4] = {ew.x, ew.y, ew.z, ew.w};
        uint32_t o[4];
#pragma unroll
        for (int w = 0; w < 4; ++w) {
          const int c0 = x * 8 + 2 * w;
          const float s0 = fast_sigmoid(gt[c0]), s1 = fast_sigmoid(gt[c0 + 1]);
          o[w] = pack_bf16x2(bf16_lo(ewords[w]) + v[c0] * s0, bf16_hi(ewords[w]) + v[c0 + 1] * s1);
        }
        ov[x] = make_uint4(o[0], o[1], o[2], o[3]);
      }
    }
  }
}

// Tile t < T0: correction tile (row block t / nt0, 256 output columns t % nt0);
// T0 <= t < T0 + T1: gate tile (row block (t-T0) / nt1, 128 features).  Tiles
// are handed out in this order by a global counter, so every gate tile's row
// block was handed out (to a running CTA) before it.
// FUSED: the same kernel also runs verification (verify_stream.cuh): warp 3
// streams the logits into a shared-memory ring, warps 8-15 reduce it, warp 16 folds the keys.  Packed rows then become available while the
// kernel runs, so the tile queue is decoded in phases -- phase q holds the
// correction tiles of row block q followed by the gate tiles of row block
// q - kGateLag -- and the producer resolves each tile against the published
// per-block row counts before loading it.  R (and the last partial block) is
// known once every sequence is finalised.
constexpr int kGateLag = 4;

template <bool FUSED>
__global__ void __launch_bounds__(FUSED ? THREADS_FUSED : THREADS, 1)
    cond_kernel(const __grid_constant__ CUtensorMap tmApack, const __grid_constant__ CUtensorMap tmWc,
                const __grid_constant__ CUtensorMap tmR, const __grid_constant__ CUtensorMap tmE,
                const __grid_constant__ CUtensorMap tmWv, const __grid_constant__ CUtensorMap tmWg,
                const CondParams p, const VerifyStreamParams vp) {
  extern __shared__ uint8_t dsmem[];
  __shared__ __align__(8) uint64_t bar_full[STAGES];
  __shared__ __align__(8) uint64_t bar_empty[STAGES];
  __shared__ __align__(8) uint64_t bar_tfull[2];
  __shared__ __align__(8) uint64_t bar_tempty[2];
  __shared__ __align__(8) uint64_t bar_tile_full[TILE_SLOTS];
  __shared__ __align__(8) uint64_t bar_tile_empty[TILE_SLOTS];
  __shared__ int s_tile[TILE_SLOTS];
  __shared__ int s_rows[TILE_SLOTS];  // valid rows of the tile (FUSED)
  __shared__ uint32_t s_tmem;
  __shared__ volatile int s_abort;
  __shared__ VerifyStreamSmem vsm;

  constexpr int NST = FUSED ? STAGES_FUSED : STAGES;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int d = p.d;
  const int nt0 = d / 256, nt1 = d / 128;
  const int R = FUSED ? 0 : *(volatile const int32_t*)p.R;
  const int tiles_m = (R + BM - 1) / BM;
  const int T0 = FUSED ? 0 : (p.do_correct ? tiles_m * nt0 : 0);
  const int T = FUSED ? 0 : T0 + (p.do_gate ? tiles_m * nt1 : 0);
  if (!FUSED && T == 0) return;  // nothing to condition
  uint32_t* tile_queue = p.sync + kSyncTileQueue;
  uint32_t* gemv_next = p.sync + kSyncGemvNext;
  uint32_t* gemv_done = p.sync + kSyncGemvDone;
  uint32_t* block_done = p.block_done;
  const bool need_ge = p.do_gate && !p.e_dense;

  if (tid == 0) {
    s_abort = 0;
    for (int s = 0; s < NST; ++s) {
      mbar_init(smem_u32(&bar_full[s]), 1);
      mbar_init(smem_u32(&bar_empty[s]), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(smem_u32(&bar_tfull[a]), 1);
      mbar_init(smem_u32(&bar_tempty[a]), 4);  // one arrival per epilogue warp
    }
    for (int a = 0; a < TILE_SLOTS; ++a) {
      mbar_init(smem_u32(&bar_tile_full[a]), 1);
      mbar_init(smem_u32(&bar_tile_empty[a]), 5);  // MMA thread + four epilogue warps
    }
    if constexpr (FUSED) vs_init(vsm);
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    if (p.do_correct) {
      tma_prefetch_desc(&tmApack);
      tma_prefetch_desc(&tmWc);
    }
    if (p.do_gate) {
      tma_prefetch_desc(&tmR);
      tma_prefetch_desc(&tmWv);
      tma_prefetch_desc(&tmWg);
      if (p.e_dense) tma_prefetch_desc(&tmE);
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
  const int kb_half = d / BK;

  if (warp == 0) {
    // ---------------- tile scheduler + TMA producer ----------------
    if (lane == 0) {
      uint32_t it = 0;
      bool ok = true;
      for (uint32_t lt = 0;; ++lt) {
        const uint32_t slot = lt % TILE_SLOTS, sph = (lt / TILE_SLOTS) & 1u;
        int t, rows = BM, m0, n0;
        bool corr, done = false;
        if (!FUSED) {
          t = (int)atomicAdd(tile_queue, 1u);
          done = t >= T;
          corr = t < T0;
          const int tt = corr ? t : t - T0;
          m0 = (corr ? tt / nt0 : tt / nt1) * BM;
          n0 = corr ? (tt % nt0) * 256 : (tt % nt1) * 128;
        } else {
          // next valid tile of the phased queue
          for (;;) {
            t = (int)atomicAdd(tile_queue, 1u);
            const int q = t / (nt0 + nt1), r = t % (nt0 + nt1);
            corr = r < nt0;
            const int m = corr ? q : q - kGateLag;
            n0 = corr ? r * 256 : (r - nt0) * 128;
            m0 = m * BM;
            if (m < 0) continue;  // gate slots of the first phases
            if (m >= p.max_blocks) {  // beyond any possible packed row
              if (!corr) {
                done = true;
                break;
              }
              continue;
            }
            // wait until block m is complete, or verification is over
            int state = 0;  // 1 valid, 2 past the last block
            const unsigned long long t_start = global_ns();
            for (uint32_t it2 = 0; state == 0; ++it2) {
              const uint32_t ready = ld_acquire(p.block_ready + m);
              if (ready >= (uint32_t)BM) {
                state = 1;
              } else if (ld_acquire(p.sync + kSyncSeqDone) >= (uint32_t)vp.B) {
                const int Rf = (int)ld_acquire(p.sync + kSyncRowCount);
                if (m0 >= Rf) state = 2;
                else if (ready >= (uint32_t)(Rf - m0)) { state = 1; rows = Rf - m0; }
              }
              if (state == 0) {
                __nanosleep(128);
                if ((it2 & 63u) == 63u && (s_abort || global_ns() - t_start > kWaitLimitNs)) break;
              }
            }
            if (state == 0) {
              ok = false;
              break;
            }
            if (state == 2) {
              // Block m is past the last packed row.  Gate tiles come in
              // increasing block order, so a gate tile past the end means
              // nothing valid is left; a correction tile past the end may
              // still be followed by valid gate tiles of earlier blocks.
              if (!corr) {
                done = true;
                break;
              }
              continue;
            }
            break;
          }
          if (!ok) break;
        }
        if (!mbar_wait_bounded(smem_u32(&bar_tile_empty[slot]), sph ^ 1u, &s_abort)) {
          ok = false;
          break;
        }
        s_tile[slot] = done ? -1 : t;
        s_rows[slot] = rows;
        mbar_arrive(smem_u32(&bar_tile_full[slot]));
        if (done) break;
        const int nkb = corr ? 2 * kb_half : kb_half + (p.e_dense ? kb_half : 0);
        if (!corr && p.do_correct) {
          // the r rows of this block are written by the correction epilogues
          if (!wait_counter(block_done + m0 / BM, (uint32_t)(4 * nt0), &s_abort)) {
            ok = false;
            break;
          }
          fence_proxy_async_global();
        }
        for (int kb = 0; kb < nkb; ++kb, ++it) {
          const uint32_t s = it % NST, ph = (it / NST) & 1u;
          if (!mbar_wait_bounded(smem_u32(&bar_empty[s]), ph ^ 1u, &s_abort)) {
            ok = false;
            break;
          }
          const uint32_t a_dst = base + s * STAGE_BYTES, b_dst = a_dst + A_BYTES;
          const uint32_t full = smem_u32(&bar_full[s]);
          if (corr) {
            mbar_arrive_expect_tx(full, A_BYTES + B_BYTES);
            tma_load_2d(a_dst, &tmApack, kb * BK, m0, full);  // [m; u] rows
            tma_load_2d(b_dst, &tmWc, kb * BK, n0, full);     // W_c rows n0..n0+255
          } else if (kb < kb_half) {
            mbar_arrive_expect_tx(full, A_BYTES + B_BYTES);
            tma_load_2d(a_dst, &tmR, kb * BK, m0, full);                     // r rows
            tma_load_2d(b_dst, &tmWv, kb * BK, n0, full);                    // W_v rows
            tma_load_2d(b_dst + B_BYTES / 2, &tmWg, d + kb * BK, n0, full);  // W_g[:, d:2d] rows
          } else {
            mbar_arrive_expect_tx(full, A_BYTES + B_BYTES / 2);
            tma_load_2d(a_dst, &tmE, (kb - kb_half) * BK, m0, full);                     // e rows
            tma_load_2d(b_dst + B_BYTES / 2, &tmWg, (kb - kb_half) * BK, n0, full);  // W_g[:, :d]
          }
        }
        if (!ok) break;
      }
      if (!ok) {
        raise_abort(&s_abort, p.status);
        volatile int never = 0;  // drain this CTA's own copies still in flight
        const uint32_t first = it > NST ? it - NST : 0;
        for (uint32_t k = first; k < it; ++k)
          mbar_wait_bounded(smem_u32(&bar_full[k % NST]), (k / NST) & 1u, &never);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      uint32_t it = 0;
      bool ok = true;
      for (uint32_t lt = 0;; ++lt) {
        const uint32_t slot = lt % TILE_SLOTS, sph = (lt / TILE_SLOTS) & 1u;
        if (!mbar_wait_bounded(smem_u32(&bar_tile_full[slot]), sph, &s_abort)) {
          ok = false;
          break;
        }
        const int t = s_tile[slot];
        mbar_arrive(smem_u32(&bar_tile_empty[slot]));
        if (t < 0) break;
        const bool corr = FUSED ? (t % (nt0 + nt1)) < nt0 : t < T0;
        const int nkb = corr ? 2 * kb_half : kb_half + (p.e_dense ? kb_half : 0);
        const uint32_t acc = lt & 1u, aph = (lt >> 1) & 1u;
        if (!mbar_wait_bounded(smem_u32(&bar_tempty[acc]), aph ^ 1u, &s_abort)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem + acc * ACC_COLS;
        for (int kb = 0; kb < nkb; ++kb, ++it) {
          const uint32_t s = it % NST, ph = (it / NST) & 1u;
          if (!mbar_wait_bounded(smem_u32(&bar_full[s]), ph, &s_abort)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a_base = base + s * STAGE_BYTES, b_base = a_base + A_BYTES;
          const bool e_part = !corr && kb >= kb_half;
          // K16 steps advance the start address by 32 bytes: + 2 in the descriptor's address field
          const uint64_t adesc0 = sw128_kmajor_desc(a_base);
          const uint64_t bdesc0 = sw128_kmajor_desc(e_part ? b_base + B_BYTES / 2 : b_base);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            if (!e_part)
              tc_mma_bf16(d_tmem, adesc0 + 2u * k, bdesc0 + 2u * k, IDESC_N256, (kb > 0 || k > 0) ? 1u : 0u);
            else
              tc_mma_bf16(d_tmem + 128u, adesc0 + 2u * k, bdesc0 + 2u * k, IDESC_N128, 1u);
          }
          tc_commit(smem_u32(&bar_empty[s]));
        }
        tc_commit(smem_u32(&bar_tfull[acc]));  // accumulator ready (also after a failure)
        if (!ok) break;
      }
      if (!ok) raise_abort(&s_abort, p.status);
    }
    __syncwarp();
  } else if (FUSED && warp == 3) {
    // ---------------- logits stream into the verification ring ----------------
    if (lane == 0) vs_producer(vp, vsm, base + NST * STAGE_BYTES, &s_abort);
    __syncwarp();
  } else if (FUSED && warp == 2) {
    // ---------------- sequence finaliser (bulk copies through staging) ----------------
    vs_finalizer(vp, vsm, base + NST * STAGE_BYTES + kRingBufs * kChunkBytes, blockIdx.x, gridDim.x, lane, &s_abort);
  } else if (warp == 2 || warp == 3) {
    // ---------------- W_g[:, :d] e for a broadcast e (idle warps) ----------------
    if (need_ge) gate_bias_rows(p, d, lane, gemv_next, gemv_done);
  } else if (warp >= 16) {
    // ---------------- verification bookkeeping (FUSED only) ----------------
    if constexpr (FUSED)
      if (lane == 0) vs_bookkeeper(vp, vsm, &s_abort);
    __syncwarp();
  } else if (warp >= 8) {
    // ---------------- verification (FUSED only: warps 8-15) ----------------
    if constexpr (FUSED)
      vs_consumer(vp, vsm, reinterpret_cast<const uint4*>(dsmem + (base + NST * STAGE_BYTES - smem_u32(dsmem))),
                  warp - 8, lane, &s_abort);
  } else if (warp >= 4) {
    // ---------------- epilogue ----------------
    const int q = (warp - 4) * 32 + lane;  // tile row = TMEM lane
    const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
    // In the fused kernel the epilogue warps have nothing to do until the
    // first rows are packed: they compute W_g[:, :d] e meanwhile.
    if (FUSED && need_ge) gate_bias_rows(p, d, lane, gemv_next, gemv_done);
    bool have_ge = !need_ge;
    for (uint32_t lt = 0;; ++lt) {
      const uint32_t slot = lt % TILE_SLOTS, sph = (lt / TILE_SLOTS) & 1u;
      bool ok = warp_wait(smem_u32(&bar_tile_full[slot]), sph, &s_abort);
      if (!ok) {
        if (lane == 0) raise_abort(&s_abort, p.status);
        break;
      }
      const int t = s_tile[slot];
      const int tile_rows = s_rows[slot];
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&bar_tile_empty[slot]));
      if (t < 0) break;
      bool corr;
      int m0, n0;
      if (FUSED) {
        const int q2 = t / (nt0 + nt1), r = t % (nt0 + nt1);
        corr = r < nt0;
        m0 = (corr ? q2 : q2 - kGateLag) * BM;
        n0 = corr ? r * 256 : (r - nt0) * 128;
      } else {
        corr = t < T0;
        const int tt = corr ? t : t - T0;
        m0 = (corr ? tt / nt0 : tt / nt1) * BM;
        n0 = corr ? (tt % nt0) * 256 : (tt % nt1) * 128;
      }
      const uint32_t acc = lt & 1u, aph = (lt >> 1) & 1u;
      ok = warp_wait(smem_u32(&bar_tfull[acc]), aph, &s_abort);
      tc_fence_after();
      if (!ok) {
        if (lane == 0) raise_abort(&s_abort, p.status);
        break;
      }
      if (s_abort) break;
      if (!corr && !have_ge) {
        int got = 1;
        if (lane == 0) got = wait_counter(gemv_done, (uint32_t)d, &s_abort) ? 1 : 0;
        got = __shfl_sync(0xFFFFFFFFu, got, 0);
        if (!got) {
          if (lane == 0) raise_abort(&s_abort, p.status);
          break;
        }
        have_ge = true;
      }
      const int g = m0 + q;
      const bool valid = FUSED ? q < tile_rows : g < R;
      const uint32_t taddr = tmem + acc * ACC_COLS + lane_base;
      if (corr) {
        epilogue_correction(p, taddr, g, valid, n0, d);
        if (p.do_gate) {
          // Publish this warp's 32 rows of the (row block, column block) of r
          // to the gate tiles: one count per epilogue warp, no wait.
          __threadfence();
          fence_proxy_async_global();
          __syncwarp();
          if (lane == 0) atomicAdd(block_done + m0 / BM, 1u);
        }
      } else {
        epilogue_gate(p, taddr, g, valid, n0, d);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&bar_tempty[acc]));
    }
    // out of tiles: help finish W_g[:, :d] e (the rows left on the counter)
    if (!FUSED && need_ge && !s_abort) gate_bias_rows(p, d, lane, gemv_next, gemv_done);
  }
  // ---------------- teardown ----------------
  tc_fence_before();
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

// ---------------------------------------------------------------------------
// CTA-pair projections: tcgen05.mma.cta_group::2, M = 256 over two SMs
// ---------------------------------------------------------------------------
// The same tiles as cond_kernel<false> with twice the rows: a cluster of two
// CTAs takes a 256-row pair tile, each CTA staging its own 128 rows of A and
// half of the N = 256 weight tile (correction: W_c rows n0.. and n0+128..;
// gate: the W_v rows in the leader, the matching W_g[:, d:2d] rows in the
// follower).  A stage is 128 deep in K (two 64-element swizzle boxes per
// operand, 64 KB per SM): three stages fit.  Each stage costs a fixed
// handshake (full wait, commit, empty wait, copies issued), which deeper
// stages amortise: at B = 256 the kernel took 251.9 us with seven 64-deep
// stages, 245.3 us with three 128-deep ones, 283 us with two 192-deep ones
// and 434 us with fourteen 32-deep ones.
// The leader's MMA thread issues M256 N256 K16 MMAs that read both CTAs'
// shared memory and accumulate into both CTAs' tensor memory (each CTA's
// TMEM lanes are its own 128 rows); its commits arrive on both CTAs'
// barriers (multicast).  Stage-full barriers live in the leader and count the
// bytes of both CTAs' copies.  The leader takes tiles from the global queue
// and hands each to the follower through the follower's shared memory.  A
// broadcast e only (per-position e takes cond_kernel).  Every wait is bounded.
constexpr int PSTAGES = 3;
constexpr int P_THREADS = 256;
constexpr int PBK = 2 * BK;                      // k-block depth of a stage: two swizzle boxes
constexpr int P_BOX_BYTES = 128 * BK * 2;        // 16 KB: one 128-row, 64-element box
constexpr int P_A_BYTES = 2 * P_BOX_BYTES;       // 32 KB: this CTA's 128 rows
constexpr int P_B_BYTES = 2 * P_BOX_BYTES;       // 32 KB: this CTA's half of the weight tile
constexpr int P_STAGE_BYTES = P_A_BYTES + P_B_BYTES;
constexpr int P_SMEM_BYTES = PSTAGES * P_STAGE_BYTES + 1024;  // + slack for 1024-B alignment
constexpr uint32_t IDESC_M256_N256 = idesc_bf16_f32(256, 256);
// Pair blocks (256 packed rows) per group of the tile order: inside a group
// the weight tile is the outer index, so the pairs that start together share
// weight tiles as well as row blocks (measured: 260 against 264 us for
// row-block-major order at config 5).
constexpr int kGroupBlocks = 4;
constexpr int P_TILE_SLOTS = 3;  // tile indices in flight: the leader publishes one tile ahead

__global__ void __launch_bounds__(P_THREADS, 1)
    cond_pair_kernel(const __grid_constant__ CUtensorMap tmApack, const __grid_constant__ CUtensorMap tmWc,
                     const __grid_constant__ CUtensorMap tmR, const __grid_constant__ CUtensorMap tmWv,
                     const __grid_constant__ CUtensorMap tmWg, const CondParams p) {
  extern __shared__ uint8_t dsmem[];
  __shared__ __align__(8) uint64_t bar_full[PSTAGES];             // leader: both CTAs' bytes of a stage
  __shared__ __align__(8) uint64_t bar_empty[PSTAGES];            // stage free (leader's commit, both CTAs)
  __shared__ __align__(8) uint64_t bar_tfull[2];                  // accumulator ready (both CTAs)
  __shared__ __align__(8) uint64_t bar_tempty[2];                 // leader: eight epilogue warps done
  __shared__ __align__(8) uint64_t bar_tile_full[P_TILE_SLOTS];   // tile index published (both CTAs)
  __shared__ __align__(8) uint64_t bar_tile_empty[P_TILE_SLOTS];  // leader: ten readers done
  __shared__ int s_tile[P_TILE_SLOTS];
  __shared__ uint32_t s_tmem;
  __shared__ volatile int s_abort;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t rank = cluster_rank();
  const bool leader = rank == 0;  // issues the pair's MMAs and runs the tile queue
  const int d = p.d;
  const int nt0 = d / 256, nt1 = d / 128;
  pdl_launch_dependents();
  uint32_t* tile_queue = p.sync + kSyncTileQueue;
  uint32_t* gemv_next = p.sync + kSyncGemvNext;
  uint32_t* gemv_done = p.sync + kSyncGemvDone;
  uint32_t* block_done = p.block_done;
  const bool need_ge = p.do_gate;  // broadcast e

  if (tid == 0) {
    s_abort = 0;
    for (int s = 0; s < PSTAGES; ++s) {
      mbar_init(smem_u32(&bar_full[s]), 1);  // the leader's expect_tx
      mbar_init(smem_u32(&bar_empty[s]), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(smem_u32(&bar_tfull[a]), 1);
      mbar_init(smem_u32(&bar_tempty[a]), 8);  // four epilogue warps in each CTA
    }
    for (int a = 0; a < P_TILE_SLOTS; ++a) {
      mbar_init(smem_u32(&bar_tile_full[a]), 1);
      mbar_init(smem_u32(&bar_tile_empty[a]), 10);  // MMA + 4 epilogue warps; producer + 4 epilogue warps
    }
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    if (p.do_correct) {
      tma_prefetch_desc(&tmApack);
      tma_prefetch_desc(&tmWc);
    }
    if (p.do_gate) {
      tma_prefetch_desc(&tmR);
      tma_prefetch_desc(&tmWv);
      tma_prefetch_desc(&tmWg);
    }
  }
  if (warp == 2) {
    tmem_alloc_pair(smem_u32(&s_tmem), TMEM_COLS);  // one warp of each CTA of the pair
    tmem_relinquish_pair();
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // both CTAs' barriers initialised before any remote arrive
  tc_fence_after();
  const uint32_t tmem = s_tmem;
  const uint32_t base = (smem_u32(dsmem) + 1023u) & ~1023u;
  const int kb_half = d / PBK;
  // The set-up above may overlap the end of the previous kernel (programmatic
  // dependent launch).  R, the packed rows and the row map are its outputs:
  // every role that reads them waits here first.  The gate-bias GEMV (warps
  // 2-3) reads only the inputs and starts at once.  With R = 0 the queue's
  // first claim already ends every role.
  int R = 0, T0 = 0, T1 = 0, X = 0, T = 0, pairs_m = 0;
  if (warp != 2 && warp != 3) {
    pdl_wait();
    R = *(volatile const int32_t*)p.R;
    pairs_m = (R + 2 * BM - 1) / (2 * BM);
    T0 = p.do_correct ? pairs_m * nt0 : 0;
    T1 = p.do_gate ? pairs_m * nt1 : 0;
    // the last wave: work units (a gate tile's worth of MMAs) beyond the
    // whole waves of the pairs
    const int last_wave = (2 * T0 + T1) % (int)(gridDim.x / 2);
    X = last_wave <= p.split_max ? min(last_wave, T1) : 0;
    T = T0 + T1 + X;
  }
  // Tile t: correction tiles first, then gate tiles; within each kind, groups
  // of kGroupBlocks pair blocks with the weight tile outer inside a group.
  // When the last wave of the queue would keep only a few pairs busy (at
  // most split_max tiles), its X gate tiles come as two K halves each (2X
  // queue entries, the halves of a tile next to each other), so that twice
  // as many pairs share it.  At B = 256 (12 pair blocks, 768 units on 76
  // pairs, 8 in the last wave) the kernel went from 245.8-247.9 to
  // 241.7-243.8 us.  Splitting 16 or 38 tiles whatever the last wave made
  // B = 128 slower (141.4 -> 159.8 us), where splitting 4 or 8 left it
  // unchanged.
  struct Tile {
    bool corr;
    int m0, n0;    // this CTA's first row; first output column (correction) or feature (gate)
    int kb0, nkb;  // k-blocks of PBK
    int split;     // -1, or the split tile (0..X-1) whose K half `half` this is
    int half;
  };
  auto decode = [&](int t) {
    Tile x;
    x.corr = t < T0;
    int tt = x.corr ? t : t - T0;
    x.kb0 = 0;
    x.nkb = x.corr ? 2 * kb_half : kb_half;
    x.split = -1;
    x.half = 0;
    if (!x.corr && tt >= T1 - X) {
      const int j = tt - (T1 - X);
      x.split = j >> 1;
      x.half = j & 1;
      tt = T1 - X + x.split;
      x.nkb = kb_half / 2;
      x.kb0 = x.half * x.nkb;
    }
    const int nt = x.corr ? nt0 : nt1;
    const int g = tt / (kGroupBlocks * nt), w = tt - g * kGroupBlocks * nt;
    const int glen = min(kGroupBlocks, pairs_m - g * kGroupBlocks);
    const int pb = g * kGroupBlocks + w % glen;  // pair block
    x.m0 = pb * 2 * BM + (int)rank * BM;         // this CTA's rows
    x.n0 = (w / glen) * (x.corr ? 256 : 128);
    return x;
  };
  // the leader's barriers as seen from either CTA
  auto leader_addr = [&](const void* local) { return map_rank(smem_u32(local), 0); };

  if (warp == 0) {
    // ---------------- tile hand-off + TMA producer (both CTAs) ----------------
    if (lane == 0) {
      uint32_t it = 0;
      bool ok = true;
      // While more tiles remain than there are pairs, the leader publishes
      // tile lt + 1 (from the queue) before it loads tile lt, so the next
      // index is already waiting in both CTAs when their producers and the MMA
      // reach the tile switch; near the end of the queue it claims the next
      // tile at the switch, so that no pair holds a tile while others go idle.
      auto publish = [&](uint32_t l, int t) -> bool {
        const uint32_t slot = l % P_TILE_SLOTS, sph = (l / P_TILE_SLOTS) & 1u;
        if (!mbar_wait_cluster_bounded(smem_u32(&bar_tile_empty[slot]), sph ^ 1u, &s_abort)) return false;
        s_tile[slot] = t;
        st_remote_u32(map_rank(smem_u32(&s_tile[slot]), 1), (uint32_t)t);
        mbar_arrive(smem_u32(&bar_tile_full[slot]));
        mbar_arrive_remote(map_rank(smem_u32(&bar_tile_full[slot]), 1));  // release orders the store
        return true;
      };
      auto dequeue = [&]() {
        const int t = (int)atomicAdd(tile_queue, 1u);
        return t < T ? t : -1;
      };
      const int pairs = (int)(gridDim.x / 2);
      if (leader && !publish(0, dequeue())) ok = false;
      for (uint32_t lt = 0; ok; ++lt) {
        const uint32_t slot = lt % P_TILE_SLOTS, sph = (lt / P_TILE_SLOTS) & 1u;
        int t;
        bool ahead = false;  // the leader published tile lt + 1 already
        if (leader) {
          t = s_tile[slot];  // published before
          ahead = t >= 0 && t + pairs < T;
          if (ahead && !publish(lt + 1, dequeue())) {
            ok = false;
            break;
          }
        } else {
          if (!mbar_wait_cluster_bounded(smem_u32(&bar_tile_full[slot]), sph, &s_abort)) {
            ok = false;
            break;
          }
          t = s_tile[slot];
          mbar_arrive_remote(leader_addr(&bar_tile_empty[slot]));
        }
        if (t < 0) break;
        const Tile x = decode(t);
        const bool corr = x.corr;
        const int m0 = x.m0, n0 = x.n0;
        if (!corr && p.do_correct) {
          // the r rows of this CTA's block are written by the correction epilogues
          if (!wait_counter(block_done + m0 / BM, (uint32_t)(4 * nt0), &s_abort)) {
            ok = false;
            break;
          }
          fence_proxy_async_global();
        }
        for (int kb = x.kb0; kb < x.kb0 + x.nkb; ++kb, ++it) {
          const uint32_t s = it % PSTAGES, ph = (it / PSTAGES) & 1u;
          if (!mbar_wait_bounded(smem_u32(&bar_empty[s]), ph ^ 1u, &s_abort)) {
            ok = false;
            break;
          }
          const uint32_t a_dst = base + s * P_STAGE_BYTES, b_dst = a_dst + P_A_BYTES;
          const uint32_t full = leader_addr(&bar_full[s]);
          if (leader) mbar_arrive_expect_tx(smem_u32(&bar_full[s]), 2 * P_STAGE_BYTES);  // both CTAs' bytes
          // [m; u] or r rows; this CTA's half of the weight tile: W_c rows n0..
          // (leader) or n0 + 128.. (follower), or the W_v rows (leader) and the
          // matching W_g[:, d:2d] rows (follower); each as two 64-element boxes
          const CUtensorMap* mb = corr ? &tmWc : (leader ? &tmWv : &tmWg);
          const int xb = (corr || leader) ? kb * PBK : d + kb * PBK;
          const int yb = corr ? n0 + (int)rank * 128 : n0;
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            tma_load_2d_pair(a_dst + (uint32_t)h * P_BOX_BYTES, corr ? &tmApack : &tmR, kb * PBK + h * BK, m0, full);
            tma_load_2d_pair(b_dst + (uint32_t)h * P_BOX_BYTES, mb, xb + h * BK, yb, full);
          }
        }
        if (!ok) break;
        if (leader && !ahead && !publish(lt + 1, dequeue())) ok = false;  // near the end: claim at the switch
      }
      if (!ok) {
        raise_abort(&s_abort, p.status);
        if (leader) {
          volatile int never = 0;  // wait for the copies in flight into the pair's stages
          const uint32_t first = it > PSTAGES ? it - PSTAGES : 0;
          for (uint32_t k = first; k < it; ++k)
            mbar_wait_bounded(smem_u32(&bar_full[k % PSTAGES]), (k / PSTAGES) & 1u, &never);
        }
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---------------- MMA issuer (leader) ----------------
    if (leader && lane == 0) {
      uint32_t it = 0;
      bool ok = true;
      for (uint32_t lt = 0;; ++lt) {
        const uint32_t slot = lt % P_TILE_SLOTS, sph = (lt / P_TILE_SLOTS) & 1u;
        if (!mbar_wait_bounded(smem_u32(&bar_tile_full[slot]), sph, &s_abort)) {
          ok = false;
          break;
        }
        const int t = s_tile[slot];
        mbar_arrive(smem_u32(&bar_tile_empty[slot]));
        if (t < 0) break;
        const int nkb = decode(t).nkb;
        const uint32_t acc = lt & 1u, aph = (lt >> 1) & 1u;
        if (!mbar_wait_cluster_bounded(smem_u32(&bar_tempty[acc]), aph ^ 1u, &s_abort)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem + acc * ACC_COLS;
        for (int kb = 0; kb < nkb; ++kb, ++it) {
          const uint32_t s = it % PSTAGES, ph = (it / PSTAGES) & 1u;
          if (!mbar_wait_bounded(smem_u32(&bar_full[s]), ph, &s_abort)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a_base = base + s * P_STAGE_BYTES, b_base = a_base + P_A_BYTES;
          // K16 steps advance the start address by 32 bytes (+ 2 in the
          // descriptor's address field) inside a box, by the box's 16 KB (+ 1024)
          // from the first box to the second
          const uint64_t adesc0 = sw128_kmajor_desc(a_base), bdesc0 = sw128_kmajor_desc(b_base);
#pragma unroll
          for (int k = 0; k < PBK / 16; ++k) {
            const uint64_t step = (uint64_t)((k / (BK / 16)) * (P_BOX_BYTES >> 4) + 2 * (k % (BK / 16)));
            tc_mma_pair(d_tmem, adesc0 + step, bdesc0 + step, IDESC_M256_N256, (kb > 0 || k > 0) ? 1u : 0u);
          }
          tc_commit_pair(smem_u32(&bar_empty[s]));  // stage free in both CTAs
        }
        tc_commit_pair(smem_u32(&bar_tfull[acc]));  // accumulator ready (also after a failure)
        if (!ok) break;
      }
      if (!ok) raise_abort(&s_abort, p.status);
    }
    __syncwarp();
  } else if (warp == 2 || warp == 3) {
    // ---------------- W_g[:, :d] e for the broadcast e (idle warps) ----------------
    if (need_ge) gate_bias_rows(p, d, lane, gemv_next, gemv_done);
  } else {
    // ---------------- epilogue (warps 4-7 of both CTAs) ----------------
    const int q = (warp - 4) * 32 + lane;  // tile row = TMEM lane
    const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
    bool have_ge = !need_ge;
    for (uint32_t lt = 0;; ++lt) {
      const uint32_t slot = lt % P_TILE_SLOTS, sph = (lt / P_TILE_SLOTS) & 1u;
      bool ok = warp_wait_cluster(smem_u32(&bar_tile_full[slot]), sph, &s_abort);
      if (!ok) {
        if (lane == 0) raise_abort(&s_abort, p.status);
        break;
      }
      const int t = s_tile[slot];
      __syncwarp();
      if (lane == 0) {
        if (leader) mbar_arrive(smem_u32(&bar_tile_empty[slot]));
        else mbar_arrive_remote(leader_addr(&bar_tile_empty[slot]));
      }
      if (t < 0) break;
      const Tile x = decode(t);
      const bool corr = x.corr;
      const int m0 = x.m0, n0 = x.n0;
      const uint32_t acc = lt & 1u, aph = (lt >> 1) & 1u;
      ok = warp_wait(smem_u32(&bar_tfull[acc]), aph, &s_abort);
      tc_fence_after();
      if (!ok) {
        if (lane == 0) raise_abort(&s_abort, p.status);
        break;
      }
      if (s_abort) break;
      if (!corr && !have_ge) {
        int got = 1;
        if (lane == 0) got = wait_counter(gemv_done, (uint32_t)d, &s_abort) ? 1 : 0;
        got = __shfl_sync(0xFFFFFFFFu, got, 0);
        if (!got) {
          if (lane == 0) raise_abort(&s_abort, p.status);
          break;
        }
        have_ge = true;
      }
      const int g = m0 + q;
      const bool valid = g < R;
      const uint32_t taddr = tmem + acc * ACC_COLS + lane_base;
      if (corr) {
        epilogue_correction(p, taddr, g, valid, n0, d);
        if (p.do_gate) {
          __threadfence();
          fence_proxy_async_global();
          __syncwarp();
          if (lane == 0) atomicAdd(block_done + m0 / BM, 1u);
        }
      } else if (x.split < 0) {
        epilogue_gate(p, taddr, g, valid, n0, d);
      } else {
        // A K half: this row's accumulator goes to the half's slot ([column][row]
        // per CTA, so that a warp's stores are contiguous); the warp that counts
        // second on the ticket of its 32 rows adds the other half's slot and
        // runs the epilogue.  Fence before the count, fence after it (the
        // last-arriver pattern): no wait on the other pair.
        const size_t slot_floats = (size_t)2 * BM * 128;
        float* own = p.split_part + ((size_t)(x.split * 2 + x.half) * 2 + rank) * slot_floats + q;
        const float* other = p.split_part + ((size_t)(x.split * 2 + (x.half ^ 1)) * 2 + rank) * slot_floats + q;
        for (int cc = 0; cc < 8; ++cc) {
          float c[32];
          tmem_ld_32cols(taddr + (uint32_t)(cc * 32), c);
#pragma unroll
          for (int i = 0; i < 32; ++i) __stcg(own + (cc * 32 + i) * 128, c[i]);
        }
        __threadfence();
        __syncwarp();
        uint32_t before = 0;
        if (lane == 0) {
          before = atomicAdd(p.split_ticket + x.split * 8 + (int)rank * 4 + (warp - 4), 1u);
          __threadfence();
        }
        before = __shfl_sync(0xFFFFFFFFu, before, 0);
        __syncwarp();
        if (before == 1u) epilogue_gate(p, taddr, g, valid, n0, d, other);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if (leader) mbar_arrive(smem_u32(&bar_tempty[acc]));
        else mbar_arrive_remote(leader_addr(&bar_tempty[acc]));
      }
    }
    // out of tiles: help finish W_g[:, :d] e (the rows left on the counter)
    if (need_ge && !s_abort) gate_bias_rows(p, d, lane, gemv_next, gemv_done);
  }
  // ---------------- teardown ----------------
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // the peer is done with this CTA's shared and tensor memory
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc_pair(tmem, TMEM_COLS);
  }
}

// One thread runs the pipelined kernels' bounded waits on a condition the
// caller controls (retrace_wait_selftest): kind 0 waits until *flag >= target
// (the counter wait), kind 1 for an mbarrier phase that completes only if
// target == 0 (the phase wait).  An expired wait sets the status flag, as in
// the kernels, and the kernel returns.
__global__ void wait_selftest_kernel(int kind, const uint32_t* flag, uint32_t target, uint32_t* status) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ volatile int s_abort;
  if (threadIdx.x != 0) return;
  s_abort = 0;
  bool ok;
  if (kind == 0) {
    ok = wait_counter(flag, target, &s_abort);
  } else {
    mbar_init(smem_u32(&bar), 1);
    fence_mbar_init();
    if (target == 0) mbar_arrive(smem_u32(&bar));  // phase 0 completes: the wait returns at once
    ok = mbar_wait_bounded(smem_u32(&bar), 0, &s_abort);
  }
  if (!ok) atomicOr(status, kFlagWaitTimeout);
}

// ---------------------------------------------------------------------------
// Small R (B (K-1) <= kSwapMaxRows conditioned rows): the weights on the M side
// ---------------------------------------------------------------------------
// With few rows the 256-row pair tiles are mostly padding and only d/256
// correction tiles exist, so a handful of SMs stream the weights.  Here the
// GEMMs run transposed: c^T = W_c [m; u]^T and [v; g_r]^T = [W_v; W_g,r] r^T,
// the weights as the A operand in 128-row tiles (M = 128, no padding), the
// rows as B in tiles of up to 256 (N = R rounded up to 16, read on the
// device), and the K range split so that one resident wave of CTAs streams
// the weights.  Each CTA writes its fp32 partial [split][row][feature]; a
// reduction kernel sums the splits in a fixed order (results repeat bit for
// bit) and applies the epilogue.
constexpr int SW_STAGES = 4;
constexpr int SW_THREADS = 256;

// How a GEMM of R rows is cut, the same in the GEMM and its reduction: N
// tiles of up to 256 rows, work = weight tiles x N tiles, each split `grid /
// work` ways along K (no empty split).
struct SwapPlan {
  int nrows, ntiles, work, splits, kb_split;
};
__device__ __forceinline__ SwapPlan swap_plan(int R, int mtiles, int nkb, int grid) {
  SwapPlan s;
  s.nrows = (R + 15) / 16 * 16;
  s.ntiles = (s.nrows + 255) / 256;
  s.work = mtiles * s.ntiles;
  int splits = s.work > 0 ? grid / s.work : 1;
  if (splits < 1) splits = 1;
  if (splits > nkb) splits = nkb;
  s.kb_split = (nkb + splits - 1) / splits;
  s.splits = (nkb + s.kb_split - 1) / s.kb_split;
  return s;
}

struct SwapParams {
  const int32_t* R;
  int nkb;        // k-blocks of the reduction
  int mtiles;     // 128-row weight tiles in all
  int mt_a;       // tiles taken from map A (the others from map A2)
  int a2_x0;      // column offset of map A2's operand (d: the r half of W_g)
  int box_n;      // rows of a B box (min(256, the largest R rounded to 16))
  uint32_t tmem_cols;
  uint32_t stage_stride;  // bytes per pipeline stage (A tile + B box, 1024-aligned)
  float* part;            // [splits][nrows][mtiles * 128]
  uint32_t* status;
};

__global__ void __launch_bounds__(SW_THREADS, 1)
    swap_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmA2,
                     const __grid_constant__ CUtensorMap tmB, const SwapParams p) {
  extern __shared__ uint8_t dsmem[];
  __shared__ __align__(8) uint64_t bar_full[SW_STAGES];
  __shared__ __align__(8) uint64_t bar_empty[SW_STAGES];
  __shared__ __align__(8) uint64_t bar_acc;
  __shared__ uint32_t s_tmem;
  __shared__ volatile int s_abort;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  pdl_launch_dependents();
  if (threadIdx.x == 0) {
    s_abort = 0;
    for (int s = 0; s < SW_STAGES; ++s) {
      mbar_init(smem_u32(&bar_full[s]), 1);
      mbar_init(smem_u32(&bar_empty[s]), 1);
    }
    mbar_init(smem_u32(&bar_acc), 1);
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmA2);
    tma_prefetch_desc(&tmB);
  }
  if (warp == 2) {
    tmem_alloc(smem_u32(&s_tmem), p.tmem_cols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s_tmem;
  const uint32_t base = (smem_u32(dsmem) + 1023u) & ~1023u;
  pdl_wait();  // R and the activation rows come from the previous kernels
  const int R = *(volatile const int32_t*)p.R;
  const SwapPlan pl = swap_plan(R, p.mtiles, p.nkb, (int)gridDim.x);
  const int c = blockIdx.x;
  const bool active = c < pl.work * pl.splits;
  const int sp = c % pl.splits, w = c / pl.splits;
  const int mt = w / (pl.ntiles > 0 ? pl.ntiles : 1), nt = w - mt * (pl.ntiles > 0 ? pl.ntiles : 1);
  const int kb0 = sp * pl.kb_split, kb1 = min(p.nkb, kb0 + pl.kb_split);
  const int tn = active ? min(256, pl.nrows - nt * 256) : 0;  // rows of this N tile (MMA N)

  if (!active) {
    // nothing to do: fall through to the teardown
  } else if (warp == 0) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      const bool second = mt >= p.mt_a;
      const CUtensorMap* ma = second ? &tmA2 : &tmA;
      const int ay = (second ? mt - p.mt_a : mt) * 128, ax0 = second ? p.a2_x0 : 0;
      const uint32_t tx = (uint32_t)(BM * BK * 2) + (uint32_t)p.box_n * BK * 2;
      int kb = kb0;
      for (; kb < kb1; ++kb) {
        const int i = kb - kb0;
        const uint32_t s = (uint32_t)(i % SW_STAGES), ph = (uint32_t)((i / SW_STAGES) & 1);
        if (!mbar_wait_bounded(smem_u32(&bar_empty[s]), ph ^ 1u, &s_abort)) break;
        const uint32_t a_dst = base + s * p.stage_stride, b_dst = a_dst + (uint32_t)(BM * BK * 2);
        mbar_arrive_expect_tx(smem_u32(&bar_full[s]), tx);
        tma_load_2d(a_dst, ma, ax0 + kb * BK, ay, smem_u32(&bar_full[s]));
        tma_load_2d(b_dst, &tmB, kb * BK, nt * 256, smem_u32(&bar_full[s]));
      }
      if (kb < kb1) {  // a wait expired: flag it, let the copies in flight land
        raise_abort(&s_abort, p.status);
        volatile int never = 0;
        const int first = kb - kb0 > SW_STAGES ? kb - kb0 - SW_STAGES : 0;
        for (int i = first; i < kb - kb0; ++i)
          mbar_wait_bounded(smem_u32(&bar_full[i % SW_STAGES]), (uint32_t)((i / SW_STAGES) & 1), &never);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16_f32(128, tn);
      bool ok = true;
      for (int kb = kb0; kb < kb1; ++kb) {
        const int i = kb - kb0;
        const uint32_t s = (uint32_t)(i % SW_STAGES), ph = (uint32_t)((i / SW_STAGES) & 1);
        if (!mbar_wait_bounded(smem_u32(&bar_full[s]), ph, &s_abort)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t a_base = base + s * p.stage_stride, b_base = a_base + (uint32_t)(BM * BK * 2);
        const uint64_t adesc0 = sw128_kmajor_desc(a_base), bdesc0 = sw128_kmajor_desc(b_base);
#pragma unroll
        for (int k = 0; k < BK / 16; ++k)
          tc_mma_bf16(tmem, adesc0 + 2u * k, bdesc0 + 2u * k, idesc, (i > 0 || k > 0) ? 1u : 0u);
        tc_commit(smem_u32(&bar_empty[s]));
      }
      tc_commit(smem_u32(&bar_acc));  // accumulator ready (also after a failure)
      if (!ok) raise_abort(&s_abort, p.status);
    }
    __syncwarp();
  } else if (warp >= 4) {
    // ---------------- epilogue: the partial of this (weight tile, N tile, split) ----------------
    const int q = (warp - 4) * 32 + lane;  // weight row of the tile = TMEM lane
    const bool ok = warp_wait(smem_u32(&bar_acc), 0u, &s_abort);
    tc_fence_after();
    if (ok && !s_abort) {
      const uint32_t taddr = tmem + ((uint32_t)((warp & 3) * 32) << 16);
      const long long mtot = (long long)p.mtiles * 128;
      float* out = p.part + ((long long)sp * pl.nrows + nt * 256) * mtot + mt * 128 + q;
      for (int c0 = 0; c0 < tn; c0 += 32) {
        float v[32];
        tmem_ld_32cols(taddr + (uint32_t)c0, v);
#pragma unroll
        for (int j = 0; j < 32; ++j)
          if (c0 + j < tn) out[(long long)(c0 + j) * mtot] = v[j];  // 32 lanes: 128 contiguous bytes
      }
    } else if (!ok && lane == 0) {
      raise_abort(&s_abort, p.status);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, p.tmem_cols);
  }
}

struct SwapReduceParams {
  int d;
  const int32_t* R;
  // the GEMM's cut (swap_plan): weight tiles, k-blocks, grid
  int mtiles, nkb, grid;
  const float* part;  // [splits][nrows][mtiles * 128]
  // correction: r = m + beta * c
  const __nv_bfloat16* apack;  // m = the first d columns of each packed row
  float beta;
  __nv_bfloat16* r_out;
  int compact_out;
  // gate: e~ = e + v * sigmoid(g_r + ge)
  const __nv_bfloat16* e;
  const float* ge;
  __nv_bfloat16* e_out;
  const int32_t* rowmap;
  // W_g[:, :d] e for a broadcast e, before the wait (it reads inputs only)
  int do_gemv;
  CondParams gemv;
  uint32_t* gemv_next;
  uint32_t* gemv_done;
};

// r rows of the packed correction (Eq. 7): eight features per thread; the
// splits summed in order.  Before it waits for the correction GEMM, every
// warp takes rows of the gate-bias GEMV W_g[:, :d] e, which thereby overlaps
// the GEMM.
__global__ void __launch_bounds__(256) swap_reduce_correction_kernel(const SwapReduceParams p) {
  pdl_launch_dependents();
  if (p.do_gemv) gate_bias_rows(p.gemv, p.d, threadIdx.x & 31, p.gemv_next, p.gemv_done);
  pdl_wait();
  const int R = *(volatile const int32_t*)p.R;
  const SwapPlan pl = swap_plan(R, p.mtiles, p.nkb, p.grid);
  const int d = p.d, vpr = d / 8;
  const long long n_units = (long long)R * vpr;
  for (long long u = blockIdx.x * (long long)blockDim.x + threadIdx.x; u < n_units;
       u += (long long)gridDim.x * blockDim.x) {
    const int g = (int)(u / vpr), n = (int)(u - (long long)g * vpr) * 8;
    float c[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) c[j] = 0.f;
    for (int s = 0; s < pl.splits; ++s) {
      const float4* src = reinterpret_cast<const float4*>(p.part + ((long long)s * pl.nrows + g) * d + n);
      const float4 x0 = __ldcg(src), x1 = __ldcg(src + 1);
      c[0] += x0.x; c[1] += x0.y; c[2] += x0.z; c[3] += x0.w;
      c[4] += x1.x; c[5] += x1.y; c[6] += x1.z; c[7] += x1.w;
    }
    const uint4 mw = __ldcg(reinterpret_cast<const uint4*>(p.apack + (long long)g * 2 * d + n));
    const uint32_t mwords[4] = {mw.x, mw.y, mw.z, mw.w};
    uint32_t o[4];
#pragma unroll
    for (int w = 0; w < 4; ++w)
      o[w] = pack_bf16x2(bf16_lo(mwords[w]) + p.beta * c[2 * w], bf16_hi(mwords[w]) + p.beta * c[2 * w + 1]);
    const long long orow = p.compact_out ? g : __ldcg(p.rowmap + g);
    *reinterpret_cast<uint4*>(p.r_out + orow * d + n) = make_uint4(o[0], o[1], o[2], o[3]);
  }
}

// W_g[:, :d] e alone (a gate-only call: no correction kernel to overlap it
// with), by the same per-row code, so the bits match the correction path's.
__global__ void __launch_bounds__(256) swap_gemv_kernel(const SwapReduceParams p) {
  pdl_launch_dependents();
  gate_bias_rows(p.gemv, p.d, threadIdx.x & 31, p.gemv_next, p.gemv_done);
  // Complete only after the previous kernel: the next kernel's programmatic
  // wait, which covers this kernel alone, then covers that one too.  One CTA
  // waiting is enough (the grid completes with its last CTA); the others
  // leave and free their SM for the next kernel.
  if (blockIdx.x == 0) pdl_wait();
}

// e~ rows of the gated fusion (Eq. 8), broadcast e: v in features 0..d-1 of
// the partials, the r half of the gate in d..2d-1.
__global__ void __launch_bounds__(256) swap_reduce_gate_kernel(const SwapReduceParams p) {
  pdl_launch_dependents();
  pdl_wait();
  const int R = *(volatile const int32_t*)p.R;
  const SwapPlan pl = swap_plan(R, p.mtiles, p.nkb, p.grid);
  const int d = p.d, vpr = d / 8;
  const long long n_units = (long long)R * vpr;
  for (long long u = blockIdx.x * (long long)blockDim.x + threadIdx.x; u < n_units;
       u += (long long)gridDim.x * blockDim.x) {
    const int g = (int)(u / vpr), n = (int)(u - (long long)g * vpr) * 8;
    float v[8], gt[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) v[j] = gt[j] = 0.f;
    for (int s = 0; s < pl.splits; ++s) {
      const float* row = p.part + ((long long)s * pl.nrows + g) * 2 * d;
      const float4* vs = reinterpret_cast<const float4*>(row + n);
      const float4* gs = reinterpret_cast<const float4*>(row + d + n);
      const float4 v0 = __ldcg(vs), v1 = __ldcg(vs + 1), g0 = __ldcg(gs), g1 = __ldcg(gs + 1);
      v[0] += v0.x; v[1] += v0.y; v[2] += v0.z; v[3] += v0.w;
      v[4] += v1.x; v[5] += v1.y; v[6] += v1.z; v[7] += v1.w;
      gt[0] += g0.x; gt[1] += g0.y; gt[2] += g0.z; gt[3] += g0.w;
      gt[4] += g1.x; gt[5] += g1.y; gt[6] += g1.z; gt[7] += g1.w;
    }
    const float4 b0 = __ldcg(reinterpret_cast<const float4*>(p.ge + n));
    const float4 b1 = __ldcg(reinterpret_cast<const float4*>(p.ge + n) + 1);
    gt[0] += b0.x; gt[1] += b0.y; gt[2] += b0.z; gt[3] += b0.w;
    gt[4] += b1.x; gt[5] += b1.y; gt[6] += b1.z; gt[7] += b1.w;
    const uint4 ew = __ldg(reinterpret_cast<const uint4*>(p.e + n));
    const uint32_t ewords[4] = {ew.x, ew.y, ew.z, ew.w};
    uint32_t o[4];
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const float s0 = fast_sigmoid(gt[2 * w]), s1 = fast_sigmoid(gt[2 * w + 1]);
      o[w] = pack_bf16x2(bf16_lo(ewords[w]) + v[2 * w] * s0, bf16_hi(ewords[w]) + v[2 * w + 1] * s1);
    }
    const long long orow = __ldcg(p.rowmap + g);
    *reinterpret_cast<uint4*>(p.e_out + orow * d + n) = make_uint4(o[0], o[1], o[2], o[3]);
  }
}

// ---------------------------------------------------------------------------
// Small R in one N tile (at most 256 rows): split-K clusters, no reduction launch
// ---------------------------------------------------------------------------
// The S K-splits of one weight tile run as one cluster of S CTAs.  Each CTA
// accumulates its k-range in TMEM as swap_gemm_kernel does, moves the fp32
// partial into its own shared memory (the drained pipeline stages), and after
// a cluster barrier sums its slice of the rows over the S partials through
// distributed shared memory, in rank order (results repeat bit for bit), and
// applies the epilogue: r = m + beta c (Eq. 7) for the correction tiles of
// W_c, or the gated fusion e~ = e + v sigmoid(g_r + W_g[:, :d] e) (Eq. 8)
// for the gate tiles, whose 128 weight rows stack 64 rows of W_v over the
// same 64 rows of W_g[:, d:2d] (v and g_r of a feature in TMEM lanes f and
// 64 + f).  Nothing goes through global partials and no reduction kernel
// follows.  The partial is stored row-major ([row][feature]) so that both
// the TMEM drain and the cluster's reads move whole 128- and 256-byte rows.
struct SwapClusterParams {
  const int32_t* R;
  int d;
  int nkb;     // 64-deep k-blocks of the GEMM
  int S;       // K splits = cluster size
  int gate;    // 0: correction tiles of W_c (128 features); 1: stacked [W_v; W_g,r] tiles (64 features)
  int tile_n;  // rows of the B box (the largest R rounded to 16, at most 256)
  uint32_t tmem_cols;
  uint32_t stage_stride;
  // correction epilogue
  const __nv_bfloat16* apack;  // m = the first d columns of each packed row
  float beta;
  __nv_bfloat16* r_out;
  int compact_out;
  // gate epilogue (broadcast e; ge = W_g[:, :d] e, complete before this launch)
  const __nv_bfloat16* e;
  const float* ge;
  __nv_bfloat16* e_out;
  const int32_t* rowmap;
  uint32_t* status;
};

__global__ void __launch_bounds__(SW_THREADS, 1)
    swap_cluster_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmA2,
                        const __grid_constant__ CUtensorMap tmB, const SwapClusterParams p) {
  extern __shared__ uint8_t dsmem[];
  __shared__ __align__(8) uint64_t bar_full[SW_STAGES];
  __shared__ __align__(8) uint64_t bar_empty[SW_STAGES];
  __shared__ __align__(8) uint64_t bar_acc;
  __shared__ uint32_t s_tmem;
  __shared__ volatile int s_abort;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int S = p.S, d = p.d;
  const uint32_t rank = cluster_rank();
  const int mt = (int)(blockIdx.x / (unsigned)S);  // weight tile of this cluster
  pdl_launch_dependents();
  if (threadIdx.x == 0) {
    s_abort = 0;
    for (int s = 0; s < SW_STAGES; ++s) {
      mbar_init(smem_u32(&bar_full[s]), 1);
      mbar_init(smem_u32(&bar_empty[s]), 1);
    }
    mbar_init(smem_u32(&bar_acc), 1);
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmA2);
    tma_prefetch_desc(&tmB);
  }
  if (warp == 2) {
    tmem_alloc(smem_u32(&s_tmem), p.tmem_cols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s_tmem;
  const uint32_t base = (smem_u32(dsmem) + 1023u) & ~1023u;
  // the partial [row][128 features], in the drained pipeline stages (the same offset in every CTA)
  float* P = reinterpret_cast<float*>(dsmem + (base - smem_u32(dsmem)));
  const int kb0 = (int)((long long)rank * p.nkb / S), kb1 = (int)((long long)(rank + 1) * p.nkb / S);
  // The weight boxes of the first stages are inputs: the producer issues them
  // before the wait on the previous kernel, and their row boxes after it.
  const uint32_t tx = (uint32_t)(BM * BK * 2) + (uint32_t)p.tile_n * BK * 2;
  const int npre = min(SW_STAGES, kb1 - kb0);
  auto load_a = [&](int kb, uint32_t a_dst, uint32_t bar) {
    if (p.gate) {  // rows 0-63: W_v rows f0..; rows 64-127: the same rows of W_g[:, d:2d]
      tma_load_2d(a_dst, &tmA, kb * BK, mt * 64, bar);
      tma_load_2d(a_dst + (uint32_t)(64 * BK * 2), &tmA2, d + kb * BK, mt * 64, bar);
    } else {
      tma_load_2d(a_dst, &tmA, kb * BK, mt * 128, bar);
    }
  };
  if (warp == 0 && lane == 0) {
    for (int i = 0; i < npre; ++i) {  // every stage is free at the start
      const uint32_t a_dst = base + (uint32_t)i * p.stage_stride;
      mbar_arrive_expect_tx(smem_u32(&bar_full[i]), tx);
      load_a(kb0 + i, a_dst, smem_u32(&bar_full[i]));
    }
  }
  pdl_wait();  // R and the activation rows come from the previous kernels
  const int R = *(volatile const int32_t*)p.R;
  const int nrows = (R + 15) / 16 * 16;  // MMA N (at most tile_n)
  const bool work = R > 0;

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      // the row boxes of the stages issued above (also without work: their
      // barriers expect them; the boxes stay inside the tensor map)
      for (int i = 0; i < npre; ++i)
        tma_load_2d(base + (uint32_t)i * p.stage_stride + (uint32_t)(BM * BK * 2), &tmB, (kb0 + i) * BK, 0,
                    smem_u32(&bar_full[i]));
      int kb = kb0 + npre;
      if (work) {
        for (; kb < kb1; ++kb) {
          const int i = kb - kb0;
          const uint32_t s = (uint32_t)(i % SW_STAGES), ph = (uint32_t)((i / SW_STAGES) & 1);
          if (!mbar_wait_bounded(smem_u32(&bar_empty[s]), ph ^ 1u, &s_abort)) break;
          const uint32_t a_dst = base + s * p.stage_stride, b_dst = a_dst + (uint32_t)(BM * BK * 2);
          mbar_arrive_expect_tx(smem_u32(&bar_full[s]), tx);
          load_a(kb, a_dst, smem_u32(&bar_full[s]));
          tma_load_2d(b_dst, &tmB, kb * BK, 0, smem_u32(&bar_full[s]));
        }
      }
      if (!work || kb < kb1) {
        // no MMA consumes the stages (no rows), or a wait expired: let the
        // copies in flight land before the stages are reused or released
        if (work) raise_abort(&s_abort, p.status);
        volatile int never = 0;
        const int issued = kb - kb0;
        const int first = issued > SW_STAGES ? issued - SW_STAGES : 0;
        for (int i = first; i < issued; ++i)
          mbar_wait_bounded(smem_u32(&bar_full[i % SW_STAGES]), (uint32_t)((i / SW_STAGES) & 1), &never);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      if (work) {
        const uint32_t idesc = idesc_bf16_f32(128, nrows);
        bool ok = true;
        for (int kb = kb0; kb < kb1; ++kb) {
          const int i = kb - kb0;
          const uint32_t s = (uint32_t)(i % SW_STAGES), ph = (uint32_t)((i / SW_STAGES) & 1);
          if (!mbar_wait_bounded(smem_u32(&bar_full[s]), ph, &s_abort)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a_base = base + s * p.stage_stride, b_base = a_base + (uint32_t)(BM * BK * 2);
          const uint64_t adesc0 = sw128_kmajor_desc(a_base), bdesc0 = sw128_kmajor_desc(b_base);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k)
            tc_mma_bf16(tmem, adesc0 + 2u * k, bdesc0 + 2u * k, idesc, (i > 0 || k > 0) ? 1u : 0u);
          tc_commit(smem_u32(&bar_empty[s]));
        }
        if (!ok) raise_abort(&s_abort, p.status);
      }
      tc_commit(smem_u32(&bar_acc));  // accumulator ready (also without work or after a failure)
    }
    __syncwarp();
  } else if (warp >= 4) {
    // ---------------- epilogue warps: the partial into shared memory ----------------
    const int q = (warp - 4) * 32 + lane;  // weight row of the tile = TMEM lane = feature
    const bool ok = warp_wait(smem_u32(&bar_acc), 0u, &s_abort);
    tc_fence_after();
    if (!ok && lane == 0) raise_abort(&s_abort, p.status);
    if (ok && work && !s_abort) {
      const uint32_t taddr = tmem + ((uint32_t)((warp & 3) * 32) << 16);
      for (int c0 = 0; c0 < nrows; c0 += 32) {
        float v[32];
        tmem_ld_32cols(taddr + (uint32_t)c0, v);
#pragma unroll
        for (int j = 0; j < 32; ++j)
          if (c0 + j < nrows) P[(c0 + j) * 128 + q] = v[j];  // a warp stores 128 contiguous bytes
      }
    }
  }
  // ---------------- the cluster's sum and the epilogue ----------------
  tc_fence_before();
  __syncthreads();
  const bool go = work && !s_abort;  // every role is done: the same in every thread of the CTA
  cluster_sync_all();  // every partial of the cluster is in shared memory
  if (go) {
    const float* Pr[8];
#pragma unroll
    for (int s = 0; s < 8; ++s) Pr[s] = map_rank_ptr(P, (uint32_t)(s < S ? s : 0));
    const int g0 = (int)((long long)rank * R / S), g1 = (int)((long long)(rank + 1) * R / S);
    if (!p.gate) {
      // r[g, n0 + f] = m + beta * c for this CTA's rows: four features per
      // thread (16-byte partial loads, a warp 512 bytes of a row)
      const int n0 = mt * 128;
      for (int u = threadIdx.x; u < (g1 - g0) * 32; u += SW_THREADS) {
        const int g = g0 + u / 32, f = (u % 32) * 4;
        float4 x[8];
#pragma unroll
        for (int s = 0; s < 8; ++s)  // all loads first, then the sums in rank order
          x[s] = s < S ? *reinterpret_cast<const float4*>(Pr[s] + g * 128 + f) : make_float4(0.f, 0.f, 0.f, 0.f);
        const uint2 mw = __ldcg(reinterpret_cast<const uint2*>(p.apack + (long long)g * 2 * d + n0 + f));
        const long long orow = p.compact_out ? g : __ldcg(p.rowmap + g);
        float c0 = 0.f, c1 = 0.f, c2 = 0.f, c3 = 0.f;
#pragma unroll
        for (int s = 0; s < 8; ++s) {
          if (s < S) {
            c0 += x[s].x;
            c1 += x[s].y;
            c2 += x[s].z;
            c3 += x[s].w;
          }
        }
        *reinterpret_cast<uint2*>(p.r_out + orow * d + n0 + f) =
            make_uint2(pack_bf16x2(bf16_lo(mw.x) + p.beta * c0, bf16_hi(mw.x) + p.beta * c1),
                       pack_bf16x2(bf16_lo(mw.y) + p.beta * c2, bf16_hi(mw.y) + p.beta * c3));
      }
    } else {
      // e~[g, f0 + f] = e + v sigmoid(g_r + ge) for this CTA's rows: four
      // features per thread
      const int f0 = mt * 64;
      for (int u = threadIdx.x; u < (g1 - g0) * 16; u += SW_THREADS) {
        const int g = g0 + u / 16, f = (u % 16) * 4;
        float4 xv[8], xa[8];
#pragma unroll
        for (int s = 0; s < 8; ++s) {  // all loads first, then the sums in rank order
          xv[s] = s < S ? *reinterpret_cast<const float4*>(Pr[s] + g * 128 + f) : make_float4(0.f, 0.f, 0.f, 0.f);
          xa[s] = s < S ? *reinterpret_cast<const float4*>(Pr[s] + g * 128 + 64 + f) : make_float4(0.f, 0.f, 0.f, 0.f);
        }
        const float4 gb = __ldcg(reinterpret_cast<const float4*>(p.ge + f0 + f));
        const uint2 ew = __ldg(reinterpret_cast<const uint2*>(p.e + f0 + f));
        const long long orow = __ldcg(p.rowmap + g);
        float v0 = 0.f, v1 = 0.f, v2 = 0.f, v3 = 0.f, a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
#pragma unroll
        for (int s = 0; s < 8; ++s) {
          if (s < S) {
            v0 += xv[s].x;
            v1 += xv[s].y;
            v2 += xv[s].z;
            v3 += xv[s].w;
            a0 += xa[s].x;
            a1 += xa[s].y;
            a2 += xa[s].z;
            a3 += xa[s].w;
          }
        }
        a0 += gb.x;
        a1 += gb.y;
        a2 += gb.z;
        a3 += gb.w;
        *reinterpret_cast<uint2*>(p.e_out + orow * d + f0 + f) =
            make_uint2(pack_bf16x2(bf16_lo(ew.x) + v0 * fast_sigmoid(a0), bf16_hi(ew.x) + v1 * fast_sigmoid(a1)),
                       pack_bf16x2(bf16_lo(ew.y) + v2 * fast_sigmoid(a2), bf16_hi(ew.y) + v3 * fast_sigmoid(a3)));
      }
    }
  }
  cluster_sync_all();  // no CTA leaves while the others read its shared memory
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, p.tmem_cols);
  }
}

template <bool FUSED>
cudaError_t ensure_smem_attr() {
  static std::atomic<int> done[64];
  int dev = 0;
  cudaError_t err = cudaGetDevice(&dev);
  if (err != cudaSuccess) return err;
  if (!done[dev & 63].load(std::memory_order_acquire)) {
    err = cudaFuncSetAttribute(cond_kernel<FUSED>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               FUSED ? SMEM_BYTES_FUSED : SMEM_BYTES);
    if (err != cudaSuccess) return err;
    done[dev & 63].store(1, std::memory_order_release);
  }
  return cudaSuccess;
}

}  // namespace

cudaError_t launch_wait_selftest(int kind, const uint32_t* flag, uint32_t target, uint32_t* status,
                                 cudaStream_t stream) {
  wait_selftest_kernel<<<1, 32, 0, stream>>>(kind, flag, target, status);
  return cudaGetLastError();
}

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

static cudaError_t launch_cond_pair(const TcCondArgs& a, int clusters, cudaStream_t stream) {
  const long long rmax = (long long)a.B * (a.K - 1);
  const uint64_t d = (uint64_t)a.d;
  CUtensorMap mApack, mWc, mR, mWv, mWg;
  // Maps of operands a call does not use point at a used buffer (never read).
  const void* apack = a.do_correct ? a.apack : a.rpack;
  const void* wc = a.do_correct ? a.Wc : a.Wv;
  const void* rp = a.do_gate ? a.rpack : a.apack;
  const void* wv = a.do_gate ? a.Wv : a.Wc;
  const void* wg = a.do_gate ? a.Wg : a.Wc;
  if (encode_tensor_map_2d(&mApack, apack, a.do_correct ? 2 * d : d, (uint64_t)rmax, (a.do_correct ? 4 : 2) * d, BK, BM) != CUDA_SUCCESS ||
      encode_tensor_map_2d(&mWc, wc, a.do_correct ? 2 * d : d, d, (a.do_correct ? 4 : 2) * d, BK, 128) != CUDA_SUCCESS ||
      encode_tensor_map_2d(&mR, rp, d, (uint64_t)rmax, 2 * (a.r_row_stride ? (uint64_t)a.r_row_stride : d), BK, BM) != CUDA_SUCCESS ||
      encode_tensor_map_2d(&mWv, wv, a.do_gate ? d : 2 * d, d, (a.do_gate ? 2 : 4) * d, BK, 128) != CUDA_SUCCESS ||
      encode_tensor_map_2d(&mWg, wg, 2 * d, d, 4 * d, BK, 128) != CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  CondParams p{};
  p.d = a.d;
  p.do_correct = a.do_correct;
  p.do_gate = a.do_gate;
  p.R = a.R;
  p.rowmap = a.rowmap;
  p.apack = reinterpret_cast<const __nv_bfloat16*>(a.apack);
  p.beta = a.beta;
  p.r_out = reinterpret_cast<__nv_bfloat16*>(a.r_out);
  p.compact_out = a.compact_out;
  p.e = reinterpret_cast<const __nv_bfloat16*>(a.e);
  p.e_dense = 0;
  p.Wg = reinterpret_cast<const __nv_bfloat16*>(a.Wg);
  p.ge = a.ge;
  p.e_out = reinterpret_cast<__nv_bfloat16*>(a.e_out);
  p.sync = a.sync;
  p.block_done = a.sync + kSyncBlocks;
  p.block_ready = a.sync + kSyncBlocks + blocks_max(a.B, a.K);
  p.split_part = a.split_part;
  p.split_ticket = a.sync + kSyncBlocks + 2 * blocks_max(a.B, a.K);
  p.split_max = (a.split_part && a.do_gate) ? kPairSplitTiles : 0;
  p.status = a.status;
  // clusters of two CTAs; set-up may overlap the previous kernel's end
  return launch_dependent(cond_pair_kernel, dim3(2 * (unsigned)clusters), dim3(P_THREADS), P_SMEM_BYTES, stream, 2,
                          mApack, mWc, mR, mWv, mWg, p);
}

// The CTA-pair kernel: broadcast e (or no gate), and a device that can keep
// at least one pair of its CTAs resident.  Returns the pair count (0: use
// cond_kernel).
static int pair_clusters(const TcCondArgs& a, long long tiles_max_pairs, cudaError_t* err) {
  *err = cudaSuccess;
  if (a.do_gate && a.e_dense) return 0;
  static std::atomic<int> max_clusters[64];  // per device; 0: not yet known; -1: none fits
  int dev = 0;
  if ((*err = cudaGetDevice(&dev)) != cudaSuccess) return 0;
  if (max_clusters[dev & 63].load(std::memory_order_acquire) == 0) {
    if ((*err = cudaFuncSetAttribute(cond_pair_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, P_SMEM_BYTES)) !=
        cudaSuccess)
      return 0;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(2, 1, 1);
    cfg.blockDim = dim3(P_THREADS, 1, 1);
    cfg.dynamicSmemBytes = P_SMEM_BYTES;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    if ((*err = cudaOccupancyMaxActiveClusters(&n, cond_pair_kernel, &cfg)) != cudaSuccess) return 0;
    max_clusters[dev & 63].store(n > 0 ? n : -1, std::memory_order_release);
  }
  const int n = max_clusters[dev & 63].load(std::memory_order_acquire);
  if (n <= 0) return 0;
  // every pair when the gate-bias GEMV is needed: pairs without tiles compute it
  if (a.do_gate) return n;
  return (int)(tiles_max_pairs < n ? tiles_max_pairs : n);
}

// The small-R path (B (K-1) <= kSwapMaxRows, broadcast e or no gate): each
// GEMM as split-K tiles of 128 weight rows against the R rows, then its
// reduction kernel; four launches, each waiting on the one before inside the
// kernel, which cut the work from the R they read.
static cudaError_t launch_cond_swap(const TcCondArgs& a, cudaStream_t stream) {
  const long long rmax = (long long)a.B * (a.K - 1);
  const int d = a.d;
  const int rows_max = (int)((rmax + 15) / 16 * 16);
  const int box_n = rows_max < 256 ? rows_max : 256;
  const int ntiles_max = (rows_max + 255) / 256;
  DeviceInfo info;
  cudaError_t err = device_info(&info);
  if (err != cudaSuccess) return err;
  static std::atomic<int> attr_done[64];
  const int max_smem = SW_STAGES * (BM * BK * 2 + 256 * BK * 2) + 1024;
  if (!attr_done[info.device & 63].load(std::memory_order_acquire)) {
    err = cudaFuncSetAttribute(swap_gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, max_smem);
    if (err != cudaSuccess) return err;
    attr_done[info.device & 63].store(1, std::memory_order_release);
  }
  const uint32_t stage_stride = (uint32_t)((BM * BK * 2 + box_n * BK * 2 + 1023) / 1024 * 1024);
  const int smem = SW_STAGES * (int)stage_stride + 1024;
  uint32_t tmem_cols = 32;
  while ((int)tmem_cols < box_n) tmem_cols <<= 1;
  // One resident wave when it can carry every work tile: a split's CTA
  // streams its whole K range, so a second wave would double the time.
  static std::atomic<int> occ_cache[64][256 / 16 + 1];
  int occ = occ_cache[info.device & 63][box_n / 16].load(std::memory_order_relaxed);
  if (occ == 0) {
    err = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, swap_gemm_kernel, SW_THREADS, (size_t)smem);
    if (err != cudaSuccess) return err;
    if (occ < 1) occ = 1;
    occ_cache[info.device & 63][box_n / 16].store(occ, std::memory_order_relaxed);
  }
  int resident = info.sm_count * occ;
  if (resident > kSwapMaxCtas) resident = kSwapMaxCtas;
  const uint64_t du = (uint64_t)d;
  auto params = [&](SwapParams& sp, int mtiles, int nkb) {
    sp.R = a.R;
    sp.nkb = nkb;
    sp.mtiles = mtiles;
    sp.box_n = box_n;
    sp.tmem_cols = tmem_cols;
    sp.stage_stride = stage_stride;
    sp.part = a.part;
    sp.status = a.status;
    const int work_max = mtiles * ntiles_max;
    return work_max > resident ? work_max : resident;  // the grid
  };
  SwapReduceParams rp{};
  rp.d = d;
  rp.R = a.R;
  rp.part = a.part;
  rp.rowmap = a.rowmap;
  const int red_grid = info.sm_count * 4;
  const bool gemv = a.do_gate && !a.e_dense;
  if (a.do_correct) {
    CUtensorMap mA, mB;
    if (encode_tensor_map_2d(&mA, a.Wc, 2 * du, du, 4 * du, BK, 128) != CUDA_SUCCESS ||
        encode_tensor_map_2d(&mB, a.apack, 2 * du, (uint64_t)rmax, 4 * du, BK, (uint32_t)box_n) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
    SwapParams sp{};
    const int grid = params(sp, d / 128, 2 * d / BK);
    sp.mt_a = d / 128;
    sp.a2_x0 = 0;
    err = launch_dependent(swap_gemm_kernel, dim3((unsigned)grid), dim3(SW_THREADS), (size_t)smem, stream, 1u, mA,
                           mA, mB, sp);
    if (err != cudaSuccess) return err;
    rp.mtiles = sp.mtiles;
    rp.nkb = sp.nkb;
    rp.grid = grid;
    rp.do_gemv = gemv ? 1 : 0;  // overlapping the correction GEMM
    rp.gemv.d = d;
    rp.gemv.e = reinterpret_cast<const __nv_bfloat16*>(a.e);
    rp.gemv.Wg = reinterpret_cast<const __nv_bfloat16*>(a.Wg);
    rp.gemv.ge = a.ge;
    rp.gemv_next = a.sync + kSyncGemvNext;
    rp.gemv_done = a.sync + kSyncGemvDone;
    rp.apack = reinterpret_cast<const __nv_bfloat16*>(a.apack);
    rp.beta = a.beta;
    rp.r_out = reinterpret_cast<__nv_bfloat16*>(a.r_out);
    rp.compact_out = a.compact_out;
    err = launch_dependent(swap_reduce_correction_kernel, dim3((unsigned)red_grid), dim3(256), 0, stream, 1u, rp);
    if (err != cudaSuccess) return err;
  }
  if (a.do_gate) {
    const uint64_t rstride = 2 * (a.r_row_stride ? (uint64_t)a.r_row_stride : du);
    CUtensorMap mA, mA2, mB;
    if (encode_tensor_map_2d(&mA, a.Wv, du, du, 2 * du, BK, 128) != CUDA_SUCCESS ||
        encode_tensor_map_2d(&mA2, a.Wg, 2 * du, du, 4 * du, BK, 128) != CUDA_SUCCESS ||
        encode_tensor_map_2d(&mB, a.rpack, du, (uint64_t)rmax, rstride, BK, (uint32_t)box_n) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
    if (gemv && !a.do_correct) {  // no correction kernel to overlap the GEMV with
      SwapReduceParams gp{};
      gp.d = d;
      gp.gemv.d = d;
      gp.gemv.e = reinterpret_cast<const __nv_bfloat16*>(a.e);
      gp.gemv.Wg = reinterpret_cast<const __nv_bfloat16*>(a.Wg);
      gp.gemv.ge = a.ge;
      gp.gemv_next = a.sync + kSyncGemvNext;
      gp.gemv_done = a.sync + kSyncGemvDone;
      err = launch_dependent(swap_gemv_kernel, dim3((unsigned)red_grid), dim3(256), 0, stream, 1u, gp);
      if (err != cudaSuccess) return err;
    }
    SwapParams sp{};
    const int grid = params(sp, 2 * d / 128, d / BK);
    sp.mt_a = d / 128;  // W_v rows first, then the r half of W_g
    sp.a2_x0 = d;
    err = launch_dependent(swap_gemm_kernel, dim3((unsigned)grid), dim3(SW_THREADS), (size_t)smem, stream, 1u, mA,
                           mA2, mB, sp);
    if (err != cudaSuccess) return err;
    rp.mtiles = sp.mtiles;
    rp.nkb = sp.nkb;
    rp.grid = grid;
    rp.do_gemv = 0;
    rp.e = reinterpret_cast<const __nv_bfloat16*>(a.e);
    rp.ge = a.ge;
    rp.e_out = reinterpret_cast<__nv_bfloat16*>(a.e_out);
    err = launch_dependent(swap_reduce_gate_kernel, dim3((unsigned)red_grid), dim3(256), 0, stream, 1u, rp);
    if (err != cudaSuccess) return err;
  }
  return cudaSuccess;
}

// Clusters of S CTAs of swap_cluster_kernel that the device holds at once
// with `smem` bytes each (0: none), cached per device, S and shared memory.
static int swap_cluster_capacity(int dev, int S, int smem, cudaError_t* err) {
  static std::atomic<int> cache[64][9][17];  // [device][S][smem in 16 KB steps]; 0: not yet known, -1: none
  std::atomic<int>& slot = cache[dev & 63][S][smem >> 14];
  int n = slot.load(std::memory_order_acquire);
  if (n == 0) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)S, 1, 1);
    cfg.blockDim = dim3(SW_THREADS, 1, 1);
    cfg.dynamicSmemBytes = (size_t)smem;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = (unsigned)S;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int m = 0;
    if ((*err = cudaOccupancyMaxActiveClusters(&m, swap_cluster_kernel, &cfg)) != cudaSuccess) return 0;
    n = m > 0 ? m : -1;
    slot.store(n, std::memory_order_release);
  }
  return n > 0 ? n : 0;
}

// The small-R GEMMs as split-K clusters with the reduction inside
// (swap_cluster_kernel): one N tile (at most 256 possible rows) and, for
// each GEMM, a cluster size S <= 8 whose clusters all fit in one wave with
// one CTA per SM.  Returns cudaErrorNotSupported (nothing launched) where
// that does not hold.
static cudaError_t launch_cond_swap_cluster(const TcCondArgs& a, cudaStream_t stream) {
  const long long rmax = (long long)a.B * (a.K - 1);
  const int d = a.d;
  const int rows_max = (int)((rmax + 15) / 16 * 16);
  if (rows_max > 256 || d % 128 != 0) return cudaErrorNotSupported;
  const int tile_n = rows_max;
  DeviceInfo info;
  cudaError_t err = device_info(&info);
  if (err != cudaSuccess) return err;
  const int dev = info.device;
  const uint32_t stage_stride = (uint32_t)((BM * BK * 2 + tile_n * BK * 2 + 1023) / 1024 * 1024);
  // at least half of an SM's shared memory: one CTA per SM, so the K splits
  // of one wave stream over distinct SMs
  int smem = SW_STAGES * (int)stage_stride + 1024;
  if (smem < 117 * 1024) smem = 117 * 1024;
  static std::atomic<int> attr_done[64];
  if (!attr_done[dev & 63].load(std::memory_order_acquire)) {
    err = cudaFuncSetAttribute(swap_cluster_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               SW_STAGES * (BM * BK * 2 + 256 * BK * 2) + 1024);
    if (err != cudaSuccess) return err;
    attr_done[dev & 63].store(1, std::memory_order_release);
  }
  // the largest S <= 8 with every cluster of the GEMM resident at once and
  // at least SW_STAGES k-blocks per split
  auto pick = [&](int work, int nkb, int* S_out, int* clusters) -> cudaError_t {
    *S_out = 0;
    for (int S = 8; S >= 1; --S) {
      if (nkb / S < SW_STAGES) continue;
      const int cap = swap_cluster_capacity(dev, S, smem, &err);
      if (err != cudaSuccess) return err;
      if (work <= cap) {
        *S_out = S;
        *clusters = cap;
        return cudaSuccess;
      }
    }
    return cudaSuccess;
  };
  int Sc = 1, cc = 0, Sg = 1, cg = 0;
  if (a.do_correct && (err = pick(d / 128, 2 * d / BK, &Sc, &cc)) != cudaSuccess) return err;
  if (a.do_gate && (err = pick(d / 64, d / BK, &Sg, &cg)) != cudaSuccess) return err;
  (void)cc;
  (void)cg;
  if ((a.do_correct && Sc == 0) || (a.do_gate && Sg == 0)) return cudaErrorNotSupported;
  uint32_t tmem_cols = 32;
  while ((int)tmem_cols < tile_n) tmem_cols <<= 1;
  const uint64_t du = (uint64_t)d;
  SwapClusterParams sp{};
  sp.R = a.R;
  sp.d = d;
  sp.tile_n = tile_n;
  sp.tmem_cols = tmem_cols;
  sp.stage_stride = stage_stride;
  sp.rowmap = a.rowmap;
  sp.status = a.status;
  // W_g[:, :d] e in its own many-warp kernel, launched after the correction
  // GEMM so that it runs beside it (alone, before the GEMM, it was slower:
  // its stream is latency-bound); it ends with a programmatic wait, so the
  // gate launch after it also waits for the correction.
  auto launch_gemv = [&]() {
    SwapReduceParams gp{};
    gp.d = d;
    gp.gemv.d = d;
    gp.gemv.e = reinterpret_cast<const __nv_bfloat16*>(a.e);
    gp.gemv.Wg = reinterpret_cast<const __nv_bfloat16*>(a.Wg);
    gp.gemv.ge = a.ge;
    gp.gemv_next = a.sync + kSyncGemvNext;
    gp.gemv_done = a.sync + kSyncGemvDone;
    return launch_dependent(swap_gemv_kernel, dim3((unsigned)(info.sm_count * 4)), dim3(256), 0, stream, 1u, gp);
  };
  if (a.do_correct) {
    CUtensorMap mA, mB;
    if (encode_tensor_map_2d(&mA, a.Wc, 2 * du, du, 4 * du, BK, 128) != CUDA_SUCCESS ||
        encode_tensor_map_2d(&mB, a.apack, 2 * du, (uint64_t)rmax, 4 * du, BK, (uint32_t)tile_n) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
    SwapClusterParams c = sp;
    c.nkb = 2 * d / BK;
    c.S = Sc;
    c.gate = 0;
    c.apack = reinterpret_cast<const __nv_bfloat16*>(a.apack);
    c.beta = a.beta;
    c.r_out = reinterpret_cast<__nv_bfloat16*>(a.r_out);
    c.compact_out = a.compact_out;
    err = launch_dependent(swap_cluster_kernel, dim3((unsigned)(d / 128 * Sc)), dim3(SW_THREADS), (size_t)smem,
                           stream, (unsigned)Sc, mA, mA, mB, c);
    if (err != cudaSuccess) return err;
  }
  if (a.do_gate) {
    const uint64_t rstride = 2 * (a.r_row_stride ? (uint64_t)a.r_row_stride : du);
    CUtensorMap mA, mA2, mB;
    if (encode_tensor_map_2d(&mA, a.Wv, du, du, 2 * du, BK, 64) != CUDA_SUCCESS ||
        encode_tensor_map_2d(&mA2, a.Wg, 2 * du, du, 4 * du, BK, 64) != CUDA_SUCCESS ||
        encode_tensor_map_2d(&mB, a.rpack, du, (uint64_t)rmax, rstride, BK, (uint32_t)tile_n) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
    if ((err = launch_gemv()) != cudaSuccess) return err;
    SwapClusterParams g = sp;
    g.nkb = d / BK;
    g.S = Sg;
    g.gate = 1;
    g.e = reinterpret_cast<const __nv_bfloat16*>(a.e);
    g.ge = a.ge;
    g.e_out = reinterpret_cast<__nv_bfloat16*>(a.e_out);
    err = launch_dependent(swap_cluster_kernel, dim3((unsigned)(d / 64 * Sg)), dim3(SW_THREADS), (size_t)smem,
                           stream, (unsigned)Sg, mA, mA2, mB, g);
    if (err != cudaSuccess) return err;
  }
  return cudaSuccess;
}

cudaError_t launch_cond_tc(const TcCondArgs& a, cudaStream_t stream) {
  const long long rmax = (long long)a.B * (a.K - 1);
  if (rmax <= 0 || (!a.do_correct && !a.do_gate)) return cudaSuccess;
  if (a.part && !(a.do_gate && a.e_dense)) {
    const cudaError_t e1 = launch_cond_swap_cluster(a, stream);
    return e1 == cudaErrorNotSupported ? launch_cond_swap(a, stream) : e1;
  }
  const long long tiles_max_pairs =
      (rmax + 2 * BM - 1) / (2 * BM) * ((a.do_correct ? a.d / 256 : 0) + (a.do_gate ? a.d / 128 : 0));
  cudaError_t err;
  const int clusters = pair_clusters(a, tiles_max_pairs, &err);
  if (err != cudaSuccess) return err;
  if (clusters > 0) return launch_cond_pair(a, clusters, stream);
  err = ensure_smem_attr<false>();
  if (err != cudaSuccess) return err;
  const uint64_t d = (uint64_t)a.d;
  CUtensorMap mApack, mWc, mR, mE, mWv, mWg;
  // Maps of operands a call does not use point at a used buffer (never read).
  const void* apack = a.do_correct ? a.apack : a.rpack;
  const void* wc = a.do_correct ? a.Wc : a.Wv;
  const void* rp = a.do_gate ? a.rpack : a.apack;
  const void* erows = (a.do_gate && a.e_dense) ? a.epack : rp;
  const void* wv = a.do_gate ? a.Wv : a.Wc;
  const void* wg = a.do_gate ? a.Wg : a.Wc;
  if (encode_tensor_map_2d(&mApack, apack, a.do_correct ? 2 * d : d, (uint64_t)rmax, (a.do_correct ? 4 : 2) * d, BK, BM) != CUDA_SUCCESS ||
      encode_tensor_map_2d(&mWc, wc, a.do_correct ? 2 * d : d, d, (a.do_correct ? 4 : 2) * d, BK, 256) != CUDA_SUCCESS ||
      encode_tensor_map_2d(&mR, rp, d, (uint64_t)rmax, 2 * (a.r_row_stride ? (uint64_t)a.r_row_stride : d), BK, BM) != CUDA_SUCCESS ||
      encode_tensor_map_2d(&mE, erows, d, (uint64_t)rmax, 2 * d, BK, BM) != CUDA_SUCCESS ||
      encode_tensor_map_2d(&mWv, wv, a.do_gate ? d : 2 * d, d, (a.do_gate ? 2 : 4) * d, BK, 128) != CUDA_SUCCESS ||
      encode_tensor_map_2d(&mWg, wg, 2 * d, d, 4 * d, BK, 128) != CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  CondParams p{};
  p.d = a.d;
  p.do_correct = a.do_correct;
  p.do_gate = a.do_gate;
  p.R = a.R;
  p.rowmap = a.rowmap;
  p.apack = reinterpret_cast<const __nv_bfloat16*>(a.apack);
  p.beta = a.beta;
  p.r_out = reinterpret_cast<__nv_bfloat16*>(a.r_out);
  p.compact_out = a.compact_out;
  p.e = reinterpret_cast<const __nv_bfloat16*>(a.e_dense ? a.epack : a.e);
  p.e_dense = a.e_dense;
  p.Wg = reinterpret_cast<const __nv_bfloat16*>(a.Wg);
  p.ge = a.ge;
  p.e_out = reinterpret_cast<__nv_bfloat16*>(a.e_out);
  p.sync = a.sync;
  p.block_done = a.sync + kSyncBlocks;
  p.block_ready = a.sync + kSyncBlocks + blocks_max(a.B, a.K);
  p.status = a.status;
  DeviceInfo info{0, 148};
  err = device_info(&info);
  if (err != cudaSuccess) return err;
  const long long tiles_max = (rmax + BM - 1) / BM * ((a.do_correct ? a.d / 256 : 0) + (a.do_gate ? a.d / 128 : 0));
  // every SM when the broadcast-e GEMV is needed: CTAs without tiles compute it
  const bool need_ge = a.do_gate && !a.e_dense;
  const unsigned grid = (unsigned)(need_ge || tiles_max >= info.sm_count ? info.sm_count : tiles_max);
  VerifyStreamParams vp{};
  cond_kernel<false><<<grid, THREADS, SMEM_BYTES, stream>>>(mApack, mWc, mR, mE, mWv, mWg, p, vp);
  return cudaGetLastError();
}

}  // namespace retrace

namespace retrace {

bool round_fused_supported(const TcRoundArgs& a) {
  // contiguous logits with rows of at least one stream chunk, so that a chunk
  // is one contiguous copy and spans at most two rows
  return tc_supported(RETRACE_BF16, a.d) && 4 * a.d <= kStageBytes && ((uintptr_t)a.logits % 16 == 0) && a.V % 8 == 0 &&
         a.V >= 8 * kChunkSlots && a.row_stride == a.V && a.batch_stride == (long long)(a.K + 1) * a.V &&
         a.K >= 2 && (long long)a.B * (a.K + 1) * (a.V / 8) < (1ll << 32) - kChunkSlots;
}

cudaError_t launch_round_tc(const TcRoundArgs& a, cudaStream_t stream) {
  cudaError_t err = ensure_smem_attr<true>();
  if (err != cudaSuccess) return err;
  const uint64_t d = (uint64_t)a.d;
  const long long rmax = (long long)a.B * (a.K - 1);
  CUtensorMap mApack, mWc, mR, mE, mWv, mWg;
  if (encode_tensor_map_2d(&mApack, a.apack, 2 * d, (uint64_t)rmax, 4 * d, BK, BM) != CUDA_SUCCESS ||
      encode_tensor_map_2d(&mWc, a.Wc, 2 * d, d, 4 * d, BK, 256) != CUDA_SUCCESS ||
      encode_tensor_map_2d(&mR, a.rpack, d, (uint64_t)rmax, 2 * d, BK, BM) != CUDA_SUCCESS ||
      encode_tensor_map_2d(&mE, a.e_dense ? a.epack : a.rpack, d, (uint64_t)rmax, 2 * d, BK, BM) != CUDA_SUCCESS ||
      encode_tensor_map_2d(&mWv, a.Wv, d, d, 2 * d, BK, 128) != CUDA_SUCCESS ||
      encode_tensor_map_2d(&mWg, a.Wg, 2 * d, d, 4 * d, BK, 128) != CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  const long long blocks = blocks_max(a.B, a.K);
  CondParams p{};
  p.d = a.d;
  p.do_correct = 1;
  p.do_gate = 1;
  p.R = reinterpret_cast<const int32_t*>(a.sync + kSyncRowCount);
  p.rowmap = a.rowmap;
  p.apack = reinterpret_cast<const __nv_bfloat16*>(a.apack);
  p.beta = a.beta;
  p.r_out = reinterpret_cast<__nv_bfloat16*>(a.rpack);
  p.compact_out = 1;
  p.e = reinterpret_cast<const __nv_bfloat16*>(a.e_dense ? a.epack : a.e);
  p.e_dense = a.e_dense;
  p.Wg = reinterpret_cast<const __nv_bfloat16*>(a.Wg);
  p.ge = a.ge;
  p.e_out = reinterpret_cast<__nv_bfloat16*>(a.e_out);
  p.sync = a.sync;
  p.block_done = a.sync + kSyncBlocks;
  p.block_ready = a.sync + kSyncBlocks + blocks;
  p.max_blocks = (int)blocks;
  p.status = a.status;

  VerifyStreamParams vp{};
  vp.logits = reinterpret_cast<const __nv_bfloat16*>(a.logits);
  vp.B = a.B;
  vp.K = a.K;
  vp.V = a.V;
  vp.draft = a.draft;
  vp.accept_len = a.accept_len;
  vp.committed = a.committed;
  vp.bonus = a.bonus;
  vp.target_argmax = a.target_argmax;
  vp.n_out = a.n_out;
  vp.keys = a.keys;
  vp.tickets = a.tickets;
  vp.e = reinterpret_cast<const __nv_bfloat16*>(a.e);
  vp.e_batch_stride = a.e_batch_stride;
  vp.e_pos_stride = a.e_pos_stride;
  vp.e_out = reinterpret_cast<__nv_bfloat16*>(a.e_out);
  vp.d = a.d;
  vp.hD = reinterpret_cast<const __nv_bfloat16*>(a.hD);
  vp.hT = reinterpret_cast<const __nv_bfloat16*>(a.hT);
  vp.e_dense = a.e_dense;
  vp.apack = reinterpret_cast<__nv_bfloat16*>(a.apack);
  vp.epack = reinterpret_cast<__nv_bfloat16*>(a.epack);
  vp.rowmap = a.rowmap;
  vp.R_count = a.sync + kSyncRowCount;
  vp.rows_ready = a.sync + kSyncBlocks + blocks;
  vp.seq_done = a.sync + kSyncSeqDone;
  vp.slots_per_row = a.V / 8;
  vp.total_slots = (long long)a.B * (a.K + 1) * vp.slots_per_row;
  vp.total_chunks = (uint32_t)((vp.total_slots + kChunkSlots - 1) / kChunkSlots);
  vp.chunk_next = a.sync + kSyncChunkNext;
  vp.status = a.status;

  DeviceInfo info{0, 148};
  err = device_info(&info);
  if (err != cudaSuccess) return err;
  const long long grid = info.sm_count;
  // Cooperative: every CTA's share of the logits feeds other CTAs' tiles, so
  // all CTAs must be resident together (one per SM); the launch fails
  // instead of starting if they cannot be.
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(THREADS_FUSED);
  cfg.dynamicSmemBytes = SMEM_BYTES_FUSED;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, cond_kernel<true>, mApack, mWc, mR, mE, mWv, mWg, p, vp);
}

}  // namespace retrace
