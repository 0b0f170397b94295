// Greedy verification of a draft block (ReTrace Algorithm 1, Verify and
// commit steps; greedy decoding = top_k 1).
//
// The [B, K+1, V] logits are one flat stream of B*(K+1) rows.  The rows are
// cut into "slots" (16-byte vectors: 8 bf16 or 4 fp32; single elements on the
// unaligned path) and the slot range is split evenly over the grid, so every
// CTA streams the same number of bytes whatever B, K and V are.  A CTA reduces
// each row segment it owns to one 64-bit (value, ~index) key and folds it into
// the row's key with atomicMax.  The last CTA to finish a sequence (per-
// sequence arrival ticket; nothing ever waits) decodes its K+1 argmaxes,
// finds the first mismatch with a warp ballot and writes the accepted length,
// committed tokens and bonus, resets the keys and ticket to zero for the next
// call and, inside a fused round, copies the unconditioned drafter inputs.
//
// The outputs depend only on rows 0..A_b of each sequence.  The windowed
// schedule runs the same kernel as a chain of passes over row windows
// [i0, i1), with no finalisers and no tickets: a pass only folds keys.  Each
// later pass (launched programmatically dependent) first rebuilds its live
// list, the sequences whose draft tokens matched every row so far, from the
// previous window's keys and the previous live list (every CTA the same list,
// in sequence order, by a block scan; CTA 0 publishes it for the next pass).
// The sequences that mismatched in the previous window are decided there and
// then: accepted length, outputs (spread over the CTAs) and their packed-row
// offsets, after the rows of the sequences decided in earlier windows.  The
// pass then streams only the listed sequences' rows.  Rows past the window
// holding the first mismatch are never read.  verify_finish_kernel decides
// the sequences of the last window the same way and does the row copies.  A one-pass round that packs rows for fewer sequences than
// there are SMs leaves its copies to verify_copy_kernel, spread over the grid.
#include <atomic>

#include "common.cuh"
#include "internal.h"

namespace retrace {
namespace {

constexpr int kThreads = 512;
constexpr int kUnroll = 4;
// Least logits bytes per active CTA: small problems spread one row or so per
// CTA instead of streaming several rows one after another on a few CTAs.
constexpr long long kMinCtaBytes = 4096;

struct VerifyParams {
  const void* logits;
  int B, K, V;
  long long row_stride, batch_stride;
  const int32_t* draft;
  int32_t* accept_len;
  int32_t* committed;
  int32_t* bonus;
  int32_t* target_argmax;
  int32_t* n_out;
  unsigned long long* keys;
  uint32_t* tickets;
  int slots_per_row;
  long long total_slots;
  const void* e;
  long long e_batch_stride, e_pos_stride;
  void* e_out;
  int d;
  const void* hD;
  const void* hT;
  int e_dense;
  void* apack;
  void* epack;
  int32_t* rowmap;
  int32_t* R_count;
  int cond_copy;
  // Row window of this pass ([0, K+1) in one pass).  A later pass of the
  // windowed schedule (i0 > 0) rebuilds its live list from the keys of the
  // previous window [pi0, i0) of the previous live list.
  int i0, i1, pi0;
  int windowed;              // a pass of the windowed schedule: keys only, no finalisers
  const int32_t* live_in;    // previous pass's live list (NULL: 0..B-1)
  const uint32_t* count_in;  // its length (NULL: B)
  const uint32_t* base_in;   // packed rows claimed by the sequences decided before (NULL: 0)
  int32_t* live_out;         // CTA 0 publishes this pass's live list here
  uint32_t* count_out;
  uint32_t* base_out;        // ... and the packed rows claimed by the sequences decided so far
  // verify_finish_kernel: the passes' counters, zeroed with the keys by its last CTA out
  uint32_t* pass_counts;
  int n_counts;
  uint32_t* exits;           // CTAs out (zero between calls)
  int defer_copies;          // the finaliser leaves the copies to verify_copy_kernel
  int32_t* pack_off;         // [B] first packed row of each sequence (deferred copies)
};

// 16-byte vector helpers: the maximum of the vector's elements and element q.
template <typename T>
struct Vec;
template <>
struct Vec<__nv_bfloat16> {
  static constexpr int E = 8;
  __device__ static __forceinline__ float vmax(const uint4& v) {
    const __nv_bfloat162 a = *reinterpret_cast<const __nv_bfloat162*>(&v.x);
    const __nv_bfloat162 b = *reinterpret_cast<const __nv_bfloat162*>(&v.y);
    const __nv_bfloat162 c = *reinterpret_cast<const __nv_bfloat162*>(&v.z);
    const __nv_bfloat162 d = *reinterpret_cast<const __nv_bfloat162*>(&v.w);
    const __nv_bfloat162 m = __hmax2(__hmax2(a, b), __hmax2(c, d));
    return fmaxf(__low2float(m), __high2float(m));
  }
  __device__ static __forceinline__ float elem(const uint4& v, int q) {
    const uint32_t w = (q < 2) ? v.x : (q < 4) ? v.y : (q < 6) ? v.z : v.w;
    return (q & 1) ? bf16_hi(w) : bf16_lo(w);
  }
};
template <>
struct Vec<float> {
  static constexpr int E = 4;
  __device__ static __forceinline__ float vmax(const uint4& v) {
    return fmaxf(fmaxf(__uint_as_float(v.x), __uint_as_float(v.y)),
                 fmaxf(__uint_as_float(v.z), __uint_as_float(v.w)));
  }
  __device__ static __forceinline__ float elem(const uint4& v, int q) {
    const uint32_t w = (q == 0) ? v.x : (q == 1) ? v.y : (q == 2) ? v.z : v.w;
    return __uint_as_float(w);
  }
};

// Key of this thread's share of row slots [v0, v1).
template <typename T, bool VEC>
__device__ __forceinline__ unsigned long long segment_key(const T* __restrict__ rowp, int v0,
                                                          int v1, int V) {
  unsigned long long key = 0ull;
  if constexpr (VEC) {
    constexpr int E = Vec<T>::E;
    const int full = V / E;  // complete 16-byte slots in the row
    const int hi = v1 < full ? v1 : full;
    const uint4* __restrict__ vp = reinterpret_cast<const uint4*>(rowp);
    float best = -INFINITY;
    int best_slot = -1;
    uint4 best_vec = make_uint4(0, 0, 0, 0);
    for (int s = v0 + (int)threadIdx.x; s < hi; s += kUnroll * kThreads) {
      uint4 x[kUnroll];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const int q = s + u * kThreads;
        if (q < hi) x[u] = __ldcs(vp + q);
      }
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const int q = s + u * kThreads;
        if (q < hi) {
          const float m = Vec<T>::vmax(x[u]);
          // strictly greater keeps the earliest slot among equal maxima
          if (m > best || best_slot < 0) {
            best = m;
            best_slot = q;
            best_vec = x[u];
          }
        }
      }
    }
    if (best_slot >= 0) {
#pragma unroll
      for (int q = 0; q < E; ++q) {
        if (Vec<T>::elem(best_vec, q) == best) {
          key = make_key(best, (uint32_t)(best_slot * E + q));
          break;
        }
      }
    }
    // Trailing partial slot (V not a multiple of E), read element by element.
    if (v1 > full && threadIdx.x == 0) {
      for (int v = full * E; v < V; ++v) key = umax64(key, make_key(to_f32<T>(rowp[v]), (uint32_t)v));
    }
  } else {
    for (int v = v0 + (int)threadIdx.x; v < v1; v += kThreads)
      key = umax64(key, make_key(to_f32<T>(rowp[v]), (uint32_t)v));
  }
  return key;
}

__device__ __forceinline__ unsigned long long block_max_key(unsigned long long key,
                                                            unsigned long long* s_red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  key = warp_max_key(key);
  if (lane == 0) s_red[warp] = key;
  __syncthreads();
  if (warp == 0) {
    unsigned long long k = (lane < kThreads / 32) ? s_red[lane] : 0ull;
    k = warp_max_key(k);
    if (lane == 0) s_red[0] = k;
  }
  __syncthreads();
  return s_red[0];
}

// Row copies of the finalising CTA go through shared memory with cp.async,
// four 16-byte vectors per thread in flight (32 KB per CTA; more would make
// this kernel spill at its two-CTAs-per-SM register budget).
constexpr int kCopyStage = 4;
constexpr int kCopyStageBytes = kCopyStage * kThreads * 16;

// Copy of rows [j0, K) of sequence b into e_out: rows j < j_m from the
// aligned drafter states m_j = hD[b, A+1+j] (the overwrite ablation), the
// others from the drafter inputs e.
template <typename T>
__device__ void copy_rows(const VerifyParams& p, int b, int A, int j0, int j_m, uint4* staging) {
  const int K = p.K, d = p.d;
  const long long rows = K - j0;
  if (rows <= 0) return;
  T* dst = reinterpret_cast<T*>(p.e_out) + ((long long)b * K + j0) * d;
  const T* src_b = reinterpret_cast<const T*>(p.e) + (long long)b * p.e_batch_stride;
  const T* m_b = reinterpret_cast<const T*>(p.hD) + ((long long)b * K + A + 1) * d;  // row j: m_b + j*d
  const bool vec = ((d * (int)sizeof(T)) % 16 == 0) && ((uintptr_t)dst % 16 == 0) &&
                   ((uintptr_t)src_b % 16 == 0) && ((p.e_pos_stride * (long long)sizeof(T)) % 16 == 0) &&
                   (j_m <= j0 || (uintptr_t)p.hD % 16 == 0);
  if (vec) {
    const int vpr = d * (int)sizeof(T) / 16;
    copy_vectors_staged<kCopyStage>(
        rows * vpr,
        staging,
        [&](long long i) {
          const long long j = j0 + i / vpr, q = i % vpr;
          const T* row = (j < j_m) ? m_b + j * d : src_b + j * p.e_pos_stride;
          return reinterpret_cast<const uint4*>(row) + q;
        },
        [&](long long i) { return reinterpret_cast<uint4*>(dst) + i; });
  } else {
    for (long long i = threadIdx.x; i < rows * d; i += kThreads) {
      const long long j = j0 + i / d, q = i % d;
      dst[i] = (j < j_m) ? m_b[j * d + q] : src_b[j * p.e_pos_stride + q];
    }
  }
}

// Packs sequence b's conditioned rows for the tensor-core projections: the
// shifted draft states and target states [m_j; u_j] = [hD[b, A+1+j]; hT[b, A+j]]
// (Eq. 4-5) and, for per-position e, e[b, j]; rows land at a block of n_b rows
// claimed with one atomic (row order across sequences does not matter: every
// packed row carries its position in rowmap).
__device__ void pack_sequence_rows(const VerifyParams& p, int b, int A, int nb, int* s_off, uint4* staging) {
  const int K = p.K, d = p.d;
  if (threadIdx.x == 0) *s_off = atomicAdd(p.R_count, nb);
  __syncthreads();
  const int off = *s_off;
  for (int j = threadIdx.x; j < nb; j += kThreads) p.rowmap[off + j] = b * K + j;
  const int vpr = d / 8;  // 16-byte vectors per bf16 row
  const long long base = (long long)b * K;
  const uint4* hD = reinterpret_cast<const uint4*>(p.hD);
  const uint4* hT = reinterpret_cast<const uint4*>(p.hT);
  uint4* out = reinterpret_cast<uint4*>(p.apack);
  copy_vectors_staged<kCopyStage>(
      (long long)nb * 2 * vpr, staging,
      [&](long long i) {
        const long long j = i / (2 * vpr), c = i - j * 2 * vpr;
        return (c < vpr) ? hD + (base + A + 1 + j) * vpr + c : hT + (base + A + j) * vpr + c - vpr;
      },
      [&](long long i) { return out + (long long)off * 2 * vpr + i; });
  if (p.e_dense) {
    const uint4* e = reinterpret_cast<const uint4*>(p.e);
    uint4* eo = reinterpret_cast<uint4*>(p.epack);
    copy_vectors_staged<kCopyStage>((long long)nb * vpr, staging, [&](long long i) { return e + base * vpr + i; },
                                    [&](long long i) { return eo + (long long)off * vpr + i; });
  }
}

// Copies of sequence b once A is known: the unconditioned rows of e_out and
// the packing of the conditioned ones (in a fused round).
template <typename T>
__device__ void copy_sequence(const VerifyParams& p, int b, int A, int* s_off, uint4* staging) {
  const int nb = (p.K - 1 - A) > 0 ? (p.K - 1 - A) : 0;
  if (p.e_out) {
    if (p.cond_copy == kCondCopyKeep) copy_rows<T>(p, b, A, nb, 0, staging);
    else if (p.cond_copy == kCondCopyE) copy_rows<T>(p, b, A, 0, 0, staging);
    else copy_rows<T>(p, b, A, 0, nb, staging);
  }
  if (p.R_count && nb > 0) pack_sequence_rows(p, b, A, nb, s_off, staging);
}

// Outputs of sequence b once its accepted length A and the argmaxes s_t[0..A]
// are known: committed tokens, accepted length, bonus, n_b and (unless a
// later kernel does them) the copies.  The argmax keys of rows 0..rows-1 are
// reset for the next call.
template <typename T>
__device__ void finish_sequence(const VerifyParams& p, int b, int A, int rows, const int* s_t, int* s_off,
                                uint4* staging) {
  const int K = p.K, K1 = K + 1;
  for (int i = threadIdx.x; i < K1; i += kThreads) {
    const long long o = (long long)b * K1 + i;
    p.committed[o] = (i <= A) ? s_t[i] : -1;
    if (p.target_argmax) p.target_argmax[o] = s_t[i];
    if (i < rows) p.keys[o] = 0ull;
  }
  const int nb = (K - 1 - A) > 0 ? (K - 1 - A) : 0;
  if (threadIdx.x == 0) {
    p.accept_len[b] = A;
    p.bonus[b] = s_t[A];
    if (p.n_out) p.n_out[b] = nb;
    if (p.defer_copies && p.R_count) p.pack_off[b] = nb > 0 ? atomicAdd(p.R_count, nb) : 0;
  }
  if (!p.defer_copies) copy_sequence<T>(p, b, A, s_off, staging);
}

// Every row of sequence b has its key (one pass): the first mismatch by
// ballot, then the outputs.
template <typename T>
__device__ void finalize_sequence(const VerifyParams& p, int b, int* s_t, int* s_A, uint4* staging) {
  const int K = p.K, K1 = K + 1;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int i = threadIdx.x; i < K1; i += kThreads)
    s_t[i] = (int)key_index(__ldcg(&p.keys[(long long)b * K1 + i]));
  __syncthreads();
  if (warp == 0) {
    int A = K;
    for (int base = 0; base < K; base += 32) {
      const int i = base + lane;
      const bool mismatch = (i < K) && (s_t[i] != p.draft[(long long)b * K + i]);
      const unsigned bal = __ballot_sync(0xFFFFFFFFu, mismatch);
      if (bal) {
        A = base + __ffs(bal) - 1;
        break;
      }
    }
    if (lane == 0) *s_A = A;
  }
  __syncthreads();
  const int A = *s_A;
  if (threadIdx.x == 0) p.tickets[b] = 0u;
  finish_sequence<T>(p, b, A, K1, s_t, s_A + 1, staging);
}

// Exclusive prefix sum over the CTA (kThreads threads, in thread order) of
// one value per thread; *total receives the sum.  s_warp holds kThreads / 32
// + 1 ints.  Every thread of the CTA must call it.
__device__ __forceinline__ int block_exclusive_scan(int v, int* s_warp, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int y = __shfl_up_sync(0xFFFFFFFFu, x, off);
    if (lane >= off) x += y;
  }
  if (lane == 31) s_warp[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int w = lane < kThreads / 32 ? s_warp[lane] : 0;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int y = __shfl_up_sync(0xFFFFFFFFu, w, off);
      if (lane >= off) w += y;
    }
    if (lane < kThreads / 32) s_warp[lane] = w;  // inclusive warp totals
  }
  __syncthreads();
  const int excl = x - v + (warp > 0 ? s_warp[warp - 1] : 0);
  *total = s_warp[kThreads / 32 - 1];
  __syncthreads();  // s_warp may be reused by the next call
  return excl;
}

// Outputs of sequence b, decided with accepted length A after a windowed
// pass (every row 0..A has its key): committed tokens, accepted length,
// bonus, n_b and the first packed row `off` of its n_b conditioned rows.
// The CTA's threads share the K + 1 committed slots.
__device__ void write_decided(const VerifyParams& p, int b, int A, int off) {
  const int K = p.K, K1 = K + 1;
  for (int i = threadIdx.x; i < K1; i += kThreads) {
    const long long o = (long long)b * K1 + i;
    p.committed[o] = i <= A ? (int)key_index(__ldcg(&p.keys[o])) : -1;
  }
  if (threadIdx.x == 0) {
    const int nb = max(0, K - 1 - A);
    p.accept_len[b] = A;
    p.bonus[b] = (int)key_index(__ldcg(&p.keys[(long long)b * K1 + A]));
    if (p.n_out) p.n_out[b] = nb;
    if (p.R_count) p.pack_off[b] = off;
  }
}

// Decides the window [w0, w1) of a windowed verification for the n sequences
// of `list` (NULL: 0..n-1), the same in every CTA.  s_first[l] = the first
// row of the window (rows below K only) whose argmax differs from the draft
// token, as an offset from w0, or w1 - w0 if none: the sequence goes on (to
// the next window) unless the window ends the block (w1 = K + 1, then A = K).
// The sequences that end here take consecutive packed rows in list order
// after `base`; s_off[l] receives their offsets.  Their outputs are written by
// CTA l mod grid.  Returns the rows they claim; fills s_live (with the going-
// on sequences, in order) and *n_live when s_live is not NULL.
__device__ int decide_window(const VerifyParams& p, const int32_t* list, int n, int w0, int w1, int base,
                             int* s_first, int* s_off, int* s_live, int* n_live, int* s_warp) {
  const int K = p.K, K1 = K + 1;
  const int wp = w1 - w0;
  const bool last = w1 == K1;
  for (int l = threadIdx.x; l < n; l += kThreads) s_first[l] = wp;
  __syncthreads();
  for (int idx = threadIdx.x; idx < n * wp; idx += kThreads) {
    const int l = idx / wp, r = idx - l * wp, i = w0 + r;
    const int b = list ? __ldcg(list + l) : l;
    if (i < K && (int)key_index(__ldcg(&p.keys[(long long)b * K1 + i])) != __ldg(p.draft + (long long)b * K + i))
      atomicMin(&s_first[l], r);
  }
  __syncthreads();
  int rows = 0, nl = 0;
  for (int c0 = 0; c0 < n; c0 += kThreads) {
    const int l = c0 + (int)threadIdx.x;
    const int first = l < n ? s_first[l] : 0;
    const bool goes_on = l < n && first == wp && !last;
    const int A = w0 + min(first, K - w0);  // first == wp in the last window: A = K
    const int nb = (l < n && !goes_on) ? max(0, K - 1 - A) : 0;
    int chunk;
    const int off = block_exclusive_scan(nb, s_warp, &chunk);
    if (l < n) s_off[l] = base + rows + off;
    rows += chunk;
    if (s_live) {
      const int pos = block_exclusive_scan(goes_on ? 1 : 0, s_warp, &chunk);
      if (goes_on) s_live[nl + pos] = list ? __ldcg(list + l) : l;
      nl += chunk;
    }
  }
  __syncthreads();
  for (int l = blockIdx.x; l < n; l += gridDim.x) {
    const int first = s_first[l];
    if (first == wp && !last) continue;  // goes on
    write_decided(p, list ? __ldcg(list + l) : l, w0 + min(first, K - w0), s_off[l]);
  }
  if (n_live) *n_live = nl;
  return rows;
}

// Start of a later pass of the windowed schedule: decides the previous
// window [pi0, i0) for the previous pass's live sequences, then builds this
// pass's live list in s_live (CTA 0 publishes it, with the packed rows
// claimed so far, for the next pass and the finish kernel).  s_stage holds 3 B
// ints.  Returns the list's length.
__device__ int begin_later_pass(const VerifyParams& p, int* s_stage, int* s_warp) {
  const int n_prev = p.count_in ? (int)__ldcg(p.count_in) : p.B;
  const int base = p.base_in ? (int)__ldcg(p.base_in) : 0;
  int* s_first = s_stage;
  int* s_off = s_stage + p.B;
  int* s_live = s_stage + 2 * p.B;
  int n = 0;
  const int rows = decide_window(p, p.live_in, n_prev, p.pi0, p.i0, base, s_first, s_off, s_live, &n, s_warp);
  if (blockIdx.x == 0) {
    for (int l = threadIdx.x; l < n; l += kThreads) p.live_out[l] = s_live[l];
    if (threadIdx.x == 0) {
      *p.count_out = (uint32_t)n;
      *p.base_out = (uint32_t)(base + rows);
    }
  }
  __syncthreads();
  return n;
}

template <typename T, bool VEC>
__global__ void __launch_bounds__(kThreads, 2) verify_kernel(const VerifyParams p) {
  __shared__ unsigned long long s_red[kThreads / 32];
  __shared__ int s_t[kMaxK + 1];
  __shared__ int s_A[2];  // accepted length, packed-row offset
  __shared__ int s_last;
  extern __shared__ uint4 s_stage[];  // kCopyStage * kThreads vectors: row copies of the finaliser
  pdl_launch_dependents();  // the next kernel may take SMs as this grid's CTAs finish

  long long n_live = p.B;
  const int* s_list = nullptr;  // the pass's live sequences (NULL: 0..B-1)
  if (p.windowed && p.i0 > 0) {
    // a later pass: the previous pass's keys decide which sequences go on
    __shared__ int s_warp[kThreads / 32 + 1];
    pdl_wait();
    n_live = begin_later_pass(p, reinterpret_cast<int*>(s_stage), s_warp);
    s_list = reinterpret_cast<int*>(s_stage) + 2 * p.B;
  }
  const long long VV = p.slots_per_row;
  const int K1 = p.K + 1, W = p.i1 - p.i0;
  const long long per_seq = (long long)W * VV;
  const long long T_ = n_live * per_seq;
  // Active CTAs: at least kMinCtaBytes of logits each, no more than there are slots.
  const long long by_bytes = (T_ * (VEC ? 16 : (long long)sizeof(T)) + kMinCtaBytes - 1) / kMinCtaBytes;
  const long long G = min((long long)gridDim.x, min(by_bytes, T_));
  const long long c = blockIdx.x;

  long long s = c < G ? c * T_ / G : 0;
  const long long s_end = c < G ? (c + 1) * T_ / G : 0;
  while (s < s_end) {
    const long long vrow = s / VV;  // row of the pass: sequence vrow / W, window row vrow % W
    const long long l = vrow / W;
    const int b = s_list ? s_list[l] : (int)l;
    const int i = p.i0 + (int)(vrow - l * W);
    const long long seg_end = min(s_end, (vrow + 1) * VV);
    const int v0 = (int)(s - vrow * VV), v1 = (int)(seg_end - vrow * VV);
    const T* rowp = reinterpret_cast<const T*>(p.logits) + (long long)b * p.batch_stride +
                    (long long)i * p.row_stride;

    unsigned long long key = segment_key<T, VEC>(rowp, v0, v1, p.V);
    key = block_max_key(key, s_red);
    if (threadIdx.x == 0) atomicMax(&p.keys[(long long)b * K1 + i], key);
    s = seg_end;

    if (!p.windowed && (s == s_end || s % per_seq == 0)) {
      // This CTA has folded in all of its rows of sequence b.  The CTAs that
      // own slots of b are those from the owner of its first slot to the
      // owner of its last (every active CTA range is non-empty: G <= T_).
      const long long first = l * per_seq, last = first + per_seq - 1;
      const long long c_first = ((first + 1) * G - 1) / T_;
      const long long c_last = ((last + 1) * G - 1) / T_;
      const uint32_t count = (uint32_t)(c_last - c_first + 1);
      if (threadIdx.x == 0) {
        __threadfence();
        const uint32_t prev = atomicAdd(&p.tickets[b], 1u);
        s_last = (prev == count - 1u);
      }
      __syncthreads();
      if (s_last) {
        __threadfence();
        finalize_sequence<T>(p, b, s_t, s_A, s_stage);
      }
      __syncthreads();
    }
  }
}

// One row segment of the copies after verification, by one warp of 32
// lanes: `kind` 0 is the e~ row of position j (e, or m_j in the overwrite
// variant), 1 and 2 the m_j and u_j halves of its packed row, 3 its packed e
// row.  A is sequence b's accepted length, pack0 its first packed row.
// Nothing is copied where the item does not apply (a conditioned e~ row,
// which the conditioning kernels write; the packed halves of an
// unconditioned position).  CV: 16-byte vectors, kCopyBatch in flight per
// lane; elements otherwise.
constexpr int kCopyBatch = 8;
template <typename T, bool CV>
__device__ __forceinline__ void copy_segment(const VerifyParams& p, int b, int j, int kind, int A, long long pack0) {
  const int K = p.K, d = p.d;
  const int nb = (K - 1 - A) > 0 ? (K - 1 - A) : 0;
  const int lane = threadIdx.x & 31;
  const long long pos = (long long)b * K + j;
  const T* e = reinterpret_cast<const T*>(p.e);
  const T* hD = reinterpret_cast<const T*>(p.hD);
  const T* hT = reinterpret_cast<const T*>(p.hT);
  const T* src;
  T* dst;
  if (kind == 0) {
    if (p.cond_copy == kCondCopyKeep && j < nb) return;  // the conditioning kernels write it
    src = (p.cond_copy == kCondCopyM && j < nb) ? hD + (pos + A + 1) * d
                                                : e + (long long)b * p.e_batch_stride + (long long)j * p.e_pos_stride;
    dst = reinterpret_cast<T*>(p.e_out) + pos * d;
  } else {
    if (j >= nb) return;
    const long long row = pack0 + j;
    if (kind == 1) {
      src = hD + (pos + A + 1) * d;
      dst = reinterpret_cast<T*>(p.apack) + row * 2 * d;
      if (lane == 0) p.rowmap[row] = (int32_t)pos;
    } else if (kind == 2) {
      src = hT + (pos + A) * d;
      dst = reinterpret_cast<T*>(p.apack) + row * 2 * d + d;
    } else {
      src = e + pos * d;
      dst = reinterpret_cast<T*>(p.epack) + row * d;
    }
  }
  if constexpr (CV) {
    const int vpr = d * (int)sizeof(T) / 16;
    const uint4* s4 = reinterpret_cast<const uint4*>(src);
    uint4* d4 = reinterpret_cast<uint4*>(dst);
    for (int v0 = 0; v0 < vpr; v0 += 32 * kCopyBatch) {
      uint4 x[kCopyBatch];
#pragma unroll
      for (int k = 0; k < kCopyBatch; ++k) {
        const int v = v0 + k * 32 + lane;
        if (v < vpr) x[k] = __ldcs(s4 + v);
      }
#pragma unroll
      for (int k = 0; k < kCopyBatch; ++k) {
        const int v = v0 + k * 32 + lane;
        if (v < vpr) d4[v] = x[k];
      }
    }
  } else {
    for (int v = lane; v < d; v += 32) dst[v] = src[v];
  }
}

// The copies of a windowed verification, after its last pass (accept_len
// and the packed-row offsets hold every sequence's values by then).  Work
// items are row segments: (sequence b, position j, segment), the segments in
// order the row of e_out (when this position's e_out row is written here: e,
// or m_j in the overwrite variant), then, for conditioned positions of a
// packing round, the halves m_j and u_j of the packed row and the packed e
// row.  Each warp takes items in turn and copies one with its 32 lanes, each
// lane kCopyBatch 16-byte vectors in flight at a time (elements when CV is
// false); inactive items cost one decode.
template <typename T, bool CV>
__global__ void __launch_bounds__(kThreads, 2) verify_copy_kernel(const VerifyParams p) {
  pdl_launch_dependents();
  pdl_wait();
  const int K = p.K;
  const bool pack = p.R_count != nullptr;
  const int nseg = (p.e_out ? 1 : 0) + (pack ? (p.e_dense ? 3 : 2) : 0);
  const long long items = (long long)p.B * K * nseg;
  const long long warps = (long long)gridDim.x * (kThreads / 32);
  for (long long it = (long long)blockIdx.x * (kThreads / 32) + (threadIdx.x >> 5); it < items; it += warps) {
    const long long u = it / nseg;
    const int seg = (int)(it - u * nseg);
    const int b = (int)(u / K), j = (int)(u - (long long)b * K);
    const int kind = p.e_out ? seg : seg + 1;
    const int A = __ldg(p.accept_len + b);
    copy_segment<T, CV>(p, b, j, kind, A, kind > 0 ? (long long)__ldg(p.pack_off + b) : 0ll);
  }
}

// The end of a windowed verification, after its last pass.  Decides the
// sequences of the last window (decide_window over the last pass's live list,
// the same in every CTA; their outputs spread over the CTAs), sets R, and the
// last CTA to finish with the keys zeroes them and the passes' counters for
// the next call.  Then the row copies as in verify_copy_kernel: the
// unconditioned rows of e~ and the packed [m; u] (and e) rows, each warp one
// row segment at a time; a sequence decided by an earlier pass gives its
// accepted length and first packed row from accept_len and pack_off.  s_dyn
// holds 4 B ints.
template <typename T, bool CV>
__global__ void __launch_bounds__(kThreads, 2) verify_finish_kernel(const VerifyParams p) {
  extern __shared__ int s_dyn[];
  __shared__ int s_warp[kThreads / 32 + 1];
  __shared__ int s_last;
  pdl_launch_dependents();
  pdl_wait();
  const int B = p.B, K = p.K, K1 = K + 1;
  // after a single pass (no live lists) every sequence is decided here
  const int n_last = p.count_in ? (int)__ldcg(p.count_in) : B;
  const int base = p.base_in ? (int)__ldcg(p.base_in) : 0;
  int* s_first = s_dyn;         // [n_last]
  int* s_off = s_dyn + B;       // [n_last]
  int* s_mapA = s_dyn + 2 * B;  // [B]: accepted length of the sequences decided here, -1 for the others
  int* s_mapO = s_dyn + 3 * B;  // [B]: their first packed row
  for (int b = threadIdx.x; b < B; b += kThreads) s_mapA[b] = -1;
  __syncthreads();
  const int rows = decide_window(p, p.live_in, n_last, p.i0, K1, base, s_first, s_off, nullptr, nullptr, s_warp);
  for (int l = threadIdx.x; l < n_last; l += kThreads) {
    const int b = p.live_in ? __ldcg(p.live_in + l) : l;
    s_mapA[b] = p.i0 + min(s_first[l], K - p.i0);
    s_mapO[b] = s_off[l];
  }
  if (blockIdx.x == 0 && threadIdx.x == 0 && p.R_count) *p.R_count = base + rows;
  // every read of the keys above is done: the last CTA out resets them
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    s_last = atomicAdd(p.exits, 1u) == gridDim.x - 1u;
  }
  __syncthreads();
  if (s_last) {
    __threadfence();
    for (long long i = threadIdx.x; i < (long long)B * K1; i += kThreads) p.keys[i] = 0ull;
    if (threadIdx.x == 0) {
      for (int k = 0; k < p.n_counts; ++k) p.pass_counts[k] = 0u;
      *p.exits = 0u;
    }
  }
  // the row copies
  const bool pack = p.R_count != nullptr;
  const int nseg = (p.e_out ? 1 : 0) + (pack ? (p.e_dense ? 3 : 2) : 0);
  const long long items = (long long)B * K * nseg;
  const long long warps = (long long)gridDim.x * (kThreads / 32);
  for (long long it = (long long)blockIdx.x * (kThreads / 32) + (threadIdx.x >> 5); it < items; it += warps) {
    const long long u = it / nseg;
    const int seg = (int)(it - u * nseg);
    const int b = (int)(u / K), j = (int)(u - (long long)b * K);
    const int kind = p.e_out ? seg : seg + 1;  // 0 e_out row, 1 m half, 2 u half, 3 packed e
    const int Ah = s_mapA[b];
    const int A = Ah >= 0 ? Ah : __ldcg(p.accept_len + b);
    const long long off = kind == 0 ? 0ll : (long long)(Ah >= 0 ? s_mapO[b] : __ldcg(p.pack_off + b));
    copy_segment<T, CV>(p, b, j, kind, A, off);
  }
}

std::atomic<int> g_schedule{RETRACE_VERIFY_AUTO};
// Row windows from this batch-row size (B * V * element size) up: measured
// against one pass, windows win from B = 40-56 rows of 151936 bf16 logits
// when 2-7 draft tokens are accepted on average (the paper's acceptance
// lengths), from B = 72-96 when the acceptance is uniform over 0..K.
constexpr long long kWindowMinBatchRowBytes = 16ll << 20;
// Largest batch of the windowed schedule: every CTA keeps its decisions and
// live lists, up to 4 B ints, in 32 KB of shared memory.
constexpr int kWindowMaxB = kCopyStageBytes / 16;

// Row windows of the windowed schedule: the first kWindowRows rows, then
// windows half as long again as the one before (fewer, longer passes as the
// live sequences thin out), the last one stretched to row K when what would
// remain is shorter than half a window.  Writes the window starts (n + 1
// entries, the last = K1) and returns the number of passes n (1: one window
// holds every row).
inline int window_bounds(int K1, int* start) {
  int n = 0, i = 0, w = kWindowRows;
  start[0] = 0;
  while (i < K1 && n < kMaxWindowPasses) {
    int e = i + w;
    if (e >= K1 || 2 * (K1 - e) < w || n == kMaxWindowPasses - 1) e = K1;
    start[++n] = e;
    i = e;
    w += w / 2;
  }
  return n;
}

}  // namespace

int verify_windows(int B, int K, int V, int elem_bytes, bool have_workspace, bool argmax_out, int* start) {
  const int K1 = K + 1;
  const int n = window_bounds(K1, start);
  const int mode = g_schedule.load(std::memory_order_relaxed);
  const long long wave = (long long)B * V * elem_bytes;
  const bool windowed = have_workspace && !argmax_out && B > 0 && B <= kWindowMaxB && n > 1 &&
                        (mode == RETRACE_VERIFY_WINDOWS || (mode == RETRACE_VERIFY_AUTO && wave >= kWindowMinBatchRowBytes));
  if (windowed) return n;
  start[0] = 0;
  start[1] = K1;
  return 1;
}

namespace {

// Copies in 16-byte vectors for every tensor a verification copies.
inline bool copies_vectorised(const VerifyArgs& a, size_t es) {
  auto al = [](const void* q) { return (uintptr_t)q % 16 == 0; };
  return (a.d * es) % 16 == 0 && (!a.e_out || (al(a.e) && al(a.e_out))) &&
         (a.e_pos_stride * (long long)es) % 16 == 0 && (a.e_batch_stride * (long long)es) % 16 == 0 &&
         (a.cond_copy != kCondCopyM || al(a.hD)) &&
         (!a.R_count || (al(a.hD) && al(a.hT) && al(a.apack) && (!a.e_dense || al(a.epack))));
}

// verify_copy_kernel after the last pass (programmatically dependent): the
// 16-byte path when every copied tensor allows it.
template <typename T>
cudaError_t launch_copies(const VerifyArgs& a, const VerifyParams& p, long long grid, cudaStream_t stream) {
  const bool cv = copies_vectorised(a, sizeof(T));
  auto kern = cv ? verify_copy_kernel<T, true> : verify_copy_kernel<T, false>;
  return launch_dependent(kern, dim3((unsigned)grid), dim3(kThreads), 0, stream, 1u, p);
}

// verify_finish_kernel after the last windowed pass (programmatically
// dependent), with the 16-byte copy path when every copied tensor allows it.
template <typename T>
cudaError_t launch_finish(const VerifyArgs& a, const VerifyParams& p, long long grid, cudaStream_t stream) {
  const bool cv = copies_vectorised(a, sizeof(T));
  auto kern = cv ? verify_finish_kernel<T, true> : verify_finish_kernel<T, false>;
  return launch_dependent(kern, dim3((unsigned)grid), dim3(kThreads), (size_t)4 * a.B * sizeof(int), stream, 1u, p);
}

template <typename T, bool VEC>
cudaError_t launch_typed(const VerifyArgs& a, cudaStream_t stream) {
  DeviceInfo info;
  cudaError_t err = device_info(&info);
  if (err != cudaSuccess) return err;
  // Per device, filled by the first call (concurrent first calls may both
  // fill it; both set the same attribute and store the same value).
  static std::atomic<int> occ_cache[64];
  int occ = occ_cache[info.device & 63].load(std::memory_order_acquire);
  if (occ == 0) {
    err = cudaFuncSetAttribute(verify_kernel<T, VEC>, cudaFuncAttributeMaxDynamicSharedMemorySize, kCopyStageBytes);
    if (err != cudaSuccess) return err;
    err = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, verify_kernel<T, VEC>, kThreads, kCopyStageBytes);
    if (err != cudaSuccess) return err;
    if (occ < 1) occ = 1;
    occ_cache[info.device & 63].store(occ, std::memory_order_release);
  }
  VerifyParams p;
  p.logits = a.logits;
  p.B = a.B;
  p.K = a.K;
  p.V = a.V;
  p.row_stride = a.row_stride;
  p.batch_stride = a.batch_stride;
  p.draft = a.draft;
  p.accept_len = a.accept_len;
  p.committed = a.committed;
  p.bonus = a.bonus;
  p.target_argmax = a.target_argmax;
  p.n_out = a.n_out;
  p.keys = a.keys;
  p.tickets = a.tickets;
  const int E = VEC ? 16 / (int)sizeof(T) : 1;
  p.slots_per_row = (a.V + E - 1) / E;
  p.total_slots = (long long)a.B * (a.K + 1) * p.slots_per_row;
  p.e = a.e;
  p.e_batch_stride = a.e_batch_stride;
  p.e_pos_stride = a.e_pos_stride;
  p.e_out = a.e_out;
  p.d = a.d;
  p.hD = a.hD;
  p.hT = a.hT;
  p.e_dense = a.e_dense;
  p.apack = a.apack;
  p.epack = a.epack;
  p.rowmap = a.rowmap;
  p.R_count = a.R_count;
  p.cond_copy = a.cond_copy;
  p.i0 = 0;
  p.i1 = a.K + 1;
  p.pi0 = 0;
  p.windowed = 0;
  p.base_in = nullptr;
  p.base_out = nullptr;
  p.live_in = nullptr;
  p.count_in = nullptr;
  p.live_out = nullptr;
  p.count_out = nullptr;
  p.pass_counts = nullptr;
  p.n_counts = 0;
  p.exits = nullptr;
  p.defer_copies = 0;
  p.pack_off = a.pack_off;
  const int K1 = a.K + 1;
  int start[kMaxWindowPasses + 1];
  const int n_pass = verify_windows(a.B, a.K, a.V, (int)sizeof(T), a.live != nullptr, a.target_argmax != nullptr, start);
  const bool windowed = n_pass > 1;
  const long long grid_full = (long long)info.sm_count * occ;
  if (!windowed) {
    // Enough CTAs to fill every SM at full occupancy, but at least kMinCtaBytes of
    // logits per CTA so that small batches do not pay for idle CTAs (the
    // kernel trims its active CTAs the same way).
    const long long bytes = (long long)a.B * K1 * a.V * (long long)sizeof(T);
    long long grid = grid_full;
    const long long by_bytes = (bytes + kMinCtaBytes - 1) / kMinCtaBytes;
    if (by_bytes < grid) grid = by_bytes;
    if (grid > p.total_slots) grid = p.total_slots;
    if (grid < 1) grid = 1;
    // Row packing for the tensor-core projections with fewer sequences than
    // SMs: each finaliser would copy its sequence's rows on one SM after the
    // stream has ended, and the per-sequence arrival tickets of a few
    // sequences shared by every CTA serialise the end of the pass.  So the
    // pass only folds keys (as a window [0, K+1) of the windowed schedule),
    // and verify_finish_kernel decides every sequence, writes the outputs
    // and does the copies over its grid (target_argmax, every row's argmax,
    // stays with the finalisers).
    const bool defer = a.R_count && a.B < info.sm_count;
    if (defer && !a.target_argmax && a.live && a.pass_counts && a.B <= kWindowMaxB) {
      p.windowed = 1;
      verify_kernel<T, VEC><<<(unsigned)grid, kThreads, kCopyStageBytes, stream>>>(p);
      err = cudaGetLastError();
      if (err != cudaSuccess) return err;
      p.i0 = 0;
      p.live_in = nullptr;  // every sequence, no packed rows claimed before
      p.count_in = nullptr;
      p.base_in = nullptr;
      p.pass_counts = a.pass_counts + 1;
      p.n_counts = 2 * kMaxWindowPasses + 1;
      p.exits = a.pass_counts;
      long long fgrid = ((long long)a.B * a.K * 3 + 15) / 16;  // about a warp per row segment
      if (fgrid > grid_full) fgrid = grid_full;
      return launch_finish<T>(a, p, fgrid < 1 ? 1 : fgrid, stream);
    }
    p.defer_copies = defer ? 1 : 0;
    verify_kernel<T, VEC><<<(unsigned)grid, kThreads, kCopyStageBytes, stream>>>(p);
    err = cudaGetLastError();
    if (err != cudaSuccess || !defer) return err;
    const long long copy_grid = ((long long)a.B * a.K * 4 + 15) / 16;  // a warp per row segment
    return launch_copies<T>(a, p, copy_grid < grid_full ? copy_grid : grid_full, stream);
  }
  // Windowed: pass k reads rows [start[k], start[k+1]) of the sequences whose
  // draft tokens matched every earlier row.  Each pass after the first waits
  // for its predecessor inside the kernel (programmatic dependent launch),
  // rebuilds the live list from the previous window's keys and sizes its
  // work from it; pass k publishes its list for pass k + 1 (two buffers in
  // turn).  verify_finish_kernel writes the outputs and does the copies.
  // Counters: pass_counts[0] CTAs out of the finish kernel, [k] the length of
  // pass k's live list, [kMaxWindowPasses + 1 + k] the packed rows claimed by
  // the sequences decided before pass k's window.
  uint32_t* bases = a.pass_counts + kMaxWindowPasses + 1;
  p.windowed = 1;
  for (int k = 0; k < n_pass; ++k) {
    p.i0 = start[k];
    p.i1 = start[k + 1];
    p.pi0 = k > 0 ? start[k - 1] : 0;
    p.live_in = k <= 1 ? nullptr : a.live + (size_t)((k - 1) & 1) * a.B;  // pass 0 holds every sequence
    p.count_in = k <= 1 ? nullptr : a.pass_counts + (k - 1);
    p.base_in = k <= 1 ? nullptr : bases + (k - 1);
    p.live_out = k == 0 ? nullptr : a.live + (size_t)(k & 1) * a.B;
    p.count_out = k == 0 ? nullptr : a.pass_counts + k;
    p.base_out = k == 0 ? nullptr : bases + k;
    if (k == 0) {
      verify_kernel<T, VEC><<<(unsigned)grid_full, kThreads, kCopyStageBytes, stream>>>(p);
      err = cudaGetLastError();
    } else {
      err = launch_dependent(verify_kernel<T, VEC>, dim3((unsigned)grid_full), dim3(kThreads), kCopyStageBytes,
                             stream, 1u, p);
    }
    if (err != cudaSuccess) return err;
  }
  // the finish kernel decides the last window [start[n-1], K+1) for the last pass's live list
  p.i0 = start[n_pass - 1];
  p.live_in = a.live + (size_t)((n_pass - 1) & 1) * a.B;
  p.count_in = a.pass_counts + (n_pass - 1);
  p.base_in = bases + (n_pass - 1);
  p.pass_counts = a.pass_counts + 1;
  p.n_counts = 2 * kMaxWindowPasses + 1;  // every live count and base after the exit counter
  p.exits = a.pass_counts;
  return launch_finish<T>(a, p, grid_full, stream);
}

}  // namespace

cudaError_t launch_verify_copies(const VerifyArgs& a, retrace_dtype dtype, cudaStream_t stream) {
  DeviceInfo info;
  cudaError_t err = device_info(&info);
  if (err != cudaSuccess) return err;
  VerifyParams p{};
  p.B = a.B;
  p.K = a.K;
  p.V = a.V;
  p.accept_len = a.accept_len;
  p.e = a.e;
  p.e_batch_stride = a.e_batch_stride;
  p.e_pos_stride = a.e_pos_stride;
  p.e_out = a.e_out;
  p.d = a.d;
  p.hD = a.hD;
  p.hT = a.hT;
  p.e_dense = a.e_dense;
  p.apack = a.apack;
  p.epack = a.epack;
  p.rowmap = a.rowmap;
  p.R_count = a.R_count;
  p.cond_copy = a.cond_copy;
  p.pack_off = a.pack_off;
  const long long grid = (long long)info.sm_count * 2;
  return dtype == RETRACE_BF16 ? launch_copies<__nv_bfloat16>(a, p, grid, stream)
                               : launch_copies<float>(a, p, grid, stream);
}

int set_verify_schedule(int mode) {
  if (mode != RETRACE_VERIFY_AUTO && mode != RETRACE_VERIFY_FULL && mode != RETRACE_VERIFY_WINDOWS) return -1;
  return g_schedule.exchange(mode);
}

cudaError_t launch_verify(const VerifyArgs& a, retrace_dtype dtype, cudaStream_t stream) {
  const size_t es = dtype == RETRACE_BF16 ? 2 : 4;
  const bool vec = ((uintptr_t)a.logits % 16 == 0) && ((a.row_stride * (long long)es) % 16 == 0) &&
                   ((a.batch_stride * (long long)es) % 16 == 0);
  if (dtype == RETRACE_BF16)
    return vec ? launch_typed<__nv_bfloat16, true>(a, stream)
               : launch_typed<__nv_bfloat16, false>(a, stream);
  return vec ? launch_typed<float, true>(a, stream) : launch_typed<float, false>(a, stream);
}

}  // namespace retrace
