// Stochastic verification of a draft block (speculative sampling) at
// temperature T with top-k / top-p filtering (Appendix "Evaluation Protocol":
// T = 1, top_p = 0.95, top_k = 20).  The paper keeps the underlying
// verification unchanged; the rule implemented is standard speculative
// sampling on the filtered distributions p (target) and q (drafter):
// accept x_i iff u_i q_i(x_i) < p_i(x_i); at the first rejection A draw the
// appended token from max(0, p_A - q_A) (renormalised; p_A if that is zero),
// else the bonus from p_K; draws are inverse-CDF in the filtered order.
//
// Only the top_k logits of a row enter its filtered distribution, so the
// row's full softmax is never formed:
//   sampled_topk_kernel      one CTA per row (target rows, then drafter rows):
//                            elements above a proven lower bound of the row's
//                            k-th largest (a sample's k-th largest, then the
//                            best warp's k-th largest candidate) go to per-warp
//                            buffers; the CTA merges the warps' lists by rank;
//   sampled_finalize_kernel  one CTA per sequence: the filtered
//                            probabilities of the draft tokens from the sorted
//                            lists (eight positions at a time, one per warp),
//                            the accept tests in order, the draw, and for a
//                            round the copies and packing of e~ and [m; u].
// The outputs depend only on the target rows 0..A_b and the drafter rows
// 0..min(A_b, K-1).  In the windowed schedule the pair of kernels runs once
// per row window, over the sequences that accepted every earlier draft (live
// lists in the workspace); the copies and packing then follow in the greedy
// path's copy kernel.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "common.cuh"
#include "internal.h"

namespace retrace {
namespace {

constexpr int kThreads = 512;
constexpr int kWarps = kThreads / 32;
constexpr int kTrigger = kMaxTopK;       // a warp's buffer is cut to its top k once it holds more keys
constexpr int kBuf = kTrigger + 32 * 8;  // candidate keys per warp: the trigger + one bf16 chunk of the warp

struct TopkParams {
  const void* tlogits;
  long long t_row, t_batch;
  const void* dlogits;
  long long d_row, d_batch;
  int B, K, V, k;
  unsigned long long* keys;  // [B (2K+1), kMaxTopK]: target rows b*(K+1)+i, then drafter rows
  // Row window of this pass ([0, K+1) in one pass): target rows [i0, i1) and
  // drafter rows [i0, min(i1, K)) of the listed sequences (NULL: 0..B-1;
  // count_in NULL: B of them, else written by the previous pass).
  int i0, i1;
  const int32_t* live_in;
  const uint32_t* count_in;
};

// The largest key whose value is below v: every element of value >= v beats it.
__device__ __forceinline__ unsigned long long below_value(float v) {
  return ((unsigned long long)ordered_bits(v) << 32) - 1ull;
}

template <typename T>
struct Chunk;  // one lane's share of a chunk (16 bytes): raw bits, partial maxima, candidate masks
template <>
struct Chunk<__nv_bfloat16> {
  static constexpr int E = 8;
  using Part = __nv_bfloat162;  // two running maxima
  uint4 w;
  __device__ Part part() const {
    const __nv_bfloat162 a = *reinterpret_cast<const __nv_bfloat162*>(&w.x);
    const __nv_bfloat162 b = *reinterpret_cast<const __nv_bfloat162*>(&w.y);
    const __nv_bfloat162 c = *reinterpret_cast<const __nv_bfloat162*>(&w.z);
    const __nv_bfloat162 d = *reinterpret_cast<const __nv_bfloat162*>(&w.w);
    return __hmax2(__hmax2(a, b), __hmax2(c, d));
  }
  static __device__ Part combine(Part a, Part b) { return __hmax2(a, b); }
  static __device__ float finish(Part m) { return fmaxf(__low2float(m), __high2float(m)); }
  static __device__ Part lowest() { return __floats2bfloat162_rn(-INFINITY, -INFINITY); }
  // bit e set iff element e >= tv
  __device__ unsigned mask(float tv) const {
    const uint32_t q[4] = {w.x, w.y, w.z, w.w};
    unsigned m = 0;
#pragma unroll
    for (int h = 0; h < 4; ++h) {
      m |= (bf16_lo(q[h]) >= tv ? 1u : 0u) << (2 * h);
      m |= (bf16_hi(q[h]) >= tv ? 1u : 0u) << (2 * h + 1);
    }
    return m;
  }
  __device__ float value(int e) const {
    const uint32_t x = e < 2 ? w.x : e < 4 ? w.y : e < 6 ? w.z : w.w;
    return (e & 1) ? bf16_hi(x) : bf16_lo(x);
  }
  __device__ void load(const __nv_bfloat16* p) { w = __ldcs(reinterpret_cast<const uint4*>(p)); }
  __device__ void fill() { w = make_uint4(0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u); }  // -inf
  __device__ void set_single(float v) { w = make_uint4(pack_bf16x2(v, -INFINITY), 0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u); }
};
template <>
struct Chunk<float> {
  static constexpr int E = 4;
  using Part = float;
  float4 w;
  __device__ Part part() const { return fmaxf(fmaxf(w.x, w.y), fmaxf(w.z, w.w)); }
  static __device__ Part combine(Part a, Part b) { return fmaxf(a, b); }
  static __device__ float finish(Part m) { return m; }
  static __device__ Part lowest() { return -INFINITY; }
  __device__ unsigned mask(float tv) const {
    return (w.x >= tv ? 1u : 0u) | (w.y >= tv ? 2u : 0u) | (w.z >= tv ? 4u : 0u) | (w.w >= tv ? 8u : 0u);
  }
  __device__ float value(int e) const { return e == 0 ? w.x : e == 1 ? w.y : e == 2 ? w.z : w.w; }
  __device__ void load(const float* p) { w = __ldcs(reinterpret_cast<const float4*>(p)); }
  __device__ void fill() { w = make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY); }
  __device__ void set_single(float v) { w = make_float4(v, -INFINITY, -INFINITY, -INFINITY); }
};

// Ranks the warp's `n` buffered keys (distinct) and keeps the largest
// min(n, k) in descending order at the front of the buffer; returns their
// count.  Lane-parallel rank counting (every key's rank is the number of
// larger keys); the thresholds keep n small.
__device__ int warp_compact(unsigned long long* buf, unsigned long long* tmp, int n, int k, int lane) {
  for (int a = lane; a < n; a += 32) {
    const unsigned long long x = buf[a];
    int rank = 0;
    for (int c = 0; c < n; ++c) rank += buf[c] > x ? 1 : 0;
    if (rank < k) tmp[rank] = x;
  }
  __syncwarp();
  const int m = n < k ? n : k;
  for (int a = lane; a < m; a += 32) buf[a] = tmp[a];
  __syncwarp();
  return m;
}

// One CTA per row; warp w scans a contiguous part of it, U chunks (16 bytes
// per lane each) per step.  Elements are kept as candidates only above a
// proven lower bound of the row's k-th largest key: first the k-th largest
// of a sample (every lane's maximum over its first U chunks: each is an
// element of the row), then any warp's k-th largest candidate so far (the
// maximum of both in s_thr).  One vote per step on the packed maxima decides whether
// any element can pass (the common case: none); otherwise a ballot per chunk
// skips the chunks without one, and the lanes that have some append them, by
// bit mask, to the warp's buffer with shared-memory atomics.  A buffer that
// passes a trigger is cut to its top k.  The row's top k are merged from the
// warps' sorted lists.
struct TopkSmem {
  unsigned long long buf[kWarps][kBuf];
  unsigned long long tmp[kWarps][kMaxTopK];
  float sample[kThreads];
  int n[kWarps];
  unsigned long long thr;
};

// The top-k list of one row x into p.keys slot `row` (the whole CTA).
template <typename T>
__device__ __forceinline__ void topk_row(const TopkParams& p, const T* x, int row, TopkSmem& sm) {
  using CT = Chunk<T>;
  using Part = typename CT::Part;
  constexpr int E = CT::E;
  constexpr int U = 4;
  auto& s_buf = sm.buf;
  auto& s_tmp = sm.tmp;
  auto& s_sample = sm.sample;
  auto& s_n = sm.n;
  auto& s_thr = sm.thr;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int V = p.V, k = p.k;
  unsigned long long* buf = s_buf[warp];
  unsigned long long* tmp = s_tmp[warp];
  if (lane == 0) s_n[warp] = 0;
  const unsigned FULL = 0xFFFFFFFFu;
  const bool vec = (V % E == 0) && ((uintptr_t)x % 16 == 0);
  const int per = vec ? E : 1;  // elements of the row per lane per chunk
  const int span = 32 * per;
  const int nchunks = (V + span - 1) / span;
  const int c0 = (int)((long long)nchunks * warp / kWarps), c1 = (int)((long long)nchunks * (warp + 1) / kWarps);
  // k <= kMaxTopK = kTrigger: a compaction leaves at most kTrigger keys, so
  // the buffer has room for the next chunk
  const int trigger = kTrigger;
  const unsigned valid_bits = vec ? (1u << E) - 1u : 1u;  // the scalar path fills elements 1.. with -inf

  // chunk c of this lane: valid iff c < c1 and its first element is in the row
  auto load_checked = [&](CT (&ch)[U], int c) {
#pragma unroll
    for (int q = 0; q < U; ++q) {
      const int base = (c + q) * span + lane * per;
      ch[q].fill();
      if (c + q < c1 && base < V) {
        if (vec) ch[q].load(x + base);
        else ch[q].set_single(to_f32(x[base]));
      }
    }
  };
  // U chunks that lie inside the row and the warp's range (the main loop)
  auto load_full = [&](CT (&ch)[U], int c) {
    const T* ptr = x + c * span + lane * per;
#pragma unroll
    for (int q = 0; q < U; ++q) {
      if (vec) ch[q].load(ptr + q * span);
      else ch[q].set_single(to_f32(ptr[q * span]));
    }
  };
  auto process = [&](const CT (&ch)[U], int c, bool full) {
    const unsigned long long t = *(volatile unsigned long long*)&s_thr;
    const float tv = t ? key_value(t) : -INFINITY;
    Part m = ch[0].part();
#pragma unroll
    for (int q = 1; q < U; ++q) m = CT::combine(m, ch[q].part());
    // invalid chunks hold -inf; they can pass only with no bound at all
    if (!__any_sync(FULL, CT::finish(m) >= tv)) return;
#pragma unroll
    for (int q = 0; q < U; ++q) {
      const int base = (c + q) * span + lane * per;
      const bool has = CT::finish(ch[q].part()) >= tv && (full || (c + q < c1 && base < V));
      if (!__ballot_sync(FULL, has)) continue;
      const unsigned bits = has ? ch[q].mask(tv) & valid_bits : 0u;
      for (unsigned r = bits; r; r &= r - 1) {
        const int e = __ffs(r) - 1;
        const unsigned long long key = make_key(ch[q].value(e), (uint32_t)(base + e));
        if (key > t) buf[atomicAdd(&s_n[warp], 1)] = key;
      }
      __syncwarp();
      int n = *(volatile int*)&s_n[warp];
      if (n > trigger) {  // keep the top k so far (kBuf leaves room for one more chunk)
        n = warp_compact(buf, tmp, n, k, lane);
        if (lane == 0) s_n[warp] = n;
        if (n >= k && lane == 0) atomicMax(&s_thr, buf[k - 1]);
        __syncwarp();
      }
    }
  };

  CT ch[U];
  load_checked(ch, c0);
  {
    // Sampling: each lane's maximum over its first U chunks, sorted within
    // the warp (bitonic, by shuffles); warp 0 merges the 16 sorted lists up
    // to the k-th largest, a lower bound of the row's k-th largest.
    Part m = ch[0].part();
#pragma unroll
    for (int q = 1; q < U; ++q) m = CT::combine(m, ch[q].part());
    float v = CT::finish(m);
    if (v != v) v = -INFINITY;  // all-NaN lane: no sample
#pragma unroll
    for (int size = 2; size <= 32; size <<= 1) {
#pragma unroll
      for (int stride = size >> 1; stride > 0; stride >>= 1) {
        const float o = __shfl_xor_sync(FULL, v, stride);
        const bool keep_max = ((lane & size) == 0) == ((lane & stride) == 0);  // descending at size 32
        v = keep_max ? fmaxf(v, o) : fminf(v, o);
      }
    }
    s_sample[threadIdx.x] = v;
    if (threadIdx.x == 0) s_thr = 0ull;
    __syncthreads();
    if (warp == 0) {
      int pos = 0;
      float head = lane < kWarps ? s_sample[lane * 32] : -INFINITY;
      float best = -INFINITY;
      for (int r = 0; r < k; ++r) {
        best = head;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) best = fmaxf(best, __shfl_xor_sync(FULL, best, off));
        const unsigned own = __ballot_sync(FULL, head == best);
        if (lane == __ffs(own) - 1) {
          ++pos;
          head = pos < 32 ? s_sample[lane * 32 + pos] : -INFINITY;
        }
      }
      if (lane == 0) s_thr = best > -INFINITY ? below_value(best) : 0ull;
    }
    __syncthreads();
  }
  process(ch, c0, false);
  // chunks [0, nfull) lie wholly inside the row
  const int cfull = c1 < V / span ? c1 : V / span;
  int c = c0 + U;
  for (; c + U <= cfull; c += U) {
    load_full(ch, c);
    process(ch, c, true);
  }
  for (; c < c1; c += U) {
    load_checked(ch, c);
    process(ch, c, false);
  }
  int n = warp_compact(buf, tmp, *(volatile int*)&s_n[warp], k, lane);
  if (lane == 0) s_n[warp] = n;
  __syncthreads();
  // Merge the warps' sorted lists: lane w of warp 0 holds the head of list w;
  // the largest head is the next key of the row.
  if (warp == 0) {
    unsigned long long* out = p.keys + (long long)row * kMaxTopK;
    int pos = 0;
    const int len = lane < kWarps ? s_n[lane] : 0;
    for (int r = 0; r < k; ++r) {
      const unsigned long long head = pos < len ? s_buf[lane][pos] : 0ull;
      const unsigned long long best = warp_max_key(head);
      if (lane == 0) out[r] = best;  // 0 once every list is exhausted (V < k)
      if (head == best && best != 0ull) ++pos;
    }
  }
}

// One row per CTA (the first pass: every row of the window), or a grid of
// resident CTAs looping over the rows of a later pass (its live count is
// known only on the device; a grid of the whole batch's rows would spend
// whole waves of CTAs that only find they have nothing to do).  The rows of
// a pass: the window's target rows of each listed sequence, then its drafter
// rows; `row` is the row's slot in p.keys.
template <typename T, bool LOOP>
__global__ void __launch_bounds__(kThreads, 3) sampled_topk_kernel(const TopkParams p) {
  __shared__ TopkSmem sm;
  pdl_launch_dependents();  // the finalize kernel may take SMs as these CTAs finish
  int n_live = p.B;
  if (p.count_in) {  // a later pass: the previous finalize wrote the live list
    pdl_wait();
    n_live = (int)__ldcg(p.count_in);
  }
  const int wt = p.i1 - p.i0, wd = min(p.i1, p.K) - p.i0;
  const int rows = n_live * (wt + wd);  // B (2K+1) at most, below 2^31
  auto row_of = [&](int r0, const T*& x) -> int {
    if (r0 < n_live * wt) {
      const int l = r0 / wt, i = p.i0 + (r0 - l * wt);
      const int b = p.live_in ? __ldg(p.live_in + l) : l;
      x = reinterpret_cast<const T*>(p.tlogits) + b * p.t_batch + i * p.t_row;
      return b * (p.K + 1) + i;
    }
    const int r = r0 - n_live * wt, l = r / wd, i = p.i0 + (r - l * wd);
    const int b = p.live_in ? __ldg(p.live_in + l) : l;
    x = reinterpret_cast<const T*>(p.dlogits) + b * p.d_batch + i * p.d_row;
    return p.B * (p.K + 1) + b * p.K + i;
  };
  if constexpr (!LOOP) {
    if ((int)blockIdx.x >= rows) return;
    const T* x;
    const int row = row_of(blockIdx.x, x);
    topk_row<T>(p, x, row, sm);
  } else {
    for (int r0 = blockIdx.x; r0 < rows; r0 += gridDim.x) {
      const T* x;
      const int row = row_of(r0, x);
      topk_row<T>(p, x, row, sm);
      __syncthreads();  // the row's shared buffers are read to the end before the next row
    }
  }
}

struct FinalizeParams {
  const unsigned long long* keys;
  int B, K, V, k;
  float inv_T, top_p;
  const int32_t* draft;
  const float* uniforms;
  int32_t* accept_len;
  int32_t* committed;
  int32_t* bonus;
  // a whole round (optional): n, copies of the unconditioned rows of e~, and
  // the packed [m; u] rows of the tensor-core projections
  int32_t* n_out;
  const void* e;
  long long e_batch_stride, e_pos_stride;
  void* e_out;
  int d, elem;
  const void* hD;
  const void* hT;
  int e_dense;
  void* apack;
  void* epack;
  int32_t* rowmap;
  int32_t* R_count;
  // Windowed schedule: accept tests over rows [i0, min(i1, K)) of the listed
  // sequences (live_in NULL: 0..B-1, count_in NULL: B); a sequence that
  // accepts them all, with rows left, goes to live_out.  The last pass's last
  // CTA out zeroes the passes' counters.  With defer_copies the finaliser
  // only claims the packed rows (pack_off) and a later kernel copies.
  int i0, i1;
  const int32_t* live_in;
  const uint32_t* count_in;
  int32_t* live_out;
  uint32_t* count_out;
  uint32_t* pass_counts;
  int n_counts;
  uint32_t* exits;
  int defer_copies;
  int32_t* pack_off;
};

// The filtered distribution of one row, lane j holding entries j and 32 + j
// of the sorted list: weight (0 beyond the top-p cut) and token (-1 if none).
struct RowDist {
  float w[2];
  int tok[2];
  float total;  // sum of the kept weights
};

__device__ RowDist row_dist(const FinalizeParams& p, long long row, int lane) {
  const unsigned FULL = 0xFFFFFFFFu;
  const unsigned long long* keys = p.keys + row * kMaxTopK;
  RowDist r;
  const float v0 = key_value(keys[0]);
  float w[2];
  int tok[2];
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int j = 32 * h + lane;
    const unsigned long long key = j < p.k ? keys[j] : 0ull;
    tok[h] = key ? (int)key_index(key) : -1;
    w[h] = key ? expf((key_value(key) - v0) * p.inv_T) : 0.f;
  }
  // softmax over the top k, then the shortest prefix reaching top_p
  float z = w[0] + w[1];
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) z += __shfl_xor_sync(FULL, z, off);
  float c0 = w[0];  // inclusive prefix over entries 0..31
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const float t = __shfl_up_sync(FULL, c0, off);
    if (lane >= off) c0 += t;
  }
  const float s0 = __shfl_sync(FULL, c0, 31);
  float c1 = w[1];
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const float t = __shfl_up_sync(FULL, c1, off);
    if (lane >= off) c1 += t;
  }
  c1 += s0;
  // entry j is kept iff the prefix before it is below top_p
  const float before0 = c0 - w[0], before1 = c1 - w[1];
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const float before = h == 0 ? before0 : before1;
    const bool keep = tok[h] >= 0 && before < p.top_p * z;
    r.w[h] = keep ? w[h] : 0.f;
    r.tok[h] = keep ? tok[h] : -1;
  }
  float t = r.w[0] + r.w[1];
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) t += __shfl_xor_sync(FULL, t, off);
  r.total = t;
  return r;
}

// Probability of token y under the row distribution (same value on every lane).
__device__ float dist_prob(const RowDist& r, int y) {
  const unsigned FULL = 0xFFFFFFFFu;
  float w = (r.tok[0] == y ? r.w[0] : 0.f) + (r.tok[1] == y ? r.w[1] : 0.f);
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) w += __shfl_xor_sync(FULL, w, off);
  return w / r.total;
}

// Inverse-CDF draw over entries in list order with weights wt (this lane's
// two entries): the first entry whose inclusive cumulative weight exceeds
// u * total; the last kept entry if rounding leaves none.
__device__ int draw(const RowDist& r, const float wt[2], float u, int lane) {
  const unsigned FULL = 0xFFFFFFFFu;
  float c0 = wt[0];
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const float t = __shfl_up_sync(FULL, c0, off);
    if (lane >= off) c0 += t;
  }
  const float s0 = __shfl_sync(FULL, c0, 31);
  float c1 = wt[1];
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const float t = __shfl_up_sync(FULL, c1, off);
    if (lane >= off) c1 += t;
  }
  c1 += s0;
  const float total = __shfl_sync(FULL, c1, 31);
  const float target = u * total;
  const unsigned b0 = __ballot_sync(FULL, wt[0] > 0.f && c0 > target);
  const unsigned b1 = __ballot_sync(FULL, wt[1] > 0.f && c1 > target);
  int src, h;
  if (b0) {
    src = __ffs(b0) - 1;
    h = 0;
  } else if (b1) {
    src = __ffs(b1) - 1;
    h = 1;
  } else {  // last entry with weight
    const unsigned l0 = __ballot_sync(FULL, wt[0] > 0.f), l1 = __ballot_sync(FULL, wt[1] > 0.f);
    if (l1) {
      src = 31 - __clz(l1);
      h = 1;
    } else {
      src = 31 - __clz(l0);
      h = 0;
    }
  }
  const int t0 = __shfl_sync(FULL, r.tok[0], src), t1 = __shfl_sync(FULL, r.tok[1], src);
  return h == 0 ? t0 : t1;
}

// One CTA per sequence.  The accept tests need only p_i(x_i) and q_i(x_i):
// the warps compute them for eight positions at a time, one position each,
// and thread 0 takes the decisions in order, so the chain of dependent
// distributions is one per chunk instead of one per position.  Warp 0 then
// draws the appended token; every thread writes the outputs and, for a round,
// copies and packs rows.
__device__ void sampled_finalize_sequence(const FinalizeParams& p, int b) {
  constexpr int kFinWarps = 8;
  __shared__ int s_A, s_y, s_off;
  __shared__ float s_px[kFinWarps], s_qx[kFinWarps];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int K = p.K, K1 = K + 1;
  const int32_t* dr = p.draft + (long long)b * K;
  const long long tbase = (long long)b * K1, dbase = (long long)p.B * K1 + (long long)b * K;
  const float* u = p.uniforms + (long long)b * K1;
  // rows before i0 were accepted in earlier passes
  int A = p.i1 == K1 ? K : -1;  // -1: every row of the window accepted, rows left
  const int hi = min(p.i1, K);
  for (int c0 = p.i0; c0 < hi; c0 += kFinWarps) {
    const int i = c0 + warp;
    if (i < hi) {
      const int x = dr[i];
      float px = -1.f, qx = 0.f;  // px < 0: a token outside [0, V) is rejected
      if (x >= 0 && x < p.V) {
        const RowDist pt = row_dist(p, tbase + i, lane);
        const RowDist qd = row_dist(p, dbase + i, lane);
        px = dist_prob(pt, x);
        qx = dist_prob(qd, x);
      }
      if (lane == 0) {
        s_px[warp] = px;
        s_qx[warp] = qx;
      }
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      int a = -1;
      for (int j = 0; j < kFinWarps && c0 + j < hi; ++j) {
        if (!(s_px[j] >= 0.f && u[c0 + j] * s_qx[j] < s_px[j])) {
          a = c0 + j;
          break;
        }
      }
      s_A = a;
    }
    __syncthreads();
    const int a = s_A;
    if (a >= 0) {
      A = a;
      break;
    }
  }
  if (A < 0) {  // every draft of the window accepted: on to the next pass
    if (threadIdx.x == 0) p.live_out[atomicAdd(p.count_out, 1u)] = b;
    return;
  }
  if (warp == 0) {
    const RowDist pt = row_dist(p, tbase + A, lane);
    int y;
    if (A < K) {
      // residual max(0, p - q) over the target's kept tokens
      const RowDist qd = row_dist(p, dbase + A, lane);
      float res[2];
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        // q of this lane's token: every lane looks it up in the drafter's list
        float qw = 0.f;
        for (int s2 = 0; s2 < 32; ++s2) {
          const int t0 = __shfl_sync(0xFFFFFFFFu, qd.tok[0], s2), t1 = __shfl_sync(0xFFFFFFFFu, qd.tok[1], s2);
          const float w0 = __shfl_sync(0xFFFFFFFFu, qd.w[0], s2), w1 = __shfl_sync(0xFFFFFFFFu, qd.w[1], s2);
          if (pt.tok[h] >= 0 && t0 == pt.tok[h]) qw = w0;
          if (pt.tok[h] >= 0 && t1 == pt.tok[h]) qw = w1;
        }
        res[h] = pt.tok[h] >= 0 ? fmaxf(0.f, pt.w[h] / pt.total - qw / qd.total) : 0.f;
      }
      float rs = res[0] + res[1];
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) rs += __shfl_xor_sync(0xFFFFFFFFu, rs, off);
      y = rs > 0.f ? draw(pt, res, u[K], lane) : draw(pt, pt.w, u[K], lane);
    } else {
      y = draw(pt, pt.w, u[K], lane);
    }
    if (lane == 0) {
      s_y = y;
      const int nb = K - 1 - A > 0 ? K - 1 - A : 0;
      s_off = (p.R_count && nb > 0) ? atomicAdd(p.R_count, nb) : 0;
      if (p.defer_copies && p.R_count) p.pack_off[b] = s_off;
    }
  }
  __syncthreads();
  const int y = s_y;
  for (int i = threadIdx.x; i < K1; i += blockDim.x) {
    const long long o = (long long)b * K1 + i;
    p.committed[o] = i < A ? dr[i] : (i == A ? y : -1);
  }
  const int nb = K - 1 - A > 0 ? K - 1 - A : 0;
  if (threadIdx.x == 0) {
    p.accept_len[b] = A;
    p.bonus[b] = y;
    if (p.n_out) p.n_out[b] = nb;
  }
  if (!p.e_out || p.defer_copies) return;
  // rows j >= n_b keep the drafter input, bit for bit
  const long long base_row = (long long)b * K;
  const char* e_b = static_cast<const char*>(p.e) + b * p.e_batch_stride * p.elem;
  const long long rows = K - nb;
  const bool vec = (p.d * p.elem) % 16 == 0 && (uintptr_t)e_b % 16 == 0 && (uintptr_t)p.e_out % 16 == 0 &&
                   (p.e_pos_stride * p.elem) % 16 == 0;
  if (vec) {
    const int vpr = p.d * p.elem / 16;
    const long long pos_vec = p.e_pos_stride * p.elem / 16;
    const uint4* src = reinterpret_cast<const uint4*>(e_b);
    uint4* dst = reinterpret_cast<uint4*>(p.e_out) + (base_row + nb) * vpr;
    copy_vectors(rows * vpr, [&](long long i) { return __ldg(src + (nb + i / vpr) * pos_vec + i % vpr); },
                 [&](long long i, const uint4& v) { dst[i] = v; });
  } else if (p.elem == 2) {
    const uint16_t* src = reinterpret_cast<const uint16_t*>(e_b);
    uint16_t* dst = reinterpret_cast<uint16_t*>(p.e_out) + (base_row + nb) * p.d;
    for (long long i = threadIdx.x; i < rows * p.d; i += blockDim.x) {
      const long long j = nb + i / p.d, c = i % p.d;
      dst[i] = src[j * p.e_pos_stride + c];
    }
  } else {
    const uint32_t* src = reinterpret_cast<const uint32_t*>(e_b);
    uint32_t* dst = reinterpret_cast<uint32_t*>(p.e_out) + (base_row + nb) * p.d;
    for (long long i = threadIdx.x; i < rows * p.d; i += blockDim.x) {
      const long long j = nb + i / p.d, c = i % p.d;
      dst[i] = src[j * p.e_pos_stride + c];
    }
  }
  if (!p.R_count || nb == 0) return;
  // packed rows [m_j; u_j] = [hD[b, A+1+j]; hT[b, A+j]] (Eq. 4-5), and e[b, j]
  // for a per-position e; the tensor-core path is bf16 with 16-byte rows
  const int off = s_off;
  const int vpr = p.d / 8;
  const uint4* e_v = reinterpret_cast<const uint4*>(e_b);
  const long long pos_vec = p.e_pos_stride / 8;
  for (int j = threadIdx.x; j < nb; j += blockDim.x) p.rowmap[off + j] = b * K + j;
  const uint4* hD = reinterpret_cast<const uint4*>(p.hD);
  const uint4* hT = reinterpret_cast<const uint4*>(p.hT);
  uint4* ap = reinterpret_cast<uint4*>(p.apack);
  copy_vectors(
      (long long)nb * 2 * vpr,
      [&](long long i) {
        const long long j = i / (2 * vpr), c = i % (2 * vpr);
        return c < vpr ? __ldg(hD + (base_row + A + 1 + j) * vpr + c) : __ldg(hT + (base_row + A + j) * vpr + c - vpr);
      },
      [&](long long i, const uint4& v) { ap[(long long)off * 2 * vpr + i] = v; });
  if (p.e_dense) {
    uint4* ep = reinterpret_cast<uint4*>(p.epack);
    copy_vectors((long long)nb * vpr, [&](long long i) { return __ldg(e_v + (i / vpr) * pos_vec + i % vpr); },
                 [&](long long i, const uint4& v) { ep[(long long)off * vpr + i] = v; });
  }
}

__global__ void __launch_bounds__(256) sampled_finalize_kernel(const FinalizeParams p) {
  pdl_launch_dependents();
  pdl_wait();  // the sorted lists come from the top-k kernel
  const int n_live = p.count_in ? (int)__ldcg(p.count_in) : p.B;
  if ((int)blockIdx.x < n_live) {
    sampled_finalize_sequence(p, p.live_in ? __ldg(p.live_in + blockIdx.x) : (int)blockIdx.x);
  }
  if (p.exits && threadIdx.x == 0) {  // the last pass's last CTA out resets the live counters
    __threadfence();
    if (atomicAdd(p.exits, 1u) == gridDim.x - 1u) {
      for (int k = 0; k < p.n_counts; ++k) p.pass_counts[k] = 0u;
      *p.exits = 0u;
    }
  }
}

}  // namespace

cudaError_t launch_verify_sampled(const SampledArgs& a, retrace_dtype dtype, cudaStream_t stream) {
  if (a.B <= 0) return cudaSuccess;
  TopkParams tp{};
  tp.tlogits = a.tlogits;
  tp.t_row = a.t_row;
  tp.t_batch = a.t_batch;
  tp.dlogits = a.dlogits;
  tp.d_row = a.d_row;
  tp.d_batch = a.d_batch;
  tp.B = a.B;
  tp.K = a.K;
  tp.V = a.V;
  tp.k = a.top_k;
  tp.keys = a.keys;
  FinalizeParams fp{};
  fp.keys = a.keys;
  fp.B = a.B;
  fp.K = a.K;
  fp.V = a.V;
  fp.k = a.top_k;
  fp.inv_T = 1.f / a.temperature;
  fp.top_p = a.top_p;
  fp.draft = a.draft;
  fp.uniforms = a.uniforms;
  fp.accept_len = a.accept_len;
  fp.committed = a.committed;
  fp.bonus = a.bonus;
  fp.n_out = a.n_out;
  fp.e = a.e;
  fp.e_batch_stride = a.e_batch_stride;
  fp.e_pos_stride = a.e_pos_stride;
  fp.e_out = a.e_out;
  fp.d = a.d;
  fp.elem = dtype == RETRACE_BF16 ? 2 : 4;
  fp.hD = a.hD;
  fp.hT = a.hT;
  fp.e_dense = a.e_dense;
  fp.apack = a.apack;
  fp.epack = a.epack;
  fp.rowmap = a.rowmap;
  fp.R_count = a.R_count;
  fp.pack_off = a.pack_off;
  // The outputs depend only on the target rows 0..A_b and the drafter rows
  // 0..min(A_b, K-1): the same row windows as greedy verification.  Pass k
  // scans the window's rows of the sequences that accepted every earlier
  // draft (top-k kernel), then runs their accept tests (finalize kernel).
  int start[kMaxWindowPasses + 1];
  const int n_pass = verify_windows(a.B, a.K, a.V, (int)fp.elem, a.live != nullptr, false, start);
  DeviceInfo info;
  cudaError_t e0 = device_info(&info);
  if (e0 != cudaSuccess) return e0;
  // Copies after the last pass, balanced over the grid: always with windows;
  // in one pass when it packs rows for fewer sequences than SMs (otherwise
  // each finalising CTA copies its own sequence's rows).
  const bool defer = a.e_out && (n_pass > 1 || (a.R_count && a.B < info.sm_count));
  const long long topk_resident = (long long)info.sm_count * 3;  // __launch_bounds__(kThreads, 3)
  fp.defer_copies = defer ? 1 : 0;
  for (int k = 0; k < n_pass; ++k) {
    const bool last = k == n_pass - 1;
    tp.i0 = fp.i0 = start[k];
    tp.i1 = fp.i1 = start[k + 1];
    tp.live_in = fp.live_in = k == 0 ? nullptr : a.live + (size_t)((k - 1) & 1) * a.B;
    tp.count_in = fp.count_in = k == 0 ? nullptr : a.pass_counts + k;
    fp.live_out = last ? nullptr : a.live + (size_t)(k & 1) * a.B;
    fp.count_out = last ? nullptr : a.pass_counts + k + 1;
    fp.pass_counts = last && n_pass > 1 ? a.pass_counts + 1 : nullptr;
    fp.n_counts = last ? n_pass - 1 : 0;
    fp.exits = last && n_pass > 1 ? a.pass_counts : nullptr;
    const int wt = tp.i1 - tp.i0, wd = (tp.i1 < a.K ? tp.i1 : a.K) - tp.i0;
    // the first pass: one CTA per row; later passes: resident CTAs looping
    const long long rows_max = (long long)a.B * (wt + wd);
    const long long grid_n = k == 0 ? rows_max : (rows_max < topk_resident ? rows_max : topk_resident);
    const dim3 grid((unsigned)(grid_n > 0 ? grid_n : 1));
    cudaError_t err;
    auto topk = k == 0 ? (dtype == RETRACE_BF16 ? sampled_topk_kernel<__nv_bfloat16, false>
                                                 : sampled_topk_kernel<float, false>)
                       : (dtype == RETRACE_BF16 ? sampled_topk_kernel<__nv_bfloat16, true>
                                                 : sampled_topk_kernel<float, true>);
    if (k == 0) {
      topk<<<grid, kThreads, 0, stream>>>(tp);
      err = cudaGetLastError();
    } else {
      err = launch_dependent(topk, grid, dim3(kThreads), 0, stream, 1, tp);
    }
    if (err != cudaSuccess) return err;
    err = launch_dependent(sampled_finalize_kernel, dim3((unsigned)a.B), dim3(256), 0, stream, 1, fp);
    if (err != cudaSuccess) return err;
  }
  if (!defer) return cudaSuccess;
  // the row copies and packing, balanced over the grid
  VerifyArgs c{};
  c.B = a.B;
  c.K = a.K;
  c.V = a.V;
  c.accept_len = a.accept_len;
  c.e = a.e;
  c.e_batch_stride = a.e_batch_stride;
  c.e_pos_stride = a.e_pos_stride;
  c.e_out = a.e_out;
  c.d = a.d;
  c.hD = a.hD;
  c.hT = a.hT;
  c.e_dense = a.e_dense;
  c.apack = a.apack;
  c.epack = a.epack;
  c.rowmap = a.rowmap;
  c.R_count = a.R_count;
  c.pack_off = a.pack_off;
  c.cond_copy = kCondCopyKeep;
  return launch_verify_copies(c, dtype, stream);
}

}  // namespace retrace
