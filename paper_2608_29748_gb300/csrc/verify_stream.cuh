// Greedy verification streamed through shared memory, for the fused round kernel.
//
// Same computation as verify.cu (Algorithm 1 Verify and commit steps), laid
// out so that verification can share every SM with the tensor-core warps:
//   * the contiguous [B, K+1, V] bf16 logits are cut into 8 KB chunks, and
//     the chunks into groups of eight that CTAs take in order from a global
//     counter, so faster SMs take more of them and sequences complete in
//     order while the kernel runs;
//   * one producer thread per CTA streams its groups' chunks with bulk TMA
//     copies (cp.async.bulk) into a ring of shared-memory buffers, which keeps
//     a fixed number of bytes in flight independent of the thread count;
//   * consumer warp w takes every eighth chunk of the CTA whole (ring buffer
//     w): it loads the chunk into registers, releases the buffer, reduces each
//     row segment to a 64-bit (value, ~index) key with shuffles and posts the
//     keys in a shared-memory record; consumers never touch global memory;
//   * the CTA's bookkeeper warp takes the records in order, keeps a running
//     key per row, folds it into the row's global key (atomicMax) when the row
//     changes, and when the CTA moves past a sequence adds the number of the
//     sequence's chunks it read to the sequence's arrival count;
//   * sequence b is finalised by the finaliser warp of CTA b mod G once its
//     arrival count reaches the number of chunks it overlaps (independent of
//     which CTAs read them); a fixed owner spreads the copies evenly;
//   * the finaliser computes the first mismatch by ballot, writes the committed
//     tokens and bonus, and moves the rows with bulk TMA copies through a
//     staging buffer: copies of the unconditioned drafter inputs, and packing
//     of the conditioned rows [m_j; u_j] = [hD[b, A+1+j]; hT[b, A+j]] (Eq. 4-5)
//     for the projections, which it then publishes per 128-row block.
// Every wait is bounded and taken by one lane, its outcome shared by shuffle;
// there is no barrier a failed wait could leave half-arrived.
#pragma once

#include "common.cuh"

namespace retrace {

// One ring buffer per consumer warp: warp w consumes exactly the chunks that
// land in buffer w, so it waits on every phase of its buffer's barriers in
// order (a phase-parity wait must never be more than one phase ahead).
constexpr int kConsumerWarps = 8;
constexpr int kRingBufs = kConsumerWarps;
constexpr int kChunkSlots = 512;  // 16-byte slots per chunk (8 KB)
constexpr int kChunkBytes = kChunkSlots * 16;
constexpr int kStageBytes = 16384;
constexpr int kRecords = 64;      // chunk key records between consumers and the bookkeeper
constexpr int kGroupChunks = 16;  // chunks per grab of the global counter (128 KB)
constexpr uint32_t kNoChunk = 0xFFFFFFFFu;  // end of a CTA's stream

struct VerifyStreamParams {
  const __nv_bfloat16* logits;  // contiguous [B, K+1, V]
  int B, K, V;
  const int32_t* draft;
  int32_t* accept_len;
  int32_t* committed;
  int32_t* bonus;
  int32_t* target_argmax;  // optional
  int32_t* n_out;          // optional
  unsigned long long* keys;
  uint32_t* tickets;
  const __nv_bfloat16* e;
  long long e_batch_stride, e_pos_stride;  // (0, 0) broadcast or (K*d, d) dense
  __nv_bfloat16* e_out;
  int d;
  const __nv_bfloat16* hD;
  const __nv_bfloat16* hT;
  int e_dense;
  __nv_bfloat16* apack;
  __nv_bfloat16* epack;
  int32_t* rowmap;
  uint32_t* R_count;
  uint32_t* rows_ready;  // per 128-row block of packed rows
  uint32_t* seq_done;
  uint32_t* chunk_next;  // global counter of chunk groups handed out
  long long total_slots;  // B (K+1) V / 8, below 2^32
  uint32_t total_chunks;
  int slots_per_row;  // V / 8 (V a multiple of 8, V >= 8 * kChunkSlots)
  uint32_t* status;
};


struct VerifyStreamSmem {
  uint64_t full[kRingBufs];
  uint64_t empty[kRingBufs];
  uint64_t stage_bar;
  uint32_t chunk_of[kRingBufs];  // chunk held by each buffer (kNoChunk: end of stream)
  // record of the CTA's it-th chunk in slot it % kRecords: the keys of its
  // first row and of the next row (if the chunk reaches it) and the chunk;
  // key0 != 0 marks a full slot
  unsigned long long rec_key0[kRecords];
  unsigned long long rec_key1[kRecords];
  uint32_t rec_chunk[kRecords];
};

__device__ __forceinline__ float vs_max8(const uint4& v) {
  const __nv_bfloat162 a = *reinterpret_cast<const __nv_bfloat162*>(&v.x);
  const __nv_bfloat162 b = *reinterpret_cast<const __nv_bfloat162*>(&v.y);
  const __nv_bfloat162 c = *reinterpret_cast<const __nv_bfloat162*>(&v.z);
  const __nv_bfloat162 d = *reinterpret_cast<const __nv_bfloat162*>(&v.w);
  const __nv_bfloat162 m = __hmax2(__hmax2(a, b), __hmax2(c, d));
  return fmaxf(__low2float(m), __high2float(m));
}

__device__ __forceinline__ float vs_elem(const uint4& v, int q) {
  const uint32_t w = (q < 2) ? v.x : (q < 4) ? v.y : (q < 6) ? v.z : v.w;
  return (q & 1) ? bf16_hi(w) : bf16_lo(w);
}

__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
               "l"(src), "r"(bytes), "r"(bar)
               : "memory");
}

__device__ void vs_init(VerifyStreamSmem& sm) {
  for (int i = 0; i < kRingBufs; ++i) {
    mbar_init(smem_u32(&sm.full[i]), 1);
    mbar_init(smem_u32(&sm.empty[i]), 1);  // one consumer warp per chunk
  }

  for (int i = 0; i < kRecords; ++i) sm.rec_key0[i] = sm.rec_key1[i] = 0ull;
  for (int i = 0; i < kRingBufs; ++i) sm.chunk_of[i] = kNoChunk;
  mbar_init(smem_u32(&sm.stage_bar), 1);
}

// Chunks overlapping sequence b (a chunk that straddles two sequences counts
// for both): the arrival count that completes the sequence.
__device__ __forceinline__ uint32_t seq_chunks(const VerifyStreamParams& p, int b) {
  const long long per_seq = (long long)(p.K + 1) * p.slots_per_row;
  const long long first = (long long)b * per_seq, last = first + per_seq - 1;
  return (uint32_t)(last / kChunkSlots - first / kChunkSlots + 1);
}

// Producer (one thread): takes groups of chunks from the global counter in
// order and streams them into the ring; then hands every consumer an
// end-of-stream buffer.
__device__ void vs_producer(const VerifyStreamParams& p, VerifyStreamSmem& sm, uint32_t ring, volatile int* abort) {
  uint32_t it = 0;
  bool ok = true;
  const uint32_t groups = (p.total_chunks + kGroupChunks - 1) / kGroupChunks;
  // two group indices requested ahead, so the counter's latency stays hidden
  uint32_t g_next = atomicAdd(p.chunk_next, 1u);
  uint32_t g_after = atomicAdd(p.chunk_next, 1u);
  while (ok && g_next < groups) {
    const uint32_t g = g_next;
    g_next = g_after;
    g_after = atomicAdd(p.chunk_next, 1u);
    const uint32_t c_end = min((g + 1) * kGroupChunks, p.total_chunks);
    for (uint32_t c = g * kGroupChunks; c < c_end; ++c, ++it) {
      const uint32_t s = it % kRingBufs, ph = (it / kRingBufs) & 1u;
      if (!mbar_wait_bounded(smem_u32(&sm.empty[s]), ph ^ 1u, abort)) {
        ok = false;
        break;
      }
      const long long base = (long long)c * kChunkSlots;
      const uint32_t bytes = (uint32_t)min((long long)kChunkSlots, p.total_slots - base) * 16u;
      sm.chunk_of[s] = c;  // published by the arrive below
      mbar_arrive_expect_tx(smem_u32(&sm.full[s]), bytes);
      bulk_load(ring + s * kChunkBytes, p.logits + base * 8, bytes, smem_u32(&sm.full[s]));
    }
  }
  for (int e = 0; ok && e < kRingBufs; ++e, ++it) {  // end of stream, one buffer per consumer
    const uint32_t s = it % kRingBufs, ph = (it / kRingBufs) & 1u;
    if (!mbar_wait_bounded(smem_u32(&sm.empty[s]), ph ^ 1u, abort)) {
      ok = false;
      break;
    }
    sm.chunk_of[s] = kNoChunk;
    mbar_arrive(smem_u32(&sm.full[s]));  // completes the phase without bytes
  }
  if (!ok) {
    *abort = 1;
    atomicOr(p.status, kFlagWaitTimeout);
    volatile int never = 0;  // drain this CTA's own copies still in flight
    const uint32_t first = it > kRingBufs ? it - kRingBufs : 0;
    for (uint32_t k = first; k < it; ++k)
      mbar_wait_bounded(smem_u32(&sm.full[k % kRingBufs]), (k / kRingBufs) & 1u, &never);
  }
}

__device__ __forceinline__ void bulk_store(void* dst, uint32_t src, uint32_t bytes) {
  asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(dst), "r"(src), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

// Lane 0: loads `n` rows of `bytes` into the staging buffer (one bulk copy
// each, at staging + k * bytes) and waits for them.  Bounded.
__device__ __forceinline__ bool stage_rows(VerifyStreamSmem& sm, uint32_t staging, const void* const* src, int n,
                                           uint32_t bytes, uint32_t* uses, volatile int* abort) {
  const uint32_t bar = smem_u32(&sm.stage_bar);
  mbar_arrive_expect_tx(bar, bytes * (uint32_t)n);
  for (int k = 0; k < n; ++k) bulk_load(staging + (uint32_t)k * bytes, src[k], bytes, bar);
  const bool ok = mbar_wait_bounded(bar, *uses & 1u, abort);
  ++*uses;
  return ok;
}

// Finalises sequence b (one warp): Algorithm 1 commit step, the unconditioned
// inputs e~ = e, and the packed rows of the projections.
__device__ bool vs_finalize(const VerifyStreamParams& p, VerifyStreamSmem& sm, uint32_t staging, int b, int lane,
                            uint32_t* uses, volatile int* abort) {
  const int K = p.K, K1 = K + 1, d = p.d;
  const unsigned FULL = 0xFFFFFFFFu;
  const unsigned long long* keys = p.keys + (long long)b * K1;
  int A = K;
  for (int base = 0; base < K; base += 32) {
    const int i = base + lane;
    bool mismatch = false;
    if (i < K) mismatch = (int)key_index(__ldcg(keys + i)) != p.draft[(long long)b * K + i];
    const unsigned bal = __ballot_sync(FULL, mismatch);
    if (bal) {
      A = base + __ffs(bal) - 1;
      break;
    }
  }
  const int tA = (int)key_index(__ldcg(keys + A));
  for (int i = lane; i < K1; i += 32) {
    const long long o = (long long)b * K1 + i;
    const int t = (int)key_index(__ldcg(keys + i));
    p.committed[o] = (i <= A) ? t : -1;
    if (p.target_argmax) p.target_argmax[o] = t;
  }
  __syncwarp();
  for (int i = lane; i < K1; i += 32) p.keys[(long long)b * K1 + i] = 0ull;
  const int nb = (K - 1 - A) > 0 ? (K - 1 - A) : 0;
  int off = 0;
  if (lane == 0) {
    p.accept_len[b] = A;
    p.bonus[b] = tA;
    if (p.n_out) p.n_out[b] = nb;
    p.tickets[b] = 0u;
    if (nb > 0) off = (int)atomicAdd(p.R_count, (uint32_t)nb);
  }
  off = __shfl_sync(FULL, off, 0);
  for (int j = lane; j < nb; j += 32) p.rowmap[off + j] = b * K + j;
  const uint32_t row_bytes = (uint32_t)d * 2u;
  const long long base_row = (long long)b * K;
  int ok = 1;
  if (lane == 0) {
    // rows j >= nb keep the drafter input: e~ = e
    if (!p.e_dense) {
      const void* src[1] = {p.e};
      ok = stage_rows(sm, staging, src, 1, row_bytes, uses, abort);
      for (int j = nb; ok && j < K; ++j) bulk_store(p.e_out + (base_row + j) * d, staging, row_bytes);
      bulk_commit();
      bulk_wait_read();
    } else {
      for (int j = nb; ok && j < K; ++j) {
        const void* src[1] = {p.e + (base_row + j) * d};
        ok = stage_rows(sm, staging, src, 1, row_bytes, uses, abort);
        if (ok) bulk_store(p.e_out + (base_row + j) * d, staging, row_bytes);
        bulk_commit();
        bulk_wait_read();
      }
    }
    // packed rows: [m_j; u_j] = [hD[b, A+1+j]; hT[b, A+j]] (Eq. 4-5), e rows for a dense e
    for (int j = 0; ok && j < nb; ++j) {
      const void* src[2] = {p.hD + (base_row + A + 1 + j) * d, p.hT + (base_row + A + j) * d};
      ok = stage_rows(sm, staging, src, 2, row_bytes, uses, abort);
      if (ok) bulk_store(p.apack + (long long)(off + j) * 2 * d, staging, 2 * row_bytes);
      bulk_commit();
      bulk_wait_read();
      if (ok && p.e_dense) {
        const void* esrc[1] = {p.e + (base_row + j) * d};
        ok = stage_rows(sm, staging, esrc, 1, row_bytes, uses, abort);
        if (ok) bulk_store(p.epack + (long long)(off + j) * d, staging, row_bytes);
        bulk_commit();
        bulk_wait_read();
      }
    }
    bulk_wait_all();
    // the packed rows were written by the async proxy; order them before the
    // generic release that publishes them
    asm volatile("fence.proxy.async.global;" ::: "memory");
  }
  ok = __shfl_sync(FULL, ok, 0);
  if (!ok) return false;
  __threadfence();
  __syncwarp();
  if (lane == 0) {
    for (int g = off; g < off + nb;) {
      const int blk = g / 128;
      const int end = (blk + 1) * 128 < off + nb ? (blk + 1) * 128 : off + nb;
      atomicAdd(p.rows_ready + blk, (uint32_t)(end - g));
      g = end;
    }
    __threadfence();
    atomicAdd(p.seq_done, 1u);
  }
  return true;
}

// Bookkeeper (lane 0 of one warp): this CTA's chunk records in order.
__device__ void vs_bookkeeper(const VerifyStreamParams& p, VerifyStreamSmem& sm, volatile int* abort) {
  const uint32_t VV = (uint32_t)p.slots_per_row, K1 = (uint32_t)p.K + 1u;
  long long cur_row = -1;
  unsigned long long cur_key = 0ull;
  int cur_seq = -1;
  uint32_t cur_cnt = 0, counted = kNoChunk;  // chunks of cur_seq read; the last one counted
  bool ok = true;
  // The CTA is done with cur_seq: its row keys, folded in before, are
  // released with its chunk count.
  auto leave = [&]() {
    __threadfence();
    atomicAdd(&p.tickets[cur_seq], cur_cnt);
  };
  auto visit = [&](uint32_t r, unsigned long long key, uint32_t c) {
    if ((long long)r == cur_row) {
      cur_key = umax64(cur_key, key);
    } else {
      if (cur_row >= 0) atomicMax(&p.keys[cur_row], cur_key);
      const int seq = (int)(r / K1);
      if (seq != cur_seq) {
        if (cur_seq >= 0) leave();
        cur_seq = seq;
        cur_cnt = 0;
        counted = kNoChunk;
      }
      cur_row = r;
      cur_key = key;
    }
    if (c != counted) {
      ++cur_cnt;
      counted = c;
    }
  };
  for (uint32_t it = 0;; ++it) {
    const uint32_t slot = it % kRecords;
    unsigned long long key0 = 0ull;
    ok = spin_until([&] { return (key0 = *(volatile unsigned long long*)&sm.rec_key0[slot]) != 0ull; }, abort, 0);
    if (!ok) break;
    __threadfence_block();
    const unsigned long long key1 = *(volatile unsigned long long*)&sm.rec_key1[slot];
    const uint32_t c = *(volatile uint32_t*)&sm.rec_chunk[slot];
    __threadfence_block();
    *(volatile unsigned long long*)&sm.rec_key0[slot] = 0ull;  // slot free again
    if (c == kNoChunk) break;
    const uint32_t base = c * (uint32_t)kChunkSlots;
    const uint32_t n = (uint32_t)min((long long)kChunkSlots, p.total_slots - base);
    const uint32_t row0 = base / VV;
    const uint32_t split = min((uint32_t)kChunkSlots, (row0 + 1u) * VV - base);
    visit(row0, key0, c);
    if (n > split) visit(row0 + 1u, key1, c);
  }
  if (ok && cur_row >= 0) {
    atomicMax(&p.keys[cur_row], cur_key);
    leave();
  }
  if (!ok) {
    *abort = 1;
    atomicOr(p.status, kFlagWaitTimeout);
  }
}

__device__ __forceinline__ uint32_t vs_ld_acquire(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Finaliser warp of CTA `cta`: sequences cta, cta + G, ... in order, each once
// all of its chunks are in.
__device__ void vs_finalizer(const VerifyStreamParams& p, VerifyStreamSmem& sm, uint32_t staging, int cta, int ncta,
                             int lane, volatile int* abort) {
  const unsigned FULL = 0xFFFFFFFFu;
  uint32_t uses = 0;
  for (int b = cta; b < p.B; b += ncta) {
    int ok = 1;
    if (lane == 0) {
      const uint32_t need = seq_chunks(p, b);
      ok = spin_until([&] { return vs_ld_acquire(p.tickets + b) >= need; }, abort, 256) ? 1 : 0;
    }
    ok = __shfl_sync(FULL, ok, 0);
    __syncwarp();     // the other lanes after lane 0's acquire
    __threadfence();  // every lane: the row keys of all CTAs that read the sequence
    if (!ok || !vs_finalize(p, sm, staging, b, lane, &uses, abort)) {
      if (lane == 0) {
        *abort = 1;
        atomicOr(p.status, kFlagWaitTimeout);
      }
      return;
    }
  }
}

// Warp argmax of per-lane (best value, first slot, vector): returns the key
// (value, lowest element index) of the warp's maximum for a row whose first
// slot is `row_start`; identical on every lane.  Float max first, then the
// lowest slot among the lanes holding it, then that lane resolves the element.
__device__ __forceinline__ unsigned long long vs_warp_key(float best, int slot, const uint4& vec, long long base,
                                                          long long row_start) {
  const unsigned FULL = 0xFFFFFFFFu;
  float m = best;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(FULL, m, o));
  int cand = (slot >= 0 && best == m) ? slot : 0x7FFFFFFF;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) cand = min(cand, __shfl_xor_sync(FULL, cand, o));
  if (cand == 0x7FFFFFFF) return 0ull;  // no slot of this row in the warp's share
  unsigned long long key = 0ull;
  if (slot == cand) {
    const long long slot_in_row = base + slot - row_start;
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      if (vs_elem(vec, q) == m) {
        key = make_key(m, (uint32_t)(slot_in_row * 8 + q));
        break;
      }
    }
  }
  const unsigned owner = __ballot_sync(FULL, slot == cand);
  return __shfl_sync(FULL, key, __ffs(owner) - 1);
}

// Posts the record of the CTA's it-th chunk (lane 0; bounded wait for the
// bookkeeper to free the slot).
__device__ __forceinline__ bool vs_post(VerifyStreamSmem& sm, uint32_t it, unsigned long long key0,
                                        unsigned long long key1, uint32_t c, volatile int* abort) {
  const uint32_t slot = it % kRecords;
  if (!spin_until([&] { return *(volatile unsigned long long*)&sm.rec_key0[slot] == 0ull; }, abort, 32))
    return false;  // the bookkeeper is behind
  *(volatile unsigned long long*)&sm.rec_key1[slot] = key1;
  *(volatile uint32_t*)&sm.rec_chunk[slot] = c;
  __threadfence_block();
  *(volatile unsigned long long*)&sm.rec_key0[slot] = key0;
  return true;
}

// Consumer warp w (0..7): every eighth chunk of this CTA (ring buffer w), whole.
__device__ void vs_consumer(const VerifyStreamParams& p, VerifyStreamSmem& sm, const uint4* ring, int w, int lane,
                            volatile int* abort) {
  const unsigned FULL = 0xFFFFFFFFu;
  const uint32_t VV = (uint32_t)p.slots_per_row;
  bool failed = false;
  for (uint32_t it = (uint32_t)w;; it += kConsumerWarps) {
    const uint32_t s = it % kRingBufs, ph = (it / kRingBufs) & 1u;  // s == w
    int ok = 1;
    uint32_t c = kNoChunk;
    if (lane == 0) {
      ok = mbar_wait_bounded(smem_u32(&sm.full[s]), ph, abort) ? 1 : 0;
      if (ok) c = *(volatile uint32_t*)&sm.chunk_of[s];  // after the acquire
    }
    ok = __shfl_sync(FULL, ok, 0);
    c = __shfl_sync(FULL, c, 0);
    __syncwarp();  // the other lanes' reads of the buffer after lane 0's acquire
    if (!ok) {
      failed = true;
      break;
    }
    if (c == kNoChunk) {  // end of stream: pass it on to the bookkeeper
      if (lane == 0) ok = vs_post(sm, it, 1ull, 0ull, kNoChunk, abort) ? 1 : 0;
      failed = __shfl_sync(FULL, ok, 0) == 0;
      break;
    }
    // The whole chunk into registers, then the buffer goes back at once.
    uint4 x[kChunkSlots / 32];
    const uint4* buf = ring + (size_t)s * kChunkSlots;
#pragma unroll
    for (int q = 0; q < kChunkSlots / 32; ++q) x[q] = buf[q * 32 + lane];
    __syncwarp();
    if (lane == 0) mbar_arrive(smem_u32(&sm.empty[s]));
    const uint32_t base = c * (uint32_t)kChunkSlots;
    const int n = (int)min((long long)kChunkSlots, p.total_slots - base);
    const uint32_t row_start = base / VV * VV;
    const int split = (int)min((uint32_t)kChunkSlots, row_start + VV - base);  // slots in the first row
    float b0 = -INFINITY, b1 = -INFINITY;
    int s0 = -1, s1 = -1;
    uint4 v0 = make_uint4(0, 0, 0, 0), v1 = make_uint4(0, 0, 0, 0);
#pragma unroll
    for (int q = 0; q < kChunkSlots / 32; ++q) {
      const int local = q * 32 + lane;
      if (local < n) {
        const float m = vs_max8(x[q]);
        if (local < split) {
          if (m > b0 || s0 < 0) {  // earliest slot among equal maxima
            b0 = m;
            s0 = local;
            v0 = x[q];
          }
        } else if (m > b1 || s1 < 0) {
          b1 = m;
          s1 = local;
          v1 = x[q];
        }
      }
    }
    const unsigned long long key0 = vs_warp_key(b0, s0, v0, base, row_start);
    const unsigned long long key1 = (n > split) ? vs_warp_key(b1, s1, v1, base, row_start + VV) : 0ull;
    if (lane == 0) ok = vs_post(sm, it, key0, key1, c, abort) ? 1 : 0;
    ok = __shfl_sync(FULL, ok, 0);
    if (!ok) {
      failed = true;
      break;
    }
  }
  if (failed && lane == 0) {
    *abort = 1;
    atomicOr(p.status, kFlagWaitTimeout);
  }
}

}  // namespace retrace
