// Host-side declarations shared by the libretrace translation units.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include <algorithm>
#include <atomic>

#include "../../include/retrace.h"

namespace retrace {

constexpr int kMaxK = 1024;  // largest draft block the kernels accept

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Workspace layout (all offsets 256-byte aligned):
//   status   uint32 [64]        [0] device status word
//   sync     uint32 [32+blocks] counters of a conditioning pass (row count, tile queue,
//                               gate-bias progress, per-128-row-block progress)
//   keys     uint64 [B*(K+1)]   per-row argmax keys, zero between calls
//   tickets  uint32 [B]         per-sequence CTA arrival counters, zero between calls
//   live     int32  [2*B]       windowed verification: live sequence lists of two passes
//   poff     int32  [B]         windowed verification: first packed row of each sequence
//   counts   uint32 [2(1+passes)] windowed verification: [0] CTAs out of the finish
//                               kernel, [k] sequences live into pass k, [17 + k] packed
//                               rows claimed before pass k's window; zero between calls
//   ge       fp32   [d]         W_g[:, :d] e for a broadcast e
//   r        elem   [R_max, d]  compacted corrected signal, R_max = B*(K-1)
//   apack    elem   [R_max, 2d] packed [m; u] rows (tensor-core path)
//   epack    elem   [R_max, d]  packed per-position e rows (tensor-core path, dense e)
//   rowmap   int32  [R_max]     packed row g -> position b*K + j
//   lrz      fp32   [S, R_max, 64]  low-rank path: split partials of the latent P m
//   lrt      fp32   [S, R_max, 32]  low-rank path: split partials of B_c[:, 64:] u
//   lrrho    elem   [R_max, 64]     low-rank path: corrected latent rho
constexpr int kLowRankLatent = 64;      // rank of the rejected-suffix latents
constexpr int kLowRankCorrection = 32;  // rank of the target-aware correction
constexpr int kLowRankSplits = 8;       // split-K parts per half of the [m; u] reduction
//   skeys    uint64 [B*(2K+1), 64]  sampled verification: top-k keys per target and drafter row
//   swp      fp32                   split partials of the small-R conditioning GEMMs, or the
//                                   K halves of the CTA-pair kernel's split gate tiles
constexpr int kMaxTopK = 64;            // largest top_k of sampled verification
constexpr int kWindowRows = 4;          // rows per pass of windowed verification
constexpr int kMaxWindowPasses = 16;    // most passes of windowed verification
// Small-R conditioning (at most kSwapMaxRows packed rows): the GEMMs as
// split-K tiles of 128 weight rows against N tiles of up to 256 rows, one
// grid of at most max(kSwapMaxCtas, work tiles) CTAs, each writing an fp32
// partial of at most 128 x min(256, rows) values.  Taken while the gate
// GEMM's work tiles (2d/128 x N tiles) fit in kSwapMaxCtas.
constexpr int kSwapMaxRows = 1024;
constexpr int kSwapMaxCtas = 256;
inline size_t swap_part_bytes(long long B, long long K, long long d) {
  const long long rmax = B * (K > 1 ? K - 1 : 0);
  if (rmax <= 0 || rmax > kSwapMaxRows || d <= 0) return 0;
  const long long rows = (rmax + 15) / 16 * 16;
  const long long ntiles = (rows + 255) / 256;
  if ((2 * d / 128) * ntiles > kSwapMaxCtas) return 0;
  const long long box = rows < 256 ? rows : 256;
  return (size_t)(kSwapMaxCtas * 128 * box * 4);
}
// CTA-pair conditioning (every other bf16 shape with d a multiple of 256): a
// last wave of at most kPairSplitTiles gate tiles runs as two K halves per
// tile on two pairs.  Each half writes its fp32 accumulator (two CTAs x 128
// rows x 256 columns) to the same region as the small-R partials, and counts
// on one ticket per CTA and epilogue warp in the sync area.
constexpr int kPairSplitTiles = 8;
inline size_t pair_split_bytes(long long B, long long K, long long d, size_t elem) {
  const long long rmax = B * (K > 1 ? K - 1 : 0);
  if (rmax <= 0 || elem != 2 || d <= 0 || d % 256 != 0 || swap_part_bytes(B, K, d) != 0) return 0;
  return (size_t)kPairSplitTiles * 2 * 2 * 128 * 256 * 4;
}
struct WsLayout {
  size_t status, sync, sync_bytes, keys, tickets, live, poff, counts, ge, r, apack, epack, rowmap, lrz, lrt, lrrho, skeys, swp, total;
};

inline WsLayout ws_layout(long long B, long long K, long long d, size_t elem) {
  WsLayout L;
  const long long rmax0 = B * (K > 1 ? K - 1 : 0);
  const size_t rmax = (size_t)(rmax0 > 0 ? rmax0 : 1);
  const size_t dd = (size_t)(d > 0 ? d : 1);
  size_t off = 0;
  L.status = off;
  off = align_up(off + 64 * 4, 256);
  L.sync = off;
  // 2 x blocks_max, then the split tickets
  L.sync_bytes = align_up((size_t)(32 + 2 * ((rmax + 255) / 256 * 2) + 8 * kPairSplitTiles) * 4, 256);
  off += L.sync_bytes;
  L.keys = off;
  off = align_up(off + (size_t)(B * (K + 1)) * 8, 256);
  L.tickets = off;
  off = align_up(off + (size_t)B * 4, 256);
  L.live = off;
  off = align_up(off + (size_t)B * 2 * 4, 256);
  L.poff = off;
  off = align_up(off + (size_t)B * 4, 256);
  L.counts = off;
  off = align_up(off + (size_t)2 * (kMaxWindowPasses + 1) * 4, 256);
  L.ge = off;
  off = align_up(off + dd * 4, 256);
  L.r = off;
  off = align_up(off + rmax * dd * elem, 256);
  L.apack = off;
  off = align_up(off + rmax * 2 * dd * elem, 256);
  L.epack = off;
  off = align_up(off + rmax * dd * elem, 256);
  L.rowmap = off;
  off = align_up(off + rmax * 4, 256);
  L.lrz = off;
  off = align_up(off + (size_t)kLowRankSplits * rmax * kLowRankLatent * 4, 256);
  L.lrt = off;
  off = align_up(off + (size_t)kLowRankSplits * rmax * kLowRankCorrection * 4, 256);
  L.lrrho = off;
  off = align_up(off + rmax * kLowRankLatent * elem, 256);
  L.skeys = off;
  off = align_up(off + (size_t)(B * (2 * K + 1)) * kMaxTopK * 8, 256);
  L.swp = off;
  off = align_up(off + std::max(swap_part_bytes(B, K, d), pair_split_bytes(B, K, d, elem)), 256);
  L.total = off;
  return L;
}

// Launches `kernel` so that it may start while the previous kernel in the
// stream finishes (programmatic dependent launch; the kernel calls pdl_wait
// before reading that kernel's outputs), optionally as clusters of
// `cluster_x` CTAs along x.
template <typename... KArgs, typename... Args>
cudaError_t launch_dependent(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                             unsigned cluster_x, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  unsigned n = 0;
  attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[n].val.programmaticStreamSerializationAllowed = 1;
  ++n;
  if (cluster_x > 1) {
    attr[n].id = cudaLaunchAttributeClusterDimension;
    attr[n].val.clusterDim.x = cluster_x;
    attr[n].val.clusterDim.y = 1;
    attr[n].val.clusterDim.z = 1;
    ++n;
  }
  cfg.attrs = attr;
  cfg.numAttrs = n;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args&&>(args)...);
}

struct DeviceInfo {
  int device;
  int sm_count;
};
cudaError_t device_info(DeviceInfo* out);

// ---- verification -----------------------------------------------------------
struct VerifyArgs {
  const void* logits;
  int B, K, V;
  long long row_stride, batch_stride;  // elements
  const int32_t* draft;
  int32_t* accept_len;
  int32_t* committed;
  int32_t* bonus;
  int32_t* target_argmax;  // optional
  int32_t* n_out;          // optional
  unsigned long long* keys;
  uint32_t* tickets;
  // Optional fused copy of the unconditioned rows j >= n_b of e_out from e.
  const void* e;
  long long e_batch_stride, e_pos_stride;
  void* e_out;
  int d;
  // Optional fused packing of the conditioned rows for the tensor-core GEMMs
  // (bf16, 16-byte aligned rows): each finalised sequence claims n_b rows of
  // the packed buffers with an atomic on *R_count (zero before the launch).
  const void* hD;
  const void* hT;
  int e_dense;
  void* apack;     // [R_max, 2d]: [m; u] rows
  void* epack;     // [R_max, d]: e rows (dense e only)
  int32_t* rowmap; // [R_max]: packed row -> b*K + j
  int32_t* R_count;
  // Windowed schedule (NULL live: one pass over every row only): two live
  // lists of B sequences and the passes' counters, from the workspace.
  int32_t* live;
  uint32_t* pass_counts;
  int32_t* pack_off;
  // Rows j < n_b of e_out in the copy above (no packing then): kCondCopyKeep
  // leaves them to the conditioning kernels, kCondCopyE writes e (no
  // conditioning), kCondCopyM writes m_j = hD[b, A_b+1+j] (overwrite).
  int cond_copy;
};
constexpr int kCondCopyKeep = 0;
constexpr int kCondCopyE = 1;
constexpr int kCondCopyM = 2;
cudaError_t launch_verify(const VerifyArgs& a, retrace_dtype dtype, cudaStream_t stream);
// The copies of a windowed verification after its last pass (accept_len and
// pack_off complete): unconditioned rows of e_out and the packed rows, from
// the copy fields of `a` (B, K, d, accept_len, e..., cond_copy, pack_off).
cudaError_t launch_verify_copies(const VerifyArgs& a, retrace_dtype dtype, cudaStream_t stream);
int set_verify_schedule(int mode);  // RETRACE_VERIFY_*; previous mode, or -1
// Row windows greedy verification takes for this call: writes the window
// starts (n + 1 entries, at most kMaxWindowPasses + 1) and returns the number
// of passes n (1: the one-pass schedule).
int verify_windows(int B, int K, int V, int elem_bytes, bool have_workspace, bool argmax_out, int* start);

// Stochastic verification (speculative sampling on top-k / top-p filtered
// distributions at temperature T).
struct SampledArgs {
  const void* tlogits;  // [B, K+1, V]
  long long t_row, t_batch;
  const void* dlogits;  // [B, K, V]
  long long d_row, d_batch;
  int B, K, V;
  const int32_t* draft;
  const float* uniforms;  // [B, K+1]
  float temperature, top_p;
  int top_k;
  int32_t* accept_len;
  int32_t* committed;
  int32_t* bonus;
  unsigned long long* keys;  // [B (2K+1), kMaxTopK]
  // a whole round (optional, e_out != NULL): n, the unconditioned rows of e~
  // copied from e (rows a multiple of 16 bytes, 16-byte aligned), and with
  // R_count the packed rows of the tensor-core projections
  int32_t* n_out;
  const void* e;
  long long e_batch_stride, e_pos_stride;  // elements
  void* e_out;
  int d;
  const void* hD;
  const void* hT;
  int e_dense;
  void* apack;
  void* epack;
  int32_t* rowmap;
  int32_t* R_count;
  // Windowed schedule (NULL live: one pass): live lists, pass counters and
  // packed-row offsets from the workspace, as for greedy verification.
  int32_t* live;
  uint32_t* pass_counts;
  int32_t* pack_off;
};
cudaError_t launch_verify_sampled(const SampledArgs& a, retrace_dtype dtype, cudaStream_t stream);

// ---- conditioning -----------------------------------------------------------
// Row plan used by every conditioning kernel: sequence b owns n_b rows, where
// n_b = max(0, K-1-A_b) from accept_len (n_from_accept) or clamp(n[b], 0, K-1).
struct RowSource {
  const int32_t* counts;  // accept_len or n
  int n_from_accept;
};

// FFMA path (fp32, and bf16 shapes the tensor-core path does not take).
struct CorrectArgs {
  const void* hD;
  const void* hT;
  const void* Wc;
  float beta;
  int B, K, d;
  RowSource rows;
  void* r_out;        // compact [R, d] (compact_out) or [B, K, d]
  int compact_out;
  int raw;            // 1: r = m (no correction; W_c is not read)
};
cudaError_t launch_correct_simt(const CorrectArgs& a, retrace_dtype dtype, cudaStream_t stream);

struct GateArgs {
  const void* e;
  int e_dense;  // 0: broadcast vector [d]; 1: dense [B, K, d]
  const void* r;
  int r_compact;  // r rows are compact [R, d] (1) or [B, K, d] (0)
  const void* Wv;
  const void* Wg;
  const float* ge;  // W_g[:, :d] e for broadcast e (device, fp32), else null
  int B, K, d;
  RowSource rows;
  void* e_out;  // [B, K, d]
};
cudaError_t launch_gate_simt(const GateArgs& a, retrace_dtype dtype, cudaStream_t stream);
cudaError_t launch_gate_bias(const void* Wg, const void* e, int d, float* ge, retrace_dtype dtype,
                             cudaStream_t stream);

// Tensor-core path (bf16, d a multiple of 256).
struct PackArgs {
  int B, K, d;
  RowSource rows;
  int mode;          // 0: [m; u] rows from hD (src0) / hT (src1); 1: r rows from src0 [B, K, d]
  const void* src0;
  const void* src1;
  const void* e;     // dense e [B, K, d] to pack (if e_dense)
  int e_dense;
  void* apack;       // mode 0: [R_max, 2d]; mode 1: [R_max, d]
  void* epack;       // [R_max, d]
  int32_t* rowmap;   // [R_max]
  int32_t* R;        // row count out
};
cudaError_t launch_pack(const PackArgs& a, cudaStream_t stream);

// Counters of one conditioning pass (uint32, zeroed before each pass):
//   [kSyncRowCount]   packed rows claimed / R
//   [kSyncTileQueue]  next tile of the dynamic schedule
//   [kSyncGemvNext]   next row of W_g[:, :d] e;  [kSyncGemvDone] rows written
//   [kSyncSeqDone]    sequences finalised (fused round)
//   [kSyncChunkNext]  next group of logits chunks to stream (fused round)
//   [kSyncBlocks ...]            per 128-row block: correction epilogue warps done
//   [kSyncBlocks + blocks ...]   per 128-row block: packed rows published (fused round)
//   [kSyncBlocks + 2 blocks ...] per split gate tile, CTA of the pair and epilogue warp:
//                                K halves finished (CTA-pair kernel; 8 kPairSplitTiles)
constexpr int kSyncRowCount = 0;
constexpr int kSyncTileQueue = 1;
constexpr int kSyncGemvNext = 2;
constexpr int kSyncGemvDone = 3;
constexpr int kSyncSeqDone = 4;
constexpr int kSyncChunkNext = 5;
constexpr int kSyncBlocks = 32;

// 128-row blocks of the largest packed-row count, rounded up to whole pairs
// (the CTA-pair kernel counts per 128-row block over 256-row pair tiles).
inline long long blocks_max(long long B, long long K) {
  const long long rmax = B * (K > 1 ? K - 1 : 0);
  return (rmax + 255) / 256 * 2;
}

struct TcCondArgs {
  int B, K, d;
  int do_correct, do_gate;
  // correction: r = m + beta * W_c [m; u] over the packed [m; u] rows
  const void* apack;
  const void* Wc;
  float beta;
  void* r_out;
  int compact_out;  // 1: r_out is compact [R_max, d]; 0: r_out is [B, K, d] (rows via rowmap)
  // gate: e~ = e + (W_v r) .* sigmoid(W_g [e; r]) over the compact r rows
  const void* rpack;
  long long r_row_stride;  // elements between rpack rows (0: d)
  const void* e;
  const void* epack;
  int e_dense;
  const void* Wv;
  const void* Wg;
  float* ge;  // [d] scratch for W_g[:, :d] e (broadcast e)
  void* e_out;
  const int32_t* R;
  const int32_t* rowmap;
  uint32_t* sync;
  uint32_t* status;
  // small-R path (B (K-1) <= kSwapMaxRows): fp32 split partials, swap_part_bytes (NULL: not taken)
  float* part;
  // CTA-pair path: fp32 accumulators of the split gate tiles, pair_split_bytes (NULL: no split tiles)
  float* split_part;
};
cudaError_t launch_cond_tc(const TcCondArgs& a, cudaStream_t stream);
// The bounded waits of the pipelined kernels on a caller-controlled condition.
cudaError_t launch_wait_selftest(int kind, const uint32_t* flag, uint32_t target, uint32_t* status,
                                 cudaStream_t stream);

// Low-rank conditioning (rank-64 latents, rank-32 correction; broadcast e).
struct LowRankArgs {
  int B, K, d;
  retrace_dtype dtype;
  float beta;
  const void* hD;
  const void* hT;
  const void* e;   // [d]
  const void* P;   // [64, d]
  const void* Bc;  // [32, 64 + d]
  const void* Ac;  // [64, 32]
  const void* Wv;  // [d, 64]
  const void* Wg;  // [d, d + 64]
  const int32_t* accept_len;
  void* e_out;
  float* ge;  // [d]: W_g[:, :d] e
  // tensor-core path: rows packed by the verification kernel
  const void* apack;
  const int32_t* rowmap;
  const int32_t* R;
  float* zpart;
  float* tpart;
  void* rho;
  uint32_t* gemv_next;  // zero before the call
  uint32_t* status;
};
bool lowrank_tc_supported(retrace_dtype dtype, int d);
cudaError_t launch_lowrank(const LowRankArgs& a, bool tc, cudaStream_t stream);

// The whole round in one persistent launch: verification warps and
// tensor-core warps share every SM (bf16, d a multiple of 256, 16-byte
// aligned logits rows, K >= 2).
struct TcRoundArgs {
  const void* logits;
  int B, K, V, d;
  long long row_stride, batch_stride;
  const int32_t* draft;
  int32_t* accept_len;
  int32_t* committed;
  int32_t* bonus;
  int32_t* target_argmax;
  int32_t* n_out;
  unsigned long long* keys;
  uint32_t* tickets;
  const void* hD;
  const void* hT;
  const void* e;
  int e_dense;
  long long e_batch_stride, e_pos_stride;
  const void* Wc;
  const void* Wv;
  const void* Wg;
  float beta;
  void* e_out;
  void* apack;
  void* epack;
  void* rpack;
  float* ge;
  int32_t* rowmap;
  uint32_t* sync;
  uint32_t* status;
};
bool round_fused_supported(const TcRoundArgs& a);
cudaError_t launch_round_tc(const TcRoundArgs& a, cudaStream_t stream);

// Writes n_out and the rows j >= n_b (zeros for r, a copy of e for e_out).
cudaError_t launch_fill_rows(int B, int K, int d, RowSource rows, int32_t* n_out, void* zero_dst,
                             const void* e, int e_dense, void* e_dst, retrace_dtype dtype,
                             cudaStream_t stream);

// Whether the tensor-core path handles this conditioning shape.
bool tc_supported(retrace_dtype dtype, int d);

// Sets the thread-local message returned by retrace_last_error().
void set_last_error(const char* msg);

// cuTensorMapEncodeTiled through the runtime's driver entry point.
CUresult encode_tensor_map_2d(CUtensorMap* map, const void* base, uint64_t inner, uint64_t rows,
                              uint64_t row_stride_bytes, uint32_t box_inner, uint32_t box_rows);

}  // namespace retrace
