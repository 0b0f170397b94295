// Host-side declarations shared by the libretrace translation units.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "../../include/retrace.h"

namespace retrace {

constexpr int kMaxK = 1024;  // largest draft block the kernels accept

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Workspace layout (all offsets 256-byte aligned):
//   status   uint32 [64]        device status word (+ spare)
//   keys     uint64 [B*(K+1)]   per-row argmax keys, zero between calls
//   tickets  uint32 [B]         per-sequence CTA arrival counters, zero between calls
//   ge       fp32   [d]         W_g[:, :d] e for a broadcast e
//   r        elem   [R_max, d]  compacted corrected signal, R_max = B*(K-1)
struct WsLayout {
  size_t status, keys, tickets, ge, r, total;
};

inline WsLayout ws_layout(long long B, long long K, long long d, size_t elem) {
  WsLayout L;
  size_t off = 0;
  L.status = off;
  off = align_up(off + 64 * 4, 256);
  L.keys = off;
  off = align_up(off + (size_t)(B * (K + 1)) * 8, 256);
  L.tickets = off;
  off = align_up(off + (size_t)B * 4, 256);
  L.ge = off;
  off = align_up(off + (size_t)(d > 0 ? d : 1) * 4, 256);
  L.r = off;
  long long rmax = B * (K > 1 ? K - 1 : 0);
  off = align_up(off + (size_t)(rmax > 0 ? rmax : 1) * (size_t)(d > 0 ? d : 1) * elem, 256);
  L.total = off;
  return L;
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
};
cudaError_t launch_verify(const VerifyArgs& a, retrace_dtype dtype, cudaStream_t stream);

// ---- conditioning -----------------------------------------------------------
// Row plan used by every conditioning kernel: sequence b owns n_b rows, where
// n_b = max(0, K-1-A_b) from accept_len (n_from_accept) or clamp(n[b], 0, K-1).
struct RowSource {
  const int32_t* counts;  // accept_len or n
  int n_from_accept;
};

struct CorrectArgs {
  const void* hD;
  const void* hT;
  const void* Wc;
  float beta;
  int B, K, d;
  RowSource rows;
  void* r_out;        // compact [R, d] (compact_out) or [B, K, d]
  int compact_out;
};
cudaError_t launch_correct(const CorrectArgs& a, retrace_dtype dtype, cudaStream_t stream);

struct GateArgs {
  const void* e;
  int e_dense;  // 0: broadcast vector [d]; 1: dense [B, K, d]
  const void* r;
  int r_compact;  // r rows are compact [R, d] (1) or [B, K, d] (0)
  long long r_rows;  // rows of the r buffer (for the tensor map)
  const void* Wv;
  const void* Wg;
  const float* ge;  // W_g[:, :d] e for broadcast e (device, fp32), else null
  int B, K, d;
  RowSource rows;
  void* e_out;  // [B, K, d]
};
cudaError_t launch_gate(const GateArgs& a, retrace_dtype dtype, cudaStream_t stream);
cudaError_t launch_gate_bias(const void* Wg, const void* e, int d, float* ge, retrace_dtype dtype,
                             cudaStream_t stream);

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
