// C ABI of libretrace (declared in include/retrace.h): argument checks,
// workspace layout, tensor-map encoding and the launch sequence of a round.
#include <stdarg.h>
#include <stdio.h>

#include <mutex>
#include <unordered_map>

#include "internal.h"

namespace retrace {

cudaError_t device_info(DeviceInfo* out) {
  static std::atomic<int> sm_cache[64];  // 0: not yet read (threads may race to fill it)
  int dev = 0;
  cudaError_t err = cudaGetDevice(&dev);
  if (err != cudaSuccess) return err;
  int sm = sm_cache[dev & 63].load(std::memory_order_relaxed);
  if (sm == 0) {
    err = cudaDeviceGetAttribute(&sm, cudaDevAttrMultiProcessorCount, dev);
    if (err != cudaSuccess) return err;
    sm_cache[dev & 63].store(sm, std::memory_order_relaxed);
  }
  out->device = dev;
  out->sm_count = sm;
  return cudaSuccess;
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn encode_fn() {
  static std::atomic<EncodeTiledFn> fn{nullptr};
  EncodeTiledFn f = fn.load(std::memory_order_acquire);
  if (!f) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess) {
      f = reinterpret_cast<EncodeTiledFn>(p);
      fn.store(f, std::memory_order_release);
    }
  }
  return f;
}

// bf16 2D tensor [rows, inner], 128-byte swizzle, box {box_inner, box_rows}.
CUresult encode_tensor_map_2d(CUtensorMap* map, const void* base, uint64_t inner, uint64_t rows,
                              uint64_t row_stride_bytes, uint32_t box_inner, uint32_t box_rows) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return CUDA_ERROR_NOT_FOUND;
  const cuuint64_t dims[2] = {inner, rows};
  const cuuint64_t strides[1] = {row_stride_bytes};
  const cuuint32_t box[2] = {box_inner, box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
}

}  // namespace retrace

using namespace retrace;

namespace {

thread_local char g_err[512] = "";

retrace_status fail(retrace_status s, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
  return s;
}

retrace_status cuda_fail(cudaError_t e, const char* what) {
  return fail(RETRACE_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

#define RT_CUDA(expr, what)                      \
  do {                                           \
    cudaError_t e_ = (expr);                     \
    if (e_ != cudaSuccess) return cuda_fail(e_, what); \
  } while (0)

size_t elem_size(retrace_dtype t) { return t == RETRACE_BF16 ? 2 : 4; }
bool dtype_ok(retrace_dtype t) { return t == RETRACE_BF16 || t == RETRACE_F32; }
bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

retrace_status check_ws(const void* ws, size_t ws_bytes, size_t need) {
  if (!ws) return fail(RETRACE_ERR_WORKSPACE, "workspace pointer is NULL");
  if (((uintptr_t)ws & 255u) != 0) return fail(RETRACE_ERR_WORKSPACE, "workspace must be 256-byte aligned");
  if (ws_bytes < need)
    return fail(RETRACE_ERR_WORKSPACE, "workspace too small: %zu bytes given, %zu needed", ws_bytes, need);
  return RETRACE_OK;
}

// The regions that must be zero between calls (sync counters, argmax keys,
// tickets, pass counters) lie before L.ge, at offsets that depend on B and K
// (the live lists and packed-row offsets between them hold data).  A call of
// another (B, K) than the previous call on the same workspace would find some
// of them over the previous layout's data, so it first re-zeroes
// [256, max(old, new) L.ge) -- the status word at 0 is kept.  The previous
// shape of each workspace is kept here, on the host, in enqueue order (calls
// on one workspace are ordered on one stream); retrace_workspace_init
// forgets it.
struct WsMemo {
  long long B, K;
  size_t zero_end;
};
static std::mutex g_ws_mu;
static std::unordered_map<uintptr_t, WsMemo> g_ws_memo;

retrace_status prepare_ws(void* ws, size_t ws_bytes, const WsLayout& L, long long B, long long K,
                          cudaStream_t stream) {
  size_t clear_end = 0;
  {
    std::lock_guard<std::mutex> lock(g_ws_mu);
    auto it = g_ws_memo.find((uintptr_t)ws);
    if (it == g_ws_memo.end()) {
      g_ws_memo[(uintptr_t)ws] = WsMemo{B, K, L.ge};
    } else if (it->second.B != B || it->second.K != K) {
      clear_end = it->second.zero_end > L.ge ? it->second.zero_end : L.ge;
      it->second = WsMemo{B, K, L.ge};
    }
  }
  if (clear_end > ws_bytes) clear_end = ws_bytes;
  if (clear_end > 256)
    RT_CUDA(cudaMemsetAsync(static_cast<char*>(ws) + 256, 0, clear_end - 256, stream),
            "cudaMemsetAsync(workspace, shape change)");
  return RETRACE_OK;
}

void forget_ws(const void* ws) {
  std::lock_guard<std::mutex> lock(g_ws_mu);
  g_ws_memo.erase((uintptr_t)ws);
}

retrace_status check_verify_args(const void* logits, retrace_dtype dtype, int B, int K, int V,
                                 int64_t rs, int64_t bs, const int32_t* draft,
                                 const int32_t* accept_len, const int32_t* committed,
                                 const int32_t* bonus) {
  if (!dtype_ok(dtype)) return fail(RETRACE_ERR_INVALID_ARG, "unknown dtype %d", (int)dtype);
  if (B < 0 || K < 0 || V < 1) return fail(RETRACE_ERR_INVALID_ARG, "bad shape B=%d K=%d V=%d", B, K, V);
  if (K > kMaxK) return fail(RETRACE_ERR_UNSUPPORTED, "K=%d exceeds the supported maximum %d", K, kMaxK);
  if (B == 0) return RETRACE_OK;
  if (!logits || (!draft && K > 0) || !accept_len || !committed || !bonus)
    return fail(RETRACE_ERR_INVALID_ARG, "NULL tensor pointer");
  if (rs < V) return fail(RETRACE_ERR_INVALID_ARG, "logits_row_stride %lld < V %d", (long long)rs, V);
  if (bs < (int64_t)(K + 1) * rs)
    return fail(RETRACE_ERR_INVALID_ARG, "logits_batch_stride %lld < (K+1)*row_stride", (long long)bs);
  return RETRACE_OK;
}

retrace_status check_cond_shape(retrace_dtype dtype, int B, int K, int d) {
  if (!dtype_ok(dtype)) return fail(RETRACE_ERR_INVALID_ARG, "unknown dtype %d", (int)dtype);
  if (B < 0 || K < 1 || d < 1) return fail(RETRACE_ERR_INVALID_ARG, "bad shape B=%d K=%d d=%d", B, K, d);
  if (K > kMaxK) return fail(RETRACE_ERR_UNSUPPORTED, "K=%d exceeds the supported maximum %d", K, kMaxK);
  if ((long long)B * K * (long long)d >= (1LL << 31) * 8LL)
    return fail(RETRACE_ERR_UNSUPPORTED, "B*K*d too large");
  if ((long long)B * K >= (1LL << 31)) return fail(RETRACE_ERR_UNSUPPORTED, "B*K too large");
  return RETRACE_OK;
}

retrace_status e_mode(int64_t ebs, int64_t eps, int K, int d, int* dense) {
  if (ebs == 0 && eps == 0) {
    *dense = 0;
    return RETRACE_OK;
  }
  if (eps == d && ebs == (int64_t)K * d) {
    *dense = 1;
    return RETRACE_OK;
  }
  return fail(RETRACE_ERR_UNSUPPORTED,
              "e strides (%lld, %lld): only (0, 0) (broadcast) or (K*d, d) (dense) are supported",
              (long long)ebs, (long long)eps);
}

uint32_t* status_word(void* ws) { return reinterpret_cast<uint32_t*>(ws); }

// Workspace pointers of the windowed schedule of sampled verification.
void sampled_workspace(SampledArgs* a, char* w, const WsLayout& L) {
  a->live = reinterpret_cast<int32_t*>(w + L.live);
  a->pass_counts = reinterpret_cast<uint32_t*>(w + L.counts);
  a->pack_off = reinterpret_cast<int32_t*>(w + L.poff);
}

// Workspace pointers of the greedy verification kernels.
void verify_workspace(VerifyArgs* a, char* w, const WsLayout& L) {
  a->keys = reinterpret_cast<unsigned long long*>(w + L.keys);
  a->tickets = reinterpret_cast<uint32_t*>(w + L.tickets);
  a->live = reinterpret_cast<int32_t*>(w + L.live);
  a->pass_counts = reinterpret_cast<uint32_t*>(w + L.counts);
  a->pack_off = reinterpret_cast<int32_t*>(w + L.poff);
}


retrace_status check_sampling(int B, int K, int V, const void* draft_logits, int64_t draft_row_stride,
                              int64_t draft_batch_stride, const float* uniforms, float temperature, int top_k,
                              float top_p) {
  if (K < 1) return fail(RETRACE_ERR_INVALID_ARG, "K must be >= 1");
  if (B > 0 && (!draft_logits || !uniforms)) return fail(RETRACE_ERR_INVALID_ARG, "NULL tensor pointer");
  if (draft_row_stride < V || draft_batch_stride < (int64_t)K * draft_row_stride)
    return fail(RETRACE_ERR_INVALID_ARG, "draft logits strides (%lld, %lld) below [B, K, V] packing",
                (long long)draft_row_stride, (long long)draft_batch_stride);
  if (!(temperature > 0.f) || temperature > 3.0e38f)
    return fail(RETRACE_ERR_INVALID_ARG, "temperature must be positive and finite");
  if (top_k < 1 || top_k > kMaxTopK || top_k > V)
    return fail(RETRACE_ERR_INVALID_ARG, "top_k must be in [1, min(64, V)], got %d", top_k);
  if (!(top_p > 0.f && top_p <= 1.f)) return fail(RETRACE_ERR_INVALID_ARG, "top_p must be in (0, 1]");
  return RETRACE_OK;
}

// Tensors of the conditioning step shared by the rounds.
struct ConditioningArgs {
  const void* hD;
  const void* hT;
  const void* e;
  int64_t e_batch_stride, e_pos_stride;
  int e_dense;
  const void* Wc;
  const void* Wv;
  const void* Wg;
  float beta;
  void* e_out;
};

// Correction (Eq. 6-7) and gated fusion (Eq. 8) of the rows j < n_b, after a
// verification kernel has written accept_len and the unconditioned rows of
// e_out and, on the tensor-core path, packed the [m; u] rows.  Records
// phase_events[2] after the correction (after both projections on the
// tensor-core path, which runs them in one launch).
retrace_status enqueue_conditioning(const ConditioningArgs& c, retrace_dtype dtype, int B, int K, int d,
                                    bool tc, bool raw, const int32_t* accept_len, void* ws, const WsLayout& L,
                                    const cudaEvent_t* phase_events, cudaStream_t stream) {
  char* w = reinterpret_cast<char*>(ws);
  float* ge = reinterpret_cast<float*>(w + L.ge);
  void* r_ws = w + L.r;
  const RowSource rows{accept_len, 1};
  if (tc) {
    uint32_t* sync = reinterpret_cast<uint32_t*>(w + L.sync);
    TcCondArgs a{};
    a.B = B;
    a.K = K;
    a.d = d;
    a.do_correct = raw ? 0 : 1;
    a.do_gate = 1;
    a.apack = w + L.apack;
    a.Wc = c.Wc;
    a.beta = c.beta;
    a.r_out = r_ws;
    a.compact_out = 1;
    // raw: r = m is the first half of each packed [m; u] row
    a.rpack = raw ? w + L.apack : r_ws;
    a.r_row_stride = raw ? 2LL * d : 0;
    a.e = c.e;
    a.epack = w + L.epack;
    a.e_dense = c.e_dense;
    a.Wv = c.Wv;
    a.Wg = c.Wg;
    a.ge = ge;
    a.e_out = c.e_out;
    a.R = reinterpret_cast<int32_t*>(sync + kSyncRowCount);
    a.rowmap = reinterpret_cast<int32_t*>(w + L.rowmap);
    a.sync = sync;
    a.status = status_word(ws);
    a.part = swap_part_bytes(B, K, d) ? reinterpret_cast<float*>(reinterpret_cast<char*>(ws) + L.swp) : nullptr;
    a.split_part = pair_split_bytes(B, K, d, 2) ? reinterpret_cast<float*>(w + L.swp) : nullptr;
    RT_CUDA(launch_cond_tc(a, stream), "conditioning kernel launch");
    if (phase_events) RT_CUDA(cudaEventRecord(phase_events[2], stream), "cudaEventRecord");
  } else {
    CorrectArgs ca{c.hD, c.hT, c.Wc, c.beta, B, K, d, rows, r_ws, 1, raw ? 1 : 0};
    RT_CUDA(launch_correct_simt(ca, dtype, stream), "correction kernel launch");
    if (phase_events) RT_CUDA(cudaEventRecord(phase_events[2], stream), "cudaEventRecord");
    if (!c.e_dense) RT_CUDA(launch_gate_bias(c.Wg, c.e, d, ge, dtype, stream), "gate bias kernel launch");
    GateArgs ga{c.e, c.e_dense, r_ws, 1, c.Wv, c.Wg, c.e_dense ? nullptr : ge, B, K, d, rows, c.e_out};
    RT_CUDA(launch_gate_simt(ga, dtype, stream), "gate kernel launch");
  }
  return RETRACE_OK;
}
}  // namespace

void retrace::set_last_error(const char* msg) { snprintf(g_err, sizeof(g_err), "%s", msg); }

extern "C" {

const char* retrace_last_error(void) { return g_err; }

const char* retrace_version(void) { return "retrace 0.1.0 sm_103a"; }

int retrace_set_verify_schedule(int mode) { return set_verify_schedule(mode); }

int retrace_verify_plan(int B, int K, int V, retrace_dtype dtype, int target_argmax, int* window_starts) {
  if (B < 0 || K < 0 || V < 1 || K > kMaxK || (dtype != RETRACE_BF16 && dtype != RETRACE_F32)) return -1;
  int start[kMaxWindowPasses + 1];
  const int n = verify_windows(B, K, V, (int)elem_size(dtype), true, target_argmax != 0, start);
  if (window_starts)
    for (int k = 0; k <= n; ++k) window_starts[k] = start[k];
  return n;
}

size_t retrace_workspace_bytes(int B, int K, int V, int d, retrace_dtype dtype) {
  if (B < 0 || K < 0 || V < 1 || d < 0 || !dtype_ok(dtype)) return 0;
  return ws_layout(B, K, d, elem_size(dtype)).total;
}

retrace_status retrace_workspace_init(void* ws, size_t ws_bytes, cudaStream_t stream) {
  g_err[0] = '\0';
  if (!ws || ws_bytes == 0) return fail(RETRACE_ERR_INVALID_ARG, "NULL or empty workspace");
  RT_CUDA(cudaMemsetAsync(ws, 0, ws_bytes, stream), "cudaMemsetAsync(workspace)");
  forget_ws(ws);
  return RETRACE_OK;
}

retrace_status retrace_workspace_check(const void* ws, size_t ws_bytes, uint32_t* device_flags,
                                       cudaStream_t stream) {
  g_err[0] = '\0';
  if (!ws || ws_bytes < 4 || !device_flags) return fail(RETRACE_ERR_INVALID_ARG, "bad arguments");
  RT_CUDA(cudaStreamSynchronize(stream), "cudaStreamSynchronize");
  RT_CUDA(cudaMemcpy(device_flags, ws, 4, cudaMemcpyDeviceToHost), "cudaMemcpy(status)");
  if (*device_flags) return fail(RETRACE_ERR_DEVICE, "device status flags 0x%x", *device_flags);
  return RETRACE_OK;
}

retrace_status retrace_verify(const void* logits, retrace_dtype dtype, int B, int K, int V,
                              int64_t logits_row_stride, int64_t logits_batch_stride,
                              const int32_t* draft, int32_t* accept_len, int32_t* committed,
                              int32_t* bonus, int32_t* target_argmax, void* ws, size_t ws_bytes,
                              cudaStream_t stream) {
  g_err[0] = '\0';
  retrace_status st = check_verify_args(logits, dtype, B, K, V, logits_row_stride,
                                        logits_batch_stride, draft, accept_len, committed, bonus);
  if (st != RETRACE_OK || B == 0) return st;
  const WsLayout L = ws_layout(B, K, 0, elem_size(dtype));
  if ((st = check_ws(ws, ws_bytes, L.ge)) != RETRACE_OK) return st;
  if ((st = prepare_ws(ws, ws_bytes, L, B, K, stream)) != RETRACE_OK) return st;
  VerifyArgs a{};
  a.logits = logits;
  a.B = B;
  a.K = K;
  a.V = V;
  a.row_stride = logits_row_stride;
  a.batch_stride = logits_batch_stride;
  a.draft = draft;
  a.accept_len = accept_len;
  a.committed = committed;
  a.bonus = bonus;
  a.target_argmax = target_argmax;
  verify_workspace(&a, reinterpret_cast<char*>(ws), L);
  RT_CUDA(launch_verify(a, dtype, stream), "verify kernel launch");
  return RETRACE_OK;
}

retrace_status retrace_align_refine(const void* hD, const void* hT, retrace_dtype dtype, int B, int K,
                                    int d, const int32_t* accept_len, const void* Wc, float beta,
                                    void* r_out, int32_t* n_out, void* ws, size_t ws_bytes,
                                    cudaStream_t stream) {
  g_err[0] = '\0';
  retrace_status st = check_cond_shape(dtype, B, K, d);
  if (st != RETRACE_OK || B == 0) return st;
  if (!hD || !hT || !accept_len || !Wc || !r_out || !n_out)
    return fail(RETRACE_ERR_INVALID_ARG, "NULL tensor pointer");
  const WsLayout L = ws_layout(B, K, d, elem_size(dtype));
  if ((st = check_ws(ws, ws_bytes, L.total)) != RETRACE_OK) return st;
  if ((st = prepare_ws(ws, ws_bytes, L, B, K, stream)) != RETRACE_OK) return st;
  const RowSource rows{accept_len, 1};
  RT_CUDA(launch_fill_rows(B, K, d, rows, n_out, r_out, nullptr, 0, nullptr, dtype, stream),
          "fill kernel launch");
  const bool tc = tc_supported(dtype, d) && aligned16(hD) && aligned16(hT) && aligned16(Wc) && aligned16(r_out);
  if (tc) {
    char* w = reinterpret_cast<char*>(ws);
    uint32_t* sync = reinterpret_cast<uint32_t*>(w + L.sync);
    int32_t* R = reinterpret_cast<int32_t*>(sync + kSyncRowCount);
    int32_t* rowmap = reinterpret_cast<int32_t*>(w + L.rowmap);
    RT_CUDA(cudaMemsetAsync(sync, 0, L.sync_bytes, stream), "cudaMemsetAsync(sync)");
    PackArgs pk{B, K, d, rows, 0, hD, hT, nullptr, 0, w + L.apack, nullptr, rowmap, R};
    RT_CUDA(launch_pack(pk, stream), "pack kernel launch");
    TcCondArgs a{};
    a.B = B;
    a.K = K;
    a.d = d;
    a.do_correct = 1;
    a.apack = w + L.apack;
    a.Wc = Wc;
    a.beta = beta;
    a.r_out = r_out;
    a.compact_out = 0;
    a.R = R;
    a.rowmap = rowmap;
    a.sync = sync;
    a.status = status_word(ws);
    a.part = swap_part_bytes(B, K, d) ? reinterpret_cast<float*>(reinterpret_cast<char*>(ws) + L.swp) : nullptr;
    RT_CUDA(launch_cond_tc(a, stream), "correction kernel launch");
  } else {
    CorrectArgs a{hD, hT, Wc, beta, B, K, d, rows, r_out, 0};
    RT_CUDA(launch_correct_simt(a, dtype, stream), "correction kernel launch");
  }
  return RETRACE_OK;
}

retrace_status retrace_gate_fuse(const void* e, int64_t e_batch_stride, int64_t e_pos_stride,
                                 const void* r, const int32_t* n, const void* Wv, const void* Wg,
                                 retrace_dtype dtype, int B, int K, int d, void* e_out, void* ws,
                                 size_t ws_bytes, cudaStream_t stream) {
  g_err[0] = '\0';
  retrace_status st = check_cond_shape(dtype, B, K, d);
  if (st != RETRACE_OK || B == 0) return st;
  if (!e || !r || !n || !Wv || !Wg || !e_out) return fail(RETRACE_ERR_INVALID_ARG, "NULL tensor pointer");
  int dense = 0;
  if ((st = e_mode(e_batch_stride, e_pos_stride, K, d, &dense)) != RETRACE_OK) return st;
  const WsLayout L = ws_layout(B, K, d, elem_size(dtype));
  if ((st = check_ws(ws, ws_bytes, L.total)) != RETRACE_OK) return st;
  if ((st = prepare_ws(ws, ws_bytes, L, B, K, stream)) != RETRACE_OK) return st;
  char* w = reinterpret_cast<char*>(ws);
  float* ge = reinterpret_cast<float*>(w + L.ge);
  const RowSource rows{n, 0};
  RT_CUDA(launch_fill_rows(B, K, d, rows, nullptr, nullptr, e, dense, e_out, dtype, stream),
          "fill kernel launch");
  const bool tc = tc_supported(dtype, d) && aligned16(e) && aligned16(r) && aligned16(Wv) &&
                  aligned16(Wg) && aligned16(e_out);
  if (tc) {
    uint32_t* sync = reinterpret_cast<uint32_t*>(w + L.sync);
    int32_t* R = reinterpret_cast<int32_t*>(sync + kSyncRowCount);
    int32_t* rowmap = reinterpret_cast<int32_t*>(w + L.rowmap);
    RT_CUDA(cudaMemsetAsync(sync, 0, L.sync_bytes, stream), "cudaMemsetAsync(sync)");
    PackArgs pk{B, K, d, rows, 1, r, nullptr, e, dense, w + L.r, w + L.epack, rowmap, R};
    RT_CUDA(launch_pack(pk, stream), "pack kernel launch");
    TcCondArgs a{};
    a.B = B;
    a.K = K;
    a.d = d;
    a.do_gate = 1;
    a.rpack = w + L.r;
    a.e = e;
    a.epack = w + L.epack;
    a.e_dense = dense;
    a.Wv = Wv;
    a.Wg = Wg;
    a.ge = ge;
    a.e_out = e_out;
    a.R = R;
    a.rowmap = rowmap;
    a.sync = sync;
    a.status = status_word(ws);
    a.part = swap_part_bytes(B, K, d) ? reinterpret_cast<float*>(reinterpret_cast<char*>(ws) + L.swp) : nullptr;
    a.split_part = pair_split_bytes(B, K, d, 2) ? reinterpret_cast<float*>(w + L.swp) : nullptr;
    RT_CUDA(launch_cond_tc(a, stream), "gate kernel launch");
  } else {
    if (!dense) RT_CUDA(launch_gate_bias(Wg, e, d, ge, dtype, stream), "gate bias kernel launch");
    GateArgs a{e, dense, r, 0, Wv, Wg, dense ? nullptr : ge, B, K, d, rows, e_out};
    RT_CUDA(launch_gate_simt(a, dtype, stream), "gate kernel launch");
  }
  return RETRACE_OK;
}

retrace_status retrace_round(const void* logits, int64_t logits_row_stride,
                             int64_t logits_batch_stride, const int32_t* draft, const void* hD,
                             const void* hT, const void* e, int64_t e_batch_stride,
                             int64_t e_pos_stride, const void* Wc, const void* Wv, const void* Wg,
                             float beta, retrace_dtype dtype, int B, int K, int V, int d,
                             int32_t* accept_len, int32_t* committed, int32_t* bonus,
                             int32_t* target_argmax, int32_t* n_out, void* e_out, void* ws,
                             size_t ws_bytes, uint32_t flags, const cudaEvent_t* phase_events,
                             cudaStream_t stream) {
  g_err[0] = '\0';
  const uint32_t kAblations = RETRACE_COND_RAW | RETRACE_COND_OVERWRITE | RETRACE_COND_NONE;
  if (flags & ~(RETRACE_ROUND_OVERLAP | kAblations)) return fail(RETRACE_ERR_INVALID_ARG, "unknown flag bits");
  const uint32_t ablation = flags & kAblations;
  if (ablation & (ablation - 1)) return fail(RETRACE_ERR_INVALID_ARG, "at most one RETRACE_COND_* flag");
  if ((flags & RETRACE_ROUND_OVERLAP) && ablation)
    return fail(RETRACE_ERR_UNSUPPORTED, "RETRACE_ROUND_OVERLAP runs the corrected method only");
  retrace_status st = check_verify_args(logits, dtype, B, K, V, logits_row_stride,
                                        logits_batch_stride, draft, accept_len, committed, bonus);
  if (st != RETRACE_OK) return st;
  if ((st = check_cond_shape(dtype, B, K, d)) != RETRACE_OK) return st;
  if (B == 0) return RETRACE_OK;
  // the tensors each variant reads
  const bool need_gate = ablation == 0 || ablation == RETRACE_COND_RAW;
  const bool need_wc = ablation == 0;
  if (!hD || !hT || !e || !e_out || (need_wc && !Wc) || (need_gate && (!Wv || !Wg)))
    return fail(RETRACE_ERR_INVALID_ARG, "NULL tensor pointer");
  int dense = 0;
  if ((st = e_mode(e_batch_stride, e_pos_stride, K, d, &dense)) != RETRACE_OK) return st;
  const WsLayout L = ws_layout(B, K, d, elem_size(dtype));
  if ((st = check_ws(ws, ws_bytes, L.total)) != RETRACE_OK) return st;
  if ((st = prepare_ws(ws, ws_bytes, L, B, K, stream)) != RETRACE_OK) return st;
  char* w = reinterpret_cast<char*>(ws);
  float* ge = reinterpret_cast<float*>(w + L.ge);
  void* r_ws = w + L.r;

  const bool tc = need_gate && tc_supported(dtype, d) && aligned16(hD) && aligned16(hT) &&
                  aligned16(Wc) && aligned16(Wv) && aligned16(Wg) && aligned16(e) && aligned16(e_out);
  if ((flags & RETRACE_ROUND_OVERLAP) && !tc)
    return fail(RETRACE_ERR_UNSUPPORTED, "RETRACE_ROUND_OVERLAP: bf16 with d a multiple of 256 and 16-byte aligned tensors only");
  uint32_t* sync = reinterpret_cast<uint32_t*>(w + L.sync);
  int32_t* R = reinterpret_cast<int32_t*>(sync + kSyncRowCount);
  int32_t* rowmap = reinterpret_cast<int32_t*>(w + L.rowmap);

  if (phase_events) RT_CUDA(cudaEventRecord(phase_events[0], stream), "cudaEventRecord");
  // The verification kernel packs the conditioned rows as sequences finish;
  // they claim packed rows from a counter that starts at zero.
  if (tc) RT_CUDA(cudaMemsetAsync(sync, 0, L.sync_bytes, stream), "cudaMemsetAsync(sync)");
  if (tc) {
    TcRoundArgs ra{};
    ra.logits = logits;
    ra.B = B;
    ra.K = K;
    ra.V = V;
    ra.d = d;
    ra.row_stride = logits_row_stride;
    ra.batch_stride = logits_batch_stride;
    ra.draft = draft;
    ra.accept_len = accept_len;
    ra.committed = committed;
    ra.bonus = bonus;
    ra.target_argmax = target_argmax;
    ra.n_out = n_out;
    ra.keys = reinterpret_cast<unsigned long long*>(w + L.keys);
    ra.tickets = reinterpret_cast<uint32_t*>(w + L.tickets);
    ra.hD = hD;
    ra.hT = hT;
    ra.e = e;
    ra.e_dense = dense;
    ra.e_batch_stride = e_batch_stride;
    ra.e_pos_stride = e_pos_stride;
    ra.Wc = Wc;
    ra.Wv = Wv;
    ra.Wg = Wg;
    ra.beta = beta;
    ra.e_out = e_out;
    ra.apack = w + L.apack;
    ra.epack = w + L.epack;
    ra.rpack = r_ws;
    ra.ge = ge;
    ra.rowmap = rowmap;
    ra.sync = sync;
    ra.status = status_word(ws);
    if (flags & RETRACE_ROUND_OVERLAP) {
      if (!round_fused_supported(ra))
        return fail(RETRACE_ERR_UNSUPPORTED, "RETRACE_ROUND_OVERLAP: shape or layout outside the overlapped kernel");
      // verification and both projections overlap inside one launch
      RT_CUDA(launch_round_tc(ra, stream), "round kernel launch");
      if (phase_events) {
        for (int k = 1; k < 4; ++k) RT_CUDA(cudaEventRecord(phase_events[k], stream), "cudaEventRecord");
      }
      return RETRACE_OK;
    }
  }
  VerifyArgs va{};
  va.logits = logits;
  va.B = B;
  va.K = K;
  va.V = V;
  va.row_stride = logits_row_stride;
  va.batch_stride = logits_batch_stride;
  va.draft = draft;
  va.accept_len = accept_len;
  va.committed = committed;
  va.bonus = bonus;
  va.target_argmax = target_argmax;
  va.n_out = n_out;
  verify_workspace(&va, w, L);
  va.e = e;
  va.e_batch_stride = e_batch_stride;
  va.e_pos_stride = e_pos_stride;
  va.e_out = e_out;
  va.d = d;
  va.hD = hD;
  va.cond_copy = ablation == RETRACE_COND_NONE ? kCondCopyE
                 : ablation == RETRACE_COND_OVERWRITE ? kCondCopyM
                                                      : kCondCopyKeep;
  if (tc) {
    va.hT = hT;
    va.e_dense = dense;
    va.apack = w + L.apack;
    va.epack = w + L.epack;
    va.rowmap = rowmap;
    va.R_count = R;
  }
  RT_CUDA(launch_verify(va, dtype, stream), "verify kernel launch");
  if (phase_events) RT_CUDA(cudaEventRecord(phase_events[1], stream), "cudaEventRecord");

  if (!need_gate) {
    // overwrite / no conditioning: verification already wrote every row of e_out
    if (phase_events) {
      for (int k = 2; k < 4; ++k) RT_CUDA(cudaEventRecord(phase_events[k], stream), "cudaEventRecord");
    }
    return RETRACE_OK;
  }
  ConditioningArgs c{hD, hT, e, e_batch_stride, e_pos_stride, dense, Wc, Wv, Wg, beta, e_out};
  if ((st = enqueue_conditioning(c, dtype, B, K, d, tc, ablation == RETRACE_COND_RAW, accept_len, ws, L,
                                 phase_events, stream)) != RETRACE_OK)
    return st;
  if (phase_events) RT_CUDA(cudaEventRecord(phase_events[3], stream), "cudaEventRecord");
  return RETRACE_OK;
}

retrace_status retrace_wait_selftest(int kind, const uint32_t* flag, uint32_t target, void* ws, size_t ws_bytes,
                                    cudaStream_t stream) {
  g_err[0] = '\0';
  if (kind != 0 && kind != 1) return fail(RETRACE_ERR_INVALID_ARG, "kind must be 0 (counter) or 1 (mbarrier)");
  if (kind == 0 && !flag) return fail(RETRACE_ERR_INVALID_ARG, "NULL flag");
  retrace_status st = check_ws(ws, ws_bytes, 256);
  if (st != RETRACE_OK) return st;
  RT_CUDA(launch_wait_selftest(kind, flag, target, status_word(ws), stream), "wait self-test launch");
  return RETRACE_OK;
}

retrace_status retrace_verify_sampled(const void* target_logits, int64_t target_row_stride,
                                      int64_t target_batch_stride, const void* draft_logits,
                                      int64_t draft_row_stride, int64_t draft_batch_stride,
                                      retrace_dtype dtype, int B, int K, int V, const int32_t* draft,
                                      const float* uniforms, float temperature, int top_k, float top_p,
                                      int32_t* accept_len, int32_t* committed, int32_t* bonus, void* ws,
                                      size_t ws_bytes, cudaStream_t stream) {
  g_err[0] = '\0';
  retrace_status st = check_verify_args(target_logits, dtype, B, K, V, target_row_stride,
                                        target_batch_stride, draft, accept_len, committed, bonus);
  if (st != RETRACE_OK) return st;
  if ((st = check_sampling(B, K, V, draft_logits, draft_row_stride, draft_batch_stride, uniforms, temperature,
                           top_k, top_p)) != RETRACE_OK)
    return st;
  if (B == 0) return RETRACE_OK;
  const WsLayout Lw = ws_layout(B, K, 1, elem_size(dtype));
  if ((st = check_ws(ws, ws_bytes, Lw.total)) != RETRACE_OK) return st;
  if ((st = prepare_ws(ws, ws_bytes, Lw, B, K, stream)) != RETRACE_OK) return st;
  SampledArgs a{};
  a.tlogits = target_logits;
  a.t_row = target_row_stride;
  a.t_batch = target_batch_stride;
  a.dlogits = draft_logits;
  a.d_row = draft_row_stride;
  a.d_batch = draft_batch_stride;
  a.B = B;
  a.K = K;
  a.V = V;
  a.draft = draft;
  a.uniforms = uniforms;
  a.temperature = temperature;
  a.top_k = top_k;
  a.top_p = top_p;
  a.accept_len = accept_len;
  a.committed = committed;
  a.bonus = bonus;
  a.keys = reinterpret_cast<unsigned long long*>(reinterpret_cast<char*>(ws) + Lw.skeys);
  sampled_workspace(&a, reinterpret_cast<char*>(ws), Lw);
  RT_CUDA(launch_verify_sampled(a, dtype, stream), "sampled verification launch");
  return RETRACE_OK;
}

retrace_status retrace_round_sampled(const void* target_logits, int64_t target_row_stride,
                                     int64_t target_batch_stride, const void* draft_logits,
                                     int64_t draft_row_stride, int64_t draft_batch_stride,
                                     const int32_t* draft, const float* uniforms, float temperature,
                                     int top_k, float top_p, const void* hD, const void* hT, const void* e,
                                     int64_t e_batch_stride, int64_t e_pos_stride, const void* Wc,
                                     const void* Wv, const void* Wg, float beta, retrace_dtype dtype, int B,
                                     int K, int V, int d, int32_t* accept_len, int32_t* committed,
                                     int32_t* bonus, int32_t* n_out, void* e_out, void* ws, size_t ws_bytes,
                                     const cudaEvent_t* phase_events, cudaStream_t stream) {
  g_err[0] = '\0';
  retrace_status st = check_verify_args(target_logits, dtype, B, K, V, target_row_stride,
                                        target_batch_stride, draft, accept_len, committed, bonus);
  if (st != RETRACE_OK) return st;
  if ((st = check_sampling(B, K, V, draft_logits, draft_row_stride, draft_batch_stride, uniforms, temperature,
                           top_k, top_p)) != RETRACE_OK)
    return st;
  if ((st = check_cond_shape(dtype, B, K, d)) != RETRACE_OK) return st;
  if (B == 0) return RETRACE_OK;
  if (!hD || !hT || !e || !e_out || !Wc || !Wv || !Wg) return fail(RETRACE_ERR_INVALID_ARG, "NULL tensor pointer");
  int dense = 0;
  if ((st = e_mode(e_batch_stride, e_pos_stride, K, d, &dense)) != RETRACE_OK) return st;
  const WsLayout L = ws_layout(B, K, d, elem_size(dtype));
  if ((st = check_ws(ws, ws_bytes, L.total)) != RETRACE_OK) return st;
  if ((st = prepare_ws(ws, ws_bytes, L, B, K, stream)) != RETRACE_OK) return st;
  char* w = reinterpret_cast<char*>(ws);
  const bool tc = tc_supported(dtype, d) && aligned16(hD) && aligned16(hT) && aligned16(Wc) && aligned16(Wv) &&
                  aligned16(Wg) && aligned16(e) && aligned16(e_out);
  uint32_t* sync = reinterpret_cast<uint32_t*>(w + L.sync);

  if (phase_events) RT_CUDA(cudaEventRecord(phase_events[0], stream), "cudaEventRecord");
  // the finalize kernel packs the conditioned rows behind a counter at zero
  if (tc) RT_CUDA(cudaMemsetAsync(sync, 0, L.sync_bytes, stream), "cudaMemsetAsync(sync)");
  SampledArgs a{};
  a.tlogits = target_logits;
  a.t_row = target_row_stride;
  a.t_batch = target_batch_stride;
  a.dlogits = draft_logits;
  a.d_row = draft_row_stride;
  a.d_batch = draft_batch_stride;
  a.B = B;
  a.K = K;
  a.V = V;
  a.draft = draft;
  a.uniforms = uniforms;
  a.temperature = temperature;
  a.top_k = top_k;
  a.top_p = top_p;
  a.accept_len = accept_len;
  a.committed = committed;
  a.bonus = bonus;
  a.keys = reinterpret_cast<unsigned long long*>(w + L.skeys);
  sampled_workspace(&a, w, L);
  a.n_out = n_out;
  a.e = e;
  a.e_batch_stride = e_batch_stride;
  a.e_pos_stride = e_pos_stride;
  a.e_out = e_out;
  a.d = d;
  if (tc) {
    a.hD = hD;
    a.hT = hT;
    a.e_dense = dense;
    a.apack = w + L.apack;
    a.epack = w + L.epack;
    a.rowmap = reinterpret_cast<int32_t*>(w + L.rowmap);
    a.R_count = reinterpret_cast<int32_t*>(sync + kSyncRowCount);
  }
  RT_CUDA(launch_verify_sampled(a, dtype, stream), "sampled verification launch");
  if (phase_events) RT_CUDA(cudaEventRecord(phase_events[1], stream), "cudaEventRecord");
  ConditioningArgs c{hD, hT, e, e_batch_stride, e_pos_stride, dense, Wc, Wv, Wg, beta, e_out};
  if ((st = enqueue_conditioning(c, dtype, B, K, d, tc, false, accept_len, ws, L, phase_events, stream)) !=
      RETRACE_OK)
    return st;
  if (phase_events) RT_CUDA(cudaEventRecord(phase_events[3], stream), "cudaEventRecord");
  return RETRACE_OK;
}

retrace_status retrace_round_lowrank(const void* logits, int64_t logits_row_stride,
                                     int64_t logits_batch_stride, const int32_t* draft,
                                     const void* hD, const void* hT, const void* e, const void* P,
                                     const void* Bc, const void* Ac, const void* Wv, const void* Wg,
                                     float beta, retrace_dtype dtype, int B, int K, int V, int d,
                                     int32_t* accept_len, int32_t* committed, int32_t* bonus,
                                     int32_t* target_argmax, int32_t* n_out, void* e_out, void* ws,
                                     size_t ws_bytes, const cudaEvent_t* phase_events,
                                     cudaStream_t stream) {
  g_err[0] = '\0';
  retrace_status st = check_verify_args(logits, dtype, B, K, V, logits_row_stride,
                                        logits_batch_stride, draft, accept_len, committed, bonus);
  if (st != RETRACE_OK) return st;
  if ((st = check_cond_shape(dtype, B, K, d)) != RETRACE_OK) return st;
  if (B == 0) return RETRACE_OK;
  if (!hD || !hT || !e || !P || !Bc || !Ac || !Wv || !Wg || !e_out)
    return fail(RETRACE_ERR_INVALID_ARG, "NULL tensor pointer");
  const WsLayout Lw = ws_layout(B, K, d, elem_size(dtype));
  if ((st = check_ws(ws, ws_bytes, Lw.total)) != RETRACE_OK) return st;
  if ((st = prepare_ws(ws, ws_bytes, Lw, B, K, stream)) != RETRACE_OK) return st;
  char* w = reinterpret_cast<char*>(ws);
  const bool tc = lowrank_tc_supported(dtype, d) && aligned16(hD) && aligned16(hT) && aligned16(e) &&
                  aligned16(P) && aligned16(Bc) && aligned16(Ac) && aligned16(Wv) && aligned16(Wg) &&
                  aligned16(e_out);
  uint32_t* sync = reinterpret_cast<uint32_t*>(w + Lw.sync);
  int32_t* R = reinterpret_cast<int32_t*>(sync + kSyncRowCount);
  int32_t* rowmap = reinterpret_cast<int32_t*>(w + Lw.rowmap);

  if (phase_events) RT_CUDA(cudaEventRecord(phase_events[0], stream), "cudaEventRecord");
  if (tc) RT_CUDA(cudaMemsetAsync(sync, 0, Lw.sync_bytes, stream), "cudaMemsetAsync(sync)");
  VerifyArgs va{};
  va.logits = logits;
  va.B = B;
  va.K = K;
  va.V = V;
  va.row_stride = logits_row_stride;
  va.batch_stride = logits_batch_stride;
  va.draft = draft;
  va.accept_len = accept_len;
  va.committed = committed;
  va.bonus = bonus;
  va.target_argmax = target_argmax;
  va.n_out = n_out;
  verify_workspace(&va, w, Lw);
  va.e = e;
  va.e_batch_stride = 0;
  va.e_pos_stride = 0;
  va.e_out = e_out;
  va.d = d;
  va.hD = hD;
  va.cond_copy = kCondCopyKeep;
  if (tc) {  // the finalising CTA of each sequence packs its [m; u] rows
    va.hT = hT;
    va.apack = w + Lw.apack;
    va.epack = w + Lw.epack;
    va.rowmap = rowmap;
    va.R_count = R;
  }
  RT_CUDA(launch_verify(va, dtype, stream), "verify kernel launch");
  if (phase_events) RT_CUDA(cudaEventRecord(phase_events[1], stream), "cudaEventRecord");

  LowRankArgs la{};
  la.B = B;
  la.K = K;
  la.d = d;
  la.dtype = dtype;
  la.beta = beta;
  la.hD = hD;
  la.hT = hT;
  la.e = e;
  la.P = P;
  la.Bc = Bc;
  la.Ac = Ac;
  la.Wv = Wv;
  la.Wg = Wg;
  la.accept_len = accept_len;
  la.e_out = e_out;
  la.ge = reinterpret_cast<float*>(w + Lw.ge);
  la.apack = w + Lw.apack;
  la.rowmap = rowmap;
  la.R = R;
  la.zpart = reinterpret_cast<float*>(w + Lw.lrz);
  la.tpart = reinterpret_cast<float*>(w + Lw.lrt);
  la.rho = w + Lw.lrrho;
  la.gemv_next = sync + kSyncGemvNext;
  la.status = status_word(ws);
  RT_CUDA(launch_lowrank(la, tc, stream), "low-rank conditioning launch");
  if (phase_events) {
    for (int k = 2; k < 4; ++k) RT_CUDA(cudaEventRecord(phase_events[k], stream), "cudaEventRecord");
  }
  return RETRACE_OK;
}

}  // extern "C"
