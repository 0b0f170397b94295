// retrace_verify_noalloc: greedy verification for callers that cannot
// allocate device memory.
//
// Who needs this: code that is handed only its input and output buffers and
// has no way to obtain scratch memory -- for example a custom operator inside
// a host framework that owns every device allocation and passes none through
// its operator interface, or a serving loop that reserved its whole memory
// budget at start-up and forbids further cudaMalloc calls while requests run.
// retrace_verify needs a caller-provided workspace for its per-row argmax
// keys and per-sequence arrival counters; this entry point keeps them in a
// fixed array that is part of the library image instead.
//
// The array lives in device memory for as long as the library is loaded, on
// every GPU the process uses the library on.  Its size bounds the batch:
// B * (K + 1) keys of 8 bytes (rounded up to 256 bytes) plus B counters of 4
// bytes must fit in kNoAllocScratchBytes.
#include <stdio.h>

#include <mutex>

#include "internal.h"

namespace retrace {
namespace {

constexpr size_t kNoAllocScratchBytes = RETRACE_NOALLOC_SCRATCH_BYTES;
constexpr int kMaxDevices = 64;

// The scratch itself.  In host code this name is only a stand-in for the
// device symbol; the device address comes from cudaGetSymbolAddress below.
static __device__ __align__(256) unsigned char g_scratch[kNoAllocScratchBytes];

std::mutex g_setup_mutex;

// Device address of g_scratch per device, with the identity of the context it
// was looked up in.  A device reset destroys the primary context and the
// module with it; a new context loads the module again, possibly elsewhere,
// so an address is only reused while the same context is current.
struct ScratchEntry {
  void* addr;
  unsigned long long ctx_id;
};
ScratchEntry g_scratch_entry[kMaxDevices] = {};

typedef CUresult (*CtxGetCurrentFn)(CUcontext*);
typedef CUresult (*CtxGetIdFn)(CUcontext, unsigned long long*);

// Unique identifier of the context current on this thread, through the
// driver entry points the runtime exposes; 0 when there is none or the
// driver cannot tell (the address is then looked up on every call).
unsigned long long current_context_id() {
  static CtxGetCurrentFn get_current = nullptr;  // resolved under g_setup_mutex
  static CtxGetIdFn get_id = nullptr;
  static bool resolved = false;
  if (!resolved) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_current = reinterpret_cast<CtxGetCurrentFn>(p);
    p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_id = reinterpret_cast<CtxGetIdFn>(p);
    resolved = true;
  }
  if (!get_current || !get_id) return 0;
  CUcontext ctx = nullptr;
  unsigned long long id = 0;
  if (get_current(&ctx) != CUDA_SUCCESS || ctx == nullptr) return 0;
  if (get_id(ctx, &id) != CUDA_SUCCESS) return 0;
  return id;
}

// Errors are reported through retrace_last_error(), like every other entry point.
retrace_status fail(retrace_status s, const char* msg) {
  set_last_error(msg);
  return s;
}

// Device address of g_scratch on the current device: looked up with
// cudaGetSymbolAddress the first time, and again whenever the current context
// differs from the one the cached address came from.
cudaError_t scratch_address(int dev, void** out) {
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  ScratchEntry& e = g_scratch_entry[dev];
  const unsigned long long id = current_context_id();
  if (!e.addr || id == 0 || e.ctx_id != id) {
    void* p = nullptr;
    const cudaError_t err = cudaGetSymbolAddress(&p, g_scratch);  // makes the primary context current if needed
    if (err != cudaSuccess) return err;
    e.addr = p;
    e.ctx_id = current_context_id();
  }
  *out = e.addr;
  return cudaSuccess;
}

}  // namespace
}  // namespace retrace

using namespace retrace;

extern "C" retrace_status retrace_verify_noalloc(const void* logits, retrace_dtype dtype, int B, int K,
                                                 int V, int64_t logits_row_stride,
                                                 int64_t logits_batch_stride, const int32_t* draft,
                                                 int32_t* accept_len, int32_t* committed,
                                                 int32_t* bonus, int32_t* target_argmax,
                                                 cudaStream_t stream) {
  set_last_error("");
  if (dtype != RETRACE_BF16 && dtype != RETRACE_F32) return fail(RETRACE_ERR_INVALID_ARG, "unknown dtype");
  if (B < 0 || K < 0 || V < 1) return fail(RETRACE_ERR_INVALID_ARG, "bad shape: need B >= 0, K >= 0, V >= 1");
  if (K > kMaxK) return fail(RETRACE_ERR_UNSUPPORTED, "K exceeds the supported maximum of 1024");
  if (B == 0) return RETRACE_OK;
  if (!logits || (!draft && K > 0) || !accept_len || !committed || !bonus)
    return fail(RETRACE_ERR_INVALID_ARG, "NULL tensor pointer");
  if (logits_row_stride < V || logits_batch_stride < (int64_t)(K + 1) * logits_row_stride)
    return fail(RETRACE_ERR_INVALID_ARG, "logits strides smaller than the [B, K+1, V] shape");
  const size_t keys_bytes = align_up((size_t)B * (size_t)(K + 1) * 8, 256);
  const size_t need = keys_bytes + (size_t)B * 4;
  if (need > kNoAllocScratchBytes) {
    char msg[200];
    snprintf(msg, sizeof(msg),
             "batch too large for the fixed scratch: B*(K+1) keys and B counters need %zu bytes, "
             "the limit is %zu (RETRACE_NOALLOC_SCRATCH_BYTES)",
             need, kNoAllocScratchBytes);
    return fail(RETRACE_ERR_UNSUPPORTED, msg);
  }
  int dev = 0;
  cudaError_t err = cudaGetDevice(&dev);
  if (err != cudaSuccess) return fail(RETRACE_ERR_CUDA, cudaGetErrorString(err));
  if (dev < 0 || dev >= kMaxDevices) return fail(RETRACE_ERR_UNSUPPORTED, "device ordinal beyond 63");
  void* scratch = nullptr;
  err = scratch_address(dev, &scratch);
  if (err != cudaSuccess) return fail(RETRACE_ERR_CUDA, cudaGetErrorString(err));

  // The kernel expects its keys and counters to start at zero.  It leaves them
  // zero when it completes, but a call that never ran to the end (an error in
  // between) would not, so clear the part this call uses every time.
  err = cudaMemsetAsync(scratch, 0, need, stream);
  if (err != cudaSuccess) return fail(RETRACE_ERR_CUDA, cudaGetErrorString(err));

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
  a.keys = reinterpret_cast<unsigned long long*>(scratch);
  a.tickets = reinterpret_cast<uint32_t*>(reinterpret_cast<char*>(scratch) + keys_bytes);
  err = launch_verify(a, dtype, stream);
  if (err != cudaSuccess) return fail(RETRACE_ERR_CUDA, cudaGetErrorString(err));
  return RETRACE_OK;
}
