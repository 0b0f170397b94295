/*
 * retrace.h — C ABI of libretrace, the GB300 (sm_103a) per-round hot path of
 * ReTrace: Rejected-Trajectory Conditioning for Speculative Decoding
 * (arXiv 2608.29748).
 *
 * One ReTrace decoding round (Algorithm 1 of the paper) is, on the data path:
 *
 *   1. greedy verification of a K-token draft block against the target's
 *      verify logits (Algorithm 1 "Verify" step; greedy decoding = top-k 1,
 *      Appendix "Evaluation Protocol"): row-wise argmax, first mismatch,
 *      accepted length A, committed tokens and the correction/bonus token;
 *   2. alignment of the rejected suffix (Eq. 3-5) and target-aware
 *      correction r = m + beta * W_c [m; u]   (Eq. 6-7);
 *   3. gated residual conditioning of the next block's drafter inputs
 *      e~ = e + (W_v r) .* sigmoid(W_g [e; r])   (Eq. 8).
 *
 * Index conventions (0-based; the paper is 1-based).
 *   K      draft tokens per block (the paper's block size "B").
 *   B      number of independent sequences in the batch.
 *   V      vocabulary size;  d  hidden size (target and drafter share it).
 *   logits[b, i, :] for i = 0..K is the target's distribution at draft slot i:
 *          row i scores draft token i, row K scores the bonus position.
 *   hD[b, k, :]  drafter final-layer state of draft slot k   (paper h^D_{t,k+1}).
 *   hT[b, k, :]  target final-layer state at the position of draft slot k
 *                (paper h^T_{t,k+1}); its logits score slot k+1.
 *   A_b          accepted length, 0..K.  First rejected slot is A_b (paper r_t = A_t+1).
 *   n_b = max(0, K-1-A_b)   number of carried rows (Eq. 4 range, Algorithm 1 reset rule).
 *   For j < n_b:  m[b,j] = hD[b, A_b+1+j]  (Eq. 4),  u[b,j] = hT[b, A_b+j]  (Eq. 5).
 *   Rows j >= n_b carry nothing: m = u = r = 0 and e~[b,j] = e[b,j].
 *   e[b, j, :] for j = 0..K-1 are the drafter inputs of the K proposal positions
 *   (paper positions 1..K); the anchor (paper position 0) is never modified.
 *
 * Weight layout follows y = W x as the equations write it (row-major [out, in]):
 *   W_c [d, 2d]  columns 0..d-1 act on m, d..2d-1 on u              (Eq. 6)
 *   W_v [d, d]                                                     (Eq. 8)
 *   W_g [d, 2d]  columns 0..d-1 act on e, d..2d-1 on r              (Eq. 8)
 *   No biases: the equations have none.
 *
 * Precision.  RETRACE_BF16: every floating tensor (logits, hD, hT, e, weights,
 * r, e~) is bfloat16; products accumulate in fp32; r is rounded once to bf16
 * (round-to-nearest-even) before the gate projection; the gate, sigmoid and
 * residual run in fp32; e~ is rounded once to bf16.  RETRACE_F32: fp32
 * everywhere, plain FFMA accumulation (no TF32).
 *
 * Conventions common to every entry point.
 *   Ownership   every pointer is caller-owned DEVICE memory unless stated; the
 *               library allocates no device memory.  Scratch comes from the
 *               caller's workspace `ws` (size from retrace_workspace_bytes).
 *   Layout      row-major, last dimension contiguous.  16-byte alignment of
 *               every tensor base enables the vector paths; unaligned inputs
 *               take a scalar path on the GPU.  Outputs must not overlap inputs.
 *   Async       all work is enqueued on `stream` (NULL = legacy default stream);
 *               no entry point synchronises the host except
 *               retrace_workspace_check.
 *   Workspace   `ws` must be zeroed once by retrace_workspace_init before its
 *               first use.  Every successful call leaves the workspace ready for
 *               the next call, also of another shape (a workspace sized for the
 *               largest shape serves every smaller one): a call whose (B, K)
 *               differs from the previous call's on the same workspace first
 *               re-zeroes the workspace's small counter regions (one
 *               cudaMemsetAsync; the library keeps each workspace's last shape
 *               on the host, in call order).  A CUDA graph replays what was
 *               captured, so between replays and calls of other shapes on the
 *               same workspace call retrace_workspace_init (or give each shape
 *               its own workspace).  Calls sharing one workspace must be ordered
 *               on one stream (or otherwise serialised); after an error status,
 *               call retrace_workspace_init again.
 *   Errors      arguments are checked on the host before anything is enqueued;
 *               a bad argument returns a status and enqueues nothing.  A CUDA
 *               launch error returns RETRACE_ERR_CUDA.  Kernels never trap: a
 *               device-side wait that exceeds its bound sets a flag in `ws`
 *               that retrace_workspace_check reports.  retrace_last_error()
 *               gives a thread-local message for the last failing call.
 *   Semantics   NaN logits are outside the contract (result unspecified).  A
 *               draft token outside [0, V) never matches, so the block is
 *               rejected there.  Ties in the argmax resolve to the lowest
 *               vocabulary index; -0 and +0 compare equal.
 */
#ifndef RETRACE_H_
#define RETRACE_H_

#include <stddef.h>
#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  RETRACE_OK = 0,
  RETRACE_ERR_INVALID_ARG = 1, /* null pointer, negative size, bad stride        */
  RETRACE_ERR_UNSUPPORTED = 2, /* valid but not implemented (e.g. strided e)    */
  RETRACE_ERR_WORKSPACE = 3,   /* ws missing, misaligned or smaller than needed  */
  RETRACE_ERR_CUDA = 4,        /* a CUDA runtime call or launch failed           */
  RETRACE_ERR_DEVICE = 5       /* a kernel reported a bounded-wait expiry        */
} retrace_status;

typedef enum { RETRACE_F32 = 0, RETRACE_BF16 = 1 } retrace_dtype;

/* Thread-local, NUL-terminated description of the last non-OK status returned
 * on this thread ("" if none).  Owned by the library; valid until the next call
 * on the same thread. */
const char* retrace_last_error(void);

/* Library version string, e.g. "retrace 0.1.0 sm_103a". */
const char* retrace_version(void);

/* Bytes of workspace that every entry point below needs for a batch of this
 * shape (one size covers verify, align_refine, gate_fuse and round).  Pure host
 * arithmetic; returns 0 for invalid shapes (negative sizes or V < 1). */
size_t retrace_workspace_bytes(int B, int K, int V, int d, retrace_dtype dtype);

/* Zero `ws_bytes` bytes of the workspace on `stream` (cudaMemsetAsync).  Must
 * precede the first use of a workspace and follow any non-OK status. */
retrace_status retrace_workspace_init(void* ws, size_t ws_bytes, cudaStream_t stream);

/* Synchronises `stream`, then reads the device status word of `ws` into
 * *device_flags (0 = no kernel reported a problem; bit 0 = a bounded wait in a
 * tensor-core kernel expired).  Returns RETRACE_ERR_DEVICE if any bit is set. */
retrace_status retrace_workspace_check(const void* ws, size_t ws_bytes,
                                       uint32_t* device_flags, cudaStream_t stream);

/* Greedy verification of one draft block per sequence (Algorithm 1, Verify and
 * commit steps; greedy = top_k 1).
 *   logits        [B, K+1, V] of `dtype`; element (b,i,v) at
 *                 b*logits_batch_stride + i*logits_row_stride + v (elements).
 *                 Requires logits_row_stride >= V and
 *                 logits_batch_stride >= (K+1)*logits_row_stride.
 *   draft         [B, K] int32 draft tokens (may be NULL when K = 0).
 *   accept_len    [B] int32 out: A_b = first i < K with argmax(logits[b,i]) !=
 *                 draft[b,i], else K.
 *   committed     [B, K+1] int32 out: draft[b, 0..A_b-1], then the correction
 *                 (A_b < K) or bonus (A_b = K) token argmax(logits[b, A_b]);
 *                 positions after A_b are -1.
 *   bonus         [B] int32 out: argmax(logits[b, A_b]) (= committed[b, A_b]).
 *   target_argmax [B, K+1] int32 out, optional (NULL to skip).
 * B = 0 is a no-op.  K >= 0, V >= 1. */
retrace_status retrace_verify(const void* logits, retrace_dtype dtype, int B, int K, int V,
                              int64_t logits_row_stride, int64_t logits_batch_stride,
                              const int32_t* draft, int32_t* accept_len, int32_t* committed,
                              int32_t* bonus, int32_t* target_argmax, void* ws,
                              size_t ws_bytes, cudaStream_t stream);

/* Schedules of verification (every entry point that verifies, greedy or at
 * temperature T).  They differ in the rows they read, never in the results.
 *   RETRACE_VERIFY_FULL     one pass over every row of every sequence.
 *   RETRACE_VERIFY_WINDOWS  passes over row windows: rows [0, 4), then
 *                           windows half as long again as the one before
 *                           (4, 6, 9, ... rows; at most 16 passes; a short
 *                           remainder joins the last window).  Pass k reads
 *                           its window only for the sequences whose draft
 *                           tokens matched (greedy) or were accepted (at
 *                           temperature T) in every earlier row, so rows past
 *                           the window of the first mismatch are never read.
 *                           Applies when target_argmax is NULL (every row is
 *                           an output otherwise) and K+1 > 5; other calls take
 *                           the full pass.  retrace_verify_plan gives the
 *                           windows.
 *   RETRACE_VERIFY_AUTO     (default) WINDOWS where it applies and one row of
 *                           the whole batch is at least 16 MiB (B * V *
 *                           element size), FULL otherwise (each extra pass
 *                           costs a few microseconds, which small batches
 *                           do not win back).
 * Process-wide.  Returns the previous mode, or -1 (nothing changes) for an
 * unknown one. */
#define RETRACE_VERIFY_AUTO 0
#define RETRACE_VERIFY_FULL 1
#define RETRACE_VERIFY_WINDOWS 2
int retrace_set_verify_schedule(int mode);

/* The greedy verification schedule a call with this shape takes under the
 * current mode, given a workspace: returns the number of passes n (1 = the
 * one-pass schedule; -1 for an invalid shape or dtype) and, when
 * window_starts is not NULL, writes the n + 1 window boundaries (at most 17
 * entries: pass k reads rows [window_starts[k], window_starts[k+1]) of the
 * sequences that matched every row before it).  A windowed greedy round
 * launches n verification kernels plus one for the row copies (one kernel in
 * one pass); at temperature T, 2n kernels (top-k scan and accept tests per
 * pass) plus the copies (two in one pass).  Host arithmetic only. */
int retrace_verify_plan(int B, int K, int V, retrace_dtype dtype, int target_argmax, int* window_starts);

/* Rejected-trajectory alignment and target-aware correction (Eq. 3-7,
 * Algorithm 1 carry/reset steps).
 *   hD, hT      [B, K, d] of `dtype`, contiguous.
 *   accept_len  [B] int32 (device), values in [0, K]; values outside are
 *               clamped to that range.
 *   Wc          [d, 2d] of `dtype`, row-major.
 *   beta        correction strength (1.0 at inference; 0 gives the "raw
 *               conditioning" ablation).
 *   r_out       [B, K, d] of `dtype` out: r[b,j] = m + beta*W_c[m;u] for
 *               j < n_b, zero rows for j >= n_b (Eq. 4-5 zero padding).
 *   n_out       [B] int32 out: n_b = max(0, K-1-A_b).
 * K >= 1, d >= 1. */
retrace_status retrace_align_refine(const void* hD, const void* hT, retrace_dtype dtype, int B,
                                    int K, int d, const int32_t* accept_len, const void* Wc,
                                    float beta, void* r_out, int32_t* n_out, void* ws,
                                    size_t ws_bytes, cudaStream_t stream);

/* Gated residual conditioning (Eq. 8).
 *   e           drafter inputs of the K proposal positions.  Two layouts:
 *               (e_batch_stride, e_pos_stride) = (0, 0): one vector [d]
 *               broadcast to every position (the DFlash mask embedding);
 *               (K*d, d): dense [B, K, d].  Other strides: UNSUPPORTED.
 *   r, n        [B, K, d] corrected signal and [B] row counts, as produced
 *               by retrace_align_refine; rows j >= n_b of r are not read.
 *   Wv [d, d], Wg [d, 2d] of `dtype`.
 *   e_out       [B, K, d] out: e + (Wv r) .* sigmoid(Wg [e; r]) for j < n_b,
 *               e bit-exactly for j >= n_b.
 * K >= 1, d >= 1. */
retrace_status retrace_gate_fuse(const void* e, int64_t e_batch_stride, int64_t e_pos_stride,
                                 const void* r, const int32_t* n, const void* Wv, const void* Wg,
                                 retrace_dtype dtype, int B, int K, int d, void* e_out,
                                 void* ws, size_t ws_bytes, cudaStream_t stream);

/* Flags of retrace_round.  With none set the round computes the method as
 * written (corrected conditioning, gated).  The three conditioning variants of
 * the component ablation (Sec. "Component Ablation", Table 3; Appendix
 * "Ablation Settings") build the same aligned signal m_j = hD[b, A_b+1+j] and
 * differ in how it enters the next block; at most one of them may be set:
 *   RETRACE_COND_RAW        raw conditioning, gated: no correction, r = m
 *                           (Eq. 8 applied to the aligned drafter states).
 *   RETRACE_COND_OVERWRITE  raw conditioning, overwrite: e~_j = m_j for
 *                           j < n_b (the mask inputs are replaced).
 *   RETRACE_COND_NONE       no conditioning (the DFlash row): e~ = e.
 * Rows j >= n_b keep e bit-exactly in every variant, and n_out still reports
 * n_b.  Wc, Wv and Wg are not read where the variant does not use them (they
 * may be NULL then).
 *   RETRACE_ROUND_OVERLAP   run verification and both projections in one
 *                           persistent launch whose warps overlap the logits
 *                           stream with the tensor-core work (the corrected
 *                           method only: bf16, d a multiple of 256, 16-byte
 *                           aligned contiguous [B, K+1, V] logits with V a
 *                           multiple of 8 and V >= 4096, K >= 2, 4d <= 16384).
 *                           Same results bit for bit; other shapes or an
 *                           ablation flag return RETRACE_ERR_UNSUPPORTED.
 *                           Experimental: measured slower than the default
 *                           round (about 2.4x the time at B = 256); the
 *                           default round never takes it.
 * Unknown bits, or two ablation flags together, return
 * RETRACE_ERR_INVALID_ARG. */
#define RETRACE_ROUND_OVERLAP 0x1u
#define RETRACE_COND_RAW 0x2u
#define RETRACE_COND_OVERWRITE 0x4u
#define RETRACE_COND_NONE 0x8u

/* One full round on one stream: verify, then align/refine and gated fusion of
 * the rejected suffix into the next block's inputs (Algorithm 1).  Arguments
 * have the meaning given above; r stays inside `ws` (compacted to the R =
 * sum_b n_b conditioned rows) and is not returned.  No host synchronisation.
 *   n_out          [B] int32 out, optional (NULL to skip).
 *   target_argmax  [B, K+1] int32 out, optional.
 *   flags          0, or the RETRACE_ROUND_* / RETRACE_COND_* bits above.
 *   phase_events   optional array of 4 cudaEvent_t recorded on `stream`
 *                  before verification, after it, after the correction
 *                  projection and after the gated fusion (NULL to skip).
 * K >= 1, V >= 1, d >= 1. */
retrace_status retrace_round(const void* logits, int64_t logits_row_stride,
                             int64_t logits_batch_stride, const int32_t* draft, const void* hD,
                             const void* hT, const void* e, int64_t e_batch_stride,
                             int64_t e_pos_stride, const void* Wc, const void* Wv, const void* Wg,
                             float beta, retrace_dtype dtype, int B, int K, int V, int d,
                             int32_t* accept_len, int32_t* committed, int32_t* bonus,
                             int32_t* target_argmax, int32_t* n_out, void* e_out, void* ws,
                             size_t ws_bytes, uint32_t flags, const cudaEvent_t* phase_events,
                             cudaStream_t stream);

/* Stochastic verification of a draft block at temperature T with top-k /
 * top-p filtering (the paper samples at T = 1 with top_p = 0.95 and
 * top_k = 20, Appendix "Evaluation Protocol", and keeps the underlying
 * verification, which it does not state).  The rule implemented is standard
 * speculative sampling on the filtered distributions:
 *   p_i, q_i   softmax(logits / T) of target row i and drafter row i,
 *              restricted to the top_k logits (the lower index first among
 *              equal values), renormalised, then to the shortest prefix of
 *              them whose probability reaches top_p, renormalised;
 *   accept     draft token x_i iff uniforms[b, i] * q_i(x_i) < p_i(x_i) (a
 *              token outside [0, V) is rejected); A_b = the first rejection;
 *   draw       with uniforms[b, K], inverse CDF over the filtered list (in
 *              descending probability): from max(0, p_A - q_A), renormalised
 *              (from p_A if it is zero), when A_b < K, else from p_K.
 * Outputs as in retrace_verify, with the drawn token as committed[b, A_b]
 * and bonus[b].  Uniforms are the caller's random numbers, in [0, 1).
 *   target_logits  [B, K+1, V]; draft_logits [B, K, V] (the drafter's logits
 *                  of the proposals), both `dtype`, V contiguous, strides in
 *                  elements.
 *   temperature > 0, 1 <= top_k <= 64 and top_k <= V, 0 < top_p <= 1.
 * The conditioning of the next block is unchanged: retrace_align_refine and
 * retrace_gate_fuse take this call's accept_len (retrace_round_sampled runs
 * both steps as one round). */
retrace_status retrace_verify_sampled(const void* target_logits, int64_t target_row_stride,
                                      int64_t target_batch_stride, const void* draft_logits,
                                      int64_t draft_row_stride, int64_t draft_batch_stride,
                                      retrace_dtype dtype, int B, int K, int V, const int32_t* draft,
                                      const float* uniforms, float temperature, int top_k, float top_p,
                                      int32_t* accept_len, int32_t* committed, int32_t* bonus, void* ws,
                                      size_t ws_bytes, cudaStream_t stream);

/* One round at temperature T: the stochastic verification of
 * retrace_verify_sampled, then the corrected, gated conditioning of the
 * rejected suffix (Eq. 4-8) exactly as retrace_round computes it, with A_b the
 * sampled accepted length (Algorithm 1 with its acceptance test replaced by
 * speculative sampling; the paper evaluates at T = 1).  Arguments are those of
 * retrace_verify_sampled followed by those of retrace_round; there is no
 * target_argmax output and no flags.  The finalize kernel writes the rows
 * j >= n_b of e_out and, on the tensor-core path (bf16, d a multiple of 256,
 * 16-byte aligned tensors), packs the conditioned rows for one persistent
 * conditioning launch.
 *   phase_events  optional 4 events: before verification, after it, after the
 *                 correction (after both projections on the tensor-core
 *                 path), after the gated fusion.
 * temperature > 0, 1 <= top_k <= 64 and top_k <= V, 0 < top_p <= 1, K >= 1,
 * V >= 1, d >= 1. */
retrace_status retrace_round_sampled(const void* target_logits, int64_t target_row_stride,
                                     int64_t target_batch_stride, const void* draft_logits,
                                     int64_t draft_row_stride, int64_t draft_batch_stride,
                                     const int32_t* draft, const float* uniforms, float temperature,
                                     int top_k, float top_p, const void* hD, const void* hT, const void* e,
                                     int64_t e_batch_stride, int64_t e_pos_stride, const void* Wc,
                                     const void* Wv, const void* Wg, float beta, retrace_dtype dtype, int B,
                                     int K, int V, int d, int32_t* accept_len, int32_t* committed,
                                     int32_t* bonus, int32_t* n_out, void* e_out, void* ws, size_t ws_bytes,
                                     const cudaEvent_t* phase_events, cudaStream_t stream);

/* Ranks of the low-rank conditioning path (Appendix "Concurrent-Serving
 * Experiment": rank-64 rejected-suffix latents, rank-32 correction). */
#define RETRACE_LOWRANK_LATENT 64
#define RETRACE_LOWRANK_CORRECTION 32

/* One round with the low-rank realisation of the conditioning path
 * (Appendix "Concurrent-Serving Experiment").  The paper names its parts
 * (rank-64 rejected-suffix latents, input-side latent residual fusion, a
 * rank-32 target-aware correction, a one-round lifetime) without equations;
 * the reading implemented here is Eq. 6-8 with the d-wide signal replaced by
 * a rank-64 latent.  For each conditioned row j < n_b, with
 * m = hD[b, A_b+1+j] and u = hT[b, A_b+j] (Eq. 4-5):
 *     z   = P m                                   (the latent)
 *     rho = z + beta * A_c (B_c [z; u])           (rank-32 correction)
 *     e~  = e + (W_v rho) .* sigmoid(W_g [e; rho])
 * z and rho are rounded to bf16 (bf16 dtype); rows j >= n_b keep e exactly.
 * Verification outputs are those of retrace_round.
 *   e     [d], the broadcast drafter input (the DFlash mask embedding); a
 *         per-position e is not supported by this form.
 *   P     [64, d];  B_c [32, 64 + d] (columns 0..63 act on z);  A_c [64, 32];
 *   W_v   [d, 64];  W_g [d, d + 64] (columns 0..d-1 act on e); all `dtype`,
 *         row-major.
 *   phase_events  optional 4 events: before verification, after it, after
 *         the latent projections, after the fusion.
 * Tensor cores for bf16 with d a multiple of 128 and 16-byte aligned tensors;
 * an FFMA kernel otherwise.  K >= 1, V >= 1, d >= 1. */
retrace_status retrace_round_lowrank(const void* logits, int64_t logits_row_stride,
                                     int64_t logits_batch_stride, const int32_t* draft,
                                     const void* hD, const void* hT, const void* e, const void* P,
                                     const void* Bc, const void* Ac, const void* Wv, const void* Wg,
                                     float beta, retrace_dtype dtype, int B, int K, int V, int d,
                                     int32_t* accept_len, int32_t* committed, int32_t* bonus,
                                     int32_t* target_argmax, int32_t* n_out, void* e_out, void* ws,
                                     size_t ws_bytes, const cudaEvent_t* phase_events,
                                     cudaStream_t stream);

/* Self-test of the bounded device waits.  The pipelined tensor-core kernels
 * wait on mbarrier phases and on counters that other CTAs raise, and none of
 * those waits may spin forever: each gives up after about one second, sets
 * bit 0 of the workspace status word (reported by retrace_workspace_check),
 * and its kernel returns normally, so the CUDA context stays usable.  This
 * call runs the same wait code in one thread on a condition the caller
 * controls:
 *   kind 0  waits until the device word *flag >= target (the counter wait);
 *   kind 1  waits for an mbarrier phase that completes only if target == 0
 *           (the phase wait; flag is not read and may be NULL).
 * A condition that is already met returns at once; one that never becomes
 * true takes the full bound and sets the flag.  Only the status word of `ws`
 * (at least 256 bytes, 256-byte aligned) is written; call
 * retrace_workspace_init before reusing the workspace after a set flag. */
retrace_status retrace_wait_selftest(int kind, const uint32_t* flag, uint32_t target, void* ws, size_t ws_bytes,
                                     cudaStream_t stream);

/* Size in bytes of the fixed device scratch used by retrace_verify_noalloc. */
#define RETRACE_NOALLOC_SCRATCH_BYTES 65536

/* Greedy verification for callers that cannot allocate device memory.
 *
 * The paper has no counterpart to this entry point; it exists for callers that
 * are handed only their input and output buffers and have no way to obtain
 * scratch memory (for example a custom operator whose host framework owns all
 * device allocations and passes none through, or a serving loop that reserved
 * its whole memory budget up front and must not call cudaMalloc while it runs).
 * It computes exactly what retrace_verify computes, with the same arguments
 * minus the workspace: the per-row argmax keys and per-sequence counters live
 * in a fixed array of RETRACE_NOALLOC_SCRATCH_BYTES bytes inside the library,
 * which every GPU that uses the library keeps until the process exits.
 *
 *   Limit      8 * B * (K+1) bytes (rounded up to a multiple of 256) plus
 *              4 * B bytes must not exceed RETRACE_NOALLOC_SCRATCH_BYTES
 *              (B = 256, K = 16 needs 35,840 bytes); a larger batch returns
 *              RETRACE_ERR_UNSUPPORTED and enqueues nothing.
 *   Set-up     the first call on each device looks up the array's device
 *              address (cudaGetSymbolAddress) with that device current; make
 *              that first call before any stream capture on the device.  The
 *              address is kept per device together with the identity of the
 *              context it belongs to: after a device reset (cudaDeviceReset)
 *              the next call looks it up again, so that call too should come
 *              before any capture.
 *   Schedule   always one pass over every row (RETRACE_VERIFY_FULL): the
 *              row-window schedule keeps live lists in the workspace, which
 *              this entry point does not have.  At large batches it is
 *              therefore slower than retrace_verify with a workspace and
 *              target_argmax NULL, which reads only the windows up to each
 *              sequence's first mismatch.
 *   Sharing    every call on a device uses the same array and clears the part
 *              it needs (cudaMemsetAsync on `stream`) before its kernel runs.
 *              Calls whose work may overlap on the GPU (different streams with
 *              no ordering between them) race on the array and give wrong
 *              results: order them on one stream.
 *   Memory     calls no cudaMalloc, cudaFree or other allocating routine. */
retrace_status retrace_verify_noalloc(const void* logits, retrace_dtype dtype, int B, int K, int V,
                                      int64_t logits_row_stride, int64_t logits_batch_stride,
                                      const int32_t* draft, int32_t* accept_len,
                                      int32_t* committed, int32_t* bonus,
                                      int32_t* target_argmax, cudaStream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* RETRACE_H_ */
