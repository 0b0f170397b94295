// Conditioning projections on the CUDA cores (FFMA, fp32 accumulation).
//
// This path serves fp32 workloads (which must not use TF32) and bf16 shapes
// the tensor-core kernels do not take (hidden size not a multiple of 256 or
// unaligned tensors).  Same arithmetic as the tensor-core path:
//   correction  r = m + beta * W_c [m; u]                (Eq. 6-7)
//   gate        e~ = e + (W_v r) .* sigmoid(W_g [e; r])  (Eq. 8)
// with the operand rows gathered through the device-side row plan.
#include "common.cuh"
#include "internal.h"
#include "plan.cuh"

namespace retrace {
namespace {

constexpr int kNT = 256;
constexpr int TM = 32, TN = 64, TK = 32;

struct SimtCorrectParams {
  const void* hD;
  const void* hT;
  const void* Wc;
  float beta;
  int B, K, d;
  RowSource rows;
  void* out;
  int compact_out;
  int raw;  // r = m: no accumulation, W_c not read
};

struct SimtGateParams {
  const void* e;
  int e_dense;
  const void* r;
  int r_compact;
  const void* Wv;
  const void* Wg;
  const float* ge;
  int B, K, d;
  RowSource rows;
  void* out;
};

// Threads form a 16 x 16 grid; thread (ty, tx) owns rows 2ty..2ty+1 and
// columns 4tx..4tx+3 of the 32 x 64 output tile.
template <typename T>
__global__ void __launch_bounds__(kNT) simt_correct_kernel(const SimtCorrectParams p) {
  __shared__ int s_b[TM], s_j[TM], s_nb[TM], s_scan[kNT / 32 + 1];
  __shared__ long long s_m[TM], s_u[TM];
  __shared__ float As[TM][TK + 1];
  __shared__ float Bs[TN][TK + 1];

  const long long m0 = (long long)blockIdx.x * TM;
  const int n0 = blockIdx.y * TN;
  const int R = plan_tile<kNT, TM>(p.rows, p.B, p.K, m0, s_b, s_j, s_nb, s_scan);
  if (m0 >= R) return;
  const int K = p.K, d = p.d, tid = threadIdx.x;
  if (tid < TM) {
    const int b = s_b[tid];
    if (b >= 0) {
      const int A = K - 1 - s_nb[tid];
      s_m[tid] = ((long long)b * K + A + 1 + s_j[tid]) * d;  // m_j = hD[b, A+1+j]
      s_u[tid] = ((long long)b * K + A + s_j[tid]) * d;      // u_j = hT[b, A+j]
    } else {
      s_m[tid] = -1;
      s_u[tid] = -1;
    }
  }
  __syncthreads();
  const T* hD = reinterpret_cast<const T*>(p.hD);
  const T* hT = reinterpret_cast<const T*>(p.hT);
  const T* Wc = reinterpret_cast<const T*>(p.Wc);
  const int ty = tid / 16, tx = tid % 16;
  float acc[2][4] = {};
  const int K2 = 2 * d;
  for (int k0 = 0; k0 < (p.raw ? 0 : K2); k0 += TK) {
    for (int idx = tid; idx < TM * TK; idx += kNT) {
      const int r = idx / TK, kk = idx % TK, k = k0 + kk;
      float v = 0.f;
      if (s_m[r] >= 0 && k < K2) v = (k < d) ? to_f32(hD[s_m[r] + k]) : to_f32(hT[s_u[r] + k - d]);
      As[r][kk] = v;
    }
    for (int idx = tid; idx < TN * TK; idx += kNT) {
      const int c = idx / TK, kk = idx % TK, k = k0 + kk, n = n0 + c;
      Bs[c][kk] = (n < d && k < K2) ? to_f32(Wc[(long long)n * K2 + k]) : 0.f;
    }
    __syncthreads();
#pragma unroll 8
    for (int kk = 0; kk < TK; ++kk) {
      const float a0 = As[2 * ty][kk], a1 = As[2 * ty + 1][kk];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float bq = Bs[4 * tx + q][kk];
        acc[0][q] = fmaf(a0, bq, acc[0][q]);
        acc[1][q] = fmaf(a1, bq, acc[1][q]);
      }
    }
    __syncthreads();
  }
  T* out = reinterpret_cast<T*>(p.out);
#pragma unroll
  for (int rr = 0; rr < 2; ++rr) {
    const int r = 2 * ty + rr;
    const int b = s_b[r];
    if (b < 0) continue;
    const long long orow = p.compact_out ? (m0 + r) : ((long long)b * K + s_j[r]);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int n = n0 + 4 * tx + q;
      if (n >= d) continue;
      const T m = hD[s_m[r] + n];
      out[orow * d + n] = p.raw ? m : from_f32<T>(to_f32(m) + p.beta * acc[rr][q]);
    }
  }
}

template <typename T>
__global__ void __launch_bounds__(kNT) simt_gate_kernel(const SimtGateParams p) {
  __shared__ int s_b[TM], s_j[TM], s_nb[TM], s_scan[kNT / 32 + 1];
  __shared__ long long s_r[TM], s_e[TM];
  __shared__ float As[TM][TK + 1];
  __shared__ float Bv[TN][TK + 1];
  __shared__ float Bg[TN][TK + 1];

  const long long m0 = (long long)blockIdx.x * TM;
  const int n0 = blockIdx.y * TN;
  const int R = plan_tile<kNT, TM>(p.rows, p.B, p.K, m0, s_b, s_j, s_nb, s_scan);
  if (m0 >= R) return;
  const int K = p.K, d = p.d, tid = threadIdx.x;
  if (tid < TM) {
    const int b = s_b[tid];
    if (b >= 0) {
      const long long pos = (long long)b * K + s_j[tid];
      s_r[tid] = (p.r_compact ? (m0 + tid) : pos) * d;
      s_e[tid] = p.e_dense ? pos * d : 0;
    } else {
      s_r[tid] = -1;
      s_e[tid] = 0;
    }
  }
  __syncthreads();
  const T* r = reinterpret_cast<const T*>(p.r);
  const T* e = reinterpret_cast<const T*>(p.e);
  const T* Wv = reinterpret_cast<const T*>(p.Wv);
  const T* Wg = reinterpret_cast<const T*>(p.Wg);
  const int ty = tid / 16, tx = tid % 16;
  const long long ldg = 2LL * d;
  float av[2][4] = {}, ag[2][4] = {};
  // v = W_v r and the r half of the gate, W_g[:, d:2d] r.
  for (int k0 = 0; k0 < d; k0 += TK) {
    for (int idx = tid; idx < TM * TK; idx += kNT) {
      const int rr = idx / TK, kk = idx % TK, k = k0 + kk;
      As[rr][kk] = (s_r[rr] >= 0 && k < d) ? to_f32(r[s_r[rr] + k]) : 0.f;
    }
    for (int idx = tid; idx < TN * TK; idx += kNT) {
      const int c = idx / TK, kk = idx % TK, k = k0 + kk, n = n0 + c;
      const bool ok = n < d && k < d;
      Bv[c][kk] = ok ? to_f32(Wv[(long long)n * d + k]) : 0.f;
      Bg[c][kk] = ok ? to_f32(Wg[(long long)n * ldg + d + k]) : 0.f;
    }
    __syncthreads();
#pragma unroll 8
    for (int kk = 0; kk < TK; ++kk) {
      const float a0 = As[2 * ty][kk], a1 = As[2 * ty + 1][kk];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float bv = Bv[4 * tx + q][kk], bg = Bg[4 * tx + q][kk];
        av[0][q] = fmaf(a0, bv, av[0][q]);
        av[1][q] = fmaf(a1, bv, av[1][q]);
        ag[0][q] = fmaf(a0, bg, ag[0][q]);
        ag[1][q] = fmaf(a1, bg, ag[1][q]);
      }
    }
    __syncthreads();
  }
  // Per-position e: the e half of the gate, W_g[:, 0:d] e.
  if (p.e_dense) {
    for (int k0 = 0; k0 < d; k0 += TK) {
      for (int idx = tid; idx < TM * TK; idx += kNT) {
        const int rr = idx / TK, kk = idx % TK, k = k0 + kk;
        As[rr][kk] = (s_r[rr] >= 0 && k < d) ? to_f32(e[s_e[rr] + k]) : 0.f;
      }
      for (int idx = tid; idx < TN * TK; idx += kNT) {
        const int c = idx / TK, kk = idx % TK, k = k0 + kk, n = n0 + c;
        Bg[c][kk] = (n < d && k < d) ? to_f32(Wg[(long long)n * ldg + k]) : 0.f;
      }
      __syncthreads();
#pragma unroll 8
      for (int kk = 0; kk < TK; ++kk) {
        const float a0 = As[2 * ty][kk], a1 = As[2 * ty + 1][kk];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const float bg = Bg[4 * tx + q][kk];
          ag[0][q] = fmaf(a0, bg, ag[0][q]);
          ag[1][q] = fmaf(a1, bg, ag[1][q]);
        }
      }
      __syncthreads();
    }
  }
  T* out = reinterpret_cast<T*>(p.out);
#pragma unroll
  for (int rr = 0; rr < 2; ++rr) {
    const int row = 2 * ty + rr;
    const int b = s_b[row];
    if (b < 0) continue;
    const long long orow = (long long)b * K + s_j[row];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int n = n0 + 4 * tx + q;
      if (n >= d) continue;
      const float g = ag[rr][q] + (p.e_dense ? 0.f : p.ge[n]);
      const float ev = to_f32(e[s_e[row] + n]);
      const float gate = 1.f / (1.f + expf(-g));
      out[orow * d + n] = from_f32<T>(ev + av[rr][q] * gate);
    }
  }
}

// ---------------------------------------------------------------------------
// Few rows (B (K-1) <= kRowsMax): one warp per output feature
// ---------------------------------------------------------------------------
// With a handful of rows the 32 x 64 tiles above leave all but d/64 SMs idle
// and walk the reduction in 32-deep steps, one load latency each.  Here each
// warp owns one output feature n and all rows: its lanes stride the
// reduction index (coalesced loads of the weight row, the operand rows read
// through L1), each lane keeps kRowGroup row sums, and a butterfly of
// shuffles adds the lanes in a fixed order (results repeat bit for bit).
// The rows are taken kRowGroup at a time (the weight row is re-read per
// group), and each lane issues the loads of kBatch reduction steps for the
// weight and every row of the group before it multiplies.
constexpr int kRowsMax = 32;  // one plan tile
constexpr int kRowGroup = 8;
constexpr int kBatch = 4;  // reduction steps per lane with their loads issued together
constexpr int kRowsWarps = kNT / 32;

__device__ __forceinline__ float warp_sum(float s) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xFFFFFFFFu, s, off);
  return s;
}

template <typename T>
__global__ void __launch_bounds__(kNT) simt_rows_correct_kernel(const SimtCorrectParams p) {
  __shared__ int s_b[kRowsMax], s_j[kRowsMax], s_nb[kRowsMax], s_scan[kNT / 32 + 1];
  __shared__ long long s_m[kRowsMax], s_u[kRowsMax];
  const int R = plan_tile<kNT, kRowsMax>(p.rows, p.B, p.K, 0, s_b, s_j, s_nb, s_scan);
  const int K = p.K, d = p.d, tid = threadIdx.x, lane = tid & 31;
  if (tid < kRowsMax) {
    const int b = s_b[tid];
    const int A = K - 1 - s_nb[tid];
    s_m[tid] = b >= 0 ? ((long long)b * K + A + 1 + s_j[tid]) * d : 0;  // m_j = hD[b, A+1+j]
    s_u[tid] = b >= 0 ? ((long long)b * K + A + s_j[tid]) * d : 0;      // u_j = hT[b, A+j]
  }
  __syncthreads();
  const int n = blockIdx.x * kRowsWarps + (tid >> 5);
  if (n >= d) return;
  const T* hD = reinterpret_cast<const T*>(p.hD);
  const T* hT = reinterpret_cast<const T*>(p.hT);
  const T* w = reinterpret_cast<const T*>(p.Wc) + (long long)n * 2 * d;
  T* out = reinterpret_cast<T*>(p.out);
  const int nrows = R < kRowsMax ? R : kRowsMax;
  for (int g0 = 0; g0 < nrows; g0 += kRowGroup) {
    const int gn = nrows - g0 < kRowGroup ? nrows - g0 : kRowGroup;
    float acc[kRowGroup];
#pragma unroll
    for (int q = 0; q < kRowGroup; ++q) acc[q] = 0.f;
    if (!p.raw) {
      // c = W_c [m; u]: the m half (k < d), then the u half
      for (int half = 0; half < 2; ++half) {
        const T* wh = w + half * d;
        const T* src[kRowGroup];
#pragma unroll
        for (int q = 0; q < kRowGroup; ++q) {  // rows past the group repeat its first (discarded)
          const int row = g0 + (q < gn ? q : 0);
          src[q] = half == 0 ? hD + s_m[row] : hT + s_u[row];
        }
        for (int k0 = lane; k0 < d; k0 += 32 * kBatch) {
          float wk[kBatch], x[kRowGroup][kBatch];
#pragma unroll
          for (int u = 0; u < kBatch; ++u) {
            const int k = k0 + 32 * u;
            wk[u] = k < d ? to_f32(wh[k]) : 0.f;
#pragma unroll
            for (int q = 0; q < kRowGroup; ++q) x[q][u] = k < d ? to_f32(src[q][k]) : 0.f;
          }
#pragma unroll
          for (int q = 0; q < kRowGroup; ++q)
#pragma unroll
            for (int u = 0; u < kBatch; ++u) acc[q] = fmaf(wk[u], x[q][u], acc[q]);
        }
      }
#pragma unroll
      for (int q = 0; q < kRowGroup; ++q) acc[q] = warp_sum(acc[q]);
    }
    if (lane < gn) {
      float a = acc[0];
#pragma unroll
      for (int q = 1; q < kRowGroup; ++q)
        if (lane == q) a = acc[q];
      const int row = g0 + lane;
      const long long orow = p.compact_out ? row : ((long long)s_b[row] * K + s_j[row]);
      const T m = hD[s_m[row] + n];
      out[orow * d + n] = p.raw ? m : from_f32<T>(to_f32(m) + p.beta * a);
    }
  }
}

template <typename T>
__global__ void __launch_bounds__(kNT) simt_rows_gate_kernel(const SimtGateParams p) {
  __shared__ int s_b[kRowsMax], s_j[kRowsMax], s_nb[kRowsMax], s_scan[kNT / 32 + 1];
  __shared__ long long s_r[kRowsMax], s_e[kRowsMax];
  const int R = plan_tile<kNT, kRowsMax>(p.rows, p.B, p.K, 0, s_b, s_j, s_nb, s_scan);
  const int K = p.K, d = p.d, tid = threadIdx.x, lane = tid & 31;
  if (tid < kRowsMax) {
    const int b = s_b[tid];
    const long long pos = b >= 0 ? (long long)b * K + s_j[tid] : 0;
    s_r[tid] = (p.r_compact ? tid : pos) * d;
    s_e[tid] = p.e_dense ? pos * d : 0;
  }
  __syncthreads();
  const int n = blockIdx.x * kRowsWarps + (tid >> 5);
  if (n >= d) return;
  const T* r = reinterpret_cast<const T*>(p.r);
  const T* e = reinterpret_cast<const T*>(p.e);
  const T* wv = reinterpret_cast<const T*>(p.Wv) + (long long)n * d;
  const T* wg = reinterpret_cast<const T*>(p.Wg) + (long long)n * 2 * d;
  T* out = reinterpret_cast<T*>(p.out);
  const int nrows = R < kRowsMax ? R : kRowsMax;
  for (int g0 = 0; g0 < nrows; g0 += kRowGroup) {
    const int gn = nrows - g0 < kRowGroup ? nrows - g0 : kRowGroup;
    float av[kRowGroup], ag[kRowGroup];
#pragma unroll
    for (int q = 0; q < kRowGroup; ++q) av[q] = ag[q] = 0.f;
    // v = W_v r and the r half of the gate, W_g[:, d:2d] r
    const T* rs[kRowGroup];
    const T* es[kRowGroup];
#pragma unroll
    for (int q = 0; q < kRowGroup; ++q) {  // rows past the group repeat its first (discarded)
      const int row = g0 + (q < gn ? q : 0);
      rs[q] = r + s_r[row];
      es[q] = e + s_e[row];
    }
    for (int k0 = lane; k0 < d; k0 += 32 * kBatch) {
      float wvk[kBatch], wgk[kBatch], x[kRowGroup][kBatch];
#pragma unroll
      for (int u = 0; u < kBatch; ++u) {
        const int k = k0 + 32 * u;
        wvk[u] = k < d ? to_f32(wv[k]) : 0.f;
        wgk[u] = k < d ? to_f32(wg[d + k]) : 0.f;
#pragma unroll
        for (int q = 0; q < kRowGroup; ++q) x[q][u] = k < d ? to_f32(rs[q][k]) : 0.f;
      }
#pragma unroll
      for (int q = 0; q < kRowGroup; ++q)
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {
          av[q] = fmaf(wvk[u], x[q][u], av[q]);
          ag[q] = fmaf(wgk[u], x[q][u], ag[q]);
        }
    }
    // per-position e: the e half of the gate, W_g[:, 0:d] e
    if (p.e_dense) {
      for (int k0 = lane; k0 < d; k0 += 32 * kBatch) {
        float wk[kBatch], x[kRowGroup][kBatch];
#pragma unroll
        for (int u = 0; u < kBatch; ++u) {
          const int k = k0 + 32 * u;
          wk[u] = k < d ? to_f32(wg[k]) : 0.f;
#pragma unroll
          for (int q = 0; q < kRowGroup; ++q) x[q][u] = k < d ? to_f32(es[q][k]) : 0.f;
        }
#pragma unroll
        for (int q = 0; q < kRowGroup; ++q)
#pragma unroll
          for (int u = 0; u < kBatch; ++u) ag[q] = fmaf(wk[u], x[q][u], ag[q]);
      }
    }
#pragma unroll
    for (int q = 0; q < kRowGroup; ++q) {
      av[q] = warp_sum(av[q]);
      ag[q] = warp_sum(ag[q]);
    }
    if (lane < gn) {
      float v = av[0], gs = ag[0];
#pragma unroll
      for (int q = 1; q < kRowGroup; ++q)
        if (lane == q) {
          v = av[q];
          gs = ag[q];
        }
      const int row = g0 + lane;
      const long long orow = (long long)s_b[row] * K + s_j[row];
      const float g = gs + (p.e_dense ? 0.f : p.ge[n]);
      const float ev = to_f32(e[s_e[row] + n]);
      const float gate = 1.f / (1.f + expf(-g));
      out[orow * d + n] = from_f32<T>(ev + v * gate);
    }
  }
}

// ge[i] = sum_k W_g[i, k] e[k] over the e half (k < d), one warp per output.
template <typename T>
__global__ void __launch_bounds__(256) gate_bias_kernel(const T* __restrict__ Wg,
                                                        const T* __restrict__ e, int d,
                                                        float* __restrict__ ge) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int i = blockIdx.x * 8 + warp;
  if (i >= d) return;
  const T* w = Wg + (long long)i * 2 * d;
  float s = 0.f;
  for (int k = lane; k < d; k += 32) s = fmaf(to_f32(w[k]), to_f32(e[k]), s);
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xFFFFFFFFu, s, off);
  if (lane == 0) ge[i] = s;
}

// One CTA per position (b, j): n_out[b], and rows j >= n_b of the zero / copy targets.
template <typename T>
__global__ void __launch_bounds__(256) fill_rows_kernel(int B, int K, int d, RowSource rows,
                                                        int32_t* n_out, T* zero_dst, const T* e,
                                                        int e_dense, T* e_dst) {
  const int b = (int)(blockIdx.x / (unsigned)K), j = (int)(blockIdx.x % (unsigned)K);
  const int nb = rows_of(rows, b, K);
  if (j == 0 && threadIdx.x == 0 && n_out) n_out[b] = nb;
  if (j < nb) return;
  const long long row = ((long long)b * K + j) * d;
  const T* src = e + (e_dense ? row : 0);
  for (int k = threadIdx.x; k < d; k += blockDim.x) {
    if (zero_dst) zero_dst[row + k] = from_f32<T>(0.f);
    if (e_dst) e_dst[row + k] = src[k];
  }
}

template <typename T>
cudaError_t correct_typed(const CorrectArgs& a, cudaStream_t stream) {
  SimtCorrectParams p{a.hD, a.hT, a.Wc, a.beta, a.B, a.K, a.d, a.rows, a.r_out, a.compact_out, a.raw};
  const long long rmax = (long long)a.B * (a.K - 1);
  if (rmax <= 0) return cudaSuccess;
  if (rmax <= kRowsMax) {
    simt_rows_correct_kernel<T><<<(unsigned)((a.d + kRowsWarps - 1) / kRowsWarps), kNT, 0, stream>>>(p);
    return cudaGetLastError();
  }
  dim3 grid((unsigned)((rmax + TM - 1) / TM), (unsigned)((a.d + TN - 1) / TN));
  simt_correct_kernel<T><<<grid, kNT, 0, stream>>>(p);
  return cudaGetLastError();
}

template <typename T>
cudaError_t gate_typed(const GateArgs& a, cudaStream_t stream) {
  SimtGateParams p{a.e, a.e_dense, a.r, a.r_compact, a.Wv, a.Wg, a.ge, a.B, a.K, a.d, a.rows, a.e_out};
  const long long rmax = (long long)a.B * (a.K - 1);
  if (rmax <= 0) return cudaSuccess;
  if (rmax <= kRowsMax) {
    simt_rows_gate_kernel<T><<<(unsigned)((a.d + kRowsWarps - 1) / kRowsWarps), kNT, 0, stream>>>(p);
    return cudaGetLastError();
  }
  dim3 grid((unsigned)((rmax + TM - 1) / TM), (unsigned)((a.d + TN - 1) / TN));
  simt_gate_kernel<T><<<grid, kNT, 0, stream>>>(p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_correct_simt(const CorrectArgs& a, retrace_dtype dtype, cudaStream_t stream) {
  return dtype == RETRACE_BF16 ? correct_typed<__nv_bfloat16>(a, stream) : correct_typed<float>(a, stream);
}

cudaError_t launch_gate_simt(const GateArgs& a, retrace_dtype dtype, cudaStream_t stream) {
  return dtype == RETRACE_BF16 ? gate_typed<__nv_bfloat16>(a, stream) : gate_typed<float>(a, stream);
}

cudaError_t launch_gate_bias(const void* Wg, const void* e, int d, float* ge, retrace_dtype dtype,
                             cudaStream_t stream) {
  const unsigned grid = (unsigned)((d + 7) / 8);
  if (dtype == RETRACE_BF16)
    gate_bias_kernel<__nv_bfloat16><<<grid, 256, 0, stream>>>(
        reinterpret_cast<const __nv_bfloat16*>(Wg), reinterpret_cast<const __nv_bfloat16*>(e), d, ge);
  else
    gate_bias_kernel<float><<<grid, 256, 0, stream>>>(reinterpret_cast<const float*>(Wg),
                                                      reinterpret_cast<const float*>(e), d, ge);
  return cudaGetLastError();
}

cudaError_t launch_fill_rows(int B, int K, int d, RowSource rows, int32_t* n_out, void* zero_dst,
                             const void* e, int e_dense, void* e_dst, retrace_dtype dtype,
                             cudaStream_t stream) {
  if (B <= 0 || K <= 0) return cudaSuccess;
  dim3 grid((unsigned)((long long)B * K));
  if (dtype == RETRACE_BF16)
    fill_rows_kernel<__nv_bfloat16><<<grid, 256, 0, stream>>>(
        B, K, d, rows, n_out, reinterpret_cast<__nv_bfloat16*>(zero_dst),
        reinterpret_cast<const __nv_bfloat16*>(e), e_dense, reinterpret_cast<__nv_bfloat16*>(e_dst));
  else
    fill_rows_kernel<float><<<grid, 256, 0, stream>>>(B, K, d, rows, n_out,
                                                      reinterpret_cast<float*>(zero_dst),
                                                      reinterpret_cast<const float*>(e), e_dense,
                                                      reinterpret_cast<float*>(e_dst));
  return cudaGetLastError();
}

}  // namespace retrace
