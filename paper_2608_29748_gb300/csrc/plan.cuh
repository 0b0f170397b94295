// Conditioned-row plan, computed on the device by every conditioning CTA.
//
// Sequence b contributes n_b = max(0, K-1-A_b) rows (Eq. 4 range; Algorithm 1
// resets the carry when A_b >= K-1).  The R = sum_b n_b rows are numbered
// contiguously in sequence order (exclusive prefix sum of n_b).  Each CTA owns
// a tile of TILE_M consecutive row numbers and needs, for every row of its
// tile, the sequence b, the position j < n_b and n_b itself.  The scan is
// cheap (B integers) and is redone per CTA, so no separate planning kernel or
// host round trip sits between verification and the projections.
#pragma once

#include "common.cuh"
#include "internal.h"

namespace retrace {

__device__ __forceinline__ int rows_of(const RowSource& rs, int b, int K) {
  const int c = rs.counts[b];
  if (rs.n_from_accept) {
    const int A = c < 0 ? 0 : (c > K ? K : c);
    const int n = K - 1 - A;
    return n > 0 ? n : 0;
  }
  const int cap = K - 1 > 0 ? K - 1 : 0;
  return c < 0 ? 0 : (c > cap ? cap : c);
}

// Fills s_b/s_j/s_nb for rows [m0, m0 + TILE_M) (s_b = -1 past the last row)
// and returns R.  s_scan needs NT/32 + 1 ints.  Must be called by all NT
// threads of the CTA.
template <int NT, int TILE_M>
__device__ int plan_tile(const RowSource& rs, int B, int K, long long m0, int* s_b, int* s_j,
                         int* s_nb, int* s_scan) {
  constexpr int NW = NT / 32;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  for (int q = tid; q < TILE_M; q += NT) {
    s_b[q] = -1;
    s_j[q] = 0;
    s_nb[q] = 0;
  }
  __syncthreads();
  long long running = 0;
  for (int base = 0; base < B; base += NT) {
    const int b = base + tid;
    const int nb = (b < B) ? rows_of(rs, b, K) : 0;
    int x = nb;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int y = __shfl_up_sync(0xFFFFFFFFu, x, off);
      if (lane >= off) x += y;
    }
    if (lane == 31) s_scan[warp] = x;
    __syncthreads();
    if (warp == 0) {
      int w = (lane < NW) ? s_scan[lane] : 0;
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const int y = __shfl_up_sync(0xFFFFFFFFu, w, off);
        if (lane >= off) w += y;
      }
      if (lane < NW) s_scan[lane] = w;  // inclusive warp totals
      if (lane == NW - 1) s_scan[NW] = w;
    }
    __syncthreads();
    const int incl = x + (warp > 0 ? s_scan[warp - 1] : 0);
    const long long off = running + (incl - nb);
    const long long lo = off > m0 ? off : m0;
    const long long hi = (off + nb) < (m0 + TILE_M) ? (off + nb) : (m0 + TILE_M);
    for (long long g = lo; g < hi; ++g) {
      const int q = (int)(g - m0);
      s_b[q] = b;
      s_j[q] = (int)(g - off);
      s_nb[q] = nb;
    }
    running += s_scan[NW];
    __syncthreads();
  }
  return (int)running;
}

}  // namespace retrace
