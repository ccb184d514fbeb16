// Device pieces shared by the selection kernels (k_select.cu, k_round0.cu):
// the pool choice of Eq. (4) and deterministic block scans.
#pragma once

#include "common.cuh"

namespace gmc {
namespace sel {

constexpr int HBINS = 2048;

__device__ __forceinline__ bool key_before(long long ua, int ja, long long ub, int jb) {
  return ua > ub || (ua == ub && ja < jb);
}

__device__ __forceinline__ unsigned lanemask_lt() {
  unsigned m;
  asm("mov.u32 %0, %%lanemask_lt;" : "=r"(m));
  return m;
}

// Monotone 11-bit bucket of a positive 64-bit gain: exponent and 5 mantissa bits.
__device__ __forceinline__ int gain_bucket(long long u) {
  const int lz = __clzll(u);                                      // 1..63 for 0 < u < 2^63
  const unsigned long long top = (unsigned long long)u << lz;     // leading one at bit 63
  return (63 - lz) * 32 + (int)((top >> 58) & 31);
}

// Block-wide exclusive scan of one int per thread (deterministic).  Every
// thread of the block must call it.
__device__ inline int block_exclusive_scan(int v, int* wsum, int* total) {
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = blockDim.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(FULL, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) wsum[w] = x;
  __syncthreads();
  if (w == 0) {
    int t = lane < nw ? wsum[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(FULL, t, o);
      if (lane >= o) t += y;
    }
    if (lane < nw) wsum[lane] = t;  // inclusive prefix of warp totals
  }
  __syncthreads();
  const int before = (w > 0 ? wsum[w - 1] : 0) + x - v;
  const int tot = wsum[nw - 1];
  __syncthreads();
  if (total) *total = tot;
  return before;
}

// Shared-memory scratch of select_pool.
struct PoolScratch {
  int* hist;              // [HBINS]
  int* bnd;               // [N]
  unsigned char* inpool;  // [N], all zero on entry and on return
  int* wsum;              // [32]
  int* scal;              // [4]
};

// Pool of one round: the min(P, #{u_i > 0}) tokens with sel[i] == 0 of largest
// gain u (fixed point), ties to the lower index.  A histogram over an
// exponent/mantissa bucket finds the boundary bucket; tokens inside it are
// ranked exactly.  Slots are numbered in ascending token order: pool[0..Pt).
// poolslot (optional) receives the slot of every pool token.  Returns Pt.
// Every thread of the block must call it; the result does not depend on
// thread scheduling.
__device__ inline int select_pool(const long long* u, const unsigned char* sel, int N, int P,
                                  PoolScratch w, int* pool, short* poolslot) {
  for (int k = threadIdx.x; k < HBINS; k += blockDim.x) w.hist[k] = 0;
  if (threadIdx.x == 0) w.scal[3] = 0;
  __syncthreads();
  for (int j = threadIdx.x; j < N; j += blockDim.x) {
    const long long v = u[j];
    if (!sel[j] && v > 0) atomicAdd(&w.hist[gain_bucket(v)], 1);
  }
  __syncthreads();
  {
    // Every thread sums a contiguous range of bins; the thread whose range
    // holds the P-th largest candidate finds the boundary bin inside it.
    const int per = (HBINS + blockDim.x - 1) / blockDim.x;
    const int h0 = min(HBINS, (int)threadIdx.x * per), h1 = min(HBINS, h0 + per);
    int part = 0;
    for (int h = h0; h < h1; ++h) part += w.hist[h];
    int npos = 0;
    const int below = block_exclusive_scan(part, w.wsum, &npos);
    const int above = npos - below - part;  // candidates in higher bins
    if (npos <= P) {
      if (threadIdx.x == 0) {
        w.scal[0] = -1;    // every candidate is in the pool
        w.scal[1] = npos;  // count above the boundary bucket
        w.scal[2] = npos;  // pool size
      }
    } else if (above < P && above + part >= P) {
      int cum = above;
      int bstar = h0;
      for (int h = h1 - 1; h >= h0; --h) {
        const int hc = w.hist[h];
        if (cum + hc >= P) { bstar = h; break; }
        cum += hc;
      }
      w.scal[0] = bstar;
      w.scal[1] = cum;
      w.scal[2] = P;
    }
  }
  __syncthreads();
  const int Pt = w.scal[2];
  const int bstar = w.scal[0];
  if (Pt > 0) {
    for (int j = threadIdx.x; j < N; j += blockDim.x) {
      const long long v = u[j];
      if (sel[j] || v <= 0) continue;
      const int k = gain_bucket(v);
      if (k > bstar) w.inpool[j] = 1;
      else if (k == bstar) w.bnd[atomicAdd(&w.scal[3], 1)] = j;
    }
    __syncthreads();
    if (bstar >= 0) {
      const int nb = w.scal[3], need = Pt - w.scal[1];
      for (int q = threadIdx.x; q < nb; q += blockDim.x) {
        const int j = w.bnd[q];
        const long long v = u[j];
        int rank = 0;
        for (int q2 = 0; q2 < nb; ++q2) {
          const int j2 = w.bnd[q2];
          rank += key_before(u[j2], j2, v, j);
        }
        if (rank < need) w.inpool[j] = 1;
      }
    }
    __syncthreads();
    const int per = (N + blockDim.x - 1) / blockDim.x;
    const int j0 = threadIdx.x * per, j1 = min(N, j0 + per);
    int mine = 0;
    for (int j = j0; j < j1; ++j) mine += w.inpool[j];
    int slot = block_exclusive_scan(mine, w.wsum, nullptr);
    for (int j = j0; j < j1; ++j)
      if (w.inpool[j]) {
        pool[slot] = j;
        if (poolslot) poolslot[j] = (short)slot;
        w.inpool[j] = 0;
        ++slot;
      }
  }
  __syncthreads();
  return Pt;
}

// Rank of pool slot k among the Pt slots by (score desc, token asc).
__device__ __forceinline__ int score_rank(const long long* s, const int* pool, int Pt, int k) {
  const long long sk = s[k];
  const int jk = pool[k];
  int rank = 0;
  for (int q = 0; q < Pt; ++q) rank += key_before(s[q], pool[q], sk, jk);
  return rank;
}

}  // namespace sel
}  // namespace gmc
