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
  int* hist;  // [HBINS], all zero on entry and on return
  int* bnd;   // [N]
  int* tmp;   // [P]  pool tokens in arrival order
  int* wsum;  // [32]
  int* scal;  // [5]
};

// Warp-aggregated append: every lane with `want` gets a distinct index from
// *counter (order within the warp by lane).  All lanes of the warp call it.
__device__ __forceinline__ int warp_append(bool want, int* counter) {
  const unsigned m = __ballot_sync(FULL, want);
  const int leader = m ? __ffs(m) - 1 : 0;  // lowest appending lane
  int base = 0;
  if (m && (int)(threadIdx.x & 31) == leader) base = atomicAdd(counter, __popc(m));
  base = __shfl_sync(FULL, base, leader);
  return base + __popc(m & lanemask_lt());
}

// Position of x among n distinct ints a[0..n) (the number smaller than x),
// counted by the 8 lanes of an aligned group (mask gm); every group lane gets it.
__device__ __forceinline__ int group_rank_of(const int* a, int n, int x, int gl, unsigned gm) {
  int c = 0;
  for (int k = gl; k < n; k += 8) c += a[k] < x;
  c += __shfl_xor_sync(gm, c, 1);
  c += __shfl_xor_sync(gm, c, 2);
  c += __shfl_xor_sync(gm, c, 4);
  return c;
}

// Pool of one round: the min(P, #{u_i > 0}) tokens with sel[i] == 0 of largest
// gain u (fixed point), ties to the lower index.  A histogram over an
// exponent/mantissa bucket finds the boundary bucket; tokens inside it are
// ranked exactly.  Pool tokens arrive in any order and take the slot of their
// rank by token index, so slots ascend with the token: pool[0..Pt).
// poolslot (optional) receives the slot of every pool token.  Returns Pt.
// Every thread of the block must call it (blockDim a multiple of 32, N
// rounded up to the block is walked by whole warps); the result does not
// depend on thread scheduling.
__device__ inline int select_pool(const long long* u, const unsigned char* sel, int N, int P,
                                  PoolScratch w, int* pool, short* poolslot) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = blockDim.x >> 5;
  if (threadIdx.x < 5) w.scal[threadIdx.x] = 0;
  for (int j = threadIdx.x; j < N; j += blockDim.x) {
    const long long v = u[j];
    if (!sel[j] && v > 0) atomicAdd(&w.hist[gain_bucket(v)], 1);
  }
  __syncthreads();
  {
    // Every thread owns a contiguous range of buckets (zeroed again here); the
    // thread whose range holds the P-th largest candidate finds the boundary
    // bucket inside it.
    const int per = (HBINS + blockDim.x - 1) / blockDim.x;
    const int h0 = min(HBINS, (int)threadIdx.x * per), h1 = min(HBINS, h0 + per);
    int part = 0;
    for (int h = h0; h < h1; ++h) part += w.hist[h];
    int x = part;  // inclusive prefix within the warp
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(FULL, x, o);
      if (lane >= o) x += y;
    }
    if (lane == 31) w.wsum[wid] = x;
    __syncthreads();
    int t = lane < nw ? w.wsum[lane] : 0;  // warp totals, prefix over warps by shuffles
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(FULL, t, o);
      if (lane >= o) t += y;
    }
    const int npos = __shfl_sync(FULL, t, 31);
    const int wbefore = wid > 0 ? __shfl_sync(FULL, t, wid - 1) : 0;
    const int above = npos - (wbefore + x);  // candidates in higher buckets
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
    for (int h = h0; h < h1; ++h) w.hist[h] = 0;
  }
  __syncthreads();
  const int Pt = w.scal[2];
  const int bstar = w.scal[0];
  if (Pt > 0) {
    for (int j0 = wid * 32; j0 < N; j0 += nw * 32) {  // whole warps: aggregated appends
      const int j = j0 + lane;
      int k = -1;
      if (j < N) {
        const long long v = u[j];
        if (!sel[j] && v > 0) k = gain_bucket(v);
      }
      const bool up = k > bstar, at = k >= 0 && k == bstar;
      const int pu = warp_append(up, &w.scal[4]);
      const int pb = warp_append(at, &w.scal[3]);
      if (up) w.tmp[pu] = j;
      if (at) w.bnd[pb] = j;
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
        if (rank < need) w.tmp[w.scal[1] + rank] = j;  // after the tokens above the bucket
      }
    }
    __syncthreads();
    // slot = rank by token index: one 8-lane group per pool token
    const int gl = lane & 7;
    const unsigned gm = 0xFFu << (lane & 24);
    for (int k0 = threadIdx.x >> 3; k0 < Pt; k0 += blockDim.x >> 3) {
      const int j = w.tmp[k0];
      const int slot = group_rank_of(w.tmp, Pt, j, gl, gm);
      if (gl == 0) {
        pool[slot] = j;
        if (poolslot) poolslot[j] = (short)slot;
      }
    }
  }
  __syncthreads();
  return Pt;
}

// Rank of pool slot k among the Pt slots by (score desc, token asc), counted by
// the 8 lanes of an aligned group (mask gm).
__device__ __forceinline__ int group_score_rank(const long long* s, const int* pool, int Pt, int k,
                                                int gl, unsigned gm) {
  const long long sk = s[k];
  const int jk = pool[k];
  int rank = 0;
  for (int q = gl; q < Pt; q += 8) rank += key_before(s[q], pool[q], sk, jk);
  rank += __shfl_xor_sync(gm, rank, 1);
  rank += __shfl_xor_sync(gm, rank, 2);
  rank += __shfl_xor_sync(gm, rank, 4);
  return rank;
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
