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
// The next 11 mantissa bits: within one bucket, monotone in the gain.
__device__ __forceinline__ int gain_subbucket(long long u) {
  const unsigned long long top = (unsigned long long)u << __clzll(u);
  return (int)((top >> 47) & 2047);
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
constexpr int CBINS = 64;       // coarse bins: the binary exponent of a gain
struct PoolScratch {
  int* hist;           // [HBINS] fine bins, all zero on entry and on return
  int* coarse;         // [CBINS] coarse bins, all zero on entry and on return
  int* bnd;            // [N]  tokens of the boundary bin, ascending
  short* key;          // [N]  bucket of every token (-1: not a candidate)
  unsigned char* pk;   // [N]  boundary tokens that enter the pool
  int* wsum;           // [32]
  int* scal;           // [8]
  long long* bval;     // optional [bcap]: the boundary bucket's gains, staged when the
                       // gains are in global memory (nullptr: read them in place)
  int bcap;
  int* sortbuf;        // optional [scap], scap a power of two: a boundary bucket of more
                       // than SORT_MIN gains is sorted there instead of ranked
  int scap;
};
constexpr int SORT_MIN = 128;

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
// gain u (fixed point), ties to the lower index.  pool[0..Pt) lists the tokens
// above the boundary bucket (below) by index, then the boundary bucket's
// entering tokens by index; poolslot (optional) receives the slot of every
// pool token.  The slots are a deterministic function of the gains, the same
// in every block that calls this with the same data.  Returns Pt.
//
// Every gain gets an 11-bit bucket (exponent, 5 mantissa bits; monotone in u).
// One pass counts the buckets and their exponents (64 coarse bins, counted
// once per warp and exponent); every warp then finds the boundary bucket
// holding the P-th largest gain from the coarse bins and the 32 fine bins of
// one exponent.  Warp w owns 32-token chunks [w * nc, (w + 1) * nc) (lane =
// token within a chunk, so every shared access is conflict-free); ballots
// order the tokens above the boundary bucket and those inside it by index,
// and one scan of the per-warp counts places them: no shared counter,
// nothing that depends on thread scheduling.  Tokens inside the boundary
// bucket are ranked exactly by (u desc, index asc).
// ids (optional): ties are broken by the lower ids[j] instead of the lower j
// (the batch kernel ranks pool slots by (score desc, token asc)).  REFINE
// (the wide solver's long prefixes) splits a large boundary bucket once more
// (below); the standard solvers leave it out, it costs them registers.
// Every thread of the block must call it; blockDim is a multiple of 32.
// bstar_out (optional): the boundary bucket, or -1 when every candidate entered.
template <bool REFINE = false>
__device__ inline int select_pool(const long long* u, const unsigned char* sel, int N, int P,
                                  PoolScratch w, int* pool, short* poolslot,
                                  const int* ids = nullptr, int* bstar_out = nullptr) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = blockDim.x >> 5;
  const int nc = (N + 32 * nw - 1) / (32 * nw);  // chunks per warp
  const unsigned lt = lanemask_lt();
  // 1. bucket of every candidate (-1: selected or zero gain), histograms; the
  //    gains of four chunks are loaded before any of their atomics
  for (int c0 = 0; c0 < nc; c0 += 4) {
    long long vv[4];
    bool cand[4];
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      const int j = (wid * nc + c0 + t) * 32 + lane;
      const bool in = c0 + t < nc && j < N;
      vv[t] = in ? u[j] : 0;
      cand[t] = in && !sel[j];
    }
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      if (c0 + t >= nc) break;  // uniform over the warp
      const int j = (wid * nc + c0 + t) * 32 + lane;
      int kb = -1;
      if (j < N) {
        if (cand[t] && vv[t] > 0) {
          kb = gain_bucket(vv[t]);
          atomicAdd(&w.hist[kb], 1);
        }
        w.key[j] = (short)kb;
      }
      // exponents: one atomic per warp and distinct exponent
      const int e = kb >= 0 ? kb >> 5 : -1;
      const unsigned same = __match_any_sync(FULL, e);
      if (e >= 0 && (same & lt) == 0) atomicAdd(&w.coarse[e], __popc(same));
    }
  }
  __syncthreads();
  // 2. boundary bucket, found by every warp alike: coarse bins from the top,
  //    then the fine bins of the boundary exponent
  int bstar, above, Pt;
  {
    const int hi = CBINS - 1 - 2 * lane;  // this lane's two coarse bins: hi, hi - 1
    const int c0 = w.coarse[hi], c1 = w.coarse[hi - 1];
    int incl = c0 + c1;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(FULL, incl, o);
      if (lane >= o) incl += y;
    }
    const int npos = __shfl_sync(FULL, incl, 31);
    if (npos <= P) {
      bstar = -1;    // every candidate is in the pool
      above = npos;  // tokens above the boundary bucket
      Pt = npos;
    } else {
      const unsigned reach = __ballot_sync(FULL, incl >= P);
      const int L = __ffs(reach) - 1;  // first lane whose prefix reaches P
      int excl = __shfl_sync(FULL, incl - c0 - c1, L);
      const int l0 = __shfl_sync(FULL, c0, L);
      int cb = CBINS - 1 - 2 * L;
      if (excl + l0 < P) {
        excl += l0;
        cb -= 1;
      }
      const int f = cb * 32 + 31 - lane;  // fine bins of that exponent, top first
      const int fc = w.hist[f];
      int fi = fc;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(FULL, fi, o);
        if (lane >= o) fi += y;
      }
      const int Lf = __ffs(__ballot_sync(FULL, excl + fi >= P)) - 1;
      bstar = __shfl_sync(FULL, f, Lf);               // boundary bucket
      above = __shfl_sync(FULL, excl + fi - fc, Lf);  // tokens in higher buckets
      Pt = P;
    }
  }
  // 3. tokens above / inside the boundary bucket, by index: per-warp counts,
  //    one scan, then the placements (tmp: above, bnd: boundary bucket)
  int cu = 0, ca = 0;
  for (int c = 0; c < nc; ++c) {
    const int j = (wid * nc + c) * 32 + lane;
    const int kb = j < N ? w.key[j] : -1;
    cu += __popc(__ballot_sync(FULL, kb > bstar));
    ca += __popc(__ballot_sync(FULL, kb >= 0 && kb == bstar));
  }
  if (lane == 0) w.wsum[wid] = (cu << 16) | ca;  // cu, ca < 2^15: N <= 8192
  __syncthreads();
  // every warp has read the histograms: clear the bins this thread counted
  for (int c = 0; c < nc; ++c) {
    const int j = (wid * nc + c) * 32 + lane;
    const int kb = j < N ? w.key[j] : -1;
    if (kb >= 0) {
      w.hist[kb] = 0;
      w.coarse[kb >> 5] = 0;
    }
  }
  int pre, nb;
  {
    const int x = lane < nw ? w.wsum[lane] : 0;
    int incl = x;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(FULL, incl, o);
      if (lane >= o) incl += y;
    }
    pre = __shfl_sync(FULL, incl - x, wid);  // this warp's offsets (packed)
    nb = __shfl_sync(FULL, incl, 31) & 0xFFFF;
  }
  int pu = pre >> 16, pa = pre & 0xFFFF;
  for (int c = 0; c < nc; ++c) {
    const int j = (wid * nc + c) * 32 + lane;
    const int kb = j < N ? w.key[j] : -1;
    const bool up = kb > bstar, at = kb >= 0 && kb == bstar;
    const unsigned bu = __ballot_sync(FULL, up), ba = __ballot_sync(FULL, at);
    if (up) {
      const int slot = pu + __popc(bu & lt);
      pool[slot] = j;
      if (poolslot) poolslot[j] = (short)slot;
    }
    if (at) w.bnd[pa + __popc(ba & lt)] = j;
    pu += __popc(bu);
    pa += __popc(ba);
  }
  if (bstar >= 0) {
    __syncthreads();
    // 4. the boundary bucket's tokens that enter, ranked exactly by (u desc,
    //    index asc); they take the slots after the tokens above, by index
    int need = Pt - above;
    const bool staged = w.bval && nb <= w.bcap;  // uniform over the block
    if (staged) {
      for (int q = threadIdx.x; q < nb; q += blockDim.x) w.bval[q] = u[w.bnd[q]];
      __syncthreads();
    }
    // A large bucket is sorted by (u desc, id asc) (bitonic, in shared
    // memory) and its first `need` tokens enter.  Otherwise a large bucket
    // (near-equal gains) is split once more by the next 11 mantissa bits: the
    // tokens of higher sub-buckets enter, those of lower ones do not, and only
    // the boundary sub-bucket is ranked exactly.
    // pk[q]: 1 enters, 0 does not, 2 undecided (ranked below).
    const bool sorted = w.sortbuf && nb > SORT_MIN && nb <= w.scap;  // uniform over the block
    const bool refine = REFINE && nb > 512 && !sorted;                        // uniform
    if (sorted) {
      int n2 = 1;
      while (n2 < nb) n2 <<= 1;
      for (int q = threadIdx.x; q < n2; q += blockDim.x) w.sortbuf[q] = q < nb ? q : -1;
      __syncthreads();
      // a before c: c is padding, or (u, id) of a comes first
      auto before = [&](int a, int c) {
        if (a < 0) return false;
        if (c < 0) return true;
        const int ja = w.bnd[a], jc = w.bnd[c];
        return key_before(staged ? w.bval[a] : u[ja], ids ? ids[ja] : ja,
                          staged ? w.bval[c] : u[jc], ids ? ids[jc] : jc);
      };
      for (int k = 2; k <= n2; k <<= 1)
        for (int jj = k >> 1; jj > 0; jj >>= 1) {
          for (int i = threadIdx.x; i < n2; i += blockDim.x) {
            const int ixj = i ^ jj;
            if (ixj > i) {
              const int a = w.sortbuf[i], c = w.sortbuf[ixj];
              const bool af = before(a, c);
              if (((i & k) == 0) != af) {  // out of order for this half's direction
                w.sortbuf[i] = c;
                w.sortbuf[ixj] = a;
              }
            }
          }
          __syncthreads();
        }
      for (int q = threadIdx.x; q < nb; q += blockDim.x) w.pk[q] = 0;
      __syncthreads();
      for (int q = threadIdx.x; q < need; q += blockDim.x) w.pk[w.sortbuf[q]] = 1;
      __syncthreads();
    }
    if (refine) {
      for (int q = threadIdx.x; q < nb; q += blockDim.x)
        atomicAdd(&w.hist[gain_subbucket(staged ? w.bval[q] : u[w.bnd[q]])], 1);
      __syncthreads();
      if (wid == 0) {  // the sub-bucket holding the need-th largest: 64 bins per lane, top first
        int cnt = 0;
        for (int t = 0; t < 64; ++t) cnt += w.hist[2047 - (lane * 64 + t)];
        int incl = cnt;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const int y = __shfl_up_sync(FULL, incl, o);
          if (lane >= o) incl += y;
        }
        const int L = __ffs(__ballot_sync(FULL, incl >= need)) - 1;  // need <= nb: L >= 0
        if (lane == L) {
          int acc = incl - cnt, sb = 2047 - lane * 64;
          for (int t = 0; t < 64; ++t, --sb) {
            const int c = w.hist[sb];
            if (acc + c >= need) break;
            acc += c;
          }
          w.scal[0] = sb;   // boundary sub-bucket
          w.scal[1] = acc;  // tokens in higher sub-buckets
        }
      }
      __syncthreads();
      const int sb = w.scal[0];
      for (int q = threadIdx.x; q < nb; q += blockDim.x) {
        const int sk = gain_subbucket(staged ? w.bval[q] : u[w.bnd[q]]);
        w.pk[q] = sk > sb ? 1 : (sk == sb ? 2 : 0);
      }
      need -= w.scal[1];
      __syncthreads();
    }
    for (int q = threadIdx.x; q < (sorted ? 0 : nb); q += blockDim.x) {
      if (refine && w.pk[q] != 2) continue;
      const int j = w.bnd[q];
      const long long v = staged ? w.bval[q] : u[j];
      const int id = ids ? ids[j] : j;
      int rank = 0;
      for (int q2 = 0; q2 < nb; ++q2) {
        if (refine && w.pk[q2] != 2) continue;  // only the boundary sub-bucket competes
        const int j2 = w.bnd[q2];
        rank += key_before(staged ? w.bval[q2] : u[j2], ids ? ids[j2] : j2, v, id);
      }
      // refine: pk still marks who competes, so the verdict waits in key[q]
      // (the tokens' bucket keys are no longer read)
      if (refine) w.key[q] = (short)(rank < need);
      else w.pk[q] = rank < need;
    }
    __syncthreads();
    if (refine) {  // the verdicts, and the sub-buckets cleared (every thread has read them)
      for (int q = threadIdx.x; q < nb; q += blockDim.x) {
        if (w.pk[q] == 2) w.pk[q] = (unsigned char)w.key[q];
        w.hist[gain_subbucket(staged ? w.bval[q] : u[w.bnd[q]])] = 0;
      }
      __syncthreads();
    }
    // slots in index order: each entering token counts the entering ones
    // before it (a small bucket), or a block scan of the entering flags over
    // contiguous ranges (a large one: its barriers cost less than the counts)
    if (nb <= 256) {
      for (int q = threadIdx.x; q < nb; q += blockDim.x) {
        if (!w.pk[q]) continue;
        int before = 0;
        for (int q2 = 0; q2 < q; ++q2) before += w.pk[q2];
        const int j = w.bnd[q];
        pool[above + before] = j;
        if (poolslot) poolslot[j] = (short)(above + before);
      }
    } else {
      const int per = (nb + (int)blockDim.x - 1) / (int)blockDim.x;
      const int q0 = min(nb, (int)threadIdx.x * per), q1 = min(nb, q0 + per);
      int c = 0;
      for (int q = q0; q < q1; ++q) c += w.pk[q];
      int before = block_exclusive_scan(c, w.wsum, nullptr);
      for (int q = q0; q < q1; ++q) {
        if (!w.pk[q]) continue;
        const int j = w.bnd[q];
        pool[above + before] = j;
        if (poolslot) poolslot[j] = (short)(above + before);
        ++before;
      }
    }
  }
  __syncthreads();
  if (bstar_out) *bstar_out = bstar;
  return Pt;
}

// Pool of a later round from a window of buckets below the previous boundary.
//
// A round takes its batch out of the candidates and can only lower the other
// gains (the coverage b_m grows), so the P-th largest gain of the next round is
// at most the P-th largest of this one: its bucket lies at or below the last
// boundary bucket `hint`.  One pass loads the gains (load(j), stored into u[j]
// for later readers), counts the candidates above a window of WBINS buckets
// that ends WTOP buckets above the hint and histograms the ones inside it;
// every warp finds the boundary bucket from the window alone.  The tokens in
// or above the boundary bucket (at most WCAP) are listed in any order and
// ranked exactly by (u desc, index asc); a pool token's slot is its rank, so
// the pool is the same in every block that calls this with the same gains and
// hint.  Three block barriers; a thread's loads of a pass are all issued before
// its atomics.
//
// Returns Pt and sets *hint to the new boundary bucket (-1 once every
// candidate enters); returns -1 when the boundary is not inside the window or
// more than WCAP tokens reach it (the caller then runs select_pool on u, which
// is complete on return).  With *hint < 0 it returns -1 at once and loads
// nothing.  Every thread gets the same answer.  Every thread of the block must
// call it.
constexpr int WBINS = 128;  // window buckets: 4 per lane of one warp
constexpr int WTOP = 8;     // window buckets above the hint
constexpr int WCAP = 256;   // candidates ranked exactly
constexpr int WU = 4;       // tokens a thread handles per pass step
struct WindowScratch {
  int* win;        // [WBINS + 4] window bins (top bucket first) and 4 counters;
                   // all zero on entry and on return
  long long* cu;   // [WCAP] candidates' gains
  int* cj;         // [WCAP] candidates' tokens
};

template <class Load>
__device__ inline int select_pool_window(Load load, long long* u, const unsigned char* sel, int N,
                                         int P, WindowScratch w, int* pool, short* poolslot,
                                         int* hint) {
  const int lane = threadIdx.x & 31;
  const int h = *hint;
  if (h < 0) return -1;  // uniform: every thread holds the same hint
  const int top = h + WTOP;             // highest window bucket (bin 0)
  int* cnt = w.win + WBINS;             // 0: above the window, 1: positive, 2: listed
  const int step = (int)blockDim.x;
  // 1. gains, window histogram, counts above the window and of positive candidates
  int npos_w = 0, nabove_w = 0;
  for (int j0 = (int)threadIdx.x - lane; j0 < N; j0 += WU * step) {  // warp-uniform
    long long v[WU];
    unsigned char sl[WU];
#pragma unroll
    for (int t = 0; t < WU; ++t) {
      const int j = j0 + t * step + lane;
      v[t] = j < N ? load(j) : 0;
      sl[t] = j < N ? sel[j] : 1;
    }
#pragma unroll
    for (int t = 0; t < WU; ++t) {
      const int j = j0 + t * step + lane;
      if (j < N) u[j] = v[t];
      const int kb = !sl[t] && v[t] > 0 ? gain_bucket(v[t]) : -1;
      const int bin = top - kb;
      if (kb >= 0 && bin >= 0 && bin < WBINS) atomicAdd(&w.win[bin], 1);
      npos_w += __popc(__ballot_sync(FULL, kb >= 0));
      nabove_w += __popc(__ballot_sync(FULL, kb > top));
    }
  }
  if (lane == 0) {
    if (nabove_w) atomicAdd(&cnt[0], nabove_w);
    if (npos_w) atomicAdd(&cnt[1], npos_w);
  }
  __syncthreads();
  // 2. boundary bucket, found by every warp alike
  const int npos = cnt[1], nabove = cnt[0];
  int bstar = -1, ncand = npos, Pt = npos;
  bool miss = false;
  if (npos > P) {
    Pt = P;
    if (nabove >= P) {
      miss = true;  // the boundary is above the window
    } else {
      const int4 c4 = reinterpret_cast<const int4*>(w.win)[lane];  // bins 4 lane .. 4 lane + 3
      const int s4 = c4.x + c4.y + c4.z + c4.w;
      int incl = s4;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(FULL, incl, o);
        if (lane >= o) incl += y;
      }
      const int need = P - nabove;
      const unsigned reach = __ballot_sync(FULL, incl >= need);
      if (!reach) {
        miss = true;  // the boundary is below the window
      } else {
        const int L = __ffs(reach) - 1;
        int acc = __shfl_sync(FULL, incl - s4, L);
        const int b0 = __shfl_sync(FULL, c4.x, L), b1 = __shfl_sync(FULL, c4.y, L);
        const int b2 = __shfl_sync(FULL, c4.z, L), b3 = __shfl_sync(FULL, c4.w, L);
        int t = 0;
        if (acc + b0 < need) {
          acc += b0;
          t = 1;
          if (acc + b1 < need) {
            acc += b1;
            t = 2;
            if (acc + b2 < need) {
              acc += b2;
              t = 3;
            }
          }
        }
        const int bt = t == 0 ? b0 : t == 1 ? b1 : t == 2 ? b2 : b3;
        bstar = top - (4 * L + t);
        ncand = nabove + acc + bt;  // every candidate in or above the boundary bucket
        miss = ncand > WCAP;
      }
    }
  } else {
    miss = npos > WCAP;
  }
  if (miss) {
    __syncthreads();  // every warp has read the bins
    for (int q = threadIdx.x; q < WBINS + 4; q += blockDim.x) w.win[q] = 0;
    __syncthreads();
    return -1;
  }
  // 3. list the candidates in or above the boundary bucket (any order); a
  //    thread reads back only the gains it stored itself
  for (int j0 = (int)threadIdx.x - lane; j0 < N; j0 += WU * step) {
    long long v[WU];
    unsigned want = 0;
#pragma unroll
    for (int t = 0; t < WU; ++t) {
      const int j = j0 + t * step + lane;
      v[t] = j < N ? u[j] : 0;
      if (j < N && !sel[j] && v[t] > 0 && gain_bucket(v[t]) >= bstar) want |= 1u << t;
    }
    unsigned bal[WU];
    int tot = 0;
#pragma unroll
    for (int t = 0; t < WU; ++t) {
      bal[t] = __ballot_sync(FULL, (want >> t) & 1u);
      tot += __popc(bal[t]);
    }
    if (tot) {  // warp-uniform: one atomic per warp and step
      int base = 0;
      if (lane == 0) base = atomicAdd(&cnt[2], tot);
      base = __shfl_sync(FULL, base, 0);
      const unsigned lt = lanemask_lt();
#pragma unroll
      for (int t = 0; t < WU; ++t) {
        if ((want >> t) & 1u) {
          const int at = base + __popc(bal[t] & lt);
          w.cu[at] = v[t];
          w.cj[at] = j0 + t * step + lane;
        }
        base += __popc(bal[t]);
      }
    }
  }
  __syncthreads();
  // 4. rank every candidate among them (4 lanes each); slot = rank
  for (int q = threadIdx.x; q < WBINS + 4; q += blockDim.x) w.win[q] = 0;
  for (int base = ((int)threadIdx.x - lane) >> 2; base < ncand; base += blockDim.x >> 2) {
    const int q = base + (lane >> 2), gl = lane & 3;
    int rank = 0;
    long long v = 0;
    int jq = 0;
    if (q < ncand) {
      v = w.cu[q];
      jq = w.cj[q];
#pragma unroll 4
      for (int q2 = gl; q2 < ncand; q2 += 4) rank += key_before(w.cu[q2], w.cj[q2], v, jq);
    }
    rank += __shfl_xor_sync(FULL, rank, 1);
    rank += __shfl_xor_sync(FULL, rank, 2);
    if (q < ncand && gl == 0 && rank < Pt) {
      pool[rank] = jq;
      if (poolslot) poolslot[jq] = (short)rank;
    }
  }
  __syncthreads();
  *hint = Pt == P ? bstar : -1;
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
