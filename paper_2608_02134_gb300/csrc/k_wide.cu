// Wide selection: the batched responsibility solver (Sec. 3.3, Eq. (4);
// appendix Eq. (cond-responsibility) and its totality rule) with every round
// on the whole GPU, for candidate pools above GMC_MAX_POOL and visual counts
// above GMC_MAX_N: the long-prefix path (b = 512, pool 4b = 2048, N = 15,876;
// Table "Shared GMC configuration", long-prefix row), whose gains the paper
// evaluates in chunks over the whole M x N client matrix.
//
// Round t (support S_t, coverage b_m = max_{j in S_t} Cbar_mj, 0 for S empty):
//   R_mi = [Cbar_mi - b_m]_+,  u_i = sum_m R_mi
//   pool = the min(4b, #{u_i > 0}) unselected tokens of largest u (ties: lower index)
//   rho_m. = softmax over the pool of R_m. / (resp_temp * max_pool R_m. + resp_eps)
//   s_i = sum_m rho_mi R_mi; the top min(b, |pool|, K - |S|) pool tokens by s
//   enter S (ties: lower index); an empty pool fills the budget in ascending
//   index order.
// Four kernels per round:
//   k_w_pool    one block per image: the pool of the current gains (the
//               histogram selection of select_common.cuh, gains read from
//               global memory);
//   k_w_rho     warp per client row: the row's responsibilities over the pool,
//               summed into the scores in 64-bit fixed point.  The dense first
//               round gathers the row at the pool tokens into shared memory;
//               later rounds walk the row's survivor list three times (max,
//               normaliser, scores: the temperature depends on the row's max);
//   k_w_batch   one block per image: a bitonic sort of the pool by (score
//               desc, token asc) gives the batch;
//   k_w_filter  warp per client row: the new coverage b_m, the row's
//               survivors {i : Cbar_mi > b_m} compacted in place (values over
//               Cbar, tokens in scol), the next round's gains summed per block
//               in shared memory and added with one 64-bit atomic per column.
// Entries with Cbar_mi <= b_m have zero residual for the rest of the solve, so
// dropping them is exact.  Every sum is an integer (fixed point), so the
// result does not depend on the order blocks run in.  ceil(K / b) rounds are
// launched; a round whose pool is empty, or that starts with the budget met,
// does nothing.  k_w_final then fills the budget in ascending order if needed,
// writes the ascending support and the diagnostics.
#include <algorithm>

#include "common.cuh"
#include "kernels.cuh"
#include "select_common.cuh"

namespace gmc {

namespace {
constexpr int WROWS = 8;      // warps (client rows) per responsibility block
constexpr int FROWS = 16;     // warps per filter block (one block per SM: the next gains of
                              // N tokens take 8 N bytes of shared memory)
constexpr int WP_THREADS = 1024;
constexpr int W_BCAP = 4096;  // boundary-bucket gains the pool kernel stages in shared memory

// Rows of image b: grounded [0, MG), appearance [MG, MG + MV), spatial after;
// 0 rows for an image whose text offsets are invalid.
__device__ __forceinline__ int wide_rows(const WideGeom& g, int b, int* MG) {
  if (g.uniform) {
    *MG = g.Mstride;
    return g.Mstride;
  }
  const TextGeom tg = text_geom(g.toff, b, g.B, g.Tmax, nullptr);
  if (tg.T == 0) {
    *MG = 0;
    return 0;
  }
  *MG = g.HV * tg.T;
  return *MG + g.MV + g.L2;
}

__device__ __forceinline__ int bank_of(int m, int MG, int MV) {
  return m < MG ? 0 : (m < MG + MV ? 1 : 2);
}

// gains read and written by round rnd: round 0 reads the column sums u0
__device__ __forceinline__ const long long* gains_in(const WideState& w, const long long* u0,
                                                     int rnd) {
  return rnd == 0 ? u0 : (rnd % 2 == 1 ? w.u1 : w.u2);
}
__device__ __forceinline__ long long* gains_out(const WideState& w, int rnd) {
  return rnd % 2 == 0 ? w.u1 : w.u2;
}
}  // namespace

// ---- pool ------------------------------------------------------------------------
// WIN: pools of at most WCAP / 2 tokens take the window pool (the boundary
// bucket of a round lies at or below the last one), with the gains staged in
// shared memory; the full histogram pool runs in round 0, when the window
// misses, and for larger pools (a separate instance, without the window's
// registers).
template <bool WIN>
__global__ void __launch_bounds__(WP_THREADS, 1) k_w_pool(WideState w, WideGeom g, int P, int rnd,
                                                       const long long* __restrict__ u0,
                                                       const int32_t* __restrict__ order,
                                                       TraceView tv) {
  constexpr bool win = WIN;
  grid_dep_wait();
  extern __shared__ __align__(16) char sm_wp[];
  const int b = blockIdx.x, N = g.N, K = g.K;
  const long long* ucur = gains_in(w, u0, rnd) + (size_t)b * N;
  long long* unext = gains_out(w, rnd) + (size_t)b * N;
  int32_t* info = w.info + b * INFO_W;
  // the scores and next gains of this round start at zero
  for (int k = threadIdx.x; k < P; k += blockDim.x) w.sc[(size_t)b * P + k] = 0;
  for (int j = threadIdx.x; j < N; j += blockDim.x) unext[j] = 0;
  if (rnd == 0) {
    for (int j = threadIdx.x; j < N; j += blockDim.x) w.stamp[(size_t)b * N + j] = 0;
    if (threadIdx.x < 4) w.fv[(size_t)b * 4 + threadIdx.x] = 0;
  }
  int MG;
  const int Mb = wide_rows(g, b, &MG);
  const int S = rnd == 0 ? 0 : info[1], rd = rnd == 0 ? 0 : info[2];
  int hint = rnd == 0 || !win ? -1 : info[5];  // the last round's boundary bucket
  __syncthreads();  // every thread has read info before thread 0 rewrites it
  if (rnd == 0 && threadIdx.x == 0) {
    info[1] = 0;
    info[2] = 0;
  }
  // nothing to do once the budget is met, after a round with an empty pool,
  // or for an invalid image
  if (Mb == 0 || S >= K || rd < rnd) {
    if (threadIdx.x == 0) info[0] = 0;
    return;
  }
  sel::PoolScratch ps;
  char* p = sm_wp;
  ps.hist = reinterpret_cast<int*>(p);       p += sizeof(int) * sel::HBINS;
  ps.bnd = reinterpret_cast<int*>(p);        p += sizeof(int) * (size_t)N;
  ps.wsum = reinterpret_cast<int*>(p);       p += sizeof(int) * 32;
  ps.scal = reinterpret_cast<int*>(p);       p += sizeof(int) * 8;
  ps.coarse = reinterpret_cast<int*>(p);     p += sizeof(int) * sel::CBINS;
  int* pool = reinterpret_cast<int*>(p);     p += sizeof(int) * (size_t)P;
  ps.key = reinterpret_cast<short*>(p);      p += sizeof(short) * (size_t)N;
  ps.pk = reinterpret_cast<unsigned char*>(p); p += (size_t)N;
  unsigned char* selz = reinterpret_cast<unsigned char*>(p); p += (size_t)N;
  p = reinterpret_cast<char*>((reinterpret_cast<uintptr_t>(p) + 15) & ~static_cast<uintptr_t>(15));
  ps.bval = reinterpret_cast<long long*>(p);  // the boundary bucket's gains
  ps.bcap = min(N, W_BCAP);
  p += sizeof(long long) * (size_t)ps.bcap;
  ps.sortbuf = reinterpret_cast<int*>(p);     // and their order
  ps.scap = W_BCAP;
  p += sizeof(int) * (size_t)W_BCAP;
  sel::WindowScratch ws{};
  long long* ug = nullptr;  // win: the gains, staged for the pool's passes
  if (win) {
    p = reinterpret_cast<char*>((reinterpret_cast<uintptr_t>(p) + 15) & ~static_cast<uintptr_t>(15));
    ug = reinterpret_cast<long long*>(p);     p += sizeof(long long) * (size_t)N;
    ws.cu = reinterpret_cast<long long*>(p);  p += sizeof(long long) * sel::WCAP;
    ws.cj = reinterpret_cast<int*>(p);        p += sizeof(int) * sel::WCAP;
    ws.win = reinterpret_cast<int*>(p);
    for (int q = threadIdx.x; q < sel::WBINS + 4; q += blockDim.x) ws.win[q] = 0;
  }
  for (int j = threadIdx.x; j < N; j += blockDim.x) {
    selz[j] = 0;
    if (tv.base) tv.gains(b, rd, N)[j] = ucur[j];
    if (win && hint < 0) ug[j] = ucur[j];  // else the window pool's first pass stages them
  }
  for (int h = threadIdx.x; h < sel::HBINS; h += blockDim.x) ps.hist[h] = 0;
  if (threadIdx.x < sel::CBINS) ps.coarse[threadIdx.x] = 0;
  __syncthreads();
  for (int q = threadIdx.x; q < S; q += blockDim.x) selz[order[(size_t)b * K + q]] = 1;
  __syncthreads();
  int Pt = -1;
  if constexpr (WIN)
    Pt = sel::select_pool_window([&](int j) { return ucur[j]; }, ug, selz, N, P, ws, pool, nullptr,
                                 &hint);
  if (Pt < 0) Pt = sel::select_pool<true>(win ? ug : ucur, selz, N, P, ps, pool, nullptr, nullptr, &hint);
  for (int k = threadIdx.x; k < P; k += blockDim.x) w.pool[(size_t)b * P + k] = k < Pt ? pool[k] : -1;
  if (threadIdx.x == 0) {
    info[0] = Pt;
    info[3] = S;
    info[4] = rd;
    info[5] = hint;
  }
  if (tv.base && Pt > 0) {
    int32_t* tp = tv.at<int32_t>(b, tv.off_pool) + (size_t)rd * tv.pool_size;
    for (int k = threadIdx.x; k < tv.pool_size; k += blockDim.x) tp[k] = k < Pt ? pool[k] : -1;
  }
}

// ---- responsibilities ----------------------------------------------------------------
// DENSE: the first round (b = 0, rows are the dense client rows); otherwise
// rows are survivor lists with coverage bcov.
template <bool DENSE>
__global__ void __launch_bounds__(32 * WROWS) k_w_rho(WideState w, WideGeom g, int P,
                                                      const float* __restrict__ C,
                                                      const uint16_t* __restrict__ scol,
                                                      float resp_temp, float resp_eps, int fx_exp,
                                                      const int32_t* fexp) {
  grid_dep_wait();
  extern __shared__ __align__(16) char sm_wr[];
  const int b = blockIdx.y, N = g.N;
  const int Pt = w.info[b * INFO_W];
  if (Pt == 0) return;
  int MG;
  const int Mb = wide_rows(g, b, &MG);
  const int m0 = blockIdx.x * WROWS;
  if (m0 >= Mb) return;
  const float fxs = ldexpf(1.f, fexp ? fexp[b] : fx_exp);
  long long* sblk = reinterpret_cast<long long*>(sm_wr);  // [P]
  char* p = sm_wr + sizeof(long long) * (size_t)P;
  const int32_t* gpool = w.pool + (size_t)b * P;
  for (int k = threadIdx.x; k < P; k += blockDim.x) sblk[k] = 0;
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, m = m0 + wid;
  if (DENSE) {
    float* Rw = reinterpret_cast<float*>(p) + (size_t)wid * P;  // this warp's row at the pool
    __syncthreads();
    if (m < Mb) {
      const float* row = C + ((size_t)b * g.Mstride + m) * N;
      float rmax = 0.f;
      int nf = 0;
      for (int k = lane; k < Pt; k += 32) {
        const float R = row[gpool[k]];  // b = 0: the residual is the client value
        Rw[k] = R;
        if (R > 0.f) {
          rmax = fmaxf(rmax, R);
          ++nf;
        }
      }
      rmax = warp_max(rmax);
      nf = warp_sum_int(nf);
      if (nf > 0) {
        // softmax of R / tau shifted by its largest logit rmax / tau
        const float tau = resp_temp * rmax + resp_eps;
        const float e0 = expf(-rmax / tau);  // a pool token with R = 0
        float z = 0.f;
        for (int k = lane; k < Pt; k += 32)
          if (Rw[k] > 0.f) z += expf((Rw[k] - rmax) / tau);
        z = warp_sum(z) + (float)(Pt - nf) * e0;
        const float invz = 1.f / z;
        for (int k = lane; k < Pt; k += 32) {
          const float R = Rw[k];
          if (R > 0.f)
            atomicAdd((unsigned long long*)&sblk[k],
                      (unsigned long long)to_fix(expf((R - rmax) / tau) * invz * R, fxs));
        }
      }
    }
  } else {
    short* pslot = reinterpret_cast<short*>(p);  // [N] pool slot of every token or -1
    for (int j = threadIdx.x; j < N; j += blockDim.x) pslot[j] = -1;
    __syncthreads();
    for (int k = threadIdx.x; k < Pt; k += blockDim.x) pslot[gpool[k]] = (short)k;
    __syncthreads();
    if (m < Mb) {
      const size_t row = (size_t)b * g.Mstride + m;
      const int n = w.cnt[row];
      const float bm = w.bcov[row];
      const float* vals = C + row * N;
      const uint16_t* cols = scol + row * N;
      // pass 1: the largest pool residual and the number of pool entries
      float rmax = 0.f;
      int nf = 0;
      for (int e = lane; e < n; e += 32) {
        const int k = pslot[cols[e]];
        if (k >= 0) {
          rmax = fmaxf(rmax, vals[e] - bm);
          ++nf;
        }
      }
      rmax = warp_max(rmax);
      nf = warp_sum_int(nf);
      if (nf > 0) {
        const float tau = resp_temp * rmax + resp_eps;
        const float e0 = expf(-rmax / tau);  // pool tokens without a survivor here: R = 0
        float z = 0.f;
        for (int e = lane; e < n; e += 32)
          if (pslot[cols[e]] >= 0) z += expf((vals[e] - bm - rmax) / tau);
        z = warp_sum(z) + (float)(Pt - nf) * e0;
        const float invz = 1.f / z;
        for (int e = lane; e < n; e += 32) {
          const int k = pslot[cols[e]];
          if (k >= 0) {
            const float R = vals[e] - bm;
            atomicAdd((unsigned long long*)&sblk[k],
                      (unsigned long long)to_fix(expf((R - rmax) / tau) * invz * R, fxs));
          }
        }
      }
    }
  }
  __syncthreads();
  for (int k = threadIdx.x; k < Pt; k += blockDim.x)
    if (sblk[k]) atomicAdd((unsigned long long*)&w.sc[(size_t)b * P + k], (unsigned long long)sblk[k]);
}

// ---- batch -----------------------------------------------------------------------------
__global__ void __launch_bounds__(WP_THREADS) k_w_batch(WideState w, WideGeom g, int P, int NP,
                                                        int bsz, int32_t* order, TraceView tv) {
  grid_dep_wait();
  extern __shared__ __align__(16) char sm_wb[];
  const int b = blockIdx.x, K = g.K;
  int32_t* info = w.info + b * INFO_W;
  const int Pt = info[0];
  if (Pt == 0) return;
  const int S = info[3], rd = info[4];
  const int nb = min(bsz, min(Pt, K - S));
  long long* ks = reinterpret_cast<long long*>(sm_wb);   // [NP] scores
  int* kj = reinterpret_cast<int*>(ks + NP);             // [NP] tokens
  if (Pt <= sel::WCAP) {
    // a small pool: every slot's exact rank by (score desc, token asc) is its
    // place in the batch (the order the histogram selection and the sort
    // below give)
    for (int k = threadIdx.x; k < Pt; k += blockDim.x) {
      ks[k] = w.sc[(size_t)b * P + k];
      kj[k] = w.pool[(size_t)b * P + k];
    }
    __syncthreads();
    for (int k = threadIdx.x; k < Pt; k += blockDim.x) {
      const long long sk = ks[k];
      const int jk = kj[k];
      int r = 0;
      for (int q = 0; q < Pt; ++q) r += sel::key_before(ks[q], kj[q], sk, jk);
      if (r < nb) {
        w.batch[(size_t)b * P + r] = jk;
        w.stamp[(size_t)b * g.N + jk] = rd + 1;
        order[(size_t)b * K + S + r] = jk;
      }
    }
    if (threadIdx.x == 0) {
      info[1] = S + nb;
      info[2] = rd + 1;
      if (tv.base) tv.at<int32_t>(b, tv.off_round_end)[rd] = S + nb;
    }
    return;
  }
  // The batch is the top nb of the pool by (score desc, token asc): the
  // histogram selection over the pool slots with the tokens as tie-breakers.
  // Scores of zero are no candidates there; if fewer than nb are positive,
  // the bitonic sort below orders the whole pool instead.
  {
    char* p = reinterpret_cast<char*>(kj + NP);
    sel::PoolScratch ps{};
    ps.hist = reinterpret_cast<int*>(p);       p += sizeof(int) * sel::HBINS;
    ps.bnd = reinterpret_cast<int*>(p);        p += sizeof(int) * (size_t)NP;
    ps.wsum = reinterpret_cast<int*>(p);       p += sizeof(int) * 32;
    ps.scal = reinterpret_cast<int*>(p);       p += sizeof(int) * 8;
    ps.coarse = reinterpret_cast<int*>(p);     p += sizeof(int) * sel::CBINS;
    int* top = reinterpret_cast<int*>(p);      p += sizeof(int) * (size_t)NP;
    ps.key = reinterpret_cast<short*>(p);      p += sizeof(short) * (size_t)NP;
    ps.pk = reinterpret_cast<unsigned char*>(p); p += (size_t)NP;
    unsigned char* none = reinterpret_cast<unsigned char*>(p); p += (size_t)NP;
    p = reinterpret_cast<char*>((reinterpret_cast<uintptr_t>(p) + 15) & ~static_cast<uintptr_t>(15));
    ps.sortbuf = reinterpret_cast<int*>(p);  // [NP], NP a power of two
    ps.scap = NP;
    for (int k = threadIdx.x; k < Pt; k += blockDim.x) {
      ks[k] = w.sc[(size_t)b * P + k];
      kj[k] = w.pool[(size_t)b * P + k];
      none[k] = 0;
    }
    for (int h = threadIdx.x; h < sel::HBINS; h += blockDim.x) ps.hist[h] = 0;
    if (threadIdx.x < sel::CBINS) ps.coarse[threadIdx.x] = 0;
    __syncthreads();
    const int got = sel::select_pool<true>(ks, none, Pt, nb, ps, top, nullptr, kj);
    if (got == nb) {  // uniform over the block
      for (int q = threadIdx.x; q < nb; q += blockDim.x) {
        const int j = kj[top[q]];
        w.batch[(size_t)b * P + q] = j;
        w.stamp[(size_t)b * g.N + j] = rd + 1;
        order[(size_t)b * K + S + q] = j;
      }
      if (threadIdx.x == 0) {
        info[1] = S + nb;
        info[2] = rd + 1;
        if (tv.base) tv.at<int32_t>(b, tv.off_round_end)[rd] = S + nb;
      }
      return;
    }
    __syncthreads();
  }
  for (int k = threadIdx.x; k < NP; k += blockDim.x) {
    const bool in = k < Pt;
    ks[k] = in ? w.sc[(size_t)b * P + k] : -1;  // padding sorts after every pool entry
    kj[k] = in ? w.pool[(size_t)b * P + k] : 0x7fffffff;
  }
  __syncthreads();
  // bitonic sort into (score desc, token asc); NP is a power of two
  for (int size = 2; size <= NP; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int t = threadIdx.x; t < NP / 2; t += blockDim.x) {
        const int lo = 2 * t - (t & (stride - 1));  // first index of the pair
        const int hi = lo + stride;
        const bool desc_block = (lo & size) == 0;   // this run sorts in key order
        const long long sa = ks[lo], sb = ks[hi];
        const int ja = kj[lo], jb = kj[hi];
        const bool b_first = sel::key_before(sb, jb, sa, ja);
        if (b_first == desc_block) {
          ks[lo] = sb; ks[hi] = sa;
          kj[lo] = jb; kj[hi] = ja;
        }
      }
      __syncthreads();
    }
  }
  for (int q = threadIdx.x; q < nb; q += blockDim.x) {
    const int j = kj[q];
    w.batch[(size_t)b * P + q] = j;
    w.stamp[(size_t)b * g.N + j] = rd + 1;
    order[(size_t)b * K + S + q] = j;
  }
  if (threadIdx.x == 0) {
    info[1] = S + nb;
    info[2] = rd + 1;
    if (tv.base) tv.at<int32_t>(b, tv.off_round_end)[rd] = S + nb;
  }
}

// ---- coverage update, survivor compaction, next gains ---------------------------------
template <bool DENSE>
__global__ void __launch_bounds__(32 * FROWS) k_w_filter(WideState w, WideGeom g, int P, int rnd,
                                                         float* C, uint16_t* scol, int fx_exp,
                                                         const int32_t* fexp, int rpw,
                                                         TraceView tv) {
  grid_dep_wait();
  extern __shared__ unsigned long long uacc[];  // [N] this block's part of the next gains
  const int b = blockIdx.y, N = g.N;
  const int32_t* info = w.info + b * INFO_W;
  const int Pt = info[0];
  if (Pt == 0) return;
  int MG;
  const int Mb = wide_rows(g, b, &MG);
  const int m0 = blockIdx.x * FROWS * rpw;
  if (m0 >= Mb) return;
  const int S = info[3], rd = info[4];
  const int nb = info[1] - S;  // the batch kernel has run: info[1] = S + nb
  const float fxs = ldexpf(1.f, fexp ? fexp[b] : fx_exp);
  const int32_t* batch = w.batch + (size_t)b * P;
  const int32_t* stamp = w.stamp + (size_t)b * N;
  long long* unext = gains_out(w, rnd) + (size_t)b * N;
  __shared__ long long fb[3];
  if (threadIdx.x < 3) fb[threadIdx.x] = 0;
  for (int j = threadIdx.x; j < N; j += blockDim.x) uacc[j] = 0;
  __syncthreads();
  const int lane = threadIdx.x & 31;
  const unsigned lt = sel::lanemask_lt();
  for (int ir = 0; ir < rpw; ++ir) {
    const int m = m0 + (threadIdx.x >> 5) + FROWS * ir;
    if (m >= Mb) break;
    const size_t row = (size_t)b * g.Mstride + m;
    float* vals = C + row * N;
    uint16_t* cols = scol + row * N;
    int wr = 0;
    float bnew;
    if (DENSE) {
      bnew = 0.f;
      for (int t = lane; t < nb; t += 32) bnew = fmaxf(bnew, vals[batch[t]]);
      bnew = warp_max(bnew);
      const long long fb_new = to_fix(bnew, fxs);
      float rowmax = 0.f;
      if ((N & 3) == 0) {
        // 8 x 16 bytes per lane in flight; all loads of a step issued before
        // any survivor is written back in place (survivors land below the
        // step's end).  Lane l's float4 holds tokens 4 k4 .. 4 k4 + 3, so the
        // survivors are written lane by lane: ascending token order.
        const float4* row4 = reinterpret_cast<const float4*>(vals);
        const int n4 = N >> 2;
        for (int b4 = 0; b4 < n4; b4 += 32 * 8) {
          float4 buf[8];
#pragma unroll
          for (int u = 0; u < 8; ++u) {
            const int k4 = b4 + u * 32 + lane;
            buf[u] = k4 < n4 ? row4[k4] : make_float4(0.f, 0.f, 0.f, 0.f);
          }
          __syncwarp();
#pragma unroll
          for (int u = 0; u < 8; ++u) {
            const int k4 = b4 + u * 32 + lane;
            const float c4[4] = {buf[u].x, buf[u].y, buf[u].z, buf[u].w};
            int pre = 0, tot = 0;
#pragma unroll
            for (int e2 = 0; e2 < 4; ++e2) {
              rowmax = fmaxf(rowmax, c4[e2]);
              const unsigned bal = __ballot_sync(FULL, k4 < n4 && c4[e2] > bnew);
              pre += __popc(bal & lt);
              tot += __popc(bal);
            }
            int pos = wr + pre;
            if (k4 < n4) {
#pragma unroll
              for (int e2 = 0; e2 < 4; ++e2)
                if (c4[e2] > bnew) {
                  const int k = 4 * k4 + e2;
                  vals[pos] = c4[e2];
                  cols[pos] = (uint16_t)k;
                  atomicAdd(&uacc[k], (unsigned long long)(to_fix(c4[e2], fxs) - fb_new));
                  ++pos;
                }
            }
            wr += tot;
          }
          __syncwarp();
        }
      } else
      // 8 loads per lane in flight; all loads of a step issued before any
      // survivor is written back in place (survivors land below the step's end)
      for (int base = 0; base < N; base += 32 * 8) {
        float c[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const int k = base + u * 32 + lane;
          c[u] = k < N ? vals[k] : 0.f;
        }
        __syncwarp();
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const int k = base + u * 32 + lane;
          rowmax = fmaxf(rowmax, c[u]);
          const bool keep = k < N && c[u] > bnew;
          const unsigned bal = __ballot_sync(FULL, keep);
          if (keep) {
            const int pos = wr + __popc(bal & lt);
            vals[pos] = c[u];
            cols[pos] = (uint16_t)k;
            atomicAdd(&uacc[k], (unsigned long long)(to_fix(c[u], fxs) - fb_new));
          }
          wr += __popc(bal);
        }
      }
      rowmax = warp_max(rowmax);
      if (lane == 0) {
        atomicAdd((unsigned long long*)&fb[bank_of(m, MG, g.MV)],
                  (unsigned long long)to_fix(rowmax, fxs));
        if (tv.base) atomicAdd(tv.cover(b, rd), (unsigned long long)fb_new);
      }
    } else {
      const int n = w.cnt[row];
      bnew = w.bcov[row];
      for (int e = lane; e < n; e += 32)
        if (stamp[cols[e]] == rd + 1) bnew = fmaxf(bnew, vals[e]);
      bnew = warp_max(bnew);
      const long long fb_new = to_fix(bnew, fxs);
      constexpr int FU = 4;  // chunks of 32 entries loaded before any is written back
      for (int e00 = 0; e00 < n; e00 += 32 * FU) {
        float cc[FU];
        int jj[FU];
#pragma unroll
        for (int u = 0; u < FU; ++u) {
          const int e = e00 + 32 * u + lane;
          cc[u] = 0.f;
          jj[u] = 0;
          if (e < n) {
            cc[u] = vals[e];
            jj[u] = cols[e];
          }
        }
        __syncwarp();
#pragma unroll
        for (int u = 0; u < FU; ++u) {
          const bool keep = e00 + 32 * u + lane < n && cc[u] > bnew;
          const unsigned bal = __ballot_sync(FULL, keep);
          if (keep) {
            const int pos = wr + __popc(bal & lt);
            vals[pos] = cc[u];
            cols[pos] = (uint16_t)jj[u];
            atomicAdd(&uacc[jj[u]], (unsigned long long)(to_fix(cc[u], fxs) - fb_new));
          }
          wr += __popc(bal);
        }
      }
      if (lane == 0 && tv.base) atomicAdd(tv.cover(b, rd), (unsigned long long)fb_new);
    }
    if (lane == 0) {
      w.bcov[row] = bnew;
      w.cnt[row] = wr;
    }
  }
  __syncthreads();
  if (DENSE && threadIdx.x < 3 && fb[threadIdx.x])
    atomicAdd((unsigned long long*)&w.fv[(size_t)b * 4 + threadIdx.x], (unsigned long long)fb[threadIdx.x]);
  unsigned long long* ub = reinterpret_cast<unsigned long long*>(unext);
  for (int j = threadIdx.x; j < N; j += blockDim.x)
    if (uacc[j]) atomicAdd(&ub[j], uacc[j]);
}

// ---- fill, ascending support, diagnostics ------------------------------------------------
__global__ void __launch_bounds__(WP_THREADS) k_w_final(WideState w, WideGeom g, int fx_exp,
                                                        const int32_t* fexp, int32_t* order,
                                                        int32_t* support, int32_t* slot,
                                                        int32_t* out_idx, uint32_t* status,
                                                        TraceView tv) {
  grid_dep_wait();
  extern __shared__ unsigned char selz[];  // [N]
  __shared__ int wsum[32];
  __shared__ long long fb[3];
  const int b = blockIdx.x, N = g.N, K = g.K;
  int MG;
  const int Mb = wide_rows(g, b, &MG);
  if (Mb == 0) return;
  const int32_t* info = w.info + b * INFO_W;
  const int S = info[1], rd = info[2];
  for (int j = threadIdx.x; j < N; j += blockDim.x) selz[j] = 0;
  if (threadIdx.x < 3) fb[threadIdx.x] = 0;
  __syncthreads();
  for (int q = threadIdx.x; q < S; q += blockDim.x) selz[order[(size_t)b * K + q]] = 1;
  __syncthreads();
  // contiguous tokens per thread for the ordered scans below
  const int per = (N + blockDim.x - 1) / blockDim.x;
  const int j0 = min(N, (int)threadIdx.x * per), j1 = min(N, j0 + per);
  const int filled = S < K ? K - S : 0;
  if (filled > 0) {  // zero-gain fill: the first K - S unselected tokens, ascending
    int c = 0;
    for (int j = j0; j < j1; ++j) c += selz[j] ? 0 : 1;
    int pos = sel::block_exclusive_scan(c, wsum, nullptr);
    for (int j = j0; j < j1; ++j) {
      if (selz[j]) continue;
      if (pos < filled) {
        order[(size_t)b * K + S + pos] = j;
        selz[j] = 1;
      }
      ++pos;
    }
    __syncthreads();
  }
  {  // the support in ascending token order
    int c = 0;
    for (int j = j0; j < j1; ++j) c += selz[j] ? 1 : 0;
    int cnt = 0;
    int pos = sel::block_exclusive_scan(c, wsum, &cnt);
    for (int j = j0; j < j1; ++j) {
      const bool on = selz[j] != 0;
      slot[(size_t)b * N + j] = on ? pos : -1;
      if (on && pos < K) {
        support[(size_t)b * K + pos] = j;
        if (out_idx) out_idx[(size_t)b * K + pos] = j;
      }
      pos += on ? 1 : 0;
    }
    if (threadIdx.x == 0 && cnt != K) set_status(status, GMC_STATUS_INTERNAL);
  }
  if (!tv.base) return;
  const int e = fexp ? fexp[b] : fx_exp;
  const float fxs = ldexpf(1.f, e);
  if (rd > 0) {  // F_b(S) from the final coverage of every row (the fill adds nothing)
    long long f[3] = {0, 0, 0};
    for (int m = threadIdx.x; m < Mb; m += blockDim.x)
      f[bank_of(m, MG, g.MV)] += to_fix(w.bcov[(size_t)b * g.Mstride + m], fxs);
    for (int q = 0; q < 3; ++q)
      if (f[q]) atomicAdd((unsigned long long*)&fb[q], (unsigned long long)f[q]);
  }
  __syncthreads();
  const int rounds = rd + (filled > 0 ? 1 : 0);
  if (threadIdx.x == 0) {
    gmc_trace_header* hd = tv.header(b);
    hd->K = K;
    hd->rounds = rounds;
    hd->filled = filled;
    const double inv = ldexp(1.0, -e);
    for (int q = 0; q < 3; ++q) {
      hd->F_S[q] = (float)((double)fb[q] * inv);
      hd->F_V[q] = (float)((double)w.fv[(size_t)b * 4 + q] * inv);
    }
  }
  int32_t* to = tv.at<int32_t>(b, tv.off_order);
  for (int q = threadIdx.x; q < K; q += blockDim.x) to[q] = order[(size_t)b * K + q];
  int32_t* te = tv.at<int32_t>(b, tv.off_round_end);
  for (int q = rd + threadIdx.x; q < tv.rounds_max; q += blockDim.x) te[q] = K;
  int32_t* tp = tv.at<int32_t>(b, tv.off_pool);
  for (size_t q = (size_t)rd * tv.pool_size + threadIdx.x; q < (size_t)tv.rounds_max * tv.pool_size;
       q += blockDim.x)
    tp[q] = -1;
}

// ---------------------------------------------------------------------------------------
int wide_rounds(int K, const gmc_params& p) { return (K + p.batch_b - 1) / p.batch_b; }

cudaError_t launch_wide_select(const WideState& w, const WideGeom& g, const gmc_params& p,
                               int fx_exp, const int32_t* fexp, float* C, uint16_t* scol,
                               const long long* u0, int32_t* order, int32_t* support,
                               int32_t* slot, int32_t* out_idx, uint32_t* status,
                               const TraceView& tv, cudaStream_t st) {
  static int sms = 0;
  cudaError_t e;
  if (sms == 0) {
    int dev = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
      return e;
  }
  const int P = p.pool_mult * p.batch_b, N = g.N;
  int NP = 1;
  while (NP < P) NP <<= 1;
  const size_t psm = sizeof(int) * (sel::HBINS + (size_t)N + 32 + 8 + sel::CBINS + P) +
                     sizeof(short) * (size_t)N + 2 * (size_t)N + 16 +
                     sizeof(long long) * (size_t)std::min(N, W_BCAP) +
                     sizeof(int) * (size_t)W_BCAP + 64;
  const size_t rsm_dense = sizeof(long long) * (size_t)P + sizeof(float) * (size_t)WROWS * P;
  const size_t rsm_sparse = sizeof(long long) * (size_t)P + sizeof(short) * (size_t)N;
  const size_t bsm = (sizeof(long long) + sizeof(int)) * (size_t)NP +
                     sizeof(int) * (sel::HBINS + 2 * (size_t)NP + 32 + 8 + sel::CBINS) +
                     sizeof(short) * (size_t)NP + 2 * (size_t)NP + sizeof(int) * (size_t)NP + 80;
  const size_t fsm = sizeof(unsigned long long) * (size_t)N;
  // the window pool's extra shared memory: the staged gains and its scratch
  const size_t wsm = 16 + sizeof(long long) * ((size_t)N + sel::WCAP) + sizeof(int) * sel::WCAP +
                     sizeof(int) * (sel::WBINS + 4);
  const int win = P <= sel::WCAP / 2 && psm + wsm <= 227 * 1024 ? 1 : 0;
  const size_t psm_w = psm + (win ? wsm : 0);
  const void* kpool = win ? (const void*)k_w_pool<true> : (const void*)k_w_pool<false>;
  if ((e = set_smem_limit(kpool, psm_w)) != cudaSuccess) return e;
  if ((e = set_smem_limit((const void*)k_w_rho<true>, rsm_dense)) != cudaSuccess) return e;
  if ((e = set_smem_limit((const void*)k_w_rho<false>, rsm_sparse)) != cudaSuccess) return e;
  if ((e = set_smem_limit((const void*)k_w_batch, bsm)) != cudaSuccess) return e;
  if ((e = set_smem_limit((const void*)k_w_filter<true>, fsm)) != cudaSuccess) return e;
  if ((e = set_smem_limit((const void*)k_w_filter<false>, fsm)) != cudaSuccess) return e;
  // filters: one row per warp while the blocks fit on the GPU about twice, four
  // beyond (each block ends with an atomic per column it touched: fewer, longer
  // blocks add fewer; 4 measured best on the long-prefix document)
  const long long fblocks = (long long)g.B * ceil_div(g.Mstride, FROWS);
  const int rpw = fblocks > 2LL * sms ? 4 : 1;
  const dim3 rgrid(ceil_div(g.Mstride, WROWS), g.B);
  const dim3 fgrid(ceil_div(g.Mstride, FROWS * rpw), g.B);
  const int R = wide_rounds(g.K, p);
  for (int rnd = 0; rnd < R; ++rnd) {
    if (win)
      launch_k(k_w_pool<true>, g.B, WP_THREADS, psm_w, st, 1, w, g, P, rnd, u0,
               (const int32_t*)order, tv);
    else
      launch_k(k_w_pool<false>, g.B, WP_THREADS, psm_w, st, 1, w, g, P, rnd, u0,
               (const int32_t*)order, tv);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    if (rnd == 0)
      launch_k(k_w_rho<true>, rgrid, 32 * WROWS, rsm_dense, st, 1, w, g, P, (const float*)C,
               (const uint16_t*)scol, p.resp_temp, p.resp_eps, fx_exp, fexp);
    else
      launch_k(k_w_rho<false>, rgrid, 32 * WROWS, rsm_sparse, st, 1, w, g, P, (const float*)C,
               (const uint16_t*)scol, p.resp_temp, p.resp_eps, fx_exp, fexp);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    launch_k(k_w_batch, g.B, WP_THREADS, bsm, st, 1, w, g, P, NP, p.batch_b, order, tv);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    if (rnd == 0)
      launch_k(k_w_filter<true>, fgrid, 32 * FROWS, fsm, st, 1, w, g, P, rnd, C, scol, fx_exp,
               fexp, rpw, tv);
    else
      launch_k(k_w_filter<false>, fgrid, 32 * FROWS, fsm, st, 1, w, g, P, rnd, C, scol, fx_exp,
               fexp, rpw, tv);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  launch_k(k_w_final, g.B, WP_THREADS, (size_t)N, st, 1, w, g, fx_exp, fexp, order, support, slot,
           out_idx, status, tv);
  return cudaGetLastError();
}

}  // namespace gmc
