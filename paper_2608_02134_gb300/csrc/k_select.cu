// Batched responsibility selection (Sec. 3.3, Eq. (4); appendix Eq.
// (cond-responsibility) and its totality rule), one thread-block cluster per image.
//
// Round t with support S_t and coverage b_m = max_{j in S_t} Cbar_mj (0 for S empty):
//   R_mi = [Cbar_mi - b_m]_+,  u_i = sum_m R_mi
//   pool = the min(pool_size, #{u_i > 0}) unselected tokens of largest u (ties: lower index)
//   rho_m. = softmax over the pool of R_m. / (resp_temp * max_pool R_m. + resp_eps)
//   s_i = sum_m rho_mi R_mi; the top min(b, |pool|, K - |S|) pool tokens by s enter S
//   (ties: lower index); an empty pool fills the budget in ascending index order.
//
// Work-efficient residual form.  An entry with Cbar_mi <= b_m has R_mi = 0 now
// and in every later round (b only grows), so it never contributes to a gain,
// a responsibility or a coverage update again.  After the first (dense) round
// each client row keeps only its "survivors" {i : Cbar_mi > b_m}, compacted in
// place, and every later round touches only those.  This is exact, not an
// approximation: the skipped entries are exactly the zero residuals.  (A
// pool member with R_mi = 0 still counts exp(0) = 1 in row m's softmax
// denominator; the kernel adds those terms explicitly.)
//
// Parallel layout.  The CS CTAs of a cluster split the client rows; each CTA
// keeps its rows' coverage b_m and survivor counts in shared memory and the
// survivor lists in global memory (in place over Cbar).  Gains and scores are
// summed in 64-bit fixed point, so the reductions across warps and CTAs
// (shared / distributed-shared-memory atomics) are exact and deterministic.
// Every CTA holds the same selected-set bitmap and derives the same control
// decisions, so all CTAs run the same number of cluster barriers.
#include <cooperative_groups.h>

#include "common.cuh"
#include "kernels.cuh"

namespace cg = cooperative_groups;

namespace gmc {

constexpr int SEL_THREADS = 512;
constexpr int SEL_MAX_CS = 16;

struct SelArgs {
  int B, N, K, Mstride, H, Tmax, L2;
  const int32_t* toff;  // compress path: per-image text lengths; select path: nullptr
  int uniform_rows;     // select path: every image has Mstride rows, all in bank 0
  int P, bsz;
  float resp_temp, resp_eps;
  int fx_exp;
  const int32_t* fexp;  // per-image fixed-point exponents (select path) or nullptr
  float* C;
  uint16_t* scol;
  const long long* u0;
  int32_t* order;
  int32_t* support;
  int32_t* slot;
  int32_t* out_idx;
  uint32_t* status;
  TraceView tv;
};

struct SelSmem {
  long long* u_part;   // [N]   this CTA's partial gains (fixed point)
  long long* u_slice;  // [SL]  reduced gains of this CTA's token slice
  long long* cand_u;   // [CS][P] candidates pushed by every CTA
  int* cand_j;         // [CS][P]
  int* ncand;          // [CS]
  int* pool;           // [P]
  long long* s_acc;    // [P]   cluster-wide scores
  long long* s_loc;    // [P]   this CTA's partial scores
  int* batch;          // [P]
  int* inb;            // [P]   pool slot is in the batch
  short* poolslot;     // [N]   pool slot of a token or -1
  unsigned char* sel;  // [N]   selected flags
  float* bcov;         // [RPC] coverage b_m of this CTA's rows
  int* cnt;            // [RPC] survivor count (-1: row still dense)
  long long* fb;       // [8]   bank sums F_S[3], F_V[3] (fixed point)
  int* scal;           // [8]   S count, Pt, nb, rounds, filled, nloc
};

__host__ __device__ inline size_t sel_smem_bytes(int N, int CS, int P, int RPC, SelSmem* o,
                                                 char* base) {
  size_t off = 0;
  auto take = [&](size_t bytes) {
    size_t at = off;
    off += (bytes + 15) & ~(size_t)15;
    return base ? base + at : nullptr;
  };
  const int SL = (N + CS - 1) / CS;
  char* p;
  p = take(sizeof(long long) * N);      if (o) o->u_part = (long long*)p;
  p = take(sizeof(long long) * SL);     if (o) o->u_slice = (long long*)p;
  p = take(sizeof(long long) * CS * P); if (o) o->cand_u = (long long*)p;
  p = take(sizeof(int) * CS * P);       if (o) o->cand_j = (int*)p;
  p = take(sizeof(int) * CS);           if (o) o->ncand = (int*)p;
  p = take(sizeof(int) * P);            if (o) o->pool = (int*)p;
  p = take(sizeof(long long) * P);      if (o) o->s_acc = (long long*)p;
  p = take(sizeof(long long) * P);      if (o) o->s_loc = (long long*)p;
  p = take(sizeof(int) * P);            if (o) o->batch = (int*)p;
  p = take(sizeof(int) * P);            if (o) o->inb = (int*)p;
  p = take(sizeof(short) * N);          if (o) o->poolslot = (short*)p;
  p = take(N);                          if (o) o->sel = (unsigned char*)p;
  p = take(sizeof(float) * RPC);        if (o) o->bcov = (float*)p;
  p = take(sizeof(int) * RPC);          if (o) o->cnt = (int*)p;
  p = take(sizeof(long long) * 8);      if (o) o->fb = (long long*)p;
  p = take(sizeof(int) * 8);            if (o) o->scal = (int*)p;
  return off;
}

__device__ __forceinline__ bool key_before(long long ua, int ja, long long ub, int jb) {
  return ua > ub || (ua == ub && ja < jb);
}

__device__ __forceinline__ unsigned lanemask_lt() {
  unsigned m;
  asm("mov.u32 %0, %%lanemask_lt;" : "=r"(m));
  return m;
}

__global__ void __launch_bounds__(SEL_THREADS, 1) k_select(SelArgs a) {
  extern __shared__ __align__(16) char sm_sel[];
  cg::cluster_group cluster = cg::this_cluster();
  const int CS = (int)cluster.num_blocks();
  const int r = (int)cluster.block_rank();
  const int b = blockIdx.x / CS;
  const int N = a.N, P = a.P;
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = blockDim.x >> 5;

  // Image geometry: rows [0, MG) grounded, [MG, MG+N) appearance, rest spatial.
  int Mb, MG;
  bool valid = true;
  if (a.uniform_rows) {
    Mb = a.Mstride;
    MG = Mb;  // everything reported as bank 0
  } else {
    const TextGeom tg = text_geom(a.toff, b, a.B, a.Tmax, nullptr);
    valid = tg.T > 0;
    MG = a.H * tg.T;
    Mb = MG + N + a.L2;
  }
  const int RPC = (a.Mstride + CS - 1) / CS;
  const int mlo = r * RPC, mhi = min(Mb, mlo + RPC);
  const int SL = (N + CS - 1) / CS;
  const int jlo = r * SL, jhi = min(N, jlo + SL);
  const int K = a.K;

  SelSmem s;
  sel_smem_bytes(N, CS, P, RPC, &s, sm_sel);
  const int e = a.fexp ? a.fexp[b] : a.fx_exp;
  const float fxs = ldexpf(1.f, e);
  float* Cimg = a.C + (size_t)b * a.Mstride * N;
  uint16_t* Simg = a.scol + (size_t)b * a.Mstride * N;

  for (int j = threadIdx.x; j < N; j += blockDim.x) {
    s.u_part[j] = 0;
    s.poolslot[j] = -1;
    s.sel[j] = 0;
  }
  for (int j = jlo + threadIdx.x; j < jhi; j += blockDim.x) s.u_slice[j - jlo] = a.u0[(size_t)b * N + j];
  for (int k = threadIdx.x; k < P; k += blockDim.x) s.s_acc[k] = 0;
  for (int q = threadIdx.x; q < RPC; q += blockDim.x) {
    s.bcov[q] = 0.f;
    s.cnt[q] = -1;
  }
  if (threadIdx.x < 8) {
    s.fb[threadIdx.x] = 0;
    s.scal[threadIdx.x] = 0;
  }
  cluster.sync();
  if (!valid) return;  // uniform across the cluster: nobody touches this CTA again

  const int rounds_max = (K + a.bsz - 1) / a.bsz + 1;
  int S_count = 0, rnd = 0, filled = 0;
  bool done = false;
  while (!done) {
    // ---- A: local candidates of this CTA's token slice -------------------
    int npos_local = 0;
    for (int j = jlo + threadIdx.x; j < jhi; j += blockDim.x) {
      const long long uj = s.u_slice[j - jlo];
      if (s.sel[j] || uj <= 0) continue;
      int rank = 0;
      for (int k = jlo; k < jhi; ++k) {
        const long long uk = s.u_slice[k - jlo];
        rank += (!s.sel[k] && uk > 0 && key_before(uk, k, uj, j));
      }
      ++npos_local;
      if (rank < P) {
        for (int c = 0; c < CS; ++c) {
          cluster.map_shared_rank(s.cand_u, c)[r * P + rank] = uj;
          cluster.map_shared_rank(s.cand_j, c)[r * P + rank] = j;
        }
      }
    }
    {
      __shared__ int cnt_sh;
      if (threadIdx.x == 0) cnt_sh = 0;
      __syncthreads();
      if (npos_local) atomicAdd(&cnt_sh, npos_local);
      __syncthreads();
      if (threadIdx.x == 0) {
        const int nloc = min(P, cnt_sh);
        s.scal[5] = nloc;
        for (int c = 0; c < CS; ++c) cluster.map_shared_rank(s.ncand, c)[r] = nloc;
      }
    }
    cluster.sync();  // B1: every CTA's candidates are visible everywhere

    // ---- B: global pool ranks; reset this CTA's gain partials ------------
    int total = 0;
    for (int c = 0; c < CS; ++c) total += s.ncand[c];
    const int Pt = min(P, total);
    const int nloc = s.scal[5];
    for (int k = threadIdx.x; k < nloc; k += blockDim.x) {
      const long long uk = s.cand_u[r * P + k];
      const int jk = s.cand_j[r * P + k];
      int grank = 0;
      for (int c = 0; c < CS; ++c) {
        const int nc = s.ncand[c];
        for (int q = 0; q < nc; ++q)
          grank += key_before(s.cand_u[c * P + q], s.cand_j[c * P + q], uk, jk);
      }
      if (grank < Pt)
        for (int c = 0; c < CS; ++c) cluster.map_shared_rank(s.pool, c)[grank] = jk;
    }
    for (int j = threadIdx.x; j < N; j += blockDim.x) s.u_part[j] = 0;
    cluster.sync();  // B2: the pool is visible everywhere

    if (Pt == 0) {
      // Zero-gain remainder: fill in ascending source order (F unchanged).
      const int need = K - S_count;
      if (wid == 0) {
        int taken = 0;
        for (int base = 0; base < N && taken < need; base += 32) {
          const int j = base + lane;
          const bool free_ = j < N && !s.sel[j];
          const unsigned m = __ballot_sync(FULL, free_);
          const int pos = taken + __popc(m & lanemask_lt());
          if (free_ && pos < need) {
            s.sel[j] = 1;
            if (r == 0) a.order[(size_t)b * K + S_count + pos] = j;
          }
          taken += __popc(m);
        }
      }
      if (r == 0 && a.tv.base && threadIdx.x == 0) {
        int32_t* tp = a.tv.at<int32_t>(b, a.tv.off_pool) + (size_t)rnd * a.tv.pool_size;
        for (int k = 0; k < a.tv.pool_size; ++k) tp[k] = -1;
        a.tv.at<int32_t>(b, a.tv.off_round_end)[rnd] = K;
      }
      filled = need;
      S_count = K;
      ++rnd;
      __syncthreads();
      break;
    }

    // ---- C: responsibilities over the pool -------------------------------
    for (int k = threadIdx.x; k < Pt; k += blockDim.x) {
      s.poolslot[s.pool[k]] = (short)k;
      s.s_loc[k] = 0;
    }
    __syncthreads();
    for (int m = mlo + wid; m < mhi; m += nw) {
      const int q = m - mlo;
      const float bm = s.bcov[q];
      const int n = s.cnt[q];
      const float* crow = Cimg + (size_t)m * N;
      const uint16_t* jrow = Simg + (size_t)m * N;
      // pass 1: max residual and number of positive pool entries
      float rmax = 0.f;
      int npool = 0;
      if (n < 0) {
        for (int k = lane; k < Pt; k += 32) {
          const float R = crow[s.pool[k]] - bm;
          if (R > 0.f) { rmax = fmaxf(rmax, R); ++npool; }
        }
      } else {
        for (int k = lane; k < n; k += 32) {
          if (s.poolslot[jrow[k]] >= 0) {
            const float R = crow[k] - bm;
            rmax = fmaxf(rmax, R);
            ++npool;
          }
        }
      }
      rmax = warp_max(rmax);
      npool = warp_sum_int(npool);
      if (npool == 0) continue;
      const float tau = a.resp_temp * rmax + a.resp_eps;
      // pass 2: softmax denominator (zero-residual pool entries add exp(0) = 1)
      float z = 0.f;
      if (n < 0) {
        for (int k = lane; k < Pt; k += 32) {
          const float R = crow[s.pool[k]] - bm;
          if (R > 0.f) z += expf(R / tau);
        }
      } else {
        for (int k = lane; k < n; k += 32)
          if (s.poolslot[jrow[k]] >= 0) z += expf((crow[k] - bm) / tau);
      }
      z = warp_sum(z) + (float)(Pt - npool);
      const float invz = 1.f / z;
      // pass 3: s_i += rho_mi R_mi
      if (n < 0) {
        for (int k = lane; k < Pt; k += 32) {
          const float R = crow[s.pool[k]] - bm;
          if (R > 0.f)
            atomicAdd((unsigned long long*)&s.s_loc[k],
                      (unsigned long long)to_fix(expf(R / tau) * invz * R, fxs));
        }
      } else {
        for (int k = lane; k < n; k += 32) {
          const int ps = s.poolslot[jrow[k]];
          if (ps >= 0) {
            const float R = crow[k] - bm;
            atomicAdd((unsigned long long*)&s.s_loc[ps],
                      (unsigned long long)to_fix(expf(R / tau) * invz * R, fxs));
          }
        }
      }
    }
    __syncthreads();
    for (int k = threadIdx.x; k < Pt; k += blockDim.x) {
      const unsigned long long v = (unsigned long long)s.s_loc[k];
      if (v)
        for (int c = 0; c < CS; ++c)
          atomicAdd((unsigned long long*)cluster.map_shared_rank(s.s_acc, c) + k, v);
    }
    cluster.sync();  // B3: the scores are complete everywhere

    // ---- D: batch, coverage update, survivor filter, next gains ----------
    const int nb = min(a.bsz, min(Pt, K - S_count));
    for (int k = threadIdx.x; k < Pt; k += blockDim.x) {
      const long long sk = s.s_acc[k];
      const int jk = s.pool[k];
      int rank = 0;
      for (int q = 0; q < Pt; ++q) rank += key_before(s.s_acc[q], s.pool[q], sk, jk);
      s.inb[k] = rank < nb;
      if (rank < nb) s.batch[rank] = jk;
    }
    __syncthreads();
    for (int q = threadIdx.x; q < nb; q += blockDim.x) {
      s.sel[s.batch[q]] = 1;
      if (r == 0) a.order[(size_t)b * K + S_count + q] = s.batch[q];
    }
    if (r == 0 && a.tv.base && threadIdx.x == 0) {
      int32_t* tp = a.tv.at<int32_t>(b, a.tv.off_pool) + (size_t)rnd * a.tv.pool_size;
      for (int k = 0; k < a.tv.pool_size; ++k) tp[k] = k < Pt ? s.pool[k] : -1;
      a.tv.at<int32_t>(b, a.tv.off_round_end)[rnd] = S_count + nb;
    }
    const bool dense_round = (rnd == 0);
    for (int m = mlo + wid; m < mhi; m += nw) {
      const int q = m - mlo;
      const float bm = s.bcov[q];
      const int n = s.cnt[q];
      float* crow = Cimg + (size_t)m * N;
      uint16_t* jrow = Simg + (size_t)m * N;
      float bnew = bm;
      if (n < 0) {
        for (int t = lane; t < nb; t += 32) bnew = fmaxf(bnew, crow[s.batch[t]]);
      } else {
        for (int k = lane; k < n; k += 32) {
          const int ps = s.poolslot[jrow[k]];
          if (ps >= 0 && s.inb[ps]) bnew = fmaxf(bnew, crow[k]);
        }
      }
      bnew = warp_max(bnew);
      const long long fb_new = to_fix(bnew, fxs);
      const int len = n < 0 ? N : n;
      int w = 0;
      float rowmax = 0.f;
      for (int base = 0; base < len; base += 32) {
        const int k = base + lane;
        float c = 0.f;
        int j = 0;
        if (k < len) {
          c = crow[k];
          j = n < 0 ? k : jrow[k];
        }
        rowmax = fmaxf(rowmax, c);
        const bool keep = k < len && c > bnew;
        const unsigned msk = __ballot_sync(FULL, keep);
        __syncwarp();  // every lane has read its entry before any lane overwrites one
        if (keep) {
          const int pos = w + __popc(msk & lanemask_lt());
          crow[pos] = c;
          jrow[pos] = (uint16_t)j;
          atomicAdd((unsigned long long*)&s.u_part[j],
                    (unsigned long long)(to_fix(c, fxs) - fb_new));
        }
        w += __popc(msk);
      }
      if (lane == 0) {
        s.bcov[q] = bnew;
        s.cnt[q] = w;
      }
      if (dense_round) {
        rowmax = warp_max(rowmax);
        if (lane == 0) {
          const int bank = m < MG ? 0 : (m < MG + N ? 1 : 2);
          atomicAdd((unsigned long long*)&s.fb[3 + bank], (unsigned long long)to_fix(rowmax, fxs));
        }
      }
    }
    __syncthreads();
    for (int k = threadIdx.x; k < Pt; k += blockDim.x) {
      s.poolslot[s.pool[k]] = -1;
      s.s_acc[k] = 0;
    }
    S_count += nb;
    ++rnd;
    if (S_count >= K) break;
    if (rnd >= rounds_max) {  // cannot happen (each round adds >= 1 token); guard the loop
      if (threadIdx.x == 0) set_status(a.status, GMC_STATUS_INTERNAL);
      break;
    }
    cluster.sync();  // B4: every CTA's gain partials are complete

    // ---- E: reduce this CTA's token slice of the gains --------------------
    for (int j = jlo + threadIdx.x; j < jhi; j += blockDim.x) {
      long long t = 0;
      for (int c = 0; c < CS; ++c) t += cluster.map_shared_rank(s.u_part, c)[j];
      s.u_slice[j - jlo] = t;
    }
    // Only a block barrier: the next remote writes (candidates) target arrays
    // nobody reads now, and u_part is reset only after B1.
    __syncthreads();
  }

  // ---- final: coverage per bank, sorted support, trace ---------------------
  {
    long long f0 = 0, f1 = 0, f2 = 0;
    for (int m = mlo + threadIdx.x; m < mhi; m += blockDim.x) {
      const long long v = to_fix(s.bcov[m - mlo], fxs);
      if (m < MG) f0 += v; else if (m < MG + N) f1 += v; else f2 += v;
    }
    long long* fb0 = cluster.map_shared_rank(s.fb, 0);
    if (f0) atomicAdd((unsigned long long*)&fb0[0], (unsigned long long)f0);
    if (f1) atomicAdd((unsigned long long*)&fb0[1], (unsigned long long)f1);
    if (f2) atomicAdd((unsigned long long*)&fb0[2], (unsigned long long)f2);
    __syncthreads();
    if (r != 0 && threadIdx.x < 3 && s.fb[3 + threadIdx.x])
      atomicAdd((unsigned long long*)&fb0[3 + threadIdx.x], (unsigned long long)s.fb[3 + threadIdx.x]);
  }
  cluster.sync();
  if (r != 0) return;
  // ascending support and slot map (one warp, ballot prefix over the flags)
  if (wid == 0) {
    int cnt = 0;
    for (int base = 0; base < N; base += 32) {
      const int j = base + lane;
      const bool on = j < N && s.sel[j];
      const unsigned m = __ballot_sync(FULL, on);
      const int pos = cnt + __popc(m & lanemask_lt());
      if (j < N) a.slot[(size_t)b * N + j] = on ? pos : -1;
      if (on && pos < K) {
        a.support[(size_t)b * K + pos] = j;
        if (a.out_idx) a.out_idx[(size_t)b * K + pos] = j;
      }
      cnt += __popc(m);
    }
    if (lane == 0 && cnt != K) set_status(a.status, GMC_STATUS_INTERNAL);
  }
  if (a.tv.base) {
    if (threadIdx.x == 0) {
      gmc_trace_header* hd = a.tv.header(b);
      hd->K = K;
      hd->rounds = rnd;
      hd->filled = filled;
      const double inv = ldexp(1.0, -e);
      for (int q = 0; q < 3; ++q) {
        hd->F_S[q] = (float)((double)s.fb[q] * inv);
        hd->F_V[q] = (float)((double)s.fb[3 + q] * inv);
      }
      hd->c_B = -1.f;  // not computed by this build
    }
    int32_t* to = a.tv.at<int32_t>(b, a.tv.off_order);
    for (int q = threadIdx.x; q < K; q += blockDim.x) to[q] = a.order[(size_t)b * K + q];
    int32_t* te = a.tv.at<int32_t>(b, a.tv.off_round_end);
    for (int q = rnd + threadIdx.x; q < a.tv.rounds_max; q += blockDim.x) te[q] = K;
    int32_t* tp = a.tv.at<int32_t>(b, a.tv.off_pool);
    for (size_t q = (size_t)rnd * a.tv.pool_size + threadIdx.x;
         q < (size_t)a.tv.rounds_max * a.tv.pool_size; q += blockDim.x)
      tp[q] = -1;
  }
}

static int g_num_sms = 0;

cudaError_t launch_select(int B, int N, int K, int M, const int32_t* toff, int H, int T, int L2,
                          const gmc_params& p, int fx_exp, const int32_t* fexp, float* C,
                          uint16_t* scol, const long long* u0, int32_t* order, int32_t* support,
                          int32_t* slot, int32_t* out_idx, uint32_t* status, const TraceView& tv,
                          cudaStream_t st) {
  cudaError_t e;
  if (g_num_sms == 0) {
    int dev = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&g_num_sms, cudaDevAttrMultiProcessorCount, dev)) !=
        cudaSuccess)
      return e;
    if ((e = cudaFuncSetAttribute(k_select, cudaFuncAttributeNonPortableClusterSizeAllowed, 1)) !=
        cudaSuccess)
      return e;
  }
  SelArgs a;
  a.B = B; a.N = N; a.K = K; a.Mstride = M; a.H = H; a.Tmax = T; a.L2 = L2;
  a.toff = toff;
  a.uniform_rows = (H == 0);
  a.P = p.pool_mult * p.batch_b;
  a.bsz = p.batch_b;
  a.resp_temp = p.resp_temp;
  a.resp_eps = p.resp_eps;
  a.fx_exp = fx_exp;
  a.fexp = fexp;
  a.C = C; a.scol = scol; a.u0 = u0;
  a.order = order; a.support = support; a.slot = slot; a.out_idx = out_idx;
  a.status = status;
  a.tv = tv;
  int CS = 1;
  while (CS * 2 <= SEL_MAX_CS && (long long)B * CS * 2 <= g_num_sms) CS *= 2;
  for (; CS >= 1; CS /= 2) {
    const int RPC = (M + CS - 1) / CS;
    const size_t smem = sel_smem_bytes(N, CS, a.P, RPC, nullptr, nullptr);
    if (smem > 227 * 1024) continue;
    if ((e = set_smem_limit((const void*)k_select, smem)) != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(B * CS);
    cfg.blockDim = dim3(SEL_THREADS);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = CS;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int nclusters = 0;
    e = cudaOccupancyMaxActiveClusters(&nclusters, (void*)k_select, &cfg);
    if (e != cudaSuccess || nclusters < 1) {
      cudaGetLastError();
      continue;
    }
    return cudaLaunchKernelEx(&cfg, k_select, a);
  }
  return cudaErrorInvalidConfiguration;
}

}  // namespace gmc
