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
// place, and later rounds touch only those.  This is exact, not an
// approximation: the skipped entries are exactly the zero residuals.  (A pool
// member with R_mi = 0 still counts in row m's softmax denominator; the
// kernel adds those terms explicitly.  Every softmax is shifted by its row's
// largest logit, so no exponential exceeds 1 for any temperature.)  Survivor lists start
// in global memory (in place over Cbar, row-major, processed by 8-lane groups)
// and move into the CTA's shared memory as soon as they all fit there, sorted
// by token ("flat mode"): then the responsibilities and the coverage update
// read only the pool's and the batch's token segments, and the gain update
// sums every token's residuals in registers.
//
// The first round (dense, S empty) runs over the whole GPU (k_round0.cu); this
// kernel continues from round 1 with the survivor lists it left.
//
// Parallel layout.  The CS CTAs of a cluster split the client rows; each CTA
// keeps its rows' coverage b_m, survivor counts and lists.  Gains and scores
// are summed in 64-bit fixed point, so every reduction (shared-memory atomics
// inside a CTA, distributed-shared-memory atomics across the cluster) is
// exact and order-independent: the solver is deterministic.  Per round:
//   pool:   every CTA selects the same pool from the full gain vector
//           (histogram + exact tie ranking, see select_pool);
//   scores: every CTA adds its rows' responsibility-weighted residuals into
//           the score array of every CTA of the cluster; every CTA then picks
//           the same batch;
//   gains:  every CTA adds its rows' residuals for the next round into the
//           owner of each token (token j belongs to CTA j / ceil(N / CS)); after
//           the barrier every CTA reads the full gain vector from the owners.
//           The owners' buffers alternate between rounds, so a buffer is
//           cleared only after every CTA has read it.
// Two cluster barriers per round; all control decisions are derived from data
// every CTA holds identically, so all CTAs run the same barriers.
#include <cooperative_groups.h>

#include "common.cuh"
#include "kernels.cuh"
#include "select_common.cuh"

namespace cg = cooperative_groups;

namespace gmc {

namespace {
constexpr int SEL_THREADS = 512;
constexpr int SEL_WARPS = SEL_THREADS / 32;
constexpr int SEL_MAX_CS = 16;
constexpr int HBINS = sel::HBINS;
constexpr int UNR = 4;     // entries in flight per lane in a sweep
constexpr int PCL = 8;     // pool entries a lane keeps in registers (8 lanes x 8 >= pool of 64)
constexpr int DEADROW = 0xFFFF;  // flat mode: row id of an entry whose residual is zero
constexpr int FU = 4;      // flat mode: entries a thread loads ahead in a walk
constexpr int CU = 8;      // flat mode: entries a thread moves per compaction chunk
constexpr int COMPACT_EVERY = 4;  // flat mode: rounds between compactions of the survivor lists
constexpr size_t SMEM_LIMIT = 227 * 1024;

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
  int images;           // images per prompt (> 1: the first round seeded one token per image)
  int cap;              // survivor entries that fit in shared memory
  int rpc;              // rows one CTA can own
  R0State r0;           // state after the first round
};

struct SelSmem {
  unsigned long long* gacc;  // [SL] gains of the tokens this CTA owns: every CTA of
                             // the cluster adds the changes of its rows (
                             // the buffer is read in a round's pool and changed
                             // after that round's score barrier)
  long long* u_full;    // [N]  gains of the current round (every CTA)
  int* hist;            // [HBINS]
  int* coarse;          // [CBINS]
  unsigned char* pk;    // [N]  select_pool: boundary tokens that enter
  short* key;           // [N]  select_pool: bucket of every token
  int* bnd;             // [N]  tokens in the boundary histogram bin
  unsigned char* sel;   // [N]
  short* poolslot;      // [N]  pool slot of a token or -1
  int* pool;            // [P]
  long long* s_acc;     // [P]  cluster-wide scores, pushed by every CTA
  unsigned long long* sw;  // [SEL_WARPS][P] per-warp partial scores
  int* batch;           // [P]
  int* inb;             // [P]
  int* wsum;            // [32] scan scratch
  float* bcov;          // [RPC] coverage b_m of this CTA's rows
  int* cnt;             // [RPC] survivors (-1: row still dense)
  int* rmaxb;           // [RPC] flat mode: bits of the row's largest pool residual
  int* npl;             // [RPC] flat mode: pool entries of the row
  unsigned long long* z64;  // [RPC] flat mode: softmax denominator (fixed point 2^40)
  int* bnb;             // [RPC] flat mode: bits of the row's largest batch value
  long long* bfix;      // [RPC] flat mode: coverage in fixed point
  long long* bfold;     // [RPC] flat mode: coverage in fixed point before the round's batch
  int* cstart;          // [N+1] flat mode: first entry of every token
  int* win;             // [WBINS + 4] select_pool_window: window bins and counters
  long long* wcu;       // [WCAP] select_pool_window: candidates' gains
  int* wcj;             // [WCAP] select_pool_window: candidates' tokens
  long long* fb;        // [8]  F_S[3], F_V[3] (fixed point)
  int* scal;            // [16] Bstar, c_hi, Pt, nbnd, cursor, global rows left
  float* svals;         // [cap]
  uint16_t* scols;      // [cap]
  uint16_t* srows;      // [cap] flat mode: row of every entry (DEADROW: residual zero)
};

enum { SC_BSTAR = 0, SC_CHI, SC_PT, SC_NBND, SC_CURSOR, SC_GLOBAL, SC_NEED };

__host__ __device__ inline size_t sel_fixed_bytes(int N, int P, int RPC, int gwords, SelSmem* o,
                                                  char* base) {
  size_t off = 0;
  auto take = [&](size_t bytes) {
    size_t at = off;
    off += (bytes + 15) & ~(size_t)15;
    return base ? base + at : nullptr;
  };
  char* p;
  p = take(sizeof(unsigned long long) * gwords);  if (o) o->gacc = (unsigned long long*)p;
  p = take(sizeof(long long) * N);  if (o) o->u_full = (long long*)p;
  p = take(sizeof(int) * HBINS);    if (o) o->hist = (int*)p;
  p = take(sizeof(int) * sel::CBINS);  if (o) o->coarse = (int*)p;
  p = take(N);                      if (o) o->pk = (unsigned char*)p;
  p = take(sizeof(short) * N);      if (o) o->key = (short*)p;
  p = take(sizeof(int) * N);        if (o) o->bnd = (int*)p;
  p = take(N);                      if (o) o->sel = (unsigned char*)p;
  p = take(sizeof(short) * N);      if (o) o->poolslot = (short*)p;
  p = take(sizeof(int) * P);        if (o) o->pool = (int*)p;
  p = take(sizeof(long long) * P);  if (o) o->s_acc = (long long*)p;
  p = take(sizeof(unsigned long long) * SEL_WARPS * P);  if (o) o->sw = (unsigned long long*)p;
  p = take(sizeof(int) * P);        if (o) o->batch = (int*)p;
  p = take(sizeof(int) * P);        if (o) o->inb = (int*)p;
  p = take(sizeof(int) * 32);       if (o) o->wsum = (int*)p;
  p = take(sizeof(float) * RPC);    if (o) o->bcov = (float*)p;
  p = take(sizeof(int) * RPC);      if (o) o->cnt = (int*)p;
  p = take(sizeof(int) * RPC);      if (o) o->rmaxb = (int*)p;
  p = take(sizeof(int) * RPC);      if (o) o->npl = (int*)p;
  p = take(sizeof(unsigned long long) * RPC); if (o) o->z64 = (unsigned long long*)p;
  p = take(sizeof(int) * RPC);      if (o) o->bnb = (int*)p;
  p = take(sizeof(long long) * RPC);  if (o) o->bfix = (long long*)p;
  p = take(sizeof(long long) * RPC);  if (o) o->bfold = (long long*)p;
  p = take(sizeof(int) * (N + 1));  if (o) o->cstart = (int*)p;
  p = take(sizeof(int) * (sel::WBINS + 4));  if (o) o->win = (int*)p;
  p = take(sizeof(long long) * sel::WCAP);   if (o) o->wcu = (long long*)p;
  p = take(sizeof(int) * sel::WCAP);         if (o) o->wcj = (int*)p;
  p = take(sizeof(long long) * 8);  if (o) o->fb = (long long*)p;
  p = take(sizeof(int) * 16);       if (o) o->scal = (int*)p;
  return off;
}

// Fire-and-forget 64-bit add into the shared memory of CTA `rank` of the
// cluster at the offset of local shared-memory address `local` (no value is
// returned, so the issuing thread does not wait for the remote round trip;
// the next cluster barrier orders it before every later read).
__device__ __forceinline__ void red_add_cluster(const void* local, int rank,
                                                unsigned long long v) {
  const uint32_t la = (uint32_t)__cvta_generic_to_shared(local);
  uint32_t ra;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(ra) : "r"(la), "r"(rank));
  asm volatile("red.shared::cluster.add.u64 [%0], %1;" ::"r"(ra), "l"(v) : "memory");
}

using sel::key_before;
using sel::lanemask_lt;
using sel::block_exclusive_scan;

// Reductions inside an aligned group of G = 8 lanes (mask `gm`).
constexpr int G = 8;
__device__ __forceinline__ float group_max(float v, unsigned gm) {
#pragma unroll
  for (int o = G / 2; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(gm, v, o));
  return v;
}
__device__ __forceinline__ float group_sum(float v, unsigned gm) {
#pragma unroll
  for (int o = G / 2; o > 0; o >>= 1) v += __shfl_xor_sync(gm, v, o);
  return v;
}
__device__ __forceinline__ int group_sum(int v, unsigned gm) {
#pragma unroll
  for (int o = G / 2; o > 0; o >>= 1) v += __shfl_xor_sync(gm, v, o);
  return v;
}

}  // namespace

__global__ void __launch_bounds__(SEL_THREADS, 1) k_select(SelArgs a) {
  grid_dep_wait();
  extern __shared__ __align__(16) char sm_sel[];
  cg::cluster_group cluster = cg::this_cluster();
  const int CS = (int)cluster.num_blocks();
  const int r = (int)cluster.block_rank();
  const int b = blockIdx.x / CS;
  const int N = a.N, P = a.P, K = a.K;
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
  const int RPC = a.rpc;  // capacity of the per-row arrays of one CTA
  // token j's next-round gain is summed in CTA j / SL (its owner)
  const int SL = (N + CS - 1) / CS;

  SelSmem s;
  const size_t fixed = sel_fixed_bytes(N, P, RPC, SL, &s, sm_sel);
  s.svals = reinterpret_cast<float*>(sm_sel + fixed);
  s.scols = reinterpret_cast<uint16_t*>(sm_sel + fixed + sizeof(float) * (size_t)a.cap);
  s.srows = s.scols + a.cap;
  const int e = a.fexp ? a.fexp[b] : a.fx_exp;
  const float fxs = ldexpf(1.f, e);
  float* Cimg = a.C + (size_t)b * a.Mstride * N;
  uint16_t* Simg = a.scol + (size_t)b * a.Mstride * N;

  // state after the rounds run on the whole GPU (k_round0.cu); a first round
  // with an empty pool leaves the gains of the empty support and nothing
  // selected
  const int rd0 = valid ? a.r0.info[b * INFO_W + 2] : 0;  // rounds done
  const int Pt0 = rd0;                                // > 0: the rounds left survivor lists
  const int nb0 = rd0 > 0 ? a.r0.info[b * INFO_W + 1] : 0;  // tokens selected so far
  // boundary bucket of the last pool (-1: none; the next pool is then found
  // over every bucket)
  int phint = rd0 > 0 ? a.r0.info[b * INFO_W + 5] : -1;
  for (int j = threadIdx.x; j < N; j += blockDim.x) {
    s.u_full[j] = rd0 > 0 ? a.r0.ugain[(size_t)b * N + j] : a.u0[(size_t)b * N + j];
    s.poolslot[j] = -1;
    s.sel[j] = 0;
  }
  for (int k = threadIdx.x; k < P; k += blockDim.x) s.s_acc[k] = 0;
  for (int q = threadIdx.x; q < SL; q += blockDim.x) {  // the gains of the tokens this CTA owns
    const int j = r * SL + q;
    s.gacc[q] = j < N ? (unsigned long long)(rd0 > 0 ? a.r0.ugain[(size_t)b * N + j]
                                                     : a.u0[(size_t)b * N + j])
                      : 0ull;
  }
  for (int h = threadIdx.x; h < HBINS; h += blockDim.x) s.hist[h] = 0;  // select_pool keeps it zero
  if (threadIdx.x < sel::CBINS) s.coarse[threadIdx.x] = 0;
  for (int q = threadIdx.x; q < sel::WBINS + 4; q += blockDim.x) s.win[q] = 0;
  if (threadIdx.x < 8) s.fb[threadIdx.x] = 0;
  if (threadIdx.x < 16) s.scal[threadIdx.x] = 0;
  if (threadIdx.x == 0) s.scal[SC_GLOBAL] = 1;
  // Rows are dealt to the CTAs in turn (CTA r holds rows r, r + CS, ...):
  // every CTA gets the same mix of grounded, appearance and spatial rows and
  // of the image's regions, so the work of every phase is about even.
  __syncthreads();
  const int nrows = Mb > r ? (Mb - r + CS - 1) / CS : 0;
  auto grow = [&](int q) { return q * CS + r; };  // client row of local row q
  for (int q = threadIdx.x; q < RPC; q += blockDim.x) {
    const bool have = Pt0 > 0 && q < nrows;
    s.bcov[q] = have ? a.r0.bcov[(size_t)b * a.Mstride + grow(q)] : 0.f;
    s.cnt[q] = have ? a.r0.cnt[(size_t)b * a.Mstride + grow(q)] : 0;
    s.bfix[q] = 0;
    s.rmaxb[q] = 0;
    s.npl[q] = 0;
    s.z64[q] = 0;
    s.bnb[q] = 0;
  }
  __syncthreads();
  for (int q = threadIdx.x; q < nb0; q += blockDim.x) s.sel[a.order[(size_t)b * K + q]] = 1;
  cluster.sync();
  if (!valid) return;  // uniform across the cluster

  // Move this CTA's survivor lists from global into shared memory once they
  // all fit, sorted by token (a counting sort): the entries of token j are
  // [cstart[j], cstart[j+1]).  The order inside a token's segment depends on
  // the schedule; nothing computed from it does (integer and max reductions).
  auto migrate = [&]() {
    if (!s.scal[SC_GLOBAL] || nrows >= DEADROW) return;  // row ids are stored in 16 bits
    // entry offsets of the rows (contiguous rows per thread), then every entry
    // of the CTA handled by one thread: all its global loads are in flight at once
    const int rper = (nrows + blockDim.x - 1) / blockDim.x;
    const int q0 = min(nrows, (int)threadIdx.x * rper), q1 = min(nrows, q0 + rper);
    int mine = 0;
    for (int q = q0; q < q1; ++q) mine += s.cnt[q];
    int tot = 0;
    int at = block_exclusive_scan(mine, s.wsum, &tot);
    if (tot > a.cap) return;  // uniform over the block
    int* rp = reinterpret_cast<int*>(s.bfix);  // [nrows + 1]; bfix is set at the end
    for (int q = q0; q < q1; ++q) {
      rp[q] = at;
      at += s.cnt[q];
    }
    if (threadIdx.x == 0) rp[nrows] = tot;
    for (int j = threadIdx.x; j < N; j += blockDim.x) s.bnd[j] = 0;
    __syncthreads();
    // row of entry e: the last q with rp[q] <= e
    auto row_of = [&](int e) {
      int lo = 0, hi = nrows;  // rp[lo] <= e < rp[hi]
      while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (rp[mid] <= e) lo = mid; else hi = mid;
      }
      return lo;
    };
    constexpr int MU = 4;  // entries per thread in flight
    for (int e0 = threadIdx.x; e0 < tot; e0 += MU * blockDim.x) {
      int jj[MU];
#pragma unroll
      for (int u = 0; u < MU; ++u) {
        const int e = e0 + u * (int)blockDim.x;
        jj[u] = -1;
        if (e < tot) {
          const int q = row_of(e);
          jj[u] = Simg[(size_t)grow(q) * N + (e - rp[q])];
        }
      }
#pragma unroll
      for (int u = 0; u < MU; ++u)
        if (jj[u] >= 0) atomicAdd(&s.bnd[jj[u]], 1);
    }
    __syncthreads();
    {
      const int per = (N + blockDim.x - 1) / blockDim.x;
      const int j0 = min(N, (int)threadIdx.x * per), j1 = min(N, j0 + per);
      int c = 0;
      for (int j = j0; j < j1; ++j) c += s.bnd[j];
      int at2 = block_exclusive_scan(c, s.wsum, nullptr);
      for (int j = j0; j < j1; ++j) {
        const int n = s.bnd[j];
        s.cstart[j] = at2;
        s.bnd[j] = at2;  // fill cursor of token j
        at2 += n;
      }
      if (threadIdx.x == 0) s.cstart[N] = tot;
    }
    __syncthreads();
    for (int e0 = threadIdx.x; e0 < tot; e0 += MU * blockDim.x) {
      int jj[MU], qq[MU];
      float vv[MU];
#pragma unroll
      for (int u = 0; u < MU; ++u) {
        const int e = e0 + u * (int)blockDim.x;
        jj[u] = -1;
        qq[u] = 0;
        vv[u] = 0.f;
        if (e < tot) {
          const int q = row_of(e);
          const size_t g = (size_t)grow(q) * N + (e - rp[q]);
          qq[u] = q;
          jj[u] = Simg[g];
          vv[u] = Cimg[g];
        }
      }
#pragma unroll
      for (int u = 0; u < MU; ++u)
        if (jj[u] >= 0) {
          const int pos = atomicAdd(&s.bnd[jj[u]], 1);
          s.svals[pos] = vv[u];
          s.scols[pos] = (uint16_t)jj[u];
          s.srows[pos] = (uint16_t)qq[u];
        }
    }
    __syncthreads();  // rp (over bfix) is no longer read
    for (int q = threadIdx.x; q < nrows; q += blockDim.x) s.bfix[q] = to_fix(s.bcov[q], fxs);
    __syncthreads();
    if (threadIdx.x == 0) {
      s.scal[SC_CURSOR] = tot;
      s.scal[SC_GLOBAL] = 0;
    }
    __syncthreads();
  };
  if (Pt0 > 0) migrate();

  const int rounds_max = (K + a.bsz - 1) / a.bsz + 1 + (a.images > 1 ? 1 : 0);
  // add v to token j's gain for the round after `rnd` at the token's owner
  // (exact: 64-bit integer atomics, order-independent)
  auto gain_add = [&](int j, unsigned long long v, int rnd_now) {
    const int o = j / SL;
    unsigned long long* at = s.gacc + (j - o * SL);
    if (CS > 1) red_add_cluster(at, o, v); else atomicAdd(at, v);
  };
  // add v to pool slot k's score in every CTA of the cluster
  auto score_push = [&](int k, unsigned long long v, int c0, int cstep) {
    for (int c = c0; c < CS; c += cstep) red_add_cluster(s.s_acc + k, c, v);
  };
  int S_count = nb0, rnd = rd0, filled = 0;
  // token j's gain for the round after the last one, at its owner
  auto gain_at = [&](int j) -> const unsigned long long* {
    const int o = j / SL;
    const unsigned long long* at = s.gacc + (j - o * SL);
    return CS > 1 ? cluster.map_shared_rank(at, o) : at;
  };
  auto read_gains = [&]() {
    constexpr int GU = 4;  // remote loads in flight per thread
    for (int j0 = threadIdx.x; j0 < N; j0 += GU * blockDim.x) {
      unsigned long long v[GU];
#pragma unroll
      for (int t = 0; t < GU; ++t) {
        const int j = j0 + t * (int)blockDim.x;
        v[t] = j < N ? *gain_at(j) : 0ull;
      }
#pragma unroll
      for (int t = 0; t < GU; ++t) {
        const int j = j0 + t * (int)blockDim.x;
        if (j < N) s.u_full[j] = (long long)v[t];
      }
    }
    __syncthreads();
  };
  bool remote_gains = false;  // this round's gains are still at their owners
  const int sub = lane / G, gl = lane % G;
  const int gid = wid * (32 / G) + sub, ngrp = nw * (32 / G);  // 8-lane groups of the block
  const unsigned gm = 0xFFu << (sub * G);
  const unsigned lt = lanemask_lt() & gm;
  while (S_count < K) {
    if (rnd >= rounds_max) {  // cannot happen (each round adds >= 1 token); guard the loop
      if (threadIdx.x == 0) set_status(a.status, GMC_STATUS_INTERNAL);
      break;
    }
    // ---- pool of this round ------------------------------------------------------
    // (u_full is complete once either pool routine returns)
    int Pt;
    if (remote_gains)
      Pt = sel::select_pool_window([&](int j) { return (long long)*gain_at(j); }, s.u_full, s.sel,
                                   N, P, sel::WindowScratch{s.win, s.wcu, s.wcj}, s.pool,
                                   s.poolslot, &phint);
    else
      Pt = sel::select_pool_window([&](int j) { return s.u_full[j]; }, s.u_full, s.sel, N, P,
                                   sel::WindowScratch{s.win, s.wcu, s.wcj}, s.pool, s.poolslot,
                                   &phint);
    remote_gains = false;
    if (Pt < 0) {
      sel::PoolScratch pw{s.hist, s.coarse, s.bnd, s.key, s.pk, s.wsum, s.scal + 8};
      Pt = sel::select_pool(s.u_full, s.sel, N, P, pw, s.pool, s.poolslot, nullptr, &phint);
    }
    if (r == 0 && a.tv.base)  // certificate input: the gains this round starts from
      for (int j = threadIdx.x; j < N; j += blockDim.x) a.tv.gains(b, rnd, N)[j] = s.u_full[j];
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
    for (int k = threadIdx.x; k < SEL_WARPS * Pt; k += blockDim.x) s.sw[k] = 0;
    if (r == 0 && a.tv.base && threadIdx.x < a.tv.pool_size) {
      int32_t* tp = a.tv.at<int32_t>(b, a.tv.off_pool) + (size_t)rnd * a.tv.pool_size;
      tp[threadIdx.x] = threadIdx.x < Pt ? s.pool[threadIdx.x] : -1;
    }
    __syncthreads();

    // ---- flat mode (every list of this CTA in shared memory, sorted by token):
    // the responsibilities touch only the pool tokens' segments, one 8-lane
    // group per pool token; per-row values are order-independent (max of positive floats
    // as integers, fixed-point sums), so nothing depends on the schedule.
    const bool flat = !s.scal[SC_GLOBAL];
    const float z_one = 1099511627776.f;  // 2^40: fixed-point scale of the softmax denominators
    const float z_inv = 1.f / z_one;
    if (flat) {
      // largest pool residual and number of pool entries of every row
      for (int k = gid; k < Pt; k += ngrp) {
        const int j = s.pool[k];
        for (int p = s.cstart[j] + gl; p < s.cstart[j + 1]; p += G) {
          const int q = s.srows[p];
          if (q == DEADROW) continue;
          atomicMax(&s.rmaxb[q], __float_as_int(s.svals[p] - s.bcov[q]));
          atomicAdd(&s.npl[q], 1);
        }
      }
      __syncthreads();
      // softmax denominators shifted by the row's largest logit (every term at
      // most 1, so at most 2^40 * pool size), exact in 2^-40
      for (int k = gid; k < Pt; k += ngrp) {
        const int j = s.pool[k];
        for (int p = s.cstart[j] + gl; p < s.cstart[j + 1]; p += G) {
          const int q = s.srows[p];
          if (q == DEADROW) continue;
          const float rmax = __int_as_float(s.rmaxb[q]);
          const float tau = a.resp_temp * rmax + a.resp_eps;
          atomicAdd(&s.z64[q], (unsigned long long)to_fix(
                                   expf(((s.svals[p] - s.bcov[q]) - rmax) / tau), z_one));
        }
      }
      __syncthreads();
      // s_k = sum_m rho_mk R_mk: one group owns pool slot k and adds its sum
      // into every CTA's scores
      for (int k = gid; k < Pt; k += ngrp) {
        const int j = s.pool[k];
        unsigned long long acc = 0;
        for (int p = s.cstart[j] + gl; p < s.cstart[j + 1]; p += G) {
          const int q = s.srows[p];
          if (q == DEADROW) continue;
          const float rmax = __int_as_float(s.rmaxb[q]);
          const float tau = a.resp_temp * rmax + a.resp_eps;
          // pool tokens without an entry in row q have R = 0
          const float z =
              fix_to_float(s.z64[q]) * z_inv + (float)(Pt - s.npl[q]) * expf(-rmax / tau);
          const float R = s.svals[p] - s.bcov[q];
          acc += (unsigned long long)to_fix(expf((R - rmax) / tau) / z * R, fxs);
        }
#pragma unroll
        for (int o = G / 2; o > 0; o >>= 1) acc += __shfl_xor_sync(gm, acc, o);
        if (acc) score_push(k, acc, gl, G);  // the group's lanes share the CTAs
      }
    }
    if (!flat) {
    // ---- responsibilities of this CTA's rows over the pool (8-lane group per row)
    // One sweep of the row finds its pool entries; each lane keeps up to PCL of
    // them in registers for the softmax (more: a second sweep).
    for (int q0 = wid * (32 / G); q0 < nrows; q0 += nw * (32 / G)) {
      const int q = q0 + sub;
      const int n = q < nrows ? s.cnt[q] : 0;
      const float bm = q < nrows ? s.bcov[q] : 0.f;
      const float* vals = Cimg + (size_t)grow(q) * N;
      const uint16_t* cols = Simg + (size_t)grow(q) * N;
      float rmax = 0.f;
      int npool = 0, ncache = 0, mine = 0;  // mine: pool entries this lane saw
      float cv[PCL] = {};
      int cs[PCL] = {};
      bool spill = false;
      for (int k0 = gl; k0 < n; k0 += UNR * G) {
        int cc[UNR];
        float vv[UNR];
#pragma unroll
        for (int u = 0; u < UNR; ++u) {
          const int k = k0 + u * G;
          cc[u] = k < n ? (int)cols[k] : -1;
          vv[u] = k < n ? vals[k] : 0.f;
        }
#pragma unroll
        for (int u = 0; u < UNR; ++u) {
          const int ps = cc[u] >= 0 ? s.poolslot[cc[u]] : -1;
          if (ps >= 0) {
            rmax = fmaxf(rmax, vv[u] - bm);
#pragma unroll
            for (int t = 0; t < PCL; ++t)
              if (t == mine) {
                cv[t] = vv[u];
                cs[t] = ps;
              }
            spill |= mine >= PCL;
            ++mine;
          }
        }
      }
      rmax = group_max(rmax, gm);
      npool = group_sum(mine, gm);
      const bool any_spill = __any_sync(gm, spill);
      ncache = mine < PCL ? mine : PCL;
      if (npool > 0) {
        // softmax shifted by the row's largest logit (exponentials at most 1)
        const float tau = a.resp_temp * rmax + a.resp_eps;
        float z = 0.f;
        if (!any_spill) {
#pragma unroll
          for (int t = 0; t < PCL; ++t)
            if (t < ncache) z += expf(((cv[t] - bm) - rmax) / tau);
        } else {
          for (int k = gl; k < n; k += G)
            if (s.poolslot[cols[k]] >= 0) z += expf(((vals[k] - bm) - rmax) / tau);
        }
        z = group_sum(z, gm) + (float)(Pt - npool) * expf(-rmax / tau);  // R = 0 entries
        const float invz = 1.f / z;
        if (!any_spill) {
#pragma unroll
          for (int t = 0; t < PCL; ++t)
            if (t < ncache) {
              const float R = cv[t] - bm;
              atomicAdd(&s.sw[wid * Pt + cs[t]],
                        (unsigned long long)to_fix(expf((R - rmax) / tau) * invz * R, fxs));
            }
        } else {
          for (int k = gl; k < n; k += G) {
            const int ps = s.poolslot[cols[k]];
            if (ps >= 0) {
              const float R = vals[k] - bm;
              atomicAdd(&s.sw[wid * Pt + ps],
                        (unsigned long long)to_fix(expf((R - rmax) / tau) * invz * R, fxs));
            }
          }
        }
      }
    }
    }
    __syncthreads();
    if (!flat)
      for (int q = threadIdx.x; q < Pt * CS; q += blockDim.x) {  // (slot, target CTA) pairs
        const int k = q / CS, c = q - k * CS;
        unsigned long long v = 0;
        for (int w2 = 0; w2 < SEL_WARPS; ++w2) v += s.sw[w2 * Pt + k];
        if (v) score_push(k, v, c, CS);
      }
    cluster.sync();  // every CTA's scores have reached every CTA's s_acc, and every
                     // CTA has read this round's gains

    // ---- batch, coverage update, survivor filter, next gains ------------------
    const int nb = min(a.bsz, min(Pt, K - S_count));
    for (int k = gid; k < Pt; k += ngrp) {  // 8 lanes rank each pool token
      const int rank = sel::group_score_rank(s.s_acc, s.pool, Pt, k, gl, gm);
      if (gl == 0) {
        s.inb[k] = rank < nb;
        if (rank < nb) s.batch[rank] = s.pool[k];
      }
    }
    __syncthreads();
    for (int q = threadIdx.x; q < nb; q += blockDim.x) {
      s.sel[s.batch[q]] = 1;
      if (r == 0) a.order[(size_t)b * K + S_count + q] = s.batch[q];
    }
    if (r == 0 && a.tv.base && threadIdx.x == 0)
      a.tv.at<int32_t>(b, a.tv.off_round_end)[rnd] = S_count + nb;
    if (flat) {
      // coverage update: largest batch value per row, one 8-lane group per batch token
      for (int k = gid; k < nb; k += ngrp) {
        const int j = s.batch[k];
        for (int p = s.cstart[j] + gl; p < s.cstart[j + 1]; p += G) {
          const int q = s.srows[p];
          if (q != DEADROW) atomicMax(&s.bnb[q], __float_as_int(s.svals[p]));
        }
      }
      __syncthreads();
      for (int q = threadIdx.x; q < nrows; q += blockDim.x) {
        const float bn = fmaxf(s.bcov[q], __int_as_float(s.bnb[q]));
        s.bcov[q] = bn;
        s.bfold[q] = s.bfix[q];
        s.bfix[q] = to_fix(bn, fxs);
        s.bnb[q] = 0;
        s.rmaxb[q] = 0;
        s.npl[q] = 0;
        s.z64[q] = 0;
      }
      for (int j = threadIdx.x; j < N; j += blockDim.x) s.bnd[j] = 0;  // live entries per token
      __syncthreads();
      // survivor filter (dead entries marked in place) and the changes of the
      // gains: an entry's residual moves from C - b_old to C - b_new, or to zero
      // when it dies (exact: integers modulo 2^64; nothing for rows whose
      // coverage stayed).  Each thread walks a contiguous slice (an odd length
      // keeps a warp's threads on distinct banks) and sums every token's
      // changes in a register
      const int tot = s.scal[SC_CURSOR];
      const int per = ((tot + SEL_THREADS - 1) / SEL_THREADS) | 1;
      const int p0s = min(tot, (int)threadIdx.x * per), p1s = min(tot, p0s + per);
      int jc = -1, nj = 0, mylive = 0;
      unsigned long long acc = 0;
      for (int p0 = p0s; p0 < p1s; p0 += FU) {
        int qq[FU], jj[FU];
        float cc[FU];
#pragma unroll
        for (int u = 0; u < FU; ++u) {
          const bool in = p0 + u < p1s;
          qq[u] = in ? (int)s.srows[p0 + u] : DEADROW;
          jj[u] = in ? (int)s.scols[p0 + u] : 0;
          cc[u] = in ? s.svals[p0 + u] : 0.f;
        }
#pragma unroll
        for (int u = 0; u < FU; ++u) {
          if (qq[u] == DEADROW) continue;
          if (jj[u] != jc) {
            if (acc) gain_add(jc, acc, rnd);
            if (nj) atomicAdd(&s.bnd[jc], nj);
            jc = jj[u];
            acc = 0;
            nj = 0;
          }
          const int q = qq[u];
          if (cc[u] > s.bcov[q]) {
            acc += (unsigned long long)(s.bfold[q] - s.bfix[q]);
            ++nj;
            ++mylive;
          } else {
            acc += (unsigned long long)(s.bfold[q] - to_fix(cc[u], fxs));
            s.srows[p0 + u] = (uint16_t)DEADROW;
          }
        }
      }
      if (acc) gain_add(jc, acc, rnd);
      if (nj) atomicAdd(&s.bnd[jc], nj);
      // Every fourth round every CTA drops its dead entries: the live entries
      // move down in order (token-major order is kept) and the token segments
      // restart at the prefix sums of the live counts.  The same round in every
      // CTA: a compaction in one CTA alone would hold the others at the next
      // cluster barrier.
      int live = 0;
      block_exclusive_scan(mylive, s.wsum, &live);
      if (rnd % COMPACT_EVERY == 0 && live < tot) {  // live, tot: block-wide values
        {
          const int perj = (N + SEL_THREADS - 1) / SEL_THREADS;
          const int j0 = min(N, (int)threadIdx.x * perj), j1 = min(N, j0 + perj);
          int c = 0;
          for (int j = j0; j < j1; ++j) c += s.bnd[j];
          int at = block_exclusive_scan(c, s.wsum, nullptr);
          for (int j = j0; j < j1; ++j) {
            s.cstart[j] = at;
            at += s.bnd[j];
          }
          if (threadIdx.x == 0) s.cstart[N] = live;
        }
        // chunks of 32 CU entries per warp, entry seg + 32 u + lane read by
        // lane (bank-conflict free); ballots keep the order.  Every thread reads
        // before the scan's barriers and writes after them, always at or below
        // the source.
        int dst = 0;
        const unsigned lt = (1u << lane) - 1u;
        for (int base = 0; base < tot; base += SEL_THREADS * CU) {
          const int seg = base + wid * (32 * CU);
          uint16_t mq[CU], mj[CU];
          float mc[CU];
          unsigned bal[CU];
          int wcount = 0;
#pragma unroll
          for (int u = 0; u < CU; ++u) {
            const int p = seg + u * 32 + lane;
            const bool in = p < tot;
            mq[u] = in ? s.srows[p] : (uint16_t)DEADROW;
            mj[u] = in ? s.scols[p] : (uint16_t)0;
            mc[u] = in ? s.svals[p] : 0.f;
            bal[u] = __ballot_sync(FULL, mq[u] != DEADROW);
            wcount += __popc(bal[u]);
          }
          int chunk_live = 0;
          int off = dst + block_exclusive_scan(lane == 0 ? wcount : 0, s.wsum, &chunk_live);
          off = __shfl_sync(FULL, off, 0);
#pragma unroll
          for (int u = 0; u < CU; ++u) {
            if ((bal[u] >> lane) & 1u) {
              const int d = off + __popc(bal[u] & lt);
              s.srows[d] = mq[u];
              s.scols[d] = mj[u];
              s.svals[d] = mc[u];
            }
            off += __popc(bal[u]);
          }
          dst += chunk_live;
        }
        __syncthreads();
        if (threadIdx.x == 0) s.scal[SC_CURSOR] = dst;
      }
    }
    if (!flat) {
    for (int q0 = wid * (32 / G); q0 < nrows; q0 += nw * (32 / G)) {
      const int q = q0 + sub;
      const int n = q < nrows ? s.cnt[q] : 0;
      const float bm = q < nrows ? s.bcov[q] : 0.f;
      float* vals = Cimg + (size_t)grow(q) * N;
      uint16_t* cols = Simg + (size_t)grow(q) * N;
      float bnew = bm;
      for (int k0 = gl; k0 < n; k0 += UNR * G) {
        int cc[UNR];
        float vv[UNR];
#pragma unroll
        for (int u = 0; u < UNR; ++u) {
          const int k = k0 + u * G;
          cc[u] = k < n ? (int)cols[k] : -1;
          vv[u] = k < n ? vals[k] : 0.f;
        }
#pragma unroll
        for (int u = 0; u < UNR; ++u) {
          const int ps = cc[u] >= 0 ? s.poolslot[cc[u]] : -1;
          if (ps >= 0 && s.inb[ps]) bnew = fmaxf(bnew, vv[u]);
        }
      }
      bnew = group_max(bnew, gm);
      const long long fb_new = to_fix(bnew, fxs), fb_old = to_fix(bm, fxs);
      // a row whose coverage stayed keeps its list and changes no gain; in the
      // others an entry's residual moves from C - b_old to C - b_new, or to zero
      // when it dies (exact: integers modulo 2^64)
      const int nch = bnew > bm ? n : 0;  // uniform over the group
      int w = n - nch;
      for (int base = 0; base < nch; base += UNR * G) {
        float c[UNR];
        int jj[UNR];
#pragma unroll
        for (int u = 0; u < UNR; ++u) {
          const int k = base + u * G + gl;
          c[u] = k < n ? vals[k] : 0.f;
          jj[u] = k < n ? (int)cols[k] : 0;
        }
        __syncwarp(gm);  // the group has read all UNR*G entries before any overwrite
#pragma unroll
        for (int u = 0; u < UNR; ++u) {
          const int k = base + u * G + gl;
          const bool keep = k < n && c[u] > bnew;
          const unsigned msk = __ballot_sync(gm, keep);
          if (k < n) {
            const long long d = keep ? fb_old - fb_new : fb_old - to_fix(c[u], fxs);
            if (d) gain_add(jj[u], (unsigned long long)d, rnd);
          }
          if (keep) {
            const int pos = w + __popc(msk & lt);
            vals[pos] = c[u];
            cols[pos] = (uint16_t)jj[u];
          }
          w += __popc(msk);
        }
      }
      if (gl == 0 && q < nrows) {
        s.bcov[q] = bnew;
        s.cnt[q] = w;
      }
    }
    }
    __syncthreads();
    if (a.tv.base) {  // certificate input: F(S) after this round, this CTA's rows
      long long f = 0;
      for (int q = threadIdx.x; q < nrows; q += blockDim.x) f += to_fix(s.bcov[q], fxs);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) f += __shfl_xor_sync(FULL, f, o);
      if (lane == 0 && f) atomicAdd(a.tv.cover(b, rnd), (unsigned long long)f);
    }
    for (int k = threadIdx.x; k < Pt; k += blockDim.x) {
      s.poolslot[s.pool[k]] = -1;
      s.s_acc[k] = 0;
    }
    if (!flat) migrate();
    S_count += nb;
    ++rnd;
    if (S_count >= K) break;
    cluster.sync();  // every contribution to the new gains has reached its owner

    // ---- gains of the next round, read from their owners ----------------------
    // With a cluster and a boundary hint the pool's first pass reads them
    // (remote_gains); otherwise they are copied here.
    remote_gains = CS > 1;
    if (!remote_gains || phint < 0) {
      read_gains();
      remote_gains = false;
    }
  }

  // ---- final: coverage per bank, sorted support, trace ---------------------
  {
    long long f0 = 0, f1 = 0, f2 = 0;
    for (int q = threadIdx.x; q < nrows; q += blockDim.x) {
      const int m = grow(q);
      const long long v = to_fix(s.bcov[q], fxs);
      if (m < MG) f0 += v; else if (m < MG + N) f1 += v; else f2 += v;
    }
    long long* fb0 = cluster.map_shared_rank(s.fb, 0);
    if (f0) atomicAdd((unsigned long long*)&fb0[0], (unsigned long long)f0);
    if (f1) atomicAdd((unsigned long long*)&fb0[1], (unsigned long long)f1);
    if (f2) atomicAdd((unsigned long long*)&fb0[2], (unsigned long long)f2);
  }
  cluster.sync();
  if (r != 0) return;
  {  // the support in ascending token order: contiguous tokens per thread, one block scan
    const int per = (N + blockDim.x - 1) / blockDim.x;
    const int j0 = min(N, (int)threadIdx.x * per), j1 = min(N, j0 + per);
    int c = 0;
    for (int j = j0; j < j1; ++j) c += s.sel[j] ? 1 : 0;
    int cnt = 0;
    int pos = block_exclusive_scan(c, s.wsum, &cnt);
    for (int j = j0; j < j1; ++j) {
      const bool on = s.sel[j] != 0;
      a.slot[(size_t)b * N + j] = on ? pos : -1;
      if (on && pos < K) {
        a.support[(size_t)b * K + pos] = j;
        if (a.out_idx) a.out_idx[(size_t)b * K + pos] = j;
      }
      pos += on ? 1 : 0;
    }
    if (threadIdx.x == 0 && cnt != K) set_status(a.status, GMC_STATUS_INTERNAL);
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
        hd->F_V[q] = (float)((double)a.r0.fv[(size_t)b * 4 + q] * inv);
      }
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

// Batched certificate (Sec. 4.1 Eq. (6); appendix Eq. (cond-batched-bound)),
// computed only for the diagnostics trace from what the solver recorded there:
// round t's gains u^t and F(S) after it.  U_t, the sum of the K largest gains
// of the tokens not selected before round t, comes from the K-th largest gain
// theta (binary search on the fixed-point value, counting on the whole
// block): U_t = sum_{u > theta} u + (K - #{u > theta}) theta, exactly.
// c_B = 1 - prod_t (1 - q_t) over the rounds with U_t > 0,
// q_t = (F_t - F_{t-1}) / U_t.  One block per image.
__global__ void __launch_bounds__(256) k_certificate(int N, int K, TraceView tv) {
  grid_dep_wait();
  extern __shared__ __align__(16) char sm_cert[];
  long long* g = reinterpret_cast<long long*>(sm_cert);               // [N]
  unsigned char* done = reinterpret_cast<unsigned char*>(g + N);      // [N] selected before t
  __shared__ long long red[8];
  __shared__ unsigned long long red2[8];
  const int b = blockIdx.x;
  gmc_trace_header* hd = tv.header(b);
  const int R = hd->rounds;
  const int32_t* order = tv.at<int32_t>(b, tv.off_order);
  const int32_t* rend = tv.at<int32_t>(b, tv.off_round_end);
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  for (int j = threadIdx.x; j < N; j += blockDim.x) done[j] = 0;
  // block sum of (count, value) over the unselected tokens with g > x (or >= x)
  auto count_ge = [&](long long x) {
    long long c = 0;
    for (int j = threadIdx.x; j < N; j += blockDim.x) c += (!done[j] && g[j] >= x);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(FULL, c, o);
    __syncthreads();
    if (lane == 0) red[wid] = c;
    __syncthreads();
    long long t = 0;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) t += red[w];
    return t;
  };
  double prod = 1.0, Fprev = 0.0;
  const double inv = 1.0;  // q_t is a ratio of two fixed-point values: the scale cancels
  for (int t = 0; t < R; ++t) {
    __syncthreads();
    const int before = t > 0 ? rend[t - 1] : 0;
    for (int q = threadIdx.x; q < before; q += blockDim.x) done[order[q]] = 1;
    const long long* gt = tv.gains(b, t, N);
    for (int j = threadIdx.x; j < N; j += blockDim.x) g[j] = gt[j] < 0 ? 0 : gt[j];
    __syncthreads();
    // theta = the largest x with #{u >= x} >= K (0 when fewer than K tokens
    // remain).  Every gain is at most the fixed-point total mass, below 2^62, so
    // the search range [0, 2^62] halves in at most 63 steps
    long long lo = 0, hi = 1LL << 62;
    if (count_ge(0) >= K) {
      for (int it = 0; it < 64 && lo < hi; ++it) {
        const long long mid = lo + (hi - lo + 1) / 2;
        if (count_ge(mid) >= K) lo = mid; else hi = mid - 1;
      }
    }
    const long long theta = lo;
    // sum and count of the gains above theta
    unsigned long long sv = 0;
    long long cv = 0;
    for (int j = threadIdx.x; j < N; j += blockDim.x)
      if (!done[j] && g[j] > theta) {
        sv += (unsigned long long)g[j];
        ++cv;
      }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      sv += __shfl_xor_sync(FULL, sv, o);
      cv += __shfl_xor_sync(FULL, cv, o);
    }
    __syncthreads();
    if (lane == 0) {
      red2[wid] = sv;
      red[wid] = cv;
    }
    __syncthreads();
    unsigned long long S = 0;
    long long C = 0;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) {
      S += red2[w];
      C += red[w];
    }
    const long long remain = count_ge(0);
    const double U = remain >= K ? (double)S + (double)(K - C) * (double)theta : (double)S;
    const double F = (double)*tv.cover(b, t) * inv;
    if (U > 0.0) {
      prod *= 1.0 - (F - Fprev) / U;
      Fprev = F;
    }
  }
  if (threadIdx.x == 0) hd->c_B = (float)(1.0 - prod);
}

static int g_num_sms = 0;

static cudaError_t num_sms() {
  if (g_num_sms) return cudaSuccess;
  int dev = 0, n = 0;
  cudaError_t e;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
  if ((e = cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
    return e;
  if ((e = cudaFuncSetAttribute(k_select, cudaFuncAttributeNonPortableClusterSizeAllowed, 1)) !=
      cudaSuccess)
    return e;
  g_num_sms = n;
  return cudaSuccess;
}

// The largest cluster launch_select tries (images x CTAs within the SMs) has
// the smallest per-CTA state; the state of any smaller one is larger.
static int first_cluster_size(int B) {
  int CS = 1;
  while (CS * 2 <= SEL_MAX_CS && (long long)B * CS * 2 <= g_num_sms) CS *= 2;
  return CS;
}

bool select_fits(int B, int N, int M, int P) {
  if (num_sms() != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  const int CS = first_cluster_size(B);
  const int RPC = (M + CS - 1) / CS;
  const int gwords = (CS > 1 ? 2 : 1) * ((N + CS - 1) / CS);
  return sel_fixed_bytes(N, P, RPC, gwords, nullptr, nullptr) + 1024 <= SMEM_LIMIT;
}

cudaError_t launch_select(const R0State& r0, int B, int N, int K, int M, const int32_t* toff, int H, int T, int L2,
                          const gmc_params& p, int fx_exp, const int32_t* fexp, float* C,
                          uint16_t* scol, const long long* u0, int32_t* order, int32_t* support,
                          int32_t* slot, int32_t* out_idx, uint32_t* status, const TraceView& tv,
                          cudaStream_t st, int I) {
  cudaError_t e;
  if ((e = num_sms()) != cudaSuccess) return e;
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
  a.r0 = r0;
  a.images = I;
  for (int CS = first_cluster_size(B); CS >= 1; CS /= 2) {
    // Row capacity of one CTA: rows are dealt in turn, so ceil(M / CS) each
    const int RPC = (M + CS - 1) / CS;
    const int gwords = (CS > 1 ? 2 : 1) * ((N + CS - 1) / CS);
    const size_t fixed = sel_fixed_bytes(N, a.P, RPC, gwords, nullptr, nullptr);
    if (fixed + 1024 > SMEM_LIMIT) continue;
    a.rpc = RPC;
    // the rest of the shared memory holds survivor entries (value, token, row: 8 bytes)
    a.cap = (int)((SMEM_LIMIT - fixed - 16) / 8);
    a.cap &= ~7;
    const size_t smem = fixed + (size_t)a.cap * 8 + 16;
    if ((e = set_smem_limit((const void*)k_select, smem)) != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(B * CS);
    cfg.blockDim = dim3(SEL_THREADS);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
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
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;  // see grid_dep_wait
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.numAttrs = 2;
    if ((e = cudaLaunchKernelEx(&cfg, k_select, a)) != cudaSuccess || !tv.base) return e;
    // diagnostics trace: the batched certificate from the recorded rounds
    return launch_certificate(B, N, K, tv, st);
  }
  return cudaErrorInvalidConfiguration;
}

cudaError_t launch_certificate(int B, int N, int K, const TraceView& tv, cudaStream_t st) {
  const size_t csm = (sizeof(long long) + 1) * (size_t)N;
  cudaError_t e;
  if ((e = set_smem_limit((const void*)k_certificate, csm)) != cudaSuccess) return e;
  launch_k(k_certificate, B, 256, csm, st, 1, N, K, tv);
  return cudaGetLastError();
}

}  // namespace gmc
