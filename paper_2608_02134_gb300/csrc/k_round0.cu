// The first (dense) round of the batched responsibility solver (Eq. (4)) over
// the whole GPU.  With S empty, b_m = 0 and the gains are the column sums of
// Cbar (computed while the clients were built).  Three kernels:
//   k_r0_pool   one block per image: the pool of the largest gains;
//   k_r0_rho    warp per client row: responsibilities over the pool, summed
//               into the scores in 64-bit fixed point (global atomics);
//   k_r0_filter warp per client row: the batch (top scores), the coverage
//               b_m = max over the batch, and the row's survivors
//               {i : Cbar_mi > b_m} compacted in place; the next round's gains
//               are summed in fixed point (global atomics).
// The next sparse_gpu_rounds(N) rounds run the same three steps over the survivor
// lists left in place by the previous round (row m: values Cbar[m][0..cnt_m),
// tokens scol[m][0..cnt_m), ascending):
//   k_rg_pool   the pool of the current gains among the unselected tokens;
//   k_rg_rho    warp per row: the row's pool entries are found through a
//               token -> pool slot table; pool tokens without a survivor in
//               the row have R = 0 and still count in its softmax denominator;
//   k_rg_filter warp per row: batch, coverage over the batch's entries, the
//               survivors compacted in place, the next gains.
// While many survivors remain, a whole-GPU round is cheaper than a round of
// the cluster kernel (16 SMs).  Every reduction is an integer sum, so the
// result does not depend on the order blocks run in.  The cluster kernel
// (k_select) continues from the first round not done here; info[b] carries the
// pool size, the tokens selected so far and the rounds done.
#include "common.cuh"
#include "kernels.cuh"
#include "select_common.cuh"

namespace gmc {

namespace {
// Warps per block of the responsibility and filter kernels (ROWS, a template
// parameter: 16 for one image, 8 for a batch; the responsibility kernels take
// one row per warp).  The filters take `rpw` rows per warp (rows m0 + w +
// ROWS * i).  More rows
// per block mean fewer global atomics for the next gains (one per block and
// column) but less parallelism: one row per warp is faster while the blocks
// fit on the GPU at once, four when there are many more blocks than that.
int filter_rows_per_warp(int B, int M, int rows) {
  static int sms = 0;
  if (sms == 0) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
      cudaGetLastError();
      sms = 152;
    }
  }
  const long long blocks = (long long)B * ceil_div(M, rows);
  return blocks > 32LL * sms ? 4 : 1;
}
}

__global__ void __launch_bounds__(512) k_r0_pool(const long long* __restrict__ u0, int B, int N,
                                                   int P, const int32_t* toff, int Tmax, int I,
                                                   int32_t* pool0, int32_t* info, long long* s0,
                                                   long long* u1, long long* fv, uint32_t* status,
                                                   TraceView tv) {
  grid_dep_wait();
  extern __shared__ __align__(16) char sm_r0p[];
  const int b = blockIdx.x;
  // the accumulators of the next two kernels start at zero; nothing selected yet
  for (int k = threadIdx.x; k < P; k += blockDim.x) s0[(size_t)b * P + k] = 0;
  for (int j = threadIdx.x; j < N; j += blockDim.x) u1[(size_t)b * N + j] = 0;
  if (threadIdx.x < 4) fv[(size_t)b * 4 + threadIdx.x] = 0;
  if (threadIdx.x == 0) {
    info[b * INFO_W + 1] = 0;
    info[b * INFO_W + 2] = 0;
    info[b * INFO_W + 3] = 0;
    info[b * INFO_W + 4] = 0;
    info[b * INFO_W + 5] = -1;  // boundary bucket of the last pool: none yet
  }
  if (toff && text_geom(toff, b, B, Tmax, nullptr).T == 0) {
    if (threadIdx.x == 0) info[b * INFO_W] = 0;
    return;
  }
  sel::PoolScratch w{};  // gains in shared memory: no boundary staging
  char* p = sm_r0p;
  long long* ug = reinterpret_cast<long long*>(p);  p += sizeof(long long) * (size_t)N;
  w.hist = reinterpret_cast<int*>(p);       p += sizeof(int) * sel::HBINS;
  w.bnd = reinterpret_cast<int*>(p);        p += sizeof(int) * N;
  w.wsum = reinterpret_cast<int*>(p);       p += sizeof(int) * 32;
  w.scal = reinterpret_cast<int*>(p);       p += sizeof(int) * 8;
  w.coarse = reinterpret_cast<int*>(p);     p += sizeof(int) * sel::CBINS;
  int* pool = reinterpret_cast<int*>(p);    p += sizeof(int) * P;
  w.key = reinterpret_cast<short*>(p);     p += sizeof(short) * (size_t)N;
  w.pk = reinterpret_cast<unsigned char*>(p); p += (size_t)N;
  unsigned char* selz = reinterpret_cast<unsigned char*>(p);
  for (int j = threadIdx.x; j < N; j += blockDim.x) {
    selz[j] = 0;
    ug[j] = u0[(size_t)b * N + j];  // the gains in shared memory: select_pool reads them often
    if (tv.base) tv.gains(b, 0, N)[j] = ug[j];
  }
  for (int h = threadIdx.x; h < sel::HBINS; h += blockDim.x) w.hist[h] = 0;
  if (threadIdx.x < sel::CBINS) w.coarse[threadIdx.x] = 0;
  __syncthreads();
  if (I > 1) {
    // several images: the first round only seeds S with each image's token of
    // largest singleton gain (ties to the lower index), one warp per image;
    // the filter takes them as its batch
    const int lane = threadIdx.x & 31, Ng = N / I;
    for (int k = threadIdx.x >> 5; k < I; k += blockDim.x >> 5) {
      long long bv = -1;
      int bj = 0x7fffffff;
      for (int j = k * Ng + lane; j < (k + 1) * Ng; j += 32)
        if (ug[j] > bv) {  // j ascending within a lane: the first maximum is kept
          bv = ug[j];
          bj = j;
        }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const long long ov = __shfl_xor_sync(FULL, bv, o);
        const int oj = __shfl_xor_sync(FULL, bj, o);
        if (ov > bv || (ov == bv && oj < bj)) {
          bv = ov;
          bj = oj;
        }
      }
      if (lane == 0) pool0[(size_t)b * P + k] = bj;
    }
    for (int k = I + threadIdx.x; k < P; k += blockDim.x) pool0[(size_t)b * P + k] = -1;
    if (threadIdx.x == 0) info[b * INFO_W] = I;
    return;
  }
  int bstar = -1;
  const int Pt = sel::select_pool(ug, selz, N, P, w, pool, nullptr, nullptr, &bstar);
  for (int k = threadIdx.x; k < P; k += blockDim.x) pool0[(size_t)b * P + k] = k < Pt ? pool[k] : -1;
  if (threadIdx.x == 0) {
    info[b * INFO_W] = Pt;
    info[b * INFO_W + 5] = bstar;
  }
}

template <int ROWS>
__global__ void __launch_bounds__(32 * ROWS) k_r0_rho(
    const float* __restrict__ C, int B, int N, int Mstride, int H, int L2, const int32_t* toff,
    int Tmax, int uniform_rows, const int32_t* __restrict__ pool0, const int32_t* __restrict__ info,
    int P, float resp_temp, float resp_eps, int fx_exp, const int32_t* fexp, int I, long long* s0) {
  grid_dep_wait();
  if (I > 1) return;  // a seed round: no responsibilities
  __shared__ int pool[GMC_MAX_POOL];
  __shared__ long long sblk[GMC_MAX_POOL];
  const int b = blockIdx.y;
  const int Pt = info[b * INFO_W];
  if (Pt == 0) return;
  int Mb = Mstride;
  if (!uniform_rows) Mb = H * text_geom(toff, b, B, Tmax, nullptr).T + N + L2;
  const int m0 = blockIdx.x * ROWS;
  if (m0 >= Mb) return;
  const float fxs = ldexpf(1.f, fexp ? fexp[b] : fx_exp);
  for (int k = threadIdx.x; k < P; k += blockDim.x) {
    pool[k] = pool0[(size_t)b * P + k];
    sblk[k] = 0;
  }
  __syncthreads();
  const int lane = threadIdx.x & 31, m = m0 + (threadIdx.x >> 5);
  if (m < Mb) {
    const float* row = C + ((size_t)b * Mstride + m) * N;
    float Rd[GMC_MAX_POOL / 32];
    float rmax = 0.f;
    int npool = 0;
#pragma unroll
    for (int u = 0; u < GMC_MAX_POOL / 32; ++u) {
      const int k = lane + 32 * u;
      Rd[u] = k < Pt ? row[pool[k]] : 0.f;  // b = 0: the residual is the client value
      if (Rd[u] > 0.f) { rmax = fmaxf(rmax, Rd[u]); ++npool; }
    }
    rmax = warp_max(rmax);
    npool = warp_sum_int(npool);
    if (npool > 0) {
      // softmax of R / tau shifted by its largest logit rmax / tau: every
      // exponential is at most 1, whatever resp_temp
      const float tau = resp_temp * rmax + resp_eps;
      const float e0 = expf(-rmax / tau);  // a pool token with R = 0
      float z = 0.f;
#pragma unroll
      for (int u = 0; u < GMC_MAX_POOL / 32; ++u)
        if (Rd[u] > 0.f) z += expf((Rd[u] - rmax) / tau);
      z = warp_sum(z) + (float)(Pt - npool) * e0;
      const float invz = 1.f / z;
#pragma unroll
      for (int u = 0; u < GMC_MAX_POOL / 32; ++u)
        if (Rd[u] > 0.f)
          atomicAdd((unsigned long long*)&sblk[lane + 32 * u],
                    (unsigned long long)to_fix(expf((Rd[u] - rmax) / tau) * invz * Rd[u], fxs));
    }
  }
  __syncthreads();
  for (int k = threadIdx.x; k < Pt; k += blockDim.x)
    if (sblk[k]) atomicAdd((unsigned long long*)&s0[(size_t)b * P + k], (unsigned long long)sblk[k]);
}

template <int ROWS>
__global__ void __launch_bounds__(32 * ROWS) k_r0_filter(
    float* C, uint16_t* scol, int B, int N, int K, int Mstride, int H, int L2,
    const int32_t* toff, int Tmax, int uniform_rows, const int32_t* __restrict__ pool0,
    int32_t* info, const long long* __restrict__ s0, int P, int bsz, int fx_exp,
    const int32_t* fexp, long long* u1, float* bcov, int32_t* cnt, long long* fv,
    int32_t* order, int rpw, int I, TraceView tv) {
  grid_dep_wait();
  __shared__ int pool[GMC_MAX_POOL];
  __shared__ long long sc[GMC_MAX_POOL];
  __shared__ int batch[GMC_MAX_POOL];
  __shared__ long long fb[3];
  // the block's contributions to the next gains, one global atomic per column at the end
  extern __shared__ unsigned long long uacc[];  // [N]
  const int b = blockIdx.y;
  const int Pt = info[b * INFO_W];
  if (Pt == 0) return;
  int Mb = Mstride, MG = Mstride;
  if (!uniform_rows) {
    MG = H * text_geom(toff, b, B, Tmax, nullptr).T;
    Mb = MG + N + L2;
  }
  const int m0 = blockIdx.x * ROWS * rpw;
  if (m0 >= Mb) return;
  const float fxs = ldexpf(1.f, fexp ? fexp[b] : fx_exp);
  const int nb = I > 1 ? Pt : min(bsz, min(Pt, K));  // a seed round takes its whole pool
  for (int k = threadIdx.x; k < Pt; k += blockDim.x) {
    pool[k] = pool0[(size_t)b * P + k];
    sc[k] = s0[(size_t)b * P + k];
  }
  if (threadIdx.x < 3) fb[threadIdx.x] = 0;
  for (int j = threadIdx.x; j < N; j += blockDim.x) uacc[j] = 0;
  __syncthreads();
  {
    const int lane = threadIdx.x & 31, gl = lane & 7;
    const unsigned gm = 0xFFu << (lane & 24);
    for (int k = threadIdx.x >> 3; k < Pt; k += blockDim.x >> 3) {  // 8 lanes per pool token
      const int rank = I > 1 ? k : sel::group_score_rank(sc, pool, Pt, k, gl, gm);
      if (gl == 0 && rank < nb) batch[rank] = pool[k];
    }
  }
  __syncthreads();
  if (blockIdx.x == 0) {  // record the first batch once per image
    for (int q = threadIdx.x; q < nb; q += blockDim.x) order[(size_t)b * K + q] = batch[q];
    if (threadIdx.x == 0) {
      info[b * INFO_W + 1] = nb;  // selected so far
      info[b * INFO_W + 2] = 1;   // rounds done
    }
    if (tv.base) {
      int32_t* tp = tv.at<int32_t>(b, tv.off_pool);
      for (int k = threadIdx.x; k < tv.pool_size; k += blockDim.x) tp[k] = k < Pt ? pool[k] : -1;
      if (threadIdx.x == 0) tv.at<int32_t>(b, tv.off_round_end)[0] = nb;
    }
  }
  const int lane = threadIdx.x & 31;
  for (int ir = 0; ir < rpw; ++ir) {
    const int m = m0 + (threadIdx.x >> 5) + ROWS * ir;
    if (m >= Mb) break;
    float* vals = C + ((size_t)b * Mstride + m) * N;
    uint16_t* cols = scol + ((size_t)b * Mstride + m) * N;
    float bnew = 0.f;
    for (int t = lane; t < nb; t += 32) bnew = fmaxf(bnew, vals[batch[t]]);
    bnew = warp_max(bnew);
    const long long fb_new = to_fix(bnew, fxs);
    int w = 0;
    float rowmax = 0.f;
    const unsigned lt = sel::lanemask_lt();
    if ((N & 3) == 0) {
      // 32 lanes x 8 float4 = 1024 columns per step; all loads issued before any
      // survivor is written back in place
      const float4* row4 = reinterpret_cast<const float4*>(vals);
      const int n4 = N >> 2;
      for (int base4 = 0; base4 < n4; base4 += 32 * 8) {
        float4 buf[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const int k4 = base4 + u * 32 + lane;
          buf[u] = k4 < n4 ? row4[k4] : make_float4(0.f, 0.f, 0.f, 0.f);
        }
        __syncwarp();
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const int k4 = base4 + u * 32 + lane;
          const float c4[4] = {buf[u].x, buf[u].y, buf[u].z, buf[u].w};
          // survivors before this lane's: one ballot per element of the float4
          int pre = 0, tot = 0;
#pragma unroll
          for (int e2 = 0; e2 < 4; ++e2) {
            rowmax = fmaxf(rowmax, c4[e2]);
            const unsigned bal = __ballot_sync(FULL, k4 < n4 && c4[e2] > bnew);
            pre += __popc(bal & lt);
            tot += __popc(bal);
          }
          int pos = w + pre;
          if (k4 < n4) {
#pragma unroll
            for (int e2 = 0; e2 < 4; ++e2)
              if (c4[e2] > bnew) {
                const int j = 4 * k4 + e2;
                vals[pos] = c4[e2];
                cols[pos] = (uint16_t)j;
                atomicAdd(&uacc[j], (unsigned long long)(to_fix(c4[e2], fxs) - fb_new));
                ++pos;
              }
          }
          w += tot;
        }
        __syncwarp();
      }
    } else {
      for (int base = 0; base < N; base += 32) {
        const int k = base + lane;
        const float c = k < N ? vals[k] : 0.f;
        rowmax = fmaxf(rowmax, c);
        const bool keep = k < N && c > bnew;
        const unsigned msk = __ballot_sync(FULL, keep);
        __syncwarp();
        if (keep) {
          const int pos = w + __popc(msk & sel::lanemask_lt());
          vals[pos] = c;
          cols[pos] = (uint16_t)k;
          atomicAdd(&uacc[k], (unsigned long long)(to_fix(c, fxs) - fb_new));
        }
        w += __popc(msk);
      }
    }
    rowmax = warp_max(rowmax);
    if (lane == 0) {
      bcov[(size_t)b * Mstride + m] = bnew;
      cnt[(size_t)b * Mstride + m] = w;
      const int bank = m < MG ? 0 : (m < MG + N ? 1 : 2);
      atomicAdd((unsigned long long*)&fb[bank], (unsigned long long)to_fix(rowmax, fxs));
      if (tv.base) atomicAdd(tv.cover(b, 0), (unsigned long long)fb_new);  // F after the round
    }
  }
  __syncthreads();
  if (threadIdx.x < 3 && fb[threadIdx.x])
    atomicAdd((unsigned long long*)&fv[(size_t)b * 4 + threadIdx.x], (unsigned long long)fb[threadIdx.x]);
  unsigned long long* ub = reinterpret_cast<unsigned long long*>(u1 + (size_t)b * N);
  for (int j = threadIdx.x; j < N; j += blockDim.x)
    if (uacc[j]) atomicAdd(&ub[j], uacc[j]);
}

// ---- sparse rounds on the whole GPU -------------------------------------------

__global__ void __launch_bounds__(512) k_rg_pool(const long long* __restrict__ ucur,
                                                   long long* unext, int B, int N, int K, int P,
                                                   const int32_t* toff, int Tmax,
                                                   const int32_t* __restrict__ order,
                                                   int32_t* pool0, int32_t* info, long long* sc,
                                                   TraceView tv) {
  grid_dep_wait();
  extern __shared__ __align__(16) char sm_rgp[];
  const int b = blockIdx.x;
  for (int k = threadIdx.x; k < P; k += blockDim.x) sc[(size_t)b * P + k] = 0;
  // the next gains start from these: the filter adds only the changes of the
  // rows whose coverage grows
  for (int j = threadIdx.x; j < N; j += blockDim.x) unext[(size_t)b * N + j] = ucur[(size_t)b * N + j];
  const int S = info[b * INFO_W + 1], rd = info[b * INFO_W + 2];
  // nothing to do here once the budget is met or when the first round found
  // no gain: the cluster kernel handles those cases
  const bool skip = (toff && text_geom(toff, b, B, Tmax, nullptr).T == 0) || rd == 0 || S >= K;
  if (skip) {
    if (threadIdx.x == 0) info[b * INFO_W] = 0;
    return;
  }
  sel::PoolScratch w{};  // gains in shared memory: no boundary staging
  char* p = sm_rgp;
  sel::WindowScratch ws;
  ws.win = reinterpret_cast<int*>(p);       p += sizeof(int) * (sel::WBINS + 4);
  ws.cu = reinterpret_cast<long long*>(p);  p += sizeof(long long) * sel::WCAP;
  ws.cj = reinterpret_cast<int*>(p);        p += sizeof(int) * sel::WCAP;
  long long* ug = reinterpret_cast<long long*>(p);  p += sizeof(long long) * (size_t)N;
  w.hist = reinterpret_cast<int*>(p);       p += sizeof(int) * sel::HBINS;
  w.bnd = reinterpret_cast<int*>(p);        p += sizeof(int) * N;
  w.wsum = reinterpret_cast<int*>(p);       p += sizeof(int) * 32;
  w.scal = reinterpret_cast<int*>(p);       p += sizeof(int) * 8;
  w.coarse = reinterpret_cast<int*>(p);     p += sizeof(int) * sel::CBINS;
  int* pool = reinterpret_cast<int*>(p);    p += sizeof(int) * P;
  w.key = reinterpret_cast<short*>(p);     p += sizeof(short) * (size_t)N;
  w.pk = reinterpret_cast<unsigned char*>(p); p += (size_t)N;
  unsigned char* self = reinterpret_cast<unsigned char*>(p);
  // the gains in shared memory (select_pool reads them often): copied here
  // without a boundary hint, else by the window pool's first pass
  int hint = info[b * INFO_W + 5];
  const long long* ub = ucur + (size_t)b * N;
  for (int j = threadIdx.x; j < N; j += blockDim.x) {
    self[j] = 0;
    if (hint < 0) ug[j] = ub[j];
  }
  for (int h = threadIdx.x; h < sel::HBINS; h += blockDim.x) w.hist[h] = 0;
  if (threadIdx.x < sel::CBINS) w.coarse[threadIdx.x] = 0;
  for (int q = threadIdx.x; q < sel::WBINS + 4; q += blockDim.x) ws.win[q] = 0;
  __syncthreads();
  for (int q = threadIdx.x; q < S; q += blockDim.x) self[order[(size_t)b * K + q]] = 1;
  __syncthreads();
  int Pt = sel::select_pool_window([&](int j) { return ub[j]; }, ug, self, N, P, ws, pool,
                                   nullptr, &hint);
  if (Pt < 0) Pt = sel::select_pool(ug, self, N, P, w, pool, nullptr, nullptr, &hint);
  if (tv.base)
    for (int j = threadIdx.x; j < N; j += blockDim.x) tv.gains(b, rd, N)[j] = ug[j];
  for (int k = threadIdx.x; k < P; k += blockDim.x) pool0[(size_t)b * P + k] = k < Pt ? pool[k] : -1;
  if (threadIdx.x == 0) {
    info[b * INFO_W + 5] = hint;
    info[b * INFO_W] = Pt;
    info[b * INFO_W + 3] = S;
    info[b * INFO_W + 4] = rd;
  }
  if (tv.base && Pt > 0) {
    int32_t* tp = tv.at<int32_t>(b, tv.off_pool) + (size_t)rd * tv.pool_size;
    for (int k = threadIdx.x; k < tv.pool_size; k += blockDim.x) tp[k] = k < Pt ? pool[k] : -1;
  }
}

template <int ROWS>
__global__ void __launch_bounds__(32 * ROWS) k_rg_rho(
    const float* __restrict__ C, const uint16_t* __restrict__ scol,
    const float* __restrict__ bcov, const int32_t* __restrict__ cnt, int B, int N, int Mstride,
    int H, int L2, const int32_t* toff, int Tmax, int uniform_rows,
    const int32_t* __restrict__ pool0, const int32_t* __restrict__ info, int P, float resp_temp,
    float resp_eps, int fx_exp, const int32_t* fexp, long long* sc) {
  grid_dep_wait();
  __shared__ long long sblk[GMC_MAX_POOL];
  __shared__ int fslot[ROWS][GMC_MAX_POOL];  // a row's pool entries: slot and residual
  __shared__ float fres[ROWS][GMC_MAX_POOL];
  extern __shared__ short pslot[];              // [N] pool slot of every token or -1
  const int b = blockIdx.y;
  const int Pt = info[b * INFO_W];
  if (Pt == 0) return;
  int Mb = Mstride;
  if (!uniform_rows) Mb = H * text_geom(toff, b, B, Tmax, nullptr).T + N + L2;
  const int m0 = blockIdx.x * ROWS;
  if (m0 >= Mb) return;
  const float fxs = ldexpf(1.f, fexp ? fexp[b] : fx_exp);
  for (int j = threadIdx.x; j < N; j += blockDim.x) pslot[j] = -1;
  for (int k = threadIdx.x; k < P; k += blockDim.x) sblk[k] = 0;
  __syncthreads();
  for (int k = threadIdx.x; k < Pt; k += blockDim.x) pslot[pool0[(size_t)b * P + k]] = (short)k;
  __syncthreads();
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, m = m0 + w;
  if (m < Mb) {
    const size_t row = (size_t)b * Mstride + m;
    const int n = cnt[row];
    const float bm = bcov[row];
    const float* vals = C + row * N;
    const uint16_t* cols = scol + row * N;
    const unsigned lt = sel::lanemask_lt();
    int nf = 0;
    float rmax = 0.f;
    constexpr int RU = 4;  // chunks of 32 entries whose loads are in flight together
    for (int e00 = 0; e00 < n; e00 += 32 * RU) {
      int ps[RU];
      float R[RU];
#pragma unroll
      for (int u = 0; u < RU; ++u) {
        const int e = e00 + 32 * u + lane;
        ps[u] = e < n ? (int)cols[e] : -1;
      }
#pragma unroll
      for (int u = 0; u < RU; ++u) {
        if (ps[u] >= 0) ps[u] = pslot[ps[u]];
        R[u] = ps[u] >= 0 ? vals[e00 + 32 * u + lane] - bm : 0.f;  // > 0: exceeds its coverage
      }
#pragma unroll
      for (int u = 0; u < RU; ++u) {
        const unsigned bal = __ballot_sync(FULL, ps[u] >= 0);
        if (ps[u] >= 0) {
          const int at = nf + __popc(bal & lt);
          fslot[w][at] = ps[u];
          fres[w][at] = R[u];
          rmax = fmaxf(rmax, R[u]);
        }
        nf += __popc(bal);
      }
    }
    rmax = warp_max(rmax);
    __syncwarp();
    if (nf > 0) {
      // softmax shifted by the largest logit (exponentials at most 1)
      const float tau = resp_temp * rmax + resp_eps;
      const float e0 = expf(-rmax / tau);  // pool tokens without a survivor here: R = 0
      float z = 0.f;
      for (int q = lane; q < nf; q += 32) z += expf((fres[w][q] - rmax) / tau);
      z = warp_sum(z) + (float)(Pt - nf) * e0;
      const float invz = 1.f / z;
      for (int q = lane; q < nf; q += 32) {
        const float R = fres[w][q];
        atomicAdd((unsigned long long*)&sblk[fslot[w][q]],
                  (unsigned long long)to_fix(expf((R - rmax) / tau) * invz * R, fxs));
      }
    }
  }
  __syncthreads();
  for (int k = threadIdx.x; k < Pt; k += blockDim.x)
    if (sblk[k]) atomicAdd((unsigned long long*)&sc[(size_t)b * P + k], (unsigned long long)sblk[k]);
}

template <int ROWS>
__global__ void __launch_bounds__(32 * ROWS) k_rg_filter(
    float* C, uint16_t* scol, int B, int N, int K, int Mstride, int H, int L2,
    const int32_t* toff, int Tmax, int uniform_rows, const int32_t* __restrict__ pool0,
    int32_t* info, const long long* __restrict__ sc0, int P, int bsz, int fx_exp,
    const int32_t* fexp, long long* unext, float* bcov, int32_t* cnt, int32_t* order, int rpw,
    TraceView tv) {
  grid_dep_wait();
  __shared__ int pool[GMC_MAX_POOL];
  __shared__ long long sc[GMC_MAX_POOL];
  __shared__ int batch[GMC_MAX_POOL];
  extern __shared__ unsigned long long uacc[];  // [N] then the batch flags [N] (bytes)
  unsigned char* inb = reinterpret_cast<unsigned char*>(uacc + N);
  const int b = blockIdx.y;
  const int Pt = info[b * INFO_W];
  if (Pt == 0) return;
  int Mb = Mstride;
  if (!uniform_rows) Mb = H * text_geom(toff, b, B, Tmax, nullptr).T + N + L2;
  const int m0 = blockIdx.x * ROWS * rpw;
  if (m0 >= Mb) return;
  const int S = info[b * INFO_W + 3], rd = info[b * INFO_W + 4];
  const float fxs = ldexpf(1.f, fexp ? fexp[b] : fx_exp);
  const int nb = min(bsz, min(Pt, K - S));
  for (int k = threadIdx.x; k < Pt; k += blockDim.x) {
    pool[k] = pool0[(size_t)b * P + k];
    sc[k] = sc0[(size_t)b * P + k];
  }
  for (int j = threadIdx.x; j < N; j += blockDim.x) {
    uacc[j] = 0;
    inb[j] = 0;
  }
  __syncthreads();
  {
    const int lane = threadIdx.x & 31, gl = lane & 7;
    const unsigned gm = 0xFFu << (lane & 24);
    for (int k = threadIdx.x >> 3; k < Pt; k += blockDim.x >> 3) {  // 8 lanes per pool token
      const int rank = sel::group_score_rank(sc, pool, Pt, k, gl, gm);
      if (gl == 0 && rank < nb) batch[rank] = pool[k];
    }
  }
  __syncthreads();
  for (int q = threadIdx.x; q < nb; q += blockDim.x) inb[batch[q]] = 1;
  if (blockIdx.x == 0) {  // record the batch once per image
    for (int q = threadIdx.x; q < nb; q += blockDim.x) order[(size_t)b * K + S + q] = batch[q];
    if (threadIdx.x == 0) {
      info[b * INFO_W + 1] = S + nb;
      info[b * INFO_W + 2] = rd + 1;
      if (tv.base) tv.at<int32_t>(b, tv.off_round_end)[rd] = S + nb;
    }
  }
  __syncthreads();
  const int lane = threadIdx.x & 31;
  for (int ir = 0; ir < rpw; ++ir) {
    const int m = m0 + (threadIdx.x >> 5) + ROWS * ir;
    if (m >= Mb) break;
    const size_t row = (size_t)b * Mstride + m;
    const int n = cnt[row];
    float* vals = C + row * N;
    uint16_t* cols = scol + row * N;
    // The list is walked FU chunks of 32 entries at a time, every load of the
    // chunks issued before the first use (and, below, before any survivor is
    // written back in place: a chunk's survivors land below its end).
    constexpr int FU = 4;
    const float bold = bcov[row];
    float bnew = bold;
    for (int e00 = 0; e00 < n; e00 += 32 * FU) {
      int jj[FU];
#pragma unroll
      for (int u = 0; u < FU; ++u) {
        const int e = e00 + 32 * u + lane;
        jj[u] = e < n ? (int)cols[e] : -1;
      }
#pragma unroll
      for (int u = 0; u < FU; ++u)
        if (jj[u] >= 0 && inb[jj[u]]) bnew = fmaxf(bnew, vals[e00 + 32 * u + lane]);
    }
    bnew = warp_max(bnew);
    const long long fb_new = to_fix(bnew, fxs);
    if (!(bnew > bold)) {  // no batch entry above the coverage: row and gains unchanged
      if (lane == 0 && tv.base) atomicAdd(tv.cover(b, rd), (unsigned long long)fb_new);
      continue;
    }
    const long long fb_old = to_fix(bold, fxs);
    const unsigned lt = sel::lanemask_lt();
    int wr = 0;
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
      __syncwarp();  // the chunks are read before any survivor moves down into them
#pragma unroll
      for (int u = 0; u < FU; ++u) {
        const bool in = e00 + 32 * u + lane < n;
        const bool keep = in && cc[u] > bnew;
        const unsigned bal = __ballot_sync(FULL, keep);
        // the entry's residual moves from C - b_old to C - b_new, or to zero
        // (exact: integers modulo 2^64)
        if (in)
          atomicAdd(&uacc[jj[u]], (unsigned long long)(keep ? fb_old - fb_new
                                                             : fb_old - to_fix(cc[u], fxs)));
        if (keep) {
          const int pos = wr + __popc(bal & lt);
          vals[pos] = cc[u];
          cols[pos] = (uint16_t)jj[u];
        }
        wr += __popc(bal);
      }
    }
    if (lane == 0) {
      bcov[row] = bnew;
      cnt[row] = wr;
      if (tv.base) atomicAdd(tv.cover(b, rd), (unsigned long long)fb_new);  // F after the round
    }
  }
  __syncthreads();
  unsigned long long* ub = reinterpret_cast<unsigned long long*>(unext + (size_t)b * N);
  for (int j = threadIdx.x; j < N; j += blockDim.x)
    if (uacc[j]) atomicAdd(&ub[j], uacc[j]);
}

// The responsibility and filter launches of every whole-GPU round, ROWS rows per block.
template <int ROWS>
static cudaError_t launch_rounds_rows(const R0State& r0, int B, int N, int K, int M,
                                      const int32_t* toff, int H, int T, int L2,
                                      const gmc_params& p, int fx_exp, const int32_t* fexp,
                                      float* C, uint16_t* scol, int32_t* order, const TraceView& tv,
                                      cudaStream_t st, int I, size_t smem) {
  const int P = p.pool_mult * p.batch_b;
  const int uniform = (H == 0);
  cudaError_t e;
  dim3 grid(ceil_div(M, ROWS), B);
  launch_k(k_r0_rho<ROWS>, grid, 32 * ROWS, 0, st, 1, C, B, N, M, H, L2, toff, T, uniform, r0.pool,
           r0.info, P, p.resp_temp, p.resp_eps, fx_exp, fexp, I, r0.s0);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  const size_t fsm = sizeof(unsigned long long) * (size_t)N;
  if ((e = set_smem_limit((const void*)k_r0_filter<ROWS>, fsm)) != cudaSuccess) return e;
  const int rpw = filter_rows_per_warp(B, M, ROWS);
  const dim3 fgrid(ceil_div(M, ROWS * rpw), B);
  launch_k(k_r0_filter<ROWS>, fgrid, 32 * ROWS, fsm, st, 1, C, scol, B, N, K, M, H, L2, toff, T,
           uniform, r0.pool, r0.info, r0.s0, P, p.batch_b, fx_exp, fexp, r0.u1, r0.bcov, r0.cnt,
           r0.fv, order, rpw, I, tv);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  // sparse rounds: gains alternate between u1 and u2
  // the pool kernel's layout is round 0's after the window scratch
  const size_t psm = smem + sizeof(int) * (sel::WBINS + 4) + 12 * (size_t)sel::WCAP;
  if ((e = set_smem_limit((const void*)k_rg_pool, psm)) != cudaSuccess) return e;
  const size_t rsm = sizeof(short) * (size_t)N;
  if ((e = set_smem_limit((const void*)k_rg_rho<ROWS>, rsm)) != cudaSuccess) return e;
  const size_t gsm = sizeof(unsigned long long) * (size_t)N + (size_t)N;
  if ((e = set_smem_limit((const void*)k_rg_filter<ROWS>, gsm)) != cudaSuccess) return e;
  for (int rr = 1; rr <= sparse_gpu_rounds(N); ++rr) {
    long long* ucur = rr % 2 == 1 ? r0.u1 : r0.u2;
    long long* unext = rr % 2 == 1 ? r0.u2 : r0.u1;
    launch_k(k_rg_pool, B, 512, psm, st, 1, (const long long*)ucur, unext, B, N, K, P,
             uniform ? nullptr : toff, T, (const int32_t*)order, r0.pool, r0.info, r0.s0, tv);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    launch_k(k_rg_rho<ROWS>, grid, 32 * ROWS, rsm, st, 1, (const float*)C, (const uint16_t*)scol,
             (const float*)r0.bcov, (const int32_t*)r0.cnt, B, N, M, H, L2, toff, T, uniform,
             (const int32_t*)r0.pool, (const int32_t*)r0.info, P, p.resp_temp, p.resp_eps, fx_exp,
             fexp, r0.s0);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    launch_k(k_rg_filter<ROWS>, fgrid, 32 * ROWS, gsm, st, 1, C, scol, B, N, K, M, H, L2, toff, T,
             uniform, (const int32_t*)r0.pool, r0.info, (const long long*)r0.s0, P, p.batch_b,
             fx_exp, fexp, unext, r0.bcov, r0.cnt, order, rpw, tv);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  return cudaSuccess;
}

cudaError_t launch_round0(const R0State& r0, int B, int N, int K, int M, const int32_t* toff,
                          int H, int T, int L2, const gmc_params& p, int fx_exp,
                          const int32_t* fexp, float* C, uint16_t* scol, const long long* u0,
                          int32_t* order, uint32_t* status, const TraceView& tv,
                          cudaStream_t st, int I) {
  const int P = p.pool_mult * p.batch_b;
  cudaError_t e;
  const size_t smem =
      sizeof(long long) * (size_t)N + sizeof(int) * (sel::HBINS + N + 32 + 8 + sel::CBINS + P) +
      4 * (size_t)N + 64;
  if ((e = set_smem_limit((const void*)k_r0_pool, smem)) != cudaSuccess) return e;
  const int uniform = (H == 0);
  launch_k(k_r0_pool, B, 512, smem, st, 1, u0, B, N, P, uniform ? nullptr : toff, T, I, r0.pool, r0.info,
                                  r0.s0, r0.u1, r0.fv, status, tv);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  // one image: 16 rows per block (fewer, larger blocks finish the rounds
  // sooner); a batch: 8
  if (B == 1)
    return launch_rounds_rows<16>(r0, B, N, K, M, toff, H, T, L2, p, fx_exp, fexp, C, scol, order,
                                  tv, st, I, smem);
  return launch_rounds_rows<8>(r0, B, N, K, M, toff, H, T, L2, p, fx_exp, fexp, C, scol, order, tv,
                               st, I, smem);
}

}  // namespace gmc
