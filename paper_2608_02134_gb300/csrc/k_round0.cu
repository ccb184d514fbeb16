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
// Every reduction is an integer sum, so the result does not depend on the
// order blocks run in.  The cluster kernel (k_select) continues from round 1.
#include "common.cuh"
#include "kernels.cuh"
#include "select_common.cuh"

namespace gmc {

namespace {
constexpr int R0_ROWS = 8;  // rows per block (one warp each)
}

__global__ void __launch_bounds__(512) k_r0_pool(const long long* __restrict__ u0, int B, int N,
                                                   int P, const int32_t* toff, int Tmax,
                                                   int32_t* pool0, int32_t* info, long long* s0,
                                                   long long* u1, long long* fv, uint32_t* status) {
  grid_dep_wait();
  extern __shared__ __align__(16) char sm_r0p[];
  const int b = blockIdx.x;
  // the accumulators of the next two kernels start at zero
  for (int k = threadIdx.x; k < P; k += blockDim.x) s0[(size_t)b * P + k] = 0;
  for (int j = threadIdx.x; j < N; j += blockDim.x) u1[(size_t)b * N + j] = 0;
  if (threadIdx.x < 4) fv[(size_t)b * 4 + threadIdx.x] = 0;
  if (toff && text_geom(toff, b, B, Tmax, nullptr).T == 0) {
    if (threadIdx.x == 0) info[b * 4] = 0;
    return;
  }
  sel::PoolScratch w;
  char* p = sm_r0p;
  w.hist = reinterpret_cast<int*>(p);       p += sizeof(int) * sel::HBINS;
  w.bnd = reinterpret_cast<int*>(p);        p += sizeof(int) * N;
  w.wsum = reinterpret_cast<int*>(p);       p += sizeof(int) * 32;
  w.scal = reinterpret_cast<int*>(p);       p += sizeof(int) * 8;
  int* pool = reinterpret_cast<int*>(p);    p += sizeof(int) * P;
  w.tmp = reinterpret_cast<int*>(p);        p += sizeof(int) * P;
  unsigned char* selz = reinterpret_cast<unsigned char*>(p);
  for (int j = threadIdx.x; j < N; j += blockDim.x) selz[j] = 0;
  for (int h = threadIdx.x; h < sel::HBINS; h += blockDim.x) w.hist[h] = 0;
  __syncthreads();
  const int Pt = sel::select_pool(u0 + (size_t)b * N, selz, N, P, w, pool, nullptr);
  for (int k = threadIdx.x; k < P; k += blockDim.x) pool0[(size_t)b * P + k] = k < Pt ? pool[k] : -1;
  if (threadIdx.x == 0) info[b * 4] = Pt;
}

__global__ void __launch_bounds__(32 * R0_ROWS) k_r0_rho(
    const float* __restrict__ C, int B, int N, int Mstride, int H, int L2, const int32_t* toff,
    int Tmax, int uniform_rows, const int32_t* __restrict__ pool0, const int32_t* __restrict__ info,
    int P, float resp_temp, float resp_eps, int fx_exp, const int32_t* fexp, long long* s0) {
  grid_dep_wait();
  __shared__ int pool[GMC_MAX_POOL];
  __shared__ long long sblk[GMC_MAX_POOL];
  const int b = blockIdx.y;
  const int Pt = info[b * 4];
  if (Pt == 0) return;
  int Mb = Mstride;
  if (!uniform_rows) Mb = H * text_geom(toff, b, B, Tmax, nullptr).T + N + L2;
  const int m0 = blockIdx.x * R0_ROWS;
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
      const float tau = resp_temp * rmax + resp_eps;
      float z = 0.f;
#pragma unroll
      for (int u = 0; u < GMC_MAX_POOL / 32; ++u)
        if (Rd[u] > 0.f) z += expf(Rd[u] / tau);
      z = warp_sum(z) + (float)(Pt - npool);
      const float invz = 1.f / z;
#pragma unroll
      for (int u = 0; u < GMC_MAX_POOL / 32; ++u)
        if (Rd[u] > 0.f)
          atomicAdd((unsigned long long*)&sblk[lane + 32 * u],
                    (unsigned long long)to_fix(expf(Rd[u] / tau) * invz * Rd[u], fxs));
    }
  }
  __syncthreads();
  for (int k = threadIdx.x; k < Pt; k += blockDim.x)
    if (sblk[k]) atomicAdd((unsigned long long*)&s0[(size_t)b * P + k], (unsigned long long)sblk[k]);
}

__global__ void __launch_bounds__(32 * R0_ROWS) k_r0_filter(
    float* C, uint16_t* scol, int B, int N, int K, int Mstride, int H, int L2,
    const int32_t* toff, int Tmax, int uniform_rows, const int32_t* __restrict__ pool0,
    int32_t* info, const long long* __restrict__ s0, int P, int bsz, int fx_exp,
    const int32_t* fexp, long long* u1, float* bcov, int32_t* cnt, long long* fv,
    int32_t* order, TraceView tv) {
  grid_dep_wait();
  __shared__ int pool[GMC_MAX_POOL];
  __shared__ long long sc[GMC_MAX_POOL];
  __shared__ int batch[GMC_MAX_POOL];
  __shared__ long long fb[3];
  // the block's contributions to the next gains, one global atomic per column at the end
  extern __shared__ unsigned long long uacc[];  // [N]
  const int b = blockIdx.y;
  const int Pt = info[b * 4];
  if (Pt == 0) return;
  int Mb = Mstride, MG = Mstride;
  if (!uniform_rows) {
    MG = H * text_geom(toff, b, B, Tmax, nullptr).T;
    Mb = MG + N + L2;
  }
  const int m0 = blockIdx.x * R0_ROWS;
  if (m0 >= Mb) return;
  const float fxs = ldexpf(1.f, fexp ? fexp[b] : fx_exp);
  const int nb = min(bsz, min(Pt, K));
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
      const int rank = sel::group_score_rank(sc, pool, Pt, k, gl, gm);
      if (gl == 0 && rank < nb) batch[rank] = pool[k];
    }
  }
  __syncthreads();
  if (blockIdx.x == 0) {  // record the first batch once per image
    for (int q = threadIdx.x; q < nb; q += blockDim.x) order[(size_t)b * K + q] = batch[q];
    if (threadIdx.x == 0) info[b * 4 + 1] = nb;
    if (tv.base) {
      int32_t* tp = tv.at<int32_t>(b, tv.off_pool);
      for (int k = threadIdx.x; k < tv.pool_size; k += blockDim.x) tp[k] = k < Pt ? pool[k] : -1;
      if (threadIdx.x == 0) tv.at<int32_t>(b, tv.off_round_end)[0] = nb;
    }
  }
  const int lane = threadIdx.x & 31, m = m0 + (threadIdx.x >> 5);
  if (m < Mb) {
    float* vals = C + ((size_t)b * Mstride + m) * N;
    uint16_t* cols = scol + ((size_t)b * Mstride + m) * N;
    float bnew = 0.f;
    for (int t = lane; t < nb; t += 32) bnew = fmaxf(bnew, vals[batch[t]]);
    bnew = warp_max(bnew);
    const long long fb_new = to_fix(bnew, fxs);
    int w = 0;
    float rowmax = 0.f;
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
          int kc = 0;
#pragma unroll
          for (int e2 = 0; e2 < 4; ++e2) {
            rowmax = fmaxf(rowmax, c4[e2]);
            kc += (k4 < n4 && c4[e2] > bnew);
          }
          int pre = kc;
#pragma unroll
          for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(FULL, pre, o);
            if (lane >= o) pre += y;
          }
          const int tot = __shfl_sync(FULL, pre, 31);
          int pos = w + pre - kc;
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
    }
  }
  __syncthreads();
  if (threadIdx.x < 3 && fb[threadIdx.x])
    atomicAdd((unsigned long long*)&fv[(size_t)b * 4 + threadIdx.x], (unsigned long long)fb[threadIdx.x]);
  unsigned long long* ub = reinterpret_cast<unsigned long long*>(u1 + (size_t)b * N);
  for (int j = threadIdx.x; j < N; j += blockDim.x)
    if (uacc[j]) atomicAdd(&ub[j], uacc[j]);
}

cudaError_t launch_round0(const R0State& r0, int B, int N, int K, int M, const int32_t* toff,
                          int H, int T, int L2, const gmc_params& p, int fx_exp,
                          const int32_t* fexp, float* C, uint16_t* scol, const long long* u0,
                          int32_t* order, uint32_t* status, const TraceView& tv,
                          cudaStream_t st) {
  const int P = p.pool_mult * p.batch_b;
  cudaError_t e;
  const size_t smem = sizeof(int) * (sel::HBINS + N + 32 + 8 + 2 * P) + (size_t)N + 64;
  if ((e = set_smem_limit((const void*)k_r0_pool, smem)) != cudaSuccess) return e;
  const int uniform = (H == 0);
  launch_k(k_r0_pool, B, 512, smem, st, 1, u0, B, N, P, uniform ? nullptr : toff, T, r0.pool, r0.info,
                                  r0.s0, r0.u1, r0.fv, status);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  dim3 grid(ceil_div(M, R0_ROWS), B);
  launch_k(k_r0_rho, grid, 32 * R0_ROWS, 0, st, 1, C, B, N, M, H, L2, toff, T, uniform, r0.pool, r0.info,
                                          P, p.resp_temp, p.resp_eps, fx_exp, fexp, r0.s0);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  const size_t fsm = sizeof(unsigned long long) * (size_t)N;
  if ((e = set_smem_limit((const void*)k_r0_filter, fsm)) != cudaSuccess) return e;
  launch_k(k_r0_filter, grid, 32 * R0_ROWS, fsm, st, 1, C, scol, B, N, K, M, H, L2, toff, T, uniform, r0.pool,
                                             r0.info, r0.s0, P, p.batch_b, fx_exp, fexp, r0.u1,
                                             r0.bcov, r0.cnt, r0.fv, order, tv);
  return cudaGetLastError();
}

}  // namespace gmc
