// Client matrix Cbar (appendix Eq. (cond-coverage)) and its column sums.
//
// Rows of image b, in this order:
//   grounded   (h, t), h-major:  beta_G * omega_h * nu_t * ||u_i^{h,t}|| / sum_j ||u_j^{h,t}||
//              (zero when the row has no energy: an inactive client)
//   appearance m = 0..N-1:       beta_V / N * softmax_i(cos_mi / tau_v)
//   spatial    l = 0..L*L-1:     beta_S / L^2 * softmax_i(-||p_i - l_l||^2 / tau_s)
// with p_i = ((r+.5)/gh, (c+.5)/gw) and landmarks ((a+.5)/L, (b+.5)/L).
// The column sums u0_i = sum_m Cbar_mi (the singleton gains of the empty
// support) are accumulated in 64-bit fixed point, so they are exact sums of
// the fp32 entries and independent of the order the blocks finish in.
#include "common.cuh"
#include "kernels.cuh"

namespace gmc {

struct RowInfo {
  int kind;       // 0 grounded, 1 appearance, 2 spatial, -1 none
  size_t src;     // grounded: A row offset; appearance: cos row offset
  size_t zrow;    // grounded: ||Z_h||^2 row offset
  float scale;    // multiplies the unnormalised value
  float shift;    // appearance: row max of the cosine; spatial: smallest distance^2
  float sg2;      // grounded: sigma_h^2
  float ly, lx;   // spatial: landmark coordinates
};

__global__ void __launch_bounds__(256) k_build_clients(
    const float* __restrict__ A, const float* __restrict__ rs, int nRS, const float* __restrict__ zn2,
    const float* __restrict__ sigma, const float* __restrict__ omega,
    const float* __restrict__ cos, const int32_t* toff, int B, int N, int Tmax, int H, int M,
    int gh, int gw, int L, float beta_G, float beta_V, float beta_S, float tau_v, float tau_s,
    float wq, float fx_scale, int check, float* C, long long* u0, uint32_t* status) {
  __shared__ RowInfo ri[ROWS_PER_BLOCK];
  const int b = blockIdx.y;
  const TextGeom tg = text_geom(toff, b, B, Tmax, status);
  if (tg.T == 0) return;
  const int Tb = tg.T, MG = H * Tb, Mb = MG + N + L * L;
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int r0 = blockIdx.x * ROWS_PER_BLOCK;
  if (r0 >= Mb) return;
  {
    const int m = r0 + w;
    RowInfo inf{-1, 0, 0, 0.f, 0.f, 0.f, 0.f, 0.f};
    if (m < MG) {
      const int h = m / Tb, t = m % Tb;
      float rsv = 0.f;  // parts over key splits, fixed order
      for (int q = 0; q < nRS; ++q) rsv += rs[(((size_t)b * H + h) * nRS + q) * Tmax + t];
      const float nu = (t == Tb - 1 ? wq : 1.f) / ((float)(Tb - 1) + wq);
      const float sg = sigma[(size_t)b * H + h];
      inf.kind = 0;
      inf.src = (((size_t)b * H + h) * Tmax + t) * N;
      inf.zrow = ((size_t)b * H + h) * N;
      inf.scale = rsv > 0.f ? beta_G * omega[(size_t)b * H + h] * nu / rsv : 0.f;
      inf.sg2 = sg * sg;
    } else if (m < MG + N) {
      const int a = m - MG;
      const float* row = cos + ((size_t)b * N + a) * N;
      float mx = -INFINITY;
      for (int j = lane; j < N; j += 32) mx = fmaxf(mx, row[j]);
      mx = warp_max(mx);
      float z = 0.f;
      for (int j = lane; j < N; j += 32) z += expf((row[j] - mx) / tau_v);
      z = warp_sum(z);
      inf.kind = 1;
      inf.src = ((size_t)b * N + a) * N;
      inf.scale = beta_V / ((float)N * z);
      inf.shift = mx;
    } else if (m < Mb) {
      const int l = m - MG - N;
      const int la = l / L, lb = l % L;
      const float ly = (la + 0.5f) / L, lx = (lb + 0.5f) / L;
      float mn = INFINITY;
      for (int j = lane; j < N; j += 32) {
        const float dy = ((j / gw) + 0.5f) / gh - ly, dx = ((j % gw) + 0.5f) / gw - lx;
        mn = fminf(mn, dy * dy + dx * dx);
      }
      mn = -warp_max(-mn);
      float z = 0.f;
      for (int j = lane; j < N; j += 32) {
        const float dy = ((j / gw) + 0.5f) / gh - ly, dx = ((j % gw) + 0.5f) / gw - lx;
        z += expf(-(dy * dy + dx * dx - mn) / tau_s);
      }
      z = warp_sum(z);
      inf.kind = 2;
      inf.scale = beta_S / ((float)(L * L) * z);
      inf.shift = mn;
      inf.ly = ly;
      inf.lx = lx;
    }
    if (lane == 0) ri[w] = inf;
  }
  __syncthreads();
  const int nrows = min(ROWS_PER_BLOCK, Mb - r0);
  const float itv = 1.f / tau_v, its = 1.f / tau_s;
  for (int j = threadIdx.x; j < N; j += blockDim.x) {
    long long colsum = 0;
    const int jr = j / gw;
    const float py = (jr + 0.5f) / gh, px = ((j - jr * gw) + 0.5f) / gw;
    for (int q = 0; q < nrows; ++q) {
      const RowInfo& inf = ri[q];
      float v = 0.f;
      if (inf.kind == 0) {
        v = A[inf.src + j] * sqrtf(zn2[inf.zrow + j] + inf.sg2) * inf.scale;
      } else if (inf.kind == 1) {
        v = expf((cos[inf.src + j] - inf.shift) * itv) * inf.scale;
      } else if (inf.kind == 2) {
        const float dy = py - inf.ly, dx = px - inf.lx;
        v = expf((inf.shift - (dy * dy + dx * dx)) * its) * inf.scale;
      }
      if (check && !isfinite(v)) set_status(status, GMC_STATUS_NONFINITE);
      C[((size_t)b * M + r0 + q) * N + j] = v;
      colsum += to_fix(v, fx_scale);
    }
    if (colsum) atomicAdd(reinterpret_cast<unsigned long long*>(u0 + (size_t)b * N + j),
                          (unsigned long long)colsum);
  }
}

cudaError_t launch_build_clients(const Dims& dm, const gmc_params& p, int fx_exp, Scratch& s,
                                 cudaStream_t st) {
  dim3 grid(ceil_div(dm.M, ROWS_PER_BLOCK), dm.B);
  k_build_clients<<<grid, 32 * ROWS_PER_BLOCK, 0, st>>>(
      s.A, s.rs, s.nRS, s.zn2, s.sigma, s.omega, s.cos, dm.toff, dm.B, dm.N, dm.T, dm.H, dm.M, dm.gh,
      dm.gw, dm.L, p.beta_G, p.beta_V, p.beta_S, p.tau_v, p.tau_s, p.terminal_q_weight,
      ldexpf(1.f, fx_exp), p.check_mode, s.C, s.u0, s.status);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// gmc_select on caller clients: per-image total mass -> fixed-point exponent,
// then fixed-point column sums.
// ---------------------------------------------------------------------------
__global__ void k_sel_total(const float* __restrict__ C, int M, int N, int nblk, double* part,
                            uint32_t* status) {
  __shared__ double red[32];
  const int b = blockIdx.y;
  const size_t n = (size_t)M * N;
  const size_t per = (n + nblk - 1) / nblk;
  const size_t lo = per * blockIdx.x, hi = min(n, lo + per);
  const float* base = C + (size_t)b * n;
  double s = 0.0;
  bool bad = false;
  for (size_t k = lo + threadIdx.x; k < hi; k += blockDim.x) {
    const float v = base[k];
    bad |= !isfinite(v) || v < 0.f;
    s += v;
  }
  if (bad) set_status(status, GMC_STATUS_NONFINITE);
  s = block_reduce(s, red, OpAdd(), 0.0);
  if (threadIdx.x == 0) part[(size_t)b * nblk + blockIdx.x] = s;
}

__global__ void k_sel_exp(const double* part, int nblk, int B, int32_t* fexp) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  double tot = 0.0;
  for (int k = 0; k < nblk; ++k) tot += part[(size_t)b * nblk + k];
  int e = 61;
  if (tot > 0.0 && isfinite(tot)) e = 61 - (int)ceil(log2(tot));
  fexp[b] = max(-60, min(120, e));
}

__global__ void __launch_bounds__(256) k_sel_colsum(const float* __restrict__ C, int M, int N,
                                                    const int32_t* fexp, long long* u0) {
  const int b = blockIdx.y;
  const int r0 = blockIdx.x * ROWS_PER_BLOCK;
  const int nrows = min(ROWS_PER_BLOCK, M - r0);
  const float sc = ldexpf(1.f, fexp[b]);
  for (int j = threadIdx.x; j < N; j += blockDim.x) {
    long long cs = 0;
    for (int q = 0; q < nrows; ++q) {
      const float v = C[((size_t)b * M + r0 + q) * N + j];
      cs += to_fix(fmaxf(v, 0.f), sc);
    }
    if (cs) atomicAdd(reinterpret_cast<unsigned long long*>(u0 + (size_t)b * N + j),
                      (unsigned long long)cs);
  }
}

cudaError_t launch_select_prep(const float* C, int B, int M, int N, Scratch& s, cudaStream_t st) {
  k_sel_total<<<dim3(s.nSel, B), 256, 0, st>>>(C, M, N, s.nSel, s.selpart, s.status);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  k_sel_exp<<<ceil_div(B, 128), 128, 0, st>>>(s.selpart, s.nSel, B, s.fexp);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  k_sel_colsum<<<dim3(ceil_div(M, ROWS_PER_BLOCK), B), 256, 0, st>>>(C, M, N, s.fexp, s.u0);
  return cudaGetLastError();
}

}  // namespace gmc
