// Client matrix Cbar (appendix Eq. (cond-coverage)) and its column sums.
//
// Rows of image b, in this order:
//   grounded   (v, h, t), view-major then h-major:
//              beta_v * omega_h * nu_t * ||u_i^{v,h,t}|| / sum_j ||u_j^{v,h,t}||
//              (v = 0 the current view with beta_G, then the historical views
//              sharing beta_hist; zero when the row has no energy: an inactive
//              client)
//   appearance m = 0..MV-1:      beta_V / MV * softmax_i(app_mi / tau_v), where
//                                app is the N x N cosine matrix (MV = N, exact
//                                bank) or the bounded bank's M_V x N projected
//                                cosines x~_{c(m)} . x~_i (long prefixes)
//   spatial    l = 0..I*L*L-1:   beta_S / (I L^2) * softmax_i(-||p_i - l_l||^2 / tau_s)
// with p_i = ((r+.5)/gh, (c+.5)/gw) and landmarks ((a+.5)/L, (b+.5)/L).  A
// prompt with I > 1 images holds them one after another (Ng = gh * gw tokens
// each): an appearance row and the landmark grid of image k (rows k L^2 ..)
// cover image k's tokens only, in that image's own coordinates; grounded rows
// cover every visual token.
// The spatial softmax separates over the grid: ||p_i - l||^2 = dy_r^2 + dx_c^2,
// so its smallest distance is min dy^2 + min dx^2 and its normaliser is
// (sum_r exp(-dy_r^2 / tau_s)) (sum_c exp(-dx_c^2 / tau_s)) (each factor
// shifted by its own minimum): gh + gw terms instead of N.  The appearance
// row's max and normaliser come from one online pass over the cosine row.
// The column sums u0_i = sum_m Cbar_mi (the singleton gains of the empty
// support) are accumulated in 64-bit fixed point, so they are exact sums of
// the fp32 entries and independent of the order the blocks finish in.
// A block's eight rows are nearly always of one kind -- eight consecutive
// queries of one head (which share the factor sqrt(||Z_h[i]||^2 + sigma_h^2)
// of every column), eight consecutive appearance rows, or eight landmarks:
// those blocks keep their rows' constants in registers and compute the
// shared factor once per column; a mixed block takes the generic loop.  Both
// evaluate the same expressions, so the entries are the same.
#include "common.cuh"
#include "kernels.cuh"

namespace gmc {

struct RowInfo {
  int kind;        // 0 grounded, 1 appearance, 2 spatial, -1 none
  const float* x;  // grounded: A row; appearance: cosine row; else nullptr
  const float* z;  // grounded: ||Z_h||^2 row; else nullptr
  float scale;     // multiplies the unnormalised value
  float shift;     // appearance: row max of the cosine; spatial: smallest distance^2
  float sg2;       // grounded: sigma_h^2
  float ly, lx;    // spatial: landmark coordinates
  int lo, hi;      // columns the row covers (its image; every column for grounded rows)
};

// Online (max, sum of exp((x - max) / tau)) of a row, one lane's share: 8
// loads in flight at a time; the running sum is rescaled when a group of 8
// raises the max.
__device__ __forceinline__ void row_softmax_stats(const float* row, int N, float itau, int lane,
                                                  float& m, float& z) {
  m = -INFINITY;
  z = 0.f;
  for (int j0 = lane; j0 < N; j0 += 32 * 8) {
    float x[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) x[u] = j0 + 32 * u < N ? row[j0 + 32 * u] : -INFINITY;
    float m8 = x[0];
#pragma unroll
    for (int u = 1; u < 8; ++u) m8 = fmaxf(m8, x[u]);
    if (m8 > m) {
      z = m == -INFINITY ? 0.f : z * expf((m - m8) * itau);
      m = m8;
    }
#pragma unroll
    for (int u = 0; u < 8; ++u) z += x[u] == -INFINITY ? 0.f : expf((x[u] - m) * itau);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {  // merge the lanes' (max, sum) pairs
    const float om = __shfl_xor_sync(FULL, m, o), oz = __shfl_xor_sync(FULL, z, o);
    const float nm = fmaxf(m, om);
    z = (z == 0.f ? 0.f : z * expf((m - nm) * itau)) + (oz == 0.f ? 0.f : oz * expf((om - nm) * itau));
    m = nm;
  }
}

__global__ void __launch_bounds__(256, 4) k_build_clients(
    const ViewRows vw, int nRS, const float* __restrict__ omega,
    const float* __restrict__ app, int MV, const int32_t* toff, int B, int N, int Tmax, int H, int M,
    int gh, int gw, int L, float beta_V, float beta_S, float tau_v, float tau_s,
    float wq, float fx_scale, int check, int I, float* C, long long* u0, uint32_t* status,
    int part) {
  grid_dep_wait();
  __shared__ RowInfo ri[ROWS_PER_BLOCK];
  const int b = blockIdx.y;
  const TextGeom tg = text_geom(toff, b, B, Tmax, status);
  if (tg.T == 0) return;
  const int Tb = tg.T, MG = vw.n * H * Tb, Mb = MG + MV + I * L * L;
  const int Ng = N / I;  // tokens of one image
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  // part 0: every row; 1: the grounded rows [0, MG); 2: the appearance and
  // spatial rows [MG, Mb) (built beside the message slice and the heads)
  const int rbeg = part == 2 ? MG : 0, rend = part == 1 ? MG : Mb;
  const int r0 = rbeg + blockIdx.x * ROWS_PER_BLOCK;
  if (r0 >= rend) return;
  {
    const int m = r0 + w;
    RowInfo inf{-1, nullptr, nullptr, 0.f, 0.f, 0.f, 0.f, 0.f, 0, N};
    if (m >= rend) {
      // past this launch's rows
    } else if (m < MG) {
      const int v = m / (H * Tb), hm = m - v * H * Tb;  // view, then (h, t) h-major
      const int h = hm / Tb, t = hm % Tb;
      float rsv = 0.f;  // parts over key splits, fixed order
      for (int q = 0; q < nRS; ++q) rsv += vw.rs[v][(((size_t)b * H + h) * nRS + q) * Tmax + t];
      const float nu = (t == Tb - 1 ? wq : 1.f) / ((float)(Tb - 1) + wq);
      const float sg = vw.sigma[v][(size_t)b * H + h];
      inf.kind = 0;
      inf.x = vw.A[v] + (((size_t)b * H + h) * Tmax + t) * N;
      inf.z = vw.zn2[v] + ((size_t)b * H + h) * N;
      inf.scale = rsv > 0.f ? vw.beta[v] * omega[(size_t)b * H + h] * nu / rsv : 0.f;
      inf.sg2 = sg * sg;
    } else if (m < MG + MV) {
      const int a = m - MG;
      const float* row = app + ((size_t)b * MV + a) * N;
      inf.lo = (a / Ng) * Ng;  // the row's own image (one image when the bank is bounded)
      inf.hi = inf.lo + Ng;
      float mx, z;
      row_softmax_stats(row + inf.lo, Ng, 1.f / tau_v, lane, mx, z);
      inf.kind = 1;
      inf.x = row;
      inf.scale = beta_V / ((float)MV * z);
      inf.shift = mx;
    } else if (m < Mb) {
      const int lg = m - MG - MV;
      const int l = lg % (L * L);  // landmark of image lg / L^2
      inf.lo = (lg / (L * L)) * Ng;
      inf.hi = inf.lo + Ng;
      const int la = l / L, lb = l % L;
      const float ly = (la + 0.5f) / L, lx = (lb + 0.5f) / L;
      float mny = INFINITY, mnx = INFINITY;
      for (int r = lane; r < gh; r += 32) {
        const float dy = (r + 0.5f) / gh - ly;
        mny = fminf(mny, dy * dy);
      }
      for (int c = lane; c < gw; c += 32) {
        const float dx = (c + 0.5f) / gw - lx;
        mnx = fminf(mnx, dx * dx);
      }
      mny = -warp_max(-mny);
      mnx = -warp_max(-mnx);
      float zy = 0.f, zx = 0.f;
      for (int r = lane; r < gh; r += 32) {
        const float dy = (r + 0.5f) / gh - ly;
        zy += expf(-(dy * dy - mny) / tau_s);
      }
      for (int c = lane; c < gw; c += 32) {
        const float dx = (c + 0.5f) / gw - lx;
        zx += expf(-(dx * dx - mnx) / tau_s);
      }
      zy = warp_sum(zy);
      zx = warp_sum(zx);
      inf.kind = 2;
      inf.scale = beta_S / ((float)(I * L * L) * (zy * zx));
      inf.shift = mny + mnx;
      inf.ly = ly;
      inf.lx = lx;
    }
    if (lane == 0) ri[w] = inf;
  }
  __shared__ int umode;  // 0 generic, 1 grounded (one head), 2 appearance, 3 spatial
  __syncthreads();
  const int nrows = min(ROWS_PER_BLOCK, rend - r0);
  const float itv = 1.f / tau_v, its = 1.f / tau_s;
  if (threadIdx.x == 0) {
    int mode = 0;
    if (nrows == ROWS_PER_BLOCK && !check) {
      const RowInfo& f = ri[0];
      bool same = true;
      for (int q = 1; q < ROWS_PER_BLOCK; ++q) {
        const RowInfo& g = ri[q];
        same = same && g.kind == f.kind && g.lo == f.lo && g.hi == f.hi;
        if (f.kind == 0) same = same && g.z == f.z && g.sg2 == f.sg2 && g.x == f.x + (size_t)q * N;
        if (f.kind == 1) same = same && g.x == f.x + (size_t)q * N;
      }
      if (same && f.kind >= 0) mode = f.kind + 1;
    }
    umode = mode;
  }
  __syncthreads();
  const int mode = umode;
  float* Crow = C + ((size_t)b * M + r0) * N;
  unsigned long long* ucol = reinterpret_cast<unsigned long long*>(u0 + (size_t)b * N);
  if (mode == 1) {  // grounded rows of one head: x * sqrt(||Z_h[i]||^2 + sigma_h^2) * scale
    const float* x0 = ri[0].x;
    const float* zr = ri[0].z;
    const float sg2 = ri[0].sg2;
    float sc[ROWS_PER_BLOCK];
#pragma unroll
    for (int q = 0; q < ROWS_PER_BLOCK; ++q) sc[q] = ri[q].scale;
    for (int j = threadIdx.x; j < N; j += blockDim.x) {
      float xv[ROWS_PER_BLOCK];
#pragma unroll
      for (int q = 0; q < ROWS_PER_BLOCK; ++q) xv[q] = x0[(size_t)q * N + j];
      const float g = sqrtf(zr[j] + sg2);
      long long colsum = 0;
#pragma unroll
      for (int q = 0; q < ROWS_PER_BLOCK; ++q) {
        const float v = xv[q] * g * sc[q];
        Crow[(size_t)q * N + j] = v;
        colsum += to_fix(v, fx_scale);
      }
      if (colsum) atomicAdd(ucol + j, (unsigned long long)colsum);
    }
    return;
  }
  if (mode == 2) {  // appearance rows: exp((x - row max) / tau_v) * scale on the row's image
    const float* x0 = ri[0].x;
    const int lo = ri[0].lo, hi = ri[0].hi;
    float sh[ROWS_PER_BLOCK], sc[ROWS_PER_BLOCK];
#pragma unroll
    for (int q = 0; q < ROWS_PER_BLOCK; ++q) {
      sh[q] = ri[q].shift;
      sc[q] = ri[q].scale;
    }
    for (int j = threadIdx.x; j < N; j += blockDim.x) {
      const bool in = j >= lo && j < hi;
      float xv[ROWS_PER_BLOCK];
#pragma unroll
      for (int q = 0; q < ROWS_PER_BLOCK; ++q) xv[q] = in ? x0[(size_t)q * N + j] : 0.f;
      long long colsum = 0;
#pragma unroll
      for (int q = 0; q < ROWS_PER_BLOCK; ++q) {
        const float v = in ? expf((xv[q] - sh[q]) * itv) * sc[q] : 0.f;
        Crow[(size_t)q * N + j] = v;
        colsum += to_fix(v, fx_scale);
      }
      if (colsum) atomicAdd(ucol + j, (unsigned long long)colsum);
    }
    return;
  }
  if (mode == 3) {  // landmark rows: exp((smallest d^2 - ||p_i - l||^2) / tau_s) * scale
    const int lo = ri[0].lo, hi = ri[0].hi;
    float sh[ROWS_PER_BLOCK], sc[ROWS_PER_BLOCK], ly[ROWS_PER_BLOCK], lx[ROWS_PER_BLOCK];
#pragma unroll
    for (int q = 0; q < ROWS_PER_BLOCK; ++q) {
      sh[q] = ri[q].shift;
      sc[q] = ri[q].scale;
      ly[q] = ri[q].ly;
      lx[q] = ri[q].lx;
    }
    for (int j = threadIdx.x; j < N; j += blockDim.x) {
      const bool in = j >= lo && j < hi;
      const int jl = j % Ng, jr = jl / gw;  // position in its own image's grid
      const float py = (jr + 0.5f) / gh, px = ((jl - jr * gw) + 0.5f) / gw;
      long long colsum = 0;
#pragma unroll
      for (int q = 0; q < ROWS_PER_BLOCK; ++q) {
        const float dy = py - ly[q], dx = px - lx[q];
        const float v = in ? expf((sh[q] - (dy * dy + dx * dx)) * its) * sc[q] : 0.f;
        Crow[(size_t)q * N + j] = v;
        colsum += to_fix(v, fx_scale);
      }
      if (colsum) atomicAdd(ucol + j, (unsigned long long)colsum);
    }
    return;
  }
  for (int j = threadIdx.x; j < N; j += blockDim.x) {
    long long colsum = 0;
    const int jl = j % Ng, jr = jl / gw;  // position in its own image's grid
    const float py = (jr + 0.5f) / gh, px = ((jl - jr * gw) + 0.5f) / gw;
    // every row's operands are loaded before any is used
    float xv[ROWS_PER_BLOCK], zv[ROWS_PER_BLOCK];
#pragma unroll
    for (int q = 0; q < ROWS_PER_BLOCK; ++q) {
      const RowInfo& inf = ri[q];
      xv[q] = q < nrows && inf.x ? inf.x[j] : 0.f;
      zv[q] = q < nrows && inf.z ? inf.z[j] : 0.f;
    }
#pragma unroll
    for (int q = 0; q < ROWS_PER_BLOCK; ++q) {
      if (q >= nrows) break;
      const RowInfo& inf = ri[q];
      float v = 0.f;
      if (j < inf.lo || j >= inf.hi) {
        v = 0.f;  // another image's token
      } else if (inf.kind == 0) {
        v = xv[q] * sqrtf(zv[q] + inf.sg2) * inf.scale;
      } else if (inf.kind == 1) {
        v = expf((xv[q] - inf.shift) * itv) * inf.scale;
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
                                 const ViewRows& views, const float* app, cudaStream_t st,
                                 int part) {
  const int rows = part == 0 ? dm.M
                 : part == 1 ? dm.V * dm.H * dm.T
                             : dm.MV + dm.I * dm.L * dm.L;
  dim3 grid(ceil_div(rows, ROWS_PER_BLOCK), dm.B);
  launch_k(k_build_clients, grid, 32 * ROWS_PER_BLOCK, 0, st, 1,
      views, s.nRS, s.omega, app, dm.MV, dm.toff, dm.B, dm.N, dm.T, dm.H, dm.M, dm.gh,
      dm.gw, dm.L, p.beta_V, p.beta_S, p.tau_v, p.tau_s, p.terminal_q_weight,
      ldexpf(1.f, fx_exp), p.check_mode, dm.I, s.C, s.u0, s.status, part);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// gmc_select on caller clients: per-image total mass -> fixed-point exponent,
// then fixed-point column sums.
// ---------------------------------------------------------------------------
__global__ void k_sel_total(const float* __restrict__ C, int M, int N, int nblk, double* part,
                            uint32_t* status) {
  grid_dep_wait();
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
  grid_dep_wait();
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
  grid_dep_wait();
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
  launch_k(k_sel_total, dim3(s.nSel, B), 256, 0, st, 1, C, M, N, s.nSel, s.selpart, s.status);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  launch_k(k_sel_exp, ceil_div(B, 128), 128, 0, st, 1, s.selpart, s.nSel, B, s.fexp);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  launch_k(k_sel_colsum, dim3(ceil_div(M, ROWS_PER_BLOCK), B), 256, 0, st, 1, C, M, N, s.fexp, s.u0);
  return cudaGetLastError();
}

}  // namespace gmc
