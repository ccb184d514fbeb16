// Head patterns, farthest-first head clusters, head weights and message energy
// (appendix Eq. (cond-head-pattern), (cond-head-weight), (cond-grounded-energy)).
//
// The pattern of head h stacks its atoms u_i^{h,t} = A[h,t,i] [Z_h[i]; sigma_h]
// over all (t, i), scaled to unit mean atom norm.  Only inner products of
// patterns are needed, and they factor per token:
//   <U_h, U_g> = sum_i (Z_h[i].Z_g[i] + sigma_h sigma_g) sum_t A[h,t,i] A[g,t,i]
// so the H x H Gram is accumulated token block by token block without ever
// forming the (T N (r+1))-long patterns.  The mean atom norm of head h is
// sum_t rs[h,t] / (T N) (rs from the message kernel).
#include "common.cuh"
#include "kernels.cuh"

namespace gmc {

constexpr int HG_TC = 32;                       // queries per staged chunk
constexpr int HG_RS = HG_TC * HG_TOK + 1;       // padded row stride of a staged head

__device__ __forceinline__ float query_weight(int t, int Tb, float wq) {
  return (t == Tb - 1 ? wq : 1.f) / ((float)(Tb - 1) + wq);
}

// Per block: HG_TOK tokens, all head pairs (h <= g).  Writes the block's part
// of the pattern Gram (fp64) and W2[h,i] = sum_t nu_t A[h,t,i]^2.
__global__ void k_head_stats(const float* __restrict__ A, const float* __restrict__ Z,
                             const float* __restrict__ sigma, const int32_t* toff, int B, int N,
                             int Tmax, int H, float wq, double* hgpart, int nHG, float* W2,
                             uint32_t* status) {
  extern __shared__ float sm_hs[];
  const int b = blockIdx.y;
  const TextGeom tg = text_geom(toff, b, B, Tmax, status);
  if (tg.T == 0) return;
  const int Tb = tg.T;
  const int npairs = H * (H + 1) / 2;
  float* Ablk = sm_hs;                          // [H][HG_RS]
  float* acc = Ablk + (size_t)H * HG_RS;        // [npairs][HG_TOK]
  float* w2 = acc + (size_t)npairs * HG_TOK;    // [H][HG_TOK]
  unsigned short* pairs = reinterpret_cast<unsigned short*>(w2 + H * HG_TOK);  // [npairs]
  const int i0 = blockIdx.x * HG_TOK;
  for (int p = threadIdx.x; p < npairs * HG_TOK; p += blockDim.x) acc[p] = 0.f;
  for (int p = threadIdx.x; p < H * HG_TOK; p += blockDim.x) w2[p] = 0.f;
  if (threadIdx.x == 0) {
    int p = 0;
    for (int h = 0; h < H; ++h)
      for (int g = h; g < H; ++g) pairs[p++] = (unsigned short)(h * 256 + g);
  }
  for (int t0 = 0; t0 < Tb; t0 += HG_TC) {
    const int tc = min(HG_TC, Tb - t0);
    __syncthreads();
    for (int idx = threadIdx.x; idx < H * HG_TC * HG_TOK; idx += blockDim.x) {
      const int h = idx / (HG_TC * HG_TOK), tt = (idx / HG_TOK) % HG_TC, ii = idx % HG_TOK;
      float v = 0.f;
      if (tt < tc && i0 + ii < N) v = A[(((size_t)b * H + h) * Tmax + t0 + tt) * N + i0 + ii];
      Ablk[h * HG_RS + tt * HG_TOK + ii] = v;
    }
    __syncthreads();
    for (int p = threadIdx.x; p < npairs; p += blockDim.x) {
      const int h = pairs[p] >> 8, g = pairs[p] & 255;
      const float* ah = Ablk + h * HG_RS;
      const float* ag = Ablk + g * HG_RS;
#pragma unroll
      for (int ii = 0; ii < HG_TOK; ++ii) {
        float s = 0.f;
        for (int tt = 0; tt < tc; ++tt) s = fmaf(ah[tt * HG_TOK + ii], ag[tt * HG_TOK + ii], s);
        acc[p * HG_TOK + ii] += s;
      }
    }
    for (int q = threadIdx.x; q < H * HG_TOK; q += blockDim.x) {
      const int h = q / HG_TOK, ii = q % HG_TOK;
      const float* ah = Ablk + h * HG_RS;
      float s = 0.f;
      for (int tt = 0; tt < tc; ++tt) {
        const float a = ah[tt * HG_TOK + ii];
        s = fmaf(query_weight(t0 + tt, Tb, wq) * a, a, s);
      }
      w2[q] += s;
    }
  }
  __syncthreads();
  double* out = hgpart + ((size_t)b * nHG + blockIdx.x) * H * H;
  for (int p = threadIdx.x; p < npairs; p += blockDim.x) {
    const int h = pairs[p] >> 8, g = pairs[p] & 255;
    const float sh = sigma[(size_t)b * H + h], sgv = sigma[(size_t)b * H + g];
    double v = 0.0;
    for (int ii = 0; ii < HG_TOK; ++ii) {
      const int i = i0 + ii;
      if (i >= N) break;
      const float4 zh = reinterpret_cast<const float4*>(Z)[((size_t)b * H + h) * N + i];
      const float4 zg = reinterpret_cast<const float4*>(Z)[((size_t)b * H + g) * N + i];
      const double w = (double)zh.x * zg.x + (double)zh.y * zg.y + (double)zh.z * zg.z +
                       (double)zh.w * zg.w + (double)sh * sgv;
      v += w * acc[p * HG_TOK + ii];
    }
    out[h * H + g] = v;
    out[g * H + h] = v;
  }
  for (int q = threadIdx.x; q < H * HG_TOK; q += blockDim.x) {
    const int h = q / HG_TOK, i = i0 + q % HG_TOK;
    if (i < N) W2[((size_t)b * H + h) * N + i] = w2[q];
  }
}

// One block per image: reduce the Gram, then one warp runs farthest-first
// clustering and the head weights (two heads per lane, H <= 64).
// Ties: the first centre is the lowest-index largest pattern, each next centre
// the lowest-index head of smallest max-cosine, and a head joins the earliest
// centre among equally similar ones.
__device__ __forceinline__ void warp_argbest(double& v, int& idx, bool want_max) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const double ov = __shfl_xor_sync(FULL, v, o);
    const int oi = __shfl_xor_sync(FULL, idx, o);
    const bool better = want_max ? (ov > v || (ov == v && oi < idx))
                                 : (ov < v || (ov == v && oi < idx));
    if (oi >= 0 && (idx < 0 || better)) { v = ov; idx = oi; }
  }
}

// The pattern Gram: sum of the token-block partials, one warp per (image, entry),
// lanes over the blocks (fixed order, so the sum is reproducible).
__global__ void k_hg_reduce(const double* __restrict__ hgpart, int nHG, int B, int HH, double* HG) {
  const int w = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (w >= B * HH) return;
  const int b = w / HH, p = w % HH;
  double s = 0.0;
  for (int k = lane; k < nHG; k += 32) s += hgpart[((size_t)b * nHG + k) * HH + p];
  s = warp_sum(s);
  if (lane == 0) HG[(size_t)b * HH + p] = s;
}

__global__ void k_head_cluster(const double* __restrict__ HGred,
                               const float* __restrict__ rs, const int32_t* toff, int B, int N,
                               int Tmax, int H, int max_clusters, float head_eps, float* omega,
                               TraceView tv, uint32_t* status) {
  extern __shared__ double sm_hc[];
  const int b = blockIdx.x;
  const TextGeom tg = text_geom(toff, b, B, Tmax, status);
  if (tg.T == 0) return;
  double* HG = sm_hc;            // [H*H]
  double* cs = HG + H * H;       // [H*H] pattern cosines
  double* pre = cs + H * H;      // [H]
  for (int p = threadIdx.x; p < H * H; p += blockDim.x) HG[p] = HGred[(size_t)b * H * H + p];
  __syncthreads();
  for (int h = threadIdx.x; h < H; h += blockDim.x) {
    double s1 = 0.0;
    for (int t = 0; t < tg.T; ++t) s1 += rs[((size_t)b * H + h) * Tmax + t];
    const double mean = s1 / ((double)tg.T * N);
    pre[h] = (mean > 0.0 && HG[h * H + h] > 0.0) ? sqrt(HG[h * H + h]) / mean : 0.0;
  }
  for (int p = threadIdx.x; p < H * H; p += blockDim.x) {
    const int h = p / H, g = p % H;
    const double a = HG[h * H + h], c = HG[g * H + g];
    cs[p] = (a > 0.0 && c > 0.0) ? HG[p] / sqrt(a * c) : 0.0;
  }
  __syncthreads();
  if (threadIdx.x >= 32) return;
  const int lane = threadIdx.x;
  const int h0 = lane, h1 = lane + 32;  // this lane's heads (if < H)
  const int nc = min(max_clusters, H);
  int centres[GMC_MAX_HEADS];
  bool c0 = false, c1 = false;  // is h0 / h1 a centre
  {
    double v = -1.0;
    int idx = -1;
    if (h0 < H) { v = pre[h0]; idx = h0; }
    if (h1 < H && (idx < 0 || pre[h1] > v)) { v = pre[h1]; idx = h1; }
    warp_argbest(v, idx, true);
    centres[0] = idx;
  }
  c0 = (h0 == centres[0]);
  c1 = (h1 == centres[0]);
  for (int c = 1; c < nc; ++c) {
    double v = 0.0;
    int idx = -1;
    for (int q = 0; q < 2; ++q) {
      const int h = q ? h1 : h0;
      if (h >= H || (q ? c1 : c0)) continue;
      double mc = -INFINITY;
      for (int k = 0; k < c; ++k) mc = fmax(mc, cs[h * H + centres[k]]);
      if (idx < 0 || mc < v) { v = mc; idx = h; }
    }
    warp_argbest(v, idx, false);
    centres[c] = idx;
    c0 |= (h0 == idx);
    c1 |= (h1 == idx);
  }
  int as0 = 0, as1 = 0;
  for (int q = 0; q < 2; ++q) {
    const int h = q ? h1 : h0;
    if (h >= H) continue;
    int bk = 0;
    for (int k = 1; k < nc; ++k)
      if (cs[h * H + centres[k]] > cs[h * H + centres[bk]]) bk = k;
    if (q) as1 = bk; else as0 = bk;
  }
  // every lane needs every head's cluster: gather through shuffles
  auto cluster_of = [&](int g) {
    const int src = g & 31;
    const int a0 = __shfl_sync(FULL, as0, src), a1 = __shfl_sync(FULL, as1, src);
    return g < 32 ? a0 : a1;
  };
  int asg[GMC_MAX_HEADS];
  for (int g = 0; g < H; ++g) asg[g] = cluster_of(g);
  int C = 0;
  double inv0 = 0.0, inv1 = 0.0;
  double invsum[GMC_MAX_HEADS];
  for (int k = 0; k < nc; ++k) {
    int cnt = 0;
    for (int g = 0; g < H; ++g) cnt += asg[g] == k;
    if (cnt == 0) { invsum[k] = 0.0; continue; }
    ++C;
    // ||sum_{g in k} u_g||^2 = sum over pairs in the cluster, rows split over lanes
    double part = 0.0;
    for (int q = 0; q < 2; ++q) {
      const int g = q ? h1 : h0;
      if (g >= H || asg[g] != k) continue;
      for (int g2 = 0; g2 < H; ++g2)
        if (asg[g2] == k) part += cs[g * H + g2];
    }
    const double nrm2 = warp_sum(part);
    const double nrm = nrm2 > 0.0 ? sqrt(nrm2) : 0.0;
    double mine = 0.0;
    for (int q = 0; q < 2; ++q) {
      const int h = q ? h1 : h0;
      if (h >= H || asg[h] != k) continue;
      double dot = 0.0;
      for (int g = 0; g < H; ++g)
        if (asg[g] == k) dot += cs[h * H + g];
      const double dh = 1.0 - (nrm > 0.0 ? dot / nrm : 0.0);
      const double inv = 1.0 / (dh + head_eps);
      if (q) inv1 = inv; else inv0 = inv;
      mine += inv;
    }
    invsum[k] = warp_sum(mine);
  }
  if (h0 < H) omega[(size_t)b * H + h0] = (float)(inv0 / invsum[as0] / C);
  if (h1 < H) omega[(size_t)b * H + h1] = (float)(inv1 / invsum[as1] / C);
  if (tv.base) {
    if (lane == 0) tv.header(b)->n_clusters = C;
    int32_t* tc = tv.at<int32_t>(b, tv.off_centres);
    for (int k = lane; k < max_clusters; k += 32) tc[k] = k < nc ? centres[k] : -1;
    int32_t* ta = tv.at<int32_t>(b, tv.off_head_assign);
    float* to = tv.at<float>(b, tv.off_omega);
    if (h0 < H) { ta[h0] = as0; to[h0] = (float)(inv0 / invsum[as0] / C); }
    if (h1 < H) { ta[h1] = as1; to[h1] = (float)(inv1 / invsum[as1] / C); }
  }
}

// e_i = (sum_h omega_h g_h(i)^2 sum_t nu_t A[h,t,i]^2)^{1/2}, ebar_i = e_i / mean(e)
// (uniform 1 if the mean vanishes).  One block per image.
__global__ void k_energy(const float* __restrict__ omega, const float* __restrict__ zn2,
                         const float* __restrict__ sigma, const float* __restrict__ W2,
                         const int32_t* toff, int B, int N, int Tmax, int H, float* ebar,
                         TraceView tv, uint32_t* status) {
  __shared__ double red[32];
  const int b = blockIdx.x;
  const TextGeom tg = text_geom(toff, b, B, Tmax, status);
  if (tg.T == 0) return;
  double local = 0.0;
  for (int i = threadIdx.x; i < N; i += blockDim.x) {
    float e2 = 0.f;
    for (int h = 0; h < H; ++h) {
      const size_t o = ((size_t)b * H + h) * N + i;
      const float sg = sigma[(size_t)b * H + h];
      e2 = fmaf(omega[(size_t)b * H + h] * (zn2[o] + sg * sg), W2[o], e2);
    }
    const float e = sqrtf(e2);
    ebar[(size_t)b * N + i] = e;
    local += e;
  }
  const double tot = block_reduce(local, red, OpAdd(), 0.0);
  const double mean = tot / N;
  for (int i = threadIdx.x; i < N; i += blockDim.x) {
    const size_t o = (size_t)b * N + i;
    const float v = mean > 0.0 ? (float)(ebar[o] / mean) : 1.f;
    ebar[o] = v;
    if (tv.base) tv.at<float>(b, tv.off_ebar)[i] = v;
  }
}

cudaError_t launch_heads(const Dims& dm, const gmc_params& p, Scratch& s, const TraceView& tv,
                         cudaStream_t st) {
  const int H = dm.H, npairs = H * (H + 1) / 2;
  size_t smem = sizeof(float) * ((size_t)H * HG_RS + (size_t)npairs * HG_TOK + H * HG_TOK) +
                sizeof(unsigned short) * npairs + 16;
  cudaError_t e = set_smem_limit((const void*)k_head_stats, smem);
  if (e != cudaSuccess) return e;
  k_head_stats<<<dim3(s.nHG, dm.B), 256, smem, st>>>(s.A, s.Z, s.sigma, dm.toff, dm.B, dm.N, dm.T,
                                                     H, p.terminal_q_weight, s.hgpart, s.nHG,
                                                     s.W2, s.status);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  const int warps = dm.B * H * H;
  k_hg_reduce<<<ceil_div(warps * 32, 256), 256, 0, st>>>(s.hgpart, s.nHG, dm.B, H * H, s.HG);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  size_t smem2 = sizeof(double) * (2 * (size_t)H * H + H);
  if ((e = set_smem_limit((const void*)k_head_cluster, smem2)) != cudaSuccess) return e;
  k_head_cluster<<<dm.B, 128, smem2, st>>>(s.HG, s.rs, dm.toff, dm.B, dm.N, dm.T, H,
                                          p.max_head_clusters, p.head_eps, s.omega, tv, s.status);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  k_energy<<<dm.B, 1024, 0, st>>>(s.omega, s.zn2, s.sigma, s.W2, dm.toff, dm.B, dm.N, dm.T, H,
                                  s.ebar, tv, s.status);
  return cudaGetLastError();
}

}  // namespace gmc
