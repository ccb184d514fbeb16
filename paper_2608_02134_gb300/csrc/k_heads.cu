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

// One block per image: reduce the Gram, farthest-first clustering, omega_h.
// Ties: the first centre is the lowest-index largest pattern, each next centre
// the lowest-index head of smallest max-cosine, and a head joins the earliest
// centre among equally similar ones.
__global__ void k_head_cluster(const double* __restrict__ hgpart, int nHG,
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
  for (int p = threadIdx.x; p < H * H; p += blockDim.x) {
    double s = 0.0;
    for (int k = 0; k < nHG; ++k) s += hgpart[((size_t)b * nHG + k) * H * H + p];
    HG[p] = s;
  }
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
  if (threadIdx.x != 0) return;
  int centres[GMC_MAX_HEADS];
  int assign[GMC_MAX_HEADS];
  bool is_c[GMC_MAX_HEADS];
  const int nc = min(max_clusters, H);
  int first = 0;
  for (int h = 1; h < H; ++h)
    if (pre[h] > pre[first]) first = h;
  for (int h = 0; h < H; ++h) is_c[h] = false;
  centres[0] = first;
  is_c[first] = true;
  for (int c = 1; c < nc; ++c) {
    int best = -1;
    double bv = 0.0;
    for (int h = 0; h < H; ++h) {
      if (is_c[h]) continue;
      double mc = -INFINITY;
      for (int k = 0; k < c; ++k) mc = fmax(mc, cs[h * H + centres[k]]);
      if (best < 0 || mc < bv) { best = h; bv = mc; }
    }
    centres[c] = best;
    is_c[best] = true;
  }
  int count[GMC_MAX_HEADS];
  for (int k = 0; k < nc; ++k) count[k] = 0;
  for (int h = 0; h < H; ++h) {
    int bk = 0;
    for (int k = 1; k < nc; ++k)
      if (cs[h * H + centres[k]] > cs[h * H + centres[bk]]) bk = k;
    assign[h] = bk;
    count[bk]++;
  }
  int C = 0;
  for (int k = 0; k < nc; ++k) C += count[k] > 0;
  for (int k = 0; k < nc; ++k) {
    if (count[k] == 0) continue;
    double nrm2 = 0.0;  // ||sum_{g in c} u_g||^2
    for (int g = 0; g < H; ++g)
      if (assign[g] == k)
        for (int g2 = 0; g2 < H; ++g2)
          if (assign[g2] == k) nrm2 += cs[g * H + g2];
    const double nrm = nrm2 > 0.0 ? sqrt(nrm2) : 0.0;
    double invsum = 0.0;
    for (int h = 0; h < H; ++h) {
      if (assign[h] != k) continue;
      double dot = 0.0;
      for (int g = 0; g < H; ++g)
        if (assign[g] == k) dot += cs[h * H + g];
      const double dh = 1.0 - (nrm > 0.0 ? dot / nrm : 0.0);
      pre[h] = 1.0 / (dh + head_eps);  // reuse: inverse-dispersion weight
      invsum += pre[h];
    }
    for (int h = 0; h < H; ++h)
      if (assign[h] == k) omega[(size_t)b * H + h] = (float)(pre[h] / invsum / C);
  }
  if (tv.base) {
    gmc_trace_header* hd = tv.header(b);
    hd->n_clusters = C;
    int32_t* tc = tv.at<int32_t>(b, tv.off_centres);
    for (int k = 0; k < max_clusters; ++k) tc[k] = k < nc ? centres[k] : -1;
    int32_t* ta = tv.at<int32_t>(b, tv.off_head_assign);
    float* to = tv.at<float>(b, tv.off_omega);
    for (int h = 0; h < H; ++h) {
      ta[h] = assign[h];
      to[h] = omega[(size_t)b * H + h];
    }
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
  size_t smem2 = sizeof(double) * (2 * (size_t)H * H + H);
  if ((e = set_smem_limit((const void*)k_head_cluster, smem2)) != cudaSuccess) return e;
  k_head_cluster<<<dm.B, 128, smem2, st>>>(s.hgpart, s.nHG, s.rs, dm.toff, dm.B, dm.N, dm.T, H,
                                          p.max_head_clusters, p.head_eps, s.omega, tv, s.status);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  k_energy<<<dm.B, 1024, 0, st>>>(s.omega, s.zn2, s.sigma, s.W2, dm.toff, dm.B, dm.N, dm.T, H,
                                  s.ebar, tv, s.status);
  return cudaGetLastError();
}

}  // namespace gmc
