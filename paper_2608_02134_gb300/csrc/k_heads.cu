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
constexpr int HG_HB = 4;                        // heads per register tile side

__device__ __forceinline__ float query_weight(int t, int Tb, float wq) {
  return (t == Tb - 1 ? wq : 1.f) / ((float)(Tb - 1) + wq);
}

__device__ __forceinline__ int pair_index(int h, int g, int H) {  // h <= g, h-major
  return h * H - h * (h - 1) / 2 + (g - h);
}

// Per block: TOK tokens (8, or 9 where that puts one image's blocks in one wave), all head
// pairs (h <= g).  Writes the block's part
// of the pattern Gram (an fp32 sum over its TOK tokens, stored as fp64 for
// the cross-block sum) and W2[h,i] = sum_t nu_t A[h,t,i]^2.  The per-token
// sums over queries are register tiles of 4 x 4 head pairs: 8 shared loads
// feed 16 FMAs.
template <int TOK>
__global__ void k_head_stats(const float* __restrict__ A, const float* __restrict__ Z,
                             const float* __restrict__ sigma, const int32_t* toff, int B, int N,
                             int Tmax, int H, float wq, double* hgpart, int nHG, float* W2,
                             uint32_t* status) {
  grid_dep_wait();
  constexpr int RS = HG_TC * TOK + 2;  // row stride of a staged head: 4 rows apart land 8 banks apart
  extern __shared__ float sm_hs[];
  __shared__ float sgm[GMC_MAX_HEADS];  // sigma_h of the image
  const int b = blockIdx.y;
  const TextGeom tg = text_geom(toff, b, B, Tmax, status);
  if (tg.T == 0) return;
  for (int h = threadIdx.x; h < H; h += blockDim.x) sgm[h] = sigma[(size_t)b * H + h];
  const int Tb = tg.T;
  const int npairs = H * (H + 1) / 2;
  const int nhb = (H + HG_HB - 1) / HG_HB, Hp = nhb * HG_HB;
  const int ntiles = nhb * (nhb + 1) / 2;
  float* Abuf = sm_hs;                          // [2][Hp][RS], rows >= H stay zero
  float* acc = Abuf + 2 * (size_t)Hp * RS;   // [2][npairs][TOK], one per block half
  float* w2 = acc + 2 * (size_t)npairs * TOK;  // [2][H][TOK]
  float4* zs = reinterpret_cast<float4*>(w2 + 2 * H * TOK);  // [H][TOK] probe values
  unsigned short* tiles = reinterpret_cast<unsigned short*>(zs + H * TOK);  // [ntiles]
  const int i0 = blockIdx.x * TOK;
  for (int p = threadIdx.x; p < 2 * npairs * TOK; p += blockDim.x) acc[p] = 0.f;
  for (int p = threadIdx.x; p < 2 * H * TOK; p += blockDim.x) w2[p] = 0.f;
  for (int p = H * RS + threadIdx.x; p < Hp * RS; p += blockDim.x) {
    Abuf[p] = 0.f;
    Abuf[(size_t)Hp * RS + p] = 0.f;
  }
  if (threadIdx.x == 0) {
    int p = 0;
    for (int hb = 0; hb < nhb; ++hb)
      for (int gb = hb; gb < nhb; ++gb) tiles[p++] = (unsigned short)(hb * 256 + gb);
  }
  // the block's probe values Z_h[i] for every head (used by the output step)
  for (int q = threadIdx.x; q < H * TOK; q += blockDim.x) {
    const int h = q / TOK, i = i0 + q % TOK;
    zs[q] = i < N ? reinterpret_cast<const float4*>(Z)[((size_t)b * H + h) * N + i]
                  : make_float4(0.f, 0.f, 0.f, 0.f);
  }
  // Queries in pairs of HG_TC-chunks: both are staged, then the two halves of
  // the block work on one chunk each into their own sums.  The TOK tokens
  // of one (head, query) row are read as 16-byte loads when the rows of A
  // start on 16 bytes (N % 4 == 0) and the block is not the ragged last one
  // (the padded shared rows are not 16-byte aligned, so these go through
  // registers); otherwise as 4-byte cp.async copies.
  const bool vec = TOK % 4 == 0 && (N & 3) == 0 && i0 + TOK <= N;
  auto stage = [&](int t0, float* buf) {
    const int tc = min(HG_TC, Tb - t0);
    if (vec) {
      constexpr int V = TOK / 4;  // 16-byte pieces per row
      for (int idx = threadIdx.x; idx < H * HG_TC * V; idx += blockDim.x) {
        const int h = idx / (HG_TC * V), tt = (idx / V) % HG_TC, v = idx % V;
        float* dst = buf + h * RS + tt * TOK + 4 * v;
        float4 x = make_float4(0.f, 0.f, 0.f, 0.f);
        if (tt < tc)
          x = *reinterpret_cast<const float4*>(A + (((size_t)b * H + h) * Tmax + t0 + tt) * N + i0 +
                                               4 * v);
        dst[0] = x.x;
        dst[1] = x.y;
        dst[2] = x.z;
        dst[3] = x.w;
      }
    } else {
      for (int idx = threadIdx.x; idx < H * HG_TC * TOK; idx += blockDim.x) {
        const int h = idx / (HG_TC * TOK), tt = (idx / TOK) % HG_TC, ii = idx % TOK;
        const bool in = tt < tc && i0 + ii < N;
        const float* src = in ? A + (((size_t)b * H + h) * Tmax + t0 + tt) * N + i0 + ii : A;
        cp_async4(buf + h * RS + tt * TOK + ii, src, in);
      }
    }
    cp_async_commit();
  };
  const int hsz = blockDim.x / 2, half = threadIdx.x / hsz, ht = threadIdx.x % hsz;
  float* accH = acc + (size_t)half * npairs * TOK;
  float* w2H = w2 + (size_t)half * H * TOK;
  for (int tp = 0; tp < Tb; tp += 2 * HG_TC) {
    __syncthreads();  // both buffers are free
    stage(tp, Abuf);
    stage(tp + HG_TC, Abuf + (size_t)Hp * RS);
    cp_async_wait<0>();
    __syncthreads();
    const int t0 = tp + half * HG_TC;
    const int tc = max(0, min(HG_TC, Tb - t0));
    const float* Ablk = Abuf + (size_t)half * Hp * RS;
    for (int task = ht; task < ntiles * TOK; task += hsz) {
      const int tile = task / TOK, ii = task % TOK;
      const int hb = tiles[tile] >> 8, gb = tiles[tile] & 255;
      const float* ah = Ablk + (size_t)hb * HG_HB * RS + ii;
      const float* ag = Ablk + (size_t)gb * HG_HB * RS + ii;
      float sacc[HG_HB][HG_HB];
#pragma unroll
      for (int u = 0; u < HG_HB; ++u)
#pragma unroll
        for (int v = 0; v < HG_HB; ++v) sacc[u][v] = 0.f;
      for (int tt = 0; tt < tc; ++tt) {
        float x[HG_HB], y[HG_HB];
#pragma unroll
        for (int u = 0; u < HG_HB; ++u) {
          x[u] = ah[u * RS + tt * TOK];
          y[u] = ag[u * RS + tt * TOK];
        }
#pragma unroll
        for (int u = 0; u < HG_HB; ++u)
#pragma unroll
          for (int v = 0; v < HG_HB; ++v) sacc[u][v] = fmaf(x[u], y[v], sacc[u][v]);
      }
#pragma unroll
      for (int u = 0; u < HG_HB; ++u)
#pragma unroll
        for (int v = 0; v < HG_HB; ++v) {
          const int h = hb * HG_HB + u, g = gb * HG_HB + v;
          if (h <= g && g < H) accH[pair_index(h, g, H) * TOK + ii] += sacc[u][v];
        }
    }
    for (int q = ht; q < H * TOK; q += hsz) {
      const int h = q / TOK, ii = q % TOK;
      const float* ah = Ablk + h * RS;
      float sw = 0.f;
      for (int tt = 0; tt < tc; ++tt) {
        const float a = ah[tt * TOK + ii];
        sw = fmaf(query_weight(t0 + tt, Tb, wq) * a, a, sw);
      }
      w2H[q] += sw;
    }
  }
  __syncthreads();
  double* out = hgpart + ((size_t)b * nHG + blockIdx.x) * H * H;
  for (int p = threadIdx.x; p < H * H; p += blockDim.x) {
    const int h = p / H, g = p % H;
    if (h > g) continue;
    const int pi = pair_index(h, g, H);
    const float sh = sgm[h], sgv = sgm[g];
    float v = 0.f;
    for (int ii = 0; ii < TOK; ++ii) {
      const int i = i0 + ii;
      if (i >= N) break;
      const float4 zh = zs[h * TOK + ii];
      const float4 zg = zs[g * TOK + ii];
      const float w = fmaf(zh.x, zg.x, fmaf(zh.y, zg.y, fmaf(zh.z, zg.z, fmaf(zh.w, zg.w, sh * sgv))));
      v = fmaf(w, acc[pi * TOK + ii] + acc[((size_t)npairs + pi) * TOK + ii], v);
    }
    out[h * H + g] = v;
    out[g * H + h] = v;
  }
  for (int q = threadIdx.x; q < H * TOK; q += blockDim.x) {
    const int h = q / TOK, i = i0 + q % TOK;
    if (i < N) W2[((size_t)b * H + h) * N + i] = w2[q] + w2[H * TOK + q];
  }
}

// Ties: the first centre is the lowest-index largest pattern, each next centre
// the lowest-index head of smallest max-cosine, and a head joins the earliest
// centre among equally similar ones.
__device__ __forceinline__ void warp_argbest(float& v, int& idx, bool want_max) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float ov = __shfl_xor_sync(FULL, v, o);
    const int oi = __shfl_xor_sync(FULL, idx, o);
    const bool better = want_max ? (ov > v || (ov == v && oi < idx))
                                 : (ov < v || (ov == v && oi < idx));
    if (oi >= 0 && (idx < 0 || better)) { v = ov; idx = oi; }
  }
}

// Farthest-first head clusters and head weights of image b from its reduced
// pattern Gram (fp64 sums, read past L1: other blocks wrote them).  The
// cosines, dispersions and weights are fp32: the weights enter as
// 1 / (dispersion + head_eps) with head_eps = 0.05 by default, far above the
// fp32 rounding of a cosine.  One block of 256 threads, one warp for the
// centres (two heads per lane, H <= 64).
__device__ void cluster_heads(const double* hgb, int b, int T, int N, int H, int max_clusters,
                              float head_eps, float* omega, const TraceView& tv, float* sm,
                              const ViewGrams& vg) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  float* cs = sm;                       // [H*H] pattern cosines
  float* pre = cs + H * H;              // [H]   pattern norm / mean atom norm
  float* dot = pre + H;                 // [H]   1/||U_h||, later h's cosine sum in its cluster
  float* inv = dot + H;                 // [H]   1 / (dispersion + eps)
  float* csum = inv + H;                // [GMC_MAX_HEADS] 1 / norm of a cluster's sum
  float* isum = csum + GMC_MAX_HEADS;   // [GMC_MAX_HEADS]
  int* asg = reinterpret_cast<int*>(isum + GMC_MAX_HEADS);  // [H] cluster of every head
  int* cent = asg + H;                  // [GMC_MAX_HEADS] centres
  int* ccnt = cent + GMC_MAX_HEADS;     // [GMC_MAX_HEADS] cluster sizes
  const float TN = (float)T * (float)N;
  if (vg.n > 1) {
    // patterns over the views (Eq. (cond-head-pattern)): with U_h^v the view's
    // atoms over their mean norm m_v[h] = sum_t rs_v[h,t] / (T N),
    // <u_h, u_g> = sum_v beta_v G_v[h][g] / (m_v[h] m_v[g])
    const int HE = H * H + H;
    for (int h = threadIdx.x; h < H; h += blockDim.x) {
      float a = 0.f;
      for (int v = 0; v < vg.n; ++v) {
        const double* hv = vg.HG[v] + (size_t)b * HE;
        const float m = (float)__ldcg(&hv[H * H + h]) / TN;
        if (m > 0.f) a += vg.beta[v] * (float)__ldcg(&hv[h * H + h]) / (m * m);
      }
      pre[h] = a > 0.f ? sqrtf(a) : 0.f;
      dot[h] = a > 0.f ? 1.f / sqrtf(a) : 0.f;
    }
    __syncthreads();
    for (int p = threadIdx.x; p < H * H; p += blockDim.x) {
      const int h = p / H, g = p % H;
      float x = 0.f;
      for (int v = 0; v < vg.n; ++v) {
        const double* hv = vg.HG[v] + (size_t)b * HE;
        const float mh = (float)__ldcg(&hv[H * H + h]) / TN, mg = (float)__ldcg(&hv[H * H + g]) / TN;
        if (mh > 0.f && mg > 0.f) x += vg.beta[v] * (float)__ldcg(&hv[p]) / (mh * mg);
      }
      cs[p] = x * dot[h] * dot[g];
    }
    __syncthreads();
  } else {
    for (int h = threadIdx.x; h < H; h += blockDim.x) {
      const float a = (float)__ldcg(&hgb[h * H + h]);
      const float mean = (float)__ldcg(&hgb[H * H + h]) / TN;  // sum_t rs / (T N)
      pre[h] = (mean > 0.f && a > 0.f) ? sqrtf(a) / mean : 0.f;
      dot[h] = a > 0.f ? 1.f / sqrtf(a) : 0.f;  // 1 / ||U_h||, 0 for a zero pattern
    }
    __syncthreads();
    for (int p = threadIdx.x; p < H * H; p += blockDim.x) {
      const int h = p / H, g = p % H;
      cs[p] = (float)__ldcg(&hgb[p]) * dot[h] * dot[g];
    }
    __syncthreads();
  }
  const int nc = min(max_clusters, H);
  if (wid == 0) {  // farthest-first centres, two heads per lane (H <= 64)
    const int h0 = lane, h1 = lane + 32;
    bool c0 = false, c1 = false;  // is h0 / h1 a centre
    float mc0 = -INFINITY, mc1 = -INFINITY;  // largest cosine of h0 / h1 to a centre
    int newest;                              // the latest centre (the same in every lane)
    {
      float v = -1.f;
      int idx = -1;
      if (h0 < H) { v = pre[h0]; idx = h0; }
      if (h1 < H && (idx < 0 || pre[h1] > v)) { v = pre[h1]; idx = h1; }
      warp_argbest(v, idx, true);
      if (lane == 0) cent[0] = idx;
      c0 = (h0 == idx);
      c1 = (h1 == idx);
      newest = idx;
    }
    for (int c = 1; c < nc; ++c) {
      if (h0 < H) mc0 = fmaxf(mc0, cs[h0 * H + newest]);
      if (h1 < H) mc1 = fmaxf(mc1, cs[h1 * H + newest]);
      float v = 0.f;
      int idx = -1;
      for (int q = 0; q < 2; ++q) {
        const int h = q ? h1 : h0;
        if (h >= H || (q ? c1 : c0)) continue;
        const float mc = q ? mc1 : mc0;
        if (idx < 0 || mc < v) { v = mc; idx = h; }
      }
      warp_argbest(v, idx, false);
      if (lane == 0) cent[c] = idx;
      c0 |= (h0 == idx);
      c1 |= (h1 == idx);
      newest = idx;
    }
  }
  __syncthreads();
  // each head joins its most similar centre (the earliest among equals)
  for (int h = threadIdx.x; h < H; h += blockDim.x) {
    int bk = 0;
    for (int k = 1; k < nc; ++k)
      if (cs[h * H + cent[k]] > cs[h * H + cent[bk]]) bk = k;
    asg[h] = bk;
  }
  __syncthreads();
  // sums over heads as warp trees (two heads per lane, fixed order)
  const int nw = blockDim.x >> 5;
  for (int h = wid; h < H; h += nw) {
    float d = 0.f;
    if (lane < H && asg[lane] == asg[h]) d += cs[h * H + lane];
    if (lane + 32 < H && asg[lane + 32] == asg[h]) d += cs[h * H + lane + 32];
    d = warp_sum(d);
    if (lane == 0) dot[h] = d;
  }
  __syncthreads();
  // ||sum_{g in k} u_g||^2 (in cosine units) = sum over the cluster's dot values
  for (int k = wid; k < nc; k += nw) {
    float sk = 0.f;
    int n = 0;
    if (lane < H && asg[lane] == k) { sk += dot[lane]; ++n; }
    if (lane + 32 < H && asg[lane + 32] == k) { sk += dot[lane + 32]; ++n; }
    sk = warp_sum(sk);
    n = warp_sum_int(n);
    if (lane == 0) {
      csum[k] = sk > 0.f ? rsqrtf(sk) : 0.f;  // 1 / ||sum_{g in k} u_g||
      ccnt[k] = n;
    }
  }
  __syncthreads();
  for (int h = threadIdx.x; h < H; h += blockDim.x) {
    const float dh = 1.f - dot[h] * csum[asg[h]];
    inv[h] = 1.f / (dh + head_eps);
  }
  __syncthreads();
  for (int k = wid; k < nc; k += nw) {
    float sk = 0.f;
    if (lane < H && asg[lane] == k) sk += inv[lane];
    if (lane + 32 < H && asg[lane + 32] == k) sk += inv[lane + 32];
    sk = warp_sum(sk);
    if (lane == 0) isum[k] = sk;
  }
  __syncthreads();
  int C = 0;
  for (int k = 0; k < nc; ++k) C += ccnt[k] > 0;
  for (int h = threadIdx.x; h < H; h += blockDim.x) {
    const float w = inv[h] / isum[asg[h]] / (float)C;
    omega[(size_t)b * H + h] = w;
    if (tv.base) {
      tv.at<int32_t>(b, tv.off_head_assign)[h] = asg[h];
      tv.at<float>(b, tv.off_omega)[h] = w;
    }
  }
  if (tv.base) {
    if (threadIdx.x == 0) tv.header(b)->n_clusters = C;
    int32_t* tc = tv.at<int32_t>(b, tv.off_centres);
    for (int k = threadIdx.x; k < max_clusters; k += blockDim.x) tc[k] = k < nc ? cent[k] : -1;
  }
}

// The pattern Gram of image blockIdx.y: sum of the token-block partials, one
// warp per entry, lanes over the blocks (fixed order, so the sum is
// reproducible); further warps sum every head's atom norms sum_t rs[h,t] (rs
// in nRS parts per query).  HG[b] holds the H*H Gram followed by the H
// atom-norm totals.  The image's last block to finish (ticket zeroed with the
// status word) clusters the heads.
__global__ void __launch_bounds__(256) k_hg_reduce(const double* __restrict__ hgpart, int nHG,
                                                     int B, int N, int H,
                                                     const float* __restrict__ rs, int nRS,
                                                     const int32_t* toff, int Tmax, double* HG,
                                                     uint32_t* tick, int max_clusters,
                                                     float head_eps, float* omega, TraceView tv,
                                                     int cluster, const ViewGrams vg,
                                                     uint32_t* status) {
  grid_dep_wait();
  extern __shared__ float sm_hc[];
  __shared__ int last;
  const int lane = threadIdx.x & 31, b = blockIdx.y;
  const int HH = H * H, HE = HH + H;
  const TextGeom tg = text_geom(toff, b, B, Tmax, status);
  if (tg.T == 0) return;  // uniform over the image
  const int p = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (p < HE) {
    double s = 0.0;
    if (p < HH) {
      for (int k = lane; k < nHG; k += 32) s += hgpart[((size_t)b * nHG + k) * HH + p];
    } else {
      const int h = p - HH;
      const float* r = rs + ((size_t)b * H + h) * nRS * Tmax;
      for (int k = lane; k < nRS * Tmax; k += 32)
        if (k % Tmax < tg.T) s += r[k];
    }
    s = warp_sum(s);
    if (lane == 0) HG[(size_t)b * HE + p] = s;
  }
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) last = atomicAdd(&tick[b], 1u) == gridDim.x - 1;
  __syncthreads();
  if (!last || !cluster) return;  // a historical view's Gram waits for the current view's call
  __threadfence();
  cluster_heads(HG + (size_t)b * HE, b, tg.T, N, H, max_clusters, head_eps, omega, tv, sm_hc, vg);
}

// Dynamic shared memory of k_head_stats for H heads: both staged query
// chunks, both halves' pair sums and query-weighted squares, the probe values
// and the tile list.
static size_t head_stats_smem(int H, int tok) {
  const int npairs = H * (H + 1) / 2;
  const int nhb = (H + HG_HB - 1) / HG_HB;
  const int rs = HG_TC * tok + 2;
  return sizeof(float) * (2 * (size_t)nhb * HG_HB * rs + 2 * (size_t)npairs * tok + 2 * H * tok) +
         sizeof(float4) * H * tok + sizeof(unsigned short) * (nhb * (nhb + 1) / 2) + 16;
}

int head_tokens(int B, int N, int H) {
  static int sms = 0;
  if (sms == 0) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
      cudaGetLastError();
      sms = 152;
    }
  }
  const long long b8 = (long long)B * ceil_div(N, 8), b9 = (long long)B * ceil_div(N, 9);
  return b8 > sms && b9 <= sms && head_stats_smem(H, 9) <= 227 * 1024 ? 9 : 8;
}

// Whether the head statistics of H heads fit one block's shared memory
// (227 KB on sm_103a): H <= 56.
bool heads_supported(int H) { return H >= 1 && head_stats_smem(H, 8) <= 227 * 1024; }

cudaError_t launch_heads(const Dims& dm, const gmc_params& p, Scratch& s, const TraceView& tv,
                         cudaStream_t st, int cluster, const ViewGrams* views) {
  const int H = dm.H;
  const int tok = s.hgtok;
  const size_t smem = head_stats_smem(H, tok);
  const void* kf = tok == 9 ? (const void*)k_head_stats<9> : (const void*)k_head_stats<8>;
  cudaError_t e = set_smem_limit(kf, smem);
  if (e != cudaSuccess) return e;
  if (tok == 9)
    launch_k(k_head_stats<9>, dim3(s.nHG, dm.B), 512, smem, st, 1, s.A, s.Z, s.sigma, dm.toff, dm.B,
             dm.N, dm.T, H, p.terminal_q_weight, s.hgpart, s.nHG, s.W2, s.status);
  else
    launch_k(k_head_stats<8>, dim3(s.nHG, dm.B), 512, smem, st, 1, s.A, s.Z, s.sigma, dm.toff, dm.B,
             dm.N, dm.T, H, p.terminal_q_weight, s.hgpart, s.nHG, s.W2, s.status);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  const size_t smem2 = sizeof(float) * ((size_t)H * H + 3 * H + 2 * GMC_MAX_HEADS) +
                       sizeof(int) * (H + 2 * GMC_MAX_HEADS);
  if ((e = set_smem_limit((const void*)k_hg_reduce, smem2)) != cudaSuccess) return e;
  launch_k(k_hg_reduce, dim3(ceil_div(H * H + H, 8), dm.B), 256, smem2, st, 1,
           (const double*)s.hgpart, s.nHG, dm.B, dm.N, H, (const float*)s.rs, s.nRS, dm.toff, dm.T,
           s.HG, s.tick3, p.max_head_clusters, p.head_eps, s.omega, tv, cluster,
           views ? *views : ViewGrams{}, s.status);
  return cudaGetLastError();
}

}  // namespace gmc
