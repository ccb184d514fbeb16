// Population assignment (appendix Eq. (cond-assignment), (cond-population-gate)).
//
// For a discarded token i, delta_i is the gap between its largest and
// second-largest cosine to the support (0 when |S| = 1); Delta_bar is the mean
// gap over the discarded tokens (0 when none is discarded);
//   s_x = 1 - exp(-(Delta_bar / gate_scale)^gate_pow)
//   g_i = exp(-(delta_i / ambig_margin)^gate_pow)
//   pi(i) = argmax_{j in S} cos_ij + lambda_p s_x g_i exp(-||p_i - p_j||^2 / tau_s)
// (ties to the lowest j); selected tokens represent themselves.  With I > 1
// images per prompt (Ng = N / I tokens each, one after another) token i's
// candidates, its gap and its coordinates are those of its own image.  The
// population weights are m_i = (1 - alpha s_x) + alpha s_x ebar_i.  Token i
// also sets bit i of its carrier's membership bitmap (atomicOr: the bitmap
// does not depend on the order of the writes), which the transport reads
// instead of scanning the whole assignment.
//
// Layout.  A block takes AT = 32 consecutive tokens, one per lane, and its
// ASSIGN_WARPS warps split the support (warp w: entries w, w + 8, ...).  The
// cosines of support entry k with the block's tokens are one contiguous
// 128-byte segment: row S_k of the symmetric N x N cosine matrix, or row k of
// the K x N support cosines of long prefixes (cs mode).  So both passes read
// exactly K x N values, coalesced, and no lane divides or gathers per entry:
// the support's images and grid coordinates are staged once per block.  The
// warps' partial results (top two cosines; best kappa and its entry, ties to
// the lower entry) are merged in shared memory.
#include "common.cuh"
#include "kernels.cuh"

namespace gmc {

namespace {
constexpr int AT = 32;  // tokens per block (one per lane)
constexpr int AU = 8;   // support entries each lane loads before using them

// Cosine row of support entry k (token j) for image b: its cosines with every token.
__device__ __forceinline__ const float* support_row(const float* cos, int cs_mode, int b, int N,
                                                    int K, int k, int j) {
  return cs_mode ? cos + ((size_t)b * K + k) * N : cos + ((size_t)b * N + j) * N;
}
}  // namespace

// Pass 1: delta_i per discarded token; per-block partial sums of delta and counts.
// Also the message energy of every token (appendix Eq. (cond-grounded-energy)):
//   e_i = (sum_h omega_h g_h(i)^2 sum_t nu_t A[h,t,i]^2)^{1/2},  g_h(i)^2 = ||Z_h[i]||^2 + sigma_h^2,
// and per-block sums of e (the mean normalises ebar in pass 2).  The last block
// of an image to finish (ticket) adds the block partials in a fixed order and
// stores Delta_bar, s_x and the mean energy for pass 2.
__global__ void __launch_bounds__(32 * ASSIGN_WARPS) k_assign_gap(
    const float* __restrict__ cos, int cs_mode, const int32_t* __restrict__ support,
    const int32_t* __restrict__ slot, const int32_t* toff, int B, int N, int K, int Tmax, int H,
    const float* __restrict__ omega, const float* __restrict__ zn2,
    const float* __restrict__ sigma, const float* __restrict__ W2, float* energy, float* epart,
    float* delta, double* dpart, int nA, float gate_scale, float gate_pow, int I, uint32_t* tick,
    float* gatev, uint32_t* status) {
  grid_dep_wait();
  __shared__ float pm1[ASSIGN_WARPS][AT], pm2[ASSIGN_WARPS][AT], pe2[ASSIGN_WARPS][AT];
  __shared__ int pnc[ASSIGN_WARPS][AT];
  __shared__ int last;
  extern __shared__ int sS[];  // [K] support, then [K] its images
  int* sImg = sS + K;
  const int b = blockIdx.y;
  const TextGeom tg = text_geom(toff, b, B, Tmax, status);
  if (tg.T == 0) return;
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int Ng = N / I;
  const int i = blockIdx.x * AT + lane;
  for (int k = threadIdx.x; k < K; k += blockDim.x) {
    const int j = support[(size_t)b * K + k];
    sS[k] = j;
    sImg[k] = j / Ng;
  }
  __syncthreads();
  const bool tok = i < N;
  const int img = tok ? i / Ng : -1;
  // top two cosines of this lane's token over the warp's share of the support
  float m1 = -INFINITY, m2 = -INFINITY;
  int nc = 0;
  for (int k0 = w; k0 < K; k0 += ASSIGN_WARPS * AU) {
    float v[AU];
    bool ok[AU];
#pragma unroll
    for (int u = 0; u < AU; ++u) {
      const int k = k0 + ASSIGN_WARPS * u;
      ok[u] = tok && k < K && sImg[k] == img;
      v[u] = ok[u] ? support_row(cos, cs_mode, b, N, K, k, sS[k])[i] : 0.f;
    }
#pragma unroll
    for (int u = 0; u < AU; ++u) {
      if (!ok[u]) continue;
      ++nc;
      if (v[u] > m1) { m2 = m1; m1 = v[u]; } else if (v[u] > m2) { m2 = v[u]; }
    }
  }
  // the message energy's head terms, the heads split over the warps
  float e2w = 0.f;
  if (tok)
    for (int h = w; h < H; h += ASSIGN_WARPS) {
      const size_t o = ((size_t)b * H + h) * N + i;
      const float sg = sigma[(size_t)b * H + h];
      e2w = fmaf(omega[(size_t)b * H + h] * (zn2[o] + sg * sg), W2[o], e2w);
    }
  pm1[w][lane] = m1;
  pm2[w][lane] = m2;
  pnc[w][lane] = nc;
  pe2[w][lane] = e2w;
  __syncthreads();
  if (w == 0) {
    // merge the warps' top two (order-independent) and their energy terms (fixed order)
    float e2 = e2w;
    for (int q = 1; q < ASSIGN_WARPS; ++q) {
      const float b1 = pm1[q][lane], b2 = pm2[q][lane];
      const float hi = fmaxf(m1, b1);
      m2 = fmaxf(fminf(m1, b1), fmaxf(m2, b2));
      m1 = hi;
      nc += pnc[q][lane];
      e2 += pe2[q][lane];
    }
    float e = 0.f;
    double dv = 0.0;
    int dc = 0;
    if (tok) {
      e = sqrtf(e2);
      energy[(size_t)b * N + i] = e;
      const bool disc = slot[(size_t)b * N + i] < 0;
      const float d = disc && nc > 1 ? m1 - m2 : 0.f;
      delta[(size_t)b * N + i] = d;
      if (disc) {
        dv = d;
        dc = 1;
      }
    }
    // block partials in a fixed order: the lanes by a shuffle tree
    dv = warp_sum(dv);
    dc = warp_sum_int(dc);
    e = warp_sum(e);
    if (lane == 0) {
      dpart[((size_t)b * nA + blockIdx.x) * 2 + 0] = dv;
      dpart[((size_t)b * nA + blockIdx.x) * 2 + 1] = (double)dc;
      epart[(size_t)b * nA + blockIdx.x] = e;
      __threadfence();
      last = atomicAdd(&tick[b], 1u) == (unsigned)(nA - 1);
    }
  }
  __syncthreads();
  if (last && w == 0) {  // the partials in a fixed order (fp32: at most 2 N per image)
    __threadfence();
    float s = 0.f, c = 0.f, et = 0.f;
    for (int q = lane; q < nA; q += 32) {
      s += (float)__ldcg(&dpart[((size_t)b * nA + q) * 2 + 0]);
      c += (float)__ldcg(&dpart[((size_t)b * nA + q) * 2 + 1]);
      et += __ldcg(&epart[(size_t)b * nA + q]);
    }
    s = warp_sum(s);
    c = warp_sum(c);
    et = warp_sum(et);
    if (lane == 0) {
      const float db = c > 0.f ? s / c : 0.f;
      gatev[(size_t)b * 4 + 0] = db;
      gatev[(size_t)b * 4 + 1] = 1.f - expf(-powf(db / gate_scale, gate_pow));
      gatev[(size_t)b * 4 + 2] = et / (float)N;
    }
  }
}

// Pass 2: s_x, the gated spatial assignment, and the population weights.
__global__ void __launch_bounds__(32 * ASSIGN_WARPS) k_assign_pick(
    const float* __restrict__ cos, int cs_mode, const int32_t* __restrict__ support,
    const int32_t* __restrict__ slot, const float* __restrict__ delta,
    const float* __restrict__ gatev, const float* __restrict__ energy, const int32_t* toff,
    int B, int N, int K, int Tmax, int gh, int gw, float gate_pow, float ambig_margin,
    float lambda_p, float tau_s, float alpha, int I, int32_t* pi, float* mass, uint32_t* mbits,
    TraceView tv, uint32_t* status) {
  grid_dep_wait();
  __shared__ float pbest[ASSIGN_WARPS][AT];
  __shared__ int pk[ASSIGN_WARPS][AT];
  extern __shared__ int sS[];  // [K] support, [K] images, [K] y and [K] x coordinates
  int* sImg = sS + K;
  float* spy = reinterpret_cast<float*>(sImg + K);
  float* spx = spy + K;
  const int b = blockIdx.y;
  const TextGeom tg = text_geom(toff, b, B, Tmax, status);
  if (tg.T == 0) return;
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int Ng = N / I;
  for (int k = threadIdx.x; k < K; k += blockDim.x) {
    const int j = support[(size_t)b * K + k];
    const int im = j / Ng, jl = j - im * Ng;  // coordinates in its own image's grid
    sS[k] = j;
    sImg[k] = im;
    spy[k] = ((jl / gw) + 0.5f) / gh;
    spx[k] = ((jl % gw) + 0.5f) / gw;
  }
  const float dbar = gatev[(size_t)b * 4 + 0], sxg = gatev[(size_t)b * 4 + 1];
  const float emean = gatev[(size_t)b * 4 + 2];
  __syncthreads();
  if (blockIdx.x == 0 && threadIdx.x == 0 && tv.base) {
    tv.header(b)->s_x = sxg;
    tv.header(b)->delta_bar = dbar;
  }
  const int i = blockIdx.x * AT + lane;
  const bool tok = i < N;
  const bool disc = tok && slot[(size_t)b * N + i] < 0;
  const int img = tok ? i / Ng : -1, il = tok ? i - img * Ng : 0;
  const float piy = ((il / gw) + 0.5f) / gh, pix = ((il % gw) + 0.5f) / gw;
  float coef = 0.f;
  if (disc) {
    const float gi = expf(-powf(delta[(size_t)b * N + i] / ambig_margin, gate_pow));
    coef = lambda_p * sxg * gi;
  }
  float best = -INFINITY;
  int bk = 0x7fffffff;
  if (disc) {
    for (int k0 = w; k0 < K; k0 += ASSIGN_WARPS * AU) {
      float v[AU];
      bool ok[AU];
#pragma unroll
      for (int u = 0; u < AU; ++u) {
        const int k = k0 + ASSIGN_WARPS * u;
        ok[u] = k < K && sImg[k] == img;  // a carrier of the token's own image
        v[u] = ok[u] ? support_row(cos, cs_mode, b, N, K, k, sS[k])[i] : 0.f;
      }
#pragma unroll
      for (int u = 0; u < AU; ++u) {
        if (!ok[u]) continue;
        const int k = k0 + ASSIGN_WARPS * u;
        float x = v[u];
        if (coef > 0.f) {
          const float dy = spy[k] - piy, dx = spx[k] - pix;
          x += coef * expf(-(dy * dy + dx * dx) / tau_s);
        }
        if (x > best) { best = x; bk = k; }  // k ascending within a warp: first maximum kept
      }
    }
  }
  pbest[w][lane] = best;
  pk[w][lane] = bk;
  __syncthreads();
  if (w != 0 || !tok) return;
  for (int q = 1; q < ASSIGN_WARPS; ++q) {
    const float ob = pbest[q][lane];
    const int ok = pk[q][lane];
    if (ob > best || (ob == best && ok < bk)) { best = ob; bk = ok; }
  }
  const float eb = emean > 0.f ? energy[(size_t)b * N + i] / emean : 1.f;
  const float m = (1.f - alpha * sxg) + alpha * sxg * eb;
  int choice = i;
  if (disc) {
    if (bk >= K) {  // no comparable value (non-finite cosines): the image's first carrier
      int first = 0;
      for (int k = 0; k < K; ++k)
        if (sImg[k] == img) { first = k; break; }
      bk = first;
      set_status(status, GMC_STATUS_NONFINITE);
    }
    choice = sS[bk];
  }
  pi[(size_t)b * N + i] = choice;
  mass[(size_t)b * N + i] = m;
  const int nw = (N + 31) >> 5;
  const int ks = slot[(size_t)b * N + choice];  // choice is in the support
  atomicOr(&mbits[((size_t)b * K + ks) * nw + (i >> 5)], 1u << (i & 31));
  if (tv.base) {
    tv.at<int32_t>(b, tv.off_pi)[i] = choice;
    tv.at<float>(b, tv.off_mass)[i] = m;
    tv.at<float>(b, tv.off_ebar)[i] = eb;
  }
}

int assign_blocks(int N) { return ceil_div(N, AT); }

cudaError_t launch_assign(const Dims& dm, const gmc_params& p, Scratch& s, const TraceView& tv,
                          cudaStream_t st, const float* cs) {
  // cosines of every token with each support entry: rows S_k of the N x N
  // matrix, or the K x N support cosines of long prefixes
  const float* src = cs ? cs : s.cos;
  const int cs_mode = cs ? 1 : 0;
  dim3 grid(s.nA, dm.B);
  const size_t gsm = 2 * sizeof(int) * (size_t)dm.K;
  const size_t psm = 4 * sizeof(int) * (size_t)dm.K;
  cudaError_t e0;
  if ((e0 = set_smem_limit((const void*)k_assign_gap, gsm)) != cudaSuccess) return e0;
  if ((e0 = set_smem_limit((const void*)k_assign_pick, psm)) != cudaSuccess) return e0;
  launch_k(k_assign_gap, grid, 32 * ASSIGN_WARPS, gsm, st, 1,
      src, cs_mode, s.support, s.slot, dm.toff, dm.B, dm.N, dm.K, dm.T, dm.H, s.omega, s.zn2,
      s.sigma, s.W2, s.ebar, s.epart, s.delta, s.dpart, s.nA, p.gate_scale, p.gate_pow, dm.I,
      s.tick2, s.gatev, s.status);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  launch_k(k_assign_pick, grid, 32 * ASSIGN_WARPS, psm, st, 1,
      src, cs_mode, s.support, s.slot, s.delta, s.gatev, s.ebar, dm.toff, dm.B, dm.N, dm.K, dm.T,
      dm.gh, dm.gw, p.gate_pow, p.ambig_margin, p.assign_spatial_w, p.tau_s,
      p.pop_strength, dm.I, s.pi, s.mass, s.mbits, tv, s.status);
  return cudaGetLastError();
}

}  // namespace gmc
