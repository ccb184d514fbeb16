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
// The cosines come from the N x N matrix at the support's columns, or (cs
// mode, long prefixes) from the N x K support cosines, column k holding the
// k-th selected token: the same values, read as contiguous rows.
#include "common.cuh"
#include "kernels.cuh"

namespace gmc {

// Pass 1: delta_i per discarded token; per-block partial sums of delta and counts.
// Also the message energy of every token (appendix Eq. (cond-grounded-energy)):
//   e_i = (sum_h omega_h g_h(i)^2 sum_t nu_t A[h,t,i]^2)^{1/2},  g_h(i)^2 = ||Z_h[i]||^2 + sigma_h^2,
// lanes over the heads, and per-block sums of e (the mean normalises ebar in pass 2).
// The last block of an image to finish (ticket) adds the block partials in a
// fixed order and stores Delta_bar, s_x and the mean energy for pass 2.
__global__ void k_assign_gap(const float* __restrict__ cos, int cs_mode,
                             const int32_t* __restrict__ support,
                             const int32_t* __restrict__ slot, const int32_t* toff, int B, int N,
                             int K, int Tmax, int H, const float* __restrict__ omega,
                             const float* __restrict__ zn2, const float* __restrict__ sigma,
                             const float* __restrict__ W2, float* energy, float* epart,
                             float* delta, double* dpart, int nA, float gate_scale,
                             float gate_pow, int I, uint32_t* tick, float* gatev,
                             uint32_t* status) {
  grid_dep_wait();
  __shared__ double sd[ASSIGN_WARPS];
  __shared__ int sc[ASSIGN_WARPS];
  __shared__ float se[ASSIGN_WARPS];
  __shared__ int last;
  extern __shared__ int sS[];  // the support of the image, staged once per block
  const int b = blockIdx.y;
  const TextGeom tg = text_geom(toff, b, B, Tmax, status);
  if (tg.T == 0) return;
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int i = blockIdx.x * ASSIGN_WARPS + w;
  for (int k = threadIdx.x; k < K; k += blockDim.x) sS[k] = support[(size_t)b * K + k];
  __syncthreads();
  float e = 0.f;
  if (i < N) {
    float e2 = 0.f;
    for (int h = lane; h < H; h += 32) {
      const size_t o = ((size_t)b * H + h) * N + i;
      const float sg = sigma[(size_t)b * H + h];
      e2 = fmaf(omega[(size_t)b * H + h] * (zn2[o] + sg * sg), W2[o], e2);
    }
    e = sqrtf(warp_sum(e2));
    if (lane == 0) energy[(size_t)b * N + i] = e;
  }
  double dv = 0.0;
  int dc = 0;
  if (i < N && slot[(size_t)b * N + i] < 0) {
    const float* row = cos + ((size_t)b * N + i) * (cs_mode ? K : N);
    const int32_t* S = sS;
    const int Ng = N / I, img = i / Ng;
    float m1 = -INFINITY, m2 = -INFINITY;
    int ncomp = 0;  // carriers of token i's image
    for (int k = lane; k < K; k += 32) {
      if (S[k] / Ng != img) continue;
      ++ncomp;
      const float v = row[cs_mode ? k : S[k]];
      if (v > m1) { m2 = m1; m1 = v; } else if (v > m2) { m2 = v; }
    }
    ncomp = warp_sum_int(ncomp);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float b1 = __shfl_xor_sync(FULL, m1, o), b2 = __shfl_xor_sync(FULL, m2, o);
      const float hi = fmaxf(m1, b1);
      m2 = fmaxf(fminf(m1, b1), fmaxf(m2, b2));
      m1 = hi;
    }
    const float d = ncomp > 1 ? m1 - m2 : 0.f;
    if (lane == 0) delta[(size_t)b * N + i] = d;
    dv = d;
    dc = 1;
  } else if (i < N && lane == 0) {
    delta[(size_t)b * N + i] = 0.f;
  }
  if (lane == 0) {
    sd[w] = dv;
    sc[w] = dc;
    se[w] = e;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    double s = 0.0;
    int c = 0;
    float es = 0.f;
    for (int q = 0; q < ASSIGN_WARPS; ++q) {
      s += sd[q];
      c += sc[q];
      es += se[q];
    }
    dpart[((size_t)b * nA + blockIdx.x) * 2 + 0] = s;
    dpart[((size_t)b * nA + blockIdx.x) * 2 + 1] = (double)c;
    epart[(size_t)b * nA + blockIdx.x] = es;
    __threadfence();
    last = atomicAdd(&tick[b], 1u) == (unsigned)(nA - 1);
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
__global__ void k_assign_pick(const float* __restrict__ cos, int cs_mode,
                              const int32_t* __restrict__ support,
                              const int32_t* __restrict__ slot, const float* __restrict__ delta,
                              const float* __restrict__ gatev, const float* __restrict__ energy,
                              const int32_t* toff, int B, int N, int K, int Tmax, int gh, int gw,
                              float gate_pow, float ambig_margin, float lambda_p, float tau_s,
                              float alpha, int I,
                              int32_t* pi, float* mass, uint32_t* mbits, TraceView tv,
                              uint32_t* status) {
  grid_dep_wait();
  extern __shared__ int sS[];  // the support of the image, staged once per block
  const int b = blockIdx.y;
  const TextGeom tg = text_geom(toff, b, B, Tmax, status);
  if (tg.T == 0) return;
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  for (int k = threadIdx.x; k < K; k += blockDim.x) sS[k] = support[(size_t)b * K + k];
  const float dbar = gatev[(size_t)b * 4 + 0], sx = gatev[(size_t)b * 4 + 1];
  const float emean = gatev[(size_t)b * 4 + 2];
  __syncthreads();
  if (blockIdx.x == 0 && threadIdx.x == 0 && tv.base) {
    tv.header(b)->s_x = sx;
    tv.header(b)->delta_bar = dbar;
  }
  const int i = blockIdx.x * ASSIGN_WARPS + w;
  if (i >= N) return;
  const float eb = emean > 0.f ? energy[(size_t)b * N + i] / emean : 1.f;
  const float m = (1.f - alpha * sx) + alpha * sx * eb;
  int choice = i;
  if (slot[(size_t)b * N + i] < 0) {
    const float gi = expf(-powf(delta[(size_t)b * N + i] / ambig_margin, gate_pow));
    const float coef = lambda_p * sx * gi;
    const int Ng = N / I, img = i / Ng, il = i - img * Ng;  // coordinates in its own grid
    const float piy = ((il / gw) + 0.5f) / gh, pix = ((il % gw) + 0.5f) / gw;
    const float* row = cos + ((size_t)b * N + i) * (cs_mode ? K : N);
    const int32_t* S = sS;
    float best = -INFINITY;
    int bk = 0x7fffffff;
    for (int k = lane; k < K; k += 32) {
      const int j = S[k];
      if (j / Ng != img) continue;  // a carrier of another image
      float v = row[cs_mode ? k : j];
      if (coef > 0.f) {
        const int jl = j - img * Ng;
        const float dy = ((jl / gw) + 0.5f) / gh - piy, dx = ((jl % gw) + 0.5f) / gw - pix;
        v += coef * expf(-(dy * dy + dx * dx) / tau_s);
      }
      if (v > best) { best = v; bk = k; }  // k ascending within a lane: first max kept
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float ob = __shfl_xor_sync(FULL, best, o);
      const int ok = __shfl_xor_sync(FULL, bk, o);
      if (ob > best || (ob == best && ok < bk)) { best = ob; bk = ok; }
    }
    if (bk >= K) {  // no comparable value (non-finite cosines): the image's first carrier
      int first = K;
      for (int k = lane; k < K; k += 32)
        if (S[k] / Ng == img) { first = k; break; }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) first = min(first, __shfl_xor_sync(FULL, first, o));
      bk = first < K ? first : 0;
      if (lane == 0) set_status(status, GMC_STATUS_NONFINITE);
    }
    choice = S[bk];
  }
  if (lane == 0) {
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
}

cudaError_t launch_assign(const Dims& dm, const gmc_params& p, Scratch& s, const TraceView& tv,
                          cudaStream_t st, const float* cs) {
  const float* src = cs ? cs : s.cos;
  const int cs_mode = cs ? 1 : 0;
  dim3 grid(s.nA, dm.B);
  const size_t smem = sizeof(int) * (size_t)dm.K;
  cudaError_t e0;
  if ((e0 = set_smem_limit((const void*)k_assign_gap, smem)) != cudaSuccess) return e0;
  if ((e0 = set_smem_limit((const void*)k_assign_pick, smem)) != cudaSuccess) return e0;
  launch_k(k_assign_gap, grid, 32 * ASSIGN_WARPS, smem, st, 1,
      src, cs_mode, s.support, s.slot, dm.toff, dm.B, dm.N, dm.K, dm.T, dm.H, s.omega, s.zn2, s.sigma,
      s.W2, s.ebar, s.epart, s.delta, s.dpart, s.nA, p.gate_scale, p.gate_pow, dm.I, s.tick2,
      s.gatev, s.status);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  launch_k(k_assign_pick, grid, 32 * ASSIGN_WARPS, smem, st, 1,
      src, cs_mode, s.support, s.slot, s.delta, s.gatev, s.ebar, dm.toff, dm.B, dm.N, dm.K, dm.T,
      dm.gh, dm.gw, p.gate_pow, p.ambig_margin, p.assign_spatial_w, p.tau_s,
      p.pop_strength, dm.I, s.pi, s.mass, s.mbits, tv, s.status);
  return cudaGetLastError();
}

}  // namespace gmc
