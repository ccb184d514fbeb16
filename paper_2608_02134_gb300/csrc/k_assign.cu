// Population assignment (appendix Eq. (cond-assignment), (cond-population-gate)).
//
// For a discarded token i, delta_i is the gap between its largest and
// second-largest cosine to the support (0 when |S| = 1); Delta_bar is the mean
// gap over the discarded tokens (0 when none is discarded);
//   s_x = 1 - exp(-(Delta_bar / gate_scale)^gate_pow)
//   g_i = exp(-(delta_i / ambig_margin)^gate_pow)
//   pi(i) = argmax_{j in S} cos_ij + lambda_p s_x g_i exp(-||p_i - p_j||^2 / tau_s)
// (ties to the lowest j); selected tokens represent themselves.  The
// population weights are m_i = (1 - alpha s_x) + alpha s_x ebar_i.  Token i
// also sets bit i of its carrier's membership bitmap (atomicOr: the bitmap
// does not depend on the order of the writes), which the transport reads
// instead of scanning the whole assignment.
#include "common.cuh"
#include "kernels.cuh"

namespace gmc {

// Pass 1: delta_i per discarded token; per-block partial sums of delta and counts.
// Also the message energy of every token (appendix Eq. (cond-grounded-energy)):
//   e_i = (sum_h omega_h g_h(i)^2 sum_t nu_t A[h,t,i]^2)^{1/2},  g_h(i)^2 = ||Z_h[i]||^2 + sigma_h^2,
// lanes over the heads, and per-block sums of e (the mean normalises ebar in pass 2).
__global__ void k_assign_gap(const float* __restrict__ cos, const int32_t* __restrict__ support,
                             const int32_t* __restrict__ slot, const int32_t* toff, int B, int N,
                             int K, int Tmax, int H, const float* __restrict__ omega,
                             const float* __restrict__ zn2, const float* __restrict__ sigma,
                             const float* __restrict__ W2, float* energy, float* epart,
                             float* delta, double* dpart, int nA, uint32_t* status) {
  __shared__ double sd[ASSIGN_WARPS];
  __shared__ int sc[ASSIGN_WARPS];
  __shared__ float se[ASSIGN_WARPS];
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
    const float* row = cos + ((size_t)b * N + i) * N;
    const int32_t* S = sS;
    float m1 = -INFINITY, m2 = -INFINITY;
    for (int k = lane; k < K; k += 32) {
      const float v = row[S[k]];
      if (v > m1) { m2 = m1; m1 = v; } else if (v > m2) { m2 = v; }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float b1 = __shfl_xor_sync(FULL, m1, o), b2 = __shfl_xor_sync(FULL, m2, o);
      const float hi = fmaxf(m1, b1);
      m2 = fmaxf(fminf(m1, b1), fmaxf(m2, b2));
      m1 = hi;
    }
    const float d = K > 1 ? m1 - m2 : 0.f;
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
  }
}

// Pass 2: s_x, the gated spatial assignment, and the population weights.
__global__ void k_assign_pick(const float* __restrict__ cos, const int32_t* __restrict__ support,
                              const int32_t* __restrict__ slot, const float* __restrict__ delta,
                              const double* __restrict__ dpart, int nA,
                              const float* __restrict__ energy, const float* __restrict__ epart,
                              int nE, const int32_t* toff, int B, int N,
                              int K, int Tmax, int gh, int gw, float gate_scale, float gate_pow,
                              float ambig_margin, float lambda_p, float tau_s, float alpha,
                              int32_t* pi, float* mass, uint32_t* mbits, TraceView tv,
                              uint32_t* status) {
  __shared__ float gate[3];      // dbar, s_x, mean energy
  extern __shared__ int sS[];  // the support of the image, staged once per block
  const int b = blockIdx.y;
  const TextGeom tg = text_geom(toff, b, B, Tmax, status);
  if (tg.T == 0) return;
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  for (int k = threadIdx.x; k < K; k += blockDim.x) sS[k] = support[(size_t)b * K + k];
  if (w == 0) {  // the partials in a fixed order (every block the same)
    double s = 0.0, c = 0.0, et = 0.0;
    for (int q = lane; q < nA; q += 32) {
      s += dpart[((size_t)b * nA + q) * 2 + 0];
      c += dpart[((size_t)b * nA + q) * 2 + 1];
    }
    for (int q = lane; q < nE; q += 32) et += epart[(size_t)b * nE + q];  // message energies
    s = warp_sum(s);
    c = warp_sum(c);
    et = warp_sum(et);
    if (lane == 0) {
      const float db = c > 0.0 ? (float)(s / c) : 0.f;
      gate[0] = db;
      gate[1] = 1.f - expf(-powf(db / gate_scale, gate_pow));
      gate[2] = (float)(et / N);
    }
  }
  __syncthreads();
  const float dbar = gate[0], sx = gate[1];
  const float emean = gate[2];
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
    const float piy = ((i / gw) + 0.5f) / gh, pix = ((i % gw) + 0.5f) / gw;
    const float* row = cos + ((size_t)b * N + i) * N;
    const int32_t* S = sS;
    float best = -INFINITY;
    int bk = 0x7fffffff;
    for (int k = lane; k < K; k += 32) {
      const int j = S[k];
      float v = row[j];
      if (coef > 0.f) {
        const float dy = ((j / gw) + 0.5f) / gh - piy, dx = ((j % gw) + 0.5f) / gw - pix;
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
                          cudaStream_t st) {
  dim3 grid(s.nA, dm.B);
  const size_t smem = sizeof(int) * (size_t)dm.K;
  cudaError_t e0;
  if ((e0 = set_smem_limit((const void*)k_assign_gap, smem)) != cudaSuccess) return e0;
  if ((e0 = set_smem_limit((const void*)k_assign_pick, smem)) != cudaSuccess) return e0;
  k_assign_gap<<<grid, 32 * ASSIGN_WARPS, smem, st>>>(
      s.cos, s.support, s.slot, dm.toff, dm.B, dm.N, dm.K, dm.T, dm.H, s.omega, s.zn2, s.sigma,
      s.W2, s.ebar, s.epart, s.delta, s.dpart, s.nA, s.status);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  k_assign_pick<<<grid, 32 * ASSIGN_WARPS, smem, st>>>(
      s.cos, s.support, s.slot, s.delta, s.dpart, s.nA, s.ebar, s.epart, s.nE, dm.toff, dm.B,
      dm.N, dm.K, dm.T,
      dm.gh, dm.gw, p.gate_scale, p.gate_pow, p.ambig_margin, p.assign_spatial_w, p.tau_s,
      p.pop_strength, s.pi, s.mass, s.mbits, tv, s.status);
  return cudaGetLastError();
}

}  // namespace gmc
