// Cosine matrix of the boundary states, cos_ij = (h_i . h_j) / (n_i n_j) with
// n_i = max(||h_i||, eps): the appearance clients of appendix Eq.
// (cond-aux-clients) and the assignment cosines of Eq. (cond-assignment).
//
// This is the fp32-input path: a CUDA-core tiled contraction in fp32 (exact
// fp32 inputs need exact fp32 products; the tensor cores would round them).
// The bf16 path runs on tcgen05 (k_gram_tc.cu).
#include "common.cuh"
#include "kernels.cuh"

namespace gmc {

constexpr int GT = 64;   // output tile
constexpr int GK = 16;   // k step

template <typename Tin>
__global__ void __launch_bounds__(256) k_gram_simt(const Tin* __restrict__ hidden,
                                                   const float* __restrict__ rn,
                                                   const int32_t* toff, int B, int N, int K,
                                                   int Tmax, int D, float* cos, uint32_t* status) {
  grid_dep_wait();
  __shared__ float As[GK][GT + 4];
  __shared__ float Bs[GK][GT + 4];
  const int b = blockIdx.z;
  const TextGeom tg = text_geom(toff, b, B, Tmax, status);
  if (tg.T == 0) return;
  const SeqIdx sq(b, N, K, tg.off, tg.T);
  const int row0 = blockIdx.y * GT, col0 = blockIdx.x * GT;
  const int tx = threadIdx.x % 16, ty = threadIdx.x / 16;
  float acc[4][4] = {};
  for (int k0 = 0; k0 < D; k0 += GK) {
    for (int e = threadIdx.x; e < GT * GK; e += 256) {
      const int r = e / GK, kk = e % GK;
      const int k = k0 + kk;
      const int ia = row0 + r, ib = col0 + r;
      As[kk][r] = (ia < N && k < D) ? to_f32(hidden[sq.hidden_row(ia, D) + k]) : 0.f;
      Bs[kk][r] = (ib < N && k < D) ? to_f32(hidden[sq.hidden_row(ib, D) + k]) : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < GK; ++kk) {
      float a[4], bb[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        a[u] = As[kk][ty * 4 + u];
        bb[u] = Bs[kk][tx * 4 + u];
      }
#pragma unroll
      for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int v = 0; v < 4; ++v) acc[u][v] = fmaf(a[u], bb[v], acc[u][v]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    const int i = row0 + ty * 4 + u;
    if (i >= N) continue;
    const float ri = rn[(size_t)b * N + i];
#pragma unroll
    for (int v = 0; v < 4; ++v) {
      const int j = col0 + tx * 4 + v;
      if (j < N) cos[((size_t)b * N + i) * N + j] = acc[u][v] * ri * rn[(size_t)b * N + j];
    }
  }
}

cudaError_t launch_gram_simt(const Dims& dm, const void* hidden, Scratch& s, cudaStream_t st) {
  dim3 grid(ceil_div(dm.N, GT), ceil_div(dm.N, GT), dm.B);
  if (dm.dtype == GMC_BF16)
    launch_k(k_gram_simt<__nv_bfloat16>, grid, 256, 0, st, 1, (const __nv_bfloat16*)hidden, s.rn, dm.toff,
                                                     dm.B, dm.N, dm.K, dm.T, dm.D, s.cos,
                                                     s.status);
  else
    launch_k(k_gram_simt<float>, grid, 256, 0, st, 1, (const float*)hidden, s.rn, dm.toff, dm.B, dm.N,
                                             dm.K, dm.T, dm.D, s.cos, s.status);
  return cudaGetLastError();
}

cudaError_t launch_gram(const Dims& dm, const void* hidden, Scratch& s, cudaStream_t st) {
  // bf16 states with at least one full 128-row tile: tcgen05.  Problems whose
  // 128 x 256 tiles on or above the diagonal fill the GPU at least once (the
  // document page, serving batches) run the general kernel in symmetric mode
  // (k_gemm_tc.cu); a single smaller image runs the split-contraction Gram of
  // k_gram_tc.cu, which keeps more SMs busy at that size.  fp32 states (exact
  // fp32 products) and tiny grids: the CUDA-core kernel above.
  if (!gram_tc_supported(dm)) return launch_gram_simt(dm, hidden, s, st);
  static int sms = 0;
  if (sms == 0) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
      cudaGetLastError();
      sms = 152;
    }
  }
  if (dm.N >= 256 && gemm_sym_ctas(dm.N, dm.B) >= sms) {
    GemmArgs g{};
    g.B = dm.B; g.M = dm.N; g.Nn = dm.N; g.Kd = dm.D;
    g.a_img = dm.N; g.b_img = dm.N; g.a_text = 1; g.b_text = 1;
    g.toff = dm.toff; g.Tmax = dm.T;
    g.rscale = s.rn; g.cscale = s.rn;
    g.C = s.cos; g.c_img = (long long)dm.N * dm.N; g.ldc = dm.N;
    g.status = s.status;
    g.sym = 1;
    const long long rows = (long long)dm.B * (dm.N + dm.T);
    return launch_gemm_tc(g, hidden, rows, dm.D, hidden, rows, dm.D, st);
  }
  return launch_gram_tc(dm, hidden, s, st);
}

}  // namespace gmc
