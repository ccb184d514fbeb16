// Native boundary attention slice (appendix Eq. (cond-native-message)) and the
// grounded-client row sums of Eq. (2).
//
// For image b, head h and text query t the scores are
//   s_k = q_{t,h} . k_{k,kv(h)} / sqrt(d)  over the N visual keys and text keys 0..t,
// A[h,t,i] = softmax(s)_i for the visual columns i < N (no renormalisation over
// the visual keys), and rs[h,t] = sum_i A[h,t,i] g_h(i) with
// g_h(i) = ||[Z_h[i]; sigma_h]|| = sqrt(||Z_h[i]||^2 + sigma_h^2).
#include "common.cuh"
#include "kernels.cuh"

namespace gmc {

// One block per (query t, head h, image b); the scores of the row stay in
// shared memory.  The query is staged once; each thread owns keys k = tid + j*blockDim.
template <typename Tin>
__global__ void k_message(const Tin* __restrict__ keys, const Tin* __restrict__ queries,
                          const float* __restrict__ zn2, const float* __restrict__ sigma,
                          const int32_t* toff, int B, int N, int K, int Tmax, int H, int Hkv,
                          int d, float* A, float* rs, uint32_t* status) {
  grid_dep_wait();
  extern __shared__ float sm_msg[];  // [d] query, then [N + Tmax] scores
  __shared__ float red[32];
  const int t = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const TextGeom tg = text_geom(toff, b, B, Tmax, status);
  if (tg.T == 0 || t >= tg.T) return;
  const SeqIdx sq(b, N, K, tg.off, tg.T);
  const int HD = Hkv * d, g = h / (H / Hkv);
  float* q = sm_msg;
  float* sc = sm_msg + d;
  const Tin* qrow = queries + ((size_t)tg.off + t) * H * d + (size_t)h * d;
  for (int k = threadIdx.x; k < d; k += blockDim.x) q[k] = to_f32(qrow[k]);
  __syncthreads();
  const float scale = rsqrtf((float)d);
  const int nkeys = N + t + 1;  // causal: every visual key and text keys 0..t
  float mx = -INFINITY;
  for (int k = threadIdx.x; k < nkeys; k += blockDim.x) {
    const Tin* kr = keys + sq.key_row(k, HD) + (size_t)g * d;
    float acc = 0.f;
    for (int c = 0; c < d; ++c) acc = fmaf(q[c], to_f32(kr[c]), acc);
    const float s = acc * scale;
    sc[k] = s;
    mx = fmaxf(mx, s);
  }
  mx = block_reduce(mx, red, OpMax(), -INFINITY);
  float sum = 0.f;
  for (int k = threadIdx.x; k < nkeys; k += blockDim.x) sum += expf(sc[k] - mx);
  sum = block_reduce(sum, red, OpAdd(), 0.f);
  const float inv = 1.f / sum;
  const float sg = sigma[(size_t)b * H + h];
  const float sg2 = sg * sg;
  const float* zr = zn2 + ((size_t)b * H + h) * N;
  float* arow = A + (((size_t)b * H + h) * Tmax + t) * N;
  float usum = 0.f;
  for (int i = threadIdx.x; i < N; i += blockDim.x) {
    const float a = expf(sc[i] - mx) * inv;
    arow[i] = a;
    usum = fmaf(a, sqrtf(zr[i] + sg2), usum);
  }
  usum = block_reduce(usum, red, OpAdd(), 0.f);
  if (threadIdx.x == 0) rs[((size_t)b * H + h) * Tmax + t] = usum;
}

cudaError_t launch_message(const Dims& dm, const void* keys, const void* queries, Scratch& s,
                           cudaStream_t st, int* launches) {
  // bf16 with d in {64, 128} and a full 128-key tile: tcgen05 (k_message_tc.cu);
  // fp32 inputs and other shapes: the CUDA-core kernel above.
  if (message_tc_supported(dm)) return launch_message_tc(dm, keys, queries, s, st, launches);
  if (launches) *launches = 1;
  dim3 grid(dm.T, dm.H, dm.B);
  size_t smem = sizeof(float) * (dm.d + dm.N + dm.T);
  cudaError_t e;
  if (dm.dtype == GMC_BF16) {
    if ((e = set_smem_limit((const void*)k_message<__nv_bfloat16>, smem)) != cudaSuccess) return e;
    launch_k(k_message<__nv_bfloat16>, grid, 256, smem, st, 1,
        (const __nv_bfloat16*)keys, (const __nv_bfloat16*)queries, s.zn2, s.sigma, dm.toff, dm.B,
        dm.N, dm.K, dm.T, dm.H, dm.Hkv, dm.d, s.A, s.rs, s.status);
  } else {
    if ((e = set_smem_limit((const void*)k_message<float>, smem)) != cudaSuccess) return e;
    launch_k(k_message<float>, grid, 256, smem, st, 1, (const float*)keys, (const float*)queries, s.zn2,
                                              s.sigma, dm.toff, dm.B, dm.N, dm.K, dm.T, dm.H,
                                              dm.Hkv, dm.d, s.A, s.rs, s.status);
  }
  return cudaGetLastError();
}

}  // namespace gmc
