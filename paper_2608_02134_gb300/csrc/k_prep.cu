// Per-token preparation: boundary-state norms, probe values and the mass
// coordinate, and the K = N identity copy.
#include "common.cuh"
#include "kernels.cuh"

namespace gmc {

// ||h_i|| for every visual row: x_i = h_i / max(||h_i||, eps) (appendix
// "Population assignment and transport") and rms(h_i) = ||h_i|| / sqrt(D) for the
// RMS restoration R_j of Eq. (5).  One warp per row, 16-byte loads; each lane
// sums D / 32 squares in fp32 (relative error ~1e-6 at D = 4096), the warp tree
// adds the lane sums.
template <typename Tin>
__global__ void k_rownorm(const Tin* __restrict__ hidden, const int32_t* toff, int B, int N,
                          int K, int Tmax, int D, float norm_eps, float* rn, float* rmsh,
                          uint32_t* status) {
  const int b = blockIdx.y;
  const TextGeom tg = text_geom(toff, b, B, Tmax, status);
  if (tg.T == 0) return;
  const int lane = threadIdx.x & 31;
  const int i = blockIdx.x * ROWS_PER_BLOCK + (threadIdx.x >> 5);
  if (i >= N) return;
  const SeqIdx sq(b, N, K, tg.off, tg.T);
  const Tin* row = hidden + sq.hidden_row(i, D);
  constexpr int V = 16 / sizeof(Tin);
  float acc = 0.f;
  for (int k = lane * V; k < D; k += 32 * V) {
    uint4 raw = *reinterpret_cast<const uint4*>(row + k);
    const Tin* e = reinterpret_cast<const Tin*>(&raw);
#pragma unroll
    for (int v = 0; v < V; ++v) {
      const float x = to_f32(e[v]);
      acc = fmaf(x, x, acc);
    }
  }
  acc = warp_sum(acc);
  if (lane == 0) {
    const float n = sqrtf(acc);
    if (rn) rn[(size_t)b * N + i] = 1.f / fmaxf(n, norm_eps);
    rmsh[(size_t)b * N + i] = sqrtf(acc / (float)D);
  }
}

// Z_h[i] = V_{kv(h)}[i] W_h (Eq. (1): (V_h O_h) P with W_h = O_h P), ||Z_h[i]||^2,
// and per-block partial sums of ||Z_h||_F^2.  A block covers ROWS_PER_BLOCK
// tokens and every head; warp per (token, head) with lanes over the head dim.
template <typename Tin>
__global__ void k_probe(const Tin* __restrict__ keys, const float* __restrict__ W,
                        const int32_t* toff, int B, int N, int K, int Tmax, int H, int Hkv, int d,
                        float* Z, float* zn2, float* sigpart, int nP, uint32_t* status) {
  extern __shared__ float sm_probe[];  // [ROWS_PER_BLOCK][H]
  const int b = blockIdx.y;
  const TextGeom tg = text_geom(toff, b, B, Tmax, status);
  if (tg.T == 0) return;
  const SeqIdx sq(b, N, K, tg.off, tg.T);
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = blockDim.x >> 5;
  const int i0 = blockIdx.x * ROWS_PER_BLOCK;
  const int grp = H / Hkv, HD = Hkv * d;
  for (int p = wid; p < ROWS_PER_BLOCK * H; p += nw) {
    const int ii = p / H, h = p % H, i = i0 + ii;
    float z0 = 0.f, z1 = 0.f, z2 = 0.f, z3 = 0.f;
    if (i < N) {
      const Tin* v = keys + sq.value_row(i, HD) + (size_t)(h / grp) * d;
      const float4* w4 = reinterpret_cast<const float4*>(W + (size_t)h * d * 4);
      for (int k = lane; k < d; k += 32) {
        float x = to_f32(v[k]);
        float4 w = w4[k];
        z0 = fmaf(x, w.x, z0);
        z1 = fmaf(x, w.y, z1);
        z2 = fmaf(x, w.z, z2);
        z3 = fmaf(x, w.w, z3);
      }
      z0 = warp_sum(z0); z1 = warp_sum(z1); z2 = warp_sum(z2); z3 = warp_sum(z3);
      if (lane == 0) {
        const size_t o = ((size_t)b * H + h) * N + i;
        reinterpret_cast<float4*>(Z)[o] = make_float4(z0, z1, z2, z3);
        zn2[o] = z0 * z0 + z1 * z1 + z2 * z2 + z3 * z3;
      }
    }
    if (lane == 0) sm_probe[ii * H + h] = z0 * z0 + z1 * z1 + z2 * z2 + z3 * z3;
  }
  __syncthreads();
  for (int h = threadIdx.x; h < H; h += blockDim.x) {
    float s = 0.f;
    for (int ii = 0; ii < ROWS_PER_BLOCK; ++ii) s += sm_probe[ii * H + h];  // fixed order
    sigpart[((size_t)b * nP + blockIdx.x) * H + h] = s;
  }
}

// sigma_h = sqrt(lambda_mass) * max(||Z_h||_F / sqrt(N r), eps_mass), Eq. (1).
// One warp per (image, head); partials summed in a fixed order.
__global__ void k_sigma(const float* sigpart, int nP, int B, int N, int H, float lambda_mass,
                        float eps_mass, float* sigma) {
  const int w = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (w >= B * H) return;
  const int b = w / H, h = w % H;
  double s = 0.0;
  for (int p = lane; p < nP; p += 32) s += sigpart[((size_t)b * nP + p) * H + h];
  s = warp_sum(s);
  if (lane == 0) {
    double fro = sqrt(s);
    double v = sqrt((double)lambda_mass) * fmax(fro / sqrt((double)N * 4.0), (double)eps_mass);
    sigma[(size_t)b * H + h] = (float)v;
  }
}

// K == N: the unmodified execution.  One block per output row copies the
// hidden row, both K/V rows and the position ids; out_idx = 0..N-1.
template <typename Tin>
__global__ void k_identity(const Tin* __restrict__ hidden, const Tin* __restrict__ keys,
                           const int32_t* __restrict__ pos, const int32_t* toff, int B, int N,
                           int Tmax, int D, int HD, int32_t* out_idx, Tin* out_hidden,
                           Tin* out_kv, int32_t* out_pos, uint32_t* status) {
  const int b = blockIdx.y, r = blockIdx.x;
  const TextGeom tg = text_geom(toff, b, B, Tmax, status);
  if (tg.T == 0 || r >= N + tg.T) return;
  const SeqIdx sq(b, N, N, tg.off, tg.T);
  const uint4* src = reinterpret_cast<const uint4*>(hidden + sq.hidden_row(r, D));
  uint4* dst = reinterpret_cast<uint4*>(out_hidden + sq.out_hidden_row(r, D));
  const int nv = D * (int)sizeof(Tin) / 16;
  for (int k = threadIdx.x; k < nv; k += blockDim.x) dst[k] = src[k];
  const int nkv = HD * (int)sizeof(Tin) / 16;
  for (int w = 0; w < 2; ++w) {
    const uint4* ks = reinterpret_cast<const uint4*>(
        keys + (w == 0 ? sq.key_row(r, HD) : sq.value_row(r, HD)));
    uint4* kd = reinterpret_cast<uint4*>(out_kv + sq.out_kv_row(w, r, HD));
    for (int k = threadIdx.x; k < nkv; k += blockDim.x) kd[k] = ks[k];
  }
  if (threadIdx.x < 3) out_pos[sq.out_pos(threadIdx.x, r)] = pos[sq.pos(threadIdx.x, r)];
  if (threadIdx.x == 0 && r < N) out_idx[(size_t)b * N + r] = r;
}

cudaError_t launch_rownorm(const Dims& dm, const void* hidden, float norm_eps, Scratch& s,
                           cudaStream_t st) {
  dim3 grid(ceil_div(dm.N, ROWS_PER_BLOCK), dm.B);
  if (dm.dtype == GMC_BF16)
    k_rownorm<__nv_bfloat16><<<grid, 32 * ROWS_PER_BLOCK, 0, st>>>(
        (const __nv_bfloat16*)hidden, dm.toff, dm.B, dm.N, dm.K, dm.T, dm.D, norm_eps, s.rn,
        s.rmsh, s.status);
  else
    k_rownorm<float><<<grid, 32 * ROWS_PER_BLOCK, 0, st>>>((const float*)hidden, dm.toff, dm.B,
                                                           dm.N, dm.K, dm.T, dm.D, norm_eps, s.rn,
                                                           s.rmsh, s.status);
  return cudaGetLastError();
}

cudaError_t launch_rms_rows(const Dims& dm, const void* hidden, float* rmsh, uint32_t* status,
                            cudaStream_t st) {
  dim3 grid(ceil_div(dm.N, ROWS_PER_BLOCK), dm.B);
  if (dm.dtype == GMC_BF16)
    k_rownorm<__nv_bfloat16><<<grid, 32 * ROWS_PER_BLOCK, 0, st>>>(
        (const __nv_bfloat16*)hidden, dm.toff, dm.B, dm.N, dm.K, dm.T, dm.D, 1e-12f, nullptr,
        rmsh, status);
  else
    k_rownorm<float><<<grid, 32 * ROWS_PER_BLOCK, 0, st>>>((const float*)hidden, dm.toff, dm.B,
                                                           dm.N, dm.K, dm.T, dm.D, 1e-12f,
                                                           nullptr, rmsh, status);
  return cudaGetLastError();
}

cudaError_t launch_probe(const Dims& dm, const void* keys, const float* W, const gmc_params& p,
                         Scratch& s, cudaStream_t st) {
  dim3 grid(s.nP, dm.B);
  size_t smem = sizeof(float) * ROWS_PER_BLOCK * dm.H;
  if (dm.dtype == GMC_BF16)
    k_probe<__nv_bfloat16><<<grid, 256, smem, st>>>((const __nv_bfloat16*)keys, W, dm.toff, dm.B,
                                                    dm.N, dm.K, dm.T, dm.H, dm.Hkv, dm.d, s.Z,
                                                    s.zn2, s.sigpart, s.nP, s.status);
  else
    k_probe<float><<<grid, 256, smem, st>>>((const float*)keys, W, dm.toff, dm.B, dm.N, dm.K,
                                            dm.T, dm.H, dm.Hkv, dm.d, s.Z, s.zn2, s.sigpart,
                                            s.nP, s.status);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const int warps = dm.B * dm.H;
  k_sigma<<<ceil_div(warps * 32, 256), 256, 0, st>>>(s.sigpart, s.nP, dm.B, dm.N, dm.H,
                                                     p.lambda_mass, p.eps_mass, s.sigma);
  return cudaGetLastError();
}

cudaError_t launch_identity(const Dims& dm, const void* hidden, const void* keys,
                            const int32_t* pos, int32_t* out_idx, void* out_hidden, void* out_kv,
                            int32_t* out_pos, uint32_t* status, cudaStream_t st) {
  dim3 grid(dm.N + dm.T, dm.B);
  const int HD = dm.Hkv * dm.d;
  if (dm.dtype == GMC_BF16)
    k_identity<__nv_bfloat16><<<grid, 128, 0, st>>>(
        (const __nv_bfloat16*)hidden, (const __nv_bfloat16*)keys, pos, dm.toff, dm.B, dm.N, dm.T,
        dm.D, HD, out_idx, (__nv_bfloat16*)out_hidden, (__nv_bfloat16*)out_kv, out_pos, status);
  else
    k_identity<float><<<grid, 128, 0, st>>>((const float*)hidden, (const float*)keys, pos,
                                            dm.toff, dm.B, dm.N, dm.T, dm.D, HD, out_idx,
                                            (float*)out_hidden, (float*)out_kv, out_pos, status);
  return cudaGetLastError();
}

}  // namespace gmc
