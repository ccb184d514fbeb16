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
                          long long* u0, uint32_t* status) {
  grid_dep_wait();
  const int b = blockIdx.y;
  // the client build's column sums start at zero (this kernel opens the
  // branch of the path that builds the appearance and spatial rows)
  if (u0 && threadIdx.x < ROWS_PER_BLOCK && blockIdx.x * ROWS_PER_BLOCK + (int)threadIdx.x < N)
    u0[(size_t)b * N + blockIdx.x * ROWS_PER_BLOCK + threadIdx.x] = 0;
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
// per-block partial sums of ||Z_h||_F^2, and
// sigma_h = sqrt(lambda_mass) * max(||Z_h||_F / sqrt(N r), eps_mass) (Eq. (1)).
// A block covers PR_TOK tokens of one KV group: the values and the group's
// W_h are staged in shared memory, one thread per (token, head) computes the
// four probe coordinates.  The last block of an image to finish (a ticket per
// image, zeroed with the status word) sums the partials in a fixed order.
// With Qp (the tensor-core message slice follows), the blocks of KV group g
// also write the group's packed text queries first: Qp [B][Hkv][RQ][d], row
// j*T_b + t holding query head g*grp + j at text position t, rows >= grp*T_b
// zero (block pb: rows pb, pb + nP, ...).
constexpr int PR_TOK = PROBE_TOK;

template <typename Tin>
__global__ void __launch_bounds__(256) k_probe(
    const Tin* __restrict__ keys, const float* __restrict__ W, const int32_t* toff, int B, int N,
    int K, int Tmax, int H, int Hkv, int d, float lambda_mass, float eps_mass, float* Z,
    float* zn2, float* sigpart, int nP, float* sigma, uint32_t* tick,
    const __nv_bfloat16* __restrict__ queries, int RQ, __nv_bfloat16* Qp, uint32_t* status) {
  grid_dep_wait();
  extern __shared__ float4 sm_probe4[];
  __shared__ int last;
  const int b = blockIdx.z, g = blockIdx.y, pb = blockIdx.x;
  const TextGeom tg = text_geom(toff, b, B, Tmax, status);
  if (Qp) {
    const int grp = H / Hkv, nv = d / 8;  // 16-byte pieces per row
    for (int idx = threadIdx.x;; idx += blockDim.x) {
      const int row = pb + (idx / nv) * nP, q = idx % nv;
      if (row >= RQ) break;  // row grows with idx
      uint4 v = make_uint4(0, 0, 0, 0);
      if (tg.T > 0 && row < grp * tg.T) {
        const int j = row / tg.T, t = row % tg.T;
        v = reinterpret_cast<const uint4*>(queries + ((size_t)tg.off + t) * H * d +
                                           (size_t)(g * grp + j) * d)[q];
      }
      reinterpret_cast<uint4*>(Qp + (((size_t)b * Hkv + g) * RQ + row) * d)[q] = v;
    }
  }
  if (tg.T == 0) return;  // uniform over the image
  const SeqIdx sq(b, N, K, tg.off, tg.T);
  const int grp = H / Hkv, HD = Hkv * d, i0 = pb * PR_TOK;
  float4* Ws = sm_probe4;                                    // [grp][d + 1]
  float* Vs = reinterpret_cast<float*>(Ws + grp * (d + 1));  // [PR_TOK][d + 1] (padded rows)
  float* zs = Vs + PR_TOK * (d + 1);                         // [PR_TOK][grp]
  const float4* W4 = reinterpret_cast<const float4*>(W) + (size_t)g * grp * d;
  // W_h rows by cp.async, the values through registers four loads at a time:
  // every copy of the block is in flight before the first one lands
  for (int idx = threadIdx.x; idx < grp * d; idx += blockDim.x)
    cp_async16(&Ws[(idx / d) * (d + 1) + idx % d], &W4[idx]);
  cp_async_commit();
  constexpr int VE = 16 / sizeof(Tin);  // elements per 16-byte load
  const int nld = PR_TOK * d / VE;
  for (int idx0 = 0; idx0 < nld; idx0 += 4 * (int)blockDim.x) {  // uniform over the block
    uint4 raw[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int idx = idx0 + u * (int)blockDim.x + (int)threadIdx.x;
      const int ii = idx / (d / VE), k = (idx % (d / VE)) * VE, i = i0 + ii;
      raw[u] = make_uint4(0, 0, 0, 0);
      if (idx < nld && i < N)
        raw[u] = *reinterpret_cast<const uint4*>(keys + sq.value_row(i, HD) + (size_t)g * d + k);
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int idx = idx0 + u * (int)blockDim.x + (int)threadIdx.x;
      if (idx >= nld) continue;
      const int ii = idx / (d / VE), k = (idx % (d / VE)) * VE;
      const Tin* e = reinterpret_cast<const Tin*>(&raw[u]);
#pragma unroll
      for (int q = 0; q < VE; ++q) Vs[ii * (d + 1) + k + q] = to_f32(e[q]);
    }
  }
  cp_async_wait<0>();
  __syncthreads();
  for (int task = threadIdx.x; task < PR_TOK * grp; task += blockDim.x) {
    const int ii = task / grp, jh = task % grp, i = i0 + ii;
    const float* v = Vs + ii * (d + 1);
    const float4* w = Ws + jh * (d + 1);
    // four coordinates loaded ahead of their FMAs; even and odd k accumulate
    // apart and are added once at the end (d is a multiple of 4)
    float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f, b0 = 0.f, b1 = 0.f, b2 = 0.f, b3 = 0.f;
#pragma unroll 2
    for (int k = 0; k < d; k += 4) {
      float x[4];
      float4 c[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        x[u] = v[k + u];
        c[u] = w[k + u];
      }
#pragma unroll
      for (int u = 0; u < 4; u += 2) {
        a0 = fmaf(x[u], c[u].x, a0);
        a1 = fmaf(x[u], c[u].y, a1);
        a2 = fmaf(x[u], c[u].z, a2);
        a3 = fmaf(x[u], c[u].w, a3);
        b0 = fmaf(x[u + 1], c[u + 1].x, b0);
        b1 = fmaf(x[u + 1], c[u + 1].y, b1);
        b2 = fmaf(x[u + 1], c[u + 1].z, b2);
        b3 = fmaf(x[u + 1], c[u + 1].w, b3);
      }
    }
    const float z0 = a0 + b0, z1 = a1 + b1, z2 = a2 + b2, z3 = a3 + b3;
    const float n2 = z0 * z0 + z1 * z1 + z2 * z2 + z3 * z3;
    if (i < N) {
      const size_t o = ((size_t)b * H + g * grp + jh) * N + i;
      reinterpret_cast<float4*>(Z)[o] = make_float4(z0, z1, z2, z3);
      zn2[o] = n2;
    }
    zs[ii * grp + jh] = i < N ? n2 : 0.f;
  }
  __syncthreads();
  // per head of the group: eight threads sum every eighth token, a fixed
  // shuffle tree adds the eight
  for (int jh0 = 0; jh0 < grp; jh0 += (int)blockDim.x / 8) {  // uniform over the block
    const int jh = jh0 + (int)threadIdx.x / 8, pt = threadIdx.x & 7;
    float sacc = 0.f;
    if (jh < grp)
      for (int ii = pt; ii < PR_TOK; ii += 8) sacc += zs[ii * grp + jh];
    sacc += __shfl_xor_sync(FULL, sacc, 4);
    sacc += __shfl_xor_sync(FULL, sacc, 2);
    sacc += __shfl_xor_sync(FULL, sacc, 1);
    if (jh < grp && pt == 0) sigpart[((size_t)b * nP + pb) * H + g * grp + jh] = sacc;
  }
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) last = atomicAdd(&tick[b], 1u) == (unsigned)(nP * Hkv - 1);
  __syncthreads();
  if (!last) return;
  __threadfence();
  // the image's partials: eight threads per head sum every eighth partial
  // (read past L1: other blocks wrote them), a fixed shuffle tree adds the
  // eight (fp32: the partials are fp32 sums already)
  const float* sp = sigpart + (size_t)b * nP * H;
  const int part = threadIdx.x & 7;
  for (int h0 = 0; h0 < H; h0 += (int)blockDim.x / 8) {  // uniform over the block
    const int h = h0 + (int)threadIdx.x / 8;
    float sacc = 0.f;
    if (h < H) {
#pragma unroll 4
      for (int q = part; q < nP; q += 8) sacc += __ldcg(&sp[(size_t)q * H + h]);
    }
    sacc += __shfl_xor_sync(FULL, sacc, 4);
    sacc += __shfl_xor_sync(FULL, sacc, 2);
    sacc += __shfl_xor_sync(FULL, sacc, 1);
    if (h < H && part == 0)
      sigma[(size_t)b * H + h] =
          sqrtf(lambda_mass) * fmaxf(sqrtf(sacc) / sqrtf((float)N * 4.f), eps_mass);
  }
}

// K == N: the unmodified execution.  One block per output row copies the
// hidden row, both K/V rows and the position ids; out_idx = 0..N-1.
template <typename Tin>
__global__ void k_identity(const Tin* __restrict__ hidden, const Tin* __restrict__ keys,
                           const int32_t* __restrict__ pos, const int32_t* toff, int B, int N,
                           int Tmax, int D, int HD, int32_t* out_idx, Tin* out_hidden,
                           Tin* out_kv, int32_t* out_pos, uint32_t* status, PrefixKV pf) {
  grid_dep_wait();
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
  for (int l = 0; l < pf.n; ++l)  // dense prefix layers: unchanged as well
    for (int w = 0; w < 2; ++w) {
      const Tin* kl = static_cast<const Tin*>(pf.keys[l]);
      const uint4* ks = reinterpret_cast<const uint4*>(
          kl + (w == 0 ? sq.key_row(r, HD) : sq.value_row(r, HD)));
      uint4* kd = reinterpret_cast<uint4*>(static_cast<Tin*>(pf.out[l]) + sq.out_kv_row(w, r, HD));
      for (int k = threadIdx.x; k < nkv; k += blockDim.x) kd[k] = ks[k];
    }
  if (threadIdx.x < 3) out_pos[sq.out_pos(threadIdx.x, r)] = pos[sq.pos(threadIdx.x, r)];
  if (threadIdx.x == 0 && r < N) out_idx[(size_t)b * N + r] = r;
}

cudaError_t launch_rownorm(const Dims& dm, const void* hidden, float norm_eps, Scratch& s,
                           cudaStream_t st) {
  dim3 grid(ceil_div(dm.N, ROWS_PER_BLOCK), dm.B);
  if (dm.dtype == GMC_BF16)
    launch_k(k_rownorm<__nv_bfloat16>, grid, 32 * ROWS_PER_BLOCK, 0, st, 1,
        (const __nv_bfloat16*)hidden, dm.toff, dm.B, dm.N, dm.K, dm.T, dm.D, norm_eps, s.rn,
        s.rmsh, s.u0, s.status);
  else
    launch_k(k_rownorm<float>, grid, 32 * ROWS_PER_BLOCK, 0, st, 1, (const float*)hidden, dm.toff, dm.B,
                                                           dm.N, dm.K, dm.T, dm.D, norm_eps, s.rn,
                                                           s.rmsh, s.u0, s.status);
  return cudaGetLastError();
}

cudaError_t launch_rms_rows(const Dims& dm, const void* hidden, float* rmsh, uint32_t* status,
                            cudaStream_t st) {
  dim3 grid(ceil_div(dm.N, ROWS_PER_BLOCK), dm.B);
  if (dm.dtype == GMC_BF16)
    launch_k(k_rownorm<__nv_bfloat16>, grid, 32 * ROWS_PER_BLOCK, 0, st, 1,
        (const __nv_bfloat16*)hidden, dm.toff, dm.B, dm.N, dm.K, dm.T, dm.D, 1e-12f, nullptr,
        rmsh, nullptr, status);
  else
    launch_k(k_rownorm<float>, grid, 32 * ROWS_PER_BLOCK, 0, st, 1, (const float*)hidden, dm.toff, dm.B,
                                                           dm.N, dm.K, dm.T, dm.D, 1e-12f,
                                                           nullptr, rmsh, nullptr, status);
  return cudaGetLastError();
}

cudaError_t launch_probe(const Dims& dm, const void* keys, const float* W, const void* queries,
                         const gmc_params& p, Scratch& s, cudaStream_t st) {
  const bool pack = message_tc_supported(dm);  // the packed queries of the tensor-core slice
  const int RQ = pack ? message_rq(dm) : 0;
  __nv_bfloat16* Qp = pack ? s.Qp : nullptr;
  const __nv_bfloat16* q16 = static_cast<const __nv_bfloat16*>(queries);
  const int grp = dm.H / dm.Hkv;
  dim3 grid(s.nP, dm.Hkv, dm.B);
  const size_t smem = sizeof(float4) * grp * (dm.d + 1) +
                      sizeof(float) * ((size_t)PR_TOK * (dm.d + 1) + (size_t)PR_TOK * grp);
  cudaError_t e;
  if (dm.dtype == GMC_BF16) {
    if ((e = set_smem_limit((const void*)k_probe<__nv_bfloat16>, smem)) != cudaSuccess) return e;
    launch_k(k_probe<__nv_bfloat16>, grid, 256, smem, st, 1,
        (const __nv_bfloat16*)keys, W, dm.toff, dm.B, dm.N, dm.K, dm.T, dm.H, dm.Hkv, dm.d,
        p.lambda_mass, p.eps_mass, s.Z, s.zn2, s.sigpart, s.nP, s.sigma, s.tick, q16, RQ, Qp,
        s.status);
  } else {
    if ((e = set_smem_limit((const void*)k_probe<float>, smem)) != cudaSuccess) return e;
    launch_k(k_probe<float>, grid, 256, smem, st, 1, (const float*)keys, W, dm.toff, dm.B, dm.N, dm.K,
                                            dm.T, dm.H, dm.Hkv, dm.d, p.lambda_mass, p.eps_mass,
                                            s.Z, s.zn2, s.sigpart, s.nP, s.sigma, s.tick,
                                            q16, RQ, Qp, s.status);
  }
  return cudaGetLastError();
}

cudaError_t launch_identity(const Dims& dm, const void* hidden, const void* keys,
                            const int32_t* pos, int32_t* out_idx, void* out_hidden, void* out_kv,
                            int32_t* out_pos, uint32_t* status, cudaStream_t st,
                            const PrefixKV* prefix) {
  dim3 grid(dm.N + dm.T, dm.B);
  const int HD = dm.Hkv * dm.d;
  PrefixKV pf{};
  if (prefix) pf = *prefix;
  if (dm.dtype == GMC_BF16)
    launch_k(k_identity<__nv_bfloat16>, grid, 128, 0, st, 1,
        (const __nv_bfloat16*)hidden, (const __nv_bfloat16*)keys, pos, dm.toff, dm.B, dm.N, dm.T,
        dm.D, HD, out_idx, (__nv_bfloat16*)out_hidden, (__nv_bfloat16*)out_kv, out_pos, status, pf);
  else
    launch_k(k_identity<float>, grid, 128, 0, st, 1, (const float*)hidden, (const float*)keys, pos,
                                            dm.toff, dm.B, dm.N, dm.T, dm.D, HD, out_idx,
                                            (float*)out_hidden, (float*)out_kv, out_pos, status, pf);
  return cudaGetLastError();
}

}  // namespace gmc
