// Population transport (Sec. 3.4, Eq. (5); appendix Eq. (cond-transport)) and
// physical compaction (Algorithm 1 step 6; appendix "Index map and physical
// token accounting").
//
// Carrier j = support[k] receives the cluster C_j = {i : pi(i) = j}:
//   M_j = sum_{i in C_j} m_i,  c_j = M_j^-1 sum_{i in C_j} m_i h_i   (fp32 accumulation)
//   h~_j = c_j * rms(h_j) / (rms(c_j) + eps)                          (one cast to the
//                                                                     output type, RNE)
// and is written to compact row k.  Members are summed in ascending source
// order, so the result does not depend on scheduling.  Text rows, K/V rows
// and position ids are gathered bit-exactly at the kept sequence rows
// [support ascending ; N .. N+T_b-1].
#include "common.cuh"
#include "kernels.cuh"

namespace gmc {

constexpr int TR_VEC = 8;  // elements per thread per row
constexpr int TR_ILP = 4;  // member rows in flight per thread

template <typename Tin> struct Vec8;
template <> struct Vec8<__nv_bfloat16> {
  static __device__ __forceinline__ void load(const __nv_bfloat16* p, float* v) {
    const uint4 raw = *reinterpret_cast<const uint4*>(p);
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&raw);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float2 f = __bfloat1622float2(h[q]);
      v[2 * q] = f.x;
      v[2 * q + 1] = f.y;
    }
  }
  static __device__ __forceinline__ void store(__nv_bfloat16* p, const float* v) {
    uint4 raw;
    __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&raw);
#pragma unroll
    for (int q = 0; q < 4; ++q) h[q] = __floats2bfloat162_rn(v[2 * q], v[2 * q + 1]);
    *reinterpret_cast<uint4*>(p) = raw;
  }
};
template <> struct Vec8<float> {
  static __device__ __forceinline__ void load(const float* p, float* v) {
    const float4 a = *reinterpret_cast<const float4*>(p);
    const float4 c = *reinterpret_cast<const float4*>(p + 4);
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
    v[4] = c.x; v[5] = c.y; v[6] = c.z; v[7] = c.w;
  }
  static __device__ __forceinline__ void store(float* p, const float* v) {
    *reinterpret_cast<float4*>(p) = make_float4(v[0], v[1], v[2], v[3]);
    *reinterpret_cast<float4*>(p + 4) = make_float4(v[4], v[5], v[6], v[7]);
  }
};

template <typename Tin>
__global__ void __launch_bounds__(1024) k_transport(
    const Tin* __restrict__ hidden, const int32_t* __restrict__ support,
    const int32_t* __restrict__ pi, const float* __restrict__ mass,
    const float* __restrict__ rmsh, const int32_t* toff, int B, int N, int K, int Tmax, int D,
    float rms_eps, int check, Tin* out_hidden, uint32_t* status) {
  __shared__ int members[1024];
  __shared__ int wcount[32];
  __shared__ double red[32];
  const int b = blockIdx.y, k = blockIdx.x;
  const TextGeom tg = text_geom(toff, b, B, Tmax, status);
  if (tg.T == 0) return;
  const SeqIdx sq(b, N, K, tg.off, tg.T);
  const int j = support[(size_t)b * K + k];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
  const int e0 = threadIdx.x * TR_VEC;
  const bool active = e0 < D;
  float acc[TR_VEC];
#pragma unroll
  for (int q = 0; q < TR_VEC; ++q) acc[q] = 0.f;
  float Msum = 0.f;
  for (int base = 0; base < N; base += blockDim.x) {
    const int i = base + threadIdx.x;
    const bool mine = i < N && pi[(size_t)b * N + i] == j;
    const unsigned bal = __ballot_sync(FULL, mine);
    if (lane == 0) wcount[w] = __popc(bal);
    __syncthreads();
    int before = 0, total = 0;
    for (int q = 0; q < nw; ++q) {
      before += q < w ? wcount[q] : 0;
      total += wcount[q];
    }
    if (mine) {
      unsigned lt;
      asm("mov.u32 %0, %%lanemask_lt;" : "=r"(lt));
      members[before + __popc(bal & lt)] = i;
    }
    __syncthreads();
    // ascending source order; TR_ILP member rows are loaded before any is added
    for (int q0 = 0; q0 < total; q0 += TR_ILP) {
      float v[TR_ILP][TR_VEC], wg[TR_ILP];
#pragma unroll
      for (int u = 0; u < TR_ILP; ++u) {
        wg[u] = 0.f;
        if (q0 + u < total) {
          const int src = members[q0 + u];
          wg[u] = mass[(size_t)b * N + src];
          if (active) Vec8<Tin>::load(hidden + sq.hidden_row(src, D) + e0, v[u]);
        }
      }
#pragma unroll
      for (int u = 0; u < TR_ILP; ++u)
        if (q0 + u < total) {
          Msum += wg[u];
          if (active) {
#pragma unroll
            for (int t = 0; t < TR_VEC; ++t) acc[t] = fmaf(wg[u], v[u][t], acc[t]);
          }
        }
    }
    __syncthreads();
  }
  const float invM = 1.f / Msum;
  float ssf = 0.f;
#pragma unroll
  for (int t = 0; t < TR_VEC; ++t) {
    acc[t] *= invM;
    if (active) ssf = fmaf(acc[t], acc[t], ssf);
  }
  const double ss = block_reduce((double)ssf, red, OpAdd(), 0.0);
  const float rc = (float)sqrt(ss / D);
  const float scale = rmsh[(size_t)b * N + j] / (rc + rms_eps);
  if (active) {
    float v[TR_VEC];
#pragma unroll
    for (int t = 0; t < TR_VEC; ++t) {
      v[t] = acc[t] * scale;
      if (check && !isfinite(v[t])) set_status(status, GMC_STATUS_NONFINITE);
    }
    Vec8<Tin>::store(out_hidden + sq.out_hidden_row(k, D) + e0, v);
  }
}

// Gather of the kept rows: text hidden rows, K/V rows, position ids and out_idx.
template <typename Tin>
__global__ void k_compact(const Tin* __restrict__ hidden, const Tin* __restrict__ keys,
                          const int32_t* __restrict__ pos, const int32_t* __restrict__ support,
                          const int32_t* toff, int B, int N, int K, int Tmax, int D, int HD,
                          int32_t* out_idx, Tin* out_hidden, Tin* out_kv, int32_t* out_pos,
                          uint32_t* status) {
  const int b = blockIdx.y, r = blockIdx.x;
  const TextGeom tg = text_geom(toff, b, B, Tmax, status);
  if (tg.T == 0 || r >= K + tg.T) return;
  const SeqIdx sq(b, N, K, tg.off, tg.T);
  const int src = r < K ? support[(size_t)b * K + r] : N + (r - K);
  if (r >= K) {
    const uint4* s = reinterpret_cast<const uint4*>(hidden + sq.hidden_row(src, D));
    uint4* d = reinterpret_cast<uint4*>(out_hidden + sq.out_hidden_row(r, D));
    for (int q = threadIdx.x; q < D * (int)sizeof(Tin) / 16; q += blockDim.x) d[q] = s[q];
  }
  const int nkv = HD * (int)sizeof(Tin) / 16;
  for (int w = 0; w < 2; ++w) {
    const uint4* s = reinterpret_cast<const uint4*>(
        keys + (w == 0 ? sq.key_row(src, HD) : sq.value_row(src, HD)));
    uint4* d = reinterpret_cast<uint4*>(out_kv + sq.out_kv_row(w, r, HD));
    for (int q = threadIdx.x; q < nkv; q += blockDim.x) d[q] = s[q];
  }
  if (threadIdx.x < 3) out_pos[sq.out_pos(threadIdx.x, r)] = pos[sq.pos(threadIdx.x, src)];
  if (threadIdx.x == 0 && r < K) out_idx[(size_t)b * K + r] = src;
}

cudaError_t launch_transport(const Dims& dm, const gmc_params& p, const void* hidden,
                             const void* keys, const int32_t* pos, const int32_t* support,
                             const int32_t* pi, const float* mass, const float* rmsh,
                             int32_t* out_idx, void* out_hidden, void* out_kv, int32_t* out_pos,
                             uint32_t* status, cudaStream_t st) {
  const int threads = ((ceil_div(dm.D, TR_VEC) + 31) / 32) * 32;
  dim3 g1(dm.K, dm.B);
  dim3 g2(dm.K + dm.T, dm.B);
  const int HD = dm.Hkv * dm.d;
  if (dm.dtype == GMC_BF16) {
    k_transport<__nv_bfloat16><<<g1, threads, 0, st>>>(
        (const __nv_bfloat16*)hidden, support, pi, mass, rmsh, dm.toff, dm.B, dm.N, dm.K, dm.T,
        dm.D, p.rms_eps, p.check_mode, (__nv_bfloat16*)out_hidden, status);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    k_compact<__nv_bfloat16><<<g2, 128, 0, st>>>(
        (const __nv_bfloat16*)hidden, (const __nv_bfloat16*)keys, pos, support, dm.toff, dm.B,
        dm.N, dm.K, dm.T, dm.D, HD, out_idx, (__nv_bfloat16*)out_hidden, (__nv_bfloat16*)out_kv,
        out_pos, status);
  } else {
    k_transport<float><<<g1, threads, 0, st>>>((const float*)hidden, support, pi, mass, rmsh,
                                               dm.toff, dm.B, dm.N, dm.K, dm.T, dm.D, p.rms_eps,
                                               p.check_mode, (float*)out_hidden, status);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    k_compact<float><<<g2, 128, 0, st>>>((const float*)hidden, (const float*)keys, pos, support,
                                         dm.toff, dm.B, dm.N, dm.K, dm.T, dm.D, HD, out_idx,
                                         (float*)out_hidden, (float*)out_kv, out_pos, status);
  }
  return cudaGetLastError();
}

}  // namespace gmc
