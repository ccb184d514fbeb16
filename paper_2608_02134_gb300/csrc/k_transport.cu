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

// Exclusive scan of one int per thread over the block (every thread calls it).
__device__ inline int sel_block_scan(int v, int* wsum, int* total) {
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(FULL, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) wsum[w] = x;
  __syncthreads();
  int before = 0, tot = 0;
  for (int q = 0; q < nw; ++q) {
    const int c = wsum[q];
    before += q < w ? c : 0;
    tot += c;
  }
  __syncthreads();
  *total = tot;
  return before + x - v;
}
// Raw 8-element slices of a row, kept in registers while more member rows are
// in flight (a cluster can hold dozens of members: each batch is one memory
// round trip).
template <typename Tin> struct Raw8;
template <> struct Raw8<__nv_bfloat16> {
  static constexpr int ILP = 16;  // member rows in flight per thread (4 registers each)
  uint4 r;
  __device__ __forceinline__ void load(const __nv_bfloat16* p) { r = *reinterpret_cast<const uint4*>(p); }
  __device__ __forceinline__ void to_f32(float* v) const {
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&r);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float2 f = __bfloat1622float2(h[q]);
      v[2 * q] = f.x;
      v[2 * q + 1] = f.y;
    }
  }
};
template <> struct Raw8<float> {
  static constexpr int ILP = 8;  // 8 registers each
  float4 a, c;
  __device__ __forceinline__ void load(const float* p) {
    a = *reinterpret_cast<const float4*>(p);
    c = *reinterpret_cast<const float4*>(p + 4);
  }
  __device__ __forceinline__ void to_f32(float* v) const {
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
    v[4] = c.x; v[5] = c.y; v[6] = c.z; v[7] = c.w;
  }
};

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

constexpr int TR_WIN = 4;  // tokens per thread in one membership window

// One block per output row r of an image:
//   r < K:  carrier j = support[r]: its members (pi(i) = j, ascending source
//           order), M_j, c_j, RMS restoration, the compact hidden row; plus the
//           carrier's K/V rows, position ids and out_idx;
//   r >= K: text row N + (r - K): hidden, K/V and position ids copied.
// Members are found in windows of TR_WIN * blockDim tokens: every thread reads
// TR_WIN consecutive assignments, a block scan of the counts orders them.
template <typename Tin, int MAXT>
__global__ void __launch_bounds__(MAXT) k_transport(
    const Tin* __restrict__ hidden, const Tin* __restrict__ keys, const int32_t* __restrict__ pos,
    const int32_t* __restrict__ support, const int32_t* __restrict__ pi,
    const float* __restrict__ mass, const float* __restrict__ rmsh, const int32_t* toff, int B,
    int N, int K, int Tmax, int D, int HD, float rms_eps, int check, int32_t* out_idx,
    Tin* out_hidden, Tin* out_kv, int32_t* out_pos, uint32_t* status) {
  __shared__ int members[TR_WIN * MAXT];
  __shared__ int wsum[32];
  __shared__ float red[32];
  const int b = blockIdx.y, r = blockIdx.x;
  const TextGeom tg = text_geom(toff, b, B, Tmax, status);
  if (tg.T == 0 || r >= K + tg.T) return;
  const SeqIdx sq(b, N, K, tg.off, tg.T);
  // the first membership window's assignments are loaded with the carrier id
  int pw[TR_WIN];
  if (r < K) {
#pragma unroll
    for (int u = 0; u < TR_WIN; ++u) {
      const int i = threadIdx.x * TR_WIN + u;
      pw[u] = i < N ? pi[(size_t)b * N + i] : -1;
    }
  }
  const int src = r < K ? support[(size_t)b * K + r] : N + (r - K);
  // K/V rows, position ids, out_idx of the kept row (bit-exact gathers)
  {
    const int nkv = HD * (int)sizeof(Tin) / 16;
    for (int q = threadIdx.x; q < 2 * nkv; q += blockDim.x) {
      const int w = q >= nkv, e = q - w * nkv;
      const uint4* sp = reinterpret_cast<const uint4*>(
          keys + (w == 0 ? sq.key_row(src, HD) : sq.value_row(src, HD)));
      reinterpret_cast<uint4*>(out_kv + sq.out_kv_row(w, r, HD))[e] = sp[e];
    }
    if (threadIdx.x < 3) out_pos[sq.out_pos(threadIdx.x, r)] = pos[sq.pos(threadIdx.x, src)];
    if (threadIdx.x == 0 && r < K) out_idx[(size_t)b * K + r] = src;
  }
  if (r >= K) {  // text row
    const uint4* sp = reinterpret_cast<const uint4*>(hidden + sq.hidden_row(src, D));
    uint4* dp = reinterpret_cast<uint4*>(out_hidden + sq.out_hidden_row(r, D));
    for (int q = threadIdx.x; q < D * (int)sizeof(Tin) / 16; q += blockDim.x) dp[q] = sp[q];
    return;
  }
  const int j = src;
  const float rms_j = rmsh[(size_t)b * N + j];
  const int e0 = threadIdx.x * TR_VEC;
  const bool active = e0 < D;
  float acc[TR_VEC];
#pragma unroll
  for (int q = 0; q < TR_VEC; ++q) acc[q] = 0.f;
  float Msum = 0.f;
  const int win = TR_WIN * blockDim.x;
  for (int base = 0; base < N; base += win) {
    const int t0 = base + threadIdx.x * TR_WIN;
    int mine[TR_WIN], cnt = 0;
#pragma unroll
    for (int u = 0; u < TR_WIN; ++u) {
      const int i = t0 + u;
      const int pv = base == 0 ? pw[u] : (i < N ? pi[(size_t)b * N + i] : -1);
      mine[u] = (i < N && pv == j) ? i : -1;
      cnt += mine[u] >= 0;
    }
    int total = 0;
    int at = sel_block_scan(cnt, wsum, &total);
#pragma unroll
    for (int u = 0; u < TR_WIN; ++u)
      if (mine[u] >= 0) members[at++] = mine[u];
    __syncthreads();
    // ascending source order; ILP member rows are loaded before any is added
    constexpr int ILP = MAXT > 512 ? Raw8<Tin>::ILP / 4 : Raw8<Tin>::ILP;  // registers per thread
    for (int q0 = 0; q0 < total; q0 += ILP) {
      Raw8<Tin> raw[ILP];
      float wg[ILP];
#pragma unroll
      for (int u = 0; u < ILP; ++u) {
        wg[u] = 0.f;
        if (q0 + u < total) {
          const int m = members[q0 + u];
          wg[u] = mass[(size_t)b * N + m];
          if (active) raw[u].load(hidden + sq.hidden_row(m, D) + e0);
        }
      }
#pragma unroll
      for (int u = 0; u < ILP; ++u)
        if (q0 + u < total) {
          Msum += wg[u];
          if (active) {
            float v[TR_VEC];
            raw[u].to_f32(v);
#pragma unroll
            for (int t = 0; t < TR_VEC; ++t) acc[t] = fmaf(wg[u], v[t], acc[t]);
          }
        }
    }
    __syncthreads();  // members is refilled by the next window
  }
  const float invM = 1.f / Msum;
  float ss = 0.f;
#pragma unroll
  for (int t = 0; t < TR_VEC; ++t) {
    acc[t] *= invM;
    if (active) ss = fmaf(acc[t], acc[t], ss);
  }
  ss = block_reduce(ss, red, OpAdd(), 0.f);
  const float rc = sqrtf(ss / (float)D);
  const float scale = rms_j / (rc + rms_eps);
  if (active) {
    float v[TR_VEC];
#pragma unroll
    for (int t = 0; t < TR_VEC; ++t) {
      v[t] = acc[t] * scale;
      if (check && !isfinite(v[t])) set_status(status, GMC_STATUS_NONFINITE);
    }
    Vec8<Tin>::store(out_hidden + sq.out_hidden_row(r, D) + e0, v);
  }
}

cudaError_t launch_transport(const Dims& dm, const gmc_params& p, const void* hidden,
                             const void* keys, const int32_t* pos, const int32_t* support,
                             const int32_t* pi, const float* mass, const float* rmsh,
                             int32_t* out_idx, void* out_hidden, void* out_kv, int32_t* out_pos,
                             uint32_t* status, cudaStream_t st) {
  const int threads = max(128, ((ceil_div(dm.D, TR_VEC) + 31) / 32) * 32);
  dim3 grid(dm.K + dm.T, dm.B);
  const int HD = dm.Hkv * dm.d;
  auto go = [&](auto kernel, const auto* h, const auto* k, auto* oh, auto* okv) {
    kernel<<<grid, threads, 0, st>>>(h, k, pos, support, pi, mass, rmsh, dm.toff, dm.B, dm.N, dm.K,
                                     dm.T, dm.D, HD, p.rms_eps, p.check_mode, out_idx, oh, okv,
                                     out_pos, status);
  };
  if (dm.dtype == GMC_BF16) {
    using T = __nv_bfloat16;
    if (threads <= 512)
      go(k_transport<T, 512>, (const T*)hidden, (const T*)keys, (T*)out_hidden, (T*)out_kv);
    else
      go(k_transport<T, 1024>, (const T*)hidden, (const T*)keys, (T*)out_hidden, (T*)out_kv);
  } else {
    if (threads <= 512)
      go(k_transport<float, 512>, (const float*)hidden, (const float*)keys, (float*)out_hidden,
         (float*)out_kv);
    else
      go(k_transport<float, 1024>, (const float*)hidden, (const float*)keys, (float*)out_hidden,
         (float*)out_kv);
  }
  return cudaGetLastError();
}

}  // namespace gmc
