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
// [support ascending ; N .. N+T_b-1], and so are the K/V rows of the dense
// prefix layers when the caller passes them (the cached path).
#include "common.cuh"
#include "kernels.cuh"

#include <cooperative_groups.h>
#include <algorithm>

namespace gmc {
namespace cg = cooperative_groups;

constexpr int TR_VEC = 8;       // elements per thread per row (one 16-B bf16 chunk)
constexpr int TR_THREADS = 128;  // threads per CTA
constexpr int TR_WIN = 16;       // assignments per thread in one membership window
constexpr int TR_MAXS = 8;       // CTAs per output row (portable cluster size)
constexpr int TR_KVS = 2;        // K/V 16-B units per thread and row staged asynchronously
constexpr int TR_FW = 4;         // bitmap words per thread of the single-pass membership scan

// Raw 8-element slices of a row, kept in registers while more member rows are
// in flight (a cluster can hold dozens of members: each batch is one memory
// round trip).
template <typename Tin> struct Raw8;
template <> struct Raw8<__nv_bfloat16> {
  static constexpr int ILP = 8;  // member rows in flight per thread (4 registers each)
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
  static constexpr int ILP = 4;  // 8 registers each
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
  static __device__ __forceinline__ void store(__nv_bfloat16* p, const float* v) {
    uint4 raw;
    __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&raw);
#pragma unroll
    for (int q = 0; q < 4; ++q) h[q] = __floats2bfloat162_rn(v[2 * q], v[2 * q + 1]);
    *reinterpret_cast<uint4*>(p) = raw;
  }
};
template <> struct Vec8<float> {
  static __device__ __forceinline__ void store(float* p, const float* v) {
    *reinterpret_cast<float4*>(p) = make_float4(v[0], v[1], v[2], v[3]);
    *reinterpret_cast<float4*>(p + 4) = make_float4(v[4], v[5], v[6], v[7]);
  }
};

// CTAs per output row: the row's D/8 chunks split so a CTA holds at most 128.
inline int transport_split(int D) {
  return std::min(TR_MAXS, std::max(1, ceil_div(D / TR_VEC, TR_THREADS)));
}

// A cluster of S CTAs per row index r of an image (CTA rank = slice of D):
//   r < K:    carrier j = support[r]: its members (pi(i) = j, ascending source
//             order), M_j, c_j over the CTA's slice, the slice's sum of squares
//             sent to every CTA of the row through distributed shared memory
//             (summed in rank order, so every slice applies the same RMS
//             scale), the compact hidden row r; plus the carrier's K/V rows,
//             position ids and out_idx;
//   r < T_b:  text row N + r copied to output row K + r (hidden, K/V and
//             position ids), beside the carrier's work.
// Members are found in windows of TR_WIN * TR_THREADS tokens, as one 32-bit
// mask per 32 tokens: read from the carrier's membership bitmap when the
// assignment kernel wrote one (mbits != nullptr), else built by ballots over
// the assignment (token base + u * TR_THREADS + tid read by thread tid,
// coalesced).  The masks' counts, scanned in token order, place every member
// in ascending source order.  With a bitmap of at most TR_FW words per
// thread (N <= 16384), every word is read at once (thread t: words TR_FW t ..)
// and one scan places all members when they fit one window: long prefixes
// have thousands of carriers with a few members each, and the windows'
// barriers would dominate.
template <typename Tin>
__global__ void __launch_bounds__(TR_THREADS, 7) k_transport(
    const Tin* __restrict__ hidden, const Tin* __restrict__ keys, const int32_t* __restrict__ pos,
    const int32_t* __restrict__ support, const int32_t* __restrict__ pi,
    const float* __restrict__ mass, const float* __restrict__ rmsh,
    const uint32_t* __restrict__ mbits, const int32_t* toff, int B, int N, int K, int Tmax, int D,
    int HD, int S, float rms_eps, int check, int32_t* out_idx, Tin* out_hidden, Tin* out_kv,
    int32_t* out_pos, uint32_t* status, PrefixKV pf) {
  grid_dep_wait();
  constexpr int NW = TR_THREADS / 32;
  constexpr int NM = TR_WIN * NW;  // 32-token masks per window
  static_assert(NM * 32 == TR_WIN * TR_THREADS, "one mask per 32 tokens of a window");
  constexpr int ILP = Raw8<Tin>::ILP;
  __shared__ uint16_t members[TR_WIN * TR_THREADS];  // N <= 8192
  __shared__ int cnt[TR_WIN * NW + 1];
  __shared__ unsigned balw[TR_WIN * NW];
  __shared__ float red[NW];
  __shared__ float ss_all[TR_MAXS];
  // bit-exact gathers land here while the membership scan runs: text hidden
  // slice (2 units), text K/V, carrier K/V; position ids of both rows
  __shared__ uint4 stage[2 + 2 * TR_KVS][TR_THREADS];
  __shared__ int stpos[2][4];
  const int b = blockIdx.y, r = blockIdx.x / S, part = blockIdx.x % S;
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const bool car = r < K;
  // loads that do not depend on the text geometry are issued first: the first
  // membership window (bitmap words or assignments) and the carrier id
  const int nwd = (N + 31) >> 5;
  const uint32_t* bits = mbits ? mbits + ((size_t)b * K + r) * nwd : nullptr;
  int pw[TR_WIN];
  uint32_t bw = 0;
  const bool single = bits && nwd <= TR_FW * TR_THREADS;  // uniform over the cluster
  uint32_t fw[TR_FW];
#pragma unroll
  for (int q = 0; q < TR_FW; ++q) fw[q] = 0u;
  if (car) {
    if (single) {
#pragma unroll
      for (int q = 0; q < TR_FW; ++q) {
        const int x = TR_FW * (int)threadIdx.x + q;
        if (x < nwd) fw[q] = bits[x];
      }
    } else if (bits) {
      if (threadIdx.x < NM && threadIdx.x < nwd) bw = bits[threadIdx.x];
    } else {
#pragma unroll
      for (int u = 0; u < TR_WIN; ++u) {
        const int i = u * TR_THREADS + threadIdx.x;
        pw[u] = i < N ? pi[(size_t)b * N + i] : -1;
      }
    }
  }
  const int j = car ? support[(size_t)b * K + r] : 0;
  const TextGeom tg = text_geom(toff, b, B, Tmax, status);
  // every condition below is uniform over the cluster (one row per cluster)
  if (tg.T == 0) return;
  const bool txt = r < tg.T;
  if (!car && !txt) return;
  const SeqIdx sq(b, N, K, tg.off, tg.T);
  const int nkv = HD * (int)sizeof(Tin) / 16;
  // K/V rows (this CTA's share) and position ids of kept sequence row src:
  // the first TR_KVS units per thread are copied into shared memory without
  // waiting (cp.async); they are written to output row dst at the end
  auto kv_src = [&](int src, int q) {
    const int wv = q >= nkv, e = q - wv * nkv;
    return reinterpret_cast<const uint4*>(
               keys + (wv == 0 ? sq.key_row(src, HD) : sq.value_row(src, HD))) + e;
  };
  auto kv_dst = [&](int dst, int q) {
    const int wv = q >= nkv, e = q - wv * nkv;
    return reinterpret_cast<uint4*>(out_kv + sq.out_kv_row(wv, dst, HD)) + e;
  };
  auto stage_kv_pos = [&](int src, int slot) {
#pragma unroll
    for (int t = 0; t < TR_KVS; ++t) {
      const int q = part * TR_THREADS + threadIdx.x + t * S * TR_THREADS;
      if (q < 2 * nkv) cp_async16(&stage[2 + slot * TR_KVS + t][threadIdx.x], kv_src(src, q));
    }
    if (part == 0 && threadIdx.x < 3)
      cp_async4(&stpos[slot][threadIdx.x], pos + sq.pos(threadIdx.x, src), true);
  };
  auto flush_kv_pos = [&](int src, int dst, int slot) {
#pragma unroll
    for (int t = 0; t < TR_KVS; ++t) {
      const int q = part * TR_THREADS + threadIdx.x + t * S * TR_THREADS;
      if (q < 2 * nkv) *kv_dst(dst, q) = stage[2 + slot * TR_KVS + t][threadIdx.x];
    }
    for (int q = part * TR_THREADS + threadIdx.x + TR_KVS * S * TR_THREADS; q < 2 * nkv;
         q += S * TR_THREADS)
      *kv_dst(dst, q) = *kv_src(src, q);
    if (part == 0 && threadIdx.x < 3) out_pos[sq.out_pos(threadIdx.x, dst)] = stpos[slot][threadIdx.x];
  };
  // the dense prefix layers' K/V of kept row src, written to output row dst;
  // the loads of PL layers are in flight together
  auto copy_prefix = [&](int src, int dst) {
    constexpr int PL = 8;
    for (int l0 = 0; l0 < pf.n; l0 += PL)
      for (int q = part * TR_THREADS + threadIdx.x; q < 2 * nkv; q += S * TR_THREADS) {
        const int wv = q >= nkv, e = q - wv * nkv;
        const size_t ro = wv == 0 ? sq.key_row(src, HD) : sq.value_row(src, HD);
        const size_t wo = sq.out_kv_row(wv, dst, HD);
        uint4 v[PL];
#pragma unroll
        for (int u = 0; u < PL; ++u)
          if (l0 + u < pf.n)
            v[u] = reinterpret_cast<const uint4*>(static_cast<const Tin*>(pf.keys[l0 + u]) + ro)[e];
#pragma unroll
        for (int u = 0; u < PL; ++u)
          if (l0 + u < pf.n) reinterpret_cast<uint4*>(static_cast<Tin*>(pf.out[l0 + u]) + wo)[e] = v[u];
      }
  };
  // this CTA's slice of D, in 8-element chunks
  const int nch = D / TR_VEC, cper = ceil_div(nch, S);
  const int c = part * cper + threadIdx.x;
  const bool active = threadIdx.x < cper && c < nch;
  const int e0 = c * TR_VEC;
  constexpr int U = TR_VEC * (int)sizeof(Tin) / 16;  // 16-B units per chunk
  if (txt) {  // text row N + r -> output row K + r
    if (active) {
      const uint4* sp = reinterpret_cast<const uint4*>(hidden + sq.hidden_row(N + r, D) + e0);
#pragma unroll
      for (int q = 0; q < U; ++q) cp_async16(&stage[q][threadIdx.x], sp + q);
    }
    stage_kv_pos(N + r, 0);
  }
  if (car) stage_kv_pos(j, 1);
  cp_async_commit();
  // the staged rows are written out by the thread that staged them
  auto flush_all = [&]() {
    cp_async_wait<0>();
    if (txt) {
      if (active) {
        uint4* dp = reinterpret_cast<uint4*>(out_hidden + sq.out_hidden_row(K + r, D) + e0);
#pragma unroll
        for (int q = 0; q < U; ++q) dp[q] = stage[q][threadIdx.x];
      }
      flush_kv_pos(N + r, K + r, 0);
      copy_prefix(N + r, K + r);
    }
    if (car) {
      flush_kv_pos(j, r, 1);
      copy_prefix(j, r);
    }
  };
  if (!car) {
    flush_all();
    return;
  }
  // first phase of the cluster barrier: every CTA of the row has started
  // before any writes into its shared memory (waited on just before that)
  if (S > 1) asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
  if (part == 0 && threadIdx.x == 0) out_idx[(size_t)b * K + r] = j;
  const float rms_j = rmsh[(size_t)b * N + j];
  float acc[TR_VEC];
#pragma unroll
  for (int q = 0; q < TR_VEC; ++q) acc[q] = 0.f;
  float Msum = 0.f;
  // ascending source order; ILP member rows are loaded before any is added
  auto accumulate = [&](int total) {
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
  };
  bool scanned = false;
  if (single) {
    // counts of this thread's words, a block scan in thread (= token) order
    int c = 0;
#pragma unroll
    for (int q = 0; q < TR_FW; ++q) c += __popc(fw[q]);
    int incl = c;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(FULL, incl, o);
      if (lane >= o) incl += y;
    }
    if (lane == 31) cnt[w] = incl;
    __syncthreads();
    int before = 0, total = 0;
#pragma unroll
    for (int q = 0; q < NW; ++q) {
      before += q < w ? cnt[q] : 0;
      total += cnt[q];
    }
    if (total <= TR_WIN * TR_THREADS) {  // uniform over the block
      int pos = before + incl - c;
#pragma unroll
      for (int q = 0; q < TR_FW; ++q) {
        uint32_t m = fw[q];
        const int t0 = 32 * (TR_FW * (int)threadIdx.x + q);
        while (m) {
          const int bit = __ffs(m) - 1;
          members[pos++] = (uint16_t)(t0 + bit);
          m &= m - 1u;
        }
      }
      __syncthreads();
      accumulate(total);
      scanned = true;
    }
    __syncthreads();  // cnt is reused by the windows
  }
  for (int base = 0; base < (scanned ? 0 : N); base += TR_WIN * TR_THREADS) {
    // mask x of the window covers tokens base + 32 x .. base + 32 x + 31
    if (bits) {
      if (threadIdx.x < NM) {
        const int x = (base >> 5) + threadIdx.x;
        const uint32_t m = base == 0 ? bw : (x < nwd ? bits[x] : 0u);
        cnt[threadIdx.x] = __popc(m);
        balw[threadIdx.x] = m;
      }
    } else {
#pragma unroll
      for (int u = 0; u < TR_WIN; ++u) {
        const int i = base + u * TR_THREADS + threadIdx.x;
        const int pv = base == 0 ? pw[u] : (i < N ? pi[(size_t)b * N + i] : -1);
        const unsigned bal = __ballot_sync(FULL, i < N && pv == j);
        if (lane == 0) {  // u * TR_THREADS + 32 w = 32 (u * NW + w)
          cnt[u * NW + w] = __popc(bal);
          balw[u * NW + w] = bal;
        }
      }
    }
    __syncthreads();
    if (w == 0) {  // exclusive scan of the mask counts, in token order
      constexpr int PER = (TR_WIN * NW + 31) / 32;
      int loc[PER], sum = 0;
#pragma unroll
      for (int q = 0; q < PER; ++q) {
        const int x = lane * PER + q;
        loc[q] = x < TR_WIN * NW ? cnt[x] : 0;
        sum += loc[q];
      }
      int incl = sum;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(FULL, incl, o);
        if (lane >= o) incl += y;
      }
      int run = incl - sum;
#pragma unroll
      for (int q = 0; q < PER; ++q) {
        const int x = lane * PER + q;
        if (x < TR_WIN * NW) cnt[x] = run;
        run += loc[q];
      }
      if (lane == 31) cnt[TR_WIN * NW] = incl;
    }
    __syncthreads();
    const unsigned lt = (1u << lane) - 1u;
#pragma unroll
    for (int u = 0; u < TR_WIN; ++u) {
      const unsigned bal = balw[u * NW + w];
      if (bal >> lane & 1u)
        members[cnt[u * NW + w] + __popc(bal & lt)] =
            (uint16_t)(base + u * TR_THREADS + threadIdx.x);
    }
    const int total = cnt[TR_WIN * NW];
    __syncthreads();
    accumulate(total);
    __syncthreads();  // members and cnt are refilled by the next window
  }
  const float invM = 1.f / Msum;
  float ss = 0.f;
#pragma unroll
  for (int t = 0; t < TR_VEC; ++t) {
    acc[t] *= invM;
    if (active) ss = fmaf(acc[t], acc[t], ss);
  }
  ss = block_reduce(ss, red, OpAdd(), 0.f);
  float sst = ss;
  if (S > 1) {
    // the slice sum goes to slot `part` of every CTA of the row; one barrier
    // phase publishes the stores, then each CTA adds the S slots in rank order
    asm volatile("barrier.cluster.wait.aligned;" ::: "memory");
    if (threadIdx.x < S) *cg::this_cluster().map_shared_rank(&ss_all[part], threadIdx.x) = ss;
    asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
    asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
    sst = 0.f;
    for (int q = 0; q < S; ++q) sst += ss_all[q];
  }
  const float rc = sqrtf(sst / (float)D);
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
  flush_all();
}

cudaError_t launch_transport(const Dims& dm, const gmc_params& p, const void* hidden,
                             const void* keys, const int32_t* pos, const int32_t* support,
                             const int32_t* pi, const float* mass, const float* rmsh,
                             const uint32_t* mbits, int32_t* out_idx, void* out_hidden,
                             void* out_kv, int32_t* out_pos, uint32_t* status, cudaStream_t st,
                             const PrefixKV* prefix) {
  const int S = transport_split(dm.D);
  PrefixKV pf{};
  if (prefix) pf = *prefix;
  const int HD = dm.Hkv * dm.d;
  // mbits: the carrier membership bitmaps, or nullptr to scan the assignment
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(std::max(dm.K, dm.T) * S, dm.B);
  cfg.blockDim = dim3(TR_THREADS);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = S;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;  // see grid_dep_wait
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.numAttrs = 2;
  if (dm.dtype == GMC_BF16) {
    using T = __nv_bfloat16;
    return cudaLaunchKernelEx(&cfg, k_transport<T>, (const T*)hidden, (const T*)keys, pos, support,
                              pi, mass, rmsh, mbits, (const int32_t*)dm.toff, dm.B, dm.N, dm.K, dm.T,
                              dm.D, HD, S, p.rms_eps, p.check_mode, out_idx, (T*)out_hidden,
                              (T*)out_kv, out_pos, status, pf);
  }
  return cudaLaunchKernelEx(&cfg, k_transport<float>, (const float*)hidden, (const float*)keys,
                            pos, support, pi, mass, rmsh, mbits, (const int32_t*)dm.toff, dm.B,
                            dm.N,
                            dm.K, dm.T, dm.D, HD, S, p.rms_eps, p.check_mode, out_idx,
                            (float*)out_hidden, (float*)out_kv, out_pos, status, pf);
}

}  // namespace gmc
