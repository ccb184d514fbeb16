// Native boundary attention slice on the tcgen05 tensor cores (bf16 path).
//
// For image b and key/value head g, the rows of the A operand are the text
// queries of the query heads of group g, packed as (j, t) -> j*T_b + t, and the
// B operand runs over the image's keys (N visual rows, then T_b text rows).
// A CTA owns 128 query rows and one split: a contiguous range of 128-key
// tiles.  Two launches:
//   statistics: online softmax statistics (max, sum of exp) per query row over
//           the split's keys it may see (all visual keys and text keys 0..t,
//           scale 1/sqrt(d)), written per split;
//   write:  the splits' statistics merged in a fixed order, then for the
//           split's visual keys i < N A[h,t,i] = exp(s_i - max) / sum, and the
//           split's part of rs[h,t] = sum_i A[h,t,i] g_h(i) with
//           g_h(i) = sqrt(||Z_h[i]||^2 + sigma_h^2).
// Recomputing the logits costs one more small MMA pass and avoids writing and
// re-reading raw scores; the splits put every SM to work on one image.  This
// is appendix Eq. (cond-native-message): the visual slice of the native causal
// softmax, not renormalised over the image.
//
// Roles: warp 8 / lane 0 loads the query tile once and streams key tiles with
// TMA through a 4-stage ring; warp 9 / lane 0 issues tcgen05.mma into two
// 128-column TMEM accumulators (double buffered); warps 0..7 read the
// accumulators (warp w: TMEM lanes 32*(w%4).., columns 64*(w/4)..) and do the
// softmax arithmetic.  Every wait is clock-bounded.
#include <cooperative_groups.h>

#include "common.cuh"
#include "kernels.cuh"
#include "tc.cuh"

namespace cg = cooperative_groups;

namespace gmc {

cudaError_t make_tmap_bf16(CUtensorMap* map, const void* base, uint64_t row_elems, uint64_t rows,
                           uint64_t pitch_elems, uint32_t box_rows);

namespace {
constexpr int BM = 128, BK = 64, STAGES = 2;
constexpr int SPLIT_TARGET_CTAS = 152;  // one wave of one CTA per SM on a 152-SM GB300
constexpr int TILE_BYTES = BM * BK * 2;
constexpr int EPI_WARPS = 16, THREADS = 32 * (EPI_WARPS + 2);
constexpr int EPI_PARTS = EPI_WARPS / 4;  // 32-column parts of a tile (warp w: lane quarter w % 4)
constexpr long long WAIT_CYCLES = 4000000000LL;

struct MsgCtl {
  uint64_t qfull;
  uint64_t full[STAGES];
  uint64_t empty[STAGES];
  uint64_t accf[2];
  uint64_t acce[2];
  uint32_t tmem;
  volatile int abort;
  float stat_m[EPI_PARTS][BM];
  float stat_l[EPI_PARTS][BM];
  float rsum[EPI_PARTS][BM];
};

// Fused kernel: 16 epilogue warps (warp w reads TMEM lanes 32*(w%4).. and the
// 32-column quarter w/4 of every tile), then the TMA producer and MMA warps.
constexpr int FE_WARPS = 16, FT_THREADS = 32 * (FE_WARPS + 2);

constexpr int FUSED_MAX_CLUSTER = 8;  // portable cluster size

// Control block of the fused kernel: barriers, this CTA's per-row statistics
// and the statistics of every split of the cluster.
struct FusedCtl {
  uint64_t qfull;
  uint64_t full[STAGES];
  uint64_t empty[STAGES];
  uint64_t accdone;
  uint32_t tmem;
  volatile int abort;
  float stat_m[4][BM];
  float stat_l[4][BM];
  float rsum[4][BM];
  // every split's statistics per query row (base-2 max, sum), written into
  // each CTA of the cluster by the split that owns them
  float all_m[FUSED_MAX_CLUSTER][BM];
  float all_l[FUSED_MAX_CLUSTER][BM];
};

__device__ __forceinline__ void fused_epi_barrier() {
  asm volatile("bar.sync 1, %0;" ::"n"(FE_WARPS * 32) : "memory");
}
constexpr int FUSED_MAX_TILES = 4;     // key tiles a CTA keeps in TMEM (4 x 128 columns)
constexpr int FUSED_STAGE_BYTES = FE_WARPS * 32 * 32 * 4;  // one 32 x 32 fp32 tile per warp

// Bytes before the control block: the operand tiles (query tile and key ring)
// while the MMAs run, then the epilogue warps' staging tiles.
__host__ __device__ inline size_t fused_region_bytes(int nkb) {
  const size_t ops = (size_t)nkb * TILE_BYTES * (1 + STAGES);
  return ops > (size_t)FUSED_STAGE_BYTES ? ops : (size_t)FUSED_STAGE_BYTES;
}

struct MsgSplit {
  int kt_per;  // key tiles per split
  int n;       // splits
};

MsgSplit msg_split(int B, int Hkv, int RQ, int N, int T) {
  const int nkt = (N + T + BM - 1) / BM;
  const int base = (RQ / BM) * Hkv * B;
  const int target = SPLIT_TARGET_CTAS / base > 1 ? SPLIT_TARGET_CTAS / base : 1;
  MsgSplit sp;
  sp.kt_per = (nkt + target - 1) / target;
  sp.n = (nkt + sp.kt_per - 1) / sp.kt_per;
  return sp;
}

size_t msg_smem_bytes(int nkb) {
  return 1024 + (size_t)nkb * TILE_BYTES * (1 + STAGES) + sizeof(MsgCtl);
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(tc::smem_u32(bar)) : "memory");
}
__device__ __forceinline__ void epi_barrier() {
  asm volatile("bar.sync 1, %0;" ::"n"(EPI_WARPS * 32) : "memory");
}
}  // namespace

__global__ void __launch_bounds__(THREADS, 1)
    k_message_tc(const __grid_constant__ CUtensorMap qmap, const __grid_constant__ CUtensorMap kmap,
                 const int32_t* toff, int B, int N, int Tmax, int H, int Hkv, int d, int RQ,
                 int mode, int kt_per, int nsplit, float2* part,
                 const float* __restrict__ zn2, const float* __restrict__ sigma, float* A,
                 float* rs, uint32_t* status) {
  grid_dep_wait();
  extern __shared__ uint8_t sm_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(sm_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const int nkb = d / BK;
  uint8_t* Qs = base;
  uint8_t* Ks = base + (size_t)nkb * TILE_BYTES;
  MsgCtl* ctl = reinterpret_cast<MsgCtl*>(base + (size_t)nkb * TILE_BYTES * (1 + STAGES));

  const int b = blockIdx.z / nsplit, split = blockIdx.z % nsplit, g = blockIdx.y, tile = blockIdx.x;
  const TextGeom tg = text_geom(toff, b, B, Tmax, status);
  const int grp = H / Hkv;
  if (tg.T == 0 || tile * BM >= grp * tg.T) return;  // uniform per CTA
  const int Tb = tg.T;
  const int nkeys = N + Tb;
  const int nkt = ceil_div(nkeys, BM);
  const int c0 = split * kt_per, c1 = min(nkt, c0 + kt_per);
  const int iters = max(0, c1 - c0);  // an image with fewer keys than the widest one
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int qrow0 = (int)(((size_t)b * Hkv + g) * RQ + (size_t)tile * BM);
  const int krow0 = (int)(2 * ((size_t)b * N + tg.off));

  if (threadIdx.x == 0) {
    tc::mbar_init(&ctl->qfull, 1);
    for (int s = 0; s < STAGES; ++s) {
      tc::mbar_init(&ctl->full[s], 1);
      tc::mbar_init(&ctl->empty[s], 1);
    }
    for (int q = 0; q < 2; ++q) {
      tc::mbar_init(&ctl->accf[q], 1);
      tc::mbar_init(&ctl->acce[q], EPI_WARPS);
    }
    ctl->abort = 0;
    tc::fence_mbar_init();
    tc::prefetch_tmap(&qmap);
    tc::prefetch_tmap(&kmap);
  }
  if (warp == 0) {
    tc::tmem_alloc(&ctl->tmem, 256);
    tc::tmem_relinquish();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = ctl->tmem;
  const long long deadline = clock64() + WAIT_CYCLES;

  if (warp == EPI_WARPS) {  // ---------------- TMA producer
    int issued = 0;
    if (lane == 0) {
      tc::mbar_arrive_expect_tx(&ctl->qfull, nkb * TILE_BYTES);
      for (int kb = 0; kb < nkb; ++kb)
        tc::tma_load_2d(Qs + kb * TILE_BYTES, &qmap, kb * BK, qrow0, &ctl->qfull);
      for (int it = 0; it < iters; ++it) {
        const int s = it % STAGES, c = c0 + it;
        const uint32_t ph = (uint32_t)(it / STAGES) & 1u;
        if (it >= STAGES && !tc::mbar_wait(&ctl->empty[s], ph ^ 1u, deadline)) {
          ctl->abort = 1;
          break;
        }
        if (ctl->abort) break;
        tc::mbar_arrive_expect_tx(&ctl->full[s], nkb * TILE_BYTES);
        for (int kb = 0; kb < nkb; ++kb)
          tc::tma_load_2d(Ks + ((size_t)s * nkb + kb) * TILE_BYTES, &kmap, g * d + kb * BK,
                          krow0 + c * BM, &ctl->full[s]);
        ++issued;
      }
      if (ctl->abort) {  // drain copies still landing in this CTA's shared memory
        const long long d2 = clock64() + WAIT_CYCLES;
        tc::mbar_wait(&ctl->qfull, 0, d2);
        for (int it = (issued > STAGES ? issued - STAGES : 0); it < issued; ++it)
          if (!tc::mbar_wait(&ctl->full[it % STAGES], (uint32_t)(it / STAGES) & 1u, d2)) break;
      }
    }
    __syncwarp();
  } else if (warp == EPI_WARPS + 1) {  // ---------------- MMA issuer
    if (lane == 0) {
      const uint32_t idesc = tc::idesc_bf16_f32(BM, BM);
      bool ok = tc::mbar_wait(&ctl->qfull, 0, deadline);
      for (int it = 0; ok && it < iters; ++it) {
        const int s = it % STAGES, buf = it & 1;
        if (!tc::mbar_wait(&ctl->full[s], (uint32_t)(it / STAGES) & 1u, deadline) ||
            (it >= 2 && !tc::mbar_wait(&ctl->acce[buf], (uint32_t)((it >> 1) - 1) & 1u, deadline))) {
          ok = false;
          break;
        }
        tc::fence_after_sync();
        const uint32_t dst = tmem + (uint32_t)(buf * BM);
        for (int kb = 0; kb < nkb; ++kb) {
          const uint64_t ad = tc::desc_sw128_kmajor(Qs + kb * TILE_BYTES);
          const uint64_t bd = tc::desc_sw128_kmajor(Ks + ((size_t)s * nkb + kb) * TILE_BYTES);
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk)
            tc::mma_bf16(dst, ad + 2 * kk, bd + 2 * kk, idesc, (kb | kk) != 0);
        }
        tc::mma_commit(&ctl->empty[s]);
        tc::mma_commit(&ctl->accf[buf]);
      }
      if (!ok) ctl->abort = 1;
    }
    __syncwarp();
  } else {  // ---------------- epilogue warps 0..7
    const int quarter = warp & 3, cpart = warp >> 2;  // TMEM lane quarter, 32-column part
    const int r = quarter * 32 + lane;           // tile row == TMEM lane
    const int R = tile * BM + r;                 // packed row
    const bool valid = R < grp * Tb;
    const int j = valid ? R / Tb : 0, t = valid ? R % Tb : 0;
    const int h = g * grp + j;
    const float scale = rsqrtf((float)d);
    const float sg = sigma[(size_t)b * H + h];
    const float sg2 = sg * sg;
    const float* zr = zn2 + ((size_t)b * H + h) * N;
    float* arow = A + (((size_t)b * H + h) * Tmax + t) * N;
    const int kvis = N + t + 1;                  // keys this query may see
    float2* prow = part + ((((size_t)b * Hkv + g) * RQ) + (size_t)tile * BM + r) * nsplit;
    float m = -INFINITY, l = 0.f, rsum = 0.f, M = 0.f, invL = 0.f;
    if (mode == 1 && valid) {  // merge the splits' statistics in a fixed order
      M = -INFINITY;
      for (int q = 0; q < nsplit; ++q) M = fmaxf(M, prow[q].x);
      float L = 0.f;
      for (int q = 0; q < nsplit; ++q) {
        const float2 st = prow[q];
        if (st.x > -INFINITY) L += st.y * expf(st.x - M);
      }
      invL = 1.f / L;
    }
    for (int it = 0; it < iters; ++it) {
      const int buf = it & 1, c = c0 + it;
      bool ok = tc::mbar_wait(&ctl->accf[buf], (uint32_t)(it >> 1) & 1u, deadline);
      ok = __all_sync(FULL, ok && !ctl->abort);
      float v[32];
      if (ok) {
        tc::fence_after_sync();
        const uint32_t ta = tmem + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(buf * BM + cpart * 32);
        tc::tmem_ld32(ta, v);
      }
      tc::fence_before_sync();
      __syncwarp();
      if (lane == 0) mbar_arrive(&ctl->acce[buf]);
      if (!ok) continue;
      const int k0 = c * BM + cpart * 32;
      if (mode == 0) {  // running max / sum over the visible keys
        float mt = -INFINITY;
#pragma unroll
        for (int q = 0; q < 32; ++q) {
          v[q] *= scale;
          if (k0 + q < kvis) mt = fmaxf(mt, v[q]);
        }
        if (mt > -INFINITY) {
          const float mn = fmaxf(m, mt);
          float acc = l * expf(m - mn);
#pragma unroll
          for (int q = 0; q < 32; ++q)
            if (k0 + q < kvis) acc += expf(v[q] - mn);
          l = acc;
          m = mn;
        }
      } else if (valid && k0 < N) {  // normalised visual columns
        const int nv = min(32, N - k0);
        if (nv == 32 && (N & 3) == 0) {
#pragma unroll
          for (int q = 0; q < 32; q += 4) {
            const float4 z = *reinterpret_cast<const float4*>(zr + k0 + q);
            float4 o;
            o.x = expf(v[q] * scale - M) * invL;
            o.y = expf(v[q + 1] * scale - M) * invL;
            o.z = expf(v[q + 2] * scale - M) * invL;
            o.w = expf(v[q + 3] * scale - M) * invL;
            *reinterpret_cast<float4*>(arow + k0 + q) = o;
            rsum = fmaf(o.x, sqrtf(z.x + sg2), rsum);
            rsum = fmaf(o.y, sqrtf(z.y + sg2), rsum);
            rsum = fmaf(o.z, sqrtf(z.z + sg2), rsum);
            rsum = fmaf(o.w, sqrtf(z.w + sg2), rsum);
          }
        } else {
#pragma unroll
          for (int q = 0; q < 32; ++q)  // unrolled: v stays in registers
            if (q < nv) {
              const float p = expf(v[q] * scale - M) * invL;
              arow[k0 + q] = p;
              rsum = fmaf(p, sqrtf(zr[k0 + q] + sg2), rsum);
            }
        }
      }
    }
    if (mode == 0) {  // combine the column parts of every row, in a fixed order
      ctl->stat_m[cpart][r] = m;
      ctl->stat_l[cpart][r] = l;
      epi_barrier();
      if (cpart == 0 && !ctl->abort) {
        float Mc = -INFINITY;
#pragma unroll
        for (int q = 0; q < EPI_PARTS; ++q) Mc = fmaxf(Mc, ctl->stat_m[q][r]);
        float Lc = 0.f;
        if (Mc > -INFINITY) {
#pragma unroll
          for (int q = 0; q < EPI_PARTS; ++q) {
            const float mq = ctl->stat_m[q][r];
            if (mq > -INFINITY) Lc += ctl->stat_l[q][r] * expf(mq - Mc);
          }
        }
        prow[split] = make_float2(Mc, Lc);
      }
    } else {
      ctl->rsum[cpart][r] = rsum;
      epi_barrier();
      if (cpart == 0 && valid && !ctl->abort) {
        float sum = 0.f;
#pragma unroll
        for (int q = 0; q < EPI_PARTS; ++q) sum += ctl->rsum[q][r];
        rs[(((size_t)b * H + h) * nsplit + split) * Tmax + t] = sum;
      }
    }
  }
  if (threadIdx.x == 0 && ctl->abort) set_status(status, GMC_STATUS_TIMEOUT);
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 0) tc::tmem_dealloc(tmem, 256);
}

// Single-launch variant: the key splits of one query tile form a thread-block
// cluster.  Every CTA keeps its split's logits in TMEM (at most FUSED_MAX_TILES
// 128-column tiles), publishes its per-row (max, sum) in shared memory, and
// after one cluster barrier merges all splits' statistics in a fixed order
// (distributed shared memory) before writing A and its part of rs from the
// resident logits.  Same results as the two launches of k_message_tc.
__global__ void __launch_bounds__(FT_THREADS, 1)
    k_message_fused(const __grid_constant__ CUtensorMap qmap, const __grid_constant__ CUtensorMap kmap,
                    const int32_t* toff, int B, int N, int Tmax, int H, int Hkv, int d, int RQ,
                    int kt_per, int nsplit, uint32_t tmem_cols, const float* __restrict__ zn2,
                    const float* __restrict__ sigma, float* A, float* rs, uint32_t* status) {
  grid_dep_wait();
  extern __shared__ uint8_t sm_raw[];
  cg::cluster_group cluster = cg::this_cluster();
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(sm_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const int nkb = d / BK;
  uint8_t* Qs = base;
  uint8_t* Ks = base + (size_t)nkb * TILE_BYTES;
  FusedCtl* ctl = reinterpret_cast<FusedCtl*>(base + fused_region_bytes(nkb));
  // g_h(i) of the CTA's query heads and visual keys, [head - j_lo][key - c0*BM]
  float* gs = reinterpret_cast<float*>(ctl + 1);
  const int gstr = kt_per * BM + 1;  // odd row stride: rows of different heads in distinct banks

  const int b = blockIdx.z / nsplit, split = (int)cluster.block_rank(), g = blockIdx.y,
            tile = blockIdx.x;
  const TextGeom tg = text_geom(toff, b, B, Tmax, status);
  const int grp = H / Hkv;
  if (tg.T == 0 || tile * BM >= grp * tg.T) return;  // uniform over the cluster (same b, tile)
  // cluster barrier phase 1: this CTA has started (its shared memory may be
  // written by the others once every CTA has arrived)
  asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
  const int Tb = tg.T;
  const int nkt = ceil_div(N + Tb, BM);
  const int c0 = split * kt_per, c1 = min(nkt, c0 + kt_per);
  const int iters = max(0, c1 - c0);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int qrow0 = (int)(((size_t)b * Hkv + g) * RQ + (size_t)tile * BM);
  const int krow0 = (int)(2 * ((size_t)b * N + tg.off));

  if (threadIdx.x == 0) {
    tc::mbar_init(&ctl->qfull, 1);
    for (int s = 0; s < STAGES; ++s) {
      tc::mbar_init(&ctl->full[s], 1);
      tc::mbar_init(&ctl->empty[s], 1);
    }
    tc::mbar_init(&ctl->accdone, 1);
    ctl->abort = 0;
    tc::fence_mbar_init();
    tc::prefetch_tmap(&qmap);
    tc::prefetch_tmap(&kmap);
  }
  if (warp == 0) {
    tc::tmem_alloc(&ctl->tmem, tmem_cols);
    tc::tmem_relinquish();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = ctl->tmem;
  const long long deadline = clock64() + WAIT_CYCLES;
  const float c2 = rsqrtf((float)d) * 1.44269504f;  // 1/sqrt(d) in base-2 units (log2 e)
  const int quarter = warp & 3, cq = (warp >> 2) & 3;  // lane quarter, column quarter
  const int r = quarter * 32 + lane;  // tile row == TMEM lane (epilogue warps)
  const int R = tile * BM + r;
  const bool valid = R < grp * Tb;
  const int j = valid ? R / Tb : 0, t = valid ? R % Tb : 0;
  const int h = g * grp + j;
  const int kvis = N + t + 1;

  if (warp == FE_WARPS) {  // ---------------- TMA producer
    int issued = 0;
    if (lane == 0) {
      tc::mbar_arrive_expect_tx(&ctl->qfull, nkb * TILE_BYTES);
      for (int kb = 0; kb < nkb; ++kb)
        tc::tma_load_2d(Qs + kb * TILE_BYTES, &qmap, kb * BK, qrow0, &ctl->qfull);
      for (int it = 0; it < iters; ++it) {
        const int s = it % STAGES;
        const uint32_t ph = (uint32_t)(it / STAGES) & 1u;
        if (it >= STAGES && !tc::mbar_wait(&ctl->empty[s], ph ^ 1u, deadline)) {
          ctl->abort = 1;
          break;
        }
        if (ctl->abort) break;
        tc::mbar_arrive_expect_tx(&ctl->full[s], nkb * TILE_BYTES);
        for (int kb = 0; kb < nkb; ++kb)
          tc::tma_load_2d(Ks + ((size_t)s * nkb + kb) * TILE_BYTES, &kmap, g * d + kb * BK,
                          krow0 + (c0 + it) * BM, &ctl->full[s]);
        ++issued;
      }
      if (ctl->abort) {  // drain copies still landing in this CTA's shared memory
        const long long d2 = clock64() + WAIT_CYCLES;
        tc::mbar_wait(&ctl->qfull, 0, d2);
        for (int it = (issued > STAGES ? issued - STAGES : 0); it < issued; ++it)
          if (!tc::mbar_wait(&ctl->full[it % STAGES], (uint32_t)(it / STAGES) & 1u, d2)) break;
      }
    }
    __syncwarp();
  } else if (warp == FE_WARPS + 1) {  // ---------------- MMA issuer: tile it -> columns it*128
    if (lane == 0) {
      const uint32_t idesc = tc::idesc_bf16_f32(BM, BM);
      bool ok = tc::mbar_wait(&ctl->qfull, 0, deadline);
      for (int it = 0; ok && it < iters; ++it) {
        const int s = it % STAGES;
        if (!tc::mbar_wait(&ctl->full[s], (uint32_t)(it / STAGES) & 1u, deadline)) {
          ok = false;
          break;
        }
        tc::fence_after_sync();
        const uint32_t dst = tmem + (uint32_t)(it * BM);
        for (int kb = 0; kb < nkb; ++kb) {
          const uint64_t ad = tc::desc_sw128_kmajor(Qs + kb * TILE_BYTES);
          const uint64_t bd = tc::desc_sw128_kmajor(Ks + ((size_t)s * nkb + kb) * TILE_BYTES);
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk)
            tc::mma_bf16(dst, ad + 2 * kk, bd + 2 * kk, idesc, (kb | kk) != 0);
        }
        tc::mma_commit(&ctl->empty[s]);
      }
      if (!ok) ctl->abort = 1;
      tc::mma_commit(&ctl->accdone);  // also with no tile or on abort
    }
    __syncwarp();
  }

  asm volatile("barrier.cluster.wait.aligned;" ::: "memory");  // every CTA has started

  // ---- epilogue warps: g_h(i) for the CTA's heads and visual keys (while the
  // MMAs run), then this split's statistics -----------------------------------
  const int j_lo = tile * BM / Tb, j_hi = (min(grp * Tb, tile * BM + BM) - 1) / Tb;
  const int key0 = c0 * BM, nvis = max(0, min(c1 * BM, N) - key0);
  if (warp < FE_WARPS) {
    for (int e = threadIdx.x; e < (j_hi - j_lo + 1) * nvis; e += FE_WARPS * 32) {
      const int jj = e / nvis, kk = e % nvis, hh = g * grp + j_lo + jj;
      const float sg = sigma[(size_t)b * H + hh];
      gs[jj * gstr + kk] = sqrtf(zn2[((size_t)b * H + hh) * N + key0 + kk] + sg * sg);
    }
  }
  bool ok = true;
  float mtile[FUSED_MAX_TILES];  // per 32-column block: the max its exponentials are taken at
  if (warp < FE_WARPS) {
    ok = tc::mbar_wait(&ctl->accdone, 0, deadline);
    ok = __all_sync(FULL, ok && !ctl->abort);
    tc::fence_after_sync();
    float m = -INFINITY, l = 0.f;
#pragma unroll
    for (int it = 0; it < FUSED_MAX_TILES; ++it) {
      mtile[it] = -INFINITY;
      if (!ok || it >= iters) continue;  // uniform over the warp
      float v[32];
      const uint32_t ta = tmem + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(it * BM + cq * 32);
      tc::tmem_ld32(ta, v);
      const int k0 = (c0 + it) * BM + cq * 32;
      float vmax = -INFINITY;
#pragma unroll
      for (int q = 0; q < 32; ++q)
        if (k0 + q < kvis) vmax = fmaxf(vmax, v[q]);
      // exp(x) = 2^(x log2 e): logits s = v / sqrt(d) in base-2 units are
      // v * c2; 2^(v c2 - mt) replaces the logits in TMEM and the write pass
      // rescales it (c2 > 0, so the block max of v c2 is vmax c2)
      const float mt = vmax * c2;
      float lt = 0.f;
#pragma unroll
      for (int q = 0; q < 32; ++q) {
        v[q] = (vmax > -INFINITY && k0 + q < kvis) ? exp2f(fmaf(v[q], c2, -mt)) : 0.f;
        lt += v[q];
      }
      tc::tmem_st32(ta, v);
      if (vmax > -INFINITY) {
        const float mn = fmaxf(m, mt);
        l = l * exp2f(m - mn) + lt * exp2f(mt - mn);
        m = mn;
      }
      mtile[it] = vmax > -INFINITY ? mt : -INFINITY;
    }
    ctl->stat_m[cq][r] = m;
    ctl->stat_l[cq][r] = l;
    fused_epi_barrier();
    if (cq == 0) {  // the four column quarters of the row, in order
      float Mc = -INFINITY;
#pragma unroll
      for (int q = 0; q < 4; ++q) Mc = fmaxf(Mc, ctl->stat_m[q][r]);
      float Lc = 0.f;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float mq = ctl->stat_m[q][r];
        if (mq > -INFINITY) Lc += ctl->stat_l[q][r] * exp2f(mq - Mc);
      }
      for (int q = 0; q < nsplit; ++q) {  // into every CTA of the cluster, this split's slot
        cluster.map_shared_rank(&ctl->all_m[split][0], q)[r] = Mc;
        cluster.map_shared_rank(&ctl->all_l[split][0], q)[r] = Lc;
      }
    }
  }
  cluster.sync();  // every split's statistics are in every CTA (release / acquire)

  if (warp < FE_WARPS) {
    // merge the splits in a fixed order, then the normalised visual columns
    float M = -INFINITY, L = 0.f;
    for (int q = 0; q < nsplit; ++q) M = fmaxf(M, ctl->all_m[q][r]);
    for (int q = 0; q < nsplit; ++q) {
      const float mq = ctl->all_m[q][r];
      if (mq > -INFINITY) L += ctl->all_l[q][r] * exp2f(mq - M);
    }
    const float invL = 1.f / L;
    const float* grow = gs + (valid ? j - j_lo : 0) * gstr;
    float* stg = reinterpret_cast<float*>(base) + warp * 32 * 32;  // the operands are consumed
    float rsum = 0.f;
#pragma unroll
    for (int it = 0; it < FUSED_MAX_TILES; ++it) {
      if (!ok || it >= iters) continue;  // uniform over the warp
      const int k0 = (c0 + it) * BM + cq * 32;
      if (k0 >= N) continue;  // uniform over the warp
      float v[32];
      tc::tmem_ld32(tmem + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(it * BM + cq * 32), v);
      const float f = mtile[it] > -INFINITY ? exp2f(mtile[it] - M) * invL : 0.f;
      const int nv = min(32, N - k0), kk0 = k0 - key0;
#pragma unroll
      for (int q = 0; q < 32; ++q) {
        v[q] *= f;
        if (q < nv) rsum = fmaf(v[q], grow[kk0 + q], rsum);
      }
      // transpose through shared memory: row = lane going in, eight lanes per
      // 128-byte row segment going out (16-byte chunks XOR-swizzled by row)
#pragma unroll
      for (int c4 = 0; c4 < 8; ++c4)
        *reinterpret_cast<float4*>(stg + lane * 32 + ((c4 ^ (lane & 7)) << 2)) =
            make_float4(v[4 * c4], v[4 * c4 + 1], v[4 * c4 + 2], v[4 * c4 + 3]);
      __syncwarp();
      const int c4 = lane & 7, col = k0 + 4 * c4;
#pragma unroll
      for (int rr = 0; rr < 32; rr += 4) {
        const int row = rr + (lane >> 3);
        const float4 o = *reinterpret_cast<const float4*>(stg + row * 32 + ((c4 ^ (row & 7)) << 2));
        const int Rw = tile * BM + quarter * 32 + row;
        if (Rw >= grp * Tb || col >= N) continue;
        float* arow = A + (((size_t)b * H + g * grp + Rw / Tb) * Tmax + Rw % Tb) * N;
        if ((N & 3) == 0 && col + 4 <= N) {
          *reinterpret_cast<float4*>(arow + col) = o;
        } else {
          arow[col] = o.x;
          if (col + 1 < N) arow[col + 1] = o.y;
          if (col + 2 < N) arow[col + 2] = o.z;
          if (col + 3 < N) arow[col + 3] = o.w;
        }
      }
      __syncwarp();  // the next block reuses the staging tile
    }
    ctl->rsum[cq][r] = rsum;
    fused_epi_barrier();
    if (cq == 0 && valid && ok)
      rs[(((size_t)b * H + h) * nsplit + split) * Tmax + t] =
          ((ctl->rsum[0][r] + ctl->rsum[1][r]) + ctl->rsum[2][r]) + ctl->rsum[3][r];
  }
  if (threadIdx.x == 0 && ctl->abort) set_status(status, GMC_STATUS_TIMEOUT);
  // no CTA touches another's shared memory after the cluster barrier
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 0) tc::tmem_dealloc(tmem, tmem_cols);
}

bool message_tc_supported(const Dims& dm) {
  return dm.dtype == GMC_BF16 && dm.N >= BM && (dm.d == 64 || dm.d == 128);
}

int message_rq(const Dims& dm) { return ceil_div((dm.H / dm.Hkv) * dm.T, BM) * BM; }

int message_splits(const Dims& dm) {
  return message_tc_supported(dm) ? msg_split(dm.B, dm.Hkv, message_rq(dm), dm.N, dm.T).n : 1;
}

// The packed queries Qp are written by the probe kernel, launched before this
// one on the same stream (k_prep.cu).
cudaError_t launch_message_tc(const Dims& dm, const void* keys, const void* queries, Scratch& s,
                              cudaStream_t st, int* launches) {
  (void)queries;
  if (launches) *launches = 1;
  const int RQ = message_rq(dm);
  cudaError_t e;
  CUtensorMap qmap, kmap;
  if ((e = make_tmap_bf16(&qmap, s.Qp, dm.d, (uint64_t)dm.B * dm.Hkv * RQ, dm.d, BM)) != cudaSuccess)
    return e;
  // keys of every image, addressed from the buffer start; the declared row
  // count is an upper bound, every box read lies inside the image's K block or
  // the V block that follows it.
  if ((e = make_tmap_bf16(&kmap, keys, (uint64_t)dm.Hkv * dm.d,
                          2ull * dm.B * (uint64_t)(dm.N + dm.T), (uint64_t)dm.Hkv * dm.d, BM)) !=
      cudaSuccess)
    return e;
  const int nkb = dm.d / BK;
  const size_t smem = msg_smem_bytes(nkb);
  if ((e = set_smem_limit((const void*)k_message_tc, smem)) != cudaSuccess) return e;
  const MsgSplit sp = msg_split(dm.B, dm.Hkv, RQ, dm.N, dm.T);
  dim3 grid(RQ / BM, dm.Hkv, dm.B * sp.n);
  const size_t fsmem = 1024 + fused_region_bytes(nkb) + sizeof(FusedCtl) +
                       sizeof(float) * (size_t)(dm.H / dm.Hkv) * (sp.kt_per * BM + 1);
  if (sp.kt_per <= FUSED_MAX_TILES && sp.n <= FUSED_MAX_CLUSTER && fsmem <= 227 * 1024) {
    uint32_t cols = 32;
    while (cols < (uint32_t)(sp.kt_per * BM)) cols *= 2;
    if ((e = set_smem_limit((const void*)k_message_fused, fsmem)) != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = dim3(FT_THREADS);
    cfg.dynamicSmemBytes = fsmem;
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 1;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = sp.n;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int ncl = 0;
    if (cudaOccupancyMaxActiveClusters(&ncl, (void*)k_message_fused, &cfg) == cudaSuccess && ncl > 0) {
      attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;  // see grid_dep_wait
      attr[1].val.programmaticStreamSerializationAllowed = 1;
      cfg.numAttrs = 2;
      return cudaLaunchKernelEx(&cfg, k_message_fused, qmap, kmap, dm.toff, dm.B, dm.N, dm.T, dm.H,
                                dm.Hkv, dm.d, RQ, sp.kt_per, sp.n, cols, (const float*)s.zn2,
                                (const float*)s.sigma, s.A, s.rs, s.status);
    }
    cudaGetLastError();  // no co-resident cluster: the two launches below
  }
  if (launches) *launches = 2;
  for (int mode = 0; mode < 2; ++mode) {
    launch_k(k_message_tc, grid, THREADS, smem, st, 1, qmap, kmap, dm.toff, dm.B, dm.N, dm.T, dm.H, dm.Hkv,
                                              dm.d, RQ, mode, sp.kt_per, sp.n, s.mpart, s.zn2,
                                              s.sigma, s.A, s.rs, s.status);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace gmc
