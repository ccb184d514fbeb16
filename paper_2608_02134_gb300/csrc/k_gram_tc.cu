// Cosine matrix of the boundary states on the tcgen05 tensor cores (bf16 path).
//
// cos_ij = (h_i . h_j) / (n_i n_j): the appearance clients of appendix Eq.
// (cond-aux-clients) and the assignment cosines of Eq. (cond-assignment).  The
// Gram runs on the raw bf16 states with fp32 accumulation in tensor memory and
// is normalised afterwards in fp32 (the states are never rounded after
// normalisation).
//
// A cluster of two CTAs computes one 128 x 128 tile of the upper triangle
// (I <= J) and writes it and its mirror; the CTAs split the contraction over
// D in two halves (one SM streams half the operand bytes, twice as many SMs
// work).  In each CTA warp 0 / lane 0 streams 64-wide K slices of both row
// blocks with TMA (128-byte swizzle) through a 6-stage mbarrier ring; warp 1 /
// lane 0 issues tcgen05.mma (M = N = 128, K = 16) into a 128-column TMEM
// accumulator; warps 2 and 3 stage the tile's reciprocal row and column norms.
// Then each CTA parks the column half its peer finishes in its own shared
// memory, and finishes its half with the peer's partial read over distributed
// shared memory: one fp32 addition of two partials, the same value in both
// orders.  The epilogue runs on all 16 warps: warp w reads TMEM lane quarter
// w % 4 and 16 of the half's 64 columns.  The last, ragged tile of an image is shifted inward (start
// N - 128) so every TMA box lies inside the image's own rows; it stores only
// the rows and columns the previous tile does not own.
#include <cooperative_groups.h>

#include "common.cuh"
#include "kernels.cuh"
#include "tc.cuh"

namespace cg = cooperative_groups;

namespace gmc {

namespace {
constexpr int BM = 128, BK = 64, STAGES = 6;
constexpr int GRAM_THREADS = 512;  // 16 warps: 4 TMEM lane quarters x 4 column groups
constexpr int TILE_BYTES = BM * BK * 2;  // 16 KiB per operand per stage
constexpr long long WAIT_CYCLES = 4000000000LL;  // about two seconds

struct GramCtl {
  uint64_t full[STAGES];
  uint64_t empty[STAGES];
  uint64_t done;
  uint32_t tmem;
  volatile int abort;
  float rnr[BM];  // reciprocal norms of the tile's rows
  float rnc[BM];  // and of its columns
};

constexpr size_t GRAM_SMEM = 1024 + 2 * STAGES * TILE_BYTES + sizeof(GramCtl);
}  // namespace

__global__ void __launch_bounds__(GRAM_THREADS, 1)
    k_gram_tc(const __grid_constant__ CUtensorMap tmap, const int32_t* toff, int B, int N,
              int Tmax, int D, const float* __restrict__ rn, float* cos, uint32_t* status) {
  grid_dep_wait();
  extern __shared__ uint8_t sm_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(sm_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* tilesA = base;
  uint8_t* tilesB = base + STAGES * TILE_BYTES;
  GramCtl* ctl = reinterpret_cast<GramCtl*>(base + 2 * STAGES * TILE_BYTES);

  cg::cluster_group cluster = cg::this_cluster();
  const int kpart = (int)cluster.block_rank();  // 0 or 1: which half of the contraction
  const int b = blockIdx.y;
  const TextGeom tg = text_geom(toff, b, B, Tmax, status);
  if (tg.T == 0) return;  // uniform over the cluster
  const int nt = ceil_div(N, BM);
  int t = blockIdx.x >> 1, I = 0;
  while (t >= nt - I) {
    t -= nt - I;
    ++I;
  }
  const int J = I + t;
  const int r0 = min(I * BM, N - BM), c0 = min(J * BM, N - BM);
  const int row_base = (int)((size_t)b * N + tg.off);  // first visual row of the image
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nk_all = ceil_div(D, BK), kh = (nk_all + 1) / 2;
  const int kb0 = kpart * kh, nk = max(0, min(nk_all, kb0 + kh) - kb0);  // this CTA's K slices

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      tc::mbar_init(&ctl->full[s], 1);
      tc::mbar_init(&ctl->empty[s], 1);
    }
    tc::mbar_init(&ctl->done, 1);
    ctl->abort = 0;
    tc::fence_mbar_init();
    tc::prefetch_tmap(&tmap);
  }
  if (warp == 0) {
    tc::tmem_alloc(&ctl->tmem, 128);
    tc::tmem_relinquish();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = ctl->tmem;
  const long long deadline = clock64() + WAIT_CYCLES;
  int issued = 0;  // producer: stages loaded

  if (warp == 0) {
    if (lane == 0) {
      for (int kb = 0; kb < nk; ++kb) {
        const int s = kb % STAGES;
        const uint32_t ph = (uint32_t)(kb / STAGES) & 1u;
        if (kb >= STAGES && !tc::mbar_wait(&ctl->empty[s], ph ^ 1u, deadline)) {
          ctl->abort = 1;
          break;
        }
        if (ctl->abort) break;
        tc::mbar_arrive_expect_tx(&ctl->full[s], 2 * TILE_BYTES);
        tc::tma_load_2d(tilesA + s * TILE_BYTES, &tmap, (kb0 + kb) * BK, row_base + r0, &ctl->full[s]);
        tc::tma_load_2d(tilesB + s * TILE_BYTES, &tmap, (kb0 + kb) * BK, row_base + c0, &ctl->full[s]);
        ++issued;
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = tc::idesc_bf16_f32(BM, BM);
      for (int kb = 0; kb < nk; ++kb) {
        const int s = kb % STAGES;
        const uint32_t ph = (uint32_t)(kb / STAGES) & 1u;
        if (!tc::mbar_wait(&ctl->full[s], ph, deadline)) {
          ctl->abort = 1;
          break;
        }
        tc::fence_after_sync();
        const uint64_t ad = tc::desc_sw128_kmajor(tilesA + s * TILE_BYTES);
        const uint64_t bd = tc::desc_sw128_kmajor(tilesB + s * TILE_BYTES);
#pragma unroll
        for (int kk = 0; kk < BK / 16; ++kk)
          tc::mma_bf16(tmem, ad + 2 * kk, bd + 2 * kk, idesc, (kb | kk) != 0);
        tc::mma_commit(&ctl->empty[s]);
      }
      tc::mma_commit(&ctl->done);  // also on abort, so the epilogue wakes up
    }
    __syncwarp();
  } else if (warp < 4) {
    // reciprocal norms of the tile's rows (warp 2) and columns (warp 3)
    const int o = warp == 2 ? r0 : c0;
    float* dst = warp == 2 ? ctl->rnr : ctl->rnc;
    for (int q = lane; q < BM; q += 32) dst[q] = rn[(size_t)b * N + o + q];
  }

  bool ok = tc::mbar_wait(&ctl->done, 0, deadline) && !ctl->abort;
  ok = __syncthreads_and(ok);  // also publishes the norms
  tc::fence_after_sync();
  const int quarter = warp & 3, grp = warp >> 2;
  const int row = quarter * 32 + lane;  // this thread's TMEM lane = tile row
  // the column half the peer finishes, column-major [64][128] in the (now idle)
  // operand ring; a CTA without K slices contributes zeros
  float* park = reinterpret_cast<float*>(tilesA);
  const uint32_t trow = tmem + ((uint32_t)(quarter * 32) << 16);
  if (ok) {
    float v[16];
    if (nk > 0) {
      tc::tmem_ld16(trow + (uint32_t)((1 - kpart) * 64 + grp * 16), v);
    } else {
#pragma unroll
      for (int q = 0; q < 16; ++q) v[q] = 0.f;
    }
#pragma unroll
    for (int q = 0; q < 16; ++q) park[(grp * 16 + q) * BM + row] = v[q];
  }
  tc::fence_before_sync();
  cluster.sync();  // both parked halves are complete
  tc::fence_after_sync();
  if (ok) {
    const float* peer = cluster.map_shared_rank(park, 1 - kpart);
    const int i = r0 + row;  // output row
    const bool own_row = i >= I * BM;
    const float ri = ctl->rnr[row];
    float v[16];
    if (nk > 0) {
      tc::tmem_ld16(trow + (uint32_t)(kpart * 64 + grp * 16), v);
    } else {
#pragma unroll
      for (int q = 0; q < 16; ++q) v[q] = 0.f;
    }
    const int jl = kpart * 64 + grp * 16;  // first column of this warp, within the tile
    const int j0 = c0 + jl;
#pragma unroll
    for (int q = 0; q < 16; ++q)
      v[q] = (v[q] + peer[(grp * 16 + q) * BM + row]) * ri * ctl->rnc[jl + q];
    // own rows: the warp's 32 x 16 block goes through shared memory (padded
    // rows), then every store instruction writes two 64-byte row segments
    float* st = reinterpret_cast<float*>(tilesB) + warp * (32 * 17);
#pragma unroll
    for (int q = 0; q < 16; ++q) st[lane * 17 + q] = v[q];
    __syncwarp();
#pragma unroll 4
    for (int k = 0; k < 16; ++k) {
      const int rr = 2 * k + (lane >> 4), cq = lane & 15;  // block row, column
      const int ii = r0 + quarter * 32 + rr, jj = j0 + cq;
      if (ii >= I * BM && jj >= J * BM) cos[((size_t)b * N + ii) * N + jj] = st[rr * 17 + cq];
    }
    if (I != J) {  // mirror: row j of the transposed block, coalesced over the warp's lanes
#pragma unroll
      for (int q = 0; q < 16; ++q) {
        const int j = j0 + q;
        if (own_row && j >= J * BM) cos[((size_t)b * N + j) * N + i] = v[q];
      }
    }
  }
  cluster.sync();  // the peer has read this CTA's parked half
  if (!ok && threadIdx.x == 0) set_status(status, GMC_STATUS_TIMEOUT);
  if (warp == 0 && lane == 0 && !ok) {
    // drain TMA copies still in flight into this CTA's shared memory
    const long long d2 = clock64() + WAIT_CYCLES;
    for (int kb = (issued > STAGES ? issued - STAGES : 0); kb < issued; ++kb)
      if (!tc::mbar_wait(&ctl->full[kb % STAGES], (uint32_t)(kb / STAGES) & 1u, d2)) break;
  }
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 0) tc::tmem_dealloc(tmem, 128);
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

// 2-D bf16 tensor map: rows of `row_elems` elements, `rows` rows, row pitch
// `pitch_elems`; box = 64 elements x `box_rows` rows, 128-byte swizzle.
cudaError_t make_tmap_bf16(CUtensorMap* map, const void* base, uint64_t row_elems, uint64_t rows,
                           uint64_t pitch_elems, uint32_t box_rows) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return cudaErrorNotSupported;
  const cuuint64_t dims[2] = {row_elems, rows};
  const cuuint64_t strides[1] = {pitch_elems * 2};
  const cuuint32_t box[2] = {64, box_rows};
  const cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

bool gram_tc_supported(const Dims& dm) {
  return dm.dtype == GMC_BF16 && dm.N >= BM && dm.D >= BK;
}

cudaError_t launch_gram_tc(const Dims& dm, const void* hidden, Scratch& s, cudaStream_t st) {
  CUtensorMap map;
  // Rows of every image are addressed from the buffer start; the declared row
  // count is an upper bound (B * (N + T)), every box read lies inside the
  // image's visual rows.
  cudaError_t e = make_tmap_bf16(&map, hidden, (uint64_t)dm.D,
                                 (uint64_t)dm.B * (uint64_t)(dm.N + dm.T), (uint64_t)dm.D, BM);
  if (e != cudaSuccess) return e;
  if ((e = set_smem_limit((const void*)k_gram_tc, GRAM_SMEM)) != cudaSuccess) return e;
  const int nt = ceil_div(dm.N, BM);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * (nt * (nt + 1) / 2), dm.B);
  cfg.blockDim = dim3(GRAM_THREADS);
  cfg.dynamicSmemBytes = GRAM_SMEM;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;  // see grid_dep_wait
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, k_gram_tc, map, dm.toff, dm.B, dm.N, dm.T, dm.D,
                            (const float*)s.rn, s.cos, s.status);
}

}  // namespace gmc
