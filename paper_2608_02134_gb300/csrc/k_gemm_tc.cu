// General C = diag(r) (A B^T) diag(c) on the tcgen05 tensor cores (bf16 operands,
// fp32 accumulation in tensor memory, fp32 output): the dense contractions of
// the long-prefix path.
//
//   * the fixed rank-r Rademacher projection of the boundary states, y_i = R h_i
//     (A = visual hidden rows, B = R, no scaling);
//   * the bounded appearance bank's cosines x~_{c(m)} . x~_i over the projected
//     unit states (A, B = the states split into bf16 hi/lo terms, laid out so
//     one product over 3r columns sums hi.hi + hi.lo + lo.hi);
//   * the support cosines of the assignment, cos(h_{S_k}, h_i), as K x N rows
//     (A = the selected rows gathered, B = the visual hidden rows, scaled by
//     the reciprocal norms of both).
//   * the cosine Gram of the boundary states for large or batched problems
//     (symmetric mode: A = B = the visual rows, scaled by their reciprocal
//     norms; only tiles on or above the diagonal are computed).
// (Appendix "Appearance and spatial clients", last paragraph; the cost notes
// after Algorithm 1: the bounded bank and the chunked N x K assignment product;
// Eq. (cond-aux-clients), (cond-assignment) for the cosines.)
//
// One CTA computes one 128 x BN output tile (BN = 128 or 256, one TMEM column
// per output column).  Warp 0 / lane 0 streams 64-wide K slices of the A and B
// row blocks with TMA (128-byte swizzle) through an mbarrier ring of ST stages
// (4; 2 when the grid holds more tiles than SMs: two CTAs then share an SM and
// one's epilogue overlaps the other's products); warp
// 1 / lane 0 issues tcgen05.mma (M = 128, N = BN, K = 16).  Then all 8 warps
// drain TMEM: warp w reads lane quarter w % 4 and half w / 4 of the columns in
// 32-column chunks, applies the row and column scales and stores each chunk
// through a padded 32 x 32 shared-memory transpose, so every store
// instruction writes one 128-byte row segment.  Ragged edges: TMA fills K
// columns past the operands' extents with zeros.  The last row block of an
// operand with at least one full tile of rows is shifted inward (start M - 128,
// likewise Nn - BN) so every box lies inside the image's own rows -- the
// hidden states' visual rows are followed by text rows whose count only the
// device knows -- and stores only the rows and columns the previous tile does
// not own; a smaller operand reads zeros past its declared rows.  Symmetric
// mode (M == Nn, A and B the same rows): the grid enumerates the tiles that
// hold an entry with j >= i; a tile stores its own entries and, from
// registers (coalesced over the lanes), the mirror C[j][i] of each entry
// j > i whose own tile is not computed -- every entry is written exactly
// once, so the result does not depend on the order of the stores.  Every
// mbarrier wait is bounded (about two seconds); on timeout the kernel records
// GMC_STATUS_TIMEOUT, drains its copies and frees its tensor memory.
#include "common.cuh"
#include "kernels.cuh"
#include "tc.cuh"

namespace gmc {

namespace {
constexpr int GM = 128, GK = 64, GSTAGES = 4;  // ring stages: at most GSTAGES
constexpr int G_THREADS = 256;
constexpr int GA_BYTES = GM * GK * 2;  // 16 KiB per stage
constexpr long long G_WAIT = 4000000000LL;

struct GemmCtl {
  uint64_t full[GSTAGES];
  uint64_t empty[GSTAGES];
  uint64_t done;
  uint32_t tmem;
  volatile int abort;
};

// Symmetric mode: tile (I, J) (rows 128 I.., columns BN J..) is computed when it
// holds an entry with j >= i.
template <int BN> __host__ __device__ __forceinline__ bool sym_tile(int I, int J) {
  return BN * J + BN - 1 >= GM * I;
}
template <int BN> __host__ __device__ __forceinline__ int sym_first_col(int I) {
  const int x = GM * I - (BN - 1);
  return x <= 0 ? 0 : (x + BN - 1) / BN;
}

template <int BN, int ST> constexpr size_t gemm_smem() {
  return 1024 + (size_t)ST * (GA_BYTES + BN * GK * 2) + sizeof(GemmCtl) + sizeof(float) * (GM + BN);
}
}  // namespace

template <int BN, int ST>
__global__ void __launch_bounds__(G_THREADS, ST == 2 ? 2 : 1)
    k_gemm_tc(const __grid_constant__ CUtensorMap amap, const __grid_constant__ CUtensorMap bmap,
              GemmArgs g) {
  grid_dep_wait();
  constexpr int B_BYTES = BN * GK * 2;
  extern __shared__ uint8_t sm_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(sm_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* tilesA = base;
  uint8_t* tilesB = base + ST * GA_BYTES;
  GemmCtl* ctl = reinterpret_cast<GemmCtl*>(base + ST * (GA_BYTES + B_BYTES));
  float* rs = reinterpret_cast<float*>(ctl + 1);  // [GM] row scales of the tile
  float* cs = rs + GM;                            // [BN] column scales

  const int b = blockIdx.z;
  // consecutive CTAs share a B tile (m_fast: the larger operand is B and stays
  // in L2 while the A tiles stream past it) or an A tile
  int tI = g.m_fast ? blockIdx.x : blockIdx.y, tJ = g.m_fast ? blockIdx.y : blockIdx.x;
  if (g.sym) {  // blockIdx.x enumerates the computed tiles, row block by row block
    const int nJ = ceil_div(g.Nn, BN);
    int t = blockIdx.x;
    tI = 0;
    while (t >= nJ - sym_first_col<BN>(tI)) {
      t -= nJ - sym_first_col<BN>(tI);
      ++tI;
    }
    tJ = sym_first_col<BN>(tI) + t;
  }
  const int n0 = tJ * BN, m0 = tI * GM;
  // the tile as loaded: shifted inward at the ragged end
  const int ml = g.M >= GM ? min(m0, g.M - GM) : m0;
  const int nl = g.Nn >= BN ? min(n0, g.Nn - BN) : n0;
  int arow = (int)((long long)b * g.a_img), brow = (int)((long long)b * g.b_img);
  if (g.a_text || g.b_text) {
    const TextGeom tg = text_geom(g.toff, b, g.B, g.Tmax, g.status);
    if (tg.T == 0) return;  // uniform over the block
    if (g.a_text) arow += tg.off;
    if (g.b_text) brow += tg.off;
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nk = ceil_div(g.Kd, GK);

  if (threadIdx.x == 0) {
    for (int s = 0; s < ST; ++s) {
      tc::mbar_init(&ctl->full[s], 1);
      tc::mbar_init(&ctl->empty[s], 1);
    }
    tc::mbar_init(&ctl->done, 1);
    ctl->abort = 0;
    tc::fence_mbar_init();
    tc::prefetch_tmap(&amap);
    tc::prefetch_tmap(&bmap);
  }
  if (warp == 0) {
    tc::tmem_alloc(&ctl->tmem, BN);
    tc::tmem_relinquish();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = ctl->tmem;
  const long long deadline = clock64() + G_WAIT;
  int issued = 0;

  if (warp == 0) {
    if (lane == 0) {
      for (int kb = 0; kb < nk; ++kb) {
        const int s = kb % ST;
        const uint32_t ph = (uint32_t)(kb / ST) & 1u;
        if (kb >= ST && !tc::mbar_wait(&ctl->empty[s], ph ^ 1u, deadline)) {
          ctl->abort = 1;
          break;
        }
        if (ctl->abort) break;
        tc::mbar_arrive_expect_tx(&ctl->full[s], GA_BYTES + B_BYTES);
        tc::tma_load_2d(tilesA + s * GA_BYTES, &amap, kb * GK, arow + ml, &ctl->full[s]);
        tc::tma_load_2d(tilesB + s * B_BYTES, &bmap, kb * GK, brow + nl, &ctl->full[s]);
        ++issued;
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = tc::idesc_bf16_f32(GM, BN);
      for (int kb = 0; kb < nk; ++kb) {
        const int s = kb % ST;
        const uint32_t ph = (uint32_t)(kb / ST) & 1u;
        if (!tc::mbar_wait(&ctl->full[s], ph, deadline)) {
          ctl->abort = 1;
          break;
        }
        tc::fence_after_sync();
        const uint64_t ad = tc::desc_sw128_kmajor(tilesA + s * GA_BYTES);
        const uint64_t bd = tc::desc_sw128_kmajor(tilesB + s * B_BYTES);
#pragma unroll
        for (int kk = 0; kk < GK / 16; ++kk)
          tc::mma_bf16(tmem, ad + 2 * kk, bd + 2 * kk, idesc, (kb | kk) != 0);
        tc::mma_commit(&ctl->empty[s]);
      }
      tc::mma_commit(&ctl->done);  // also on abort, so the epilogue wakes up
    }
    __syncwarp();
  } else {
    // scales of the tile's rows and columns (1 where none is given)
    for (int q = threadIdx.x - 64; q < GM + BN; q += G_THREADS - 64) {
      float v = 1.f;
      if (q < GM) {
        const int m = ml + q;
        if (g.rscale && m < g.M) v = g.rscale[(size_t)b * g.M + m];
        rs[q] = v;
      } else {
        const int n = nl + q - GM;
        if (g.cscale && n < g.Nn) v = g.cscale[(size_t)b * g.Nn + n];
        cs[q - GM] = v;
      }
    }
  }

  bool ok = tc::mbar_wait(&ctl->done, 0, deadline) && !ctl->abort;
  ok = __syncthreads_and(ok);  // also publishes the scales
  tc::fence_after_sync();
  if (ok && nk > 0) {
    const int quarter = warp & 3, half = warp >> 2;
    const int row = quarter * 32 + lane;  // this thread's TMEM lane = tile row
    const float r = rs[row];
    // the operand ring is idle now: a padded 32 x 33 staging block per warp
    float* st = reinterpret_cast<float*>(tilesA) + warp * (32 * 33);
    const uint32_t trow = tmem + ((uint32_t)(quarter * 32) << 16);
    float* Cimg = g.C + (size_t)b * g.c_img;
#pragma unroll 1
    for (int c = 0; c < BN / 64; ++c) {
      const int cl = half * (BN / 2) + c * 32;  // first column of the chunk, within the tile
      float v[32];
      tc::tmem_ld32(trow + (uint32_t)cl, v);
#pragma unroll
      for (int q = 0; q < 32; ++q) {
        v[q] *= r * cs[cl + q];
        st[lane * 33 + q] = v[q];
      }
      if (g.sym) {  // mirrors of owned entries j > i whose own tile is not computed
        const int i = ml + row;
        const bool own_i = i >= m0 && i < g.M;
#pragma unroll  // fully: v stays in registers
        for (int q = 0; q < 32; ++q) {
          const int j = nl + cl + q;
          if (own_i && j >= n0 && j < g.Nn && j > i && !sym_tile<BN>(j / GM, i / BN))
            Cimg[(size_t)j * g.ldc + i] = v[q];
        }
      }
      __syncwarp();
      const int col = nl + cl + lane;
      const bool col_ok = col >= n0 && col < g.Nn;  // owned by this tile
#pragma unroll 4
      for (int rr = 0; rr < 32; ++rr) {
        const int m = ml + quarter * 32 + rr;
        if (m >= m0 && m < g.M && col_ok) Cimg[(size_t)m * g.ldc + col] = st[rr * 33 + lane];
      }
      __syncwarp();
    }
  }
  if (!ok && threadIdx.x == 0) set_status(g.status, GMC_STATUS_TIMEOUT);
  if (warp == 0 && lane == 0 && !ok) {
    // drain TMA copies still in flight into this CTA's shared memory
    const long long d2 = clock64() + G_WAIT;
    for (int kb = (issued > ST ? issued - ST : 0); kb < issued; ++kb)
      if (!tc::mbar_wait(&ctl->full[kb % ST], (uint32_t)(kb / ST) & 1u, d2)) break;
  }
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 0) tc::tmem_dealloc(tmem, BN);
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
template <int BN, int ST>
static cudaError_t launch_gemm_st(const CUtensorMap& am, const CUtensorMap& bm, const GemmArgs& g,
                                  dim3 grid, cudaStream_t st) {
  const size_t smem = gemm_smem<BN, ST>();
  cudaError_t e;
  if ((e = set_smem_limit((const void*)k_gemm_tc<BN, ST>, smem)) != cudaSuccess) return e;
  launch_k(k_gemm_tc<BN, ST>, grid, G_THREADS, smem, st, 1, am, bm, g);
  return cudaGetLastError();
}

template <int BN>
static cudaError_t launch_gemm_bn(const GemmArgs& g, const void* A, long long a_rows, int lda,
                                  const void* Bm, long long b_rows, int ldb, cudaStream_t st) {
  CUtensorMap am, bm;
  cudaError_t e = make_tmap_bf16(&am, A, (uint64_t)g.Kd, (uint64_t)a_rows, (uint64_t)lda, GM);
  if (e != cudaSuccess) return e;
  if ((e = make_tmap_bf16(&bm, Bm, (uint64_t)g.Kd, (uint64_t)b_rows, (uint64_t)ldb, BN)) !=
      cudaSuccess)
    return e;
  dim3 grid(ceil_div(g.Nn, BN), ceil_div(g.M, GM), g.B);
  if (g.m_fast) grid = dim3(ceil_div(g.M, GM), ceil_div(g.Nn, BN), g.B);
  if (g.sym) grid = dim3(gemm_sym_ctas(g.M, 1), 1, g.B);  // the computed tiles of every image
  static int sms = 0;
  if (sms == 0 && cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, 0) != cudaSuccess) {
    cudaGetLastError();
    sms = 152;
  }
  // more tiles than SMs: two CTAs per SM with two stages each
  if ((long long)grid.x * grid.y * grid.z > sms) return launch_gemm_st<BN, 2>(am, bm, g, grid, st);
  return launch_gemm_st<BN, GSTAGES>(am, bm, g, grid, st);
}

int gemm_sym_ctas(int N, int B) {  // symmetric Grams use 128 x 256 tiles (N > 128)
  int nt = 0;
  for (int I = 0; I < ceil_div(N, GM); ++I) nt += ceil_div(N, 256) - sym_first_col<256>(I);
  return nt * B;
}

cudaError_t launch_gemm_tc(const GemmArgs& g, const void* A, long long a_rows, int lda,
                           const void* Bm, long long b_rows, int ldb, cudaStream_t st) {
  if (g.M < 1 || g.Nn < 1 || g.Kd < 1 || g.B < 1) return cudaErrorInvalidValue;
  if (g.sym && (g.M != g.Nn || g.Nn <= 128 || g.m_fast)) return cudaErrorInvalidValue;
  // an operand addressed from the hidden states (a_text / b_text) must hold a
  // full box of rows, so the shifted last box stays inside the image's visual
  // rows (the buffer may end right after the last image's text rows)
  if ((g.a_text && g.M < GM) || (g.b_text && g.Nn < (g.Nn <= 128 ? 128 : 256)))
    return cudaErrorInvalidValue;
  if (g.Nn <= 128) return launch_gemm_bn<128>(g, A, a_rows, lda, Bm, b_rows, ldb, st);
  return launch_gemm_bn<256>(g, A, a_rows, lda, Bm, b_rows, ldb, st);
}

}  // namespace gmc
