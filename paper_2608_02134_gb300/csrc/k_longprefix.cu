// Long prefixes: the bounded appearance bank (appendix "Appearance and spatial
// clients", last paragraph; the cost notes after Algorithm 1; Table "Shared GMC
// configuration", long-prefix row: rank 128, M_V <= 4096, b = 512).
//
// The appearance states are the boundary states under a fixed rank-r
// Rademacher map R, normalised: x~_i = R h_i / max(||R h_i||, eps) (the product
// R h_i runs on the tensor cores, k_gemm_tc.cu).  The appearance clients are
// the M_V = min(N, 4096) uniformly spaced tokens c(m) = floor(m N / M_V); row
// m of the bank is softmax_i(x~_{c(m)} . x~_i / tau_v), beta_V / M_V each.
//
// k_lp_norm turns y_i = R h_i into the operands of that cosine product.  A
// unit state in fp32 is split exactly into bf16 terms x = hi + lo + e with
// hi = bf16(x), lo = bf16(x - hi) and |e| <= 2^-17 |x|; the rows
//   Xa_i = [hi_i | hi_i | lo_i],  Xb_i = [hi_i | lo_i | hi_i]   (3r columns)
// give Xa_c . Xb_i = hi.hi + hi.lo + lo.hi, which is x~_c . x~_i up to the lo.lo
// and e terms (about 2^-16 of |x~_c||x~_i| at worst, far below a bf16 product
// of the unsplit states): the bf16 tensor cores compute the projected cosines
// to nearly fp32 accuracy.  XaC holds Xa at the client tokens.
//
// k_gather_support copies the selected rows of the boundary states (and their
// reciprocal norms) into a dense [K][D] block, the second operand of the N x K
// support-cosine product of the assignment (Eq. (cond-assignment) needs
// cos(h_i, h_j) for j in S only).
#include "common.cuh"
#include "kernels.cuh"

namespace gmc {

__global__ void __launch_bounds__(256) k_lp_norm(const float* __restrict__ Y, int B, int N, int r,
                                                 int MV, float norm_eps, __nv_bfloat16* Xa,
                                                 __nv_bfloat16* Xb, __nv_bfloat16* XaC) {
  grid_dep_wait();
  const int b = blockIdx.y;
  const int lane = threadIdx.x & 31;
  const int i = blockIdx.x * 8 + (threadIdx.x >> 5);
  if (i >= N) return;
  const float* y = Y + ((size_t)b * N + i) * r;
  float ss = 0.f;
  for (int k = lane; k < r; k += 32) ss = fmaf(y[k], y[k], ss);
  ss = warp_sum(ss);
  const float inv = 1.f / fmaxf(sqrtf(ss), norm_eps);
  // client slot of this token: m = ceil(i M_V / N) when floor(m N / M_V) == i
  const long long mq = ((long long)i * MV + N - 1) / N;
  const bool client = mq < MV && (mq * N) / MV == i;
  const size_t w = 3 * (size_t)r;
  __nv_bfloat16* a = Xa + ((size_t)b * N + i) * w;
  __nv_bfloat16* bb = Xb + ((size_t)b * N + i) * w;
  __nv_bfloat16* c = client ? XaC + ((size_t)b * MV + mq) * w : nullptr;
  for (int k = lane; k < r; k += 32) {
    const float x = y[k] * inv;
    const __nv_bfloat16 hi = __float2bfloat16_rn(x);
    const __nv_bfloat16 lo = __float2bfloat16_rn(x - __bfloat162float(hi));
    a[k] = hi;
    a[r + k] = hi;
    a[2 * r + k] = lo;
    bb[k] = hi;
    bb[r + k] = lo;
    bb[2 * r + k] = hi;
    if (c) {
      c[k] = hi;
      c[r + k] = hi;
      c[2 * r + k] = lo;
    }
  }
}

cudaError_t launch_lp_norm(const Dims& dm, float norm_eps, const float* Y, __nv_bfloat16* Xa,
                           __nv_bfloat16* Xb, __nv_bfloat16* XaC, uint32_t* status,
                           cudaStream_t st) {
  (void)status;
  launch_k(k_lp_norm, dim3(ceil_div(dm.N, 8), dm.B), 256, 0, st, 1, Y, dm.B, dm.N, dm.rank, dm.MV,
           norm_eps, Xa, Xb, XaC);
  return cudaGetLastError();
}

// Hs[b][k][:] = visual hidden row S_b[k] of image b; rnS[b][k] = its reciprocal norm.
__global__ void __launch_bounds__(256) k_gather_support(
    const uint4* __restrict__ hidden, const int32_t* __restrict__ support,
    const float* __restrict__ rn, const int32_t* toff, int B, int N, int K, int Tmax, int D8,
    uint4* Hs, float* rnS, uint32_t* status) {
  grid_dep_wait();
  const int b = blockIdx.y, k = blockIdx.x;
  const TextGeom tg = text_geom(toff, b, B, Tmax, status);
  if (tg.T == 0) return;
  const int j = support[(size_t)b * K + k];
  if (j < 0 || j >= N) {  // the solver always writes a valid support
    if (threadIdx.x == 0) set_status(status, GMC_STATUS_INTERNAL);
    return;
  }
  const uint4* src = hidden + ((size_t)b * N + tg.off + j) * D8;
  uint4* dst = Hs + ((size_t)b * K + k) * D8;
  for (int q = threadIdx.x; q < D8; q += blockDim.x) dst[q] = src[q];
  if (threadIdx.x == 0) rnS[(size_t)b * K + k] = rn[(size_t)b * N + j];
}

cudaError_t launch_gather_support(const Dims& dm, const void* hidden, const int32_t* support,
                                  const float* rn, __nv_bfloat16* Hs, float* rnS, uint32_t* status,
                                  cudaStream_t st) {
  // bf16 rows of D elements, D a multiple of 8: D / 8 16-byte units
  launch_k(k_gather_support, dim3(dm.K, dm.B), 256, 0, st, 1, (const uint4*)hidden, support, rn,
           dm.toff, dm.B, dm.N, dm.K, dm.T, dm.D / 8, (uint4*)Hs, rnS, status);
  return cudaGetLastError();
}

}  // namespace gmc
