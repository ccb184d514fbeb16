// Device helpers shared by the GMC kernels (sm_103a).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace gmc {

constexpr unsigned FULL = 0xffffffffu;

__device__ __forceinline__ float to_f32(float x) { return x; }
__device__ __forceinline__ float to_f32(__nv_bfloat16 x) { return __bfloat162float(x); }

template <typename T> __device__ __forceinline__ T from_f32(float x);
template <> __device__ __forceinline__ float from_f32<float>(float x) { return x; }
template <> __device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float x) {
  return __float2bfloat16_rn(x);  // round to nearest even
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(FULL, v, o);
  return v;
}
__device__ __forceinline__ double warp_sum(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(FULL, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(FULL, v, o));
  return v;
}
__device__ __forceinline__ int warp_sum_int(int v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(FULL, v, o);
  return v;
}

// Block-wide reductions; `scratch` holds >= 32 elements.  Every thread gets the result.
template <typename T, typename Op>
__device__ __forceinline__ T block_reduce(T v, T* scratch, Op op, T ident) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = op(v, __shfl_xor_sync(FULL, v, o));
  __syncthreads();
  if (lane == 0) scratch[wid] = v;
  __syncthreads();
  T r = ident;
  for (int w = 0; w < nw; ++w) r = op(r, scratch[w]);  // fixed order: deterministic
  __syncthreads();
  return r;
}
struct OpAdd { template <typename T> __device__ T operator()(T a, T b) const { return a + b; } };
struct OpMax { __device__ float operator()(float a, float b) const { return fmaxf(a, b); } };

// Fixed-point accumulation: a value x >= 0 is held as round(x * 2^e) in a
// 64-bit integer.  Integer sums do not depend on the order of the additions,
// so every gain / score reduction below is deterministic however the threads
// are scheduled, and exact for terms >= 2^-(e-24).
// x * 2^e rounded to the nearest integer (ties to even), for 0 <= x * 2^e < 2^63
// (every caller converts a non-negative value).  A 64-bit float-to-integer
// conversion runs on the narrow fp64 pipe of this GPU, so the value is split
// into two 32-bit conversions: v = x * 2^e is exact (power-of-two scale),
// hi = floor(v / 2^32) and lo = v - hi 2^32 are exact floats (v >= 2^32 makes v
// a multiple of 2^9), and only lo can carry a fraction.
__device__ __forceinline__ long long to_fix(float x, float scale) {
  const float v = x * scale;
  const float hi = floorf(v * 2.3283064365386963e-10f);  // 2^-32
  const float lo = fmaf(hi, -4294967296.f, v);             // exact
  return (long long)(((unsigned long long)__float2uint_rz(hi) << 32) + __float2uint_rn(lo));
}

// A non-negative 64-bit fixed-point integer as fp32 (within one ulp; the same
// on every call) without the fp64-pipe conversion.
__device__ __forceinline__ float fix_to_float(unsigned long long q) {
  return fmaf(__uint2float_rn((unsigned)(q >> 32)), 4294967296.f, __uint2float_rn((unsigned)q));
}
__device__ __forceinline__ double from_fix(long long q, double inv_scale) {
  return (double)q * inv_scale;
}

// 4-byte asynchronous global -> shared copy; a false predicate writes zero
// (source size 0, nothing is read from src).
__device__ __forceinline__ void cp_async4(void* smem, const void* src, bool pred) {
  const unsigned sa = (unsigned)__cvta_generic_to_shared(smem);
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;" ::"r"(sa), "l"(src),
               "r"(pred ? 4 : 0)
               : "memory");
}
__device__ __forceinline__ void cp_async16(void* smem, const void* src) {
  const unsigned sa = (unsigned)__cvta_generic_to_shared(smem);
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(sa), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}
template <int Pending>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(Pending) : "memory");
}

// Programmatic dependent launch: every kernel of the path is launched so it may
// begin while the previous kernel on its stream is still running, and its
// first statement waits here until that kernel has completed and its writes
// are visible.  Only the launch and the block set-up overlap; no memory is
// touched before the wait.  Without the launch attribute the wait returns at
// once.
__device__ __forceinline__ void grid_dep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

__device__ __forceinline__ void set_status(uint32_t* status, uint32_t bit) {
  if (status) atomicOr(status, bit);
}

__host__ __device__ __forceinline__ int ceil_div(int a, int b) { return (a + b - 1) / b; }

// Per-image text geometry.  text_offsets == nullptr: uniform T.
struct TextGeom {
  int off;  // text rows before this image (sum of T_b' for b' < b)
  int T;    // text rows of this image; 0 marks an image whose offsets are invalid
};
// An image with 1 <= T_b <= Tmax and offsets inside [0, B*Tmax] is valid; any
// other one sets GMC_STATUS_TEXT_LEN and is skipped by every kernel (T = 0).
__device__ __forceinline__ TextGeom text_geom(const int32_t* text_offsets, int b, int B, int Tmax,
                                              uint32_t* status) {
  TextGeom g;
  if (text_offsets) {
    g.off = text_offsets[b];
    g.T = text_offsets[b + 1] - g.off;
    if (g.T < 1 || g.T > Tmax || g.off < 0 || (long long)g.off + g.T > (long long)B * Tmax) {
      set_status(status, 0x4u);
      g.off = 0;
      g.T = 0;
    }
  } else {
    g.off = b * Tmax;
    g.T = Tmax;
  }
  return g;
}

}  // namespace gmc
