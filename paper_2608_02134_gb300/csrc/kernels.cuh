// Internal interface between the C-ABI layer (gmc_api.cu) and the kernel
// translation units.  Nothing here is exported from libgmc.so.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "../../include/gmc.h"

namespace gmc {

// Shapes of one call; every per-image buffer is strided by T (= T_max).
constexpr int MAX_VIEWS = 4;  // message views: the current one and up to 3 historical ones

struct Dims {
  int B, N, T, H, Hkv, d, D, K, gh, gw, L;  // L = landmarks per side
  int V;                                    // message views (1: the current view only)
  int I;                                    // images per prompt (N = I * gh * gw)
  int MV;                                   // appearance rows: N (exact bank) or the bounded bank's M_V
  int M;                                    // V*H*T + MV + I*L*L: client rows per prompt (max)
  int dtype;                                // GMC_F32 / GMC_BF16
  const int32_t* toff;                      // device text offsets or nullptr
  int rank;                                 // long prefixes: rows r of the Rademacher map (0: exact bank)
};

// Trace record layout passed by value to kernels (byte offsets, 0 = absent).
struct TraceView {
  char* base;  // nullptr: no trace
  size_t stride, off_order, off_round_end, off_pool, off_centres, off_head_assign, off_omega,
      off_pi, off_ebar, off_mass, off_gains, off_cover;
  int rounds_max, pool_size;
  __device__ __forceinline__ char* rec(int b) const { return base + (size_t)b * stride; }
  __device__ __forceinline__ gmc_trace_header* header(int b) const {
    return reinterpret_cast<gmc_trace_header*>(rec(b));
  }
  template <typename T> __device__ __forceinline__ T* at(int b, size_t off) const {
    return reinterpret_cast<T*>(rec(b) + off);
  }
  // round rd's gains row and F(S) slot (certificate inputs)
  __device__ __forceinline__ long long* gains(int b, int rd, int N) const {
    return at<long long>(b, off_gains) + (size_t)rd * N;
  }
  __device__ __forceinline__ unsigned long long* cover(int b, int rd) const {
    return at<unsigned long long>(b, off_cover) + rd;
  }
};

// The grounded rows' inputs of every message view (view 0 = current), by value
// to the client builder: row (v, h, t) of image b is
// beta[v] * omega_h * nu_t * ||u_i^{v,h,t}|| / sum_j ||u_j^{v,h,t}||.
struct ViewRows {
  int n;
  const float* A[MAX_VIEWS];
  const float* rs[MAX_VIEWS];
  const float* zn2[MAX_VIEWS];
  const float* sigma[MAX_VIEWS];
  float beta[MAX_VIEWS];
};

// The head-pattern Grams of every view for the clustering (view 0 = current):
// HG[v] holds [B][H*H + H] (Gram, then sum_t rs[h,t] per head).
struct ViewGrams {
  int n;
  const double* HG[MAX_VIEWS];
  float beta[MAX_VIEWS];
};

// Dense prefix layers gathered at the kept rows with the compaction (passed
// by value to the transport and identity kernels; n = 0: none).
struct PrefixKV {
  int n;
  const void* keys[GMC_MAX_PREFIX_LAYERS];
  void* out[GMC_MAX_PREFIX_LAYERS];
};

// Device scratch carved out of the caller's workspace.
struct Scratch {
  uint32_t* status;
  float* A;          // [B][H][T][N]   native attention slice (visual columns)
  float* rs;         // [B][H][nRS][T] parts of sum_i ||u_i^{h,t}|| over key splits (sum: 0 = inactive row)
  float2* mpart;     // [B][Hkv][RQ][nRS] per-split softmax (max, sum) of the packed query rows
  float* Z;          // [B][H][N][4]   probe values Z_h[i]
  float* zn2;        // [B][H][N]      ||Z_h[i]||^2
  float* sigpart;    // [B][nP][H]     block partials of ||Z_h||_F^2
  uint32_t* tick;    // [B]            last-block tickets of the probe (zeroed with status)
  uint32_t* tick2;   // [B]            last-block tickets of the assignment gap pass (same)
  uint32_t* tick3;   // [B]            last-block tickets of the head-Gram reduction (same)
  float* gatev;      // [B][4]         Delta_bar, s_x, mean message energy
  float* sigma;      // [B][H]         mass coordinate sigma_h
  double* hgpart;    // [B][nHG][H*H]  block partials of the head-pattern Gram
  double* HG;        // [B][H*H + H]   head-pattern Gram, then sum_t rs[h,t] per head
  float* W2;         // [B][H][N]      sum_t nu_t A[h,t,i]^2
  float* omega;      // [B][H]
  float* ebar;       // [B][N]  message energy e_i (the assignment divides by its mean)
  float* rn;         // [B][N]         1 / max(||h_i||, eps)
  float* rmsh;       // [B][N]         rms(h_i)
  float* cos;        // [B][N][N]      cosine of boundary states
  float* C;          // [B][M][N]      client matrix, then in-place residual survivor values
  uint16_t* scol;    // [B][M][N]      survivor token index
  long long* u0;     // [B][N]         fixed-point column sums of C
  int32_t* support;  // [B][K]         ascending
  int32_t* slot;     // [B][N]         position in support or -1
  int32_t* order;    // [B][K]         selection order
  float* delta;      // [B][N]
  double* dpart;     // [B][nA][2]     partial sums of delta and counts over discarded tokens
  float* epart;      // [B][nE]        block sums of the message energies e_i
  int32_t* pi;       // [B][N]
  uint32_t* mbits;   // [B][K][ceil(N/32)] members of each carrier slot, bit i = token i
  float* mass;       // [B][N]
  double* selpart;   // [B][64]        select-path total mass partials
  int32_t* fexp;     // [B]            select-path fixed-point exponents
  __nv_bfloat16* Qp; // [B][Hkv][RQ][d] packed text queries of each KV group (tcgen05 path)
  int nP, nHG, nA, nSel, nE, nRS;
  int hgtok;         // tokens per head-statistics block (nHG = ceil(N / hgtok))
  // Message views: A, rs, mpart, Z, zn2, sigpart, sigma, hgpart, HG, W2, Qp, the
  // probe tickets (tick) and the head-Gram tickets (tick3) hold V consecutive
  // per-view blocks; the pointers above address view 0 (the current view).
  int V, B;
  size_t vA, vrs, vmp, vZ, vzn, vsp, vsg, vhp, vHG, vW2, vQp;  // elements per view
  Scratch view(int v) const {
    Scratch t = *this;
    t.A += v * vA; t.rs += v * vrs; t.mpart += v * vmp; t.Z += v * vZ; t.zn2 += v * vzn;
    t.sigpart += v * vsp; t.sigma += v * vsg; t.hgpart += v * vhp; t.HG += v * vHG;
    t.W2 += v * vW2; t.Qp += v * vQp; t.tick += (size_t)v * B; t.tick3 += (size_t)v * B;
    return t;
  }
};

constexpr int ROWS_PER_BLOCK = 8;  // rownorm / probe / client builder blocks
int head_tokens(int B, int N, int H);  // tokens per head-statistics block: 8, or 9 where
                                      // that puts every block in one wave
constexpr int ASSIGN_WARPS = 16;   // warps per assignment block (32 tokens, one per lane)
int assign_blocks(int N);          // assignment blocks per image
constexpr int PROBE_TOK = 32;       // tokens per probe block

// Launch wrappers.  Each returns the first CUDA error it saw.
cudaError_t launch_rownorm(const Dims&, const void* hidden, float norm_eps, Scratch&, cudaStream_t);
cudaError_t launch_probe(const Dims&, const void* keys, const float* W, const void* queries,
                         const gmc_params&, Scratch&,
                         cudaStream_t);
cudaError_t launch_message(const Dims&, const void* keys, const void* queries, Scratch&,
                           cudaStream_t, int* launches = nullptr);
cudaError_t launch_heads(const Dims&, const gmc_params&, Scratch&, const TraceView&, cudaStream_t,
                         int cluster = 1, const ViewGrams* views = nullptr);
bool heads_supported(int H);  // the head statistics of H heads fit a block (H <= 56)
cudaError_t launch_gram(const Dims&, const void* hidden, Scratch&, cudaStream_t);
// app: the appearance rows' cosines, [B][MV][N] (the exact bank passes the
// N x N cosine matrix, MV = N)
// part: 0 every row, 1 the grounded rows, 2 the appearance and spatial rows
// (the column sums s.u0 start at zero: k_rownorm clears them)
cudaError_t launch_build_clients(const Dims&, const gmc_params&, int fx_exp, Scratch&,
                                 const ViewRows& views, const float* app,
                                 cudaStream_t, int part = 0);
// State left by the first (dense) selection round, run over the whole GPU.
// Rounds of the solver run on the whole GPU before the cluster kernel takes
// over: the dense first round, then sparse_gpu_rounds(N) sparse rounds (an
// even count: the cluster kernel starts from the gains in u1).  Larger images
// keep more survivors per round, so more rounds stay on the whole GPU; the
// counts were chosen by measurement.
__host__ __device__ inline int sparse_gpu_rounds(int N) { return N > 2048 ? 8 : 4; }

// per-image words of R0State::info
constexpr int INFO_W = 8;

struct R0State {
  int32_t* pool;   // [B][P]  pool of the current whole-GPU round (-1 padded)
  int32_t* info;   // [B][INFO_W]  pool size of the current round, tokens selected so far,
                   //         rounds done, tokens selected before the current round,
                   //         rounds done before the current round (the last two are
                   //         snapshots the pool kernel takes, read by every filter block
                   //         while block 0 advances the running counts)
  long long* s0;   // [B][P]  scores of the current round (fixed point)
  long long* u1;   // [B][N]  gains (fixed point), written by rounds 0, 2, ...
  long long* u2;   // [B][N]  gains written by rounds 1, 3, ...
  long long* ugain;  // u1 or u2: the gains the cluster kernel starts from
  float* bcov;     // [B][M]  coverage b_m after the last whole-GPU round
  int32_t* cnt;    // [B][M]  survivors per row (lists in place over Cbar / scol)
  long long* fv;   // [B][4]  F_b(V) per bank (fixed point)
};
cudaError_t launch_round0(const R0State&, int B, int N, int K, int M, const int32_t* toff, int H,
                          int T, int L2, const gmc_params&, int fx_exp, const int32_t* fexp,
                          float* C, uint16_t* scol, const long long* u0, int32_t* order,
                          uint32_t* status, const TraceView&, cudaStream_t, int I = 1);
cudaError_t launch_select(const R0State&, int B, int N, int K, int M, const int32_t* toff, int H, int T, int L2,
                          const gmc_params&, int fx_exp, const int32_t* fexp_per_image, float* C,
                          uint16_t* scol, const long long* u0, int32_t* order, int32_t* support,
                          int32_t* slot, int32_t* out_idx, uint32_t* status, const TraceView&,
                          cudaStream_t, int I = 1);
cudaError_t launch_select_prep(const float* C, int B, int M, int N, Scratch&, cudaStream_t);
// Whether the cluster solver's per-CTA state (a copy of every token's gain,
// bucket and pool slot, and its share of the client rows) fits one CTA's
// shared memory for this problem on this device; where it does not, every
// round runs on the whole GPU (launch_wide_select).
bool select_fits(int B, int N, int M, int P);
// Batched certificate c_B of the trace from the recorded rounds (one block per image).
cudaError_t launch_certificate(int B, int N, int K, const TraceView&, cudaStream_t);
// cs: nullptr (cosines read from the N x N matrix at the support's columns) or
// the support cosines [B][N][K], column k holding the k-th selected token
cudaError_t launch_assign(const Dims&, const gmc_params&, Scratch&, const TraceView&,
                          cudaStream_t, const float* cs = nullptr);
cudaError_t launch_transport(const Dims&, const gmc_params&, const void* hidden, const void* keys,
                             const int32_t* pos, const int32_t* support, const int32_t* pi,
                             const float* mass, const float* rmsh, const uint32_t* mbits,
                             int32_t* out_idx, void* out_hidden, void* out_kv, int32_t* out_pos,
                             uint32_t* status, cudaStream_t, const PrefixKV* prefix = nullptr);
cudaError_t launch_identity(const Dims&, const void* hidden, const void* keys, const int32_t* pos,
                            int32_t* out_idx, void* out_hidden, void* out_kv, int32_t* out_pos,
                            uint32_t* status, cudaStream_t, const PrefixKV* prefix = nullptr);
cudaError_t launch_rms_rows(const Dims&, const void* hidden, float* rmsh, uint32_t* status,
                            cudaStream_t);

}  // namespace gmc

namespace gmc {
// Element offsets of one image's rows in the ABI layouts (see include/gmc.h).
struct SeqIdx {
  size_t s;   // b*N + off_b: first input sequence row of the image
  size_t o;   // b*K + off_b: first output row of the image
  int R, Ro;  // N + T_b, K + T_b
  __host__ __device__ SeqIdx(int b, int N, int K, int off, int Tb)
      : s((size_t)b * N + off), o((size_t)b * K + off), R(N + Tb), Ro(K + Tb) {}
  __host__ __device__ size_t hidden_row(int r, int D) const { return (s + r) * (size_t)D; }
  __host__ __device__ size_t key_row(int r, int HD) const { return (2 * s + r) * (size_t)HD; }
  __host__ __device__ size_t value_row(int r, int HD) const { return (2 * s + R + r) * (size_t)HD; }
  __host__ __device__ size_t pos(int axis, int r) const { return 3 * s + (size_t)axis * R + r; }
  __host__ __device__ size_t out_hidden_row(int r, int D) const { return (o + r) * (size_t)D; }
  __host__ __device__ size_t out_kv_row(int which, int r, int HD) const {
    return (2 * o + (size_t)which * Ro + r) * (size_t)HD;
  }
  __host__ __device__ size_t out_pos(int axis, int r) const { return 3 * o + (size_t)axis * Ro + r; }
};
}  // namespace gmc

namespace gmc {
// Argument checks shared by the entry points (gmc_api.cu): every parameter in
// its documented range; the problem's shape within this build's limits
// (GMC_OK, GMC_ERR_ARG or GMC_ERR_UNSUPPORTED).
bool params_ok(const gmc_params& p, int max_pool = GMC_MAX_POOL);
int check_problem(const gmc_problem* prob, int N, int T, int d, int D, int max_n = GMC_MAX_N);
}  // namespace gmc

namespace gmc {
// Raise a kernel's dynamic shared-memory limit when a launch needs more than
// the 48 KB default (idempotent; remembers the largest value set per kernel).
cudaError_t set_smem_limit(const void* func, size_t bytes);
}  // namespace gmc

namespace gmc {
// Launch `kernel` on `st` with programmatic stream serialization: it may be
// scheduled while the previous kernel on the stream is still running, and its
// first statement (grid_dep_wait) orders every memory access after that
// kernel.  cluster_x > 1 adds a thread-block cluster of that size along x.
template <typename... P, typename... A>
cudaError_t launch_k(void (*kernel)(P...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                     int cluster_x, A... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  int n = 0;
  attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[n].val.programmaticStreamSerializationAllowed = 1;
  ++n;
  if (cluster_x > 1) {
    attr[n].id = cudaLaunchAttributeClusterDimension;
    attr[n].val.clusterDim.x = cluster_x;
    attr[n].val.clusterDim.y = 1;
    attr[n].val.clusterDim.z = 1;
    ++n;
  }
  cfg.attrs = attr;
  cfg.numAttrs = n;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}
}  // namespace gmc

namespace gmc {
cudaError_t launch_gram_simt(const Dims&, const void* hidden, Scratch&, cudaStream_t);
cudaError_t launch_gram_tc(const Dims&, const void* hidden, Scratch&, cudaStream_t);
bool gram_tc_supported(const Dims&);
cudaError_t launch_message_tc(const Dims&, const void* keys, const void* queries, Scratch&,
                              cudaStream_t, int* launches = nullptr);
bool message_tc_supported(const Dims&);
int message_rq(const Dims&);  // packed query rows per (image, KV group)
int message_splits(const Dims&);  // key splits of the message slice (parts of rs)
}  // namespace gmc

namespace gmc {
// C = diag(rscale) (A B^T) diag(cscale) on the tensor cores (k_gemm_tc.cu):
// A and B bf16, K-major rows of Kd elements; C fp32.  Image b's A rows start at
// row b * a_img (+ the image's text offset when a_text: the hidden layout, b*N +
// off_b) of A's tensor map, its B rows likewise; its C block at b * c_img.
struct GemmArgs {
  int B, M, Nn, Kd;          // images, rows, columns, contraction length
  long long a_img, b_img;    // operand rows between images (0: shared by every image)
  int a_text, b_text;        // add the image's text offset to the A / B row
  const int32_t* toff;       // text offsets (nullptr: uniform Tmax)
  int Tmax;
  const float* rscale;       // [B][M] or nullptr
  const float* cscale;       // [B][Nn] or nullptr
  float* C;                  // output
  long long c_img, ldc;      // elements between images / rows of C
  uint32_t* status;
  int sym;                   // 1: C symmetric (A, B the same rows, M == Nn > 128): tiles on
                             // or above the diagonal computed, the rest mirrored
  int m_fast;                // 1: consecutive CTAs walk the row tiles (B is the larger operand)
};
int gemm_sym_ctas(int N, int B);  // CTAs of the symmetric mode for N x N Grams of B images
// a_rows / b_rows: rows declared in the operand's tensor map (reads past them
// return zeros); lda / ldb: row pitch in elements (a multiple of 8).
cudaError_t launch_gemm_tc(const GemmArgs&, const void* A, long long a_rows, int lda,
                           const void* Bm, long long b_rows, int ldb, cudaStream_t);
cudaError_t make_tmap_bf16(CUtensorMap* map, const void* base, uint64_t row_elems, uint64_t rows,
                           uint64_t pitch_elems, uint32_t box_rows);

// Long prefixes (k_longprefix.cu): the projected unit states split into bf16
// hi/lo terms (Xa = [hi|hi|lo], Xb = [hi|lo|hi], XaC = Xa at the M_V uniformly
// spaced client tokens floor(m N / M_V)), and the selected rows gathered for
// the support cosines.
cudaError_t launch_lp_norm(const Dims&, float norm_eps, const float* Y, __nv_bfloat16* Xa,
                           __nv_bfloat16* Xb, __nv_bfloat16* XaC, uint32_t* status, cudaStream_t);
cudaError_t launch_gather_support(const Dims&, const void* hidden, const int32_t* support,
                                  const float* rn, __nv_bfloat16* Hs, float* rnS, uint32_t* status,
                                  cudaStream_t);

// Wide selection (k_wide.cu): every round of the batched responsibility solver
// on the whole GPU, for pools above GMC_MAX_POOL and visual counts above
// GMC_MAX_N (the long-prefix path: b = 512, N = 15,876).
struct WideState {
  int32_t* pool;    // [B][P]   pool of the current round (-1 padded)
  long long* sc;    // [B][P]   its scores (fixed point)
  int32_t* batch;   // [B][P]   the current round's batch, in score order
  int32_t* stamp;   // [B][N]   1 + the round a token entered the support (0: not yet)
  int32_t* info;    // [B][INFO_W] as R0State::info
  long long* u1;    // [B][N]   gains written by rounds 0, 2, ...
  long long* u2;    // [B][N]   gains written by rounds 1, 3, ...
  float* bcov;      // [B][M]   coverage b_m
  int32_t* cnt;     // [B][M]   survivors per row
  long long* fv;    // [B][4]   F_b(V) per bank (fixed point)
};
struct WideGeom {
  int B, N, K, Mstride;  // client rows per image (stride)
  int HV, Tmax, MV, L2;  // grounded rows per text token, appearance rows, spatial rows
  const int32_t* toff;
  int uniform;           // gmc_select: every image has Mstride rows, all in bank 0
};
int wide_rounds(int K, const gmc_params&);  // whole-GPU rounds launched: ceil(K / b)
cudaError_t launch_wide_select(const WideState&, const WideGeom&, const gmc_params&, int fx_exp,
                               const int32_t* fexp, float* C, uint16_t* scol, const long long* u0,
                               int32_t* order, int32_t* support, int32_t* slot, int32_t* out_idx,
                               uint32_t* status, const TraceView&, cudaStream_t);
}  // namespace gmc
