// C-ABI entry points of libgmc.so (declared and documented in include/gmc.h):
// argument validation, workspace carving and the launch sequence of one call.
#include <math.h>
#include <string.h>

#include <atomic>
#include <mutex>
#include <unordered_map>

#include "common.cuh"
#include "kernels.cuh"

using namespace gmc;

namespace gmc {

cudaError_t set_smem_limit(const void* func, size_t bytes) {
  static std::mutex mu;
  static std::unordered_map<const void*, size_t> done;
  if (bytes <= 48 * 1024) return cudaSuccess;
  std::lock_guard<std::mutex> lk(mu);
  auto it = done.find(func);
  if (it != done.end() && it->second >= bytes) return cudaSuccess;
  cudaError_t e =
      cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
  if (e == cudaSuccess) done[func] = bytes;
  return e;
}

bool params_ok(const gmc_params& p, int max_pool) {
  return p.batch_b >= 1 && p.pool_mult >= 1 && (long long)p.pool_mult * p.batch_b <= max_pool &&
         p.resp_temp > 0.f && p.resp_eps >= 0.f && p.tau_v > 0.f && p.tau_s > 0.f &&
         p.beta_G >= 0.f && p.beta_V >= 0.f && p.beta_S >= 0.f && p.landmarks >= 1 &&
         p.landmarks <= 64 && p.max_head_clusters >= 1 &&
         p.max_head_clusters <= GMC_MAX_HEADS && p.head_eps > 0.f && p.terminal_q_weight > 0.f &&
         p.lambda_mass >= 0.f && p.eps_mass > 0.f && p.gate_scale > 0.f && p.gate_pow > 0.f &&
         p.ambig_margin > 0.f && p.pop_strength >= 0.f && p.pop_strength <= 1.f &&
         p.rms_eps >= 0.f && p.norm_eps > 0.f && (p.check_mode == 0 || p.check_mode == 1);
}

// Shape checks shared by gmc_compress / gmc_transport / gmc_transport_noalloc.
int check_problem(const gmc_problem* prob, int N, int T, int d, int D, int max_n) {
  if (!prob) return GMC_ERR_ARG;
  const int I = prob->images < 1 ? 1 : prob->images;  // images per prompt
  if (prob->B < 1 || prob->grid_h < 1 || prob->grid_w < 1 || N < 1 ||
      (long long)prob->grid_h * prob->grid_w * I != N || T < 1 || d < 1 || D < 1 ||
      prob->Hkv < 1)
    return GMC_ERR_ARG;
  if (prob->dtype != GMC_F32 && prob->dtype != GMC_BF16) return GMC_ERR_ARG;
  if (N > max_n || D > 8192 || d > 1024) return GMC_ERR_UNSUPPORTED;
  if (prob->dtype == GMC_BF16 && (d % 8 != 0 || D % 8 != 0)) return GMC_ERR_UNSUPPORTED;
  if (prob->dtype == GMC_F32 && (d % 4 != 0 || D % 8 != 0)) return GMC_ERR_UNSUPPORTED;
  return GMC_OK;
}

}  // namespace gmc

namespace {

constexpr size_t ALIGN = 256;

struct Carver {
  char* base;
  size_t off = 0;
  template <typename T> T* take(size_t count) {
    const size_t at = off;
    off += (count * sizeof(T) + ALIGN - 1) & ~(ALIGN - 1);
    return base ? reinterpret_cast<T*>(base + at) : nullptr;
  }
};

// The long-prefix path: bf16 states, one image per prompt, at least 256 visual
// tokens (a full 128 x 256 tile of the support cosines), a rank that keeps the
// split states' rows 16-byte aligned, a device map.
int check_long_prefix(const gmc_problem* prob, const gmc_long_prefix* lp) {
  if (!lp->rademacher || ((uintptr_t)lp->rademacher % 16) != 0 || lp->rank < 8 ||
      lp->rank % 8 != 0 || lp->max_clients < 1)
    return GMC_ERR_ARG;
  if (lp->rank > GMC_MAX_RANK || prob->dtype != GMC_BF16 || (prob->images > 1) ||
      prob->grid_h * prob->grid_w < 256)
    return GMC_ERR_UNSUPPORTED;
  return GMC_OK;
}

// K = min{N, max{K_r, I}} (Sec. 3.1); K_r < 1 asks for the minimum
int effective_K(int K, int N, int I = 1) {
  const int k = K < I ? I : K;
  return k < 1 ? 1 : (k > N ? N : k);
}
int images_of(const gmc_problem* prob) { return prob->images < 1 ? 1 : prob->images; }

bool aligned(const void* p, size_t a) { return ((uintptr_t)p % a) == 0; }

Dims make_dims(const gmc_problem* prob, const gmc_params& p, int N, int T, int H, int d, int D,
               int K, int V = 1) {
  Dims dm;
  dm.B = prob->B; dm.N = N; dm.T = T; dm.H = H; dm.Hkv = prob->Hkv; dm.d = d; dm.D = D;
  dm.K = K; dm.gh = prob->grid_h; dm.gw = prob->grid_w; dm.L = p.landmarks;
  dm.V = V;
  dm.I = images_of(prob);
  dm.MV = N;
  dm.rank = 0;
  dm.M = V * H * T + dm.MV + dm.I * p.landmarks * p.landmarks;
  dm.dtype = prob->dtype;
  dm.toff = prob->text_offsets;
  return dm;
}

// Long prefixes: the bounded appearance bank has min(N, max_clients) rows.
Dims long_dims(Dims dm, const gmc_params& p, const gmc_long_prefix& lp) {
  dm.MV = lp.max_clients < dm.N ? lp.max_clients : dm.N;
  dm.rank = lp.rank;
  dm.M = dm.V * dm.H * dm.T + dm.MV + dm.I * p.landmarks * p.landmarks;
  return dm;
}

// Scratch of the long-prefix path and its wide solver (carved after the rest).
struct LongScratch {
  float* Y;             // [B][N][r]   projected states R h_i
  __nv_bfloat16* Xa;    // [B][N][3r]  [hi | hi | lo] of the unit projected states
  __nv_bfloat16* Xb;    // [B][N][3r]  [hi | lo | hi]
  __nv_bfloat16* XaC;   // [B][MV][3r] Xa at the appearance clients
  float* app;           // [B][MV][N]  projected cosines of the appearance clients
  __nv_bfloat16* Hs;    // [B][K][D]   selected visual rows
  float* rnS;           // [B][K]      their reciprocal norms
  float* cs;            // [B][K][N]   support cosines (row k: every token against S_k)
  WideState w;
};

void carve_wide(Carver& c, size_t B, size_t N, size_t M, size_t P, WideState* w) {
  w->pool = c.take<int32_t>(B * P);
  w->sc = c.take<long long>(B * P);
  w->batch = c.take<int32_t>(B * P);
  w->stamp = c.take<int32_t>(B * N);
  w->info = c.take<int32_t>(B * INFO_W);
  w->u1 = c.take<long long>(B * N);
  w->u2 = c.take<long long>(B * N);
  w->bcov = c.take<float>(B * M);
  w->cnt = c.take<int32_t>(B * M);
  w->fv = c.take<long long>(B * 4);
}

R0State carve_round0(Carver& c, size_t B, size_t N, size_t M);

// Words of the per-call zeroed status block: status, probe tickets (per
// view), assignment tickets, head-Gram tickets (per view), membership bitmaps.
size_t status_words(const Dims& dm) {
  return 4 + (2 * (size_t)dm.V + 1) * dm.B + (size_t)dm.B * dm.K * ceil_div(dm.N, 32);
}

// Workspace of gmc_compress.  base == nullptr only measures.
size_t carve_compress(const Dims& dm, Scratch* s, char* base, R0State* r0s = nullptr,
                      LongScratch* ls = nullptr, int pool = 0) {
  Carver c{base};
  Scratch t{};
  const size_t B = dm.B, N = dm.N, H = dm.H, T = dm.T, M = dm.M, K = dm.K;
  t.nP = ceil_div(dm.N, PROBE_TOK);
  t.hgtok = head_tokens(dm.B, dm.N, dm.H);
  t.nHG = ceil_div(dm.N, t.hgtok);
  t.nA = assign_blocks(dm.N);
  t.nE = t.nA;  // energy block sums come from the assignment gap kernel
  t.nSel = 0;
  const size_t V = dm.V;
  t.V = dm.V;
  t.B = dm.B;
  // status word, the probe (per view), assignment and head-Gram (per view)
  // tickets of every image, then the carrier membership bitmaps: one block,
  // zeroed by one memset per call
  t.status = c.take<uint32_t>(status_words(dm));
  t.tick = t.status + 4;
  t.tick2 = t.tick + V * B;
  t.tick3 = t.tick2 + B;
  t.mbits = t.tick3 + V * B;
  t.gatev = c.take<float>(B * 4);
  t.nRS = message_splits(dm);
  t.vA = B * H * T * N;
  t.vrs = B * H * (size_t)t.nRS * T;
  t.vmp = B * dm.Hkv * (size_t)message_rq(dm) * t.nRS;
  t.vZ = B * H * N * 4;
  t.vzn = B * H * N;
  t.vsp = B * t.nP * H;
  t.vsg = B * H;
  t.vhp = B * t.nHG * H * H;
  t.vHG = B * (H * H + H);
  t.vW2 = B * H * N;
  t.vQp = B * dm.Hkv * (size_t)message_rq(dm) * dm.d;
  t.A = c.take<float>(V * t.vA);
  t.rs = c.take<float>(V * t.vrs);
  t.mpart = c.take<float2>(V * t.vmp);
  t.Z = c.take<float>(V * t.vZ);
  t.zn2 = c.take<float>(V * t.vzn);
  t.sigpart = c.take<float>(V * t.vsp);
  t.sigma = c.take<float>(V * t.vsg);
  t.hgpart = c.take<double>(V * t.vhp);
  t.HG = c.take<double>(V * t.vHG);
  t.W2 = c.take<float>(V * t.vW2);
  t.omega = c.take<float>(B * H);
  t.ebar = c.take<float>(B * N);
  t.rn = c.take<float>(B * N);
  t.rmsh = c.take<float>(B * N);
  t.cos = dm.rank ? nullptr : c.take<float>(B * N * N);
  t.C = c.take<float>(B * M * N);
  t.scol = c.take<uint16_t>(B * M * N);
  t.u0 = c.take<long long>(B * N);
  t.support = c.take<int32_t>(B * K);
  t.slot = c.take<int32_t>(B * N);
  t.order = c.take<int32_t>(B * K);
  t.delta = c.take<float>(B * N);
  t.dpart = c.take<double>(B * t.nA * 2);
  t.epart = c.take<float>(B * t.nE);
  t.pi = c.take<int32_t>(B * N);
  t.mass = c.take<float>(B * N);
  t.selpart = nullptr;
  t.fexp = nullptr;
  t.Qp = c.take<__nv_bfloat16>(V * t.vQp);
  if (s) *s = t;
  if (dm.rank) {  // long prefixes: bounded bank, support cosines, wide solver
    LongScratch l{};
    const size_t r = dm.rank, MV = dm.MV;
    l.Y = c.take<float>(B * N * r);
    l.Xa = c.take<__nv_bfloat16>(B * N * 3 * r);
    l.Xb = c.take<__nv_bfloat16>(B * N * 3 * r);
    l.XaC = c.take<__nv_bfloat16>(B * MV * 3 * r);
    l.app = c.take<float>(B * MV * N);
    l.Hs = c.take<__nv_bfloat16>(B * K * dm.D);
    l.rnS = c.take<float>(B * K);
    l.cs = c.take<float>(B * N * K);
    carve_wide(c, B, N, M, (size_t)pool, &l.w);
    if (ls && base) *ls = l;
    return c.off;
  }
  R0State r0 = carve_round0(c, B, N, M);
  if (r0s && base) *r0s = r0;
  // the wide solver's state, for problems whose cluster-solver state does not
  // fit one CTA's shared memory (a few words per token and client row)
  WideState w{};
  carve_wide(c, B, N, M, GMC_MAX_POOL, &w);
  if (ls && base) ls->w = w;
  return c.off;
}

R0State carve_round0(Carver& c, size_t B, size_t N, size_t M) {
  R0State r;
  r.pool = c.take<int32_t>(B * GMC_MAX_POOL);
  r.info = c.take<int32_t>(B * INFO_W);
  r.s0 = c.take<long long>(B * GMC_MAX_POOL);
  r.u1 = c.take<long long>(B * N);
  r.u2 = c.take<long long>(B * N);
  r.ugain = sparse_gpu_rounds((int)N) % 2 == 0 ? r.u1 : r.u2;
  r.bcov = c.take<float>(B * M);
  r.cnt = c.take<int32_t>(B * M);
  r.fv = c.take<long long>(B * 4);
  return r;
}

int fixed_point_exponent(double total) {
  if (!(total > 0.0) || !isfinite(total)) return 61;
  int e = 61 - (int)ceil(log2(total));
  return e < -60 ? -60 : (e > 120 ? 120 : e);
}

int fill_trace_layout(int B, const gmc_params& p, int N, int H, int K, gmc_trace_layout* o,
                      int images = 1) {
  if (B < 1 || N < 1 || H < 0 || K < 1) return GMC_ERR_ARG;
  gmc_trace_layout L{};
  // responsibility rounds, a zero-gain fill, and a seed round for several images
  L.rounds_max = (K + p.batch_b - 1) / p.batch_b + 1 + (images > 1 ? 1 : 0);
  L.pool_size = p.pool_mult * p.batch_b;
  size_t off = sizeof(gmc_trace_header);
  auto take = [&](size_t bytes) {
    size_t at = off;
    off += (bytes + 15) & ~(size_t)15;
    return at;
  };
  L.off_order = take(4 * (size_t)K);
  L.off_round_end = take(4 * (size_t)L.rounds_max);
  L.off_pool = take(4 * (size_t)L.rounds_max * L.pool_size);
  L.off_centres = take(4 * (size_t)p.max_head_clusters);
  L.off_head_assign = take(4 * (size_t)H);
  L.off_omega = take(4 * (size_t)H);
  L.off_pi = take(4 * (size_t)N);
  L.off_ebar = take(4 * (size_t)N);
  L.off_mass = take(4 * (size_t)N);
  L.off_gains = take(8 * (size_t)L.rounds_max * N);
  L.off_cover = take(8 * (size_t)L.rounds_max);
  L.bytes_per_image = (off + 15) & ~(size_t)15;
  *o = L;
  return GMC_OK;
}

TraceView make_trace_view(void* trace, const gmc_trace_layout& L) {
  TraceView tv{};
  tv.base = (char*)trace;
  tv.stride = L.bytes_per_image;
  tv.off_order = L.off_order;
  tv.off_round_end = L.off_round_end;
  tv.off_pool = L.off_pool;
  tv.off_centres = L.off_centres;
  tv.off_head_assign = L.off_head_assign;
  tv.off_omega = L.off_omega;
  tv.off_pi = L.off_pi;
  tv.off_ebar = L.off_ebar;
  tv.off_mass = L.off_mass;
  tv.off_gains = L.off_gains;
  tv.off_cover = L.off_cover;
  tv.rounds_max = L.rounds_max;
  tv.pool_size = L.pool_size;
  return tv;
}

int cuda_fail(cudaError_t e) {
  if (e == cudaSuccess) return GMC_OK;
  cudaGetLastError();
  return GMC_ERR_CUDA;
}

#define GMC_TRY(expr)                         \
  do {                                        \
    cudaError_t _e = (expr);                  \
    if (_e != cudaSuccess) return cuda_fail(_e); \
  } while (0)

std::atomic<uint64_t> g_launches{0};

// Stage timing for benchmarks: events on the call's own stream.
struct Profiler {
  static constexpr int MAXEV = 16;
  std::mutex mu;
  bool on = false, valid = false;
  cudaEvent_t ev[MAXEV] = {};
  const char* names[MAXEV] = {};
  int n = 0;
  cudaError_t begin(cudaStream_t st) {
    n = 0;
    valid = false;
    if (!on) return cudaSuccess;
    if (!ev[0])
      for (int k = 0; k < MAXEV; ++k) {
        cudaError_t e = cudaEventCreate(&ev[k]);
        if (e != cudaSuccess) return e;
      }
    return cudaEventRecord(ev[n++], st);
  }
  cudaError_t mark(const char* name, cudaStream_t st) {
    if (!on || n >= MAXEV) return cudaSuccess;
    names[n - 1] = name;
    return cudaEventRecord(ev[n++], st);
  }
};
Profiler g_prof;

// A second stream per device for the branch of the path that does not depend
// on the message slice (row norms -> cosine Gram), forked from and joined back
// into the caller's stream with events.  Created on first use on each device;
// calls are serialised by the host lock of gmc_compress.
struct SideStream {
  cudaStream_t st = nullptr;
  cudaEvent_t fork = nullptr, join = nullptr;
  cudaEvent_t aux = nullptr;  // gmc_compress_host: the hidden states' copy has landed
};
SideStream g_side[64];

cudaError_t side_stream(SideStream** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  SideStream& sd = g_side[dev];
  if (!sd.st) {
    if ((e = cudaStreamCreateWithFlags(&sd.st, cudaStreamNonBlocking)) != cudaSuccess) return e;
    if ((e = cudaEventCreateWithFlags(&sd.fork, cudaEventDisableTiming)) != cudaSuccess) return e;
    if ((e = cudaEventCreateWithFlags(&sd.join, cudaEventDisableTiming)) != cudaSuccess) return e;
    if ((e = cudaEventCreateWithFlags(&sd.aux, cudaEventDisableTiming)) != cudaSuccess) return e;
  }
  *out = &sd;
  return cudaSuccess;
}

#define GMC_STAGE(name, nkernels, expr)              \
  do {                                               \
    GMC_TRY(expr);                                   \
    g_launches += (nkernels);                        \
    GMC_TRY(g_prof.mark(name, st));                  \
  } while (0)

}  // namespace

extern "C" {

void gmc_default_params(gmc_params* p) {
  if (!p) return;
  p->batch_b = 16;
  p->pool_mult = 4;
  p->resp_temp = 0.1f;
  p->resp_eps = 1e-12f;
  p->tau_v = 0.2f;
  p->tau_s = 0.02f;
  p->beta_G = 0.5f;
  p->beta_V = 0.5f;
  p->beta_S = 0.25f;
  p->landmarks = 16;
  p->max_head_clusters = 4;
  p->head_eps = 0.05f;
  p->terminal_q_weight = 2.f;
  p->lambda_mass = 1.f;
  p->eps_mass = 1e-8f;
  p->assign_spatial_w = 0.5f;
  p->gate_scale = 0.08f;
  p->gate_pow = 8.f;
  p->ambig_margin = 0.05f;
  p->pop_strength = 0.5f;
  p->rms_eps = 1e-6f;
  p->norm_eps = 1e-12f;
  p->check_mode = 0;
}

const char* gmc_error_string(int code) {
  switch (code) {
    case GMC_OK: return "GMC_OK";
    case GMC_ERR_ARG: return "GMC_ERR_ARG: invalid argument";
    case GMC_ERR_UNSUPPORTED: return "GMC_ERR_UNSUPPORTED: shape outside this build's limits";
    case GMC_ERR_WORKSPACE: return "GMC_ERR_WORKSPACE: workspace too small";
    case GMC_ERR_CUDA: return "GMC_ERR_CUDA: CUDA launch or query failed";
    default: return "GMC: unknown code";
  }
}

const char* gmc_version(void) { return "gmc 0.1.0 sm_103a"; }

size_t gmc_workspace_size_views(const gmc_problem* prob, int n_views, int N, int T, int H, int d,
                                int D, int K) {
  if (check_problem(prob, N, T, d, D) != GMC_OK || H < 1 || H > GMC_MAX_HEADS ||
      H % prob->Hkv != 0 || !heads_supported(H) || n_views < 0 || n_views > GMC_MAX_VIEWS - 1)
    return 0;
  gmc_params p;
  gmc_default_params(&p);
  const Dims dm =
      make_dims(prob, p, N, T, H, d, D, effective_K(K, N, images_of(prob)), 1 + n_views);
  return carve_compress(dm, nullptr, nullptr);
}

size_t gmc_workspace_size(const gmc_problem* prob, int N, int T, int H, int d, int D, int K) {
  return gmc_workspace_size_views(prob, 0, N, T, H, d, D, K);
}

int gmc_get_trace_layout(const gmc_problem* prob, const gmc_params* params, int N, int T, int H,
                         int K, gmc_trace_layout* out) {
  if (!prob || !out || T < 1) return GMC_ERR_ARG;
  gmc_params p;
  if (params) p = *params; else gmc_default_params(&p);
  if (!params_ok(p, GMC_MAX_POOL_WIDE)) return GMC_ERR_ARG;
  return fill_trace_layout(prob->B, p, N, H, effective_K(K, N, images_of(prob)), out,
                           images_of(prob));
}

size_t gmc_trace_size(const gmc_problem* prob, const gmc_params* params, int N, int T, int H,
                      int K) {
  gmc_trace_layout L;
  if (gmc_get_trace_layout(prob, params, N, T, H, K, &L) != GMC_OK) return 0;
  return (size_t)prob->B * L.bytes_per_image;
}

// The whole step, or (out_clients != nullptr) its steps up to the client
// matrix, copied into out_clients.
static int compress_impl(const gmc_problem* prob, const gmc_params* params,
                         const gmc_views* views, const gmc_prefix_kv* prefix,
                         const void* hidden, const void* keys,
                         const void* queries, const int32_t* pos_ids, const float* vo_probe,
                         int N, int T, int H, int d, int D, int K, int32_t* out_idx,
                         void* out_hidden, void* out_kv, int32_t* out_pos, void* workspace,
                         size_t ws_bytes, void* trace, gmc_stream_t stream_,
                         float* out_clients = nullptr, const gmc_long_prefix* lp = nullptr) {
  int rc = check_problem(prob, N, T, d, D, lp ? GMC_MAX_N_LONG : GMC_MAX_N);
  if (rc != GMC_OK) return rc;
  if (H < 1 || H % prob->Hkv != 0) return GMC_ERR_ARG;
  if (H > GMC_MAX_HEADS || !heads_supported(H)) return GMC_ERR_UNSUPPORTED;
  gmc_params p;
  if (params) p = *params; else gmc_default_params(&p);
  if (!params_ok(p, lp ? GMC_MAX_POOL_WIDE : GMC_MAX_POOL)) return GMC_ERR_ARG;
  if (lp) {
    rc = check_long_prefix(prob, lp);
    if (rc != GMC_OK) return rc;
  }
  if (!hidden || !keys || !queries || !pos_ids || !vo_probe || !workspace ||
      (!out_clients && (!out_idx || !out_hidden || !out_kv || !out_pos)))
    return GMC_ERR_ARG;
  if (out_clients && !aligned(out_clients, 16)) return GMC_ERR_ARG;
  if (!aligned(hidden, 16) || !aligned(keys, 16) || !aligned(queries, 16) ||
      !aligned(vo_probe, 16) || !aligned(out_hidden, 16) || !aligned(out_kv, 16) ||
      !aligned(workspace, ALIGN) || (trace && !aligned(trace, 16)))
    return GMC_ERR_ARG;
  // message views: view 0 is the call's own, then the historical ones
  const int nh = views ? views->n : 0;
  if (nh < 0 || nh > GMC_MAX_VIEWS - 1) return GMC_ERR_ARG;
  if (nh > 0 && !(views->beta_hist >= 0.f)) return GMC_ERR_ARG;
  const int V = 1 + nh;
  const void* vkeys[GMC_MAX_VIEWS] = {keys};
  const void* vqueries[GMC_MAX_VIEWS] = {queries};
  const float* vprobe[GMC_MAX_VIEWS] = {vo_probe};
  float vbeta[GMC_MAX_VIEWS] = {p.beta_G};
  for (int v = 1; v < V; ++v) {
    vkeys[v] = views->keys[v - 1];
    vqueries[v] = views->queries[v - 1];
    vprobe[v] = views->vo_probe[v - 1];
    vbeta[v] = views->beta_hist / (float)nh;
    if (!vkeys[v] || !vqueries[v] || !vprobe[v] || !aligned(vkeys[v], 16) ||
        !aligned(vqueries[v], 16) || !aligned(vprobe[v], 16))
      return GMC_ERR_ARG;
  }
  // dense prefix layers (cached path), gathered with the compaction
  PrefixKV pf{};
  if (prefix && !out_clients) {
    if (prefix->n_layers < 0 || prefix->n_layers > GMC_MAX_PREFIX_LAYERS) return GMC_ERR_ARG;
    pf.n = prefix->n_layers;
    for (int l = 0; l < pf.n; ++l) {
      pf.keys[l] = prefix->keys[l];
      pf.out[l] = prefix->out_kv[l];
      if (!pf.keys[l] || !pf.out[l] || !aligned(pf.keys[l], 16) || !aligned(pf.out[l], 16))
        return GMC_ERR_ARG;
    }
  }
  const int Ke = effective_K(K, N, images_of(prob));
  Dims dm = make_dims(prob, p, N, T, H, d, D, Ke, V);
  if (lp) dm = long_dims(dm, p, *lp);
  Scratch s;
  R0State r0;
  LongScratch ls{};
  const size_t need =
      carve_compress(dm, &s, (char*)workspace, &r0, &ls, p.pool_mult * p.batch_b);
  if (ws_bytes < need) return GMC_ERR_WORKSPACE;
  // every selection round on the whole GPU: long prefixes, and problems whose
  // cluster-solver state (a copy per token and a share of the client rows in
  // each CTA) does not fit one CTA's shared memory; that solver seeds no
  // per-image tokens, so a multi-image prompt must fit the cluster solver
  const bool wide =
      lp != nullptr || (!out_clients && Ke != N &&
                        !select_fits(dm.B, N, dm.M, p.pool_mult * p.batch_b));
  if (wide && dm.I > 1) return GMC_ERR_UNSUPPORTED;
  cudaStream_t st = (cudaStream_t)stream_;
  gmc_trace_layout L;
  TraceView tv{};
  if (trace) {
    fill_trace_layout(dm.B, p, N, H, Ke, &L, dm.I);
    tv = make_trace_view(trace, L);
    GMC_TRY(cudaMemsetAsync(trace, 0, (size_t)dm.B * L.bytes_per_image, st));
  }
  std::lock_guard<std::mutex> lk(g_prof.mu);
  // status, tickets, membership bitmaps
  GMC_TRY(cudaMemsetAsync(s.status, 0, sizeof(uint32_t) * status_words(dm), st));
  if (Ke == N && !out_clients) {  // K = N returns the unmodified execution
    GMC_TRY(launch_identity(dm, hidden, keys, pos_ids, out_idx, out_hidden, out_kv, out_pos,
                            s.status, st, &pf));
    g_launches += 1;
    return GMC_OK;
  }
  double mass = (double)p.beta_G + p.beta_V + p.beta_S;
  if (nh > 0) mass += views->beta_hist;
  const int fx = fixed_point_exponent(mass);
  Scratch sv[GMC_MAX_VIEWS];
  ViewRows vr{};
  ViewGrams vg{};
  vr.n = vg.n = V;
  for (int v = 0; v < V; ++v) {
    sv[v] = s.view(v);
    vr.A[v] = sv[v].A;
    vr.rs[v] = sv[v].rs;
    vr.zn2[v] = sv[v].zn2;
    vr.sigma[v] = sv[v].sigma;
    vr.beta[v] = vg.beta[v] = vbeta[v];
    vg.HG[v] = sv[v].HG;
  }
  // every view's probe and message slice; the historical views' head Grams,
  // then the current view's, whose last block clusters the heads over all views
  auto probes = [&]() -> cudaError_t {
    for (int v = 0; v < V; ++v) {
      const cudaError_t e = launch_probe(dm, vkeys[v], vprobe[v], vqueries[v], p, sv[v], st);
      if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
  };
  int msg_k = 0;  // message-slice launches of the call
  auto messages = [&]() -> cudaError_t {
    for (int v = 0; v < V; ++v) {
      int n = 0;
      const cudaError_t e = launch_message(dm, vkeys[v], vqueries[v], sv[v], st, &n);
      if (e != cudaSuccess) return e;
      msg_k += n;
    }
    return cudaSuccess;
  };
  auto heads = [&]() -> cudaError_t {
    for (int v = 1; v < V; ++v) {
      const cudaError_t e = launch_heads(dm, p, sv[v], tv, st, 0, nullptr);
      if (e != cudaSuccess) return e;
    }
    return launch_heads(dm, p, sv[0], tv, st, 1, V > 1 ? &vg : nullptr);
  };
  GMC_TRY(g_prof.begin(st));  // k_rownorm zeroes the column sums u0 of the client build
  // the appearance branch: cosine Gram, or on long prefixes the projection,
  // the split unit states and the bounded bank's cosines
  auto project = [&](cudaStream_t q) -> cudaError_t {
    GemmArgs g{};
    g.B = dm.B; g.M = N; g.Nn = dm.rank; g.Kd = D;
    g.a_img = N; g.b_img = 0; g.a_text = 1; g.b_text = 0;
    g.toff = dm.toff; g.Tmax = T;
    g.C = ls.Y; g.c_img = (long long)N * dm.rank; g.ldc = dm.rank;
    g.status = s.status;
    cudaError_t e = launch_gemm_tc(g, hidden, (long long)dm.B * (N + T), D, lp->rademacher,
                                   dm.rank, D, q);
    if (e != cudaSuccess) return e;
    return launch_lp_norm(dm, p.norm_eps, ls.Y, ls.Xa, ls.Xb, ls.XaC, s.status, q);
  };
  auto app_cos = [&](cudaStream_t q) -> cudaError_t {
    GemmArgs g{};
    g.B = dm.B; g.M = dm.MV; g.Nn = N; g.Kd = 3 * dm.rank;
    g.a_img = dm.MV; g.b_img = N; g.toff = dm.toff; g.Tmax = T;
    g.C = ls.app; g.c_img = (long long)dm.MV * N; g.ldc = N;
    g.status = s.status;
    return launch_gemm_tc(g, ls.XaC, (long long)dm.B * dm.MV, 3 * dm.rank, ls.Xb,
                          (long long)dm.B * N, 3 * dm.rank, q);
  };
  if (g_prof.on) {  // stage timing: every stage in turn on the caller's stream
    GMC_STAGE("rownorm", 1, launch_rownorm(dm, hidden, p.norm_eps, s, st));
    GMC_STAGE("probe", V, probes());
    GMC_STAGE("message", msg_k, messages());
    GMC_STAGE("heads", 2 * V, heads());
    if (lp) {
      GMC_STAGE("project", 2, project(st));
      GMC_STAGE("app_cos", 1, app_cos(st));
    } else {
      GMC_STAGE("gram", 1, launch_gram(dm, hidden, s, st));
    }
  } else {
    // row norms and the cosine Gram run beside probe -> message -> heads
    SideStream* sd = nullptr;
    GMC_TRY(side_stream(&sd));
    GMC_TRY(cudaEventRecord(sd->fork, st));
    GMC_TRY(cudaStreamWaitEvent(sd->st, sd->fork, 0));
    GMC_STAGE("rownorm", 1, launch_rownorm(dm, hidden, p.norm_eps, s, sd->st));
    if (lp) {
      GMC_STAGE("project", 2, project(sd->st));
      GMC_STAGE("app_cos", 1, app_cos(sd->st));
    } else {
      GMC_STAGE("gram", 1, launch_gram(dm, hidden, s, sd->st));
    }
    // the appearance and spatial rows need only the cosines: built here,
    // beside the message slice and the heads
    GMC_STAGE("clients_aux", 1,
              launch_build_clients(dm, p, fx, s, vr, lp ? ls.app : s.cos, sd->st, 2));
    GMC_TRY(cudaEventRecord(sd->join, sd->st));
    GMC_STAGE("probe", V, probes());
    GMC_STAGE("message", msg_k, messages());
    GMC_STAGE("heads", 2 * V, heads());
    GMC_TRY(cudaStreamWaitEvent(st, sd->join, 0));
  }
  // every view's grounded rows count as head rows of the client layout
  const int HV = H * V;
  // the grounded rows (every row when stages are timed one after another)
  GMC_STAGE("clients", 1,
            launch_build_clients(dm, p, fx, s, vr, lp ? ls.app : s.cos, st, g_prof.on ? 0 : 1));
  if (out_clients) {  // staged call: the client matrix, before selection compacts it in place
    GMC_TRY(cudaMemcpyAsync(out_clients, s.C, sizeof(float) * dm.B * (size_t)dm.M * N,
                            cudaMemcpyDeviceToDevice, st));
    return GMC_OK;
  }
  const int LS = dm.I * p.landmarks * p.landmarks;  // spatial rows: a landmark grid per image
  if (wide) {
    WideGeom wg{};
    wg.B = dm.B; wg.N = N; wg.K = Ke; wg.Mstride = dm.M;
    wg.HV = HV; wg.Tmax = T; wg.MV = dm.MV; wg.L2 = LS;
    wg.toff = dm.toff; wg.uniform = 0;
    GMC_STAGE("select", 4 * wide_rounds(Ke, p) + 1,
              launch_wide_select(ls.w, wg, p, fx, nullptr, s.C, s.scol, s.u0, s.order, s.support,
                                 s.slot, nullptr, s.status, tv, st));
    if (tv.base) {
      GMC_TRY(launch_certificate(dm.B, N, Ke, tv, st));
      g_launches += 1;
    }
  } else {
    GMC_STAGE("rounds_gpu", 3 + 3 * sparse_gpu_rounds(N),
              launch_round0(r0, dm.B, N, Ke, dm.M, dm.toff, HV, T, LS, p, fx, nullptr, s.C,
                            s.scol, s.u0, s.order, s.status, tv, st, dm.I));
    GMC_STAGE("select", 1,
              launch_select(r0, dm.B, N, Ke, dm.M, dm.toff, HV, T, LS, p, fx, nullptr, s.C,
                            s.scol, s.u0, s.order, s.support, s.slot, nullptr, s.status, tv, st,
                            dm.I));
  }
  if (lp) {
    // the support cosines of the assignment (Eq. (cond-assignment)), K x N:
    // row k holds the cosines of every token with the k-th selected one
    auto support_cos = [&]() -> cudaError_t {
      cudaError_t e = launch_gather_support(dm, hidden, s.support, s.rn, ls.Hs, ls.rnS, s.status, st);
      if (e != cudaSuccess) return e;
      GemmArgs g{};
      g.B = dm.B; g.M = Ke; g.Nn = N; g.Kd = D;
      g.a_img = Ke; g.b_img = N; g.a_text = 0; g.b_text = 1;
      g.toff = dm.toff; g.Tmax = T;
      g.rscale = ls.rnS; g.cscale = s.rn;
      g.C = ls.cs; g.c_img = (long long)N * Ke; g.ldc = N;
      g.status = s.status;
      g.m_fast = 1;  // the hidden rows (B) are the large operand
      return launch_gemm_tc(g, ls.Hs, (long long)dm.B * Ke, D, hidden, (long long)dm.B * (N + T),
                            D, st);
    };
    GMC_STAGE("support_cos", 2, support_cos());
    GMC_STAGE("assign", 2, launch_assign(dm, p, s, tv, st, ls.cs));
    GMC_STAGE("transport", 1,
              launch_transport(dm, p, hidden, keys, pos_ids, s.support, s.pi, s.mass, s.rmsh,
                               s.mbits, out_idx, out_hidden, out_kv, out_pos, s.status, st, &pf));
    g_prof.valid = g_prof.on;
    return GMC_OK;
  }
  GMC_STAGE("assign", 2, launch_assign(dm, p, s, tv, st));
  GMC_STAGE("transport", 1,
            launch_transport(dm, p, hidden, keys, pos_ids, s.support, s.pi, s.mass, s.rmsh,
                             s.mbits, out_idx, out_hidden, out_kv, out_pos, s.status, st, &pf));
  g_prof.valid = g_prof.on;
  return GMC_OK;
}

int gmc_compress(const gmc_problem* prob, const gmc_params* params, const void* hidden,
                 const void* keys, const void* queries, const int32_t* pos_ids,
                 const float* vo_probe, int N, int T, int H, int d, int D, int K,
                 int32_t* out_idx, void* out_hidden, void* out_kv, int32_t* out_pos,
                 void* workspace, size_t ws_bytes, void* trace, gmc_stream_t stream_) {
  return compress_impl(prob, params, nullptr, nullptr, hidden, keys, queries, pos_ids, vo_probe,
                       N, T, H, d, D, K, out_idx, out_hidden, out_kv, out_pos, workspace,
                       ws_bytes, trace, stream_);
}

int gmc_compress_host(const gmc_problem* prob, const gmc_params* params, const gmc_host_io* io,
                      int N, int T, int H, int d, int D, int K, void* workspace, size_t ws_bytes,
                      void* trace, gmc_stream_t stream_) {
  if (!prob || !io) return GMC_ERR_ARG;
  if (!io->hidden || !io->d_hidden || !io->keys || !io->d_keys || !io->queries ||
      !io->d_queries || !io->pos_ids || !io->d_pos_ids || !io->vo_probe || !io->d_vo_probe ||
      !io->d_out_idx || !io->out_idx || !io->d_out_hidden || !io->out_hidden || !io->d_out_kv ||
      !io->out_kv || !io->d_out_pos || !io->out_pos)
    return GMC_ERR_ARG;
  if (!io->hidden_bytes || !io->keys_bytes || !io->queries_bytes || !io->pos_ids_bytes ||
      !io->vo_probe_bytes || !io->out_idx_bytes || !io->out_hidden_bytes || !io->out_kv_bytes ||
      !io->out_pos_bytes)
    return GMC_ERR_ARG;
  // the problem is checked before any copy is enqueued
  if (gmc_workspace_size(prob, N, T, H, d, D, K) == 0) return GMC_ERR_ARG;
  cudaStream_t st = (cudaStream_t)stream_;
  SideStream* sd = nullptr;
  GMC_TRY(side_stream(&sd));
  // the hidden states on the side stream, after the caller's earlier work on `stream`
  GMC_TRY(cudaEventRecord(sd->fork, st));
  GMC_TRY(cudaStreamWaitEvent(sd->st, sd->fork, 0));
  GMC_TRY(cudaMemcpyAsync(io->d_hidden, io->hidden, io->hidden_bytes, cudaMemcpyHostToDevice,
                          sd->st));
  GMC_TRY(cudaMemcpyAsync(io->d_keys, io->keys, io->keys_bytes, cudaMemcpyHostToDevice, st));
  GMC_TRY(cudaMemcpyAsync(io->d_queries, io->queries, io->queries_bytes, cudaMemcpyHostToDevice,
                          st));
  GMC_TRY(cudaMemcpyAsync(io->d_vo_probe, io->vo_probe, io->vo_probe_bytes,
                          cudaMemcpyHostToDevice, st));
  GMC_TRY(cudaMemcpyAsync(io->d_pos_ids, io->pos_ids, io->pos_ids_bytes, cudaMemcpyHostToDevice,
                          st));
  // Only the pipelined path reads the hidden states after its side stream has
  // joined; the identity (K = N) and the stage-timed runs read them on `stream`.
  const bool pipelined = !g_prof.on && effective_K(K, N, images_of(prob)) != N;
  if (!pipelined) {
    GMC_TRY(cudaEventRecord(sd->aux, sd->st));
    GMC_TRY(cudaStreamWaitEvent(st, sd->aux, 0));
  }
  const int rc = compress_impl(prob, params, nullptr, nullptr, io->d_hidden, io->d_keys,
                               io->d_queries, io->d_pos_ids, io->d_vo_probe, N, T, H, d, D, K,
                               io->d_out_idx, io->d_out_hidden, io->d_out_kv, io->d_out_pos,
                               workspace, ws_bytes, trace, stream_);
  if (rc != GMC_OK) return rc;
  GMC_TRY(cudaMemcpyAsync(io->out_idx, io->d_out_idx, io->out_idx_bytes, cudaMemcpyDeviceToHost,
                          st));
  GMC_TRY(cudaMemcpyAsync(io->out_hidden, io->d_out_hidden, io->out_hidden_bytes,
                          cudaMemcpyDeviceToHost, st));
  GMC_TRY(cudaMemcpyAsync(io->out_kv, io->d_out_kv, io->out_kv_bytes, cudaMemcpyDeviceToHost, st));
  GMC_TRY(cudaMemcpyAsync(io->out_pos, io->d_out_pos, io->out_pos_bytes, cudaMemcpyDeviceToHost,
                          st));
  return GMC_OK;
}

int gmc_compress_views(const gmc_problem* prob, const gmc_params* params, const gmc_views* views,
                       const void* hidden, const void* keys, const void* queries,
                       const int32_t* pos_ids, const float* vo_probe, int N, int T, int H, int d,
                       int D, int K, int32_t* out_idx, void* out_hidden, void* out_kv,
                       int32_t* out_pos, void* workspace, size_t ws_bytes, void* trace,
                       gmc_stream_t stream_) {
  return compress_impl(prob, params, views, nullptr, hidden, keys, queries, pos_ids, vo_probe, N,
                       T, H, d, D, K, out_idx, out_hidden, out_kv, out_pos, workspace, ws_bytes,
                       trace, stream_);
}

int gmc_compress_ex(const gmc_problem* prob, const gmc_params* params, const gmc_views* views,
                    const gmc_prefix_kv* prefix, const void* hidden, const void* keys,
                    const void* queries, const int32_t* pos_ids, const float* vo_probe, int N,
                    int T, int H, int d, int D, int K, int32_t* out_idx, void* out_hidden,
                    void* out_kv, int32_t* out_pos, void* workspace, size_t ws_bytes,
                    void* trace, gmc_stream_t stream_) {
  return compress_impl(prob, params, views, prefix, hidden, keys, queries, pos_ids, vo_probe, N,
                       T, H, d, D, K, out_idx, out_hidden, out_kv, out_pos, workspace, ws_bytes,
                       trace, stream_);
}

size_t gmc_workspace_size_long(const gmc_problem* prob, const gmc_params* params,
                               const gmc_long_prefix* lp, int n_views, int N, int T, int H, int d,
                               int D, int K) {
  if (!lp || check_problem(prob, N, T, d, D, GMC_MAX_N_LONG) != GMC_OK ||
      check_long_prefix(prob, lp) != GMC_OK || H < 1 || H > GMC_MAX_HEADS ||
      H % prob->Hkv != 0 || !heads_supported(H) || n_views < 0 || n_views > GMC_MAX_VIEWS - 1)
    return 0;
  gmc_params p;
  if (params) p = *params; else gmc_default_params(&p);
  if (!params_ok(p, GMC_MAX_POOL_WIDE)) return 0;
  Dims dm = make_dims(prob, p, N, T, H, d, D, effective_K(K, N, images_of(prob)), 1 + n_views);
  dm = long_dims(dm, p, *lp);
  return carve_compress(dm, nullptr, nullptr, nullptr, nullptr, p.pool_mult * p.batch_b);
}

int gmc_compress_long(const gmc_problem* prob, const gmc_params* params,
                      const gmc_long_prefix* lp, const gmc_views* views,
                      const gmc_prefix_kv* prefix, const void* hidden, const void* keys,
                      const void* queries, const int32_t* pos_ids, const float* vo_probe, int N,
                      int T, int H, int d, int D, int K, int32_t* out_idx, void* out_hidden,
                      void* out_kv, int32_t* out_pos, void* workspace, size_t ws_bytes,
                      void* trace, gmc_stream_t stream_) {
  if (!lp) return GMC_ERR_ARG;
  return compress_impl(prob, params, views, prefix, hidden, keys, queries, pos_ids, vo_probe, N,
                       T, H, d, D, K, out_idx, out_hidden, out_kv, out_pos, workspace, ws_bytes,
                       trace, stream_, nullptr, lp);
}

int gmc_clients_long(const gmc_problem* prob, const gmc_params* params, const gmc_long_prefix* lp,
                     const gmc_views* views, const void* hidden, const void* keys,
                     const void* queries, const int32_t* pos_ids, const float* vo_probe, int N,
                     int T, int H, int d, int D, int K, float* out_clients, void* workspace,
                     size_t ws_bytes, void* trace, gmc_stream_t stream_) {
  if (!out_clients || !lp) return GMC_ERR_ARG;
  return compress_impl(prob, params, views, nullptr, hidden, keys, queries, pos_ids, vo_probe, N,
                       T, H, d, D, K, nullptr, nullptr, nullptr, nullptr, workspace, ws_bytes,
                       trace, stream_, out_clients, lp);
}

int gmc_clients(const gmc_problem* prob, const gmc_params* params, const gmc_views* views,
                const void* hidden, const void* keys, const void* queries, const int32_t* pos_ids,
                const float* vo_probe, int N, int T, int H, int d, int D, int K,
                float* out_clients, void* workspace, size_t ws_bytes, void* trace,
                gmc_stream_t stream_) {
  if (!out_clients) return GMC_ERR_ARG;
  return compress_impl(prob, params, views, nullptr, hidden, keys, queries, pos_ids, vo_probe, N,
                       T, H, d, D, K, nullptr, nullptr, nullptr, nullptr, workspace, ws_bytes,
                       trace, stream_, out_clients);
}

// ---------------------------------------------------------------------------
// gmc_select
// ---------------------------------------------------------------------------
static size_t carve_select(int B, int M, int N, int K, Scratch* s, char* base,
                           R0State* r0s = nullptr, int wide_pool = 0, WideState* ws = nullptr) {
  Carver c{base};
  Scratch t{};
  t.nSel = 64;
  t.status = c.take<uint32_t>(4);
  t.C = c.take<float>((size_t)B * M * N);
  t.scol = c.take<uint16_t>((size_t)B * M * N);
  t.u0 = c.take<long long>((size_t)B * N);
  t.order = c.take<int32_t>((size_t)B * K);
  t.support = c.take<int32_t>((size_t)B * K);
  t.slot = c.take<int32_t>((size_t)B * N);
  t.selpart = c.take<double>((size_t)B * t.nSel);
  t.fexp = c.take<int32_t>((size_t)B);
  if (s) *s = t;
  // the wide solver's state: pools above GMC_MAX_POOL, and problems whose
  // cluster-solver state does not fit one CTA's shared memory
  WideState w{};
  carve_wide(c, (size_t)B, (size_t)N, (size_t)M, (size_t)(wide_pool > 0 ? wide_pool : GMC_MAX_POOL),
             &w);
  if (ws && base) *ws = w;
  if (wide_pool > 0) return c.off;
  R0State r0 = carve_round0(c, (size_t)B, (size_t)N, (size_t)M);
  if (r0s && base) *r0s = r0;
  return c.off;
}

// gmc_select runs the wide solver when the pool exceeds GMC_MAX_POOL (and, at
// run time, when the cluster solver's state does not fit; see select_fits)
static int select_wide_pool(const gmc_params& p) {
  const int P = p.pool_mult * p.batch_b;
  return P > GMC_MAX_POOL ? P : 0;
}

size_t gmc_select_workspace_size(int B, int M, int N, int K, const gmc_params* params) {
  gmc_params p;
  if (params) p = *params; else gmc_default_params(&p);
  if (!params_ok(p, GMC_MAX_POOL_WIDE)) return 0;
  const int wp = select_wide_pool(p);
  if (B < 1 || M < 1 || N < 1 || N > (wp ? GMC_MAX_N_LONG : GMC_MAX_N) || K < 1 || K > N) return 0;
  return carve_select(B, M, N, K, nullptr, nullptr, nullptr, wp);
}

int gmc_select(const float* clients, int B, int M, int N, int K, const gmc_params* params,
               int32_t* out_idx, void* workspace, size_t ws_bytes, void* trace,
               gmc_stream_t stream_) {
  if (!clients || !out_idx || !workspace || B < 1 || M < 1 || N < 1 || K < 1 || K > N)
    return GMC_ERR_ARG;
  if (!aligned(workspace, ALIGN) || (trace && !aligned(trace, 16))) return GMC_ERR_ARG;
  gmc_params p;
  if (params) p = *params; else gmc_default_params(&p);
  if (!params_ok(p, GMC_MAX_POOL_WIDE)) return GMC_ERR_ARG;
  const int wp = select_wide_pool(p);
  if (N > (wp ? GMC_MAX_N_LONG : GMC_MAX_N)) return GMC_ERR_UNSUPPORTED;
  Scratch s;
  R0State r0;
  WideState w{};
  const size_t need = carve_select(B, M, N, K, &s, (char*)workspace, &r0, wp, &w);
  if (ws_bytes < need) return GMC_ERR_WORKSPACE;
  cudaStream_t st = (cudaStream_t)stream_;
  TraceView tv{};
  if (trace) {
    gmc_trace_layout L;
    fill_trace_layout(B, p, N, 0, K, &L);
    tv = make_trace_view(trace, L);
    GMC_TRY(cudaMemsetAsync(trace, 0, (size_t)B * L.bytes_per_image, st));
  }
  GMC_TRY(cudaMemsetAsync(s.status, 0, sizeof(uint32_t), st));
  GMC_TRY(cudaMemcpyAsync(s.C, clients, sizeof(float) * B * (size_t)M * N,
                          cudaMemcpyDeviceToDevice, st));
  GMC_TRY(cudaMemsetAsync(s.u0, 0, sizeof(long long) * B * (size_t)N, st));
  GMC_TRY(launch_select_prep(s.C, B, M, N, s, st));
  if (wp || !select_fits(B, N, M, p.pool_mult * p.batch_b)) {
    WideGeom wg{};
    wg.B = B; wg.N = N; wg.K = K; wg.Mstride = M;
    wg.HV = 0; wg.Tmax = 1; wg.MV = 0; wg.L2 = 0;
    wg.toff = nullptr; wg.uniform = 1;
    GMC_TRY(launch_wide_select(w, wg, p, 0, s.fexp, s.C, s.scol, s.u0, s.order, s.support, s.slot,
                               out_idx, s.status, tv, st));
    g_launches += 3 + 4 * wide_rounds(K, p) + 1;
    if (tv.base) {
      GMC_TRY(launch_certificate(B, N, K, tv, st));
      g_launches += 1;
    }
    return GMC_OK;
  }
  GMC_TRY(launch_round0(r0, B, N, K, M, nullptr, 0, 1, 0, p, 0, s.fexp, s.C, s.scol, s.u0,
                        s.order, s.status, tv, st));
  GMC_TRY(launch_select(r0, B, N, K, M, nullptr, 0, 1, 0, p, 0, s.fexp, s.C, s.scol, s.u0,
                        s.order, s.support, s.slot, out_idx, s.status, tv, st));
  g_launches += 7 + 3 * sparse_gpu_rounds(N);
  return GMC_OK;
}

// ---------------------------------------------------------------------------
// gmc_cosine
// ---------------------------------------------------------------------------
size_t gmc_cosine_workspace_size(const gmc_problem* prob, int N) {
  if (!prob || prob->B < 1 || N < 1) return 0;
  Carver c{nullptr};
  c.take<uint32_t>(4);
  c.take<float>((size_t)prob->B * N * 2);
  return c.off;
}

int gmc_cosine(const gmc_problem* prob, const gmc_params* params, const void* hidden, int N,
               int T, int D, float* out_cos, void* workspace, size_t ws_bytes,
               gmc_stream_t stream_) {
  int rc = check_problem(prob, N, T, 8, D);
  if (rc != GMC_OK) return rc;
  gmc_params p;
  if (params) p = *params; else gmc_default_params(&p);
  if (!params_ok(p)) return GMC_ERR_ARG;
  if (!hidden || !out_cos || !workspace) return GMC_ERR_ARG;
  if (!aligned(hidden, 16) || !aligned(out_cos, 16) || !aligned(workspace, ALIGN))
    return GMC_ERR_ARG;
  if (ws_bytes < gmc_cosine_workspace_size(prob, N)) return GMC_ERR_WORKSPACE;
  Carver c{(char*)workspace};
  Scratch s{};
  s.status = c.take<uint32_t>(4);
  s.rn = c.take<float>((size_t)prob->B * N);
  s.rmsh = c.take<float>((size_t)prob->B * N);
  s.cos = out_cos;
  cudaStream_t st = (cudaStream_t)stream_;
  const Dims dm = make_dims(prob, p, N, T, 0, 8, D, 1);
  GMC_TRY(cudaMemsetAsync(s.status, 0, sizeof(uint32_t), st));
  GMC_TRY(launch_rownorm(dm, hidden, p.norm_eps, s, st));
  GMC_TRY(launch_gram(dm, hidden, s, st));
  g_launches += 2;
  return GMC_OK;
}

// ---------------------------------------------------------------------------
// gmc_transport
// ---------------------------------------------------------------------------
size_t gmc_transport_workspace_size(const gmc_problem* prob, int N, int T, int K) {
  if (!prob || prob->B < 1 || N < 1 || T < 1 || K < 1 || K > N) return 0;
  Carver c{nullptr};
  c.take<uint32_t>(4);
  c.take<float>((size_t)prob->B * N);
  return c.off;
}

int gmc_transport(const gmc_problem* prob, const gmc_params* params, const void* hidden,
                  const void* keys, const int32_t* pos_ids, const int32_t* support,
                  const int32_t* assign, const float* weights, int N, int T, int d, int D, int K,
                  int32_t* out_idx, void* out_hidden, void* out_kv, int32_t* out_pos,
                  void* workspace, size_t ws_bytes, gmc_stream_t stream_) {
  int rc = check_problem(prob, N, T, d, D);
  if (rc != GMC_OK) return rc;
  if (K < 1 || K > N) return GMC_ERR_ARG;
  gmc_params p;
  if (params) p = *params; else gmc_default_params(&p);
  if (!params_ok(p)) return GMC_ERR_ARG;
  if (!hidden || !keys || !pos_ids || !support || !assign || !weights || !out_idx ||
      !out_hidden || !out_kv || !out_pos || !workspace)
    return GMC_ERR_ARG;
  if (!aligned(hidden, 16) || !aligned(keys, 16) || !aligned(out_hidden, 16) ||
      !aligned(out_kv, 16) || !aligned(workspace, ALIGN))
    return GMC_ERR_ARG;
  if (ws_bytes < gmc_transport_workspace_size(prob, N, T, K)) return GMC_ERR_WORKSPACE;
  Carver c{(char*)workspace};
  uint32_t* status = c.take<uint32_t>(4);
  float* rmsh = c.take<float>((size_t)prob->B * N);
  cudaStream_t st = (cudaStream_t)stream_;
  const Dims dm = make_dims(prob, p, N, T, 0, d, D, K);
  GMC_TRY(cudaMemsetAsync(status, 0, sizeof(uint32_t), st));
  GMC_TRY(launch_rms_rows(dm, hidden, rmsh, status, st));
  GMC_TRY(launch_transport(dm, p, hidden, keys, pos_ids, support, assign, weights, rmsh, nullptr,
                           out_idx, out_hidden, out_kv, out_pos, status, st));
  g_launches += 3;
  return GMC_OK;
}

int gmc_profile_enable(int on) {
  std::lock_guard<std::mutex> lk(g_prof.mu);
  g_prof.on = on != 0;
  g_prof.valid = false;
  return GMC_OK;
}

int gmc_profile_read(float* ms, const char** names, int max) {
  std::lock_guard<std::mutex> lk(g_prof.mu);
  if (!g_prof.valid || g_prof.n < 2) return -1;
  if (cudaEventSynchronize(g_prof.ev[g_prof.n - 1]) != cudaSuccess) return cuda_fail(cudaErrorUnknown), -1;
  const int ns = g_prof.n - 1;
  for (int k = 0; k < ns && k < max; ++k) {
    float t = 0.f;
    cudaEventElapsedTime(&t, g_prof.ev[k], g_prof.ev[k + 1]);
    if (ms) ms[k] = t;
    if (names) names[k] = g_prof.names[k];
  }
  return ns;
}

uint64_t gmc_launch_count(void) { return g_launches.load(); }

int gmc_read_status(const void* workspace, uint32_t* status, gmc_stream_t stream_) {
  if (!workspace || !status) return GMC_ERR_ARG;
  cudaStream_t st = (cudaStream_t)stream_;
  GMC_TRY(cudaStreamSynchronize(st));
  GMC_TRY(cudaMemcpy(status, workspace, sizeof(uint32_t), cudaMemcpyDeviceToHost));
  return GMC_OK;
}

}  // extern "C"
