// gmc_transport_noalloc: the transport + compaction entry point for callers
// that cannot allocate device memory.
//
// Some callers run where cudaMalloc (or any allocator) is off limits: an
// inference-engine plugin whose enqueue() may only launch work into memory
// the engine already owns, code running while a framework captures a CUDA
// graph (allocation breaks or invalidates the capture), or a serving process
// whose memory pool is sized once at start-up and must never grow.  Those
// callers can still pass their input and output tensors, but not a workspace.
// This variant keeps its scratch (one status word and the per-row RMS of the
// visual states) in a fixed array in the library's own device memory.
//
// The array is a file-scope __device__ variable, so every GPU that loads
// libgmc.so holds it (GMC_NOALLOC_MAX_ROWS floats + 256 bytes) until the
// process exits.  In host code its name is only a host-side stand-in; the
// device address is fetched with cudaGetSymbolAddress on the first call made
// in a given CUDA context (the device's primary context, or whichever
// context is current) and cached for that context.  A context that replaces
// it -- for example the new primary context after cudaDeviceReset -- gets
// its own look-up on its first call.
#include <cuda.h>  // CUcontext: the cache key (the driver entry point is found at run time)

#include <mutex>

#include "common.cuh"
#include "kernels.cuh"

using namespace gmc;

namespace {

constexpr size_t kStatusBytes = 256;  // status word, padded so the row array stays aligned

static __device__ __align__(256) unsigned char
    g_noalloc_scratch[kStatusBytes + sizeof(float) * GMC_NOALLOC_MAX_ROWS];

constexpr int kMaxDevices = 256;
std::mutex g_setup_mu;
struct CachedAddress {
  CUcontext ctx;  // context the address belongs to
  void* addr;
};
CachedAddress g_scratch_addr[kMaxDevices] = {};

using CtxGetCurrentFn = CUresult (*)(CUcontext*);

// cuCtxGetCurrent through the runtime's driver entry point table (the
// library does not link libcuda directly).  nullptr if unavailable.
CtxGetCurrentFn ctx_get_current() {
  static CtxGetCurrentFn fn = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q = cudaDriverEntryPointSymbolNotFound;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) !=
            cudaSuccess ||
        q != cudaDriverEntryPointSuccess) {
      cudaGetLastError();
      return (CtxGetCurrentFn) nullptr;
    }
    return reinterpret_cast<CtxGetCurrentFn>(p);
  }();
  return fn;
}

// Device address of the scratch array in the current context: looked up by
// the first call in a context (cudaGetSymbolAddress also creates the device's
// primary context if none is current yet), reused while that context stays
// current.  Without the driver entry point every call looks it up.
cudaError_t scratch_address(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lk(g_setup_mu);
  CUcontext ctx = nullptr;
  const CtxGetCurrentFn get = ctx_get_current();
  const bool known = get && get(&ctx) == CUDA_SUCCESS && ctx != nullptr;
  CachedAddress& c = g_scratch_addr[dev];
  if (!known || !c.addr || c.ctx != ctx) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess) return e;
    // the look-up made the device's primary context current if none was
    if (get && !known && get(&ctx) != CUDA_SUCCESS) ctx = nullptr;
    c.addr = p;
    c.ctx = ctx;
  }
  *out = c.addr;
  return cudaSuccess;
}

bool ok_align(const void* p, size_t a) { return ((uintptr_t)p % a) == 0; }

}  // namespace

extern "C" int gmc_transport_noalloc(const gmc_problem* prob, const gmc_params* params,
                                     const void* hidden, const void* keys,
                                     const int32_t* pos_ids, const int32_t* support,
                                     const int32_t* assign, const float* weights, int N, int T,
                                     int d, int D, int K, int32_t* out_idx, void* out_hidden,
                                     void* out_kv, int32_t* out_pos, uint32_t* device_status,
                                     gmc_stream_t stream_) {
  // the checks of gmc_transport, plus the size of the fixed scratch
  const int rc = check_problem(prob, N, T, d, D);
  if (rc != GMC_OK) return rc;
  if (K < 1 || K > N) return GMC_ERR_ARG;
  if ((long long)prob->B * N > GMC_NOALLOC_MAX_ROWS) return GMC_ERR_UNSUPPORTED;
  gmc_params p;
  if (params) p = *params; else gmc_default_params(&p);
  if (!params_ok(p)) return GMC_ERR_ARG;
  if (!hidden || !keys || !pos_ids || !support || !assign || !weights || !out_idx ||
      !out_hidden || !out_kv || !out_pos)
    return GMC_ERR_ARG;
  if (!ok_align(hidden, 16) || !ok_align(keys, 16) || !ok_align(out_hidden, 16) ||
      !ok_align(out_kv, 16) || (device_status && !ok_align(device_status, 4)))
    return GMC_ERR_ARG;
  void* base = nullptr;
  cudaError_t e = scratch_address(&base);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return GMC_ERR_CUDA;
  }
  uint32_t* status = device_status ? device_status : reinterpret_cast<uint32_t*>(base);
  float* rmsh = reinterpret_cast<float*>(static_cast<char*>(base) + kStatusBytes);
  cudaStream_t st = (cudaStream_t)stream_;
  Dims dm;
  dm.B = prob->B; dm.N = N; dm.T = T; dm.H = 0; dm.Hkv = prob->Hkv; dm.d = d; dm.D = D;
  dm.K = K; dm.gh = prob->grid_h; dm.gw = prob->grid_w; dm.L = p.landmarks;
  dm.V = 1; dm.I = 1; dm.M = N; dm.dtype = prob->dtype; dm.toff = prob->text_offsets;
  if ((e = cudaMemsetAsync(status, 0, sizeof(uint32_t), st)) != cudaSuccess ||
      (e = launch_rms_rows(dm, hidden, rmsh, status, st)) != cudaSuccess ||
      (e = launch_transport(dm, p, hidden, keys, pos_ids, support, assign, weights, rmsh,
                            nullptr, out_idx, out_hidden, out_kv, out_pos, status, st)) != cudaSuccess) {
    cudaGetLastError();
    return GMC_ERR_CUDA;
  }
  return GMC_OK;
}
