// Forward pass that allocates no device memory.  Meant for callers that cannot
// call cudaMalloc themselves -- for instance code running inside a framework or
// an allocator-owned process where every device allocation must go through a
// pool it does not control, or a host thread that must not synchronise the
// device the way cudaMalloc can.  It runs the SIMT (CUDA-core) kernels with the
// caller's device weights, and takes all of its workspace from one file-scope
// device array that every GPU loading this library holds until the process
// exits.
#include <mutex>

#include "trackfit_internal.h"

// SIMT workspace (chunks of whole tracks) followed by the error counters.
#define TF_NOALLOC_SCRATCH_BYTES (32u << 20)
static __device__ __align__(256) unsigned char g_noalloc_scratch[TF_NOALLOC_SCRATCH_BYTES];

bool tf_derive(const trackfit_config_t* c, tf_shape* s, tf_blob_off* o);
size_t tf_simt_bytes_per_track(const tf_shape& s);
int tf_simt_forward_explicit(const tf_shape& s, const tf_blob_off& o, const float* W, float* ws, int64_t ws_tracks,
                             unsigned long long* err, const float* hits, const int32_t* n_hits, int64_t B,
                             float* out, cudaStream_t st);

namespace {
constexpr int kMaxDevices = 64;
std::mutex g_mu;
void* g_addr[kMaxDevices] = {nullptr};

// Device address of the scratch array on the current device.  Host code only
// sees a host-side stand-in for the symbol, so the address is looked up once
// per device (with that device current) and cached.
int scratch_address(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return TRACKFIT_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_addr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return TRACKFIT_ERR_CUDA;
    g_addr[dev] = p;
  }
  *out = g_addr[dev];
  return TRACKFIT_OK;
}
}  // namespace

extern "C" int trackfit_forward_noalloc(const trackfit_config_t* cfg, const float* weights, const float* hits,
                                        const int32_t* n_hits, int64_t n_tracks, float* out_params,
                                        void* stream) {
  tf_nvtx_range nvtx_range("trackfit_forward_noalloc");
  tf_shape s;
  tf_blob_off o;
  if (!cfg || !weights || !hits || !n_hits || !out_params || n_tracks <= 0) return TRACKFIT_ERR_INVALID_ARG;
  if (!tf_derive(cfg, &s, &o)) return TRACKFIT_ERR_UNSUPPORTED;
  const uintptr_t mis = reinterpret_cast<uintptr_t>(hits) | reinterpret_cast<uintptr_t>(out_params) |
                        reinterpret_cast<uintptr_t>(n_hits) | reinterpret_cast<uintptr_t>(weights);
  if (mis & 15u) return TRACKFIT_ERR_INVALID_ARG;
  const size_t counter_bytes = 256;
  const size_t per_track = tf_simt_bytes_per_track(s);
  const int64_t fit = (int64_t)((TF_NOALLOC_SCRATCH_BYTES - counter_bytes) / per_track);
  if (fit < 1) return TRACKFIT_ERR_UNSUPPORTED;   // one track's workspace exceeds the array
  int64_t chunk = fit;
  if (chunk > 65535) chunk = 65535;
  if (chunk * s.T > 65535LL * 64) chunk = 65535LL * 64 / s.T;
  void* base = nullptr;
  int st = scratch_address(&base);
  if (st != TRACKFIT_OK) return st;
  cudaStream_t cs = reinterpret_cast<cudaStream_t>(stream);
  unsigned long long* err = reinterpret_cast<unsigned long long*>(static_cast<unsigned char*>(base) +
                                                                  TF_NOALLOC_SCRATCH_BYTES - counter_bytes);
  // the array keeps the previous call's contents: the counter must start at zero
  if (cudaMemsetAsync(err, 0, sizeof(unsigned long long), cs) != cudaSuccess) return TRACKFIT_ERR_CUDA;
  return tf_simt_forward_explicit(s, o, weights, static_cast<float*>(base), chunk, err, hits, n_hits, n_tracks,
                                  out_params, cs);
}
