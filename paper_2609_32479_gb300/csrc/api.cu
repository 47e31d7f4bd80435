// Host side of the C-ABI (include/trackfit.h): validation, weight upload,
// workspace, dispatch to the SIMT or tcgen05 kernel path, error counters.
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <new>

#include "trackfit_internal.h"

// The CUDA error behind this thread's last TRACKFIT_ERR_CUDA / ERR_OOM.
static thread_local char g_last_error[160] = "";

void tf_note_cuda(cudaError_t e, const char* where) {
  std::snprintf(g_last_error, sizeof(g_last_error), "%s: %s (%s)", where, cudaGetErrorName(e), cudaGetErrorString(e));
}

int tf_status_from_cuda(cudaError_t e) {
  if (e == cudaSuccess) return TRACKFIT_OK;
  tf_note_cuda(e, "CUDA call");
  if (e == cudaErrorMemoryAllocation) return TRACKFIT_ERR_OOM;
  return TRACKFIT_ERR_CUDA;
}

extern "C" const char* trackfit_last_error(void) { return g_last_error; }

// Allocation bookkeeping for the test hook trackfit_debug_alloc (host side; the
// counters are not meant for concurrent use).
static int64_t g_live_allocs = 0, g_attempted = 0, g_fail_countdown = 0;

cudaError_t tf_malloc(void** p, size_t bytes) {
  ++g_attempted;
  if (g_fail_countdown > 0 && --g_fail_countdown == 0) {
    *p = nullptr;
    return cudaErrorMemoryAllocation;
  }
  const cudaError_t e = cudaMalloc(p, bytes);
  if (e == cudaSuccess) ++g_live_allocs;
  return e;
}

void tf_free(void* p) {
  if (!p) return;
  if (cudaFree(p) == cudaSuccess) --g_live_allocs;
}

extern "C" int64_t trackfit_debug_alloc(int64_t fail_nth, int64_t* attempted) {
  if (attempted) *attempted = g_attempted;
  g_attempted = 0;
  g_fail_countdown = fail_nth > 0 ? fail_nth : 0;
  return g_live_allocs;
}

extern "C" int trackfit_debug_wait_limit(trackfit_t h, int64_t limit_ns, int32_t hold_tile) {
  if (!h) return TRACKFIT_ERR_INVALID_ARG;
  if (h->rows) {   // the packed-row path: the limit only (it has no loader hand-over to hold)
    if (limit_ns < 0 || hold_tile != -1) return limit_ns < 0 || hold_tile < -1 ? TRACKFIT_ERR_INVALID_ARG
                                                                               : TRACKFIT_ERR_UNSUPPORTED;
    return tf_rows_wait_limit(h, limit_ns);
  }
  return tf_tc_wait_limit(h, limit_ns, hold_tile);
}

static bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Fill the shape summary and blob offsets; false if cfg is outside the supported set.
static bool derive(const trackfit_config_t* c, tf_shape* s, tf_blob_off* o) {
  if (!c || c->abi_version != TRACKFIT_ABI_VERSION) return false;
  if (c->n_features < 1 || c->n_features > TRACKFIT_MAX_FEATURES || c->n_fourier != TRACKFIT_MAX_FOURIER) return false;
  const bool attn = c->topology == TRACKFIT_TOPOLOGY_ATTENTION;
  if (c->topology != TRACKFIT_TOPOLOGY_MERGE && c->topology != TRACKFIT_TOPOLOGY_CONCAT && !attn) return false;
  if (c->max_hits < 1 || c->max_hits > TF_MAX_HITS) return false;
  if (c->d_model < 16 || c->d_model > 256 || (c->d_model % 16) != 0) return false;
  if (attn) {
    if (c->d_hidden < 16 || c->d_hidden > 1024 || (c->d_hidden % 16) != 0) return false;
    if (c->n_heads < 1 || (c->d_model % c->n_heads) != 0) return false;
    const int dh = c->d_model / c->n_heads;
    if ((dh % 8) != 0 || dh > 64) return false;
    if (c->pool != TRACKFIT_POOL_MEAN) return false;
  } else if (c->d_hidden != 3 * c->d_model / 2) {
    return false;
  }
  if (c->n_layers < 1 || c->n_layers > TF_MAX_LAYERS) return false;
  if (c->head_hidden != 128) return false;
  if (c->n_quantiles < 1 || c->n_quantiles > 15 || (c->n_quantiles % 2) == 0) return false;
  if (c->precision != TRACKFIT_FP32 && c->precision != TRACKFIT_BF16_PROJ && c->precision != TRACKFIT_FP16_PROJ)
    return false;
  if (c->pool != TRACKFIT_POOL_MEAN && c->pool != TRACKFIT_POOL_ENDPOINTS) return false;
  if (!(c->rms_eps > 0.0f) || !std::isfinite(c->rms_eps)) return false;
  for (int f = 0; f < c->n_features; ++f)
    if (!(c->feat_max[f] > c->feat_min[f]) || !std::isfinite(c->feat_max[f]) || !std::isfinite(c->feat_min[f]))
      return false;
  for (int k = 0; k < TRACKFIT_MAX_FOURIER; ++k)
    if (!std::isfinite(c->fourier_scale[k])) return false;
  s->T = c->max_hits;
  s->F = c->n_features;
  s->K = c->n_fourier;
  s->E = 2 * s->F * s->K;
  s->D = c->d_model;
  s->H = c->d_hidden;
  s->L = c->n_layers;
  s->topology = c->topology;
  s->NH = attn ? c->n_heads : 0;
  s->P = (c->pool == TRACKFIT_POOL_MEAN && c->topology != TRACKFIT_TOPOLOGY_CONCAT) ? s->D : 2 * s->H;
  s->Hh = c->head_hidden;
  s->NQ = c->n_quantiles;
  s->Q = 5 * c->n_quantiles;
  s->precision = c->precision;
  s->pool = c->pool;
  s->rms_eps = c->rms_eps;
  for (int f = 0; f < s->F; ++f) {
    s->feat_min[f] = c->feat_min[f];
    const double inv = 1.0 / ((double)c->feat_max[f] - (double)c->feat_min[f]);
    s->feat_inv_range[f] = (float)inv;
    s->feat_inv_lo[f] = (float)(inv - (double)s->feat_inv_range[f]);
    s->feat_min_d[f] = c->feat_min[f];
    s->feat_range_d[f] = (double)c->feat_max[f] - (double)c->feat_min[f];
  }
  for (int k = 0; k < s->K; ++k) s->scale[k] = c->fourier_scale[k];
  const size_t D = s->D, H = s->H, E = s->E, P = s->P, Hh = s->Hh, Q = s->Q;
  size_t p = 0;
  o->emb_w1 = p; p += D * E;
  o->emb_b1 = p; p += D;
  o->emb_w2 = p; p += D * D;
  o->emb_b2 = p; p += D;
  for (int l = 0; l < s->L; ++l) {
    tf_layer_off& y = o->layer[l];
    y.g2 = 0;
    if (attn) {   // g_1 W_qkv b_qkv W_o b_o g_2 W_1 b_1 W_2 b_2
      y.g = p; p += D;
      y.w_in = p; p += 3 * D * D;
      y.b_in = p; p += 3 * D;
      y.w_m = p; p += D * D;
      y.b_m = p; p += D;
      y.g2 = p; p += D;
      y.w1 = p; p += H * D;
      y.b1 = p; p += H;
      y.w2 = p; p += D * H;
      y.b2 = p; p += D;
      continue;
    }
    if (s->topology == TRACKFIT_TOPOLOGY_CONCAT) {   // W_in[4H][I_l] b_in[4H]
      const size_t I = l == 0 ? D : 2 * H;
      y.g = y.w_m = y.b_m = y.w1 = y.b1 = y.w2 = y.b2 = 0;
      y.w_in = p; p += 4 * H * I;
      y.b_in = p; p += 4 * H;
      continue;
    }
    y.g = p; p += D;
    y.w_in = p; p += (4 * H + D) * D;
    y.b_in = p; p += 4 * H + D;
    y.w_m = p; p += D * 2 * H;
    y.b_m = p; p += D;
    y.w1 = p; p += D * D;
    y.b1 = p; p += D;
    y.w2 = p; p += D * D;
    y.b2 = p; p += D;
  }
  o->head_g = p; p += P;
  o->head_w1 = p; p += Hh * P;
  o->head_b1 = p; p += Hh;
  o->head_w2 = p; p += Q * Hh;
  o->head_b2 = p; p += Q;
  o->total = p;
  return true;
}

extern "C" size_t trackfit_weight_count(const trackfit_config_t* cfg) {
  tf_shape s;
  tf_blob_off o;
  if (!derive(cfg, &s, &o)) return 0;
  return o.total;
}

extern "C" const char* trackfit_strerror(int status) {
  switch (status) {
    case TRACKFIT_OK: return "ok";
    case TRACKFIT_ERR_INVALID_ARG: return "invalid argument";
    case TRACKFIT_ERR_UNSUPPORTED: return "unsupported configuration";
    case TRACKFIT_ERR_CUDA: return "CUDA error";
    case TRACKFIT_ERR_OOM: return "out of device memory";
    case TRACKFIT_ERR_BAD_HITS: return "tracks with hit counts outside [1, max_hits]";
    case TRACKFIT_ERR_TIMEOUT: return "a bounded device wait expired";
    default: return "unknown status";
  }
}

static void prof_collect(trackfit_ctx* h) {
  for (int i = 0; i < h->prof_n; ++i) {
    float ms = 0.0f;
    cudaEventSynchronize(h->prof_ev[2 * i + 1]);
    if (cudaEventElapsedTime(&ms, h->prof_ev[2 * i], h->prof_ev[2 * i + 1]) == cudaSuccess) h->prof_ms += ms;
    ++h->prof_launches;
  }
  h->prof_n = 0;
}

void tf_prof_begin(trackfit_ctx* h, cudaStream_t st) {
  if (!h->prof_on) return;
  if (h->prof_n == 64) prof_collect(h);
  cudaEventRecord(h->prof_ev[2 * h->prof_n], st);
}

void tf_prof_end(trackfit_ctx* h, cudaStream_t st) {
  if (!h->prof_on) return;
  cudaEventRecord(h->prof_ev[2 * h->prof_n + 1], st);
  ++h->prof_n;
}

extern "C" int trackfit_profile(trackfit_t h, int enable) {
  if (!h) return TRACKFIT_ERR_INVALID_ARG;
  if (enable && !h->prof_on) {
    for (int i = 0; i < 2 * 64; ++i)
      if (cudaEventCreate(&h->prof_ev[i]) != cudaSuccess) return TRACKFIT_ERR_CUDA;
  }
  if (!enable && h->prof_on) {
    prof_collect(h);
    for (int i = 0; i < 2 * 64; ++i) cudaEventDestroy(h->prof_ev[i]);
  }
  h->prof_on = enable ? 1 : 0;
  h->prof_n = 0;
  h->prof_ms = 0.0;
  h->prof_launches = 0;
  return TRACKFIT_OK;
}

extern "C" int trackfit_profile_read(trackfit_t h, double* kernel_ms, int64_t* launches) {
  if (!h || !kernel_ms || !launches) return TRACKFIT_ERR_INVALID_ARG;
  if (h->prof_on) prof_collect(h);
  *kernel_ms = h->prof_ms;
  *launches = h->prof_launches;
  h->prof_ms = 0.0;
  h->prof_launches = 0;
  return TRACKFIT_OK;
}

extern "C" void trackfit_destroy(trackfit_t h) {
  if (!h) return;
  if (h->prof_on) trackfit_profile(h, 0);
  tf_tc_destroy(h);
  tf_rows_destroy(h);
  tf_free(h->d_w);
  tf_free(h->d_err);
  tf_free(h->ws);
  tf_free(h->pk_n);
  tf_free(h->st_hits);
  tf_free(h->st_n);
  tf_free(h->st_out);
  for (int i = 0; i < h->cp_nev; ++i) cudaEventDestroy(h->cp_ev[i]);
  if (h->cp_stream) cudaStreamDestroy(h->cp_stream);
  delete h;
}

extern "C" int trackfit_create(const trackfit_config_t* cfg, const float* weights, size_t n_weights,
                               trackfit_t* out) {
  tf_nvtx_range nvtx_range("trackfit_create");
  if (!cfg || !weights || !out) return TRACKFIT_ERR_INVALID_ARG;
  tf_shape s;
  tf_blob_off o;
  if (cfg->abi_version != TRACKFIT_ABI_VERSION) return TRACKFIT_ERR_UNSUPPORTED;
  if (!derive(cfg, &s, &o)) return TRACKFIT_ERR_UNSUPPORTED;
  if (n_weights != o.total) return TRACKFIT_ERR_INVALID_ARG;
  trackfit_ctx* h = new (std::nothrow) trackfit_ctx();
  if (!h) return TRACKFIT_ERR_OOM;
  h->cfg = *cfg;
  h->s = s;
  h->off = o;
  h->path = TF_PATH_SIMT;
  int st = tf_status_from_cuda(tf_malloc((void**)&h->d_w, o.total * sizeof(float)));
  if (st == TRACKFIT_OK) st = tf_status_from_cuda(cudaMemcpy(h->d_w, weights, o.total * sizeof(float), cudaMemcpyHostToDevice));
  if (st == TRACKFIT_OK) st = tf_status_from_cuda(tf_malloc((void**)&h->d_err, 4 * sizeof(unsigned long long)));
  if (st == TRACKFIT_OK) st = tf_status_from_cuda(cudaMemset(h->d_err, 0, 4 * sizeof(unsigned long long)));
  if (st == TRACKFIT_OK) st = tf_simt_workspace(h);
  if (st == TRACKFIT_OK) st = tf_status_from_cuda(tf_malloc((void**)&h->pk_n, TF_PACKED_CHUNK * sizeof(int32_t)));
  if (st == TRACKFIT_OK && tf_tc_supported(s)) {
    st = tf_tc_create(h, weights);
    if (st == TRACKFIT_OK) h->path = TF_PATH_TC;
  } else if (st == TRACKFIT_OK && tf_rows_supported(s)) {
    st = tf_rows_create(h, weights);
    if (st == TRACKFIT_OK) h->path = TF_PATH_ROWS;
  }
  if (st == TRACKFIT_OK) st = tf_status_from_cuda(cudaDeviceSynchronize());
  if (st != TRACKFIT_OK) {
    trackfit_destroy(h);
    return st;
  }
  *out = h;
  return TRACKFIT_OK;
}

extern "C" const char* trackfit_path_name(trackfit_t h) {
  if (!h) return "none";
  const bool tc = h->path == TF_PATH_TC, rows = h->path == TF_PATH_ROWS;
  if (h->s.precision == TRACKFIT_FP16_PROJ) return tc ? "tcgen05-fp16" : rows ? "tcgen05-rows-fp16" : "simt-fp16";
  if (h->s.precision == TRACKFIT_BF16_PROJ) return tc ? "tcgen05-bf16" : rows ? "tcgen05-rows-bf16" : "simt-bf16";
  return "simt-fp32";
}

extern "C" int trackfit_set_path(trackfit_t h, int path) {
  if (!h) return TRACKFIT_ERR_INVALID_ARG;
  if (path == 1) {
    h->path = TF_PATH_SIMT;
    return TRACKFIT_OK;
  }
  if (path != 0) return TRACKFIT_ERR_INVALID_ARG;
  h->path = (h->tc != nullptr) ? TF_PATH_TC : (h->rows != nullptr) ? TF_PATH_ROWS : TF_PATH_SIMT;
  return TRACKFIT_OK;
}

extern "C" int trackfit_forward_ex(trackfit_t h, const float* hits, const int32_t* n_hits, int64_t n_tracks,
                                   float* out_params, float* out_q, float* out_pool, void* stream) {
  tf_nvtx_range nvtx_range("trackfit_forward_ex");
  if (!h || !hits || !n_hits || !out_params) return TRACKFIT_ERR_INVALID_ARG;
  if (n_tracks <= 0) return TRACKFIT_ERR_INVALID_ARG;
  if (!aligned16(hits) || !aligned16(out_params) || !aligned16(n_hits)) return TRACKFIT_ERR_INVALID_ARG;
  if ((out_q && !aligned16(out_q)) || (out_pool && !aligned16(out_pool))) return TRACKFIT_ERR_INVALID_ARG;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (h->path == TF_PATH_TC) return tf_tc_forward(h, hits, n_hits, n_tracks, out_params, out_q, out_pool, st);
  if (h->path == TF_PATH_ROWS) return tf_rows_forward(h, hits, n_hits, n_tracks, out_params, out_q, out_pool, st);
  return tf_simt_forward(h, hits, n_hits, n_tracks, out_params, out_q, out_pool, st);
}

// Per-track hit counts of a packed batch: n_b = offsets[b + 1] - offsets[b] when
// the track's rows lie inside the hit array and 1 <= n_b <= T, else 0 (an
// invalid track: NaN row, counted, and none of its rows read).
__global__ void counts_from_offsets(const int64_t* __restrict__ offs, int64_t B, int64_t n_rows, int T,
                                    int32_t* __restrict__ n) {
  const int64_t b = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (b >= B) return;
  const int64_t lo = offs[b], hi = offs[b + 1], d = hi - lo;
  n[b] = (lo >= 0 && hi <= n_rows && d >= 1 && d <= T) ? (int32_t)d : 0;
}

extern "C" int trackfit_forward_packed(trackfit_t h, const float* hits, int64_t n_hit_rows, const int64_t* offsets,
                                       int64_t n_tracks, float* out_params, void* stream) {
  tf_nvtx_range nvtx_range("trackfit_forward_packed");
  if (!h || !hits || !offsets || !out_params || n_tracks <= 0 || n_hit_rows < 0) return TRACKFIT_ERR_INVALID_ARG;
  if (!aligned16(hits) || !aligned16(offsets) || !aligned16(out_params)) return TRACKFIT_ERR_INVALID_ARG;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  for (int64_t c0 = 0; c0 < n_tracks; c0 += TF_PACKED_CHUNK) {
    const int64_t nb = (n_tracks - c0 < TF_PACKED_CHUNK) ? n_tracks - c0 : TF_PACKED_CHUNK;
    counts_from_offsets<<<(unsigned)((nb + 255) / 256), 256, 0, st>>>(offsets + c0, nb, n_hit_rows, h->s.T, h->pk_n);
    if (cudaPeekAtLastError() != cudaSuccess) return TRACKFIT_ERR_CUDA;
    const int r =
        h->path == TF_PATH_TC
            ? tf_tc_forward(h, hits, h->pk_n, nb, out_params + c0 * 5, nullptr, nullptr, st, offsets + c0)
        : h->path == TF_PATH_ROWS
            ? tf_rows_forward(h, hits, h->pk_n, nb, out_params + c0 * 5, nullptr, nullptr, st, offsets + c0)
            : tf_simt_forward(h, hits, h->pk_n, nb, out_params + c0 * 5, nullptr, nullptr, st, offsets + c0);
    if (r != TRACKFIT_OK) return r;
  }
  return TRACKFIT_OK;
}

extern "C" int trackfit_forward(trackfit_t h, const float* hits, const int32_t* n_hits, int64_t n_tracks,
                                float* out_params, void* stream) {
  return trackfit_forward_ex(h, hits, n_hits, n_tracks, out_params, nullptr, nullptr, stream);
}

extern "C" int trackfit_forward_host(trackfit_t h, const float* hits_host, const int32_t* n_hits_host,
                                     int64_t n_tracks, float* out_host, void* stream) {
  tf_nvtx_range nvtx_range("trackfit_forward_host");
  if (!h || !hits_host || !n_hits_host || !out_host || n_tracks <= 0) return TRACKFIT_ERR_INVALID_ARG;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const size_t row = (size_t)h->s.T * 5;
  if (n_tracks > h->st_cap) {
    cudaStreamSynchronize(st);
    tf_free(h->st_hits);
    tf_free(h->st_n);
    tf_free(h->st_out);
    h->st_hits = nullptr;
    h->st_n = nullptr;
    h->st_out = nullptr;
    h->st_cap = 0;
    int s1 = tf_status_from_cuda(tf_malloc((void**)&h->st_hits, n_tracks * row * sizeof(float)));
    if (s1 == TRACKFIT_OK) s1 = tf_status_from_cuda(tf_malloc((void**)&h->st_n, ((n_tracks + 3) / 4) * 4 * sizeof(int32_t)));
    if (s1 == TRACKFIT_OK) s1 = tf_status_from_cuda(tf_malloc((void**)&h->st_out, n_tracks * 5 * sizeof(float)));
    if (s1 != TRACKFIT_OK) {   // keep nothing of a failed set-up
      tf_free(h->st_hits);
      tf_free(h->st_n);
      tf_free(h->st_out);
      h->st_hits = nullptr;
      h->st_n = nullptr;
      h->st_out = nullptr;
      return s1;
    }
    h->st_cap = n_tracks;
  }
  // Copies overlap the compute: chunk k + 1's inputs travel on the handle's copy
  // stream while chunk k runs on the caller's stream, and each chunk's outputs
  // travel back behind it.
  if (!h->cp_stream) {
    if (cudaStreamCreateWithFlags(&h->cp_stream, cudaStreamNonBlocking) != cudaSuccess) {
      h->cp_stream = nullptr;
      return TRACKFIT_ERR_CUDA;
    }
    for (int i = 0; i < TF_HOST_EVENTS; ++i) {
      if (cudaEventCreateWithFlags(&h->cp_ev[i], cudaEventDisableTiming) != cudaSuccess) {   // all or nothing
        for (int j = 0; j < h->cp_nev; ++j) cudaEventDestroy(h->cp_ev[j]);
        h->cp_nev = 0;
        cudaStreamDestroy(h->cp_stream);
        h->cp_stream = nullptr;
        return TRACKFIT_ERR_CUDA;
      }
      ++h->cp_nev;
    }
  }
  cudaStream_t cs = h->cp_stream;
  cudaEvent_t* ev = h->cp_ev;
  const int64_t chunk = TF_HOST_CHUNK;
  const int64_t n_chunks = (n_tracks + chunk - 1) / chunk;
  // chunk k's events: in(k) (its inputs have landed), done(k) (its outputs are
  // computed), from a ring (each is waited for before it is recorded again)
  auto ev_in = [&](int64_t k) { return ev[1 + (2 * k) % (TF_HOST_EVENTS - 2)]; };
  auto ev_done = [&](int64_t k) { return ev[2 + (2 * k) % (TF_HOST_EVENTS - 2)]; };
  auto send = [&](int64_t k) -> cudaError_t {   // chunk k's inputs, on the copy stream
    const int64_t c0 = k * chunk, nb = (n_tracks - c0 < chunk) ? n_tracks - c0 : chunk;
    cudaError_t r = cudaMemcpyAsync(h->st_hits + c0 * row, hits_host + c0 * row, nb * row * sizeof(float),
                                    cudaMemcpyHostToDevice, cs);
    if (r == cudaSuccess)
      r = cudaMemcpyAsync(h->st_n + c0, n_hits_host + c0, nb * sizeof(int32_t), cudaMemcpyHostToDevice, cs);
    if (r == cudaSuccess) r = cudaEventRecord(ev_in(k), cs);
    return r;
  };
  // the staging buffers may still be read by earlier work on the caller's stream
  cudaError_t e = cudaEventRecord(ev[0], st);
  if (e == cudaSuccess) e = cudaStreamWaitEvent(cs, ev[0], 0);
  if (e == cudaSuccess) e = send(0);
  for (int64_t k = 0; k < n_chunks && e == cudaSuccess; ++k) {
    // chunk k + 1's inputs are queued on the copy stream before that stream waits
    // for chunk k's outputs, so they travel while chunk k computes
    if (k + 1 < n_chunks) e = send(k + 1);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(st, ev_in(k), 0);
    if (e != cudaSuccess) break;
    const int64_t c0 = k * chunk, nb = (n_tracks - c0 < chunk) ? n_tracks - c0 : chunk;
    const int r = trackfit_forward(h, h->st_hits + c0 * row, h->st_n + c0, nb, h->st_out + c0 * 5, stream);
    if (r != TRACKFIT_OK) {
      cudaStreamSynchronize(cs);
      return r;
    }
    e = cudaEventRecord(ev_done(k), st);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(cs, ev_done(k), 0);
    if (e == cudaSuccess)
      e = cudaMemcpyAsync(out_host + c0 * 5, h->st_out + c0 * 5, nb * 5 * sizeof(float), cudaMemcpyDeviceToHost, cs);
  }
  const cudaError_t e2 = cudaStreamSynchronize(cs);
  if (e == cudaSuccess) e = e2;
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return tf_status_from_cuda(e);
  // the results are only as good as the device's own checks: read (and reset)
  // the error counters, as trackfit_device_errors does
  int64_t n_bad = 0;
  return trackfit_device_errors(h, stream, &n_bad);
}

extern "C" int trackfit_device_errors(trackfit_t h, void* stream, int64_t* n_bad) {
  if (!h || !n_bad) return TRACKFIT_ERR_INVALID_ARG;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  unsigned long long v[4] = {0, 0, 0, 0};
  cudaError_t e = cudaMemcpyAsync(v, h->d_err, sizeof(v), cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  if (e == cudaSuccess) e = cudaMemsetAsync(h->d_err, 0, sizeof(v), st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return TRACKFIT_ERR_CUDA;
  *n_bad = (int64_t)v[0];
  if (v[1] != 0) return TRACKFIT_ERR_TIMEOUT;
  return v[0] ? TRACKFIT_ERR_BAD_HITS : TRACKFIT_OK;
}

extern "C" int trackfit_debug_scan(const float* a, const float* b, const float* x, const int32_t* n_hits,
                                   int64_t n_tracks, int32_t T, int32_t C, float* h_fwd, float* h_bwd,
                                   void* stream) {
  if (!a || !b || !x || !n_hits || !h_fwd || !h_bwd) return TRACKFIT_ERR_INVALID_ARG;
  if (n_tracks <= 0 || T < 1 || T > TF_MAX_HITS || C < 1) return TRACKFIT_ERR_INVALID_ARG;
  return tf_simt_debug_scan(a, b, x, n_hits, n_tracks, T, C, h_fwd, h_bwd,
                            reinterpret_cast<cudaStream_t>(stream));
}

extern "C" int trackfit_debug_schedule(const trackfit_config_t* cfg, int64_t* counts, int32_t n_counts,
                                       uint8_t* codes, int64_t codes_cap) {
  if (!cfg || !counts) return TRACKFIT_ERR_INVALID_ARG;
  tf_shape s;
  tf_blob_off o;
  if (!derive(cfg, &s, &o)) return TRACKFIT_ERR_UNSUPPORTED;
  if (!tf_tc_supported(s)) return TRACKFIT_ERR_UNSUPPORTED;
  return tf_tc_schedule_counts(s, counts, n_counts, codes, codes_cap);
}

extern "C" int trackfit_debug_umma(trackfit_t h, const uint16_t* A, const uint16_t* Bkn, int32_t K, float* D,
                                   void* stream) {
  if (!h || !A || !Bkn || !D) return TRACKFIT_ERR_INVALID_ARG;
  if (!aligned16(A) || !aligned16(Bkn) || !aligned16(D)) return TRACKFIT_ERR_INVALID_ARG;
  return tf_tc_probe(h, A, Bkn, K, D, reinterpret_cast<cudaStream_t>(stream));
}

// Validation and blob offsets for callers outside this file (no-allocation entry point).
bool tf_derive(const trackfit_config_t* c, tf_shape* s, tf_blob_off* o) { return derive(c, s, o); }
