// Internal declarations shared by the host API and the kernel translation units.
#pragma once

#include <cuda_runtime.h>
#include <nvtx3/nvToolsExt.h>
#include <stdint.h>
#include <stddef.h>

#include "trackfit.h"

// An NVTX range over an entry point's host-side work (its launches included), so
// that timeline tools show each call; with no tool attached a push and a pop cost
// a few instructions.
struct tf_nvtx_range {
  explicit tf_nvtx_range(const char* name) { nvtxRangePushA(name); }
  ~tf_nvtx_range() { nvtxRangePop(); }
  tf_nvtx_range(const tf_nvtx_range&) = delete;
  tf_nvtx_range& operator=(const tf_nvtx_range&) = delete;
};

#define TF_MAX_LAYERS 16
#define TF_MAX_HITS 64
#define TF_PACKED_CHUNK 1048576
#define TF_HOST_CHUNK 262144  // tracks per copy / compute step of trackfit_forward_host
#define TF_HOST_EVENTS 10

// Offsets (in floats) of every tensor inside the fp32 weight blob.
// ATTENTION layers reuse the names: g = g_1, w_in/b_in = W_qkv/b_qkv, w_m/b_m =
// W_o/b_o, g2 = g_2, w1/b1 and w2/b2 the MLP.
struct tf_layer_off {
  size_t g, w_in, b_in, w_m, b_m, w1, b1, w2, b2, g2;
};
struct tf_blob_off {
  size_t emb_w1, emb_b1, emb_w2, emb_b2;
  tf_layer_off layer[TF_MAX_LAYERS];
  size_t head_g, head_w1, head_b1, head_w2, head_b2;
  size_t total;
};

// Shape summary derived from the public config.
struct tf_shape {
  int T, F, K, E, D, H, L, P, Hh, NQ, Q, precision, pool, topology, NH;
  float rms_eps;
  // 1 / (max - min) as the unevaluated sum feat_inv_range + feat_inv_lo of two floats
  float feat_min[TRACKFIT_MAX_FEATURES], feat_inv_range[TRACKFIT_MAX_FEATURES], feat_inv_lo[TRACKFIT_MAX_FEATURES];
  double feat_min_d[TRACKFIT_MAX_FEATURES], feat_range_d[TRACKFIT_MAX_FEATURES];
  float scale[TRACKFIT_MAX_FOURIER];
};

struct tf_tc_state;    // tcgen05 fused path (tc_forward.cu)
struct tf_rows_state;  // tcgen05 packed-row path (rows.cu)

enum { TF_PATH_SIMT = 0, TF_PATH_TC = 1, TF_PATH_ROWS = 2 };

struct trackfit_ctx {
  trackfit_config_t cfg;
  tf_shape s;
  tf_blob_off off;
  int path;
  float* d_w;                    // fp32 weight blob on the device
  unsigned long long* d_err;     // [0] tracks with bad n_hits, [1] expired bounded waits
  // SIMT workspace (one chunk of tracks at a time)
  float* ws;
  size_t ws_bytes;
  int64_t ws_tracks;
  // packed input: per-track hit counts derived from the offsets, one chunk of
  // TF_PACKED_CHUNK tracks at a time
  int32_t* pk_n;
  // host-buffer staging
  float* st_hits;
  int32_t* st_n;
  float* st_out;
  int64_t st_cap;
  cudaStream_t cp_stream;        // copies of trackfit_forward_host (created on first use)
  cudaEvent_t cp_ev[TF_HOST_EVENTS];
  int cp_nev;
  tf_tc_state* tc;
  tf_rows_state* rows;
  // optional timing of the main compute kernel (trackfit_profile)
  int prof_on;
  int prof_n;
  cudaEvent_t prof_ev[2 * 64];
  double prof_ms;
  int64_t prof_launches;
};

// Record the start / end of the main kernel of one forward when profiling is on.
void tf_prof_begin(trackfit_ctx* h, cudaStream_t st);
void tf_prof_end(trackfit_ctx* h, cudaStream_t st);

// simt.cu
int tf_simt_workspace(trackfit_ctx* h);
// offs (may be null): packed input, track b's hits are rows offs[b] .. of hits
int tf_simt_forward(trackfit_ctx* h, const float* hits, const int32_t* n_hits, int64_t B,
                    float* out, float* out_q, float* out_pool, cudaStream_t st, const int64_t* offs = nullptr);
int tf_simt_head(const tf_shape& s, const tf_blob_off& o, const float* W, const float* pooled,
                 const int32_t* n_hits, int64_t B, float* out, float* out_q, float* out_pool,
                 unsigned long long* err, cudaStream_t st);
int tf_simt_head_batched(const tf_shape& s, const tf_blob_off& o, const float* W, const float* pooled,
                         const int32_t* n_hits, int64_t B, float* ws, float* out, float* out_q, float* out_pool,
                         unsigned long long* err, cudaStream_t st);
int tf_simt_debug_scan(const float* a, const float* b, const float* x, const int32_t* n_hits,
                       int64_t B, int T, int C, float* hf, float* hb, cudaStream_t st);

// tc_forward.cu
bool tf_tc_supported(const tf_shape& s);
int tf_tc_schedule_counts(const tf_shape& s, int64_t* counts, int n, uint8_t* codes, int64_t cap);
int tf_tc_create(trackfit_ctx* h, const float* host_w);
void tf_tc_destroy(trackfit_ctx* h);
int tf_tc_forward(trackfit_ctx* h, const float* hits, const int32_t* n_hits, int64_t B,
                  float* out, float* out_q, float* out_pool, cudaStream_t st, const int64_t* offs = nullptr);

int tf_tc_wait_limit(trackfit_ctx* h, int64_t limit_ns, int hold_tile);
int tf_tc_probe(trackfit_ctx* h, const uint16_t* A, const uint16_t* Bkn, int K, float* D, cudaStream_t st);

// rows.cu
bool tf_rows_supported(const tf_shape& s);
int tf_rows_create(trackfit_ctx* h, const float* host_w);
void tf_rows_destroy(trackfit_ctx* h);
int tf_rows_forward(trackfit_ctx* h, const float* hits, const int32_t* n_hits, int64_t B, float* out,
                    float* out_q, float* out_pool, cudaStream_t st, const int64_t* offs = nullptr);
int tf_rows_wait_limit(trackfit_ctx* h, int64_t limit_ns);

// api.cu
int tf_status_from_cuda(cudaError_t e);
// Record e as the calling thread's last CUDA error (trackfit_last_error), with
// where it happened.
void tf_note_cuda(cudaError_t e, const char* where);
// Every device allocation of a handle goes through these two (counted; a test
// hook can make one fail as if the device were out of memory).  tf_free
// accepts null.
cudaError_t tf_malloc(void** p, size_t bytes);
void tf_free(void* p);
