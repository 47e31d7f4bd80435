/*
 * trackfit.h -- C-ABI of the GB300 (sm_103a) batched inference library for the
 * bidirectional minGRU track-fit encoder of "Fast and Precise Learned
 * Charged-Particle Trajectory Regression at the LHC".
 *
 * Problem statement (Sec. 3, first paragraph): the model maps the hit sequence
 * of one track, ordered by measurement time, to the five perigee parameters
 * (d0, z0, phi, theta, q/p) at the point of closest approach to the beam axis.
 * This library runs that map for a batch of independent tracks (Sec. 4,
 * "embarrassingly parallel across tracks").  The encoder computed is:
 *
 *   per hit   : u = min-max normalised features, e = [sin(pi s_k u_f), cos(pi s_k u_f)]
 *               (Sec. 3.2, 16-scale Fourier featurisation), x0 = W_e2 SiLU(W_e1 e + b_e1) + b_e2
 *   per layer : x_hat = RMSNorm(x) g ; [p_zf, n_f, p_zb, n_b, p_g] = W_in x_hat + b_in
 *               forward and reverse scans h_t = h_{t-1} + z_t (n_t - h_{t-1}), z = sigma(p_z)
 *               (Sec. 3.2, Eq. 2), masked to the track's hits, zero initial state
 *               x' = x + (W_m [h_f; h_b] + b_m) * sigma(p_g)
 *               x  = x' + W_2 SiLU(W_1 x' + b_1) + b_2        (padded hits set to 0)
 *   per track : p = mean of x over the track's hits (or, pool = ENDPOINTS, the
 *               forward state at the last hit and the reverse state at the first
 *               hit, Sec. 3.2); q = W_h2 SiLU(W_h1 RMSNorm(p) g_h + b_h1) + b_h2,
 *               35 = 5 parameters x 7 quantiles; output = the median quantile
 *               (Sec. 3.2-3.3).
 *
 * Precision: TRACKFIT_FP32 computes everything in fp32.  TRACKFIT_BF16_PROJ rounds
 * the operands of every per-hit matrix product (Fourier vector, embedding hidden,
 * x_hat, [h_f; h_b], x', MLP hidden, and the weights of those products) to bf16
 * and accumulates in fp32; gates, scan state, residual stream, pooling and the
 * head stay fp32 (Sec. 3.5: reduced-precision projections, fp32 recurrence).
 * TRACKFIT_FP16_PROJ is the same with fp16 operands, the format Sec. 3.5 names.
 *
 * Threading: a handle may be used from one host thread at a time and on one
 * stream at a time (it owns a device workspace).  Different handles are
 * independent.
 */
#ifndef TRACKFIT_H
#define TRACKFIT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define TRACKFIT_ABI_VERSION 3
#define TRACKFIT_MAX_FEATURES 16
#define TRACKFIT_MAX_FOURIER 16

typedef enum {
  TRACKFIT_OK = 0,
  TRACKFIT_ERR_INVALID_ARG = 1,  /* NULL pointer, n_tracks <= 0, misaligned pointer, bad sizes */
  TRACKFIT_ERR_UNSUPPORTED = 2,  /* configuration outside what the kernels implement */
  TRACKFIT_ERR_CUDA = 3,         /* a CUDA runtime call or kernel launch failed */
  TRACKFIT_ERR_OOM = 4,          /* device allocation failed (create only) */
  TRACKFIT_ERR_BAD_HITS = 5,     /* device-side: tracks with n_hits outside [1, max_hits] */
  TRACKFIT_ERR_TIMEOUT = 6       /* device-side: a bounded wait inside a kernel expired */
} trackfit_status;

typedef enum { TRACKFIT_FP32 = 0, TRACKFIT_BF16_PROJ = 1, TRACKFIT_FP16_PROJ = 2 } trackfit_precision;
typedef enum { TRACKFIT_POOL_MEAN = 0, TRACKFIT_POOL_ENDPOINTS = 1 } trackfit_pool;
/* Layer topology.  MERGE: each layer pre-norms its input, projects it to the
 * gates, candidates and an output gate, scans, merges the two directions with
 * the output gate and an MLP into a d_model-wide residual stream (the form given
 * with the task).  CONCAT: the paper's own (Sec. 3.2): each layer projects its
 * input to the forward and reverse gates and candidates, scans, and the two
 * directions' states, concatenated (2 d_hidden wide), are the next layer's input
 * and the readout's; no norm inside the encoder.  ATTENTION: the Transformer of
 * the paper's encoder comparison (App. A.3, Tab. A.1): per layer, pre-norm
 * multi-head self-attention over the track's own hits and a pre-norm SiLU MLP of
 * hidden width d_hidden, each added to a d_model-wide residual stream; no
 * positional encoding; mean pooling. */
typedef enum {
  TRACKFIT_TOPOLOGY_MERGE = 0,
  TRACKFIT_TOPOLOGY_CONCAT = 1,
  TRACKFIT_TOPOLOGY_ATTENTION = 2
} trackfit_topology;

/* Encoder shape.  Supported: abi_version = 3, 1 <= n_features <= 16 per hit (the
 * task's configs use 5: x, y, z [mm], r [mm], phi [rad]; the paper's model 15, its
 * last three the seed features of trackfit_seed), n_fourier = 16, 1 <= max_hits
 * <= 64, d_model in {16, 32, ..., 256} (multiple of 16), d_hidden = 3 * d_model / 2
 * (MERGE, CONCAT) or, ATTENTION, the MLP width, a multiple of 16 in [16, 1024],
 * 1 <= n_layers <= 16, head_hidden = 128, n_quantiles odd <= 15.  n_heads is read
 * for ATTENTION only: d_model / n_heads a multiple of 8, at most 64 (ATTENTION
 * pools by the mean).  feat_min/feat_max (first n_features entries) are fixed min-max
 * constants (feat_max > feat_min); fourier_scale[k] = s_k, the feature argument is
 * pi * s_k * u; rms_eps > 0.  The fused tensor-core path runs 16-bit-operand
 * MERGE configs with 5 features, mean pooling and d_model 128 or 256; the
 * packed-row tensor-core path runs 16-bit-operand CONCAT and ATTENTION configs
 * (valid hits only, one tensor-core product per matrix of Sec. 3.2 / App. A.3);
 * everything else runs on the CUDA cores. */
typedef struct {
  int32_t abi_version;
  int32_t max_hits;
  int32_t n_features;
  int32_t n_fourier;
  int32_t d_model;
  int32_t d_hidden;
  int32_t n_layers;
  int32_t head_hidden;
  int32_t n_quantiles;
  int32_t precision;  /* trackfit_precision */
  int32_t pool;       /* trackfit_pool */
  int32_t topology;   /* trackfit_topology */
  int32_t n_heads;    /* attention heads (ATTENTION) */
  float feat_min[TRACKFIT_MAX_FEATURES];
  float feat_max[TRACKFIT_MAX_FEATURES];
  float fourier_scale[TRACKFIT_MAX_FOURIER];
  float rms_eps;
} trackfit_config_t;

typedef struct trackfit_ctx* trackfit_t;

/* Size of the encoder of Sec. 3.2 for cfg (the paper's model: 0.64 M parameters).
 * Number of fp32 values in the weight blob for cfg (0 if cfg is NULL or
 * unsupported).  Blob order, every matrix in PyTorch [out][in] row-major order,
 * with D = d_model, H = d_hidden, E = 2 * n_features * n_fourier,
 * P = D (MERGE with mean pooling, ATTENTION) or 2H (endpoints, or CONCAT), Hh = head_hidden,
 * Q = 5 * n_quantiles:
 *   W_e1[D][E] b_e1[D] W_e2[D][D] b_e2[D]
 *   MERGE, per layer: g[D] W_in[4H+D][D] b_in[4H+D] (row blocks z_f, n_f, z_b, n_b, gate)
 *              W_m[D][2H] (columns: forward states, then reverse) b_m[D]
 *              W_1[D][D] b_1[D] W_2[D][D] b_2[D]
 *   CONCAT, per layer l: W_in[4H][I_l] b_in[4H] (row blocks z_f, n_f, z_b, n_b), I_0 = D,
 *              I_l = 2H after (columns: forward states, then reverse)
 *   ATTENTION, per layer: g_1[D] W_qkv[3D][D] b_qkv[3D] (row blocks q, k, v; head h
 *              owns rows h D/n_heads .. of each block) W_o[D][D] b_o[D] g_2[D]
 *              W_1[H][D] b_1[H] W_2[D][H] b_2[D]
 *   g_h[P] W_h1[Hh][P] b_h1[Hh] W_h2[Q][Hh] b_h2[Q]   (Q rows parameter-major: [5][7]) */
size_t trackfit_weight_count(const trackfit_config_t* cfg);

/* Load a trained encoder (Sec. 3.2: Fourier featurisation, dense embedding,
 * bidirectional minGRU layers, RMSNorm and the quantile head) for inference.
 * With 16-bit operand precision the weights of the per-hit products are
 * converted once here (Sec. 3.5: reduced-precision projection weights).
 * Validate cfg, copy the host fp32 weights to the device (converted and repacked
 * for the kernels) and allocate the handle's workspace.  Synchronous; launches no
 * work on any user stream.  The caller keeps ownership of `weights` and may free
 * it on return.  Errors: INVALID_ARG (NULL, n_weights != trackfit_weight_count),
 * UNSUPPORTED (cfg outside the supported set), OOM, CUDA.  *out is set only on
 * success. */
int trackfit_create(const trackfit_config_t* cfg, const float* weights, size_t n_weights,
                    trackfit_t* out);

/* The fit itself (Sec. 3, problem statement): each track's hit sequence, in
 * measurement-time order, to its five perigee parameters, for a batch of
 * independent tracks in one call (Sec. 4: the fit is embarrassingly parallel
 * across tracks; Sec. 3.5: tracks run packed, without padding, inside the
 * kernels).  The output is the median of the 7 quantiles of each parameter
 * (Sec. 3.3).
 * Run the encoder on n_tracks tracks, asynchronously on `stream` (a cudaStream_t;
 * NULL = the legacy default stream).  No host synchronisation, no allocation.
 *   hits       device, [n_tracks][max_hits][5] fp32, row-major, 16-byte aligned;
 *              hit t of track b is valid for t < n_hits[b]; padded entries are
 *              never read into the result (they may hold NaN).
 *   n_hits     device, [n_tracks] int32.
 *   out_params device, [n_tracks][5] fp32 (d0, z0, phi, theta, q/p), 16-byte aligned.
 * The caller owns all three buffers.  Host-side checks (NULL, n_tracks <= 0,
 * alignment) return INVALID_ARG and launch nothing; launch failures return CUDA.
 * A track with n_hits outside [1, max_hits] gets a NaN row and is counted in the
 * device error counter (trackfit_device_errors). */
int trackfit_forward(trackfit_t h, const float* hits, const int32_t* n_hits, int64_t n_tracks,
                     float* out_params, void* stream);

/* As trackfit_forward, and optionally also writes (each pointer may be NULL)
 * the head's full quantile output (Sec. 3.3: 7 quantiles per parameter) and the
 * pooled track vector it reads (Sec. 3.2):
 *   out_quantiles device [n_tracks][5][7] fp32: all head outputs (Sec. 3.2-3.3);
 *   out_pooled    device [n_tracks][P] fp32: the pooled vector before the head. */
int trackfit_forward_ex(trackfit_t h, const float* hits, const int32_t* n_hits, int64_t n_tracks,
                        float* out_params, float* out_quantiles, float* out_pooled, void* stream);

/* The fit of trackfit_forward on the packed, unpadded layout the paper deploys
 * (Sec. 3.5: tracks run packed, without padding): no padding rows cross HBM.
 *   hits        device [n_hit_rows][5] fp32 (x, y, z [mm], r [mm], phi [rad]),
 *               the hits of all tracks back to back, 16-byte aligned.
 *   n_hit_rows  rows in hits (bounds every track's rows).
 *   offsets     device [n_tracks + 1] int64, 16-byte aligned: track b's hits are
 *               rows offsets[b] .. offsets[b + 1] - 1, in measurement-time order.
 *   out_params  device [n_tracks][5] fp32, as trackfit_forward.
 * A track whose row range is empty, longer than max_hits, or outside
 * [0, n_hit_rows) gets a NaN row and is counted in the device error counter;
 * none of its rows is read.  Results are bit-identical to trackfit_forward on
 * the same tracks padded to max_hits.  Asynchronous on `stream`; no host
 * synchronisation, no allocation (the per-track counts go to a buffer the
 * handle allocated at create, in chunks of 1,048,576 tracks).  Errors:
 * INVALID_ARG (NULL, n_tracks <= 0, n_hit_rows < 0, misalignment), CUDA. */
int trackfit_forward_packed(trackfit_t h, const float* hits, int64_t n_hit_rows, const int64_t* offsets,
                            int64_t n_tracks, float* out_params, void* stream);

/* The fit of trackfit_forward with the data movement a deployment pays (Sec. 4.2
 * times the whole forward from the hits to the parameters).
 * End-to-end variant with HOST buffers: copies hits [n_tracks][max_hits][5] and
 * n_hits [n_tracks] to the device, runs the encoder and copies out_params
 * [n_tracks][5] back, all on `stream`, and returns after the stream has finished
 * this work (synchronous).  The batch moves in steps of 262,144 tracks: a
 * step's inputs are copied on a stream of the handle's own while the previous
 * step computes on `stream` (only the first step's copy is not hidden), and
 * its outputs are copied back behind it.  Pinned
 * (page-locked) host memory makes the copies asynchronous and lets them
 * overlap; pageable memory works too.  The device staging
 * buffers are owned by the handle and grow on demand (this call may allocate).
 * Errors as trackfit_forward, plus OOM.  Before returning it reads and resets the
 * device error counters (as trackfit_device_errors): TRACKFIT_ERR_BAD_HITS when
 * tracks had hit counts outside [1, max_hits] (their rows are NaN, the others
 * valid), TRACKFIT_ERR_TIMEOUT when a bounded device wait expired (the output is
 * not valid). */
int trackfit_forward_host(trackfit_t h, const float* hits_host, const int32_t* n_hits_host,
                          int64_t n_tracks, float* out_params_host, void* stream);

/* Validity of a batch's results.  The problem statement (Sec. 3) defines a
 * track by its hits; a track with no hit, or with more hits than max_hits, has
 * no defined fit and gets a NaN row, counted here.
 * Read and reset the device error counters: synchronises `stream`, returns the
 * number of tracks with invalid n_hits since the last call in *n_bad, and
 * returns TRACKFIT_ERR_TIMEOUT if a bounded device wait expired (else OK or
 * BAD_HITS when *n_bad > 0). */
int trackfit_device_errors(trackfit_t h, void* stream, int64_t* n_bad);

/* Name of the kernel path the handle runs: "simt-fp32", "simt-bf16",
 * "simt-fp16", "tcgen05-bf16", "tcgen05-fp16", "tcgen05-rows-bf16" or
 * "tcgen05-rows-fp16".  Static string, owned by the library. */
const char* trackfit_path_name(trackfit_t h);

/* Select the kernel path: 0 = automatic (the fused tcgen05 path for the
 * BF16_PROJ / FP16_PROJ MERGE configs it supports: mean pooling, d_model 128 or
 * 256; the packed-row tcgen05 path for 16-bit CONCAT and ATTENTION configs; SIMT
 * otherwise), 1 = force the SIMT path.  Returns UNSUPPORTED if the requested path
 * cannot run this configuration. */
int trackfit_set_path(trackfit_t h, int path);

/* Timing hook: with enable = 1 every forward records CUDA events on its stream
 * around the main compute kernel (the fused tcgen05 kernel, every product
 * launch of the packed-row tcgen05 path, or the SIMT layer sequence);
 * trackfit_profile_read synchronises on them, returns the summed
 * kernel time in milliseconds and the number of timed launches since the last
 * read, and resets both.  enable = 0 releases the events. */
int trackfit_profile(trackfit_t h, int enable);
int trackfit_profile_read(trackfit_t h, double* kernel_ms, int64_t* launches);

/* Release a loaded encoder (the counterpart of trackfit_create; the paper's
 * model lives for the whole job, Sec. 4.2).
 * Free everything the handle owns.  Accepts NULL.  The caller must make sure no
 * work using the handle is still running on any stream. */
void trackfit_destroy(trackfit_t h);

/* Static description of a status code. */
const char* trackfit_strerror(int status);

/* The CUDA error behind the calling thread's last TRACKFIT_ERR_CUDA or
 * TRACKFIT_ERR_OOM, with the step it came from ("" if none yet).  The string is
 * owned by the library and valid until the thread's next failing call. */
const char* trackfit_last_error(void);

/* Test hook: masked bidirectional linear recurrence h_t = a_t h_{t-1} + b_t x_t
 * (Eq. 2 written as a linear recurrence, with a = 1 - z, b = z, x = n) on the device.
 * a, b, x, h_fwd, h_bwd: device [n_tracks][T][C] fp32; n_hits device [n_tracks].
 * Steps t >= n_hits[b] carry the state and output 0; the reverse scan starts at
 * t = n_hits[b] - 1.  Asynchronous on `stream`. */
int trackfit_debug_scan(const float* a, const float* b, const float* x, const int32_t* n_hits,
                        int64_t n_tracks, int32_t T, int32_t C, float* h_fwd, float* h_bwd,
                        void* stream);

/* Test hook, host only (no GPU needed): per-tile totals of the tensor-core
 * path's block schedule for cfg, from the same expansion the fused kernel uses.
 * counts (host, n_counts >= 6): [0] 128 x 64 weight blocks, [1] MMA instructions
 * (128 x 128 x 16 each), [2] operand hand-overs the issuer waits for from the
 * epilogue (W_E), [3] state hand-overs (W_H), [4] accumulator commits the
 * epilogue waits for (C_ACC), [5] state-buffer commits (C_HB).  codes (host,
 * optional, NULL when codes_cap is 0): the first codes_cap blocks' hand-overs in
 * issue order, one byte each: wait (0 none, 1 W_E, 2 W_H) | commit (0 none,
 * 1 C_ACC, 2 C_HB) << 2.  Returns TRACKFIT_ERR_UNSUPPORTED when cfg does not run
 * on the tensor-core path, TRACKFIT_ERR_INVALID_ARG for NULL pointers, n_counts
 * < 6, or codes_cap > 0 with codes NULL. */
int trackfit_debug_schedule(const trackfit_config_t* cfg, int64_t* counts, int32_t n_counts, uint8_t* codes,
                            int64_t codes_cap);

/* Test hook for the tensor-core operand layouts: D = A * B on one 128 x 128
 * tile through the same TMA, shared-memory descriptor and tensor-memory path as
 * the fused kernel.  A device bf16 bits [128][K] row-major (K-major), Bkn device
 * bf16 bits [K][128] row-major, D device fp32 [128][128]; K in {64, 128, 192,
 * 256}; all 16-byte aligned.  h supplies the device error counter.
 * Asynchronous on `stream`; requires an sm_100-family GPU. */
int trackfit_debug_umma(trackfit_t h, const uint16_t* A, const uint16_t* Bkn, int32_t K, float* D,
                        void* stream);

/* The analytic seed of Sec. 3.1, on the device in fp64 (the paper keeps the seed
 * in float64 to avoid a cancellation in the beam-line transport at high
 * momentum).  Per track: the seed triplet (the first hit, then each first later
 * hit more than 10 mm (3-D) from the previous seed hit: there are no
 * detector-volume identifiers in these inputs, and the distance keeps two hits
 * of one surface out of a triplet), the circle through the triplet's transverse
 * points by the conformal map, its point closest to the beam line, the charge
 * from the turning direction, theta from the first and third seed hit, and the
 * perigee (d0, z0, phi0, theta, q/p) with p_T = 0.299792458 B R / 1000 GeV.  Per
 * hit: the three residual features of Sec. 3.1 against that helix, asinh(du),
 * asinh(dv) and s_helix, where the foot point is the helix point whose normal
 * plane holds the hit (Newton's method), du and dv the hit's coordinates there
 * along U = z x t / |z x t| and V = t x U (the curvilinear frame), s the 3-D
 * path length from the perigee, lengths in mm (asinh scale 1 mm).
 *   hits         device [n_tracks][max_hits][hit_stride] fp32, x, y, z [mm] first.
 *   hit_stride   floats per hit row (>= 3; 5 for the task's inputs, 15 for the paper's).
 *   n_hits       device [n_tracks] int32.
 *   b_field      the solenoid field B_z in tesla (> 0).
 *   seed_out     device [n_tracks][5] fp64: the seed perigee; a NaN row where a
 *                track has fewer than three hits so spaced, or n_hits outside
 *                [0, max_hits].
 *   features_out device fp32 or NULL: hit t of track b gets its three residual
 *                features at features_out[(b max_hits + t) feat_stride + 0..2],
 *                zero on padded hits and on tracks without a seed (feat_stride 3:
 *                an array [n_tracks][max_hits][3]; feat_stride = hit_stride with
 *                features_out pointing at column 12 of the hit array: the last
 *                three of the paper's 15 encoder features, written in place).
 *   feat_stride  >= 3.
 * All pointers 16-byte aligned; the caller owns every buffer.  Asynchronous on
 * `stream`; allocates nothing.  Errors: INVALID_ARG (NULL, n_tracks <= 0,
 * max_hits outside [1, 64], hit_stride or feat_stride below 3, b_field not > 0,
 * misalignment), CUDA. */
int trackfit_seed(const float* hits, int32_t hit_stride, const int32_t* n_hits, int64_t n_tracks,
                  int32_t max_hits, double b_field, double* seed_out, float* features_out,
                  int32_t feat_stride, void* stream);

/* Decode of the heads' corrections against the seed (Sec. 3.3): d0, z0, theta
 * additive, phi additive and wrapped to (-pi, pi], q/p from the scale-free
 * residual r: q/p = q/p_seed + r (|q/p_seed| + 0.02 / GeV).
 *   seed         device [n_tracks][5] fp64 (trackfit_seed's output).
 *   corrections  device [n_tracks][5] fp32 (the heads' median outputs).
 *   out_params   device [n_tracks][5] fp32 (computed in fp64, then rounded).
 * 16-byte aligned; asynchronous on `stream`; allocates nothing.  Errors:
 * INVALID_ARG (NULL, n_tracks <= 0, misalignment), CUDA. */
int trackfit_decode(const double* seed, const float* corrections, int64_t n_tracks, float* out_params,
                    void* stream);

/* Test hook for the failure path of the fused tensor-core kernel's bounded
 * waits (every wait for a hand-over inside that kernel gives up after a time
 * limit, records TRACKFIT_ERR_TIMEOUT in the handle's device error counters,
 * and the kernel drains its copies and products and returns instead of
 * hanging).  For this handle's later forwards: limit_ns > 0 replaces the 2 s
 * limit (0 restores it); hold_tile >= 0 makes the loader warp of the first CTA
 * hold back its hand-over of the metadata of its hold_tile-th tile for twice the
 * limit (or until a wait has given up), so that the epilogue's wait for it
 * expires; -1 holds nothing.  The outputs of a forward that timed out are not
 * valid; trackfit_device_errors reports TRACKFIT_ERR_TIMEOUT and resets the
 * counters, after which the handle is usable again.  Host side only; launches
 * nothing.  On a handle of the packed-row tensor-core path (16-bit CONCAT and
 * ATTENTION configs) only the limit applies: hold_tile must be -1 there.
 * Errors: INVALID_ARG (NULL handle, limit_ns < 0, hold_tile < -1), UNSUPPORTED
 * (the handle runs the CUDA-core path, which has no waits, or hold_tile >= 0 on
 * the packed-row path). */
int trackfit_debug_wait_limit(trackfit_t h, int64_t limit_ns, int32_t hold_tile);

/* Test hook for allocation failures (host side, not thread-safe): every device
 * allocation the library makes for a handle (trackfit_create, the staging
 * buffers of trackfit_forward_host) is counted.  fail_nth > 0 makes the
 * fail_nth-th allocation from now on fail as if the device were out of memory
 * (the call then returns TRACKFIT_ERR_OOM after freeing what it had allocated);
 * 0 arms nothing.  Returns the number of device allocations the library holds
 * now; *attempted (may be NULL) receives the allocations attempted since the
 * previous call. */
int64_t trackfit_debug_alloc(int64_t fail_nth, int64_t* attempted);

/* Forward pass that allocates no device memory, for callers that cannot call
 * cudaMalloc (code whose device memory is owned by an outer framework or pool,
 * or that must not let an allocation synchronise the device).  The paper has no
 * counterpart: it is a deployment variant of the CUDA-core (SIMT) path.
 *   cfg        host, as for trackfit_create (any supported precision / pooling).
 *   weights    device, the fp32 blob of trackfit_weight_count(cfg) values in the
 *              layout documented there, 16-byte aligned (used as given, no repack).
 *   hits, n_hits, n_tracks, out_params: as for trackfit_forward.
 * All workspace comes from one file-scope device array of 32 MiB that every GPU
 * loading this library keeps until the process exits; the batch is processed in
 * chunks of whole tracks that fit in it.  A configuration whose workspace for a
 * single track exceeds 32 MiB returns TRACKFIT_ERR_UNSUPPORTED.  The first call
 * on a device looks up the array's device address (cudaGetSymbolAddress) with
 * that device current; make that first call before any stream capture.  Every
 * call shares the array: calls that overlap on the GPU (different streams or
 * devices' contexts sharing it concurrently) race and must be serialised by the
 * caller.  Tracks with n_hits outside [1, max_hits] get NaN rows (no counter is
 * read back).  Asynchronous on `stream`; makes no cudaMalloc / cudaFree call.
 * Errors: INVALID_ARG (NULL, n_tracks <= 0, misalignment), UNSUPPORTED, CUDA. */
int trackfit_forward_noalloc(const trackfit_config_t* cfg, const float* weights, const float* hits,
                             const int32_t* n_hits, int64_t n_tracks, float* out_params, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* TRACKFIT_H */
