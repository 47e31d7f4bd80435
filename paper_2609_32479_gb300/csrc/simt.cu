// SIMT (CUDA-core) kernel path: the production path for TRACKFIT_FP32 configs
// and a second, independent GPU implementation of the BF16_PROJ arithmetic.
//
// Layout: the batch is processed in chunks of whole tracks; inside a chunk every
// per-hit tensor is row-major [tracks * max_hits][channels] in the handle's
// workspace.  Padded rows are computed and then excluded by select (their
// residual rows are forced to 0, the scans and pooling skip them).
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <math.h>

#include "attention.cuh"
#include "trackfit_internal.h"

namespace {

enum { EPI_STORE = 0, EPI_SILU = 1, EPI_PROJ = 2, EPI_GATE_RES = 3, EPI_RES_MASK = 4, EPI_MASK = 5 };

__device__ __forceinline__ float sigm(float x) { return 1.0f / (1.0f + expf(-x)); }
__device__ __forceinline__ float silu(float x) { return x * sigm(x); }
__device__ __forceinline__ float bf16r(float x) { return __bfloat162float(__float2bfloat16_rn(x)); }
__device__ __forceinline__ float fp16r(float x) { return __half2float(__float2half_rn(x)); }

__device__ __forceinline__ bool row_valid(int r, int T, const int32_t* n_hits) {
  int b = r / T, t = r - b * T;
  int n = n_hits[b];
  return n >= 1 && n <= T && t < n;
}

struct GemmArgs {
  const float* A; int lda;      // [R][lda], first K columns used
  const float* W;               // [N][K] row-major (PyTorch [out][in])
  const float* bias;            // [N]
  float* C; int ldc;            // [R][ldc]
  int R, N, K;
  int rnd;                      // round both operands on load: 0 none, 1 bf16, 2 fp16
  int epi;
  const float* res; int ldr;    // residual input (GATE_RES, RES_MASK)
  const float* gate; int ldg;   // sigmoid gate values (GATE_RES)
  int H;                        // hidden width (PROJ: which columns are gates)
  const int32_t* n_hits; int T; // padding mask (MASK, RES_MASK)
};

constexpr int BM = 64, BN = 64, BK = 16;

// C = epilogue(A W^T + bias); 256 threads, 4x4 outputs per thread.
__global__ void __launch_bounds__(256) gemm_kernel(GemmArgs g) {
  __shared__ float As[BK][BM + 4];
  __shared__ float Ws[BK][BN + 4];
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  const int row0 = blockIdx.y * BM, col0 = blockIdx.x * BN;
  float acc[4][4] = {};
  for (int k0 = 0; k0 < g.K; k0 += BK) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      int idx = tid + i * 256, m = idx >> 4, k = idx & 15;
      int r = row0 + m, kk = k0 + k;
      float a = (r < g.R && kk < g.K) ? g.A[(size_t)r * g.lda + kk] : 0.0f;
      int n = col0 + m;
      float w = (n < g.N && kk < g.K) ? g.W[(size_t)n * g.K + kk] : 0.0f;
      if (g.rnd == 1) { a = bf16r(a); w = bf16r(w); }
      if (g.rnd == 2) { a = fp16r(a); w = fp16r(w); }
      As[k][m] = a;
      Ws[k][m] = w;
    }
    __syncthreads();
#pragma unroll
    for (int k = 0; k < BK; ++k) {
      float a[4], w[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) { a[i] = As[k][ty * 4 + i]; w[i] = Ws[k][tx * 4 + i]; }
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], w[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    int r = row0 + ty * 4 + i;
    if (r >= g.R) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      int n = col0 + tx * 4 + j;
      if (n >= g.N) continue;
      float v = acc[i][j] + g.bias[n];
      switch (g.epi) {
        case EPI_SILU: v = silu(v); break;
        case EPI_PROJ: {
          bool is_gate = (n < g.H) || (n >= 2 * g.H && n < 3 * g.H) || (n >= 4 * g.H);
          if (is_gate) v = sigm(v);
        } break;
        case EPI_GATE_RES: v = g.res[(size_t)r * g.ldr + n] + v * g.gate[(size_t)r * g.ldg + n]; break;
        case EPI_RES_MASK:
          v = row_valid(r, g.T, g.n_hits) ? g.res[(size_t)r * g.ldr + n] + v : 0.0f;
          break;
        case EPI_MASK: v = row_valid(r, g.T, g.n_hits) ? v : 0.0f; break;
        default: break;
      }
      g.C[(size_t)r * g.ldc + n] = v;
    }
  }
}

// Fourier features (Sec. 3.2): one thread per (hit row, feature).  The argument
// s_k * u is formed in fp64 and reduced modulo 2 before the fp32 sinpi/cospi, so
// the fp32 result carries no argument error from the up-to-32x scale.  With a
// packed input (offs), row r = b T + t reads hit offs[b] + t for t < n_hits[b]
// and is zero otherwise (padding rows are excluded by select later).
__global__ void fourier_kernel(const float* __restrict__ hits, int64_t rows, float* __restrict__ e,
                               tf_shape s, const int64_t* __restrict__ offs, const int32_t* __restrict__ n_hits) {
  int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (i >= rows * s.F) return;
  int64_t r = i / s.F;
  int f = (int)(i - r * s.F);
  float v;
  if (offs) {
    const int64_t b = r / s.T, t = r - b * s.T;
    const int n = n_hits[b];
    v = (n >= 1 && n <= s.T && t < n) ? hits[(offs[b] + t) * s.F + f] : 0.0f;
  } else {
    v = hits[r * s.F + f];
  }
  double u = ((double)v - s.feat_min_d[f]) / s.feat_range_d[f];
  float* o = e + r * s.E + f * 2 * s.K;
  for (int k = 0; k < s.K; ++k) {
    double a = u * (double)s.scale[k];
    a -= 2.0 * rint(0.5 * a);
    float af = (float)a;
    o[k] = sinpif(af);
    o[s.K + k] = cospif(af);
  }
}

// x_hat = x / sqrt(mean(x^2) + eps) * g, one warp per row.
__global__ void rmsnorm_kernel(const float* __restrict__ x, int64_t rows, int D, const float* __restrict__ gain,
                               float eps, float* __restrict__ y) {
  int64_t r = blockIdx.x * (int64_t)(blockDim.x / 32) + threadIdx.x / 32;
  int lane = threadIdx.x & 31;
  if (r >= rows) return;
  const float* xr = x + r * D;
  float ss = 0.0f;
  for (int c = lane; c < D; c += 32) ss = fmaf(xr[c], xr[c], ss);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  float inv = 1.0f / sqrtf(ss / (float)D + eps);
  for (int c = lane; c < D; c += 32) y[r * D + c] = xr[c] * inv * gain[c];
}

// Bidirectional minGRU scans of one layer (Sec. 3.2, Eq. 2): one thread per
// (track, channel); z already passed through the sigmoid by the projection.
__global__ void mingru_scan_kernel(const float* __restrict__ pr, int ldp, const int32_t* __restrict__ n_hits,
                                   int64_t B, int T, int H, float* __restrict__ y) {
  int c = blockIdx.x * blockDim.x + threadIdx.x;
  int64_t b = blockIdx.y;
  if (c >= H || b >= B) return;
  int n = n_hits[b];
  if (n < 1 || n > T) n = 0;
  const float* p = pr + b * T * (int64_t)ldp;
  float* yo = y + b * T * (int64_t)(2 * H);
  float h = 0.0f;
  for (int t = 0; t < T; ++t) {
    if (t < n) {
      float z = p[t * ldp + c], cand = p[t * ldp + H + c];
      h = fmaf(z, cand - h, h);
      yo[t * 2 * H + c] = h;
    } else {
      yo[t * 2 * H + c] = 0.0f;
    }
  }
  h = 0.0f;
  for (int t = T - 1; t >= 0; --t) {
    if (t < n) {
      float z = p[t * ldp + 2 * H + c], cand = p[t * ldp + 3 * H + c];
      h = fmaf(z, cand - h, h);
      yo[t * 2 * H + H + c] = h;
    } else {
      yo[t * 2 * H + H + c] = 0.0f;
    }
  }
}

// Generic masked linear recurrence h_t = a_t h_{t-1} + b_t x_t, both directions.
__global__ void linear_scan_kernel(const float* __restrict__ a, const float* __restrict__ bb,
                                   const float* __restrict__ x, const int32_t* __restrict__ n_hits, int64_t B,
                                   int T, int C, float* __restrict__ hf, float* __restrict__ hb) {
  int c = blockIdx.x * blockDim.x + threadIdx.x;
  int64_t b = blockIdx.y;
  if (c >= C || b >= B) return;
  int n = n_hits[b];
  if (n < 0) n = 0;
  if (n > T) n = T;
  int64_t base = b * T * (int64_t)C + c;
  float h = 0.0f;
  for (int t = 0; t < T; ++t) {
    int64_t i = base + (int64_t)t * C;
    if (t < n) { h = fmaf(a[i], h, bb[i] * x[i]); hf[i] = h; } else { hf[i] = 0.0f; }
  }
  h = 0.0f;
  for (int t = T - 1; t >= 0; --t) {
    int64_t i = base + (int64_t)t * C;
    if (t < n) { h = fmaf(a[i], h, bb[i] * x[i]); hb[i] = h; } else { hb[i] = 0.0f; }
  }
}

// Pooling and head (Sec. 3.2-3.3): one 128-thread block per track.  With
// pooled_in the pooled vectors [B][P] are given (the packed-row path pools in its
// scan or pooling kernel) and x, y are not read.
__global__ void __launch_bounds__(128) pool_head_kernel(const float* __restrict__ pooled_in,
                                                        const float* __restrict__ x, const float* __restrict__ y,
                                                        const int32_t* __restrict__ n_hits, int64_t B, tf_shape s,
                                                        const float* __restrict__ gh, const float* __restrict__ w1,
                                                        const float* __restrict__ b1, const float* __restrict__ w2,
                                                        const float* __restrict__ b2, float* __restrict__ out,
                                                        float* __restrict__ out_q, float* __restrict__ out_pool,
                                                        unsigned long long* err) {
  __shared__ float pv[2 * 384];
  __shared__ float hid[256];
  __shared__ float red[4];
  __shared__ float qv[5 * 15];
  const int64_t b = blockIdx.x;
  const int tid = threadIdx.x;
  const int T = s.T, H = s.H, P = s.P;
  int n = n_hits[b];
  const bool bad = n < 1 || n > T;
  if (bad) {
    if (tid == 0) atomicAdd(err, 1ull);
    n = 1;
  }
  if (pooled_in) {
    for (int c = tid; c < P; c += blockDim.x) pv[c] = bad ? 0.0f : pooled_in[b * P + c];
  } else if (s.pool == TRACKFIT_POOL_MEAN) {   // x: [rows][P] (P = D, or 2H for CONCAT)
    for (int c = tid; c < P; c += blockDim.x) {
      float acc = 0.0f;
      for (int t = 0; t < n; ++t) acc += x[(b * T + t) * P + c];
      pv[c] = acc / (float)n;
    }
  } else {
    for (int c = tid; c < H; c += blockDim.x) {
      pv[c] = y[(b * T + (n - 1)) * 2 * H + c];
      pv[H + c] = y[(b * T) * 2 * H + H + c];
    }
  }
  __syncthreads();
  float ss = 0.0f;
  for (int c = tid; c < P; c += blockDim.x) ss = fmaf(pv[c], pv[c], ss);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  if ((tid & 31) == 0) red[tid >> 5] = ss;
  __syncthreads();
  float tot = 0.0f;
  for (int i = 0; i < (int)(blockDim.x >> 5); ++i) tot += red[i];
  const float inv = 1.0f / sqrtf(tot / (float)P + s.rms_eps);
  if (out_pool)
    for (int c = tid; c < P; c += blockDim.x) out_pool[b * P + c] = bad ? NAN : pv[c];
  __syncthreads();
  for (int c = tid; c < P; c += blockDim.x) pv[c] = pv[c] * inv * gh[c];
  __syncthreads();
  for (int j = tid; j < s.Hh; j += blockDim.x) {
    float acc = b1[j];
    const float* wr = w1 + (size_t)j * P;
    for (int c = 0; c < P; ++c) acc = fmaf(wr[c], pv[c], acc);
    hid[j] = silu(acc);
  }
  __syncthreads();
  for (int o = tid; o < s.Q; o += blockDim.x) {
    float acc = b2[o];
    const float* wr = w2 + (size_t)o * s.Hh;
    for (int j = 0; j < s.Hh; ++j) acc = fmaf(wr[j], hid[j], acc);
    qv[o] = bad ? NAN : acc;
    if (out_q) out_q[b * s.Q + o] = qv[o];
  }
  __syncthreads();
  if (tid < 5) out[b * 5 + tid] = qv[tid * s.NQ + s.NQ / 2];
}

// Per hit row: E (Fourier) + U + X + XH + PR + Y + X1, with U = D and PR = 4H + D,
// Y = 2H (recurrent topologies) or U = H (the MLP), PR = 3D (q, k, v) and Y = D
// (the attention output) for ATTENTION.
// The head's last step on given quantiles qv [B][Q]: invalid tracks (count
// outside [1, T]) get NaN rows and are counted; the medians go to out, the
// quantiles and the pooled vectors to the optional exports.
__global__ void head_finish_kernel(const float* __restrict__ qv, const float* __restrict__ pooled,
                                   const int32_t* __restrict__ n_hits, int64_t B, tf_shape s, float* __restrict__ out,
                                   float* __restrict__ out_q, float* __restrict__ out_pool, unsigned long long* err) {
  const int64_t b = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (b >= B) return;
  const int n = n_hits[b];
  const bool bad = n < 1 || n > s.T;
  if (bad) atomicAdd(err, 1ull);
  for (int p = 0; p < 5; ++p) out[b * 5 + p] = bad ? NAN : qv[b * s.Q + p * s.NQ + s.NQ / 2];
  if (out_q)
    for (int o = 0; o < s.Q; ++o) out_q[b * s.Q + o] = bad ? NAN : qv[b * s.Q + o];
  if (out_pool)
    for (int c = 0; c < s.P; ++c) out_pool[b * s.P + c] = bad ? NAN : pooled[b * s.P + c];
}

size_t ws_floats_per_track(const tf_shape& s) {
  const size_t D = s.D, H = s.H;
  const size_t row = s.topology == TRACKFIT_TOPOLOGY_ATTENTION ? H + 7 * D : 5 * D + 6 * H;
  return (size_t)s.T * (s.E + row);
}

int launch_gemm(const GemmArgs& g, cudaStream_t st) {
  dim3 grid((g.N + BN - 1) / BN, (g.R + BM - 1) / BM);
  gemm_kernel<<<grid, 256, 0, st>>>(g);
  return cudaPeekAtLastError() == cudaSuccess ? TRACKFIT_OK : TRACKFIT_ERR_CUDA;
}

}  // namespace

int tf_simt_workspace(trackfit_ctx* h) {
  const size_t budget = (size_t)1 << 30;
  size_t per = ws_floats_per_track(h->s) * sizeof(float);
  int64_t n = (int64_t)(budget / per);
  if (n < 1) n = 1;
  if (n > 65535) n = 65535;                       // grid.y limit of the scan launch
  if (n * h->s.T > 65535LL * 64) n = 65535LL * 64 / h->s.T;   // grid.y limit of the GEMM
  h->ws_tracks = n;
  h->ws_bytes = per * (size_t)n;
  return tf_status_from_cuda(tf_malloc((void**)&h->ws, h->ws_bytes));
}

// The whole SIMT forward over chunks of ws_tracks tracks, with the workspace and
// the device error counter supplied by the caller.  prof (may be null) is the
// handle whose timing hook brackets each chunk's kernels.
int tf_simt_run(const tf_shape& s, const tf_blob_off& o, const float* W, float* ws, int64_t ws_tracks,
                unsigned long long* err, const float* hits, const int32_t* n_hits, int64_t B, float* out,
                float* out_q, float* out_pool, cudaStream_t st, trackfit_ctx* prof, const int64_t* offs) {
  const int rnd = s.precision;   // TRACKFIT_FP32 = 0, BF16_PROJ = 1, FP16_PROJ = 2
  const bool attn = s.topology == TRACKFIT_TOPOLOGY_ATTENTION;
  const int D = s.D, H = s.H, PD = attn ? 3 * s.D : 4 * s.H + s.D;
  const int UW = attn ? s.H : s.D, YW = attn ? s.D : 2 * s.H;
  // the attention CTA's dynamic shared memory, when above the default 48 KB
  if (attn && tf_attn::allow_smem<float>(s.T, s.D, s.NH) != cudaSuccess) return TRACKFIT_ERR_CUDA;
  for (int64_t c0 = 0; c0 < B; c0 += ws_tracks) {
    const int64_t nb = (B - c0 < ws_tracks) ? B - c0 : ws_tracks;
    const int64_t R = nb * s.T;
    float* EB = ws;
    float* U = EB + R * s.E;
    float* X = U + R * UW;
    float* XH = X + R * D;
    float* PR = XH + R * D;
    float* Y = PR + R * PD;
    float* X1 = Y + R * YW;
    const float* hc = offs ? hits : hits + c0 * s.T * 5;
    const int64_t* oc = offs ? offs + c0 : nullptr;
    const int32_t* nc = n_hits + c0;
    if (prof) tf_prof_begin(prof, st);
    int64_t nthreads = R * s.F;
    fourier_kernel<<<(unsigned)((nthreads + 255) / 256), 256, 0, st>>>(hc, R, EB, s, oc, nc);
    GemmArgs g{};
    g.R = (int)R;
    g.rnd = rnd;
    g.n_hits = nc;
    g.T = s.T;
    g.H = H;
    // embedding: U = SiLU(W_e1 e + b_e1); X = mask(W_e2 U + b_e2)
    g.A = EB; g.lda = s.E; g.W = W + o.emb_w1; g.bias = W + o.emb_b1; g.C = U; g.ldc = D;
    g.N = D; g.K = s.E; g.epi = EPI_SILU;
    if (launch_gemm(g, st)) return TRACKFIT_ERR_CUDA;
    g.A = U; g.lda = D; g.W = W + o.emb_w2; g.bias = W + o.emb_b2; g.C = X; g.ldc = D;
    g.N = D; g.K = D; g.epi = EPI_MASK;
    if (launch_gemm(g, st)) return TRACKFIT_ERR_CUDA;
    for (int l = 0; l < s.L; ++l) {
      const tf_layer_off& lo = o.layer[l];
      if (s.topology == TRACKFIT_TOPOLOGY_CONCAT) {
        // Sec. 3.2: the layer input (the embedding, then the previous layer's
        // concatenated states) projected to the gates and candidates, the two
        // scans, their states concatenated in Y (the next layer's input: the
        // projection reads Y before the scan overwrites it, in stream order)
        const int I = l == 0 ? D : 2 * H;
        g.A = l == 0 ? X : Y; g.lda = I; g.W = W + lo.w_in; g.bias = W + lo.b_in; g.C = PR; g.ldc = 4 * H;
        g.N = 4 * H; g.K = I; g.epi = EPI_PROJ;
        if (launch_gemm(g, st)) return TRACKFIT_ERR_CUDA;
        dim3 sg((H + 127) / 128, (unsigned)nb);
        mingru_scan_kernel<<<sg, 128, 0, st>>>(PR, 4 * H, nc, nb, s.T, H, Y);
        continue;
      }
      if (attn) {
        // App. A.3: x' = x + W_o attention(RMSNorm(x) g_1 W_qkv^T + b_qkv) + b_o,
        // x <- x' + W_2 SiLU(RMSNorm(x') g_2 W_1^T + b_1) + b_2, padded rows 0
        rmsnorm_kernel<<<(unsigned)((R + 7) / 8), 256, 0, st>>>(X, R, D, W + lo.g, s.rms_eps, XH);
        g.A = XH; g.lda = D; g.W = W + lo.w_in; g.bias = W + lo.b_in; g.C = PR; g.ldc = 3 * D;
        g.N = 3 * D; g.K = D; g.epi = EPI_STORE;
        if (launch_gemm(g, st)) return TRACKFIT_ERR_CUDA;
        if (tf_attn::launch<float>(PR, 3 * D, nullptr, nc, nb, s.T, D, s.NH, Y, D, st) != cudaSuccess)
          return TRACKFIT_ERR_CUDA;
        g.A = Y; g.lda = D; g.W = W + lo.w_m; g.bias = W + lo.b_m; g.C = X1; g.ldc = D;
        g.N = D; g.K = D; g.epi = EPI_RES_MASK; g.res = X; g.ldr = D;
        if (launch_gemm(g, st)) return TRACKFIT_ERR_CUDA;
        rmsnorm_kernel<<<(unsigned)((R + 7) / 8), 256, 0, st>>>(X1, R, D, W + lo.g2, s.rms_eps, XH);
        g.A = XH; g.lda = D; g.W = W + lo.w1; g.bias = W + lo.b1; g.C = U; g.ldc = H;
        g.N = H; g.K = D; g.epi = EPI_SILU;
        if (launch_gemm(g, st)) return TRACKFIT_ERR_CUDA;
        g.A = U; g.lda = H; g.W = W + lo.w2; g.bias = W + lo.b2; g.C = X; g.ldc = D;
        g.N = D; g.K = H; g.epi = EPI_RES_MASK; g.res = X1; g.ldr = D;
        if (launch_gemm(g, st)) return TRACKFIT_ERR_CUDA;
        continue;
      }
      rmsnorm_kernel<<<(unsigned)((R + 7) / 8), 256, 0, st>>>(X, R, D, W + lo.g, s.rms_eps, XH);
      g.A = XH; g.lda = D; g.W = W + lo.w_in; g.bias = W + lo.b_in; g.C = PR; g.ldc = PD;
      g.N = PD; g.K = D; g.epi = EPI_PROJ;
      if (launch_gemm(g, st)) return TRACKFIT_ERR_CUDA;
      dim3 sg((H + 127) / 128, (unsigned)nb);
      mingru_scan_kernel<<<sg, 128, 0, st>>>(PR, PD, nc, nb, s.T, H, Y);
      if (s.pool == TRACKFIT_POOL_ENDPOINTS && l == s.L - 1) break;
      g.A = Y; g.lda = 2 * H; g.W = W + lo.w_m; g.bias = W + lo.b_m; g.C = X1; g.ldc = D;
      g.N = D; g.K = 2 * H; g.epi = EPI_GATE_RES; g.res = X; g.ldr = D; g.gate = PR + 4 * H; g.ldg = PD;
      if (launch_gemm(g, st)) return TRACKFIT_ERR_CUDA;
      g.A = X1; g.lda = D; g.W = W + lo.w1; g.bias = W + lo.b1; g.C = U; g.ldc = D;
      g.N = D; g.K = D; g.epi = EPI_SILU;
      if (launch_gemm(g, st)) return TRACKFIT_ERR_CUDA;
      g.A = U; g.lda = D; g.W = W + lo.w2; g.bias = W + lo.b2; g.C = X; g.ldc = D;
      g.N = D; g.K = D; g.epi = EPI_RES_MASK; g.res = X1; g.ldr = D;
      if (launch_gemm(g, st)) return TRACKFIT_ERR_CUDA;
    }
    // mean pooling reads the last layer's output: X (MERGE) or the states Y (CONCAT)
    const float* xm = s.topology == TRACKFIT_TOPOLOGY_CONCAT ? Y : X;
    pool_head_kernel<<<(unsigned)nb, 128, 0, st>>>(nullptr, xm, Y, nc, nb, s, W + o.head_g, W + o.head_w1, W + o.head_b1,
                                                    W + o.head_w2, W + o.head_b2, out + c0 * 5,
                                                    out_q ? out_q + c0 * s.Q : nullptr,
                                                    out_pool ? out_pool + c0 * s.P : nullptr, err);
    if (prof) tf_prof_end(prof, st);
    if (cudaPeekAtLastError() != cudaSuccess) return TRACKFIT_ERR_CUDA;
  }
  return TRACKFIT_OK;
}

int tf_simt_forward(trackfit_ctx* h, const float* hits, const int32_t* n_hits, int64_t B, float* out,
                    float* out_q, float* out_pool, cudaStream_t st, const int64_t* offs) {
  return tf_simt_run(h->s, h->off, h->d_w, h->ws, h->ws_tracks, h->d_err, hits, n_hits, B, out, out_q, out_pool, st,
                     h, offs);
}

int tf_simt_debug_scan(const float* a, const float* b, const float* x, const int32_t* n_hits, int64_t B, int T,
                       int C, float* hf, float* hb, cudaStream_t st) {
  dim3 grid((C + 127) / 128, (unsigned)B);
  linear_scan_kernel<<<grid, 128, 0, st>>>(a, b, x, n_hits, B, T, C, hf, hb);
  return cudaPeekAtLastError() == cudaSuccess ? TRACKFIT_OK : TRACKFIT_ERR_CUDA;
}

// The forward with caller-supplied workspace and error counter (the
// no-allocation entry point): no quantile or pooled export, no timing hook.
int tf_simt_forward_explicit(const tf_shape& s, const tf_blob_off& o, const float* W, float* ws, int64_t ws_tracks,
                             unsigned long long* err, const float* hits, const int32_t* n_hits, int64_t B,
                             float* out, cudaStream_t st) {
  return tf_simt_run(s, o, W, ws, ws_tracks, err, hits, n_hits, B, out, nullptr, nullptr, st, nullptr, nullptr);
}

size_t tf_simt_bytes_per_track(const tf_shape& s) { return ws_floats_per_track(s) * sizeof(float); }

// The head of Sec. 3.2-3.3 on given pooled vectors [B][P] as three batched
// steps over all tracks: RMSNorm, the tiled product with W_h1 (SiLU), the tiled
// product with W_h2, then the medians.  ws: B (P + 128 + Q) floats.
int tf_simt_head_batched(const tf_shape& s, const tf_blob_off& o, const float* W, const float* pooled,
                         const int32_t* n_hits, int64_t B, float* ws, float* out, float* out_q, float* out_pool,
                         unsigned long long* err, cudaStream_t st) {
  float* pn = ws;
  float* hid = pn + B * s.P;
  float* qv = hid + B * s.Hh;
  rmsnorm_kernel<<<(unsigned)((B + 7) / 8), 256, 0, st>>>(pooled, B, s.P, W + o.head_g, s.rms_eps, pn);
  GemmArgs g{};
  g.R = (int)B;
  g.rnd = 0;
  g.A = pn; g.lda = s.P; g.W = W + o.head_w1; g.bias = W + o.head_b1; g.C = hid; g.ldc = s.Hh;
  g.N = s.Hh; g.K = s.P; g.epi = EPI_SILU;
  if (launch_gemm(g, st)) return TRACKFIT_ERR_CUDA;
  g.A = hid; g.lda = s.Hh; g.W = W + o.head_w2; g.bias = W + o.head_b2; g.C = qv; g.ldc = s.Q;
  g.N = s.Q; g.K = s.Hh; g.epi = EPI_STORE;
  if (launch_gemm(g, st)) return TRACKFIT_ERR_CUDA;
  head_finish_kernel<<<(unsigned)((B + 255) / 256), 256, 0, st>>>(qv, pooled, n_hits, B, s, out, out_q, out_pool, err);
  return cudaPeekAtLastError() == cudaSuccess ? TRACKFIT_OK : TRACKFIT_ERR_CUDA;
}

// The head of Sec. 3.2-3.3 on given pooled vectors [B][P]: out [B][5], optional
// quantiles [B][Q] and the pooled export (NaN rows for invalid tracks).
int tf_simt_head(const tf_shape& s, const tf_blob_off& o, const float* W, const float* pooled,
                 const int32_t* n_hits, int64_t B, float* out, float* out_q, float* out_pool,
                 unsigned long long* err, cudaStream_t st) {
  pool_head_kernel<<<(unsigned)B, 128, 0, st>>>(pooled, nullptr, nullptr, n_hits, B, s, W + o.head_g, W + o.head_w1,
                                                 W + o.head_b1, W + o.head_w2, W + o.head_b2, out, out_q, out_pool,
                                                 err);
  return cudaPeekAtLastError() == cudaSuccess ? TRACKFIT_OK : TRACKFIT_ERR_CUDA;
}
