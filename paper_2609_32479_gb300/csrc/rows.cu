// Packed-row tensor-core path for the paper's own topology (Sec. 3.2: concatenated
// directions, endpoint or mean readout) and for the Transformer encoder of its
// encoder comparison (App. A.3), with 16-bit operands (Sec. 3.5: fp16 projections,
// fp32 accumulation and recurrence).
//
// Layout: only valid hits are stored (Sec. 3.5, packed and unpadded).  Track b's
// hit t is row row0[b] + t of every per-hit matrix; row0 is the exclusive prefix
// sum of the valid hit counts (a track whose count is outside [1, max_hits] has
// no rows and a NaN output).  Every per-hit matrix product is one launch of
// row_gemm_kernel over all rows of a chunk:
//   C[row][n] = epilogue(sum_k A[row][k] W[n][k])
// A (16-bit activations, [rows][K]) and W (16-bit weights, PyTorch [N][K]) are
// both K-major, TMA-staged with 128-byte swizzle; the fp32 accumulator lives in
// tensor memory with lane = row, column = output channel, so one epilogue thread
// owns one hit row: bias, SiLU, the sigmoid of the update gates, the residual
// addition and the RMSNorm of the next pre-norm block (a reduction over the row)
// are applied in registers and the results leave in the precision their consumer
// reads (16-bit operands for the next product, fp32 for the residual stream and
// the scans).  Between products run the CUDA-core kernels that are not
// contractions: the Fourier featurisation, the gated scans along each track (the
// concatenation topology) and the attention within each track (the Transformer),
// the pooling and the head.
//
// Kernel roles (192 threads, one CTA per SM, persistent over 128-row x Nt tiles):
//   warp 0     TMA producer (one elected lane): A and W chunks of 64 k into a ring of stages
//   warp 1     MMA issuer (one elected lane) and TMEM owner: two accumulator buffers
//   warps 2-9  epilogue, TMEM lane quadrant = warp % 4, column half = (warp - 2) / 4
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cudaTypedefs.h>
#include <math.h>

#include <cstring>
#include <map>
#include <type_traits>
#include <vector>

#include "attention.cuh"
#include "sm100_ptx.cuh"
#include "trackfit_internal.h"

using namespace sm100;

namespace {

constexpr int RG_THREADS = 320;
constexpr int RG_EPI_WARPS = 8;                   // two per TMEM lane quadrant, each half of a tile's columns
constexpr int RG_ROWS = 128;                      // rows per tile (MMA M)
constexpr int RG_KC = 64;                         // k per stage (one 128-byte swizzle row of 16-bit values)
constexpr int RG_A_BYTES = RG_ROWS * RG_KC * 2;   // 16 KB
constexpr int RG_MAX_NT = 256;                    // MMA N per tile (two buffers fill the 512 TMEM columns)
constexpr int RG_SMEM_BUDGET = 158 * 1024;        // the ring of stages
constexpr int RG_MISC = 2048;                     // RMSNorm partial sums
constexpr int RG_STG_BUFS = 4;                    // staging buffers per epilogue warp (stores in flight)
constexpr int RG_STG_WARP = RG_STG_BUFS * 2048;   // each a 32 x 16 fp32 (or 16-bit) box
constexpr int RG_MAX_STAGES = 8;
constexpr uint64_t RG_WAIT_NS = 2000000000ull;
constexpr uint64_t RG_DRAIN_NS = 200000000ull;
constexpr size_t RG_WS_BUDGET = (size_t)4 << 30;  // workspace bytes of one handle

// epilogues
enum {
  EP_F32 = 0,        // out32 = v
  EP_PROJ = 1,       // out32 = v: the pre-activations of z_f, n_f, z_b, n_b (the scan applies the sigmoid)
  EP_16 = 2,         // out16 = v
  EP_SILU16 = 3,     // out16 = SiLU(v)
  EP_NORM = 4,       // x = v (+ res): out32 = x, out16 = RMSNorm(x) g
  EP_RES = 5         // out32 = res + v
};

struct RowGemm {
  CUtensorMap ta;             // A [cap][K] 16-bit, box 64 x 128, 128-byte swizzle
  CUtensorMap tw;             // W [N][K] 16-bit, box 64 x Nt, 128-byte swizzle
  CUtensorMap to32;           // out32 [cap][N] fp32, box 16 x 32 (stores)
  CUtensorMap to16;           // out16 [cap][N] 16-bit, box 16 x 32 (stores)
  const int64_t* n_rows;      // device: rows of this chunk
  int K, N, Nt, n_ntiles, kchunks, stages;
  int epi;
  uint32_t idesc;
  const float* bias;          // [N]
  const float* res;           // EP_NORM (optional), EP_RES: fp32 [rows][N]
  const float* gain;          // EP_NORM: [N]
  float rms_eps;
  float* out32;               // fp32 [rows][N]
  void* out16;                // 16-bit [rows][N]
  int fp16;                   // 16-bit format of A, W and out16: 1 fp16, 0 bf16
  int64_t cap;                // rows of the workspace (the row count is clamped to it)
  unsigned long long* err;    // [1]: expired bounded waits
  uint64_t wait_ns;
};

struct RgBars {
  uint64_t full[RG_MAX_STAGES], empty[RG_MAX_STAGES];
  uint64_t acc_full[2], acc_empty[2], drain;
  uint64_t ssb[4];            // RMSNorm: the two warps of a lane quadrant exchange their partial sums
  uint32_t tmem_base;
  int abort;
  int never;                  // a flag nothing sets: for the waits at exit that must not give up on abort
};

// sigma(x) = 1 / (1 + e^-x) with the hardware exponential (ex2 of -x log2 e) and
// the hardware reciprocal (two MUFU operations, no branch): a few ulp of fp32, far
// below the 16-bit rounding of the operands it feeds (e^-x = inf for x < -88
// gives 1 / inf = 0).
__device__ __forceinline__ float sigm(float x) { return __fdividef(1.0f, 1.0f + __expf(-x)); }

__device__ __forceinline__ uint32_t pack16(float a, float b, int fp16) {   // a -> low half
  if (fp16) {
    const __half2 h = __floats2half2_rn(a, b);
    return *reinterpret_cast<const uint32_t*>(&h);
  }
  const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<const uint32_t*>(&h);
}

}  // namespace

namespace {

// ------------------------------------------------------------------ the GEMM
__device__ __forceinline__ void sts4(uint32_t addr, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
  asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(a), "r"(b), "r"(c), "r"(d) : "memory");
}

// Output of a warp's 32 rows, 16 columns (one box) at a time, fp32 or 16-bit:
// every lane writes its row's 16 values into one of the warp's staging buffers,
// then one lane stores the [32][16] boxes of a group of two with TMA.  The
// buffers use the tensor maps' swizzled layouts (fp32 rows of 64 bytes: 16-byte
// piece c of row r at c ^ ((r >> 1) & 3); 16-bit rows of 32 bytes: piece c at
// c ^ ((r >> 2) & 1)), so the 8 lanes of a quarter warp write 8 different bank
// groups.  Two groups of two buffers alternate; a group's buffers are rewritten
// only after the stores that read them two groups earlier have finished reading.
struct Emit {
  uint32_t stg;     // this warp's staging area (RG_STG_BUFS = 4 buffers of 2 KB)
  int group;        // groups flushed so far
  __device__ __forceinline__ uint32_t buf(int slot) const {
    return stg + (uint32_t)((((group & 1) << 1) + slot) * 2048);
  }
  __device__ __forceinline__ void begin(int lane) {
    if (lane == 0) bulk_wait_read_keep(1);
    __syncwarp();
  }
  __device__ __forceinline__ void put(const RowGemm& g, int lane, int slot, const float (&v)[16], bool is32) {
    if (is32) {
      const uint32_t a = buf(slot) + lane * 64;
      const int sw = (lane >> 1) & 3;
#pragma unroll
      for (int j = 0; j < 4; ++j)
        sts4(a + 16 * (j ^ sw), __float_as_uint(v[4 * j]), __float_as_uint(v[4 * j + 1]),
             __float_as_uint(v[4 * j + 2]), __float_as_uint(v[4 * j + 3]));
    } else {
      const uint32_t a = buf(slot) + lane * 32;
      const int sw = (lane >> 2) & 1;
#pragma unroll
      for (int j = 0; j < 2; ++j)
        sts4(a + 16 * (j ^ sw), pack16(v[8 * j], v[8 * j + 1], g.fp16), pack16(v[8 * j + 2], v[8 * j + 3], g.fp16),
             pack16(v[8 * j + 4], v[8 * j + 5], g.fp16), pack16(v[8 * j + 6], v[8 * j + 7], g.fp16));
    }
  }
  // count (1 or 2) boxes at columns nb0, nb0 + 16 of rows row .. row + 31
  __device__ __forceinline__ void flush(const RowGemm& g, int lane, bool is32, int nb0, int count, int row) {
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) {
      const CUtensorMap* m = is32 ? &g.to32 : &g.to16;
      tma_store_2d(m, buf(0), nb0, row);
      if (count > 1) tma_store_2d(m, buf(1), nb0 + 16, row);
      bulk_commit();
    }
    ++group;
  }
};


__device__ void rg_fail(const RowGemm& g, RgBars* b) {
  if (atomicExch(&b->abort, 1) == 0) atomicAdd(g.err + 1, 1ull);
}

__global__ void __launch_bounds__(RG_THREADS, 1) row_gemm_kernel(const __grid_constant__ RowGemm g) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  const int stage_bytes = RG_A_BYTES + g.Nt * 128;
  RgBars* bars = reinterpret_cast<RgBars*>(smem_raw + (base - raw) + (size_t)g.stages * stage_bytes);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < g.stages; ++s) {
      mbar_init(smem_u32(&bars->full[s]), 1);
      mbar_init(smem_u32(&bars->empty[s]), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(smem_u32(&bars->acc_full[b]), 1);
      mbar_init(smem_u32(&bars->acc_empty[b]), RG_EPI_WARPS);   // one arrival per epilogue warp
    }
    for (int q = 0; q < 4; ++q) mbar_init(smem_u32(&bars->ssb[q]), 2);
    mbar_init(smem_u32(&bars->drain), 1);
    bars->abort = 0;
    bars->never = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&bars->tmem_base), 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars->tmem_base;
  const int64_t rows = *g.n_rows < g.cap ? *g.n_rows : g.cap;
  const int64_t total = ((rows + RG_ROWS - 1) / RG_ROWS) * g.n_ntiles;
  volatile int* abort = &bars->abort;
  volatile int* never = &bars->never;

  if (warp == 0 && lane == 0) {
    // ---------------- TMA producer
    uint32_t armed[RG_MAX_STAGES];
    for (int s = 0; s < RG_MAX_STAGES; ++s) armed[s] = 0;
    int s = 0;
    uint32_t ph = 0;
    for (int64_t t = blockIdx.x; t < total && !*abort; t += gridDim.x) {
      const int m0 = (int)(t / g.n_ntiles) * RG_ROWS, n0 = (int)(t % g.n_ntiles) * g.Nt;
      for (int kc = 0; kc < g.kchunks; ++kc) {
        if (!mbar_wait(smem_u32(&bars->empty[s]), ph ^ 1u, abort, g.wait_ns)) {
          rg_fail(g, bars);
          break;
        }
        const uint32_t a_s = base + (uint32_t)(s * stage_bytes), fb = smem_u32(&bars->full[s]);
        mbar_arrive_expect_tx(fb, (uint32_t)stage_bytes);
        tma_load_2d(a_s, &g.ta, fb, kc * RG_KC, m0);
        tma_load_2d(a_s + RG_A_BYTES, &g.tw, fb, kc * RG_KC, n0);
        ++armed[s];
        if (++s == g.stages) {
          s = 0;
          ph ^= 1u;
        }
      }
    }
    // no copy may land after the CTA has gone: wait for the last phase armed on
    // every stage (already complete on the normal path)
    for (int i = 0; i < g.stages; ++i)
      if (armed[i] && !mbar_wait(smem_u32(&bars->full[i]), (armed[i] - 1) & 1u, never, RG_DRAIN_NS))
        rg_fail(g, bars);
  } else if (warp == 1 && lane == 0) {
    // ---------------- MMA issuer
    int s = 0;
    uint32_t ph = 0;
    int acc_k = 0;
    bool issued = false;
    for (int64_t t = blockIdx.x; t < total && !*abort; t += gridDim.x) {
      const int buf = acc_k & 1;
      const uint32_t aph = (uint32_t)(acc_k >> 1) & 1u;
      if (!mbar_wait(smem_u32(&bars->acc_empty[buf]), aph ^ 1u, abort, g.wait_ns)) {
        rg_fail(g, bars);
        break;
      }
      tc_fence_after();
      const uint32_t d = tmem + (uint32_t)(buf * RG_MAX_NT);
      bool ok = true;
      for (int kc = 0; kc < g.kchunks; ++kc) {
        if (!mbar_wait(smem_u32(&bars->full[s]), ph, abort, g.wait_ns)) {
          rg_fail(g, bars);
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t a_s = base + (uint32_t)(s * stage_bytes), w_s = a_s + RG_A_BYTES;
#pragma unroll
        for (int k = 0; k < RG_KC / 16; ++k)
          umma_f16(d, sdesc_sw128(a_s + 32 * k, 16, 1024), sdesc_sw128(w_s + 32 * k, 16, 1024), g.idesc,
                   (kc | k) ? 1u : 0u);
        issued = true;
        umma_commit(smem_u32(&bars->empty[s]));
        if (++s == g.stages) {
          s = 0;
          ph ^= 1u;
        }
      }
      if (!ok) break;
      umma_commit(smem_u32(&bars->acc_full[buf]));
      ++acc_k;
    }
    // every MMA complete before TMEM is freed
    if (issued) {
      umma_commit(smem_u32(&bars->drain));
      if (!mbar_wait(smem_u32(&bars->drain), 0, never, RG_DRAIN_NS)) rg_fail(g, bars);
    }
  } else if (warp >= 2) {
    // ---------------- epilogue: this warp's 32 rows and half of the columns of each tile
    const int q = warp & 3, hs = (warp - 2) >> 2;
    // misc: RMSNorm partial sums [2][2][128]
    const uint32_t misc = base + (uint32_t)(g.stages * stage_bytes) + 1024u;
    float* ssx = reinterpret_cast<float*>(smem_raw + (misc - raw));
    Emit emit{misc + (uint32_t)RG_MISC + (uint32_t)((warp - 2) * RG_STG_WARP), 0};
    static_assert(RG_STG_BUFS == 4, "the epilogue's staging rotates two groups of two buffers");
    const int U = g.Nt / 16, ub = hs ? (U + 1) / 2 : 0, ue = hs ? U : (U + 1) / 2;
    int acc_k = 0, norms = 0;
    for (int64_t t = blockIdx.x; t < total; t += gridDim.x) {
      const int buf = acc_k & 1;
      const uint32_t aph = (uint32_t)(acc_k >> 1) & 1u;
      if (!mbar_wait(smem_u32(&bars->acc_full[buf]), aph, abort, g.wait_ns)) {
        if (lane == 0) rg_fail(g, bars);
        break;
      }
      tc_fence_after();
      const int64_t row = (t / g.n_ntiles) * RG_ROWS + 32 * q + lane;
      const int rbox = (int)((t / g.n_ntiles) * RG_ROWS + 32 * q);   // first row of this warp's boxes
      const int n0 = (int)(t % g.n_ntiles) * g.Nt;
      const bool live = row < rows;
      const uint32_t tq = tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(buf * RG_MAX_NT);
      // one pass over this warp's 16-column units, the next unit's TMEM load in
      // flight while the current one is processed.  mode 0: the epilogue; 1: the
      // residual stream of EP_NORM and its sum of squares; 2: its normed operand.
      auto pass = [&](int mode, float inv) -> float {
        const bool is32 = mode == 1 || (mode == 0 && g.epi != EP_16 && g.epi != EP_SILU16);
        // EP_NORM's first pass writes x = res + (acc + b) back over the accumulator,
        // so the second pass reads x from TMEM instead of forming it again
        const bool x_in_tmem = mode == 2;
        const bool use_res = g.res && live && !x_in_tmem;
        // a unit's residual (64 bytes of the thread's row) is prefetched into L1
        // together with that unit's TMEM load, one unit ahead
        auto prefetch_res = [&](int u) {
          if (use_res) asm volatile("prefetch.global.L1 [%0];" ::"l"(g.res + row * g.N + n0 + 16 * u));
        };
        float ss = 0.0f, cur[16], nxt[16];
        if (ub < ue) {
          tmem_ld16(tq + 16 * ub, cur);
          prefetch_res(ub);
          tmem_ld_wait();
        }
        for (int u = ub; u < ue; ++u) {
          const int slot = (u - ub) & 1;
          if (slot == 0) emit.begin(lane);
          if (u + 1 < ue) {
            tmem_ld16(tq + 16 * (u + 1), nxt);
            prefetch_res(u + 1);
          }
          const int nb = n0 + 16 * u;
          if (!x_in_tmem) {
            const float4* bb = reinterpret_cast<const float4*>(g.bias + nb);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              const float4 w = __ldg(bb + i);
              cur[4 * i] += w.x;
              cur[4 * i + 1] += w.y;
              cur[4 * i + 2] += w.z;
              cur[4 * i + 3] += w.w;
            }
          }
          if (use_res) {   // x + (acc + b)
            const float4* rr = reinterpret_cast<const float4*>(g.res + row * g.N + nb);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              const float4 a = rr[i];
              cur[4 * i] = a.x + cur[4 * i];
              cur[4 * i + 1] = a.y + cur[4 * i + 1];
              cur[4 * i + 2] = a.z + cur[4 * i + 2];
              cur[4 * i + 3] = a.w + cur[4 * i + 3];
            }
          }
          if (mode == 1) {
            tmem_st16(tq + 16 * u, cur);   // x for the second pass (not the unit being loaded)
#pragma unroll
            for (int i = 0; i < 16; ++i) ss = fmaf(cur[i], cur[i], ss);
          } else if (mode == 2) {
            const float4* gn = reinterpret_cast<const float4*>(g.gain + nb);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              const float4 w = __ldg(gn + i);
              cur[4 * i] = cur[4 * i] * inv * w.x;
              cur[4 * i + 1] = cur[4 * i + 1] * inv * w.y;
              cur[4 * i + 2] = cur[4 * i + 2] * inv * w.z;
              cur[4 * i + 3] = cur[4 * i + 3] * inv * w.w;
            }
          } else if (g.epi == EP_SILU16) {
#pragma unroll
            for (int i = 0; i < 16; ++i) cur[i] = cur[i] * sigm(cur[i]);
          }
          emit.put(g, lane, slot, cur, is32);
          if (slot == 1 || u + 1 == ue) emit.flush(g, lane, is32, nb - 16 * slot, slot + 1, rbox);
          if (u + 1 < ue) {
            tmem_ld_wait();
#pragma unroll
            for (int i = 0; i < 16; ++i) cur[i] = nxt[i];
          }
        }
        return ss;
      };
      bool ok = true;
      if (g.epi == EP_NORM) {
        // the row's sum of squares: this warp's half, then the partner's through
        // shared memory (double-buffered by tile) and a two-arrival barrier
        const int par = norms & 1;
        ssx[(par * 2 + hs) * 128 + 32 * q + lane] = pass(1, 0.0f);
        tmem_st_wait();   // x is in TMEM before the second pass reads it
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&bars->ssb[q]));
        ok = mbar_wait(smem_u32(&bars->ssb[q]), (uint32_t)par, abort, g.wait_ns);
        if (ok) {
          const float tot = ssx[(par * 2) * 128 + 32 * q + lane] + ssx[(par * 2 + 1) * 128 + 32 * q + lane];
          pass(2, 1.0f / sqrtf(tot / (float)g.N + g.rms_eps));
        } else if (lane == 0) {
          rg_fail(g, bars);
        }
        ++norms;
      } else {
        pass(0, 0.0f);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&bars->acc_empty[buf]));
      ++acc_k;
      if (!ok) break;
    }
    if (lane == 0) bulk_wait_all();   // every store done before the CTA leaves
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

}  // namespace

namespace {

// ------------------------------------------------------------------ row plan
// row0[b] = sum of the valid hit counts of tracks < b (a count outside [1, T]
// counts 0); row0[B] = the chunk's rows.  Three launches: block totals, one CTA
// scanning the totals, each block's scan.
constexpr int PLAN_NT = 1024;

__device__ __forceinline__ int64_t valid_count(const int32_t* n_hits, int64_t b, int64_t B, int T) {
  if (b >= B) return 0;
  const int n = n_hits[b];
  return (n >= 1 && n <= T) ? n : 0;
}

// inclusive scan of one value per thread over the CTA (PLAN_NT threads)
__device__ int64_t cta_inclusive_scan(int64_t v, int64_t* warp_tot) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int64_t u = __shfl_up_sync(0xffffffffu, v, o);
    if (lane >= o) v += u;
  }
  if (lane == 31) warp_tot[warp] = v;
  __syncthreads();
  if (warp == 0) {
    int64_t w = warp_tot[lane];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int64_t u = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += u;
    }
    warp_tot[lane] = w;
  }
  __syncthreads();
  const int64_t r = v + (warp ? warp_tot[warp - 1] : 0);
  __syncthreads();
  return r;
}

__global__ void __launch_bounds__(PLAN_NT) plan_totals(const int32_t* __restrict__ n_hits, int64_t B, int T,
                                                       int64_t* __restrict__ tot) {
  __shared__ int64_t wt[32];
  const int64_t b = blockIdx.x * (int64_t)PLAN_NT + threadIdx.x;
  const int64_t s = cta_inclusive_scan(valid_count(n_hits, b, B, T), wt);
  if (threadIdx.x == PLAN_NT - 1) tot[blockIdx.x] = s;
}

__global__ void __launch_bounds__(PLAN_NT) plan_scan_totals(int64_t* __restrict__ tot, int nblk) {
  __shared__ int64_t wt[32];
  __shared__ int64_t last;
  int64_t carry = 0;
  for (int i0 = 0; i0 < nblk; i0 += PLAN_NT) {   // exclusive scan in place
    const int i = i0 + threadIdx.x;
    const int64_t v = i < nblk ? tot[i] : 0;
    const int64_t s = cta_inclusive_scan(v, wt);
    if (i < nblk) tot[i] = carry + s - v;
    if (threadIdx.x == PLAN_NT - 1) last = s;
    __syncthreads();
    carry += last;
    __syncthreads();
  }
  if (threadIdx.x == 0) tot[nblk] = carry;   // the total after the offsets
}

__global__ void __launch_bounds__(PLAN_NT) plan_rows(const int32_t* __restrict__ n_hits, int64_t B, int T,
                                                     const int64_t* __restrict__ tot, int64_t* __restrict__ row0) {
  __shared__ int64_t wt[32];
  const int64_t b = blockIdx.x * (int64_t)PLAN_NT + threadIdx.x;
  const int64_t v = valid_count(n_hits, b, B, T);
  const int64_t s = cta_inclusive_scan(v, wt) + tot[blockIdx.x];
  if (b < B) row0[b] = s - v;
  if (b == B - 1) row0[B] = s;
}

// ------------------------------------------------------------------ Fourier rows
// Sec. 3.2: u = (v - min) / (max - min) per feature, then sin(pi s_k u) and
// cos(pi s_k u) for the 16 scales, feature-major ([f][sin k, cos k]).  One thread
// per (track, hit, feature); the 2 n_fourier values leave as 16-bit operands of
// the embedding product.  Hit rows: padded hits[b][t] or packed hits[offs[b] + t].
// fp32 only (fp64 is slow on this part): v - min (TwoSum) times the two-float
// 1 / (max - min) and s_k (TwoProduct) give the argument as an unevaluated sum
// of two floats, reduced modulo 2 exactly, so the sine and cosine carry only the
// final fp32 rounding of the argument.  When s_{k+3} = 2 s_k for every k (the
// scales 2^(k/3)), the scales k = 0-2, 6-8, 12-14 are evaluated and the others
// follow by one double-angle step (2 s c, (c - s)(c + s)).
template <typename T16>
__global__ void fourier_rows_kernel(const float* __restrict__ hits, const int64_t* __restrict__ offs,
                                    const int32_t* __restrict__ n_hits, int64_t B, tf_shape s,
                                    const int64_t* __restrict__ row0, int doubling, T16* __restrict__ e) {
  const int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (i >= B * s.T * s.F) return;
  const int64_t b = i / (s.T * s.F);
  const int r = (int)(i - b * s.T * s.F), t = r / s.F, f = r - t * s.F;
  const int n = n_hits[b];
  if (n < 1 || n > s.T || t >= n) return;
  const float v = offs ? hits[(offs[b] + t) * s.F + f] : hits[(b * s.T + t) * s.F + f];
  const float mn = -s.feat_min[f], ih = s.feat_inv_range[f];
  const float dh = v + mn;
  const float bv = dh - v;
  const float dl = (v - (dh - bv)) + (mn - bv);
  const float uh = dh * ih;
  const float ul = fmaf(dh, ih, -uh) + fmaf(dh, s.feat_inv_lo[f], dl * ih);
  float sv[TRACKFIT_MAX_FOURIER], cv[TRACKFIT_MAX_FOURIER];
#pragma unroll
  for (int k = 0; k < TRACKFIT_MAX_FOURIER; ++k) {
    if (doubling && (k % 6) >= 3) {   // s_k = 2 s_{k-3}
      sv[k] = 2.0f * sv[k - 3] * cv[k - 3];
      cv[k] = (cv[k - 3] - sv[k - 3]) * (cv[k - 3] + sv[k - 3]);
      continue;
    }
    const float sk = s.scale[k];
    const float xh = uh * sk;
    const float xl = fmaf(uh, sk, -xh) + ul * sk;
    const float r = (xh - 2.0f * rintf(0.5f * xh)) + xl;
    sv[k] = sinpif(r);
    cv[k] = cospif(r);
  }
  // the feature's 32 values (64 bytes, 16-byte aligned) in four vector stores
  uint4* o = reinterpret_cast<uint4*>(e + (row0[b] + t) * s.E + f * 2 * TRACKFIT_MAX_FOURIER);
  const int h16 = sizeof(T16) == 2 && std::is_same<T16, __half>::value;
#pragma unroll
  for (int q = 0; q < 2; ++q) {
    o[q] = make_uint4(pack16(sv[8 * q], sv[8 * q + 1], h16), pack16(sv[8 * q + 2], sv[8 * q + 3], h16),
                      pack16(sv[8 * q + 4], sv[8 * q + 5], h16), pack16(sv[8 * q + 6], sv[8 * q + 7], h16));
    o[2 + q] = make_uint4(pack16(cv[8 * q], cv[8 * q + 1], h16), pack16(cv[8 * q + 2], cv[8 * q + 3], h16),
                          pack16(cv[8 * q + 4], cv[8 * q + 5], h16), pack16(cv[8 * q + 6], cv[8 * q + 7], h16));
  }
}

// ------------------------------------------------------------------ scans
// The two gated scans of one concatenation layer (Sec. 3.2, Eq. 2) over each
// track's rows: z_t = sigma(p_z), h_t = (1 - z_t) h_{t-1} + z_t n_t forward, the
// same backward with the reverse gates (the projection stores the
// pre-activations; the sigmoid runs here, in a kernel bound by HBM).  One thread per (track,
// channel).  y16 (optional): the concatenated states [h_f | h_b] per row as the
// next layer's 16-bit operand.  pooled (optional, the last layer): endpoints, the
// forward state at the last hit and the reverse state at the first, or the mean
// of [h_f | h_b] over the hits.
template <typename T16>
__global__ void concat_scan_rows_kernel(const float* __restrict__ pr, const int64_t* __restrict__ row0,
                                        const int32_t* __restrict__ n_hits, int64_t B, int T, int H,
                                        T16* __restrict__ y16, float* __restrict__ pooled, int pool) {
  const int64_t b = blockIdx.x;
  const int c = blockIdx.y * blockDim.x + threadIdx.x;
  if (b >= B || c >= H) return;
  const int n = n_hits[b];
  if (n < 1 || n > T) return;
  const int64_t r0 = row0[b];
  const int ldp = 4 * H;
  // the two directions are independent chains: step t forward and step n - 1 - t
  // backward run together, each in hit order for its own direction
  float hf = 0.0f, hb = 0.0f, sf = 0.0f, sb = 0.0f;
  for (int t = 0; t < n; ++t) {
    const float* pf = pr + (r0 + t) * ldp;
    const float* pb = pr + (r0 + n - 1 - t) * ldp;
    const float zf = pf[c], nf = pf[H + c], zb = pb[2 * H + c], nb = pb[3 * H + c];
    hf = fmaf(sigm(zf), nf - hf, hf);
    hb = fmaf(sigm(zb), nb - hb, hb);
    if (y16) {
      tf_attn::put(y16 + (r0 + t) * 2 * H + c, hf);
      tf_attn::put(y16 + (r0 + n - 1 - t) * 2 * H + H + c, hb);
    }
    sf += hf;
    sb += hb;
  }
  if (pooled) {
    pooled[b * 2 * H + c] = pool == TRACKFIT_POOL_ENDPOINTS ? hf : sf / (float)n;
    pooled[b * 2 * H + H + c] = pool == TRACKFIT_POOL_ENDPOINTS ? hb : sb / (float)n;
  }
}

// Mean over each track's rows of the last layer's output x [rows][D] (the
// Transformer's readout); one thread per (track, channel), hits in order.
__global__ void pool_mean_rows_kernel(const float* __restrict__ x, const int64_t* __restrict__ row0,
                                      const int32_t* __restrict__ n_hits, int64_t B, int T, int D,
                                      float* __restrict__ pooled) {
  const int64_t b = blockIdx.x;
  const int c = blockIdx.y * blockDim.x + threadIdx.x;
  if (b >= B || c >= D) return;
  const int n = n_hits[b];
  if (n < 1 || n > T) return;
  const int64_t r0 = row0[b];
  float acc = 0.0f;
  for (int t = 0; t < n; ++t) acc += x[(r0 + t) * D + c];
  pooled[b * D + c] = acc / (float)n;
}

}  // namespace

// ------------------------------------------------------------------ host side
struct tf_rows_state {
  int fp16;
  int nsm;
  uint16_t* w16;            // every product's weights, 16-bit, back to back
  float* hws;               // the head's workspace, chunk x (P + 128 + Q) floats
  float* vec;               // the products' bias and gain vectors, each 16-byte aligned
  int doubling;             // fourier_scale[k + 3] == 2 fourier_scale[k] for every k
  int64_t chunk, cap;       // tracks per chunk; rows of the workspace (chunk * max_hits)
  int64_t* row0;            // [chunk + 1]
  int64_t* tot;             // [chunk / 1024 + 1]
  uint16_t *a0, *hs16, *xy16, *o16;
  float *p32, *x32, *x1, *pooled;
  RowGemm e1, e2;
  RowGemm lay[TF_MAX_LAYERS][4];
  size_t smem;
  uint64_t wait_ns;
};

namespace {

PFN_cuTensorMapEncodeTiled_v12000 rows_encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

// 16-bit matrix [rows][cols] row-major -> tensor map of 64-column x box_rows boxes
// with 128-byte swizzle (out-of-range elements read as zero).
bool rows_map(CUtensorMap* m, const void* ptr, uint64_t rows, uint64_t cols, uint32_t box_rows, int fp16) {
  auto fn = rows_encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {64, box_rows};
  cuuint32_t es[2] = {1, 1};
  return fn(m, fp16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr),
            dims, strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Output matrix [rows][cols] row-major (fp32, or 16-bit) -> tensor map of
// 16-column x 32-row boxes for the epilogue's TMA stores, swizzled over the box
// row (64 bytes for fp32, 32 bytes for 16-bit).
bool out_map(CUtensorMap* m, const void* ptr, uint64_t rows, uint64_t cols, int bytes, int fp16) {
  auto fn = rows_encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * (uint64_t)bytes};
  cuuint32_t box[2] = {16, 32};
  cuuint32_t es[2] = {1, 1};
  const CUtensorMapDataType t = bytes == 4 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32
                                : fp16     ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16
                                           : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
  return fn(m, t, 2, const_cast<void*>(ptr), dims, strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
            bytes == 4 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_32B,
            CU_TENSOR_MAP_L2_PROMOTION_NONE,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// The store maps of a product whose output pointers are set.
bool finish_gemm(RowGemm& g, const tf_rows_state* r) {
  const bool need32 = g.epi == EP_F32 || g.epi == EP_PROJ || g.epi == EP_RES || g.epi == EP_NORM;
  const bool need16 = g.epi == EP_16 || g.epi == EP_SILU16 || g.epi == EP_NORM;
  if (need32 != (g.out32 != nullptr) || need16 != (g.out16 != nullptr)) return false;
  return (!g.out32 || out_map(&g.to32, g.out32, (uint64_t)r->cap, (uint64_t)g.N, 4, r->fp16)) &&
         (!g.out16 || out_map(&g.to16, g.out16, (uint64_t)r->cap, (uint64_t)g.N, 2, r->fp16));
}

// The MMA N of one tile: N itself up to 256, else the smallest equal split into
// multiples of 16 (0 if there is none).
int tile_n(int N) {
  for (int parts = (N + RG_MAX_NT - 1) / RG_MAX_NT; parts <= N / 16; ++parts)
    if (N % parts == 0 && (N / parts) % 16 == 0) return N / parts;
  return 0;
}

// alignment slack, the ring of stages, the barriers (one 1 KB block), the
// exchange area of the epilogue warps, their staging buffers
size_t gemm_smem(const RowGemm& g) {
  return 1024 + (size_t)g.stages * (RG_A_BYTES + g.Nt * 128) + 1024 + RG_MISC + RG_EPI_WARPS * RG_STG_WARP;
}

// A [cap][K] (16-bit, row stride K) times W [N][K]; the epilogue's pointers are set by the caller.
bool make_gemm(RowGemm& g, const tf_rows_state* r, const void* A, int K, const uint16_t* W, int N, int epi) {
  std::memset(&g, 0, sizeof(g));
  g.K = K;
  g.N = N;
  g.Nt = tile_n(N);
  if (!g.Nt || (K % 8) != 0) return false;
  g.n_ntiles = N / g.Nt;
  g.kchunks = (K + RG_KC - 1) / RG_KC;
  const int stage = RG_A_BYTES + g.Nt * 128;
  g.stages = (int)((RG_SMEM_BUDGET - 1024) / stage);
  if (g.stages > RG_MAX_STAGES) g.stages = RG_MAX_STAGES;
  if (g.stages < 2) return false;
  g.epi = epi;
  g.idesc = idesc_f16(RG_ROWS, g.Nt, r->fp16 ? 0u : 1u, false, false);
  g.fp16 = r->fp16;
  g.wait_ns = RG_WAIT_NS;
  return rows_map(&g.ta, A, (uint64_t)r->cap, (uint64_t)K, RG_ROWS, r->fp16) &&
         rows_map(&g.tw, W, (uint64_t)N, (uint64_t)K, (uint32_t)g.Nt, r->fp16);
}

// One product over the chunk's rows; the handle's timing hook (trackfit_profile)
// brackets every product launch of this path.
int launch_gemm(trackfit_ctx* h, RowGemm& g, const int64_t* n_rows, cudaStream_t st) {
  const tf_rows_state* r = h->rows;
  g.n_rows = n_rows;
  g.cap = r->cap;
  g.err = h->d_err;
  g.wait_ns = r->wait_ns;
  tf_prof_begin(h, st);
  row_gemm_kernel<<<r->nsm, RG_THREADS, gemm_smem(g), st>>>(g);
  tf_prof_end(h, st);
  const cudaError_t e = cudaPeekAtLastError();
  if (e == cudaSuccess) return TRACKFIT_OK;
  tf_note_cuda(e, "row_gemm_kernel launch");
  return TRACKFIT_ERR_CUDA;
}

uint16_t to16(float f, int fp16) {
  if (fp16) {
    const __half v = __float2half_rn(f);
    return *reinterpret_cast<const uint16_t*>(&v);
  }
  const __nv_bfloat16 v = __float2bfloat16_rn(f);
  return *reinterpret_cast<const uint16_t*>(&v);
}

}  // namespace

bool tf_rows_supported(const tf_shape& s) {
  if (s.precision != TRACKFIT_BF16_PROJ && s.precision != TRACKFIT_FP16_PROJ) return false;
  if (s.topology != TRACKFIT_TOPOLOGY_CONCAT && s.topology != TRACKFIT_TOPOLOGY_ATTENTION) return false;
  if (tile_n(s.D) != s.D) return false;   // the row-wide epilogues need a whole row in one tile
  // CONCAT: the sigmoid of the update-gate blocks is chosen per 16 columns
  if (s.topology == TRACKFIT_TOPOLOGY_CONCAT) return (s.H % 16) == 0 && tile_n(4 * s.H) != 0;
  return tile_n(3 * s.D) != 0 && tile_n(s.H) != 0;
}

void tf_rows_destroy(trackfit_ctx* h) {
  tf_rows_state* r = h->rows;
  if (!r) return;
  tf_free(r->w16);
  tf_free(r->hws);
  tf_free(r->vec);
  tf_free(r->row0);
  tf_free(r->tot);
  tf_free(r->a0);
  tf_free(r->hs16);
  tf_free(r->xy16);
  tf_free(r->o16);
  tf_free(r->p32);
  tf_free(r->x32);
  tf_free(r->x1);
  tf_free(r->pooled);
  delete r;
  h->rows = nullptr;
}

int tf_rows_wait_limit(trackfit_ctx* h, int64_t limit_ns) {
  if (!h->rows) return TRACKFIT_ERR_UNSUPPORTED;
  h->rows->wait_ns = limit_ns > 0 ? (uint64_t)limit_ns : RG_WAIT_NS;
  return TRACKFIT_OK;
}

int tf_rows_create(trackfit_ctx* h, const float* host_w) {
  const tf_shape& s = h->s;
  const tf_blob_off& o = h->off;
  tf_rows_state* r = new (std::nothrow) tf_rows_state();
  if (!r) return TRACKFIT_ERR_OOM;
  h->rows = r;   // freed by tf_rows_destroy on any failure below
  r->fp16 = s.precision == TRACKFIT_FP16_PROJ;
  r->wait_ns = RG_WAIT_NS;
  r->doubling = 1;
  for (int k = 0; k + 3 < TRACKFIT_MAX_FOURIER; ++k)
    if (s.scale[k + 3] != 2.0f * s.scale[k]) r->doubling = 0;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&r->nsm, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return TRACKFIT_ERR_CUDA;
  const bool attn = s.topology == TRACKFIT_TOPOLOGY_ATTENTION;
  const size_t D = s.D, H = s.H, E = s.E;
  // the 16-bit weights of every product: (blob offset, N, K)
  struct Mat { size_t off, n, k, at; };
  std::vector<Mat> mats;
  mats.push_back({o.emb_w1, D, E, 0});
  mats.push_back({o.emb_w2, D, D, 0});
  for (int l = 0; l < s.L; ++l) {
    const tf_layer_off& lo = o.layer[l];
    if (attn) {
      mats.push_back({lo.w_in, 3 * D, D, 0});
      mats.push_back({lo.w_m, D, D, 0});
      mats.push_back({lo.w1, H, D, 0});
      mats.push_back({lo.w2, D, H, 0});
    } else {
      mats.push_back({lo.w_in, 4 * H, l == 0 ? D : 2 * H, 0});
    }
  }
  size_t n16 = 0;
  for (Mat& m : mats) {
    m.at = n16;
    n16 += (m.n * m.k + 63) / 64 * 64;   // 128-byte aligned starts
  }
  std::vector<uint16_t> w(n16, 0);
  for (const Mat& m : mats)
    for (size_t i = 0; i < m.n * m.k; ++i) w[m.at + i] = to16(host_w[m.off + i], r->fp16);
  int st = tf_status_from_cuda(tf_malloc((void**)&r->w16, n16 * 2));
  if (st == TRACKFIT_OK) st = tf_status_from_cuda(cudaMemcpy(r->w16, w.data(), n16 * 2, cudaMemcpyHostToDevice));
  if (st != TRACKFIT_OK) return st;
  // workspace, sized for whole chunks of full-length tracks
  const size_t hsw = attn ? (H > D ? H : D) : D;
  const size_t xyw = attn ? D : (2 * H > D ? 2 * H : D);
  const size_t pw = attn ? 3 * D : 4 * H;
  const size_t row_bytes = 2 * (E + hsw + xyw + (attn ? D : 0)) + 4 * (pw + (attn ? 2 * D : 0));
  const size_t track_bytes = (size_t)s.T * row_bytes + 4 * (2 * (size_t)s.P + s.Hh + s.Q) + 16;
  int64_t chunk = (int64_t)(RG_WS_BUDGET / track_bytes);
  if (chunk > 4194304) chunk = 4194304;
  chunk = chunk / PLAN_NT * PLAN_NT;
  if (chunk < PLAN_NT) return TRACKFIT_ERR_UNSUPPORTED;
  r->chunk = chunk;
  r->cap = chunk * s.T;
  const size_t cap = (size_t)r->cap;
  auto alloc = [&](void** p, size_t bytes) {
    if (st == TRACKFIT_OK) st = tf_status_from_cuda(tf_malloc(p, bytes));
  };
  alloc((void**)&r->row0, (chunk + 1) * sizeof(int64_t));
  alloc((void**)&r->tot, (chunk / PLAN_NT + 2) * sizeof(int64_t));
  alloc((void**)&r->a0, cap * E * 2);
  alloc((void**)&r->hs16, cap * hsw * 2);
  alloc((void**)&r->xy16, cap * xyw * 2);
  alloc((void**)&r->p32, cap * pw * 4);
  alloc((void**)&r->pooled, (size_t)chunk * s.P * 4);
  alloc((void**)&r->hws, (size_t)chunk * (s.P + s.Hh + s.Q) * 4);
  if (attn) {
    alloc((void**)&r->o16, cap * D * 2);
    alloc((void**)&r->x32, cap * D * 4);
    alloc((void**)&r->x1, cap * D * 4);
  }
  if (st != TRACKFIT_OK) return st;
  // 16-byte aligned copies of the bias and gain vectors the epilogues read
  std::map<size_t, size_t> at;
  std::vector<float> hv;
  auto want = [&](size_t off, size_t n) {
    if (at.count(off)) return;
    at[off] = hv.size();
    hv.insert(hv.end(), host_w + off, host_w + off + n);
    hv.resize((hv.size() + 3) / 4 * 4, 0.0f);
  };
  want(o.emb_b1, D);
  want(o.emb_b2, D);
  for (int l = 0; l < s.L; ++l) {
    const tf_layer_off& lo = o.layer[l];
    if (!attn) {
      want(lo.b_in, 4 * H);
      continue;
    }
    want(lo.g, D);
    want(lo.b_in, 3 * D);
    want(lo.b_m, D);
    want(lo.g2, D);
    want(lo.b1, H);
    want(lo.b2, D);
  }
  st = tf_status_from_cuda(tf_malloc((void**)&r->vec, hv.size() * 4));
  if (st == TRACKFIT_OK) st = tf_status_from_cuda(cudaMemcpy(r->vec, hv.data(), hv.size() * 4, cudaMemcpyHostToDevice));
  if (st != TRACKFIT_OK) return st;
  auto V = [&](size_t off) -> const float* { return r->vec + at[off]; };
  // the products of one chunk
  const uint16_t* w16 = r->w16;
  size_t mi = 0;
  bool ok = make_gemm(r->e1, r, r->a0, (int)E, w16 + mats[mi++].at, (int)D, EP_SILU16);
  r->e1.bias = V(o.emb_b1);
  r->e1.out16 = r->hs16;
  ok = ok && make_gemm(r->e2, r, r->hs16, (int)D, w16 + mats[mi++].at, (int)D, attn ? EP_NORM : EP_16);
  r->e2.bias = V(o.emb_b2);
  r->e2.out16 = r->xy16;
  if (attn) {   // x = embedding; the first layer's pre-norm operand
    r->e2.out32 = r->x32;
    r->e2.gain = V(o.layer[0].g);
    r->e2.rms_eps = s.rms_eps;
  }
  for (int l = 0; l < s.L && ok; ++l) {
    const tf_layer_off& lo = o.layer[l];
    RowGemm* g = r->lay[l];
    if (!attn) {   // Sec. 3.2: the layer input (D, then 2H wide) to z_f, n_f, z_b, n_b
      ok = make_gemm(g[0], r, r->xy16, l == 0 ? (int)D : (int)(2 * H), w16 + mats[mi++].at, (int)(4 * H), EP_PROJ);
      g[0].bias = V(lo.b_in);
      g[0].out32 = r->p32;
      continue;
    }
    // App. A.3: qkv of the normed stream; x' = x + W_o o + b_o and its pre-norm;
    // SiLU(W_1 .. + b_1); x = x' + W_2 u + b_2 and the next layer's pre-norm
    ok = make_gemm(g[0], r, r->xy16, (int)D, w16 + mats[mi++].at, (int)(3 * D), EP_F32) &&
         make_gemm(g[1], r, r->o16, (int)D, w16 + mats[mi++].at, (int)D, EP_NORM) &&
         make_gemm(g[2], r, r->xy16, (int)D, w16 + mats[mi++].at, (int)H, EP_SILU16) &&
         make_gemm(g[3], r, r->hs16, (int)H, w16 + mats[mi++].at, (int)D, l + 1 < s.L ? EP_NORM : EP_RES);
    g[0].bias = V(lo.b_in);
    g[0].out32 = r->p32;
    g[1].bias = V(lo.b_m);
    g[1].res = r->x32;
    g[1].gain = V(lo.g2);
    g[1].rms_eps = s.rms_eps;
    g[1].out32 = r->x1;
    g[1].out16 = r->xy16;
    g[2].bias = V(lo.b1);
    g[2].out16 = r->hs16;
    g[3].bias = V(lo.b2);
    g[3].res = r->x1;
    g[3].out32 = r->x32;
    if (l + 1 < s.L) {
      g[3].gain = V(o.layer[l + 1].g);
      g[3].rms_eps = s.rms_eps;
      g[3].out16 = r->xy16;
    }
  }
  ok = ok && finish_gemm(r->e1, r) && finish_gemm(r->e2, r);
  for (int l = 0; l < s.L && ok; ++l)
    for (int k = 0; k < (attn ? 4 : 1) && ok; ++k) ok = finish_gemm(r->lay[l][k], r);
  if (!ok) return TRACKFIT_ERR_CUDA;
  r->smem = gemm_smem(r->e1);
  auto upd = [&](const RowGemm& g) { r->smem = gemm_smem(g) > r->smem ? gemm_smem(g) : r->smem; };
  upd(r->e2);
  for (int l = 0; l < s.L; ++l)
    for (int k = 0; k < (attn ? 4 : 1); ++k) upd(r->lay[l][k]);
  if (cudaFuncSetAttribute(row_gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)r->smem) != cudaSuccess)
    return TRACKFIT_ERR_CUDA;
  {   // one CTA of every product must fit on an SM (registers, shared memory)
    int per_sm = 0;
    const cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, row_gemm_kernel, RG_THREADS, r->smem);
    if (e != cudaSuccess) return tf_status_from_cuda(e);
    if (per_sm < 1) {
      tf_note_cuda(cudaErrorLaunchOutOfResources, "row_gemm_kernel occupancy");
      return TRACKFIT_ERR_UNSUPPORTED;
    }
  }
  if (attn && (tf_attn::allow_smem<__half>(s.T, s.D, s.NH) != cudaSuccess ||
               tf_attn::allow_smem<__nv_bfloat16>(s.T, s.D, s.NH) != cudaSuccess))
    return TRACKFIT_ERR_CUDA;
  return TRACKFIT_OK;
}

namespace {

template <typename T16>
int rows_chunk(trackfit_ctx* h, const float* hits, const int64_t* offs, const int32_t* nc, int64_t nb, float* out,
               float* out_q, float* out_pool, cudaStream_t st) {
  tf_rows_state* r = h->rows;
  const tf_shape& s = h->s;
  unsigned long long* err = h->d_err;   // bad-track counter of the head
  const bool attn = s.topology == TRACKFIT_TOPOLOGY_ATTENTION;
  const int nblk = (int)((nb + PLAN_NT - 1) / PLAN_NT);
  plan_totals<<<nblk, PLAN_NT, 0, st>>>(nc, nb, s.T, r->tot);
  plan_scan_totals<<<1, PLAN_NT, 0, st>>>(r->tot, nblk);
  plan_rows<<<nblk, PLAN_NT, 0, st>>>(nc, nb, s.T, r->tot, r->row0);
  const int64_t* nrows = r->row0 + nb;
  const int64_t nf = nb * s.T * s.F;
  fourier_rows_kernel<T16><<<(unsigned)((nf + 255) / 256), 256, 0, st>>>(hits, offs, nc, nb, s, r->row0, r->doubling,
                                                                         reinterpret_cast<T16*>(r->a0));
  {
    const cudaError_t e = cudaPeekAtLastError();   // the plan and Fourier launches
    if (e != cudaSuccess) {
      tf_note_cuda(e, "row plan / Fourier launch");
      return TRACKFIT_ERR_CUDA;
    }
  }
  if (launch_gemm(h, r->e1, nrows, st) || launch_gemm(h, r->e2, nrows, st)) return TRACKFIT_ERR_CUDA;
  for (int l = 0; l < s.L; ++l) {
    RowGemm* g = r->lay[l];
    if (!attn) {
      if (launch_gemm(h, g[0], nrows, st)) return TRACKFIT_ERR_CUDA;
      const bool last = l + 1 == s.L;
      dim3 grid((unsigned)nb, (unsigned)((s.H + 127) / 128));
      concat_scan_rows_kernel<T16><<<grid, 128, 0, st>>>(r->p32, r->row0, nc, nb, s.T, s.H,
                                                         last ? nullptr : reinterpret_cast<T16*>(r->xy16),
                                                         last ? r->pooled : nullptr, s.pool);
      continue;
    }
    if (launch_gemm(h, g[0], nrows, st)) return TRACKFIT_ERR_CUDA;
    const cudaError_t ea =
        tf_attn::launch<T16>(r->p32, 3 * s.D, r->row0, nc, nb, s.T, s.D, s.NH, reinterpret_cast<T16*>(r->o16), s.D, st);
    if (ea != cudaSuccess) {
      tf_note_cuda(ea, "track_attention_kernel launch");
      return TRACKFIT_ERR_CUDA;
    }
    if (launch_gemm(h, g[1], nrows, st) || launch_gemm(h, g[2], nrows, st) ||
        launch_gemm(h, g[3], nrows, st))
      return TRACKFIT_ERR_CUDA;
  }
  if (attn) {
    dim3 grid((unsigned)nb, (unsigned)((s.D + 127) / 128));
    pool_mean_rows_kernel<<<grid, 128, 0, st>>>(r->x32, r->row0, nc, nb, s.T, s.D, r->pooled);
  }
  return tf_simt_head_batched(s, h->off, h->d_w, r->pooled, nc, nb, r->hws, out, out_q, out_pool, err, st);
}

}  // namespace

int tf_rows_forward(trackfit_ctx* h, const float* hits, const int32_t* n_hits, int64_t B, float* out,
                    float* out_q, float* out_pool, cudaStream_t st, const int64_t* offs) {
  tf_rows_state* r = h->rows;
  const tf_shape& s = h->s;
  for (int64_t c0 = 0; c0 < B; c0 += r->chunk) {
    const int64_t nb = B - c0 < r->chunk ? B - c0 : r->chunk;
    const float* hc = offs ? hits : hits + c0 * s.T * s.F;
    const int64_t* oc = offs ? offs + c0 : nullptr;
    const int e = r->fp16 ? rows_chunk<__half>(h, hc, oc, n_hits + c0, nb, out + c0 * 5,
                                               out_q ? out_q + c0 * s.Q : nullptr,
                                               out_pool ? out_pool + c0 * s.P : nullptr, st)
                          : rows_chunk<__nv_bfloat16>(h, hc, oc, n_hits + c0, nb, out + c0 * 5,
                                                      out_q ? out_q + c0 * s.Q : nullptr,
                                                      out_pool ? out_pool + c0 * s.P : nullptr, st);
    if (e != TRACKFIT_OK) return e;
  }
  return TRACKFIT_OK;
}
