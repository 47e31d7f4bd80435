// Multi-head self-attention within each track: the token mixing of the
// Transformer encoder in the paper's encoder comparison (App. A.3, Tab. A.1: full
// attention over a track's hits, no causal mask).  Per head h of width
// dh = D / NH, query hit t of track b attends to the track's n valid hits:
//   o_t = sum_j softmax_j(q_t . k_j / sqrt(dh)) v_j.
// q, k, v are the fp32 outputs of the qkv projection; scores, softmax and the
// weighted sum run in fp32.
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <stdint.h>

namespace tf_attn {

__device__ __forceinline__ void put(float* p, float v) { *p = v; }
__device__ __forceinline__ void put(__half* p, float v) { *p = __float2half_rn(v); }
__device__ __forceinline__ void put(__nv_bfloat16* p, float v) { *p = __float2bfloat16_rn(v); }

constexpr int THREADS = 128;   // 4 warps; warp w takes heads w, w + 4, ...

// Dynamic shared memory of one CTA: the track's keys and values, T rows of 2 D + 1
// floats (the odd row stride puts key j's channel c in bank (j + c) mod 32).
__host__ __device__ inline size_t smem_bytes(int T, int D) { return (size_t)T * (2 * D + 1) * sizeof(float); }

// One CTA per track.  qkv: rows [q | k | v] of width 3 D at stride ldq; track b's
// hit t is row row0[b] + t (packed rows) or b T + t (padded rows, row0 null).
// o: the attention output, row-aligned with qkv at stride ldo.  With padded rows
// the rows t >= n of a track (all of them for a track whose count is outside
// [1, T]) are written 0; packed rows have no padding.
template <typename OutT>
__global__ void __launch_bounds__(THREADS) track_attention_kernel(const float* __restrict__ qkv, int ldq,
                                                                  const int64_t* __restrict__ row0,
                                                                  const int32_t* __restrict__ n_hits, int64_t B,
                                                                  int T, int D, int NH, OutT* __restrict__ o,
                                                                  int ldo) {
  extern __shared__ float kv[];
  const int64_t b = blockIdx.x;
  if (b >= B) return;
  int n = n_hits[b];
  if (n < 1 || n > T) n = 0;
  const int64_t r0 = row0 ? row0[b] : b * (int64_t)T;
  const int ks = 2 * D + 1;
  for (int i = threadIdx.x; i < n * 2 * D; i += THREADS) {
    const int j = i / (2 * D), c = i - j * (2 * D);
    kv[j * ks + c] = qkv[(r0 + j) * ldq + D + c];
  }
  if (!row0) {   // padded layout: zero the padding rows
    for (int i = threadIdx.x; i < (T - n) * D; i += THREADS) {
      const int t = n + i / D, c = i % D;
      put(o + (r0 + t) * ldo + c, 0.0f);
    }
  }
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int dh = D / NH;
  const float scale = rsqrtf((float)dh);
  for (int h = warp; h < NH; h += THREADS / 32) {
    const int c0 = h * dh;
    for (int t = 0; t < n; ++t) {
      const float* q = qkv + (r0 + t) * ldq + c0;
      const float qa = lane < dh ? q[lane] : 0.0f;
      const float qb = lane + 32 < dh ? q[lane + 32] : 0.0f;
      // lane j scores keys j and j + 32
      float s0 = 0.0f, s1 = 0.0f;
      const float* k0 = kv + lane * ks + c0;
      const float* k1 = kv + (lane + 32) * ks + c0;
      for (int c = 0; c < dh; ++c) {
        const float qc = __shfl_sync(0xffffffffu, c < 32 ? qa : qb, c & 31);
        if (lane < n) s0 = fmaf(qc, k0[c], s0);
        if (lane + 32 < n) s1 = fmaf(qc, k1[c], s1);
      }
      s0 = lane < n ? s0 * scale : -INFINITY;
      s1 = lane + 32 < n ? s1 * scale : -INFINITY;
      float m = fmaxf(s0, s1);
#pragma unroll
      for (int w = 16; w > 0; w >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, w));
      const float p0 = lane < n ? expf(s0 - m) : 0.0f;
      const float p1 = lane + 32 < n ? expf(s1 - m) : 0.0f;
      float z = p0 + p1;
#pragma unroll
      for (int w = 16; w > 0; w >>= 1) z += __shfl_xor_sync(0xffffffffu, z, w);
      const float inv = 1.0f / z;
      float oa = 0.0f, ob = 0.0f;   // channels c0 + lane and c0 + lane + 32
      for (int j = 0; j < n; ++j) {
        const float pj = __shfl_sync(0xffffffffu, j < 32 ? p0 : p1, j & 31);
        const float* v = kv + j * ks + D + c0;
        if (lane < dh) oa = fmaf(pj, v[lane], oa);
        if (lane + 32 < dh) ob = fmaf(pj, v[lane + 32], ob);
      }
      OutT* orow = o + (r0 + t) * ldo + c0;
      if (lane < dh) put(orow + lane, oa * inv);
      if (lane + 32 < dh) put(orow + lane + 32, ob * inv);
    }
  }
}

}  // namespace tf_attn
