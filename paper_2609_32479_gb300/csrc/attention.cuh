// Multi-head self-attention within each track: the token mixing of the
// Transformer encoder in the paper's encoder comparison (App. A.3, Tab. A.1: full
// attention over a track's hits, no causal mask).  Per head h of width
// dh = D / NH, query hit t of track b attends to the track's n valid hits:
//   o_t = sum_j softmax_j(q_t . k_j / sqrt(dh)) v_j.
// q, k, v are the fp32 outputs of the qkv projection; scores, softmax and the
// weighted sum run in fp32.
//
// One CTA per track stages the track's keys and values in shared memory, each
// head's slice of a row padded by 4 floats so that the heads fall in different
// banks; thread i takes the (head, query) items i, i + 64, ... (head = item / n,
// query = item % n), keeps its query and its output (dh values each) in
// registers and reads every key and value of its head as a broadcast within the
// threads of that head.  With n hits a track keeps n x heads threads busy (52 at
// 13 hits and 4 heads, of 64).  The softmax takes two passes
// over the keys: the scores (kept in registers, up to KMAX = 32 or 64 keys) and
// their maximum, then the exponentials, their sum and the weighted values.
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <stdint.h>

namespace tf_attn {

__device__ __forceinline__ void put(float* p, float v) { *p = v; }
__device__ __forceinline__ void put(__half* p, float v) { *p = __float2half_rn(v); }
__device__ __forceinline__ void put(__nv_bfloat16* p, float v) { *p = __float2bfloat16_rn(v); }

// One head's output row o[0 .. DH) = acc * inv in 16-byte stores (DH is a
// multiple of 8; a row that does not start on a 16-byte boundary, which a
// workspace carved at an odd offset could give, is written value by value);
// each value is rounded as put() rounds it.
template <int DH>
__device__ __forceinline__ void put_row(float* o, const float (&acc)[DH], float inv) {
  if (reinterpret_cast<uintptr_t>(o) & 15u) {
#pragma unroll
    for (int i = 0; i < DH; ++i) put(o + i, acc[i] * inv);
    return;
  }
#pragma unroll
  for (int i = 0; i < DH; i += 4)
    *reinterpret_cast<float4*>(o + i) = make_float4(acc[i] * inv, acc[i + 1] * inv, acc[i + 2] * inv, acc[i + 3] * inv);
}
template <int DH>
__device__ __forceinline__ void put_row(__half* o, const float (&acc)[DH], float inv) {
  if (reinterpret_cast<uintptr_t>(o) & 15u) {
#pragma unroll
    for (int i = 0; i < DH; ++i) put(o + i, acc[i] * inv);
    return;
  }
#pragma unroll
  for (int i = 0; i < DH; i += 8) {
    uint4 w;
    __half2 h0 = __floats2half2_rn(acc[i] * inv, acc[i + 1] * inv), h1 = __floats2half2_rn(acc[i + 2] * inv, acc[i + 3] * inv);
    __half2 h2 = __floats2half2_rn(acc[i + 4] * inv, acc[i + 5] * inv), h3 = __floats2half2_rn(acc[i + 6] * inv, acc[i + 7] * inv);
    w.x = *reinterpret_cast<uint32_t*>(&h0);
    w.y = *reinterpret_cast<uint32_t*>(&h1);
    w.z = *reinterpret_cast<uint32_t*>(&h2);
    w.w = *reinterpret_cast<uint32_t*>(&h3);
    *reinterpret_cast<uint4*>(o + i) = w;
  }
}
template <int DH>
__device__ __forceinline__ void put_row(__nv_bfloat16* o, const float (&acc)[DH], float inv) {
  if (reinterpret_cast<uintptr_t>(o) & 15u) {
#pragma unroll
    for (int i = 0; i < DH; ++i) put(o + i, acc[i] * inv);
    return;
  }
#pragma unroll
  for (int i = 0; i < DH; i += 8) {
    uint4 w;
    __nv_bfloat162 h0 = __floats2bfloat162_rn(acc[i] * inv, acc[i + 1] * inv);
    __nv_bfloat162 h1 = __floats2bfloat162_rn(acc[i + 2] * inv, acc[i + 3] * inv);
    __nv_bfloat162 h2 = __floats2bfloat162_rn(acc[i + 4] * inv, acc[i + 5] * inv);
    __nv_bfloat162 h3 = __floats2bfloat162_rn(acc[i + 6] * inv, acc[i + 7] * inv);
    w.x = *reinterpret_cast<uint32_t*>(&h0);
    w.y = *reinterpret_cast<uint32_t*>(&h1);
    w.z = *reinterpret_cast<uint32_t*>(&h2);
    w.w = *reinterpret_cast<uint32_t*>(&h3);
    *reinterpret_cast<uint4*>(o + i) = w;
  }
}

constexpr int THREADS = 64;   // a track: heads x hits items (52 at 13 hits and 4 heads)

// Shared memory of one CTA: keys and values, T rows x NH heads x (dh + 4) floats each.
__host__ __device__ inline size_t smem_bytes(int T, int D, int NH) {
  return (size_t)2 * T * (D + 4 * NH) * sizeof(float);
}

// qkv: rows [q | k | v] of width 3 D at stride ldq; track b's hit t is row
// row0[b] + t (packed rows) or b T + t (padded rows, row0 null).  o: the attention
// output at stride ldo, row-aligned with qkv.  With padded rows the rows t >= n of
// a track (all of them for a track whose count is outside [1, T]) are written 0.
template <int DH, int KMAX, typename OutT>
__global__ void __launch_bounds__(THREADS) track_attention_kernel(const float* __restrict__ qkv, int ldq,
                                                                  const int64_t* __restrict__ row0,
                                                                  const int32_t* __restrict__ n_hits, int64_t B,
                                                                  int T, int D, int NH, OutT* __restrict__ o,
                                                                  int ldo) {
  extern __shared__ float4 sm4[];
  float* sm = reinterpret_cast<float*>(sm4);
  const int64_t b = blockIdx.x;
  if (b >= B) return;
  int n = n_hits[b];
  if (n < 1 || n > T) n = 0;
  const int64_t r0 = row0 ? row0[b] : b * (int64_t)T;
  const int hs = DH + 4, rs = NH * hs;   // padded head slice, row of one matrix
  float* ks = sm;
  float* vs = sm + (size_t)T * rs;
  const int w4 = (2 * D) / 4;            // float4s of k and v per row
  for (int i = threadIdx.x; i < n * w4; i += THREADS) {
    const int j = i / w4, c = 4 * (i - j * w4);
    const int m = c >= D, cc = c - m * D, h = cc / DH, e = cc - h * DH;
    *reinterpret_cast<float4*>((m ? vs : ks) + j * rs + h * hs + e) =
        *reinterpret_cast<const float4*>(qkv + (r0 + j) * ldq + D + c);
  }
  if (!row0) {   // padded layout: zero the padding rows
    for (int i = threadIdx.x; i < (T - n) * D; i += THREADS) {
      const int t = n + i / D, c = i % D;
      put(o + (r0 + t) * ldo + c, 0.0f);
    }
  }
  __syncthreads();
  const float scale = rsqrtf((float)DH);
  for (int it = threadIdx.x; it < NH * n; it += THREADS) {
    const int h = it / n, t = it - h * n;
    const float* qr = qkv + (r0 + t) * ldq + h * DH;
    float q[DH], acc[DH];
#pragma unroll
    for (int i = 0; i < DH; i += 4) {
      const float4 a = *reinterpret_cast<const float4*>(qr + i);
      q[i] = a.x;
      q[i + 1] = a.y;
      q[i + 2] = a.z;
      q[i + 3] = a.w;
      acc[i] = acc[i + 1] = acc[i + 2] = acc[i + 3] = 0.0f;
    }
    const float* kh = ks + h * hs;
    const float* vh = vs + h * hs;
    // the scores four keys at a time: four independent chains, each summed over
    // the head's dimensions in order (rows past the last key are read from the
    // last key's row and their scores dropped, so every read stays within the
    // track's keys)
    float sc[KMAX];
    float m = -INFINITY;
#pragma unroll
    for (int j0 = 0; j0 < KMAX; j0 += 4) {
      if (j0 >= n) break;
      const float* k0 = kh + j0 * rs;
      const float* k1 = kh + min(j0 + 1, n - 1) * rs;
      const float* k2 = kh + min(j0 + 2, n - 1) * rs;
      const float* k3 = kh + min(j0 + 3, n - 1) * rs;
      float s0 = 0.0f, s1 = 0.0f, s2 = 0.0f, s3 = 0.0f;
#pragma unroll
      for (int i = 0; i < DH; i += 4) {
        const float4 a0 = *reinterpret_cast<const float4*>(k0 + i);
        const float4 a1 = *reinterpret_cast<const float4*>(k1 + i);
        const float4 a2 = *reinterpret_cast<const float4*>(k2 + i);
        const float4 a3 = *reinterpret_cast<const float4*>(k3 + i);
        s0 = fmaf(q[i], a0.x, s0);
        s1 = fmaf(q[i], a1.x, s1);
        s2 = fmaf(q[i], a2.x, s2);
        s3 = fmaf(q[i], a3.x, s3);
        s0 = fmaf(q[i + 1], a0.y, s0);
        s1 = fmaf(q[i + 1], a1.y, s1);
        s2 = fmaf(q[i + 1], a2.y, s2);
        s3 = fmaf(q[i + 1], a3.y, s3);
        s0 = fmaf(q[i + 2], a0.z, s0);
        s1 = fmaf(q[i + 2], a1.z, s1);
        s2 = fmaf(q[i + 2], a2.z, s2);
        s3 = fmaf(q[i + 2], a3.z, s3);
        s0 = fmaf(q[i + 3], a0.w, s0);
        s1 = fmaf(q[i + 3], a1.w, s1);
        s2 = fmaf(q[i + 3], a2.w, s2);
        s3 = fmaf(q[i + 3], a3.w, s3);
      }
      sc[j0] = s0 * scale;
      m = fmaxf(m, sc[j0]);
      if (j0 + 1 < n) {
        sc[j0 + 1] = s1 * scale;
        m = fmaxf(m, sc[j0 + 1]);
      }
      if (j0 + 2 < n) {
        sc[j0 + 2] = s2 * scale;
        m = fmaxf(m, sc[j0 + 2]);
      }
      if (j0 + 3 < n) {
        sc[j0 + 3] = s3 * scale;
        m = fmaxf(m, sc[j0 + 3]);
      }
    }
    float l = 0.0f;
#pragma unroll
    for (int j = 0; j < KMAX; ++j) {
      if (j >= n) break;
      const float p = expf(sc[j] - m);
      l += p;
      const float* vr = vh + j * rs;
#pragma unroll
      for (int i = 0; i < DH; i += 4) {
        const float4 v = *reinterpret_cast<const float4*>(vr + i);
        acc[i] = fmaf(p, v.x, acc[i]);
        acc[i + 1] = fmaf(p, v.y, acc[i + 1]);
        acc[i + 2] = fmaf(p, v.z, acc[i + 2]);
        acc[i + 3] = fmaf(p, v.w, acc[i + 3]);
      }
    }
    const float inv = 1.0f / l;
    put_row<DH>(o + (r0 + t) * ldo + h * DH, acc, inv);
  }
}

// Launch for the head width D / NH (a multiple of 8 up to 64; anything else is
// rejected when the handle is created).
template <typename OutT>
inline cudaError_t launch(const float* qkv, int ldq, const int64_t* row0, const int32_t* n_hits, int64_t B, int T,
                          int D, int NH, OutT* o, int ldo, cudaStream_t st) {
  const size_t sm = smem_bytes(T, D, NH);
  const unsigned g = (unsigned)B;
#define TF_ATTN_CASE(DHV)                                                                                  \
  case DHV:                                                                                                \
    if (T <= 32)                                                                                           \
      track_attention_kernel<DHV, 32, OutT><<<g, THREADS, sm, st>>>(qkv, ldq, row0, n_hits, B, T, D, NH, o, ldo); \
    else                                                                                                   \
      track_attention_kernel<DHV, 64, OutT><<<g, THREADS, sm, st>>>(qkv, ldq, row0, n_hits, B, T, D, NH, o, ldo); \
    break;
  switch (D / NH) {
    TF_ATTN_CASE(8)
    TF_ATTN_CASE(16)
    TF_ATTN_CASE(24)
    TF_ATTN_CASE(32)
    TF_ATTN_CASE(40)
    TF_ATTN_CASE(48)
    TF_ATTN_CASE(56)
    TF_ATTN_CASE(64)
    default: return cudaErrorInvalidValue;
  }
#undef TF_ATTN_CASE
  return cudaPeekAtLastError();
}

// The dynamic shared memory of the launches above for tracks of T hits at width D.
template <typename OutT>
inline cudaError_t allow_smem(int T, int D, int NH) {
  const int sm = (int)smem_bytes(T, D, NH);
  if (sm <= 48 * 1024) return cudaSuccess;
#define TF_ATTN_ATTR(DHV)                                                                                    \
  case DHV:                                                                                                  \
    return T <= 32 ? cudaFuncSetAttribute(track_attention_kernel<DHV, 32, OutT>,                             \
                                          cudaFuncAttributeMaxDynamicSharedMemorySize, sm)                   \
                   : cudaFuncSetAttribute(track_attention_kernel<DHV, 64, OutT>,                             \
                                          cudaFuncAttributeMaxDynamicSharedMemorySize, sm);
  switch (D / NH) {
    TF_ATTN_ATTR(8)
    TF_ATTN_ATTR(16)
    TF_ATTN_ATTR(24)
    TF_ATTN_ATTR(32)
    TF_ATTN_ATTR(40)
    TF_ATTN_ATTR(48)
    TF_ATTN_ATTR(56)
    TF_ATTN_ATTR(64)
    default: return cudaErrorInvalidValue;
  }
#undef TF_ATTN_ATTR
}

}  // namespace tf_attn
