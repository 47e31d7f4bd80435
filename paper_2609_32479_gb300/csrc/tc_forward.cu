// tcgen05 path: one persistent, warp-specialised kernel runs the whole encoder
// forward (embedding, every minGRU layer, pooling) for the 16-bit-operand
// configs; head_kernel then applies the regression head to the pooled vectors.
//
// Orientation: every per-hit matrix product is computed transposed,
//   D[channel][hit] = W[channel][k] * Act[k][hit],
// with the weights as the M=128 operand (K-major, TMA-staged from L2/HBM with
// 128-byte swizzle) and the activations of one tile of 128 packed hits as the
// N=128 operand (MN-major, written by the epilogue warps straight into shared
// memory).  The fp32 accumulator lives in tensor memory with lane = channel and
// column = hit, so each epilogue thread owns one channel and walks the hits of
// its tracks in order: the gated scans of Eq. 2 run in registers without any
// cross-thread exchange.
//
// Tile: 128 hit columns = two 64-column slabs; each slab holds whole tracks
// (packed by best fit, unpadded).  Warp roles (608 threads):
//   warp 0       TMA producer of weight blocks (warp-wide loop, one elected lane issues)
//   warp 1       tcgen05.mma issuer (warp-wide loop, one elected lane issues), TMEM owner
//   warps 2..17  epilogue: TMEM lane quadrant = warp % 4, 32-column segment = (warp-2)/4
//   warp 18      loader: column metadata and Fourier operand of the next tile
// TMEM (512 columns): R0,R1 = merge accumulators, then x' with the MLP2 product
// accumulated onto it (d_model rows); R2,R3 = z and n of one scan chunk, then the
// output-gate projection, then MLP1 (and the embedding's first product).
// The fp32 residual stream of the tile lives in a per-CTA global scratch slab
// (L2-resident), never in HBM-sized intermediates.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cudaTypedefs.h>
#include <math.h>

#include <cstring>
#include <new>
#include <vector>

#include "sm100_ptx.cuh"
#include "trackfit_internal.h"

using namespace sm100;

namespace {

constexpr int NT = 608;                   // warp 0 TMA, warp 1 MMA issuer, warps 2..17 epilogue, warp 18 loader
constexpr int NE = 512;                   // epilogue threads
constexpr int SEGW = 32;                  // hit columns per epilogue thread (half a slab)
constexpr int TILE = 128;
constexpr int SLAB = 64;
constexpr int MAX_TRK_SLAB = 16;
constexpr int MAX_TRK_TILE = 2 * MAX_TRK_SLAB;
constexpr int A_BLOCK = 128 * 64 * 2;     // one 128-row x 64-k 16-bit weight block
constexpr int A_STAGE = 2 * A_BLOCK;      // a pipeline stage holds two consecutive blocks
constexpr int MAX_SCHED = 2048;           // schedule entries per tile
constexpr int EB_BYTES = 160 * 256;       // Fourier operand: 160 k-rows x 128 hits bf16
constexpr int MISC_BYTES = 10240;
constexpr int SCHED_BYTES = 2 * MAX_SCHED * 4;   // both schedule tables, copied to shared memory
constexpr int MAX_STAGES = 8;
constexpr int SEG = 1024;                 // tracks per packing segment
constexpr int64_t MAXB = 4194304;         // tracks per launch chunk
constexpr int64_t POOL_TRACKS = 1048576;  // tracks per launch chunk when the pooled means go to the internal buffer
constexpr uint64_t WAIT_NS = 2000000000ull;   // bounded-wait limit (a handle's test hook may lower it)
constexpr uint64_t DRAIN_NS = 200000000ull;
constexpr int B_SBO = 2048;               // k-group stride of the MN-major activation operand
constexpr int B_LBO = 1024;               // 64-hit atom stride

enum { MAP_E1 = 0, MAP_E2, MAP_IN, MAP_M, MAP_1, MAP_2, NMAPS };
enum { BSEL_XB = 0, BSEL_HB = 1 };
// Hand-overs around a schedule block: before its first MMA the issuer waits for
// the epilogue's next hand-over on e_bar (W_E; two barriers used alternately) or
// eh_bar (W_H); after its last MMA it commits to acc_bar (C_ACC; two barriers
// used alternately) or hb_bar (C_HB).
enum { W_NONE = 0, W_E = 1, W_H = 2 };
enum { C_NONE = 0, C_ACC = 1, C_HB = 2 };
// bits of an MMA schedule entry
constexpr uint32_t S_NK4 = 1u << 16, S_ACC = 1u << 17, S_C_ACC = 1u << 18, S_C_HB = 1u << 19, S_W_E = 1u << 20,
                   S_W_H = 1u << 21;
enum { F_FIRST = 1, F_LAST = 2, F_VALID = 4 };

struct TcParams {
  CUtensorMap tm[NMAPS];
  const float* hits;
  const int64_t* offs;   // packed input: track b's hits are rows offs[b] .. of hits (null: padded [B][T][5])
  const int32_t* n_hits;
  float* out;
  float* out_q;
  float* pool;   // [B][D] pooled means (the caller's buffer or an internal one)
  float* xs;
  const int32_t* slab_start;   // slab s = tracks order[slab_start[s] .. slab_start[s + 1])
  const int32_t* order;        // tracks in packing order
  const int32_t* n_slabs;
  const uint32_t* sched_p;   // per block: map | col/64 << 4 | row << 8
  const uint32_t* sched_m;   // per block: b offset | bsel << 13 | tcol/128 << 14 | S_* flags
  int n_sched;
  const float* b_e1;
  const float* b_e2;
  const float* g;
  const float* b_in;
  const float* b_m;
  const float* b_1;
  const float* b_2;
  unsigned long long* err;
  uint64_t wait_ns;     // limit of every bounded wait
  int hold_tile;        // test hook: CTA 0's loader holds this tile's metadata hand-over (-1: none)
  int T, D, H, L, NDC, ROWS_IN, NQ, Q, nst;
  uint32_t idesc;
  int off_xb, off_hb, off_a, off_misc;
  int fp16;
  float rms_eps;
  float feat_min[5], feat_inv_hi[5], feat_inv_lo[5], scale[16];
  int scale_doubling;   // scale[k + 3] == 2 scale[k] for every k: Fourier by angle doubling
  uint8_t* fbuf;        // per CTA two Fourier operands (HB byte images) written by the loader warp
};

// Column metadata of one tile, written by the loader warp one tile ahead (two
// buffers, alternating by tile).
struct TileMeta {
  int slot_track[MAX_TRK_TILE], slot_n[MAX_TRK_TILE];
  uint8_t col_flags[TILE], col_slot[TILE];
  // per column half h, 32-column word w: bit j = column 64h + 32w + j starts a
  // track (first), ends one (last), holds a hit (valid)
  uint32_t m_first[2][2], m_last[2][2], m_valid[2][2];
};
struct Misc {
  uint64_t full[MAX_STAGES], empty[MAX_STAGES];
  uint64_t acc_bar[2], e_bar[2], hb_bar, eh_bar, drain_bar;
  uint64_t meta_full[2], meta_free[2];   // loader -> epilogue, epilogue -> loader
  uint32_t tmem_base;
  int abort_flag;
  TileMeta meta[2];
  uint8_t col_tpos[TILE];   // the loader's own
  alignas(16) float part[4][TILE];
  float carry[2][128];   // [slab][channel]: scan states between a slab's column segments
  alignas(16) float rinv[NE / 32][32];   // per epilogue warp: 1 / RMS of its 32 columns
  float hs[TILE][5];   // the loader's own
};
static_assert(sizeof(Misc) <= MISC_BYTES, "misc region too small");

__device__ __forceinline__ float sigm(float x) { return __fdividef(1.0f, 1.0f + __expf(-x)); }
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ float rcp_approx(float x) {
  float y;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
constexpr float LOG2E_F = 1.4426950408889634f;
__device__ __forceinline__ float silu(float x) { return x * sigm(x); }
// The MLP's SiLU inside the fused kernel uses one MUFU operation per value
// instead of two (ex2 and rcp), from SiLU(x) = (x / 2)(1 + tanh(x / 2)):
// tanh.approx has a relative error of about 2^-11, and the result is rounded
// to a 16-bit operand right away (measured: no change in the error against the
// oracle).  The output gate does not: its value scales the merge into the fp32
// residual stream, where that error showed up on every track, so it takes the
// two-operation sigmoid, as do the scan gates (a = 1 - sigma there also needs
// relative accuracy as sigma -> 1).  (A reciprocal by Newton steps on the FMA
// pipe instead of rcp was measured slower: these epilogues are bound by issued
// instructions more than by the MUFU unit.)  sigm_pre takes its argument
// already scaled by -log2 e, with the bias folded in by one FMA.
__device__ __forceinline__ float sigm_pre(float t) { return rcp_approx(1.0f + ex2_approx(t)); }
__device__ __forceinline__ float tanh_approx(float x) {
  float y;
  asm("tanh.approx.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
// SiLU(v + b) in that form, with hb = b / 2: the half argument (v + b) / 2 comes
// from one FMA, bit for bit the value of halving the rounded sum (halving is exact)
__device__ __forceinline__ float silu_tb(float v, float hb) {
  const float h = fmaf(v, 0.5f, hb);
  return fmaf(h, tanh_approx(h), h);
}

// Operand conversion (round to nearest even): bf16, or fp16 when FP16 is set.
template <bool FP16>
__device__ __forceinline__ uint32_t pack2(float a, float b) {   // a -> low half (lower column)
  if constexpr (FP16) {
    __half2 v = __floats2half2_rn(a, b);
    return *reinterpret_cast<uint32_t*>(&v);
  } else {
    __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
    return *reinterpret_cast<uint32_t*>(&v);
  }
}

// Byte offset, inside an MN-major 128-byte-swizzled operand with 128 columns, of
// the 16-byte chunk that holds columns [8*n8, 8*n8+8) of k-row k.  Atoms are 8
// k-rows x 64 columns (1 KB); the two column atoms of a k-group are adjacent.
__device__ __forceinline__ uint32_t bchunk(int k, int n8) {
  return (uint32_t)((k >> 3) * B_SBO + (n8 >> 3) * B_LBO + (k & 7) * 128 + (((n8 & 7) ^ (k & 7)) << 4));
}

__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
  asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(a), "r"(b), "r"(c), "r"(d) : "memory");
}

// Write 32 consecutive columns [n0, n0+32) of k-row k (n0 % 32 == 0) as 16-bit operands.
template <bool FP16>
__device__ __forceinline__ void store_row32(uint32_t buf, int k, int n0, const float (&v)[32]) {
#pragma unroll
  for (int c = 0; c < 4; ++c) {
    st_shared_v4(buf + bchunk(k, (n0 >> 3) + c), pack2<FP16>(v[8 * c + 0], v[8 * c + 1]),
                 pack2<FP16>(v[8 * c + 2], v[8 * c + 3]), pack2<FP16>(v[8 * c + 4], v[8 * c + 5]),
                 pack2<FP16>(v[8 * c + 6], v[8 * c + 7]));
  }
}

template <bool FP16>
__device__ __forceinline__ void store_row16(uint32_t buf, int k, int n0, const float (&v)[16]) {
#pragma unroll
  for (int c = 0; c < 2; ++c) {
    st_shared_v4(buf + bchunk(k, (n0 >> 3) + c), pack2<FP16>(v[8 * c + 0], v[8 * c + 1]),
                 pack2<FP16>(v[8 * c + 2], v[8 * c + 3]), pack2<FP16>(v[8 * c + 4], v[8 * c + 5]),
                 pack2<FP16>(v[8 * c + 6], v[8 * c + 7]));
  }
}

// The four epilogue warps of one 32-column segment (one per TMEM quadrant):
// barrier 10 + seg, 128 threads.
__device__ __forceinline__ void seg_sync(int seg) { asm volatile("bar.sync %0, 128;" ::"r"(10 + seg) : "memory"); }

// The static sequence of 128x64 weight blocks of one tile, in the order the MMA
// issuer consumes them.  f(map, row, col, nk, tmem_col, bsel, bk, acc, wait, commit):
// nk MMAs of K=16 read the block, accumulate into TMEM columns tmem_col, with
// the activation operand bsel starting at k-row bk; acc = accumulate onto the
// existing accumulator; wait / commit = hand-overs (W_*, C_*).
//
// Within a layer the scan chunks are software-pipelined: as soon as the
// epilogue has copied the z/n accumulators of chunk k into registers, the
// issuer computes z/n of chunk k+1 into the same TMEM columns, and the merge
// product of chunk k follows once its states h(k) are in shared memory.
template <class F>
__host__ __device__ inline void walk_tile(const TcParams& p, F&& f) {
  const int MT = p.D >> 7, KD = p.D >> 6;
  // the embedding's first product goes to the z/n columns, so it can run while
  // the epilogue still pools the previous tile from columns 0..
  for (int mt = 0; mt < MT; ++mt)
    for (int kc = 0; kc < 3; ++kc)
      f(MAP_E1, mt * 128, kc * 64, kc == 2 ? 2 : 4, 256 + mt * 128, BSEL_HB, kc * 64, kc > 0,
        (mt == 0 && kc == 0) ? W_E : W_NONE, (mt == MT - 1 && kc == 2) ? C_ACC : C_NONE);
  // a dense D x D product from XB into accumulator columns tcol0 + 128 mt; with
  // onto = true it accumulates onto what the columns hold (MLP2 onto x')
  auto dense = [&](int map, int r0, int tcol0, bool onto) {
    for (int mt = 0; mt < MT; ++mt)
      for (int kc = 0; kc < KD; ++kc)
        f(map, r0 + mt * 128, kc * 64, 4, tcol0 + mt * 128, BSEL_XB, kc * 64, onto || kc > 0,
          (mt == 0 && kc == 0) ? W_E : W_NONE, (mt == MT - 1 && kc == KD - 1) ? C_ACC : C_NONE);
  };
  if (MT == 1) {
    dense(MAP_E2, 0, 0, false);
  } else {   // committed per 128-channel tile, like MLP2
    for (int mt = 0; mt < 2; ++mt)
      for (int kc = 0; kc < KD; ++kc)
        f(MAP_E2, mt * 128, kc * 64, 4, mt * 128, BSEL_XB, kc * 64, kc > 0, (mt == 0 && kc == 0) ? W_E : W_NONE,
          kc == KD - 1 ? C_ACC : C_NONE);
  }
  for (int l = 0; l < p.L; ++l) {
    const int rb = l * p.ROWS_IN;
    auto zn = [&](int k) {   // z and n of scan chunk k -> TMEM columns 256.. and 384..
      for (int kc = 0; kc < KD; ++kc)
        f(MAP_IN, rb + k * 256, kc * 64, 4, 256, BSEL_XB, kc * 64, kc > 0, kc == 0 ? W_E : W_NONE, C_NONE);
      for (int kc = 0; kc < KD; ++kc)
        f(MAP_IN, rb + k * 256 + 128, kc * 64, 4, 384, BSEL_XB, kc * 64, kc > 0, W_NONE,
          kc == KD - 1 ? C_ACC : C_NONE);
    };
    if (MT == 1) {
      zn(0);
    } else {   // x_hat arrives one 128-channel tile at a time (K rows 0-127, then 128-255)
      for (int kh = 0; kh < 2; ++kh) {
        for (int kc = 2 * kh; kc < 2 * kh + 2; ++kc)
          f(MAP_IN, rb, kc * 64, 4, 256, BSEL_XB, kc * 64, kc > 0, kc == 2 * kh ? W_E : W_NONE, C_NONE);
        for (int kc = 2 * kh; kc < 2 * kh + 2; ++kc)
          f(MAP_IN, rb + 128, kc * 64, 4, 384, BSEL_XB, kc * 64, kc > 0, W_NONE,
            kc == KD - 1 ? C_ACC : C_NONE);
      }
    }
    for (int k = 0; k < p.NDC; ++k) {
      if (k + 1 < p.NDC) {
        zn(k + 1);
      } else {   // output-gate projection into the z/n columns once the last chunk is out
        for (int mt = 0; mt < MT; ++mt)
          for (int kc = 0; kc < KD; ++kc)
            f(MAP_IN, rb + p.NDC * 256 + mt * 128, kc * 64, 4, 256 + mt * 128, BSEL_XB, kc * 64, kc > 0,
              (mt == 0 && kc == 0) ? W_E : W_NONE, C_NONE);
      }
      // merge of chunk k: M[D] += W_m[:, chunk] * h(k).  The last one completes
      // the gate epilogue's inputs one 128-channel tile at a time.
      const bool last = k + 1 == p.NDC;
      for (int mt = 0; mt < MT; ++mt)
        for (int kc = 0; kc < 2; ++kc)
          f(MAP_M, l * p.D + mt * 128, k * 128 + kc * 64, 4, mt * 128, BSEL_HB, kc * 64, k > 0 || kc > 0,
            (mt == 0 && kc == 0) ? W_H : W_NONE,
            kc == 1 && (last || mt == MT - 1) ? (last ? C_ACC : C_HB) : C_NONE);
    }
    if (MT == 1) {
      dense(MAP_1, l * p.D, 256, false);   // MLP1 -> the z/n columns
      dense(MAP_2, l * p.D, 0, true);      // MLP2 accumulates onto x'
    } else {
      // d_model 256, pipelined by 128-channel tile: MLP1's first K half (x' of
      // tile 0, XB rows 0-127) starts once the gate epilogue of tile 0 is out,
      // the rest once tile 1 is; MLP2's K rows 0-127 (SiLU of tile 0) come from
      // HB, rows 128-255 (SiLU of tile 1) from XB.
      const int r1 = l * p.D;
      // MLP1 goes to the z/n columns (free once the gate epilogue of the tile has
      // read them); MLP2 accumulates onto x', which the gate epilogue left in the
      // merge columns
      for (int kc = 0; kc < 4; ++kc)
        f(MAP_1, r1, kc * 64, 4, 256, BSEL_XB, kc * 64, kc > 0, (kc & 1) ? W_NONE : W_E, kc == 3 ? C_ACC : C_NONE);
      for (int kc = 0; kc < 4; ++kc)
        f(MAP_1, r1 + 128, kc * 64, 4, 384, BSEL_XB, kc * 64, kc > 0, W_NONE, kc == 3 ? C_ACC : C_NONE);
      // MLP2: K rows 0-127 (HB) of both output tiles once the SiLU of tile 0 is
      // in, then rows 128-255 (XB), tile 0 first (the residual starts on it)
      for (int kh = 0; kh < 2; ++kh)
        for (int mt = 0; mt < 2; ++mt)
          for (int kc = 2 * kh; kc < 2 * kh + 2; ++kc)
            f(MAP_2, r1 + mt * 128, kc * 64, 4, mt * 128, kh == 0 ? BSEL_HB : BSEL_XB, kc * 64, true,
              (mt == 0 && kc == 2 * kh) ? W_E : W_NONE, kc == 3 ? C_ACC : C_NONE);
    }
  }
}

__device__ __forceinline__ void set_abort(Misc* m, unsigned long long* err) {
  if (atomicExch(&m->abort_flag, 1) == 0) atomicAdd(err + 1, 1ull);
}

// ------------------------------------------------------------------ epilogue
struct ECtx {
  const TcParams* p;
  Misc* m;
  const TileMeta* md;   // metadata of the tile being processed
  uint32_t xb, hb, tq;
  float* xs;
  // quadrant q (TMEM lanes / channels 32q..), column segment seg = 32-column
  // quarter of the tile (slab half = seg / 2, position in the slab sub = seg % 2)
  int q, lane, seg, half, sub, c, col0, te, e, MT;
};

// The two epilogue warps that share a quadrant and a slab hand a recurrence state
// from the slab's first 32 columns to the second, or back in the reverse
// direction: barrier 2 + 2q + half, 64 threads, both warps synchronising once
// per hand-over.  (The leading warp must not merely arrive: a warp that could
// arrive twice before its partner synchronises would complete a barrier
// instance on its own and leave the partner's last one unmatched.  In normal
// operation the state-buffer wait keeps the leader within one hand-over, but
// after an expired wait every wait fails fast and that bound is gone; with a
// synchronisation on both sides the two warps pair up whatever the waits do.
// The partner reaches its side before its own scan, so the leader, which
// scans first, seldom waits.)
__device__ __forceinline__ void carry_pass(const ECtx& x) {
  asm volatile("bar.sync %0, 64;" ::"r"(2 + 2 * x.q + x.half) : "memory");
}
__device__ __forceinline__ void carry_wait(const ECtx& x) {
  asm volatile("bar.sync %0, 64;" ::"r"(2 + 2 * x.q + x.half) : "memory");
}

// silu(acc + b) of the 128-channel tile mt -> k-rows row0 + c of buf (b: the
// thread's channel's bias, loaded before the wait for the product)
template <bool FP16>
__device__ __forceinline__ void ep_silu_mt(const ECtx& x, float b, int mt, uint32_t tcol, uint32_t buf, int row0) {
  float v[32];
  tmem_ld32(x.tq + tcol + mt * 128 + x.col0, v);
  tmem_ld_wait();
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = silu_tb(v[i], 0.5f * b);
  store_row32<FP16>(buf, row0 + x.c, x.col0, v);
}
// silu(acc + bias) of the embedding's first product (accumulator columns
// 256 + mt*128) -> XB rows [mt*128 + c], all tiles read under one TMEM wait;
// the biases are loaded before the wait for the product (wait_first)
template <bool FP16, int MT, class W>
__device__ __forceinline__ void ep_silu_t(const ECtx& x, const float* bias, W&& wait_first) {
  float bv[MT];
#pragma unroll
  for (int mt = 0; mt < MT; ++mt) bv[mt] = bias[mt * 128 + x.c];
  wait_first();
  float v[MT][32];
#pragma unroll
  for (int mt = 0; mt < MT; ++mt) tmem_ld32(x.tq + 256 + mt * 128 + x.col0, v[mt]);
  tmem_ld_wait();
#pragma unroll
  for (int mt = 0; mt < MT; ++mt) {
    const float b = bv[mt];
#pragma unroll
    for (int i = 0; i < 32; ++i) v[mt][i] = silu(v[mt][i] + b);
    store_row32<FP16>(x.xb, mt * 128 + x.c, x.col0, v[mt]);
  }
}
template <bool FP16, class W>
__device__ __forceinline__ void ep_silu(const ECtx& x, const float* bias, W&& wait_first) {
  if (x.MT == 2)
    ep_silu_t<FP16, 2>(x, bias, wait_first);
  else
    ep_silu_t<FP16, 1>(x, bias, wait_first);
}

// X = acc + bias (a layer's accumulator already holds x' plus the MLP2 product).
// X goes to the per-CTA scratch (read back once, by the next layer's gate
// epilogue) and the RMS-normalised x_hat to XB (recomputing X from TMEM); the
// last layer's X is mean-pooled instead (ep_pool).
// Sum of v over the 32 lanes for 16 columns at once: afterwards lane L holds the
// total of column L & 15 (both halves of the warp hold the same 16 totals).
__device__ __forceinline__ float reduce_scatter16(float (&v)[16], int lane) {
#pragma unroll
  for (int off = 8; off >= 1; off >>= 1) {
    const bool upper = (lane & off) != 0;
#pragma unroll
    for (int i = 0; i < off; ++i) {
      const float send = upper ? v[i] : v[i + off];
      const float keep = upper ? v[i + off] : v[i];
      v[i] = keep + __shfl_xor_sync(0xffffffffu, send, off);
    }
  }
  return v[0] + __shfl_xor_sync(0xffffffffu, v[0], 16);
}

template <bool FP16, int MT, class W, class S>
__device__ __forceinline__ void ep_residual_t(const ECtx& x, const float* bias, const float* gain, W&& wait_tile,
                                              S&& signal_tile) {
  // bias and gain of the thread's channels, loaded before the wait for the
  // first tile's product so that their latency hides behind it
  const TcParams& p = *x.p;
  constexpr int D = 128 * MT;   // d_model
  const uint32_t vm = x.md->m_valid[x.half][x.sub];   // bit i: column col0 + i holds a hit
  // X = acc + bias (the accumulator already holds x' + MLP for a layer, the
  // embedding product for the embedding).  Pad columns are not cleared in X:
  // their x_hat is 0 (their inverse RMS is set to 0), so every product gives
  // them its bias, and their values stay finite and in their own columns (the
  // products and norms are per column, the scans restart at each track's ends,
  // pooling skips them).  The products complete one 128-channel tile at a time,
  // each waited for in turn (wait_tile): tile 0 is summed while tile 1 is still
  // being computed, and x_hat is handed over per tile (signal_tile) so the next
  // products can start on its K rows.  Only the sums of squares stand between
  // the last product and the first hand-over: X goes to the scratch after both
  // hand-overs (each thread later reads back only its own values, and the
  // accumulator columns still hold X until the next layer's first merge, which
  // waits for this thread's scan hand-over).
  float bias_v[MT], gain_v[MT];
#pragma unroll
  for (int mt = 0; mt < MT; ++mt) {
    bias_v[mt] = bias[mt * 128 + x.c];
    gain_v[mt] = gain[mt * 128 + x.c];
  }
  float sq[32];
#pragma unroll
  for (int i = 0; i < 32; ++i) sq[i] = 0.0f;
#pragma unroll
  for (int mt = 0; mt < MT; ++mt) {
    wait_tile();
#pragma unroll
    for (int hh = 0; hh < 2; ++hh) {
      float v[16];
      tmem_ld16(x.tq + mt * 128 + x.col0 + 16 * hh, v);
      tmem_ld_wait();
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        const float val = v[i] + bias_v[mt];
        sq[16 * hh + i] = fmaf(val, val, sq[16 * hh + i]);
      }
    }
  }
#pragma unroll
  for (int hh = 0; hh < 2; ++hh) {
    float h16[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) h16[i] = sq[16 * hh + i];
    const float t = reduce_scatter16(h16, x.lane);
    if (x.lane < 16) x.m->part[x.q][x.col0 + 16 * hh + x.lane] = t;
  }
  // the column sums over all channels: the four quadrants' partial sums of this
  // segment's columns; every warp then forms the 32 inverse RMS values itself
  // (the same sum in the same order, so the four copies are identical) in a
  // slice of its own
  seg_sync(x.seg);
  float* rw = x.m->rinv[x.e];
  {
    const int c = x.col0 + x.lane;
    const float t = x.m->part[0][c] + x.m->part[1][c] + x.m->part[2][c] + x.m->part[3][c];
    rw[x.lane] = ((vm >> x.lane) & 1u) ? 1.0f / sqrtf(t / (float)D + p.rms_eps) : 0.0f;
  }
  __syncwarp();
#pragma unroll
  for (int mt = 0; mt < MT; ++mt) {
    const float g = gain_v[mt];
#pragma unroll
    for (int hh = 0; hh < 2; ++hh) {
      const int c0 = x.col0 + 16 * hh;
      float v[16], rv[16];
      tmem_ld16(x.tq + mt * 128 + c0, v);
      const float4* rp = reinterpret_cast<const float4*>(rw + 16 * hh);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float4 r4 = rp[i];
        rv[4 * i] = r4.x;
        rv[4 * i + 1] = r4.y;
        rv[4 * i + 2] = r4.z;
        rv[4 * i + 3] = r4.w;
      }
      tmem_ld_wait();
#pragma unroll
      for (int i = 0; i < 16; ++i) v[i] = (v[i] + bias_v[mt]) * g * rv[i];
      store_row16<FP16>(x.xb, mt * 128 + x.c, c0, v);
    }
    signal_tile();   // x_hat of this tile is in XB
  }
  // the residual stream to the scratch (a warp's store: one 128-byte line)
#pragma unroll
  for (int mt = 0; mt < MT; ++mt) {
#pragma unroll
    for (int hh = 0; hh < 2; ++hh) {
      const int c0 = x.col0 + 16 * hh;
      float v[16];
      tmem_ld16(x.tq + mt * 128 + c0, v);
      tmem_ld_wait();
      float* xp = x.xs + (size_t)c0 * D + mt * 128 + x.c;
#pragma unroll
      for (int i = 0; i < 16; ++i) xp[(size_t)i * D] = v[i] + bias_v[mt];
    }
  }
}

template <bool FP16, class W, class S>
__device__ __forceinline__ void ep_residual(const ECtx& x, const float* bias, const float* gain, W&& wait_tile,
                                            S&& signal_tile) {
  if (x.MT == 2)
    ep_residual_t<FP16, 2>(x, bias, gain, wait_tile, signal_tile);
  else
    ep_residual_t<FP16, 1>(x, bias, gain, wait_tile, signal_tile);
}

// Masked mean pooling of the last layer's output X = acc + bias.  The warp of
// quadrant q, slab half and segment sub pools channel tile mt = sub (channels
// 128 mt + 32 q + lane) over all 64 columns of the slab, each track's hits summed
// in order from its first; with d_model 128 the sub = 1 warps have no tile.
// The column loops stay rolled: this runs once per tile, and its code is cold.
__device__ __forceinline__ void ep_pool(const ECtx& x, const float* bias) {
  const TcParams& p = *x.p;
  const int mt = x.sub;
  if (mt >= x.MT) return;
  // after an expired wait the tile's metadata may not have been handed over:
  // no stores indexed by it
  if (*reinterpret_cast<volatile int*>(&x.m->abort_flag)) return;
  const int D = p.D, ch = mt * 128 + x.c;
  const float bv = bias[ch];
  const uint8_t* flags = x.md->col_flags;
  float run = 0.0f;
#pragma unroll 1
  for (int k = 0; k < 4; ++k) {   // 16-column groups of the slab
    const int c0 = SLAB * x.half + 16 * k;
    const uint32_t vm = x.md->m_valid[x.half][k >> 1] >> (16 * (k & 1));
    float v[16];
    tmem_ld16(x.tq + mt * 128 + c0, v);
    tmem_ld_wait();
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const float val = ((vm >> i) & 1u) ? v[i] + bv : 0.0f;
      const int fl = flags[c0 + i];
      run = (fl & F_FIRST) ? val : run + val;
      if (fl & F_LAST) {
        const int s = x.md->col_slot[c0 + i];
        p.pool[(size_t)x.md->slot_track[s] * D + ch] = run / (float)x.md->slot_n[s];
      }
    }
  }
}

// X of the thread's channel in tile mt and its 32 columns, read back from the
// scratch; issued before the wait for the gate's inputs so the loads' latency
// hides behind it.
__device__ __forceinline__ void gate_x_load(const ECtx& x, int mt, float (&xv)[32]) {
  const int D = x.p->D;
  const float* xp = x.xs + (size_t)x.col0 * D + mt * 128 + x.c;
#pragma unroll
  for (int i = 0; i < 32; ++i) xv[i] = xp[(size_t)i * D];
}
// x' = X + (M + b_m) * sigma(p_g + b_g) for the 128-channel tile mt -> TMEM columns
// 128 mt.. (in place of the merge accumulator; MLP2 accumulates onto it) and XB
// rows 128 mt + c.
template <bool FP16>
__device__ __forceinline__ void ep_gate(const ECtx& x, int mt, const float (&xv)[32], float bm, float bg) {
  const int ch_g = mt * 128 + x.c;
  const float cg = -bg * LOG2E_F;
#pragma unroll
  for (int hh = 0; hh < 2; ++hh) {
    const int c0 = x.col0 + 16 * hh;
    float mv[16], gv[16];
    tmem_ld16(x.tq + mt * 128 + c0, mv);
    tmem_ld16(x.tq + 256 + mt * 128 + c0, gv);
    tmem_ld_wait();
#pragma unroll
    for (int i = 0; i < 16; ++i) mv[i] = fmaf(mv[i] + bm, sigm_pre(fmaf(gv[i], -LOG2E_F, cg)), xv[16 * hh + i]);
    tmem_st16(x.tq + mt * 128 + c0, mv);   // x' where MLP2 will accumulate
    store_row16<FP16>(x.xb, ch_g, c0, mv);
  }
  tmem_st_wait();
}

// Scan chunk of one layer.  The chunk holds 64 channels of both directions:
// TMEM lanes 0-63 (quadrants 0, 1) run the forward recurrence over the hits in
// time order, lanes 64-127 (quadrants 2, 3) the reverse one.  Each thread owns a
// 32-column segment; the two segments of a slab run one after the other, the
// leading one handing its final state to the other (carry_pass / carry_wait).  The
// z/n accumulators are first copied to registers (scan_load) so the issuer can
// reuse their TMEM columns for the next chunk while the gates and the recurrence
// run; the states then go to HB.
__device__ __forceinline__ void scan_load(const ECtx& x, float (&z)[32], float (&n)[32]) {
  tmem_ld32(x.tq + 256 + x.col0, z);
  tmem_ld32(x.tq + 384 + x.col0, n);
  tmem_ld_wait();
}
// The gates, independent across hits, in the form h_t = a_t h_{t-1} + b_t of the
// linear scan: with s = sigma(z + b_z) = 1 / (1 + e), e = 2^(-(z + b_z) log2 e),
// a = 1 - s = e s (no cancellation as s -> 1) and b = s (n + b_n).  Where the
// recurrence restarts (a track's first hit forward, its last in reverse) a = 0.
// a replaces z, b replaces n.
__device__ __forceinline__ void scan_gates(const ECtx& x, float (&z)[32], float (&n)[32], float bz, float bn) {
  const uint32_t rm = x.q < 2 ? x.md->m_first[x.half][x.sub] : x.md->m_last[x.half][x.sub];
  const float cz = -bz * LOG2E_F;
#pragma unroll
  for (int j = 0; j < 32; ++j) {
    const float e = ex2_approx(fmaf(z[j], -LOG2E_F, cz));
    const float sg = rcp_approx(1.0f + e);
    z[j] = (rm & (1u << j)) ? 0.0f : e * sg;
    n[j] = sg * (n[j] + bn);
  }
}
// Eq. 2 per channel over this thread's 32 columns (one FMA per hit on the serial
// path), the states replacing z.  Tracks fill a slab from its first column, so
// padding only trails the last track: the forward state is never read after it,
// and in reverse the last track's end restarts the state (a = 0 there: the
// finite state coming from the padding is multiplied away).  Values left in
// padding columns stay in padding columns (every product and norm is per
// column) and stay finite (their x_hat is 0), so they need no clearing here.
template <bool FP16>
__device__ __forceinline__ void scan_chain_store(const ECtx& x, float (&a)[32], const float (&b)[32]) {
  const bool fwd = x.q < 2;
  const bool leads = fwd ? x.sub == 0 : x.sub == 1;
  float h = 0.0f;
  if (!leads) {
    carry_wait(x);
    h = x.m->carry[x.half][x.c];
  }
  if (fwd) {
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      h = fmaf(a[j], h, b[j]);
      a[j] = h;
    }
  } else {
#pragma unroll
    for (int j = 31; j >= 0; --j) {
      h = fmaf(a[j], h, b[j]);
      a[j] = h;
    }
  }
  if (leads) {
    x.m->carry[x.half][x.c] = h;
    carry_pass(x);
  }
  store_row32<FP16>(x.hb, x.c, x.col0, a);
}

// Tile set-up, run one tile ahead by the loader warp while the epilogue warps
// work on the current tile: the column metadata of the tile's two slabs (into
// the metadata buffer md), the features of its hits, and the Fourier operand
// (the B operand of the embedding's first product) as the byte image of HB in
// the CTA's global buffer fb, from which the epilogue copies it at tile start.
template <bool FP16>
__device__ __forceinline__ void load_tile(const TcParams& p, Misc* m, TileMeta* md, uint8_t* fb, int tile,
                                          int n_slabs, int lane) {
  for (int c = lane; c < TILE; c += 32) md->col_flags[c] = 0;
  __syncwarp();
  int ns = 0;
  for (int hf = 0; hf < 2; ++hf) {
    const int s = 2 * tile + hf;
    if (s >= n_slabs) break;
    const int b0 = p.slab_start[s];
    const int cnt = p.slab_start[s + 1] - b0;
    int n = 0, trk = 0;
    if (lane < cnt) {
      trk = p.order[b0 + lane];
      n = p.n_hits[trk];
      if (n < 1 || n > p.T) n = 0;   // rejected by the packer's validity check: no columns
    }
    int incl = n;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += y;
    }
    if (lane < cnt) {
      const int slot = ns + lane;
      const int c0 = SLAB * hf + incl - n;
      md->slot_track[slot] = trk;
      md->slot_n[slot] = n;
      for (int t = 0; t < n; ++t) {
        const int col = c0 + t;
        md->col_flags[col] = (uint8_t)(F_VALID | (t == 0 ? F_FIRST : 0) | (t == n - 1 ? F_LAST : 0));
        md->col_slot[col] = (uint8_t)slot;
        m->col_tpos[col] = (uint8_t)t;
      }
    }
    ns += cnt;
  }
  __syncwarp();
  if (lane < 4) {   // column bitmasks
    const int hf = lane >> 1, w = lane & 1;
    uint32_t fm = 0, lm = 0, vm = 0;
    for (int j = 0; j < 32; ++j) {
      const int f = md->col_flags[SLAB * hf + 32 * w + j];
      fm |= (uint32_t)((f & F_FIRST) != 0) << j;
      lm |= (uint32_t)((f & F_LAST) != 0) << j;
      vm |= (uint32_t)((f & F_VALID) != 0) << j;
    }
    md->m_first[hf][w] = fm;
    md->m_last[hf][w] = lm;
    md->m_valid[hf][w] = vm;
  }
  for (int idx = lane; idx < TILE * 5; idx += 32) {
    const int col = idx / 5, f = idx - col * 5;
    float v = 0.0f;
    if (md->col_flags[col] & F_VALID) {
      const size_t trk = (size_t)md->slot_track[md->col_slot[col]];
      const size_t row = p.offs ? (size_t)p.offs[trk] + m->col_tpos[col] : trk * p.T + m->col_tpos[col];
      v = p.hits[row * 5 + f];
    }
    m->hs[col][f] = v;
  }
  __syncwarp();
  // u = (v - min) / (max - min) and the argument s_k * u as unevaluated sums of
  // two floats (error-free TwoSum / TwoProduct with fma), reduced modulo 2
  // exactly, so sin(pi s_k u) carries only the final fp32 rounding.
  auto arg = [&](int col, int f, float sk) -> float {
    const float v = m->hs[col][f], mn = -p.feat_min[f];
    const float dh = v + mn;
    const float bv = dh - v;
    const float dl = (v - (dh - bv)) + (mn - bv);
    const float uh = dh * p.feat_inv_hi[f];
    const float ul = fmaf(dh, p.feat_inv_hi[f], -uh) + fmaf(dh, p.feat_inv_lo[f], dl * p.feat_inv_hi[f]);
    const float xh = uh * sk;
    const float xl = fmaf(uh, sk, -xh) + ul * sk;
    return (xh - 2.0f * rintf(0.5f * xh)) + xl;
  };
  auto put = [&](int row, int g, const float (&v)[8]) {
    *reinterpret_cast<uint4*>(fb + bchunk(row, g)) =
        make_uint4(pack2<FP16>(v[0], v[1]), pack2<FP16>(v[2], v[3]), pack2<FP16>(v[4], v[5]), pack2<FP16>(v[6], v[7]));
  };
  // one work item = 8 columns of one feature and one evaluated scale, stored as
  // 16-byte chunks of the operand.  With s_{k+3} = 2 s_k, sin/cos are evaluated
  // for the scales k = 0-2, 6-8, 12-14 only and the others follow by one step of
  // the double angle identities (2 s c, (c - s)(c + s)), so no value is more than
  // one doubling (a few ulp) from an evaluated one.
  const int n_eval = p.scale_doubling ? 9 : 16;
  for (int it = lane; it < (TILE / 8) * 5 * n_eval; it += 32) {
    const int g = it % (TILE / 8), fk = it / (TILE / 8), f = fk % 5, bi = fk / 5;
    const int kb = p.scale_doubling ? (bi / 3) * 6 + bi % 3 : bi;
    float sn[8], cs[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int col = 8 * g + j;
      sn[j] = 0.0f;
      cs[j] = 0.0f;
      if (md->col_flags[col] & F_VALID) {
        const float r = arg(col, f, p.scale[kb]);
        sn[j] = sinpif(r);
        cs[j] = cospif(r);
      }
    }
    put(f * 32 + kb, g, sn);
    put(f * 32 + 16 + kb, g, cs);
    if (p.scale_doubling && kb + 3 < 16) {
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const float s2 = 2.0f * sn[j] * cs[j], c2 = (cs[j] - sn[j]) * (cs[j] + sn[j]);
        sn[j] = s2;
        cs[j] = c2;
      }
      put(f * 32 + kb + 3, g, sn);
      put(f * 32 + 16 + kb + 3, g, cs);
    }
  }
}

// Tile start on the epilogue side: the Fourier operand from the CTA's global
// buffer into HB (five 16-byte chunks per thread, all loads in flight at once).
// The loads bypass L1 (ld.global.cg): the buffer is rewritten by the loader warp
// every other tile, and a line of an earlier tile's operand must not be served
// from L1.  The loads (fourier_fetch) can be issued before HB is free; the
// stores (fourier_put) only after.
static_assert(EB_BYTES == 5 * 16 * NE, "one chunk per thread per round");
__device__ __forceinline__ void fourier_fetch(const ECtx& x, const uint8_t* fb, uint4 (&v)[5]) {
#pragma unroll
  for (int r = 0; r < 5; ++r) v[r] = __ldcg(reinterpret_cast<const uint4*>(fb) + r * NE + x.te);
}
__device__ __forceinline__ void fourier_put(const ECtx& x, const uint4 (&v)[5]) {
#pragma unroll
  for (int r = 0; r < 5; ++r) st_shared_v4(x.hb + 16 * (r * NE + x.te), v[r].x, v[r].y, v[r].z, v[r].w);
}

template <bool FP16>
__global__ void __launch_bounds__(NT, 1) tc_forward_kernel(const __grid_constant__ TcParams p) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (base - raw);
  const uint32_t xb = base + p.off_xb, hb = base + p.off_hb, ab = base + p.off_a;
  Misc* m = reinterpret_cast<Misc*>(gbase + p.off_misc);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t full0 = smem_u32(&m->full[0]), empty0 = smem_u32(&m->empty[0]);
  const uint32_t acc_bar0 = smem_u32(&m->acc_bar[0]), acc_bar1 = smem_u32(&m->acc_bar[1]);
  const uint32_t e_bar0 = smem_u32(&m->e_bar[0]), e_bar1 = smem_u32(&m->e_bar[1]);
  const uint32_t hb_bar = smem_u32(&m->hb_bar), eh_bar = smem_u32(&m->eh_bar);
  const uint32_t drain_bar = smem_u32(&m->drain_bar);

  if (threadIdx.x == 0) {
    for (int s = 0; s < p.nst; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, 1);
    }
    mbar_init(acc_bar0, 1);
    mbar_init(acc_bar1, 1);
    mbar_init(e_bar0, NE / 32);   // one arrival per epilogue warp
    mbar_init(e_bar1, NE / 32);
    mbar_init(hb_bar, 1);
    mbar_init(eh_bar, NE / 32);
    mbar_init(drain_bar, 1);
    for (int b = 0; b < 2; ++b) {
      mbar_init(smem_u32(&m->meta_full[b]), 1);
      mbar_init(smem_u32(&m->meta_free[b]), NE / 32);
    }
    m->abort_flag = 0;
    fence_mbar_init();
  }
  uint32_t* sched_s = reinterpret_cast<uint32_t*>(gbase + p.off_misc + MISC_BYTES);   // [2][MAX_SCHED]
  for (int i = threadIdx.x; i < p.n_sched; i += blockDim.x) {
    sched_s[i] = p.sched_p[i];
    sched_s[MAX_SCHED + i] = p.sched_m[i];
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&m->tmem_base), 512);
    tmem_relinquish();
  }
  if (warp == 0 && lane == 0)
    for (int i = 0; i < NMAPS; ++i) prefetch_tmap(&p.tm[i]);
  static_assert(NT == 608 && NE == 512 && SEGW == 32, "warp roles assume 19 warps");
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = m->tmem_base;
  const int n_slabs = *p.n_slabs;
  const int n_tiles = (n_slabs + 1) >> 1;
  volatile int* abort = &m->abort_flag;

  if (warp == 0) {
    // TMA producer: two consecutive 16 KB weight blocks per stage, in schedule
    // order (the CTA's block sequence runs on across tiles; a final odd block
    // occupies a stage alone).  The whole warp walks the schedule and waits; one
    // elected lane issues (a loop run by a lone lane issues far slower).
    uint32_t stage = 0, phase = 0;
    bool ok = true;
    int issued = 0, half = 0;
    int my_tiles = 0;
    for (int t = blockIdx.x; t < n_tiles; t += gridDim.x) ++my_tiles;
    const int total = my_tiles * p.n_sched;
    for (int t = blockIdx.x; t < n_tiles && ok; t += gridDim.x) {
      for (int i = 0; i < p.n_sched; ++i) {
        const uint32_t e = sched_s[i];
        if (half == 0) {
          const bool got = mbar_wait(empty0 + 8 * stage, phase ^ 1u, abort, p.wait_ns);
          if (!__all_sync(0xffffffffu, got)) {
            if (lane == 0) set_abort(m, p.err);
            ok = false;
            break;
          }
        }
        if (elect_one()) {
          if (half == 0) mbar_arrive_expect_tx(full0 + 8 * stage, issued + 1 < total ? A_STAGE : A_BLOCK);
          tma_load_2d(ab + stage * A_STAGE + half * A_BLOCK, &p.tm[e & 15u], full0 + 8 * stage,
                      (int)((e >> 4) & 15u) * 64, (int)(e >> 8));
        }
        __syncwarp();
        ++issued;
        if (++half == 2) {
          half = 0;
          if (++stage == (uint32_t)p.nst) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
    }
    if (!ok) {
      // let the copies already issued land before the CTA can exit
      volatile int never = 0;
      const int used = (issued + 1) / 2;
      for (int k = 0; k < p.nst && k < used; ++k) {
        const int i = used - 1 - k;
        mbar_wait(full0 + 8 * (i % p.nst), (uint32_t)((i / p.nst) & 1), &never, DRAIN_NS);
      }
    }
  } else if (warp == 1) {
    // MMA issuer, run by the whole warp with one elected lane issuing.  One
    // iteration per stage (two consecutive schedule blocks, 8 MMAs): the stage's
    // barrier is tested without blocking first, and both blocks go out in one
    // elected run unless an epilogue hand-over falls between them, so the
    // per-iteration bookkeeping stays short next to the tensor pipe's queue.
    uint32_t stage = 0, phase = 0, eh_phase = 0, e_k = 0, e_phase0 = 0, e_phase1 = 0;
    bool ok = true;
    int my_tiles = 0;
    for (int t = blockIdx.x; t < n_tiles; t += gridDim.x) ++my_tiles;
    const int total = my_tiles * p.n_sched;
    const int n_stages = (total + 1) >> 1;
    const uint64_t a_desc0 = sdesc_sw128(ab, 16, 1024);
    const uint64_t b_desc_xb = sdesc_sw128(xb, B_LBO, B_SBO), b_desc_hb = sdesc_sw128(hb, B_LBO, B_SBO);
    constexpr uint32_t BSTEP = (2 * B_SBO) >> 4;
    const uint32_t* sm_tab = sched_s + MAX_SCHED;
    const uint32_t idesc = p.idesc;
    auto wait_bar = [&](uint32_t bar, uint32_t& ph, bool spin) -> bool {
      const bool got = spin ? mbar_wait_spin(bar, ph, abort, p.wait_ns) : mbar_wait(bar, ph, abort, p.wait_ns);
      if (!__all_sync(0xffffffffu, got)) {
        if (lane == 0) set_abort(m, p.err);
        return false;
      }
      ph ^= 1u;
      return true;
    };
    auto handover = [&](uint32_t e) -> bool {
      if (e & S_W_E) {   // the k-th W_E hand-over arrives on e_bar[k % 2]
        const bool got = (e_k & 1u) ? wait_bar(e_bar1, e_phase1, false) : wait_bar(e_bar0, e_phase0, false);
        if (!got) return false;
        ++e_k;
      } else if (!wait_bar(eh_bar, eh_phase, false)) {
        return false;
      }
      tc_fence_after();
      return true;
    };
    // The k-th accumulator commit goes to acc_bar[k % 2] (some commits come in
    // pairs with no epilogue hand-over between them; see the epilogue).  The
    // count is kept by the whole warp: the barrier of a block's commit, and the
    // count advanced past it.
    uint32_t acc_k = 0;
    auto acc_for = [&](uint32_t e) -> uint32_t {
      const uint32_t b = (acc_k & 1u) ? acc_bar1 : acc_bar0;
      if (e & S_C_ACC) ++acc_k;
      return b;
    };
    // the MMAs and group commits of one block (elected lane only)
    auto issue = [&](uint32_t e, uint64_t ad, uint32_t acc_b) {
      const uint64_t bd = ((e >> 13) & 1u ? b_desc_hb : b_desc_xb) + (uint64_t)(e & 0x1FFFu);
      const uint32_t d = tmem + ((e >> 14) & 3u) * 128u;
      const uint32_t nk4 = e & S_NK4;
      umma_f16(d, ad, bd, idesc, e & S_ACC);
      umma_f16(d, ad + 2, bd + BSTEP, idesc, 1u);
      umma_f16_if(d, ad + 4, bd + 2 * BSTEP, idesc, 1u, nk4);
      umma_f16_if(d, ad + 6, bd + 3 * BSTEP, idesc, 1u, nk4);
      umma_commit_if(acc_b, e & S_C_ACC);
      umma_commit_if(hb_bar, e & S_C_HB);
    };
    int i0 = 0;   // schedule index of the stage's first block
    for (int sg = 0; sg < n_stages; ++sg) {
      int i1 = i0 + 1;
      if (i1 == p.n_sched) i1 = 0;
      const bool two = 2 * sg + 1 < total;
      const uint32_t e0 = sm_tab[i0], e1 = two ? sm_tab[i1] : 0u;
      i0 = i1 + 1;
      if (i0 >= p.n_sched) i0 -= p.n_sched;
      const uint32_t ab0 = acc_for(e0), ab1 = acc_for(e1);   // (e1 = 0 commits nothing)
      if ((e0 & (S_W_E | S_W_H)) && !(ok = handover(e0))) break;
      if (!mbar_test_wait(full0 + 8 * stage, phase)) {
        uint32_t ph = phase;
        if (!(ok = wait_bar(full0 + 8 * stage, ph, false))) break;
      }
      tc_fence_after();
      const uint64_t ad0 = a_desc0 + (uint64_t)((stage * A_STAGE) >> 4);
      const uint64_t ad1 = ad0 + (uint64_t)(A_BLOCK >> 4);
      const uint32_t empty = empty0 + 8 * stage;
      if (e1 & (S_W_E | S_W_H)) {   // a hand-over between the two blocks
        if (elect_one()) issue(e0, ad0, ab0);
        __syncwarp();
        if (!(ok = handover(e1))) break;
        if (elect_one()) {
          issue(e1, ad1, ab1);
          umma_commit(empty);
        }
        __syncwarp();
      } else {
        if (elect_one()) {
          issue(e0, ad0, ab0);
          if (two) issue(e1, ad1, ab1);
          umma_commit(empty);
        }
        __syncwarp();
      }
      if (++stage == (uint32_t)p.nst) {
        stage = 0;
        phase ^= 1u;
      }
    }
    // no MMA may still run when TMEM is released (the elected lane is the one
    // that issued them)
    if (elect_one()) umma_commit(drain_bar);
    __syncwarp();
    volatile int never = 0;
    mbar_wait(drain_bar, 0, &never, DRAIN_NS);
  } else if (warp < 2 + NE / 32) {
    ECtx x;
    x.p = &p;
    x.m = m;
    x.xb = xb;
    x.hb = hb;
    x.e = warp - 2;
    x.q = warp & 3;
    x.seg = x.e >> 2;
    x.half = x.seg >> 1;
    x.sub = x.seg & 1;
    x.lane = lane;
    x.c = 32 * x.q + lane;
    x.col0 = SEGW * x.seg;
    x.te = threadIdx.x - 64;
    x.MT = p.D >> 7;
    x.tq = tmem + ((uint32_t)(32 * x.q) << 16);
    x.xs = p.xs + (size_t)blockIdx.x * TILE * p.D;
    uint32_t acc_ph0 = 0, acc_ph1 = 0, hb_phase = 0;
    // The epilogue warps run decoupled: each makes its shared-memory operand
    // writes visible to the async proxy, orders its TMEM reads and arrives on the
    // hand-over barrier itself (e_bar and eh_bar count one arrival per warp), and
    // each polls the MMA commits itself.  Some consecutive hand-overs do not wait
    // for the issuer in between (gate tile 0 then 1, SiLU 0 then 1, x_hat 0 then
    // 1), so a warp can arrive for the next one before a slower warp has arrived
    // for the current one; on a single counting barrier that arrival would
    // complete the current phase early.  The W_E hand-overs therefore alternate
    // between two barriers: a warp is never more than one hand-over ahead of
    // another (the one after a pair waits for a product that needs both).  The
    // accumulator commits come in such pairs too (the last merge's two channel
    // tiles, MLP1's, MLP2's, the embedding's second product): a warp that starts
    // its wait for the first of a pair after the second has landed would see the
    // phase parity flipped twice, so they alternate between two barriers as
    // well (a warp is never two commits behind: the issuer makes commit k + 2
    // only after a hand-over that every warp gives after its wait for commit k).
    // A failed wait sets the abort flag and every later wait fails fast, but no
    // warp leaves the loop early: all warps keep taking the same sequence of named
    // barriers (the column-norm exchanges, the segment hand-overs), so none of
    // them can be left waiting.
    auto signal_to = [&](uint32_t bar, bool wrote_operands) {
      if (wrote_operands) fence_proxy_async_smem();   // costly: only after operand writes
      tc_fence_before();
      __syncwarp();
      if (x.lane == 0) mbar_arrive(bar);
    };
    uint32_t e_k = 0;   // W_E hand-overs so far: the next goes to e_bar[e_k % 2]
    auto signal_e = [&](bool wrote_operands) {
      signal_to((e_k & 1u) ? e_bar1 : e_bar0, wrote_operands);
      ++e_k;
    };
    auto signal = [&]() { signal_e(true); };
    auto wait_on = [&](uint32_t bar, uint32_t& ph) {
      const bool got = mbar_wait(bar, ph, abort, p.wait_ns);   // try_wait: suspends instead of polling
      if (!__all_sync(0xffffffffu, got) && x.lane == 0) set_abort(m, p.err);
      ph ^= 1u;
      tc_fence_after();
    };
    uint32_t acc_k = 0;   // accumulator commits waited for so far: the next is on acc_bar[acc_k % 2]
    auto wait_acc = [&]() {
      if (acc_k & 1u)
        wait_on(acc_bar1, acc_ph1);
      else
        wait_on(acc_bar0, acc_ph0);
      ++acc_k;
    };
    const uint8_t* fbuf = p.fbuf + (size_t)blockIdx.x * 2 * EB_BYTES;
    uint32_t meta_ph[2] = {0u, 0u};
    // tile start: the loader's metadata and Fourier operand of the CTA's i-th tile
    // the loads wait for the loader's hand-over of tile i; the stores, after
    // which the operand is handed to the issuer, need HB free
    auto tile_fetch = [&](int i, uint4 (&v)[5]) {
      const int b = i & 1;
      wait_on(smem_u32(&m->meta_full[b]), meta_ph[b]);
      fourier_fetch(x, fbuf + b * EB_BYTES, v);
    };
    auto tile_put = [&](const uint4 (&v)[5]) {
      fourier_put(x, v);
      signal();
    };
    auto tile_in = [&](int i) {
      uint4 v[5];
      tile_fetch(i, v);
      tile_put(v);
    };
    if ((int)blockIdx.x < n_tiles) tile_in(0);
    int i = 0;
    for (int t = blockIdx.x; t < n_tiles; t += gridDim.x, ++i) {
      x.md = &m->meta[i & 1];
      ep_silu<FP16>(x, p.b_e1, wait_acc);
      signal();
      ep_residual<FP16>(x, p.b_e2, p.g, wait_acc, signal);   // embedding output X0
      for (int l = 0; l < p.L; ++l) {
        for (int dc = 0; dc < p.NDC; ++dc) {
          // biases are loaded before the wait so their latency hides behind it
          const size_t rb = (size_t)l * p.ROWS_IN + dc * 256;
          const float bz = p.b_in[rb + x.c], bn = p.b_in[rb + 128 + x.c];
          wait_acc();
          float z[32], n[32];
          scan_load(x, z, n);
          signal_e(false);   // the z/n columns are free for the next chunk
          scan_gates(x, z, n, bz, bn);
          // HB still feeds the merge of the previous chunk (the gate hand-over
          // covers the last merge of the previous layer)
          if (dc > 0) wait_on(hb_bar, hb_phase);
          scan_chain_store<FP16>(x, z, n);
          signal_to(eh_bar, true);
        }
        // gate and MLP1 epilogues one 128-channel tile at a time (the issuer
        // pipelines the next tile's products behind each); with d_model 256 the
        // SiLU of tile 0 goes to HB (MLP1 still reads XB rows 0-127 then)
        // the biases of the thread's channels are loaded ahead of the waits
        const float* b1 = p.b_1 + (size_t)l * p.D;
        const float* bmp = p.b_m + (size_t)l * p.D;
        const float* bgp = p.b_in + (size_t)l * p.ROWS_IN + p.NDC * 256;
        const float bm0 = bmp[x.c], bg0 = bgp[x.c], b10 = b1[x.c];
        float xg[32];
        gate_x_load(x, 0, xg);
        wait_acc();
        ep_gate<FP16>(x, 0, xg, bm0, bg0);
        signal();
        if (x.MT == 2) {
          const float bm1 = bmp[128 + x.c], bg1 = bgp[128 + x.c], b11 = b1[128 + x.c];
          gate_x_load(x, 1, xg);
          wait_acc();
          ep_gate<FP16>(x, 1, xg, bm1, bg1);
          signal();
          wait_acc();
          ep_silu_mt<FP16>(x, b10, 0, 256, x.hb, 0);
          signal();
          wait_acc();
          ep_silu_mt<FP16>(x, b11, 1, 256, x.xb, 128);
          signal();
        } else {
          wait_acc();
          ep_silu_mt<FP16>(x, b10, 0, 256, x.xb, 0);
          signal();
        }
        if (l + 1 < p.L) {
          ep_residual<FP16>(x, p.b_2 + (size_t)l * p.D, p.g + (size_t)(l + 1) * p.D, wait_acc, signal);
        } else {
          // once both output tiles of the last MLP2 have completed, HB and XB
          // are free: the next tile's Fourier operand (fetched before the
          // waits) goes in and its first product (into the z/n columns) runs
          // while this tile is pooled
          const bool more = t + (int)gridDim.x < n_tiles;
          uint4 fv[5];
          if (more) tile_fetch(i + 1, fv);
          wait_acc();
          if (x.MT == 2) wait_acc();
          if (more) tile_put(fv);
          ep_pool(x, p.b_2 + (size_t)l * p.D);
          signal_to(smem_u32(&m->meta_free[i & 1]), false);   // this tile's metadata is no longer read
        }
      }
    }
  } else {
    // loader warp: tile set-up one tile ahead of the epilogue
    uint8_t* fbuf = p.fbuf + (size_t)blockIdx.x * 2 * EB_BYTES;
    uint32_t free_ph[2] = {0u, 0u};
    int i = 0;
    for (int t = blockIdx.x; t < n_tiles; t += gridDim.x, ++i) {
      const int b = i & 1;
      if (i >= 2) {   // buffer b last held the metadata of tile i - 2
        const bool got = mbar_wait(smem_u32(&m->meta_free[b]), free_ph[b], abort, p.wait_ns);
        if (!__all_sync(0xffffffffu, got) && lane == 0) set_abort(m, p.err);
        free_ph[b] ^= 1u;
      }
      load_tile<FP16>(p, m, &m->meta[b], fbuf + b * EB_BYTES, t, n_slabs, lane);
      __threadfence_block();
      __syncwarp();
      if (i == p.hold_tile && blockIdx.x == 0) {
        // test hook: hold this hand-over past the waiters' limit (at most twice
        // the limit, and no longer once a wait has given up), so that the
        // epilogue's wait for it expires; the metadata itself is complete
        const uint64_t t0 = globaltimer();
        while (!*abort && globaltimer() - t0 < 2 * p.wait_ns) {
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&m->meta_full[b]));
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// ------------------------------------------------------------------ schedule
// One thread expands walk_tile into the compact per-block entries read by the
// producer and the MMA issuer (identical for every tile).
__global__ void build_schedule(const __grid_constant__ TcParams p, uint32_t* sp, uint32_t* sm, int* count) {
  int n = 0;
  walk_tile(p, [&](int map, int row, int col, int nk, int tcol, int bsel, int bk, int acc, int wait, int commit) {
    if (n < MAX_SCHED) {
      sp[n] = (uint32_t)map | ((uint32_t)(col >> 6) << 4) | ((uint32_t)row << 8);
      sm[n] = (uint32_t)(((bk >> 3) * B_SBO) >> 4) | ((uint32_t)bsel << 13) | ((uint32_t)(tcol >> 7) << 14) |
              (nk == 4 ? S_NK4 : 0u) | (acc ? S_ACC : 0u) | (commit == C_ACC ? S_C_ACC : 0u) |
              (commit == C_HB ? S_C_HB : 0u) | (wait == W_E ? S_W_E : 0u) | (wait == W_H ? S_W_H : 0u);
    }
    ++n;
  });
  *count = n;
}

// ------------------------------------------------------------------ packing
// Packing of one segment of up to SEG tracks into slabs of at most SLAB hits and
// MAX_TRK_SLAB tracks (one warp per segment, decisions by lane 0 so the order is
// deterministic): best fit over length buckets, each slab taking the longest
// remaining track that still fits until none does; tracks with an invalid hit
// count take a slot but no columns, at the end.  A track's results do not
// depend on where it is packed.  Writes the segment's slice of the packing order
// and the order positions where its slabs start.
__global__ void __launch_bounds__(32) plan_pack(const int32_t* __restrict__ n_hits, int64_t B, int T,
                                                int32_t* __restrict__ seg_count, int32_t* __restrict__ seg_slabs,
                                                int32_t* __restrict__ order) {
  __shared__ int32_t cnt[SLAB + 1], pos[SLAB + 2];
  __shared__ int16_t len_of[SEG], items[SEG];
  const int seg = blockIdx.x, lane = threadIdx.x;
  const int64_t b0 = (int64_t)seg * SEG;
  const int nt = (int)((b0 + SEG < B) ? SEG : B - b0);
  for (int i = lane; i <= SLAB; i += 32) cnt[i] = 0;
  __syncwarp();
  for (int i = lane; i < nt; i += 32) {
    int v = n_hits[b0 + i];
    if (v < 1 || v > T) v = 0;
    len_of[i] = (int16_t)v;
  }
  __syncwarp();
  if (lane == 0) {
    for (int i = 0; i < nt; ++i) ++cnt[len_of[i]];
    pos[0] = 0;
    for (int l = 0; l <= SLAB; ++l) pos[l + 1] = pos[l] + cnt[l];
    for (int i = 0; i < nt; ++i) items[pos[len_of[i]]++] = (int16_t)i;   // pos[l] -> end of bucket l
    int32_t* out = seg_slabs + (size_t)seg * (SEG + 1);
    int o = 0, ns = 0, cap = SLAB, ntr = 0;
    int remaining = nt - cnt[0];
    out[ns++] = (int32_t)b0;
    int top = T < SLAB ? T : SLAB;
    while (remaining > 0) {
      int l = cap < top ? cap : top;
      while (l >= 1 && cnt[l] == 0) --l;
      if (l >= 1 && ntr < MAX_TRK_SLAB) {
        order[b0 + o++] = (int32_t)(b0 + items[pos[l] - cnt[l]]);   // bucket l, next in track order
        --cnt[l];
        cap -= l;
        ++ntr;
        --remaining;
      } else {   // the slab is full: start the next one
        out[ns++] = (int32_t)(b0 + o);
        cap = SLAB;
        ntr = 0;
      }
    }
    for (int k = 0; k < cnt[0]; ++k) {   // invalid tracks
      if (ntr == MAX_TRK_SLAB) {
        out[ns++] = (int32_t)(b0 + o);
        ntr = 0;
      }
      order[b0 + o++] = (int32_t)(b0 + items[pos[0] - cnt[0] + k]);
      ++ntr;
    }
    if (o == 0) ns = 0;   // (an empty segment cannot occur: nt >= 1)
    seg_count[seg] = ns;
  }
}

// Exclusive scan of the per-segment slab counts (one block), total and sentinel.
__global__ void plan_scan(const int32_t* __restrict__ seg_count, int nseg, int64_t B, int32_t* __restrict__ seg_off,
                          int32_t* __restrict__ n_slabs, int32_t* __restrict__ slab_start) {
  __shared__ int32_t part[1024];
  const int tid = threadIdx.x;
  const int per = (nseg + 1023) / 1024;
  int32_t s = 0;
  for (int i = 0; i < per; ++i) {
    const int k = tid * per + i;
    if (k < nseg) s += seg_count[k];
  }
  part[tid] = s;
  __syncthreads();
  for (int o = 1; o < 1024; o <<= 1) {
    const int32_t v = tid >= o ? part[tid - o] : 0;
    __syncthreads();
    part[tid] += v;
    __syncthreads();
  }
  int32_t run = part[tid] - s;
  for (int i = 0; i < per; ++i) {
    const int k = tid * per + i;
    if (k < nseg) {
      seg_off[k] = run;
      run += seg_count[k];
    }
  }
  if (tid == 1023) {
    n_slabs[0] = part[1023];
    slab_start[part[1023]] = (int32_t)B;
  }
}

__global__ void plan_scatter(const int32_t* __restrict__ seg_count, const int32_t* __restrict__ seg_off,
                             const int32_t* __restrict__ seg_slabs, int32_t* __restrict__ slab_start) {
  const int seg = blockIdx.x;
  const int cnt = seg_count[seg], off = seg_off[seg];
  for (int i = threadIdx.x; i < cnt; i += blockDim.x) slab_start[off + i] = seg_slabs[(size_t)seg * (SEG + 1) + i];
}

// ------------------------------------------------------------------ UMMA probe
// D[128][128] = A[128][K] * B[K][128] through the same TMA / descriptor / TMEM
// path as the fused kernel (test hook for the operand layouts).
__global__ void __launch_bounds__(128, 1) umma_probe_kernel(const __grid_constant__ CUtensorMap tmA,
                                                            const uint16_t* __restrict__ Bkn, int K,
                                                            float* __restrict__ Dout, uint32_t idesc,
                                                            unsigned long long* err) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (base - raw);
  const uint32_t a_s = base;                 // K/64 blocks of 16 KB
  const uint32_t b_s = base + (K / 64) * A_BLOCK;
  uint64_t* bars = reinterpret_cast<uint64_t*>(gbase + (K / 64) * A_BLOCK + K * 256);
  uint32_t* tbase = reinterpret_cast<uint32_t*>(bars + 2);
  int* abortp = reinterpret_cast<int*>(bars + 3);
  const uint32_t tma_bar = smem_u32(&bars[0]), mma_bar = smem_u32(&bars[1]);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    mbar_init(tma_bar, 1);
    mbar_init(mma_bar, 1);
    *abortp = 0;
    fence_mbar_init();
  }
  if (warp == 0) {
    tmem_alloc(smem_u32(tbase), 128);
    tmem_relinquish();
  }
  // B operand written by the threads, exactly as the epilogue does
  for (int idx = threadIdx.x; idx < K * 16; idx += 128) {
    const int k = idx >> 4, n8 = idx & 15;
    const uint16_t* src = Bkn + (size_t)k * 128 + n8 * 8;
    uint32_t w[4];
    for (int i = 0; i < 4; ++i) w[i] = (uint32_t)src[2 * i] | ((uint32_t)src[2 * i + 1] << 16);
    st_shared_v4(b_s + bchunk(k, n8), w[0], w[1], w[2], w[3]);
  }
  fence_proxy_async_smem();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tbase;
  volatile int* abort = abortp;
  bool ok = true;
  if (threadIdx.x == 0) {
    mbar_arrive_expect_tx(tma_bar, (K / 64) * A_BLOCK);
    for (int kc = 0; kc < K / 64; ++kc) tma_load_2d(a_s + kc * A_BLOCK, &tmA, tma_bar, kc * 64, 0);
    ok = mbar_wait(tma_bar, 0, abort, WAIT_NS);
    if (ok) {
      tc_fence_after();
      for (int kc = 0; kc < K / 64; ++kc)
        for (int k = 0; k < 4; ++k) {
          const uint64_t ad = sdesc_sw128(a_s + kc * A_BLOCK + 32 * k, 16, 1024);
          const uint64_t bd = sdesc_sw128(b_s + ((kc * 64 + 16 * k) >> 3) * B_SBO, B_LBO, B_SBO);
          umma_f16(tmem, ad, bd, idesc, (kc || k) ? 1u : 0u);
        }
      umma_commit(mma_bar);
    } else {
      atomicAdd(err + 1, 1ull);
      *abortp = 1;
    }
  }
  __syncthreads();
  if (!*abort) {
    if (mbar_wait(mma_bar, 0, abort, WAIT_NS)) {
      tc_fence_after();
      const uint32_t tq = tmem + ((uint32_t)(32 * warp) << 16);
      for (int ch = 0; ch < 4; ++ch) {
        float v[32];
        tmem_ld32(tq + 32 * ch, v);
        tmem_ld_wait();
        for (int i = 0; i < 32; ++i) Dout[(size_t)(32 * warp + lane) * 128 + 32 * ch + i] = v[i];
      }
    } else if (lane == 0) {
      atomicAdd(err + 1, 1ull);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, 128);
  }
}

// ------------------------------------------------------------------ host side
uint16_t fp16_bits(float f) {
  const __half v = __float2half_rn(f);
  return *reinterpret_cast<const uint16_t*>(&v);
}
uint16_t bf16_bits(float f) {
  uint32_t u;
  std::memcpy(&u, &f, 4);
  if ((u & 0x7f800000u) == 0x7f800000u && (u & 0x007fffffu)) return 0x7fc0;
  u += 0x7fffu + ((u >> 16) & 1u);
  return (uint16_t)(u >> 16);
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
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

// bf16 matrix [rows][cols] row-major -> tensor map with 64 x 128 boxes, 128 B swizzle.
bool make_map(CUtensorMap* m, const void* ptr, uint64_t rows, uint64_t cols, bool fp16 = false) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {64, 128};
  cuuint32_t es[2] = {1, 1};
  return fn(m, fp16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// ------------------------------------------------------------------ head
// Pooled vector -> RMSNorm (gain g_h) -> W_h1 (D -> 128) + SiLU -> W_h2 (128 -> Q)
// for every track, fp32 on the CUDA cores (the head of Sec. 3.2).  One CTA per SM
// walks blocks of HEAD_TRK tracks with both weight matrices staged in shared
// memory once per CTA; the fused kernel leaves the pooled means in global memory.
struct HeadParams {
  const float* pool;   // [B][D] pooled means
  const int32_t* n_hits;
  int64_t B;
  int T, D, Q, NQ;
  float rms_eps;
  const float* g;     // [D]
  const float* w1t;   // [D][128]
  const float* b1;    // [128]
  const float* w2;    // [Q][128]
  const float* b2;    // [Q]
  float* out;         // [B][5]
  float* out_q;       // [B][Q] or null
  float* out_pool;    // the caller's pooled buffer (invalid tracks -> NaN) or null
  unsigned long long* err;
};
constexpr int HEAD_TRK = 32, HEAD_NT = 256;
size_t head_smem_bytes(int D, int Q) {
  return ((size_t)D * 128 + (size_t)Q * 128 + (size_t)HEAD_TRK * D + (size_t)HEAD_TRK * 128 + D + 128 + Q +
          HEAD_TRK) * 4;
}

__global__ void __launch_bounds__(HEAD_NT, 1) head_kernel(const __grid_constant__ HeadParams hp) {
  extern __shared__ float4 hsm4[];
  const int D = hp.D, Q = hp.Q;
  float* w1t = reinterpret_cast<float*>(hsm4);   // [D][128]
  float* w2 = w1t + D * 128;                      // [Q][128]
  float* xv = w2 + Q * 128;                       // [HEAD_TRK][D]
  float* hid = xv + HEAD_TRK * D;                 // [HEAD_TRK][128]
  float* gs = hid + HEAD_TRK * 128;               // [D]
  float* b1s = gs + D;                            // [128]
  float* b2s = b1s + 128;                         // [Q]
  int* bad_s = reinterpret_cast<int*>(b2s + Q);   // [HEAD_TRK]
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  for (int i = tid; i < D * 32; i += HEAD_NT) reinterpret_cast<float4*>(w1t)[i] = reinterpret_cast<const float4*>(hp.w1t)[i];
  for (int i = tid; i < Q * 32; i += HEAD_NT) reinterpret_cast<float4*>(w2)[i] = reinterpret_cast<const float4*>(hp.w2)[i];
  for (int i = tid; i < D; i += HEAD_NT) gs[i] = hp.g[i];
  for (int i = tid; i < 128; i += HEAD_NT) b1s[i] = hp.b1[i];
  for (int i = tid; i < Q; i += HEAD_NT) b2s[i] = hp.b2[i];
  __syncthreads();
  const float qnan = __int_as_float(0x7fc00000);
  const int64_t nblk = (hp.B + HEAD_TRK - 1) / HEAD_TRK;
  for (int64_t blk = blockIdx.x; blk < nblk; blk += gridDim.x) {
    const int64_t t0 = blk * HEAD_TRK;
    const int nt = (int)((hp.B - t0) < HEAD_TRK ? (hp.B - t0) : HEAD_TRK);
    // RMSNorm of each pooled vector (one warp per track); padding rows and
    // invalid tracks become zero rows whose outputs are replaced by NaN
    for (int i = warp; i < HEAD_TRK; i += HEAD_NT / 32) {
      float* row = xv + i * D;
      bool bad = true;
      if (i < nt) {
        const int n = hp.n_hits[t0 + i];
        bad = n < 1 || n > hp.T;
      }
      if (bad) {
        for (int c = lane; c < D; c += 32) row[c] = 0.0f;
        if (i < nt && hp.out_pool)
          for (int c = lane; c < D; c += 32) hp.out_pool[(t0 + i) * D + c] = qnan;
      } else {
        const float4* src = reinterpret_cast<const float4*>(hp.pool + (t0 + i) * D);
        float ss = 0.0f;
        for (int c4 = lane; c4 < D / 4; c4 += 32) {
          const float4 v = src[c4];
          reinterpret_cast<float4*>(row)[c4] = v;
          ss = fmaf(v.x, v.x, ss);
          ss = fmaf(v.y, v.y, ss);
          ss = fmaf(v.z, v.z, ss);
          ss = fmaf(v.w, v.w, ss);
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
        const float r = 1.0f / sqrtf(ss / (float)D + hp.rms_eps);
        for (int c = lane; c < D; c += 32) row[c] *= r * gs[c];
      }
      if (lane == 0) bad_s[i] = bad;
    }
    __syncthreads();
    {   // hidden units 4*j4 .. 4*j4+3 of tracks 4*tg .. 4*tg+3 (16-byte loads of
        // both operands: 8 loads per 64 FMAs); the sum over c runs in order
      const int j4 = tid & 31, tg = tid >> 5;
      float a[4][4];
#pragma unroll
      for (int r = 0; r < 4; ++r)
#pragma unroll
        for (int u = 0; u < 4; ++u) a[r][u] = b1s[4 * j4 + u];
#pragma unroll 2
      for (int c = 0; c < D; c += 4) {
        float4 w[4], xr[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) w[k] = *reinterpret_cast<const float4*>(w1t + (c + k) * 128 + 4 * j4);
#pragma unroll
        for (int r = 0; r < 4; ++r) xr[r] = *reinterpret_cast<const float4*>(xv + (4 * tg + r) * D + c);
#pragma unroll
        for (int r = 0; r < 4; ++r) {
          const float xk[4] = {xr[r].x, xr[r].y, xr[r].z, xr[r].w};
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            a[r][0] = fmaf(w[k].x, xk[k], a[r][0]);
            a[r][1] = fmaf(w[k].y, xk[k], a[r][1]);
            a[r][2] = fmaf(w[k].z, xk[k], a[r][2]);
            a[r][3] = fmaf(w[k].w, xk[k], a[r][3]);
          }
        }
      }
#pragma unroll
      for (int r = 0; r < 4; ++r)
        *reinterpret_cast<float4*>(hid + (4 * tg + r) * 128 + 4 * j4) =
            make_float4(silu(a[r][0]), silu(a[r][1]), silu(a[r][2]), silu(a[r][3]));
    }
    __syncthreads();
    // outputs; the dot product for output o starts at column 4o (mod 128), so the
    // rows of W_h2 read by one warp fall in different banks while the
    // summation order stays a function of o alone (results do not depend on a
    // track's position in the batch)
    for (int idx = tid; idx < nt * Q; idx += HEAD_NT) {
      const int i = idx / Q, o = idx - i * Q;
      const float4* w = reinterpret_cast<const float4*>(w2 + o * 128);
      const float4* hv = reinterpret_cast<const float4*>(hid + i * 128);
      float acc = 0.0f;
#pragma unroll 8
      for (int u = 0; u < 32; ++u) {
        const int j4 = (u + o) & 31;
        const float4 a4 = w[j4], h4 = hv[j4];
        acc = fmaf(a4.x, h4.x, acc);
        acc = fmaf(a4.y, h4.y, acc);
        acc = fmaf(a4.z, h4.z, acc);
        acc = fmaf(a4.w, h4.w, acc);
      }
      acc += b2s[o];
      const int64_t trk = t0 + i;
      if (bad_s[i]) acc = qnan;
      if (hp.out_q) hp.out_q[trk * Q + o] = acc;
      if (o % hp.NQ == hp.NQ / 2) hp.out[trk * 5 + o / hp.NQ] = acc;
    }
    if (tid < nt && bad_s[tid]) atomicAdd(hp.err, 1ull);
    __syncthreads();
  }
}

}  // namespace

struct tf_tc_state {
  int nsm = 0, nst = 0, NDC = 0, ROWS_IN = 0, KM = 0;
  size_t smem = 0;
  int off_xb = 0, off_hb = 0, off_a = 0, off_misc = 0;
  uint32_t idesc = 0;
  void* dev = nullptr;  // one allocation for all weights
  uint16_t *w_e1 = nullptr, *w_e2 = nullptr, *w_in = nullptr, *w_m = nullptr, *w_1 = nullptr, *w_2 = nullptr;
  float *b_e1 = nullptr, *b_e2 = nullptr, *g = nullptr, *b_in = nullptr, *b_m = nullptr, *b_1 = nullptr,
        *b_2 = nullptr, *hg = nullptr, *hw1t = nullptr, *hb1 = nullptr, *hw2 = nullptr, *hb2 = nullptr;
  int32_t *seg_count = nullptr, *seg_off = nullptr, *seg_slabs = nullptr, *slab_start = nullptr, *n_slabs = nullptr,
          *order = nullptr;
  uint32_t* sched = nullptr;   // [2][MAX_SCHED]: producer entries, then MMA entries
  int n_sched = 0;
  float* xs = nullptr;
  uint8_t* fbuf = nullptr;
  float* pool = nullptr;   // pooled means when the caller passes no buffer [POOL_TRACKS][D]
  size_t head_smem = 0;
  uint64_t wait_ns = WAIT_NS;   // test hook (trackfit_debug_wait_limit)
  int hold_tile = -1;
  CUtensorMap tm[NMAPS];
};

struct ScheduleCounter {   // a callable for walk_tile on either side
  int64_t c[6] = {0, 0, 0, 0, 0, 0};
  uint8_t* codes = nullptr;   // optional: per block wait | commit << 2, in order
  int64_t cap = 0;
  __host__ __device__ void operator()(int, int, int, int nk, int, int, int, int, int wait, int commit) {
    if (c[0] < cap) codes[c[0]] = (uint8_t)(wait | (commit << 2));
    ++c[0];
    c[1] += nk;
    c[2] += wait == W_E;
    c[3] += wait == W_H;
    c[4] += commit == C_ACC;
    c[5] += commit == C_HB;
  }
};

// Per-tile totals of the fused kernel's block schedule, from the same walk_tile
// the kernel expands (host only, no device needed): counts[0] blocks, [1] MMA
// instructions (128 x 128 x 16 each), [2] W_E and [3] W_H hand-over waits, [4]
// C_ACC and [5] C_HB commits; with codes, also each block's wait | commit << 2
// in issue order (at most cap blocks).
int tf_tc_schedule_counts(const tf_shape& s, int64_t* counts, int n, uint8_t* codes, int64_t cap) {
  if (n < 6 || (cap > 0 && !codes)) return TRACKFIT_ERR_INVALID_ARG;
  TcParams q;
  memset(&q, 0, sizeof(q));
  q.D = s.D;
  q.L = s.L;
  q.NDC = s.H / 64;
  q.ROWS_IN = q.NDC * 256 + s.D;
  ScheduleCounter c;
  c.codes = codes;
  c.cap = cap;
  walk_tile(q, c);
  for (int i = 0; i < 6; ++i) counts[i] = c.c[i];
  return TRACKFIT_OK;
}

int tf_tc_wait_limit(trackfit_ctx* h, int64_t limit_ns, int hold_tile) {
  if (!h->tc) return TRACKFIT_ERR_UNSUPPORTED;
  if (limit_ns < 0 || hold_tile < -1) return TRACKFIT_ERR_INVALID_ARG;
  h->tc->wait_ns = limit_ns > 0 ? (uint64_t)limit_ns : WAIT_NS;
  h->tc->hold_tile = hold_tile;
  return TRACKFIT_OK;
}

bool tf_tc_supported(const tf_shape& s) {
  return (s.precision == TRACKFIT_BF16_PROJ || s.precision == TRACKFIT_FP16_PROJ) && s.pool == TRACKFIT_POOL_MEAN &&
         s.topology == TRACKFIT_TOPOLOGY_MERGE && (s.D == 128 || s.D == 256) &&
         s.H % 64 == 0 && s.T <= 64 && s.Hh == 128 && s.Q <= 75 && s.F == 5 && s.K == 16;
}

void tf_tc_destroy(trackfit_ctx* h) {
  if (!h || !h->tc) return;
  tf_tc_state* t = h->tc;
  tf_free(t->dev);
  tf_free(t->seg_count);
  tf_free(t->xs);
  tf_free(t->fbuf);
  tf_free(t->pool);
  tf_free(t->sched);
  delete t;
  h->tc = nullptr;
}

int tf_tc_create(trackfit_ctx* h, const float* W) {
  const tf_shape& s = h->s;
  const tf_blob_off& o = h->off;
  tf_tc_state* t = new (std::nothrow) tf_tc_state();
  if (!t) return TRACKFIT_ERR_OOM;
  h->tc = t;
  const int D = s.D, H = s.H, L = s.L, E = s.E;
  t->NDC = H / 64;
  t->ROWS_IN = t->NDC * 256 + D;
  t->KM = t->NDC * 128;
  const bool fp16 = s.precision == TRACKFIT_FP16_PROJ;
  t->idesc = idesc_f16(128, 128, fp16 ? 0u : 1u, false, true);
  int dev = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&t->nsm, cudaDevAttrMultiProcessorCount, dev);
  int smem_optin = 0;
  cudaDeviceGetAttribute(&smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  t->off_xb = 0;
  t->off_hb = D * 256;
  t->off_a = t->off_hb + EB_BYTES;
  const int avail = smem_optin - 1024 - MISC_BYTES - SCHED_BYTES - t->off_a;
  t->nst = avail / A_STAGE;
  if (t->nst > MAX_STAGES) t->nst = MAX_STAGES;
  if (t->nst < 2) return TRACKFIT_ERR_UNSUPPORTED;
  t->off_misc = t->off_a + t->nst * A_STAGE;
  t->smem = (size_t)t->off_misc + MISC_BYTES + SCHED_BYTES + 1024;
  t->head_smem = head_smem_bytes(D, s.Q);
  if (t->head_smem > (size_t)smem_optin) return TRACKFIT_ERR_UNSUPPORTED;

  // ---- repack weights (bf16 GEMM operands, fp32 biases/head)
  const size_t n_e1 = (size_t)D * E, n_e2 = (size_t)D * D, n_in = (size_t)L * t->ROWS_IN * D,
               n_m = (size_t)L * D * t->KM, n_11 = (size_t)L * D * D;
  std::vector<uint16_t> we1(n_e1), we2(n_e2), win(n_in, 0), wm(n_m, 0), w1(n_11), w2(n_11);
  std::vector<float> bin((size_t)L * t->ROWS_IN, 0.0f), gg((size_t)L * D), bm((size_t)L * D), b1((size_t)L * D),
      b2((size_t)L * D), hw1t((size_t)s.P * 128);
  uint16_t (*cv)(float) = fp16 ? fp16_bits : bf16_bits;
  for (size_t i = 0; i < n_e1; ++i) we1[i] = cv(W[o.emb_w1 + i]);
  for (size_t i = 0; i < n_e2; ++i) we2[i] = cv(W[o.emb_w2 + i]);
  for (int l = 0; l < L; ++l) {
    const tf_layer_off& lo = o.layer[l];
    const size_t rb = (size_t)l * t->ROWS_IN;
    // scan chunk dc = 64 channels of both directions: rows 0-63 forward,
    // rows 64-127 reverse (z block, then n block); the merge columns follow
    for (int dc = 0; dc < t->NDC; ++dc) {
      for (int c = 0; c < 128; ++c) {
        const int dir = c >> 6, ch = dc * 64 + (c & 63);
        const int src_z = (dir == 0 ? 0 : 2 * H) + ch, src_n = (dir == 0 ? H : 3 * H) + ch;
        for (int k = 0; k < D; ++k) {
          win[(rb + dc * 256 + c) * D + k] = cv(W[lo.w_in + (size_t)src_z * D + k]);
          win[(rb + dc * 256 + 128 + c) * D + k] = cv(W[lo.w_in + (size_t)src_n * D + k]);
        }
        bin[rb + dc * 256 + c] = W[lo.b_in + src_z];
        bin[rb + dc * 256 + 128 + c] = W[lo.b_in + src_n];
        for (int r = 0; r < D; ++r)
          wm[((size_t)l * D + r) * t->KM + dc * 128 + c] = cv(W[lo.w_m + (size_t)r * 2 * H + dir * H + ch]);
      }
    }
    for (int c = 0; c < D; ++c) {
      for (int k = 0; k < D; ++k)
        win[(rb + t->NDC * 256 + c) * D + k] = cv(W[lo.w_in + (size_t)(4 * H + c) * D + k]);
      bin[rb + t->NDC * 256 + c] = W[lo.b_in + 4 * H + c];
    }
    for (size_t i = 0; i < (size_t)D * D; ++i) {
      w1[(size_t)l * D * D + i] = cv(W[lo.w1 + i]);
      w2[(size_t)l * D * D + i] = cv(W[lo.w2 + i]);
    }
    for (int c = 0; c < D; ++c) {
      gg[(size_t)l * D + c] = W[lo.g + c];
      bm[(size_t)l * D + c] = W[lo.b_m + c];
      b1[(size_t)l * D + c] = W[lo.b1 + c];
      b2[(size_t)l * D + c] = W[lo.b2 + c];
    }
  }
  for (int c = 0; c < s.P; ++c)
    for (int j = 0; j < 128; ++j) hw1t[(size_t)c * 128 + j] = W[o.head_w1 + (size_t)j * s.P + c];

  // ---- one device allocation for everything the kernel reads
  struct Part {
    const void* src;
    size_t bytes;
    void** dst;
  };
  std::vector<Part> parts = {
      {we1.data(), n_e1 * 2, (void**)&t->w_e1},
      {we2.data(), n_e2 * 2, (void**)&t->w_e2},
      {win.data(), n_in * 2, (void**)&t->w_in},
      {wm.data(), n_m * 2, (void**)&t->w_m},
      {w1.data(), n_11 * 2, (void**)&t->w_1},
      {w2.data(), n_11 * 2, (void**)&t->w_2},
      {W + o.emb_b1, (size_t)D * 4, (void**)&t->b_e1},
      {W + o.emb_b2, (size_t)D * 4, (void**)&t->b_e2},
      {gg.data(), gg.size() * 4, (void**)&t->g},
      {bin.data(), bin.size() * 4, (void**)&t->b_in},
      {bm.data(), bm.size() * 4, (void**)&t->b_m},
      {b1.data(), b1.size() * 4, (void**)&t->b_1},
      {b2.data(), b2.size() * 4, (void**)&t->b_2},
      {W + o.head_g, (size_t)s.P * 4, (void**)&t->hg},
      {hw1t.data(), hw1t.size() * 4, (void**)&t->hw1t},
      {W + o.head_b1, (size_t)128 * 4, (void**)&t->hb1},
      {W + o.head_w2, (size_t)s.Q * 128 * 4, (void**)&t->hw2},
      {W + o.head_b2, (size_t)s.Q * 4, (void**)&t->hb2},
  };
  size_t total = 0;
  for (auto& pt : parts) total += (pt.bytes + 255) & ~(size_t)255;
  if (tf_malloc((void**)&t->dev, total) != cudaSuccess) return TRACKFIT_ERR_OOM;
  size_t off = 0;
  for (auto& pt : parts) {
    *pt.dst = static_cast<char*>(t->dev) + off;
    if (cudaMemcpy(*pt.dst, pt.src, pt.bytes, cudaMemcpyHostToDevice) != cudaSuccess) return TRACKFIT_ERR_CUDA;
    off += (pt.bytes + 255) & ~(size_t)255;
  }
  // ---- packing buffers and the per-CTA residual scratch
  const int nseg_max = (int)((MAXB + SEG - 1) / SEG);
  const size_t plan_ints = (size_t)nseg_max * 2 + (size_t)nseg_max * (SEG + 1) + (size_t)MAXB + 2 + 64 + (size_t)MAXB;
  if (tf_malloc((void**)&t->seg_count, plan_ints * 4) != cudaSuccess) return TRACKFIT_ERR_OOM;
  t->seg_off = t->seg_count + nseg_max;
  t->seg_slabs = t->seg_off + nseg_max;
  t->slab_start = t->seg_slabs + (size_t)nseg_max * (SEG + 1);
  t->n_slabs = t->slab_start + MAXB + 2;
  t->order = t->n_slabs + 64;
  if (tf_malloc((void**)&t->xs, (size_t)t->nsm * TILE * D * sizeof(float)) != cudaSuccess) return TRACKFIT_ERR_OOM;
  if (tf_malloc((void**)&t->fbuf, (size_t)t->nsm * 2 * EB_BYTES) != cudaSuccess) return TRACKFIT_ERR_OOM;
  if (tf_malloc((void**)&t->pool, (size_t)POOL_TRACKS * D * sizeof(float)) != cudaSuccess) return TRACKFIT_ERR_OOM;
  // ---- tensor maps
  bool ok = make_map(&t->tm[MAP_E1], t->w_e1, D, E, fp16) && make_map(&t->tm[MAP_E2], t->w_e2, D, D, fp16) &&
            make_map(&t->tm[MAP_IN], t->w_in, (uint64_t)L * t->ROWS_IN, D, fp16) &&
            make_map(&t->tm[MAP_M], t->w_m, (uint64_t)L * D, t->KM, fp16) &&
            make_map(&t->tm[MAP_1], t->w_1, (uint64_t)L * D, D, fp16) &&
            make_map(&t->tm[MAP_2], t->w_2, (uint64_t)L * D, D, fp16);
  if (!ok) return TRACKFIT_ERR_CUDA;
  // ---- the per-tile block schedule, expanded once on the device
  {
    TcParams q;
    std::memset(&q, 0, sizeof(q));
    q.D = D;
    q.L = L;
    q.NDC = t->NDC;
    q.ROWS_IN = t->ROWS_IN;
    int* d_count = nullptr;
    if (tf_malloc((void**)&t->sched, 2 * MAX_SCHED * sizeof(uint32_t) + 16) != cudaSuccess) return TRACKFIT_ERR_OOM;
    d_count = reinterpret_cast<int*>(t->sched + 2 * MAX_SCHED);
    build_schedule<<<1, 1>>>(q, t->sched, t->sched + MAX_SCHED, d_count);
    if (cudaMemcpy(&t->n_sched, d_count, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess) return TRACKFIT_ERR_CUDA;
    if (t->n_sched < 1 || t->n_sched > MAX_SCHED) return TRACKFIT_ERR_UNSUPPORTED;
  }
  if (cudaFuncSetAttribute(tc_forward_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)t->smem) !=
          cudaSuccess ||
      cudaFuncSetAttribute(tc_forward_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)t->smem) !=
          cudaSuccess ||
      cudaFuncSetAttribute(head_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)t->head_smem) !=
          cudaSuccess)
    return TRACKFIT_ERR_CUDA;
  return TRACKFIT_OK;
}

int tf_tc_forward(trackfit_ctx* h, const float* hits, const int32_t* n_hits, int64_t B, float* out, float* out_q,
                  float* out_pool, cudaStream_t st, const int64_t* offs) {
  tf_tc_state* t = h->tc;
  const tf_shape& s = h->s;
  TcParams p;
  std::memset(&p, 0, sizeof(p));
  for (int i = 0; i < NMAPS; ++i) p.tm[i] = t->tm[i];
  p.xs = t->xs;
  p.fbuf = t->fbuf;
  p.slab_start = t->slab_start;
  p.order = t->order;
  p.n_slabs = t->n_slabs;
  p.sched_p = t->sched;
  p.sched_m = t->sched + MAX_SCHED;
  p.n_sched = t->n_sched;
  p.b_e1 = t->b_e1;
  p.b_e2 = t->b_e2;
  p.g = t->g;
  p.b_in = t->b_in;
  p.b_m = t->b_m;
  p.b_1 = t->b_1;
  p.b_2 = t->b_2;
  p.err = h->d_err;
  p.wait_ns = t->wait_ns;
  p.hold_tile = t->hold_tile;
  p.T = s.T;
  p.D = s.D;
  p.H = s.H;
  p.L = s.L;
  p.NDC = t->NDC;
  p.ROWS_IN = t->ROWS_IN;
  p.NQ = s.NQ;
  p.Q = s.Q;
  p.nst = t->nst;
  p.idesc = t->idesc;
  p.off_xb = t->off_xb;
  p.off_hb = t->off_hb;
  p.off_a = t->off_a;
  p.off_misc = t->off_misc;
  p.rms_eps = s.rms_eps;
  p.fp16 = s.precision == TRACKFIT_FP16_PROJ;
  for (int f = 0; f < 5; ++f) {
    const double inv = 1.0 / s.feat_range_d[f];
    p.feat_min[f] = s.feat_min[f];
    p.feat_inv_hi[f] = (float)inv;
    p.feat_inv_lo[f] = (float)(inv - (double)p.feat_inv_hi[f]);
  }
  for (int k = 0; k < 16; ++k) p.scale[k] = s.scale[k];
  p.scale_doubling = 1;
  for (int k = 0; k + 3 < 16; ++k)
    if (s.scale[k + 3] != 2.0f * s.scale[k]) p.scale_doubling = 0;
  HeadParams hp;
  std::memset(&hp, 0, sizeof(hp));
  hp.T = s.T;
  hp.D = s.D;
  hp.Q = s.Q;
  hp.NQ = s.NQ;
  hp.rms_eps = s.rms_eps;
  hp.g = t->hg;
  hp.w1t = t->hw1t;
  hp.b1 = t->hb1;
  hp.w2 = t->hw2;
  hp.b2 = t->hb2;
  hp.err = h->d_err;
  // without a caller buffer the pooled means go to the internal one, which
  // bounds the launch chunk
  const int64_t chunk = out_pool ? MAXB : POOL_TRACKS;
  for (int64_t c0 = 0; c0 < B; c0 += chunk) {
    const int64_t nb = (B - c0 < chunk) ? B - c0 : chunk;
    const int nseg = (int)((nb + SEG - 1) / SEG);
    plan_pack<<<nseg, 32, 0, st>>>(n_hits + c0, nb, s.T, t->seg_count, t->seg_slabs, t->order);
    plan_scan<<<1, 1024, 0, st>>>(t->seg_count, nseg, nb, t->seg_off, t->n_slabs, t->slab_start);
    plan_scatter<<<nseg, 128, 0, st>>>(t->seg_count, t->seg_off, t->seg_slabs, t->slab_start);
    p.hits = offs ? hits : hits + c0 * s.T * 5;
    p.offs = offs ? offs + c0 : nullptr;
    p.n_hits = n_hits + c0;
    p.out = out + c0 * 5;
    p.out_q = out_q ? out_q + c0 * s.Q : nullptr;
    p.pool = out_pool ? out_pool + c0 * s.P : t->pool;
    tf_prof_begin(h, st);
    if (p.fp16)
      tc_forward_kernel<true><<<t->nsm, NT, t->smem, st>>>(p);
    else
      tc_forward_kernel<false><<<t->nsm, NT, t->smem, st>>>(p);
    tf_prof_end(h, st);
    hp.pool = p.pool;
    hp.n_hits = p.n_hits;
    hp.B = nb;
    hp.out = p.out;
    hp.out_q = p.out_q;
    hp.out_pool = out_pool ? p.pool : nullptr;
    head_kernel<<<t->nsm, HEAD_NT, t->head_smem, st>>>(hp);
    if (cudaPeekAtLastError() != cudaSuccess) return TRACKFIT_ERR_CUDA;
  }
  return TRACKFIT_OK;
}

// UMMA layout probe: A device bf16 [128][K] (K-major), Bkn device bf16 [K][128],
// D device fp32 [128][128]; K in {64, 128, 192, 256}.  Synchronous.
int tf_tc_probe(trackfit_ctx* h, const uint16_t* A, const uint16_t* Bkn, int K, float* D, cudaStream_t st) {
  if (K < 64 || K > 256 || (K % 64) != 0) return TRACKFIT_ERR_INVALID_ARG;
  CUtensorMap m;
  if (!make_map(&m, A, 128, (uint64_t)K)) return TRACKFIT_ERR_CUDA;
  const size_t smem = (size_t)(K / 64) * A_BLOCK + (size_t)K * 256 + 64 + 1024;
  if (cudaFuncSetAttribute(umma_probe_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
    return TRACKFIT_ERR_CUDA;
  umma_probe_kernel<<<1, 128, smem, st>>>(m, Bkn, K, D, idesc_f16(128, 128, 1u, false, true), h->d_err);
  if (cudaPeekAtLastError() != cudaSuccess) return TRACKFIT_ERR_CUDA;
  return TRACKFIT_OK;
}
