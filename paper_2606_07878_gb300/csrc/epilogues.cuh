// GEMM epilogues: TMEM -> registers -> fused element-wise work -> global memory.
// Each epilogue thread owns one accumulator row (TMEM lane) of a 128 x BN tile and walks its
// columns 32 at a time.
#pragma once
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "tc_gemm.cuh"

namespace still {

// Element offset of (batch b, row r, column c) as an affine function of their div/mod parts.
struct AffineMap {
  int32_t bdiv = 1, rdiv = 1 << 30, cdiv = 1 << 30;
  int64_t b1 = 0, b0 = 0, r1 = 0, r0 = 0, c1 = 0, c0 = 0, k = 0;
  __device__ __forceinline__ int64_t at(int b, int r, int c) const {
    return (int64_t)(b / bdiv) * b1 + (int64_t)(b % bdiv) * b0 + (int64_t)(r / rdiv) * r1 +
           (int64_t)(r % rdiv) * r0 + (int64_t)(c / cdiv) * c1 + (int64_t)(c % cdiv) * c0 + k;
  }
};

// OUT_HILO: bf16 hi and lo = bf16(x - hi); OUT_HILO16: the same in fp16 (about 22 bits).
enum OutKind : int32_t { OUT_F32 = 0, OUT_BF16 = 1, OUT_HILO = 2, OUT_HILO16 = 3 };

__device__ __forceinline__ void split_hilo(float x, __nv_bfloat16& hi, __nv_bfloat16& lo) {
  hi = __float2bfloat16_rn(x);
  lo = __float2bfloat16_rn(x - __bfloat162float(hi));
}

// GELU with the exact (erf) form, 0.5 x (1 + erf(x / sqrt 2)) (App. A, Feed-forward).
__device__ __forceinline__ float gelu_erf(float x) {
  return 0.5f * x * (1.0f + erff(x * 0.70710678118654752f));
}

__device__ __forceinline__ uint32_t pack_bf16x2(float a, float b) {
  __nv_bfloat162 v = __floats2bfloat162_rn(a, b);  // a -> low half, b -> high half
  return *reinterpret_cast<uint32_t*>(&v);
}

// hi/lo split of two values, packed: hi = bf16(x), lo = bf16(x - hi)
__device__ __forceinline__ void split_pack(float a, float b, uint32_t& hi, uint32_t& lo) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  const float2 hf = __bfloat1622float2(h);
  const __nv_bfloat162 l = __floats2bfloat162_rn(a - hf.x, b - hf.y);
  hi = *reinterpret_cast<const uint32_t*>(&h);
  lo = *reinterpret_cast<const uint32_t*>(&l);
}

// hi/lo split of two values in fp16 (11-bit significands: about 22 bits together):
// hi = fp16(x), lo = fp16(x - hi), packed.
__device__ __forceinline__ void split_pack_f16(float a, float b, uint32_t& hi, uint32_t& lo) {
  const __half2 h = __floats2half2_rn(a, b);
  const float2 hf = __half22float2(h);
  const __half2 l = __floats2half2_rn(a - hf.x, b - hf.y);
  hi = *reinterpret_cast<const uint32_t*>(&h);
  lo = *reinterpret_cast<const uint32_t*>(&l);
}

// 32 floats -> 32 bf16 packed in 4 x uint4
__device__ __forceinline__ void pack_bf16x32(const float (&v)[32], uint4 (&o)[4]) {
#pragma unroll
  for (int q = 0; q < 4; ++q)
    o[q] = make_uint4(pack_bf16x2(v[8 * q], v[8 * q + 1]), pack_bf16x2(v[8 * q + 2], v[8 * q + 3]),
                      pack_bf16x2(v[8 * q + 4], v[8 * q + 5]),
                      pack_bf16x2(v[8 * q + 6], v[8 * q + 7]));
}

// 32 floats -> hi and lo bf16, each packed in 4 x uint4
__device__ __forceinline__ void pack_hilo_x32(const float (&v)[32], uint4 (&h4)[4],
                                              uint4 (&l4)[4]) {
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    uint32_t h[4], l[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) split_pack(v[8 * q + 2 * k], v[8 * q + 2 * k + 1], h[k], l[k]);
    h4[q] = make_uint4(h[0], h[1], h[2], h[3]);
    l4[q] = make_uint4(l[0], l[1], l[2], l[3]);
  }
}

__device__ __forceinline__ void pack_hilo16_x32(const float (&v)[32], uint4 (&h4)[4],
                                                uint4 (&l4)[4]) {
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    uint32_t h[4], l[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) split_pack_f16(v[8 * q + 2 * k], v[8 * q + 2 * k + 1], h[k], l[k]);
    h4[q] = make_uint4(h[0], h[1], h[2], h[3]);
    l4[q] = make_uint4(l[0], l[1], l[2], l[3]);
  }
}

// 16 floats -> 4 x uint4 (fp32 bits)
__device__ __forceinline__ void pack_f32x16(const float* v, uint4 (&o)[4]) {
#pragma unroll
  for (int q = 0; q < 4; ++q)
    o[q] = make_uint4(__float_as_uint(v[4 * q]), __float_as_uint(v[4 * q + 1]),
                      __float_as_uint(v[4 * q + 2]), __float_as_uint(v[4 * q + 3]));
}

// General epilogue: v = acc * alpha [* colscale(c)] [* rowscale(r)] [+ bias(c)]
//   -> [sum-of-squares partial] -> [GELU] -> [+ residual (split 0)] -> store (f32/bf16/hi-lo)
// colscale / rowscale are read from vectors of ready factors (see launch_inv_norms).
// Sums of squares are written as partials, never accumulated atomically, so that results do
// not depend on scheduling: per (vector, tile, half-warp) one slot, ss_parts slots per vector.
// Split-K partial results go to out + split * split_stride and are reduced in a fixed order by
// the consumer.
// Host contract: csm, resm and (when vec_ok) om are contiguous in c (c0 == 1) with cdiv a
// multiple of 32, so every 32-column chunk maps to 32 consecutive elements; ss_seg is a
// multiple of the tile width.
struct EpiAffine {
  static constexpr int kWarps = 8;  // two per lane quarter: alternating 32-column chunks
  static constexpr int kStages = 0;  // default pipeline depth
  static constexpr int kStoreBufs = 1;
  int32_t kind = OUT_F32;
  void* out = nullptr;
  int64_t lo_off = 0;  // OUT_HILO: lo element offset from hi
  AffineMap om;
  float alpha = 1.f;
  const float* bias = nullptr;  // indexed by column
  const float* col_scale = nullptr;
  AffineMap csm;  // (b, 0, c) -> index
  const float* row_scale = nullptr;
  AffineMap rsm;  // (b, r, 0) -> index
  int32_t gelu = 0;
  int32_t res_kind = 0;  // 0 none, 1 f32, 2 bf16
  const void* res = nullptr;
  AffineMap resm;
  float* sumsq = nullptr;  // partial sums of v^2 over segments of ss_seg columns
  AffineMap ssm;           // (b, r, c / ss_seg) -> vector index
  int32_t ss_seg = 1 << 30;
  int32_t ss_parts = 2;    // slots per vector = 2 * ss_seg / tile width
  // Vectors in blocks of ss_block consecutive indices, stored part-major (see launch_inv_norms),
  // so that a warp's 32 rows write 32 consecutive floats of one part.
  int64_t ss_block = 1;
  int64_t split_stride = 0;
  int32_t vec_ok = 0;  // host: om.c0 == 1, cdiv % 32 == 0, 16-B aligned rows
  // OUT_F32 through TMA stores: the output is the 3-D view (col, row, batch) given to the
  // launcher (boxes of 32 x 32 fp32, 128-byte swizzled staging); rows / columns past the view
  // are clipped by the copy engine.
  int32_t tma_f32 = 0;
  int32_t tile_cols_ = 256;  // the tile width BN, set by the launcher

  // The residual rows of this warp's columns are pulled into L2 while the main loop runs.
  __device__ void prefetch(const GemmParams& p, const TileCoord& tc, int row, int half) const {
    if (res_kind == 0 || tc.split != 0) return;
    const int r = tc.tm * kBM + row;
    if (r >= p.M) return;
    const int esz = res_kind == 1 ? 4 : 2;
    for (int cc = 32 * half; cc < tile_cols_; cc += 64) {
      const int c0 = tc.tn * tile_cols_ + cc;
      if (c0 >= p.N) break;
      const char* base = static_cast<const char*>(res) + resm.at(tc.b, r, c0) * esz;
      for (int off = 0; off < 32 * esz; off += 32) prefetch_l2(base + off);  // per 32-B sector
    }
  }

  __device__ void operator()(const GemmParams& p, const TileCoord& tc, int row, uint32_t taddr,
                             int half, uint4* stage, const CUtensorMap* tmc) const {
    const int r = tc.tm * kBM + row;
    const bool rvalid = r < p.M;
    float rscale = alpha;
    if (row_scale != nullptr && rvalid) rscale *= row_scale[rsm.at(tc.b, r, 0)];
    float ss = 0.f;
    for (int cc = 32 * half; cc < tile_cols_; cc += 64) {
      float v[32];
      tmem_ld32(taddr + (uint32_t)cc, v);
      const int c0 = tc.tn * tile_cols_ + cc;
      if (c0 >= p.N) continue;  // uniform across the warp
      const int nv = min(32, p.N - c0);
#pragma unroll
      for (int e = 0; e < 32; ++e) v[e] *= rscale;
      // Residual rows read coalesced by the whole warp (before the invalid-row exit: every
      // lane takes part). Not on the TMA-store path, whose staging area may still be in use.
      const bool res_vec = res_kind != 0 && tc.split == 0 && vec_ok && !tma_f32 && nv == 32;
      float resv[32];
      if (res_vec) {
        const int64_t o = rvalid ? resm.at(tc.b, r, c0) : 0;
        if (res_kind == 1) {
          uint4 u[8];
          warp_load_rows<8>(stage, static_cast<const float*>(res) + o, rvalid, u);
#pragma unroll
          for (int q = 0; q < 8; ++q) {
            resv[4 * q] = __uint_as_float(u[q].x);
            resv[4 * q + 1] = __uint_as_float(u[q].y);
            resv[4 * q + 2] = __uint_as_float(u[q].z);
            resv[4 * q + 3] = __uint_as_float(u[q].w);
          }
        } else {
          uint4 u[4];
          warp_load_rows<4>(stage, static_cast<const __nv_bfloat16*>(res) + o, rvalid, u);
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const uint32_t w[4] = {u[q].x, u[q].y, u[q].z, u[q].w};
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w[k]));
              resv[8 * q + 2 * k] = f.x;
              resv[8 * q + 2 * k + 1] = f.y;
            }
          }
        }
      }
      if (!rvalid) {  // keep the warp-collective stores; the row itself is not written
        if (tma_f32)
          store32_tma(tc, row, c0, v, stage, tmc);
        else
          store32(p, tc.b, r, c0, v, tc.split, false, stage);
        continue;
      }
      if (col_scale != nullptr) {
        const float* cs = col_scale + csm.at(tc.b, 0, c0);
#pragma unroll
        for (int e = 0; e < 32; ++e)
          if (e < nv) v[e] *= cs[e];
      }
      if (bias != nullptr) {
#pragma unroll
        for (int e = 0; e < 32; ++e)
          if (e < nv) v[e] += bias[c0 + e];
      }
      if (sumsq != nullptr) {
#pragma unroll
        for (int e = 0; e < 32; ++e)
          if (e < nv) ss += v[e] * v[e];
      }
      if (gelu) {
#pragma unroll
        for (int e = 0; e < 32; ++e) v[e] = gelu_erf(v[e]);
      }
      if (res_vec) {
#pragma unroll
        for (int e = 0; e < 32; ++e) v[e] += resv[e];
      } else if (res_kind != 0 && tc.split == 0) {
        const int64_t o = resm.at(tc.b, r, c0);
        if (res_kind == 1) {
          const float* rp = static_cast<const float*>(res) + o;
#pragma unroll
          for (int e = 0; e < 32; ++e)
            if (e < nv) v[e] += rp[e];
        } else {
          const __nv_bfloat16* rp = static_cast<const __nv_bfloat16*>(res) + o;
#pragma unroll
          for (int e = 0; e < 32; ++e)
            if (e < nv) v[e] += __bfloat162float(rp[e]);
        }
      }
      if (tma_f32)
        store32_tma(tc, row, c0, v, stage, tmc);
      else
        store32(p, tc.b, r, c0, v, tc.split, rvalid, stage);
    }
    if (sumsq != nullptr && rvalid) {
      const int c_tile = tc.tn * tile_cols_;
      const int slot = ((c_tile % ss_seg) / tile_cols_) * 2 + half;
      const int64_t vec = ssm.at(tc.b, r, c_tile / ss_seg);
      sumsq[(vec / ss_block) * ss_parts * ss_block + slot * ss_block + vec % ss_block] = ss;
    }
  }

  // Warp-collective: this warp's 32 rows x 32 fp32 columns as one TMA box.
  __device__ __forceinline__ void store32_tma(const TileCoord& tc, int row, int c0,
                                              const float (&v)[32], uint4* stage,
                                              const CUtensorMap* tmc) const {
    const int lane = threadIdx.x & 31;
    if (lane == 0) bulk_wait_read();  // the previous box has left the staging area
    __syncwarp();
    uint4* my = stage + lane * 8;  // 128 B per row; 16-B chunk q lands at q ^ (row & 7)
#pragma unroll
    for (int q = 0; q < 8; ++q)
      my[q ^ (lane & 7)] = make_uint4(__float_as_uint(v[4 * q]), __float_as_uint(v[4 * q + 1]),
                                      __float_as_uint(v[4 * q + 2]), __float_as_uint(v[4 * q + 3]));
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) {
      tma_store_3d(tmc, stage, c0, tc.tm * kBM + row, tc.b);
      bulk_commit();
    }
  }

  // Warp-collective on the vector path (every lane calls it; invalid rows store nothing).
  __device__ __forceinline__ void store32(const GemmParams& p, int b, int r, int c0,
                                          const float (&v)[32], int split, bool rvalid,
                                          uint4* stage) const {
    const bool full = vec_ok && (c0 + 32 <= p.N);  // uniform across the warp
    const int64_t so = (int64_t)split * split_stride;
    if (full) {
      const int64_t o = rvalid ? om.at(b, r, c0) + so : 0;
      uint4 a4[4], b4[4];
      if (kind == OUT_F32) {
        float* dst = static_cast<float*>(out) + o;
        pack_f32x16(v, a4);
        pack_f32x16(v + 16, b4);
        warp_store64(stage, a4, dst, rvalid);
        warp_store64(stage, b4, dst + 16, rvalid);
      } else if (kind == OUT_HILO || kind == OUT_HILO16) {
        __nv_bfloat16* dst = static_cast<__nv_bfloat16*>(out) + o;
        if (kind == OUT_HILO)
          pack_hilo_x32(v, a4, b4);
        else
          pack_hilo16_x32(v, a4, b4);
        warp_store64(stage, a4, dst, rvalid);
        warp_store64(stage, b4, dst + lo_off, rvalid);
      } else {
        pack_bf16x32(v, a4);
        warp_store64(stage, a4, static_cast<__nv_bfloat16*>(out) + o, rvalid);
      }
      return;
    }
    if (!rvalid) return;
#pragma unroll
    for (int e = 0; e < 32; ++e) {
      const int c = c0 + e;
      if (c >= p.N) break;
      const int64_t o = om.at(b, r, c) + so;
      if (kind == OUT_F32) {
        static_cast<float*>(out)[o] = v[e];
      } else if (kind == OUT_BF16) {
        static_cast<__nv_bfloat16*>(out)[o] = __float2bfloat16_rn(v[e]);
      } else if (kind == OUT_HILO16) {
        const __half hh = __float2half_rn(v[e]);
        const __half ll = __float2half_rn(v[e] - __half2float(hh));
        reinterpret_cast<__half*>(out)[o] = hh;
        reinterpret_cast<__half*>(out)[o + lo_off] = ll;
      } else {
        __nv_bfloat16 h, l;
        split_hilo(v[e], h, l);
        static_cast<__nv_bfloat16*>(out)[o] = h;
        static_cast<__nv_bfloat16*>(out)[o + lo_off] = l;
      }
    }
  }
};

// Cache positions given as segments: position of token idx = start[k] + (idx - begin[k]) * step[k].
struct PosSegs {
  int32_t n = 0;
  int64_t begin[9] = {0};
  double start[8] = {0};
  double step[8] = {0};
};

__device__ __forceinline__ double seg_position(const PosSegs& s, int64_t idx) {
  int k = 0;
#pragma unroll 1
  while (k + 1 < s.n && idx >= s.begin[k + 1]) ++k;
  return s.start[k] + (double)(idx - s.begin[k]) * s.step[k];
}

// Key projection epilogue (cross-attention keys):
//   k~ = acc + b_K;  sumsq(token, head) += |k~|^2;  k = RoPE_c(k~, p_n)  -> hi/lo bf16.
// Columns are in "pair-chunk" order: within each 256-column tile, columns [0,128) hold the
// first elements of 128 RoPE pairs and [128,256) their partners, so a tile owns whole pairs.
// The angle p_n * omega_m is split as G_g * omega_m + i * omega_m + f * omega_m with
// delta = p_n - G_g in [0, kPosGrain), i = floor(delta) and f = delta - i: the first two
// rotations come from tables built per call in fp64 (coarse[g], fine[i]), the third (only for
// fractional positions, |f * omega_m| < 1) from Taylor series; the three are combined by the
// angle-addition formulas. Every rotation is thus accurate to fp32 rounding; forming
// delta * omega_m in fp32 instead would leave angle errors near 2e-6 rad at delta ~ 31. The
// per-token (g, delta) come from a table formed once per call in fp64 (gd[n] = (g, delta)), so
// the epilogue itself does no fp64 arithmetic.
constexpr int kPosGrain = 32;

// sin and cos of |x| <= 1 from their Taylor series about 0, through x^11 and x^12 (the first
// omitted terms are below 2e-10), by Horner's rule in fp32: no range reduction needed.
__device__ __forceinline__ void sincos_taylor(float x, float* s, float* c) {
  const float x2 = x * x;
  float ps = 1.f / 39916800.f;                  // 1/11!
  ps = fmaf(ps, -x2, 1.f / 362880.f);           // 1/9!
  ps = fmaf(ps, -x2, 1.f / 5040.f);             // 1/7!
  ps = fmaf(ps, -x2, 1.f / 120.f);              // 1/5!
  ps = fmaf(ps, -x2, 1.f / 6.f);                // 1/3!
  ps = fmaf(ps, -x2, 1.f);
  float pc = 1.f / 479001600.f;                 // 1/12!
  pc = fmaf(pc, -x2, 1.f / 3628800.f);          // 1/10!
  pc = fmaf(pc, -x2, 1.f / 40320.f);            // 1/8!
  pc = fmaf(pc, -x2, 1.f / 720.f);              // 1/6!
  pc = fmaf(pc, -x2, 1.f / 24.f);               // 1/4!
  pc = fmaf(pc, -x2, 0.5f);                     // 1/2!
  *s = x * ps;
  *c = fmaf(pc, -x2, 1.f);
}

// kFrac: some key positions are fractional (the sub-unit rotation is compiled in only then,
// so the integer-position kernel keeps its registers).
template <bool kFrac>
struct EpiRopeCT {
  // Element-wise heavy and MMA-light (K = 3d): four warps per lane quarter, each owning 32 of
  // the tile's 128 pairs, processed 16 at a time; a short pipeline suffices.
  static constexpr int kWarps = 16;
  static constexpr int kParts = kWarps / 4;
  static constexpr int kPairsPerPart = 128 / kParts;  // RoPE pairs of a tile per warp
  static constexpr int kStages = 3;
  static constexpr int kStoreBufs = 1;  // 4 KB TMA-store staging buffers per warp
  __nv_bfloat16* out = nullptr;  // [H][n][N][2D]: hi at [0, D), lo at [D, 2D) (via the TMA view)
  float* sumsq = nullptr;        // [H][n][kParts * D / 256][N] partial sums of |k~|^2 (part-major)
  const float* bias = nullptr;   // [n*D], pair-chunk order
  const float2* coarse = nullptr;  // [G][D/2]: (cos, sin)(G_g * omega_m)
  // [D/2][kPosGrain]: (cos, sin)(i * omega_m), i fastest: the 32 consecutive tokens of a warp
  // read 32 neighbouring entries of one pair's row (one 256-byte span per load)
  const float2* fine = nullptr;
  const float* omega = nullptr;    // [D/2] fp32
  const float2* gd = nullptr;      // [Ntok]: (coarse index g as float, delta)
  int32_t fp16 = 0;                // hi / lo as fp16 (about 22 bits) instead of bf16
  int32_t D = 0, nheads = 0, ncoarse = 0;
  int64_t Ntok = 0;
  int32_t tile_cols_ = 256;  // must be 256: a tile holds 128 whole RoPE pairs

  __device__ void prefetch(const GemmParams&, const TileCoord&, int, int) const {}

  __device__ void operator()(const GemmParams& p, const TileCoord& tc, int row, uint32_t taddr,
                             int half, uint4* stage, const CUtensorMap* tmc) const {
    const int r = tc.tm * kBM + row;
    const bool rvalid = r < p.M;
    const int lane = threadIdx.x & 31;
    const int row0 = tc.tm * kBM + row - lane;  // first token row of this warp
    const int c_tile = tc.tn * 256;
    const int head = c_tile / D;
    const int f_tile = c_tile % D;       // column of this tile inside the head (pair-chunk order)
    const int m_base = (f_tile / 256) * 128;  // first pair index of this tile
    const float2 gdr = rvalid ? gd[r] : make_float2(0.f, 0.f);
    const int g = max(0, min((int)gdr.x, ncoarse - 1));
    const int di = max(0, min((int)gdr.y, kPosGrain - 1));
    const float frac = gdr.y - (float)di;  // exact; 0 for integer positions
    const bool any_frac = kFrac && __any_sync(0xffffffffu, frac != 0.f);
    float ss = 0.f;
    // Part p owns pairs [p, p + 1) * kPairsPerPart of the tile, 16 at a time. With kStoreBufs = 2 the
    // staging area holds two 4 KB buffers used alternately, so one iteration's TMA stores can
    // still be reading while the next fills the other buffer.
    for (int it = 0; it < kPairsPerPart / 16; ++it) {
      const int u = kPairsPerPart * half + 16 * it;
      // tables first: their latency overlaps the TMEM loads
      const float4* crow = reinterpret_cast<const float4*>(coarse + (int64_t)g * (D / 2) + m_base + u);
      const float2* fcol = fine + (int64_t)(m_base + u) * kPosGrain + di;
      const float4* om4 = reinterpret_cast<const float4*>(omega + m_base + u);
      const float4* ba4 = reinterpret_cast<const float4*>(bias + c_tile + u);
      const float4* bb4 = reinterpret_cast<const float4*>(bias + c_tile + 128 + u);
      float4 w[4], xa[4], xb[4], cs[8];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        w[q] = any_frac ? om4[q] : make_float4(0.f, 0.f, 0.f, 0.f);
        xa[q] = ba4[q];
        xb[q] = bb4[q];
        cs[2 * q] = crow[2 * q];
        cs[2 * q + 1] = crow[2 * q + 1];
      }
      float a[16], bb[16];
      tmem_ld16x2(taddr + (uint32_t)u, taddr + (uint32_t)(128 + u), a, bb);
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float ws[4] = {w[q].x, w[q].y, w[q].z, w[q].w};
        const float bas[4] = {xa[q].x, xa[q].y, xa[q].z, xa[q].w};
        const float bbs[4] = {xb[q].x, xb[q].y, xb[q].z, xb[q].w};
        const float cc[4] = {cs[2 * q].x, cs[2 * q].z, cs[2 * q + 1].x, cs[2 * q + 1].z};
        const float sc[4] = {cs[2 * q].y, cs[2 * q].w, cs[2 * q + 1].y, cs[2 * q + 1].w};
        float cf[4], sf[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const float2 f = fcol[(4 * q + k) * kPosGrain];  // small table: L1-resident
          cf[k] = f.x;
          sf[k] = f.y;
        }
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const int e = 4 * q + k;
          const float x = a[e] + bas[k];
          const float y = bb[e] + bbs[k];
          ss += x * x + y * y;
          float cw = cc[k] * cf[k] - sc[k] * sf[k];  // cos(G w + i w)
          float sw = sc[k] * cf[k] + cc[k] * sf[k];  // sin(G w + i w)
          if (any_frac) {  // + f w, |f w| < 1
            float s3, c3;
            sincos_taylor(frac * ws[k], &s3, &c3);
            const float c2 = cw * c3 - sw * s3;
            sw = sw * c3 + cw * s3;
            cw = c2;
          }
          a[e] = x * cw - y * sw;
          bb[e] = x * sw + y * cw;
        }
      }
      // Four boxes of 32 rows x 16 bf16 (hi a, lo a, hi b, lo b), 1 KB each, stored by TMA;
      // rows past N are clipped by the copy engine.
      uint4* box = stage + (kStoreBufs == 2 ? (it & 1) * 256 : 0);
      if (lane == 0) {
        if (kStoreBufs == 2)
          bulk_wait_read1();
        else
          bulk_wait_read();
      }
      __syncwarp();
      uint4* bl = box + lane * 2;
#pragma unroll
      for (int q = 0; q < 2; ++q) {
        uint32_t h[4], l[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          if (fp16)
            split_pack_f16(a[8 * q + 2 * k], a[8 * q + 2 * k + 1], h[k], l[k]);
          else
            split_pack(a[8 * q + 2 * k], a[8 * q + 2 * k + 1], h[k], l[k]);
        }
        bl[q] = make_uint4(h[0], h[1], h[2], h[3]);
        bl[64 + q] = make_uint4(l[0], l[1], l[2], l[3]);
#pragma unroll
        for (int k = 0; k < 4; ++k)
          if (fp16)
            split_pack_f16(bb[8 * q + 2 * k], bb[8 * q + 2 * k + 1], h[k], l[k]);
          else
            split_pack(bb[8 * q + 2 * k], bb[8 * q + 2 * k + 1], h[k], l[k]);
        bl[128 + q] = make_uint4(h[0], h[1], h[2], h[3]);
        bl[192 + q] = make_uint4(l[0], l[1], l[2], l[3]);
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) {
        const int z = tc.b * nheads + head;
        const int x = f_tile + u;
        tma_store_3d(tmc, box, x, row0, z);
        tma_store_3d(tmc, box + 64, D + x, row0, z);
        tma_store_3d(tmc, box + 128, x + 128, row0, z);
        tma_store_3d(tmc, box + 192, D + x + 128, row0, z);
        bulk_commit();
      }
    }
    if (rvalid) {
      const int parts = kParts * (D / 256);
      sumsq[((int64_t)(tc.b * nheads + head) * parts + (f_tile / 256) * kParts + half) * Ntok + r] =
          ss;
    }
  }
};

// Output heads: columns [0, d) = Z_out W_key, re-rotated by the base RoPE at the output
// position of latent j; columns [d, 2d) = Z_out W_val. Rows r = h * t + j. bf16 stores into
// the caller's C_k / C_v with element strides (st, sh). rot[j][m] = (cos, sin)(p_j * omega_m),
// a table formed once per call with the angle reduced modulo 2 pi in fp64.
// Folded key path (no compactor RoPE): |k~_n|^2 = x~_n G x~_n^T with G = W~ W~^T. The GEMM
// gives Y = x~ G (rows = tokens of one KV-head, columns = the Kp entries of one cross head);
// the epilogue dots each 32-column chunk of Y with the same columns of x~ (hi + lo, read back
// from global memory) and stores the partial, part-major: part[(b * Kp/32 + chunk) * Ntok + n].
struct EpiQuad {
  static constexpr int kWarps = 8;   // two per lane quarter: alternating 32-column chunks
  static constexpr int kStages = 0;
  static constexpr int kStoreBufs = 1;
  float* part = nullptr;
  const __nv_bfloat16* xt = nullptr;  // x~ rows [hi | lo], pitch 2 Kp, of the group's first KV-head
  int64_t Ntok = 0;
  int32_t Kp = 0;
  int32_t tile_cols_ = 256;

  __device__ void prefetch(const GemmParams&, const TileCoord&, int, int) const {}

  __device__ void operator()(const GemmParams& p, const TileCoord& tc, int row, uint32_t taddr,
                             int half, uint4*, const CUtensorMap*) const {
    const int r = tc.tm * kBM + row;
    const bool rvalid = r < p.M;
    const int parts = Kp / 32;
    const __nv_bfloat16* xr =
        xt + ((int64_t)(tc.b / p.bdiv) * Ntok + (rvalid ? r : 0)) * 2 * Kp;
    for (int cc = 32 * half; cc < tile_cols_; cc += 64) {
      float v[32];
      tmem_ld32(taddr + (uint32_t)cc, v);  // warp-collective: before any per-lane exit
      const int c0 = tc.tn * tile_cols_ + cc;
      if (c0 >= p.N || !rvalid) continue;
      const uint4* hp = reinterpret_cast<const uint4*>(xr + c0);
      const uint4* lp = reinterpret_cast<const uint4*>(xr + Kp + c0);
      float acc = 0.f;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const uint4 hq = hp[q], lq = lp[q];
        const uint32_t hw[4] = {hq.x, hq.y, hq.z, hq.w}, lw[4] = {lq.x, lq.y, lq.z, lq.w};
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const float2 h2 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&hw[k]));
          const float2 l2 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&lw[k]));
          acc = fmaf(v[8 * q + 2 * k], h2.x + l2.x, acc);
          acc = fmaf(v[8 * q + 2 * k + 1], h2.y + l2.y, acc);
        }
      }
      part[((int64_t)tc.b * parts + c0 / 32) * Ntok + r] = acc;
    }
  }
};

struct EpiHeads {
  static constexpr int kWarps = 8;
  static constexpr int kStages = 0;
  static constexpr int kStoreBufs = 1;
  __nv_bfloat16* ck = nullptr;
  __nv_bfloat16* cv = nullptr;
  int64_t st = 0, sh = 0;  // element strides of [t, H, d]; d is contiguous, rows 16-B aligned
  int32_t t = 0, d = 0;
  const float2* rot = nullptr;  // [t][d/2]
  int32_t tile_cols_ = 256;

  __device__ void prefetch(const GemmParams&, const TileCoord&, int, int) const {}

  __device__ void operator()(const GemmParams& p, const TileCoord& tc, int row, uint32_t taddr,
                             int half, uint4* stage, const CUtensorMap*) const {
    const int r = tc.tm * kBM + row;
    const bool rvalid = r < p.M;
    const int h = rvalid ? r / t : 0, j = rvalid ? r % t : 0;
    const int c_tile = tc.tn * tile_cols_;
    const float2* rrow = rot + (int64_t)j * (d / 2);
    const int64_t obase = (int64_t)j * st + (int64_t)h * sh;
    const int hd = d / 2;
    for (int cc = 32 * half; cc < tile_cols_; cc += 64) {
      const int c0 = c_tile + cc;
      if (c0 >= p.N) break;
      if (c0 < d) {
        // key columns: process pairs (m, m + d/2) when visiting the first half
        if (c0 >= hd) continue;
        float a[32], b[32];
        tmem_ld32(taddr + (uint32_t)cc, a);
        tmem_ld32(taddr + (uint32_t)(cc + hd), b);
#pragma unroll
        for (int e = 0; e < 32; ++e) {
          const float2 cs = rrow[c0 + e];
          const float cw = cs.x, sw = cs.y;
          const float x = a[e], y = b[e];
          a[e] = x * cw - y * sw;
          b[e] = x * sw + y * cw;
        }
        uint4 o4[4];
        pack_bf16x32(a, o4);
        warp_store64(stage, o4, ck + obase + c0, rvalid);
        pack_bf16x32(b, o4);
        warp_store64(stage, o4, ck + obase + c0 + hd, rvalid);
      } else {
        float v[32];
        tmem_ld32(taddr + (uint32_t)cc, v);
        uint4 o4[4];
        pack_bf16x32(v, o4);
        warp_store64(stage, o4, cv + obase + (c0 - d), rvalid);
      }
    }
  }
};

}  // namespace still
