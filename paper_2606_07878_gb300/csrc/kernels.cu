// Memory-bound kernels of the compactor path: RoPE-fix strip, RoPE tables, query rotation,
// softmax, hi/lo conversion, RMSNorm, weight re-layout.
#include <algorithm>
#include <type_traits>

#include "kernels.cuh"

namespace still {

namespace {

constexpr double kTwoPi = 6.283185307179586;
constexpr double kInvTwoPi = 0.15915494309189535;
constexpr float kLog2e = 1.4426950408889634f;

// angle reduced to [-pi, pi] in fp64, then sin/cos in fp32 (|error| ~1e-7)
__device__ __forceinline__ void sincos_reduced(double ang, float* s, float* c) {
  ang -= kTwoPi * rint(ang * kInvTwoPi);
  sincosf((float)ang, s, c);
}

constexpr int kStripTok = 32;

__device__ __forceinline__ int64_t kv_offset(const KVSource& src, int64_t n, int h, bool& second) {
  second = n >= src.n_split;
  return second ? (n - src.n_split) * src.sN2 + (int64_t)h * src.sH2
                : n * src.sN + (int64_t)h * src.sH;
}

// Eight consecutive bf16 of a K / V row as fp32 (one 16-byte load when aligned).
__device__ __forceinline__ void load8(const __nv_bfloat16* p, bool vec, float (&v)[8]) {
  if (vec) {
    const uint4 u = *reinterpret_cast<const uint4*>(p);
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w[k]));
      v[2 * k] = f.x;
      v[2 * k + 1] = f.y;
    }
  } else {
#pragma unroll
    for (int e = 0; e < 8; ++e) v[e] = __bfloat162float(p[e]);
  }
}

// One CTA = 32 tokens x all KV-heads. The base-RoPE angles of the tile's tokens are formed
// once (fp64, reduced mod 2 pi) and reused by every KV-head. Keys: inverse rotation of pairs
// (m, m + d/2) (Sec. 2.2, RoPE-fix); values pass through. Writes X (bf16 hi | key lo) and XT
// (fp16 hi for all 2d features, fp16 lo for the key half; the value half's lo is exactly zero
// and is never read). Rows are moved in 16-byte pieces; the transpose for XT goes through
// shared memory with an odd word pitch (conflict-free column reads).
// Kp > 0 writes X in the layout of the folded key path instead: rows of 2 Kp elements,
// [x~ hi | x~ lo] with x~ = [unRoPE(K) | V | 1 | 0 ...] (Kp >= 2d + 1, a multiple of 64).
__global__ void __launch_bounds__(256) strip_kernel(KVSource src, int64_t N, int H, int d,
                                                    PosSegs segs, const double* __restrict__ omega,
                                                    int rope_fix, int vec, int x16, int Kp,
                                                    __nv_bfloat16* __restrict__ X,
                                                    __half* __restrict__ XT, int64_t Np,
                                                    float2* __restrict__ gd, double pmin, int G) {
  extern __shared__ __align__(16) uint8_t sm[];
  __shared__ double tpos[kStripTok];
  const int half = d / 2;
  const int ph = 2 * d + 2, pl = d + 2;  // pitches (halves) of the transpose tiles
  float2* rot = reinterpret_cast<float2*>(sm);  // [kStripTok][half]: (cos, sin)
  __half* thi = reinterpret_cast<__half*>(rot + kStripTok * half);  // [kStripTok][ph]
  __half* tlo = thi + kStripTok * ph;                                 // [kStripTok][pl]
  const int64_t n0 = (int64_t)blockIdx.x * kStripTok;
  if (threadIdx.x < kStripTok) {
    // token position (fp64) once per token; also the compactor-RoPE coarse index and residual
    const int64_t n = n0 + threadIdx.x;
    const double pos = n < N ? seg_position(segs, n) : pmin;
    tpos[threadIdx.x] = pos;
    if (n < N) {
      int g = (int)floor((pos - pmin) / (double)kPosGrain);
      g = max(0, min(g, G - 1));
      gd[n] = make_float2((float)g, (float)(pos - (pmin + (double)g * kPosGrain)));
    }
  }
  __syncthreads();
  for (int it = threadIdx.x; it < kStripTok * half; it += blockDim.x) {
    const int tok = it / half, m = it % half;
    const int64_t n = n0 + tok;
    float sw = 0.f, cw = 1.f;
    if (rope_fix && n < N) sincos_reduced(tpos[tok] * omega[m], &sw, &cw);
    rot[it] = make_float2(cw, sw);
  }
  __syncthreads();
  const int d3 = Kp > 0 ? 2 * Kp : 3 * d;  // X row pitch
  const int lo0 = Kp > 0 ? Kp : 2 * d;     // column of the key lo part
  const int64_t ld = 2 * Np;
  const int kg = half / 8, vg = d / 8;  // 8-element groups per token: key pairs, values
  for (int h = 0; h < H; ++h) {
    // keys: group g holds pairs m = 8g .. 8g + 7
    for (int it = threadIdx.x; it < kStripTok * kg; it += blockDim.x) {
      const int tok = it / kg, m0 = 8 * (it % kg);
      const int64_t n = n0 + tok;
      float a[8], b[8];
      if (n < N) {
        bool second;
        const int64_t off = kv_offset(src, n, h, second);
        const __nv_bfloat16* kr = (second ? src.K2 : src.K) + off;
        float ka[8], kb[8];
        load8(kr + m0, vec, ka);
        load8(kr + half + m0, vec, kb);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const float2 cs = rot[tok * half + m0 + e];
          a[e] = ka[e] * cs.x + kb[e] * cs.y;
          b[e] = -ka[e] * cs.y + kb[e] * cs.x;
        }
        uint32_t ah[4], al[4], bh[4], bl[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          if (x16) {
            split_pack_f16(a[2 * k], a[2 * k + 1], ah[k], al[k]);
            split_pack_f16(b[2 * k], b[2 * k + 1], bh[k], bl[k]);
          } else {
            split_pack(a[2 * k], a[2 * k + 1], ah[k], al[k]);
            split_pack(b[2 * k], b[2 * k + 1], bh[k], bl[k]);
          }
        }
        __nv_bfloat16* xr = X + ((int64_t)h * N + n) * d3;
        if (vec) {
          *reinterpret_cast<uint4*>(xr + m0) = make_uint4(ah[0], ah[1], ah[2], ah[3]);
          *reinterpret_cast<uint4*>(xr + half + m0) = make_uint4(bh[0], bh[1], bh[2], bh[3]);
          *reinterpret_cast<uint4*>(xr + lo0 + m0) = make_uint4(al[0], al[1], al[2], al[3]);
          *reinterpret_cast<uint4*>(xr + lo0 + half + m0) = make_uint4(bl[0], bl[1], bl[2], bl[3]);
        } else {
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            reinterpret_cast<uint32_t*>(xr + m0)[k] = ah[k];
            reinterpret_cast<uint32_t*>(xr + half + m0)[k] = bh[k];
            reinterpret_cast<uint32_t*>(xr + lo0 + m0)[k] = al[k];
            reinterpret_cast<uint32_t*>(xr + lo0 + half + m0)[k] = bl[k];
          }
        }
      } else {
#pragma unroll
        for (int e = 0; e < 8; ++e) a[e] = b[e] = 0.f;
      }
      __half* hr = thi + tok * ph;
      __half* lr = tlo + tok * pl;
#pragma unroll
      for (int e = 0; e < 8; e += 2) {
        const __half2 ha = __floats2half2_rn(a[e], a[e + 1]);
        const __half2 hb = __floats2half2_rn(b[e], b[e + 1]);
        const float2 fa = __half22float2(ha), fb = __half22float2(hb);
        *reinterpret_cast<__half2*>(hr + m0 + e) = ha;
        *reinterpret_cast<__half2*>(hr + half + m0 + e) = hb;
        *reinterpret_cast<__half2*>(lr + m0 + e) = __floats2half2_rn(a[e] - fa.x, a[e + 1] - fa.y);
        *reinterpret_cast<__half2*>(lr + half + m0 + e) =
            __floats2half2_rn(b[e] - fb.x, b[e + 1] - fb.y);
      }
    }
    // values: group g holds features 8g .. 8g + 7 (bf16 values are exact in fp16)
    for (int it = threadIdx.x; it < kStripTok * vg; it += blockDim.x) {
      const int tok = it / vg, f0 = 8 * (it % vg);
      const int64_t n = n0 + tok;
      float v[8];
      if (n < N) {
        bool second;
        const int64_t off = kv_offset(src, n, h, second);
        const __nv_bfloat16* vr = (second ? src.V2 : src.V) + off + f0;
        load8(vr, vec, v);
        __nv_bfloat16* xr = X + ((int64_t)h * N + n) * d3 + d + f0;
        if (x16) {  // values in fp16 (bf16 values in the fp16 range convert exactly)
#pragma unroll
          for (int e = 0; e < 8; ++e) reinterpret_cast<__half*>(xr)[e] = __float2half_rn(v[e]);
        } else if (vec) {
          *reinterpret_cast<uint4*>(xr) = *reinterpret_cast<const uint4*>(vr);
        } else {
#pragma unroll
          for (int e = 0; e < 8; ++e) xr[e] = vr[e];
        }
      } else {
#pragma unroll
        for (int e = 0; e < 8; ++e) v[e] = 0.f;
      }
      __half* hr = thi + tok * ph + d + f0;
#pragma unroll
      for (int e = 0; e < 8; e += 2)
        *reinterpret_cast<__half2*>(hr + e) = __floats2half2_rn(v[e], v[e + 1]);
    }
    if (Kp > 0) {  // folded layout: [.. | 1 | 0 ...] after the values, zeros after the key lo
      const int nc = (Kp - 2 * d) / 8, nz = (Kp - d) / 8;  // 16-byte groups per token
      for (int it = threadIdx.x; it < kStripTok * (nc + nz); it += blockDim.x) {
        const int tok = it / (nc + nz), q = it % (nc + nz);
        const int64_t n = n0 + tok;
        if (n >= N) continue;
        __nv_bfloat16* xr = X + ((int64_t)h * N + n) * d3;
        uint4 val = make_uint4(0, 0, 0, 0);
        if (q == 0) val.x = x16 ? 0x3C00u : 0x3F80u;  // 1.0 in the first element (fp16 / bf16)
        *reinterpret_cast<uint4*>(xr + (q < nc ? 2 * d + 8 * q : Kp + d + 8 * (q - nc))) = val;
      }
    }
    __syncthreads();
    // XT: feature rows of 32 tokens, 8 tokens (16 B) per store; hi rows [0, 2d), lo rows [0, d)
    constexpr int kTg = kStripTok / 8;
    const int nhi = 2 * d * kTg;
    for (int it = threadIdx.x; it < 3 * d * kTg; it += blockDim.x) {
      const bool lo = it >= nhi;
      const int q = lo ? it - nhi : it;
      const int f = q / kTg, t0 = 8 * (q % kTg);
      const __half* col = lo ? tlo + f : thi + f;
      const int pitch = lo ? pl : ph;
      uint32_t w[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const __half x0 = col[(t0 + 2 * k) * pitch], x1 = col[(t0 + 2 * k + 1) * pitch];
        const __half2 pr = __halves2half2(x0, x1);
        w[k] = *reinterpret_cast<const uint32_t*>(&pr);
      }
      __half* dst = XT + ((int64_t)h * 2 * d + f) * ld + (lo ? Np : 0) + n0 + t0;
      *reinterpret_cast<uint4*>(dst) = make_uint4(w[0], w[1], w[2], w[3]);
    }
    __syncthreads();
  }
}

// Rows [0, G): coarse[g][m] = (cos, sin)((pmin + g * kPosGrain) * w_m); then, in the next
// kPosGrain * D/2 entries, fine[m][i] = (cos, sin)(i * w_m). Angles formed and reduced in fp64.
__global__ void rope_tables_kernel(float2* coarse, float* omega, int G, int D, double pmin,
                                   const double* __restrict__ omega_c) {
  const int half = D / 2;
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (int64_t)(G + kPosGrain) * half) return;
  const int g = (int)(idx / half);
  const int64_t f = idx - (int64_t)G * half;  // index into the fine table when >= 0
  const int m = g < G ? (int)(idx % half) : (int)(f / kPosGrain);
  const double w = omega_c[m];
  float s, c;
  const double ang = g < G ? (pmin + (double)g * kPosGrain) * w : (double)(f % kPosGrain) * w;
  sincos_reduced(ang, &s, &c);
  coarse[idx] = make_float2(c, s);
  if (g == 0) omega[m] = (float)w;
}

// rot[j][m] = (cos, sin)(p_j * omega[m]), p_j = pstart + j * pstep, angle reduced in fp64;
// (1, 0) when use_rope is 0.
__global__ void heads_rot_kernel(float2* rot, int t, int hd, double pstart, double pstep,
                                 const double* __restrict__ omega, int use_rope) {
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (int64_t)t * hd) return;
  const int j = (int)(idx / hd), m = (int)(idx % hd);
  float s = 0.f, c = 1.f;
  if (use_rope) sincos_reduced((pstart + (double)j * pstep) * omega[m], &s, &c);
  rot[idx] = make_float2(c, s);
}

// Thread = (latent j, 4 consecutive pairs m); the angles are formed once and reused for every
// batch. Columns are in pair-chunk order: pair m sits at f1 = (m / 128) * 256 + m % 128 and its
// partner at f1 + 128, so four consecutive pairs are four consecutive columns.
__global__ void q_rope_kernel(const float* __restrict__ qhat, int t_max, int b0, int nb, int t,
                              int D, double qstart, double qstep, const double* omega_c,
                              int use_rope, __nv_bfloat16* __restrict__ qhl, int fp16,
                              float qscale) {
  const int half = D / 2, q4 = half / 4;
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (int64_t)t * q4) return;
  const int j = (int)(idx / q4), m0 = 4 * (int)(idx % q4);
  float s[4], c[4];
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    s[e] = 0.f;
    c[e] = 1.f;
    if (use_rope) sincos_reduced((qstart + (double)j * qstep) * omega_c[m0 + e], &s[e], &c[e]);
  }
  const int f1 = (m0 / 128) * 256 + (m0 % 128), f2 = f1 + 128;
  for (int bb = 0; bb < nb; ++bb) {
    const float* q = qhat + ((int64_t)(b0 + bb) * t_max + j) * D;
    const float4 x4 = *reinterpret_cast<const float4*>(q + f1);
    const float4 y4 = *reinterpret_cast<const float4*>(q + f2);
    const float x[4] = {x4.x, x4.y, x4.z, x4.w}, y[4] = {y4.x, y4.y, y4.z, y4.w};
    float a[4], b[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      a[e] = x[e] * c[e] - y[e] * s[e];
      b[e] = x[e] * s[e] + y[e] * c[e];
    }
    uint32_t ah[2], al[2], bh[2], bl[2];
    if (fp16) {
      split_pack_f16(a[0] * qscale, a[1] * qscale, ah[0], al[0]);
      split_pack_f16(a[2] * qscale, a[3] * qscale, ah[1], al[1]);
      split_pack_f16(b[0] * qscale, b[1] * qscale, bh[0], bl[0]);
      split_pack_f16(b[2] * qscale, b[3] * qscale, bh[1], bl[1]);
    } else {
      split_pack(a[0], a[1], ah[0], al[0]);
      split_pack(a[2], a[3], ah[1], al[1]);
      split_pack(b[0], b[1], bh[0], bl[0]);
      split_pack(b[2], b[3], bh[1], bl[1]);
    }
    __nv_bfloat16* o = qhl + ((int64_t)bb * t + j) * 2 * D;
    *reinterpret_cast<uint2*>(o + f1) = make_uint2(ah[0], ah[1]);
    *reinterpret_cast<uint2*>(o + D + f1) = make_uint2(al[0], al[1]);
    *reinterpret_cast<uint2*>(o + f2) = make_uint2(bh[0], bh[1]);
    *reinterpret_cast<uint2*>(o + D + f2) = make_uint2(bl[0], bl[1]);
  }
}

__device__ __forceinline__ void ml_combine(float& m, float& l, float m2, float l2) {
  if (m2 == -INFINITY) return;
  if (m == -INFINITY) {
    m = m2;
    l = l2;
    return;
  }
  const float M = fmaxf(m, m2);
  l = l * exp2f((m - M) * kLog2e) + l2 * exp2f((m2 - M) * kLog2e);
  m = M;
}

template <typename OutT>
__global__ void __launch_bounds__(256) softmax_kernel(const float* __restrict__ S, int64_t ncols,
                                                      int64_t ldS, OutT* __restrict__ P,
                                                      int64_t ldP) {
  __shared__ float red_m[8], red_l[8];
  const int64_t row = blockIdx.x;
  const float* s = S + row * ldS;
  float m = -INFINITY, l = 0.f;
  for (int64_t c = threadIdx.x; c < ncols; c += blockDim.x) {
    const float x = s[c];
    if (x > m) {
      l = (m == -INFINITY ? 0.f : l * exp2f((m - x) * kLog2e)) + 1.f;
      m = x;
    } else {
      l += exp2f((x - m) * kLog2e);
    }
  }
  for (int o = 16; o > 0; o >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
    const float l2 = __shfl_xor_sync(0xffffffffu, l, o);
    ml_combine(m, l, m2, l2);
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) {
    red_m[warp] = m;
    red_l[warp] = l;
  }
  __syncthreads();
  if (warp == 0) {
    m = lane < 8 ? red_m[lane] : -INFINITY;
    l = lane < 8 ? red_l[lane] : 0.f;
    for (int o = 4; o > 0; o >>= 1) {
      const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
      const float l2 = __shfl_xor_sync(0xffffffffu, l, o);
      ml_combine(m, l, m2, l2);
    }
    if (lane == 0) {
      red_m[0] = m;
      red_l[0] = l;
    }
  }
  __syncthreads();
  const float M = red_m[0], inv = 1.f / red_l[0];
  OutT* p = P + row * ldP;
  for (int64_t c = threadIdx.x; c < ldP; c += blockDim.x) {
    const float v = c < ncols ? exp2f((s[c] - M) * kLog2e) * inv : 0.f;
    if constexpr (sizeof(OutT) == 2 && std::is_same<OutT, __half>::value)
      p[c] = __float2half_rn(v);
    else
      p[c] = __float2bfloat16_rn(v);
  }
}

// Row softmax with the row held in registers: 256 threads, PER columns each (float4 groups).
// HILO: the row is written as hi at [0, ldP) and lo = OutT(p - hi) at [ldP, 2 ldP) of a row of
// pitch 2 ldP (bf16 or fp16 parts).
template <typename OutT, int PER, bool HILO = false>
__global__ void __launch_bounds__(256) softmax_reg_kernel(const float* __restrict__ S,
                                                          int64_t ncols, int64_t ldS,
                                                          OutT* __restrict__ P, int64_t ldP) {
  __shared__ float red[8];
  const int64_t row = blockIdx.x;
  const float* s = S + row * ldS;
  constexpr int G = PER / 4;
  float v[PER];
  float m = -INFINITY;
#pragma unroll
  for (int i = 0; i < G; ++i) {
    const int64_t c = (int64_t)(i * 256 + threadIdx.x) * 4;
    float4 x = make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
    if (c + 3 < ncols) {
      x = *reinterpret_cast<const float4*>(s + c);
    } else if (c < ncols) {
      x.x = s[c];
      if (c + 1 < ncols) x.y = s[c + 1];
      if (c + 2 < ncols) x.z = s[c + 2];
    }
    v[4 * i] = x.x;
    v[4 * i + 1] = x.y;
    v[4 * i + 2] = x.z;
    v[4 * i + 3] = x.w;
    m = fmaxf(m, fmaxf(fmaxf(x.x, x.y), fmaxf(x.z, x.w)));
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
  if (lane == 0) red[warp] = m;
  __syncthreads();
  m = red[0];
#pragma unroll
  for (int w = 1; w < 8; ++w) m = fmaxf(m, red[w]);
  __syncthreads();
  float l = 0.f;
#pragma unroll
  for (int k = 0; k < PER; ++k) {
    v[k] = exp2f((v[k] - m) * kLog2e);  // exp(-inf) = 0 for padding
    l += v[k];
  }
  for (int o = 16; o > 0; o >>= 1) l += __shfl_xor_sync(0xffffffffu, l, o);
  if (lane == 0) red[warp] = l;
  __syncthreads();
  l = 0.f;
#pragma unroll
  for (int w = 0; w < 8; ++w) l += red[w];
  const float inv = 1.f / l;
  OutT* prow = P + row * (HILO ? 2 * ldP : ldP);
#pragma unroll
  for (int i = 0; i < G; ++i) {
    const int64_t c = (int64_t)(i * 256 + threadIdx.x) * 4;
    if (c < ldP) {
      OutT o4[4], l4[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const float y = v[4 * i + k] * inv;
        if constexpr (std::is_same<OutT, __half>::value) {
          o4[k] = __float2half_rn(y);
          if constexpr (HILO) l4[k] = __float2half_rn(y - __half2float(o4[k]));
        } else {
          o4[k] = __float2bfloat16_rn(y);
          if constexpr (HILO) l4[k] = __float2bfloat16_rn(y - __bfloat162float(o4[k]));
        }
      }
      *reinterpret_cast<uint2*>(prow + c) = *reinterpret_cast<const uint2*>(o4);
      if constexpr (HILO) *reinterpret_cast<uint2*>(prow + ldP + c) = *reinterpret_cast<const uint2*>(l4);
    }
  }
}

// Failure-detection self-test: waits on an mbarrier that nothing arrives on, with a short
// bound. The wait expires, the kernel records DEV_WAIT_TIMEOUT in the error record and returns.
__global__ void wait_timeout_selftest_kernel(int* err, unsigned long long limit_ns) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    const uint32_t a = smem_u32(&bar);
    const uint64_t t0 = globaltimer_ns();
    bool done = false;
    while (!done && globaltimer_ns() - t0 < limit_ns) done = mbar_try_wait(a, 0) != 0;
    if (!done) dev_set_error(err, DEV_WAIT_TIMEOUT, 900);
  }
}

__global__ void omega_kernel(double* out, int half, int width, double base) {
  const int m = blockIdx.x * blockDim.x + threadIdx.x;
  if (m < half) out[m] = pow(base, -2.0 * m / width);
}

// Key-split merge of the fused cross-attention. Split s holds, per row, the unnormalised
// O_s = sum_k 2^(v_k - m_s) X_k and l_s = sum_k 2^(v_k - m_s) (v, m in log2 units). With
// M = max_s m_s:  O = sum_s 2^(m_s - M) O_s / sum_s 2^(m_s - M) l_s, summed in split order.
// One warp per row; each lane owns 4-column groups (16-byte loads).
__global__ void __launch_bounds__(256) ca_merge_kernel(const float* __restrict__ O,
                                                       const float2* __restrict__ stats,
                                                       int nsplit, int b0, int nb, int n, int t,
                                                       int d2, int f16,
                                                       __nv_bfloat16* __restrict__ PX) {
  const int64_t rows = (int64_t)nb * t;
  const int64_t rj = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (rj >= rows) return;
  float M = -INFINITY;
  for (int k = 0; k < nsplit; ++k) M = fmaxf(M, stats[k * rows + rj].x);
  float L = 0.f;
  for (int k = 0; k < nsplit; ++k) {
    const float2 st = stats[k * rows + rj];
    L += exp2f(st.x - M) * st.y;
  }
  const float invL = 1.f / L;
  const int j = (int)(rj % t), bb = (int)(rj / t);
  const int b = b0 + bb, h = b / n, i = b % n;
  const int64_t ld = 2 * (int64_t)n * d2;
  __nv_bfloat16* row = PX + ((int64_t)h * t + j) * ld + (int64_t)i * d2;
  for (int c = 4 * lane; c < d2; c += 128) {
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int k = 0; k < nsplit; ++k) {
      const float w = exp2f(stats[k * rows + rj].x - M);
      const float4 o = *reinterpret_cast<const float4*>(O + (k * rows + rj) * d2 + c);
      acc.x += w * o.x;
      acc.y += w * o.y;
      acc.z += w * o.z;
      acc.w += w * o.w;
    }
    uint32_t h01, l01, h23, l23;
    if (f16) {  // fp16 hi | lo
      split_pack_f16(acc.x * invL, acc.y * invL, h01, l01);
      split_pack_f16(acc.z * invL, acc.w * invL, h23, l23);
    } else {
      split_pack(acc.x * invL, acc.y * invL, h01, l01);
      split_pack(acc.z * invL, acc.w * invL, h23, l23);
    }
    *reinterpret_cast<uint2*>(row + c) = make_uint2(h01, h23);
    *reinterpret_cast<uint2*>(row + (int64_t)n * d2 + c) = make_uint2(l01, l23);
  }
}

__global__ void __launch_bounds__(256) rmsnorm_kernel(const void* __restrict__ in, int in_bf16,
                                                      int64_t rows, int D, int64_t ldi, float eps,
                                                      __nv_bfloat16* __restrict__ out,
                                                      int64_t ldo, int hilo) {
  const int64_t row = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= rows) return;
  auto ld = [&](int c) -> float {
    return in_bf16 ? __bfloat162float(static_cast<const __nv_bfloat16*>(in)[row * ldi + c])
                   : static_cast<const float*>(in)[row * ldi + c];
  };
  float ss = 0.f;
  for (int c = lane; c < D; c += 32) {
    const float x = ld(c);
    ss += x * x;
  }
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  const float scale = 1.f / sqrtf(ss / (float)D + eps);
  __nv_bfloat16* o = out + row * ldo;
  for (int c = lane; c < D; c += 32) {
    const float y = ld(c) * scale;
    if (hilo == 2) {  // fp16 hi | lo
      const __half hi = __float2half_rn(y);
      const __half lo = __float2half_rn(y - __half2float(hi));
      reinterpret_cast<__half*>(o)[c] = hi;
      reinterpret_cast<__half*>(o)[D + c] = lo;
    } else if (hilo) {
      __nv_bfloat16 hi, lo;
      split_hilo(y, hi, lo);
      o[c] = hi;
      o[D + c] = lo;
    } else {
      o[c] = __float2bfloat16_rn(y);
    }
  }
}

__global__ void bf16_to_f16_kernel(uint16_t* p, int64_t n) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  const __nv_bfloat16 b = *reinterpret_cast<const __nv_bfloat16*>(&p[i]);
  const __half h = __float2half_rn(__bfloat162float(b));
  p[i] = *reinterpret_cast<const uint16_t*>(&h);
}

__global__ void scale_rows_kernel(float* x, const float* inv, int64_t rows, int D) {
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= rows * D) return;
  x[idx] *= inv[idx / D];
}

__global__ void inv_norms_kernel(const float* __restrict__ parts, int64_t nvec, int nparts,
                                 int64_t block, float eps, float alpha, float* __restrict__ out) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= nvec) return;
  const float* p = parts + (i / block) * nparts * block + i % block;
  float s = 0.f;
  for (int k = 0; k < nparts; ++k) s += p[k * block];  // fixed order
  out[i] = alpha / fmaxf(sqrtf(fmaxf(s, 0.f)), eps);  // a quadratic form may round below 0
}

__global__ void transpose_kernel(const __nv_bfloat16* __restrict__ in, int64_t R, int64_t C,
                                 __nv_bfloat16* __restrict__ out, int perm_D) {
  __shared__ __nv_bfloat16 tile[32][33];
  const int64_t c0 = (int64_t)blockIdx.x * 32, r0 = (int64_t)blockIdx.y * 32;
  for (int k = threadIdx.y; k < 32; k += blockDim.y) {
    const int64_t r = r0 + k, c = c0 + threadIdx.x;
    if (r < R && c < C) {
      const int64_t src = perm_D > 0 ? pair_chunk_src((int)c, perm_D) : c;
      tile[k][threadIdx.x] = in[r * C + src];
    }
  }
  __syncthreads();
  for (int k = threadIdx.y; k < 32; k += blockDim.y) {
    const int64_t c = c0 + k, r = r0 + threadIdx.x;
    if (r < R && c < C) out[c * R + r] = tile[threadIdx.x][k];
  }
}

__global__ void bias_kernel(const __nv_bfloat16* in, const __nv_bfloat16* in2, int64_t C,
                            float* out, int perm_D) {
  const int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= C) return;
  const int64_t src = perm_D > 0 ? pair_chunk_src((int)c, perm_D) : c;
  out[c] = __bfloat162float(in[src]);
  if (in2 != nullptr) out[C + c] = __bfloat162float(in2[src]);
}

// ---------------------------------------------------------------- folded key projection

// Wt[i][c][j] = W_K,i[c][j] (c < 2d), b_K,i[j] (c = 2d), 0 (2d < c < Kp): the rows of
// W~_i = [W_K,i ; b_K,i], from the pair-chunk-ordered transposed copy WkT[i D + j][c] and
// bias bk[i D + j] (fp32 copies of bf16 values, so the conversion back is exact).
__global__ void fold_weights_kernel(const __nv_bfloat16* __restrict__ WkT,
                                    const float* __restrict__ bk, int n, int D, int d2, int Kp,
                                    __nv_bfloat16* __restrict__ Wt) {
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= (int64_t)n * Kp * D) return;
  const int j = (int)(idx % D);
  const int c = (int)((idx / D) % Kp);
  const int i = (int)(idx / ((int64_t)D * Kp));
  const int64_t col = (int64_t)i * D + j;
  __nv_bfloat16 v = __float2bfloat16_rn(0.f);
  if (c < d2)
    v = WkT[col * d2 + c];
  else if (c == d2)
    v = __float2bfloat16_rn(bk[col]);
  Wt[idx] = v;
}

// out[r] = [bf16 hi(x) | bf16 lo(x)] of fp32 rows x of width C.
__global__ void f32_hilo_kernel(const float* __restrict__ x, int64_t rows, int C,
                                __nv_bfloat16* __restrict__ out) {
  const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= rows * C) return;
  const int64_t r = idx / C;
  const int c = (int)(idx % C);
  __nv_bfloat16 hi, lo;
  split_hilo(x[idx], hi, lo);
  out[r * 2 * C + c] = hi;
  out[r * 2 * C + C + c] = lo;
}

// ----------------------------------------------------------------------- beta channel

// beta[j][h] of latent row (h, j): Z_out (hi + lo) . w, then saturation and the mass-matching
// offset (App. A, output projections and optional beta shaping). One warp per row.
__global__ void beta_kernel(const __nv_bfloat16* __restrict__ Z, int64_t rows, int t, int H,
                            int D, const float* __restrict__ w, float beta_max, float offset,
                            float* __restrict__ beta) {
  const int64_t row = (int64_t)blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
  const int lane = threadIdx.x & 31;
  if (row >= rows) return;
  const __nv_bfloat16* z = Z + row * 2 * D;
  float acc = 0.f;
  for (int c = lane; c < D; c += 32)
    acc += (__bfloat162float(z[c]) + __bfloat162float(z[D + c])) * w[c];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  if (lane == 0) {
    if (beta_max > 0.f) acc = beta_max * tanhf(acc / beta_max);
    const int h = (int)(row / t), j = (int)(row % t);
    beta[(int64_t)j * H + h] = acc + offset;
  }
}

// ----------------------------------------------------------------- biased decode attention
//
// Attention of query rows over the entries [C (t compact slots, logit bias beta) ; F (S
// uncompacted entries, bias 0)] (App. B, "Bias semantics in attention"). Grid (slot, KV-head,
// layer): the CTAs of a KV-head take its chunks of dec_chunk entries in turn (slot, slot +
// slots, ...). In a chunk each of the 16 warps holds 8 entries (4 at d = 256); a lane holds
// DPL = d/32 dimensions of its warp's keys and values in registers (coalesced loads, all issued
// up front), so the cache is read once and straight from global memory. Per query row of the
// KV-head's query heads, each warp forms its logits (warp sums of the lane partials), their max,
// weights and weighted values; the warps' (max, sum, O) are combined through shared memory and
// merged into the CTA's running row state, which is written once as the CTA's partial;
// decode_merge_kernel combines the partials in slot order.
constexpr int kDecThreads = 512;
constexpr int kDecRowGroup = 4;  // query rows per pass
// entries per warp: 8 (4 at d = 256, whose 8 dimensions per lane double the registers); 16
// warps keep more loads and more independent instruction streams in flight per SM
__host__ __device__ constexpr int dec_per_warp(int dpl) { return dpl == 8 ? 4 : 8; }
__host__ __device__ constexpr int dec_chunk(int dpl) { return dec_per_warp(dpl) * kDecThreads / 32; }

// DPL consecutive bf16 as DPL / 2 packed pairs (one 4-, 8- or 16-byte load).
template <int DPL>
__device__ __forceinline__ void load_pairs(const __nv_bfloat16* p, uint32_t (&x)[DPL / 2]) {
  if constexpr (DPL == 2) {
    x[0] = *reinterpret_cast<const uint32_t*>(p);
  } else if constexpr (DPL == 4) {
    const uint2 u = *reinterpret_cast<const uint2*>(p);
    x[0] = u.x;
    x[1] = u.y;
  } else {
    const uint4 u = *reinterpret_cast<const uint4*>(p);
    x[0] = u.x;
    x[1] = u.y;
    x[2] = u.z;
    x[3] = u.w;
  }
}

__device__ __forceinline__ float2 unpack_pair(uint32_t w) {
  return __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w));
}

// Warp sums of K values (K = 8 or 4) by recursive halving: each lane ends with the sum over all
// 32 lanes of one value, index dec_idx<K>(lane); 9 (K = 8) or 7 (K = 4) shuffles instead of
// 5 K.
template <int K>
__device__ __forceinline__ int dec_idx(int lane) {
  return K == 8 ? ((lane >> 4) & 1) * 4 + ((lane >> 3) & 1) * 2 + ((lane >> 2) & 1)
                : ((lane >> 4) & 1) * 2 + ((lane >> 3) & 1);
}

template <int K>
__device__ __forceinline__ int dec_src(int k) {  // a lane holding value k after dec_halve
  return K == 8 ? ((k >> 2) & 1) * 16 + ((k >> 1) & 1) * 8 + (k & 1) * 4
                : ((k >> 1) & 1) * 16 + (k & 1) * 8;
}

template <int K>
__device__ __forceinline__ float dec_halve(const float (&v)[K], int lane) {
  constexpr unsigned kFull = 0xffffffffu;
  float a[K / 2];
  {
    const bool up = lane & 16;
#pragma unroll
    for (int j = 0; j < K / 2; ++j) {
      const float send = up ? v[j] : v[j + K / 2];
      const float keep = up ? v[j + K / 2] : v[j];
      a[j] = keep + __shfl_xor_sync(kFull, send, 16);
    }
  }
  float c;
  if constexpr (K == 8) {
    float b[2];
    const bool up = lane & 8;
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      const float send = up ? a[j] : a[j + 2];
      const float keep = up ? a[j + 2] : a[j];
      b[j] = keep + __shfl_xor_sync(kFull, send, 8);
    }
    const bool up2 = lane & 4;
    c = (up2 ? b[1] : b[0]) + __shfl_xor_sync(kFull, up2 ? b[0] : b[1], 4);
    c += __shfl_xor_sync(kFull, c, 2);
    c += __shfl_xor_sync(kFull, c, 1);
  } else {
    const bool up = lane & 8;
    c = (up ? a[1] : a[0]) + __shfl_xor_sync(kFull, up ? a[0] : a[1], 8);
    c += __shfl_xor_sync(kFull, c, 4);
    c += __shfl_xor_sync(kFull, c, 2);
    c += __shfl_xor_sync(kFull, c, 1);
  }
  return c;
}

// Max (op 0) or sum (op 1) over the K distinct values held after dec_halve.
template <int K, int OP>
__device__ __forceinline__ float dec_across(float x) {
#pragma unroll
  for (int o = (K == 8 ? 4 : 8); o <= 16; o <<= 1) {
    const float y = __shfl_xor_sync(0xffffffffu, x, o);
    x = OP == 0 ? fmaxf(x, y) : x + y;
  }
  return x;
}

// Grid (slot, KV-head, layer): layer z's arguments are st.layer[z]; its partials start
// z * rows * slots rows into part_o / part_ml.
template <int DPL>
__global__ void __launch_bounds__(kDecThreads, 1)
    decode_chunk_kernel(const __grid_constant__ DecodeStack st, float* __restrict__ part_o,
                        float2* __restrict__ part_ml) {
  extern __shared__ float dsm[];
  constexpr int d = 32 * DPL;
  constexpr int kW = kDecThreads / 32;
  constexpr int kDecPerWarp = dec_per_warp(DPL);
  constexpr int kDecChunk = dec_chunk(DPL);
  const DecodeArgs& a = st.layer[blockIdx.z];
  const int h = blockIdx.y, slot = blockIdx.x, nslots = gridDim.x;
  {
    const int64_t lrows = (int64_t)blockIdx.z * a.nq * a.Hq * nslots;
    part_o += lrows * d;
    part_ml += lrows;
  }
  const int g = a.Hq / a.H;        // query heads per KV-head
  const int G = a.nq * g;          // query rows served by this CTA
  float* qs = dsm;                                  // [G][d]
  float* red = qs + (size_t)G * d;                  // [kW][kDecRowGroup][d + 2]
  float* acc = red + (size_t)kW * kDecRowGroup * (d + 2);  // [G][d + 2]: running O, M, L
  float* mlx = acc + (size_t)G * (d + 2);           // [kDecRowGroup][2]: next M, L
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t E = a.t + a.S;
  const int64_t nch = (E + kDecChunk - 1) / kDecChunk;
  // query rows of this KV-head: row r = (query n, head h * g + r % g), n = r / g
  for (int it = threadIdx.x; it < G * d; it += kDecThreads) {
    const int r = it / d, c = it % d;
    const int n = r / g, qh = h * g + r % g;
    qs[it] = __bfloat162float(a.q[((int64_t)n * a.Hq + qh) * d + c]);
  }
  for (int it = threadIdx.x; it < G * (d + 2); it += kDecThreads)
    acc[it] = (it % (d + 2)) == d ? -INFINITY : 0.f;
  __syncthreads();
  // This CTA's chunks: slot, slot + nslots, ... (in order), merged into acc as they come.
  for (int64_t chunk = slot; chunk < nch; chunk += nslots) {
    // this warp's keys and values (lane dims [DPL lane, +DPL)), packed bf16 pairs
    uint32_t kx[kDecPerWarp][DPL / 2], vx[kDecPerWarp][DPL / 2];
    float bias[kDecPerWarp];
    bool valid[kDecPerWarp];
#pragma unroll
    for (int k = 0; k < kDecPerWarp; ++k) {
      const int64_t e = chunk * kDecChunk + warp * kDecPerWarp + k;
      valid[k] = e < E;
      bias[k] = 0.f;
      if (valid[k]) {
        const bool comp = e < a.t;
        const int64_t off = (comp ? e * a.cst : (e - a.t) * a.fst) + (int64_t)h * d + DPL * lane;
        load_pairs<DPL>((comp ? a.Ck : a.Kf) + off, kx[k]);
        load_pairs<DPL>((comp ? a.Cv : a.Vf) + off, vx[k]);
        if (comp && a.beta != nullptr) bias[k] = a.beta[e * a.H + h];
      } else {
#pragma unroll
        for (int i = 0; i < DPL / 2; ++i) kx[k][i] = vx[k][i] = 0u;
      }
    }
    // the entry whose logit this lane will hold after the warp sums
    const int my = dec_idx<kDecPerWarp>(lane);
    float my_bias = 0.f;
    bool my_valid = false;
#pragma unroll
    for (int k = 0; k < kDecPerWarp; ++k)
      if (k == my) {
        my_bias = bias[k];
        my_valid = valid[k];
      }
    for (int r0 = 0; r0 < G; r0 += kDecRowGroup) {
      const int nr = min(kDecRowGroup, G - r0);
#pragma unroll 1
      for (int rr = 0; rr < nr; ++rr) {
        float qv[DPL];
#pragma unroll
        for (int i = 0; i < DPL; ++i) qv[i] = qs[(size_t)(r0 + rr) * d + DPL * lane + i];
        float lg[kDecPerWarp];
#pragma unroll
        for (int k = 0; k < kDecPerWarp; ++k) {
          float sdot = 0.f;
#pragma unroll
          for (int i = 0; i < DPL / 2; ++i) {
            const float2 kf = unpack_pair(kx[k][i]);
            sdot = fmaf(qv[2 * i], kf.x, fmaf(qv[2 * i + 1], kf.y, sdot));
          }
          lg[k] = sdot;
        }
        const float lsum = dec_halve<kDecPerWarp>(lg, lane);  // logit of entry `my`
        const float lgt = my_valid ? lsum * a.scale + my_bias : -INFINITY;
        const float m = dec_across<kDecPerWarp, 0>(lgt);
        const float pm = my_valid ? __expf(lgt - m) : 0.f;
        const float l = dec_across<kDecPerWarp, 1>(pm);
        float ov[DPL];
#pragma unroll
        for (int i = 0; i < DPL; ++i) ov[i] = 0.f;
#pragma unroll
        for (int k = 0; k < kDecPerWarp; ++k) {
          const float p = __shfl_sync(0xffffffffu, pm, dec_src<kDecPerWarp>(k));
#pragma unroll
          for (int i = 0; i < DPL / 2; ++i) {
            const float2 vf = unpack_pair(vx[k][i]);
            ov[2 * i] = fmaf(p, vf.x, ov[2 * i]);
            ov[2 * i + 1] = fmaf(p, vf.y, ov[2 * i + 1]);
          }
        }
        float* sl = red + ((size_t)warp * kDecRowGroup + rr) * (d + 2);
#pragma unroll
        for (int i = 0; i < DPL; ++i) sl[DPL * lane + i] = ov[i];
        if (lane == 0) {
          sl[d] = m;
          sl[d + 1] = l;
        }
      }
      __syncthreads();
      // Combine the warps' partials of this chunk and merge them into the running row state:
      // one thread per (row, column); the new (M, L) go through mlx so that no thread reads
      // a row's M after another has replaced it.
      for (int it = threadIdx.x; it < nr * d; it += kDecThreads) {
        const int rr = it / d, c = it % d;
        float Mc = -INFINITY;
#pragma unroll
        for (int w = 0; w < kW; ++w)
          Mc = fmaxf(Mc, red[((size_t)w * kDecRowGroup + rr) * (d + 2) + d]);
        float Lc = 0.f, Oc = 0.f;
#pragma unroll
        for (int w = 0; w < kW; ++w) {
          const float* sw = red + ((size_t)w * kDecRowGroup + rr) * (d + 2);
          const float wt = sw[d] == -INFINITY ? 0.f : __expf(sw[d] - Mc);
          Lc += wt * sw[d + 1];
          Oc += wt * sw[c];
        }
        float* ar = acc + (size_t)(r0 + rr) * (d + 2);
        const float Mo = ar[d], Lo = ar[d + 1];
        const float Mn = fmaxf(Mo, Mc);
        const float ao = Mo == -INFINITY ? 0.f : __expf(Mo - Mn);
        const float an = Mc == -INFINITY ? 0.f : __expf(Mc - Mn);
        ar[c] = ar[c] * ao + Oc * an;
        if (c == 0) {
          mlx[2 * rr] = Mn;
          mlx[2 * rr + 1] = Lo * ao + Lc * an;
        }
      }
      __syncthreads();
      for (int rr = threadIdx.x; rr < nr; rr += kDecThreads) {
        acc[(size_t)(r0 + rr) * (d + 2) + d] = mlx[2 * rr];
        acc[(size_t)(r0 + rr) * (d + 2) + d + 1] = mlx[2 * rr + 1];
      }
      __syncthreads();  // red, mlx and acc are reused by the next row group / chunk
    }
  }
  // this CTA's partial for every row
  for (int it = threadIdx.x; it < G * d; it += kDecThreads) {
    const int r = it / d, c = it % d;
    const int n = r / g, qh = h * g + r % g;
    const int64_t prow = ((int64_t)n * a.Hq + qh) * nslots + slot;
    const float* ar = acc + (size_t)r * (d + 2);
    part_o[prow * d + c] = ar[c];
    if (c == 0) part_ml[prow] = make_float2(ar[d], ar[d + 1]);
  }
}

// Output row (query n, query head qh): sum_s e^(m_s - M) O_s / sum_s e^(m_s - M) l_s over the
// chunk partials, in chunk order. One CTA of d threads per row, one column per thread.
__global__ void decode_merge_kernel(const __grid_constant__ DecodeStack st,
                                    const float* __restrict__ part_o,
                                    const float2* __restrict__ part_ml, int64_t rows, int nch,
                                    int d) {
  extern __shared__ float2 mls[];  // the row's (m, l) per chunk, then (weight, -)
  const int64_t row = blockIdx.x;
  const int c = threadIdx.x;
  __nv_bfloat16* __restrict__ out = st.layer[blockIdx.y].out;
  part_o += (int64_t)blockIdx.y * rows * nch * d;  // layer blockIdx.y's partials
  part_ml += (int64_t)blockIdx.y * rows * nch;
  for (int s = c; s < nch; s += blockDim.x) mls[s] = part_ml[row * nch + s];  // coalesced
  __syncthreads();
  float M = -INFINITY;
  for (int s = 0; s < nch; ++s) M = fmaxf(M, mls[s].x);
  float L = 0.f, o = 0.f;
  const float* po = part_o + row * nch * d + c;
#pragma unroll 8
  for (int s = 0; s < nch; ++s) {
    const float2 m = mls[s];
    const float w = m.x != -INFINITY ? __expf(m.x - M) : 0.f;
    L += w * m.y;
    o += w * po[(int64_t)s * d];
  }
  out[row * d + c] = __float2bfloat16_rn(o / L);
}

}  // namespace

namespace {

inline unsigned blocks_for(int64_t n, int per) { return (unsigned)((n + per - 1) / per); }

}  // namespace

size_t decode_workspace_bytes(int64_t rows, int64_t entries, int d, int layers) {
  const int chunk = dec_chunk(d / 32);
  const int64_t nch = (entries + chunk - 1) / chunk;
  const int64_t r = rows * layers;
  return (size_t)r * nch * d * 4 + 256 + (size_t)r * nch * 8 + 256;
}

cudaError_t launch_decode_biased(const DecodeStack& st, void* ws, int num_sms, cudaStream_t s) {
  if (st.n < 1 || st.n > kDecodeMaxLayers) return cudaErrorInvalidValue;
  const DecodeArgs& a = st.layer[0];  // every layer has the same shape
  const int64_t E = a.t + a.S;
  const int chunk = dec_chunk(a.d / 32);
  const int64_t nchunks = (E + chunk - 1) / chunk;
  // One wave per layer: the CTAs of a KV-head split its chunks (each CTA merges its own in
  // order).
  const int per_sm = 1;
  const int nch = (int)std::max<int64_t>(
      1, std::min<int64_t>(nchunks, (int64_t)num_sms * per_sm / std::max(1, a.H)));
  const int g = a.Hq / a.H;
  const int G = a.nq * g;
  const int64_t rows = (int64_t)a.nq * a.Hq;
  float* part_o = static_cast<float*>(ws);
  float2* part_ml = reinterpret_cast<float2*>(
      static_cast<uint8_t*>(ws) +
      (((size_t)rows * st.n * nch * a.d * 4 + 255) & ~size_t(255)));
  const size_t smem = ((size_t)G * a.d + (size_t)(kDecThreads / 32) * kDecRowGroup * (a.d + 2) +
                       (size_t)G * (a.d + 2) + 2 * kDecRowGroup) * 4;
  auto kern = a.d == 64 ? decode_chunk_kernel<2>
                        : a.d == 128 ? decode_chunk_kernel<4> : decode_chunk_kernel<8>;
  static thread_local size_t smem_set[3] = {48 * 1024, 48 * 1024, 48 * 1024};
  const int ki = a.d == 64 ? 0 : a.d == 128 ? 1 : 2;
  if (smem > smem_set[ki]) {
    cudaError_t e =
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    smem_set[ki] = smem;
  }
  kern<<<dim3(nch, a.H, st.n), kDecThreads, smem, s>>>(st, part_o, part_ml);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const size_t msm = (size_t)nch * sizeof(float2);
  if (msm > 48 * 1024) return cudaErrorInvalidValue;  // more than 6144 chunks
  decode_merge_kernel<<<dim3((unsigned)rows, st.n), a.d, msm, s>>>(st, part_o, part_ml, rows,
                                                                   nch, a.d);
  return cudaGetLastError();
}

cudaError_t launch_fold_weights(const __nv_bfloat16* WkT, const float* bk, int n, int D, int d2,
                                int Kp, __nv_bfloat16* Wt, cudaStream_t s) {
  const int64_t total = (int64_t)n * Kp * D;
  fold_weights_kernel<<<blocks_for(total, 256), 256, 0, s>>>(WkT, bk, n, D, d2, Kp, Wt);
  return cudaGetLastError();
}

cudaError_t launch_f32_hilo(const float* x, int64_t rows, int C, __nv_bfloat16* out,
                            cudaStream_t s) {
  if (rows == 0) return cudaSuccess;
  f32_hilo_kernel<<<blocks_for(rows * C, 256), 256, 0, s>>>(x, rows, C, out);
  return cudaGetLastError();
}

cudaError_t launch_beta(const __nv_bfloat16* Z, int t, int H, int D, const float* w,
                        float beta_max, float offset, float* beta, cudaStream_t s) {
  const int64_t rows = (int64_t)H * t;
  if (rows == 0) return cudaSuccess;
  beta_kernel<<<blocks_for(rows, 8), 256, 0, s>>>(Z, rows, t, H, D, w, beta_max, offset, beta);
  return cudaGetLastError();
}

cudaError_t launch_strip(const KVSource& src, int64_t N, int H, int d, const PosSegs& segs,
                         const double* omega, int rope_fix, __nv_bfloat16* X, __half* XT,
                         int64_t Np, float2* gd, double pmin, int G, int x16, int Kp,
                         cudaStream_t s) {
  if (d % 16 != 0 || Np % kStripTok != 0 || (Kp != 0 && (Kp % 64 != 0 || Kp < 2 * d + 1)))
    return cudaErrorInvalidValue;
  const size_t smem = (size_t)kStripTok * (d / 2) * sizeof(float2) +
                      (size_t)kStripTok * ((2 * d + 2) + (d + 2)) * 2;
  auto al16 = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; };
  const bool second = src.n_split < N;
  const int vec = al16(src.K) && al16(src.V) && src.sN % 8 == 0 && src.sH % 8 == 0 &&
                  (!second || (al16(src.K2) && al16(src.V2) && src.sN2 % 8 == 0 &&
                               src.sH2 % 8 == 0));
  static bool attr = false;
  if (!attr) {
    cudaFuncSetAttribute(strip_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 128 * 1024);
    attr = true;
  }
  strip_kernel<<<(unsigned)(Np / kStripTok), 256, smem, s>>>(src, N, H, d, segs, omega, rope_fix,
                                                             vec, x16, Kp, X, XT, Np, gd, pmin, G);
  return cudaGetLastError();
}

cudaError_t launch_heads_rot(float2* rot, int t, int hd, double pstart, double pstep,
                             const double* omega, int use_rope, cudaStream_t s) {
  const int64_t n = (int64_t)t * hd;
  heads_rot_kernel<<<blocks_for(n, 256), 256, 0, s>>>(rot, t, hd, pstart, pstep, omega, use_rope);
  return cudaGetLastError();
}

cudaError_t launch_rope_tables(float2* coarse, float* omega, int G, int D, double pmin,
                               const double* omega_c, cudaStream_t s) {
  const int64_t n = (int64_t)(G + kPosGrain) * (D / 2);
  rope_tables_kernel<<<blocks_for(n, 256), 256, 0, s>>>(coarse, omega, G, D, pmin, omega_c);
  return cudaGetLastError();
}

cudaError_t launch_q_rope(const float* qhat, int t_max, int b0, int nb, int t, int D,
                          double qstart, double qstep, const double* omega_c, int use_rope,
                          __nv_bfloat16* qhl, int fp16, float qscale, cudaStream_t s) {
  if (D % 256 != 0) return cudaErrorInvalidValue;
  const int64_t n = (int64_t)t * (D / 8);
  q_rope_kernel<<<blocks_for(n, 256), 256, 0, s>>>(qhat, t_max, b0, nb, t, D, qstart, qstep,
                                                    omega_c, use_rope, qhl, fp16, qscale);
  return cudaGetLastError();
}

template <typename OutT, bool HILO = false>
static bool softmax_reg(const float* S, int64_t rows, int64_t ncols, int64_t ldS, void* P,
                        int64_t ldP, cudaStream_t s) {
  const int64_t need = std::max(ldP, ncols);
  OutT* Pt = static_cast<OutT*>(P);
  if ((ldS % 4) != 0 || (ldP % 4) != 0) return false;
  if (need <= 1024)
    softmax_reg_kernel<OutT, 4, HILO><<<(unsigned)rows, 256, 0, s>>>(S, ncols, ldS, Pt, ldP);
  else if (need <= 2048)
    softmax_reg_kernel<OutT, 8, HILO><<<(unsigned)rows, 256, 0, s>>>(S, ncols, ldS, Pt, ldP);
  else if (need <= 4096)
    softmax_reg_kernel<OutT, 16, HILO><<<(unsigned)rows, 256, 0, s>>>(S, ncols, ldS, Pt, ldP);
  else if (need <= 8192)
    softmax_reg_kernel<OutT, 32, HILO><<<(unsigned)rows, 256, 0, s>>>(S, ncols, ldS, Pt, ldP);
  else if (need <= 16384)
    softmax_reg_kernel<OutT, 64, HILO><<<(unsigned)rows, 256, 0, s>>>(S, ncols, ldS, Pt, ldP);
  else
    return false;
  return true;
}

cudaError_t launch_wait_timeout_selftest(int* err, unsigned long long limit_ns, cudaStream_t s) {
  wait_timeout_selftest_kernel<<<1, 32, 0, s>>>(err, limit_ns);
  return cudaGetLastError();
}

cudaError_t launch_omega(double* out, int half, int width, double base, cudaStream_t s) {
  omega_kernel<<<blocks_for(half, 256), 256, 0, s>>>(out, half, width, base);
  return cudaGetLastError();
}

cudaError_t launch_softmax(const float* S, int64_t rows, int64_t ncols, int64_t ldS, void* P,
                           int64_t ldP, int out_fp16, cudaStream_t s) {
  if (rows == 0) return cudaSuccess;
  if (out_fp16 == 2 || out_fp16 == 3) {  // bf16 (2) or fp16 (3) hi | lo rows
    if (!(out_fp16 == 2 ? softmax_reg<__nv_bfloat16, true>(S, rows, ncols, ldS, P, ldP, s)
                        : softmax_reg<__half, true>(S, rows, ncols, ldS, P, ldP, s)))
      return cudaErrorInvalidValue;
    return cudaGetLastError();
  }
  if (out_fp16 ? softmax_reg<__half>(S, rows, ncols, ldS, P, ldP, s)
               : softmax_reg<__nv_bfloat16>(S, rows, ncols, ldS, P, ldP, s))
    return cudaGetLastError();
  if (out_fp16)
    softmax_kernel<__half><<<(unsigned)rows, 256, 0, s>>>(S, ncols, ldS,
                                                          static_cast<__half*>(P), ldP);
  else
    softmax_kernel<__nv_bfloat16><<<(unsigned)rows, 256, 0, s>>>(
        S, ncols, ldS, static_cast<__nv_bfloat16*>(P), ldP);
  return cudaGetLastError();
}

cudaError_t launch_ca_merge(const float* O, const float2* stats, int nsplit, int b0, int nb,
                            int n, int t, int d2, int f16, __nv_bfloat16* PX, cudaStream_t s) {
  const int64_t total = (int64_t)nb * t * d2;
  if (total == 0) return cudaSuccess;
  if (d2 % 4 != 0) return cudaErrorInvalidValue;
  ca_merge_kernel<<<blocks_for((int64_t)nb * t, 8), 256, 0, s>>>(O, stats, nsplit, b0, nb, n, t,
                                                                  d2, f16, PX);
  return cudaGetLastError();
}

cudaError_t launch_rmsnorm(const void* in, int in_bf16, int64_t rows, int D, int64_t ldi,
                           float eps, __nv_bfloat16* out, int64_t ldo, int hilo, cudaStream_t s) {
  rmsnorm_kernel<<<blocks_for(rows, 8), 256, 0, s>>>(in, in_bf16, rows, D, ldi, eps, out, ldo,
                                                     hilo);
  return cudaGetLastError();
}

cudaError_t launch_bf16_to_f16(void* p, int64_t n, cudaStream_t s) {
  if (n == 0) return cudaSuccess;
  bf16_to_f16_kernel<<<blocks_for(n, 256), 256, 0, s>>>(static_cast<uint16_t*>(p), n);
  return cudaGetLastError();
}

cudaError_t launch_scale_rows(float* x, const float* inv, int64_t rows, int D, cudaStream_t s) {
  scale_rows_kernel<<<blocks_for(rows * D, 256), 256, 0, s>>>(x, inv, rows, D);
  return cudaGetLastError();
}

cudaError_t launch_inv_norms(const float* parts, int64_t nvec, int nparts, int64_t block, float eps,
                             float alpha, float* out, cudaStream_t s) {
  if (block < 1) return cudaErrorInvalidValue;
  inv_norms_kernel<<<blocks_for(nvec, 256), 256, 0, s>>>(parts, nvec, nparts, block, eps, alpha,
                                                         out);
  return cudaGetLastError();
}

cudaError_t launch_transpose(const __nv_bfloat16* in, int64_t R, int64_t C, __nv_bfloat16* out,
                             int perm_D, cudaStream_t s) {
  dim3 grid(blocks_for(C, 32), blocks_for(R, 32));
  transpose_kernel<<<grid, dim3(32, 8), 0, s>>>(in, R, C, out, perm_D);
  return cudaGetLastError();
}

cudaError_t launch_bias(const __nv_bfloat16* in, const __nv_bfloat16* in2, int64_t C,
                        float* out, int perm_D, cudaStream_t s) {
  bias_kernel<<<blocks_for(C, 256), 256, 0, s>>>(in, in2, C, out, perm_D);
  return cudaGetLastError();
}

}  // namespace still
