// Cross-attention value product with the softmax applied on the fly, for sm_103a.
//
//   O[s][b](m, :) = sum over tokens k of split s:  P(m, k) X(k, :),
//   P(m, k) = exp(S[b](m, k) - M[b](m)) / L[b](m)                    (row softmax, App. A)
//
// The scores S (fp32, written by the scores GEMM) are read once: eight "transform" warps turn
// each 128 x 64 slice into fp16 probabilities directly in the 128-byte-swizzled shared-memory
// layout tcgen05.mma reads, so the probabilities never exist in global memory. X^T arrives by
// TMA as fp16 hi and lo (the lo part only for the key half of X: the value half is exact in
// fp16). Row statistics (M, L) come from the scores epilogue's per-tile partials.
//
// Each transform warp keeps the next 64-token block's scores in flight while it converts the
// current one.
//
// CTA = 2 + 8 + 8 warps: TMA producer, MMA issuer, transform warps, epilogue.
#pragma once
#include "gemm_host.cuh"

namespace still {

constexpr int kPxTransformWarps = 8;
constexpr int kPxRowSteps = kBM / (4 * kPxTransformWarps);  // 4-row steps per transform warp

// Epilogue of the P X kernel: the tile's fp32 accumulator rows go to the split's partial
// output, out + split * split_stride + om(b, r, c), with coalesced warp stores.
struct EpiPxOut {
  static constexpr int kWarps = 8;
  float* out = nullptr;
  int64_t split_stride = 0;
  AffineMap om;
  int32_t tile_cols_ = 256;

  __device__ void operator()(const GemmParams& p, const TileCoord& tc, int row, uint32_t taddr,
                             int half, uint4* stage, const CUtensorMap*) const {
    const int r = tc.tm * kBM + row;
    const bool rvalid = r < p.M;
    for (int cc = 32 * half; cc < tile_cols_; cc += 64) {
      const int c0 = tc.tn * tile_cols_ + cc;
      if (c0 >= p.N) break;  // uniform across the warp
      float v[32];
      tmem_ld32(taddr + (uint32_t)cc, v);
      float* dst = out + (rvalid ? om.at(tc.b, r, c0) + (int64_t)tc.split * split_stride : 0);
      uint4 a4[4], b4[4];
      pack_f32x16(v, a4);
      pack_f32x16(v + 16, b4);
      warp_store64(stage, a4, dst, rvalid);
      warp_store64(stage, b4, dst + 16, rvalid);
    }
  }
};

struct PxParams {
  const float* S = nullptr;      // [nb][t][ldS] scores (natural-log units)
  const float2* stats = nullptr;  // [nb * t]: (max * log2 e, 1 / sum) per row
  int64_t ldS = 0;
  int32_t t = 0, N = 0;           // rows per batch, valid tokens
  int32_t xbase_row = 0;          // X^T row of feature 0 of KV-head h0 (= h0 * 2d)
  int32_t d2 = 0;                 // 2d (rows of X^T per KV-head)
  int32_t lo_rows = 0;            // rows of X^T lo that matter (the key half, d)
  int64_t Np = 0;                 // token pitch of X^T hi / lo
  int32_t nb = 0, bdiv = 1;       // batches; KV-head of batch b = (b / bdiv)
};

// BN: output columns per tile; LOB: rows of the X^T lo box (the key half inside the tile);
// PLO: the probabilities as fp16 hi + lo (a second P tile and one more MMA pass).
template <int BN, int LOB, bool PLO = false>
struct PxSmem {
  static constexpr int kPBytes = kBM * kBK * 2;       // one P tile (fp16)
  static constexpr int kABytes = kPBytes * (PLO ? 2 : 1);  // P hi [, P lo]
  static constexpr int kBBytes = BN * kBK * 2;        // X^T hi tile
  static constexpr int kLoBytes = LOB * kBK * 2;      // X^T lo tile
  static constexpr int kStageBytes = kABytes + kBBytes + kLoBytes;
  static constexpr int kEpiBytes = EpiPxOut::kWarps * kWarpStageBytes;
  static constexpr int kStages = (232448 - kEpiBytes - 2048) / kStageBytes >= 3 ? 3 : 2;
  static constexpr int kEpiOffset = kStages * kStageBytes;
  static constexpr int kBarOffset = kEpiOffset + kEpiBytes;
  static constexpr int kBytes = kBarOffset + 256 + 1024;
  static_assert(kBytes <= 232448, "shared memory budget");
};

// The GemmParams carry M = t, N = BN-tiled output width (2d), batch = nb, ksplit; a single
// "pass" of klen = Np describes the token range (iters_total = Np / 64).
constexpr int kPxThreads = 64 + 32 * kPxTransformWarps + 32 * EpiPxOut::kWarps;

template <int BN, int LOB, bool PLO>
__global__ void __launch_bounds__(kPxThreads, 1)
    px_fused_kernel(const __grid_constant__ CUtensorMap tmXhi,
                    const __grid_constant__ CUtensorMap tmXlo,
                    const __grid_constant__ CUtensorMap tmC, const GemmParams p,
                    const PxParams px, const EpiPxOut epi) {
  using S = PxSmem<BN, LOB, PLO>;
  constexpr int kStages = S::kStages;
  constexpr int kEpiWarps = EpiPxOut::kWarps;
  constexpr int kTW = kPxTransformWarps;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + S::kBarOffset);
  uint64_t* empty = full + kStages;
  uint64_t* tfull = empty + kStages;  // [2]
  uint64_t* tempty = tfull + 2;       // [2]
  uint64_t* drain = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int first_epi = 2 + kTW;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1 + kTW);  // TMA producer arrival (+ bytes) and each transform warp
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], kEpiWarps);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
    tma_prefetch_desc(&tmXhi);
    tma_prefetch_desc(&tmXlo);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, 2 * BN);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------------------ TMA producer (X^T)
      int stage = 0;
      uint32_t phase = 0;
      uint32_t armed = 0, armed_par = 0;
      for (int tile = blockIdx.x; tile < p.ntiles && !*abort_flag; tile += gridDim.x) {
        const TileCoord tc = decode_tile(p, tile);
        const int lo_w = min(BN, max(0, px.lo_rows - tc.tn * BN));
        const int xrow = px.xbase_row + (tc.b / px.bdiv) * px.d2 + tc.tn * BN;
        int it0, it1;
        split_range(p, tc.split, it0, it1);
        for (int it = it0; it < it1; ++it) {
          if (!mbar_wait(&empty[stage], phase ^ 1)) {
            dev_set_error(p.err, DEV_WAIT_TIMEOUT, 200);
            *abort_flag = 1;
            break;
          }
          mbar_arrive_expect_tx(&full[stage], S::kBBytes + (lo_w > 0 ? S::kLoBytes : 0));
          // lo_w is either LOB or 0 (the launcher guarantees it)
          uint8_t* sb = smem + stage * S::kStageBytes + S::kABytes;
          tma_load_2d(sb, &tmXhi, &full[stage], it * kBK, xrow);
          if (lo_w > 0)
            tma_load_2d(sb + S::kBBytes, &tmXlo, &full[stage], (int32_t)(px.Np + it * kBK), xrow);
          armed |= 1u << stage;
          armed_par = (armed_par & ~(1u << stage)) | (phase << stage);
          if (++stage == kStages) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
      if (*abort_flag) {
        for (int s = 0; s < kStages; ++s)
          if (armed & (1u << s)) (void)mbar_wait(&full[s], (armed_par >> s) & 1);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ------------------------------------------------------------ MMA issuer
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      bool issued = false;
      const uint32_t idesc_hi = idesc_f16(kBM, BN, 0);
      for (int tile = blockIdx.x; tile < p.ntiles && !*abort_flag; tile += gridDim.x) {
        const TileCoord tc = decode_tile(p, tile);
        const int lo_w = min(BN, max(0, px.lo_rows - tc.tn * BN));
        const uint32_t idesc_lo = idesc_f16(kBM, lo_w > 0 ? lo_w : 16, 0);
        int it0, it1;
        split_range(p, tc.split, it0, it1);
        if (!mbar_wait(&tempty[acc], acc_phase ^ 1)) {
          dev_set_error(p.err, DEV_WAIT_TIMEOUT, 201);
          *abort_flag = 1;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(acc * BN);
        for (int it = it0; it < it1; ++it) {
          if (!mbar_wait(&full[stage], phase)) {
            dev_set_error(p.err, DEV_WAIT_TIMEOUT, 202);
            *abort_flag = 1;
            break;
          }
          tc_fence_after();
          const uint32_t sa = smem_u32(smem + stage * S::kStageBytes);
          const uint64_t ad = sdesc_k_sw128(sa);
          const uint64_t bd = sdesc_k_sw128(sa + S::kABytes);
          const uint64_t ld = sdesc_k_sw128(sa + S::kABytes + S::kBBytes);
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k)
            tc_mma_f16(d_tmem, ad + 2 * k, bd + 2 * k, idesc_hi, (it > it0 || k > 0) ? 1u : 0u);
          if constexpr (PLO) {  // + P_lo X_hi
            const uint64_t pl = sdesc_k_sw128(sa + S::kPBytes);
#pragma unroll
            for (int k = 0; k < kBK / 16; ++k) tc_mma_f16(d_tmem, pl + 2 * k, bd + 2 * k, idesc_hi, 1u);
          }
          if (lo_w > 0) {
#pragma unroll
            for (int k = 0; k < kBK / 16; ++k) tc_mma_f16(d_tmem, ad + 2 * k, ld + 2 * k, idesc_lo, 1u);
          }
          issued = true;
          tc_commit(&empty[stage]);
          if (++stage == kStages) {
            stage = 0;
            phase ^= 1;
          }
        }
        if (*abort_flag) break;
        tc_commit(&tfull[acc]);
        if (++acc == 2) {
          acc = 0;
          acc_phase ^= 1;
        }
      }
      if (*abort_flag && issued) {
        tc_commit(drain);
        (void)mbar_wait(drain, 0);
      }
    }
  } else if (warp < first_epi) {
    // -------------------------------------------------------------- transform warps
    // Warp w writes rows [16w, 16w + 16) of each P tile; a step covers 4 rows x 64 tokens,
    // 8 lanes per row, 8 tokens (one 16-byte fp16 chunk) per lane.
    const int w = warp - 2;
    const int sub = lane >> 3, chunk = lane & 7;
    constexpr float kLog2e = 1.4426950408889634f;
    int stage = 0;
    uint32_t phase = 0;
    for (int tile = blockIdx.x; tile < p.ntiles && !warp_flag(abort_flag); tile += gridDim.x) {
      const TileCoord tc = decode_tile(p, tile);
      float2 st[kPxRowSteps];
      const float* srow[kPxRowSteps];
#pragma unroll
      for (int q = 0; q < kPxRowSteps; ++q) {
        const int m = tc.tm * kBM + 4 * kPxRowSteps * w + 4 * q + sub;
        const bool ok = m < px.t;
        st[q] = ok ? px.stats[(int64_t)tc.b * px.t + m] : make_float2(0.f, 0.f);
        srow[q] = ok ? px.S + ((int64_t)tc.b * px.t + m) * px.ldS : nullptr;
      }
      int it0, it1;
      split_range(p, tc.split, it0, it1);
      // The sixteen loads of a k-block are issued together, one k-block ahead of their use:
      // while block it is converted, block it + 1 is in flight (software pipelining).
      auto load_block = [&](int it, float4 (&xo)[kPxRowSteps][2]) {
        const int k0 = it * kBK + chunk * 8;
        const bool full_k = k0 + 8 <= px.N;
#pragma unroll
        for (int q = 0; q < kPxRowSteps; ++q) {
          if (srow[q] != nullptr && full_k) {
            xo[q][0] = __ldg(reinterpret_cast<const float4*>(srow[q] + k0));
            xo[q][1] = __ldg(reinterpret_cast<const float4*>(srow[q] + k0) + 1);
          } else {
            float t8[8];
#pragma unroll
            for (int e = 0; e < 8; ++e)
              t8[e] = (srow[q] != nullptr && k0 + e < px.N) ? srow[q][k0 + e] : -INFINITY;
            xo[q][0] = make_float4(t8[0], t8[1], t8[2], t8[3]);
            xo[q][1] = make_float4(t8[4], t8[5], t8[6], t8[7]);
          }
        }
      };
      float4 x[kPxRowSteps][2], xn[kPxRowSteps][2];
      if (it0 < it1) load_block(it0, x);
      for (int it = it0; it < it1; ++it) {
        if (it + 1 < it1) load_block(it + 1, xn);
        bool ok = mbar_wait(&empty[stage], phase ^ 1);
        ok = __all_sync(0xffffffffu, ok);
        if (!ok) {
          if (lane == 0) {
            dev_set_error(p.err, DEV_WAIT_TIMEOUT, 203);
            *abort_flag = 1;
          }
          break;
        }
        uint4* a = reinterpret_cast<uint4*>(smem + stage * S::kStageBytes);
#pragma unroll
        for (int q = 0; q < kPxRowSteps; ++q) {
          const int r = 4 * kPxRowSteps * w + 4 * q + sub;  // row inside the tile
          const float v0[8] = {x[q][0].x, x[q][0].y, x[q][0].z, x[q][0].w,
                               x[q][1].x, x[q][1].y, x[q][1].z, x[q][1].w};
          float v[8];
#pragma unroll
          for (int e = 0; e < 8; ++e) v[e] = exp2f(v0[e] * kLog2e - st[q].x) * st[q].y;  // 0 for -inf
          __half2 h01 = __floats2half2_rn(v[0], v[1]), h23 = __floats2half2_rn(v[2], v[3]);
          __half2 h45 = __floats2half2_rn(v[4], v[5]), h67 = __floats2half2_rn(v[6], v[7]);
          a[r * 8 + (chunk ^ (r & 7))] =
              make_uint4(*reinterpret_cast<uint32_t*>(&h01), *reinterpret_cast<uint32_t*>(&h23),
                         *reinterpret_cast<uint32_t*>(&h45), *reinterpret_cast<uint32_t*>(&h67));
          if constexpr (PLO) {  // lo = fp16(p - hi), same swizzled position in the P_lo tile
            const float2 f01 = __half22float2(h01), f23 = __half22float2(h23);
            const float2 f45 = __half22float2(h45), f67 = __half22float2(h67);
            __half2 l01 = __floats2half2_rn(v[0] - f01.x, v[1] - f01.y);
            __half2 l23 = __floats2half2_rn(v[2] - f23.x, v[3] - f23.y);
            __half2 l45 = __floats2half2_rn(v[4] - f45.x, v[5] - f45.y);
            __half2 l67 = __floats2half2_rn(v[6] - f67.x, v[7] - f67.y);
            a[S::kPBytes / 16 + r * 8 + (chunk ^ (r & 7))] =
                make_uint4(*reinterpret_cast<uint32_t*>(&l01), *reinterpret_cast<uint32_t*>(&l23),
                           *reinterpret_cast<uint32_t*>(&l45), *reinterpret_cast<uint32_t*>(&l67));
          }
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(&full[stage]);
        if (++stage == kStages) {
          stage = 0;
          phase ^= 1;
        }
#pragma unroll
        for (int q = 0; q < kPxRowSteps; ++q) {
          x[q][0] = xn[q][0];
          x[q][1] = xn[q][1];
        }
      }
    }
  } else {
    // -------------------------------------------------------------- epilogue
    const int ew = warp - first_epi;
    const int quarter = warp & 3;
    const int half = ew >> 2;
    const int row = quarter * 32 + lane;
    uint4* stage = reinterpret_cast<uint4*>(smem + S::kEpiOffset + ew * kWarpStageBytes);
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int tile = blockIdx.x; tile < p.ntiles; tile += gridDim.x) {
      const TileCoord tc = decode_tile(p, tile);
      bool ok = mbar_wait(&tfull[acc], acc_phase);
      ok = __all_sync(0xffffffffu, ok);
      if (!ok || warp_flag(abort_flag)) {
        if (lane == 0 && !ok) {
          dev_set_error(p.err, DEV_WAIT_TIMEOUT, 204);
          *abort_flag = 1;
        }
        break;
      }
      tc_fence_after();
      const uint32_t taddr = tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(acc * BN);
      epi(p, tc, row, taddr, half, stage, &tmC);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty[acc]);
      if (++acc == 2) {
        acc = 0;
        acc_phase ^= 1;
      }
    }
    if (lane == 0) bulk_wait_all();
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, 2 * BN);
  }
}

}  // namespace still

namespace still {

// Launches px_fused_kernel: A = probabilities from S (transform warps), B = X^T hi / lo.
template <int BN, int LOB, bool PLO = false>
inline cudaError_t launch_px_fused(const Operand2D& XT, GemmParams p, const PxParams& px,
                                   EpiPxOut epi, int num_sms, cudaStream_t stream) {
  using S = PxSmem<BN, LOB, PLO>;
  if (!finalize_gemm<BN>(p, 0)) return cudaErrorInvalidValue;
  CUtensorMap thi, tlo, tc;
  if (!make_tmap(&thi, XT, BN) || !make_tmap(&tlo, XT, LOB)) return cudaErrorInvalidValue;
  std::memset(&tc, 0, sizeof(tc));
  epi.tile_cols_ = BN;
  auto kern = px_fused_kernel<BN, LOB, PLO>;
  static thread_local bool attr_set = false;
  if (!attr_set) {
    cudaError_t e =
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, S::kBytes);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  const int grid = p.ntiles < num_sms ? p.ntiles : num_sms;
  kern<<<grid, kPxThreads, S::kBytes, stream>>>(thi, tlo, tc, p, px, epi);
  return cudaGetLastError();
}

}  // namespace still
