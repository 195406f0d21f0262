// Persistent tcgen05 GEMM with split-precision passes, for sm_103a.
//
//   C[b](m, n) = sum over passes p of  A_p[b](m, :) . B_p[b](n, :)       (fp32 accumulate)
//
// A and B are 16-bit (bf16 or fp16), K-major, read by TMA in 128-byte-swizzled boxes of
// 64 elements along K. A pass names a K offset and a row offset into each operand, so a
// "hi/lo" operand stored as [hi | lo] along K gives the 2- and 3-pass products that keep
// ~fp32 accuracy on bf16 tensor cores (a_hi b_hi + a_hi b_lo + a_lo b_hi).
//
// CTA = 2 + Epi::kWarps warps: warp 0 issues TMA, warp 1 owns TMEM and issues tcgen05.mma
// (one thread), the rest run the epilogue from TMEM (Epi::kWarps / 4 per lane quarter). The accumulator is double-buffered in TMEM
// (2 x BN fp32 columns), so a tile's epilogue overlaps the next tile's main loop.
// Tiles are 128 x BN; the grid is persistent (tile += gridDim.x), m-tiles fastest so that
// CTAs running together share B tiles through L2.
#pragma once
#include "ptx.cuh"

namespace still {

constexpr int kBM = 128;
constexpr int kBK = 64;
// Epilogue warps come from the epilogue type (Epi::kWarps, a multiple of 4): kWarps / 4 warps
// share each TMEM lane quarter and split its columns ("parts").
template <class Epi>
constexpr int gemm_threads() {
  return 64 + 32 * Epi::kWarps;
}

struct GemmPass {
  int32_t a_koff, b_koff;  // K offset (elements) of this pass in A / B
  int32_t a_roff, b_roff;  // row offset of this pass in A / B
  int32_t klen;            // K extent, a multiple of 64
};

struct GemmParams {
  int32_t M, N;         // output extent per batch
  int32_t batch, bdiv;  // batch b splits as (b / bdiv, b % bdiv)
  // Row / K origin of batch b in each operand: (b / bdiv) * x1 + (b % bdiv) * x0.
  int64_t a_r1, a_r0, a_k1, a_k0;
  int64_t b_r1, b_r0, b_k1, b_k0;
  int32_t npass;
  GemmPass pass[3];
  int32_t ksplit;  // split-K factor (each split = a contiguous range of K iterations)
  // Tile order: m-tiles fastest (default; concurrent CTAs share B tiles through L2) or, with
  // n_fast, n-tiles fastest (concurrent CTAs share A tiles: for an A operand larger than L2
  // and a B operand that fits, A is then read from HBM once).
  int32_t n_fast;
  // Derived by the host launcher.
  int32_t tiles_m, tiles_n, iters_total, ntiles;
  uint32_t idesc;
  int* err;  // device error record (may be null)
};

struct TileCoord {
  int b, tm, tn, split;
};

__device__ __forceinline__ TileCoord decode_tile(const GemmParams& p, int tile) {
  TileCoord c;
  if (p.n_fast) {
    c.tn = tile % p.tiles_n;
    int r = tile / p.tiles_n;
    c.split = r % p.ksplit;
    r /= p.ksplit;
    c.tm = r % p.tiles_m;
    c.b = r / p.tiles_m;
    return c;
  }
  c.tm = tile % p.tiles_m;
  int r = tile / p.tiles_m;
  c.split = r % p.ksplit;
  r /= p.ksplit;
  c.tn = r % p.tiles_n;
  c.b = r / p.tiles_n;
  return c;
}

__device__ __forceinline__ void split_range(const GemmParams& p, int split, int& it0, int& it1) {
  it0 = (int)(((int64_t)p.iters_total * split) / p.ksplit);
  it1 = (int)(((int64_t)p.iters_total * (split + 1)) / p.ksplit);
}

// Per-epilogue-warp staging area (1024-byte aligned): 32 rows x 64 B for the LSU path (rows
// 80 B apart), or one TMA-store box of up to 4 KB.
constexpr int kStageRowU4 = 5;
constexpr int kWarpStageBytes = 4096;

template <int BN, class Epi>
struct GemmSmem {
  static constexpr int kStages = Epi::kStages > 0 ? Epi::kStages : (BN >= 256 ? 4 : 6);
  static constexpr int kABytes = kBM * kBK * 2;
  static constexpr int kBBytes = BN * kBK * 2;
  static constexpr int kStageBytes = kABytes + kBBytes;
  static constexpr int kEpiOffset = kStages * kStageBytes;  // a multiple of 1024
  static constexpr int kWarpStage = kWarpStageBytes * Epi::kStoreBufs;  // per epilogue warp
  static constexpr int kBarOffset = kEpiOffset + Epi::kWarps * kWarpStage;
  static constexpr int kBytes = kBarOffset + 256 + 1024;  // + barriers + alignment slack
  static_assert(kBytes <= 232448, "shared memory budget");
};

// Coalesced row store for one warp: lane i holds 64 bytes (v[0..3]) for its own row, to be
// written at dst (16-byte aligned) if valid. The warp exchanges them through its staging area
// so that each store instruction writes 8 rows x 64 contiguous bytes (whole 32-byte sectors).
// As warp_store64 with 32 bytes per lane: each store instruction writes 16 rows x 32 bytes.
__device__ __forceinline__ void warp_store32(uint4* stage, const uint4 (&v)[2], void* dst,
                                             bool valid) {
  const int lane = threadIdx.x & 31;
  stage[lane * 3] = v[0];
  stage[lane * 3 + 1] = v[1];
  __syncwarp();
  const unsigned long long mine = reinterpret_cast<unsigned long long>(dst);
#pragma unroll
  for (int it = 0; it < 2; ++it) {
    const int r = it * 16 + (lane >> 1), q = lane & 1;
    const unsigned long long d = __shfl_sync(0xffffffffu, mine, r);
    const int ok = __shfl_sync(0xffffffffu, valid ? 1 : 0, r);
    if (ok) reinterpret_cast<uint4*>(d)[q] = stage[r * 3 + q];
  }
  __syncwarp();
}

__device__ __forceinline__ void warp_store64(uint4* stage, const uint4 (&v)[4], void* dst,
                                             bool valid) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int q = 0; q < 4; ++q) stage[lane * kStageRowU4 + q] = v[q];
  __syncwarp();
  const unsigned long long mine = reinterpret_cast<unsigned long long>(dst);
#pragma unroll
  for (int it = 0; it < 4; ++it) {
    const int r = it * 8 + (lane >> 2), q = lane & 3;
    const unsigned long long d = __shfl_sync(0xffffffffu, mine, r);
    const int ok = __shfl_sync(0xffffffffu, valid ? 1 : 0, r);
    if (ok) reinterpret_cast<uint4*>(d)[q] = stage[r * kStageRowU4 + q];
  }
  __syncwarp();
}

// Coalesced row load for one warp, the inverse of warp_store64: lane i receives `bytes` (64 or
// 128) contiguous bytes starting at its own src (16-byte aligned), zeros when !valid. Each load
// instruction reads whole rows (8 lanes x 16 B per 128-B row); the warp's staging area
// (4 KB, rows 128 B apart, 16-B chunk q of row r at q ^ (r & 7)) does the transpose.
template <int kChunks>  // 16-byte chunks per row: 4 (64 B) or 8 (128 B)
__device__ __forceinline__ void warp_load_rows(uint4* stage, const void* src, bool valid,
                                               uint4 (&out)[kChunks]) {
  static_assert(kChunks == 4 || kChunks == 8, "64 or 128 bytes per row");
  const int lane = threadIdx.x & 31;
  const unsigned long long mine = reinterpret_cast<unsigned long long>(src);
  constexpr int kRowsPerIt = 32 / kChunks;
#pragma unroll
  for (int it = 0; it < kChunks; ++it) {
    const int r = it * kRowsPerIt + lane / kChunks, q = lane % kChunks;
    const unsigned long long s = __shfl_sync(0xffffffffu, mine, r);
    const int ok = __shfl_sync(0xffffffffu, valid ? 1 : 0, r);
    const uint4 x = ok ? reinterpret_cast<const uint4*>(s)[q] : make_uint4(0u, 0u, 0u, 0u);
    stage[r * 8 + (q ^ (r & 7))] = x;
  }
  __syncwarp();
#pragma unroll
  for (int q = 0; q < kChunks; ++q) out[q] = stage[lane * 8 + (q ^ (lane & 7))];
  __syncwarp();
}

// Epi must provide:  __device__ void prefetch(const GemmParams&, const TileCoord&, int row,
//                    int half) const  (called before the tile's accumulator is ready), and
//                    __device__ void operator()(const GemmParams&, const TileCoord&,
//                    int row_in_tile, uint32_t tmem_addr_of_this_warp_lane_quarter,
//                    int half, uint4* warp_stage, const CUtensorMap* out_map) const;
// where `half` (0 or 1) selects the 32-column chunks this warp owns: chunk c is handled by the
// warp with half == (c & 1); the functor loads TMEM and stores its own results.
// kRole only names the instantiation (one per GEMM of the launch sequence) so that profilers
// can tell the GEMMs apart; it does not change the code.
template <int BN, class Epi, int kRole>
__global__ void __launch_bounds__(gemm_threads<Epi>(), 1)
    tc_gemm_kernel(const __grid_constant__ CUtensorMap tmA,
                   const __grid_constant__ CUtensorMap tmB,
                   const __grid_constant__ CUtensorMap tmC, const GemmParams p, const Epi epi) {
  using S = GemmSmem<BN, Epi>;
  constexpr int kEpiWarps = Epi::kWarps;
  constexpr int kStages = S::kStages;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + S::kBarOffset);
  uint64_t* empty = full + kStages;
  uint64_t* tfull = empty + kStages;  // [2]
  uint64_t* tempty = tfull + 2;       // [2]
  uint64_t* drain = tempty + 2;       // [1]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], kEpiWarps);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
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
      // ------------------------------------------------------------ TMA producer
      int stage = 0;
      uint32_t phase = 0;
      uint32_t armed = 0;  // bit s: stage s armed at least once
      uint32_t armed_par = 0;
      for (int tile = blockIdx.x; tile < p.ntiles && !*abort_flag; tile += gridDim.x) {
        const TileCoord tc = decode_tile(p, tile);
        const int bo = tc.b / p.bdiv, bi = tc.b % p.bdiv;
        const int64_t ar = bo * p.a_r1 + bi * p.a_r0 + (int64_t)tc.tm * kBM;
        const int64_t ak = bo * p.a_k1 + bi * p.a_k0;
        const int64_t br = bo * p.b_r1 + bi * p.b_r0 + (int64_t)tc.tn * BN;
        const int64_t bk = bo * p.b_k1 + bi * p.b_k0;
        int it0, it1;
        split_range(p, tc.split, it0, it1);
        int pass = 0, base = 0;
        for (int it = it0; it < it1; ++it) {
          while (pass < p.npass - 1 && it >= base + p.pass[pass].klen / kBK) {
            base += p.pass[pass].klen / kBK;
            ++pass;
          }
          const GemmPass& ps = p.pass[pass];
          const int kk = (it - base) * kBK;
          if (!mbar_wait(&empty[stage], phase ^ 1)) {
            dev_set_error(p.err, DEV_WAIT_TIMEOUT, 100);
            *abort_flag = 1;
            break;
          }
          mbar_arrive_expect_tx(&full[stage], S::kStageBytes);
          uint8_t* sa = smem + stage * S::kStageBytes;
          tma_load_2d(sa, &tmA, &full[stage], (int32_t)(ak + ps.a_koff + kk),
                      (int32_t)(ar + ps.a_roff));
          tma_load_2d(sa + S::kABytes, &tmB, &full[stage], (int32_t)(bk + ps.b_koff + kk),
                      (int32_t)(br + ps.b_roff));
          armed |= 1u << stage;
          armed_par = (armed_par & ~(1u << stage)) | (phase << stage);
          if (++stage == kStages) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
      if (*abort_flag) {
        // Let every copy this thread issued land before the CTA can exit.
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
      for (int tile = blockIdx.x; tile < p.ntiles && !*abort_flag; tile += gridDim.x) {
        const TileCoord tc = decode_tile(p, tile);
        int it0, it1;
        split_range(p, tc.split, it0, it1);
        if (!mbar_wait(&tempty[acc], acc_phase ^ 1)) {
          dev_set_error(p.err, DEV_WAIT_TIMEOUT, 101);
          *abort_flag = 1;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(acc * BN);
        for (int it = it0; it < it1; ++it) {
          if (!mbar_wait(&full[stage], phase)) {
            dev_set_error(p.err, DEV_WAIT_TIMEOUT, 102);
            *abort_flag = 1;
            break;
          }
          tc_fence_after();
          const uint32_t sa = smem_u32(smem + stage * S::kStageBytes);
          const uint64_t ad = sdesc_k_sw128(sa);
          const uint64_t bd = sdesc_k_sw128(sa + S::kABytes);
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k)
            tc_mma_f16(d_tmem, ad + 2 * k, bd + 2 * k, p.idesc, (it > it0 || k > 0) ? 1u : 0u);
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
  } else {
    // -------------------------------------------------------------- epilogue (warps 2..)
    const int quarter = warp & 3;  // TMEM lanes this warp may access: [32q, 32q + 32)
    const int half = (warp - 2) >> 2;  // the "part" of the quarter's columns this warp owns
    const int row = quarter * 32 + lane;
    uint4* stage = reinterpret_cast<uint4*>(smem + S::kEpiOffset + (warp - 2) * S::kWarpStage);
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int tile = blockIdx.x; tile < p.ntiles; tile += gridDim.x) {
      const TileCoord tc = decode_tile(p, tile);
      epi.prefetch(p, tc, row, half);  // inputs that do not depend on the accumulator
      bool ok = mbar_wait(&tfull[acc], acc_phase);
      ok = __all_sync(0xffffffffu, ok);
      if (!ok || warp_flag(abort_flag)) {
        if (lane == 0 && !ok) {
          dev_set_error(p.err, DEV_WAIT_TIMEOUT, 103);
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
    if (lane == 0) bulk_wait_all();  // TMA stores issued by this warp (if any) have landed
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, 2 * BN);
  }
}

// ------------------------------------------------------------------ 2-SM form (CTA pairs)
//
// The same GEMM on clusters of two CTAs that compute a 256 x BN tile as one 2-SM
// tcgen05.mma (cta_group::2, M = 256) issued by the even CTA: CTA x holds the A rows of
// m-tile 2 m + x and rows [x BN / 2, +BN / 2) of the B tile, and each SM's tensor core reads
// the other half of B from its twin. Per SM this halves the B operand's shared-memory traffic
// and loads (the 1-SM kernel at 128 x 256 is bound by its shared memory: TMA writes and MMA
// reads of every stage, with the epilogue's staging on top). Both CTAs run the epilogue on
// their own 128 rows. Stage copies of both CTAs complete on the even CTA's full barrier; its
// commits arrive on both CTAs' empty and tfull barriers; both CTAs' epilogue warps arrive on
// its tempty barrier. An m-tile past the last one (odd count) is computed, and the epilogue
// skips its rows (they lie outside M).
template <int BN, class Epi>
struct Gemm2Smem {
  static constexpr int kStages = 4;
  static constexpr int kABytes = kBM * kBK * 2;
  static constexpr int kBBytes = (BN / 2) * kBK * 2;
  static constexpr int kStageBytes = kABytes + kBBytes;
  static constexpr int kEpiOffset = kStages * kStageBytes;  // a multiple of 1024
  static constexpr int kWarpStage = kWarpStageBytes * Epi::kStoreBufs;
  static constexpr int kBarOffset = kEpiOffset + Epi::kWarps * kWarpStage;
  static constexpr int kBytes = kBarOffset + 256 + 1024;
  static_assert(kBytes <= 232448, "shared memory budget");
};

// Tile pair t: as decode_tile over ceil(tiles_m / 2) m-tile pairs; this CTA takes 2 m + x.
__device__ __forceinline__ TileCoord decode_tile2(const GemmParams& p, int tile, int x) {
  GemmParams q = p;
  q.tiles_m = (p.tiles_m + 1) / 2;
  TileCoord c = decode_tile(q, tile);
  c.tm = 2 * c.tm + x;
  return c;
}

template <int BN, class Epi, int kRole>
__global__ void __launch_bounds__(gemm_threads<Epi>(), 1)
    tc_gemm2_kernel(const __grid_constant__ CUtensorMap tmA,
                    const __grid_constant__ CUtensorMap tmB,
                    const __grid_constant__ CUtensorMap tmC, const GemmParams p, const Epi epi) {
  using S = Gemm2Smem<BN, Epi>;
  constexpr int kEpiWarps = Epi::kWarps;
  constexpr int kStages = S::kStages;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + S::kBarOffset);  // even CTA's
  uint64_t* empty = full + kStages;
  uint64_t* tfull = empty + kStages;  // [2]
  uint64_t* tempty = tfull + 2;       // [2], even CTA's
  uint64_t* drain = tempty + 2;       // [1]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const int x = (int)(rank & 1u);
  const bool leader = x == 0;
  const uint16_t pair_mask = (uint16_t)((1u << rank) | (1u << (rank ^ 1u)));
  const int cid = (int)cluster_id_x(), ncl = (int)cluster_count_x();
  const int npairs = ((p.tiles_m + 1) / 2) * p.tiles_n * p.ksplit * p.batch;
  // the 2-SM instruction descriptor: M = 256
  const uint32_t idesc2 = (p.idesc & ~(0x1Fu << 24)) | ((uint32_t)(2 * kBM >> 4) << 24);

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], 2 * kEpiWarps);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
  }
  if (warp == 1) {
    tmem_alloc_2sm(tmem_slot, 2 * BN);
    tmem_relinquish_2sm();
  }
  tc_fence_before();
  cluster_sync();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const uint32_t l_full = cluster_map(smem_u32(full), rank & ~1u);
  const uint32_t l_tempty = cluster_map(smem_u32(tempty), rank & ~1u);

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------------------ TMA producer
      int stage = 0;
      uint32_t phase = 0;
      uint32_t armed = 0, armed_par = 0;
      bool bad = false;
      for (int tile = cid; tile < npairs && !bad && !*abort_flag; tile += ncl) {
        const TileCoord tc = decode_tile2(p, tile, x);
        const int bo = tc.b / p.bdiv, bi = tc.b % p.bdiv;
        const int64_t ar = bo * p.a_r1 + bi * p.a_r0 + (int64_t)tc.tm * kBM;
        const int64_t ak = bo * p.a_k1 + bi * p.a_k0;
        const int64_t br = bo * p.b_r1 + bi * p.b_r0 + (int64_t)tc.tn * BN + (BN / 2) * x;
        const int64_t bk = bo * p.b_k1 + bi * p.b_k0;
        int it0, it1;
        split_range(p, tc.split, it0, it1);
        int pass = 0, base = 0;
        for (int it = it0; it < it1; ++it) {
          while (pass < p.npass - 1 && it >= base + p.pass[pass].klen / kBK) {
            base += p.pass[pass].klen / kBK;
            ++pass;
          }
          const GemmPass& ps = p.pass[pass];
          const int kk = (it - base) * kBK;
          if (!mbar_wait(&empty[stage], phase ^ 1)) {
            dev_set_error(p.err, DEV_WAIT_TIMEOUT, 104);
            *abort_flag = 1;
            bad = true;
            break;
          }
          if (leader) {
            mbar_arrive_expect_tx(&full[stage], 2 * S::kStageBytes);
            armed |= 1u << stage;
            armed_par = (armed_par & ~(1u << stage)) | (phase << stage);
          }
          uint8_t* sa = smem + stage * S::kStageBytes;
          const uint32_t bar = l_full + 8u * (uint32_t)stage;
          tma_load_2d_2sm(sa, &tmA, bar, (int32_t)(ak + ps.a_koff + kk), (int32_t)(ar + ps.a_roff));
          tma_load_2d_2sm(sa + S::kABytes, &tmB, bar, (int32_t)(bk + ps.b_koff + kk),
                          (int32_t)(br + ps.b_roff));
          if (++stage == kStages) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
      // every slot released by the even CTA's MMAs before the CTA may leave
      for (int i = 0; i < kStages && !bad && !*abort_flag; ++i) {
        if (!mbar_wait(&empty[stage], phase ^ 1)) {
          dev_set_error(p.err, DEV_WAIT_TIMEOUT, 105);
          *abort_flag = 1;
          break;
        }
        if (++stage == kStages) {
          stage = 0;
          phase ^= 1;
        }
      }
      if (*abort_flag) {
        for (int s = 0; s < kStages; ++s)
          if (armed & (1u << s)) (void)mbar_wait_cluster(&full[s], (armed_par >> s) & 1);
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && leader) {
      // ------------------------------------------------------------ MMA issuer (2-SM)
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      bool issued = false;
      for (int tile = cid; tile < npairs && !*abort_flag; tile += ncl) {
        const TileCoord tc = decode_tile2(p, tile, x);
        int it0, it1;
        split_range(p, tc.split, it0, it1);
        if (!mbar_wait_cluster(&tempty[acc], acc_phase ^ 1)) {
          dev_set_error(p.err, DEV_WAIT_TIMEOUT, 106);
          *abort_flag = 1;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(acc * BN);
        for (int it = it0; it < it1; ++it) {
          if (!mbar_wait_cluster(&full[stage], phase)) {
            dev_set_error(p.err, DEV_WAIT_TIMEOUT, 107);
            *abort_flag = 1;
            break;
          }
          tc_fence_after();
          const uint32_t sa = smem_u32(smem + stage * S::kStageBytes);
          const uint64_t ad = sdesc_k_sw128(sa);
          const uint64_t bd = sdesc_k_sw128(sa + S::kABytes);
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k)
            tc_mma_f16_2sm(d_tmem, ad + 2 * k, bd + 2 * k, idesc2, (it > it0 || k > 0) ? 1u : 0u);
          issued = true;
          tc_commit_2sm_mc(&empty[stage], pair_mask);
          if (++stage == kStages) {
            stage = 0;
            phase ^= 1;
          }
        }
        if (*abort_flag) break;
        tc_commit_2sm_mc(&tfull[acc], pair_mask);
        if (++acc == 2) {
          acc = 0;
          acc_phase ^= 1;
        }
      }
      if (*abort_flag && issued) {
        tc_commit_2sm_mc(drain, (uint16_t)(1u << rank));
        (void)mbar_wait(drain, 0);
      }
    }
  } else {
    // -------------------------------------------------------------- epilogue (warps 2..)
    const int quarter = warp & 3;
    const int half = (warp - 2) >> 2;
    const int row = quarter * 32 + lane;
    uint4* stage = reinterpret_cast<uint4*>(smem + S::kEpiOffset + (warp - 2) * S::kWarpStage);
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int tile = cid; tile < npairs; tile += ncl) {
      const TileCoord tc = decode_tile2(p, tile, x);
      epi.prefetch(p, tc, row, half);
      bool ok = mbar_wait(&tfull[acc], acc_phase);
      ok = __all_sync(0xffffffffu, ok);
      if (!ok || warp_flag(abort_flag)) {
        if (lane == 0 && !ok) {
          dev_set_error(p.err, DEV_WAIT_TIMEOUT, 108);
          *abort_flag = 1;
        }
        break;
      }
      tc_fence_after();
      const uint32_t taddr = tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(acc * BN);
      epi(p, tc, row, taddr, half, stage, &tmC);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(l_tempty + 8u * (uint32_t)acc);
      if (++acc == 2) {
        acc = 0;
        acc_phase ^= 1;
      }
    }
    if (lane == 0) bulk_wait_all();
  }

  tc_fence_before();
  // No CTA frees its TMEM while the even CTA's MMAs may still write it, nor leaves while the
  // other may still copy into or arrive on its shared memory.
  cluster_sync();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_2sm(tmem_base, 2 * BN);
  }
}

}  // namespace still
