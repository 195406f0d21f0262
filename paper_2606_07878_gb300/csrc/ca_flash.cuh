// Cross-attention of one compactor layer in a single kernel, for sm_103a (App. A,
// "Cross-attention"; the compactor's latent queries attend over the cached tokens X):
//
//   S(m, k)  = scale * q_m . k_k / |k~_k|          3-pass split-bf16 tcgen05.mma, fp32 in TMEM
//   P(m, k)  = exp(S(m, k) - M(m))                   online row softmax over 256-key tiles
//   O(m, :)  = sum_k P(m, k) X(k, :) / sum_k P(m, k)
//
// A work unit is (batch b = (KV-head, cross head), two 128-row query tiles, key split) on a
// CTA pair (cluster of two): CTA x computes query tile 2 m + x. Per key tile the even CTA issues
// S for both tiles as one 2-SM MMA (tcgen05.mma.cta_group::2, M = 256) into each CTA's TMEM
// columns [0, 256); each CTA's eight softmax warps drain their S to registers and form fp16
// probabilities in the 128-byte-swizzled shared-memory layout the tensor core reads, and the
// even CTA accumulates P X^T for both into TMEM columns [256, 256 + 2d). Each CTA holds its own
// q and P rows and half of every k and X^T stage (the B operands), which halves the B traffic of
// each SM's shared memory. S and P never reach global memory. The running max is kept in log2 units and only moved (with a rescale of the
// TMEM accumulator) when a tile raises it by more than kRescaleLog2, so that P <= 2^8 fits fp16.
//
// Issue order of the tensor pipe: S_0, S_1, PX_0, S_2, PX_1, ... . PX_{j-1} runs while the
// softmax warps drain S_j, so the single S buffer costs no tensor-pipe idle time.
//
// Output per split: unnormalised O rows and (m, l) with m in log2 units; ca_merge_kernel
// combines the splits in a fixed order (bit-reproducible).
//
// EX (a block whose output feeds another block): q, k in fp16 hi | lo, probabilities as fp16
// hi + lo with one more P X pass, 128-key tiles (S in TMEM columns [0, 128)).
//
// Synchronisation inside the pair (all waits bounded): every stage's copies of both CTAs
// complete on the even CTA's full barrier (cta_group::2 TMA); its commits arrive on both CTAs'
// empty, sfull and pempty barriers; both CTAs' softmax warps arrive on its sfree and ofree
// barriers, and the odd CTA's warp 1 forwards each completion of its pfull barrier.
//
// CTA = 10 warps: 0 TMA producer, 1 MMA issuer (even CTA) or P relay (odd CTA) and TMEM
// allocation, 2..9 softmax / output.
#pragma once
#include "gemm_host.cuh"

namespace still {

struct FlashParams {
  int32_t t = 0, N = 0;     // query rows per batch, valid keys
  int32_t D = 0;            // width of one hi or lo part of q / k (multiple of 64)
  int64_t Np = 0;           // key pitch of X^T hi / lo (multiple of 64, >= N, zero padded)
  int32_t nb = 0, bdiv = 1; // batches; KV-head of batch b is h0 + b / bdiv
  int32_t xbase_row = 0;    // X^T row of feature 0 of KV-head h0
  // Q rows of batch b start at q_row0 + b * q_pitch (q_pitch 0: t). K rows of batch b start at
  // k_row0 + b * N, or at k_row0 + (b / kdiv) * N when kdiv > 0 (keys shared by kdiv batches).
  int64_t q_row0 = 0, k_row0 = 0;
  int32_t q_pitch = 0, kdiv = 0;
  int32_t tiles_m = 0, tiles_k = 0, nsplit = 1, nunits = 0;
  const float* kinv = nullptr;  // [nb][N]: scale / |k~| per key
  float* O = nullptr;           // [nsplit][nb][t][2d] unnormalised
  float2* stats = nullptr;      // [nsplit][nb][t]: (running max m in log2 units, sum l)
  int* err = nullptr;
  // One-pass scores with a top-k repair (ca_pair_kernel<true>): per (split, b, row), kTopK
  // candidates per list and kTopLists lists, as (key, c = m + log2 p of the weight used);
  // key -1 marks an empty slot.
  int* cand_key = nullptr;      // [nsplit][nb][t][kTopLists][kTopK]
  float* cand_c = nullptr;
};

constexpr int kTopK = 8;       // repair candidates per list
constexpr int kTopLists = 4;   // lists per row: (column half of its CTAs, half of the key tile)

constexpr int kFlashKeys = 256;       // keys per S tile (EX: 128)
constexpr int kFlashSoftWarps = 8;    // two per TMEM lane quarter
constexpr int kFlashThreads = 64 + 32 * kFlashSoftWarps;
constexpr float kRescaleLog2 = 8.f;

// EX (split precision, for a block whose output feeds another block): q, k as fp16 hi | lo and
// the probabilities as fp16 hi + lo (one more P X pass); key tiles of 128 so that the P_hi and
// P_lo tiles together take the shared memory of one 256-key P tile.
template <int D2, bool EX = false>
struct FlashSmem {
  static_assert(D2 == 128 || D2 == 256, "2d must be 128 or 256");
  // Per CTA of a pair: its own q rows and half of the B operand of every stage (the 2-SM MMA
  // reads the other half from the twin's shared memory at the same offset).
  static constexpr int kKeys = EX ? 128 : kFlashKeys;     // keys per S tile
  static constexpr int kQBytes = kBM * kBK * 2;            // q chunk, 16 KB
  static constexpr int kKBytes = (kKeys / 2) * kBK * 2;    // half a k chunk
  static constexpr int kXhiBytes = (D2 / 2) * kBK * 2;     // half the X^T hi chunk
  static constexpr int kXloBytes = (D2 / 4) * kBK * 2;     // half the X^T lo chunk (key half)
  static constexpr int kStageBytes = (kQBytes + kKBytes) > (kXhiBytes + kXloBytes)
                                         ? (kQBytes + kKBytes) : (kXhiBytes + kXloBytes);
  static constexpr int kStages = 4;
  static constexpr int kPChunkBytes = kBM * kBK * 2;       // 128 rows x 64 keys fp16
  static constexpr int kPChunks = kKeys / kBK;             // chunks of one P tile (hi)
  static constexpr int kPOffset = kStages * kStageBytes;
  static constexpr int kKinvOffset = kPOffset + 4 * kPChunkBytes;        // [8 warps][128] f32
  static constexpr int kXchOffset = kKinvOffset + kFlashSoftWarps * 128 * 4;  // [2][2][128] f32
  static constexpr int kBarOffset = kXchOffset + 2 * 2 * 128 * 4;
  static constexpr int kBytes = kBarOffset + 256 + 1024;
  static_assert(kXhiBytes + kXloBytes <= kStageBytes, "X chunk fits a stage");
  static_assert(kStageBytes % 1024 == 0 && kXhiBytes % 1024 == 0, "swizzle-atom alignment");
  static_assert(kBytes <= 232448, "shared memory budget");
};

struct FlashUnit {
  int b, tm, split, j0, j1;
};

// Unit u of the CTA pairs: query tiles 2 m and 2 m + 1 (m fastest), then the key split, then
// the batch; the CTA x of the pair takes query tile 2 m + x (one past the last tile, for an odd
// count, is computed and not stored).
__device__ __forceinline__ FlashUnit flash_pair_unit(const FlashParams& f, int u, uint32_t x) {
  const int mp = (f.tiles_m + 1) / 2;
  FlashUnit r;
  r.tm = 2 * (u % mp) + (int)x;
  const int q = u / mp;
  r.split = q % f.nsplit;
  r.b = q / f.nsplit;
  r.j0 = (int)(((int64_t)f.tiles_k * r.split) / f.nsplit);
  r.j1 = (int)(((int64_t)f.tiles_k * (r.split + 1)) / f.nsplit);
  return r;
}

// Number of 64-key chunks of tile j (of KEYS keys) that lie inside the padded key range [0, Np).
template <int KEYS>
__device__ __forceinline__ int flash_chunks(const FlashParams& f, int j) {
  const int64_t left = f.Np - (int64_t)j * KEYS;
  return left >= KEYS ? KEYS / kBK : (int)(left / kBK);
}

template <int D2, bool EX>
__global__ void __launch_bounds__(kFlashThreads, 1)
    ca_flash_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                    const __grid_constant__ CUtensorMap tmXhi,
                    const __grid_constant__ CUtensorMap tmXlo, const FlashParams f) {
  using S = FlashSmem<D2, EX>;
  constexpr int kKeys = S::kKeys;
  constexpr int kStages = S::kStages;
  constexpr int kOCols = D2 / 2;  // O columns per softmax warp (its half of 2d)
  constexpr int kCols = kKeys / 2;  // S columns per softmax warp (its half of the key tile)
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + S::kBarOffset);  // even CTA: stage loaded
  uint64_t* empty = full + kStages;   // stage consumed (the even CTA's commit, in both CTAs)
  uint64_t* sfull = empty + kStages;  // S tile complete in TMEM
  uint64_t* sfree = sfull + 1;        // even CTA: S tile drained in both CTAs
  uint64_t* pfull = sfree + 1;        // P tile written (and O rescaled if needed)
  uint64_t* ptwin = pfull + 1;        // even CTA: the same in the odd CTA
  uint64_t* pempty = ptwin + 1;       // PX MMA complete (P buffer free, O up to date)
  uint64_t* ofree = pempty + 1;       // even CTA: O drained in both CTAs at the end of a unit
  uint64_t* xb = ofree + 1;           // [4] row-value exchange per lane quarter
  uint64_t* drain = xb + 4;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int qchunks = f.D / kBK;
  const uint32_t rank = cluster_ctarank();
  const uint32_t qx = rank & 1u;  // query tile of the unit's pair
  const bool leader = qx == 0;    // issues the pair's MMAs
  const uint16_t pair_mask = (uint16_t)(3u << (rank & ~1u));
  const int cid = (int)cluster_id_x(), ncl = (int)cluster_count_x();

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(sfull, 1);
    mbar_init(sfree, 2 * kFlashSoftWarps);
    mbar_init(pfull, kFlashSoftWarps);
    mbar_init(ptwin, 1);
    mbar_init(pempty, 1);
    mbar_init(ofree, 2 * kFlashSoftWarps);
    for (int q = 0; q < 4; ++q) mbar_init(&xb[q], 2);
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
    tma_prefetch_desc(&tmQ);
    tma_prefetch_desc(&tmK);
    tma_prefetch_desc(&tmXhi);
    tma_prefetch_desc(&tmXlo);
  }
  if (warp == 1) {  // one warp of each CTA of the pair allocates both TMEMs together
    tmem_alloc_2sm(tmem_slot, 512);
    tmem_relinquish_2sm();
  }
  tc_fence_before();
  cluster_sync();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  // the even CTA's barriers, as seen from this CTA
  const uint32_t l_full = cluster_map(smem_u32(full), rank & ~1u);
  const uint32_t l_sfree = cluster_map(smem_u32(sfree), rank & ~1u);
  const uint32_t l_ofree = cluster_map(smem_u32(ofree), rank & ~1u);
  const uint32_t l_ptwin = cluster_map(smem_u32(ptwin), rank & ~1u);

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------------------ TMA producer
      // Both CTAs load their halves of every stage into their own shared memory; all the
      // copies complete on the even CTA's full barrier, which it arms for both.
      int stage = 0;
      uint32_t phase = 0;
      uint32_t armed = 0, armed_par = 0;
      bool bad = false;
      auto acquire = [&](uint32_t bytes) -> uint8_t* {
        if (!mbar_wait(&empty[stage], phase ^ 1)) {
          dev_set_error(f.err, DEV_WAIT_TIMEOUT, 300);
          *abort_flag = 1;
          bad = true;
          return nullptr;
        }
        if (leader) {
          mbar_arrive_expect_tx(&full[stage], 2 * bytes);
          armed |= 1u << stage;
          armed_par = (armed_par & ~(1u << stage)) | (phase << stage);
        }
        return smem + stage * S::kStageBytes;
      };
      auto advance = [&]() {
        if (++stage == kStages) {
          stage = 0;
          phase ^= 1;
        }
      };
      for (int u = cid; u < f.nunits && !bad && !*abort_flag; u += ncl) {
        const FlashUnit w = flash_pair_unit(f, u, qx);
        const int32_t qrow =
            (int32_t)(f.q_row0 + (int64_t)w.b * (f.q_pitch > 0 ? f.q_pitch : f.t)) + w.tm * kBM;
        const int32_t krow =
            (int32_t)(f.k_row0 + (int64_t)(f.kdiv > 0 ? w.b / f.kdiv : w.b) * f.N);
        // X^T rows of this CTA: hi rows [D2/2 x, +D2/2) (K~ in the even CTA, V in the odd one),
        // lo rows [D2/4 x, +D2/4) of K~
        const int32_t xrow = f.xbase_row + (w.b / f.bdiv) * D2;
        const int32_t xhi = xrow + (D2 / 2) * (int32_t)qx;
        const int32_t xlo = xrow + (D2 / 4) * (int32_t)qx;
        const int J = w.j1 - w.j0;
        for (int jj = 0; jj <= J && !bad; ++jj) {
          if (jj < J) {
            // keys [kKeys/2 x, +kKeys/2) of the tile: rows x of the S operand B
            const int32_t kr = krow + (w.j0 + jj) * kKeys + (kKeys / 2) * (int32_t)qx;
            for (int pass = 0; pass < 3 && !bad; ++pass) {
              const int32_t qoff = pass == 2 ? f.D : 0;  // (q_hi,k_hi), (q_hi,k_lo), (q_lo,k_hi)
              const int32_t koff = pass == 1 ? f.D : 0;
              for (int c = 0; c < qchunks; ++c) {
                uint8_t* sa = acquire(S::kQBytes + S::kKBytes);  // this CTA's bytes
                if (sa == nullptr) break;
                const uint32_t bar = l_full + 8u * (uint32_t)stage;
                tma_load_2d_2sm(sa, &tmQ, bar, qoff + c * kBK, qrow);
                tma_load_2d_2sm(sa + S::kQBytes, &tmK, bar, koff + c * kBK, kr);
                advance();
              }
            }
          }
          if (jj >= 1) {
            const int j = w.j0 + jj - 1;
            const int nch = flash_chunks<kKeys>(f, j);
            for (int c = 0; c < nch; ++c) {
              uint8_t* sa = acquire(S::kXhiBytes + S::kXloBytes);
              if (sa == nullptr) break;
              const int32_t x = j * kKeys + c * kBK;
              const uint32_t bar = l_full + 8u * (uint32_t)stage;
              tma_load_2d_2sm(sa, &tmXhi, bar, x, xhi);
              tma_load_2d_2sm(sa + S::kXhiBytes, &tmXlo, bar, (int32_t)(f.Np + x), xlo);
              advance();
            }
          }
        }
      }
      // every slot released by the even CTA's MMAs before the CTA may leave
      for (int i = 0; i < kStages && !bad && !*abort_flag; ++i) {
        if (!mbar_wait(&empty[stage], phase ^ 1)) {
          dev_set_error(f.err, DEV_WAIT_TIMEOUT, 301);
          *abort_flag = 1;
          bad = true;
          break;
        }
        advance();
      }
      if (bad || *abort_flag) {
        for (int s = 0; s < kStages; ++s)
          if (armed & (1u << s)) (void)mbar_wait_cluster(&full[s], (armed_par >> s) & 1);
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && !leader) {
      // ------------------------------------------------------------ odd CTA: P readiness relay
      uint32_t n = 0;
      for (int u = cid; u < f.nunits && !*abort_flag; u += ncl) {
        const FlashUnit w = flash_pair_unit(f, u, qx);
        bool bad = false;
        for (int i = 0; i < w.j1 - w.j0; ++i, ++n) {
          if (!mbar_wait(pfull, n & 1)) {
            dev_set_error(f.err, DEV_WAIT_TIMEOUT, 315);
            *abort_flag = 1;
            bad = true;
            break;
          }
          mbar_arrive_cluster(l_ptwin);
        }
        if (bad) break;
      }
    }
    if (lane == 0 && leader) {
      // ------------------------------------------------------------ MMA issuer (2-SM)
      const uint32_t idesc_s = idesc_f16(2 * kBM, kKeys, EX ? 0 : 1);  // fp16 (EX) or bf16 q, k
      const uint32_t idesc_hi = idesc_f16(2 * kBM, D2, 0);         // fp16 P, X^T hi
      const uint32_t idesc_lo = idesc_f16(2 * kBM, D2 / 2, 0);     // fp16 P, X^T lo (key half)
      const uint32_t s_tmem = tmem_base;
      const uint32_t o_tmem = tmem_base + 256;
      const uint32_t p_smem = smem_u32(smem + S::kPOffset);
      int stage = 0;
      uint32_t phase = 0;
      uint32_t n_s = 0, n_px = 0, n_units = 0;
      bool issued = false, bad = false;
      auto fail = [&](int where) {
        dev_set_error(f.err, DEV_WAIT_TIMEOUT, where);
        *abort_flag = 1;
        bad = true;
      };
      for (int u = cid; u < f.nunits && !bad && !*abort_flag; u += ncl) {
        const FlashUnit w = flash_pair_unit(f, u, qx);
        const int J = w.j1 - w.j0;
        for (int jj = 0; jj <= J && !bad; ++jj) {
          if (jj < J) {
            if (n_s > 0 && !mbar_wait_cluster(sfree, (n_s - 1) & 1)) {
              fail(310);
              break;
            }
            tc_fence_after();
            const int nst = 3 * qchunks;
            for (int st = 0; st < nst; ++st) {
              if (!mbar_wait_cluster(&full[stage], phase)) {
                fail(311);
                break;
              }
              tc_fence_after();
              const uint32_t sa = smem_u32(smem + stage * S::kStageBytes);
              const uint64_t ad = sdesc_k_sw128(sa);
              const uint64_t bd = sdesc_k_sw128(sa + S::kQBytes);
#pragma unroll
              for (int k = 0; k < kBK / 16; ++k)
                tc_mma_f16_2sm(s_tmem, ad + 2 * k, bd + 2 * k, idesc_s,
                               (st > 0 || k > 0) ? 1u : 0u);
              issued = true;
              tc_commit_2sm_mc(&empty[stage], pair_mask);
              if (++stage == kStages) {
                stage = 0;
                phase ^= 1;
              }
            }
            if (bad) break;
            tc_commit_2sm_mc(sfull, pair_mask);
            ++n_s;
          }
          if (jj >= 1) {
            const int j = w.j0 + jj - 1;
            const int nch = flash_chunks<kKeys>(f, j);
            if (jj == 1 && n_units > 0 && !mbar_wait_cluster(ofree, (n_units - 1) & 1)) {
              fail(312);
              break;
            }
            if (!mbar_wait(pfull, n_px & 1) || !mbar_wait_cluster(ptwin, n_px & 1)) {
              fail(313);
              break;
            }
            tc_fence_after();
            for (int c = 0; c < nch; ++c) {
              if (!mbar_wait_cluster(&full[stage], phase)) {
                fail(314);
                break;
              }
              tc_fence_after();
              const uint32_t sa = smem_u32(smem + stage * S::kStageBytes);
              const uint64_t pd = sdesc_k_sw128(p_smem + c * S::kPChunkBytes);
              const uint64_t hd = sdesc_k_sw128(sa);
              const uint64_t ld = sdesc_k_sw128(sa + S::kXhiBytes);
#pragma unroll
              for (int k = 0; k < kBK / 16; ++k)
                tc_mma_f16_2sm(o_tmem, pd + 2 * k, hd + 2 * k, idesc_hi,
                               (jj > 1 || c > 0 || k > 0) ? 1u : 0u);
#pragma unroll
              for (int k = 0; k < kBK / 16; ++k)
                tc_mma_f16_2sm(o_tmem, pd + 2 * k, ld + 2 * k, idesc_lo, 1u);
              if constexpr (EX) {  // + P_lo X^T hi
                const uint64_t pld =
                    sdesc_k_sw128(p_smem + (S::kPChunks + c) * S::kPChunkBytes);
#pragma unroll
                for (int k = 0; k < kBK / 16; ++k)
                  tc_mma_f16_2sm(o_tmem, pld + 2 * k, hd + 2 * k, idesc_hi, 1u);
              }
              tc_commit_2sm_mc(&empty[stage], pair_mask);
              if (++stage == kStages) {
                stage = 0;
                phase ^= 1;
              }
            }
            if (bad) break;
            tc_commit_2sm_mc(pempty, pair_mask);
            ++n_px;
          }
        }
        ++n_units;
      }
      if ((bad || *abort_flag) && issued) {
        tc_commit_2sm_mc(drain, (uint16_t)(1u << rank));
        (void)mbar_wait(drain, 0);
      }
    }
  } else {
    // -------------------------------------------------------------- softmax / output warps
    const int sw = warp - 2;
    const int quarter = warp & 3;  // TMEM lanes [32 quarter, 32 quarter + 32)
    const int half = sw >> 2;      // S columns [128 half, +128), O columns [kOCols half, +kOCols)
    const int row = quarter * 32 + lane;
    const uint32_t lane_base = tmem_base + ((uint32_t)(quarter * 32) << 16);
    float* kw = reinterpret_cast<float*>(smem + S::kKinvOffset) + sw * 128;
    float* xch = reinterpret_cast<float*>(smem + S::kXchOffset);  // [2][2][128]
    uint8_t* pbuf = smem + S::kPOffset;
    constexpr float kLog2e = 1.4426950408889634f;
    uint32_t n_sf = 0, n_pe = 0, n_pf = 0, n_x = 0;
    bool bad = false;
    auto wait_all = [&](uint64_t* bar, uint32_t parity, int where) -> bool {
      bool ok = mbar_wait(bar, parity);
      ok = __all_sync(0xffffffffu, ok);
      if (!ok) {
        if (lane == 0) {
          dev_set_error(f.err, DEV_WAIT_TIMEOUT, where);
          *abort_flag = 1;
        }
        bad = true;
      }
      return ok;
    };
    // Exchanges one value per row with the other warp of this lane quarter; returns its value.
    auto exchange = [&](float mine, int where) -> float {
      float* slot = xch + (n_x & 1) * 256;
      slot[half * 128 + row] = mine;
      __syncwarp();
      if (lane == 0) mbar_arrive(&xb[quarter]);
      const bool ok = wait_all(&xb[quarter], n_x & 1, where);
      ++n_x;
      return ok ? slot[(1 - half) * 128 + row] : mine;
    };

    for (int u = cid; u < f.nunits && !bad && !warp_flag(abort_flag); u += ncl) {
      const FlashUnit w = flash_pair_unit(f, u, qx);
      const int J = w.j1 - w.j0;
      float m_run = -INFINITY, l_part = 0.f;
      for (int jj = 0; jj < J; ++jj) {
        const int j = w.j0 + jj;
        const int key0 = j * kKeys + kCols * half;  // first key of this warp's columns
        float kv[kCols / 32];
#pragma unroll
        for (int e = 0; e < kCols / 32; ++e) {
          const int key = key0 + lane + 32 * e;
          kv[e] = key < f.N ? f.kinv[(int64_t)w.b * f.N + key] * kLog2e : 0.f;
        }
        if (!wait_all(sfull, n_sf & 1, 320)) break;
        ++n_sf;
        tc_fence_after();
        float v[kCols];
#pragma unroll
        for (int g = 0; g < kCols / 32; ++g) {
          float tmp[32];
          tmem_ld32(lane_base + (uint32_t)(kCols * half + 32 * g), tmp);
#pragma unroll
          for (int e = 0; e < 32; ++e) v[32 * g + e] = tmp[e];
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive_cluster(l_sfree);  // the even CTA's, for both CTAs
        // scale per key (log2 units), mask keys past N, tile max
#pragma unroll
        for (int e = 0; e < kCols / 32; ++e) kw[lane + 32 * e] = kv[e];
        __syncwarp();
        const int cvalid = f.N - key0;
        float mx = -INFINITY;
#pragma unroll
        for (int c = 0; c < kCols; c += 4) {
          const float4 k4 = *reinterpret_cast<const float4*>(kw + c);
          v[c] = c < cvalid ? v[c] * k4.x : -INFINITY;
          v[c + 1] = c + 1 < cvalid ? v[c + 1] * k4.y : -INFINITY;
          v[c + 2] = c + 2 < cvalid ? v[c + 2] * k4.z : -INFINITY;
          v[c + 3] = c + 3 < cvalid ? v[c + 3] * k4.w : -INFINITY;
          mx = fmaxf(mx, fmaxf(fmaxf(v[c], v[c + 1]), fmaxf(v[c + 2], v[c + 3])));
        }
        __syncwarp();
        mx = fmaxf(mx, exchange(mx, 321));
        if (bad) break;
        // Both warps of the quarter hold the same (m_run, mx), so they take the same decision.
        bool rescale = false;
        float fac = 1.f;
        if (m_run == -INFINITY) {
          m_run = mx;
        } else if (mx > m_run + kRescaleLog2) {
          fac = exp2f(m_run - mx);
          m_run = mx;
          l_part *= fac;
          rescale = true;
        }
        // probabilities (fp16, <= 2^8) into registers as packed pairs; l from the rounded values
        // (EX: hi and lo = fp16(p - hi), l from hi + lo)
        uint32_t pk[kCols / 2];
        uint32_t pkl[EX ? kCols / 2 : 1];
#pragma unroll
        for (int c = 0; c < kCols; c += 2) {
          const float p0 = exp2f(v[c] - m_run), p1 = exp2f(v[c + 1] - m_run);
          const __half2 h = __floats2half2_rn(p0, p1);
          const float2 r = __half22float2(h);
          pk[c / 2] = *reinterpret_cast<const uint32_t*>(&h);
          if constexpr (EX) {
            const __half2 lo = __floats2half2_rn(p0 - r.x, p1 - r.y);
            const float2 rl = __half22float2(lo);
            l_part += (r.x + rl.x) + (r.y + rl.y);
            pkl[c / 2] = *reinterpret_cast<const uint32_t*>(&lo);
          } else {
            l_part += r.x + r.y;
          }
        }
        // The previous PX must be complete before P is overwritten or O is rescaled.
        if (n_pf > n_pe) {
          if (!wait_all(pempty, n_pe & 1, 322)) break;
          ++n_pe;
          tc_fence_after();
        }
        // tcgen05.ld / st are warp-collective: the warp rescales when any of its rows needs it
        // (rows that do not have fac = 1).
        if (__any_sync(0xffffffffu, rescale)) {
#pragma unroll
          for (int g = 0; g < kOCols / 32; ++g) {
            const uint32_t ta = lane_base + 256u + (uint32_t)(kOCols * half + 32 * g);
            float o[32];
            tmem_ld32(ta, o);
#pragma unroll
            for (int e = 0; e < 32; ++e) o[e] *= fac;
            tmem_st32(ta, o);
          }
        }
        // P row `row`, keys [kCols half, +kCols): chunks kCols/64 * half + q of the P tile
        // (EX: the lo values in the same chunks of the second tile, kPChunks further).
#pragma unroll
        for (int q = 0; q < kCols / 64; ++q) {
          const int chunk = (kCols / 64) * half + q;
          uint4* dst = reinterpret_cast<uint4*>(pbuf + chunk * S::kPChunkBytes + row * 128);
#pragma unroll
          for (int un = 0; un < 8; ++un) {
            const int base = (64 * q + 8 * un) / 2;
            dst[un ^ (row & 7)] = make_uint4(pk[base], pk[base + 1], pk[base + 2], pk[base + 3]);
          }
          if constexpr (EX) {
            uint4* dl = reinterpret_cast<uint4*>(pbuf + (S::kPChunks + chunk) * S::kPChunkBytes +
                                                 row * 128);
#pragma unroll
            for (int un = 0; un < 8; ++un) {
              const int base = (64 * q + 8 * un) / 2;
              dl[un ^ (row & 7)] =
                  make_uint4(pkl[base], pkl[base + 1], pkl[base + 2], pkl[base + 3]);
            }
          }
        }
        fence_proxy_async_smem();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(pfull);
        ++n_pf;
      }
      if (bad) break;
      // ---- unit output: wait for the last PX, drain O, hand TMEM back, store.
      if (n_pf > n_pe) {
        if (!wait_all(pempty, n_pe & 1, 323)) break;
        ++n_pe;
      }
      tc_fence_after();
      float o[kOCols];
#pragma unroll
      for (int g = 0; g < kOCols / 32; ++g) {
        float tmp[32];
        tmem_ld32(lane_base + 256u + (uint32_t)(kOCols * half + 32 * g), tmp);
#pragma unroll
        for (int e = 0; e < 32; ++e) o[32 * g + e] = tmp[e];
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(l_ofree);
      const float l_tot = l_part + exchange(l_part, 324);
      if (bad) break;
      const int r = w.tm * kBM + row;
      if (r < f.t) {
        const int64_t orow = ((int64_t)w.split * f.nb + w.b) * f.t + r;
        float4* dst = reinterpret_cast<float4*>(f.O + orow * D2 + kOCols * half);
#pragma unroll
        for (int c = 0; c < kOCols; c += 4) dst[c / 4] = make_float4(o[c], o[c + 1], o[c + 2], o[c + 3]);
        if (half == 0) f.stats[orow] = make_float2(m_run, l_tot);
      }
    }
  }

  tc_fence_before();
  // Neither CTA frees its TMEM while the even CTA's MMAs may still write it, nor leaves while
  // the other may still copy into or arrive on its shared memory.
  cluster_sync();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_2sm(tmem_base, 512);
  }
}

// Splits the key tiles so that the units fill the SMs in near-whole waves.
inline int flash_split(int64_t base_units, int tiles_k, int num_sms, int max_split) {
  int best = 1;
  double best_cost = 1e300;
  for (int s = 1; s <= std::min(tiles_k, max_split); ++s) {
    const int64_t units = base_units * s;
    const double waves = (double)((units + num_sms - 1) / num_sms);
    const double per_unit = (double)((tiles_k + s - 1) / s) + 0.25;
    const double cost = waves * per_unit;
    if (cost < best_cost - 1e-9) {
      best_cost = cost;
      best = s;
    }
  }
  return best;
}

// Q: [nb*t][2D] bf16 (hi | lo), K: [nb*N][2D] bf16 (hi | lo), XT: [H*2d][2*Np] fp16 (hi | lo);
// EX: Q and K fp16 hi | lo, key tiles of S::kKeys = 128 (f.tiles_k counts those).
// The kernel runs on CTA pairs (clusters of two): f.nunits counts (query-tile pair, key split,
// batch) units.
template <int D2, bool EX = false>
inline cudaError_t launch_ca_flash(const Operand2D& Q, const Operand2D& K, const Operand2D& XT,
                                   const FlashParams& f, int num_sms, cudaStream_t stream) {
  using S = FlashSmem<D2, EX>;
  if (f.D <= 0 || f.D % kBK != 0 || f.t <= 0 || f.N <= 0 || f.Np % kBK != 0 || f.Np < f.N ||
      f.nunits <= 0)
    return cudaErrorInvalidValue;
  // boxes per CTA of a pair: its q rows, half of the k tile, half of the X^T hi and lo rows
  CUtensorMap tq, tk, thi, tlo;
  if (!make_tmap(&tq, Q, kBM) || !make_tmap(&tk, K, S::kKeys / 2) ||
      !make_tmap(&thi, XT, D2 / 2) || !make_tmap(&tlo, XT, D2 / 4))
    return cudaErrorInvalidValue;
  auto kern = ca_flash_kernel<D2, EX>;
  static thread_local int clusters = 0;  // resident CTA pairs (per instantiation)
  if (clusters == 0) {
    cudaError_t e =
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, S::kBytes);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t q = {};
    q.gridDim = dim3(2 * std::max(1, num_sms / 2), 1, 1);
    q.blockDim = dim3(kFlashThreads, 1, 1);
    q.dynamicSmemBytes = S::kBytes;
    cudaLaunchAttribute qa[1];
    qa[0].id = cudaLaunchAttributeClusterDimension;
    qa[0].val.clusterDim.x = 2;
    qa[0].val.clusterDim.y = 1;
    qa[0].val.clusterDim.z = 1;
    q.attrs = qa;
    q.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, kern, &q) != cudaSuccess || n < 1) {
      cudaGetLastError();
      n = num_sms / 2;
    }
    clusters = std::max(1, std::min(n, num_sms / 2));
  }
  cudaLaunchConfig_t cfg = {};
  cfg.blockDim = dim3(kFlashThreads, 1, 1);
  cfg.dynamicSmemBytes = S::kBytes;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cfg.gridDim = dim3(2 * (unsigned)std::min(f.nunits, clusters), 1, 1);
  return cudaLaunchKernelEx(&cfg, kern, tq, tk, thi, tlo, f);
}

// 2d = 512 (head dim 256): the same computation on clusters of four CTAs, two query tiles x
// two column halves; the CTAs of a query tile split the O columns and take turns computing S,
// the two CTAs of a half run their MMAs as one 2-SM MMA over both query tiles (ca_pair.cu). Q, K as for launch_ca_flash;
// XT: [H*512][2*Np] fp16 (hi | lo). f.nunits counts (query-tile pair, key split, batch) units.
// num_sms: SMs of the device (four per cluster).
// one_pass: q, k as fp16 hi | lo with S from the hi parts only (one MMA pass) and repair
// candidates in f.cand_key / f.cand_c for ca_topk_repair; else 3-pass split-bf16 scores.
cudaError_t launch_ca_pair(const Operand2D& Q, const Operand2D& K, const Operand2D& XT,
                           const FlashParams& f, int num_sms, cudaStream_t stream,
                           bool one_pass = false);
// Four-CTA clusters of that kernel that can be resident at once (its persistent grid size).
int ca_pair_clusters(int num_sms);

// Top-k repair of one-pass scores: for each (b, row), over the splits whose running max is within
// `cut` (log2 units) of the row's largest, each candidate's exact logit
// e = kinv (q_hi + q_lo) . (k_hi + k_lo) log2 e replaces the one-pass value c that the fused
// kernel used: delta = 2^(e - m) - 2^(c - m) is added to the split's l and delta X_key to its O.
// A split whose weight outside its candidates exceeds `guard` of its l is recomputed exactly
// over all its keys. Candidates below 2^-cut of the row's largest weight are left as they are.
// Deterministic: splits and candidates in a fixed order, one warp per row.
struct TopkRepairParams {
  const __half* q = nullptr;          // [nb * t][2D] fp16 hi | lo (times the q scale)
  const __half* k = nullptr;          // [nb * N][2D] fp16 hi | lo
  const float* kinv = nullptr;        // [nb][N]: logit scale / (q scale |k~|)
  const __nv_bfloat16* X = nullptr;   // KV-head h0's rows [N][3d]: hi [0, 2d), lo of K~ [2d, 3d)
  float* O = nullptr;                 // [nsplit][nb][t][2d]
  float2* stats = nullptr;            // [nsplit][nb][t]: (m log2 units, l)
  const int* cand_key = nullptr;      // [nsplit][nb][t][nlists][kTopK]
  const float* cand_c = nullptr;
  int32_t D = 0, d = 0, t = 0, N = 0, nb = 0, nsplit = 1, bdiv = 1, nlists = 0;
  int32_t tiles_k = 0, keys_per_tile = 256;  // the fused kernel's key tiles and splits
  float cut = 24.f;
  float guard = 1.f / 64.f;
};
cudaError_t launch_ca_topk_repair(const TopkRepairParams& f, int d2, cudaStream_t stream);

}  // namespace still
