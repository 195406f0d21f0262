// Cross-attention of one compactor layer for 2d = 512 (head dim 256), flash-style, for sm_103a
// (App. A, "Cross-attention"):
//
//   S(m, k)  = scale * q_m . k_k / |k~_k|          3-pass split-bf16 tcgen05.mma, fp32 in TMEM
//   P(m, k)  = 2^(S(m, k) log2e - M(m))             online row softmax over 256-key tiles
//   O(m, :)  = sum_k P(m, k) X(k, :)                unnormalised, with the row sum l per split
//
// The accumulator of a 128-row query tile over 2d = 512 columns fills a whole TMEM (512
// fp32 columns), leaving no room for S. Two CTAs therefore share each query tile: CTA half r
// keeps the O columns of features [128 r, 128 r + 128) of K~ and of V (256 columns, TMEM
// [256, 512)) and computes S for every other 256-key tile (TMEM [0, 256)). The CTA that owns
// a tile forms its fp16 probabilities, sends the tile's running row maximum to its peer as
// soon as it is decided, and copies the probability tile into the peer's shared memory with a
// bulk DSMEM copy; both CTAs then accumulate P X for their column half. S and P never reach
// global memory.
//
// A work unit (batch b = (KV-head, cross head), two 128-row query tiles, key split) runs on
// a cluster of four CTAs, rank = 2 r + x: query tile x of the pair, column half r. The two
// CTAs of one half (ranks 2 r and 2 r + 1, a CTA pair) need the same k tiles and X^T columns
// in the same order, so their MMAs run as one 2-SM tcgen05.mma (cta_group::2, M = 256)
// issued by the even CTA: each CTA holds its own query rows (or P rows) and one half of the
// keys (or of the X^T rows) of every stage, and each SM's tensor core reads the other half
// from its twin. Per SM this halves the shared-memory traffic of the B operand and its loads,
// which is what bounds the S stream at M = 128 (128-byte/clock shared memory, read by the MMA
// and written by TMA for every stage).
//
// Both CTAs apply the same running-maximum sequence (the owner's decision travels with the
// tile), so their O halves, and the row sums each accumulates from its own tiles, stay on one
// reference. The running max moves only when a tile raises it by more than kRescaleLog2
// (log2 units), so P <= 2^8 fits fp16.
//
// Tensor-pipe issue order per CTA: before each of its own S tiles j, every P X tile up to
// j - 2 (own or peer), so that a P buffer is never held behind a long S computation; the
// softmax of tile j overlaps the peer's S computation of tile j + 1.
//
// Synchronisation inside a CTA pair: every stage's copies of both CTAs complete on the even
// CTA's full barrier (cta_group::2 TMA); its MMA commits arrive on both CTAs' empty, sfull and
// pempty barriers; both CTAs' softmax warps arrive on its sfree and ofree barriers, and the
// odd CTA's warp 1 forwards each completion of its pfull barrier (its P and O rescale).
//
// Synchronisation between the two CTAs of a query tile (all waits bounded):
//   mmsg   the owner's per-row running max of a tile (st.shared::cluster + remote arrive)
//   pfull  P of the tile in this CTA's buffer and O rescaled: 8 local arrivals; for a peer
//          tile one of them expects the 64 KB that the peer's bulk copies complete
//   rfree  the peer's P X of the previous tile is done (its P buffer may be overwritten)
//   lmsg   the peer's row sum at the end of a unit
//
// Output per split: unnormalised O rows (natural feature order) and (m, l), m in log2 units;
// ca_merge_kernel combines the splits in a fixed order.
//
// CTA = 10 warps: 0 TMA producer, 1 MMA issuer (even CTA) or P relay (odd CTA) and TMEM
// allocation, 2..9 softmax / output.
#include <algorithm>

#include "ca_flash.cuh"

namespace still {

namespace {

constexpr int kPairKeys = 256;   // keys per S tile
constexpr int kPairOCols = 256;  // O columns per CTA
constexpr uint32_t kPairPBytes = kBM * kPairKeys * 2;  // one fp16 P tile, 64 KB
constexpr int kPairCluster = 4;  // CTAs per cluster: two query tiles x two column halves
// S stages of an own tile issued after the own P X tile j - 2 (all of them: P X first)
constexpr int kPxTail = 12;

struct PairSmem {
  // Per CTA: its 128 query rows and half of the keys (or of the X^T rows) of a stage; the
  // 2-SM MMA reads the other half from the twin's shared memory at the same offset.
  static constexpr int kQBytes = kBM * kBK * 2;                // q chunk, 16 KB
  static constexpr int kKBytes = (kPairKeys / 2) * kBK * 2;    // half a k chunk, 16 KB
  static constexpr int kXBox = 128 * kBK * 2;                  // one 128-row X^T box, 16 KB
  static constexpr int kXloBytes = 64 * kBK * 2;               // half the lo box, 8 KB
  static constexpr int kStageBytes = kQBytes + kKBytes;        // 32 KB
  static constexpr int kStages = 4;
  static constexpr int kPChunkBytes = kBM * kBK * 2;           // 128 rows x 64 keys fp16
  static constexpr int kPOffset = kStages * kStageBytes;
  static constexpr int kKinvOffset = kPOffset + (int)kPairPBytes;            // [8][128] f32
  static constexpr int kXchOffset = kKinvOffset + kFlashSoftWarps * 128 * 4;  // [2][2][128]
  static constexpr int kMsgOffset = kXchOffset + 2 * 2 * 128 * 4;             // [2][128] m
  static constexpr int kLslotOffset = kMsgOffset + 2 * 128 * 4;              // [128] l
  static constexpr int kBarOffset = kLslotOffset + 128 * 4;
  static constexpr int kBytes = kBarOffset + 256 + 1024;
  static_assert(kXBox + kXloBytes <= kStageBytes, "an X^T chunk fits a stage");
  static_assert(kBytes <= 232448, "shared memory budget");
};

// Owner of tile jj of a unit: the CTAs of half (jj & 1). Before its own tile jj a CTA issues
// every P X tile up to jj - 2; the remaining ones after its last own tile.
__device__ __forceinline__ bool pair_owner(int jj, uint32_t half) {
  return (uint32_t)(jj & 1) == half;
}

// Unit u of the four-CTA clusters: query tiles 2 m and 2 m + 1 (m fastest), then the key
// split, then the batch; this CTA takes query tile 2 m + x. A tile past the last one (odd
// tile count) is computed and not stored.
__device__ __forceinline__ FlashUnit pair_unit(const FlashParams& f, int u, uint32_t x) {
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

// TK: one-pass fp16 scores (q_hi . k_hi) with repair candidates; else 3-pass split-bf16.
template <bool TK>
__global__ void __launch_bounds__(kFlashThreads, 1)
    ca_pair_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                   const __grid_constant__ CUtensorMap tmX, const FlashParams f) {
  using S = PairSmem;
  constexpr int kPasses = TK ? 1 : 3;
  constexpr int kStages = S::kStages;
  constexpr int kCols = kPairKeys / 2;   // S columns per softmax warp (its half of the tile)
  constexpr int kOCols = kPairOCols / 2;  // O columns per softmax warp
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + S::kBarOffset);  // leader: stage loaded
  uint64_t* empty = full + kStages;   // stage consumed (the leader's commit, in both CTAs)
  uint64_t* sfull = empty + kStages;  // own S tile complete in TMEM
  uint64_t* sfree = sfull + 1;        // leader: own S tile drained in both CTAs
  uint64_t* pfull = sfree + 1;        // P of the tile in the local buffer, O rescaled
  uint64_t* ptwin = pfull + 1;        // leader: the same in the twin
  uint64_t* pempty = ptwin + 1;       // P X complete
  uint64_t* ofree = pempty + 1;       // leader: O drained in both CTAs at the end of a unit
  uint64_t* xb = ofree + 1;           // [4] row-value exchange per lane quarter
  uint64_t* mmsg = xb + 4;            // peer's running max of a tile (4 remote arrivals)
  uint64_t* rfree = mmsg + 1;         // peer's P X of the previous tile done (8 remote)
  uint64_t* lmsg = rfree + 1;         // peer's row sums at the end of a unit (4 remote)
  uint64_t* drain = lmsg + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int qchunks = f.D / kBK;
  const uint32_t rank = cluster_ctarank();
  const uint32_t qx = rank & 1u;      // query tile of the unit's pair
  const uint32_t chalf = rank >> 1;   // column half; S owner parity
  const uint32_t peer = rank ^ 2u;    // same query tile, other half: the P exchange
  const uint32_t twin = rank ^ 1u;    // same half, other query tile: the 2-SM MMA pair
  const bool leader = qx == 0;        // issues the pair's MMAs
  const uint16_t pair_mask = (uint16_t)((1u << rank) | (1u << twin));
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
    mbar_init(mmsg, 4);
    mbar_init(rfree, kFlashSoftWarps);
    mbar_init(lmsg, 4);
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
    tma_prefetch_desc(&tmQ);
    tma_prefetch_desc(&tmK);
    tma_prefetch_desc(&tmX);
  }
  if (warp == 1) {  // one warp of each CTA of the pair allocates both TMEMs together
    tmem_alloc_2sm(tmem_slot, 512);
    tmem_relinquish_2sm();
  }
  tc_fence_before();
  // Every CTA's barriers are initialised before any arrives on another's.
  cluster_sync();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  // the leader's barriers, as seen from this CTA
  const uint32_t l_full = cluster_map(smem_u32(full), rank & ~1u);
  const uint32_t l_sfree = cluster_map(smem_u32(sfree), rank & ~1u);
  const uint32_t l_ofree = cluster_map(smem_u32(ofree), rank & ~1u);
  const uint32_t l_ptwin = cluster_map(smem_u32(ptwin), rank & ~1u);

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------------------ TMA producer
      // Both CTAs load their halves of every stage into their own shared memory; all the
      // copies complete on the leader's full barrier, which the leader arms for both.
      int stage = 0;
      uint32_t phase = 0;
      uint32_t armed = 0, armed_par = 0;
      bool bad = false;
      auto acquire = [&](uint32_t bytes) -> uint8_t* {
        if (!mbar_wait(&empty[stage], phase ^ 1)) {
          dev_set_error(f.err, DEV_WAIT_TIMEOUT, 400);
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
      const uint32_t fbar = l_full;  // + 8 stage
      for (int u = cid; u < f.nunits && !bad && !*abort_flag; u += ncl) {
        const FlashUnit w = pair_unit(f, u, qx);
        const int32_t qrow =
            (int32_t)(f.q_row0 + (int64_t)w.b * (f.q_pitch > 0 ? f.q_pitch : f.t)) + w.tm * kBM;
        const int32_t krow =
            (int32_t)(f.k_row0 + (int64_t)(f.kdiv > 0 ? w.b / f.kdiv : w.b) * f.N);
        // this half's feature rows of X^T: K~ [128 r, +128) and V [128 r, +128). The leader
        // holds the K~ box, the twin the V box (rows 0..127 and 128..255 of the P X operand
        // B), and each half of the lo box of K~.
        const int32_t xk = f.xbase_row + (w.b / f.bdiv) * 512 + 128 * (int32_t)chalf;
        const int32_t xhi = leader ? xk : xk + 256;
        const int32_t xlo = xk + 64 * (int32_t)qx;
        const int J = w.j1 - w.j0;
        auto produce_px = [&](int i) {
          const int j = w.j0 + i;
          const int nch = flash_chunks<kPairKeys>(f, j);
          for (int c = 0; c < nch && !bad; ++c) {
            uint8_t* sa = acquire(S::kXBox + S::kXloBytes);
            if (sa == nullptr) break;
            const int32_t x = j * kPairKeys + c * kBK;
            const uint32_t bar = fbar + 8u * (uint32_t)stage;
            tma_load_2d_2sm(sa, &tmX, bar, x, xhi);  // 64-row boxes
            tma_load_2d_2sm(sa + S::kXBox / 2, &tmX, bar, x, xhi + 64);
            tma_load_2d_2sm(sa + S::kXBox, &tmX, bar, (int32_t)(f.Np + x), xlo);
            advance();
          }
        };
        int px_next = 0;
        for (int jj = 0; jj < J && !bad; ++jj) {
          if (!pair_owner(jj, chalf)) continue;
          while (px_next <= jj - 3 && !bad) produce_px(px_next++);
          const int32_t kr = krow + (w.j0 + jj) * kPairKeys;
          const int nst = kPasses * qchunks, at = max(0, nst - kPxTail);
          for (int st = 0; st < nst && !bad; ++st) {
            if (st == at)
              while (px_next <= jj - 2 && !bad) produce_px(px_next++);
            const int pass = st / qchunks, c = st % qchunks;
            const int32_t qoff = pass == 2 ? f.D : 0;  // (q_hi,k_hi), (q_hi,k_lo), (q_lo,k_hi)
            const int32_t koff = pass == 1 ? f.D : 0;
            uint8_t* sa = acquire(S::kQBytes + S::kKBytes);
            if (sa == nullptr) break;
            const uint32_t bar = fbar + 8u * (uint32_t)stage;
            tma_load_2d_2sm(sa, &tmQ, bar, qoff + c * kBK, qrow);
            // keys [128 x, +128) of the tile: rows x of the S operand B
            tma_load_2d_2sm(sa + S::kQBytes, &tmK, bar, koff + c * kBK, kr + 128 * (int32_t)qx);
            advance();
          }
        }
        while (px_next < J && !bad) produce_px(px_next++);
      }
      // Every slot released by the leader's MMAs before the CTA may leave (its copies have
      // landed and no commit arrives on its barriers after it exited).
      for (int i = 0; i < kStages && !bad && !*abort_flag; ++i) {
        if (!mbar_wait(&empty[stage], phase ^ 1)) {
          dev_set_error(f.err, DEV_WAIT_TIMEOUT, 401);
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
      // ------------------------------------------------------------ twin: P readiness relay
      // The leader's P X of a tile needs P (and the O rescale) in both CTAs: forward each
      // completion of this CTA's pfull to the leader.
      uint32_t n = 0;
      for (int u = cid; u < f.nunits && !*abort_flag; u += ncl) {
        const FlashUnit w = pair_unit(f, u, qx);
        bool bad = false;
        for (int i = 0; i < w.j1 - w.j0; ++i, ++n) {
          if (!mbar_wait(pfull, n & 1)) {
            dev_set_error(f.err, DEV_WAIT_TIMEOUT, 415);
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
      const uint32_t idesc_s = idesc_f16(2 * kBM, kPairKeys, TK ? 0 : 1);  // fp16 / bf16 q, k
      const uint32_t idesc_hi = idesc_f16(2 * kBM, kPairOCols, 0);  // fp16 P, X^T hi (K~ | V)
      const uint32_t idesc_lo = idesc_f16(2 * kBM, 128, 0);         // fp16 P, X^T lo (K~ half)
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
        const FlashUnit w = pair_unit(f, u, qx);
        const int J = w.j1 - w.j0;
        auto issue_px = [&](int i) {
          const int nch = flash_chunks<kPairKeys>(f, w.j0 + i);
          if (i == 0 && n_units > 0 && !mbar_wait_cluster(ofree, (n_units - 1) & 1)) {
            fail(412);
            return;
          }
          if (!mbar_wait(pfull, n_px & 1) || !mbar_wait_cluster(ptwin, n_px & 1)) {
            fail(413);
            return;
          }
          tc_fence_after();
          for (int c = 0; c < nch; ++c) {
            if (!mbar_wait_cluster(&full[stage], phase)) {
              fail(414);
              return;
            }
            tc_fence_after();
            const uint32_t sa = smem_u32(smem + stage * S::kStageBytes);
            const uint64_t pd = sdesc_k_sw128(p_smem + c * S::kPChunkBytes);
            const uint64_t hd = sdesc_k_sw128(sa);
            const uint64_t ld = sdesc_k_sw128(sa + S::kXBox);
#pragma unroll
            for (int k = 0; k < kBK / 16; ++k)
              tc_mma_f16_2sm(o_tmem, pd + 2 * k, hd + 2 * k, idesc_hi,
                             (i > 0 || c > 0 || k > 0) ? 1u : 0u);
#pragma unroll
            for (int k = 0; k < kBK / 16; ++k)
              tc_mma_f16_2sm(o_tmem, pd + 2 * k, ld + 2 * k, idesc_lo, 1u);
            issued = true;
            tc_commit_2sm_mc(&empty[stage], pair_mask);
            if (++stage == kStages) {
              stage = 0;
              phase ^= 1;
            }
          }
          tc_commit_2sm_mc(pempty, pair_mask);
          ++n_px;
        };
        int px_next = 0;
        for (int jj = 0; jj < J && !bad; ++jj) {
          if (!pair_owner(jj, chalf)) continue;
          while (px_next <= jj - 3 && !bad) issue_px(px_next++);
          if (bad) break;
          if (n_s > 0 && !mbar_wait_cluster(sfree, (n_s - 1) & 1)) {
            fail(410);
            break;
          }
          tc_fence_after();
          const int nst = kPasses * qchunks, at = max(0, nst - kPxTail);
          for (int st = 0; st < nst; ++st) {
            if (st == at) {
              while (px_next <= jj - 2 && !bad) issue_px(px_next++);
              if (bad) break;
            }
            if (!mbar_wait_cluster(&full[stage], phase)) {
              fail(411);
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
        while (px_next < J && !bad) issue_px(px_next++);
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
    const int half = sw >> 2;      // S columns [128 half, +128), O columns [128 half, +128)
    const int row = quarter * 32 + lane;
    const uint32_t lane_base = tmem_base + ((uint32_t)(quarter * 32) << 16);
    float* kw = reinterpret_cast<float*>(smem + S::kKinvOffset) + sw * 128;
    float* xch = reinterpret_cast<float*>(smem + S::kXchOffset);    // [2][2][128]
    float* msg = reinterpret_cast<float*>(smem + S::kMsgOffset);    // [2][128]
    float* lslot = reinterpret_cast<float*>(smem + S::kLslotOffset);  // [128]
    uint8_t* pbuf = smem + S::kPOffset;
    // the peer's copies of this CTA's message slots, barriers and P buffer
    const uint32_t r_msg = cluster_map(smem_u32(msg), peer);
    const uint32_t r_lslot = cluster_map(smem_u32(lslot), peer);
    const uint32_t r_mmsg = cluster_map(smem_u32(mmsg), peer);
    const uint32_t r_rfree = cluster_map(smem_u32(rfree), peer);
    const uint32_t r_lmsg = cluster_map(smem_u32(lmsg), peer);
    const uint32_t r_pfull = cluster_map(smem_u32(pfull), peer);
    const uint32_t r_pbuf = cluster_map(smem_u32(pbuf), peer);
    constexpr float kLog2e = 1.4426950408889634f;
    uint32_t n_sf = 0, n_pe = 0, n_pf = 0, n_x = 0;
    uint32_t n_msent = 0, n_mrecv = 0, n_l = 0;
    uint32_t g = 0;  // P tiles handled so far (both CTAs count the same sequence)
    bool bad = false;
    auto wait_all = [&](uint64_t* bar, uint32_t parity, int where, bool cluster) -> bool {
      bool ok = cluster ? mbar_wait_cluster(bar, parity) : mbar_wait(bar, parity);
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
      const bool ok = wait_all(&xb[quarter], n_x & 1, where, false);
      ++n_x;
      return ok ? slot[(1 - half) * 128 + row] : mine;
    };
    // The previous P X of this CTA is complete (its P buffer and O may be touched); tell the
    // peer, whose next P copy overwrites this buffer.
    auto prev_px_done = [&](int where) -> bool {
      if (n_pf > n_pe) {
        if (!wait_all(pempty, n_pe & 1, where, false)) return false;
        ++n_pe;
        tc_fence_after();
        __syncwarp();
        if (lane == 0) mbar_arrive_cluster(r_rfree);
      }
      return true;
    };
    auto rescale_o = [&](bool rescale, float fac) {
      // tcgen05.ld / st are warp-collective: the warp rescales when any of its rows needs it
      if (__any_sync(0xffffffffu, rescale)) {
#pragma unroll
        for (int gq = 0; gq < kOCols / 32; ++gq) {
          const uint32_t ta = lane_base + 256u + (uint32_t)(kOCols * half + 32 * gq);
          float o[32];
          tmem_ld32(ta, o);
#pragma unroll
          for (int e = 0; e < 32; ++e) o[e] *= fac;
          tmem_st32(ta, o);
        }
      }
    };

    for (int u = cid; u < f.nunits && !bad && !warp_flag(abort_flag); u += ncl) {
      const FlashUnit w = pair_unit(f, u, qx);
      const int J = w.j1 - w.j0;
      float m_run = -INFINITY, l_part = 0.f;
      // TK: the kTopK keys of this row half (own tiles) with the largest weights used
      int tk_key[TK ? kTopK : 1];
      float tk_c[TK ? kTopK : 1];
      float tk_tau = -INFINITY;  // smallest c in the list (-inf while a slot is free)
      int tk_slot = 0;           // its slot
#pragma unroll
      for (int e = 0; e < (TK ? kTopK : 1); ++e) {
        tk_key[e] = -1;
        tk_c[e] = -INFINITY;
      }
      for (int jj = 0; jj < J; ++jj, ++g) {
        const int j = w.j0 + jj;
        if (pair_owner(jj, chalf)) {
          // ---------------- own tile: softmax of S_j
          const int key0 = j * kPairKeys + kCols * half;
          float kv[kCols / 32];
#pragma unroll
          for (int e = 0; e < kCols / 32; ++e) {
            const int key = key0 + lane + 32 * e;
            kv[e] = key < f.N ? f.kinv[(int64_t)w.b * f.N + key] * kLog2e : 0.f;
          }
          if (!wait_all(sfull, n_sf & 1, 420, false)) break;
          ++n_sf;
          tc_fence_after();
          float v[kCols];
#pragma unroll
          for (int gq = 0; gq < kCols / 32; ++gq) {
            float tmp[32];
            tmem_ld32(lane_base + (uint32_t)(kCols * half + 32 * gq), tmp);
#pragma unroll
            for (int e = 0; e < 32; ++e) v[32 * gq + e] = tmp[e];
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive_cluster(l_sfree);  // the leader's, for both CTAs
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
          const float mx_own = mx;
          mx = fmaxf(mx, exchange(mx, 421));
          if (bad) break;
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
          // the tile's running max to the peer, before anything else of this tile
          if (half == 0) {
            st_cluster_f32(r_msg + (uint32_t)(((n_msent & 1) * 128 + row) * 4), m_run);
            __syncwarp();
            if (lane == 0) mbar_arrive_cluster(r_mmsg);
          }
          ++n_msent;
          uint32_t pk[kCols / 2];
#pragma unroll
          for (int c = 0; c < kCols; c += 2) {
            const float p0 = exp2f(v[c] - m_run), p1 = exp2f(v[c + 1] - m_run);
            const __half2 h = __floats2half2_rn(p0, p1);
            const float2 r2 = __half22float2(h);
            pk[c / 2] = *reinterpret_cast<const uint32_t*>(&h);
            l_part += r2.x + r2.y;
          }
          // This CTA's previous P X done (buffer, O) and the peer's (its buffer).
          if (!prev_px_done(422)) break;
          if (g > 0 && !wait_all(rfree, (g - 1) & 1, 423, true)) break;
          rescale_o(rescale, fac);
#pragma unroll
          for (int q = 0; q < kCols / 64; ++q) {
            const int chunk = (kCols / 64) * half + q;
            uint4* dst = reinterpret_cast<uint4*>(pbuf + chunk * S::kPChunkBytes + row * 128);
#pragma unroll
            for (int un = 0; un < 8; ++un) {
              const int base = (64 * q + 8 * un) / 2;
              dst[un ^ (row & 7)] = make_uint4(pk[base], pk[base + 1], pk[base + 2], pk[base + 3]);
            }
          }
          fence_proxy_async_smem();
          tc_fence_before();
          __syncwarp();
          if (lane == 0) {
            // this warp's rows of its two chunks, 4 KB each, into the peer's P buffer
#pragma unroll
            for (int q = 0; q < kCols / 64; ++q) {
              const uint32_t off =
                  (uint32_t)(((kCols / 64) * half + q) * S::kPChunkBytes + quarter * 32 * 128);
              bulk_copy_to_cluster(r_pbuf + off, pbuf + off, 32 * 128, r_pfull);
            }
            mbar_arrive(pfull);
          }
          ++n_pf;
          if constexpr (TK) {
            // This row half's weights, read back from the P tile (the tensor core and the bulk
            // copies only read it; the buffer is written again after this thread's next wait),
            // when the tile holds a logit above the list's smallest: rare once the list holds
            // the row's heavy keys.
            if (mx_own > tk_tau) {
#pragma unroll 1
              for (int q = 0; q < kCols / 64; ++q) {
                const int chunk = (kCols / 64) * half + q;
                const uint4* src =
                    reinterpret_cast<const uint4*>(pbuf + chunk * S::kPChunkBytes + row * 128);
#pragma unroll 1
                for (int un = 0; un < 8; ++un) {
                  const uint4 w4 = src[un ^ (row & 7)];
                  const uint32_t wv[4] = {w4.x, w4.y, w4.z, w4.w};
#pragma unroll
                  for (int e = 0; e < 8; ++e) {
                    const uint16_t hb = (uint16_t)(wv[e >> 1] >> (16 * (e & 1)));
                    const float p = __half2float(__ushort_as_half(hb));
                    if (p > 0.f) {
                      const float c = m_run + log2f(p);
                      if (c > tk_tau) {
                        const int key = key0 + 64 * q + 8 * un + e;
#pragma unroll
                        for (int sl = 0; sl < kTopK; ++sl)
                          if (sl == tk_slot) {
                            tk_key[sl] = key;
                            tk_c[sl] = c;
                          }
                        tk_tau = tk_c[0];
                        tk_slot = 0;
#pragma unroll
                        for (int sl = 1; sl < kTopK; ++sl)
                          if (tk_c[sl] < tk_tau) {
                            tk_tau = tk_c[sl];
                            tk_slot = sl;
                          }
                      }
                    }
                  }
                }
              }
            }
          }
        } else {
          // ---------------- peer tile: its running max, O rescale, P arrives by bulk copy
          if (!wait_all(mmsg, n_mrecv & 1, 424, true)) break;
          const float m_new = msg[(n_mrecv & 1) * 128 + row];
          ++n_mrecv;
          bool rescale = false;
          float fac = 1.f;
          if (m_run != -INFINITY && m_new != m_run) {
            fac = exp2f(m_run - m_new);
            l_part *= fac;
            rescale = true;
          }
          m_run = m_new;
          if (!prev_px_done(425)) break;
          rescale_o(rescale, fac);
          tc_fence_before();
          __syncwarp();
          if (lane == 0) {
            if (sw == 0)
              mbar_arrive_expect_tx(pfull, kPairPBytes);
            else
              mbar_arrive(pfull);
          }
          ++n_pf;
        }
      }
      if (bad) break;
      // ---- unit output: wait for the last P X, drain O, hand TMEM back, store.
      if (!prev_px_done(426)) break;
      tc_fence_after();
      float o[kOCols];
#pragma unroll
      for (int gq = 0; gq < kOCols / 32; ++gq) {
        float tmp[32];
        tmem_ld32(lane_base + 256u + (uint32_t)(kOCols * half + 32 * gq), tmp);
#pragma unroll
        for (int e = 0; e < 32; ++e) o[32 * gq + e] = tmp[e];
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(l_ofree);
      const float l_cta = l_part + exchange(l_part, 427);
      if (bad) break;
      // row sums of both CTAs, added in rank order so that both hold the same bits
      if (half == 0) {
        st_cluster_f32(r_lslot + (uint32_t)(row * 4), l_cta);
        __syncwarp();
        if (lane == 0) mbar_arrive_cluster(r_lmsg);
      }
      if (!wait_all(lmsg, n_l & 1, 428, true)) break;
      ++n_l;
      const float l_peer = lslot[row];
      const float l_tot = chalf == 0 ? l_cta + l_peer : l_peer + l_cta;
      const int r = w.tm * kBM + row;
      if (r < f.t) {
        const int64_t orow = ((int64_t)w.split * f.nb + w.b) * f.t + r;
        // local columns [0, 128): K~ features 128 r + c; [128, 256): V features
        const int feat0 = (half == 0 ? 0 : 256) + 128 * (int)chalf;
        float4* dst = reinterpret_cast<float4*>(f.O + orow * 512 + feat0);
#pragma unroll
        for (int c = 0; c < kOCols; c += 4) dst[c / 4] = make_float4(o[c], o[c + 1], o[c + 2], o[c + 3]);
        if (chalf == 0 && half == 0) f.stats[orow] = make_float2(m_run, l_tot);
        if constexpr (TK) {
          const int64_t cb = (orow * kTopLists + 2 * (int)chalf + half) * kTopK;
#pragma unroll
          for (int sl = 0; sl < kTopK; ++sl) {
            f.cand_key[cb + sl] = tk_key[sl];
            f.cand_c[cb + sl] = tk_c[sl];
          }
        }
      }
    }
  }

  tc_fence_before();
  // Neither CTA frees its TMEM while the leader's MMAs may still write it, nor leaves while
  // another CTA may still copy into or arrive on its shared memory.
  cluster_sync();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_2sm(tmem_base, 512);
  }
}

// One warp per (batch b, row r): the exact logits of the row's repair candidates replace the
// one-pass ones in every split's (O, l). See launch_ca_topk_repair.
template <int D2>
__global__ void __launch_bounds__(256) ca_topk_repair_kernel(const TopkRepairParams f) {
  constexpr float kLog2e = 1.4426950408889634f;
  constexpr int kG = D2 / 128;  // 4-column groups of O per lane
  constexpr int kQ = 8;         // 8-element q groups per lane (D <= 2048)
  const int64_t rows = (int64_t)f.nb * f.t;
  const int64_t rj = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (rj >= rows) return;
  const int b = (int)(rj / f.t);
  float M = -INFINITY;
  for (int s = 0; s < f.nsplit; ++s) M = fmaxf(M, f.stats[s * rows + rj].x);
  uint4 qh[kQ], ql[kQ];
  const __half* qrow = f.q + rj * 2 * (int64_t)f.D;
#pragma unroll
  for (int it = 0; it < kQ; ++it) {
    const int i = 8 * lane + 256 * it;
    qh[it] = i < f.D ? *reinterpret_cast<const uint4*>(qrow + i) : make_uint4(0, 0, 0, 0);
    ql[it] = i < f.D ? *reinterpret_cast<const uint4*>(qrow + f.D + i) : make_uint4(0, 0, 0, 0);
  }
  // exact logit of one key in log2 units (q_hi k_hi + q_hi k_lo + q_lo k_hi, fp32), the same
  // value in every lane
  auto logit = [&](int key) -> float {
    const __half* krow = f.k + ((int64_t)b * f.N + key) * 2 * (int64_t)f.D;
    float acc = 0.f;
#pragma unroll
    for (int it = 0; it < kQ; ++it) {
      const int i = 8 * lane + 256 * it;
      if (i < f.D) {
        const uint4 kh = *reinterpret_cast<const uint4*>(krow + i);
        const uint4 kl = *reinterpret_cast<const uint4*>(krow + f.D + i);
        const __half2* a = reinterpret_cast<const __half2*>(&qh[it]);
        const __half2* al = reinterpret_cast<const __half2*>(&ql[it]);
        const __half2* c = reinterpret_cast<const __half2*>(&kh);
        const __half2* cl = reinterpret_cast<const __half2*>(&kl);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float2 x = __half22float2(a[e]), xl = __half22float2(al[e]);
          const float2 y = __half22float2(c[e]), yl = __half22float2(cl[e]);
          acc = fmaf(x.x, y.x, fmaf(x.x, yl.x, fmaf(xl.x, y.x, acc)));
          acc = fmaf(x.y, y.y, fmaf(x.y, yl.y, fmaf(xl.y, y.y, acc)));
        }
      }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
    return acc * (f.kinv[(int64_t)b * f.N + key] * kLog2e);
  };
  const __nv_bfloat16* xbase = f.X + (int64_t)(b / f.bdiv) * f.N * 3 * f.d;
  float oacc[kG][4];
  // oacc += w * X_key (hi, plus lo on the K~ half)
  auto add_x = [&](int key, float w) {
    const __nv_bfloat16* xr = xbase + (int64_t)key * 3 * f.d;
#pragma unroll
    for (int gq = 0; gq < kG; ++gq) {
      const int col = 4 * lane + 128 * gq;
      const uint2 hv = *reinterpret_cast<const uint2*>(xr + col);
      const __nv_bfloat162* h2 = reinterpret_cast<const __nv_bfloat162*>(&hv);
      float2 x01 = __bfloat1622float2(h2[0]), x23 = __bfloat1622float2(h2[1]);
      if (col < f.d) {
        const uint2 lv = *reinterpret_cast<const uint2*>(xr + 2 * f.d + col);
        const __nv_bfloat162* l2 = reinterpret_cast<const __nv_bfloat162*>(&lv);
        const float2 l01 = __bfloat1622float2(l2[0]), l23 = __bfloat1622float2(l2[1]);
        x01.x += l01.x;
        x01.y += l01.y;
        x23.x += l23.x;
        x23.y += l23.y;
      }
      oacc[gq][0] = fmaf(w, x01.x, oacc[gq][0]);
      oacc[gq][1] = fmaf(w, x01.y, oacc[gq][1]);
      oacc[gq][2] = fmaf(w, x23.x, oacc[gq][2]);
      oacc[gq][3] = fmaf(w, x23.y, oacc[gq][3]);
    }
  };
  const int nc = f.nlists * kTopK;
  for (int s = 0; s < f.nsplit; ++s) {
    const int64_t sr = s * rows + rj;
    const float2 st = f.stats[sr];
    if (!(st.x >= M - f.cut)) continue;  // this split's weights are negligible in the row
    const int* ck = f.cand_key + sr * nc;
    const float* cc = f.cand_c + sr * nc;
#pragma unroll
    for (int gq = 0; gq < kG; ++gq) oacc[gq][0] = oacc[gq][1] = oacc[gq][2] = oacc[gq][3] = 0.f;
    float4* orow = reinterpret_cast<float4*>(f.O + sr * D2);
    float wc = 0.f;  // the candidates' one-pass weights
    for (int sl = 0; sl < nc; ++sl)
      if (ck[sl] >= 0) wc += exp2f(cc[sl] - st.x);
    if (st.y - wc > f.guard * st.y) {
      // weight spread beyond the candidates: every key of the split, exact, in key order
      const int j0 = (int)(((int64_t)f.tiles_k * s) / f.nsplit);
      const int j1 = (int)(((int64_t)f.tiles_k * (s + 1)) / f.nsplit);
      const int k1 = min(j1 * f.keys_per_tile, f.N);
      float lsum = 0.f;
      for (int key = j0 * f.keys_per_tile; key < k1; ++key) {
        const float w = exp2f(logit(key) - st.x);
        lsum += w;
        add_x(key, w);
      }
#pragma unroll
      for (int gq = 0; gq < kG; ++gq)
        orow[lane + 32 * gq] = make_float4(oacc[gq][0], oacc[gq][1], oacc[gq][2], oacc[gq][3]);
      if (lane == 0) f.stats[sr].y = lsum;
      continue;
    }
    float dl = 0.f;
    for (int sl = 0; sl < nc; ++sl) {
      const int key = ck[sl];  // warp-uniform
      if (key < 0 || !(cc[sl] >= M - f.cut)) continue;
      const float delta = exp2f(logit(key) - st.x) - exp2f(cc[sl] - st.x);
      dl += delta;
      add_x(key, delta);
    }
#pragma unroll
    for (int gq = 0; gq < kG; ++gq) {
      float4 o = orow[lane + 32 * gq];
      o.x += oacc[gq][0];
      o.y += oacc[gq][1];
      o.z += oacc[gq][2];
      o.w += oacc[gq][3];
      orow[lane + 32 * gq] = o;
    }
    if (lane == 0) f.stats[sr].y = st.y + dl;
  }
}

}  // namespace

cudaError_t launch_ca_topk_repair(const TopkRepairParams& f, int d2, cudaStream_t stream) {
  if (f.D <= 0 || f.D % 8 != 0 || f.D > 2048 || f.d * 2 != d2 || f.t <= 0 || f.nb <= 0 ||
      f.N <= 0 || f.nsplit < 1 || f.nlists < 1 || f.tiles_k < f.nsplit ||
      (int64_t)f.tiles_k * f.keys_per_tile < f.N || f.q == nullptr || f.k == nullptr ||
      f.X == nullptr || f.O == nullptr || f.stats == nullptr || f.cand_key == nullptr ||
      f.cand_c == nullptr || f.bdiv < 1)
    return cudaErrorInvalidValue;
  const int64_t rows = (int64_t)f.nb * f.t;
  const unsigned grid = (unsigned)((rows + 7) / 8);
  if (d2 == 512)
    ca_topk_repair_kernel<512><<<grid, 256, 0, stream>>>(f);
  else if (d2 == 256)
    ca_topk_repair_kernel<256><<<grid, 256, 0, stream>>>(f);
  else if (d2 == 128)
    ca_topk_repair_kernel<128><<<grid, 256, 0, stream>>>(f);
  else
    return cudaErrorInvalidValue;
  return cudaGetLastError();
}

// The persistent grid holds no more clusters than can be resident at once (a cluster needs two
// free SMs of one GPC): a cluster that waited for another to exit would start its whole share
// of the units late.
int ca_pair_clusters(int num_sms) {
  static thread_local int resident = 0;
  const int most = std::max(1, num_sms / kPairCluster);
  if (resident == 0) {
    if (cudaFuncSetAttribute(ca_pair_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             PairSmem::kBytes) != cudaSuccess) {
      cudaGetLastError();
      return most;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(kPairCluster * most, 1, 1);
    cfg.blockDim = dim3(kFlashThreads, 1, 1);
    cfg.dynamicSmemBytes = PairSmem::kBytes;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = kPairCluster;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, ca_pair_kernel<false>, &cfg) != cudaSuccess || n < 1) {
      cudaGetLastError();
      n = most;
    }
    resident = std::max(1, std::min(n, most));
  }
  return resident;
}

cudaError_t launch_ca_pair(const Operand2D& Q, const Operand2D& K, const Operand2D& XT,
                           const FlashParams& f, int num_sms, cudaStream_t stream,
                           bool one_pass) {
  using S = PairSmem;
  if (f.D <= 0 || f.D % kBK != 0 || f.t <= 0 || f.N <= 0 || f.Np % kBK != 0 || f.Np < f.N ||
      f.nunits <= 0 || (one_pass && (f.cand_key == nullptr || f.cand_c == nullptr)))
    return cudaErrorInvalidValue;
  // boxes: q 128 rows; k halves of 128 rows; X^T boxes of 64 rows (hi boxes in two copies)
  CUtensorMap tq, tk, tx;
  if (!make_tmap(&tq, Q, kBM) || !make_tmap(&tk, K, kPairKeys / 2) || !make_tmap(&tx, XT, 64))
    return cudaErrorInvalidValue;
  auto kern = one_pass ? ca_pair_kernel<true> : ca_pair_kernel<false>;
  static thread_local bool attr_set[2] = {false, false};
  if (!attr_set[one_pass]) {
    cudaError_t e =
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, S::kBytes);
    if (e != cudaSuccess) return e;
    attr_set[one_pass] = true;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.blockDim = dim3(kFlashThreads, 1, 1);
  cfg.dynamicSmemBytes = S::kBytes;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = kPairCluster;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const int clusters = std::max(1, std::min(f.nunits, ca_pair_clusters(num_sms)));
  cfg.gridDim = dim3(kPairCluster * clusters, 1, 1);
  return cudaLaunchKernelEx(&cfg, kern, tq, tk, tx, f);
}

}  // namespace still
