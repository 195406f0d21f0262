// Host runtime behind the C ABI (include/still.h): validation, weight re-layout and
// precompute, workspace planning, and the per-layer launch sequence.
//
// Per-layer sequence for one sequence of N tokens and t latents (Sec. 2.1, App. A):
//   strip      K, V -> X = [unRoPE(K) | V]  (hi/lo bf16 and hi/lo fp16 transposed)
//   tables     compactor-RoPE coarse angle table for the key positions
//   per group of (KV-head h, cross head i):
//     keyproj  k~ = X W_K,i + b_K,i -> RoPE_c -> hi/lo, |k~|^2          (2-pass GEMM, 2-SM)
//     qrope    q = RoPE_c(q^_i, p_j) -> hi/lo                         (q^ precomputed at load)
//     ca_fused S = d_l * q.k / |k~|, online softmax, O_i += P X per key split, in one kernel
//              (units of two query tiles: a CTA pair with 2-SM MMAs for head dim <= 128, a
//              cluster of four for 256)
//     repair   (head dim 256) exact logits of each row's heaviest keys
//     merge    the key splits of O_i and (m, l), in a fixed order -> hi/lo
//   VO         Z' = Z + [O_1..O_n] (W_V,i W_O,i)_i                     (3-pass GEMM)
//   SA         Z'' = Z' + Concat_i softmax(d_l q^ k^T) v . S_O          (per KV-head bank)
//   FFN        Z''' = Z'' + GELU(RMSNorm(Z'') W_1) W_2
//   heads      C_k = RoPE(Z''' W_key, p_out), C_v = Z''' W_val      (2-pass, Z''' hi/lo)
#include <algorithm>
#include <cmath>
#include <cstring>
#include <mutex>
#include <vector>

#include "../../include/still.h"
#include "gemm_host.cuh"
#include "kernels.cuh"
#include "ca_flash.cuh"

using namespace still;

namespace {

using bf16 = __nv_bfloat16;

// One compactor block's weights in the library's layouts (App. A, "Compactor blocks").
struct BlockW {
  bool has_ca = false;   // cross-attention in this block
  bf16* WkT = nullptr;   // [nD][2d]  pair-chunk order
  float* bk = nullptr;   // [nD]      pair-chunk order
  bf16* WqT = nullptr;   // [nD][D] pair-chunk order (queries formed per call only)
  float* bq = nullptr;   // [nD]    pair-chunk order (queries formed per call only)
  bf16* WvoT = nullptr;  // [D][2 * n * 2d]: (W_V,i W_O,i)^T hi | lo
  bf16* SqkT = nullptr;  // [2nD][D]
  float* sbqk = nullptr; // [2nD]
  bf16* SvT = nullptr;   // [nD][D]
  bf16* SoT = nullptr;   // [D][nD]
  bf16* W1T = nullptr;   // [F][D]
  bf16* W2T = nullptr;   // [D][F]
};

struct LayerW {
  bool loaded = false;
  still_layer_config cfg{};
  bf16* Z = nullptr;     // [H][t_max][D]
  float* qhat = nullptr; // block 0: [H][n][t_max][D] fp32, L2-normalised, pair-chunk order
  bool qhat_lazy = false; // block 0's q^ formed per call from Z (qhat unused)
  // Layers of more than one block keep W_K, W_Q, X and RMSNorm(Z) in fp16 (hi | lo where
  // split): about 22 bits against bf16 hi | lo's 16, for the amplification across blocks.
  bool f16 = false;
  std::vector<BlockW> blk;
  bf16* WhT = nullptr;   // [2d][D]
  double* omega_b = nullptr;  // [d/2] base-model RoPE frequencies (fp64)
  double* omega_c = nullptr;  // [D/2] compactor RoPE frequencies (fp64)
  // Without compactor RoPE the key projection folds into the queries (fold): the scores are
  // x~ . u with x~ = [x; 1] and u = W~ q^ (W~ = [W_K; b_K]), the key norms x~ G x~ with
  // G = W~ W~^T, so the N-token cache is never projected.
  bool fold = false;
  int Kp = 0;                 // width of x~ padded to a multiple of 64
  bf16* U = nullptr;          // [H][n][t_max][2 Kp]: u = W~_i q^ as hi | lo
  bf16* G = nullptr;          // [n][Kp][2 Kp]: W~_i W~_i^T as hi | lo
  float* wbeta = nullptr;     // [D] beta head w_beta (fp32), when set
  still_beta_config beta{};
  std::vector<void*> owned;
};

}  // namespace

// Per-kernel-class launch counts and (when enabled) CUDA-event timings.
struct Profiler {
  bool on = false;
  uint64_t mask = ~uint64_t(0);  // classes with event timing while on
  int64_t launches[STILL_K_COUNT] = {0};
  double ms[STILL_K_COUNT] = {0};
  struct Rec {
    int cls;
    cudaEvent_t a, b;
  };
  std::vector<Rec> recs;
  std::vector<cudaEvent_t> pool;
  cudaEvent_t pending = nullptr;
  int64_t untimed = 0;  // event pairs that could not be timed since the last reset

  cudaEvent_t get() {
    if (!pool.empty()) {
      cudaEvent_t e = pool.back();
      pool.pop_back();
      return e;
    }
    cudaEvent_t e = nullptr;
    cudaEventCreate(&e);
    return e;
  }
  // Inside a stream capture an event must be recorded as an external node to be recorded again
  // on every replay of the graph (a plain record there only orders the captured work).
  static void record(cudaEvent_t e, cudaStream_t s) {
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(s, &cs) == cudaSuccess && cs == cudaStreamCaptureStatusActive)
      cudaEventRecordWithFlags(e, s, cudaEventRecordExternal);
    else
      cudaEventRecord(e, s);
  }
  // Set on the calling host thread while it runs an allocation-free call: event timing creates
  // CUDA events, so it is skipped there (launch counting stays on). Per thread, so that no
  // shared state of the context is written.
  static bool& untimed_thread() {
    static thread_local bool v = false;
    return v;
  }
  void begin(int cls, cudaStream_t s) {
    ++launches[cls];
    if (!on || untimed_thread() || !((mask >> cls) & 1)) return;
    pending = get();
    record(pending, s);
  }
  void end(int cls, cudaStream_t s) {
    if (!on || pending == nullptr) return;
    cudaEvent_t b = get();
    record(b, s);
    recs.push_back(Rec{cls, pending, b});
    pending = nullptr;
  }
  bool resolve() {
    if (recs.empty()) return true;
    if (cudaDeviceSynchronize() != cudaSuccess) return false;
    for (auto& r : recs) {
      float t = 0.f;
      if (cudaEventElapsedTime(&t, r.a, r.b) != cudaSuccess) {
        cudaGetLastError();  // not a device fault: do not leave it to the next launch check
        untimed += 1;
        t = 0.f;
      }
      ms[r.cls] += t;
      pool.push_back(r.a);
      pool.push_back(r.b);
    }
    recs.clear();
    return true;
  }
  void reset() {
    resolve();
    untimed = 0;
    for (int i = 0; i < STILL_K_COUNT; ++i) {
      launches[i] = 0;
      ms[i] = 0;
    }
  }
  ~Profiler() {
    for (auto& r : recs) {
      cudaEventDestroy(r.a);
      cudaEventDestroy(r.b);
    }
    for (auto e : pool) cudaEventDestroy(e);
  }
};

struct still_ctx {
  int device = 0;
  int nsm = 0;
  int* err = nullptr;  // device error record [4]
  std::vector<LayerW> layers;
  void* ws = nullptr;
  size_t ws_bytes = 0;
  size_t ws_limit = size_t(48) << 30;
  size_t qhat_eager_limit = size_t(2) << 30;
  bool key_fold = true;  // fold W_K into the queries where the layer allows it
  Profiler prof;
};

namespace {

#define CK(x)                                            \
  do {                                                   \
    cudaError_t e_ = (x);                                \
    if (e_ != cudaSuccess) return STILL_ERR_CUDA;        \
  } while (0)

inline int64_t rup(int64_t x, int64_t a) { return (x + a - 1) / a * a; }

constexpr int kMaxFlashSplit = 16;  // key-split cap of the fused cross-attention

void free_layer(LayerW& L) {
  for (void* p : L.owned) cudaFree(p);
  L = LayerW();
}

template <typename T>
still_status dalloc(LayerW& L, T** p, size_t count) {
  void* q = nullptr;
  if (cudaMalloc(&q, std::max<size_t>(count, 1) * sizeof(T)) != cudaSuccess) return STILL_ERR_OOM;
  L.owned.push_back(q);
  *p = static_cast<T*>(q);
  return STILL_OK;
}

still_status check_cfg(const still_layer_config* c) {
  if (c == nullptr) return STILL_ERR_INVALID_ARG;
  if (c->n_kv_heads < 1 || c->head_dim < 1 || c->d_latent < 1 || c->n_cross_heads < 1 ||
      c->n_self_heads < 1 || c->t_max < 1 || c->ffn_dim < 0 || c->n_blocks < 1)
    return STILL_ERR_SHAPE;
  if (!(std::isfinite(c->rope_theta) && c->rope_theta > 0) ||
      !(std::isfinite(c->rope_theta_compactor) && c->rope_theta_compactor > 0) ||
      !std::isfinite(c->logit_scale) || !(c->rms_eps >= 0) || !(c->l2_eps > 0))
    return STILL_ERR_INVALID_ARG;
  if (c->n_blocks < 1 || c->n_blocks > 2 ||
      (c->cross_every_block != 0 && c->cross_every_block != 1) ||
      c->n_cross_heads != c->n_self_heads ||
      c->d_latent % 256 != 0 || !(c->head_dim == 64 || c->head_dim == 128 || c->head_dim == 256) ||
      c->ffn_dim % 64 != 0 || (c->compactor_rope != 0 && c->compactor_rope != 1) ||
      c->rope_fix != 1 ||
      (c->final_norm != 0 && c->final_norm != 1))
    return STILL_ERR_UNSUPPORTED;
  // Two-block layers run every block through the fused cross-attention kernel, which needs
  // 2d <= 256; the first block of a 2d = 512 layer would take the unfused split-fp16 path,
  // which the parity tests do not cover.
  if (c->n_blocks > 1 && c->head_dim == 256) return STILL_ERR_UNSUPPORTED;
  return STILL_OK;
}

// ------------------------------------------------------------------------------ GEMM helper

GemmParams gp(int M, int N, int batch = 1, int bdiv = 1) {
  GemmParams p;
  std::memset(&p, 0, sizeof(p));
  p.M = M;
  p.N = N;
  p.batch = batch;
  p.bdiv = bdiv;
  p.ksplit = 1;
  return p;
}

void add_pass(GemmParams& p, int a_koff, int b_koff, int a_roff, int b_roff, int klen) {
  p.pass[p.npass++] = GemmPass{a_koff, b_koff, a_roff, b_roff, klen};
}

Operand2D op(const void* ptr, int64_t rows, int64_t cols, int64_t pitch = -1) {
  return Operand2D{ptr, rows, cols, pitch < 0 ? cols : pitch};
}

// One GEMM of the launch sequence; CLS is its kernel class (profiling and kernel name).
template <int CLS, int BN, class Epi>
still_status run_gemm_bn(still_ctx* ctx, const Operand2D& A, const Operand2D& B, GemmParams p,
                         const Epi& e, int ab_fmt, cudaStream_t s,
                         const StoreView3D* view = nullptr) {
  p.err = ctx->err;
  ctx->prof.begin(CLS, s);
  cudaError_t r = launch_gemm<BN, CLS>(A, B, p, e, ab_fmt, ctx->nsm, s, view);
  ctx->prof.end(CLS, s);
  if (r == cudaErrorInvalidValue) return STILL_ERR_INVALID_ARG;
  return r == cudaSuccess ? STILL_OK : STILL_ERR_CUDA;
}

template <int CLS, class Epi>
still_status run_gemm(still_ctx* ctx, int bn, const Operand2D& A, const Operand2D& B,
                      GemmParams p, const Epi& e, int ab_fmt, cudaStream_t s) {
  return bn == 128 ? run_gemm_bn<CLS, 128>(ctx, A, B, p, e, ab_fmt, s)
                   : run_gemm_bn<CLS, 256>(ctx, A, B, p, e, ab_fmt, s);
}

template <int CLS, class Epi>
still_status run_gemm256(still_ctx* ctx, const Operand2D& A, const Operand2D& B, GemmParams p,
                         const Epi& e, int ab_fmt, cudaStream_t s,
                         const StoreView3D* view = nullptr) {
  return run_gemm_bn<CLS, 256>(ctx, A, B, p, e, ab_fmt, s, view);
}

// The same on CTA pairs (2-SM MMAs, 256 x 256 tiles): for the key projection, whose 1-SM form
// is bound by shared-memory traffic.
template <int CLS, class Epi>
still_status run_gemm256_2sm(still_ctx* ctx, const Operand2D& A, const Operand2D& B,
                             GemmParams p, const Epi& e, int ab_fmt, cudaStream_t s,
                             const StoreView3D* view = nullptr) {
  p.err = ctx->err;
  ctx->prof.begin(CLS, s);
  cudaError_t r = launch_gemm_2sm<256, CLS>(A, B, p, e, ab_fmt, ctx->nsm, s, view);
  ctx->prof.end(CLS, s);
  if (r == cudaErrorInvalidValue) return STILL_ERR_INVALID_ARG;
  return r == cudaSuccess ? STILL_OK : STILL_ERR_CUDA;
}

StoreView3D store_view(void* ptr, int elem_bytes, int64_t nx, int64_t ny, int64_t nz,
                       int64_t ystride, int64_t zstride, int bx, bool swz) {
  StoreView3D v;
  v.ptr = ptr;
  v.elem_bytes = elem_bytes;
  v.nx = nx;
  v.ny = ny;
  v.nz = nz;
  v.ystride = ystride;
  v.zstride = zstride;
  v.bx = bx;
  v.swizzle128 = swz;
  return v;
}

// Launch of one of the memory-bound kernels, timed under its class.
#define KLAUNCH(cls, call)                  \
  do {                                      \
    ctx->prof.begin((cls), s);              \
    cudaError_t e_ = (call);                \
    ctx->prof.end((cls), s);                \
    if (e_ != cudaSuccess) return STILL_ERR_CUDA; \
  } while (0)

#define TRY(x)                          \
  do {                                  \
    still_status st_ = (x);             \
    if (st_ != STILL_OK) return st_;    \
  } while (0)

// ------------------------------------------------------------------------------ workspace plan

struct Plan {
  int H, d, D, n, F, t;
  int64_t N, Np, tp, ldt;
  int G;
  bool flash;     // fused cross-attention kernel (2d of 128 or 256) for the last block
  int ca_units;   // (h, i) pairs per cross-attention group
  int sa_heads;   // KV-heads per self-attention group
  int sa_sub;     // self heads per scores / softmax / P.v pass (n unless one bank is too big)
  // byte offsets
  size_t oX, oXT, oCoarse, oOmega, oGD, oHrot, oPX, oZ1, oA1, oCat, oZ2, oA2, oG, oZ3;
  size_t oCA, oSA;
  size_t ca_unit_bytes, sa_unit_bytes;
  size_t kb_b, kss_b, q_b, P_b, O_b, qt_b, cand_b;  // per CA unit
  bool lazy_q;
  size_t oZn;
  size_t qk_b, sss_b, vT_b, Ssa_b, Psa_b;        // per SA bank (KV-head)
  size_t Ssah_b, Psah_b;                          // per self head (unpadded)
  size_t total;
};

size_t a256(size_t x) { return (x + 255) & ~size_t(255); }

// The self-attention value path (probabilities, values, head outputs) and the FFN run in bf16
// hi | lo rather than plain bf16. The self-attention logits d_l cos(q, k) over t latents are
// sharp enough that the rounding of its output moves the next sublayers by far more than its
// own size, and more so as d_l and t grow: emulating plain-bf16 probabilities, values and FFN
// activations on the Gemma-shaped compactor moves C_k from the output-rounding floor of 0.009
// to 0.015 x RMS (0.009 in hi | lo), and on the iterative Qwen-8B-shaped workload the plain
// path reaches 0.020 once t passes 4000. In a layer of two blocks the next block's queries
// amplify it further.
bool value_hilo(const still_layer_config&) { return true; }

// The cross-attention scores of a one-block layer of head dim 256 (the kernel on clusters of
// two CTAs) take one fp16 MMA pass (q_hi . k_hi) instead of three split-bf16 passes, and a
// repair kernel then recomputes the logits of each row's heaviest keys from the fp16 hi | lo
// operands (about 22 bits). At d_l >= 512 the rows put nearly all their weight on a few
// keys: CPU emulation of the C_k error from the cross-attention logits alone, with the k
// heaviest keys of every row repaired, gives 5.1e-4 (k = 8) and 1.5e-5 (k = 16) on the Gemma
// shape at 16k tokens, against 3.7e-3 for the three-pass split. Head dims 64 and 128 keep the
// split: there one CTA runs the softmax of every tile, a one-pass S tile takes no longer than
// that softmax, and the kernel measured slower with one pass (the Qwen-7B-shaped stack went
// from 76 to 109 ms, with 24 ms of repair).
bool one_pass_scores(const still_layer_config& c) {
  return c.n_blocks == 1 && c.head_dim == 256 && c.d_latent >= 512 && c.d_latent <= 2048;
}

bool make_plan(const still_layer_config& c, bool lazy_q, int Kp, int64_t N, int t, double pmin,
               double pmax, size_t limit, Plan& P) {
  P.H = c.n_kv_heads;
  P.d = c.head_dim;
  P.D = c.d_latent;
  P.n = c.n_cross_heads;
  P.F = c.ffn_dim;
  P.t = t;
  P.N = N;
  P.Np = rup(N, 64);
  P.tp = rup(t, 64);
  P.ldt = rup(t, 4);
  P.G = (int)std::floor((pmax - pmin) / kPosGrain) + 2;
  const int64_t H = P.H, d = P.d, D = P.D, n = P.n, F = P.F, T = t;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    size_t o = off;
    off += a256(bytes);
    return o;
  };
  P.oX = take(H * N * std::max<int64_t>(3 * d, 2 * Kp) * 2);  // Kp > 0: the folded x~ rows
  P.oXT = take(H * 2 * d * 2 * P.Np * 2);
  P.oCoarse = take((size_t)(P.G + kPosGrain) * (D / 2) * 8);  // coarse rows, then fine rows
  P.oOmega = take((D / 2) * 4);
  P.oGD = take((size_t)P.Np * 8);
  P.oHrot = take(T * (d / 2) * 8);
  P.oPX = take(H * T * 2 * n * 2 * d * 2);
  P.oZ1 = take(H * T * D * 4);
  P.oA1 = take(H * T * 2 * D * 2);
  // A block that feeds another keeps its value path in hi/lo (x2 buffers below).
  const int64_t hl = value_hilo(c) ? 2 : 1;
  P.oCat = take(H * T * n * D * 2 * hl);
  P.oZ2 = take(H * T * D * 4);
  P.oA2 = take(H * T * D * 2 * hl);
  P.oG = take(H * T * std::max<int64_t>(F, 1) * 2 * hl);
  P.oZ3 = take(H * T * D * 4);
  P.lazy_q = lazy_q;
  P.oZn = lazy_q ? take(H * T * 2 * D * 2) : 0;  // RMSNorm(Z) hi | lo for the call's t latents
  const size_t fixed = off;
  // |k~|^2 partials + inverses; the folded path needs neither k nor per-call q
  const int64_t kparts = std::max<int64_t>(EpiRopeCT<false>::kParts * (D / 256), Kp / 32);
  P.kb_b = Kp > 0 ? 0 : a256(N * 2 * D * 2);
  P.kss_b = a256(N * 4 * (kparts + 1));
  P.q_b = Kp > 0 ? 0 : a256(T * 2 * D * 2);
  // The fused kernel serves every block (a block that feeds another takes its split-precision
  // variant); 2d = 512 runs it on clusters of four CTAs whose query-tile pairs split the O
  // columns.
  P.flash = d == 64 || d == 128 || d == 256;
  P.P_b = a256(T * 8) * kMaxFlashSplit;          // per-split row statistics (m, l)
  P.O_b = a256(T * 2 * d * 4) * kMaxFlashSplit;  // per-split unnormalised O
  // one-pass scores: repair candidates (key, c) per split, row and list
  P.cand_b = one_pass_scores(c) && Kp == 0 ? 2 * a256(T * kTopLists * kTopK * 4) * kMaxFlashSplit
                                           : 0;
  // lazy q^: fp32 q~ of the unit and its sum-of-squares partials + inverse norms
  P.qt_b = lazy_q ? a256(T * D * 4) + a256(T * 4 * (2 * (D / 256) + 1)) : 0;
  P.ca_unit_bytes = P.kb_b + P.kss_b + P.q_b + P.P_b + P.O_b + P.qt_b + P.cand_b;
  P.qk_b = a256(2 * n * T * 2 * D * 2);
  P.sss_b = a256(2 * n * T * 4 * (2 * (D / 256) + 1));
  P.vT_b = a256(n * D * P.tp * 2 * hl);
  P.Ssa_b = a256(n * T * P.ldt * 4);
  P.Psa_b = a256(n * T * P.tp * 2 * hl);
  P.Ssah_b = (size_t)T * P.ldt * 4;
  P.Psah_b = (size_t)T * P.tp * 2 * hl;
  P.sa_unit_bytes = P.qk_b + P.sss_b + P.vT_b + P.Ssa_b + P.Psa_b;
  if (fixed >= limit) return false;
  const size_t avail = limit - fixed;
  // Cross-attention groups: whole KV-heads when possible, else a part of one head.
  const int64_t units_total = H * n;
  int64_t u = std::min<int64_t>(units_total, (int64_t)(avail / P.ca_unit_bytes));
  if (u < 1) return false;
  if (u >= n)
    u = (u / n) * n;
  P.ca_units = (int)u;
  int64_t sh = std::min<int64_t>(H, (int64_t)(avail / P.sa_unit_bytes));
  size_t sa_bytes;
  if (sh >= 1) {
    P.sa_heads = (int)sh;
    P.sa_sub = (int)n;
    sa_bytes = P.sa_unit_bytes * P.sa_heads;
  } else {
    // One bank at a time, its self heads in sub-groups (scores and probabilities per head).
    const size_t bank = P.qk_b + P.sss_b + P.vT_b;
    const size_t head = P.Ssah_b + P.Psah_b;
    if (avail < bank + head + 1024) return false;
    P.sa_heads = 1;
    P.sa_sub = (int)std::min<int64_t>(n, (int64_t)((avail - bank - 1024) / head));
    sa_bytes = bank + a256(P.sa_sub * P.Ssah_b) + a256(P.sa_sub * P.Psah_b);
  }
  P.oCA = off;
  P.oSA = off;  // the two phases reuse the same region
  P.total = off + std::max(P.ca_unit_bytes * P.ca_units, sa_bytes);
  return true;
}

still_status ensure_ws(still_ctx* ctx, size_t bytes) {
  if (bytes <= ctx->ws_bytes) return STILL_OK;
  if (ctx->ws != nullptr) {
    CK(cudaDeviceSynchronize());
    cudaFree(ctx->ws);
    ctx->ws = nullptr;
    ctx->ws_bytes = 0;
  }
  if (cudaMalloc(&ctx->ws, bytes) != cudaSuccess) {
    cudaGetLastError();
    return STILL_ERR_OOM;
  }
  ctx->ws_bytes = bytes;
  return STILL_OK;
}

// ------------------------------------------------------------------------------ positions

struct Positions {
  PosSegs segs;
  double pmin = 0, pmax = 0;
  bool frac = false;  // some position is not an integer
};

still_status make_positions(const still_pos_segment* h_segments, int32_t n_segments, int64_t N,
                            Positions& out) {
  out = Positions();
  if (n_segments == 0 || h_segments == nullptr) {
    if (n_segments != 0) return STILL_ERR_INVALID_ARG;
    out.segs.n = 1;
    out.segs.begin[0] = 0;
    out.segs.begin[1] = N;
    out.segs.start[0] = 0;
    out.segs.step[0] = 1;
    out.pmin = 0;
    out.pmax = (double)(N - 1);
    return STILL_OK;
  }
  if (n_segments < 0 || n_segments > 8) return STILL_ERR_UNSUPPORTED;
  int64_t acc = 0;
  double lo = INFINITY, hi = -INFINITY;
  int k = 0;
  for (int i = 0; i < n_segments; ++i) {
    const still_pos_segment& s = h_segments[i];
    if (s.count < 0 || !std::isfinite(s.start) || !std::isfinite(s.step))
      return STILL_ERR_INVALID_ARG;
    if (s.count == 0) continue;
    if (s.start != std::floor(s.start) || (s.count > 1 && s.step != std::floor(s.step)))
      out.frac = true;
    const double last = s.start + (double)(s.count - 1) * s.step;
    if (!std::isfinite(last)) return STILL_ERR_INVALID_ARG;
    lo = std::min(lo, std::min(s.start, last));
    hi = std::max(hi, std::max(s.start, last));
    out.segs.begin[k] = acc;
    out.segs.start[k] = s.start;
    out.segs.step[k] = s.step;
    ++k;
    acc += s.count;
  }
  if (acc != N || k == 0) return STILL_ERR_SHAPE;
  out.segs.n = k;
  out.segs.begin[k] = acc;
  out.pmin = lo;
  out.pmax = hi;
  return STILL_OK;
}

// ------------------------------------------------------------------------------ one sequence

struct OutSpec {
  bf16* ck;
  bf16* cv;
  int64_t st, sh;          // element strides of [t, H, d] outputs (d contiguous)
  float* beta = nullptr;   // [t][H] per-slot logit bias (optional; needs a beta head)
};

// ws_fixed / ws_fixed_bytes: when set, the call runs in that caller-provided scratch and never
// touches the context's (growable) workspace.
// Some block's latent queries are formed inside the call (block 0's when too large to keep,
// every later cross-attending block's).
bool queries_per_call(const LayerW& L) {
  return L.qhat_lazy || (L.cfg.n_blocks > 1 && L.cfg.cross_every_block);
}

int fold_kp(const LayerW& L) { return L.fold ? L.Kp : 0; }

// The fp16 hi | lo copy of W_V W_O of a block that feeds another is stored multiplied by this
// power of two: its entries (products of two weights) sit near the fp16 subnormal range.
constexpr float kWvoScale = 256.f;

still_status compact_one(still_ctx* ctx, const LayerW& L, const KVSource& src,
                         const Positions& pos, int64_t N, int t, const OutSpec& out,
                         cudaStream_t s, uint8_t* ws_fixed = nullptr,
                         size_t ws_fixed_bytes = 0) {
  const still_layer_config& c = L.cfg;
  Plan P;
  const size_t limit = ws_fixed != nullptr ? ws_fixed_bytes : ctx->ws_limit;
  if (!make_plan(c, queries_per_call(L), fold_kp(L), N, t, pos.pmin, pos.pmax, limit, P))
    return STILL_ERR_OOM;
  if (ws_fixed == nullptr) TRY(ensure_ws(ctx, P.total));
  uint8_t* ws = ws_fixed != nullptr ? ws_fixed : static_cast<uint8_t*>(ctx->ws);
  const int H = P.H, d = P.d, D = P.D, n = P.n, F = P.F;
  const int64_t Np = P.Np;
  const float scale = c.logit_scale > 0 ? (float)c.logit_scale : (float)D;
  const double qstart = pos.pmin;
  const double qstep = t > 1 ? (pos.pmax - pos.pmin) / (double)(t - 1) : 0.0;

  bf16* X = reinterpret_cast<bf16*>(ws + P.oX);
  __half* XT = reinterpret_cast<__half*>(ws + P.oXT);
  float2* coarse = reinterpret_cast<float2*>(ws + P.oCoarse);
  float* omega = reinterpret_cast<float*>(ws + P.oOmega);
  float2* gd = reinterpret_cast<float2*>(ws + P.oGD);
  float2* hrot = reinterpret_cast<float2*>(ws + P.oHrot);
  bf16* PX = reinterpret_cast<bf16*>(ws + P.oPX);
  float* Z1 = reinterpret_cast<float*>(ws + P.oZ1);
  bf16* A1 = reinterpret_cast<bf16*>(ws + P.oA1);
  bf16* cat = reinterpret_cast<bf16*>(ws + P.oCat);
  float* Z2 = reinterpret_cast<float*>(ws + P.oZ2);
  bf16* A2 = reinterpret_cast<bf16*>(ws + P.oA2);
  bf16* Gb = reinterpret_cast<bf16*>(ws + P.oG);
  void* Z3 = ws + P.oZ3;

  KLAUNCH(STILL_K_STRIP, launch_strip(src, N, H, d, pos.segs, L.omega_b, c.rope_fix, X, XT, Np,
                                      gd, pos.pmin, P.G, L.f16 ? 1 : 0, fold_kp(L), s));
  const int w_fmt = L.f16 ? 0 : 1;    // operand format of X, RMSNorm(Z), W_K and W_Q products
  const int zn_mode = L.f16 ? 2 : 1;  // RMSNorm(Z) as fp16 or bf16 hi | lo
  KLAUNCH(STILL_K_TABLES, launch_rope_tables(coarse, omega, P.G, D, pos.pmin, L.omega_c, s));
  KLAUNCH(STILL_K_TABLES, launch_heads_rot(hrot, t, d / 2, qstart, qstep, L.omega_b, c.rope_fix, s));
  bf16* Zn = P.lazy_q ? reinterpret_cast<bf16*>(ws + P.oZn) : nullptr;
  const int64_t rows = (int64_t)H * t;
  const int n2d = n * 2 * d;
  const bool z3_bf16 = (c.final_norm == 0);
  // Latent state entering a block: the bank rows L.Z (bf16, pitch t_max) for block 0, else the
  // fp32 state Z2 [H * t][D] that the previous block left.
  for (int bi = 0; bi < c.n_blocks; ++bi) {
  const BlockW& Bw = L.blk[bi];
  const bool last = bi + 1 == c.n_blocks;
  // A block whose output enters another block keeps its cross-attention, self-attention
  // value path and FFN in split precision: the next block's cross-attention queries amplify
  // any rounding there. In a two-block layer the last block keeps its value path and FFN in
  // hi | lo too, and the first block's value chains (P X, W_V W_O, RMSNorm(Z'), the
  // self-attention q, k, v, P and head outputs) are fp16 hi | lo rather than bf16 hi | lo.
  const bool exact = !last;
  const bool vexact = exact || L.f16 || value_hilo(c);
  const bool tk = !exact && P.flash && !L.fold && one_pass_scores(c);  // one-pass scores
  const bool f16v = exact && L.f16 && P.flash;
  const int vfmt = f16v ? 0 : 1;
  const int32_t vkind = f16v ? OUT_HILO16 : OUT_HILO;
  float* Za = Z2;  // this block's state after cross-attention (Z2 itself without it)
  if (Bw.has_ca) {
  const bool q_call = bi > 0 || L.qhat_lazy;  // queries formed in this call
  if (q_call) {  // RMSNorm(latent state) hi | lo for latents j < t of every KV-head bank
    if (bi == 0) {
      for (int h = 0; h < H; ++h)
        KLAUNCH(STILL_K_LOAD, launch_rmsnorm(L.Z + (size_t)h * c.t_max * D, 1, t, D, D, c.rms_eps,
                                             Zn + (size_t)h * t * 2 * D, 2 * D, zn_mode, s));
    } else {
      KLAUNCH(STILL_K_LOAD, launch_rmsnorm(Z2, 0, rows, D, D, c.rms_eps, Zn, 2 * D, zn_mode, s));
    }
  }

  // ---------------------------------------------------------------- cross-attention groups
  const int units_total = H * n;
  for (int b0 = 0; b0 < units_total;) {
    // A group is whole KV-heads [h0, h0 + nh) x all cross heads, or part of one KV-head.
    const int h0 = b0 / n, i0 = b0 % n;
    int nh, ni;
    if (i0 == 0 && P.ca_units >= n) {
      nh = std::min(P.ca_units / n, H - h0);
      ni = n;
    } else {
      nh = 1;
      ni = std::min(P.ca_units, n - i0);
    }
    const int nbl = nh * ni;
    uint8_t* g = ws + P.oCA;
    bf16* kb = reinterpret_cast<bf16*>(g);
    g += P.kb_b * nbl;
    const int kparts = L.fold ? L.Kp / 32 : EpiRopeCT<false>::kParts * (D / 256);
    float* kss = reinterpret_cast<float*>(g);        // [nbl][N][kparts]
    float* kinv = kss + (size_t)nbl * N * kparts;    // [nbl][N]
    g += P.kss_b * nbl;
    bf16* qhl = reinterpret_cast<bf16*>(g);
    g += P.q_b * nbl;
    float2* fst = reinterpret_cast<float2*>(g);  // [nsplit][nbl * t]: per-split (m, l)
    g += P.P_b * nbl;
    float* O = reinterpret_cast<float*>(g);
    g += P.O_b * nbl;
    int* cand_key = reinterpret_cast<int*>(g);  // one-pass scores: repair candidates
    float* cand_c = reinterpret_cast<float*>(g + P.cand_b / 2 * nbl);
    g += P.cand_b * nbl;
    // lazy q^: q~ [nbl][t][D] fp32 and its sum-of-squares partials / inverse norms
    float* qt = reinterpret_cast<float*>(g);
    float* qss = reinterpret_cast<float*>(g + a256((size_t)t * D * 4) * nbl);
    const float* qsrc = L.qhat;  // [.][t_max][D], batch index b0 + local
    int q_tmax = c.t_max, q_b0 = b0;
    if (q_call) {
      // q~ = RMSNorm(Z) W_Q + b_Q (2-pass), as at weight load, for this group's (h, i) only
      GemmParams p = gp(t, ni * D, nh, 1);
      p.a_r1 = t;
      add_pass(p, 0, 0, h0 * t, i0 * D, D);
      add_pass(p, D, 0, h0 * t, i0 * D, D);
      EpiAffine e;
      e.kind = OUT_F32;
      e.out = qt;
      e.om.b1 = (int64_t)ni * t * D;
      e.om.r0 = D;
      e.om.cdiv = D;
      e.om.c1 = (int64_t)t * D;
      e.om.c0 = 1;
      e.bias = Bw.bq + (size_t)i0 * D;
      e.sumsq = qss;
      e.ssm.b1 = (int64_t)ni * t;
      e.ssm.r0 = 1;
      e.ssm.c0 = t;
      e.ss_seg = D;
      e.ss_parts = 2 * (D / 256);
      e.ss_block = t;
      e.vec_ok = 1;
      TRY(run_gemm256<STILL_K_LOAD>(ctx, op(Zn, (int64_t)H * t, 2 * D), op(Bw.WqT, (int64_t)n * D, D),
                                    p, e, w_fmt, s));
      const int64_t nq = (int64_t)nbl * t;
      float* qinv = qss + nq * (2 * (D / 256));
      KLAUNCH(STILL_K_NORMS, launch_inv_norms(qss, nq, 2 * (D / 256), t, c.l2_eps, 1.f, qinv, s));
      KLAUNCH(STILL_K_NORMS, launch_scale_rows(qt, qinv, nq, D, s));
      qsrc = qt;
      q_tmax = t;
      q_b0 = 0;
    }
    if (L.fold) {
      // |k~|^2 = x~ G_i x~: Y = x~ G_i (3-pass hi / lo, K = Kp), dotted with x~ in the epilogue
      const int Kp = L.Kp;
      GemmParams p = gp((int)N, Kp, nbl, ni);
      p.a_r1 = N;    // x~ rows of KV-head h0 + b / ni
      p.b_r0 = Kp;   // G rows of cross head i0 + b % ni
      add_pass(p, 0, 0, (int)(h0 * N), i0 * Kp, Kp);
      add_pass(p, 0, Kp, (int)(h0 * N), i0 * Kp, Kp);
      add_pass(p, Kp, 0, (int)(h0 * N), i0 * Kp, Kp);
      EpiQuad e;
      e.part = kss;
      e.xt = X + (size_t)h0 * N * 2 * Kp;
      e.Ntok = N;
      e.Kp = Kp;
      TRY(run_gemm256<STILL_K_KEYPROJ>(ctx, op(X, (int64_t)H * N, 2 * Kp),
                                       op(L.G, (int64_t)n * Kp, 2 * Kp), p, e, 1, s));
    } else {  // keyproj: rows = tokens of heads [h0, h0+nh), columns = cross heads [i0, i0+ni)
      GemmParams p = gp((int)N, ni * D, nh, 1);
      p.a_r1 = N;
      p.n_fast = 1;  // X rows of a KV-head can exceed L2; the W_K block fits
      add_pass(p, 0, 0, (int)(h0 * N), i0 * D, 2 * d);
      add_pass(p, 2 * d, 0, (int)(h0 * N), i0 * D, d);
      auto fill = [&](auto& e) {
        e.out = kb;
        e.sumsq = kss;
        e.bias = Bw.bk + (size_t)i0 * D;
        e.coarse = coarse;
        e.fine = coarse + (size_t)P.G * (D / 2);
        e.omega = omega;
        e.gd = gd;
        e.D = D;
        e.nheads = ni;
        e.ncoarse = P.G;
        e.fp16 = exact || tk ? 1 : 0;  // k as fp16 hi / lo (block feeding another; one pass)
        e.Ntok = N;
      };
      const StoreView3D kv = store_view(kb, 2, 2 * D, N, nbl, 2 * D, N * 2 * D, 16, false);
      const Operand2D xop = op(X, (int64_t)H * N, 3 * d);
      const Operand2D wop = op(Bw.WkT, (int64_t)n * D, 2 * d);
      if (pos.frac) {
        EpiRopeCT<true> e;
        fill(e);
        TRY(run_gemm256_2sm<STILL_K_KEYPROJ>(ctx, xop, wop, p, e, w_fmt, s, &kv));
      } else {
        EpiRopeCT<false> e;
        fill(e);
        TRY(run_gemm256_2sm<STILL_K_KEYPROJ>(ctx, xop, wop, p, e, w_fmt, s, &kv));
      }
    }  // key projection
    // scale / |k~_n| per key (the d_l logit scale folded in)
    // A block that feeds another forms q and k as fp16 hi / lo (about 22 bits; bf16 hi / lo
    // keeps 16): its logits steer the next block's queries. q is unit-norm, so it is scaled by
    // a power of two near sqrt(D) into the fp16 normal range and the logit scale divided by it.
    const float qscale =
        exact || tk ? std::exp2(std::round(0.5 * std::log2((double)D))) : 1.f;
    KLAUNCH(STILL_K_NORMS, launch_inv_norms(kss, (int64_t)nbl * N, kparts, N, c.l2_eps,
                                            scale / qscale, kinv, s));
    if (!L.fold)
      KLAUNCH(STILL_K_QROPE, launch_q_rope(qsrc, q_tmax, q_b0, nbl, t, D, qstart, qstep,
                                           L.omega_c, c.compactor_rope, qhl,
                                           exact || tk ? 1 : 0, qscale, s));
    {
      // S, the online softmax and P X in one kernel; per-split partials merged in order.
      FlashParams fp;
      fp.t = t;
      fp.N = (int)N;
      fp.D = D;
      fp.Np = Np;
      fp.nb = nbl;
      fp.bdiv = ni;
      fp.xbase_row = h0 * 2 * d;
      fp.tiles_m = (t + kBM - 1) / kBM;
      const int fkeys = exact ? FlashSmem<256, true>::kKeys : kFlashKeys;
      fp.tiles_k = (int)((N + fkeys - 1) / fkeys);
      // a unit holds two query tiles: a CTA pair (2d <= 256) or a cluster of four (2d = 512)
      const int slots = d == 256 ? ca_pair_clusters(ctx->nsm) : ctx->nsm / 2;
      const int mt = (fp.tiles_m + 1) / 2;
      fp.nsplit = flash_split((int64_t)mt * nbl, fp.tiles_k, slots, kMaxFlashSplit);
      const int64_t nunits = (int64_t)mt * nbl * fp.nsplit;
      if (nunits > 0x7fffffff || (int64_t)nbl * N > 0x7fffffff) return STILL_ERR_UNSUPPORTED;
      fp.nunits = (int)nunits;
      fp.kinv = kinv;
      fp.O = O;
      fp.stats = fst;
      fp.err = ctx->err;
      if (tk) {
        fp.cand_key = cand_key;
        fp.cand_c = cand_c;
      }
      Operand2D qop = op(qhl, (int64_t)nbl * t, 2 * D);
      Operand2D kop = op(kb, (int64_t)nbl * N, 2 * D);
      if (L.fold) {  // q := u (precomputed, t_max rows per (h, i)), k := x~ shared per KV-head
        const int Kp = L.Kp;
        fp.D = Kp;
        fp.q_row0 = ((int64_t)h0 * n + i0) * c.t_max;
        fp.q_pitch = c.t_max;
        fp.k_row0 = (int64_t)h0 * N;
        fp.kdiv = ni;
        qop = op(L.U, (int64_t)H * n * c.t_max, 2 * Kp);
        kop = op(X, (int64_t)H * N, 2 * Kp);
      }
      const Operand2D xop = op(XT, (int64_t)H * 2 * d, 2 * Np);
      ctx->prof.begin(STILL_K_CA_FUSED, s);
      cudaError_t r =
          d == 256 ? (exact ? cudaErrorInvalidValue  // two-block layers at d = 256 are refused
                            : launch_ca_pair(qop, kop, xop, fp, ctx->nsm, s, tk))
          : exact  ? (d == 64 ? launch_ca_flash<128, true>(qop, kop, xop, fp, ctx->nsm, s)
                              : launch_ca_flash<256, true>(qop, kop, xop, fp, ctx->nsm, s))
                   : (d == 64 ? launch_ca_flash<128>(qop, kop, xop, fp, ctx->nsm, s)
                              : launch_ca_flash<256>(qop, kop, xop, fp, ctx->nsm, s));
      ctx->prof.end(STILL_K_CA_FUSED, s);
      if (r == cudaErrorInvalidValue) return STILL_ERR_INVALID_ARG;
      if (r != cudaSuccess) return STILL_ERR_CUDA;
      if (tk) {  // exact logits of each row's heaviest keys, before the split merge
        TopkRepairParams rp;
        rp.q = reinterpret_cast<const __half*>(qhl);
        rp.k = reinterpret_cast<const __half*>(kb);
        rp.kinv = kinv;
        rp.X = X + (size_t)h0 * N * 3 * d;
        rp.O = O;
        rp.stats = fst;
        rp.cand_key = cand_key;
        rp.cand_c = cand_c;
        rp.D = D;
        rp.d = d;
        rp.t = t;
        rp.N = (int)N;
        rp.nb = nbl;
        rp.nsplit = fp.nsplit;
        rp.bdiv = ni;
        rp.nlists = kTopLists;
        rp.tiles_k = fp.tiles_k;
        rp.keys_per_tile = kFlashKeys;
        KLAUNCH(STILL_K_REPAIR, launch_ca_topk_repair(rp, 2 * d, s));
      }
      KLAUNCH(STILL_K_PXSPLIT, launch_ca_merge(O, fst, fp.nsplit, b0, nbl, n, t, 2 * d,
                                               f16v ? 1 : 0, PX, s));
      b0 += nbl;
    }
  }

  // ---------------------------------------------------------------- Z' = Z + PX W_VO
  {
    GemmParams p = gp((int)rows, D);
    add_pass(p, 0, 0, 0, 0, n2d);
    add_pass(p, 0, n2d, 0, 0, n2d);
    add_pass(p, n2d, 0, 0, 0, n2d);
    EpiAffine e;
    e.kind = OUT_F32;
    e.out = Z1;
    e.om.r0 = D;
    e.om.c0 = 1;
    if (bi == 0) {  // the latent bank rows [0, t) of each KV-head (bf16)
      e.res_kind = 2;
      e.res = L.Z;
      e.resm.rdiv = t;
      e.resm.r1 = (int64_t)c.t_max * D;
      e.resm.r0 = D;
      e.resm.c0 = 1;
    } else {  // the previous block's fp32 state
      e.res_kind = 1;
      e.res = Z2;
      e.resm.r0 = D;
      e.resm.c0 = 1;
    }
    e.vec_ok = 1;
    e.alpha = f16v ? 1.f / kWvoScale : 1.f;  // the fp16 W_V W_O copy is stored scaled
    TRY(run_gemm256<STILL_K_VO>(ctx, op(PX, rows, 2 * n2d), op(Bw.WvoT, D, 2 * n2d), p, e, vfmt,
                                s));
  }
  Za = Z1;
  }  // cross-attention of block bi
  KLAUNCH(STILL_K_NORM, launch_rmsnorm(Za, 0, rows, D, D, c.rms_eps, A1, 2 * D, f16v ? 2 : 1, s));

  // ---------------------------------------------------------------- latent self-attention
  for (int h0 = 0; h0 < H; h0 += P.sa_heads) {
    const int nh = std::min(P.sa_heads, H - h0);
    uint8_t* g = ws + P.oSA;
    bf16* qk = reinterpret_cast<bf16*>(g);
    g += P.qk_b * nh;
    const int sparts = 2 * (D / 256);
    float* sss = reinterpret_cast<float*>(g);                 // [nh][2n][t][sparts]
    float* sinv = sss + (size_t)nh * 2 * n * t * sparts;       // [nh][2n][t]
    g += P.sss_b * nh;
    bf16* vT = reinterpret_cast<bf16*>(g);
    g += P.vT_b * nh;
    float* Ssa = reinterpret_cast<float*>(g);
    g += a256((size_t)nh * P.sa_sub * P.Ssah_b);
    bf16* Psa = reinterpret_cast<bf16*>(g);
    // The P.v product reads v^T columns [t, tp) of each head against zero probabilities:
    // they must hold finite values, and the region is shared with the cross-attention phase.
    if (P.tp != t) CK(cudaMemsetAsync(vT, 0, P.vT_b * nh, s));
    {  // [q~ | k~] = RMSNorm(Z') [S_Q | S_K] + [b | b]  (2-pass), |.|^2 per head
      GemmParams p = gp(nh * t, 2 * n * D);
      add_pass(p, 0, 0, h0 * t, 0, D);
      add_pass(p, D, 0, h0 * t, 0, D);
      EpiAffine e;
      e.kind = vkind;
      e.out = qk;
      e.lo_off = D;
      e.om.rdiv = t;
      e.om.r1 = (int64_t)2 * n * t * 2 * D;
      e.om.r0 = 2 * D;
      e.om.cdiv = D;
      e.om.c1 = (int64_t)t * 2 * D;
      e.om.c0 = 1;
      e.bias = Bw.sbqk;
      e.sumsq = sss;
      e.ssm.rdiv = t;
      e.ssm.r1 = (int64_t)2 * n * t;
      e.ssm.r0 = 1;
      e.ssm.c0 = t;
      e.ss_seg = D;
      e.ss_parts = sparts;
      e.ss_block = t;
      e.vec_ok = 1;
      TRY(run_gemm256<STILL_K_SA_PROJ>(ctx, op(A1, rows, 2 * D), op(Bw.SqkT, (int64_t)2 * n * D, D),
                                       p, e, vfmt, s));
    }
    KLAUNCH(STILL_K_NORMS,
            launch_inv_norms(sss, (int64_t)nh * 2 * n * t, sparts, t, c.l2_eps, 1.f, sinv, s));
    {  // v^T = S_V^T RMSNorm(Z')^T  -> [nD][nh * tp]  (hi, then lo rows when exact);
       // one batch per bank, so that each bank's t columns start on a 64-column boundary
       // and are stored by whole-row vector writes
      GemmParams p = gp(n * D, t, nh, 1);
      p.b_r1 = t;
      add_pass(p, 0, 0, 0, h0 * t, D);
      if (vexact) add_pass(p, 0, D, 0, h0 * t, D);
      EpiAffine e;
      e.kind = vexact ? vkind : OUT_BF16;
      e.lo_off = (int64_t)n * D * nh * P.tp;
      e.out = vT;
      e.om.b1 = P.tp;
      e.om.r0 = (int64_t)nh * P.tp;
      e.om.c0 = 1;
      e.vec_ok = 1;
      TRY(run_gemm256<STILL_K_SA_V>(ctx, op(Bw.SvT, (int64_t)n * D, D), op(A1, rows, 2 * D), p, e,
                                    vfmt, s));
    }
    // Self heads [i0, i0 + ns) of the nh banks per pass (all n unless one bank is too big).
    for (int i0 = 0; i0 < n; i0 += P.sa_sub) {
      const int ns = std::min(P.sa_sub, n - i0);
      {  // S = scale * q~.k~ / (|q~| |k~|)  per (bank hh, self head i0 + bi), batch hh * ns + bi
        GemmParams p = gp(t, t, nh * ns, ns);
        p.a_r1 = (int64_t)2 * n * t;
        p.a_r0 = t;
        p.b_r1 = (int64_t)2 * n * t;
        p.b_r0 = t;
        add_pass(p, 0, 0, i0 * t, (n + i0) * t, D);
        add_pass(p, 0, D, i0 * t, (n + i0) * t, D);
        add_pass(p, D, 0, i0 * t, (n + i0) * t, D);
        EpiAffine e;
        e.kind = OUT_F32;
        e.out = Ssa;
        e.om.b1 = (int64_t)t * P.ldt;
        e.om.r0 = P.ldt;
        e.om.c0 = 1;
        e.alpha = scale;
        e.row_scale = sinv;
        e.rsm.bdiv = ns;
        e.rsm.b1 = (int64_t)2 * n * t;
        e.rsm.b0 = t;
        e.rsm.r0 = 1;
        e.rsm.k = (int64_t)i0 * t;
        e.col_scale = sinv;
        e.csm.bdiv = ns;
        e.csm.b1 = (int64_t)2 * n * t;
        e.csm.b0 = t;
        e.csm.c0 = 1;
        e.csm.k = (int64_t)(n + i0) * t;
        e.vec_ok = 1;
        e.tma_f32 = 1;
        const StoreView3D sv = store_view(Ssa, 4, t, t, (int64_t)nh * ns, P.ldt,
                                          (int64_t)t * P.ldt, 32, true);
        TRY(run_gemm256<STILL_K_SA_SCORES>(ctx, op(qk, (int64_t)nh * 2 * n * t, 2 * D),
                                           op(qk, (int64_t)nh * 2 * n * t, 2 * D), p, e, vfmt, s,
                                           &sv));
      }
      KLAUNCH(STILL_K_SA_SOFTMAX,
              launch_softmax(Ssa, (int64_t)nh * ns * t, t, P.ldt, Psa, P.tp,
                             f16v ? 3 : vexact ? 2 : 0, s));
      {  // heads = P v -> concat rows (h0 + hh) * t + j, columns (i0 + bi) * D + f
        // exact: P_hi v_hi + P_hi v_lo + P_lo v_hi, concat rows of hi | lo
        const int64_t cw = vexact ? 2 * (int64_t)n * D : (int64_t)n * D;  // concat row pitch
        GemmParams p = gp(t, D, nh * ns, ns);
        p.a_r1 = (int64_t)ns * t;
        p.a_r0 = t;
        p.b_r0 = D;
        p.b_k1 = P.tp;
        add_pass(p, 0, 0, 0, i0 * D, (int)P.tp);
        if (vexact) {
          add_pass(p, 0, 0, 0, n * D + i0 * D, (int)P.tp);
          add_pass(p, (int)P.tp, 0, 0, i0 * D, (int)P.tp);
        }
        EpiAffine e;
        e.kind = vexact ? vkind : OUT_BF16;
        e.lo_off = (int64_t)n * D;
        e.out = cat;
        e.om.bdiv = ns;
        e.om.b1 = (int64_t)t * cw;
        e.om.b0 = D;
        e.om.r0 = cw;
        e.om.c0 = 1;
        e.om.k = (int64_t)h0 * t * cw + (int64_t)i0 * D;
        e.vec_ok = 1;
        TRY(run_gemm256<STILL_K_SA_PV>(
            ctx, op(Psa, (int64_t)nh * ns * t, vexact ? 2 * P.tp : P.tp),
            op(vT, (vexact ? 2 : 1) * (int64_t)n * D, (int64_t)nh * P.tp), p, e, vfmt, s));
      }
    }
  }
  {  // Z'' = Z' + concat S_O  (hi | lo concat: 2 passes)
    GemmParams p = gp((int)rows, D);
    add_pass(p, 0, 0, 0, 0, n * D);
    if (vexact) add_pass(p, n * D, 0, 0, 0, n * D);
    EpiAffine e;
    const bool direct = last && (F == 0) && z3_bf16;
    e.kind = direct ? OUT_HILO : OUT_F32;
    e.out = direct ? Z3 : static_cast<void*>(Z2);
    e.lo_off = D;
    e.om.r0 = direct ? 2 * D : D;
    e.om.c0 = 1;
    e.res_kind = 1;
    e.res = Za;  // in place when the block has no cross-attention (Za = Z2): same thread
    e.resm.r0 = D;
    e.resm.c0 = 1;
    e.vec_ok = 1;
    TRY(run_gemm256<STILL_K_SO>(ctx, op(cat, rows, (vexact ? 2 : 1) * (int64_t)n * D),
                                op(Bw.SoT, D, (int64_t)n * D), p, e, vfmt, s));
  }
  if (F > 0) {
    // vexact: RMSNorm(Z'') and GELU(.) as hi | lo, both products in 2 passes
    KLAUNCH(STILL_K_NORM, launch_rmsnorm(Z2, 0, rows, D, D, c.rms_eps, A2, vexact ? 2 * D : D,
                                         vexact ? 1 : 0, s));
    {
      GemmParams p = gp((int)rows, F);
      add_pass(p, 0, 0, 0, 0, D);
      if (vexact) add_pass(p, D, 0, 0, 0, D);
      EpiAffine e;
      e.kind = vexact ? OUT_HILO : OUT_BF16;
      e.lo_off = F;
      e.out = Gb;
      e.om.r0 = vexact ? 2 * F : F;
      e.om.c0 = 1;
      e.gelu = 1;
      e.vec_ok = 1;
      TRY(run_gemm256<STILL_K_FFN1>(ctx, op(A2, rows, vexact ? 2 * D : D), op(Bw.W1T, F, D), p, e,
                                    1, s));
    }
    {
      GemmParams p = gp((int)rows, D);
      add_pass(p, 0, 0, 0, 0, F);
      if (vexact) add_pass(p, F, 0, 0, 0, F);
      EpiAffine e;
      const bool direct = last && z3_bf16;
      e.kind = direct ? OUT_HILO : OUT_F32;
      e.out = direct ? Z3 : static_cast<void*>(Z2);
      e.lo_off = D;
      e.om.r0 = direct ? 2 * D : D;
      e.om.c0 = 1;
      e.res_kind = 1;
      e.res = Z2;
      e.resm.r0 = D;
      e.resm.c0 = 1;
      e.vec_ok = 1;
      // In place (Z2 -> Z2) is safe: each element is read and written by the same thread.
      TRY(run_gemm256<STILL_K_FFN2>(ctx, op(Gb, rows, vexact ? 2 * F : F), op(Bw.W2T, D, F), p, e,
                                    1, s));
    }
  }
  }  // block bi
  if (!z3_bf16) {
    KLAUNCH(STILL_K_NORM, launch_rmsnorm(Z2, 0, rows, D, D, c.rms_eps, reinterpret_cast<bf16*>(Z3), 2 * D, 1, s));
  }
  {  // output heads (2-pass on the hi/lo latent state) + re-rotation
    GemmParams p = gp((int)rows, 2 * d);
    add_pass(p, 0, 0, 0, 0, D);
    add_pass(p, D, 0, 0, 0, D);
    EpiHeads e;
    e.ck = out.ck;
    e.cv = out.cv;
    e.st = out.st;
    e.sh = out.sh;
    e.t = t;
    e.d = d;
    e.rot = hrot;
    const int bn = 2 * d <= 128 ? 128 : 256;
    TRY(run_gemm<STILL_K_HEADS>(ctx, bn, op(Z3, rows, 2 * D), op(L.WhT, 2 * d, D), p, e, 1, s));
  }
  if (out.beta != nullptr) {  // beta = Z_out w_beta, shaped; T = the N entries replaced
    const double off = L.beta.mass_match == 0
                           ? 0.0
                           : std::log((double)N / (double)t) +
                                 (L.beta.mass_match == 2 ? (double)L.beta.log_x : 0.0);
    KLAUNCH(STILL_K_BETA, launch_beta(reinterpret_cast<const bf16*>(Z3), t, H, D, L.wbeta,
                                       L.beta.beta_max, (float)off, out.beta, s));
  }
  return STILL_OK;
}

KVSource single_source(const void* K, const void* V, const int64_t strides_kv[3], int64_t N) {
  KVSource src;
  src.K = static_cast<const bf16*>(K);
  src.V = static_cast<const bf16*>(V);
  src.sN = strides_kv[0];
  src.sH = strides_kv[1];
  src.n_split = N;
  return src;
}

still_status check_ctx_layer(still_ctx* ctx, int32_t layer, const LayerW** L) {
  if (ctx == nullptr) return STILL_ERR_INVALID_ARG;
  if (layer < 0 || layer >= (int32_t)ctx->layers.size() || !ctx->layers[layer].loaded)
    return STILL_ERR_NOT_LOADED;
  *L = &ctx->layers[layer];
  return STILL_OK;
}

// Loads one layer: latent banks, per-block weights, output heads (App. A). Block 0's latent
// queries are precomputed when they fit the eager limit; later blocks' queries depend on the
// latent state and are formed in each call, so their W_Q and b_Q are kept.
still_status load_layer(still_ctx* ctx, int32_t layer, const still_layer_config* cfg,
                        const void* Zsrc, const still_block_weights* blocks, const void* Wkey,
                        const void* Wval, void* stream) {
  if (ctx == nullptr || layer < 0 || Zsrc == nullptr || blocks == nullptr || Wkey == nullptr ||
      Wval == nullptr)
    return STILL_ERR_INVALID_ARG;
  TRY(check_cfg(cfg));
  const still_layer_config& c = *cfg;
  const int H = c.n_kv_heads, d = c.head_dim, D = c.d_latent, n = c.n_cross_heads,
            F = c.ffn_dim, T = c.t_max, NB = c.n_blocks;
  for (int b = 0; b < NB; ++b) {
    const still_block_weights& w = blocks[b];
    const bool ca = b == 0 || c.cross_every_block;
    const void* req_ca[] = {w.Wq, w.bq, w.Wk, w.bk, w.Wv, w.Wo};
    const void* req_sa[] = {w.Sq, w.sbq, w.Sk, w.sbk, w.Sv, w.So};
    if (ca)
      for (const void* p : req_ca)
        if (p == nullptr) return STILL_ERR_INVALID_ARG;
    for (const void* p : req_sa)
      if (p == nullptr) return STILL_ERR_INVALID_ARG;
    if (F > 0 && (w.W1 == nullptr || w.W2 == nullptr)) return STILL_ERR_INVALID_ARG;
  }
  CK(cudaSetDevice(ctx->device));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if ((int32_t)ctx->layers.size() <= layer) ctx->layers.resize(layer + 1);
  LayerW& L = ctx->layers[layer];
  if (L.loaded) {
    CK(cudaStreamSynchronize(s));
    free_layer(L);
  }
  L.cfg = c;
  if (L.cfg.logit_scale == 0) L.cfg.logit_scale = D;
  const int64_t nD = (int64_t)n * D;
  L.blk.resize(NB);
  L.qhat_lazy = (size_t)H * n * T * D * sizeof(float) > ctx->qhat_eager_limit;
  L.f16 = NB > 1;
  // The folded key path: no compactor RoPE, one block whose queries are precomputed, the fused
  // kernel (2d <= 256), and a padded x~ narrower than d_l (else projecting k is cheaper).
  L.Kp = (int)rup(2 * d + 1, 64);
  L.fold = ctx->key_fold && c.compactor_rope == 0 && NB == 1 && (d == 64 || d == 128) &&
           !L.qhat_lazy && L.Kp < D;
  auto fail = [&](still_status st) {
    cudaStreamSynchronize(s);
    free_layer(L);
    return st;
  };
  still_status st = STILL_OK;
  // ---- layer-level tensors
  if ((st = dalloc(L, &L.Z, (size_t)H * T * D)) != STILL_OK ||
      (st = dalloc(L, &L.WhT, (size_t)2 * d * D)) != STILL_OK ||
      (st = dalloc(L, &L.omega_b, (size_t)d / 2)) != STILL_OK ||
      (st = dalloc(L, &L.omega_c, (size_t)D / 2)) != STILL_OK ||
      (!L.qhat_lazy && (st = dalloc(L, &L.qhat, (size_t)H * n * T * D)) != STILL_OK))
    return fail(st);
  // Without compactor RoPE its frequencies are zero: every rotation is exactly the identity.
  if (launch_omega(L.omega_b, d / 2, d, c.rope_theta, s) != cudaSuccess ||
      (c.compactor_rope ? launch_omega(L.omega_c, D / 2, D, c.rope_theta_compactor, s)
                        : cudaMemsetAsync(L.omega_c, 0, sizeof(double) * (D / 2), s)) !=
          cudaSuccess ||
      cudaMemcpyAsync(L.Z, Zsrc, sizeof(bf16) * (size_t)H * T * D, cudaMemcpyDeviceToDevice, s) !=
          cudaSuccess ||
      launch_transpose(static_cast<const bf16*>(Wkey), D, d, L.WhT, 0, s) != cudaSuccess ||
      launch_transpose(static_cast<const bf16*>(Wval), D, d, L.WhT + (size_t)d * D, 0, s) !=
          cudaSuccess)
    return fail(STILL_ERR_CUDA);

  // ---- per-block tensors
  LayerW tmp;  // temporaries of the precompute
  auto body = [&]() -> still_status {
    for (int b = 0; b < NB; ++b) {
      const still_block_weights& w = blocks[b];
      BlockW& B = L.blk[b];
      B.has_ca = b == 0 || c.cross_every_block;
      TRY(dalloc(L, &B.SqkT, (size_t)2 * nD * D));
      TRY(dalloc(L, &B.sbqk, (size_t)2 * nD));
      TRY(dalloc(L, &B.SvT, (size_t)nD * D));
      TRY(dalloc(L, &B.SoT, (size_t)D * nD));
      CK(launch_transpose(static_cast<const bf16*>(w.Sq), D, nD, B.SqkT, 0, s));
      CK(launch_transpose(static_cast<const bf16*>(w.Sk), D, nD, B.SqkT + nD * D, 0, s));
      CK(launch_bias(static_cast<const bf16*>(w.sbq), static_cast<const bf16*>(w.sbk), nD, B.sbqk,
                     0, s));
      CK(launch_transpose(static_cast<const bf16*>(w.Sv), D, nD, B.SvT, 0, s));
      CK(launch_transpose(static_cast<const bf16*>(w.So), nD, D, B.SoT, 0, s));
      // The first block of a two-block layer runs its value chains in fp16 (with the fused
      // cross-attention kernel, 2d <= 256): its self-attention weights as fp16 copies.
      const bool f16v = L.f16 && b + 1 < NB && (d == 64 || d == 128);
      if (f16v) {
        CK(launch_bf16_to_f16(B.SqkT, 2 * nD * D, s));
        CK(launch_bf16_to_f16(B.SvT, nD * D, s));
        CK(launch_bf16_to_f16(B.SoT, (int64_t)D * nD, s));
      }
      if (F > 0) {
        TRY(dalloc(L, &B.W1T, (size_t)F * D));
        TRY(dalloc(L, &B.W2T, (size_t)D * F));
        CK(launch_transpose(static_cast<const bf16*>(w.W1), D, F, B.W1T, 0, s));
        CK(launch_transpose(static_cast<const bf16*>(w.W2), F, D, B.W2T, 0, s));
      }
      if (!B.has_ca) continue;
      TRY(dalloc(L, &B.WkT, (size_t)nD * 2 * d));
      TRY(dalloc(L, &B.bk, (size_t)nD));
      TRY(dalloc(L, &B.WvoT, (size_t)D * 2 * n * 2 * d));
      CK(launch_transpose(static_cast<const bf16*>(w.Wk), 2 * d, nD, B.WkT, D, s));
      if (L.f16) CK(launch_bf16_to_f16(B.WkT, (int64_t)nD * 2 * d, s));
      CK(launch_bias(static_cast<const bf16*>(w.bk), nullptr, nD, B.bk, D, s));
      // W_Q and b_Q: kept when the block's queries are formed per call, else temporaries.
      const bool keep_q = b > 0 || L.qhat_lazy;
      LayerW& qown = keep_q ? L : tmp;
      bf16* WqT = nullptr;
      float* bq = nullptr;
      TRY(dalloc(qown, &WqT, (size_t)nD * D));
      TRY(dalloc(qown, &bq, (size_t)nD));
      CK(launch_transpose(static_cast<const bf16*>(w.Wq), D, nD, WqT, D, s));
      if (L.f16) CK(launch_bf16_to_f16(WqT, (int64_t)nD * D, s));
      CK(launch_bias(static_cast<const bf16*>(w.bq), nullptr, nD, bq, D, s));
      if (keep_q) {
        B.WqT = WqT;
        B.bq = bq;
      } else {  // q~ = RMSNorm(Z) W_Q + b_Q  (2-pass), |q~|^2 per (row, head), then L2 norm
        bf16* Zn = nullptr;
        float* qss = nullptr;
        TRY(dalloc(tmp, &Zn, (size_t)H * T * 2 * D));
        TRY(dalloc(tmp, &qss, (size_t)H * n * T * (2 * (D / 256) + 1)));
        CK(launch_rmsnorm(Zsrc, 1, (int64_t)H * T, D, D, c.rms_eps, Zn, 2 * D, L.f16 ? 2 : 1, s));
        GemmParams p = gp(H * T, (int)nD);
        add_pass(p, 0, 0, 0, 0, D);
        add_pass(p, D, 0, 0, 0, D);
        EpiAffine e;
        e.kind = OUT_F32;
        e.out = L.qhat;
        e.om.rdiv = T;
        e.om.r1 = (int64_t)n * T * D;
        e.om.r0 = D;
        e.om.cdiv = D;
        e.om.c1 = (int64_t)T * D;
        e.om.c0 = 1;
        e.bias = bq;
        e.sumsq = qss;
        e.ssm.rdiv = T;
        e.ssm.r1 = (int64_t)n * T;
        e.ssm.r0 = 1;
        e.ssm.c0 = T;
        e.ss_seg = D;
        e.ss_parts = 2 * (D / 256);
        e.ss_block = T;
        e.vec_ok = 1;
        TRY(run_gemm256<STILL_K_LOAD>(ctx, op(Zn, (int64_t)H * T, 2 * D), op(WqT, nD, D), p, e,
                                      L.f16 ? 0 : 1, s));
        const int64_t nq = (int64_t)H * n * T;
        float* qinv = qss + nq * (2 * (D / 256));
        CK(launch_inv_norms(qss, nq, 2 * (D / 256), T, c.l2_eps, 1.f, qinv, s));
        CK(launch_scale_rows(L.qhat, qinv, nq, D, s));
      }
      // W_VO,i = W_V,i W_O,i  -> stored transposed as hi | lo: WvoT[c][i*2d + f]
      bf16* WoT = nullptr;
      TRY(dalloc(tmp, &WoT, (size_t)D * nD));
      CK(launch_transpose(static_cast<const bf16*>(w.Wo), nD, D, WoT, 0, s));
      GemmParams p = gp(2 * d, D, n, 1);
      p.a_k1 = D;
      p.b_k1 = D;
      add_pass(p, 0, 0, 0, 0, D);
      EpiAffine e;
      e.kind = f16v ? OUT_HILO16 : OUT_HILO;
      e.alpha = f16v ? kWvoScale : 1.f;
      e.out = B.WvoT;
      e.lo_off = (int64_t)n * 2 * d;
      e.om.b1 = 2 * d;
      e.om.r0 = 1;
      e.om.c0 = (int64_t)2 * n * 2 * d;
      e.vec_ok = 0;
      TRY(run_gemm256<STILL_K_LOAD>(ctx, op(w.Wv, 2 * d, nD), op(WoT, D, nD), p, e, 1, s));
    }
    return STILL_OK;
  };
  st = body();
  if (st == STILL_OK && L.fold) {  // u = W~_i q^ and G_i = W~_i W~_i^T, hi | lo (block 0)
    auto fold = [&]() -> still_status {
      const BlockW& B0 = L.blk[0];
      const int Kp = L.Kp;
      bf16* Wt = nullptr;
      bf16* qhl = nullptr;
      TRY(dalloc(tmp, &Wt, (size_t)n * Kp * D));
      TRY(dalloc(tmp, &qhl, (size_t)H * n * T * 2 * D));
      TRY(dalloc(L, &L.U, (size_t)H * n * T * 2 * Kp));
      TRY(dalloc(L, &L.G, (size_t)n * Kp * 2 * Kp));
      CK(launch_fold_weights(B0.WkT, B0.bk, (int)n, D, 2 * d, Kp, Wt, s));
      CK(launch_f32_hilo(L.qhat, (int64_t)H * n * T, D, qhl, s));
      {  // U rows (h, i, m): batch b = h n + i over q^ hi | lo (2 passes) x W~_i
        GemmParams p = gp(T, Kp, H * (int)n, (int)n);
        p.a_r1 = n * T;
        p.a_r0 = T;
        p.b_r1 = 0;
        p.b_r0 = Kp;
        add_pass(p, 0, 0, 0, 0, D);
        add_pass(p, D, 0, 0, 0, D);
        EpiAffine e;
        e.kind = OUT_HILO;
        e.out = L.U;
        e.lo_off = Kp;
        e.om.b1 = n * T * 2 * Kp;
        e.om.b0 = T * 2 * Kp;
        e.om.bdiv = n;
        e.om.r0 = 2 * Kp;
        e.om.c0 = 1;
        e.vec_ok = 0;
        TRY(run_gemm256<STILL_K_LOAD>(ctx, op(qhl, (int64_t)H * n * T, 2 * D),
                                      op(Wt, (int64_t)n * Kp, D), p, e, 1, s));
      }
      {  // G_i = W~_i W~_i^T (bf16 operands, exact products)
        GemmParams p = gp(Kp, Kp, (int)n, 1);
        p.a_r1 = Kp;
        p.b_r1 = Kp;
        add_pass(p, 0, 0, 0, 0, D);
        EpiAffine e;
        e.kind = OUT_HILO;
        e.out = L.G;
        e.lo_off = Kp;
        e.om.b1 = (int64_t)Kp * 2 * Kp;
        e.om.r0 = 2 * Kp;
        e.om.c0 = 1;
        e.vec_ok = 0;
        TRY(run_gemm256<STILL_K_LOAD>(ctx, op(Wt, (int64_t)n * Kp, D), op(Wt, (int64_t)n * Kp, D),
                                      p, e, 1, s));
      }
      return STILL_OK;
    };
    st = fold();
  }
  cudaStreamSynchronize(s);
  free_layer(tmp);
  if (st != STILL_OK) return fail(st);
  L.loaded = true;
  return STILL_OK;
}

}  // namespace

// ============================================================================== fixed scratch

// Scratch of still_compact_layer_noalloc: a file-scope device array, so that the entry point
// never allocates. Every device that loads this library holds it until the process exits.
constexpr size_t kNoAllocScratchBytes = size_t(STILL_NOALLOC_SCRATCH_MIB) << 20;
static __device__ __align__(256) uint8_t g_noalloc_scratch[kNoAllocScratchBytes];

namespace {

constexpr int kMaxDevices = 64;
std::mutex g_noalloc_mu;
uint8_t* g_noalloc_ptr[kMaxDevices] = {nullptr};

// Device address of the scratch array on `device` (which must be current). The host-side name
// g_noalloc_scratch is only a stand-in symbol: kernels must be given this address instead.
still_status noalloc_scratch(int device, uint8_t** out) {
  if (device < 0 || device >= kMaxDevices) return STILL_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lk(g_noalloc_mu);
  if (g_noalloc_ptr[device] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) {
      cudaGetLastError();
      return STILL_ERR_CUDA;
    }
    g_noalloc_ptr[device] = static_cast<uint8_t*>(p);
  }
  *out = g_noalloc_ptr[device];
  return STILL_OK;
}

}  // namespace

// ============================================================================== C ABI

extern "C" {

const char* still_status_string(still_status s) {
  switch (s) {
    case STILL_OK: return "ok";
    case STILL_ERR_INVALID_ARG: return "invalid argument";
    case STILL_ERR_UNSUPPORTED: return "unsupported configuration";
    case STILL_ERR_SHAPE: return "inconsistent shape";
    case STILL_ERR_ALIGNMENT: return "misaligned pointer or stride";
    case STILL_ERR_NOT_LOADED: return "layer weights not loaded";
    case STILL_ERR_OOM: return "out of device memory or workspace limit";
    case STILL_ERR_CUDA: return "CUDA error";
    case STILL_ERR_TIMEOUT: return "device-side wait timed out";
  }
  return "unknown status";
}

still_status still_create(int device, still_ctx** out) {
  if (out == nullptr) return STILL_ERR_INVALID_ARG;
  *out = nullptr;
  int ndev = 0;
  if (cudaGetDeviceCount(&ndev) != cudaSuccess || device < 0 || device >= ndev) {
    cudaGetLastError();
    return STILL_ERR_INVALID_ARG;
  }
  CK(cudaSetDevice(device));
  int major = 0, minor = 0;
  CK(cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, device));
  CK(cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, device));
  if (major != 10 || minor != 3) return STILL_ERR_UNSUPPORTED;  // built for sm_103a only
  still_ctx* c = new still_ctx();
  c->device = device;
  if (cudaDeviceGetAttribute(&c->nsm, cudaDevAttrMultiProcessorCount, device) != cudaSuccess ||
      cudaMalloc(&c->err, 4 * sizeof(int)) != cudaSuccess ||
      cudaMemset(c->err, 0, 4 * sizeof(int)) != cudaSuccess) {
    delete c;
    return STILL_ERR_CUDA;
  }
  *out = c;
  return STILL_OK;
}

still_status still_destroy(still_ctx* ctx) {
  if (ctx == nullptr) return STILL_ERR_INVALID_ARG;
  cudaSetDevice(ctx->device);
  cudaDeviceSynchronize();
  for (auto& L : ctx->layers) free_layer(L);
  if (ctx->ws) cudaFree(ctx->ws);
  if (ctx->err) cudaFree(ctx->err);
  delete ctx;
  return STILL_OK;
}

still_status still_set_qhat_eager_limit(still_ctx* ctx, size_t bytes) {
  if (ctx == nullptr) return STILL_ERR_INVALID_ARG;
  ctx->qhat_eager_limit = bytes;
  return STILL_OK;
}

still_status still_set_key_fold(still_ctx* ctx, int32_t enable) {
  if (ctx == nullptr || (enable != 0 && enable != 1)) return STILL_ERR_INVALID_ARG;
  ctx->key_fold = enable != 0;
  return STILL_OK;
}

still_status still_set_workspace_limit(still_ctx* ctx, size_t bytes) {
  if (ctx == nullptr || bytes == 0) return STILL_ERR_INVALID_ARG;
  ctx->ws_limit = bytes;
  return STILL_OK;
}

still_status still_load_layer_weights(still_ctx* ctx, int32_t layer,
                                      const still_layer_config* cfg,
                                      const still_layer_weights* w, void* stream) {
  if (w == nullptr) return STILL_ERR_INVALID_ARG;
  if (cfg != nullptr && cfg->n_blocks != 1) return STILL_ERR_INVALID_ARG;
  const still_block_weights blk = {w->Wq, w->bq, w->Wk, w->bk, w->Wv, w->Wo, w->Sq,
                                   w->sbq, w->Sk, w->sbk, w->Sv, w->So, w->W1, w->W2};
  return load_layer(ctx, layer, cfg, w->Z, &blk, w->Wkey, w->Wval, stream);
}

still_status still_load_layer_weights_blocks(still_ctx* ctx, int32_t layer,
                                             const still_layer_config* cfg, const void* Z,
                                             const still_block_weights* blocks, const void* Wkey,
                                             const void* Wval, void* stream) {
  return load_layer(ctx, layer, cfg, Z, blocks, Wkey, Wval, stream);
}

namespace {

// noalloc: run in the library's fixed device scratch (still_compact_layer_noalloc) instead of
// the context's growable workspace, with event timing suspended on this thread.
still_status compact_layer_impl(still_ctx* ctx, int32_t layer, const void* K, const void* V,
                                const int64_t strides_kv[3],
                                const still_pos_segment* h_segments, int32_t n_segments,
                                int64_t N, int32_t t, void* Ck, void* Cv, float* beta,
                                double* h_out_pos_start, double* h_out_pos_step,
                                int64_t* h_pos_offset, void* stream, bool noalloc = false) {
  const LayerW* L = nullptr;
  TRY(check_ctx_layer(ctx, layer, &L));
  if (beta != nullptr && (L->wbeta == nullptr || (reinterpret_cast<uintptr_t>(beta) & 3)))
    return L->wbeta == nullptr ? STILL_ERR_NOT_LOADED : STILL_ERR_ALIGNMENT;
  if (K == nullptr || V == nullptr || Ck == nullptr || Cv == nullptr || strides_kv == nullptr)
    return STILL_ERR_INVALID_ARG;
  if (N < 1 || t < 1 || t > N || t > L->cfg.t_max || N > (int64_t(1) << 30))
    return STILL_ERR_SHAPE;
  if (strides_kv[2] != 1 || strides_kv[0] < 1 || strides_kv[1] < 0) return STILL_ERR_SHAPE;
  if (((reinterpret_cast<uintptr_t>(K) | reinterpret_cast<uintptr_t>(V)) & 1) ||
      ((reinterpret_cast<uintptr_t>(Ck) | reinterpret_cast<uintptr_t>(Cv)) & 15))
    return STILL_ERR_ALIGNMENT;
  Positions pos;
  TRY(make_positions(h_segments, n_segments, N, pos));
  CK(cudaSetDevice(ctx->device));
  const int H = L->cfg.n_kv_heads, d = L->cfg.head_dim;
  OutSpec o{static_cast<bf16*>(Ck), static_cast<bf16*>(Cv), (int64_t)H * d, d};
  o.beta = beta;
  if (noalloc) {
    uint8_t* scratch = nullptr;
    TRY(noalloc_scratch(ctx->device, &scratch));
    bool& untimed = Profiler::untimed_thread();
    untimed = true;
    const still_status st =
        compact_one(ctx, *L, single_source(K, V, strides_kv, N), pos, N, t, o,
                    static_cast<cudaStream_t>(stream), scratch, kNoAllocScratchBytes);
    untimed = false;
    TRY(st);  // STILL_ERR_OOM: even the smallest grouping needs more than the fixed scratch
  } else {
    TRY(compact_one(ctx, *L, single_source(K, V, strides_kv, N), pos, N, t, o,
                    static_cast<cudaStream_t>(stream)));
  }
  if (h_out_pos_start) *h_out_pos_start = pos.pmin;
  if (h_out_pos_step) *h_out_pos_step = t > 1 ? (pos.pmax - pos.pmin) / (double)(t - 1) : 0.0;
  if (h_pos_offset) *h_pos_offset = N - t;
  return STILL_OK;
}

}  // namespace

still_status still_compact_layer(still_ctx* ctx, int32_t layer, const void* K, const void* V,
                                 const int64_t strides_kv[3],
                                 const still_pos_segment* h_segments, int32_t n_segments,
                                 int64_t N, int32_t t, void* Ck, void* Cv,
                                 double* h_out_pos_start, double* h_out_pos_step,
                                 int64_t* h_pos_offset, void* stream) {
  return compact_layer_impl(ctx, layer, K, V, strides_kv, h_segments, n_segments, N, t, Ck, Cv,
                            nullptr, h_out_pos_start, h_out_pos_step, h_pos_offset, stream);
}

still_status still_compact_layer_beta(still_ctx* ctx, int32_t layer, const void* K,
                                      const void* V, const int64_t strides_kv[3],
                                      const still_pos_segment* h_segments, int32_t n_segments,
                                      int64_t N, int32_t t, void* Ck, void* Cv, float* beta,
                                      double* h_out_pos_start, double* h_out_pos_step,
                                      int64_t* h_pos_offset, void* stream) {
  if (beta == nullptr) return STILL_ERR_INVALID_ARG;
  return compact_layer_impl(ctx, layer, K, V, strides_kv, h_segments, n_segments, N, t, Ck, Cv,
                            beta, h_out_pos_start, h_out_pos_step, h_pos_offset, stream);
}

still_status still_set_beta_head(still_ctx* ctx, int32_t layer, const void* w_beta,
                                 const still_beta_config* bc, void* stream) {
  if (ctx == nullptr || w_beta == nullptr || bc == nullptr) return STILL_ERR_INVALID_ARG;
  if (layer < 0 || layer >= (int32_t)ctx->layers.size() || !ctx->layers[layer].loaded)
    return STILL_ERR_NOT_LOADED;
  if (!(bc->beta_max >= 0.f) || !std::isfinite(bc->beta_max) || bc->mass_match < 0 ||
      bc->mass_match > 2 || !std::isfinite(bc->log_x))
    return STILL_ERR_INVALID_ARG;
  LayerW& L = ctx->layers[layer];
  CK(cudaSetDevice(ctx->device));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int D = L.cfg.d_latent;
  if (L.wbeta == nullptr) TRY(dalloc(L, &L.wbeta, (size_t)D));
  CK(launch_bias(static_cast<const bf16*>(w_beta), nullptr, D, L.wbeta, 0, s));
  L.beta = *bc;
  return STILL_OK;
}

}  // extern "C"

namespace {

// The decode-time attention of n_layers layers of one shape, in one launch of the chunk kernel
// and one of the merge. Pointer arrays are host arrays of device pointers.
still_status attend_biased_impl(still_ctx* ctx, int32_t n_layers, const void* const* q,
                                int32_t nq, int32_t Hq, const void* const* Ck,
                                const void* const* Cv, const float* const* beta, int64_t t,
                                const void* const* Kfix, const void* const* Vfix, int64_t S,
                                int32_t H, int32_t d, float scale, void* const* out,
                                void* stream) {
  if (ctx == nullptr || q == nullptr || out == nullptr) return STILL_ERR_INVALID_ARG;
  if (n_layers < 1 || n_layers > kDecodeMaxLayers) return STILL_ERR_UNSUPPORTED;
  if (nq < 1 || H < 1 || Hq < H || Hq % H != 0 || t < 0 || S < 0 || t + S < 1 ||
      (t > 0 && (Ck == nullptr || Cv == nullptr)) || (S > 0 && (Kfix == nullptr || Vfix == nullptr)))
    return STILL_ERR_INVALID_ARG;
  if ((d != 64 && d != 128 && d != 256) || (int64_t)nq * (Hq / H) > 64 ||
      t + S > (int64_t(1) << 31) - 128)
    return STILL_ERR_UNSUPPORTED;
  if (!(scale >= 0.f) || !std::isfinite(scale)) return STILL_ERR_INVALID_ARG;
  DecodeStack st;
  st.n = n_layers;
  for (int l = 0; l < n_layers; ++l) {
    const void* ck = t > 0 ? Ck[l] : nullptr;
    const void* cv = t > 0 ? Cv[l] : nullptr;
    const void* kf = S > 0 ? Kfix[l] : nullptr;
    const void* vf = S > 0 ? Vfix[l] : nullptr;
    const float* b = beta != nullptr ? beta[l] : nullptr;
    if (q[l] == nullptr || out[l] == nullptr || (t > 0 && (ck == nullptr || cv == nullptr)) ||
        (S > 0 && (kf == nullptr || vf == nullptr)))
      return STILL_ERR_INVALID_ARG;
    const uintptr_t al = reinterpret_cast<uintptr_t>(q[l]) | reinterpret_cast<uintptr_t>(out[l]) |
                         reinterpret_cast<uintptr_t>(ck) | reinterpret_cast<uintptr_t>(cv) |
                         reinterpret_cast<uintptr_t>(kf) | reinterpret_cast<uintptr_t>(vf);
    if ((al & 15) || (reinterpret_cast<uintptr_t>(b) & 3)) return STILL_ERR_ALIGNMENT;
    DecodeArgs& a = st.layer[l];
    a.q = static_cast<const bf16*>(q[l]);
    a.Ck = static_cast<const bf16*>(ck);
    a.Cv = static_cast<const bf16*>(cv);
    a.beta = b;
    a.Kf = static_cast<const bf16*>(kf);
    a.Vf = static_cast<const bf16*>(vf);
    a.out = static_cast<bf16*>(out[l]);
    a.t = t;
    a.S = S;
    a.cst = (int64_t)H * d;
    a.fst = (int64_t)H * d;
    a.nq = nq;
    a.Hq = Hq;
    a.H = H;
    a.d = d;
    a.scale = scale > 0.f ? scale : 1.f / std::sqrt((float)d);
  }
  CK(cudaSetDevice(ctx->device));
  TRY(ensure_ws(ctx, decode_workspace_bytes((int64_t)nq * Hq, t + S, d, n_layers)));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  ctx->prof.begin(STILL_K_DECODE, s);
  cudaError_t r = launch_decode_biased(st, ctx->ws, ctx->nsm, s);
  ctx->prof.end(STILL_K_DECODE, s);
  ctx->prof.launches[STILL_K_DECODE] += 1;  // the merge kernel (begin counted the first)
  if (r != cudaSuccess) return STILL_ERR_CUDA;
  return STILL_OK;
}

}  // namespace

extern "C" {

still_status still_attend_biased(still_ctx* ctx, const void* q, int32_t nq, int32_t Hq,
                                 const void* Ck, const void* Cv, const float* beta, int64_t t,
                                 const void* Kfix, const void* Vfix, int64_t S, int32_t H,
                                 int32_t d, float scale, void* out, void* stream) {
  return attend_biased_impl(ctx, 1, &q, nq, Hq, &Ck, &Cv, &beta, t, &Kfix, &Vfix, S, H, d, scale,
                            &out, stream);
}

still_status still_attend_biased_stack(still_ctx* ctx, int32_t n_layers, const void* const* q,
                                       int32_t nq, int32_t Hq, const void* const* Ck,
                                       const void* const* Cv, const float* const* beta, int64_t t,
                                       const void* const* Kfix, const void* const* Vfix,
                                       int64_t S, int32_t H, int32_t d, float scale,
                                       void* const* out, void* stream) {
  return attend_biased_impl(ctx, n_layers, q, nq, Hq, Ck, Cv, beta, t, Kfix, Vfix, S, H, d,
                            scale, out, stream);
}

still_status still_compact_layer_noalloc(still_ctx* ctx, int32_t layer, const void* K,
                                         const void* V, const int64_t strides_kv[3],
                                         const still_pos_segment* h_segments,
                                         int32_t n_segments, int64_t N, int32_t t, void* Ck,
                                         void* Cv, double* h_out_pos_start,
                                         double* h_out_pos_step, int64_t* h_pos_offset,
                                         void* stream) {
  return compact_layer_impl(ctx, layer, K, V, strides_kv, h_segments, n_segments, N, t, Ck, Cv,
                            nullptr, h_out_pos_start, h_out_pos_step, h_pos_offset, stream,
                            true);
}

still_status still_compact_stack(still_ctx* ctx, int32_t n_layers, const void* const* K,
                                 const void* const* V, const int64_t strides_kv[3],
                                 const still_pos_segment* h_segments, int32_t n_segments,
                                 int64_t N, int32_t t, void* const* Ck, void* const* Cv,
                                 double* h_out_pos_start, double* h_out_pos_step,
                                 int64_t* h_pos_offset, void* stream) {
  if (ctx == nullptr || K == nullptr || V == nullptr || Ck == nullptr || Cv == nullptr ||
      n_layers < 1)
    return STILL_ERR_INVALID_ARG;
  for (int l = 0; l < n_layers; ++l) {
    const LayerW* L = nullptr;
    TRY(check_ctx_layer(ctx, l, &L));
  }
  for (int l = 0; l < n_layers; ++l)
    TRY(still_compact_layer(ctx, l, K[l], V[l], strides_kv, h_segments, n_segments, N, t, Ck[l],
                            Cv[l], h_out_pos_start, h_out_pos_step, h_pos_offset, stream));
  return STILL_OK;
}

still_status still_compact_stack_masked(still_ctx* ctx, int32_t n_layers,
                                        const uint8_t* h_compact_layer, const void* const* K,
                                        const void* const* V, const int64_t strides_kv[3],
                                        const still_pos_segment* h_segments, int32_t n_segments,
                                        int64_t N, int32_t t, void* const* Ck, void* const* Cv,
                                        double* h_out_pos_start, double* h_out_pos_step,
                                        int64_t* h_pos_offset, void* stream) {
  if (ctx == nullptr || h_compact_layer == nullptr || K == nullptr || V == nullptr ||
      Ck == nullptr || Cv == nullptr || n_layers < 1)
    return STILL_ERR_INVALID_ARG;
  for (int l = 0; l < n_layers; ++l) {
    if (!h_compact_layer[l]) continue;
    const LayerW* L = nullptr;
    TRY(check_ctx_layer(ctx, l, &L));
  }
  for (int l = 0; l < n_layers; ++l)
    if (h_compact_layer[l])
      TRY(still_compact_layer(ctx, l, K[l], V[l], strides_kv, h_segments, n_segments, N, t,
                              Ck[l], Cv[l], h_out_pos_start, h_out_pos_step, h_pos_offset,
                              stream));
  return STILL_OK;
}

// ------------------------------------------------------------------ lookahead chunked schedule

still_status still_lookahead_pass_info(int64_t k, int64_t c, int32_t t,
                                       still_lookahead_pass* out) {
  constexpr int64_t kExact = int64_t(1) << 53;  // positions stay exact in fp64
  if (out == nullptr || k < 0 || c < 1 || t < 1) return STILL_ERR_INVALID_ARG;
  if (c > kExact / t) return STILL_ERR_INVALID_ARG;
  const int64_t ct = c * t;
  if (k + 2 > kExact / ct) return STILL_ERR_INVALID_ARG;  // (k + 2) ct bounds every field
  still_lookahead_pass r;
  r.chunk_start = k * ct;
  r.chunk_len = ct;
  r.prefill_start = k == 0 ? 0 : (k + 1) * ct;
  r.prefill_len = k == 0 ? 2 * ct : ct;
  r.prefill_past = k == 0 ? 0 : (k + c) * (int64_t)t;
  r.compact_row = k * t;
  r.retained_after = (k + 1) * t + ct;
  r.logical_after = (k + 2) * ct;
  r.pos_offset_after = r.logical_after - r.retained_after;
  *out = r;
  return STILL_OK;
}

still_status still_lookahead_totals(int64_t T, int64_t c, int32_t t, int64_t* h_passes,
                                    int64_t* h_retained) {
  if (h_passes == nullptr || h_retained == nullptr || c < 1 || t < 1 || T < 1)
    return STILL_ERR_INVALID_ARG;
  if (c > (int64_t(1) << 53) / t) return STILL_ERR_INVALID_ARG;
  const int64_t ct = c * t;
  if (T % ct != 0) return STILL_ERR_SHAPE;
  still_lookahead_pass last;
  TRY(still_lookahead_pass_info(T / ct - 1, c, t, &last));
  *h_passes = T / ct;
  *h_retained = last.retained_after;
  return STILL_OK;
}

namespace {

// Packed-chunk ragged arguments of one lookahead step: sequence b holds c*t tokens at
// positions k_b*c*t + i and t output slots.
struct LookaheadArgs {
  std::vector<int64_t> cu_seq, cu_t;
  std::vector<int32_t> ts, seg_per_seq;
  std::vector<still_pos_segment> segs;
};

still_status lookahead_args(int32_t B, const int64_t* h_pass, int64_t c, int32_t t,
                            LookaheadArgs& a) {
  if (B < 1 || h_pass == nullptr) return STILL_ERR_INVALID_ARG;
  a.cu_seq.assign(B + 1, 0);
  a.cu_t.assign(B + 1, 0);
  a.ts.assign(B, t);
  a.seg_per_seq.assign(B, 1);
  a.segs.resize(B);
  for (int b = 0; b < B; ++b) {
    still_lookahead_pass ps;
    TRY(still_lookahead_pass_info(h_pass[b], c, t, &ps));
    a.cu_seq[b + 1] = a.cu_seq[b] + ps.chunk_len;
    a.cu_t[b + 1] = a.cu_t[b] + t;
    a.segs[b] = still_pos_segment{(double)ps.chunk_start, 1.0, ps.chunk_len};
  }
  return STILL_OK;
}

}  // namespace

still_status still_lookahead_compact_layer(still_ctx* ctx, int32_t layer, int32_t B,
                                           const void* K, const void* V, const int64_t* h_pass,
                                           int64_t c, int32_t t, void* Ck, void* Cv,
                                           void* stream) {
  LookaheadArgs a;
  TRY(lookahead_args(B, h_pass, c, t, a));
  return still_compact_layer_ragged(ctx, layer, K, V, a.cu_seq.data(), B, a.segs.data(),
                                    a.seg_per_seq.data(), a.ts.data(), a.cu_t.data(), Ck, Cv,
                                    nullptr, stream);
}

still_status still_lookahead_compact_stack(still_ctx* ctx, int32_t n_layers,
                                           const uint8_t* h_compact_layer, int32_t B,
                                           const void* const* K, const void* const* V,
                                           const int64_t* h_pass, int64_t c, int32_t t,
                                           void* const* Ck, void* const* Cv, void* stream) {
  if (ctx == nullptr || K == nullptr || V == nullptr || Ck == nullptr || Cv == nullptr ||
      n_layers < 1)
    return STILL_ERR_INVALID_ARG;
  LookaheadArgs a;
  TRY(lookahead_args(B, h_pass, c, t, a));
  for (int l = 0; l < n_layers; ++l) {
    if (h_compact_layer != nullptr && !h_compact_layer[l]) continue;
    const LayerW* L = nullptr;
    TRY(check_ctx_layer(ctx, l, &L));
  }
  for (int l = 0; l < n_layers; ++l) {
    if (h_compact_layer != nullptr && !h_compact_layer[l]) continue;
    TRY(still_compact_layer_ragged(ctx, l, K[l], V[l], a.cu_seq.data(), B, a.segs.data(),
                                   a.seg_per_seq.data(), a.ts.data(), a.cu_t.data(), Ck[l],
                                   Cv[l], nullptr, stream));
  }
  return STILL_OK;
}

still_status still_compact_layer_ragged(still_ctx* ctx, int32_t layer, const void* Kpacked,
                                        const void* Vpacked, const int64_t* h_cu_seqlens,
                                        int32_t B, const still_pos_segment* h_segments,
                                        const int32_t* h_seg_per_seq, const int32_t* h_t,
                                        const int64_t* h_cu_t, void* Ck, void* Cv,
                                        int64_t* h_pos_offset, void* stream) {
  const LayerW* L = nullptr;
  TRY(check_ctx_layer(ctx, layer, &L));
  if (Kpacked == nullptr || Vpacked == nullptr || h_cu_seqlens == nullptr || h_t == nullptr ||
      h_cu_t == nullptr || Ck == nullptr || Cv == nullptr || B < 1)
    return STILL_ERR_INVALID_ARG;
  if ((h_segments == nullptr) != (h_seg_per_seq == nullptr)) return STILL_ERR_INVALID_ARG;
  if (h_cu_seqlens[0] != 0 || h_cu_t[0] != 0) return STILL_ERR_SHAPE;
  for (int b = 0; b < B; ++b) {
    if (h_cu_seqlens[b + 1] < h_cu_seqlens[b] || h_cu_t[b + 1] - h_cu_t[b] != h_t[b])
      return STILL_ERR_SHAPE;
    const int64_t Nb = h_cu_seqlens[b + 1] - h_cu_seqlens[b];
    if (Nb < 1 || h_t[b] < 1 || h_t[b] > Nb || h_t[b] > L->cfg.t_max) return STILL_ERR_SHAPE;
  }
  const int H = L->cfg.n_kv_heads, d = L->cfg.head_dim;
  const int64_t row = (int64_t)H * d;
  const int64_t strides[3] = {row, d, 1};
  int seg0 = 0;
  for (int b = 0; b < B; ++b) {
    const int64_t Nb = h_cu_seqlens[b + 1] - h_cu_seqlens[b];
    const still_pos_segment* sg = h_segments ? h_segments + seg0 : nullptr;
    const int nsg = h_seg_per_seq ? h_seg_per_seq[b] : 0;
    seg0 += nsg;
    TRY(still_compact_layer(
        ctx, layer, static_cast<const bf16*>(Kpacked) + h_cu_seqlens[b] * row,
        static_cast<const bf16*>(Vpacked) + h_cu_seqlens[b] * row, strides, sg, nsg, Nb, h_t[b],
        static_cast<bf16*>(Ck) + h_cu_t[b] * row, static_cast<bf16*>(Cv) + h_cu_t[b] * row,
        nullptr, nullptr, h_pos_offset ? h_pos_offset + b : nullptr, stream));
  }
  return STILL_OK;
}

still_status still_compact_stack_ragged(still_ctx* ctx, int32_t n_layers,
                                        const void* const* Kpacked, const void* const* Vpacked,
                                        const int64_t* h_cu_seqlens, int32_t B,
                                        const still_pos_segment* h_segments,
                                        const int32_t* h_seg_per_seq, const int32_t* h_t,
                                        const int64_t* h_cu_t, void* const* Ck,
                                        void* const* Cv, int64_t* h_pos_offset, void* stream) {
  if (ctx == nullptr || Kpacked == nullptr || Vpacked == nullptr || Ck == nullptr ||
      Cv == nullptr || n_layers < 1)
    return STILL_ERR_INVALID_ARG;
  for (int l = 0; l < n_layers; ++l)
    TRY(still_compact_layer_ragged(ctx, l, Kpacked[l], Vpacked[l], h_cu_seqlens, B, h_segments,
                                   h_seg_per_seq, h_t, h_cu_t, Ck[l], Cv[l], h_pos_offset,
                                   stream));
  return STILL_OK;
}

still_status still_recompact_layer_ragged(still_ctx* ctx, int32_t layer, int32_t B,
                                          const void* Kprev, const void* Vprev,
                                          const int64_t* h_cu_prev, const int64_t* h_prev_len,
                                          const void* Knew, const void* Vnew,
                                          const int64_t* h_cu_new, int64_t ratio, void* Ck,
                                          void* Cv, int64_t* h_cu_out, int64_t* h_len_out,
                                          void* stream) {
  const LayerW* L = nullptr;
  TRY(check_ctx_layer(ctx, layer, &L));
  if (B < 1 || Kprev == nullptr || Vprev == nullptr || h_cu_prev == nullptr ||
      h_prev_len == nullptr || h_cu_new == nullptr || Ck == nullptr || Cv == nullptr ||
      h_cu_out == nullptr || ratio < 1)
    return STILL_ERR_INVALID_ARG;
  if (h_cu_prev[0] != 0 || h_cu_new[0] != 0) return STILL_ERR_SHAPE;
  const int H = L->cfg.n_kv_heads, d = L->cfg.head_dim;
  const int64_t row = (int64_t)H * d;
  // Budgets first (integers only): t_b = round((L_prev + new) / ratio).
  h_cu_out[0] = 0;
  for (int b = 0; b < B; ++b) {
    const int64_t tprev = h_cu_prev[b + 1] - h_cu_prev[b];
    const int64_t nnew = h_cu_new[b + 1] - h_cu_new[b];
    if (tprev < 1 || nnew < 0 || h_prev_len[b] < tprev) return STILL_ERR_SHAPE;
    if (nnew > 0 && (Knew == nullptr || Vnew == nullptr)) return STILL_ERR_INVALID_ARG;
    const int64_t Lr = h_prev_len[b] + nnew;
    const int64_t tb = std::max<int64_t>(1, still_budget(Lr, ratio));
    if (tb > tprev + nnew || tb > L->cfg.t_max) return STILL_ERR_SHAPE;
    h_cu_out[b + 1] = h_cu_out[b] + tb;
  }
  if (((reinterpret_cast<uintptr_t>(Ck) | reinterpret_cast<uintptr_t>(Cv)) & 15) ||
      ((reinterpret_cast<uintptr_t>(Kprev) | reinterpret_cast<uintptr_t>(Vprev)) & 1))
    return STILL_ERR_ALIGNMENT;
  CK(cudaSetDevice(ctx->device));
  for (int b = 0; b < B; ++b) {
    const int64_t tprev = h_cu_prev[b + 1] - h_cu_prev[b];
    const int64_t nnew = h_cu_new[b + 1] - h_cu_new[b];
    const int64_t Lp = h_prev_len[b];
    const int64_t N = tprev + nnew;
    const int t = (int)(h_cu_out[b + 1] - h_cu_out[b]);
    // Segment A: the previous compact slots at their output positions (evenly spaced over
    // [0, L_prev - 1]); segment B: the new tokens at L_prev .. L_prev + new - 1.
    still_pos_segment seg[2] = {
        {0.0, tprev > 1 ? (double)(Lp - 1) / (double)(tprev - 1) : 0.0, tprev},
        {(double)Lp, 1.0, nnew}};
    Positions pos;
    TRY(make_positions(seg, nnew > 0 ? 2 : 1, N, pos));
    KVSource src;
    src.K = static_cast<const bf16*>(Kprev) + h_cu_prev[b] * row;
    src.V = static_cast<const bf16*>(Vprev) + h_cu_prev[b] * row;
    src.sN = row;
    src.sH = d;
    src.K2 = nnew > 0 ? static_cast<const bf16*>(Knew) + h_cu_new[b] * row : nullptr;
    src.V2 = nnew > 0 ? static_cast<const bf16*>(Vnew) + h_cu_new[b] * row : nullptr;
    src.sN2 = row;
    src.sH2 = d;
    src.n_split = tprev;
    OutSpec o{static_cast<bf16*>(Ck) + h_cu_out[b] * row, static_cast<bf16*>(Cv) + h_cu_out[b] * row,
              row, d};
    TRY(compact_one(ctx, *L, src, pos, N, t, o, static_cast<cudaStream_t>(stream)));
    if (h_len_out) h_len_out[b] = Lp + nnew;
  }
  return STILL_OK;
}

still_status still_recompact_stack_ragged(still_ctx* ctx, int32_t n_layers, int32_t B,
                                          const void* const* Kprev, const void* const* Vprev,
                                          const int64_t* h_cu_prev, const int64_t* h_prev_len,
                                          const void* const* Knew, const void* const* Vnew,
                                          const int64_t* h_cu_new, int64_t ratio,
                                          void* const* Ck, void* const* Cv, int64_t* h_cu_out,
                                          int64_t* h_len_out, void* stream) {
  if (ctx == nullptr || n_layers < 1 || Kprev == nullptr || Vprev == nullptr ||
      Ck == nullptr || Cv == nullptr)
    return STILL_ERR_INVALID_ARG;
  for (int l = 0; l < n_layers; ++l)
    TRY(still_recompact_layer_ragged(ctx, l, B, Kprev[l], Vprev[l], h_cu_prev, h_prev_len,
                                     Knew ? Knew[l] : nullptr, Vnew ? Vnew[l] : nullptr,
                                     h_cu_new, ratio, Ck[l], Cv[l], h_cu_out, h_len_out,
                                     stream));
  return STILL_OK;
}

still_status still_workspace_size(const still_ctx* ctx, int64_t max_tokens, int32_t max_t,
                                  size_t* bytes) {
  if (ctx == nullptr || bytes == nullptr || ctx->layers.empty() || !ctx->layers[0].loaded)
    return ctx == nullptr || bytes == nullptr ? STILL_ERR_INVALID_ARG : STILL_ERR_NOT_LOADED;
  if (max_tokens < 1 || max_t < 1 || max_t > max_tokens) return STILL_ERR_SHAPE;
  Plan P;
  if (!make_plan(ctx->layers[0].cfg, queries_per_call(ctx->layers[0]), fold_kp(ctx->layers[0]),
                 max_tokens, max_t, 0.0,
                 (double)(max_tokens - 1), ctx->ws_limit, P))
    return STILL_ERR_OOM;
  *bytes = P.total;
  return STILL_OK;
}

still_status still_reserve_workspace(still_ctx* ctx, int64_t max_tokens, int32_t max_t) {
  size_t bytes = 0;
  TRY(still_workspace_size(ctx, max_tokens, max_t, &bytes));
  CK(cudaSetDevice(ctx->device));
  return ensure_ws(ctx, bytes);
}

still_status still_get_device_status(still_ctx* ctx, void* stream, int32_t* h_detail) {
  if (ctx == nullptr) return STILL_ERR_INVALID_ARG;
  CK(cudaSetDevice(ctx->device));
  cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
  int rec[4] = {0, 0, 0, 0};
  if (cudaMemcpy(rec, ctx->err, sizeof(rec), cudaMemcpyDeviceToHost) != cudaSuccess)
    return STILL_ERR_CUDA;
  if (h_detail)
    for (int i = 0; i < 4; ++i) h_detail[i] = rec[i];
  if (rec[0] != 0) cudaMemset(ctx->err, 0, sizeof(rec));
  if (e != cudaSuccess) return STILL_ERR_CUDA;
  if (rec[0] == DEV_WAIT_TIMEOUT) return STILL_ERR_TIMEOUT;
  if (rec[0] != 0) return STILL_ERR_CUDA;
  return STILL_OK;
}

still_status still_profile_enable(still_ctx* ctx, int32_t enable) {
  if (ctx == nullptr) return STILL_ERR_INVALID_ARG;
  CK(cudaSetDevice(ctx->device));
  ctx->prof.reset();
  ctx->prof.on = enable != 0;
  ctx->prof.mask = ~uint64_t(0);
  return STILL_OK;
}

still_status still_profile_enable_classes(still_ctx* ctx, uint64_t mask) {
  if (ctx == nullptr) return STILL_ERR_INVALID_ARG;
  CK(cudaSetDevice(ctx->device));
  ctx->prof.reset();
  ctx->prof.on = mask != 0;
  ctx->prof.mask = mask;
  return STILL_OK;
}

still_status still_profile_read(still_ctx* ctx, int32_t cls, int64_t* h_launches, double* h_ms) {
  if (ctx == nullptr || cls < 0 || cls >= STILL_K_COUNT) return STILL_ERR_INVALID_ARG;
  CK(cudaSetDevice(ctx->device));
  if (!ctx->prof.resolve()) return STILL_ERR_CUDA;
  if (h_launches) *h_launches = ctx->prof.launches[cls];
  if (h_ms) *h_ms = ctx->prof.ms[cls];
  return STILL_OK;
}

const char* still_kernel_class_name(int32_t cls) {
  static const char* names[STILL_K_COUNT] = {
      "strip", "rope_tables", "keyproj", "q_rope", "scores", "softmax", "px", "px_split",
      "vo", "rmsnorm", "sa_proj", "sa_v", "sa_scores", "sa_softmax", "sa_pv", "sa_out",
      "ffn1", "ffn2", "heads", "norms", "load", "ca_fused", "beta", "decode", "repair"};
  return cls >= 0 && cls < STILL_K_COUNT ? names[cls] : "unknown";
}

still_status still_selftest_wait_timeout(still_ctx* ctx, int64_t limit_us, void* stream) {
  if (ctx == nullptr || limit_us < 1 || limit_us > 2000000) return STILL_ERR_INVALID_ARG;
  CK(cudaSetDevice(ctx->device));
  CK(launch_wait_timeout_selftest(ctx->err, (unsigned long long)limit_us * 1000ull,
                                  static_cast<cudaStream_t>(stream)));
  return STILL_OK;
}

int64_t still_budget(int64_t n_tokens, int64_t ratio) {
  if (n_tokens < 0 || ratio < 1) return -1;
  return (2 * n_tokens + ratio) / (2 * ratio);
}

int64_t still_kv_bytes(int64_t n_layers, int64_t n_kv_heads, int64_t head_dim,
                       int64_t elem_bytes, int64_t n_slots) {
  return 2 * n_layers * n_kv_heads * head_dim * elem_bytes * n_slots;
}

int64_t still_param_count(const still_layer_config* cfg, int32_t t) {
  if (cfg == nullptr) return -1;
  const int64_t H = cfg->n_kv_heads, d = cfg->head_dim, D = cfg->d_latent;
  const int64_t nc = cfg->n_cross_heads, ns = cfg->n_self_heads, F = cfg->ffn_dim;
  const int64_t B = cfg->n_blocks, Bc = cfg->cross_every_block ? B : 1;
  return H * t * D + Bc * (2 * nc * D * D + 4 * d * nc * D) + B * (4 * ns * D * D) +
         B * (2 * F * D) + (2 * D * d + D);
}

}  // extern "C"
