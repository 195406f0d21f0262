/* still.h — C ABI of the Still per-layer KV-cache compactor (GB300 / sm_103a).
 *
 * The library computes the paper's per-layer compactor (Sec. 2.1, App. A)
 *
 *     g_phi^(l) : (K^(l,h), V^(l,h))_{h=1..H}  ->  (C_k^(l,h), C_v^(l,h))_{h=1..H},
 *     C_k, C_v in R^{t x d},
 *
 * on one GPU: keys are un-rotated by the base model's RoPE (RoPE-fix, Sec. 2.2), t latent
 * queries per KV-head cross-attend X = [K; V] with QK-norm, the compactor's own RoPE and logits
 * scaled by d_l (App. A, "Cross-attention"), are refined by latent self-attention and a GELU
 * FFN (one or two such blocks), and are projected by W_key / W_val; C_k is re-rotated at evenly
 * spaced output positions over the compacted range (App. B, single-pass recipe, step 5). The
 * reported configuration sets beta = 0 (Sec. 2.1); the optional per-slot bias and its
 * decode-time consumer are separate calls (still_set_beta_head, still_compact_layer_beta,
 * still_attend_biased).
 *
 * Conventions
 *  - Pointers are DEVICE pointers unless their name starts with h_ (host). All calls are
 *    stream-ordered on the given `stream` (a cudaStream_t; NULL = legacy default stream) and
 *    asynchronous unless stated. Host output arguments (h_*) are written before return.
 *  - Tensors are row-major, 16-bit values are bf16 (round-to-nearest-even when produced).
 *  - Calls never throw and never abort; every failure is a still_status. A device-side
 *    failure (a bounded wait that expired) is recorded and reported by
 *    still_get_device_status.
 *  - A context is bound to one device and is not thread-safe; use one per host thread.
 */
#ifndef STILL_H_
#define STILL_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  STILL_OK = 0,
  STILL_ERR_INVALID_ARG = 1, /* null pointer, bad enum or flag value */
  STILL_ERR_UNSUPPORTED = 2, /* a configuration this build does not implement */
  STILL_ERR_SHAPE = 3,       /* inconsistent sizes (t > N, t > t_max, N = 0, ...) */
  STILL_ERR_ALIGNMENT = 4,   /* a pointer or stride breaks the required alignment */
  STILL_ERR_NOT_LOADED = 5,  /* layer weights were never loaded */
  STILL_ERR_OOM = 6,         /* device allocation failed or workspace limit exceeded */
  STILL_ERR_CUDA = 7,        /* a CUDA runtime call failed (sticky errors included) */
  STILL_ERR_TIMEOUT = 8      /* a device-side bounded wait expired (see device status) */
} still_status;

typedef struct still_ctx still_ctx; /* opaque: weight copies, precompute, workspace */

/* One layer's compactor hyperparameters (App. A, "Canonical configuration summary").
 * Implemented: n_blocks 1 or 2, cross_every_block 0 or 1, n_cross_heads = n_self_heads,
 * d_latent % 256 == 0, head_dim in {64, 128, 256} (two blocks: 64 or 128), ffn_dim % 64 == 0
 * (or 0 = no FFN), compactor_rope 0 or 1, rope_fix = 1. Other values return
 * STILL_ERR_UNSUPPORTED. */
typedef struct {
  int32_t n_kv_heads;        /* H: KV-heads of the base model */
  int32_t head_dim;          /* d: base model head dim */
  int32_t d_latent;          /* D = d_l: compactor width; every attention head is D wide */
  int32_t n_cross_heads;     /* n_c */
  int32_t n_self_heads;      /* n_s */
  int32_t ffn_dim;           /* r * d_l, 0 = no FFN sublayer */
  int32_t n_blocks;          /* B */
  int32_t cross_every_block; /* 1 = canonical (CA in every block), 0 = resampler */
  int32_t t_max;             /* rows of each latent bank; a call uses rows [0, t) */
  int32_t final_norm;        /* RMSNorm before the output heads (0 = off, the default) */
  int32_t compactor_rope;    /* apply the compactor's RoPE in cross-attention (0: no RoPE; see
                                still_set_key_fold) */
  int32_t rope_fix;          /* un-rotate cached keys / re-rotate C_k */
  double rope_theta;         /* base model RoPE base */
  double rope_theta_compactor; /* compactor RoPE base (canonical 10) */
  double logit_scale;        /* 0 => d_latent (canonical) */
  float rms_eps;             /* RMSNorm epsilon (1e-6) */
  float l2_eps;              /* QK-norm epsilon (1e-12) */
} still_layer_config;

/* One layer's weights, device bf16, x @ W convention (row = input feature).
 * n = n_cross_heads = n_self_heads; head i of a multi-head projection is the column block
 * [i*D, (i+1)*D) of its [in, n*D] matrix, and row block i of an [n*D, D] output projection.
 *   Z    [H, t_max, D]   latent banks (App. A, "Latent queries")
 *   Wq   [D, n*D]   bq [n*D]    cross-attention query projection and bias
 *   Wk   [2d, n*D]  bk [n*D]    cross-attention key projection and bias (X = [K; V] rows)
 *   Wv   [2d, n*D]              cross-attention value projection (no bias)
 *   Wo   [n*D, D]               cross-attention output projection
 *   Sq   [D, n*D]   sbq [n*D]   self-attention query projection and bias
 *   Sk   [D, n*D]   sbk [n*D]   self-attention key projection and bias
 *   Sv   [D, n*D]               self-attention value projection
 *   So   [n*D, D]               self-attention output projection
 *   W1   [D, F]     W2 [F, D]   FFN (no biases); may be NULL when ffn_dim = 0
 *   Wkey [D, d]     Wval [D, d] output heads
 * The library copies (and re-lays out) everything it needs; the caller may free the inputs
 * after the call's stream work completes. */
typedef struct {
  const void *Z, *Wq, *bq, *Wk, *bk, *Wv, *Wo;
  const void *Sq, *sbq, *Sk, *sbk, *Sv, *So;
  const void *W1, *W2, *Wkey, *Wval;
} still_layer_weights;

/* Weights of one compactor block (App. A, "Compactor blocks"), layouts as in
 * still_layer_weights. The cross-attention fields (Wq, bq, Wk, bk, Wv, Wo) are not read for
 * blocks without cross-attention (blocks after the first when cross_every_block = 0); W1, W2
 * are not read when ffn_dim = 0. */
typedef struct {
  const void *Wq, *bq, *Wk, *bk, *Wv, *Wo;
  const void *Sq, *sbq, *Sk, *sbk, *Sv, *So;
  const void *W1, *W2;
} still_block_weights;

/* Cache positions: token i of the segment sits at start + i * step (exact fp64). Segments
 * are concatenated in order and must cover the N tokens exactly. At most 8 per call. */
typedef struct {
  double start;
  double step;
  int64_t count;
} still_pos_segment;

/* Creates a context on `device` (makes it current). */
still_status still_create(int device, still_ctx** out);
/* Frees everything the context owns. Synchronizes the device first. */
still_status still_destroy(still_ctx* ctx);
/* Static string for a status code. */
const char* still_status_string(still_status s);

/* Copies layer `layer`'s weights into the context and runs the input-independent precompute
 * (App. A: the block-1 latent query q^ = L2norm(RMSNorm(Z) W_Q + b_Q) per KV-head and
 * cross head; the value/output product W_V,i W_O,i). Replaces an earlier load of the layer. */
still_status still_load_layer_weights(still_ctx* ctx, int32_t layer,
                                      const still_layer_config* cfg,
                                      const still_layer_weights* w, void* stream);

/* still_load_layer_weights for a compactor of cfg->n_blocks (1 or 2) blocks (App. A; the
 * paper's canonical compactor has two, both with cross-attention). A block whose output feeds
 * another runs in split precision (fp16 hi / lo operand chains), since the next block's
 * cross-attention magnifies its rounding; n_blocks > 2 gives STILL_ERR_UNSUPPORTED (three
 * blocks measured past the parity bar). Z [H, t_max, D] latent banks;
 * blocks[b] the weights of block b; Wkey, Wval [D, d] output heads. Block 0's latent queries
 * depend only on Z and are precomputed here (as in still_load_layer_weights). A later
 * cross-attending block's queries L2norm(RMSNorm(Z_b) W_Q + b_Q) depend on the latent state
 * Z_b entering it and are formed inside each compaction call. still_load_layer_weights
 * requires n_blocks = 1. */
still_status still_load_layer_weights_blocks(still_ctx* ctx, int32_t layer,
                                             const still_layer_config* cfg, const void* Z,
                                             const still_block_weights* blocks,
                                             const void* Wkey, const void* Wval, void* stream);

/* Compacts one layer (Sec. 2.1; App. B single-pass recipe steps 3-5).
 *   K, V       [N, H, d] bf16 device, element strides strides_kv = {s_token, s_head, s_dim}
 *              (s_dim must be 1; rows 16-byte aligned is not required)
 *   h_segments key positions (NULL and n_segments = 0 => 0..N-1); the latent query
 *              positions and the C_k output positions are t points spaced evenly from the
 *              smallest to the largest key position, both ends included (App. A,
 *              Cross-attention; App. B, step 5).
 *   t          compact length, 1 <= t <= min(N, t_max)
 *   Ck, Cv     [t, H, d] bf16 device outputs, caller-owned, contiguous, 16-byte aligned
 *   h_out_pos_start, h_out_pos_step  (optional) output positions start + j * step
 *   h_pos_offset (optional) logical minus physical length, N - t (App. B, "Logical vs.
 *              physical cache length")
 * Returns STILL_ERR_TIMEOUT/STILL_ERR_CUDA only for failures detected at launch; use
 * still_get_device_status after synchronizing to see device-side failures. */
still_status still_compact_layer(still_ctx* ctx, int32_t layer, const void* K, const void* V,
                                 const int64_t strides_kv[3],
                                 const still_pos_segment* h_segments, int32_t n_segments,
                                 int64_t N, int32_t t, void* Ck, void* Cv,
                                 double* h_out_pos_start, double* h_out_pos_step,
                                 int64_t* h_pos_offset, void* stream);

/* Size of the fixed device scratch behind still_compact_layer_noalloc, in MiB. */
#define STILL_NOALLOC_SCRATCH_MIB 64

/* Same computation, arguments and results as still_compact_layer, for callers that cannot
 * allocate device memory at call time: a serving engine that has handed all free HBM to its
 * own pool (a cudaMalloc would fail or steal from it), a latency-critical loop that must not
 * hit cudaMalloc/cudaFree's implicit device synchronisation, or code running where the CUDA
 * allocator may not be entered. The paper has no counterpart: this is a deployment variant.
 *
 * It allocates nothing: the intermediate buffers live in one file-scope device array of
 * STILL_NOALLOC_SCRATCH_MIB MiB compiled into the library, which every GPU that loads the
 * library holds until the process exits. Weights must already be loaded (that call does
 * allocate). Sizes whose workspace cannot fit in the array even when the KV-heads are
 * processed in small groups are rejected with STILL_ERR_OOM before anything is launched
 * (the tiny 1k-token workload fits; an 8k-token, d_l = 1024 layer does not).
 *
 * The first call on each device looks up the array's device address (cudaGetSymbolAddress,
 * with that device current) and caches it; make that first call before any stream capture.
 * Every call, from every context on the device, shares the one array and leaves its last
 * contents there; the path clears what it needs zeroed on each call. Calls whose execution
 * overlaps on the GPU (different streams, or concurrent host threads) race on the array:
 * serialise them. Kernel event timing (still_profile_enable) is skipped for the kernels of
 * this call, on the calling host thread only and without changing the context's profiling
 * setting; launch counts are still recorded. A context is not thread-safe: host threads that
 * share one must serialise their calls. */
still_status still_compact_layer_noalloc(still_ctx* ctx, int32_t layer, const void* K,
                                         const void* V, const int64_t strides_kv[3],
                                         const still_pos_segment* h_segments,
                                         int32_t n_segments, int64_t N, int32_t t, void* Ck,
                                         void* Cv, double* h_out_pos_start,
                                         double* h_out_pos_step, int64_t* h_pos_offset,
                                         void* stream);

/* ---------------------------------------------------------------------------------------
 * Optional per-slot logit bias (App. A, "Output projections" and "Optional beta shaping";
 * App. B, "Bias semantics in attention"). A third head beta = Z_out w_beta, shared across
 * KV-heads like W_key and W_val, optionally shaped:
 *   saturation     beta <- beta_max * tanh(beta / beta_max)         (beta_max > 0)
 *   mass matching  beta <- beta + log(T / t)                        (mass_match = 1)
 *                  beta <- beta + log_x + log(T / t)                (mass_match = 2, log_x = log x)
 * in that order, with T the number of cached entries the t slots replace (N of the call). */
typedef struct {
  float beta_max;      /* 0: no saturation */
  int32_t mass_match;  /* 0, 1 or 2 as above */
  float log_x;         /* learnable offset log x (the paper initialises x at 1e-3) */
} still_beta_config;

/* Sets (or replaces) the beta head of a loaded layer: w_beta [d_latent] bf16 device pointer
 * (copied), shaping bc (host). STILL_ERR_NOT_LOADED if the layer is not loaded. */
still_status still_set_beta_head(still_ctx* ctx, int32_t layer, const void* w_beta,
                                 const still_beta_config* bc, void* stream);

/* still_compact_layer that also writes the per-slot bias: beta [t][H] fp32 device pointer
 * (4-byte aligned; slot j of KV-head h at j * H + h). STILL_ERR_NOT_LOADED without a beta head. */
still_status still_compact_layer_beta(still_ctx* ctx, int32_t layer, const void* K,
                                      const void* V, const int64_t strides_kv[3],
                                      const still_pos_segment* h_segments, int32_t n_segments,
                                      int64_t N, int32_t t, void* Ck, void* Cv, float* beta,
                                      double* h_out_pos_start, double* h_out_pos_step,
                                      int64_t* h_pos_offset, void* stream);

/* The consumer of a compact cache at decode time (App. B, "Bias semantics in attention"):
 * for each query row, softmax over [scale q C_k^T + beta, scale q K_fix^T] applied to
 * [C_v; V_fix], with grouped query heads (query head i reads KV-head i / (Hq / H)).
 *   q      [nq][Hq][d] bf16
 *   Ck, Cv [t][H][d] bf16 compact prefix (the layout still_compact_layer writes); t >= 0
 *   beta   [t][H] fp32 per-slot bias, or NULL for none (must be finite)
 *   Kfix, Vfix [S][H][d] bf16 uncompacted entries (RoPE already applied, as cached); S >= 0
 *   out    [nq][Hq][d] bf16
 *   scale  logit scale; 0 means 1 / sqrt(d)
 * d in {64, 128, 256}, t + S >= 1, nq * Hq / H <= 64; tensor pointers 16-byte aligned.
 * Keys are processed in chunks of 128 whose partial results are merged in a fixed order; the
 * context's workspace holds the partials (grown on demand), so calls that share a context (this
 * one and the compaction calls) must be ordered on one stream or otherwise serialised. */
still_status still_attend_biased(still_ctx* ctx, const void* q, int32_t nq, int32_t Hq,
                                 const void* Ck, const void* Cv, const float* beta, int64_t t,
                                 const void* Kfix, const void* Vfix, int64_t S, int32_t H,
                                 int32_t d, float scale, void* out, void* stream);

/* still_attend_biased for n_layers layers of one shape (the decode step of a model, App. B,
 * "Bias semantics in attention"), in one launch: every argument as above, the tensors given as
 * host arrays of n_layers device pointers (q[l], Ck[l], Cv[l], Kfix[l], Vfix[l], out[l]);
 * beta is NULL (no bias in any layer) or an array whose entries may be NULL.
 * 1 <= n_layers <= 64 (STILL_ERR_UNSUPPORTED otherwise). A single layer's cache is too small
 * for one launch to keep HBM busy; layer l's result equals still_attend_biased on layer l
 * bit for bit. */
still_status still_attend_biased_stack(still_ctx* ctx, int32_t n_layers, const void* const* q,
                                       int32_t nq, int32_t Hq, const void* const* Ck,
                                       const void* const* Cv, const float* const* beta, int64_t t,
                                       const void* const* Kfix, const void* const* Vfix,
                                       int64_t S, int32_t H, int32_t d, float scale,
                                       void* const* out, void* stream);

/* Compacts layers 0..n_layers-1 (all loaded) over the same positions: the per-layer
 * compactors share nothing at forward time (App. M, "No inter-layer compactor channel"), so
 * this is one stream-ordered launch sequence over the layer stack. K[l], V[l], Ck[l], Cv[l] are device
 * pointers (arrays of n_layers entries, host memory). */
still_status still_compact_stack(still_ctx* ctx, int32_t n_layers, const void* const* K,
                                 const void* const* V, const int64_t strides_kv[3],
                                 const still_pos_segment* h_segments, int32_t n_segments,
                                 int64_t N, int32_t t, void* const* Ck, void* const* Cv,
                                 double* h_out_pos_start, double* h_out_pos_step,
                                 int64_t* h_pos_offset, void* stream);

/* Ragged batch of B sequences packed along the token axis.
 *   Kpacked, Vpacked [sum N_b, H, d] bf16 (contiguous), h_cu_seqlens[B+1] token offsets
 *   h_segments / h_seg_per_seq: sequence b uses h_seg_per_seq[b] consecutive segments
 *     (NULL => positions 0..N_b-1 for every sequence)
 *   h_t[B] compact lengths; h_cu_t[B+1] offsets of each sequence's rows in Ck/Cv
 *   Ck, Cv [sum t_b, H, d] bf16; h_pos_offset[B] (optional) N_b - t_b.
 * Sequence b uses rows [0, t_b) of every latent bank. */
still_status still_compact_layer_ragged(still_ctx* ctx, int32_t layer, const void* Kpacked,
                                        const void* Vpacked, const int64_t* h_cu_seqlens,
                                        int32_t B, const still_pos_segment* h_segments,
                                        const int32_t* h_seg_per_seq, const int32_t* h_t,
                                        const int64_t* h_cu_t, void* Ck, void* Cv,
                                        int64_t* h_pos_offset, void* stream);

/* Ragged batch over layers 0..n_layers-1: per-layer packed K/V and Ck/Cv pointer arrays
 * (host arrays of device pointers); the other arguments as still_compact_layer_ragged. */
still_status still_compact_stack_ragged(still_ctx* ctx, int32_t n_layers,
                                        const void* const* Kpacked, const void* const* Vpacked,
                                        const int64_t* h_cu_seqlens, int32_t B,
                                        const still_pos_segment* h_segments,
                                        const int32_t* h_seg_per_seq, const int32_t* h_t,
                                        const int64_t* h_cu_t, void* const* Ck,
                                        void* const* Cv, int64_t* h_pos_offset, void* stream);

/* Iterative re-compaction (Sec. 2.3, iterative chunked compaction; here the fixed-ratio
 * form that appends new tokens to each sequence's compact cache): for each of B sequences,
 * the keys and values [previous compact cache | new tokens] are compacted again to
 * t_b = round((L_prev,b + new_b) / ratio) slots (at least 1). Previous compact slots sit at
 * their output positions, t_prev points evenly spaced over [0, L_prev - 1]; the new tokens
 * at L_prev .. L_prev + new - 1; the new slots are evenly spaced over [0, L_prev + new - 1].
 * The two parts are read in place (no concatenation copy).
 *   Kprev, Vprev [sum t_prev, H, d] bf16: sequence b at rows [h_cu_prev[b], h_cu_prev[b+1])
 *   h_prev_len[B] logical lengths already absorbed (>= t_prev)
 *   Knew, Vnew   [sum new, H, d] bf16, h_cu_new[B+1] (new_b may be 0)
 *   Ck, Cv       output [sum t_b, H, d] bf16, 16-byte aligned, disjoint from the inputs;
 *                the caller sizes them with still_budget
 *   h_cu_out[B+1] (out) row offsets of each sequence's new compact cache
 *   h_len_out[B]  (out, optional) new logical lengths. */
still_status still_recompact_layer_ragged(still_ctx* ctx, int32_t layer, int32_t B,
                                          const void* Kprev, const void* Vprev,
                                          const int64_t* h_cu_prev, const int64_t* h_prev_len,
                                          const void* Knew, const void* Vnew,
                                          const int64_t* h_cu_new, int64_t ratio, void* Ck,
                                          void* Cv, int64_t* h_cu_out, int64_t* h_len_out,
                                          void* stream);

/* still_recompact_layer_ragged over layers 0..n_layers-1 (host arrays of per-layer device
 * pointers; the offsets and lengths are shared by all layers). */
still_status still_recompact_stack_ragged(still_ctx* ctx, int32_t n_layers, int32_t B,
                                          const void* const* Kprev, const void* const* Vprev,
                                          const int64_t* h_cu_prev, const int64_t* h_prev_len,
                                          const void* const* Knew, const void* const* Vnew,
                                          const int64_t* h_cu_new, int64_t ratio,
                                          void* const* Ck, void* const* Cv, int64_t* h_cu_out,
                                          int64_t* h_len_out, void* stream);

/* Compacts only the layers l < n_layers with h_compact_layer[l] != 0, each as
 * still_compact_layer over the same positions (Sec. 2.1 and App. A "Per-layer stack and
 * mixed-attention models": in a model that mixes sliding-window and global attention, such
 * as Gemma-3, only the global-attention layers are compacted; the others keep their own
 * sliding-window cache). Skipped layers need not be loaded and their K, V, Ck, Cv entries may
 * be NULL; their buffers are not touched. h_compact_layer: host array of n_layers bytes.
 * Other arguments as still_compact_stack. */
still_status still_compact_stack_masked(still_ctx* ctx, int32_t n_layers,
                                        const uint8_t* h_compact_layer, const void* const* K,
                                        const void* const* V, const int64_t strides_kv[3],
                                        const still_pos_segment* h_segments, int32_t n_segments,
                                        int64_t N, int32_t t, void* const* Ck, void* const* Cv,
                                        double* h_out_pos_start, double* h_out_pos_step,
                                        int64_t* h_pos_offset, void* stream);

/* ---------------------------------------------------------------------------------------
 * Iterative chunked compaction with lookahead (Sec. 2.3, "Iterative chunked compaction";
 * App. B). The context arrives in chunks of c*t tokens (c the local compression ratio, t the
 * slots per chunk). Pass 0 prefills chunks 0 and 1 and compacts chunk 0; pass k > 0
 * prefills chunk k + 1 with the k compacted chunks followed by raw chunk k as its past
 * ((k + c) * t entries), then compacts chunk k to t slots. After pass k the cache holds
 * chunks 0..k compacted plus raw chunk k + 1 (the one-chunk lookahead buffer): once T tokens
 * have been compacted (T / (c t) passes) it holds T / c + c t entries. The base-model
 * prefill itself is the caller's; the library computes the schedule and the compaction. */
typedef struct {
  int64_t chunk_start;       /* first token position of the chunk this pass compacts: k*c*t  */
  int64_t chunk_len;         /* c*t                                                          */
  int64_t prefill_start;     /* first token the base model prefills in this pass             */
  int64_t prefill_len;       /* 2*c*t at pass 0, c*t after                                   */
  int64_t prefill_past;      /* cache entries the prefill attends to: 0, then (k + c)*t       */
  int64_t compact_row;       /* k*t: first row of this chunk's t slots in the compact prefix */
  int64_t retained_after;    /* (k + 1)*t + c*t cache entries after the pass                 */
  int64_t logical_after;     /* (k + 2)*c*t tokens prefilled after the pass                  */
  int64_t pos_offset_after;  /* logical_after - retained_after (App. B position offset)      */
} still_lookahead_pass;

/* Host only. Pass k >= 0 of the schedule for ratio c >= 1 and t >= 1 slots per chunk.
 * STILL_ERR_INVALID_ARG for out-of-range arguments or when a field would exceed 2^53
 * (positions must stay exact in fp64). */
still_status still_lookahead_pass_info(int64_t k, int64_t c, int32_t t,
                                       still_lookahead_pass* out);

/* Host only. Passes (T / (c t)) and retained cache entries (T / c + c t) once T tokens have
 * been compacted; T must be a positive multiple of c*t (else STILL_ERR_SHAPE). */
still_status still_lookahead_totals(int64_t T, int64_t c, int32_t t, int64_t* h_passes,
                                    int64_t* h_retained);

/* Compaction step of one lookahead pass for B sequences at once, each at its own pass
 * index: sequence b's raw chunk (c*t tokens at positions h_pass[b]*c*t + i, as the base
 * model cached them) is compacted to t slots at output positions evenly spaced over the
 * chunk. One ragged call (still_compact_layer_ragged) with one position segment per
 * sequence.
 *   K, V    [B * c*t, H, d] bf16 packed chunks, sequence b at rows [b*c*t, (b+1)*c*t)
 *   h_pass  [B] pass indices k_b >= 0 (host)
 *   Ck, Cv  [B * t, H, d] bf16 outputs, sequence b at rows [b*t, (b+1)*t); the caller
 *           appends them at row h_pass[b]*t (compact_row) of that sequence's compact prefix
 * Requires 1 <= t <= t_max of the layer. */
still_status still_lookahead_compact_layer(still_ctx* ctx, int32_t layer, int32_t B,
                                           const void* K, const void* V, const int64_t* h_pass,
                                           int64_t c, int32_t t, void* Ck, void* Cv,
                                           void* stream);

/* still_lookahead_compact_layer over the layers l < n_layers with h_compact_layer[l] != 0
 * (NULL: every layer), per-layer pointer arrays in host memory as in
 * still_compact_stack_masked. */
still_status still_lookahead_compact_stack(still_ctx* ctx, int32_t n_layers,
                                           const uint8_t* h_compact_layer, int32_t B,
                                           const void* const* K, const void* const* V,
                                           const int64_t* h_pass, int64_t c, int32_t t,
                                           void* const* Ck, void* const* Cv, void* stream);

/* Device workspace bytes a call with up to max_tokens tokens and compact length max_t needs
 * for layer 0's configuration (the context allocates it on demand and keeps it). */
still_status still_workspace_size(const still_ctx* ctx, int64_t max_tokens, int32_t max_t,
                                  size_t* bytes);

/* Allocates now the workspace a call with up to max_tokens tokens and compact length max_t
 * needs (layer 0's configuration), so that later calls of at most those sizes allocate
 * nothing. still_compact_layer and still_compact_stack enqueue work only on their stream and
 * neither allocate nor synchronize when the workspace suffices (and after one earlier call has
 * set the kernels' shared-memory attributes): such calls can be captured into a CUDA graph
 * and replayed. Kernel timing (still_profile_*) should cover only the classes needed while
 * capturing: timed launches become event nodes of the graph. */
still_status still_reserve_workspace(still_ctx* ctx, int64_t max_tokens, int32_t max_t);

/* Upper bound on the workspace the context may allocate (default 48 GiB). Calls whose
 * workspace would exceed it process the KV-heads in smaller groups, or fail with
 * STILL_ERR_OOM when even one group does not fit. */
still_status still_set_workspace_limit(still_ctx* ctx, size_t bytes);

/* Size limit, per layer, of the precomputed latent queries q^ = L2n(RMSNorm(Z) W_Q + b_Q)
 * (H * n * t_max * D fp32, App. A "Cross-attention"; input-independent, so by default formed
 * once at weight load). Layers loaded while their q^ would exceed `bytes` keep W_Q and b_Q
 * instead and form q^ for the call's t latents inside each compaction call, with the same
 * kernels and the same results. Default 2 GiB; applies to later still_load_layer_weights. */
still_status still_set_qhat_eager_limit(still_ctx* ctx, size_t bytes);

/* Layers without compactor RoPE (compactor_rope = 0) fold the key projection into the
 * queries when they have one block, 2d <= 256, precomputed queries and 2d + 1 (padded to a
 * multiple of 64) below d_latent: with x~ = [x; 1] and W~ = [W_K; b_K], the logits are
 * d_l (x~ . W~ q^) / |x~ W~| and |x~ W~|^2 = x~ (W~ W~^T) x~^T, so the cached tokens are
 * never projected to d_latent (App. A, "Cross-attention": the logits of QK-normed heads).
 * enable = 0 keeps the explicit projection for layers loaded afterwards (default 1). */
still_status still_set_key_fold(still_ctx* ctx, int32_t enable);

/* Synchronizes `stream`, then reports (and clears) the device error record:
 * STILL_ERR_TIMEOUT if a kernel's bounded wait expired, STILL_ERR_CUDA if the stream
 * reported an error. h_detail (optional, 4 ints): code, site, block, count. */
still_status still_get_device_status(still_ctx* ctx, void* stream, int32_t* h_detail);

/* Kernel classes of the launch sequence, for launch counts and timings. */
typedef enum {
  STILL_K_STRIP = 0,    /* RoPE-fix + [K; V] concat (hi/lo)                 */
  STILL_K_TABLES,       /* compactor-RoPE angle table                       */
  STILL_K_KEYPROJ,      /* k = RoPE_c(X W_K + b_K) (2-pass tcgen05 GEMM)    */
  STILL_K_QROPE,        /* q = RoPE_c(q^) at the latent query positions     */
  STILL_K_SCORES,       /* (unused: the scores are fused into STILL_K_CA_FUSED) */
  STILL_K_SOFTMAX,      /* (unused: the softmax is fused)                   */
  STILL_K_PX,           /* (unused: P X is fused)                           */
  STILL_K_PXSPLIT,      /* key-split merge of O, O -> hi/lo                 */
  STILL_K_VO,           /* Z' = Z + O (W_V W_O) (3-pass tcgen05 GEMM)       */
  STILL_K_NORM,         /* RMSNorm                                          */
  STILL_K_SA_PROJ,      /* self-attention q/k projections                   */
  STILL_K_SA_V,         /* self-attention v projection                      */
  STILL_K_SA_SCORES,    /* self-attention scores                            */
  STILL_K_SA_SOFTMAX,   /* self-attention row softmax                       */
  STILL_K_SA_PV,        /* self-attention P v                               */
  STILL_K_SO,           /* self-attention output projection + residual      */
  STILL_K_FFN1,         /* GELU(x W_1)                                      */
  STILL_K_FFN2,         /* (.) W_2 + residual                               */
  STILL_K_HEADS,        /* C_k, C_v output heads + re-rotation              */
  STILL_K_NORMS,        /* QK-norm factors from sum-of-squares partials     */
  STILL_K_LOAD,         /* weight-load precompute GEMMs                     */
  STILL_K_CA_FUSED,     /* fused scores + online softmax + P X              */
  STILL_K_BETA,         /* beta head: Z_out w_beta, shaped                  */
  STILL_K_DECODE,       /* biased decode attention (chunks + merge)         */
  STILL_K_REPAIR,       /* top-k repair of one-pass cross-attention scores  */
  STILL_K_COUNT
} still_kernel_class;

/* Starts (enable = 1) or stops kernel timing and clears the counters. While enabled, every
 * launch of the library's kernels is bracketed by a CUDA event pair on its stream. Launch
 * counts are kept whether or not timing is enabled (reset by this call). */
still_status still_profile_enable(still_ctx* ctx, int32_t enable);
/* As still_profile_enable, with event timing only for the kernel classes whose bit
 * (1 << class) is set in `mask` (0 stops timing). Timing one class costs two events per launch
 * of that class only, so a step can be timed with its dominant kernel measured inside it. */
still_status still_profile_enable_classes(still_ctx* ctx, uint64_t mask);
/* Launches and total event time (ms) of one kernel class since the last enable call.
 * Synchronizes the device when timings are pending. */
still_status still_profile_read(still_ctx* ctx, int32_t cls, int64_t* h_launches, double* h_ms);
/* Static name of a kernel class ("scores", "softmax", ...). */
const char* still_kernel_class_name(int32_t cls);

/* Failure-detection self-test (no counterpart in the paper): launches one kernel that waits,
 * for at most limit_us microseconds (1 .. 2e6), on a barrier nothing will release, exactly as
 * the library's kernels bound every wait. The wait expires, the kernel records a timeout in
 * the device error record and returns; the next still_get_device_status reports
 * STILL_ERR_TIMEOUT (and clears the record) and the context stays usable. */
still_status still_selftest_wait_timeout(still_ctx* ctx, int64_t limit_us, void* stream);

/* Compact budget t = round(N / ratio) with halves rounded up (App. J exact-results table,
 * K column: 8192 / 50 -> 164, 65536 / 50 -> 1311). Host-only. */
int64_t still_budget(int64_t n_tokens, int64_t ratio);

/* Retained KV bytes M_KV(S) = 2 L H d b S (App. B, "Deployment accounting"). Host-only. */
int64_t still_kv_bytes(int64_t n_layers, int64_t n_kv_heads, int64_t head_dim,
                       int64_t elem_bytes, int64_t n_slots);

/* Number of per-layer compactor parameters (App. D) for a configuration: bank H*t*D,
 * per CA block 2 n D^2 + 4 d n D, per SA block 4 n D^2, per FFN block 2 F D, heads
 * 2 D d + D (the D-wide beta head included, as in the paper's count). Host-only. */
int64_t still_param_count(const still_layer_config* cfg, int32_t t);

#ifdef __cplusplus
}
#endif
#endif /* STILL_H_ */
