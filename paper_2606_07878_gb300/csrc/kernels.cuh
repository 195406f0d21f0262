// Memory-bound kernels of the compactor path (launchers implemented in kernels.cu).
#pragma once
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include "epilogues.cuh"

namespace still {

// The cached tokens of one call: tokens [0, n_split) come from (K, V), tokens [n_split, N)
// from (K2, V2) (the iterative path reads [previous compact cache | new tokens] this way,
// without a concatenation copy). Element strides per token and per KV-head; d contiguous.
struct KVSource {
  const __nv_bfloat16 *K = nullptr, *V = nullptr;
  int64_t sN = 0, sH = 0;
  const __nv_bfloat16 *K2 = nullptr, *V2 = nullptr;
  int64_t sN2 = 0, sH2 = 0;
  int64_t n_split = 0;
};

// RoPE-fix and input concatenation (Sec. 2.2, App. A "Input concatenation"):
//   X[h, n]  = [unRoPE(K[n, h]) | V[n, h]]  as bf16 hi (2d) + bf16 lo of the key half (d)
//   XT[h]    = X[h]^T as fp16 hi / lo, token-contiguous, tokens padded with zeros to Np.
// X:  [H*N][3d] bf16.  XT: [H*2d][2*Np] fp16 (hi at [0, Np), lo at [Np, 2Np); lo rows of
// the value half are not written). omega: [d/2] fp64 base-model frequencies theta^(-2m/d).
// Also gd[n] = (g, p_n - (pmin + g * kPosGrain)) with g = floor((p_n - pmin) / kPosGrain)
// clamped to [0, G): the compactor-RoPE coarse index and residual of token n (n < N).
// x16: X in fp16 (hi | key lo as fp16 hi / lo, values as fp16) instead of bf16.
// Kp > 0: X rows of 2 Kp elements, [x~ hi | x~ lo] with x~ = [unRoPE(K) | V | 1 | 0 ...]
// (the folded key path; Kp a multiple of 64, >= 2d + 1).
cudaError_t launch_strip(const KVSource& src, int64_t N, int H, int d, const PosSegs& segs,
                         const double* omega, int rope_fix, __nv_bfloat16* X, __half* XT,
                         int64_t Np, float2* gd, double pmin, int G, int x16, int Kp,
                         cudaStream_t s);

// Folded key projection (no compactor RoPE): Wt [n][Kp][D] bf16, rows of W~_i = [W_K,i; b_K,i]
// padded with zero rows to Kp, columns in pair-chunk order (from WkT [nD][2d] and bk [nD]).
cudaError_t launch_fold_weights(const __nv_bfloat16* WkT, const float* bk, int n, int D, int d2,
                                int Kp, __nv_bfloat16* Wt, cudaStream_t s);

// Rows of fp32 x [rows][C] -> bf16 [rows][2C]: hi | lo.
cudaError_t launch_f32_hilo(const float* x, int64_t rows, int C, __nv_bfloat16* out,
                            cudaStream_t s);

// Per-slot logit bias from the final latent state Z ([H * t][2D] bf16 hi | lo, rows h * t + j):
// beta[j][h] = sat(Z_hi + Z_lo) . w) + offset, sat(x) = beta_max tanh(x / beta_max) when
// beta_max > 0 (App. A, output projections; optional beta shaping).
cudaError_t launch_beta(const __nv_bfloat16* Z, int t, int H, int D, const float* w,
                        float beta_max, float offset, float* beta, cudaStream_t s);

// Decode-time attention over a compact prefix with logit bias followed by uncompacted entries
// (App. B, "Bias semantics in attention").
struct DecodeArgs {
  const __nv_bfloat16* q = nullptr;   // [nq][Hq][d]
  const __nv_bfloat16* Ck = nullptr;  // slot j of KV-head h at j * cst + h * d
  const __nv_bfloat16* Cv = nullptr;
  const float* beta = nullptr;        // [t][H] or null (no bias)
  const __nv_bfloat16* Kf = nullptr;  // entry j of KV-head h at j * fst + h * d
  const __nv_bfloat16* Vf = nullptr;
  __nv_bfloat16* out = nullptr;       // [nq][Hq][d]
  int64_t t = 0, S = 0, cst = 0, fst = 0;
  int32_t nq = 0, Hq = 0, H = 0, d = 0;
  float scale = 0.f;
};
// Several layers of one shape (t, S, nq, Hq, H, d equal) in one launch of the chunk kernel and
// one of the merge: layer z's arguments are layer[z], z < n.
constexpr int kDecodeMaxLayers = 64;
struct DecodeStack {
  DecodeArgs layer[kDecodeMaxLayers];
  int32_t n = 0;
};
size_t decode_workspace_bytes(int64_t rows, int64_t entries, int d, int layers = 1);
cudaError_t launch_decode_biased(const DecodeStack& st, void* ws, int num_sms, cudaStream_t s);

// Converts n bf16 values to fp16 in place (exact within the fp16 range; values below it
// become fp16 subnormals, absolute error <= 2^-25).
cudaError_t launch_bf16_to_f16(void* p, int64_t n, cudaStream_t s);

// rot[j][m] = (cos, sin)((pstart + j * pstep) * omega[m]) for j < t, m < hd (angle reduced
// modulo 2 pi in fp64); (1, 0) when use_rope is 0. The output heads' re-rotation table.
cudaError_t launch_heads_rot(float2* rot, int t, int hd, double pstart, double pstep,
                             const double* omega, int use_rope, cudaStream_t s);

// Compactor-RoPE tables: coarse[g][m] = (cos, sin)((pmin + g * kPosGrain) * w_m) for g < G,
// then fine[m][i] = (cos, sin)(i * w_m) for i < kPosGrain at coarse + G * D/2; omega[m] = w_m
// (fp32), w_m = omega_c[m] = theta_c^(-2m/D) (fp64 table), angles reduced in fp64.
cudaError_t launch_rope_tables(float2* coarse, float* omega, int G, int D, double pmin,
                               const double* omega_c, cudaStream_t s);

// Per-call cross-attention queries: q = RoPE_c(q^, p_j) for latents j < t, batches
// b in [b0, b0 + nb) (b = h * n + i), as hi/lo bf16 [nb * t][2D]. q^ is [H*n][t_max][D] fp32
// in pair-chunk column order; p_j = qstart + j * qstep.
// fp16: hi/lo in fp16 of (q * qscale) instead of bf16 of q (qscale a power of two).
cudaError_t launch_q_rope(const float* qhat, int t_max, int b0, int nb, int t, int D,
                          double qstart, double qstep, const double* omega_c, int use_rope,
                          __nv_bfloat16* qhl, int fp16, float qscale, cudaStream_t s);

// One-block kernel whose bounded wait on an mbarrier can only expire (failure-detection test).
cudaError_t launch_wait_timeout_selftest(int* err, unsigned long long limit_ns, cudaStream_t s);

// out[m] = base^(-2m / width) in fp64, m < half.
cudaError_t launch_omega(double* out, int half, int width, double base, cudaStream_t s);

// Row softmax: S fp32 [rows][ldS] (first ncols valid) -> P [rows][ldP], zero beyond ncols.
// out_fp16: 1 = P is fp16; 0 = bf16; 2 = bf16 hi | lo: rows of pitch 2 ldP, hi at [0, ldP),
// lo = bf16(p - hi) at [ldP, 2 ldP) (ldP and ncols up to 16384); 3 = the same in fp16.
cudaError_t launch_softmax(const float* S, int64_t rows, int64_t ncols, int64_t ldS, void* P,
                           int64_t ldP, int out_fp16, cudaStream_t s);

// Key-split merge of the fused cross-attention: O [nsplit][nb][t][2d] unnormalised partials (batch
// b = b0 + local) with stats [nsplit][nb][t] = (max in log2 units, sum) -> normalised hi/lo bf16
// rows of PXcat [H*t][2 * n * 2d]: row h*t + j, columns i*2d + f (hi) and n*2d + i*2d + f (lo)
// (f16: fp16 hi | lo instead). Splits are combined in a fixed order.
cudaError_t launch_ca_merge(const float* O, const float2* stats, int nsplit, int b0, int nb,
                            int n, int t, int d2, int f16, __nv_bfloat16* PX, cudaStream_t s);

// out[i] = alpha / max(sqrt(sum_k part(i, k)), eps), summed in slot order: the L2 / QK-norm
// factor of vector i from the epilogues' sum-of-squares partials. Vectors come in blocks of
// `block` consecutive indices stored part-major: part(i, k) is at
// (i / block) * nparts * block + k * block + i % block (block = 1: [vector][part]).
cudaError_t launch_inv_norms(const float* parts, int64_t nvec, int nparts, int64_t block, float eps,
                             float alpha, float* out, cudaStream_t s);

// Non-parametric RMSNorm over rows of width D: out = x / sqrt(mean(x^2) + eps) as bf16 hi
// (and lo at +D when hilo = 1; fp16 hi and lo when hilo = 2), row pitch ldo. Input fp32 or
// bf16 (in_bf16), row pitch ldi.
cudaError_t launch_rmsnorm(const void* in, int in_bf16, int64_t rows, int D, int64_t ldi,
                           float eps, __nv_bfloat16* out, int64_t ldo, int hilo, cudaStream_t s);

// x[row] *= inv[row] for rows of width D (fp32, in place).
cudaError_t launch_scale_rows(float* x, const float* inv, int64_t rows, int D, cudaStream_t s);

// out[c][r] = in[r][src(c)] (bf16), in is [R][C] row-major; src(c) maps pair-chunk order
// back to natural order inside blocks of D columns when perm_D > 0.
cudaError_t launch_transpose(const __nv_bfloat16* in, int64_t R, int64_t C, __nv_bfloat16* out,
                             int perm_D, cudaStream_t s);

// out[c] = float(in[src(c)]) (bf16 -> fp32 with the same optional permutation); in2 (optional)
// is appended after in ([in | in2]), each of length C.
cudaError_t launch_bias(const __nv_bfloat16* in, const __nv_bfloat16* in2, int64_t C,
                        float* out, int perm_D, cudaStream_t s);

// Natural column index of pair-chunk column c inside a block of D columns.
__host__ __device__ inline int pair_chunk_src(int c, int D) {
  const int blk = c / D, f = c % D;
  const int chunk = f / 256, u = f % 256;
  const int m = chunk * 128 + (u & 127);
  return blk * D + (u < 128 ? m : D / 2 + m);
}

}  // namespace still
