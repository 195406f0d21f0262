"""fp64 CPU oracle for the Still per-layer compactor forward (test infrastructure only).

This file is TEST INFRASTRUCTURE. Only the tests, the smoke check and the bench's CPU-baseline
leg may import it. The library's compute path never calls it. It shares no code with the
CUDA path. Everything here is plain NumPy in float64, written from the paper's definitions
so that each step can be checked against the text by eye:

  * per-layer compactor g_phi: (K_h, V_h)_h -> (C_k_h, C_v_h)_h ............... Sec. 2.1
  * input X = [unRoPE(K); V] (RoPE-fix), values unrotated ...... Sec. 2.2; App. A "Input"
  * latent banks Z[h] (t x d_l), projections shared across KV-heads ...... App. A "Latent"
  * pre-norm blocks Z' = Z + CA(RMSNorm Z, X), Z'' = Z' + SA(RMSNorm Z'),
    Z''' = Z'' + FFN(RMSNorm Z'') ................................. App. A "Compactor blocks"
  * cross-attention: expanded heads (each d_l wide), q~ = Q W_Q + b_Q, k~ = X W_K + b_K,
    v = X W_V (no bias), L2 QK-norm, compactor RoPE (keys at cache positions, queries evenly
    spaced between the first and last key positions), logits x d_l, Concat(heads) W_O
    ................................................................. App. A "Cross-attention"
  * latent self-attention: same QK-norm and logit scale, no RoPE ....... App. A "Latent self"
  * FFN = GELU(x W_1) W_2 ................................................. App. A "Feed-forward"
  * C_k = Z_out W_key, C_v = Z_out W_val, C_k re-rotated at evenly spaced output positions
    ..................................................... App. A "Output projections"; App. B
  * compact budget t = round(N / c) ........ App. J exact-results table (K column)
  * position offset T - t ................................ App. B, logical vs physical length
  * beta = Z_out w_beta, saturation, mass matching ......... App. A, Output projections / beta
  * attention over [C_k; K_fix] with bias [beta; 0] .......... App. B, Bias semantics
  * iterative chunked schedule with lookahead: passes, chunks, retained cache . Sec. 2.3

Readings taken where the paper is silent (each listed with its basis in the design notes):
half-split RoPE pairs (m, m + w/2) with omega_m = base^(-2m/w); RMSNorm x/sqrt(mean x^2 + 1e-6)
without gain; L2 norm x/max(|x|, 1e-12); exact-erf GELU; no FFN biases; SA carries query/key
biases like CA; query and output positions = linspace(min pos, max pos, t), inclusive, fp64;
KV-heads independent (self-attention runs within each head's bank); beta = 0; the final
RMSNorm before the heads is off unless requested.

Parity pins live in tests/test_oracle_pins.py. The end-to-end values for random weights at
the benchmark shapes have no printed worked example in the paper: beyond the pins below they
are "parity unpinned" (brute force, invariants and the identity-init construction pin the
oracle's pieces and their composition).
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np
from scipy.special import erf


# ----------------------------------------------------------------------------- configuration

@dataclass
class Cfg:
    """Hyperparameters of one layer's compactor (App. A, "Canonical configuration summary")."""
    H: int                  # KV-heads of the base model
    d: int                  # base model head dim
    D: int                  # compactor width d_l
    n_c: int                # cross-attention heads (each D wide)
    n_s: int                # self-attention heads (each D wide)
    F: int = 0              # FFN hidden width r*d_l (0 = no FFN)
    n_blocks: int = 1       # B
    cross_every_block: bool = True   # canonical: CA in every block; resampler: first only
    self_attn: bool = True
    final_norm: bool = False
    compactor_rope: bool = True      # "when cross-attention positions are supplied"
    rope_fix: bool = True            # un-rotate cached keys before the compactor
    theta: float = 1e6               # base model RoPE base
    theta_c: float = 10.0            # compactor RoPE base (canonical 10)
    logit_scale: float | None = None  # None -> d_l (canonical); ablations: 1/sqrt(d_l), 2 d_l
    rms_eps: float = 1e-6
    l2_eps: float = 1e-12

    @property
    def scale(self) -> float:
        return float(self.D) if self.logit_scale is None else float(self.logit_scale)


def cfg_from_workload(wl: dict, **over) -> Cfg:
    c = Cfg(H=wl["H"], d=wl["d"], D=wl["D"], n_c=wl["n"], n_s=wl["n"], F=wl["F"],
            theta=wl["theta"])
    for k, v in over.items():
        setattr(c, k, v)
    return c


# ----------------------------------------------------------------------------- primitives

def budget(N: int, c: int) -> int:
    """Compact length t = round(N / c), halves rounded up, in integers (App. J table, K column)."""
    return (2 * N + c) // (2 * c)


def position_offset(logical_len: int, t: int) -> int:
    """Continuation positions are offset by logical length minus physical length (App. B)."""
    return logical_len - t


# ----------------------------------------------------------------------------- lookahead schedule

def lookahead_pass(k: int, c: int, t: int) -> dict:
    """Pass k of the iterative chunked schedule with lookahead (Sec. 2.3; App. B, iterative
    chunked compaction), chunks of ct tokens, walked through as the text describes them.

    Pass 0 prefills the first two chunks with no past and compacts chunk 0. Pass k > 0
    prefills chunk k + 1 while the past holds the k chunks already compacted (t slots each)
    followed by raw chunk k, then compacts chunk k, the one just before the new chunk.
    After pass k the cache holds chunks 0..k compacted and chunk k + 1 raw (the lookahead).
    """
    ct = c * t
    compacted_before = k                                  # chunks 0..k-1
    if k == 0:
        prefill = (0, 2 * ct)
        past = 0
    else:
        prefill = ((k + 1) * ct, ct)                      # chunk k + 1
        past = compacted_before * t + ct                  # compact prefix, then raw chunk k
    compacted_after = k + 1
    raw_after = ct                                        # chunk k + 1
    logical_after = (k + 2) * ct                          # tokens prefilled so far
    retained_after = compacted_after * t + raw_after
    return {
        "chunk_start": k * ct, "chunk_len": ct,
        "prefill_start": prefill[0], "prefill_len": prefill[1], "prefill_past": past,
        "compact_row": compacted_before * t,
        "retained_after": retained_after, "logical_after": logical_after,
        "pos_offset_after": logical_after - retained_after,
    }


def lookahead_totals(T: int, c: int, t: int) -> tuple[int, int]:
    """(passes, retained cache entries) once T tokens have been compacted: every chunk of ct
    tokens costs one pass, and the last pass leaves one raw lookahead chunk (Sec. 2.3)."""
    ct = c * t
    if T <= 0 or T % ct:
        raise ValueError("T must be a positive multiple of the chunk length c*t")
    passes = T // ct
    return passes, lookahead_pass(passes - 1, c, t)["retained_after"]


def rope_angles(pos: np.ndarray, width: int, base: float) -> np.ndarray:
    """Angles pos_n * base^(-2m/width) for the width/2 frequency pairs, fp64. [N, width/2]"""
    m = np.arange(width // 2, dtype=np.float64)
    omega = base ** (-2.0 * m / width)
    return np.multiply.outer(np.asarray(pos, dtype=np.float64), omega)


def rope(x: np.ndarray, pos: np.ndarray, base: float) -> np.ndarray:
    """Rotary embedding: pair (m, m + w/2) of row n rotated by +angle[n, m]."""
    w = x.shape[-1]
    h = w // 2
    ang = rope_angles(pos, w, base)
    c, s = np.cos(ang), np.sin(ang)
    a, b = x[..., :h], x[..., h:]
    return np.concatenate([a * c - b * s, a * s + b * c], axis=-1)


def unrope(x: np.ndarray, pos: np.ndarray, base: float) -> np.ndarray:
    """Inverse rotary embedding (RoPE-fix, Sec. 2.2): pair (m, m + w/2) rotated by -angle."""
    w = x.shape[-1]
    h = w // 2
    ang = rope_angles(pos, w, base)
    c, s = np.cos(ang), np.sin(ang)
    a, b = x[..., :h], x[..., h:]
    return np.concatenate([a * c + b * s, -a * s + b * c], axis=-1)


def rmsnorm(x: np.ndarray, eps: float) -> np.ndarray:
    """Non-parametric RMSNorm over the last axis."""
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps)


def l2norm(x: np.ndarray, eps: float) -> np.ndarray:
    """QK-norm: x / max(||x||_2, eps) over the last axis."""
    return x / np.maximum(np.linalg.norm(x, axis=-1, keepdims=True), eps)


def softmax_rows(s: np.ndarray) -> np.ndarray:
    """Row softmax, max-subtracted."""
    e = np.exp(s - s.max(axis=-1, keepdims=True))
    return e / e.sum(axis=-1, keepdims=True)


def gelu(x: np.ndarray) -> np.ndarray:
    """Exact GELU, x * Phi(x)."""
    return 0.5 * x * (1.0 + erf(x / np.sqrt(2.0)))


def linspace_positions(pmin: float, pmax: float, t: int) -> np.ndarray:
    """t positions evenly spaced over [pmin, pmax], inclusive; t = 1 gives pmin."""
    if t == 1:
        return np.array([pmin], dtype=np.float64)
    return np.linspace(pmin, pmax, t, dtype=np.float64)


def positions_from_segments(segments) -> np.ndarray:
    """Key positions from (start, step, count) segments."""
    if not segments:
        return np.zeros(0)
    return np.concatenate([s + st * np.arange(c, dtype=np.float64) for s, st, c in segments])


# ----------------------------------------------------------------------------- sublayers

def _blk(W: dict, name: str, b: int):
    return W[name if b == 0 else f"{name}@{b}"]


def cross_attention(Zn: np.ndarray, X: np.ndarray, W: dict, b: int, cfg: Cfg,
                    qpos: np.ndarray, kpos: np.ndarray, row_chunk: int = 4096) -> np.ndarray:
    """CrossAttn(Q, X) = Concat_i softmax(s q_i k_i^T) v_i . W_O   (App. A, Cross-attention).

    Zn: RMSNorm'd latents [t, D]; X: [N, 2d]. Softmax rows are independent, so rows are
    processed `row_chunk` at a time to bound memory.
    """
    D = cfg.D
    Wq, bq = _blk(W, "Wq", b), _blk(W, "bq", b)
    Wk, bk = _blk(W, "Wk", b), _blk(W, "bk", b)
    Wv, Wo = _blk(W, "Wv", b), _blk(W, "Wo", b)
    heads = []
    for i in range(cfg.n_c):
        cols = slice(i * D, (i + 1) * D)
        q = l2norm(Zn @ Wq[:, cols] + bq[cols], cfg.l2_eps)        # [t, D]
        k = l2norm(X @ Wk[:, cols] + bk[cols], cfg.l2_eps)         # [N, D]
        if cfg.compactor_rope:
            q = rope(q, qpos, cfg.theta_c)
            k = rope(k, kpos, cfg.theta_c)
        v = X @ Wv[:, cols]                                        # [N, D], no bias
        head = np.empty((Zn.shape[0], D))
        for r0 in range(0, Zn.shape[0], row_chunk):
            r1 = min(r0 + row_chunk, Zn.shape[0])
            A = softmax_rows(cfg.scale * (q[r0:r1] @ k.T))         # [rows, N]
            head[r0:r1] = A @ v
        heads.append(head)
    return np.concatenate(heads, axis=-1) @ Wo                      # [t, D]


def self_attention(Zn: np.ndarray, W: dict, b: int, cfg: Cfg) -> np.ndarray:
    """SelfAttn(Z) = Concat_i softmax(s q_i k_i^T) v_i . W_O^(sa), QK-norm, no RoPE (App. A)."""
    D = cfg.D
    Sq, sbq = _blk(W, "Sq", b), _blk(W, "sbq", b)
    Sk, sbk = _blk(W, "Sk", b), _blk(W, "sbk", b)
    Sv, So = _blk(W, "Sv", b), _blk(W, "So", b)
    heads = []
    for i in range(cfg.n_s):
        cols = slice(i * D, (i + 1) * D)
        q = l2norm(Zn @ Sq[:, cols] + sbq[cols], cfg.l2_eps)
        k = l2norm(Zn @ Sk[:, cols] + sbk[cols], cfg.l2_eps)
        v = Zn @ Sv[:, cols]
        heads.append(softmax_rows(cfg.scale * (q @ k.T)) @ v)
    return np.concatenate(heads, axis=-1) @ So


def ffn(Zn: np.ndarray, W: dict, b: int) -> np.ndarray:
    """FFN(x) = GELU(x W_1) W_2 (App. A, Feed-forward sublayer)."""
    return gelu(Zn @ _blk(W, "W1", b)) @ _blk(W, "W2", b)


# ----------------------------------------------------------------------------- compactor

def compact_head(Kh: np.ndarray, Vh: np.ndarray, Zh: np.ndarray, W: dict, cfg: Cfg,
                 kpos: np.ndarray, row_chunk: int = 4096, return_state: bool = False):
    """One KV-head: cached (K_h, V_h) [N, d] and its latent bank Z_h [t, D] -> (C_k, C_v) [t, d].

    Returns (C_k, C_v, out_positions), and the final latent state Z_out when return_state.
    """
    t = Zh.shape[0]
    pmin, pmax = float(np.min(kpos)), float(np.max(kpos))
    qpos = linspace_positions(pmin, pmax, t)           # evenly spaced latent query positions
    Kx = unrope(Kh, kpos, cfg.theta) if cfg.rope_fix else Kh
    X = np.concatenate([Kx, Vh], axis=-1)              # [N, 2d]
    Z = Zh.copy()
    for b in range(cfg.n_blocks):
        if b == 0 or cfg.cross_every_block:
            Z = Z + cross_attention(rmsnorm(Z, cfg.rms_eps), X, W, b, cfg, qpos, kpos, row_chunk)
        if cfg.self_attn:
            Z = Z + self_attention(rmsnorm(Z, cfg.rms_eps), W, b, cfg)
        if cfg.F:
            Z = Z + ffn(rmsnorm(Z, cfg.rms_eps), W, b)
    Zout = rmsnorm(Z, cfg.rms_eps) if cfg.final_norm else Z
    opos = qpos                                        # evenly spaced over the compacted range
    Ck = Zout @ W["Wkey"]
    if cfg.rope_fix:
        Ck = rope(Ck, opos, cfg.theta)                 # back into the base model's RoPE frame
    Cv = Zout @ W["Wval"]
    if return_state:
        return Ck, Cv, opos, Zout
    return Ck, Cv, opos


def beta_head(Zout: np.ndarray, w_beta: np.ndarray, beta_max: float = 0.0, mass_match: int = 0,
              log_x: float = 0.0, T: float | None = None) -> np.ndarray:
    """Per-slot logit bias of one KV-head, beta = Z_out w_beta (App. A, Output projections),
    with the optional shaping of App. A ("Optional beta shaping"), applied in that order:
      saturation     beta <- beta_max * tanh(beta / beta_max)          when beta_max > 0
      mass matching  beta <- beta + log(T / t)                        mass_match = 1
                     beta <- beta + log(x) + log(T / t), log_x = log x  mass_match = 2
    T is the number of cached tokens the t slots replace."""
    t = Zout.shape[0]
    beta = Zout @ w_beta
    if beta_max > 0:
        beta = beta_max * np.tanh(beta / beta_max)
    if mass_match:
        beta = beta + np.log(T / t) + (log_x if mass_match == 2 else 0.0)
    return beta


def biased_attention(q: np.ndarray, Ck: np.ndarray, Cv: np.ndarray, beta: np.ndarray,
                     Kfix: np.ndarray, Vfix: np.ndarray, scale: float) -> np.ndarray:
    """Attention of query rows q [m, d] over the compact prefix followed by uncompacted entries,
    with beta added to the compact-prefix logits and 0 to the others (App. B, "Bias semantics
    in attention"): softmax over [scale q C_k^T + beta, scale q K_fix^T] applied to
    [C_v; V_fix]."""
    logits = np.concatenate([scale * (q @ Ck.T) + beta[None, :], scale * (q @ Kfix.T)], axis=1)
    return softmax_rows(logits) @ np.concatenate([Cv, Vfix], axis=0)


def compact_layer(K: np.ndarray, V: np.ndarray, W: dict, cfg: Cfg, t: int,
                  kpos: np.ndarray | None = None, heads=None, row_chunk: int = 4096):
    """g_phi for one layer (Sec. 2.1): K, V [N, H, d] -> C_k, C_v [t, H, d] (fp64).

    Head h uses rows [0, t) of its latent bank W["Z"][h]. `heads` restricts the KV-heads
    computed (the others are left as NaN); KV-heads are independent.
    Returns (C_k, C_v, out_positions, position_offset).
    """
    N = K.shape[0]
    if kpos is None:
        kpos = np.arange(N, dtype=np.float64)
    kpos = np.asarray(kpos, dtype=np.float64)
    Z = np.asarray(W["Z"], dtype=np.float64)
    Ck = np.full((t, cfg.H, cfg.d), np.nan)
    Cv = np.full((t, cfg.H, cfg.d), np.nan)
    opos = None
    for h in (range(cfg.H) if heads is None else heads):
        Ck[:, h], Cv[:, h], opos = compact_head(K[:, h], V[:, h], Z[h, :t], W, cfg, kpos,
                                                row_chunk)
    return Ck, Cv, opos, position_offset(N, t)


def compact_layer_beta(K: np.ndarray, V: np.ndarray, W: dict, cfg: Cfg, t: int, w_beta,
                       beta_max: float = 0.0, mass_match: int = 0, log_x: float = 0.0,
                       kpos: np.ndarray | None = None, heads=None):
    """compact_layer plus the beta head: returns (C_k, C_v, beta [t, H]); the mass-matching
    T is the number of cached tokens N (the entries the t slots replace)."""
    N = K.shape[0]
    if kpos is None:
        kpos = np.arange(N, dtype=np.float64)
    kpos = np.asarray(kpos, dtype=np.float64)
    Z = np.asarray(W["Z"], dtype=np.float64)
    Ck = np.full((t, cfg.H, cfg.d), np.nan)
    Cv = np.full((t, cfg.H, cfg.d), np.nan)
    B = np.full((t, cfg.H), np.nan)
    for h in (range(cfg.H) if heads is None else heads):
        Ck[:, h], Cv[:, h], _, Zout = compact_head(K[:, h], V[:, h], Z[h, :t], W, cfg, kpos,
                                                   return_state=True)
        B[:, h] = beta_head(Zout, np.asarray(w_beta, dtype=np.float64), beta_max, mass_match,
                            log_x, T=N)
    return Ck, Cv, B


def as_f64(weights: dict) -> dict:
    """Widen a dict of (torch bf16 or numpy) tensors to float64 numpy arrays."""
    out = {}
    for k, v in weights.items():
        if hasattr(v, "detach"):
            import torch
            v = v.detach().to(torch.float64).cpu().numpy()
        out[k] = np.asarray(v, dtype=np.float64)
    return out


# ----------------------------------------------------------------------------- accounting

def param_count(H, d, D, t, n_blocks, n_c, n_s, r, cross_every_block, ffn_on, beta_head=True):
    """Per-layer parameter count (App. D), restated from the weight shapes of App. A.

    Counts each weight matrix (not the small biases) as laid out by the compactor: bank
    H*t*D; per CA block W_Q (D x n_c D), W_K and W_V (2d x n_c D), W_O (n_c D x D); per SA block
    S_Q, S_K, S_V (D x n_s D), S_O (n_s D x D); per FFN block W_1, W_2 (D x rD, rD x D); heads
    W_key, W_val (D x d) and w_beta (D).
    """
    bank = H * t * D
    ca = D * n_c * D + 2 * (2 * d * n_c * D) + n_c * D * D
    sa = 3 * (D * n_s * D) + n_s * D * D
    ff = 2 * (D * r * D) if ffn_on else 0
    heads = 2 * D * d + (D if beta_head else 0)
    n_ca = n_blocks if cross_every_block else 1
    return bank + n_ca * ca + n_blocks * (sa + ff) + heads


def kv_bytes(L, H, d, b, S):
    """Retained KV state M_KV(S) = 2 L H d b S bytes (App. B, Deployment accounting)."""
    return 2 * L * H * d * b * S
