"""Pins for the fp64 oracle: it is checked against things other than itself.

Each test fixes a fact that the paper or the mathematics gives: a scalar-loop restatement on
tiny inputs, closed forms, library routines, invariants of the definition, the identity-style
initialisation of App. C (an exact pass-through construction), and numbers the paper prints
(tests/golden/*.json, each with its source).
"""
import json
import os

import numpy as np
import pytest
import scipy.special
import scipy.stats
import torch

from oracle import brute
from oracle import still_oracle as O
from paper_2606_07878_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _golden(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def _tiny(**over):
    wl = dict(L=1, N=12, H=2, d=4, D=8, n=2, F=16, ts=(3,), theta=1e4, heavy=1)
    wl.update(over)
    return wl


def _weights_f64(wl, t, n_blocks=1, cross_every_block=True, seed=0):
    W = synth.gen_weights(wl, 0, t, "cpu", seed=seed, n_blocks=n_blocks)
    W = O.as_f64(W)
    # Scale weights up so that tiny widths give non-trivial attention patterns.
    return {k: v * 10.0 for k, v in W.items()}


# ------------------------------------------------------------------ brute force vs vectorised

@pytest.mark.parametrize("variant", [
    dict(),
    dict(final_norm=True),
    dict(compactor_rope=False),
    dict(F=0),
    dict(n_blocks=2),
    dict(n_blocks=2, cross_every_block=False),
    dict(logit_scale=1.0 / np.sqrt(8.0)),
    dict(self_attn=False),
])
def test_brute_force_matches_vectorised(variant):
    wl = _tiny()
    F = variant.get("F", wl["F"])
    wl["F"] = F
    nb = variant.get("n_blocks", 1)
    cfg = O.cfg_from_workload(wl, **variant)
    t = 3
    W = _weights_f64(wl, t, n_blocks=nb)
    K, V = synth.gen_kv(wl, 0, N=wl["N"], positions=torch.arange(wl["N"]) * 3.5 + 7.25)
    K, V = synth.bf16_to_f64(K), synth.bf16_to_f64(V)
    kpos = np.arange(wl["N"]) * 3.5 + 7.25
    Ck, Cv, opos, off = O.compact_layer(K, V, W, cfg, t, kpos)
    Wl = {k: v.tolist() for k, v in W.items()}
    for h in range(cfg.H):
        bk, bv = brute.compact_head_brute(K[:, h].tolist(), V[:, h].tolist(),
                                          W["Z"][h, :t].tolist(), Wl, cfg, kpos.tolist())
        np.testing.assert_allclose(Ck[:, h], np.array(bk), rtol=0, atol=1e-10)
        np.testing.assert_allclose(Cv[:, h], np.array(bv), rtol=0, atol=1e-10)
    assert off == wl["N"] - t
    assert np.all(np.isfinite(Ck)) and np.abs(Ck).max() > 1e-3


# ------------------------------------------------------------------ RoPE

def test_rope_roundtrip_and_zero_position():
    rng = np.random.default_rng(0)
    x = rng.standard_normal((64, 128))
    pos = np.concatenate([np.arange(32) * 6250.0, rng.uniform(0, 2e5, 32)])  # up to 2e5, fractional
    for base in (10.0, 1e4, 1e6):
        y = O.unrope(O.rope(x, pos, base), pos, base)
        assert np.max(np.abs(y - x)) <= 1e-14 * np.max(np.abs(x)) * 10
        np.testing.assert_array_equal(O.rope(x, np.zeros(64), base), x)


def test_rope_is_complex_multiplication():
    """Half-split RoPE: (x_m + i x_{m+w/2}) * exp(i p omega_m), omega_m = base^(-2m/w)."""
    rng = np.random.default_rng(1)
    w, base = 16, 10.0
    x = rng.standard_normal((5, w))
    pos = rng.uniform(0, 1000, 5)
    z = (x[:, : w // 2] + 1j * x[:, w // 2:])
    omega = np.array([base ** (-(2.0 * m) / w) for m in range(w // 2)])
    zr = z * np.exp(1j * pos[:, None] * omega[None, :])
    ref = np.concatenate([zr.real, zr.imag], axis=1)
    np.testing.assert_allclose(O.rope(x, pos, base), ref, atol=1e-11)
    # rotation preserves norms
    np.testing.assert_allclose(np.linalg.norm(O.rope(x, pos, base), axis=1),
                               np.linalg.norm(x, axis=1), rtol=1e-13)


# ------------------------------------------------------------------ norms, softmax, GELU

def test_softmax_rows_sum_to_one_and_match_library():
    rng = np.random.default_rng(2)
    s = rng.standard_normal((7, 300)) * 200.0          # d_l-scaled logits
    p = O.softmax_rows(s)
    np.testing.assert_allclose(p.sum(axis=1), 1.0, atol=1e-14)
    np.testing.assert_allclose(p, scipy.special.softmax(s, axis=1), rtol=1e-12, atol=1e-300)


def test_l2norm_unit_and_zero():
    rng = np.random.default_rng(3)
    x = rng.standard_normal((9, 33))
    np.testing.assert_allclose(np.linalg.norm(O.l2norm(x, 1e-12), axis=1), 1.0, atol=1e-14)
    np.testing.assert_array_equal(O.l2norm(np.zeros((2, 5)), 1e-12), 0.0)


def test_rmsnorm_closed_form():
    rng = np.random.default_rng(4)
    x = rng.standard_normal((9, 64)) * 1e-3
    eps = 1e-6
    ms = np.mean(x * x, axis=1)
    y = O.rmsnorm(x, eps)
    np.testing.assert_allclose(np.mean(y * y, axis=1), ms / (ms + eps), rtol=1e-13)
    np.testing.assert_array_equal(O.rmsnorm(np.zeros((1, 8)), eps), 0.0)


def test_gelu_is_x_times_normal_cdf():
    x = np.linspace(-8, 8, 1001)
    np.testing.assert_allclose(O.gelu(x), x * scipy.stats.norm.cdf(x), atol=1e-15)


# ------------------------------------------------------------------ cross-attention invariants

def _ca_setup(N=40, seed=5):
    wl = _tiny(N=N)
    cfg = O.cfg_from_workload(wl)
    W = _weights_f64(wl, 4, seed=seed)
    rng = np.random.default_rng(seed)
    X = rng.standard_normal((N, 2 * wl["d"]))
    Zn = O.rmsnorm(W["Z"][0, :4], cfg.rms_eps)
    return wl, cfg, W, X, Zn


def test_zero_scores_give_mean_of_projected_values():
    """W_Q = 0, b_Q = 0 -> q = 0, every logit 0 -> head_i = mean_n(X) W_V,i."""
    wl, cfg, W, X, Zn = _ca_setup()
    W = dict(W)
    W["Wq"] = np.zeros_like(W["Wq"])
    W["bq"] = np.zeros_like(W["bq"])
    kpos = np.arange(X.shape[0], dtype=float)
    qpos = O.linspace_positions(0, X.shape[0] - 1, Zn.shape[0])
    out = O.cross_attention(Zn, X, W, 0, cfg, qpos, kpos)
    D = cfg.D
    mean = np.mean(X, axis=0)
    heads = np.concatenate([mean @ W["Wv"][:, i * D:(i + 1) * D] for i in range(cfg.n_c)])
    ref = np.tile(heads @ W["Wo"], (Zn.shape[0], 1))
    np.testing.assert_allclose(out, ref, atol=1e-12)


def test_self_attention_zero_scores_give_mean_of_values():
    """S_Q = S_K = 0 and zero query/key biases -> q = k = 0 (the L2 norm keeps a zero vector
    zero), every self-attention logit 0 -> each latent receives Concat_i(mean_j v_ij) S_O with
    v_i = Zn S_V,i (App. A, Latent self-attention), compared with np.mean."""
    wl, cfg, W, X, Zn = _ca_setup()
    W = dict(W)
    for k in ("Sq", "sbq", "Sk", "sbk"):
        W[k] = np.zeros_like(W[k])
    out = O.self_attention(Zn, W, 0, cfg)
    D = cfg.D
    heads = np.concatenate([np.mean(Zn @ W["Sv"][:, i * D:(i + 1) * D], axis=0)
                            for i in range(cfg.n_s)])
    ref = np.tile(heads @ W["So"], (Zn.shape[0], 1))
    np.testing.assert_allclose(out, ref, atol=1e-12)
    # the rows of Zn differ, so a per-row (not averaged) value would not match
    assert np.abs(Zn @ W["Sv"][:, :D] - np.mean(Zn @ W["Sv"][:, :D], axis=0)).max() > 1e-3


def test_permutation_invariance():
    """Jointly permuting (K row, V row, position) leaves C_k, C_v unchanged."""
    wl = _tiny(N=30)
    cfg = O.cfg_from_workload(wl)
    W = _weights_f64(wl, 4)
    kpos = np.arange(30) * 2.0 + 5.0
    K, V = synth.gen_kv(wl, 0, N=30, positions=torch.tensor(kpos))
    K, V = synth.bf16_to_f64(K), synth.bf16_to_f64(V)
    perm = np.random.default_rng(6).permutation(30)
    a = O.compact_layer(K, V, W, cfg, 4, kpos)
    b = O.compact_layer(K[perm], V[perm], W, cfg, 4, kpos[perm])
    np.testing.assert_allclose(a[0], b[0], atol=1e-12)
    np.testing.assert_allclose(a[1], b[1], atol=1e-12)


def test_compactor_rope_translation_invariance():
    """Only p_n - p_j enters the compactor RoPE: shifting every position leaves CA unchanged."""
    wl, cfg, W, X, Zn = _ca_setup()
    N = X.shape[0]
    kpos = np.arange(N, dtype=float) * 1.5
    qpos = O.linspace_positions(kpos.min(), kpos.max(), Zn.shape[0])
    a = O.cross_attention(Zn, X, W, 0, cfg, qpos, kpos)
    b = O.cross_attention(Zn, X, W, 0, cfg, qpos + 1234.5, kpos + 1234.5)
    np.testing.assert_allclose(a, b, atol=1e-9)


# ------------------------------------------------------------------ identity-style init (App. C)

def identity_init_weights(H, d, N):
    """App. C construction with d_l = 2d, one cross head: Z = 0, W_K = 0, W_Q = 0, aligned q/k
    biases u spread evenly over all compactor frequency pairs, W_V = W_O = I, refinement
    outputs (S_O, W_2) zero, W_key = [I 0], W_val = [0 I]."""
    D = 2 * d
    rng = np.random.default_rng(11)
    u = np.full(D, 1.0 / np.sqrt(D))
    W = {
        "Z": np.zeros((H, N, D)),
        "Wq": np.zeros((D, D)), "bq": u.copy(), "Wk": np.zeros((2 * d, D)), "bk": u.copy(),
        "Wv": np.eye(2 * d, D), "Wo": np.eye(D),
        "Sq": rng.standard_normal((D, D)) * 0.02, "sbq": rng.standard_normal(D) * 0.02,
        "Sk": rng.standard_normal((D, D)) * 0.02, "sbk": rng.standard_normal(D) * 0.02,
        "Sv": rng.standard_normal((D, D)) * 0.02, "So": np.zeros((D, D)),
        "W1": rng.standard_normal((D, 4 * D)) * 0.02, "W2": np.zeros((4 * D, D)),
        "Wkey": np.concatenate([np.eye(d), np.zeros((d, d))], axis=0),
        "Wval": np.concatenate([np.zeros((d, d)), np.eye(d)], axis=0),
    }
    return W


def test_identity_init_passes_keys_and_values_through():
    H, d, N = 2, 128, 96
    W = identity_init_weights(H, d, N)
    cfg = O.Cfg(H=H, d=d, D=2 * d, n_c=1, n_s=1, F=4 * 2 * d, theta=1e4)
    wl = dict(N=N, H=H, d=d, theta=1e4, heavy=4)
    K, V = synth.gen_kv(wl, 0, N=N)
    K, V = synth.bf16_to_f64(K), synth.bf16_to_f64(V)
    Ck, Cv, opos, off = O.compact_layer(K, V, W, cfg, N)
    np.testing.assert_array_equal(opos, np.arange(N))
    assert off == 0
    np.testing.assert_allclose(Ck, K, atol=1e-9)
    np.testing.assert_allclose(Cv, V, atol=1e-9)


def test_identity_init_two_blocks_passes_through():
    """App. C for a compactor of two blocks: the later block's cross-attention output projection
    and the refinement outputs are zero, so the pass-through survives the second block whatever
    its other weights (random here). Same shape as the one-block construction above, whose
    block-diagonal attention makes the pass-through exact to rounding."""
    H, d, N = 2, 128, 96
    D = 2 * d
    W = identity_init_weights(H, d, N)
    rng = np.random.default_rng(12)
    for name, shape in (("Wq", (D, D)), ("bq", (D,)), ("Wk", (2 * d, D)), ("bk", (D,)),
                        ("Wv", (2 * d, D)), ("Sq", (D, D)), ("sbq", (D,)), ("Sk", (D, D)),
                        ("sbk", (D,)), ("Sv", (D, D)), ("W1", (D, 4 * D))):
        W[name + "@1"] = rng.standard_normal(shape) * 0.05
    for name, shape in (("Wo", (D, D)), ("So", (D, D)), ("W2", (4 * D, D))):
        W[name + "@1"] = np.zeros(shape)
    cfg = O.Cfg(H=H, d=d, D=D, n_c=1, n_s=1, F=4 * D, theta=1e4, n_blocks=2)
    wl = dict(N=N, H=H, d=d, theta=1e4, heavy=4)
    K, V = synth.gen_kv(wl, 0, N=N)
    K, V = synth.bf16_to_f64(K), synth.bf16_to_f64(V)
    Ck, Cv, _, _ = O.compact_layer(K, V, W, cfg, N)
    np.testing.assert_allclose(Ck, K, atol=1e-9)
    np.testing.assert_allclose(Cv, V, atol=1e-9)
    # a non-zero later output projection breaks it (the pin sees the second block)
    W["Wo@1"] = np.eye(D) * 0.1
    Ck2, _, _, _ = O.compact_layer(K, V, W, cfg, N)
    assert np.abs(Ck2 - K).max() > 1e-3


# ------------------------------------------------------------------ printed numbers

def test_budgets_match_paper_table():
    g = _golden("budgets.json")
    for ctx, ratio, K in g["rows"]:
        assert O.budget(g["ctx_tokens"][ctx], ratio) == K, (ctx, ratio, K)
    assert O.budget(5, 2) == 3 and O.budget(3, 2) == 2      # halves round up


def test_param_counts_match_paper():
    g = _golden("param_counts.json")
    b = g["base"]
    for c in g["cases"]:
        shapes = synth.weight_shapes(b["H"], b["d"], c["D"], c["n"], c["r"] * c["D"], c["t"],
                                     n_blocks=c["B"], cross_every_block=c["cross_every_block"])
        # Matrices only (the count ignores the small biases) plus the D-wide w_beta head.
        per_layer = sum(int(np.prod(s)) for s in shapes.values() if len(s) > 1) + c["D"]
        total = b["L"] * per_layer
        assert abs(total - c["printed_total"]) <= g["tolerance_abs"], (c["name"], total)
        assert per_layer == O.param_count(b["H"], b["d"], c["D"], c["t"], c["B"], c["n"], c["n"],
                                          c["r"], c["cross_every_block"], c["r"] > 0)


def test_kv_bytes_match_paper():
    g = _golden("kv_bytes.json")
    m = g["model"]
    assert O.kv_bytes(m["L"], m["H"], m["d"], m["b"], 1) == g["per_token_kib"] * 1024
    for S, gib in g["gib_at_tokens"]:
        assert O.kv_bytes(m["L"], m["H"], m["d"], m["b"], S) / 2**30 == pytest.approx(gib, abs=5e-4)
    for S, mib in g["mib_at_K"]:
        assert round(O.kv_bytes(m["L"], m["H"], m["d"], m["b"], S) / 2**20) == mib
    for S, gib in g["retained_gib_vllm"]:
        assert O.kv_bytes(m["L"], m["H"], m["d"], m["b"], S) / 2**30 == pytest.approx(gib, abs=5e-4)


# ------------------------------------------------------------------ lookahead schedule

def test_lookahead_schedule_matches_paper_counts():
    g = _golden("iterative_slots.json")
    t = g["t"]
    for c, tokens in g["chunk_tokens"]:
        assert O.lookahead_pass(0, c, t)["chunk_len"] == tokens
    for case in g["cases"]:
        passes, retained = O.lookahead_totals(case["T"], case["c"], t)
        if "passes" in case:
            assert passes == case["passes"], case
        if "retained" in case:
            assert retained == case["retained"], case


@pytest.mark.parametrize("c,t", [(8, 128), (3, 5), (1, 1), (32, 7)])
def test_lookahead_schedule_invariants(c, t):
    ct = c * t
    n = 20
    passes = [O.lookahead_pass(k, c, t) for k in range(n)]
    # chunks are compacted in order, each once; every token is prefilled exactly once, in order
    assert [p["chunk_start"] for p in passes] == [k * ct for k in range(n)]
    prefilled = []
    for p in passes:
        prefilled.extend(range(p["prefill_start"], p["prefill_start"] + p["prefill_len"]))
    assert prefilled == list(range((n + 1) * ct))
    for k, p in enumerate(passes):
        # by the end of the pass the chunk and one more (the lookahead) have been prefilled
        assert p["prefill_start"] + p["prefill_len"] == p["chunk_start"] + 2 * ct
        if k:
            assert p["prefill_start"] == p["chunk_start"] + ct  # the chunk just before the new one
            assert p["prefill_past"] == (k + c) * t            # (N + c) t in Sec. 2.3
        compacted = (k + 1) * ct
        assert p["retained_after"] == compacted // c + ct      # T / c + ct
        assert p["compact_row"] == k * t
        assert p["logical_after"] - p["pos_offset_after"] == p["retained_after"]
    with pytest.raises(ValueError):
        O.lookahead_totals(0, c, t)
    if ct > 1:
        with pytest.raises(ValueError):
            O.lookahead_totals(ct + 1, c, t)


# ------------------------------------------------------------------ beta channel

def test_beta_head_identity_init_and_shaping():
    rng = np.random.default_rng(5)
    Zout = rng.standard_normal((12, 32))
    # identity-style initialisation sets w_beta = 0 (App. C): no bias at all
    assert np.all(O.beta_head(Zout, np.zeros(32)) == 0)
    # ... and exact mass matching alone then gives the uniform offset log(T / t)
    np.testing.assert_allclose(O.beta_head(Zout, np.zeros(32), mass_match=1, T=600),
                               np.log(600 / 12), rtol=0, atol=1e-15)
    w = rng.standard_normal(32)
    raw = Zout @ w
    np.testing.assert_allclose(O.beta_head(Zout, w), raw, rtol=1e-15)
    sat = O.beta_head(Zout, 0.5 * w, beta_max=3.0)
    assert np.all(np.abs(sat) < 3.0) and np.all(np.sign(sat) == np.sign(raw))
    assert np.all(np.abs(sat) < np.abs(0.5 * raw))      # tanh(x) < x for x > 0
    # far below beta_max the saturation is the identity to second order
    # (relative deviation (beta / beta_max)^2 / 3 < 1e-9 here)
    np.testing.assert_allclose(O.beta_head(Zout, 1e-4 * w, beta_max=50.0), 1e-4 * raw,
                               rtol=1e-8)
    # learnable mass matching at x0 = 1e-3 starts 3 ln 10 below exact mass matching
    d = (O.beta_head(Zout, w, mass_match=2, log_x=np.log(1e-3), T=600)
         - O.beta_head(Zout, w, mass_match=1, T=600))
    np.testing.assert_allclose(d, -3 * np.log(10), rtol=1e-14)


def test_biased_attention_reduces_to_softmax_attention():
    rng = np.random.default_rng(6)
    d = 16
    q = rng.standard_normal((3, d))
    Ck, Cv = rng.standard_normal((5, d)), rng.standard_normal((5, d))
    Kf, Vf = rng.standard_normal((7, d)), rng.standard_normal((7, d))
    s = 1 / np.sqrt(d)
    out = O.biased_attention(q, Ck, Cv, np.zeros(5), Kf, Vf, s)
    K, V = np.concatenate([Ck, Kf]), np.concatenate([Cv, Vf])
    ref = scipy.special.softmax(s * q @ K.T, axis=1) @ V
    np.testing.assert_allclose(out, ref, rtol=1e-12, atol=1e-14)
    # no uncompacted entries, or no compact prefix
    np.testing.assert_allclose(O.biased_attention(q, Ck, Cv, np.zeros(5), Kf[:0], Vf[:0], s),
                               scipy.special.softmax(s * q @ Ck.T, axis=1) @ Cv, rtol=1e-12)
    np.testing.assert_allclose(O.biased_attention(q, Ck[:0], Cv[:0], np.zeros(0), Kf, Vf, s),
                               scipy.special.softmax(s * q @ Kf.T, axis=1) @ Vf, rtol=1e-12)


def test_bias_log_m_equals_m_copies_of_the_slot():
    """A compact slot carrying beta = log m attends exactly like m identical raw entries."""
    rng = np.random.default_rng(7)
    d = 8
    q = rng.standard_normal((4, d))
    Ck, Cv = rng.standard_normal((3, d)), rng.standard_normal((3, d))
    Kf, Vf = rng.standard_normal((5, d)), rng.standard_normal((5, d))
    m = np.array([1, 4, 9])
    out = O.biased_attention(q, Ck, Cv, np.log(m), Kf, Vf, 0.3)
    Kx = np.concatenate([np.repeat(Ck, m, axis=0), Kf])
    Vx = np.concatenate([np.repeat(Cv, m, axis=0), Vf])
    rows = []
    for qi in q:                      # brute force, one query at a time
        w = np.exp(0.3 * Kx @ qi - np.max(0.3 * Kx @ qi))
        rows.append(w @ Vx / w.sum())
    np.testing.assert_allclose(out, np.array(rows), rtol=1e-12, atol=1e-14)


def test_mass_matching_restores_the_prefix_share_under_uniform_attention():
    """With equal logits (q = 0), slots offset by log(T / t) take the share T / (T + S) of the
    attention that T uncompacted prefix tokens would take next to S others."""
    d, t, T, S = 8, 6, 300, 40
    rng = np.random.default_rng(8)
    Ck = rng.standard_normal((t, d))
    Cv = np.ones((t, d))
    Kf = rng.standard_normal((S, d))
    Vf = np.zeros((S, d))
    beta = O.beta_head(rng.standard_normal((t, 4)), np.zeros(4), mass_match=1, T=T)
    share = O.biased_attention(np.zeros((1, d)), Ck, Cv, beta, Kf, Vf, 1.0)[0, 0]
    assert share == pytest.approx(T / (T + S), rel=1e-13)
