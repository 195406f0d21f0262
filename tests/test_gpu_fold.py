"""GPU parity of compactors without compactor RoPE, where the key projection folds into the
queries (logits d_l (x~ . W~ q^) / |x~ W~|, norms from x~ (W~ W~^T) x~), against the fp64
oracle's explicit projection; and the explicit path for the shapes the fold does not cover."""
import math

import numpy as np
import pytest
import torch

from paper_2606_07878_gb300 import still, synth

from gpu_helpers import Runner, assert_parity, metrics, oracle_layer

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


def _small(**over):
    wl = dict(L=1, N=1000, H=2, d=128, D=256, n=2, F=512, ts=(100,), theta=1e6, heavy=4)
    wl.update(over)
    return wl


def _run(wl, t, cfg_over, fold=True):
    r = Runner.__new__(Runner)
    r.wl, r.t_max, r.dev = wl, t, DEV
    r.ctx = still.still_create(0)
    still.still_set_key_fold(r.ctx, fold)
    r.W = {0: synth.gen_weights(wl, 0, t, DEV)}
    still.still_load_layer_weights(r.ctx, 0, still.config_from_workload(wl, t, **cfg_over),
                                   r.W[0])
    return r


@pytest.mark.parametrize("over,folded", [
    (dict(d=128, D=1024, n=2, F=512), True),           # 2d + 1 -> 320 < 1024
    (dict(d=64, D=256, n=3, N=700, F=256), True),      # 192 < 256
    (dict(d=128, D=256, n=2, N=900, F=0), False),      # 320 >= 256: explicit projection
    (dict(d=256, D=512, n=1, H=1, N=300, F=0), False),  # 2d = 512: two-kernel path
    (dict(d=128, D=256, n=2, F=0, n_blocks=2), False),  # two blocks: explicit projection
])
def test_no_compactor_rope_matches_oracle(over, folded):
    wl = _small(**over)
    t = 100
    nb = wl.get("n_blocks", 1)
    r = _run(wl, t, dict(compactor_rope=0))
    try:
        K, V = synth.gen_kv(wl, 0, device=DEV)
        still.still_profile_enable(r.ctx, True)
        Ck, Cv, _ = r.layer(0, K, V, t)
        prof = still.still_profile_read(r.ctx)
        still.still_profile_enable(r.ctx, False)
        assert (prof["q_rope"][0] == 0) == folded, prof["q_rope"]
        rk, rv, _, _ = oracle_layer(wl, r.W[0], K, V, t,
                                    cfg_over=dict(compactor_rope=False, n_blocks=nb))
        assert_parity(rk, synth.bf16_to_f64(Ck), f"C_k {over}")
        assert_parity(rv, synth.bf16_to_f64(Cv), f"C_v {over}")
    finally:
        r.close()


@pytest.mark.parametrize("logit_scale", [0.0, 1.0 / math.sqrt(1024)])
def test_fold_agrees_with_explicit_projection(logit_scale):
    """The same layer with the fold on and off, at the canonical d_l logit scale and at the
    1 / sqrt(d_l) ablation."""
    wl = _small(d=128, D=1024, n=2, F=512)
    t = 100
    over = dict(compactor_rope=0, logit_scale=logit_scale)
    ra, rb = _run(wl, t, over, fold=True), _run(wl, t, over, fold=False)
    try:
        K, V = synth.gen_kv(wl, 0, device=DEV)
        Cka, Cva, _ = ra.layer(0, K, V, t)
        Ckb, Cvb, _ = rb.layer(0, K, V, t)
        ocfg = dict(compactor_rope=False, logit_scale=logit_scale or None)
        rk, rv, _, _ = oracle_layer(wl, ra.W[0], K, V, t, cfg_over=ocfg)
        for tag, Ck, Cv in (("fold", Cka, Cva), ("explicit", Ckb, Cvb)):
            assert_parity(rk, synth.bf16_to_f64(Ck), f"C_k {tag} scale={logit_scale}")
            assert_parity(rv, synth.bf16_to_f64(Cv), f"C_v {tag} scale={logit_scale}")
        err, cos = metrics(synth.bf16_to_f64(Ckb).reshape(-1, wl["d"]),
                           synth.bf16_to_f64(Cka).reshape(-1, wl["d"]))
        assert err <= 4e-2 and cos >= 0.999, (err, cos)
    finally:
        ra.close()
        rb.close()


def test_fold_keeps_parity_when_groups_split_kv_heads():
    """Smaller workspace limits split the cross-attention groups down to single (KV-head,
    cross head) units; the folded path addresses u rows and shared x~ rows per group."""
    wl = _small(d=128, D=1024, n=4, H=2, N=600, F=0)
    t = 60
    r = _run(wl, t, dict(compactor_rope=0))
    try:
        K, V = synth.gen_kv(wl, 0, device=DEV)
        rk, rv, _, _ = oracle_layer(wl, r.W[0], K, V, t, cfg_over=dict(compactor_rope=False))
        total = still.still_workspace_size(r.ctx, wl["N"], t)
        ran = []
        for frac in (1.0, 0.95, 0.9, 0.85, 0.8, 0.75, 0.7, 0.65, 0.6, 0.5, 0.4):
            still.still_set_workspace_limit(r.ctx, int(total * frac))
            Ck, Cv = r.out(t)
            try:
                still.still_compact_layer(r.ctx, 0, K, V, t, Ck, Cv)
            except still.StillError as e:
                assert e.name == "STILL_ERR_OOM", e.name
                continue
            r.check_status()
            assert_parity(rk, synth.bf16_to_f64(Ck), f"C_k limit {frac}")
            assert_parity(rv, synth.bf16_to_f64(Cv), f"C_v limit {frac}")
            ran.append(frac)
        assert len(ran) >= 3 and min(ran) <= 0.85, ran  # the cross-attention units split
    finally:
        r.close()
