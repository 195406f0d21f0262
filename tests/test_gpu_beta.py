"""GPU checks of the optional bias channel (App. A "Optional beta shaping"; App. B "Bias
semantics in attention"): the beta head against the oracle, and the biased decode attention
over [C_k; K_fix] against the oracle, through the C ABI."""
import math

import numpy as np
import pytest
import torch

from oracle import still_oracle as O
from paper_2606_07878_gb300 import still, synth

from gpu_helpers import Runner, assert_parity, metrics

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


def _small(**over):
    wl = dict(L=1, N=1000, H=2, d=128, D=256, n=2, F=512, ts=(100,), theta=1e6, heavy=4)
    wl.update(over)
    return wl


def _bf16(shape, seed, scale=1.0):
    g = torch.Generator().manual_seed(seed)
    return (scale * torch.randn(shape, generator=g)).to(torch.bfloat16).to(DEV)


@pytest.mark.parametrize("shaping", [dict(), dict(beta_max=0.05, mass_match=1),
                                     dict(mass_match=2, log_x=math.log(1e-3))])
def test_beta_head_matches_oracle(shaping):
    wl = _small()
    t = 100
    r = Runner(wl, t)
    try:
        w = _bf16((wl["D"],), 11, 0.02)
        K, V = synth.gen_kv(wl, 0, device=DEV)
        with pytest.raises(still.StillError) as e:  # no beta head yet
            still.still_compact_layer_beta(r.ctx, 0, K, V, t, *r.out(t),
                                           torch.empty((t, wl["H"]), device=DEV))
        assert e.value.name == "STILL_ERR_NOT_LOADED"
        still.still_set_beta_head(r.ctx, 0, w, **shaping)
        Ck, Cv = r.out(t)
        beta = torch.full((t, wl["H"]), float("nan"), device=DEV)
        still.still_compact_layer_beta(r.ctx, 0, K, V, t, Ck, Cv, beta)
        r.check_status()
        Ck0, Cv0, _ = r.layer(0, K, V, t)       # the compaction itself is unchanged
        assert torch.equal(Ck0, Ck) and torch.equal(Cv0, Cv)
        cfg = O.cfg_from_workload(wl)
        rk, rv, rb = O.compact_layer_beta(synth.bf16_to_f64(K), synth.bf16_to_f64(V),
                                          O.as_f64(r.W[0]), cfg, t,
                                          w.double().cpu().numpy(), **shaping)
        assert_parity(rk, synth.bf16_to_f64(Ck), "C_k")
        got = beta.double().cpu().numpy()
        offset = 0.0
        if shaping.get("mass_match"):
            offset = math.log(wl["N"] / t) + shaping.get("log_x", 0.0)
        for h in range(wl["H"]):
            err, _ = metrics((rb[:, h] - offset)[:, None], (got[:, h] - offset)[:, None])
            assert err <= 2e-2, (h, err)
    finally:
        r.close()


@pytest.mark.parametrize("nq,Hq,H,d,t,S", [(1, 32, 8, 128, 300, 77), (3, 4, 2, 64, 0, 200),
                                           (2, 16, 8, 256, 129, 0), (4, 8, 8, 128, 1, 1)])
def test_biased_decode_attention_matches_oracle(nq, Hq, H, d, t, S):
    q = _bf16((nq, Hq, d), 1)
    Ck, Cv = _bf16((t, H, d), 2), _bf16((t, H, d), 3)
    Kf, Vf = _bf16((S, H, d), 4), _bf16((S, H, d), 5)
    g = torch.Generator().manual_seed(6)
    beta = (2.0 * torch.randn((t, H), generator=g)).to(DEV)
    out = torch.empty((nq, Hq, d), dtype=torch.bfloat16, device=DEV)
    ctx = still.still_create(0)
    try:
        still.still_attend_biased(ctx, q, Ck, Cv, beta, Kf, Vf, out)
        code, det = still.still_get_device_status(ctx)
        assert code == 0, det
        f = lambda x: x.double().cpu().numpy()
        qn, ckn, cvn, kfn, vfn, bn = f(q), f(Ck), f(Cv), f(Kf), f(Vf), f(beta)
        got = f(out)
        ref = np.empty_like(got)
        for qh in range(Hq):
            h = qh // (Hq // H)
            ref[:, qh] = O.biased_attention(qn[:, qh], ckn[:, h], cvn[:, h], bn[:, h], kfn[:, h],
                                            vfn[:, h], 1 / math.sqrt(d))
        assert_parity(ref.reshape(-1, d), got.reshape(-1, d), f"out {nq, Hq, H, d, t, S}")
        # no bias is the same as zero bias
        out0 = torch.empty_like(out)
        still.still_attend_biased(ctx, q, Ck, Cv, None, Kf, Vf, out0)
        out1 = torch.empty_like(out)
        still.still_attend_biased(ctx, q, Ck, Cv, torch.zeros_like(beta), Kf, Vf, out1)
        assert torch.equal(out0, out1)
    finally:
        still.still_destroy(ctx)


def test_decode_over_a_compaction_with_beta():
    """End to end: compact a layer with a beta head, then attend over [C_k; new tokens]."""
    wl = _small(N=600)
    t = 60
    r = Runner(wl, t)
    try:
        w = _bf16((wl["D"],), 12, 0.05)
        still.still_set_beta_head(r.ctx, 0, w, beta_max=4.0, mass_match=1)
        K, V = synth.gen_kv(wl, 0, device=DEV)
        Ck, Cv = r.out(t)
        beta = torch.empty((t, wl["H"]), device=DEV)
        still.still_compact_layer_beta(r.ctx, 0, K, V, t, Ck, Cv, beta)
        Kf, Vf = synth.gen_kv(wl, 0, N=40, device=DEV, stream=9)
        q = _bf16((1, 4 * wl["H"], wl["d"]), 13)
        out = torch.empty((1, 4 * wl["H"], wl["d"]), dtype=torch.bfloat16, device=DEV)
        still.still_attend_biased(r.ctx, q, Ck, Cv, beta, Kf, Vf, out)
        r.check_status()
        f = lambda x: x.double().cpu().numpy()
        ref = np.empty((1, 4 * wl["H"], wl["d"]))
        for qh in range(4 * wl["H"]):
            h = qh // 4
            ref[:, qh] = O.biased_attention(f(q)[:, qh], f(Ck)[:, h], f(Cv)[:, h], f(beta)[:, h],
                                            f(Kf)[:, h], f(Vf)[:, h], 1 / math.sqrt(wl["d"]))
        assert_parity(ref.reshape(-1, wl["d"]), f(out).reshape(-1, wl["d"]), "out")
    finally:
        r.close()


def test_biased_decode_rejects_bad_arguments():
    ctx = still.still_create(0)
    try:
        q = _bf16((1, 6, 128), 1)
        C = _bf16((10, 4, 128), 2)
        out = torch.empty((1, 6, 128), dtype=torch.bfloat16, device=DEV)
        with pytest.raises(still.StillError) as e:  # 6 query heads over 4 KV-heads
            still.still_attend_biased(ctx, q, C, C, None, C[:0], C[:0], out)
        assert e.value.name == "STILL_ERR_INVALID_ARG"
        q2 = _bf16((1, 4, 96), 1)
        C2 = _bf16((10, 4, 96), 2)
        with pytest.raises(still.StillError) as e:  # d = 96
            still.still_attend_biased(ctx, q2, C2, C2, None, C2[:0], C2[:0],
                                      torch.empty_like(q2))
        assert e.value.name == "STILL_ERR_UNSUPPORTED"
    finally:
        still.still_destroy(ctx)


@pytest.mark.parametrize("d,t,S", [(128, 300, 77), (256, 129, 0), (64, 0, 200)])
def test_decode_stack_equals_per_layer_calls_and_oracle(d, t, S):
    """One launch over a stack of layers: every layer's result equals the single-layer call bit
    for bit (same chunking, same merge order), and layer results match the oracle."""
    L, nq, Hq, H = 5, 1, 16, 4
    q = [_bf16((nq, Hq, d), 100 + l) for l in range(L)]
    Ck = [_bf16((t, H, d), 200 + l) for l in range(L)]
    Cv = [_bf16((t, H, d), 300 + l) for l in range(L)]
    Kf = [_bf16((S, H, d), 400 + l) for l in range(L)]
    Vf = [_bf16((S, H, d), 500 + l) for l in range(L)]
    beta = [(2.0 * torch.randn((t, H), generator=torch.Generator().manual_seed(600 + l))).to(DEV)
            for l in range(L)]
    beta[2] = None  # a layer without the bias channel
    out = [torch.empty((nq, Hq, d), dtype=torch.bfloat16, device=DEV) for _ in range(L)]
    ctx = still.still_create(0)
    try:
        still.still_attend_biased_stack(ctx, q, Ck, Cv, beta, Kf, Vf, out)
        code, det = still.still_get_device_status(ctx)
        assert code == 0, det
        f = lambda x: x.double().cpu().numpy()
        for l in range(L):
            one = torch.empty_like(out[l])
            still.still_attend_biased(ctx, q[l], Ck[l], Cv[l], beta[l], Kf[l], Vf[l], one)
            assert torch.equal(one, out[l]), l
        for l in (0, 2, L - 1):
            bn = f(beta[l]) if beta[l] is not None else np.zeros((t, H))
            ref = np.empty((nq, Hq, d))
            for qh in range(Hq):
                h = qh // (Hq // H)
                ref[:, qh] = O.biased_attention(f(q[l])[:, qh], f(Ck[l])[:, h], f(Cv[l])[:, h],
                                                bn[:, h], f(Kf[l])[:, h], f(Vf[l])[:, h],
                                                1 / math.sqrt(d))
            assert_parity(ref.reshape(-1, d), f(out[l]).reshape(-1, d), f"layer {l}")
        with pytest.raises(still.StillError) as e:  # more layers than one launch takes
            still.still_attend_biased_stack(ctx, q * 13, Ck * 13, Cv * 13, None, Kf * 13,
                                            Vf * 13, out * 13)
        assert e.value.name == "STILL_ERR_UNSUPPORTED"
    finally:
        still.still_destroy(ctx)
