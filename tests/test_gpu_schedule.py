"""GPU checks of the layer mask (mixed-attention models) and the lookahead chunked schedule
(Sec. 2.3) through the C ABI: compaction results against the fp64 oracle, untouched
buffers of skipped layers, and bit-identity with the equivalent per-layer calls."""
import numpy as np
import pytest
import torch

from oracle import still_oracle as O
from paper_2606_07878_gb300 import still, synth

from gpu_helpers import Runner, assert_parity, oracle_layer

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


def _small(**over):
    wl = dict(L=1, N=1000, H=2, d=128, D=256, n=2, F=512, ts=(100,), theta=1e6, heavy=4)
    wl.update(over)
    return wl


def test_masked_stack_compacts_only_global_layers():
    """Six layers in a 5-local : 1-global interleave with two global layers (1 and 4 here);
    the sliding-window layers' buffers must stay as they were."""
    wl = _small(L=6, N=400)
    t = 40
    mask = [0, 1, 0, 0, 1, 0]
    glob = [l for l, m in enumerate(mask) if m]
    r = Runner(wl, t, layers=glob)
    try:
        Ks, Vs, Cks, Cvs = [], [], [], []
        for l in range(6):
            K, V = synth.gen_kv(wl, l, device=DEV)
            Ck, Cv = r.out(t)
            Ck.fill_(7.0)
            Cv.fill_(-3.0)
            Ks.append(K)
            Vs.append(V)
            Cks.append(Ck)
            Cvs.append(Cv)
        _, _, off = still.still_compact_stack_masked(r.ctx, mask, Ks, Vs, t, Cks, Cvs)
        r.check_status()
        assert off == 400 - t
        for l in range(6):
            if not mask[l]:
                assert torch.all(Cks[l] == 7.0) and torch.all(Cvs[l] == -3.0), l
                continue
            rk, rv, _, _ = oracle_layer(wl, r.W[l], Ks[l], Vs[l], t)
            assert_parity(rk, synth.bf16_to_f64(Cks[l]), f"C_k layer {l}")
            assert_parity(rv, synth.bf16_to_f64(Cvs[l]), f"C_v layer {l}")
            Ck1, Cv1, _ = r.layer(l, Ks[l], Vs[l], t)  # same call alone: bit-identical
            assert torch.equal(Ck1, Cks[l]) and torch.equal(Cv1, Cvs[l]), l
        # skipped layers may be NULL; an unloaded layer that is not skipped is refused
        nul = [x if m else None for x, m in zip(Ks, mask)]
        still.still_compact_stack_masked(r.ctx, mask, nul, [x if m else None for x, m in
                                                          zip(Vs, mask)], t,
                                         [x if m else None for x, m in zip(Cks, mask)],
                                         [x if m else None for x, m in zip(Cvs, mask)])
        r.check_status()
        with pytest.raises(still.StillError) as e:
            still.still_compact_stack_masked(r.ctx, [1, 1, 0, 0, 1, 0], Ks, Vs, t, Cks, Cvs)
        assert e.value.name == "STILL_ERR_NOT_LOADED"
    finally:
        r.close()


@pytest.mark.parametrize("c,t,passes", [(8, 16, [0, 3, 7]), (4, 37, [2, 0])])
def test_lookahead_pass_compaction_matches_oracle(c, t, passes):
    """Each sequence's raw chunk sits at positions k*c*t .. (k+1)*c*t - 1 of its context; the
    oracle compacts that chunk alone at those positions."""
    wl = _small()
    ct = c * t
    r = Runner(wl, t)
    try:
        chunks = []
        for b, k in enumerate(passes):
            kpos = np.arange(k * ct, (k + 1) * ct, dtype=np.float64)
            chunks.append(synth.gen_kv(wl, 0, N=ct, device=DEV, stream=b,
                                       positions=torch.tensor(kpos)) + (kpos,))
        K = torch.cat([x[0] for x in chunks]).contiguous()
        V = torch.cat([x[1] for x in chunks]).contiguous()
        Ck = torch.empty((len(passes) * t, wl["H"], wl["d"]), dtype=torch.bfloat16, device=DEV)
        Cv = torch.empty_like(Ck)
        still.still_lookahead_compact_layer(r.ctx, 0, K, V, passes, c, t, Ck, Cv)
        r.check_status()
        for b, (Kb, Vb, kpos) in enumerate(chunks):
            rk, rv, _, _ = oracle_layer(wl, r.W[0], Kb, Vb, t, kpos=kpos)
            assert_parity(rk, synth.bf16_to_f64(Ck[b * t:(b + 1) * t]), f"C_k seq {b}")
            assert_parity(rv, synth.bf16_to_f64(Cv[b * t:(b + 1) * t]), f"C_v seq {b}")
    finally:
        r.close()


def test_lookahead_stack_equals_per_layer_calls():
    wl = _small(L=3, N=256)
    c, t, passes = 8, 16, [1, 5]
    ct = c * t
    mask = [1, 0, 1]
    r = Runner(wl, t, layers=(0, 2))
    try:
        Ks, Vs, Cks, Cvs = [], [], [], []
        for l in range(3):
            parts = [synth.gen_kv(wl, l, N=ct, device=DEV, stream=b,
                                  positions=torch.arange(k * ct, (k + 1) * ct,
                                                         dtype=torch.float64))
                     for b, k in enumerate(passes)]
            Ks.append(torch.cat([p[0] for p in parts]).contiguous())
            Vs.append(torch.cat([p[1] for p in parts]).contiguous())
            Cks.append(torch.zeros((len(passes) * t, wl["H"], wl["d"]), dtype=torch.bfloat16,
                                   device=DEV))
            Cvs.append(torch.zeros_like(Cks[-1]))
        still.still_lookahead_compact_stack(r.ctx, Ks, Vs, passes, c, t, Cks, Cvs, mask=mask)
        r.check_status()
        assert torch.count_nonzero(Cks[1]) == 0 and torch.count_nonzero(Cvs[1]) == 0
        for l in (0, 2):
            Ck1 = torch.empty_like(Cks[l])
            Cv1 = torch.empty_like(Cvs[l])
            still.still_lookahead_compact_layer(r.ctx, l, Ks[l], Vs[l], passes, c, t, Ck1, Cv1)
            r.check_status()
            assert torch.equal(Ck1, Cks[l]) and torch.equal(Cv1, Cvs[l]), l
    finally:
        r.close()


def test_lookahead_rejects_bad_arguments():
    wl = _small()
    r = Runner(wl, 16)
    try:
        K, V = synth.gen_kv(wl, 0, N=128, device=DEV)
        Ck = torch.empty((16, wl["H"], wl["d"]), dtype=torch.bfloat16, device=DEV)
        Cv = torch.empty_like(Ck)
        for passes, c, t, name in [([-1], 8, 16, "STILL_ERR_INVALID_ARG"),
                                   ([0], 0, 16, "STILL_ERR_INVALID_ARG"),
                                   ([0], 8, 17, "STILL_ERR_SHAPE")]:  # t above t_max
            with pytest.raises(still.StillError) as e:
                still.still_lookahead_compact_layer(r.ctx, 0, K, V, passes, c, t, Ck, Cv)
            assert e.value.name == name, (passes, c, t)
    finally:
        r.close()
