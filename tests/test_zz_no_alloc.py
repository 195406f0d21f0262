"""still_compact_layer_noalloc: the variant for callers that cannot allocate device memory at
call time (a serving engine whose pool owns all free HBM, a loop that must not hit
cudaMalloc's implicit synchronisation). It runs in a fixed scratch array compiled into the
library and must give the same compaction as still_compact_layer.

Collected last on purpose (file name), so that a stop-at-first-failure run has already run
everything else; it also passes alone in a fresh process.
"""
import pytest
import torch

from paper_2606_07878_gb300 import still, synth

from gpu_helpers import Runner, assert_parity, oracle_layer

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


def test_noalloc_matches_allocating_entry_point_twice():
    """Where the fixed scratch holds the same grouping as the context workspace, the launch
    sequence is the same and deterministic: both calls give the allocating call's bits."""
    wl = synth.WORKLOADS["tiny_1k"]
    t = wl["ts"][0]
    r = Runner(wl, t)
    try:
        K, V = synth.gen_kv(wl, 0, device=DEV)
        Ck, Cv, info = r.layer(0, K, V, t)
        for call in range(2):
            Ck2 = torch.full_like(Ck, float("nan"))
            Cv2 = torch.full_like(Cv, float("nan"))
            info2 = still.still_compact_layer_noalloc(r.ctx, 0, K, V, t, Ck2, Cv2)
            r.check_status()
            assert info2 == info
            assert torch.equal(Ck2, Ck), f"C_k call {call}"
            assert torch.equal(Cv2, Cv), f"C_v call {call}"
    finally:
        r.close()


def test_noalloc_smaller_groups_meet_the_oracle_bar():
    """An 8k-token layer (H = 2, d = 128, d_l = 512, 4 heads, t = 256) whose cross-attention
    units fit the fixed scratch only one (KV-head, head) pair at a time, while the context
    workspace takes all eight at once: the groupings differ (more fused cross-attention
    launches), so the two entry points are compared with the oracle, on two calls in a row."""
    wl = dict(L=1, N=8192, H=2, d=128, D=512, n=4, F=1024, ts=(256,), theta=1e6, heavy=4)
    t = 256
    r = Runner(wl, t)
    try:
        K, V = synth.gen_kv(wl, 0, device=DEV)
        rk, rv, _, _ = oracle_layer(wl, r.W[0], K, V, t)
        still.still_profile_enable(r.ctx, True)
        still.still_profile_enable_classes(r.ctx, [])
        Ck, Cv, info = r.layer(0, K, V, t)
        n_alloc = still.still_profile_read(r.ctx)["ca_fused"][0]
        assert_parity(rk, synth.bf16_to_f64(Ck), "C_k allocating")
        assert_parity(rv, synth.bf16_to_f64(Cv), "C_v allocating")
        for call in range(2):
            still.still_profile_enable(r.ctx, True)
            still.still_profile_enable_classes(r.ctx, [])
            Ck2 = torch.full_like(Ck, float("nan"))
            Cv2 = torch.full_like(Cv, float("nan"))
            info2 = still.still_compact_layer_noalloc(r.ctx, 0, K, V, t, Ck2, Cv2)
            r.check_status()
            n_fixed = still.still_profile_read(r.ctx)["ca_fused"][0]
            assert info2 == info
            assert n_fixed > n_alloc, (n_fixed, n_alloc)
            assert_parity(rk, synth.bf16_to_f64(Ck2), f"C_k call {call}")
            assert_parity(rv, synth.bf16_to_f64(Cv2), f"C_v call {call}")
        still.still_profile_enable(r.ctx, False)
    finally:
        r.close()


def test_noalloc_rejects_sizes_beyond_the_scratch():
    wl = dict(synth.WORKLOADS["tiny_1k"])
    t = wl["ts"][0]
    r = Runner(wl, t)
    try:
        # 2^20 tokens: the strip buffers alone exceed the fixed scratch. The tensors are real,
        # full-size buffers, so nothing could read outside them even if the size were accepted.
        N = 1 << 20
        K = torch.zeros((N, wl["H"], wl["d"]), dtype=torch.bfloat16, device=DEV)
        V = torch.zeros_like(K)
        Ck, Cv = r.out(t)
        with pytest.raises(still.StillError) as e:
            still.still_compact_layer_noalloc(r.ctx, 0, K, V, t, Ck, Cv)
        assert e.value.name == "STILL_ERR_OOM"
        r.check_status()
    finally:
        r.close()
