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

from gpu_helpers import Runner, assert_parity

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


def test_noalloc_matches_allocating_entry_point_twice():
    wl = synth.WORKLOADS["tiny_1k"]
    t = wl["ts"][0]
    r = Runner(wl, t)
    try:
        K, V = synth.gen_kv(wl, 0, device=DEV)
        Ck, Cv, info = r.layer(0, K, V, t)
        ref_k, ref_v = synth.bf16_to_f64(Ck), synth.bf16_to_f64(Cv)
        for call in range(2):
            Ck2 = torch.full_like(Ck, float("nan"))
            Cv2 = torch.full_like(Cv, float("nan"))
            info2 = still.still_compact_layer_noalloc(r.ctx, 0, K, V, t, Ck2, Cv2)
            r.check_status()
            assert info2 == info
            assert_parity(ref_k, synth.bf16_to_f64(Ck2), f"C_k call {call}")
            assert_parity(ref_v, synth.bf16_to_f64(Cv2), f"C_v call {call}")
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
