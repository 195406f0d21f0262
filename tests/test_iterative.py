"""Iterative re-compaction: [previous compact cache | new tokens] compacted again to the fixed
ratio (Sec. 2.3; the benchmark's append-and-recompact form). The GPU call is compared with the
oracle on the same inputs; the budgets, row offsets and logical lengths exactly."""
import numpy as np
import pytest
import torch

from oracle import still_oracle as O
from paper_2606_07878_gb300 import still, synth

from gpu_helpers import Runner, assert_parity

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
RATIO = 32


def _wl():
    return dict(L=1, N=0, H=2, d=128, D=256, n=2, F=512, ts=(), theta=1e6, heavy=1)


def _prev_cache(wl, Lp, stream):
    """A synthetic previous compact cache: t_prev slots whose keys sit (rotated) at the evenly
    spaced positions of the previous round's outputs."""
    tp = O.budget(Lp, RATIO)
    pos = O.linspace_positions(0, Lp - 1, tp)
    K, V = synth.gen_kv(wl, 0, N=tp, device=DEV, positions=torch.tensor(pos), stream=stream)
    return K, V, pos


def test_recompact_one_round_matches_oracle():
    wl = _wl()
    prev_len = [2000, 3100, 1500]
    new = [256, 300, 0]
    t_out = [O.budget(a + b, RATIO) for a, b in zip(prev_len, new)]
    r = Runner(wl, max(t_out))
    try:
        prev = [_prev_cache(wl, Lp, 10 + b) for b, Lp in enumerate(prev_len)]
        newkv = []
        for b, (Lp, nn) in enumerate(zip(prev_len, new)):
            pos = np.arange(Lp, Lp + nn, dtype=np.float64)
            newkv.append(synth.gen_kv(wl, 0, N=nn, device=DEV, positions=torch.tensor(pos),
                                      stream=20 + b) + (pos,))
        Kp = torch.cat([p[0] for p in prev]).contiguous()
        Vp = torch.cat([p[1] for p in prev]).contiguous()
        Kn = torch.cat([x[0] for x in newkv]).contiguous()
        Vn = torch.cat([x[1] for x in newkv]).contiguous()
        cu_prev = np.concatenate([[0], np.cumsum([p[0].shape[0] for p in prev])]).tolist()
        cu_new = np.concatenate([[0], np.cumsum(new)]).tolist()
        Ck = torch.empty((sum(t_out), wl["H"], wl["d"]), dtype=torch.bfloat16, device=DEV)
        Cv = torch.empty_like(Ck)
        cu_out, len_out = still.still_recompact_layer_ragged(
            r.ctx, 0, Kp, Vp, cu_prev, prev_len, Kn, Vn, cu_new, RATIO, Ck, Cv)
        r.check_status()
        assert cu_out == np.concatenate([[0], np.cumsum(t_out)]).tolist()
        assert len_out == [a + b for a, b in zip(prev_len, new)]
        cfg = O.cfg_from_workload(wl)
        W = O.as_f64(r.W[0])
        for b in range(3):
            K = torch.cat([prev[b][0], newkv[b][0]])
            V = torch.cat([prev[b][1], newkv[b][1]])
            kpos = np.concatenate([prev[b][2], newkv[b][2]])
            rk, rv, opos, _ = O.compact_layer(synth.bf16_to_f64(K), synth.bf16_to_f64(V), W, cfg,
                                              t_out[b], kpos=kpos)
            np.testing.assert_allclose(opos, O.linspace_positions(0, len_out[b] - 1, t_out[b]))
            rows = slice(cu_out[b], cu_out[b + 1])
            assert_parity(rk, synth.bf16_to_f64(Ck[rows]), f"C_k seq {b}")
            assert_parity(rv, synth.bf16_to_f64(Cv[rows]), f"C_v seq {b}")
    finally:
        r.close()


def test_recompact_rounds_bookkeeping():
    """Three rounds of append + recompact on the GPU's own outputs: budgets, offsets and
    logical lengths follow the integer recurrence exactly; outputs stay finite."""
    wl = _wl()
    lens = [1200, 2500]
    chunk = 512
    ts = [O.budget(x, RATIO) for x in lens]
    r = Runner(wl, O.budget(max(lens) + 3 * chunk, RATIO))
    try:
        parts = [synth.gen_kv(wl, 0, N=n, device=DEV, stream=b) for b, n in enumerate(lens)]
        Kp = torch.cat([p[0] for p in parts]).contiguous()
        Vp = torch.cat([p[1] for p in parts]).contiguous()
        cu = np.concatenate([[0], np.cumsum(lens)]).tolist()
        Ck = torch.empty((sum(ts), wl["H"], wl["d"]), dtype=torch.bfloat16, device=DEV)
        Cv = torch.empty_like(Ck)
        still.still_compact_layer_ragged(r.ctx, 0, Kp, Vp, cu, ts, Ck, Cv)
        cu_prev = np.concatenate([[0], np.cumsum(ts)]).tolist()
        prev_len = list(lens)
        for rnd in range(3):
            new = []
            for b, Lp in enumerate(prev_len):
                pos = torch.arange(Lp, Lp + chunk, dtype=torch.float64)
                new.append(synth.gen_kv(wl, 0, N=chunk, device=DEV, positions=pos,
                                        stream=100 * (rnd + 1) + b))
            Kn = torch.cat([x[0] for x in new]).contiguous()
            Vn = torch.cat([x[1] for x in new]).contiguous()
            t_next = [O.budget(Lp + chunk, RATIO) for Lp in prev_len]
            Ck2 = torch.empty((sum(t_next), wl["H"], wl["d"]), dtype=torch.bfloat16, device=DEV)
            Cv2 = torch.empty_like(Ck2)
            cu_out, len_out = still.still_recompact_layer_ragged(
                r.ctx, 0, Ck, Cv, cu_prev, prev_len, Kn, Vn,
                [0, chunk, 2 * chunk], RATIO, Ck2, Cv2)
            r.check_status()
            assert cu_out == np.concatenate([[0], np.cumsum(t_next)]).tolist()
            assert len_out == [Lp + chunk for Lp in prev_len]
            assert torch.isfinite(Ck2.float()).all() and torch.isfinite(Cv2.float()).all()
            Ck, Cv, cu_prev, prev_len = Ck2, Cv2, cu_out, len_out
    finally:
        r.close()
