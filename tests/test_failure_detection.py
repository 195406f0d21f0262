"""Failure detection without a GPU fault: a kernel's bounded wait on a barrier that nothing
releases expires after a short limit, the kernel records the timeout and returns, the host
reads STILL_ERR_TIMEOUT from the device status, and the context keeps working."""
import pytest
import torch

from paper_2606_07878_gb300 import still, synth

from gpu_helpers import Runner, assert_parity, oracle_layer

pytestmark = pytest.mark.gpu


def test_expired_wait_is_reported_and_context_survives():
    wl = dict(synth.WORKLOADS["tiny_1k"], N=300)
    t = 30
    r = Runner(wl, t)
    try:
        code, _ = still.still_get_device_status(r.ctx)
        assert code == 0
        still.still_selftest_wait_timeout(r.ctx, 2000)  # 2 ms bound, nothing arrives
        code, detail = still.still_get_device_status(r.ctx)
        assert still.STATUS[code] == "STILL_ERR_TIMEOUT"
        assert detail[0] == 1 and detail[1] == 900 and detail[3] >= 1
        code, _ = still.still_get_device_status(r.ctx)  # the record was cleared
        assert code == 0
        K, V = synth.gen_kv(wl, 0, device="cuda:0")
        Ck, Cv, _ = r.layer(0, K, V, t)  # the context still computes correctly
        rk, rv, _, _ = oracle_layer(wl, r.W[0], K, V, t)
        assert_parity(rk, synth.bf16_to_f64(Ck), "C_k after timeout")
        assert_parity(rv, synth.bf16_to_f64(Cv), "C_v after timeout")
    finally:
        r.close()
