"""Shared helpers for the GPU parity tests: run the library, compare with the oracle."""
import json
import os

import numpy as np
import torch

from oracle import still_oracle as O
from paper_2606_07878_gb300 import still, synth

# Tolerance of the parity bar: max |err| <= 2e-2 * RMS(reference), per-row cosine >= 0.999,
# rows = one compact slot of one KV-head (length d), C_k and C_v checked separately.
ERR_REL = 2e-2
COS_MIN = 0.999


def metrics(ref: np.ndarray, got: np.ndarray):
    rms = float(np.sqrt(np.mean(ref ** 2)))
    err = float(np.max(np.abs(got - ref))) / rms
    num = np.sum(got * ref, axis=-1)
    den = np.linalg.norm(got, axis=-1) * np.linalg.norm(ref, axis=-1)
    cos = float(np.min(num / np.maximum(den, 1e-300)))
    return err, cos


def assert_parity(ref, got, what="", err_rel=ERR_REL):
    err, cos = metrics(ref, got)
    log = os.environ.get("STILL_PARITY_LOG")
    if log:
        with open(log, "a") as f:
            f.write(json.dumps({"test": os.environ.get("PYTEST_CURRENT_TEST", "").split(" ")[0],
                                "what": what, "max_err_over_rms": err, "min_row_cos": cos})
                    + "\n")
    assert np.all(np.isfinite(got)), f"{what}: non-finite output"
    assert err <= err_rel and cos >= COS_MIN, f"{what}: max|err|/RMS={err:.4e} min cos={cos:.6f}"
    return err, cos


class Runner:
    """A context with some layers loaded from synthetic weights."""

    def __init__(self, wl, t_max, layers=(0,), device="cuda:0", weights=None, cfg_over=None):
        self.wl, self.t_max, self.dev = wl, t_max, device
        self.ctx = still.still_create(0)
        self.W = {}
        for l in layers:
            W = weights if weights is not None else synth.gen_weights(wl, l, t_max, device)
            self.W[l] = W
            still.still_load_layer_weights(
                self.ctx, l, still.config_from_workload(wl, t_max, **(cfg_over or {})), W)

    def out(self, t, N=None):
        C = torch.empty((t, self.wl["H"], self.wl["d"]), dtype=torch.bfloat16, device=self.dev)
        return C, torch.empty_like(C)

    def layer(self, l, K, V, t, segments=None):
        Ck, Cv = self.out(t)
        info = still.still_compact_layer(self.ctx, l, K, V, t, Ck, Cv, segments)
        self.check_status()
        return Ck, Cv, info

    def check_status(self):
        code, det = still.still_get_device_status(self.ctx)
        assert code == 0, f"device status {still.STATUS.get(code)} {det}"

    def close(self):
        still.still_destroy(self.ctx)


def oracle_layer(wl, W, K, V, t, kpos=None, heads=None, cfg_over=None):
    cfg = O.cfg_from_workload(wl, **(cfg_over or {}))
    return O.compact_layer(synth.bf16_to_f64(K), synth.bf16_to_f64(V), O.as_f64(W), cfg, t,
                           kpos=kpos, heads=heads)
