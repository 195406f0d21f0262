"""Benchmark: compacted-context tokens/s per layer stack on GB300.

One step = still_compact_stack over every layer of the Qwen-7B-shaped workload (28 layers,
N = 8192 cached tokens, 4 KV-heads of dim 128, compactor width 1024 with 8 heads, GELU FFN
4096, t = 1024 latents, 8x) on synthetic inputs already resident in HBM. Prints one JSON line.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference] [--t T]

--impl reference times the fp64 oracle (the CPU restatement of the method) on the host cores
on a bounded sample of the same workload. Under torchrun (N > 1) every rank compacts its own
document (weak scaling, no data-path collective); the timing takes the max over ranks.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

WORKLOAD = "qwen7b_8k"

# DRAM traffic of one scores-GEMM launch from an ncu capture (profiles/), valid only for the
# kernel sources it was taken on.
TRAFFIC = {"kernel_hash": None, "bytes_per_launch": None, "profile": None}


def _csrc_hash():
    h = hashlib.sha256()
    d = os.path.join(ROOT, "paper_2606_07878_gb300", "csrc")
    for f in sorted(os.listdir(d)):
        with open(os.path.join(d, f), "rb") as fh:
            h.update(f.encode())
            h.update(fh.read())
    return h.hexdigest()[:16]


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return p["hbm_gbs"], p["bf16_tflops"], p["bf16_tflops_sustained"], "measured"
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


class ClockSampler:
    """nvidia-smi clocks / throttle reasons sampled every 200 ms during the timed region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.thread.join(timeout=2)
        sm, mx, reasons = [], 0.0, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx = max(mx, float(parts[2]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(nm)
        if not sm:
            return None
        loaded = [x for x in sm if x > 0.5 * max(sm)] or sm
        return {"sm_mhz": statistics.median(loaded), "sm_max_mhz": mx,
                "reasons": sorted(reasons), "samples": len(sm)}


def _dist():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def doc_seed(rank: int) -> int:
    """Each rank compacts its own synthetic document (weak scaling)."""
    return 1 + rank


def max_over_ranks(x: float, dist, device) -> float:
    """Max of a per-rank scalar over the job (the timing reduction; not on the data path)."""
    if dist is None:
        return x
    import torch
    tt = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(tt, op=dist.ReduceOp.MAX)
    return float(tt.item())


def throughput(world: int, tokens_per_rank: int, steps: int, ms: float) -> float:
    """Whole-job tokens/s: every rank's tokens over the slowest rank's time."""
    return world * tokens_per_rank * steps / (ms / 1e3)


def algorithmic_flops(wl, t, N):
    """Per layer per sequence (W_V folded, W_K not foldable): key projection, scores, P X,
    V/O projections, self-attention, FFN, output heads."""
    H, d, D, n, F = wl["H"], wl["d"], wl["D"], wl["n"], wl["F"]
    ca = (2 * N * H * 2 * d * n * D + 2 * t * N * H * n * D + 2 * t * N * H * n * 2 * d
          + 2 * t * H * n * 2 * d * D + 2 * t * H * n * D * D)
    sa = 6 * t * H * D * n * D + 4 * t * t * H * n * D + 2 * t * H * n * D * D
    return {"total": ca + sa + 4 * t * H * D * F + 4 * t * H * D * d,
            "scores": 2 * t * N * H * n * D}


def run_cpu_baseline(wl, t, budget_s=30.0):
    """The oracle as it stands on one (layer, KV-head) slice, extrapolated to the stack."""
    import numpy as np
    import torch

    from oracle import still_oracle as O
    from paper_2606_07878_gb300 import synth

    W = synth.gen_weights(wl, 0, t, "cpu")
    K, V = synth.gen_kv(wl, 0, device="cpu")
    cfg = O.cfg_from_workload(wl)
    Kf, Vf, Wf = synth.bf16_to_f64(K), synth.bf16_to_f64(V), O.as_f64(W)
    t0 = time.perf_counter()
    O.compact_layer(Kf, Vf, Wf, cfg, t, heads=[0])
    sec = time.perf_counter() - t0
    slices = wl["L"] * wl["H"]
    value = wl["N"] / (sec * slices)
    return {"value": value, "unit": "tokens/s", "cores": os.cpu_count(), "kind": "oracle",
            "sample": f"layer 0, KV-head 0 of {wl['L']}x{wl['H']} (t={t}, N={wl['N']}), "
                      f"{sec:.1f} s, extrapolated x{slices} to the stack",
            "seconds": sec}


def run_reference(args):
    world, rank, _ = _dist()
    if rank != 0:
        return
    from paper_2606_07878_gb300 import synth
    wl = synth.WORKLOADS[WORKLOAD]
    t = args.t
    secs = []
    for i in range(args.warmup + args.steps):
        r = run_cpu_baseline(wl, t)
        if i >= args.warmup:
            secs.append(r["seconds"])
    slices = wl["L"] * wl["H"]
    mean = sum(secs) / len(secs)
    value = wl["N"] / (mean * slices)
    line = {
        "impl": "reference", "metric": "compacted context tokens/s per layer stack",
        "value": value, "unit": "tokens/s", "n_gpus": args.gpus, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": mean * 1e3 * slices, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": f"{WORKLOAD}: 28 layers, N=8192, H_kv=4, d=128, D=1024, "
                               f"8 heads, FFN 4096, t={t}", "layers": wl["L"], "N": wl["N"],
                   "t": t},
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": os.cpu_count(),
                         "kind": "oracle",
                         "sample": f"each step: layer 0, KV-head 0 of {wl['L']}x{wl['H']}, "
                                   f"extrapolated x{slices}"},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--t", type=int, default=1024)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    args = ap.parse_args()
    if args.impl == "reference":
        run_reference(args)
        return

    import torch

    from paper_2606_07878_gb300 import still, synth

    world, rank, local = _dist()
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group(backend="nccl", device_id=torch.device(f"cuda:{local}"))
    torch.cuda.set_device(local)
    dev = f"cuda:{local}"
    wl = synth.WORKLOADS[WORKLOAD]
    L, N, H, d, t = wl["L"], wl["N"], wl["H"], wl["d"], args.t
    stream = torch.cuda.current_stream()

    ctx = still.still_create(local)
    cfg = still.config_from_workload(wl, t)
    for l in range(L):
        W = synth.gen_weights(wl, l, t, dev)
        still.still_load_layer_weights(ctx, l, cfg, W)
        del W
    Ks, Vs = [], []
    for l in range(L):
        K, V = synth.gen_kv(wl, l, device=dev, seed=doc_seed(rank))
        Ks.append(K)
        Vs.append(V)
    Cks = [torch.empty((t, H, d), dtype=torch.bfloat16, device=dev) for _ in range(L)]
    Cvs = [torch.empty_like(c) for c in Cks]
    torch.cuda.synchronize()

    def step():
        still.still_compact_stack(ctx, Ks, Vs, t, Cks, Cvs, stream=stream)

    still.still_profile_enable(ctx, True)  # warm-up also primes the timing-event pool
    for _ in range(max(args.warmup, 3)):
        step()
    code, det = still.still_get_device_status(ctx, stream)
    if code != 0:
        raise RuntimeError(f"device status {still.STATUS.get(code)} {det}")

    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    still.still_profile_enable(ctx, True)
    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize()
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for _ in range(args.steps):
        step()
    ev1.record(stream)
    torch.cuda.synchronize()
    if dist is not None:
        dist.barrier()
    ms = ev0.elapsed_time(ev1)
    prof = still.still_profile_read(ctx)
    still.still_profile_enable(ctx, False)
    clk = clocks.stop()
    code, det = still.still_get_device_status(ctx, stream)
    if code != 0:
        raise RuntimeError(f"device status {still.STATUS.get(code)} {det}")
    ms = max_over_ranks(ms, dist, dev)
    ms_step = ms / args.steps
    value = throughput(world, N, args.steps, ms)
    launches = sum(v[0] for k, v in prof.items() if k != "load")

    # ---------------------------------------------------------------- end to end (host buffers)
    hK = [k.cpu().pin_memory() for k in Ks]
    hV = [v.cpu().pin_memory() for v in Vs]
    hCk = [torch.empty((t, H, d), dtype=torch.bfloat16).pin_memory() for _ in range(L)]
    hCv = [torch.empty_like(c) for c in hCk]
    h2d = sum(k.numel() * 2 for k in hK) * 2
    d2h = sum(c.numel() * 2 for c in hCk) * 2

    def e2e_step():
        for l in range(L):
            Ks[l].copy_(hK[l], non_blocking=True)
            Vs[l].copy_(hV[l], non_blocking=True)
        still.still_compact_stack(ctx, Ks, Vs, t, Cks, Cvs, stream=stream)
        for l in range(L):
            hCk[l].copy_(Cks[l], non_blocking=True)
            hCv[l].copy_(Cvs[l], non_blocking=True)

    e2e_step()
    torch.cuda.synchronize()
    if dist is not None:
        dist.barrier()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        e2e_step()
    e1.record(stream)
    torch.cuda.synchronize()
    ems = e0.elapsed_time(e1)
    ems = max_over_ranks(ems, dist, dev)
    e2e_value = throughput(world, N, args.steps, ems)

    # ---------------------------------------------------------------- roofline (scores GEMM)
    hbm, bf16_burst, bf16_sus, src = _peaks()
    fl = algorithmic_flops(wl, t, N)
    n_sc, ms_sc = prof["scores"]
    per_launch_flops = fl["scores"] * L * args.steps / max(n_sc, 1)
    achieved = per_launch_flops / (ms_sc / max(n_sc, 1) / 1e3) / 1e12 if ms_sc > 0 else None
    traffic = None
    if TRAFFIC["kernel_hash"] == _csrc_hash():
        traffic = TRAFFIC["bytes_per_launch"]
    roof = {"bound": "tensor", "kernel": "scores (3-pass split-bf16 tcgen05 GEMM)",
            "achieved": achieved, "peak": bf16_sus, "unit": "TFLOP/s",
            "frac": achieved / bf16_sus if achieved else None, "traffic": traffic,
            "peak_source": f"{src} bf16 sustained (kernel timed inside a long step)",
            "issued_tflops": achieved * 3 if achieved else None,
            "issued_frac": achieved * 3 / bf16_sus if achieved else None,
            "flops_per_launch": per_launch_flops}
    whole = fl["total"] * L * world * args.steps / (ms / 1e3) / 1e12

    line = {
        "metric": "compacted context tokens/s per layer stack",
        "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
        "warmup": max(args.warmup, 3), "ms_per_step": ms_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": f"{WORKLOAD}: 28 layers, N=8192, H_kv=4, d=128, D=1024, "
                               f"8 heads, FFN 4096, t={t} ({N // t}x)",
                   "layers": L, "N": N, "t": t,
                   "l2": "inputs larger than L2 (28 layers of K/V = "
                         f"{sum(k.numel() for k in Ks) * 4 / 1e6:.0f} MB per step)"},
        "e2e": {"value": e2e_value, "unit": "tokens/s", "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h},
        "gpu_launches": launches,
        "roofline": roof,
        "whole_path_alg_tflops": whole,
        "kernel_ms_per_step": {k: v[1] / args.steps for k, v in prof.items()
                               if k != "load" and v[0] > 0},
        "clocks": clk,
    }
    still.still_destroy(ctx)
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cb = run_cpu_baseline(wl, t)
        cb.pop("seconds", None)
        line["cpu_baseline"] = cb
    if rank == 0:
        print(json.dumps(line))
    if dist is not None:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
