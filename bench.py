"""Benchmark: compacted-context tokens/s per layer stack on GB300.

One step = still_compact_stack over every layer of the Gemma-shaped long-context workload
(48 layers, N = 131072 cached tokens, 8 KV-heads of dim 256, compactor width 2048 with 16
heads, GELU FFN 8192, t = 655 latents, 200x) on synthetic inputs already resident in HBM.
Prints one JSON line. Other workloads (--workload) are the Qwen-shaped stacks, the canonical
compactor, the iterative re-compaction and the decode-time consumer.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference] [--t T]
                  [--workload NAME]

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

WORKLOAD = "gemma_128k"
DEFAULT_T = {"qwen7b_8k": 1024, "qwen8b_32k": 2048, "gemma_128k": 655, "tiny_1k": 128,
             "qwen3_4b_64k": 1311, "qwen7b_8k_norope": 1024}


def folded(wl):
    """Whether the library folds W_K into the queries for this workload (no compactor RoPE, one
    block, 2d <= 256, x~ = [x; 1] padded to 64 narrower than d_l); returns the padded width."""
    d, D = wl["d"], wl["D"]
    Kp = (2 * d + 1 + 63) // 64 * 64
    ok = (not wl.get("compactor_rope", 1) and wl.get("n_blocks", 1) == 1 and d in (64, 128)
          and Kp < D)
    return Kp if ok else 0


def one_pass_scores(wl):
    """Whether the library computes this workload's cross-attention scores in one fp16 pass
    with a repair of each row's heaviest logits (one block, head dim 256, 512 <= d_l <= 2048)."""
    return wl.get("n_blocks", 1) == 1 and wl["d"] == 256 and 512 <= wl["D"] <= 2048


def describe(name, wl, t):
    nb = wl.get("n_blocks", 1)
    blocks = "" if nb == 1 else (f", {nb} blocks" + (" (CA in every block)"
                                                      if wl.get("cross_every_block", 1) else ""))
    rope = "" if wl.get("compactor_rope", 1) else (
        ", no compactor RoPE" + (" (W_K folded into the queries)" if folded(wl) else ""))
    return (f"{name}: {wl['L']} layers, N={wl['N']}, H_kv={wl['H']}, d={wl['d']}, "
            f"D={wl['D']}, {wl['n']} heads, FFN {wl['F']}{blocks}{rope}, t={t} "
            f"({round(wl['N'] / t)}x)")

# DRAM traffic (read + write) per launch of the dominant kernel at a workload, from an ncu
# capture; valid only for the kernel sources it was taken on (hash of the listed sources).
# The fused cross-attention kernel (the scores GEMM entry is kept for the record: no workload
# takes it any more).
TRAFFIC = {
    "scores": [],
    # one entry per captured workload
    "ca_fused": [
        # 1.313 GB read + 0.127 GB written per launch (profiles/ca_fused_qwen7b_8k_t1024.md,
        # the CTA-pair kernel, whose source is ca_flash.cuh)
        {"files": ["ca_flash.cuh"], "kernel_hash": "362e2f1dfbf525ed",
         "bytes_per_launch": 1.4405e9, "workload": ("qwen7b_8k", 1024),
         "profile": "profiles/ca_fused_qwen7b_8k_t1024.md"},
        # the head-dim-256 kernel (source ca_pair.cu) captured on one KV-head of a 16k-token
        # cache (1.231 GB read + 0.086 GB written, profiles/ca_pair_gemma_n16k_t655.md), scaled
        # by the units of a full-size launch (2 KV-heads x 131072 tokens: x16); its traffic (k
        # read once, X^T, partials) grows in proportion
        {"files": ["ca_pair.cu"], "kernel_hash": "89e4b7a50e367c33",
         "bytes_per_launch": 16 * 1.3165e9, "workload": ("gemma_128k", 655),
         "profile": "profiles/ca_pair_gemma_n16k_t655.md"},
    ],
}


def _kernel_hash(files):
    h = hashlib.sha256()
    d = os.path.join(ROOT, "paper_2606_07878_gb300", "csrc")
    for f in files:
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
    nb = wl.get("n_blocks", 1)
    n_ca = nb if wl.get("cross_every_block", 1) else 1  # blocks with cross-attention
    # With the fold the keys are never projected: the logits contract over x~ (width Kp) and
    # the key norms are x~ G x~ (Kp^2 per token and head).
    Kp = folded(wl)
    kw = Kp if Kp else D
    kproj = 2 * N * H * n * Kp * Kp if Kp else 2 * N * H * 2 * d * n * D
    ca = (kproj + 2 * t * N * H * n * kw + 2 * t * N * H * n * 2 * d
          + 2 * t * H * n * 2 * d * D + 2 * t * H * n * D * D)
    sa = 6 * t * H * D * n * D + 4 * t * t * H * n * D + 2 * t * H * n * D * D
    # Every block's cross-attention is one fused kernel (a block that feeds another in its
    # split-precision form, P X in 2.5 passes; 2d = 512 on clusters of four CTAs).
    fused = True
    return {"total": n_ca * ca + nb * (sa + 4 * t * H * D * F) + 4 * t * H * D * d,
            "scores": n_ca * 2 * t * N * H * n * kw, "px": n_ca * 2 * t * N * H * n * 2 * d,
            "scores_gemm": 0 if fused else n_ca * 2 * t * N * H * n * D,
            # passes of P X issued over all blocks with cross-attention (the last 1.5, others 2.5)
            "px_passes": 1.5 + 2.5 * (n_ca - 1), "px_blk": 2 * t * N * H * n * 2 * d}


def run_cpu_baseline(wl, t, budget_s=30.0):
    """The oracle as it stands on a bounded slice of the workload, extrapolated to the stack.

    One (layer, KV-head) when that fits the budget (the full per-head compaction); for the
    largest shapes, the cross-attention of one cross head of one KV-head, extrapolated by the
    ratio of algorithmic flops.
    """
    from oracle import still_oracle as O
    from paper_2606_07878_gb300 import synth

    fl = algorithmic_flops(wl, t, wl["N"])
    one_head = fl["total"] / wl["H"]
    W = synth.gen_weights(wl, 0, t, "cpu")
    cfg = O.cfg_from_workload(wl, n_blocks=wl.get("n_blocks", 1),
                              compactor_rope=bool(wl.get("compactor_rope", 1)),
                              cross_every_block=bool(wl.get("cross_every_block", 1)))
    Wf = O.as_f64(W)
    if one_head < 2.5e12:
        K, V = synth.gen_kv(wl, 0, device="cpu")
        Kf, Vf = synth.bf16_to_f64(K), synth.bf16_to_f64(V)
        t0 = time.perf_counter()
        O.compact_layer(Kf, Vf, Wf, cfg, t, heads=[0])
        sec = time.perf_counter() - t0
        scale = wl["L"] * wl["H"]
        what = f"layer 0, KV-head 0 of {wl['L']}x{wl['H']}"
    else:
        import numpy as np
        K, V = synth.gen_kv(wl, 0, device="cpu")
        Kf, Vf = synth.bf16_to_f64(K)[:, 0], synth.bf16_to_f64(V)[:, 0]
        kpos = np.arange(wl["N"], dtype=np.float64)
        Wi = dict(Wf)
        D = wl["D"]
        for k in ("Wq", "Wk", "Wv"):
            Wi[k] = Wf[k][:, :D]
        for k in ("bq", "bk"):
            Wi[k] = Wf[k][:D]
        Wi["Wo"] = Wf["Wo"][:D]
        c1 = O.cfg_from_workload(wl, n_c=1)
        t0 = time.perf_counter()
        X = np.concatenate([O.unrope(Kf, kpos, cfg.theta), Vf], axis=-1)
        Zn = O.rmsnorm(Wf["Z"][0, :t], cfg.rms_eps)
        O.cross_attention(Zn, X, Wi, 0, c1, O.linspace_positions(0, wl["N"] - 1, t), kpos)
        sec = time.perf_counter() - t0
        N, d = wl["N"], wl["d"]
        sample_fl = (2 * N * 2 * d * D + 2 * t * N * D + 2 * t * N * 2 * d + 2 * t * 2 * d * D
                     + 2 * t * D * D)
        scale = fl["total"] * wl["L"] / sample_fl
        what = (f"cross-attention of 1 of {wl['n']} heads of KV-head 0, layer 0, "
                f"extrapolated by algorithmic flops")
    value = wl["N"] / (sec * scale)
    return {"value": value, "unit": "tokens/s", "cores": os.cpu_count(), "kind": "oracle",
            "sample": f"{what} (t={t}, N={wl['N']}), {sec:.1f} s, x{scale:.0f} to the stack",
            "seconds": sec, "scale": scale}


def run_reference(args):
    world, rank, _ = _dist()
    if rank != 0:
        return
    from paper_2606_07878_gb300 import synth
    name = args.workload
    wl = synth.WORKLOADS[name]
    t = args.t or DEFAULT_T[name]
    secs = []
    for i in range(args.warmup + args.steps):
        r = run_cpu_baseline(wl, t)
        if i >= args.warmup:
            secs.append(r["seconds"])
    slices = r["scale"]
    mean = sum(secs) / len(secs)
    value = wl["N"] / (mean * slices)
    # A step here is one measured slice; value and ms_per_step extrapolate it to the whole
    # stack by the slice's share of the work (labelled as such in the line).
    line = {
        "impl": "reference", "metric": "compacted context tokens/s per layer stack",
        "value": value, "unit": "tokens/s", "n_gpus": args.gpus, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": mean * 1e3 * slices, "extrapolated": True,
        "measured_slice_ms": mean * 1e3, "extrapolation_factor": slices,
        "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": describe(name, wl, t), "layers": wl["L"], "N": wl["N"], "t": t},
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": os.cpu_count(),
                         "kind": "oracle", "sample": "each step: " + r["sample"],
                         "extrapolated": True},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))


# The compact cache's consumer at decode time: one generated token of one sequence through the
# biased attention of every layer of a Qwen3-4B-shaped model (32 query heads over 8 KV-heads,
# d = 128), over the canonical compaction of a 64k context (t = 1311 slots with a bias) followed
# by one raw lookahead chunk of 4096 tokens.
DECODE = dict(L=36, H=8, Hq=32, d=128, t=1311, S=4096, nq=1)


def run_decode(args):
    """Biased decode attention (App. B, "Bias semantics in attention") over [C_k; K_fix] for
    every layer in one launch (captured as a CUDA graph); one step = one decode token through
    all layers."""
    import numpy as np
    import torch

    from oracle import still_oracle as O
    from paper_2606_07878_gb300 import still

    c = DECODE
    L, H, Hq, d, t, S, nq = c["L"], c["H"], c["Hq"], c["d"], c["t"], c["S"], c["nq"]
    dev = "cuda:0"
    torch.cuda.set_device(0)
    stream = torch.cuda.Stream()
    torch.cuda.set_stream(stream)
    g = torch.Generator(device=dev).manual_seed(3)
    rnd = lambda *shape: torch.randn(shape, generator=g, device=dev).to(torch.bfloat16)
    Cks = [rnd(t, H, d) for _ in range(L)]
    Cvs = [rnd(t, H, d) for _ in range(L)]
    betas = [torch.randn((t, H), generator=g, device=dev) for _ in range(L)]
    Kfs = [rnd(S, H, d) for _ in range(L)]
    Vfs = [rnd(S, H, d) for _ in range(L)]
    qs = [rnd(nq, Hq, d) for _ in range(L)]
    outs = [torch.empty((nq, Hq, d), dtype=torch.bfloat16, device=dev) for _ in range(L)]
    ctx = still.still_create(0)

    def step():  # every layer in one launch pair (chunks + merge)
        still.still_attend_biased_stack(ctx, qs, Cks, Cvs, betas, Kfs, Vfs, outs, stream=stream)

    still.still_profile_enable(ctx, True)
    for _ in range(max(args.warmup, 3)):
        step()
    torch.cuda.synchronize()
    still.still_profile_enable_classes(ctx, ["decode"])
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        step()
    graph.replay()
    torch.cuda.synchronize()
    clocks = ClockSampler(0)
    clocks.start()
    time.sleep(0.3)
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    steps = max(args.steps, 20)  # a step is short: time at least 20
    ev0.record(stream)
    for _ in range(steps):
        graph.replay()
    ev1.record(stream)
    torch.cuda.synchronize()
    ms = ev0.elapsed_time(ev1)
    prof = still.still_profile_read(ctx)
    still.still_profile_enable(ctx, False)
    clk = clocks.stop()
    code, det = still.still_get_device_status(ctx, stream)
    if code != 0:
        raise RuntimeError(f"device status {still.STATUS.get(code)} {det}")
    del graph
    n_dec, ms_dec = prof["decode"]  # the last replay's launches (chunk + merge)
    # Algorithmic bytes of one layer's attention: the compact slots and raw entries (K and V),
    # the bias, the query and the output; one replay covers all L layers.
    layer_bytes = (t + S) * H * d * 2 * 2 + t * H * 4 + 2 * nq * Hq * d * 2
    achieved = layer_bytes * L / (ms_dec / 1e3) / 1e9 if ms_dec > 0 else None
    hbm, _, _, src = _peaks()
    # end to end: the step's queries from pinned host memory in, outputs back to the host
    q_host = [x.cpu().pin_memory() for x in qs]
    o_host = [torch.empty((nq, Hq, d), dtype=torch.bfloat16).pin_memory() for _ in range(L)]
    ds = torch.cuda.default_stream()

    def e2e_step():
        for l in range(L):
            qs[l].copy_(q_host[l], non_blocking=True)
        still.still_attend_biased_stack(ctx, qs, Cks, Cvs, betas, Kfs, Vfs, outs, stream=ds)
        for l in range(L):
            o_host[l].copy_(outs[l], non_blocking=True)
        ds.synchronize()

    with torch.cuda.stream(ds):
        e2e_step()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        for _ in range(steps):
            e2e_step()
        e2e_s = time.perf_counter() - t0
    still.still_destroy(ctx)
    cpu = None
    if not args.no_cpu_baseline:
        f = lambda x: x.double().cpu().numpy()
        qn, ck, cv, bn, kf, vf = f(qs[0]), f(Cks[0]), f(Cvs[0]), f(betas[0]), f(Kfs[0]), f(Vfs[0])
        t0 = time.perf_counter()
        for qh in range(Hq):
            h = qh // (Hq // H)
            O.biased_attention(qn[:, qh], ck[:, h], cv[:, h], bn[:, h], kf[:, h], vf[:, h],
                               1 / np.sqrt(d))
        sec = (time.perf_counter() - t0) * L
        cpu = {"value": 1.0 / sec, "unit": "decode tokens/s", "cores": os.cpu_count(),
               "kind": "oracle", "sample": f"layer 0 of {L} (all {Hq} query heads), x{L}"}
    print(json.dumps({
        "metric": "decode tokens/s through the compact cache (biased attention over [C_k; K_fix], all layers)",
        "value": steps / (ms / 1e3), "unit": "tokens/s", "n_gpus": 1, "steps": steps,
        "warmup": max(args.warmup, 3), "ms_per_step": ms / steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": f"decode_qwen3_4b: {L} layers, {Hq} query heads over {H} KV-heads, "
                               f"d={d}, {nq} query token, t={t} compact slots with bias + "
                               f"{S} raw entries",
                   "l2": f"inputs larger than L2 ({L * layer_bytes / 1e6:.0f} MB per step)"},
        "e2e": {"value": steps / e2e_s, "unit": "tokens/s",
                "h2d_bytes_per_step": L * nq * Hq * d * 2, "d2h_bytes_per_step": L * nq * Hq * d * 2},
        "gpu_launches": n_dec * steps,  # launches per replay x timed replays
        "roofline": {"bound": "hbm", "kernel": f"decode attention over {L} layers in one "
                                                 f"launch (chunks + merge)",
                     "achieved": achieved, "peak": hbm, "unit": "GB/s",
                     "frac": achieved / hbm if achieved else None, "traffic": None,
                     "peak_source": f"{src} HBM copy bandwidth",
                     "bytes_per_launch": layer_bytes * L},
        "cpu_baseline": cpu, "clocks": clk}))


def run_iterative(args):
    """The iterative ragged serving workload: 8 sequences (lengths uniform in [8k, 32k], seed
    7), 36 Qwen-8B-shaped layers, compacted to 32x; then rounds of +8192 new tokens per
    sequence, each round re-compacting [compact | new] to the 32x budget. One step = one round
    over the whole stack; the metric is new logical tokens absorbed per second."""
    import torch

    from paper_2606_07878_gb300 import still, synth

    wl = synth.WORKLOADS["iterative_ragged"]
    L, H, d, ratio, chunk = wl["L"], wl["H"], wl["d"], wl["ratio"], wl["chunk"]
    rounds = min(args.steps, wl["rounds"])
    lens = synth.iterative_lengths(wl)
    B = len(lens)
    dev = "cuda:0"
    torch.cuda.set_device(0)
    stream = torch.cuda.current_stream()
    t_cap = still.still_budget(max(lens) + wl["rounds"] * chunk, ratio)
    ctx = still.still_create(0)
    cfg = still.config_from_workload(dict(wl, N=0), t_cap)
    for l in range(L):
        W = synth.gen_weights(wl, l, t_cap, dev)
        still.still_load_layer_weights(ctx, l, cfg, W)
        del W
    # round 0: the initial caches, compacted once (untimed set-up)
    ts = [still.still_budget(x, ratio) for x in lens]
    cu = [0]
    for x in lens:
        cu.append(cu[-1] + x)
    Cks, Cvs = [], []
    for l in range(L):
        parts = [synth.gen_kv(wl, l, N=x, device=dev, stream=b) for b, x in enumerate(lens)]
        Kp = torch.cat([p[0] for p in parts])
        Vp = torch.cat([p[1] for p in parts])
        Ck = torch.empty((sum(ts), H, d), dtype=torch.bfloat16, device=dev)
        Cv = torch.empty_like(Ck)
        still.still_compact_layer_ragged(ctx, l, Kp, Vp, cu, ts, Ck, Cv, stream=stream)
        Cks.append(Ck)
        Cvs.append(Cv)
        del Kp, Vp, parts
    cu_prev = [0]
    for x in ts:
        cu_prev.append(cu_prev[-1] + x)
    prev_len = list(lens)
    cu_new = [b * chunk for b in range(B + 1)]

    def round_inputs(r):
        """Round r's new tokens (at the positions after each sequence's logical length) and its
        output buffers."""
        Kn, Vn = [], []
        for l in range(L):
            parts = [synth.gen_kv(wl, l, N=chunk, device=dev, stream=1000 * (r + 1) + b,
                                  positions=torch.arange(prev_len[b], prev_len[b] + chunk,
                                                         dtype=torch.float64))
                     for b in range(B)]
            Kn.append(torch.cat([p[0] for p in parts]))
            Vn.append(torch.cat([p[1] for p in parts]))
        t_next = [still.still_budget(x + chunk, ratio) for x in prev_len]
        Ck2 = [torch.empty((sum(t_next), H, d), dtype=torch.bfloat16, device=dev)
               for _ in range(L)]
        Cv2 = [torch.empty_like(c) for c in Ck2]
        return Kn, Vn, Ck2, Cv2

    # untimed warm-up: the first round's recompaction, its outputs dropped (the state does not
    # advance)
    Kn, Vn, Ck2, Cv2 = round_inputs(0)
    for _ in range(max(args.warmup, 3)):
        still.still_recompact_stack_ragged(ctx, Cks, Cvs, cu_prev, prev_len, Kn, Vn, cu_new,
                                           ratio, Ck2, Cv2, stream=stream)
    del Kn, Vn, Ck2, Cv2
    total_ms = 0.0
    launches = 0
    clocks = ClockSampler(0)  # sampled over the rounds (their input generation included)
    clocks.start()
    for r in range(rounds):
        Kn, Vn, Ck2, Cv2 = round_inputs(r)
        torch.cuda.synchronize()
        still.still_profile_enable(ctx, False)  # launch counts only; no events in the timing
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        cu_out, len_out = still.still_recompact_stack_ragged(
            ctx, Cks, Cvs, cu_prev, prev_len, Kn, Vn, cu_new, ratio, Ck2, Cv2, stream=stream)
        e1.record(stream)
        torch.cuda.synchronize()
        total_ms += e0.elapsed_time(e1)
        prof = still.still_profile_read(ctx)
        launches += sum(v[0] for k, v in prof.items() if k != "load")
        Cks, Cvs, cu_prev, prev_len = Ck2, Cv2, cu_out, len_out
        del Kn, Vn
    clk = clocks.stop()
    code, det = still.still_get_device_status(ctx, stream)
    if code != 0:
        raise RuntimeError(f"device status {still.STATUS.get(code)} {det}")
    still.still_destroy(ctx)
    value = B * chunk * rounds / (total_ms / 1e3)
    print(json.dumps({
        "metric": "new logical tokens absorbed per second (iterative re-compaction, all layers)",
        "value": value, "unit": "tokens/s", "n_gpus": 1, "steps": rounds, "warmup": max(args.warmup, 3),
        "ms_per_step": total_ms / rounds, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": f"iterative_ragged: {B} sequences, lengths {lens}, {L} layers, "
                               f"H_kv={H}, d={d}, D={wl['D']}, {wl['n']} heads, "
                               f"{ratio}x, +{chunk} tokens per round",
                   "final_lengths": prev_len},
        "gpu_launches": launches, "clocks": clk,
    }))


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--t", type=int, default=0, help="compact length (default per workload)")
    ap.add_argument("--workload", default=WORKLOAD,
                    choices=sorted(DEFAULT_T) + ["iterative_ragged", "decode_qwen3_4b"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    args = ap.parse_args()
    if args.impl == "reference":
        run_reference(args)
        return
    if args.workload == "iterative_ragged":
        run_iterative(args)
        return
    if args.workload == "decode_qwen3_4b":
        run_decode(args)
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
    name = args.workload
    wl = synth.WORKLOADS[name]
    L, N, H, d = wl["L"], wl["N"], wl["H"], wl["d"]
    t = args.t or DEFAULT_T[name]
    # A dedicated stream (graph capture needs a non-default one), current for every torch op
    # below so that copies and the library's kernels are ordered on it.
    stream = torch.cuda.Stream()
    torch.cuda.set_stream(stream)

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

    # One stack step is captured into a CUDA graph and replayed (the layer-stack launch sequence
    # as one graph). The dominant kernel class, the fused cross-attention, is the only one with
    # events: its launches are bracketed by event nodes of the graph, read after the last replay.
    kname = "ca_fused"
    still.still_reserve_workspace(ctx, N, t)
    still.still_profile_enable_classes(ctx, [kname])
    graph = torch.cuda.CUDAGraph()
    torch.cuda.synchronize()
    with torch.cuda.graph(graph, stream=stream):
        step()
    graph.replay()
    torch.cuda.synchronize()
    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize()
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for _ in range(args.steps):
        graph.replay()
    ev1.record(stream)
    torch.cuda.synchronize()
    if dist is not None:
        dist.barrier()
    ms = ev0.elapsed_time(ev1)
    prof_timed = still.still_profile_read(ctx)  # the dominant kernel's launches of the last replay
    still.still_profile_enable(ctx, False)
    clk = clocks.stop()
    code, det = still.still_get_device_status(ctx, stream)
    if code != 0:
        raise RuntimeError(f"device status {still.STATUS.get(code)} {det}")
    del graph
    ms = max_over_ranks(ms, dist, dev)
    ms_step = ms / args.steps
    value = throughput(world, N, args.steps, ms)

    # Per-class breakdown: a few more steps with every launch bracketed by events (not part of
    # the timed region; the events cost about 3% of a step).
    brk = max(1, min(args.steps, 2))
    still.still_profile_enable(ctx, True)
    for _ in range(brk):
        step()
    torch.cuda.synchronize()
    prof = still.still_profile_read(ctx)
    still.still_profile_enable(ctx, False)
    # Kernel launches in the timed region: each graph replay launches what one step launches.
    launches = sum(v[0] for k, v in prof.items() if k != "load") // brk * args.steps

    # ---------------------------------------------------------------- end to end (host buffers)
    hK = [k.cpu().pin_memory() for k in Ks]
    hV = [v.cpu().pin_memory() for v in Vs]
    hCk = [torch.empty((t, H, d), dtype=torch.bfloat16).pin_memory() for _ in range(L)]
    hCv = [torch.empty_like(c) for c in hCk]
    h2d = sum(k.numel() * 2 for k in hK) * 2
    d2h = sum(c.numel() * 2 for c in hCk) * 2

    # The end-to-end step runs on the default stream (pinned-host copies measured slower on a
    # side stream on this machine).
    estream = torch.cuda.default_stream()
    torch.cuda.synchronize()
    torch.cuda.set_stream(estream)

    def e2e_step():
        for l in range(L):
            Ks[l].copy_(hK[l], non_blocking=True)
            Vs[l].copy_(hV[l], non_blocking=True)
        still.still_compact_stack(ctx, Ks, Vs, t, Cks, Cvs, stream=estream)
        for l in range(L):
            hCk[l].copy_(Cks[l], non_blocking=True)
            hCv[l].copy_(Cvs[l], non_blocking=True)

    e2e_step()
    torch.cuda.synchronize()
    if dist is not None:
        dist.barrier()
    e2e_steps = max(1, min(args.steps, 3))  # whole-stack host copies: a few steps suffice
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(estream)
    for _ in range(e2e_steps):
        e2e_step()
    e1.record(estream)
    torch.cuda.synchronize()
    ems = e0.elapsed_time(e1)
    ems = max_over_ranks(ems, dist, dev)
    e2e_value = throughput(world, N, e2e_steps, ems)

    # ---------------------------------------------------------------- roofline
    # Dominant kernel: the fused cross-attention (scores + softmax + P X). Algorithmic flops
    # count each product once; the
    # issued view counts the split-precision passes (3 for q.k, 1.5 for P X: hi + key-half lo).
    hbm, bf16_burst, bf16_sus, src = _peaks()
    fl = algorithmic_flops(wl, t, N)
    fused = kname == "ca_fused"
    n_k, ms_k = prof_timed[kname]  # one step's launches (the captured event pairs)
    alg = fl["scores"] + fl["px"] if fused else fl["scores_gemm"]
    # one fp16 pass for the scores where the library takes them (head dim 256, one block,
    # 512 <= d_l <= 2048), else three split-bf16 passes
    qk_passes = 1 if one_pass_scores(wl) else 3
    issued = (qk_passes * fl["scores"] + fl["px_passes"] * fl["px_blk"] if fused
              else 3 * fl["scores_gemm"])
    per_launch_flops = alg * L / max(n_k, 1)
    achieved = per_launch_flops / (ms_k / max(n_k, 1) / 1e3) / 1e12 if ms_k > 0 else None
    traffic = None
    for tr in TRAFFIC[kname]:
        if tr["workload"] == (name, t) and tr["kernel_hash"] == _kernel_hash(tr["files"]):
            traffic = tr["bytes_per_launch"]
    kdesc = ("ca_fused (" + ("1-pass fp16 scores with a top-k logit repair" if qk_passes == 1
                             else "3-pass split-bf16 scores")
             + " + online softmax + P X, one tcgen05 kernel"
             + ("; clusters of four CTAs: two query tiles x two O-column halves, 2-SM MMAs"
                if 2 * d == 512 else "")
             + ("; the first block's launches in split fp16 with P hi + lo)"
                if wl.get("n_blocks", 1) > 1 and wl.get("cross_every_block", 1) else ")")
             if fused else "scores (3-pass split-bf16 tcgen05 GEMM)")
    ratio = issued / alg
    roof = {"bound": "tensor", "kernel": kdesc,
            "achieved": achieved, "peak": bf16_sus, "unit": "TFLOP/s",
            "frac": achieved / bf16_sus if achieved else None, "traffic": traffic,
            "peak_source": f"{src} bf16 sustained (kernel timed inside a long step)",
            "issued_tflops": achieved * ratio if achieved else None,
            "issued_frac": achieved * ratio / bf16_sus if achieved else None,
            "flops_per_launch": per_launch_flops}
    whole = fl["total"] * L * world * args.steps / (ms / 1e3) / 1e12

    line = {
        "metric": "compacted context tokens/s per layer stack",
        "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
        "warmup": max(args.warmup, 3), "ms_per_step": ms_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": describe(name, wl, t), "layers": L, "N": N, "t": t,
                   "l2": f"inputs larger than L2 ({L} layers of K/V = "
                         f"{sum(k.numel() for k in Ks) * 4 / 1e6:.0f} MB per step)"},
        "e2e": {"value": e2e_value, "unit": "tokens/s", "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h, "steps": e2e_steps},
        "gpu_launches": launches,
        "roofline": roof,
        "whole_path_alg_tflops": whole,
        "kernel_ms_per_step": {k: v[1] / brk for k, v in prof.items()
                               if k != "load" and v[0] > 0},
        "clocks": clk,
    }
    still.still_destroy(ctx)
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cb = run_cpu_baseline(wl, t)
        cb.pop("seconds", None)
        cb.pop("scale", None)
        cb["extrapolated"] = True
        line["cpu_baseline"] = cb
    if rank == 0:
        print(json.dumps(line))
    if dist is not None:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
