"""Seeded synthetic workloads for the Still compactor: shapes, K/V caches, random weights.

This module is shared input plumbing. It draws random numbers and lays them out. It holds
none of the compactor's arithmetic (no norms, attention, projections or budgets). Both the
fp64 oracle and the CUDA path consume what it produces, and neither is imported here.

Recipe (stands in for the paper's Qwen3 / Gemma-3 caches on MCQ, RULER and similar; those
models and datasets are not available; the paper trains and evaluates on real caches, Sec. 2.4):
  * V ~ N(0, 1), rounded to bf16 (round-to-nearest-even).
  * K: raw N(0, 1); a seeded choice of `heavy` channels per (layer, KV-head) is scaled x8
    (outlier key channels); then the base model's RoPE (half-split pairs, base theta) is
    applied at the cache positions, with angles in fp64, as the frozen model would have done
    before caching the keys (Sec. 2.2); then bf16.
  * Weights: every tensor, biases and latent banks included, N(0, 0.02) then bf16, from a
    counter-derived seed per (seed, layer, tensor id).
"""
from __future__ import annotations

import torch

# Workloads, named by what they are.  L layers, N cached tokens, H KV-heads, d head dim,
# D compactor width (d_l), n heads (n_c = n_s, each D wide), F FFN hidden (0 = off),
# ts compact lengths, theta base-model RoPE base, heavy = outlier key channels.
WORKLOADS = {
    "tiny_1k": dict(L=1, N=1024, H=2, d=64, D=256, n=4, F=1024, ts=(128,), theta=1e4, heavy=4),
    "qwen7b_8k": dict(L=28, N=8192, H=4, d=128, D=1024, n=8, F=4096, ts=(1024, 256),
                      theta=1e6, heavy=4),
    "qwen8b_32k": dict(L=36, N=32768, H=8, d=128, D=1024, n=8, F=4096, ts=(2048, 512, 164),
                       theta=1e6, heavy=1),
    "gemma_128k": dict(L=48, N=131072, H=8, d=256, D=2048, n=16, F=8192, ts=(16384, 655),
                       theta=1e6, heavy=3),
    # The paper's canonical compactor on Qwen3-4B-shaped caches (36 layers, 8 KV-heads, d 128):
    # d_l = 256, two blocks with cross-attention in both, one head, no FFN; 64k context at the
    # 50x ratio (t = 1311).
    "qwen3_4b_64k": dict(L=36, N=65536, H=8, d=128, D=256, n=1, F=0, ts=(1311,), theta=1e6,
                         heavy=1, n_blocks=2, cross_every_block=1),
    # The compactor-RoPE-free ablation (App. M) of the qwen7b_8k shape: the key projection
    # folds into the queries.
    "qwen7b_8k_norope": dict(L=28, N=8192, H=4, d=128, D=1024, n=8, F=4096, ts=(1024, 256),
                             theta=1e6, heavy=4, compactor_rope=0),
    # Iterative ragged serving: 8 sequences, lengths uniform in [8k, 32k] from seed 7, then
    # 16 rounds of +8192 tokens each, re-compacted to the 32x budget.
    "iterative_ragged": dict(L=36, H=8, d=128, D=1024, n=8, F=4096, theta=1e6, heavy=1,
                             n_seq=8, ratio=32, rounds=16, chunk=8192, len_seed=7,
                             len_lo=8192, len_hi=32768),
}

WEIGHT_STD = 0.02
HEAVY_SCALE = 8.0

# Tensor ids for the seed counter (stable; never renumber).
_TENSOR_IDS = {
    "Z": 1, "Wq": 2, "bq": 3, "Wk": 4, "bk": 5, "Wv": 6, "Wo": 7,
    "Sq": 8, "sbq": 9, "Sk": 10, "sbk": 11, "Sv": 12, "So": 13,
    "W1": 14, "W2": 15, "Wkey": 16, "Wval": 17,
    "K": 40, "V": 41, "heavy": 42,
}


def _mix(*xs: int) -> int:
    """splitmix64 over a tuple of integers -> a 63-bit seed."""
    z = 0x9E3779B97F4A7C15
    for x in xs:
        z = (z + (int(x) & 0xFFFFFFFFFFFFFFFF) + 0x9E3779B97F4A7C15) & 0xFFFFFFFFFFFFFFFF
        z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & 0xFFFFFFFFFFFFFFFF
        z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & 0xFFFFFFFFFFFFFFFF
        z ^= z >> 31
    return z & 0x7FFFFFFFFFFFFFFF


def _gen(device, *key) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(_mix(*key))
    return g


def weight_shapes(H, d, D, n, F, t_max, n_blocks=1, cross_every_block=True):
    """Shapes of one layer's weights in the library's layout (x @ W convention).

    Head i of a multi-head projection is the column block [i*D, (i+1)*D) of the [in, n*D]
    matrix; the output projections are [n*D, D] with head i in row block i.  Per block b
    the names carry a suffix (b = 0 has none); without cross_every_block only block 0 has
    cross-attention weights.
    """
    shapes = {"Z": (H, t_max, D)}
    for b in range(n_blocks):
        s = "" if b == 0 else f"@{b}"
        if b == 0 or cross_every_block:
            shapes.update({
                "Wq" + s: (D, n * D), "bq" + s: (n * D,), "Wk" + s: (2 * d, n * D),
                "bk" + s: (n * D,), "Wv" + s: (2 * d, n * D), "Wo" + s: (n * D, D)})
        shapes.update({
            "Sq" + s: (D, n * D), "sbq" + s: (n * D,), "Sk" + s: (D, n * D),
            "sbk" + s: (n * D,), "Sv" + s: (D, n * D), "So" + s: (n * D, D),
        })
        if F:
            shapes.update({"W1" + s: (D, F), "W2" + s: (F, D)})
    shapes.update({"Wkey": (D, d), "Wval": (D, d)})
    return shapes


def gen_weights(wl: dict, layer: int, t_max: int, device="cpu", seed: int = 0, n_blocks=None,
                cross_every_block=None):
    """Random-init weights for one layer: N(0, 0.02) rounded to bf16, layout of weight_shapes.
    The block structure defaults to the workload's (n_blocks, cross_every_block; 1 and True)."""
    if n_blocks is None:
        n_blocks = wl.get("n_blocks", 1)
    if cross_every_block is None:
        cross_every_block = bool(wl.get("cross_every_block", 1))
    out = {}
    for name, shape in weight_shapes(wl["H"], wl["d"], wl["D"], wl["n"], wl["F"], t_max,
                                     n_blocks, cross_every_block).items():
        base, _, blk = name.partition("@")
        g = _gen(device, seed, layer, _TENSOR_IDS[base], int(blk or 0))
        x = torch.randn(shape, generator=g, device=device, dtype=torch.float32)
        out[name] = (x * WEIGHT_STD).to(torch.bfloat16)
    return out


def heavy_channels(wl: dict, layer: int, head: int, seed: int = 1):
    """Indices of the outlier key channels of (layer, KV-head): a seeded permutation prefix."""
    g = _gen("cpu", seed, layer, _TENSOR_IDS["heavy"], head)
    return torch.randperm(wl["d"], generator=g)[: wl["heavy"]]


def positions_from_segments(segments, device="cpu"):
    """Cache positions from (start, step, count) segments, in fp64."""
    parts = [s + st * torch.arange(c, dtype=torch.float64, device=device) for s, st, c in segments]
    return torch.cat(parts) if parts else torch.zeros(0, dtype=torch.float64, device=device)


def gen_kv(wl: dict, layer: int, N: int | None = None, device="cpu", seed: int = 1,
           positions=None, stream: int = 0):
    """Synthetic cached K, V [N, H, d] bf16 for one layer.

    `positions` (fp64, length N) are where the base model would have rotated the keys;
    default 0..N-1.  `stream` separates independent draws (ragged sequences, rounds).
    """
    N = wl["N"] if N is None else N
    H, d = wl["H"], wl["d"]
    if positions is None:
        positions = torch.arange(N, dtype=torch.float64, device=device)
    positions = positions.to(device=device, dtype=torch.float64)
    gk = _gen(device, seed, layer, _TENSOR_IDS["K"], stream)
    gv = _gen(device, seed, layer, _TENSOR_IDS["V"], stream)
    k = torch.randn((N, H, d), generator=gk, device=device, dtype=torch.float32)
    v = torch.randn((N, H, d), generator=gv, device=device, dtype=torch.float32)
    for h in range(H):
        idx = heavy_channels(wl, layer, h, seed).to(device)
        k[:, h, idx] *= HEAVY_SCALE
    # The frozen base model caches rotated keys: rotate pair (m, m + d/2) by pos * theta^(-2m/d).
    half = d // 2
    inv = torch.tensor([wl["theta"] ** (-2.0 * m / d) for m in range(half)],
                       dtype=torch.float64, device=device)
    ang = positions[:, None] * inv[None, :]
    c, s = torch.cos(ang)[:, None, :], torch.sin(ang)[:, None, :]
    a, b = k[..., :half].double(), k[..., half:].double()
    k = torch.cat([a * c - b * s, a * s + b * c], dim=-1)
    return k.to(torch.bfloat16), v.to(torch.bfloat16)


def iterative_lengths(wl: dict):
    """Initial lengths of the ragged sequences: uniform integers in [len_lo, len_hi], seed 7."""
    import numpy as np
    rng = np.random.default_rng(wl["len_seed"])
    return [int(x) for x in rng.integers(wl["len_lo"], wl["len_hi"] + 1, size=wl["n_seq"])]


def tiny_workload(**over):
    """A small workload for CPU and oracle tests (several tiles and a ragged tail on the GPU)."""
    wl = dict(L=1, N=200, H=2, d=64, D=256, n=2, F=512, ts=(40,), theta=1e4, heavy=4)
    wl.update(over)
    return wl


def bf16_to_f64(x: torch.Tensor):
    """Exact widening of a bf16 tensor to a float64 numpy array."""
    return x.to(torch.float64).cpu().numpy()


__all__ = ["WORKLOADS", "weight_shapes", "gen_weights", "gen_kv", "heavy_channels",
           "positions_from_segments", "iterative_lengths", "tiny_workload", "bf16_to_f64"]
