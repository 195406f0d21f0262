"""CPU checks of the benchmark's algorithmic-work accounting (the numerators of its roofline
fractions) against the formulas written out term by term, and of its workload descriptions."""
import math

import pytest

import bench
from paper_2606_07878_gb300 import synth


def _terms(wl, t, N, kw=None, kproj=None):
    H, d, D, n, F = wl["H"], wl["d"], wl["D"], wl["n"], wl["F"]
    kw = D if kw is None else kw
    kproj = 2 * N * H * 2 * d * n * D if kproj is None else kproj
    ca = (kproj + 2 * t * N * H * n * kw + 2 * t * N * H * n * 2 * d + 2 * t * H * n * 2 * d * D
          + 2 * t * H * n * D * D)
    sa = 6 * t * H * D * n * D + 4 * t * t * H * n * D + 2 * t * H * n * D * D
    return ca, sa


@pytest.mark.parametrize("name,t", [("qwen7b_8k", 1024), ("qwen8b_32k", 512),
                                    ("gemma_128k", 655), ("tiny_1k", 128)])
def test_one_block_flops(name, t):
    wl = synth.WORKLOADS[name]
    N, H, d, D, n, F = wl["N"], wl["H"], wl["d"], wl["D"], wl["n"], wl["F"]
    fl = bench.algorithmic_flops(wl, t, N)
    ca, sa = _terms(wl, t, N)
    assert fl["total"] == ca + sa + 4 * t * H * D * F + 4 * t * H * D * d
    assert fl["scores"] == 2 * t * N * H * n * D
    assert fl["px"] == 2 * t * N * H * n * 2 * d
    assert fl["px_passes"] == 1.5
    # every head size takes the fused kernel (2d = 512 on clusters of four CTAs)
    assert fl["scores_gemm"] == 0


def test_two_block_flops_count_both_blocks():
    wl = synth.WORKLOADS["qwen3_4b_64k"]
    t, N = 1311, wl["N"]
    fl = bench.algorithmic_flops(wl, t, N)
    ca, sa = _terms(wl, t, N)
    assert fl["total"] == 2 * ca + 2 * sa + 4 * t * wl["H"] * wl["D"] * wl["d"]
    assert fl["scores"] == 2 * (2 * t * N * wl["H"] * wl["n"] * wl["D"])
    assert fl["px_passes"] == 1.5 + 2.5  # the first block's P X runs with P hi + lo


def test_folded_workload_flops():
    wl = synth.WORKLOADS["qwen7b_8k_norope"]
    Kp = bench.folded(wl)
    assert Kp == 320 and Kp % 64 == 0 and Kp >= 2 * wl["d"] + 1
    t, N = 1024, wl["N"]
    fl = bench.algorithmic_flops(wl, t, N)
    ca, sa = _terms(wl, t, N, kw=Kp, kproj=2 * N * wl["H"] * wl["n"] * Kp * Kp)
    assert fl["total"] == ca + sa + 4 * t * wl["H"] * wl["D"] * wl["F"] + 4 * t * wl["H"] * wl["D"] * wl["d"]
    assert fl["scores"] == 2 * t * N * wl["H"] * wl["n"] * Kp
    # the RoPE workload of the same shape does not fold
    assert bench.folded(synth.WORKLOADS["qwen7b_8k"]) == 0
    assert "W_K folded" in bench.describe("qwen7b_8k_norope", wl, t)


def test_fold_conditions():
    base = dict(synth.WORKLOADS["qwen7b_8k_norope"])
    assert bench.folded(dict(base, d=64, D=256)) == 192          # 129 -> 192 < 256
    assert bench.folded(dict(base, d=128, D=256)) == 0           # 320 >= 256
    assert bench.folded(dict(base, d=256, D=2048)) == 0          # 2d = 512: no fused kernel
    assert bench.folded(dict(base, n_blocks=2)) == 0             # two blocks
    assert bench.folded(dict(base, compactor_rope=1)) == 0


def test_describe_names_the_shape():
    wl = synth.WORKLOADS["qwen3_4b_64k"]
    s = bench.describe("qwen3_4b_64k", wl, 1311)
    assert "2 blocks (CA in every block)" in s and "t=1311" in s and f"({round(65536 / 1311)}x)" in s
    assert math.isclose(65536 / 1311, 49.99, rel_tol=1e-3)


def test_traffic_records_name_existing_profiles_and_current_kernels():
    """Every DRAM-traffic record of the bench line points at a committed ncu summary and was
    taken on the kernel source as it is now (otherwise the bench would silently report null)."""
    import os
    for kname, recs in bench.TRAFFIC.items():
        for tr in recs:
            assert os.path.exists(os.path.join(bench.ROOT, tr["profile"])), tr["profile"]
            assert tr["kernel_hash"] == bench._kernel_hash(tr["files"]), (kname, tr["workload"])
            assert tr["bytes_per_launch"] > 0
    # the default workload has one
    assert any(tr["workload"] == (bench.WORKLOAD, bench.DEFAULT_T[bench.WORKLOAD])
               for tr in bench.TRAFFIC["ca_fused"])
