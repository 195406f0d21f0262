"""Profiling driver: compacts one layer of a synthetic workload a few times.

Small enough for kernel captures (one layer's weights and workspace, a few GB; --N and --H shrink
a large workload's cache while keeping its compactor shape), e.g.

  ncu --set full --clock-control none --kernel-name-base mangled -k regex:EpiAffineELi4E \\
      -s 1 -c 1 -o prof python -m paper_2606_07878_gb300.profile_layer --workload qwen7b_8k

Exits non-zero if the device reports an error.
"""
import argparse
import os
import sys


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--workload", default="qwen7b_8k")
    ap.add_argument("--t", type=int, default=1024)
    ap.add_argument("--repeat", type=int, default=3)
    ap.add_argument("--N", type=int, default=0, help="cached tokens (default: the workload's)")
    ap.add_argument("--H", type=int, default=0, help="KV-heads (default: the workload's)")
    args = ap.parse_args()
    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import torch

    from paper_2606_07878_gb300 import still, synth

    wl = dict(synth.WORKLOADS[args.workload])
    if args.N:
        wl["N"] = args.N
    if args.H:
        wl["H"] = args.H
    t = args.t
    dev = "cuda:0"
    ctx = still.still_create(0)
    W = synth.gen_weights(wl, 0, t, dev)
    still.still_load_layer_weights(ctx, 0, still.config_from_workload(wl, t), W)
    K, V = synth.gen_kv(wl, 0, device=dev)
    Ck = torch.empty((t, wl["H"], wl["d"]), dtype=torch.bfloat16, device=dev)
    Cv = torch.empty_like(Ck)
    for _ in range(args.repeat):
        still.still_compact_layer(ctx, 0, K, V, t, Ck, Cv)
    code, det = still.still_get_device_status(ctx)
    print("device status", still.STATUS.get(code), det)
    still.still_destroy(ctx)
    return 0 if code == 0 else 1


if __name__ == "__main__":
    sys.exit(main())
