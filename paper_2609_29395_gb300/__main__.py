"""Run GCPSL rounds of one of the synthetic workloads on the GPU.

    python -m paper_2609_29395_gb300 --workload resnet18_c8 --rounds 5

builds the workload's inputs, creates a context (CUDA graphs on, bf16
operands where the workload has them), runs the rounds and prints, per round,
the mean loss over the clusters and the number of library kernel launches.
This is also the small, fixed program that kernel profilers are pointed at:
`--rounds` bounds the launches.
"""
from __future__ import annotations

import argparse
import dataclasses
import time

import numpy as np

from . import Context, configs


def main() -> int:
    ap = argparse.ArgumentParser(prog="python -m paper_2609_29395_gb300")
    ap.add_argument("--workload", default="splitcnn_c4", choices=sorted(configs.WORKLOADS))
    ap.add_argument("--rounds", type=int, default=5)
    ap.add_argument("--eager", action="store_true", help="launch kernels one by one, no graphs")
    ap.add_argument("--images", type=int, default=0,
                    help="dataset size (default: the workload's); the round shapes stay")
    ap.add_argument("--clusters", type=int, default=0,
                    help="number of clusters C (default: the workload's)")
    args = ap.parse_args()
    w = configs.WORKLOADS[args.workload]
    if args.images:
        w = dataclasses.replace(w, n=args.images)
    if args.clusters:
        w = dataclasses.replace(w, num_clusters=args.clusters)
    ds, assign, params = configs.build_inputs(w)
    ctx = Context(w.arch, w.num_clients, w.num_clusters, assign, w.B, w.F, 4, ds.images,
                  ds.labels, ds.owner, params, bf16=w.bf16, **w.options())
    if args.eager:
        ctx.set_graph(False)
    t0 = time.perf_counter()
    counts = []
    for r in range(args.rounds):
        n0 = ctx.kernels_launched()
        loss, active = ctx.step(stats=True)
        counts.append(ctx.kernels_launched() - n0)
        print(f"round {r + 1}: mean loss {float(np.mean(loss)):.4f}, "
              f"active clients {int(np.sum(active))}, launches {counts[-1]}", flush=True)
    print(f"launches_first_round={counts[0] if counts else 0} "
          f"launches_last_round={counts[-1] if counts else 0} "
          f"wall_s={time.perf_counter() - t0:.2f}", flush=True)
    ctx.close()
    return 0


if __name__ == "__main__":
    raise SystemExit(main())
