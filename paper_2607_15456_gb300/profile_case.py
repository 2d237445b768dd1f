"""A small, fixed case of one kernel for ncu captures.

Builds a workload's latent cache for a few layers only (same batch, context lengths, heads and
ranks, so every decode launch has exactly the shape and bytes of a launch in the full
benchmark), then runs `--calls` pass-1 decode calls (and one encode call per layer), so that a
profiler can skip the warm-up launches and capture one to three of them:

    ncu --set full --clock-control none -k regex:decode_async_kernel -s 6 -c 1 \\
        python -m paper_2607_15456_gb300.profile_case --workload ouro14_rho4 --layers 2 --calls 10
"""
from __future__ import annotations

import argparse
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--workload", default="ouro14_rho4")
    ap.add_argument("--layers", type=int, default=2)
    ap.add_argument("--calls", type=int, default=10)
    args = ap.parse_args()
    import torch

    from bench import DecodeBench
    from paper_2607_15456_gb300 import lla

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    bench = DecodeBench(args.workload, dev, layers=args.layers)
    w = bench.w
    for i in range(args.calls):
        l, t = i % w.D, (i // w.D) % w.T
        lla.lla_decode_attn(bench.geom, bench.codecs[l], bench.caches[l], bench.ctx, bench.max_ctx,
                            t, bench.q[l, t], bench.cur_k[l, t], bench.cur_v[l, t], bench.out[l, t],
                            bench.ws)
    bench.encode_calls()
    torch.cuda.synchronize()
    err = lla.lla_get_device_error()
    if err:
        raise SystemExit(f"device error word {err:#x}")
    print(f"profile case done: {args.workload}, {w.D} layers, {args.calls} decode calls, "
          f"{bench.decode_bytes_per_launch()} algorithmic bytes per decode launch")


if __name__ == "__main__":
    main()
