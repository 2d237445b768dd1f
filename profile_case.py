"""Small, fixed cases of one kernel each, for ncu captures.

decode (default): builds a workload's latent cache for a few layers only (same batch, context
lengths, heads and ranks, so every decode launch has exactly the shape and bytes of a launch in
the full benchmark; `--fill random` writes N(0,1) latents instead of encoding them), then runs
`--calls` pass-1 decode calls (and one encode call per layer), so that a profiler can skip the
warm-up launches and capture one to three of them:

    ncu --set full --clock-control none -k regex:decode_async_kernel -s 6 -c 1 \\
        python profile_case.py --workload ouro14_rho4 --layers 2 --calls 10

rope: the same decode calls through lla_decode_attn_rope (RoPE after reconstruction, base 10^4):

    ncu --set full --clock-control none -k regex:decode_rope_kernel -s 6 -c 1 \\
        python profile_case.py --case rope --workload ouro14_rho4 --layers 2 --calls 10

rope_prefill: the same prompts through lla_prefill_attn_rope (key rebuild, then attention):

    ncu --set full --clock-control none -k regex:"rope_rebuild_kernel|prefill_tc_kernel" -c 2 \\
        python profile_case.py --case rope_prefill --workload ouro14_rho2 \\
        --prompts 4 --len 8192 --calls 1

loops / decoupled: the same cache through lla_decode_attn_loops (all T loops of a layer per call)
or lla_decode_attn_decoupled (rotary planes of d_rope = 64 stored first, one per layer):

    ncu --set full --clock-control none -k regex:attn2d_kernel -s 2 -c 1 \\
        python profile_case.py --case decoupled --workload ouro14_rho4 --layers 2 --calls 10

2d: LLA-2D on an LLA-2D workload's shape (`--workload2d`, the stress2d workload by default) with
`--batch` sequences (random latents written into two layers' pages; --batch 32 keeps a stress2d
layer near 1 GB, above L2; the (1152, 1920) workload's 16 sequences take 351 MB a layer):

    ncu --set full --clock-control none -k regex:attn2d_kernel -s 2 -c 1 \\
        python profile_case.py --case 2d --batch 32 --calls 8
    ncu --section SpeedOfLight --section MemoryWorkloadAnalysis --clock-control none \\
        -k regex:attn2d_big_kernel -s 2 -c 1 \\
        python profile_case.py --case 2d --workload2d ouro14_2d_rho533 --batch 16 --calls 6

prefill: encodes `--prompts` prompts of `--len` tokens of a workload's ranks (tensor-core encode,
one launch per axis), then runs `--calls` causal prefill calls over them:

    ncu --set full --clock-control none -k regex:"encode_tc_kernel|prefill_tc_kernel" -c 3 \\
        python profile_case.py --case prefill --workload ouro14_rho2 \\
        --prompts 4 --len 8192 --calls 1
"""
from __future__ import annotations

import argparse
import os
import sys

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def decode_case(args):
    import torch

    from bench import DecodeBench
    from paper_2607_15456_gb300 import lla

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    bench = DecodeBench(args.workload, dev, layers=args.layers, fill=args.fill)
    w = bench.w
    if args.case == "decoupled":
        from paper_2607_15456_gb300 import workloads as W
        d_rope = 64
        plane = lla.lla_rope_plane_bytes(d_rope)
        pos = torch.cat([torch.arange(L, dtype=torch.int32) for L in bench.lens]).to(dev)
        slots = torch.cat([bench.pt.slots(b, range(L)) for b, L in enumerate(bench.lens)]).to(dev)
        pools = []
        for l in range(w.D):
            pool = torch.empty(bench.pt.num_blocks * plane, dtype=torch.uint8, device=dev)
            k = W.normal((sum(bench.lens), d_rope), w.seed, 500, l, device=dev)
            lla.lla_encode_rope_keys(d_rope, 10000.0, lla.LLA_ROPE_HALF, pool, bench.pt.num_blocks, k, pos,
                                     slots)
            pools.append(pool)
        qr = W.normal((bench.B, w.H, d_rope), w.seed, 501, device=dev)
        ckr = W.normal((bench.B, d_rope), w.seed, 502, device=dev)
        dws = torch.zeros(lla.lla_decode_decoupled_workspace_size(bench.geom, d_rope, bench.B),
                          dtype=torch.uint8, device=dev)
    if args.case == "loops":
        lws = torch.zeros(lla.lla_decode_loops_workspace_size(bench.geom, bench.B), dtype=torch.uint8,
                          device=dev)
    for i in range(args.calls):
        l, t = i % w.D, (i // w.D) % w.T
        if args.case == "decoupled":
            lla.lla_decode_attn_decoupled(bench.geom, bench.codecs[l], bench.caches[l], pools[l], d_rope,
                                          10000.0, lla.LLA_ROPE_HALF, bench.ctx, bench.max_ctx, t,
                                          bench.q[l, t], qr, bench.cur_k[l, t], bench.cur_v[l, t], ckr,
                                          bench.out[l, t], dws)
        elif args.case == "loops":
            lla.lla_decode_attn_loops(bench.geom, bench.codecs[l], bench.caches[l], bench.ctx, bench.max_ctx,
                                      bench.q[l], bench.cur_k[l], bench.cur_v[l], bench.out[l], lws)
        elif args.case == "rope":
            lla.lla_decode_attn_rope(bench.geom, bench.codecs[l], bench.caches[l], 10000.0,
                                     lla.LLA_ROPE_HALF, bench.ctx, bench.max_ctx, t, bench.q[l, t],
                                     bench.cur_k[l, t], bench.cur_v[l, t], bench.out[l, t],
                                     bench.ws)
        else:
            lla.lla_decode_attn(bench.geom, bench.codecs[l], bench.caches[l], bench.ctx,
                                bench.max_ctx, t, bench.q[l, t], bench.cur_k[l, t],
                                bench.cur_v[l, t], bench.out[l, t], bench.ws)
    bench.encode_calls()
    torch.cuda.synchronize()
    err = lla.lla_get_device_error()
    if err:
        raise SystemExit(f"device error word {err:#x}")
    print(f"profile case done: {args.workload}, {w.D} layers, {args.calls} decode calls, "
          f"{bench.decode_bytes_per_launch()} algorithmic bytes per decode launch")


def case_2d(args):
    import torch

    from paper_2607_15456_gb300 import lla
    from paper_2607_15456_gb300 import workloads as W

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    w = W.WORKLOADS[args.workload2d]
    if not w.lla2d:
        raise SystemExit(f"{args.workload2d} is not an LLA-2D workload")
    lens = W.context_lengths(w, B=args.batch)
    pt = W.page_table(lens, w.seed, extra_tokens=1)
    table = pt.block_table.to(dev)
    geom = lla.Geometry(w.T, w.H, w.d, w.r_k, w.r_v, "bf16")
    layers = []
    for l in range(2):
        ck = W.normal((sum(lens), w.r_k), w.seed, 400, l, device=dev)
        cv = W.normal((sum(lens), w.r_v), w.seed, 401, l, device=dev)
        pool = W.pack_latent_pages(ck, cv, pt.block_table, lens, pt.num_blocks)
        del ck, cv
        codec = lla.Codec(**W.codec_tensors_2d(w.T, w.H, w.d, w.r_k, w.r_v, w.seed, l, device=dev))
        layers.append((pool, codec, lla.Cache(pool, pt.num_blocks, table, pt.max_blocks)))
    shape = (len(lens), w.H, w.d)
    q, k, v = (W.normal(shape, w.seed, 402 + i, device=dev) for i in range(3))
    out = torch.empty_like(q)
    ctx = torch.tensor(lens, dtype=torch.int32, device=dev)
    ws = torch.empty(lla.lla_decode_2d_workspace_size(geom, len(lens)), dtype=torch.uint8, device=dev)
    for i in range(args.calls):
        l, t = i % 2, (i // 2) % w.T
        lla.lla_decode_attn_2d(geom, layers[l][1], layers[l][2], ctx, max(lens), t, q, k, v, out, ws)
    torch.cuda.synchronize()
    err = lla.lla_get_device_error()
    if err:
        raise SystemExit(f"device error word {err:#x}")
    nbytes = sum(lens) * (w.r_k + w.r_v) * 2 + w.H * w.d * (w.r_k + w.r_v) * 2 + 4 * len(lens) * w.H * w.d * 2
    print(f"profile case done: LLA-2D, B={len(lens)}, {args.calls} calls, {nbytes} algorithmic bytes per call")


def prefill_case(args):
    import torch

    from paper_2607_15456_gb300 import lla
    from paper_2607_15456_gb300 import workloads as W

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    w = W.WORKLOADS[args.workload]
    T, H, d = w.T, w.H, w.d
    geom = lla.Geometry(T, H, d, w.r_k, w.r_v, "bf16")
    codec = lla.Codec(**W.codec_tensors(T, H, d, w.r_k, w.r_v, w.seed, 0, device=dev))
    lens = [args.len] * args.prompts
    pt = W.page_table(lens, w.seed, extra_tokens=0)
    pool = torch.zeros(pt.num_blocks * lla.lla_cache_block_bytes(geom), dtype=torch.uint8, device=dev)
    cache = lla.Cache(pool, pt.num_blocks, pt.block_table.to(dev), pt.max_blocks)
    N = sum(lens)
    slots = torch.cat([pt.slots(b, range(L)) for b, L in enumerate(lens)]).to(dev)
    xk = W.normal((T, N, H, d), w.seed, 300, device=dev)
    xv = W.normal((T, N, H, d), w.seed, 301, device=dev)
    lla.lla_encode(geom, codec, cache, xk, xv, slots)
    del xk, xv
    q = W.normal((N, H, d), w.seed, 302, device=dev)
    out = torch.empty_like(q)
    cu = torch.tensor([i * args.len for i in range(args.prompts + 1)], dtype=torch.int32, device=dev)
    ws = None
    if args.case == "rope_prefill":
        ws = torch.empty(lla.lla_prefill_rope_workspace_size(geom, args.prompts, args.len),
                         dtype=torch.uint8, device=dev)
    for _ in range(args.calls):
        if ws is not None:
            lla.lla_prefill_attn_rope(geom, codec, cache, 10000.0, lla.LLA_ROPE_HALF, cu, args.len, 1,
                                      q, out, ws)
        else:
            lla.lla_prefill_attn(geom, codec, cache, cu, args.len, 1, q, out)
    torch.cuda.synchronize()
    err = lla.lla_get_device_error()
    if err:
        raise SystemExit(f"device error word {err:#x}")
    pairs = args.prompts * H * args.len * (args.len + 1) // 2
    print(f"profile case done: {args.workload} prefill, {args.prompts} x {args.len} tokens, "
          f"{pairs} (query, key) pairs per call, {args.calls} calls")


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--case", choices=["decode", "rope", "loops", "decoupled", "2d", "prefill", "rope_prefill"],
                    default="decode")
    ap.add_argument("--workload", default="ouro14_rho4")
    ap.add_argument("--workload2d", default="stress2d_rho2133", help="the LLA-2D workload of --case 2d")
    ap.add_argument("--layers", type=int, default=2)
    ap.add_argument("--calls", type=int, default=10)
    ap.add_argument("--prompts", type=int, default=4)
    ap.add_argument("--len", type=int, default=8192)
    ap.add_argument("--batch", type=int, default=32)
    ap.add_argument("--fill", choices=["encode", "random"], default="encode",
                    help="decode cases: latents through lla_encode, or N(0,1) bf16 written into the pages")
    args = ap.parse_args()
    if args.case in ("decode", "rope", "loops", "decoupled"):
        decode_case(args)
    elif args.case == "2d":
        case_2d(args)
    else:
        prefill_case(args)


if __name__ == "__main__":
    main()
