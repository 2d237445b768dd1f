#!/usr/bin/env python
"""Benchmark of the LLA decode hot path on GB300.

One step = one decode step of the Ouro-shaped workload: pass 1 of the cached reconstruction
decoder over every (loop, layer) call (T*D calls of lla_decode_attn, the current token attending
with its exact loop-t K/V), then lla_encode of the B completed tokens in every layer (D calls).
Inputs (latent cache, codec, queries, current K/V) are resident in HBM when the timed region
starts; the latent cache (9.7 GB for ouro14_rho4) is far larger than L2, so no flush is needed.

Prints one JSON line (rank 0).  `value` is tokens/s over all ranks (each rank decodes its own
batch: weak scaling, no collective on the data path).  `roofline` is for the decode kernel:
algorithmic bytes per launch over its average launch time, measured with CUDA events around the
decode calls of every timed step.  `e2e` repeats the step through the C ABI with the step's
inputs copied from pinned host memory and the outputs copied back inside the timed region.
`cpu_baseline` (and `--impl reference`) time the CPU float64 oracle on a bounded sample.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

ROPE_BASE = 10000.0
METRIC = "LLA decode-attn tokens/s, Ouro-1.4B shape, rho=4; HBM GB/s as % of peak"
FALLBACK_HBM_GBS = 6800.0
NOMINAL_HBM_GBS = 8000.0


def parse_args():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=100)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    p.add_argument("--workload", default="ouro14_rho4")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--cpu-seconds", type=float, default=12.0,
                   help="target CPU time of the oracle sample")
    p.add_argument("--no-extras", action="store_true",
                   help="skip the prefill, prefill-size encode and comparator measurements")
    p.add_argument("--no-workloads", action="store_true",
                   help="skip the other workloads' decode rows, the rho = 2 workload as written and "
                        "the long prompt")
    return p.parse_args()


# ------------------------------------------------------------------------------------ helpers

def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def decode_source_hash() -> str:
    h = hashlib.sha256()
    for rel in ("paper_2607_15456_gb300/csrc/lla_decode.cu",
                "paper_2607_15456_gb300/csrc/lla_decode_async.cuh",
                "paper_2607_15456_gb300/csrc/lla_decode_common.cuh",
                "paper_2607_15456_gb300/csrc/lla_device.cuh"):
        with open(os.path.join(ROOT, rel), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def ncu_traffic(workload: str):
    """DRAM bytes per decode launch from the committed ncu summary, if it was taken on the
    current kernel source and on this workload (else None)."""
    path = os.path.join(ROOT, "profiles", "decode_traffic.json")
    try:
        with open(path) as f:
            d = json.load(f)
        ent = d.get(workload)
        if ent and ent.get("kernel_src_sha") == decode_source_hash():
            return float(ent["dram_bytes_per_launch"])
    except Exception:
        pass
    return None


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled while the timed region runs."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.rows = []
        self.proc = None
        self.t0 = self.t1 = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()
        time.sleep(0.3)

    def _read(self):
        for line in self.proc.stdout:
            self.rows.append((time.time(), line.strip()))

    def mark(self, begin: bool):
        if begin:
            self.t0 = time.time()
        else:
            self.t1 = time.time()

    def stop(self):
        if self.proc is None:
            return {"samples": 0, "note": "nvidia-smi unavailable"}
        time.sleep(0.1)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.thread.join(timeout=2)
        inside = [r for t, r in self.rows if self.t0 is not None and self.t0 <= t <= (self.t1 or t)]
        use = inside or [r for _, r in self.rows[-3:]]
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in use:
            parts = [x.strip() for x in r.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                smax.append(float(parts[1]))
            except ValueError:
                continue
            for name, val in zip(names, parts[4:8]):
                if val.lower().startswith("active"):
                    reasons.add(name)
        out = {"sm_mhz": statistics.median(sm) if sm else None,
               "sm_max_mhz": max(smax) if smax else None,
               "reasons": sorted(reasons), "samples": len(sm),
               "samples_inside_timed_region": len(inside)}
        return out


# ------------------------------------------------------------------------------- our arm

class DecodeBench:
    """One workload's model: D layers of codecs and paged latent caches, and the decode step's
    inputs.  fill="encode" writes every cached token through lla_encode from N(0,1) stacked loop
    vectors; fill="random" writes N(0,1) bf16 latents straight into the pages (the decode reads
    the same bytes either way; used where encoding millions of tokens per layer would only add
    set-up time).  extra_tokens reserves room for the tokens later steps append."""

    def __init__(self, wname: str, device, layers=None, fill="encode", extra_tokens=1):
        import torch
        from paper_2607_15456_gb300 import lla
        from paper_2607_15456_gb300 import workloads as W

        self.torch, self.lla, self.W = torch, lla, W
        w = W.WORKLOADS[wname]
        if layers is not None:  # a shallower model with the same per-launch shape (profiling)
            from dataclasses import replace
            w = replace(w, D=layers)
        self.w = w
        self.device = device
        self.fill = fill
        self.geom = lla.Geometry(w.T, w.H, w.d, w.r_k, w.r_v, w.storage)
        self.lens = W.context_lengths(w)
        self.B = len(self.lens)
        # one page table for all layers (the pages of the tokens still to come are allocated too)
        self.pt = W.page_table(self.lens, w.seed, extra_tokens=extra_tokens)
        self.table = self.pt.block_table.to(device)
        bb = lla.lla_cache_block_bytes(self.geom)
        self.codecs, self.caches, self.pools = [], [], []
        if fill == "encode":
            slots_all = torch.cat([self.pt.slots(b, range(L)) for b, L in enumerate(self.lens)])
            N = slots_all.numel()
        chunk = 1 << 17
        for l in range(w.D):
            cod = W.codec_tensors(w.T, w.H, w.d, w.r_k, w.r_v, w.seed, l, dtype=torch.bfloat16,
                                  device=device)
            codec = lla.Codec(**cod)
            if fill == "random":
                pool = W.random_pool(self.pt.num_blocks * bb, w.seed, 120, l, device=device)
            else:
                pool = torch.empty(self.pt.num_blocks * bb, dtype=torch.uint8, device=device)
            cache = lla.Cache(pool, self.pt.num_blocks, self.table, self.pt.max_blocks)
            if fill == "encode":
                for ci, n0 in enumerate(range(0, N, chunk)):
                    n1 = min(N, n0 + chunk)
                    xk = W.normal((w.T, n1 - n0, w.H, w.d), w.seed, 100, l, ci, device=device)
                    xv = W.normal((w.T, n1 - n0, w.H, w.d), w.seed, 101, l, ci, device=device)
                    lla.lla_encode(self.geom, codec, cache, xk, xv, slots_all[n0:n1].to(device))
                    del xk, xv
            self.codecs.append(codec)
            self.caches.append(cache)
            self.pools.append(pool)
        shape = (w.D, w.T, self.B, w.H, w.d)
        self.q = W.normal(shape, w.seed, 200, device=device)
        self.cur_k = W.normal(shape, w.seed, 201, device=device)
        self.cur_v = W.normal(shape, w.seed, 202, device=device)
        self.out = torch.empty(shape, dtype=torch.bfloat16, device=device)
        self.next_slots = torch.stack([self.pt.slots(b, [L])[0] for b, L in enumerate(self.lens)]).to(device)
        self.ctx = torch.tensor(self.lens, dtype=torch.int32, device=device)
        self.max_ctx = max(self.lens)
        self.ws = torch.zeros(lla.lla_decode_workspace_size(self.geom, self.B), dtype=torch.uint8,
                              device=device)
        torch.cuda.synchronize()
        lla.lla_clear_device_error()

    def decode_calls(self):
        w, lla = self.w, self.lla
        for t in range(w.T):
            for l in range(w.D):
                lla.lla_decode_attn(self.geom, self.codecs[l], self.caches[l], self.ctx,
                                    self.max_ctx, t, self.q[l, t], self.cur_k[l, t],
                                    self.cur_v[l, t], self.out[l, t], self.ws)

    def decode_calls_rope(self, base=ROPE_BASE):
        """The same pass-1 sweep with rotary positions applied after reconstruction (keys
        rebuilt on the tensor cores, lla_decode_attn_rope)."""
        w, lla = self.w, self.lla
        for t in range(w.T):
            for l in range(w.D):
                lla.lla_decode_attn_rope(self.geom, self.codecs[l], self.caches[l], base,
                                         lla.LLA_ROPE_HALF, self.ctx, self.max_ctx, t,
                                         self.q[l, t], self.cur_k[l, t], self.cur_v[l, t],
                                         self.out[l, t], self.ws)

    def decode_calls_loops(self, ws):
        """The same T x D pass-1 calls as D calls that each take all T loops of a layer in one
        pass over its latents (lla_decode_attn_loops)."""
        lla = self.lla
        for l in range(self.w.D):
            lla.lla_decode_attn_loops(self.geom, self.codecs[l], self.caches[l], self.ctx,
                                      self.max_ctx, self.q[l], self.cur_k[l], self.cur_v[l],
                                      self.out[l], ws)

    def encode_calls(self):
        # the completed token of every sequence, in every layer: its stacked loop-t keys and
        # values (one lla_encode_layers launch for all layers)
        D = self.w.D
        self.lla.lla_encode_layers(self.geom, self.codecs, self.caches,
                                   [self.cur_k[l] for l in range(D)],
                                   [self.cur_v[l] for l in range(D)], self.next_slots)

    def step(self):
        self.decode_calls()
        self.encode_calls()

    # algorithmic bytes of one decode launch: latents of every cached token of every head,
    # this loop's W_up^K and W_up^V, and q, k_cur, v_cur, out
    def decode_bytes_per_launch(self) -> int:
        w = self.w
        es = 2
        lat = sum(self.lens) * w.H * (w.r_k + w.r_v) * es
        wup = w.H * w.d * (w.r_k + w.r_v) * es
        io = 4 * self.B * w.H * w.d * 2
        return lat + wup + io

    def encode_bytes_per_launch(self) -> int:
        w = self.w
        return (w.H * w.T * w.d * (w.r_k + w.r_v) * 2 + 2 * w.T * self.B * w.H * w.d * 2
                + self.B * w.H * (w.r_k + w.r_v) * 2)


def latent_cache_bytes(w, lens, extra_tokens=1) -> int:
    """Bytes of the whole model's paged latent cache (D layers, every block of every sequence)."""
    blocks = sum(max(1, -(-(L + extra_tokens) // 64)) for L in lens)
    return w.D * blocks * w.H * 64 * (w.r_k + w.r_v) * 2


def config_dict(w, lens, world) -> dict:
    """The workload's description, printed identically by both arms of the benchmark."""
    return {
        "workload": w.name, "D": w.D, "H": w.H, "d_head": w.d, "T": w.T, "r_k": w.r_k,
        "r_v": w.r_v, "rho": round(w.rho, 4), "batch_per_gpu": len(lens),
        "context": list(w.lens), "sum_context": sum(lens), "block_tokens": 64,
        "storage": "bf16 latents and codec weights, fp32 accumulation",
        "step": f"{w.T}x{w.D} pass-1 lla_decode_attn calls + one lla_encode_layers call "
                f"encoding the {len(lens)} completed tokens in all {w.D} layers",
        "l2": "no flush: latent cache (%.1f GB) far larger than L2" % (latent_cache_bytes(w, lens) / 1e9),
        "parallelism": f"replicas x{world} (independent batches)",
    }


def max_over_ranks(values, world, device):
    """Each value's maximum over the ranks (the slowest rank sets the whole job's time); with
    one rank, the values themselves."""
    if world <= 1:
        return [float(v) for v in values]
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(v) for v in values], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(v) for v in t.tolist()]


def job_tokens_per_s(world, batch_per_rank, ms_per_step):
    """Whole-job throughput: every rank decodes its own batch of `batch_per_rank` sequences
    (replicas, weak scaling), one token each per step."""
    return world * batch_per_rank / (ms_per_step / 1e3)


def run_ours(args, rank, world, local_rank):
    import torch
    import torch.distributed as dist

    device = torch.device("cuda", local_rank)
    torch.cuda.set_device(device)
    from __graft_entry__ import build
    if rank == 0:
        build()
    if world > 1:
        dist.barrier()
    build()
    bench = DecodeBench(args.workload, device)
    w = bench.w
    lla = bench.lla
    stream = torch.cuda.current_stream()

    for _ in range(args.warmup):
        bench.step()
    torch.cuda.synchronize()
    if lla.lla_get_device_error() != 0:
        raise RuntimeError("device error during warm-up")

    K = args.steps
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(K)]
    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    sampler = ClockSampler(device.index if device.index is not None else 0)
    sampler.start()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    sampler.mark(True)
    t_start.record(stream)
    for k in range(K):
        ev[k][0].record(stream)
        bench.decode_calls()
        ev[k][1].record(stream)
        bench.encode_calls()
    t_end.record(stream)
    torch.cuda.synchronize()
    sampler.mark(False)
    if world > 1:
        dist.barrier()
    clocks = sampler.stop()
    total_ms = t_start.elapsed_time(t_end)
    dec_ms = sum(a.elapsed_time(b) for a, b in ev)
    total_ms, dec_ms = max_over_ranks([total_ms, dec_ms], world, device)
    err = lla.lla_get_device_error()
    if err != 0:
        raise RuntimeError(f"device error word {err:#x} after the timed region")

    ms_per_step = total_ms / K
    value = job_tokens_per_s(world, bench.B, ms_per_step)
    launches_dec = w.D * w.T
    dec_launch_s = dec_ms / 1e3 / (K * launches_dec)
    bytes_launch = bench.decode_bytes_per_launch()
    achieved = bytes_launch / dec_launch_s / 1e9
    peak, peak_kind = measured_peaks()
    step_bytes = launches_dec * bytes_launch + w.D * bench.encode_bytes_per_launch()

    result = {
        "metric": METRIC,
        "value": value,
        "unit": "tokens/s",
        "n_gpus": world,
        "steps": K,
        "warmup": args.warmup,
        "ms_per_step": ms_per_step,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic",
        "config": config_dict(w, bench.lens, world),
        "roofline": {
            "bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
            "frac": achieved / peak, "traffic": ncu_traffic(w.name),
            "kernel": "decode_async_kernel (lla_decode_attn)",
            "peak_source": f"{peak_kind} copy bandwidth (MEASURED_PEAKS.json hbm_gbs)"
                           if peak_kind == "measured" else "fallback 6.8 TB/s",
            "frac_of_nominal_8tbs": achieved / NOMINAL_HBM_GBS,
            "bytes_per_launch": bytes_launch,
            "avg_launch_us": dec_launch_s * 1e6,
        },
        "step_hbm_gbs": step_bytes / (ms_per_step / 1e3) / 1e9,
        "gpu_launches": K * (launches_dec + 1),
        "clocks": clocks,
    }

    if not args.no_e2e:
        result["e2e"] = run_e2e(bench, args, world)
    if not args.no_cpu_baseline and rank == 0 and world == 1:
        result["cpu_baseline"] = cpu_baseline(bench.w, bench.lens, args.cpu_seconds)
    if not args.no_extras and rank == 0:
        _extra(result, "rope_decode", run_rope_extra, bench)
        _extra(result, "loops_decode", run_loops_extra, bench)
        _extra(result, "decoupled_decode", run_decoupled_extra, bench)
        del bench
        torch.cuda.empty_cache()
        _extra(result, "prefill_encode_comparator", run_extras, device)
        torch.cuda.empty_cache()
        _extra(result, "lla2d_decode", run_2d_extra, device)
        torch.cuda.empty_cache()
    if not args.no_workloads and rank == 0:
        _extra(result, "workloads", run_workload_rows, device, ("ouro14_rho2", "ouro26_rho533", "stress_rho2133"),
               5, 2, 3.0, world == 1 and not args.no_cpu_baseline)
        torch.cuda.empty_cache()
        _extra(result, "rho2_as_written", run_rho2_as_written, device)
        torch.cuda.empty_cache()
        _extra(result, "long_prompt", run_long_prompt, device, 65536, False)
        _extra(result, "long_prompt_rope", run_long_prompt, device, 65536, True)
    return result


def _extra(result, name, fn, *args):
    """Adds one group of extra rows to the JSON line.  A failure there is reported under
    "extra_errors" (and the sticky device error word cleared so that the next group is measured
    on its own) instead of losing the headline line."""
    import torch
    try:
        result.update(fn(*args))
    except Exception as e:  # reported, never hidden
        result.setdefault("extra_errors", {})[name] = f"{type(e).__name__}: {e}"[:400]
        try:
            from paper_2607_15456_gb300 import lla
            torch.cuda.synchronize()
            lla.lla_clear_device_error()
        except Exception:
            pass


def _time_ms(fn, reps=5, warm=2):
    """Best of `reps` CUDA-event timings of fn() on the current stream, after `warm` calls."""
    import torch
    for _ in range(warm):
        fn()
    torch.cuda.synchronize()
    best = float("inf")
    for _ in range(reps):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        fn()
        b.record()
        torch.cuda.synchronize()
        best = min(best, a.elapsed_time(b))
    return best


def run_rope_extra(bench):
    """The full-RoPE decode (f1: keys rebuilt on the tensor cores and rotated at their
    positions, Sec. 3 "RoPE and reconstruction") on the headline batch: the same D x T pass-1
    sweep through lla_decode_attn_rope, against the HBM roofline of the same algorithmic bytes
    as the absorbed decode, with the key rebuild's tensor work beside it."""
    w, lla = bench.w, bench.lla
    peak, _ = measured_peaks()
    ms = _time_ms(bench.decode_calls_rope, reps=3, warm=1)
    launches = w.D * w.T
    per_launch_s = ms / 1e3 / launches
    nbytes = bench.decode_bytes_per_launch()
    rebuild_flops = 2.0 * sum(bench.lens) * w.H * w.d * w.r_k
    if lla.lla_get_device_error() != 0:
        raise RuntimeError("device error in the RoPE decode measurement")
    return {"rope_decode": {
        "workload": f"{w.name} batch, RoPE after reconstruction (base {ROPE_BASE:g}, rotate-half "
                    f"pairs), {w.D}x{w.T} pass-1 calls",
        "kernel": f"rope_tc_kernel<{w.r_k}, {w.r_v}> + rope_finish_kernel (lla_decode_attn_rope)", "bound": "hbm",
        "ms_per_sweep": ms, "avg_launch_us": per_launch_s * 1e6,
        "GB_s": nbytes / per_launch_s / 1e9, "hbm_frac": nbytes / per_launch_s / 1e9 / peak,
        "bytes_per_launch": nbytes, "key_rebuild_TFLOP_s": rebuild_flops / per_launch_s / 1e12,
        "tokens_per_s_decode_only": bench.B / (ms / 1e3)}}


def run_loops_extra(bench):
    """Multi-query decode against the shared latent (the next row after full RoPE): the step's
    T x D pass-1 calls as D calls of lla_decode_attn_loops, each reading a layer's latents once
    for all T loops.  Reported beside the headline, never as it: the paper's loops run one after
    the other, so this is the regime of loops computed together."""
    import torch
    w, lla = bench.w, bench.lla
    peak, _ = measured_peaks()
    ws = torch.zeros(lla.lla_decode_loops_workspace_size(bench.geom, bench.B), dtype=torch.uint8,
                     device=bench.device)
    ms = _time_ms(lambda: bench.decode_calls_loops(ws), reps=3, warm=1)
    per_launch_s = ms / 1e3 / w.D
    lat = sum(bench.lens) * w.H * (w.r_k + w.r_v) * 2
    nbytes = lat + w.T * (w.H * w.d * (w.r_k + w.r_v) * 2 + 4 * bench.B * w.H * w.d * 2)
    if lla.lla_get_device_error() != 0:
        raise RuntimeError("device error in the multi-loop decode measurement")
    return {"loops_decode": {
        "workload": f"{w.name} batch, all {w.T} loops of a layer per call (shared latent), "
                    f"{w.D} calls per step",
        "kernel": f"absorb2d_kernel + attn2d_kernel<{w.r_k}, {w.r_v}, 4> + finish2d_kernel (lla_decode_attn_loops)",
        "bound": "hbm",
        "ms_per_sweep": ms, "avg_launch_us": per_launch_s * 1e6,
        "GB_s": nbytes / per_launch_s / 1e9, "hbm_frac": nbytes / per_launch_s / 1e9 / peak,
        "bytes_per_launch": nbytes, "tokens_per_s_decode_only": bench.B / (ms / 1e3),
        "note": "the layer's latents cross HBM once for its T loop calls"}}


def run_decoupled_extra(bench, d_rope=64):
    """Per-head LLA with the decoupled rotary branch (App. J "Absorbed attention"; d_rope = 64 as
    in Table decoupled_char) on the headline batch: one rotary key per token and layer stored
    turned at its position, then the step's D x T pass-1 calls through lla_decode_attn_decoupled.
    Algorithmic bytes: the latents, the rotary planes once, this loop's W_up,t and the inputs and
    outputs."""
    import torch
    w, lla, W = bench.w, bench.lla, bench.W
    peak, _ = measured_peaks()
    plane = lla.lla_rope_plane_bytes(d_rope)
    Nt = sum(bench.lens)
    pos = torch.cat([torch.arange(L, dtype=torch.int32) for L in bench.lens]).to(bench.device)
    slots = torch.cat([bench.pt.slots(b, range(L)) for b, L in enumerate(bench.lens)]).to(bench.device)
    pools = []
    for l in range(w.D):
        pool = torch.empty(bench.pt.num_blocks * plane, dtype=torch.uint8, device=bench.device)
        k = W.normal((Nt, d_rope), w.seed, 500, l, device=bench.device)
        lla.lla_encode_rope_keys(d_rope, ROPE_BASE, lla.LLA_ROPE_HALF, pool, bench.pt.num_blocks, k, pos, slots)
        pools.append(pool)
        del k
    qr = W.normal((w.D, w.T, bench.B, w.H, d_rope), w.seed, 501, device=bench.device)
    ckr = W.normal((w.D, w.T, bench.B, d_rope), w.seed, 502, device=bench.device)
    ws = torch.zeros(lla.lla_decode_decoupled_workspace_size(bench.geom, d_rope, bench.B), dtype=torch.uint8,
                     device=bench.device)

    def sweep():
        for t in range(w.T):
            for l in range(w.D):
                lla.lla_decode_attn_decoupled(bench.geom, bench.codecs[l], bench.caches[l], pools[l], d_rope,
                                              ROPE_BASE, lla.LLA_ROPE_HALF, bench.ctx, bench.max_ctx, t,
                                              bench.q[l, t], qr[l, t], bench.cur_k[l, t], bench.cur_v[l, t],
                                              ckr[l, t], bench.out[l, t], ws)
    ms = _time_ms(sweep, reps=3, warm=1)
    per_launch_s = ms / 1e3 / (w.D * w.T)
    nbytes = (bench.decode_bytes_per_launch() + Nt * d_rope * 2
              + bench.B * w.H * d_rope * 2 + bench.B * d_rope * 2)
    if lla.lla_get_device_error() != 0:
        raise RuntimeError("device error in the decoupled decode measurement")
    return {"decoupled_decode": {
        "workload": f"{w.name} batch, decoupled rotary branch d_rope={d_rope} (base {ROPE_BASE:g}), "
                    f"{w.D}x{w.T} pass-1 calls",
        "kernel": f"decode_async_kernel<2, 96, 160, 128, {d_rope}> (lla_decode_attn_decoupled)",
        "bound": "hbm", "ms_per_sweep": ms, "avg_call_us": per_launch_s * 1e6,
        "GB_s": nbytes / per_launch_s / 1e9, "hbm_frac": nbytes / per_launch_s / 1e9 / peak,
        "bytes_per_call": nbytes, "tokens_per_s_decode_only": bench.B / (ms / 1e3)}}


def run_2d_extra(device):
    """LLA-2D decode (Sec. 3, "The LLA-2D variant (loop x head)": one latent per (token, layer)
    for all heads, read by the H absorbed queries of each sequence on the tensor cores) on the
    stress workload's batch and contexts at the same cache budget, (r_k, r_v) = (288, 480),
    rho_2D = 21.33: two layers' caches of random bf16 latents, cycled through 2 x T pass-1 calls
    (every call has the shape and bytes of a call of the 48-layer model), the same 2D shape on
    the headline batch of 16 sequences, and (1152, 1920), rho_2D = 5.33, on the headline batch."""
    import torch
    from paper_2607_15456_gb300 import lla
    from paper_2607_15456_gb300 import workloads as W
    peak, _ = measured_peaks()
    out = {}
    for name, wname, B in (("lla2d_decode", "stress2d_rho2133", None),
                           ("lla2d_decode_b16", "stress2d_rho2133", 16),
                           ("lla2d_decode_rho533", "ouro14_2d_rho533", None)):
        w = W.WORKLOADS[wname]
        if B is not None:  # the headline batch's contexts with the 2D shape
            lens = W.context_lengths(W.WORKLOADS["ouro14_rho4"])
        else:
            lens = W.context_lengths(w)
        B = len(lens)
        geom = lla.Geometry(w.T, w.H, w.d, w.r_k, w.r_v, "bf16")
        pt = W.page_table(lens, w.seed, extra_tokens=1)
        table = pt.block_table.to(device)
        Nt = sum(lens)
        layers = []
        for l in range(2):
            ck = W.normal((Nt, w.r_k), w.seed, 400, l, device=device)
            cv = W.normal((Nt, w.r_v), w.seed, 401, l, device=device)
            pool = W.pack_latent_pages(ck, cv, pt.block_table, lens, pt.num_blocks)
            del ck, cv
            codec = lla.Codec(**W.codec_tensors_2d(w.T, w.H, w.d, w.r_k, w.r_v, w.seed, l,
                                                   device=device))
            layers.append((pool, codec, lla.Cache(pool, pt.num_blocks, table, pt.max_blocks)))
        shape = (2, w.T, B, w.H, w.d)
        q = W.normal(shape, w.seed, 402, device=device)
        ck = W.normal(shape, w.seed, 403, device=device)
        cv = W.normal(shape, w.seed, 404, device=device)
        o = torch.empty_like(q)
        ctx = torch.tensor(lens, dtype=torch.int32, device=device)
        ws = torch.empty(lla.lla_decode_2d_workspace_size(geom, B), dtype=torch.uint8, device=device)

        def sweep():
            for t in range(w.T):
                for l in range(2):
                    lla.lla_decode_attn_2d(geom, layers[l][1], layers[l][2], ctx, max(lens), t,
                                           q[l, t], ck[l, t], cv[l, t], o[l, t], ws)
        ms = _time_ms(sweep, reps=5, warm=2)
        per_launch_s = ms / 1e3 / (2 * w.T)
        nbytes = Nt * (w.r_k + w.r_v) * 2 + w.H * w.d * (w.r_k + w.r_v) * 2 + 4 * B * w.H * w.d * 2
        if lla.lla_get_device_error() != 0:
            raise RuntimeError("device error in the LLA-2D decode measurement")
        out[name] = {
            "workload": f"LLA-2D, H={w.H}, (r_k, r_v)=({w.r_k}, {w.r_v}), rho_2D={w.rho:.2f}, "
                        f"B={B}, sum context {Nt}; 2 layers x {w.T} pass-1 calls",
            "kernel": ("absorb2d_kernel + " + ("attn2d_big_kernel" if w.r_k > 512 else "attn2d_kernel")
                       + " + finish2d_kernel (lla_decode_attn_2d)"),
            "bound": "hbm", "avg_call_us": per_launch_s * 1e6,
            "GB_s": nbytes / per_launch_s / 1e9, "hbm_frac": nbytes / per_launch_s / 1e9 / peak,
            "bytes_per_call": nbytes,
            "tokens_per_s_decode_only": B / (per_launch_s * w.D * w.T)}
        del layers, q, ck, cv, o, ws
        torch.cuda.empty_cache()
    return out


def run_extras(device):
    """The other rows of the hot path on their own workloads, each against its roofline:
    causal prefill attention and the encode of a prefilled prompt (Ouro-1.4B at rho = 2,
    4 prompts of 8192 tokens, one layer and loop per call), the same prompts' prefill at the
    headline workload's ranks (rho = 4), and the uncompressed loop-t decode comparator on the
    headline batch (D x T calls over plain K/V pages of d = 128)."""
    import torch
    from paper_2607_15456_gb300 import lla
    from paper_2607_15456_gb300 import workloads as W

    peaks = {}
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            peaks = json.load(f)
    except Exception:
        pass
    tc_peak = float(peaks.get("bf16_tflops_sustained", 1700.0))
    hbm = float(peaks.get("hbm_gbs", FALLBACK_HBM_GBS))
    out = {}

    # prefill: ouro14_rho2, 4 x 8192 tokens
    w = W.WORKLOADS["ouro14_rho2"]
    nseq, L = w.prefill
    T, H, d = w.T, w.H, w.d
    geom = lla.Geometry(T, H, d, w.r_k, w.r_v, "bf16")
    codec = lla.Codec(**W.codec_tensors(T, H, d, w.r_k, w.r_v, w.seed, 0, device=device))
    lens = [L] * nseq
    pt = W.page_table(lens, w.seed, extra_tokens=0)
    pool = torch.zeros(pt.num_blocks * lla.lla_cache_block_bytes(geom), dtype=torch.uint8, device=device)
    cache = lla.Cache(pool, pt.num_blocks, pt.block_table.to(device), pt.max_blocks)
    N = nseq * L
    slots = torch.cat([pt.slots(b, range(L)) for b in range(nseq)]).to(device)
    xk = W.normal((T, N, H, d), w.seed, 300, device=device)
    xv = W.normal((T, N, H, d), w.seed, 301, device=device)
    enc_ms = _time_ms(lambda: lla.lla_encode(geom, codec, cache, xk, xv, slots), reps=3, warm=1)
    enc_bytes = 2 * xk.numel() * 2 + H * T * d * (w.r_k + w.r_v) * 2 + N * H * (w.r_k + w.r_v) * 2
    enc_flops = 2.0 * N * H * T * d * (w.r_k + w.r_v)
    out["encode_prefill"] = {
        "workload": f"{w.name} prompt encode, {nseq}x{L} tokens, H={H}, (r_k, r_v)=({w.r_k}, {w.r_v})",
        "kernel": "encode_kernel (lla_encode)", "ms_per_call": enc_ms,
        "GB_s": enc_bytes / (enc_ms / 1e3) / 1e9, "hbm_frac": enc_bytes / (enc_ms / 1e3) / 1e9 / hbm,
        "TFLOP_s": enc_flops / (enc_ms / 1e3) / 1e12,
        "tensor_frac": enc_flops / (enc_ms / 1e3) / 1e12 / tc_peak,
        "bytes_per_call": enc_bytes, "flops_per_call": enc_flops}
    del xk, xv
    q = W.normal((N, H, d), w.seed, 302, device=device)
    o = torch.empty_like(q)
    cu = torch.tensor([i * L for i in range(nseq + 1)], dtype=torch.int32, device=device)
    pf_ms = _time_ms(lambda: lla.lla_prefill_attn(geom, codec, cache, cu, L, 1, q, o))
    pairs = nseq * H * L * (L + 1) / 2
    pf_flops = pairs * 2 * (w.r_k + w.r_v) + N * H * 2 * d * (w.r_k + w.r_v)
    out["prefill"] = {
        "workload": f"{w.name} causal prefill, {nseq}x{L} tokens, H={H}, one layer and loop",
        "kernel": "prefill_tc_kernel (lla_prefill_attn)", "bound": "tensor",
        "ms_per_call": pf_ms, "tokens_per_s": N / (pf_ms / 1e3),
        "TFLOP_s": pf_flops / (pf_ms / 1e3) / 1e12, "peak_TFLOP_s": tc_peak,
        "frac": pf_flops / (pf_ms / 1e3) / 1e12 / tc_peak,
        "peak_source": "measured sustained cuBLAS bf16 (MEASURED_PEAKS.json bf16_tflops_sustained)",
        "flops_per_call": pf_flops}
    # the same prompts with rotary positions after reconstruction: keys rebuilt and rotated
    # (tcgen05), then the causal attention over them (Sec. 3 "RoPE and reconstruction")
    ws = torch.empty(lla.lla_prefill_rope_workspace_size(geom, nseq, L), dtype=torch.uint8, device=device)
    rp_ms = _time_ms(lambda: lla.lla_prefill_attn_rope(geom, codec, cache, ROPE_BASE, lla.LLA_ROPE_HALF,
                                                       cu, L, 1, q, o, ws))
    rp_flops = (pairs * 2 * (d + w.r_v) + N * H * 2 * d * w.r_k + N * H * 2 * d * w.r_v)
    out["rope_prefill"] = {
        "workload": f"{w.name} causal prefill with RoPE after reconstruction (base {ROPE_BASE:g}), "
                    f"{nseq}x{L} tokens, H={H}, one layer and loop",
        "kernel": "rope_rebuild_kernel + prefill_tc_kernel<ROPE> (lla_prefill_attn_rope)",
        "bound": "tensor", "ms_per_call": rp_ms, "tokens_per_s": N / (rp_ms / 1e3),
        "TFLOP_s": rp_flops / (rp_ms / 1e3) / 1e12, "peak_TFLOP_s": tc_peak,
        "frac": rp_flops / (rp_ms / 1e3) / 1e12 / tc_peak, "flops_per_call": rp_flops,
        "note": "flops: 2 (d + r_v) per causal (query, key) pair, the key rebuild 2 d r_k and the "
                "output projection 2 d r_v per (token, head)"}
    del pool, cache, ws
    # the same prompts at the headline workload's ranks (rho = 4, (96, 160)): encoded, then the
    # causal prefill over them
    w4 = W.WORKLOADS["ouro14_rho4"]
    geom4 = lla.Geometry(T, H, d, w4.r_k, w4.r_v, "bf16")
    codec4 = lla.Codec(**W.codec_tensors(T, H, d, w4.r_k, w4.r_v, w4.seed, 0, device=device))
    pool = torch.zeros(pt.num_blocks * lla.lla_cache_block_bytes(geom4), dtype=torch.uint8, device=device)
    cache = lla.Cache(pool, pt.num_blocks, pt.block_table.to(device), pt.max_blocks)
    xk = W.normal((T, N, H, d), w4.seed, 300, device=device)
    xv = W.normal((T, N, H, d), w4.seed, 301, device=device)
    lla.lla_encode(geom4, codec4, cache, xk, xv, slots)
    del xk, xv
    p4_ms = _time_ms(lambda: lla.lla_prefill_attn(geom4, codec4, cache, cu, L, 1, q, o))
    p4_flops = pairs * 2 * (w4.r_k + w4.r_v) + N * H * 2 * d * (w4.r_k + w4.r_v)
    out["prefill_rho4"] = {
        "workload": f"{nseq}x{L}-token prompts at {w4.name}'s ranks (r_k, r_v)=({w4.r_k}, {w4.r_v}), "
                    f"H={H}, one layer and loop",
        "kernel": "prefill_tc_kernel (lla_prefill_attn)", "bound": "tensor",
        "ms_per_call": p4_ms, "tokens_per_s": N / (p4_ms / 1e3),
        "TFLOP_s": p4_flops / (p4_ms / 1e3) / 1e12, "peak_TFLOP_s": tc_peak,
        "frac": p4_flops / (p4_ms / 1e3) / 1e12 / tc_peak, "flops_per_call": p4_flops}
    del q, o, pool, cache

    # comparator: plain loop-t K/V of the headline batch, d = 128
    w = W.WORKLOADS["ouro14_rho4"]
    lens = W.context_lengths(w)
    B = len(lens)
    dgeom = lla.Geometry(1, w.H, w.d, w.d, w.d, "bf16")
    pt = W.page_table(lens, w.seed, extra_tokens=1)
    table = pt.block_table.to(device)
    Nt = sum(lens)
    slots = torch.cat([pt.slots(b, range(Lb)) for b, Lb in enumerate(lens)]).to(device)
    caches = []
    for t in range(w.T):  # the teacher cache holds every loop's keys and values
        pool = torch.empty(pt.num_blocks * lla.lla_cache_block_bytes(dgeom), dtype=torch.uint8, device=device)
        cache = lla.Cache(pool, pt.num_blocks, table, pt.max_blocks)
        k = W.normal((Nt, w.H, w.d), w.seed, 310, t, device=device)
        v = W.normal((Nt, w.H, w.d), w.seed, 311, t, device=device)
        lla.lla_dense_store(dgeom, cache, k, v, slots)
        caches.append((pool, cache))
        del k, v
    ctx = torch.tensor(lens, dtype=torch.int32, device=device)
    qs = W.normal((w.T, B, w.H, w.d), w.seed, 312, device=device)
    cks = W.normal((w.T, B, w.H, w.d), w.seed, 313, device=device)
    cvs = W.normal((w.T, B, w.H, w.d), w.seed, 314, device=device)
    os_ = torch.empty_like(qs)
    ws = torch.zeros(lla.lla_decode_workspace_size(dgeom, B), dtype=torch.uint8, device=device)

    def sweep():
        for _ in range(w.D):
            for t in range(w.T):
                lla.lla_dense_decode_attn(dgeom, caches[t][1], ctx, max(lens), qs[t], cks[t], cvs[t],
                                          os_[t], ws)
    cmp_ms = _time_ms(sweep, reps=3, warm=1)
    per_launch = cmp_ms / (w.D * w.T)
    cbytes = Nt * w.H * 2 * w.d * 2 + 4 * B * w.H * w.d * 2
    out["comparator"] = {
        "workload": f"{w.name} batch, uncompressed loop-t K/V (d={w.d}), {w.D}x{w.T} calls per step",
        "kernel": "decode_async_kernel<2,128,128> (lla_dense_decode_attn)",
        "tokens_per_s": B / (cmp_ms / 1e3), "ms_per_step_decode_only": cmp_ms,
        "avg_launch_us": per_launch * 1e3, "GB_s": cbytes / (per_launch / 1e3) / 1e9,
        "hbm_frac": cbytes / (per_launch / 1e3) / 1e9 / hbm, "bytes_per_launch": cbytes,
        "note": "same bytes per call as the latent cache at rho = 4 (2d = r_k + r_v); the "
                "teacher cache of the whole model is rho times the latent cache"}
    if lla.lla_get_device_error() != 0:
        raise RuntimeError("device error in the extra measurements")
    return out


def _dense_comparator(w, lens, device, reps=2):
    """The uncompressed loop-t decode (same kernel, no codec) at the workload's full batch: the T
    loop caches of one layer (N(0,1) bf16 keys and values, d = 128) resident, read by D x T
    calls per step.  A whole model's teacher cache (D x T such caches) does not fit the GPU for
    the larger workloads; every call still reads its whole cache from HBM (each is far larger
    than L2), so the per-call time is that of a resident model."""
    import torch
    from paper_2607_15456_gb300 import lla
    from paper_2607_15456_gb300 import workloads as W
    peak, _ = measured_peaks()
    B = len(lens)
    dgeom = lla.Geometry(1, w.H, w.d, w.d, w.d, "bf16")
    pt = W.page_table(lens, w.seed, extra_tokens=1)
    table = pt.block_table.to(device)
    bb = lla.lla_cache_block_bytes(dgeom)
    caches = [lla.Cache(W.random_pool(pt.num_blocks * bb, w.seed, 130, t, device=device), pt.num_blocks,
                        table, pt.max_blocks) for t in range(w.T)]
    ctx = torch.tensor(lens, dtype=torch.int32, device=device)
    qs = W.normal((w.T, B, w.H, w.d), w.seed, 131, device=device)
    out = torch.empty_like(qs)
    ws = torch.zeros(lla.lla_decode_workspace_size(dgeom, B), dtype=torch.uint8, device=device)

    def sweep():
        for _ in range(w.D):
            for t in range(w.T):
                lla.lla_dense_decode_attn(dgeom, caches[t], ctx, max(lens), qs[t], qs[t], qs[t], out[t], ws)
    ms = _time_ms(sweep, reps=reps, warm=1)
    per_launch_s = ms / 1e3 / (w.D * w.T)
    nbytes = sum(lens) * w.H * 2 * w.d * 2 + 4 * B * w.H * w.d * 2
    if lla.lla_get_device_error() != 0:
        raise RuntimeError("device error in the comparator measurement")
    whole = w.D * w.T * sum(max(1, -(-(L + 1) // 64)) for L in lens) * bb
    res = {"kernel": "decode_async_kernel<2,128,128> (lla_dense_decode_attn)",
           "ms_per_step_decode_only": ms, "tokens_per_s_decode_only": B / (ms / 1e3),
           "avg_launch_us": per_launch_s * 1e6, "GB_s": nbytes / per_launch_s / 1e9,
           "hbm_frac": nbytes / per_launch_s / 1e9 / peak, "bytes_per_launch": nbytes,
           "teacher_cache_GB": whole / 1e9,
           "note": "one layer's T loop caches resident at full batch, read D x T times per step"}
    del caches, qs, out, ws
    torch.cuda.empty_cache()
    return res


def run_workload_rows(device, names=("ouro14_rho2", "ouro26_rho533", "stress_rho2133"), steps=5,
                      warmup=2, cpu_seconds=3.0, cpu=True):
    """Decode throughput of the other Ouro-shaped workloads at full depth: D layers of latent
    caches resident (N(0,1) bf16 latents written into the pages), one step = T x D pass-1
    lla_decode_attn calls + one lla_encode_layers call, timed as the headline; beside it the
    uncompressed comparator at the same batch and the oracle on a bounded sample of the step."""
    import torch
    from paper_2607_15456_gb300 import lla
    peak, _ = measured_peaks()
    out = {}
    for name in names:
        bench = DecodeBench(name, device, fill="random")
        w = bench.w
        for _ in range(warmup):
            bench.step()
        torch.cuda.synchronize()
        stream = torch.cuda.current_stream()
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
        t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        t0.record(stream)
        for k in range(steps):
            ev[k][0].record(stream)
            bench.decode_calls()
            ev[k][1].record(stream)
            bench.encode_calls()
        t1.record(stream)
        torch.cuda.synchronize()
        if lla.lla_get_device_error() != 0:
            raise RuntimeError(f"device error in the {name} decode measurement")
        ms = t0.elapsed_time(t1) / steps
        dec_s = sum(a.elapsed_time(b) for a, b in ev) / 1e3 / (steps * w.D * w.T)
        nbytes = bench.decode_bytes_per_launch()
        rope = None
        try:  # shapes without a tensor-core key rebuild are refused before anything is enqueued
            bench.decode_calls_rope()
        except lla.LLAError as e:
            if e.status != 2:  # LLA_ERR_UNSUPPORTED
                raise
        else:
            # the same sweep with rotary positions after reconstruction (keys rebuilt on tcgen05)
            rms = _time_ms(bench.decode_calls_rope, reps=2, warm=1)
            rs = rms / 1e3 / (w.D * w.T)
            rope_k = (f"rope_tc_kernel<{w.r_k}, {w.r_v}> + rope_finish_kernel" if (w.r_k, w.r_v) != (192, 320)
                      else "decode_rope_kernel<192, 320>")
            rope = {"kernel": f"{rope_k} (lla_decode_attn_rope)", "ms_per_sweep": rms,
                    "avg_launch_us": rs * 1e6, "GB_s": nbytes / rs / 1e9, "hbm_frac": nbytes / rs / 1e9 / peak,
                    "tokens_per_s_decode_only": bench.B / (rms / 1e3)}
            if lla.lla_get_device_error() != 0:
                raise RuntimeError(f"device error in the {name} RoPE decode measurement")
        loops = None
        lws = torch.zeros(1, dtype=torch.uint8, device=device)
        try:  # the T loops of a layer in one pass over its latents, where a kernel shape exists
            lws = torch.zeros(lla.lla_decode_loops_workspace_size(bench.geom, bench.B), dtype=torch.uint8,
                              device=device)
            bench.decode_calls_loops(lws)
        except lla.LLAError as e:
            if e.status != 2:  # LLA_ERR_UNSUPPORTED
                raise
        else:
            lms = _time_ms(lambda: bench.decode_calls_loops(lws), reps=2, warm=1)
            ls_ = lms / 1e3 / w.D
            lbytes = (sum(bench.lens) * w.H * (w.r_k + w.r_v) * 2
                      + w.T * (w.H * w.d * (w.r_k + w.r_v) * 2 + 4 * bench.B * w.H * w.d * 2))
            loops = {"kernel": f"absorb2d_kernel + attn2d_kernel<{w.r_k}, {w.r_v}, 4> + finish2d_kernel (lla_decode_attn_loops)",
                     "ms_per_sweep": lms,
                     "avg_launch_us": ls_ * 1e6, "GB_s": lbytes / ls_ / 1e9, "hbm_frac": lbytes / ls_ / 1e9 / peak,
                     "bytes_per_launch": lbytes, "tokens_per_s_decode_only": bench.B / (lms / 1e3),
                     "note": "all T loops of a layer per call: the layer's latents cross HBM once"}
            if lla.lla_get_device_error() != 0:
                raise RuntimeError(f"device error in the {name} multi-loop decode measurement")
        del lws
        row = {"config": config_dict(w, bench.lens, 1), "steps": steps, "warmup": warmup,
               "kernel": "decode_async_kernel (lla_decode_attn)", "bound": "hbm",
               "ms_per_step": ms, "tokens_per_s": bench.B / (ms / 1e3),
               "avg_launch_us": dec_s * 1e6, "GB_s": nbytes / dec_s / 1e9,
               "hbm_frac": nbytes / dec_s / 1e9 / peak, "frac_of_nominal_8tbs": nbytes / dec_s / 1e9 / NOMINAL_HBM_GBS,
               "bytes_per_launch": nbytes, "traffic": ncu_traffic(name),
               "latent_cache_GB": latent_cache_bytes(w, bench.lens) / 1e9,
               "fill": "N(0,1) bf16 latents written into every page (the decode reads the same bytes "
                       "as for encoded ones)"}
        if rope is not None:
            row["rope_decode"] = rope
        if loops is not None:
            row["loops_decode"] = loops
        lens = bench.lens
        del bench
        torch.cuda.empty_cache()
        row["comparator"] = _dense_comparator(w, lens, device, reps=1 if w.B >= 128 else 2)
        if cpu:
            row["cpu_baseline"] = cpu_baseline(w, lens, cpu_seconds)
        out["decode_" + name] = row
    return out


def run_rho2_as_written(device, steps=None):
    """The rho = 2 workload as it is written: a causal prefill of 4 prompts of 8192 tokens
    through all 24 layers (lla_prefill_two_pass: each layer's pass-1 keys and values encoded, then
    the loop-major pass-2 attention over the latents), then 256 decode steps at batch 32 whose
    contexts grow from 8192 to 8447 (each step: T x D pass-1 calls, then the encode of the 32
    completed tokens in every layer).  The 4 prefilled prompts are sequences 0..3 of the batch;
    the other 28 hold N(0,1) latents.  Pass-1 captures are N(0,1) draws made before the timed
    region (one per layer); pass-2 queries are one N(0,1) draw per loop, handed to every layer."""
    import torch
    from paper_2607_15456_gb300 import lla
    from paper_2607_15456_gb300 import workloads as W
    peak, _ = measured_peaks()
    w = W.WORKLOADS["ouro14_rho2"]
    nseq, Lp = w.prefill
    steps = w.decode_steps if steps is None else steps
    bench = DecodeBench("ouro14_rho2", device, fill="random", extra_tokens=steps + 1)
    geom, pt = bench.geom, bench.pt
    N = nseq * Lp
    slots = torch.cat([pt.slots(b, range(Lp)) for b in range(nseq)]).to(device)
    cu = torch.tensor([i * Lp for i in range(nseq + 1)], dtype=torch.int32, device=device)
    caps = [(W.normal((w.T, N, w.H, w.d), w.seed, 140, l, device=device),
             W.normal((w.T, N, w.H, w.d), w.seed, 141, l, device=device)) for l in range(w.D)]
    qp = [W.normal((N, w.H, w.d), w.seed, 142, t, device=device) for t in range(w.T)]
    op = torch.empty_like(qp[0])
    # prefill tables: the 4 prompts' rows of the batch's block table
    pcaches = [lla.Cache(c.pool, c.num_blocks, bench.table[:nseq].contiguous(), c.max_blocks_per_seq)
               for c in bench.caches]
    marks = {}

    def capture(l):
        return caps[l]

    def query(l, t):
        if l == 0 and t == 0:  # phase 1 (every layer encoded) ends here
            marks["encoded"] = torch.cuda.Event(enable_timing=True)
            marks["encoded"].record()
        return qp[t], op

    def prefill():
        lla.lla_prefill_two_pass(geom, bench.codecs, pcaches, slots, cu, Lp, capture, query)

    prefill()  # warm-up (rewrites the same latents)
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    prefill()
    b.record()
    torch.cuda.synchronize()
    pf_ms = a.elapsed_time(b)
    enc_ms = a.elapsed_time(marks["encoded"])
    del caps
    torch.cuda.empty_cache()
    if lla.lla_get_device_error() != 0:
        raise RuntimeError("device error in the rho = 2 prefill")
    pairs = nseq * w.H * Lp * (Lp + 1) / 2
    attn_flops = w.D * w.T * (pairs * 2 * (w.r_k + w.r_v) + N * w.H * 2 * w.d * (w.r_k + w.r_v))
    enc_bytes = w.D * (2 * w.T * N * w.H * w.d * 2 + w.H * w.T * w.d * (w.r_k + w.r_v) * 2
                       + N * w.H * (w.r_k + w.r_v) * 2)

    # 256 decode steps, contexts L + s, the completed token of step s written at position L + s
    base = torch.tensor(bench.lens, dtype=torch.int32)
    ctx_all = torch.stack([base + s for s in range(steps)]).to(device)
    slots_all = torch.stack([torch.stack([pt.slots(bb, [L + s])[0] for bb, L in enumerate(bench.lens)])
                             for s in range(steps)]).to(device)

    def run_steps(n, ev=None):
        for s in range(n):
            bench.ctx, bench.max_ctx, bench.next_slots = ctx_all[s], max(bench.lens) + s, slots_all[s]
            if ev is not None:
                ev[s][0].record()
            bench.decode_calls()
            if ev is not None:
                ev[s][1].record()
            bench.encode_calls()

    run_steps(2)  # warm-up (the first two steps, repeated below with the same inputs)
    torch.cuda.synchronize()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    a.record()
    run_steps(steps, ev)
    b.record()
    torch.cuda.synchronize()
    if lla.lla_get_device_error() != 0:
        raise RuntimeError("device error in the rho = 2 decode steps")
    dec_total_ms = a.elapsed_time(b)
    dec_kernel_s = sum(x.elapsed_time(y) for x, y in ev) / 1e3
    lat = sum((L + s) for s in range(steps) for L in bench.lens) * w.H * (w.r_k + w.r_v) * 2
    dec_bytes = w.D * w.T * (lat + steps * (w.H * w.d * (w.r_k + w.r_v) * 2 + 4 * bench.B * w.H * w.d * 2))
    B = bench.B
    del bench, pcaches, qp, op
    torch.cuda.empty_cache()
    return {"rho2_as_written": {
        "workload": f"{w.name}: prefill {nseq}x{Lp} through {w.D} layers (two-pass, streamed layer by "
                    f"layer), then {steps} decode steps at B={B}, contexts {Lp} -> {Lp + steps - 1}",
        "prefill_ms": pf_ms, "prefill_tokens_per_s": N / (pf_ms / 1e3),
        "prefill_encode_phase_ms": enc_ms, "prefill_attention_phase_ms": pf_ms - enc_ms,
        "prefill_attention_TFLOP_s": attn_flops / ((pf_ms - enc_ms) / 1e3) / 1e12,
        "prefill_encode_GB_s": enc_bytes / (enc_ms / 1e3) / 1e9,
        "decode_steps": steps, "decode_ms_per_step": dec_total_ms / steps,
        "decode_tokens_per_s": B * steps / (dec_total_ms / 1e3),
        "decode_kernel_GB_s": dec_bytes / dec_kernel_s / 1e9,
        "decode_kernel_hbm_frac": dec_bytes / dec_kernel_s / 1e9 / peak,
        "total_s": (pf_ms + dec_total_ms) / 1e3,
        "kernels": "encode_tc_kernel + prefill_tc_kernel (lla_prefill_two_pass); decode_async_kernel + "
                   "encode_layers_kernel (decode steps)"}}


def run_long_prompt(device, L=65536, rope=False):
    """One long prompt through the streamed two-pass prefill of the rho = 2 Ouro-1.4B geometry
    (24 layers): the regime the layer-by-layer streaming exists for (App. J reaches 64k prompts
    this way).  One layer's capture is live at a time; the same N(0,1) capture tensors stand in
    for every layer's pass-1 keys and values, one N(0,1) query draw per loop for every layer."""
    import torch
    from paper_2607_15456_gb300 import lla
    from paper_2607_15456_gb300 import workloads as W
    peaks = {}
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            peaks = json.load(f)
    except Exception:
        pass
    tc_peak = float(peaks.get("bf16_tflops_sustained", 1700.0))
    w = W.WORKLOADS["ouro14_rho2"]
    geom = lla.Geometry(w.T, w.H, w.d, w.r_k, w.r_v, "bf16")
    pt = W.page_table([L], w.seed, extra_tokens=0)
    table = pt.block_table.to(device)
    bb = lla.lla_cache_block_bytes(geom)
    codecs = [lla.Codec(**W.codec_tensors(w.T, w.H, w.d, w.r_k, w.r_v, w.seed, l, device=device))
              for l in range(w.D)]
    caches = [lla.Cache(torch.empty(pt.num_blocks * bb, dtype=torch.uint8, device=device), pt.num_blocks,
                        table, pt.max_blocks) for _ in range(w.D)]
    slots = pt.slots(0, range(L)).to(device)
    cu = torch.tensor([0, L], dtype=torch.int32, device=device)
    cap = (W.normal((w.T, L, w.H, w.d), w.seed, 150, device=device),
           W.normal((w.T, L, w.H, w.d), w.seed, 151, device=device))
    qp = [W.normal((L, w.H, w.d), w.seed, 152, t, device=device) for t in range(w.T)]
    op = torch.empty_like(qp[0])
    ws = None
    if rope:
        ws = torch.empty(lla.lla_prefill_rope_workspace_size(geom, 1, L), dtype=torch.uint8, device=device)
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    lla.lla_prefill_two_pass(geom, codecs, caches, slots, cu, L, lambda l: cap, lambda l, t: (qp[t], op),
                             rope_base=ROPE_BASE if rope else None, workspace=ws)
    b.record()
    torch.cuda.synchronize()
    if lla.lla_get_device_error() != 0:
        raise RuntimeError("device error in the long-prompt prefill")
    ms = a.elapsed_time(b)
    pairs = w.H * L * (L + 1) / 2
    if rope:
        flops = w.D * w.T * (pairs * 2 * (w.d + w.r_v) + L * w.H * 2 * w.d * (w.r_k + w.r_v))
    else:
        flops = w.D * w.T * (pairs * 2 * (w.r_k + w.r_v) + L * w.H * 2 * w.d * (w.r_k + w.r_v))
    cap_gb = 2 * cap[0].numel() * 2 / 1e9
    res = {"workload": f"one {L}-token prompt, {w.name} geometry ({w.D} layers, (r_k, r_v)=({w.r_k}, {w.r_v}))"
                       + (", RoPE after reconstruction" if rope else ""),
           "kernels": ("rope_rebuild_kernel + prefill_tc_kernel<ROPE>" if rope else "prefill_tc_kernel")
                      + " + encode_tc_kernel (lla_prefill_two_pass)",
           "ms": ms, "tokens_per_s": L / (ms / 1e3), "TFLOP_s": flops / (ms / 1e3) / 1e12,
           "tensor_frac": flops / (ms / 1e3) / 1e12 / tc_peak,
           "capture_live_GB": cap_gb, "captures_of_all_layers_GB_bf16": cap_gb * w.D,
           "latent_cache_GB": w.D * pt.num_blocks * bb / 1e9,
           "note": "TFLOP/s over the whole call (the encodes included) against sustained bf16"}
    del caches, cap, qp, op, ws
    torch.cuda.empty_cache()
    return {("long_prompt_rope" if rope else "long_prompt"): res}


def run_e2e(bench, args, world):
    """Same step with the step's inputs (q, k_cur, v_cur of every call) copied from pinned
    host memory and the outputs copied back, inside the timed region.  Inputs and outputs are
    double-buffered on the device: one stream copies step k+1's inputs in and another copies
    step k-1's outputs out while step k computes."""
    import torch
    import torch.distributed as dist

    q_h = bench.q.cpu().pin_memory()
    k_h = bench.cur_k.cpu().pin_memory()
    v_h = bench.cur_v.cpu().pin_memory()
    o_h = [torch.empty(bench.out.shape, dtype=bench.out.dtype).pin_memory() for _ in range(2)]
    bufs = [(bench.q, bench.cur_k, bench.cur_v, bench.out),
            tuple(torch.empty_like(t) for t in (bench.q, bench.cur_k, bench.cur_v, bench.out))]
    main = torch.cuda.current_stream()
    copy = torch.cuda.Stream(device=bench.device)    # inputs in
    copy_out = torch.cuda.Stream(device=bench.device)  # outputs out
    K = max(1, args.steps)
    ev = lambda: torch.cuda.Event()

    def run(nsteps):
        copy.wait_stream(main)  # nothing on the copy streams starts before the timed region
        copy_out.wait_stream(main)
        copied = [None, None]   # inputs of the step using buffer i are on the device
        done = [None, None]     # the step using buffer i has finished computing
        drained = [None, None]  # the outputs of buffer i have been copied out
        for k in range(nsteps):
            i = k & 1
            q, ck, cv, out = bufs[i]
            with torch.cuda.stream(copy):
                if done[i] is not None:
                    copy.wait_event(done[i])       # step k-2 no longer reads these inputs
                q.copy_(q_h, non_blocking=True)
                ck.copy_(k_h, non_blocking=True)
                cv.copy_(v_h, non_blocking=True)
                copied[i] = ev()
                copied[i].record(copy)
            main.wait_event(copied[i])
            if drained[i] is not None:
                main.wait_event(drained[i])        # step k-2's outputs have left the buffer
            bench.q, bench.cur_k, bench.cur_v, bench.out = q, ck, cv, out
            bench.step()
            done[i] = ev()
            done[i].record(main)
            with torch.cuda.stream(copy_out):
                copy_out.wait_event(done[i])
                o_h[i].copy_(out, non_blocking=True)
                drained[i] = ev()
                drained[i].record(copy_out)
        main.wait_stream(copy)
        main.wait_stream(copy_out)

    run(max(1, args.warmup))
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(main)
    run(K)
    b.record(main)
    torch.cuda.synchronize()
    bench.q, bench.cur_k, bench.cur_v, bench.out = bufs[0]
    ms = max_over_ranks([a.elapsed_time(b)], world, bench.device)[0]
    nbytes = lambda t: t.numel() * t.element_size()
    return {"value": job_tokens_per_s(world, bench.B, ms / K), "unit": "tokens/s",
            "h2d_bytes_per_step": nbytes(q_h) + nbytes(k_h) + nbytes(v_h),
            "d2h_bytes_per_step": nbytes(o_h[0]), "ms_per_step": ms / K,
            "copies": "double-buffered; inputs and outputs on their own streams, overlapping the "
                      "neighbouring steps"}


# ----------------------------------------------------------------- oracle (CPU) timing

def oracle_step_time(w, lens, target_s: float, detail: bool = False):
    """Times the CPU oracle on a bounded sample of one decode step and extrapolates to the
    whole step.  The sample is layer 0: pass-1 decode items (loop, sequence, head) in order
    until about target_s of work, plus the encode of the B completed tokens of layer 0.  The
    oracle's time depends on shapes only, so latents and activations are N(0,1) draws.
    Returns (seconds per full step, sample description, threads), and with detail also the
    sample's own seconds and its share of the full step's work."""
    import numpy as np

    import oracle

    rng = np.random.default_rng(w.seed)
    T, H, d, rk, rv = w.T, w.H, w.d, w.r_k, w.r_v
    w_up_k = rng.standard_normal((T, d, rk)) / math.sqrt(rk)
    w_up_v = rng.standard_normal((T, d, rv)) / math.sqrt(rv)
    scale = 1 / math.sqrt(d)
    threads = oracle.max_threads()
    lat = {}

    def item(t, b):
        if b not in lat:
            lat[b] = (rng.standard_normal((lens[b], rk)), rng.standard_normal((lens[b], rv)))
        return dict(t=t, c_k=lat[b][0], c_v=lat[b][1], w_up_k=w_up_k, w_up_v=w_up_v, mu_k=None,
                    mu_v=None, q=rng.standard_normal(d), cur_k=rng.standard_normal(d),
                    cur_v=rng.standard_normal(d))

    order = [(t, b, h) for t in range(T) for b in range(len(lens)) for h in range(H)]
    work = lambda b: lens[b] + 1  # reconstruction cost per item is proportional to L + 1
    total_work = w.D * H * T * sum(lens[b] + 1 for b in range(len(lens)))
    # calibration batch: one item per thread
    done_work, secs, i = 0, 0.0, 0
    while i < len(order) and secs < target_s:
        n = threads if i == 0 else max(threads, int(threads * 4))
        batch = order[i:i + n]
        items = [item(t, b) for t, b, h in batch]
        t0 = time.perf_counter()
        oracle.decode_batch(T, d, rk, rv, scale, items, n_threads=threads)
        secs += time.perf_counter() - t0
        done_work += sum(work(b) for _, b, _ in batch)
        i += n
    # encode of the completed tokens of layer 0 (all heads, both axes)
    enc_items = [dict(x=rng.standard_normal((T, len(lens), d)), mu=None,
                      w_down=rng.standard_normal((T * d, r)) / math.sqrt(T * d))
                 for _ in range(H) for r in (rk, rv)]
    t0 = time.perf_counter()
    oracle.encode_batch(T, d, enc_items, n_threads=threads)
    enc_s = time.perf_counter() - t0
    step_s = secs * total_work / done_work + enc_s * w.D
    sample = (f"layer 0 of {w.D}: {i if i < len(order) else len(order)} of {len(order)} pass-1 "
              f"decode items (loop, sequence, head) = {done_work / (total_work / w.D):.1%} of the "
              f"layer's decode work, plus the layer's encode of {len(lens)} tokens; extrapolated "
              f"linearly to the full step (work is linear in context length x heads x loops x "
              f"layers)")
    if detail:
        sample_s = secs + enc_s
        frac = sample_s / step_s  # the sample's share of the full step's (linear) work
        return step_s, sample, threads, sample_s, frac
    return step_s, sample, threads


def cpu_baseline(w, lens, target_s):
    step_s, sample, threads = oracle_step_time(w, lens, target_s)
    return {"value": len(lens) / step_s, "unit": "tokens/s", "cores": threads, "kind": "oracle",
            "sample": sample, "seconds_per_step": step_s}


def run_reference(args, rank, world):
    """The oracle as it stands on the host cores.  Each step is one bounded sample of the
    workload's decode step (see oracle_step_time); ms_per_step is the sample's own time and
    value the throughput that sample ran at (tokens of the full step x the sample's share of the
    step's work / the sample's time), so steps x ms_per_step is the time actually measured."""
    from paper_2607_15456_gb300 import workloads as W
    w = W.WORKLOADS[args.workload]
    lens = W.context_lengths(w)
    per_step = max(2.0, min(args.cpu_seconds, 150.0 / max(1, args.steps + args.warmup)))
    for _ in range(args.warmup):
        oracle_step_time(w, lens, per_step)
    full, sample_s, share, sample, threads = [], [], [], "", 1
    t0 = time.perf_counter()
    for _ in range(args.steps):
        s_full, sample, threads, secs, frac = oracle_step_time(w, lens, per_step, detail=True)
        full.append(s_full)
        sample_s.append(secs)
        share.append(frac)
    wall = time.perf_counter() - t0
    value = len(lens) * sum(share) / sum(sample_s)
    return {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": statistics.mean(sample_s) * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": config_dict(w, lens, world),
        "extrapolated": True,
        "step_definition": "one bounded sample of the decode step per timed step; value = tokens "
                           "of the step x the sample's share of its work / the sample's time",
        "full_step_seconds_extrapolated": statistics.mean(full),
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": threads, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
        "wall_seconds": wall,
    }


def main():
    args = parse_args()
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        if rank == 0:
            print(json.dumps(run_reference(args, rank, world)), flush=True)
        return
    if world > 1:
        import torch
        import torch.distributed as dist
        torch.cuda.set_device(local_rank)
        dist.init_process_group("nccl", init_method="env://")
    result = run_ours(args, rank, world, local_rank)
    if rank == 0:
        print(json.dumps(result), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
