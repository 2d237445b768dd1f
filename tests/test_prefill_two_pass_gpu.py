"""GPU parity of lla_prefill_two_pass: the capacity decoder's two-pass prefill of a batch of
prompts through every layer, streamed layer by layer (App. A "Decoding and caching"; App. J
"Eviction and long-context prefill").

A three-layer model with a per-layer codec (with mu) and ragged prompts.  The callbacks hand over
each layer's pass-1 keys and values and each (layer, loop)'s pass-2 queries; the test checks
  * the call order: every layer's capture first (layer by layer), then the re-forward loop by
    loop, layer by layer within a loop;
  * that the latents each layer's cache holds and every (layer, loop) output equal, bit for bit,
    those of separate lla_encode and lla_prefill_attn(_rope) calls on the same inputs;
  * the outputs against the oracle (Eq. encode of the layer's captures, then causal attention over
    the explicitly reconstructed keys and values, with or without RoPE after reconstruction), on
    every row of two heads at the first and last loop of every layer: bf16 tolerance, max abs
    <= 2e-2 beyond the rounding of a bf16 output, relative L2 <= 5e-3.
"""
import math

import numpy as np
import pytest
import torch

import oracle
from helpers import assert_parity, ensure_library, f64

pytestmark = pytest.mark.gpu

DEV = "cuda"


@pytest.fixture(scope="module")
def lla():
    ensure_library()
    from paper_2607_15456_gb300 import lla as m
    m.lla_clear_device_error()
    return m


@pytest.mark.parametrize("rope", [False, True])
def test_two_pass_prefill_streams_layers_and_matches_the_oracle(lla, rope):
    from paper_2607_15456_gb300 import workloads as W
    D, T, H, d, r_k, r_v = 3, 4, 4, 128, 96, 160
    lens = [300, 130, 1]
    seed = 90
    base, pairing = 10000.0, lla.LLA_ROPE_HALF
    geom = lla.Geometry(T, H, d, r_k, r_v, "bf16")
    pt = W.page_table(lens, seed, extra_tokens=0)
    table = pt.block_table.to(DEV)
    bb = lla.lla_cache_block_bytes(geom)
    N = sum(lens)
    slots = torch.cat([pt.slots(b, range(L)) for b, L in enumerate(lens)]).to(DEV)
    cu = torch.tensor(np.cumsum([0] + lens), dtype=torch.int32, device=DEV)
    cods = [W.codec_tensors(T, H, d, r_k, r_v, seed, l, dtype=torch.bfloat16, device=DEV, with_mu=True)
            for l in range(D)]
    codecs = [lla.Codec(**c) for c in cods]

    def pools():
        return [torch.full((pt.num_blocks * bb,), 0xFF, dtype=torch.uint8, device=DEV) for _ in range(D)]

    pa, pb = pools(), pools()
    caches_a = [lla.Cache(p, pt.num_blocks, table, pt.max_blocks) for p in pa]
    caches_b = [lla.Cache(p, pt.num_blocks, table, pt.max_blocks) for p in pb]
    xk = [W.normal((T, N, H, d), seed, 100, l, device=DEV) for l in range(D)]
    xv = [W.normal((T, N, H, d), seed, 101, l, device=DEV) for l in range(D)]
    q = [[W.normal((N, H, d), seed, 102, l, t, device=DEV) for t in range(T)] for l in range(D)]
    out = [[torch.full((N, H, d), float("nan"), dtype=torch.bfloat16, device=DEV) for _ in range(T)]
           for _ in range(D)]
    ws = None
    if rope:
        ws = torch.empty(lla.lla_prefill_rope_workspace_size(geom, len(lens), max(lens)), dtype=torch.uint8,
                         device=DEV)
    order = []

    def capture(l):
        order.append(("capture", l))
        return xk[l], xv[l]

    def query(l, t):
        order.append(("query", l, t))
        return q[l][t], out[l][t]

    lla.lla_clear_device_error()
    lla.lla_prefill_two_pass(geom, codecs, caches_a, slots, cu, max(lens), capture, query,
                             rope_base=base if rope else None, rope_pairing=pairing, workspace=ws)
    torch.cuda.synchronize()
    assert lla.lla_get_device_error() == 0
    assert order == [("capture", l) for l in range(D)] + [("query", l, t) for t in range(T) for l in range(D)]

    # the same steps as separate calls
    ref = [[torch.empty_like(out[0][0]) for _ in range(T)] for _ in range(D)]
    for l in range(D):
        lla.lla_encode(geom, codecs[l], caches_b[l], xk[l], xv[l], slots)
    for t in range(T):
        for l in range(D):
            if rope:
                lla.lla_prefill_attn_rope(geom, codecs[l], caches_b[l], base, pairing, cu, max(lens), t,
                                          q[l][t], ref[l][t], ws)
            else:
                lla.lla_prefill_attn(geom, codecs[l], caches_b[l], cu, max(lens), t, q[l][t], ref[l][t])
    torch.cuda.synchronize()
    for l in range(D):
        # compare the written pages only (unwritten rows of a last page keep the poison bytes)
        assert torch.equal(pa[l], pb[l]), f"layer {l} latents"
        for t in range(T):
            assert torch.equal(out[l][t], ref[l][t]), f"layer {l} loop {t} output"

    # the oracle on its own latents
    scale = 1.0 / math.sqrt(d)
    for l in range(D):
        w = {k: (None if v is None else f64(v)) for k, v in cods[l].items()}
        xk64, xv64 = f64(xk[l]), f64(xv[l])
        for t in (0, T - 1):
            got = f64(out[l][t])
            q64 = f64(q[l][t])
            off = 0
            for b, L in enumerate(lens):
                for h in (0, H - 1):
                    ck = oracle.encode(xk64[:, off:off + L, h], w["mu_k"][h], w["w_down_k"][h])
                    cv = oracle.encode(xv64[:, off:off + L, h], w["mu_v"][h], w["w_down_v"][h])
                    args = (w["w_up_k"][h], w["w_up_v"][h], w["mu_k"][h], w["mu_v"][h], q64[off:off + L, h], scale)
                    r = (oracle.prefill_rope(t, ck, cv, *args, base, pairing) if rope
                         else oracle.prefill(t, ck, cv, *args))
                    assert_parity(got[off:off + L, h], r, "bf16", f"layer {l} loop {t} b{b} h{h}",
                                  output_rounding=True)
                off += L


def test_a_failing_callback_stops_the_prefill(lla):
    """A callback that raises: nothing after it is called or enqueued, and the error reaches the
    caller."""
    from paper_2607_15456_gb300 import workloads as W
    D, T, H, d, r_k, r_v = 2, 4, 2, 128, 96, 160
    lens = [70]
    geom = lla.Geometry(T, H, d, r_k, r_v, "bf16")
    pt = W.page_table(lens, 91, extra_tokens=0)
    table = pt.block_table.to(DEV)
    codecs = [lla.Codec(**W.codec_tensors(T, H, d, r_k, r_v, 91, l, dtype=torch.bfloat16, device=DEV))
              for l in range(D)]
    caches = [lla.Cache(torch.zeros(pt.num_blocks * lla.lla_cache_block_bytes(geom), dtype=torch.uint8,
                                    device=DEV), pt.num_blocks, table, pt.max_blocks) for _ in range(D)]
    slots = pt.slots(0, range(70)).to(DEV)
    cu = torch.tensor([0, 70], dtype=torch.int32, device=DEV)
    x = W.normal((T, 70, H, d), 91, 1, device=DEV)
    calls = []

    def capture(l):
        calls.append(l)
        if l == 1:
            raise KeyError("no capture for layer 1")
        return x, x

    with pytest.raises(KeyError):
        lla.lla_prefill_two_pass(geom, codecs, caches, slots, cu, 70, capture,
                                 lambda l, t: pytest.fail("no query after a failed capture"))
    assert calls == [0, 1]
    torch.cuda.synchronize()
    assert lla.lla_get_device_error() == 0
