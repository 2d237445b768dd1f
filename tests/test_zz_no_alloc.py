"""lla_decode_attn_noalloc: the decode call for callers that cannot allocate device memory.

Some callers cannot call cudaMalloc (a plug-in inside a host application that owns all device
memory, or a latency-critical loop that cannot afford the device synchronisation cudaMalloc
may cause).  lla_decode_attn_noalloc keeps the decode scratch in a fixed 1 MiB device array of
the library instead.  This test first leaves the shared array dirty with a call of another shape
(more sequences, other ranks), then calls the entry point through the C ABI twice in a row and
checks each result against lla_decode_attn with a caller-provided workspace.  Both run the same
kernel with the same split-KV boundaries and the same fixed-order merge, so the outputs must be
bitwise equal (stale partials or counters would show); the oracle tolerance is checked too.  It
lives in its own file, collected last, and builds its own inputs, so it passes both alone in a
fresh process and after the rest of the suite.
"""
import math

import numpy as np
import pytest
import torch

from helpers import assert_parity, ensure_library, f64

pytestmark = pytest.mark.gpu

DEV = "cuda"


def _dirty_scratch(lla, W):
    """One no-alloc call of another shape that uses more of the shared array (48 sequences at
    (192, 320)), so the checked calls below start from its leftovers."""
    T, H, d, r_k, r_v = 4, 16, 128, 192, 320
    lens = [700 + 37 * i for i in range(48)]
    geom = lla.Geometry(T, H, d, r_k, r_v, "bf16")
    codec = lla.Codec(**W.codec_tensors(T, H, d, r_k, r_v, 22, 0, dtype=torch.bfloat16, device=DEV))
    pt = W.page_table(lens, 22, extra_tokens=1)
    pool = torch.zeros(pt.num_blocks * lla.lla_cache_block_bytes(geom), dtype=torch.uint8,
                       device=DEV)
    cache = lla.Cache(pool, pt.num_blocks, pt.block_table.to(DEV), pt.max_blocks)
    N = sum(lens)
    slots = torch.cat([pt.slots(b, range(L)) for b, L in enumerate(lens)]).to(DEV)
    lla.lla_encode(geom, codec, cache, W.normal((T, N, H, d), 22, 1, device=DEV),
                   W.normal((T, N, H, d), 22, 2, device=DEV), slots)
    B = len(lens)
    assert lla.lla_decode_workspace_size(geom, B) > lla.lla_decode_workspace_size(
        lla.Geometry(T, H, d, 96, 160, "bf16"), 6)
    q = W.normal((B, H, d), 22, 3, device=DEV)
    out = torch.empty_like(q)
    lla.lla_decode_attn_noalloc(geom, codec, cache, torch.tensor(lens, dtype=torch.int32, device=DEV),
                                max(lens), 1, q, q, q, out)
    torch.cuda.synchronize()
    assert torch.isfinite(out.float()).all()


def test_noalloc_decode_matches_workspace_decode_on_two_calls():
    ensure_library()
    from paper_2607_15456_gb300 import lla
    from paper_2607_15456_gb300 import workloads as W

    lla.lla_clear_device_error()
    _dirty_scratch(lla, W)
    T, H, d, r_k, r_v = 4, 16, 128, 96, 160
    lens = [3000, 2500, 17, 64, 0, 1300]
    geom = lla.Geometry(T, H, d, r_k, r_v, "bf16")
    cod = W.codec_tensors(T, H, d, r_k, r_v, 21, 0, dtype=torch.bfloat16, device=DEV)
    codec = lla.Codec(**cod)
    pt = W.page_table(lens, 21, extra_tokens=1)
    pool = torch.zeros(pt.num_blocks * lla.lla_cache_block_bytes(geom), dtype=torch.uint8,
                       device=DEV)
    cache = lla.Cache(pool, pt.num_blocks, pt.block_table.to(DEV), pt.max_blocks)
    N = sum(lens)
    slots = torch.cat([pt.slots(b, range(L)) for b, L in enumerate(lens)]).to(DEV)
    lla.lla_encode(geom, codec, cache, W.normal((T, N, H, d), 21, 1, device=DEV),
                   W.normal((T, N, H, d), 21, 2, device=DEV), slots)
    B = len(lens)
    ctx = torch.tensor(lens, dtype=torch.int32, device=DEV)
    ws = torch.zeros(lla.lla_decode_workspace_size(geom, B), dtype=torch.uint8, device=DEV)
    lla.lla_clear_device_error()
    for call, loop in enumerate((0, 3)):
        q = W.normal((B, H, d), 21, 10, call, device=DEV)
        ck = W.normal((B, H, d), 21, 11, call, device=DEV)
        cv = W.normal((B, H, d), 21, 12, call, device=DEV)
        ref = torch.empty_like(q)
        got = torch.full_like(q, float("nan"))
        lla.lla_decode_attn(geom, codec, cache, ctx, max(lens), loop, q, ck, cv, ref, ws)
        lla.lla_decode_attn_noalloc(geom, codec, cache, ctx, max(lens), loop, q, ck, cv, got)
        torch.cuda.synchronize()
        assert torch.equal(got, ref), f"no-alloc call {call} differs from the workspace call"
        assert_parity(f64(got), f64(ref), "bf16", f"no-alloc call {call}")
    assert lla.lla_get_device_error() == 0


def test_noalloc_rejects_requests_beyond_its_scratch():
    """B x H arrival counters beyond the 1 MiB array: rejected before anything is enqueued."""
    ensure_library()
    from paper_2607_15456_gb300 import lla
    geom = lla.Geometry(4, 512, 128, 96, 160, "bf16")
    B = 1024
    assert lla.lla_decode_workspace_size(geom, B) > (1 << 20)
    fake = torch.zeros(16, dtype=torch.bfloat16, device=DEV)  # never read: the call is rejected
    cod = lla.Codec(fake, fake, fake, fake)
    cache = lla.Cache(fake, 1, torch.zeros(1, dtype=torch.int32, device=DEV), 1)
    q = torch.zeros((B, 1, 1), dtype=torch.bfloat16, device=DEV)
    with pytest.raises(lla.LLAError) as e:
        lla.lla_decode_attn_noalloc(geom, cod, cache, torch.zeros(B, dtype=torch.int32, device=DEV),
                                    0, 0, q, None, None, q)
    assert e.value.status == 6  # LLA_ERR_WORKSPACE
