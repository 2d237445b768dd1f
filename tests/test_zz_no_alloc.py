"""lla_decode_attn_noalloc: the decode call for callers that cannot allocate device memory.

Some callers cannot call cudaMalloc (a plug-in inside a host application that owns all device
memory, or a latency-critical loop that cannot afford the device synchronisation cudaMalloc
may cause).  lla_decode_attn_noalloc keeps the decode scratch in a fixed 1 MiB device array of
the library instead.  This test calls it through the C ABI twice in a row and checks each result
against lla_decode_attn with a caller-provided workspace, within the tolerance of the other
decode tests.  It lives in its own file, collected last, and builds its own inputs, so it passes
both alone in a fresh process and after the rest of the suite.
"""
import math

import numpy as np
import pytest
import torch

from helpers import assert_parity, ensure_library, f64

pytestmark = pytest.mark.gpu

DEV = "cuda"


def test_noalloc_decode_matches_workspace_decode_on_two_calls():
    ensure_library()
    from paper_2607_15456_gb300 import lla
    from paper_2607_15456_gb300 import workloads as W

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
