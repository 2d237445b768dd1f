"""GPU parity of lla_prefill_attn_rope (causal prefill with rotary positions applied after
reconstruction, Sec. 3 "RoPE and reconstruction") against the CPU float64 oracle
(oracle.prefill_rope).

The cache is filled by lla_encode from the seeded generators; the oracle rebuilds every key by
Eq. decode, rotates keys and queries at their prompt positions and runs causal softmax attention.
Two comparisons per (sequence, head): against the oracle on its own latents (bf16 storage: max
abs <= 2e-2 beyond the rounding of a bf16 output, relative L2 <= 5e-3), and against the oracle
fed the latents the GPU stored (relative L2 <= 5e-3: the kernels round rotated keys and queries
and the probabilities to bf16 tensor-core operands).  Cases: prompts shorter than a page, on page
and tile boundaries and across several query tiles, both pairings, with and without mu, the
three tensor-core rank shapes.
"""
import numpy as np
import pytest
import torch

import oracle
from helpers import assert_parity, ensure_library, f64, rel_l2
from test_decode_gpu import Scene

pytestmark = pytest.mark.gpu

DEV = "cuda"


@pytest.fixture(scope="module")
def lla():
    ensure_library()
    from paper_2607_15456_gb300 import lla as m
    m.lla_clear_device_error()
    return m


def _case(lla, r_k, r_v, io, lens, loop, with_mu, pairing, base=10000.0, H=2, seed=0):
    sc = Scene(lla, T=4, H=H, d=128, r_k=r_k, r_v=r_v, storage="bf16", io=io, lens=lens,
               seed=seed, with_mu=with_mu, extra_tokens=0)
    W = sc.W
    N = sum(lens)
    dt = torch.bfloat16 if io == "bf16" else torch.float32
    q = W.normal((N, H, 128), seed, 70, loop, dtype=dt, device=DEV)
    out = torch.full_like(q, float("nan"))
    cu = torch.tensor(np.cumsum([0] + list(lens)), dtype=torch.int32, device=DEV)
    ws = torch.empty(lla.lla_prefill_rope_workspace_size(sc.geom, len(lens), max(lens)),
                     dtype=torch.uint8, device=DEV)
    lla.lla_prefill_attn_rope(sc.geom, sc.codec, sc.cache, base, pairing, cu, max(lens), loop,
                              q, out, ws)
    torch.cuda.synchronize()
    assert lla.lla_get_device_error() == 0
    got, q64 = f64(out), f64(q)
    w = sc.w64
    off = 0
    for b, L in enumerate(lens):
        for h in range(H):
            mk = None if w["mu_k"] is None else w["mu_k"][h]
            mv = None if w["mu_v"] is None else w["mu_v"][h]
            args = (w["w_up_k"][h], w["w_up_v"][h], mk, mv, q64[off:off + L, h], sc.scale, base,
                    pairing)
            ref = oracle.prefill_rope(loop, sc.ck[b, h], sc.cv[b, h], *args)
            assert_parity(got[off:off + L, h], ref, "bf16", f"rope prefill b{b} h{h}", io=io,
                          output_rounding=True)
            gk, gv = sc.gpu_latents(b, h)
            ref2 = oracle.prefill_rope(loop, gk, gv, *args)
            assert rel_l2(got[off:off + L, h], ref2) <= 5e-3, rel_l2(got[off:off + L, h], ref2)
        off += L
    return sc


@pytest.mark.parametrize("pairing", [0, 1])
@pytest.mark.parametrize("with_mu", [False, True])
def test_rope_prefill_ragged_prompts(lla, pairing, with_mu):
    """Prompts of 1, 63, 64, 65, 200 and 300 tokens (within a page, on page and tile boundaries,
    several 128-query tiles), (96, 160), fp32 queries and outputs."""
    _case(lla, 96, 160, "fp32", [1, 63, 64, 65, 200, 300], 2, with_mu, pairing, seed=80)


@pytest.mark.parametrize("rk,rv", [(192, 320), (128, 128)])
def test_rope_prefill_rank_shapes(lla, rk, rv):
    _case(lla, rk, rv, "bf16", [130, 257], 1, True, 0, base=500000.0, seed=81)


def test_rope_prefill_long_prompt(lla):
    """One 2000-token prompt at H = 4: many query tiles, positions up to 2 x 10^3."""
    _case(lla, 96, 160, "bf16", [2000], 3, False, 0, H=4, seed=82)


def test_rope_prefill_rejects_rows_past_the_workspace(lla):
    """cu_seqlens that start past row 0 reach beyond B * max_len rows of the rotated-query
    buffer: flagged, and nothing is written out of range."""
    sc = Scene(lla, T=4, H=2, d=128, r_k=96, r_v=160, storage="bf16", io="bf16", lens=[100, 50],
               seed=83, extra_tokens=0)
    q = torch.zeros((450, 2, 128), dtype=torch.bfloat16, device=DEV)
    out = torch.zeros_like(q)
    cu = torch.tensor([300, 400, 450], dtype=torch.int32, device=DEV)  # rows 300..449
    ws = torch.empty(lla.lla_prefill_rope_workspace_size(sc.geom, 2, 100), dtype=torch.uint8,
                     device=DEV)
    lla.lla_clear_device_error()
    lla.lla_prefill_attn_rope(sc.geom, sc.codec, sc.cache, 10000.0, 0, cu, 100, 0, q, out, ws)
    torch.cuda.synchronize()
    assert lla.lla_get_device_error() & lla.LLA_DEVERR_CONTEXT
    lla.lla_clear_device_error()
