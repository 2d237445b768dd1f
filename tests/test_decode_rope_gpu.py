"""GPU parity of lla_decode_attn_rope (RoPE applied after reconstruction, Sec. 3 "RoPE and
reconstruction") against the CPU float64 oracle (oracle.decode_rope).

The caches are filled by lla_encode from the seeded generators exactly as in
test_decode_gpu.py; the oracle rebuilds every key by Eq. decode, rotates it at its position and
the query at the current token's, and runs plain softmax attention.  The GPU rebuilds keys on
the tensor cores and rotates through relative positions.  Tolerances: bf16 storage, max abs
<= 2e-2 and relative L2 <= 5e-3; against the oracle fed the GPU's own stored latents (only
accumulation order and the fp32 rotation phases differ), relative L2 <= 1e-4 for fp32 outputs.
"""
import numpy as np
import pytest
import torch

import oracle
from helpers import assert_parity, f64, rel_l2
from test_decode_gpu import DEV, Scene, _dt, lla  # noqa: F401  (lla is a fixture)

pytestmark = pytest.mark.gpu

HALF, ADJ = oracle.ROPE_HALF, oracle.ROPE_ADJACENT


def _decode_rope(sc, loop, pass1, base, pairing, key=30):
    W = sc.W
    shape = (sc.B, sc.H, sc.d)
    q = W.normal(shape, sc.seed, key, loop, dtype=_dt(sc.io), device=DEV)
    ck = W.normal(shape, sc.seed, key + 1, loop, dtype=_dt(sc.io), device=DEV) if pass1 else None
    cv = W.normal(shape, sc.seed, key + 2, loop, dtype=_dt(sc.io), device=DEV) if pass1 else None
    out = torch.empty(shape, dtype=_dt(sc.io), device=DEV)
    lens = torch.tensor(sc.lens, dtype=torch.int32, device=DEV)
    sc.lla.lla_decode_attn_rope(sc.geom, sc.codec, sc.cache, base, pairing, lens,
                                max(sc.lens + [0]), loop, q, ck, cv, out, sc.ws)
    torch.cuda.synchronize()
    return q, ck, cv, out


def _oracle(sc, loop, q, ck, cv, b, h, base, pairing, latents=None):
    c_k, c_v = latents if latents is not None else (sc.ck[b, h], sc.cv[b, h])
    w = sc.w64
    return oracle.decode_rope(loop, c_k, c_v, w["w_up_k"][h], w["w_up_v"][h],
                              None if w["mu_k"] is None else w["mu_k"][h],
                              None if w["mu_v"] is None else w["mu_v"][h],
                              f64(q[b, h]), None if ck is None else f64(ck[b, h]),
                              None if cv is None else f64(cv[b, h]), sc.scale, base, pairing)


def _check(sc, loop, pass1, base=10000.0, pairing=HALF, tight=False, pairs=None):
    q, ck, cv, out = _decode_rope(sc, loop, pass1, base, pairing)
    got = f64(out)
    pairs = pairs or [(b, h) for b in range(sc.B) for h in range(sc.H)]
    ref = np.stack([_oracle(sc, loop, q, ck, cv, b, h, base, pairing) for b, h in pairs])
    sel = np.stack([got[b, h] for b, h in pairs])
    assert_parity(sel, ref, sc.storage, f"rope decode loop {loop} pass{1 if pass1 else 2}",
                  io=sc.io, output_rounding=True)
    if tight:
        ref2 = np.stack([_oracle(sc, loop, q, ck, cv, b, h, base, pairing,
                                 latents=sc.gpu_latents(b, h)) for b, h in pairs])
        bound = 1e-4 if sc.io == "fp32" else 5e-3
        assert rel_l2(sel, ref2) <= bound, rel_l2(sel, ref2)
    return got


@pytest.mark.parametrize("pairing", [HALF, ADJ])
@pytest.mark.parametrize("with_mu", [False, True])
def test_tiny_workload_two_pass_decode(lla, pairing, with_mu):
    """T=4, H=4, (96,160), one sequence of 256 cached tokens: pass 1 over all four loops, encode
    of the completed token, pass 2 over all four loops, fp32 outputs."""
    sc = Scene(lla, with_mu=with_mu, io="fp32", seed=40)
    for t in range(sc.T):
        _check(sc, t, pass1=True, pairing=pairing, tight=True)
    sc.append_token()
    for t in range(sc.T):
        _check(sc, t, pass1=False, pairing=pairing, tight=True)
    assert lla.lla_get_device_error() == 0


@pytest.mark.parametrize("rk,rv", [(96, 160), (128, 128), (192, 320), (72, 120)])
@pytest.mark.parametrize("base", [10000.0, 1e6])
def test_ragged_batch(lla, rk, rv, base):
    """Empty (pass 1 only), one token, page-aligned, ragged tails and several pages in one
    batch, bf16 inputs and outputs, with mu."""
    sc = Scene(lla, r_k=rk, r_v=rv, io="bf16", lens=[0, 1, 63, 64, 65, 200, 513], seed=41,
               with_mu=True)
    for t in (0, 3):
        _check(sc, t, pass1=True, base=base)
    sc.append_token()
    _check(sc, 1, pass1=False, base=base, pairing=ADJ)
    assert lla.lla_get_device_error() == 0


def test_long_sequences_split_across_many_ctas(lla):
    """H=16 and a few long sequences: every (sequence, head) is split over several CTAs, so runs
    start mid-sequence (the phase of a run's first page) and partials are merged."""
    sc = Scene(lla, H=16, lens=[4000, 3100, 2049], io="bf16", seed=42, with_mu=True)
    for t in (0, 2):
        _check(sc, t, pass1=True)
    sc.append_token()
    _check(sc, 3, pass1=False, pairing=ADJ)


def test_long_sequences_split_across_many_ctas_rho2(lla):
    """The rho = 2 rank shape (192, 320): 64 KB head pages, two ring stages, W_up,t^K of 96
    TMEM columns per A slot; long sequences split over CTAs, both passes."""
    sc = Scene(lla, H=16, r_k=192, r_v=320, lens=[3000, 2100, 70], io="bf16", seed=48, with_mu=True)
    _check(sc, 1, pass1=True)
    sc.append_token()
    _check(sc, 2, pass1=False, pairing=ADJ)


def test_long_sequences_split_across_many_ctas_rho533(lla):
    """The Ouro-2.6B rank shape (72, 120): r_k is not a multiple of 16, so the key rebuild takes a
    fifth K step over zero columns of A; long sequences split over CTAs, both passes, with mu."""
    sc = Scene(lla, H=16, r_k=72, r_v=120, lens=[5000, 2100, 64, 65], io="bf16", seed=49, with_mu=True)
    _check(sc, 3, pass1=True, tight=True)
    sc.append_token()
    _check(sc, 0, pass1=False, pairing=ADJ)


def test_far_positions_keep_their_phase(lla):
    """One 30000-token sequence: relative offsets up to 3 * 10^4 rad at theta_0 = 1 take the
    phase through the 64-bit fixed-point turns; checked on fp32 outputs against the oracle."""
    sc = Scene(lla, H=2, lens=[30000], io="fp32", seed=43)
    _check(sc, 1, pass1=True, tight=True)
    _check(sc, 2, pass1=True, base=500000.0, pairing=ADJ, tight=True)


def test_many_short_sequences(lla):
    g = torch.Generator().manual_seed(44)
    lens = [int(v) for v in torch.randint(1, 141, (300,), generator=g)]
    sc = Scene(lla, H=2, lens=lens, io="bf16", seed=44)
    _check(sc, 2, pass1=True)


def test_rope_decode_is_deterministic(lla):
    sc = Scene(lla, H=8, lens=[700, 1500, 90], io="bf16", seed=45)
    a = _decode_rope(sc, 0, True, 10000.0, HALF)[3].clone()
    b = _decode_rope(sc, 0, True, 10000.0, HALF)[3]
    assert torch.equal(a, b)


def test_pass1_empty_cache_returns_current_value(lla):
    sc = Scene(lla, lens=[0, 0], io="fp32", seed=46)
    q, ck, cv, out = _decode_rope(sc, 1, True, 10000.0, HALF)
    torch.testing.assert_close(out, cv, rtol=0, atol=0)


def test_device_checks_flag_a_bad_block_id(lla):
    sc = Scene(lla, lens=[100, 200], io="bf16", seed=47)
    lla.lla_clear_device_error()
    bad = sc.table.clone()
    bad[1, 2] = sc.pt.num_blocks + 3
    cache = lla.Cache(sc.pool, sc.pt.num_blocks, bad, sc.pt.max_blocks)
    q = torch.zeros((sc.B, sc.H, sc.d), dtype=torch.bfloat16, device=DEV)
    out = torch.empty_like(q)
    lens = torch.tensor(sc.lens, dtype=torch.int32, device=DEV)
    lla.lla_decode_attn_rope(sc.geom, sc.codec, cache, 10000.0, HALF, lens, 200, 0, q, q, q,
                             out, sc.ws)
    torch.cuda.synchronize()
    assert lla.lla_get_device_error() & lla.LLA_DEVERR_BLOCK_ID
    lla.lla_clear_device_error()
    lla.lla_decode_workspace_init(sc.ws)
    assert lla.lla_get_device_error() == 0
