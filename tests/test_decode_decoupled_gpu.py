"""GPU parity of lla_encode_rope_keys and lla_decode_attn_decoupled (per-head LLA with the
decoupled rotary branch, App. J "Absorbed attention") against the CPU float64 oracle
(oracle.rope, oracle.decode_decoupled).

The latent cache comes from lla_encode as in test_decode_gpu.py; one rotary key per token (shared
by every loop and head) is stored turned at the token's position.  The oracle rebuilds every
content key by Eq. decode, joins it with the rotary key turned at its position, and runs plain
softmax attention; the GPU streams the block's rotary plane beside each head page and extends
every token's absorbed score over the rotary dimensions.  Tolerances: bf16 storage, max abs
<= 2e-2 (before the final rounding of bf16 outputs) and relative L2 <= 5e-3.
"""
import numpy as np
import pytest
import torch

import oracle
from helpers import assert_parity, f64
from test_decode_gpu import DEV, Scene, _dt, lla  # noqa: F401  (lla is a fixture)

pytestmark = pytest.mark.gpu

HALF, ADJ = oracle.ROPE_HALF, oracle.ROPE_ADJACENT


class Rotary:
    """Rotary planes for a Scene: one N(0,1) rotary key per token, stored by lla_encode_rope_keys."""

    def __init__(self, sc, d_rope, base=10000.0, pairing=HALF, key=60):
        self.sc, self.d_rope, self.base, self.pairing = sc, d_rope, base, pairing
        lla = sc.lla
        plane = lla.lla_rope_plane_bytes(d_rope)
        self.pool = torch.full((sc.pt.num_blocks * plane,), 0xFF, dtype=torch.uint8, device=DEV)
        N = sum(sc.lens)
        self.k = sc.W.normal((N, d_rope), sc.seed, key, dtype=_dt(sc.io), device=DEV)
        self.keys = []  # per sequence, float64 [L][d_rope]
        off = 0
        k64 = f64(self.k)
        for L in sc.lens:
            self.keys.append(k64[off:off + L])
            off += L
        if N:
            pos = torch.cat([torch.arange(L, dtype=torch.int32) for L in sc.lens]).to(DEV)
            lla.lla_encode_rope_keys(d_rope, base, pairing, self.pool, sc.pt.num_blocks, self.k, pos,
                                     sc.slots)
        self.ws = torch.zeros(lla.lla_decode_decoupled_workspace_size(sc.geom, d_rope, sc.B),
                              dtype=torch.uint8, device=DEV)

    def append(self, key=61):
        """The completed token's rotary key at position L_b (call before Scene.append_token)."""
        sc = self.sc
        k = sc.W.normal((sc.B, self.d_rope), sc.seed, key, dtype=_dt(sc.io), device=DEV)
        pos = torch.tensor(sc.lens, dtype=torch.int32, device=DEV)
        slots = torch.stack([sc.pt.slots(b, [L])[0] for b, L in enumerate(sc.lens)]).to(DEV)
        sc.lla.lla_encode_rope_keys(self.d_rope, self.base, self.pairing, self.pool, sc.pt.num_blocks,
                                    k, pos, slots)
        k64 = f64(k)
        self.keys = [np.concatenate([self.keys[b], k64[b:b + 1]]) for b in range(sc.B)]

    def decode(self, loop, pass1, key=70):
        sc, W = self.sc, self.sc.W
        shape = (sc.B, sc.H, sc.d)
        q = W.normal(shape, sc.seed, key, loop, dtype=_dt(sc.io), device=DEV)
        qr = W.normal((sc.B, sc.H, self.d_rope), sc.seed, key + 1, loop, dtype=_dt(sc.io), device=DEV)
        ck = W.normal(shape, sc.seed, key + 2, loop, dtype=_dt(sc.io), device=DEV) if pass1 else None
        cv = W.normal(shape, sc.seed, key + 3, loop, dtype=_dt(sc.io), device=DEV) if pass1 else None
        ckr = W.normal((sc.B, self.d_rope), sc.seed, key + 4, loop, dtype=_dt(sc.io), device=DEV) if pass1 else None
        out = torch.empty(shape, dtype=_dt(sc.io), device=DEV)
        lens = torch.tensor(sc.lens, dtype=torch.int32, device=DEV)
        sc.lla.lla_decode_attn_decoupled(sc.geom, sc.codec, sc.cache, self.pool, self.d_rope, self.base,
                                         self.pairing, lens, max(sc.lens + [0]), loop, q, qr, ck, cv, ckr,
                                         out, self.ws)
        torch.cuda.synchronize()
        return q, qr, ck, cv, ckr, out

    def oracle_decode(self, loop, q, qr, ck, cv, ckr, b, h):
        sc, w = self.sc, self.sc.w64
        return oracle.decode_decoupled(
            loop, sc.ck[b, h], sc.cv[b, h], self.keys[b], w["w_up_k"][h], w["w_up_v"][h],
            None if w["mu_k"] is None else w["mu_k"][h], None if w["mu_v"] is None else w["mu_v"][h],
            f64(q[b, h]), f64(qr[b, h]), None if ck is None else f64(ck[b, h]),
            None if cv is None else f64(cv[b, h]), None if ckr is None else f64(ckr[b]),
            sc.scale, self.base, self.pairing)


def _check(rt, loop, pass1, pairs=None):
    sc = rt.sc
    q, qr, ck, cv, ckr, out = rt.decode(loop, pass1)
    got = f64(out)
    pairs = pairs or [(b, h) for b in range(sc.B) for h in range(sc.H)]
    ref = np.stack([rt.oracle_decode(loop, q, qr, ck, cv, ckr, b, h) for b, h in pairs])
    sel = np.stack([got[b, h] for b, h in pairs])
    assert_parity(sel, ref, "bf16", f"decoupled loop {loop} pass{1 if pass1 else 2}", io=sc.io,
                  output_rounding=True)
    return got


@pytest.mark.parametrize("pairing", [HALF, ADJ])
@pytest.mark.parametrize("with_mu", [False, True])
def test_tiny_workload_two_pass_decode(lla, pairing, with_mu):
    """T=4, H=4, (96,160), d_rope=64, one sequence of 256 cached tokens: pass 1 over all four
    loops, encode of the completed token (latents and rotary key), pass 2 over all four loops;
    fp32 inputs and outputs."""
    sc = Scene(lla, with_mu=with_mu, io="fp32", seed=80)
    rt = Rotary(sc, 64, pairing=pairing)
    for t in range(sc.T):
        _check(rt, t, pass1=True)
    rt.append()
    sc.append_token()
    for t in range(sc.T):
        _check(rt, t, pass1=False)
    assert lla.lla_get_device_error() == 0


@pytest.mark.parametrize("d_rope", [32, 64, 96])
def test_ragged_batch(lla, d_rope):
    """Empty (pass 1 only), one token, page-aligned, ragged tails and several pages, H=16, bf16
    inputs and outputs, with mu."""
    sc = Scene(lla, H=16, io="bf16", lens=[0, 1, 63, 64, 65, 200, 513], seed=81, with_mu=True)
    rt = Rotary(sc, d_rope, base=500000.0)
    for t in (0, 3):
        _check(rt, t, pass1=True)
    rt.append()
    sc.append_token()
    _check(rt, 1, pass1=False)
    assert lla.lla_get_device_error() == 0


@pytest.mark.parametrize("lens", [[4000, 3100, 2049], [9000, 130, 5000]])
def test_long_sequences_split_across_many_ctas(lla, lens):
    """Units (sequence, head) of many pages split over many CTAs and merged by the finish."""
    sc = Scene(lla, H=16, lens=lens, io="bf16", seed=82, with_mu=True)
    rt = Rotary(sc, 64, pairing=ADJ)
    _check(rt, 2, pass1=True, pairs=[(b, h) for b in range(sc.B) for h in (0, 7, 15)])
    rt.append()
    sc.append_token()
    _check(rt, 0, pass1=False, pairs=[(b, h) for b in range(sc.B) for h in (3, 12)])


def test_pass1_empty_cache_returns_current_value(lla):
    sc = Scene(lla, lens=[0, 0], io="fp32", seed=83)
    rt = Rotary(sc, 32)
    q, qr, ck, cv, ckr, out = rt.decode(1, True)
    torch.testing.assert_close(out, cv, rtol=0, atol=0)


def test_decoupled_decode_is_deterministic(lla):
    sc = Scene(lla, H=8, lens=[700, 1500, 90], io="bf16", seed=84)
    rt = Rotary(sc, 64)
    a = rt.decode(0, True)[5].clone()
    b = rt.decode(0, True)[5]
    assert torch.equal(a, b)


def test_rotary_keys_are_stored_turned_at_their_positions(lla):
    """The rotary plane rows against oracle.rope (RoFormer rotation, pinned) at positions up to
    20000, in the granule layout of a K-plane; bf16 storage."""
    sc = Scene(lla, H=2, lens=[20000, 3], io="bf16", seed=85)
    for pairing in (HALF, ADJ):
        rt = Rotary(sc, 64, pairing=pairing)
        plane = rt.pool.cpu().view(sc.pt.num_blocks, 64 // 8, 64, 16)  # [block][granule][row][16 B]
        for b, positions in ((0, [0, 1, 63, 64, 12345, 19999]), (1, [0, 2])):
            for p in positions:
                blk = int(sc.pt.block_table[b, p // 64])
                raw = plane[blk, :, p % 64, :].contiguous().view(torch.bfloat16).reshape(-1)
                got = raw.to(torch.float64).numpy()
                ref = oracle.rope(rt.keys[b][p], p, rt.base, pairing)
                assert np.abs(got - ref).max() <= 2.0 ** -8 * (np.abs(ref).max() + 1e-3) + 1e-6, (b, p)
    assert lla.lla_get_device_error() == 0


def test_device_checks_flag_a_bad_block_id(lla):
    sc = Scene(lla, lens=[100, 200], io="bf16", seed=86)
    rt = Rotary(sc, 32)
    lla.lla_clear_device_error()
    bad = sc.table.clone()
    bad[1, 2] = sc.pt.num_blocks + 3
    cache = lla.Cache(sc.pool, sc.pt.num_blocks, bad, sc.pt.max_blocks)
    q = torch.zeros((sc.B, sc.H, sc.d), dtype=torch.bfloat16, device=DEV)
    qr = torch.zeros((sc.B, sc.H, 32), dtype=torch.bfloat16, device=DEV)
    kr = torch.zeros((sc.B, 32), dtype=torch.bfloat16, device=DEV)
    out = torch.empty_like(q)
    lens = torch.tensor(sc.lens, dtype=torch.int32, device=DEV)
    lla.lla_decode_attn_decoupled(sc.geom, sc.codec, cache, rt.pool, 32, 10000.0, HALF, lens, 200, 0, q,
                                  qr, q, q, kr, out, rt.ws)
    torch.cuda.synchronize()
    assert lla.lla_get_device_error() & lla.LLA_DEVERR_BLOCK_ID
    lla.lla_clear_device_error()
