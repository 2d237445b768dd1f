"""GPU parity of lla_decode_attn_loops (the decode calls of all T loops of a layer in one pass
over the shared latents) against the CPU float64 oracle: loop t of the call must equal
oracle.decode at loop t, the definition of one decode call (App. A; App. J absorbed form per
loop).  Tolerances as for lla_decode_attn: bf16 storage, max abs <= 2e-2 beyond the rounding of
a bf16 output and relative L2 <= 5e-3; with fp32 outputs, relative L2 <= 1e-4 against the oracle
fed the latents the GPU stored.  The loop-t output is also compared with lla_decode_attn at loop t:
the tensor-core kernel feeds q~ and p to the MMAs as sums of three bf16 parts (24 significant
bits, as fp32), so the two differ only in summation order (relative L2 <= 1e-5).
"""
import numpy as np
import pytest
import torch

import oracle
from helpers import assert_parity, f64, rel_l2
from test_decode_gpu import DEV, Scene, _dt, lla  # noqa: F401  (lla is a fixture)

pytestmark = pytest.mark.gpu


def _run_loops(sc, pass1, key=90):
    W = sc.W
    shape = (sc.T, sc.B, sc.H, sc.d)
    q = W.normal(shape, sc.seed, key, dtype=_dt(sc.io), device=DEV)
    ck = W.normal(shape, sc.seed, key + 1, dtype=_dt(sc.io), device=DEV) if pass1 else None
    cv = W.normal(shape, sc.seed, key + 2, dtype=_dt(sc.io), device=DEV) if pass1 else None
    out = torch.empty(shape, dtype=_dt(sc.io), device=DEV)
    # the workspace needs no initialisation: all-ones bytes (NaN floats, -1 ints) must not matter
    ws = torch.full((sc.lla.lla_decode_loops_workspace_size(sc.geom, sc.B),), 0xFF, dtype=torch.uint8,
                    device=DEV)
    lens = torch.tensor(sc.lens, dtype=torch.int32, device=DEV)
    sc.lla.lla_decode_attn_loops(sc.geom, sc.codec, sc.cache, lens, max(sc.lens + [0]), q, ck, cv,
                                 out, ws)
    torch.cuda.synchronize()
    return q, ck, cv, out, ws


def _check(sc, pass1, tight=False, pairs=None, single=True):
    q, ck, cv, out, ws = _run_loops(sc, pass1)
    got = f64(out)
    pairs = pairs or [(b, h) for b in range(sc.B) for h in range(sc.H)]
    for t in range(sc.T):
        qt = q[t]
        ckt = None if ck is None else ck[t]
        cvt = None if cv is None else cv[t]
        ref = np.stack([sc.oracle_decode(t, qt, ckt, cvt, b, h) for b, h in pairs])
        sel = np.stack([got[t, b, h] for b, h in pairs])
        assert_parity(sel, ref, sc.storage, f"loops call, loop {t}", io=sc.io, output_rounding=True)
        if tight:
            ref2 = np.stack([sc.oracle_decode(t, qt, ckt, cvt, b, h, latents=sc.gpu_latents(b, h))
                             for b, h in pairs])
            bound = 1e-4 if sc.io == "fp32" else 5e-3
            assert rel_l2(sel, ref2) <= bound, rel_l2(sel, ref2)
        if single:
            one = torch.empty_like(qt)
            lens = torch.tensor(sc.lens, dtype=torch.int32, device=DEV)
            sc.lla.lla_decode_attn(sc.geom, sc.codec, sc.cache, lens, max(sc.lens + [0]), t, qt,
                                   ckt, cvt, one, sc.ws)
            torch.cuda.synchronize()
            if sc.io == "fp32":
                assert rel_l2(got[t], f64(one)) <= 1e-5, rel_l2(got[t], f64(one))
    assert sc.lla.lla_get_device_error() == 0
    return ws


@pytest.mark.parametrize("with_mu", [False, True])
def test_tiny_workload_both_passes(lla, with_mu):
    sc = Scene(lla, with_mu=with_mu, io="fp32", seed=50)
    _check(sc, pass1=True, tight=True)
    sc.append_token()
    _check(sc, pass1=False, tight=True)


@pytest.mark.parametrize("rk,rv", [(96, 160), (128, 128), (72, 120), (192, 320)])
def test_ragged_batch(lla, rk, rv):
    sc = Scene(lla, r_k=rk, r_v=rv, io="bf16", lens=[0, 1, 63, 64, 65, 200, 513], seed=51,
               with_mu=True)
    _check(sc, pass1=True)
    sc.append_token()
    _check(sc, pass1=False)


def test_long_sequences_split_across_many_ctas(lla):
    sc = Scene(lla, H=16, lens=[4000, 3100, 2049], io="fp32", seed=52)
    pairs = [(b, h) for b in range(3) for h in (0, 5, 15)]
    _check(sc, pass1=True, pairs=pairs)


@pytest.mark.parametrize("T", [1, 2, 3])
def test_fewer_loops_than_query_slots(lla, T):
    """T < 4: the absent query slots of a unit carry zero q~ and p and write nothing."""
    sc = Scene(lla, T=T, H=3, lens=[70, 0, 130], io="fp32", seed=55, with_mu=True)
    _check(sc, pass1=True, tight=True)
    sc.append_token()
    _check(sc, pass1=False, tight=True)


@pytest.mark.parametrize("rk,rv", [(96, 160), (192, 320)])
def test_many_short_sequences_and_determinism(lla, rk, rv):
    """200 sequences x 2 heads x 4 loops: many runs per CTA; at (192, 320) a batch this large
    takes the finish without row slices, the small batches above take it with them."""
    g = torch.Generator().manual_seed(53)
    lens = [int(v) for v in torch.randint(1, 141, (200,), generator=g)]
    sc = Scene(lla, H=2, r_k=rk, r_v=rv, lens=lens, io="bf16", seed=53)
    pairs = [(b, h) for b in range(0, 200, 7) for h in range(2)]
    _check(sc, pass1=True, pairs=pairs, single=False)
    a = _run_loops(sc, True)[3].clone()
    b = _run_loops(sc, True)[3]
    assert torch.equal(a, b)


def test_pass1_empty_cache_returns_current_values(lla):
    sc = Scene(lla, lens=[0, 0], io="fp32", seed=54)
    q, ck, cv, out, ws = _run_loops(sc, True)
    torch.testing.assert_close(out, cv, rtol=0, atol=0)
