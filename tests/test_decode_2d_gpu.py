"""GPU parity of lla_encode_2d and lla_decode_attn_2d (LLA-2D, Sec. 3 "The LLA-2D variant (loop x
head)") against the CPU float64 oracle (oracle.encode_2d, oracle.decode_2d).

The oracle rebuilds every head's keys and values of loop t from the shared latent and runs plain
softmax attention per head; the GPU absorbs the up-projections per head and reads the latent once
for all heads on the tensor cores.  Tolerances: bf16 storage with fp32 accumulation, max abs
<= 2e-2 (before the final rounding of bf16 outputs, which adds up to half an ulp) and relative
L2 <= 5e-3 against the oracle on its own latents; against the oracle fed the
GPU's stored latents (only accumulation order and the bf16 operands of the two contractions
differ) relative L2 <= 5e-3 as well.
"""
import math

import numpy as np
import pytest
import torch

import oracle
from helpers import assert_parity, ensure_library, f64, rel_l2, unpack_head

pytestmark = pytest.mark.gpu

DEV = "cuda"


@pytest.fixture(scope="module")
def lla():
    ensure_library()
    from paper_2607_15456_gb300 import lla as m
    m.lla_clear_device_error()
    return m


def _dt(name):
    return torch.bfloat16 if name == "bf16" else torch.float32


class Scene2D:
    """One layer's LLA-2D codec and a paged cache (one page per block) filled by lla_encode_2d."""

    def __init__(self, lla, T=4, H=4, d=128, r_k=96, r_v=160, io="fp32", lens=(256,), seed=0,
                 with_mu=False, oracle_encode=True):
        from paper_2607_15456_gb300 import workloads as W
        self.lla, self.W = lla, W
        self.T, self.H, self.d, self.r_k, self.r_v = T, H, d, r_k, r_v
        self.io, self.lens, self.seed = io, list(lens), seed
        self.geom = lla.Geometry(T, H, d, r_k, r_v, "bf16")
        self.scale = 1.0 / math.sqrt(d)
        cod = W.codec_tensors_2d(T, H, d, r_k, r_v, seed, 0, device=DEV, with_mu=with_mu)
        self.codec = lla.Codec(**cod)
        self.w64 = {k: (None if v is None else f64(v)) for k, v in cod.items()}
        self.pt = W.page_table(self.lens, seed, extra_tokens=1)
        bb = lla.lla_cache_2d_block_bytes(self.geom)
        # all-ones bytes are NaN in bf16: a read of a row that was never written shows
        self.pool = torch.full((self.pt.num_blocks * bb,), 0xFF, dtype=torch.uint8, device=DEV)
        self.table = self.pt.block_table.to(DEV)
        self.cache = lla.Cache(self.pool, self.pt.num_blocks, self.table, self.pt.max_blocks)
        self.B = len(self.lens)
        N = sum(self.lens)
        self.x_k = W.normal((T, N, H, d), seed, 40, dtype=_dt(io), device=DEV)
        self.x_v = W.normal((T, N, H, d), seed, 41, dtype=_dt(io), device=DEV)
        if N:
            slots = torch.cat([self.pt.slots(b, range(L)) for b, L in enumerate(self.lens)])
            lla.lla_encode_2d(self.geom, self.codec, self.cache, self.x_k, self.x_v, slots.to(DEV))
        # without oracle_encode the oracle decodes the latents the GPU stored (a decode check;
        # the encode is checked by the tests that keep it)
        self.oracle_encode = oracle_encode
        xk, xv = f64(self.x_k), f64(self.x_v)
        self.ck, self.cv = [], []
        off = 0
        for L in (self.lens if oracle_encode else []):
            self.ck.append(oracle.encode_2d(xk[:, off:off + L], self.w64["mu_k"], self.w64["w_down_k"]))
            self.cv.append(oracle.encode_2d(xv[:, off:off + L], self.w64["mu_v"], self.w64["w_down_v"]))
            off += L
        self.ws = torch.empty(lla.lla_decode_2d_workspace_size(self.geom, self.B), dtype=torch.uint8,
                              device=DEV)

    def gpu_latents(self, b, L=None):
        L = self.lens[b] if L is None else L
        return unpack_head(self.pool.cpu(), 1, self.r_k, self.r_v, "bf16", self.pt.block_table[b], L, 0)

    def append_token(self, seed_key=42):
        W = self.W
        xk = W.normal((self.T, self.B, self.H, self.d), self.seed, seed_key, dtype=_dt(self.io), device=DEV)
        xv = W.normal((self.T, self.B, self.H, self.d), self.seed, seed_key + 1, dtype=_dt(self.io), device=DEV)
        slots = torch.stack([self.pt.slots(b, [L])[0] for b, L in enumerate(self.lens)]).to(DEV)
        self.lla.lla_encode_2d(self.geom, self.codec, self.cache, xk, xv, slots)
        xk64, xv64 = f64(xk), f64(xv)
        for b in (range(self.B) if self.oracle_encode else []):
            self.ck[b] = np.concatenate([self.ck[b], oracle.encode_2d(xk64[:, b:b + 1], self.w64["mu_k"],
                                                                      self.w64["w_down_k"])])
            self.cv[b] = np.concatenate([self.cv[b], oracle.encode_2d(xv64[:, b:b + 1], self.w64["mu_v"],
                                                                      self.w64["w_down_v"])])
        self.lens = [L + 1 for L in self.lens]

    def decode(self, loop, pass1, key=50, lens=None):
        W = self.W
        shape = (self.B, self.H, self.d)
        q = W.normal(shape, self.seed, key, loop, dtype=_dt(self.io), device=DEV)
        ck = W.normal(shape, self.seed, key + 1, loop, dtype=_dt(self.io), device=DEV) if pass1 else None
        cv = W.normal(shape, self.seed, key + 2, loop, dtype=_dt(self.io), device=DEV) if pass1 else None
        out = torch.empty(shape, dtype=_dt(self.io), device=DEV)
        lens = self.lens if lens is None else lens
        lt = torch.tensor(lens, dtype=torch.int32, device=DEV)
        self.lla.lla_decode_attn_2d(self.geom, self.codec, self.cache, lt, max(lens + [0]), loop, q,
                                    ck, cv, out, self.ws)
        torch.cuda.synchronize()
        return q, ck, cv, out

    def oracle_decode(self, loop, q, ck, cv, b, latents=None, heads=None):
        if latents is None:
            latents = (self.ck[b], self.cv[b]) if self.oracle_encode else self.gpu_latents(b)
        c_k, c_v = latents
        w = self.w64
        return oracle.decode_2d(loop, c_k, c_v, w["w_up_k"], w["w_up_v"], w["mu_k"], w["mu_v"],
                                f64(q[b]), None if ck is None else f64(ck[b]),
                                None if cv is None else f64(cv[b]), self.scale, heads=heads)


def _check(sc, loop, pass1, tight=False, seqs=None):
    q, ck, cv, out = sc.decode(loop, pass1)
    got = f64(out)
    seqs = list(range(sc.B)) if seqs is None else seqs
    ref = np.stack([sc.oracle_decode(loop, q, ck, cv, b) for b in seqs])
    sel = got[seqs]
    assert np.isfinite(sel).all()
    assert_parity(sel, ref, "bf16", f"2D decode loop {loop} pass{1 if pass1 else 2}", io=sc.io,
                  output_rounding=True)
    if tight:
        ref2 = np.stack([sc.oracle_decode(loop, q, ck, cv, b, latents=sc.gpu_latents(b)) for b in seqs])
        assert rel_l2(sel, ref2) <= 5e-3, rel_l2(sel, ref2)
    return got


@pytest.mark.parametrize("with_mu", [False, True])
def test_tiny_2d_encode_then_two_pass_decode(lla, with_mu):
    """T=4, H=4, 2D ranks (96, 160), one sequence of 256 tokens: encode, pass 1 over all four
    loops, encode of the completed token, pass 2 over all four loops; fp32 inputs and outputs."""
    sc = Scene2D(lla, with_mu=with_mu, seed=70)
    gk, gv = sc.gpu_latents(0)
    assert_parity(gk, sc.ck[0], "bf16", "2D K latents")
    assert_parity(gv, sc.cv[0], "bf16", "2D V latents")
    for t in range(sc.T):
        _check(sc, t, pass1=True, tight=True)
    sc.append_token()
    for t in range(sc.T):
        _check(sc, t, pass1=False, tight=True)
    assert lla.lla_get_device_error() == 0


@pytest.mark.parametrize("rk,rv,H", [(96, 160, 16), (128, 128, 8), (288, 480, 16), (288, 480, 5)])
def test_ragged_batch_every_shape(lla, rk, rv, H):
    """Empty (pass 1 only), one token, page-aligned, ragged tails and several pages in one batch,
    bf16 inputs and outputs, with mu; H = 5 leaves 11 of the 16 MMA head columns unused."""
    lens = [0, 1, 63, 64, 65, 200, 513]
    sc = Scene2D(lla, H=H, r_k=rk, r_v=rv, io="bf16", lens=lens, seed=71, with_mu=True)
    for b in (1, 4, 6):
        gk, gv = sc.gpu_latents(b)
        assert_parity(gk, sc.ck[b], "bf16", "2D K latents")
        assert_parity(gv, sc.cv[b], "bf16", "2D V latents")
    for t in (0, 3):
        _check(sc, t, pass1=True)
    sc.append_token()
    _check(sc, 1, pass1=False)
    assert lla.lla_get_device_error() == 0


def test_pass1_empty_cache_returns_current_value(lla):
    sc = Scene2D(lla, lens=[0, 0, 0], seed=72)
    q, ck, cv, out = sc.decode(2, pass1=True)
    torch.testing.assert_close(out, cv, rtol=0, atol=0)


@pytest.mark.parametrize("lens", [[4000, 3100, 2049], [20000, 9000]])
def test_long_sequences_split_across_many_ctas(lla, lens):
    """Fewer pages than CTAs (each CTA holds about one page of one sequence) and more pages than
    CTAs (runs of several pages, sequences split over many CTAs and merged by the finish); the
    oracle decodes the stored latents."""
    sc = Scene2D(lla, H=16, r_k=288, r_v=480, io="bf16", lens=lens, seed=73, with_mu=True,
                 oracle_encode=False)
    _check(sc, 0, pass1=True)
    sc.append_token()
    _check(sc, 2, pass1=False)


def test_many_short_sequences(lla):
    """300 sequences of 1 to 140 tokens: many runs per CTA and 38 finish groups of 8."""
    g = torch.Generator().manual_seed(74)
    lens = [int(v) for v in torch.randint(1, 141, (300,), generator=g)]
    sc = Scene2D(lla, H=8, r_k=288, r_v=480, io="bf16", lens=lens, seed=74, oracle_encode=False)
    _check(sc, 1, pass1=True, seqs=[0, 1, 2, 77, 150, 298, 299])


def test_2d_decode_is_deterministic(lla):
    sc = Scene2D(lla, H=16, r_k=288, r_v=480, io="bf16", lens=[700, 1500, 90], seed=75,
                 oracle_encode=False)
    a = sc.decode(0, True)[3].clone()
    b = sc.decode(0, True)[3]
    assert torch.equal(a, b)


def test_device_checks_flag_bad_block_ids_and_lengths(lla):
    sc = Scene2D(lla, lens=[100, 200], io="bf16", seed=76, oracle_encode=False)
    lla.lla_clear_device_error()
    bad = sc.table.clone()
    bad[1, 2] = sc.pt.num_blocks + 3
    cache = lla.Cache(sc.pool, sc.pt.num_blocks, bad, sc.pt.max_blocks)
    q = torch.zeros((sc.B, sc.H, sc.d), dtype=torch.bfloat16, device=DEV)
    out = torch.empty_like(q)
    lens = torch.tensor(sc.lens, dtype=torch.int32, device=DEV)
    lla.lla_decode_attn_2d(sc.geom, sc.codec, cache, lens, 200, 0, q, q, q, out, sc.ws)
    torch.cuda.synchronize()
    assert lla.lla_get_device_error() & lla.LLA_DEVERR_BLOCK_ID
    lla.lla_clear_device_error()
    # a length past max_ctx, and pass 2 over an empty sequence
    lens = torch.tensor([100, 500], dtype=torch.int32, device=DEV)
    lla.lla_decode_attn_2d(sc.geom, sc.codec, sc.cache, lens, 200, 0, q, q, q, out, sc.ws)
    torch.cuda.synchronize()
    assert lla.lla_get_device_error() & lla.LLA_DEVERR_CONTEXT
    lla.lla_clear_device_error()
    lens = torch.tensor([0, 200], dtype=torch.int32, device=DEV)
    lla.lla_decode_attn_2d(sc.geom, sc.codec, sc.cache, lens, 200, 0, q, None, None, out, sc.ws)
    torch.cuda.synchronize()
    assert lla.lla_get_device_error() & lla.LLA_DEVERR_EMPTY_PASS2
    lla.lla_clear_device_error()
    assert lla.lla_get_device_error() == 0


def test_full_size_stress2d_sampled(lla):
    """The LLA-2D stress workload at full size (H=16, (288, 480), B=128, contexts ~ U[8192,
    32768], one layer, the launch configuration the benchmark times): random N(0,1) bf16 latents
    written straight into the pages, every output finite, and sampled (sequence, head) outputs
    (the shortest and the longest sequence among them) against the oracle."""
    from paper_2607_15456_gb300 import workloads as W
    w = W.WORKLOADS["stress2d_rho2133"]
    lens = W.context_lengths(w)
    pt = W.page_table(lens, w.seed)
    N = sum(lens)
    c_k = W.normal((N, w.r_k), w.seed, 80, device=DEV)
    c_v = W.normal((N, w.r_v), w.seed, 81, device=DEV)
    pool = W.pack_latent_pages(c_k, c_v, pt.block_table, lens, pt.num_blocks)
    geom = lla.Geometry(w.T, w.H, w.d, w.r_k, w.r_v, "bf16")
    cod = W.codec_tensors_2d(w.T, w.H, w.d, w.r_k, w.r_v, w.seed, 0, device=DEV, with_mu=True)
    codec = lla.Codec(**cod)
    cache = lla.Cache(pool, pt.num_blocks, pt.block_table.to(DEV), pt.max_blocks)
    ws = torch.empty(lla.lla_decode_2d_workspace_size(geom, w.B), dtype=torch.uint8, device=DEV)
    shape = (w.B, w.H, w.d)
    q = W.normal(shape, w.seed, 82, device=DEV)
    ck = W.normal(shape, w.seed, 83, device=DEV)
    cv = W.normal(shape, w.seed, 84, device=DEV)
    out = torch.empty(shape, dtype=torch.bfloat16, device=DEV)
    lt = torch.tensor(lens, dtype=torch.int32, device=DEV)
    lla.lla_decode_attn_2d(geom, codec, cache, lt, max(lens), 1, q, ck, cv, out, ws)
    torch.cuda.synchronize()
    assert lla.lla_get_device_error() == 0
    got = f64(out)
    assert np.isfinite(got).all()
    w64 = {k: (None if v is None else f64(v)) for k, v in cod.items()}
    starts = np.concatenate([[0], np.cumsum(lens)])
    picks = [int(np.argmin(lens)), int(np.argmax(lens)), 37]
    for b in picks:
        ckb = f64(c_k[starts[b]:starts[b + 1]])
        cvb = f64(c_v[starts[b]:starts[b + 1]])
        heads = [0, 9, 15]
        ref = oracle.decode_2d(1, ckb, cvb, w64["w_up_k"], w64["w_up_v"], w64["mu_k"], w64["mu_v"],
                               f64(q[b]), f64(ck[b]), f64(cv[b]), 1 / math.sqrt(w.d), heads=heads)
        assert_parity(got[b, heads], ref, "bf16", f"2D stress sequence {b}", io="bf16",
                      output_rounding=True)


def test_large_latents_ragged_batch(lla):
    """(1152, 1920), rho_2D = 5.33 (paper Table isocache): a 384 KB page streams through the
    kernel in K-plane column chunks and V-plane row chunks; empty, one-token, page-aligned and
    ragged sequences, with mu, both passes; the stored latents against the oracle's encode."""
    sc = Scene2D(lla, H=16, r_k=1152, r_v=1920, io="bf16", lens=[0, 1, 63, 64, 65, 200], seed=76,
                 with_mu=True)
    for b in (1, 4, 5):
        gk, gv = sc.gpu_latents(b)
        assert_parity(gk, sc.ck[b], "bf16", "2D K latents")
        assert_parity(gv, sc.cv[b], "bf16", "2D V latents")
    _check(sc, 0, pass1=True)
    sc.append_token()
    _check(sc, 3, pass1=False)
    assert lla.lla_get_device_error() == 0


@pytest.mark.parametrize("lens", [[3000, 1100], [9000, 3000, 17]])
def test_large_latents_split_across_ctas(lla, lens):
    """Fewer and more pages than CTAs at (1152, 1920): runs of one sequence on many CTAs, merged
    by the finish kernel; the oracle decodes the stored latents."""
    sc = Scene2D(lla, H=16, r_k=1152, r_v=1920, io="bf16", lens=lens, seed=77, with_mu=True,
                 oracle_encode=False)
    _check(sc, 1, pass1=True)
    sc.append_token()
    _check(sc, 2, pass1=False)
    assert lla.lla_get_device_error() == 0
