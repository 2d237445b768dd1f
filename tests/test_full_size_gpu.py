"""Parity at the full sizes of the benchmark workloads, in the launch configuration bench.py times.

For each workload (Ouro-1.4B at rho = 4 and 2, Ouro-2.6B at rho = 5.33, the rho = 21.33 stress
shape) one layer of the cache is filled exactly as bench.py fills it (its batch, its context
lengths, its scattered page table), then one pass-1 decode call runs at the loop given.  The
oracle cannot take the whole batch in seconds, so outputs are sampled: the shortest and the
longest sequence and four more, each at three heads.

  * decode: the oracle is fed the latents the GPU stored (read back page by page through the
    documented layout), so only the kernel is under test; bound relative L2 <= 5e-3 on the
    sampled rows, max abs <= 2e-2 (bf16 output).
  * encode: for the sampled (sequence, head) pairs, 64 positions spread over the context are
    re-encoded by the oracle from the same inputs and compared with the stored latents.
  * prefill: the rho = 2 workload's prompts (4 x 8192 tokens), sampled rows checked as pass-2
    decodes of their causal prefixes.
  * RoPE decode: the headline batch through lla_decode_attn_rope, sampled rows against the
    oracle's RoPE decode on the stored latents.
"""
import numpy as np
import pytest
import torch

import oracle
from helpers import BLOCK, assert_parity, ensure_library, f64, unpack_head

pytestmark = pytest.mark.gpu

DEV = "cuda"


def _sample_sequences(lens, k=6):
    order = sorted(range(len(lens)), key=lambda b: lens[b])
    picks = [order[0], order[-1]]
    rng = np.random.default_rng(len(lens))
    for b in rng.permutation(len(lens)):
        if len(picks) >= k:
            break
        if int(b) not in picks:
            picks.append(int(b))
    return picks


def _compact_pages(pool, table_row, L, block_bytes):
    """CPU copy of the pages holding positions 0..L-1 of one sequence, with a table 0..n-1."""
    n = -(-L // BLOCK)
    ids = table_row[:n].to(torch.int64).to(pool.device)
    pages = pool.view(-1, block_bytes)[ids].reshape(-1).cpu()
    return pages, torch.arange(n, dtype=torch.int32)


@pytest.mark.parametrize("wname,loop", [("ouro14_rho4", 2), ("ouro14_rho2", 0),
                                        ("ouro26_rho533", 3), ("stress_rho2133", 1)])
def test_full_size_decode_and_encode_sampled(wname, loop):
    ensure_library()
    import bench
    from paper_2607_15456_gb300 import lla
    from paper_2607_15456_gb300 import workloads as W

    dev = torch.device(DEV, 0)
    db = bench.DecodeBench(wname, dev, layers=1)
    w = db.w
    lla.lla_clear_device_error()
    lla.lla_decode_attn(db.geom, db.codecs[0], db.caches[0], db.ctx, db.max_ctx, loop,
                        db.q[0, loop], db.cur_k[0, loop], db.cur_v[0, loop], db.out[0, loop], db.ws)
    torch.cuda.synchronize()
    assert lla.lla_get_device_error() == 0
    out = f64(db.out[0, loop])
    cod = {k: (None if v is None else f64(v)) for k, v in
           W.codec_tensors(w.T, w.H, w.d, w.r_k, w.r_v, w.seed, 0, dtype=torch.bfloat16).items()}
    q, ck, cv = f64(db.q[0, loop]), f64(db.cur_k[0, loop]), f64(db.cur_v[0, loop])
    bb = lla.lla_cache_block_bytes(db.geom)
    scale = 1.0 / np.sqrt(w.d)
    # the inputs bench.py encoded: chunks of 131072 tokens in sequence order
    chunk = 1 << 17
    starts = np.cumsum([0] + db.lens)
    got_rows, ref_rows = [], []
    for b in _sample_sequences(db.lens):
        L = db.lens[b]
        pages, table = _compact_pages(db.pools[0], db.pt.block_table[b], L, bb)
        positions = np.unique(np.linspace(0, L - 1, 64).astype(np.int64))
        heads = (0, w.H // 2, w.H - 1)
        # the inputs of the sampled positions, regenerating each chunk they fall in once
        xs_k = np.zeros((len(positions), w.T, w.H, w.d))
        xs_v = np.zeros_like(xs_k)
        glob = starts[b] + positions
        for ci in np.unique(glob // chunk):
            sel = np.nonzero(glob // chunk == ci)[0]
            n1 = min(int(starts[-1]), (int(ci) + 1) * chunk) - int(ci) * chunk
            offs = torch.as_tensor(glob[sel] - int(ci) * chunk, device=dev)
            for key, dst in ((100, xs_k), (101, xs_v)):
                x = W.normal((w.T, n1, w.H, w.d), w.seed, key, 0, int(ci), device=dev)
                dst[sel] = f64(x[:, offs].permute(1, 0, 2, 3))
                del x
        for h in heads:
            c_k, c_v = unpack_head(pages, w.H, w.r_k, w.r_v, w.storage, table, L, h)
            ref = oracle.decode(loop, c_k, c_v, cod["w_up_k"][h], cod["w_up_v"][h], None, None,
                                q[b, h], ck[b, h], cv[b, h], scale)
            got_rows.append(out[b, h])
            ref_rows.append(ref)
            ek = oracle.encode(xs_k[:, :, h, :].transpose(1, 0, 2), None, cod["w_down_k"][h])
            ev = oracle.encode(xs_v[:, :, h, :].transpose(1, 0, 2), None, cod["w_down_v"][h])
            assert_parity(c_k[positions], ek, "bf16", f"{wname} c_k b{b} h{h}")
            assert_parity(c_v[positions], ev, "bf16", f"{wname} c_v b{b} h{h}")
    assert_parity(np.stack(got_rows), np.stack(ref_rows), "bf16", f"{wname} decode loop {loop}")


@pytest.mark.parametrize("pairing,io", [(0, "bf16"), (1, "bf16"), (0, "fp32")])
def test_full_size_rope_decode_sampled(pairing, io):
    """The RoPE decode (lla_decode_attn_rope, base 10^4) on the headline batch as bench.py runs
    it: sampled (sequence, head) rows against oracle.decode_rope fed the stored latents.  With
    fp32 inputs and outputs the plain bound holds (max abs <= 2e-2, relative L2 <= 5e-3, no
    allowance for an output's own rounding)."""
    ensure_library()
    import bench
    from paper_2607_15456_gb300 import lla
    from paper_2607_15456_gb300 import workloads as W

    dev = torch.device(DEV, 0)
    db = bench.DecodeBench("ouro14_rho4", dev, layers=1)
    w = db.w
    loop = 1
    dt = torch.float32 if io == "fp32" else torch.bfloat16
    qi, cki, cvi = (t[0, loop].to(dt).contiguous() for t in (db.q, db.cur_k, db.cur_v))
    o = torch.empty_like(qi)
    lla.lla_clear_device_error()
    lla.lla_decode_attn_rope(db.geom, db.codecs[0], db.caches[0], 10000.0, pairing, db.ctx,
                             db.max_ctx, loop, qi, cki, cvi, o, db.ws)
    torch.cuda.synchronize()
    assert lla.lla_get_device_error() == 0
    out = f64(o)
    cod = {k: (None if v is None else f64(v)) for k, v in
           W.codec_tensors(w.T, w.H, w.d, w.r_k, w.r_v, w.seed, 0, dtype=torch.bfloat16).items()}
    q, ck, cv = f64(qi), f64(cki), f64(cvi)
    bb = lla.lla_cache_block_bytes(db.geom)
    scale = 1.0 / np.sqrt(w.d)
    got_rows, ref_rows = [], []
    for b in _sample_sequences(db.lens):
        L = db.lens[b]
        pages, table = _compact_pages(db.pools[0], db.pt.block_table[b], L, bb)
        for h in (0, w.H // 2, w.H - 1):
            c_k, c_v = unpack_head(pages, w.H, w.r_k, w.r_v, w.storage, table, L, h)
            ref = oracle.decode_rope(loop, c_k, c_v, cod["w_up_k"][h], cod["w_up_v"][h], None,
                                     None, q[b, h], ck[b, h], cv[b, h], scale, 10000.0, pairing)
            got_rows.append(out[b, h])
            ref_rows.append(ref)
    assert_parity(np.stack(got_rows), np.stack(ref_rows), "bf16", f"rope decode, full size, {io} io",
                  io=io, output_rounding=io == "bf16")


@pytest.mark.parametrize("io", ["bf16", "fp32"])
def test_full_size_prefill_sampled_rows(io):
    """Causal prefill at the benchmark's prompt size (Ouro-1.4B at rho = 2: 4 prompts of 8192
    tokens, 16 heads), in the launch configuration bench.py times.  Row i of a prompt is the
    pass-2 decode of query i over keys 0..i, so sampled rows are checked with the oracle's decode
    on the latents the GPU stored (first and last rows, rows on tile and page boundaries, and
    random rows).  bf16 queries and outputs: the bf16 bound taken before the output's own
    rounding; fp32 queries and outputs: the plain bound (max abs <= 2e-2, relative L2 <= 5e-3)."""
    ensure_library()
    from paper_2607_15456_gb300 import lla
    from paper_2607_15456_gb300 import workloads as W

    dev = torch.device(DEV, 0)
    w = W.WORKLOADS["ouro14_rho2"]
    nseq, L = w.prefill
    T, H, d = w.T, w.H, w.d
    geom = lla.Geometry(T, H, d, w.r_k, w.r_v, "bf16")
    cod = W.codec_tensors(T, H, d, w.r_k, w.r_v, w.seed, 0, device=dev)
    codec = lla.Codec(**cod)
    lens = [L] * nseq
    pt = W.page_table(lens, w.seed, extra_tokens=0)
    bb = lla.lla_cache_block_bytes(geom)
    pool = torch.zeros(pt.num_blocks * bb, dtype=torch.uint8, device=dev)
    cache = lla.Cache(pool, pt.num_blocks, pt.block_table.to(dev), pt.max_blocks)
    N = nseq * L
    slots = torch.cat([pt.slots(b, range(L)) for b in range(nseq)]).to(dev)
    lla.lla_encode(geom, codec, cache, W.normal((T, N, H, d), w.seed, 300, device=dev),
                   W.normal((T, N, H, d), w.seed, 301, device=dev), slots)
    q = W.normal((N, H, d), w.seed, 302, device=dev, dtype=torch.float32 if io == "fp32" else torch.bfloat16)
    out = torch.empty_like(q)
    cu = torch.tensor([i * L for i in range(nseq + 1)], dtype=torch.int32, device=dev)
    lla.lla_clear_device_error()
    loop = 1
    lla.lla_prefill_attn(geom, codec, cache, cu, L, loop, q, out)
    torch.cuda.synchronize()
    assert lla.lla_get_device_error() == 0
    w64 = {k: (None if v is None else f64(v)) for k, v in cod.items()}
    scale = 1.0 / np.sqrt(d)
    rng = np.random.default_rng(11)
    rows = sorted({0, 1, 63, 64, 127, 128, 129, 4095, 4096, L - 2, L - 1} |
                  set(int(x) for x in rng.integers(0, L, 6)))
    got, ref = [], []
    for b, h in ((0, 0), (3, 15), (1, 7)):
        pages, table = _compact_pages(pool, pt.block_table[b], L, bb)
        c_k, c_v = unpack_head(pages, H, w.r_k, w.r_v, "bf16", table, L, h)
        qb = f64(q[b * L:(b + 1) * L, h])
        ob = f64(out[b * L:(b + 1) * L, h])
        for i in rows:
            ref.append(oracle.decode(loop, c_k[:i + 1], c_v[:i + 1], w64["w_up_k"][h], w64["w_up_v"][h],
                                     None, None, qb[i], None, None, scale))
            got.append(ob[i])
    assert_parity(np.stack(got), np.stack(ref), "bf16", f"full-size prefill rows, {io} io", io=io,
                  output_rounding=io == "bf16")
