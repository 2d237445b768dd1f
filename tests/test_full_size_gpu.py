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
