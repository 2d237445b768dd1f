"""GPU parity of lla_encode (Eq. encode, Sec. 3) against the CPU float64 oracle.

The latents the GPU stored are read back from the paged pool through the documented layout and
compared with oracle.encode on the same inputs (bf16 storage: max abs <= 2e-2 and relative
L2 <= 5e-3; fp32 storage and fp32 x: relative L2 <= 1e-5).  The cases reach the kernel's
separate code paths: a reduction axis T*d longer than one shared-memory chunk of W_down (fp32
and bf16), ranks whose rows are not a multiple of 16 bytes (4-byte copies), token counts that
leave a ragged last tile, x in bf16 and fp32, with and without mu, a decode-step batch, and
prompts of 128 tokens or more in bf16, which take the tensor-core kernel.
"""
import pytest
import torch

import oracle
from helpers import assert_parity, ensure_library, f64, unpack_head

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


def _encode_and_compare(lla, T, H, d, r_k, r_v, storage, x_dtype, lens, with_mu, seed):
    from paper_2607_15456_gb300 import workloads as W
    geom = lla.Geometry(T, H, d, r_k, r_v, storage)
    cod = W.codec_tensors(T, H, d, r_k, r_v, seed, 0, dtype=_dt(storage), device=DEV,
                          with_mu=with_mu)
    codec = lla.Codec(**cod)
    pt = W.page_table(lens, seed, extra_tokens=0)
    bb = lla.lla_cache_block_bytes(geom)
    pool = torch.full((pt.num_blocks * bb,), 0xFF, dtype=torch.uint8, device=DEV)
    cache = lla.Cache(pool, pt.num_blocks, pt.block_table.to(DEV), pt.max_blocks)
    N = sum(lens)
    x_k = W.normal((T, N, H, d), seed, 40, dtype=_dt(x_dtype), device=DEV)
    x_v = W.normal((T, N, H, d), seed, 41, dtype=_dt(x_dtype), device=DEV)
    slots = torch.cat([pt.slots(b, range(L)) for b, L in enumerate(lens)]).to(DEV)
    lla.lla_encode(geom, codec, cache, x_k, x_v, slots)
    torch.cuda.synchronize()
    assert lla.lla_get_device_error() == 0
    w = {k: (None if v is None else f64(v)) for k, v in cod.items()}
    xk, xv = f64(x_k), f64(x_v)
    pool_cpu = pool.cpu()
    off = 0
    for b, L in enumerate(lens):
        for h in range(H):
            gk, gv = unpack_head(pool_cpu, H, r_k, r_v, storage, pt.block_table[b], L, h)
            ck = oracle.encode(xk[:, off:off + L, h, :], None if w["mu_k"] is None else w["mu_k"][h],
                               w["w_down_k"][h])
            cv = oracle.encode(xv[:, off:off + L, h, :], None if w["mu_v"] is None else w["mu_v"][h],
                               w["w_down_v"][h])
            io = "bf16" if x_dtype == "bf16" else "fp32"
            assert_parity(gk, ck, storage, f"c_k b{b} h{h}", io=io)
            assert_parity(gv, cv, storage, f"c_v b{b} h{h}", io=io)
        off += L


@pytest.mark.parametrize("storage,x_dtype", [("bf16", "bf16"), ("bf16", "fp32"), ("fp32", "fp32")])
def test_encode_reduction_axis_longer_than_one_chunk(lla, storage, x_dtype):
    # T*d = 16 * 256 = 4096: 8 chunks of W_down in bf16, 16 in fp32; token tiles of 6
    _encode_and_compare(lla, 16, 2, 256, 96, 160, storage, x_dtype, [13, 1, 7], True, 3)


@pytest.mark.parametrize("r_k,r_v", [(18, 30), (72, 120), (192, 320)])
def test_encode_rank_shapes_and_ragged_tiles(lla, r_k, r_v):
    # 37 tokens: two full tiles of 16 and a ragged tile of 5; r = 18, 30 use 4-byte copies
    _encode_and_compare(lla, 4, 3, 128, r_k, r_v, "bf16", "bf16", [20, 17], False, 4)


def test_encode_fp32_small_ranks(lla):
    _encode_and_compare(lla, 4, 2, 128, 18, 30, "fp32", "fp32", [33], True, 5)


def test_encode_decode_step_batch(lla):
    # the decode-step shape: one completed token for each of 16 sequences, all 16 heads
    _encode_and_compare(lla, 4, 16, 128, 96, 160, "bf16", "bf16", [1] * 16, False, 6)


@pytest.mark.parametrize("r_k,r_v,with_mu", [(96, 160, True), (192, 320, False), (128, 128, True)])
def test_encode_prompt_on_tensor_cores(lla, r_k, r_v, with_mu):
    # 300 tokens in three sequences: three tiles of 128 tokens, the last one ragged (44 tokens)
    _encode_and_compare(lla, 4, 3, 128, r_k, r_v, "bf16", "bf16", [130, 101, 69], with_mu, 7)


@pytest.mark.parametrize("r_k,r_v", [(192, 320), (96, 160)])
def test_encode_prompt_many_units_per_cta(lla, r_k, r_v):
    # 4200 tokens (33 tiles, the last ragged) of 8 heads with mu: every CTA of the persistent
    # kernel takes several (head, tile, column group) units, alternates its two accumulator
    # slots and crosses a head boundary (the bias mu W_down is recomputed there); at (192, 320)
    # the two column groups of the V axis read the same x tile one after the other
    _encode_and_compare(lla, 4, 8, 128, r_k, r_v, "bf16", "bf16", [2000, 1500, 700], True, 10)


def test_encode_prompt_long_reduction_on_tensor_cores(lla):
    # T*d = 16 * 256 = 4096: 64 slabs of the reduction axis through the stage ring
    _encode_and_compare(lla, 16, 2, 256, 96, 160, "bf16", "bf16", [150], True, 8)


@pytest.mark.parametrize("N,storage", [(16, "bf16"), (16, "fp32"), (200, "bf16")])
def test_encode_layers_equals_per_layer_calls(lla, N, storage):
    """lla_encode_layers writes exactly what one lla_encode call per layer writes (one launch
    for a decode batch; prompts go layer by layer through the tensor-core kernel)."""
    from paper_2607_15456_gb300 import workloads as W
    T, H, d, r_k, r_v, L = 4, 16, 128, 96, 160, 3
    geom = lla.Geometry(T, H, d, r_k, r_v, storage)
    pt = W.page_table([N], 9, extra_tokens=0)
    bb = lla.lla_cache_block_bytes(geom)
    slots = pt.slots(0, range(N)).to(DEV)
    table = pt.block_table.to(DEV)
    codecs, caches_a, caches_b, xs_k, xs_v, pools = [], [], [], [], [], []
    for l in range(L):
        cod = W.codec_tensors(T, H, d, r_k, r_v, 9, l, dtype=_dt(storage), device=DEV, with_mu=(l == 1))
        codecs.append(lla.Codec(**cod))
        for lst in (caches_a, caches_b):
            pool = torch.full((pt.num_blocks * bb,), 0xFF, dtype=torch.uint8, device=DEV)
            pools.append(pool)
            lst.append(lla.Cache(pool, pt.num_blocks, table, pt.max_blocks))
        xs_k.append(W.normal((T, N, H, d), 9, 50, l, device=DEV))
        xs_v.append(W.normal((T, N, H, d), 9, 51, l, device=DEV))
    lla.lla_clear_device_error()
    lla.lla_encode_layers(geom, codecs, caches_a, xs_k, xs_v, slots)
    for l in range(L):
        lla.lla_encode(geom, codecs[l], caches_b[l], xs_k[l], xs_v[l], slots)
    torch.cuda.synchronize()
    assert lla.lla_get_device_error() == 0
    for l in range(L):
        assert torch.equal(caches_a[l].pool, caches_b[l].pool), l
