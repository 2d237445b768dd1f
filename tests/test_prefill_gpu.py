"""GPU parity of lla_prefill_attn (causal pass-2 prefill, App. A and App. J) against the oracle.

The cache is filled by lla_encode; the oracle runs causal softmax attention over the explicitly
reconstructed K/V of every key (Eq. decode).  Two comparisons per (sequence, head):
  * against the oracle on its own latents (the full path, bf16 storage tolerance: max abs
    <= 2e-2 beyond the rounding of a bf16 output to its own format, relative L2 <= 5e-3; fp32
    storage: relative L2 <= 1e-5);
  * against the oracle fed the latents the GPU stored, so that only the attention kernel is
    under test (relative L2 <= 5e-3 with bf16 tensor-core operands, 1e-5 in fp32).
Cases reach both code paths (tcgen05 for bf16 storage with ranks multiple of 16, CUDA cores
otherwise), prompts shorter than a page, on page and tile boundaries and across several query
tiles, fp32 and bf16 queries, with and without mu.
"""
import math

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


def _prefill_case(lla, r_k, r_v, storage, io, lens, loop, with_mu, H=2, seed=0):
    sc = Scene(lla, T=4, H=H, d=128, r_k=r_k, r_v=r_v, storage=storage, io=io, lens=lens,
               seed=seed, with_mu=with_mu, extra_tokens=0)
    W = sc.W
    N = sum(lens)
    dt = torch.bfloat16 if io == "bf16" else torch.float32
    q = W.normal((N, H, 128), seed, 60, loop, dtype=dt, device=DEV)
    out = torch.full_like(q, float("nan"))
    cu = torch.tensor(np.cumsum([0] + list(lens)), dtype=torch.int32, device=DEV)
    lla.lla_prefill_attn(sc.geom, sc.codec, sc.cache, cu, max(lens), loop, q, out)
    torch.cuda.synchronize()
    assert lla.lla_get_device_error() == 0
    got, q64 = f64(out), f64(q)
    w = sc.w64
    tight = 1e-5 if storage == "fp32" else 5e-3
    off = 0
    for b, L in enumerate(lens):
        for h in range(H):
            mk = None if w["mu_k"] is None else w["mu_k"][h]
            mv = None if w["mu_v"] is None else w["mu_v"][h]
            args = (w["w_up_k"][h], w["w_up_v"][h], mk, mv, q64[off:off + L, h], sc.scale)
            ref = oracle.prefill(loop, sc.ck[b, h], sc.cv[b, h], *args)
            assert_parity(got[off:off + L, h], ref, storage, f"prefill b{b} h{h}", io=io,
                          output_rounding=True)
            gk, gv = sc.gpu_latents(b, h)
            ref2 = oracle.prefill(loop, gk, gv, *args)
            err = rel_l2(got[off:off + L, h], ref2)
            assert err <= tight, (b, h, err)
        off += L
    return got


@pytest.mark.parametrize("io", ["bf16", "fp32"])
def test_prefill_tensor_core_ragged_prompts(lla, io):
    # 1 token; one page minus one; exactly one page; one more; two tiles plus; three tiles
    _prefill_case(lla, 96, 160, "bf16", io, [1, 63, 64, 65, 130, 300], 2, True)


def test_prefill_tensor_core_rho2_ranks(lla):
    # r_v = 320: the PV product is split in two N = 160 halves
    _prefill_case(lla, 192, 320, "bf16", "bf16", [200, 129], 0, False)


def test_prefill_tensor_core_full_rank(lla):
    _prefill_case(lla, 128, 128, "bf16", "bf16", [257], 1, True)


def test_prefill_long_prompt_rescales(lla):
    # 1500 keys: many pages per tile, so row maxima grow and O is rescaled in TMEM
    _prefill_case(lla, 96, 160, "bf16", "bf16", [1500], 3, False, H=1, seed=5)


def test_prefill_cuda_core_ranks(lla):
    # r = (72, 120): not multiples of 16, served by the CUDA-core kernel
    _prefill_case(lla, 72, 120, "bf16", "bf16", [70, 5], 1, False)


def test_prefill_fp32_storage(lla):
    _prefill_case(lla, 96, 160, "fp32", "fp32", [90, 33], 0, True)


def test_prefill_rejects_bad_context(lla):
    # a prompt longer than max_len is flagged on the device; nothing is written for it
    sc = Scene(lla, T=4, H=1, d=128, r_k=96, r_v=160, storage="bf16", io="bf16", lens=[100],
               seed=9, extra_tokens=0)
    q = torch.zeros((100, 1, 128), dtype=torch.bfloat16, device=DEV)
    out = torch.zeros_like(q)
    cu = torch.tensor([0, 100], dtype=torch.int32, device=DEV)
    lla.lla_clear_device_error()
    lla.lla_prefill_attn(sc.geom, sc.codec, sc.cache, cu, 64, 0, q, out)
    torch.cuda.synchronize()
    assert lla.lla_get_device_error() & 0x2  # LLA_DEVERR_CONTEXT
    lla.lla_clear_device_error()
