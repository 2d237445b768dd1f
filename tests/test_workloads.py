"""The seeded input generators and page bookkeeping (no GPU): the page packer writes the layout
of include/lla.h that the test helper reads back, the LLA-2D codec has the recipe's shapes and
scales, and the workloads' ratios follow Eq. ratio (per head) and rho_2D (LLA-2D)."""
import math

import numpy as np
import torch

import oracle
from helpers import unpack_head
from paper_2607_15456_gb300 import workloads as W


def test_packed_pages_read_back_in_the_documented_layout():
    lens = [5, 64, 130, 0, 1]
    pt = W.page_table(lens, 3)
    N = sum(lens)
    g = torch.Generator().manual_seed(0)
    ck = torch.randn(N, 96, generator=g).to(torch.bfloat16)
    cv = torch.randn(N, 160, generator=g).to(torch.bfloat16)
    pool = W.pack_latent_pages(ck, cv, pt.block_table, lens, pt.num_blocks)
    assert pool.numel() == pt.num_blocks * 64 * (96 + 160) * 2
    off = 0
    for b, L in enumerate(lens):
        gk, gv = unpack_head(pool, 1, 96, 160, "bf16", pt.block_table[b], L, 0)
        assert np.array_equal(gk, ck[off:off + L].double().numpy())
        assert np.array_equal(gv, cv[off:off + L].double().numpy())
        off += L


def test_2d_codec_shapes_and_scales():
    c = W.codec_tensors_2d(4, 16, 128, 288, 480, seed=4, layer=0, dtype=torch.float32, with_mu=True)
    assert c["w_down_k"].shape == (4 * 16 * 128, 288) and c["w_down_v"].shape == (8192, 480)
    assert c["w_up_k"].shape == (4, 16, 128, 288) and c["w_up_v"].shape == (4, 16, 128, 480)
    assert c["mu_k"].shape == (8192,) and c["mu_k"].dtype == torch.float32
    # std 1/sqrt(T H d) and 1/sqrt(r), to a few percent over ~2.4 M draws
    assert abs(c["w_down_k"].std().item() * math.sqrt(8192) - 1) < 0.02
    assert abs(c["w_up_v"].std().item() * math.sqrt(480) - 1) < 0.02
    again = W.codec_tensors_2d(4, 16, 128, 288, 480, seed=4, layer=0, dtype=torch.float32, with_mu=True)
    assert torch.equal(c["w_up_k"], again["w_up_k"])  # seeded


def test_workload_ratios():
    for w in W.WORKLOADS.values():
        if w.lla2d:
            assert abs(w.rho - oracle.ratio_2d(w.T, w.H, w.d, w.r_k, w.r_v)) < 1e-12
        else:
            assert abs(w.rho - oracle.ratio(w.T, w.d, w.r_k, w.r_v)) < 1e-12
    assert abs(W.WORKLOADS["stress2d_rho2133"].rho - W.WORKLOADS["stress_rho2133"].rho) < 1e-12
