"""Seeded synthetic inputs shared by the tests, the benchmark and the smoke check.

This module draws random numbers and does page bookkeeping only; it computes no part of the
method.  Both the CUDA path and the CPU oracle receive exactly the tensors made here.

Workloads (the five shapes the library is measured and checked on; Ouro-shaped per App. A
"Models": T=4 loops, H=16 heads of width 128, D=24 or 48 layers):

  tiny            D=1,  H=4,  (r_k,r_v)=(96,160)  rho=4.00, B=1,   context 256, fp32 inputs
  ouro14_rho4     D=24, H=16, (96,160)  rho=4.00,  B=16,  context ~ U[2048, 4096]
  ouro14_rho2     D=24, H=16, (192,320) rho=2.00,  prefill 4 x 8192, then decode B=32
  ouro26_rho533   D=48, H=16, (72,120)  rho=5.33,  B=64,  context ~ logU[512, 16384]
  stress_rho2133  D=48, H=16, (18,30)   rho=21.33, B=128, context ~ U[8192, 32768]

and the LLA-2D variant (Sec. 3) at the per-head stress workload's cache budget: one latent per
(token, layer) of H times the per-head width, (r_k, r_v) = 16 x (18, 30) = (288, 480), the same
rho_2D = 2 T H d / (r_k + r_v) = 21.33 (Table isocache prints LLA-2D at this ratio):

  stress2d_rho2133  D=48, H=16, (288,480)  B=128, context ~ U[8192, 32768]

and LLA-2D at rho_2D = 5.33 (also printed in Table isocache), (r_k, r_v) = (1152, 1920), on the
Ouro-1.4B headline batch:

  ouro14_2d_rho533  D=24, H=16, (1152,1920) B=16, context ~ U[2048, 4096]

Recipe: activations, queries and current-token K/V are N(0,1); W_down is N(0, 1/(T d)) and
W_up,t is N(0, 1/r) (std = 1/sqrt(.)); for LLA-2D W_down is N(0, 1/(T H d)) and W_up,t,h
N(0, 1/r); mu = 0 unless asked for (then N(0,1)); seeds are the
workload's index (tiny = 0).  Context lengths are integers drawn uniformly (or log-uniformly,
floor(exp(U[ln lo, ln hi]))) over the inclusive range and are not rounded to the 64-token page
grid.  Physical blocks come from a shuffled free list, so every sequence's pages are scattered
through the pool as under a real allocator, and no page is shared between sequences.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import List, Optional, Tuple

import torch

BLOCK = 64


@dataclass(frozen=True)
class Workload:
    name: str
    D: int
    H: int
    d: int
    T: int
    r_k: int
    r_v: int
    B: int
    lens: Tuple  # ("fixed", L) | ("uniform", lo, hi) | ("loguniform", lo, hi)
    seed: int
    storage: str = "bf16"
    io: str = "bf16"
    prefill: Optional[Tuple[int, int]] = None  # (sequences, tokens each)
    decode_steps: int = 1
    lla2d: bool = False  # one latent per (token, layer) for all heads (Sec. 3, LLA-2D)

    @property
    def rho(self) -> float:
        return 2 * self.T * self.d * (self.H if self.lla2d else 1) / (self.r_k + self.r_v)


WORKLOADS = {
    "tiny": Workload("tiny", D=1, H=4, d=128, T=4, r_k=96, r_v=160, B=1, lens=("fixed", 256),
                     seed=0, storage="bf16", io="fp32"),
    "ouro14_rho4": Workload("ouro14_rho4", D=24, H=16, d=128, T=4, r_k=96, r_v=160, B=16,
                            lens=("uniform", 2048, 4096), seed=1),
    "ouro14_rho2": Workload("ouro14_rho2", D=24, H=16, d=128, T=4, r_k=192, r_v=320, B=32,
                            lens=("fixed", 8192), seed=2, prefill=(4, 8192), decode_steps=256),
    "ouro26_rho533": Workload("ouro26_rho533", D=48, H=16, d=128, T=4, r_k=72, r_v=120, B=64,
                              lens=("loguniform", 512, 16384), seed=3),
    "stress_rho2133": Workload("stress_rho2133", D=48, H=16, d=128, T=4, r_k=18, r_v=30, B=128,
                               lens=("uniform", 8192, 32768), seed=4),
    "stress2d_rho2133": Workload("stress2d_rho2133", D=48, H=16, d=128, T=4, r_k=288, r_v=480,
                                 B=128, lens=("uniform", 8192, 32768), seed=4, lla2d=True),
    "ouro14_2d_rho533": Workload("ouro14_2d_rho533", D=24, H=16, d=128, T=4, r_k=1152, r_v=1920,
                                 B=16, lens=("uniform", 2048, 4096), seed=1, lla2d=True),
}


def _gen(*key: int) -> torch.Generator:
    """CPU generator seeded from a tuple of small non-negative integers."""
    s = 0
    for k in key:
        s = (s * 1000003 + int(k) + 1) % (2**61 - 1)
    return torch.Generator().manual_seed(s)


def context_lengths(w: Workload, B: Optional[int] = None) -> List[int]:
    B = w.B if B is None else B
    g = _gen(w.seed, 1)
    kind = w.lens[0]
    if kind == "fixed":
        return [int(w.lens[1])] * B
    lo, hi = w.lens[1], w.lens[2]
    if kind == "uniform":
        return [int(v) for v in torch.randint(lo, hi + 1, (B,), generator=g)]
    if kind == "loguniform":
        u = torch.rand(B, generator=g, dtype=torch.float64)
        return [int(math.floor(math.exp(math.log(lo) + float(x) * (math.log(hi) - math.log(lo)))))
                for x in u]
    raise ValueError(kind)


def codec_tensors(T: int, H: int, d: int, r_k: int, r_v: int, seed: int, layer: int,
                  dtype=torch.bfloat16, device="cpu", with_mu: bool = False, mu_seed: int = 1):
    """W_down [H][T*d][r] ~ N(0, 1/(T d)), W_up [H][T][d][r] ~ N(0, 1/r), drawn head by head,
    axis K then V, W_down then W_up,0..T-1.  mu [H][T*d] ~ N(0, 1) fp32 when asked for."""
    g = _gen(seed, 2, layer)
    Td = T * d
    wd = {"k": torch.empty(H, Td, r_k), "v": torch.empty(H, Td, r_v)}
    wu = {"k": torch.empty(H, T, d, r_k), "v": torch.empty(H, T, d, r_v)}
    for h in range(H):
        for ax, r in (("k", r_k), ("v", r_v)):
            wd[ax][h] = torch.randn(Td, r, generator=g) / math.sqrt(Td)
            for t in range(T):
                wu[ax][h, t] = torch.randn(d, r, generator=g) / math.sqrt(r)
    out = dict(w_down_k=wd["k"], w_down_v=wd["v"], w_up_k=wu["k"], w_up_v=wu["v"],
               mu_k=None, mu_v=None)
    if with_mu:
        gm = _gen(seed, 3, layer, mu_seed)
        out["mu_k"] = torch.randn(H, Td, generator=gm)
        out["mu_v"] = torch.randn(H, Td, generator=gm)
    for k in ("w_down_k", "w_down_v", "w_up_k", "w_up_v"):
        out[k] = out[k].to(dtype).to(device).contiguous()
    for k in ("mu_k", "mu_v"):
        if out[k] is not None:
            out[k] = out[k].to(torch.float32).to(device).contiguous()
    return out


def codec_tensors_2d(T: int, H: int, d: int, r_k: int, r_v: int, seed: int, layer: int,
                     dtype=torch.bfloat16, device="cpu", with_mu: bool = False, mu_seed: int = 1):
    """LLA-2D codec of one layer: W_down [T*H*d][r] ~ N(0, 1/(T H d)) (rows ordered (t, h, e)),
    W_up [T][H][d][r] ~ N(0, 1/r), axis K then V, W_down then W_up,t,h in (t, h) order.
    mu [T*H*d] ~ N(0, 1) fp32 when asked for."""
    g = _gen(seed, 6, layer)
    S = T * H * d
    out = dict(mu_k=None, mu_v=None)
    for ax, r in (("k", r_k), ("v", r_v)):
        out["w_down_" + ax] = torch.randn(S, r, generator=g) / math.sqrt(S)
        out["w_up_" + ax] = torch.randn(T, H, d, r, generator=g) / math.sqrt(r)
    if with_mu:
        gm = _gen(seed, 7, layer, mu_seed)
        out["mu_k"] = torch.randn(S, generator=gm)
        out["mu_v"] = torch.randn(S, generator=gm)
    for k in ("w_down_k", "w_down_v", "w_up_k", "w_up_v"):
        out[k] = out[k].to(dtype).to(device).contiguous()
    for k in ("mu_k", "mu_v"):
        if out[k] is not None:
            out[k] = out[k].to(torch.float32).to(device).contiguous()
    return out


def normal(shape, seed: int, *key: int, dtype=torch.bfloat16, device="cpu") -> torch.Tensor:
    """N(0,1) tensor; drawn on `device` with a generator of that device."""
    s = _gen(seed, 4, *key).initial_seed()
    g = torch.Generator(device=device).manual_seed(s)
    return torch.randn(shape, generator=g, device=device, dtype=torch.float32).to(dtype)


@dataclass
class PageTable:
    block_table: torch.Tensor  # [B][max_blocks] int32, -1 where unused
    num_blocks: int
    max_blocks: int
    capacity: List[int] = field(default_factory=list)  # tokens each row can hold

    def slots(self, b: int, positions) -> torch.Tensor:
        """Slot ids (block * 64 + row) of the given positions of sequence b (int64, CPU)."""
        pos = torch.as_tensor(positions, dtype=torch.int64)
        blocks = self.block_table[b].to(torch.int64)[pos // BLOCK]
        return blocks * BLOCK + pos % BLOCK


def page_table(lens: List[int], seed: int, extra_tokens: int = 1, spare_blocks: int = 0,
               max_blocks: Optional[int] = None) -> PageTable:
    """Scattered physical pages: each sequence gets ceil((L + extra)/64) blocks taken in order
    from a shuffled free list of all blocks."""
    need = [max(1, -(-(L + extra_tokens) // BLOCK)) for L in lens]
    total = sum(need) + spare_blocks
    mb = max(need) if max_blocks is None else max_blocks
    perm = torch.randperm(total, generator=_gen(seed, 5)).to(torch.int32)
    table = torch.full((len(lens), mb), -1, dtype=torch.int32)
    o = 0
    for b, n in enumerate(need):
        table[b, :n] = perm[o:o + n]
        o += n
    return PageTable(table, total, mb, [n * BLOCK for n in need])


def pack_latent_pages(c_k: torch.Tensor, c_v: torch.Tensor, table: torch.Tensor, lens: List[int],
                      num_blocks: int) -> torch.Tensor:
    """A one-page-per-block cache pool (uint8, on c_k's device) holding given bf16 latents:
    c_k [N][r_k], c_v [N][r_v] of the sequences back to back, token p of sequence b in block
    table[b][p // 64], row p % 64.  Layout of include/lla.h: the K-plane in 16-byte granules of
    8 columns (granule g of row i at g*1024 + i*16), the V-plane row-major; rows past a
    sequence are zero."""
    r_k, r_v = c_k.shape[1], c_v.shape[1]
    dev = c_k.device
    page = BLOCK * (r_k + r_v) * 2
    pool = torch.zeros((num_blocks, page), dtype=torch.uint8, device=dev)
    off = 0
    for b, L in enumerate(lens):
        n = -(-L // BLOCK)
        if n == 0:
            continue
        kp = torch.zeros((n * BLOCK, r_k), dtype=torch.bfloat16, device=dev)
        vp = torch.zeros((n * BLOCK, r_v), dtype=torch.bfloat16, device=dev)
        kp[:L] = c_k[off:off + L]
        vp[:L] = c_v[off:off + L]
        kg = kp.view(n, BLOCK, r_k // 8, 8).permute(0, 2, 1, 3).contiguous().view(n, -1)
        blocks = table[b, :n].to(torch.int64).to(dev)
        pool[blocks, :BLOCK * r_k * 2] = kg.view(torch.uint8)
        pool[blocks, BLOCK * r_k * 2:] = vp.view(n, -1).view(torch.uint8)
        off += L
    return pool.view(-1)


def random_pool(num_bytes: int, seed: int, *key: int, device="cpu", chunk: int = 1 << 30) -> torch.Tensor:
    """A cache pool (uint8, num_bytes a multiple of 2) whose every bf16 element is an N(0,1)
    draw: valid latents in every position of every page, whatever the layout, for timing decode
    over a full-size cache without encoding it.  Drawn in chunks of `chunk` elements."""
    pool = torch.empty(num_bytes, dtype=torch.uint8, device=device)
    flat = pool.view(torch.bfloat16)
    s = _gen(seed, 8, *key).initial_seed()
    g = torch.Generator(device=device).manual_seed(s)
    for o in range(0, flat.numel(), chunk):
        n = min(chunk, flat.numel() - o)
        flat[o:o + n] = torch.randn(n, generator=g, device=device, dtype=torch.float32).to(torch.bfloat16)
    return pool
