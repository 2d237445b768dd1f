"""Test-side helpers: reading the paged cache layout documented in include/lla.h back into
logical latents, tolerance checks, and building the library once per session.

This file is test infrastructure.  It shares no code with the CUDA library (it re-reads the
layout from its documented formula) nor with the oracle (it does no attention arithmetic).
"""
from __future__ import annotations

import math

import numpy as np
import torch

BLOCK = 64

# Tolerances for GPU vs oracle (float64): bf16 storage with fp32 accumulation, and fp32 mode.
BF16_MAX_ABS = 2e-2
BF16_REL_L2 = 5e-3
F32_REL_L2 = 1e-5


def rel_l2(a, b) -> float:
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    den = np.linalg.norm(b.ravel())
    return float(np.linalg.norm((a - b).ravel()) / (den if den > 0 else 1.0))


def bf16_half_ulp(x):
    """Half the spacing of bf16 numbers at |x| (the largest error of rounding x to bf16)."""
    a = np.abs(np.asarray(x, dtype=np.float64))
    e = np.floor(np.log2(np.maximum(a, np.finfo(np.float32).tiny)))
    return np.ldexp(1.0, (e - 8).astype(np.int64))


def assert_parity(gpu, ref, storage: str, what: str = "", io: str = "bf16",
                  output_rounding: bool = False):
    """bf16 storage or io: max abs <= 2e-2 and relative L2 <= 5e-3; fp32: relative L2 <= 1e-5.
    With output_rounding (bf16 outputs), the max-abs bound applies to the value before its final
    rounding to bf16: |gpu - ref| <= 2e-2 + half a bf16 ulp of ref."""
    gpu = np.asarray(gpu, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert gpu.shape == ref.shape, (gpu.shape, ref.shape)
    assert np.isfinite(gpu).all(), f"{what}: non-finite GPU output"
    dev = np.abs(gpu - ref)
    if output_rounding and io == "bf16":
        dev = dev - bf16_half_ulp(ref)
    err_max = float(dev.max()) if gpu.size else 0.0
    err_l2 = rel_l2(gpu, ref)
    if storage == "bf16" or io == "bf16":
        assert err_max <= BF16_MAX_ABS and err_l2 <= BF16_REL_L2, (what, err_max, err_l2)
    else:
        assert err_l2 <= F32_REL_L2, (what, err_max, err_l2)
    return err_max, err_l2


def es_of(storage: str) -> int:
    return 2 if storage == "bf16" else 4


def granule(r: int, es: int) -> int:
    return 16 if (r * es) % 16 == 0 else 4


def unpack_head(pool_u8: torch.Tensor, H: int, r_k: int, r_v: int, storage: str,
                table_row, L: int, h: int):
    """Latents (c_k [L][r_k], c_v [L][r_v], float64 numpy) of the first L positions of one
    sequence and head, read from a CPU copy of the pool per the layout in include/lla.h."""
    es = es_of(storage)
    dt = torch.bfloat16 if storage == "bf16" else torch.float32
    hpb = BLOCK * (r_k + r_v) * es
    kplane = BLOCK * r_k * es
    gk = granule(r_k, es)
    ck = np.zeros((L, r_k))
    cv = np.zeros((L, r_v))
    for p in range(math.ceil(L / BLOCK)):
        blk = int(table_row[p])
        base = blk * H * hpb + h * hpb
        page = pool_u8[base:base + hpb]
        kp = page[:kplane].reshape(r_k * es // gk, BLOCK, gk).permute(1, 0, 2)
        kp = kp.reshape(BLOCK, r_k * es).contiguous().view(dt).to(torch.float64).numpy()
        vp = page[kplane:].reshape(BLOCK, r_v * es).contiguous().view(dt)
        vp = vp.to(torch.float64).numpy()
        n = min(BLOCK, L - p * BLOCK)
        ck[p * BLOCK:p * BLOCK + n] = kp[:n]
        cv[p * BLOCK:p * BLOCK + n] = vp[:n]
    return ck, cv


def f64(t: torch.Tensor) -> np.ndarray:
    return t.detach().to("cpu").to(torch.float64).numpy()


_built = False


def ensure_library():
    global _built
    if not _built:
        from paper_2607_15456_gb300 import build
        build.build()
        _built = True
