"""Thin Python binding of liblla (include/lla.h): argument marshalling only.

Every function here has the name of the C entry point it calls and does nothing but turn
torch tensors into device pointers, fill the ABI structs and raise ``LLAError`` on a non-zero
status.  All computation happens in the CUDA kernels of liblla.so; there is no fallback: if
the library is missing or a call fails, an exception is raised.
"""
from __future__ import annotations

import ctypes
import math
import os
from dataclasses import dataclass
from typing import Optional

import torch

from .build import LIB

LLA_BLOCK_TOKENS = 64
LLA_MAX_BATCH = 1024
LLA_BF16, LLA_F32 = 0, 1
LLA_ROPE_HALF, LLA_ROPE_ADJACENT = 0, 1
LLA_DEVERR_BLOCK_ID = 0x1
LLA_DEVERR_CONTEXT = 0x2
LLA_DEVERR_EMPTY_PASS2 = 0x4
LLA_DEVERR_TIMEOUT = 0x8
LLA_DEVERR_SLOT = 0x10

_STATUS = {0: "LLA_OK", 1: "LLA_ERR_INVALID_ARG", 2: "LLA_ERR_UNSUPPORTED", 3: "LLA_ERR_CUDA",
           4: "LLA_ERR_TIMEOUT", 5: "LLA_ERR_DEVICE_CHECK", 6: "LLA_ERR_WORKSPACE"}


class LLAError(RuntimeError):
    def __init__(self, fn: str, status: int):
        self.status = status
        super().__init__(f"{fn} returned {_STATUS.get(status, status)}")


class lla_geometry(ctypes.Structure):
    _fields_ = [("T", ctypes.c_int32), ("H", ctypes.c_int32), ("d", ctypes.c_int32),
                ("r_k", ctypes.c_int32), ("r_v", ctypes.c_int32), ("block_size", ctypes.c_int32),
                ("storage", ctypes.c_int32), ("scale", ctypes.c_float)]


class lla_codec(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in
                ("w_down_k", "w_down_v", "w_up_k", "w_up_v", "mu_k", "mu_v")]


class lla_rope(ctypes.Structure):
    _fields_ = [("base", ctypes.c_double), ("pairing", ctypes.c_int32)]


class lla_cache(ctypes.Structure):
    _fields_ = [("pool", ctypes.c_void_p), ("num_blocks", ctypes.c_int64),
                ("block_table", ctypes.c_void_p), ("max_blocks_per_seq", ctypes.c_int32)]


# lla_capture_fn and lla_query_fn of include/lla.h
CAPTURE_FN = ctypes.CFUNCTYPE(ctypes.c_int32, ctypes.c_int32, ctypes.POINTER(ctypes.c_void_p),
                              ctypes.POINTER(ctypes.c_void_p), ctypes.c_void_p, ctypes.c_void_p)
QUERY_FN = ctypes.CFUNCTYPE(ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,
                            ctypes.POINTER(ctypes.c_void_p), ctypes.POINTER(ctypes.c_void_p),
                            ctypes.c_void_p, ctypes.c_void_p)

_lib = None


def library() -> ctypes.CDLL:
    """Loads liblla.so from the package directory (built by ``__graft_entry__.build()``)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB):
            raise RuntimeError(f"liblla.so not found at {LIB}: build it first "
                               "(python -c 'import __graft_entry__ as g; g.build()')")
        lib = ctypes.CDLL(LIB)
        P, I32, I64, SZ = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t
        sig = {
            "lla_status_string": (ctypes.c_char_p, [I32]),
            "lla_version": (I32, []),
            "lla_cache_block_bytes": (I32, [P, P]),
            "lla_encode": (I32, [P, P, P, P, P, I32, P, I32, P]),
            "lla_encode_layers": (I32, [P, I32, P, P, P, P, I32, P, I32, P]),
            "lla_decode_workspace_size": (I32, [P, I32, P]),
            "lla_decode_workspace_init": (I32, [P, SZ, P]),
            "lla_decode_attn": (I32, [P, P, P, P, I32, I32, I32, P, P, P, I32, P, P, SZ, P]),
            "lla_decode_attn_noalloc": (I32, [P, P, P, P, I32, I32, I32, P, P, P, I32, P, P]),
            "lla_decode_attn_rope": (I32, [P, P, P, P, P, I32, I32, I32, P, P, P, I32, P, P, SZ,
                                           P]),
            "lla_decode_loops_workspace_size": (I32, [P, I32, P]),
            "lla_decode_attn_loops": (I32, [P, P, P, P, I32, I32, P, P, P, I32, P, P, SZ, P]),
            "lla_prefill_attn": (I32, [P, P, P, P, I32, I32, I32, P, I32, P, P]),
            "lla_prefill_rope_workspace_size": (I32, [P, I32, I32, P]),
            "lla_prefill_attn_rope": (I32, [P, P, P, P, P, I32, I32, I32, P, I32, P, P, SZ, P]),
            "lla_dense_store": (I32, [P, P, P, P, I32, P, I32, P]),
            "lla_dense_decode_attn": (I32, [P, P, P, I32, I32, P, P, P, I32, P, P, SZ, P]),
            "lla_cache_2d_block_bytes": (I32, [P, P]),
            "lla_encode_2d": (I32, [P, P, P, P, P, I32, P, I32, P]),
            "lla_decode_2d_workspace_size": (I32, [P, I32, P]),
            "lla_decode_attn_2d": (I32, [P, P, P, P, I32, I32, I32, P, P, P, I32, P, P, SZ, P]),
            "lla_rope_plane_bytes": (I32, [I32, P]),
            "lla_encode_rope_keys": (I32, [I32, P, P, I64, P, I32, P, P, I32, P]),
            "lla_decode_decoupled_workspace_size": (I32, [P, I32, I32, P]),
            "lla_decode_attn_decoupled": (I32, [P, P, P, P, I32, P, P, I32, I32, I32, P, P, P, P, P, I32,
                                                P, P, SZ, P]),
            "lla_get_device_error": (I32, [P, P]),
            "lla_clear_device_error": (I32, [P]),
            "lla_prefill_two_pass": (I32, [P, I32, P, P, I32, P, I32, P, I32, I32, I32, P, CAPTURE_FN,
                                           QUERY_FN, P, P, SZ, P]),
            "lla_set_wait_limit_ns": (I32, [ctypes.c_uint64]),
            "lla_get_wait_limit_ns": (ctypes.c_uint64, []),
        }
        for name, (res, args) in sig.items():
            fn = getattr(lib, name)
            fn.restype, fn.argtypes = res, args
        _lib = lib
    return _lib


def _check(fn: str, status: int):
    if status != 0:
        raise LLAError(fn, status)


def _ptr(t: Optional[torch.Tensor]):
    if t is None:
        return None
    if isinstance(t, int):
        return t
    if not t.is_contiguous():
        raise ValueError("tensors passed to liblla must be contiguous")
    if not t.is_cuda:
        # every buffer of the ABI is a device buffer: a host address would fault the kernel
        raise ValueError("tensors passed to liblla must be CUDA tensors")
    return t.data_ptr()


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return LLA_BF16
    if t.dtype == torch.float32:
        return LLA_F32
    raise ValueError(f"unsupported dtype {t.dtype}")


def _stream(stream) -> Optional[int]:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


@dataclass
class Geometry:
    T: int
    H: int
    d: int
    r_k: int
    r_v: int
    storage: str = "bf16"
    scale: Optional[float] = None

    def c(self) -> lla_geometry:
        scale = self.scale if self.scale is not None else 1.0 / math.sqrt(self.d)
        return lla_geometry(self.T, self.H, self.d, self.r_k, self.r_v, LLA_BLOCK_TOKENS,
                            LLA_BF16 if self.storage == "bf16" else LLA_F32, scale)

    @property
    def torch_dtype(self):
        return torch.bfloat16 if self.storage == "bf16" else torch.float32


@dataclass
class Codec:
    """Codec of one layer: w_down_* [H][T*d][r], w_up_* [H][T][d][r], mu_* [H][T*d] fp32."""
    w_down_k: torch.Tensor
    w_down_v: torch.Tensor
    w_up_k: torch.Tensor
    w_up_v: torch.Tensor
    mu_k: Optional[torch.Tensor] = None
    mu_v: Optional[torch.Tensor] = None

    def c(self) -> lla_codec:
        return lla_codec(*(_ptr(t) for t in (self.w_down_k, self.w_down_v, self.w_up_k,
                                             self.w_up_v, self.mu_k, self.mu_v)))


@dataclass
class Cache:
    """Paged cache of one layer: pool (uint8 or any dtype, 16-byte aligned), block table
    [B][max_blocks_per_seq] int32."""
    pool: torch.Tensor
    num_blocks: int
    block_table: Optional[torch.Tensor]
    max_blocks_per_seq: int

    def c(self) -> lla_cache:
        return lla_cache(_ptr(self.pool), self.num_blocks, _ptr(self.block_table),
                         self.max_blocks_per_seq)


def lla_status_string(status: int) -> str:
    return library().lla_status_string(status).decode()


def lla_version() -> int:
    return library().lla_version()


def lla_cache_block_bytes(geom: Geometry) -> int:
    out = ctypes.c_size_t(0)
    g = geom.c()
    _check("lla_cache_block_bytes",
           library().lla_cache_block_bytes(ctypes.byref(g), ctypes.byref(out)))
    return out.value


def lla_encode(geom: Geometry, codec: Codec, cache: Cache, x_k: torch.Tensor, x_v: torch.Tensor,
               slot_mapping: torch.Tensor, stream=None) -> None:
    """x_k, x_v [T][N][H][d] (bf16 or fp32); slot_mapping [N] int64."""
    g, cd, ch = geom.c(), codec.c(), cache.c()
    N = x_k.shape[1] if x_k.dim() == 4 else 0
    _check("lla_encode", library().lla_encode(
        ctypes.byref(g), ctypes.byref(cd), ctypes.byref(ch), _ptr(x_k), _ptr(x_v),
        _dtype_code(x_k), _ptr(slot_mapping), N, _stream(stream)))


def lla_encode_layers(geom: Geometry, codecs, caches, x_k, x_v, slot_mapping: torch.Tensor,
                      stream=None) -> None:
    """The same encode in several layers at once: codecs, caches, x_k, x_v are per-layer lists
    (x_k[l], x_v[l] [T][N][H][d]); slot_mapping [N] int64 is shared."""
    L = len(codecs)
    if not (len(caches) == len(x_k) == len(x_v) == L):
        raise ValueError("one codec, cache and input pair per layer")
    g = geom.c()
    cds = (lla_codec * max(L, 1))(*[c.c() for c in codecs])
    chs = (lla_cache * max(L, 1))(*[c.c() for c in caches])
    xk = (ctypes.c_void_p * max(L, 1))(*[_ptr(t) for t in x_k])
    xv = (ctypes.c_void_p * max(L, 1))(*[_ptr(t) for t in x_v])
    N = x_k[0].shape[1] if L and x_k[0].dim() == 4 else 0
    _check("lla_encode_layers", library().lla_encode_layers(
        ctypes.byref(g), L, cds, chs, xk, xv, _dtype_code(x_k[0]) if L else 0, _ptr(slot_mapping), N,
        _stream(stream)))


def lla_decode_workspace_size(geom: Geometry, B: int) -> int:
    out = ctypes.c_size_t(0)
    g = geom.c()
    _check("lla_decode_workspace_size",
           library().lla_decode_workspace_size(ctypes.byref(g), B, ctypes.byref(out)))
    return out.value


def lla_decode_workspace_init(workspace: torch.Tensor, stream=None) -> None:
    nbytes = workspace.numel() * workspace.element_size()
    _check("lla_decode_workspace_init",
           library().lla_decode_workspace_init(_ptr(workspace), nbytes, _stream(stream)))


def lla_decode_attn(geom: Geometry, codec: Codec, cache: Cache, context_lens: torch.Tensor,
                    max_ctx: int, loop: int, q: torch.Tensor, cur_k: Optional[torch.Tensor],
                    cur_v: Optional[torch.Tensor], out: torch.Tensor, workspace: torch.Tensor,
                    stream=None) -> None:
    """q, cur_k, cur_v, out [B][H][d]; cur_k = cur_v = None selects pass 2."""
    g, cd, ch = geom.c(), codec.c(), cache.c()
    B = q.shape[0]
    _check("lla_decode_attn", library().lla_decode_attn(
        ctypes.byref(g), ctypes.byref(cd), ctypes.byref(ch), _ptr(context_lens), B, max_ctx,
        loop, _ptr(q), _ptr(cur_k), _ptr(cur_v), _dtype_code(q), _ptr(out), _ptr(workspace),
        workspace.numel() * workspace.element_size(), _stream(stream)))


def lla_decode_attn_rope(geom: Geometry, codec: Codec, cache: Cache, rope_base: float,
                         rope_pairing: int, context_lens: torch.Tensor, max_ctx: int, loop: int,
                         q: torch.Tensor, cur_k: Optional[torch.Tensor],
                         cur_v: Optional[torch.Tensor], out: torch.Tensor,
                         workspace: torch.Tensor, stream=None) -> None:
    """lla_decode_attn with RoPE after reconstruction; q and cur_k pre-RoPE.  rope_pairing:
    LLA_ROPE_HALF (pairs (j, j + d/2)) or LLA_ROPE_ADJACENT (pairs (2j, 2j + 1))."""
    g, cd, ch = geom.c(), codec.c(), cache.c()
    rp = lla_rope(float(rope_base), int(rope_pairing))
    _check("lla_decode_attn_rope", library().lla_decode_attn_rope(
        ctypes.byref(g), ctypes.byref(cd), ctypes.byref(ch), ctypes.byref(rp),
        _ptr(context_lens), q.shape[0], max_ctx, loop, _ptr(q), _ptr(cur_k), _ptr(cur_v),
        _dtype_code(q), _ptr(out), _ptr(workspace), workspace.numel() * workspace.element_size(),
        _stream(stream)))


def lla_decode_loops_workspace_size(geom: Geometry, B: int) -> int:
    g = geom.c()
    out = ctypes.c_size_t()
    _check("lla_decode_loops_workspace_size",
           library().lla_decode_loops_workspace_size(ctypes.byref(g), B, ctypes.byref(out)))
    return out.value


def lla_decode_attn_loops(geom: Geometry, codec: Codec, cache: Cache, context_lens: torch.Tensor,
                          max_ctx: int, q: torch.Tensor, cur_k: Optional[torch.Tensor],
                          cur_v: Optional[torch.Tensor], out: torch.Tensor,
                          workspace: torch.Tensor, stream=None) -> None:
    """All T loops' decode calls in one pass over the latents: q, cur_k, cur_v, out [T][B][H][d]."""
    g, cd, ch = geom.c(), codec.c(), cache.c()
    _check("lla_decode_attn_loops", library().lla_decode_attn_loops(
        ctypes.byref(g), ctypes.byref(cd), ctypes.byref(ch), _ptr(context_lens), q.shape[1],
        max_ctx, _ptr(q), _ptr(cur_k), _ptr(cur_v), _dtype_code(q), _ptr(out), _ptr(workspace),
        workspace.numel() * workspace.element_size(), _stream(stream)))


def lla_decode_attn_noalloc(geom: Geometry, codec: Codec, cache: Cache,
                            context_lens: torch.Tensor, max_ctx: int, loop: int,
                            q: torch.Tensor, cur_k: Optional[torch.Tensor],
                            cur_v: Optional[torch.Tensor], out: torch.Tensor,
                            stream=None) -> None:
    """lla_decode_attn with the library's own 1 MiB device scratch instead of a caller
    workspace, for callers that cannot allocate device memory (see include/lla.h)."""
    g, cd, ch = geom.c(), codec.c(), cache.c()
    _check("lla_decode_attn_noalloc", library().lla_decode_attn_noalloc(
        ctypes.byref(g), ctypes.byref(cd), ctypes.byref(ch), _ptr(context_lens), q.shape[0],
        max_ctx, loop, _ptr(q), _ptr(cur_k), _ptr(cur_v), _dtype_code(q), _ptr(out),
        _stream(stream)))


def lla_prefill_attn(geom: Geometry, codec: Codec, cache: Cache, cu_seqlens: torch.Tensor,
                     max_len: int, loop: int, q: torch.Tensor, out: torch.Tensor,
                     stream=None) -> None:
    """q, out [Ntok][H][d]; cu_seqlens [B+1] int32."""
    g, cd, ch = geom.c(), codec.c(), cache.c()
    B = cu_seqlens.shape[0] - 1
    _check("lla_prefill_attn", library().lla_prefill_attn(
        ctypes.byref(g), ctypes.byref(cd), ctypes.byref(ch), _ptr(cu_seqlens), B, max_len, loop,
        _ptr(q), _dtype_code(q), _ptr(out), _stream(stream)))


def lla_prefill_rope_workspace_size(geom: Geometry, B: int, max_len: int) -> int:
    g = geom.c()
    out = ctypes.c_size_t()
    _check("lla_prefill_rope_workspace_size",
           library().lla_prefill_rope_workspace_size(ctypes.byref(g), B, max_len, ctypes.byref(out)))
    return out.value


def lla_prefill_attn_rope(geom: Geometry, codec: Codec, cache: Cache, rope_base: float,
                          rope_pairing: int, cu_seqlens: torch.Tensor, max_len: int, loop: int,
                          q: torch.Tensor, out: torch.Tensor, workspace: torch.Tensor,
                          stream=None) -> None:
    """lla_prefill_attn with RoPE after reconstruction; q pre-RoPE [Ntok][H][d]."""
    g, cd, ch = geom.c(), codec.c(), cache.c()
    rp = lla_rope(float(rope_base), int(rope_pairing))
    B = cu_seqlens.shape[0] - 1
    _check("lla_prefill_attn_rope", library().lla_prefill_attn_rope(
        ctypes.byref(g), ctypes.byref(cd), ctypes.byref(ch), ctypes.byref(rp), _ptr(cu_seqlens), B,
        max_len, loop, _ptr(q), _dtype_code(q), _ptr(out), _ptr(workspace),
        workspace.numel() * workspace.element_size(), _stream(stream)))


def lla_prefill_two_pass(geom: Geometry, codecs, caches, slot_mapping: torch.Tensor,
                         cu_seqlens: torch.Tensor, max_len: int, capture, query,
                         x_dtype=torch.bfloat16, io_dtype=torch.bfloat16, rope_base=None,
                         rope_pairing: int = LLA_ROPE_HALF, workspace: Optional[torch.Tensor] = None,
                         stream=None) -> None:
    """Two-pass prefill of len(cu_seqlens) - 1 prompts through len(codecs) layers, streamed layer
    by layer.  capture(layer) returns layer's pass-1 (x_k, x_v) [T][N][H][d]; query(layer, loop)
    returns (q, out) [N][H][d].  Both are called from inside the C call, in its order; the
    tensors they return are kept alive until it returns (stream order covers the rest).
    rope_base None: positions-free content path; else RoPE after reconstruction (workspace of
    lla_prefill_rope_workspace_size bytes)."""
    D = len(codecs)
    if len(caches) != D:
        raise ValueError("one cache per codec")
    cds = (lla_codec * max(D, 1))(*[c.c() for c in codecs])
    chs = (lla_cache * max(D, 1))(*[c.c() for c in caches])
    g = geom.c()
    keep, errors = [], []

    def _capture(layer, pk, pv, _stream_, _user):
        try:
            xk, xv = capture(layer)
            keep.append((xk, xv))
            pk[0], pv[0] = _ptr(xk), _ptr(xv)
            return 0
        except Exception as e:  # reported after the C call returns
            errors.append(e)
            return 1

    def _query(layer, loop, pq, po, _stream_, _user):
        try:
            q, out = query(layer, loop)
            keep.append((q, out))
            pq[0], po[0] = _ptr(q), _ptr(out)
            return 0
        except Exception as e:
            errors.append(e)
            return 1

    cb_c, cb_q = CAPTURE_FN(_capture), QUERY_FN(_query)
    rp = None if rope_base is None else lla_rope(float(rope_base), int(rope_pairing))
    xd = LLA_BF16 if x_dtype == torch.bfloat16 else LLA_F32
    iod = LLA_BF16 if io_dtype == torch.bfloat16 else LLA_F32
    B = cu_seqlens.shape[0] - 1
    st = library().lla_prefill_two_pass(
        ctypes.byref(g), D, cds, chs, xd, _ptr(slot_mapping), slot_mapping.numel(), _ptr(cu_seqlens),
        B, max_len, iod, None if rp is None else ctypes.byref(rp), cb_c, cb_q, None, _ptr(workspace),
        0 if workspace is None else workspace.numel() * workspace.element_size(), _stream(stream))
    if errors:
        raise errors[0]
    _check("lla_prefill_two_pass", st)


def lla_cache_2d_block_bytes(geom: Geometry) -> int:
    """Bytes of one LLA-2D cache block (one page of 64 tokens for all heads)."""
    out = ctypes.c_size_t(0)
    g = geom.c()
    _check("lla_cache_2d_block_bytes",
           library().lla_cache_2d_block_bytes(ctypes.byref(g), ctypes.byref(out)))
    return out.value


def lla_encode_2d(geom: Geometry, codec: Codec, cache: Cache, x_k: torch.Tensor,
                  x_v: torch.Tensor, slot_mapping: torch.Tensor, stream=None) -> None:
    """LLA-2D encode.  x_k, x_v [T][N][H][d]; codec w_down_* [T*H*d][r], mu_* [T*H*d];
    cache with one page per block."""
    g, cd, ch = geom.c(), codec.c(), cache.c()
    N = x_k.shape[1] if x_k.dim() == 4 else 0
    _check("lla_encode_2d", library().lla_encode_2d(
        ctypes.byref(g), ctypes.byref(cd), ctypes.byref(ch), _ptr(x_k), _ptr(x_v),
        _dtype_code(x_k), _ptr(slot_mapping), N, _stream(stream)))


def lla_decode_2d_workspace_size(geom: Geometry, B: int) -> int:
    out = ctypes.c_size_t(0)
    g = geom.c()
    _check("lla_decode_2d_workspace_size",
           library().lla_decode_2d_workspace_size(ctypes.byref(g), B, ctypes.byref(out)))
    return out.value


def lla_decode_attn_2d(geom: Geometry, codec: Codec, cache: Cache, context_lens: torch.Tensor,
                       max_ctx: int, loop: int, q: torch.Tensor, cur_k: Optional[torch.Tensor],
                       cur_v: Optional[torch.Tensor], out: torch.Tensor, workspace: torch.Tensor,
                       stream=None) -> None:
    """LLA-2D decode call; codec w_up_* [T][H][d][r]; q, cur_k, cur_v, out [B][H][d]."""
    g, cd, ch = geom.c(), codec.c(), cache.c()
    _check("lla_decode_attn_2d", library().lla_decode_attn_2d(
        ctypes.byref(g), ctypes.byref(cd), ctypes.byref(ch), _ptr(context_lens), q.shape[0],
        max_ctx, loop, _ptr(q), _ptr(cur_k), _ptr(cur_v), _dtype_code(q), _ptr(out),
        _ptr(workspace), workspace.numel() * workspace.element_size(), _stream(stream)))


def lla_rope_plane_bytes(d_rope: int) -> int:
    out = ctypes.c_size_t(0)
    _check("lla_rope_plane_bytes", library().lla_rope_plane_bytes(d_rope, ctypes.byref(out)))
    return out.value


def lla_encode_rope_keys(d_rope: int, rope_base: float, rope_pairing: int, rope_pool: torch.Tensor,
                         num_blocks: int, k_rope: torch.Tensor, positions: torch.Tensor,
                         slot_mapping: torch.Tensor, stream=None) -> None:
    """Rotary keys k_rope [N][d_rope], turned at positions [N] int32, into the rotary planes."""
    rp = lla_rope(float(rope_base), int(rope_pairing))
    N = k_rope.shape[0] if k_rope.dim() == 2 else 0
    _check("lla_encode_rope_keys", library().lla_encode_rope_keys(
        d_rope, ctypes.byref(rp), _ptr(rope_pool), num_blocks, _ptr(k_rope), _dtype_code(k_rope),
        _ptr(positions), _ptr(slot_mapping), N, _stream(stream)))


def lla_decode_decoupled_workspace_size(geom: Geometry, d_rope: int, B: int) -> int:
    out = ctypes.c_size_t(0)
    g = geom.c()
    _check("lla_decode_decoupled_workspace_size", library().lla_decode_decoupled_workspace_size(
        ctypes.byref(g), d_rope, B, ctypes.byref(out)))
    return out.value


def lla_decode_attn_decoupled(geom: Geometry, codec: Codec, cache: Cache, rope_pool: torch.Tensor,
                              d_rope: int, rope_base: float, rope_pairing: int,
                              context_lens: torch.Tensor, max_ctx: int, loop: int, q: torch.Tensor,
                              q_rope: torch.Tensor, cur_k: Optional[torch.Tensor],
                              cur_v: Optional[torch.Tensor], cur_k_rope: Optional[torch.Tensor],
                              out: torch.Tensor, workspace: torch.Tensor, stream=None) -> None:
    """Per-head LLA decode with the decoupled rotary branch; q, cur_k, cur_v, out [B][H][d],
    q_rope [B][H][d_rope], cur_k_rope [B][d_rope] (pass 1) or None."""
    g, cd, ch = geom.c(), codec.c(), cache.c()
    rp = lla_rope(float(rope_base), int(rope_pairing))
    _check("lla_decode_attn_decoupled", library().lla_decode_attn_decoupled(
        ctypes.byref(g), ctypes.byref(cd), ctypes.byref(ch), _ptr(rope_pool), d_rope, ctypes.byref(rp),
        _ptr(context_lens), q.shape[0], max_ctx, loop, _ptr(q), _ptr(q_rope), _ptr(cur_k), _ptr(cur_v),
        _ptr(cur_k_rope), _dtype_code(q), _ptr(out), _ptr(workspace),
        workspace.numel() * workspace.element_size(), _stream(stream)))


def lla_dense_store(geom: Geometry, cache: Cache, k: torch.Tensor, v: torch.Tensor,
                    slot_mapping: torch.Tensor, stream=None) -> None:
    """k, v [N][H][d]: plain loop-t keys and values for the uncompressed comparator."""
    g, ch = geom.c(), cache.c()
    _check("lla_dense_store", library().lla_dense_store(
        ctypes.byref(g), ctypes.byref(ch), _ptr(k), _ptr(v), _dtype_code(k), _ptr(slot_mapping),
        k.shape[0], _stream(stream)))


def lla_dense_decode_attn(geom: Geometry, cache: Cache, context_lens: torch.Tensor, max_ctx: int,
                          q: torch.Tensor, cur_k: Optional[torch.Tensor],
                          cur_v: Optional[torch.Tensor], out: torch.Tensor,
                          workspace: torch.Tensor, stream=None) -> None:
    g, ch = geom.c(), cache.c()
    _check("lla_dense_decode_attn", library().lla_dense_decode_attn(
        ctypes.byref(g), ctypes.byref(ch), _ptr(context_lens), q.shape[0], max_ctx, _ptr(q),
        _ptr(cur_k), _ptr(cur_v), _dtype_code(q), _ptr(out), _ptr(workspace),
        workspace.numel() * workspace.element_size(), _stream(stream)))


def lla_get_device_error(stream=None) -> int:
    """Returns the device error word (0 = no error) without raising."""
    word = ctypes.c_uint32(0)
    st = library().lla_get_device_error(_stream(stream), ctypes.byref(word))
    if st not in (0, 4, 5):
        raise LLAError("lla_get_device_error", st)
    return word.value


def lla_clear_device_error(stream=None) -> None:
    _check("lla_clear_device_error", library().lla_clear_device_error(_stream(stream)))


def lla_set_wait_limit_ns(nanoseconds: int) -> None:
    _check("lla_set_wait_limit_ns", library().lla_set_wait_limit_ns(int(nanoseconds)))


def lla_get_wait_limit_ns() -> int:
    return int(library().lla_get_wait_limit_ns())
