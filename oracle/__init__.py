"""CPU float64 oracle for Looped Latent Attention (LLA).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this package.  The
product path (``paper_2607_15456_gb300``) never imports it, and this package never imports
the product path: the two share no code.  Inputs reach both sides from the seeded input
generators only.

The arithmetic lives in ``lla_oracle.c`` (plain C, double precision, loops in the order of
the paper's equations); this module only converts numpy arrays to contiguous float64 and
calls it through ctypes.  Citations (paper sections and equations):

* ``ratio``                         -- Eq. ratio, rho = 2 T d / (r_k + r_v)  (Sec. 3)
* ``teacher_cache_bytes_per_token`` -- "Teacher cache" paragraph, 2 T H d scalars per layer
* ``latent_cache_bytes_per_token``  -- (r_k + r_v) H scalars per layer (Sec. 3, Eq. ratio)
* ``encode``                        -- Eq. encode, c = (x - mu) W_down
* ``reconstruct``                   -- Eq. decode, xhat_t = c W_up,t^T + mu_t
* ``attention``                     -- softmax attention over explicit K, V
* ``decode``                        -- one call of the two-pass cached reconstruction
                                       decoder (App. A, "Decoding and caching")
* ``prefill``                       -- causal pass-2 prefill over latents (App. A; App. J,
                                       "Eviction and long-context prefill")
* ``rope``                          -- rotary position embedding (RoFormer), applied after
                                       reconstruction (Sec. 3, "RoPE and reconstruction")
* ``decode_rope``, ``prefill_rope`` -- ``decode`` / ``prefill`` with every reconstructed key
                                       and the query rotated at their token positions
* ``decode_decoupled``              -- the decoupled rotary branch (App. J "Absorbed attention"):
                                       content key by Eq. decode (no rotation) joined with one
                                       rotary key per token, shared by every loop
* ``ratio_2d``, ``encode_2d``,      -- the LLA-2D variant (Sec. 3, "The LLA-2D variant (loop x
  ``decode_2d``                        head)"): one latent per (token, layer) over the
                                       loop-major (loop, head) stack, every head rebuilt from it

Parity status of every function: pinned (see ``tests/test_oracle_pins.py``).
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

import numpy as np

from .build import build_oracle, library_path

_lib = None


def _load():
    global _lib
    if _lib is None:
        # LLA_ORACLE_LIB lets the mutation test load a deliberately broken copy of the oracle
        path = os.environ.get("LLA_ORACLE_LIB") or build_oracle()
        lib = ctypes.CDLL(path)
        d, i32, i64, p = ctypes.c_double, ctypes.c_int, ctypes.c_int64, ctypes.c_void_p
        lib.lla_oracle_ratio.restype = d
        lib.lla_oracle_ratio.argtypes = [i32, i32, i32, i32]
        lib.lla_oracle_teacher_cache_bytes_per_token.restype = d
        lib.lla_oracle_teacher_cache_bytes_per_token.argtypes = [i32, i32, i32, i32, i32]
        lib.lla_oracle_latent_cache_bytes_per_token.restype = d
        lib.lla_oracle_latent_cache_bytes_per_token.argtypes = [i32, i32, i32, i32, i32]
        lib.lla_oracle_encode.restype = None
        lib.lla_oracle_encode.argtypes = [i32, i32, i32, i64, p, p, p, p]
        lib.lla_oracle_reconstruct.restype = None
        lib.lla_oracle_reconstruct.argtypes = [i32, i32, i64, p, p, p, p]
        lib.lla_oracle_attention.restype = i32
        lib.lla_oracle_attention.argtypes = [i32, i64, p, p, p, d, p]
        lib.lla_oracle_decode.restype = i32
        lib.lla_oracle_decode.argtypes = [i32, i32, i32, i32, i32, i64] + [p] * 9 + [d, p]
        lib.lla_oracle_prefill.restype = i32
        lib.lla_oracle_prefill.argtypes = [i32, i32, i32, i32, i32, i64] + [p] * 7 + [d, p]
        lib.lla_oracle_rope.restype = None
        lib.lla_oracle_rope.argtypes = [i32, i32, d, i64, p, p]
        lib.lla_oracle_decode_rope.restype = i32
        lib.lla_oracle_decode_rope.argtypes = ([i32, i32, i32, i32, i32, i64] + [p] * 9 +
                                               [d, i32, d, i64, p])
        lib.lla_oracle_prefill_rope.restype = i32
        lib.lla_oracle_prefill_rope.argtypes = ([i32, i32, i32, i32, i32, i64] + [p] * 7 +
                                                [d, i32, d, i64, p])
        lib.lla_oracle_decode_batch.restype = i32
        lib.lla_oracle_decode_batch.argtypes = [i32, i32, i32, i32, d, i64, p, i32]
        lib.lla_oracle_encode_batch.restype = i32
        lib.lla_oracle_encode_batch.argtypes = [i32, i32, i64, i64, p, i32]
        lib.lla_oracle_decode_decoupled.restype = i32
        lib.lla_oracle_decode_decoupled.argtypes = ([i32] * 6 + [i64] + [p] * 12 +
                                                    [d, i32, d, i64, p])
        lib.lla_oracle_ratio_2d.restype = d
        lib.lla_oracle_ratio_2d.argtypes = [i32, i32, i32, i32, i32]
        lib.lla_oracle_encode_2d.restype = None
        lib.lla_oracle_encode_2d.argtypes = [i32, i32, i32, i32, i64, p, p, p, p]
        lib.lla_oracle_decode_2d_head.restype = i32
        lib.lla_oracle_decode_2d_head.argtypes = [i32] * 7 + [i64] + [p] * 9 + [d, p]
        lib.lla_oracle_decode_2d_batch.restype = i32
        lib.lla_oracle_decode_2d_batch.argtypes = [i32, i32, i32, i32, i32, d, i64, p, i32]
        lib.lla_oracle_max_threads.restype = i32
        lib.lla_oracle_max_threads.argtypes = []
        _lib = lib
    return _lib


def _f64(a) -> np.ndarray:
    """Contiguous float64 copy (exact widening of float32 / bf16-valued inputs)."""
    return np.ascontiguousarray(np.asarray(a, dtype=np.float64))


def _ptr(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


# ---------------------------------------------------------------- closed forms (Eq. ratio)

def ratio(T: int, d_head: int, r_k: int, r_v: int) -> float:
    return _load().lla_oracle_ratio(T, d_head, r_k, r_v)


def teacher_cache_bytes_per_token(T: int, H: int, d_head: int, D: int, elem_bytes: int) -> float:
    return _load().lla_oracle_teacher_cache_bytes_per_token(T, H, d_head, D, elem_bytes)


def latent_cache_bytes_per_token(H: int, D: int, r_k: int, r_v: int, elem_bytes: int) -> float:
    return _load().lla_oracle_latent_cache_bytes_per_token(H, D, r_k, r_v, elem_bytes)


# ---------------------------------------------------------------- codec (Eqs. encode, decode)

def encode(x, mu, w_down) -> np.ndarray:
    """Eq. encode.  x [T][N][d], mu [T*d] or None, w_down [T*d][r] -> c [N][r]."""
    x, w_down = _f64(x), _f64(w_down)
    T, N, d = x.shape
    r = w_down.shape[1]
    assert w_down.shape[0] == T * d
    mu = None if mu is None else _f64(mu).reshape(T * d)
    c = np.zeros((N, r), dtype=np.float64)
    _load().lla_oracle_encode(T, d, r, N, _ptr(x), _ptr(mu), _ptr(w_down), _ptr(c))
    return c


def reconstruct(c, w_up_t, mu_t=None) -> np.ndarray:
    """Eq. decode at one loop.  c [N][r], w_up_t [d][r], mu_t [d] or None -> xhat [N][d]."""
    c, w_up_t = _f64(c), _f64(w_up_t)
    N, r = c.shape
    d = w_up_t.shape[0]
    mu_t = None if mu_t is None else _f64(mu_t).reshape(d)
    out = np.zeros((N, d), dtype=np.float64)
    _load().lla_oracle_reconstruct(d, r, N, _ptr(c), _ptr(w_up_t), _ptr(mu_t), _ptr(out))
    return out


def attention(q, K, V, scale: float) -> np.ndarray:
    """Softmax attention of one query q [d] over K, V [L][d]."""
    q, K, V = _f64(q), _f64(K), _f64(V)
    L, d = K.shape
    out = np.zeros(d, dtype=np.float64)
    rc = _load().lla_oracle_attention(d, L, _ptr(q), _ptr(K), _ptr(V), scale, _ptr(out))
    if rc:
        raise ValueError("attention needs at least one key")
    return out


def decode(t: int, c_k, c_v, w_up_k, w_up_v, mu_k, mu_v, q, cur_k, cur_v,
           scale: float) -> np.ndarray:
    """One decode call for one (sequence, head) at loop t.

    c_k [L][r_k], c_v [L][r_v]; w_up_k [T][d][r_k]; w_up_v [T][d][r_v]; mu_* [T*d] or None;
    q [d]; cur_k / cur_v [d] for pass 1 or None for pass 2.
    """
    w_up_k, w_up_v = _f64(w_up_k), _f64(w_up_v)
    T, d, r_k = w_up_k.shape
    r_v = w_up_v.shape[2]
    c_k = _f64(c_k).reshape(-1, r_k)
    c_v = _f64(c_v).reshape(-1, r_v)
    L = c_k.shape[0]
    mu_k = None if mu_k is None else _f64(mu_k).reshape(T * d)
    mu_v = None if mu_v is None else _f64(mu_v).reshape(T * d)
    q = _f64(q).reshape(d)
    cur_k = None if cur_k is None else _f64(cur_k).reshape(d)
    cur_v = None if cur_v is None else _f64(cur_v).reshape(d)
    out = np.zeros(d, dtype=np.float64)
    rc = _load().lla_oracle_decode(T, d, r_k, r_v, t, L, _ptr(c_k), _ptr(c_v), _ptr(w_up_k),
                                   _ptr(w_up_v), _ptr(mu_k), _ptr(mu_v), _ptr(q), _ptr(cur_k),
                                   _ptr(cur_v), scale, _ptr(out))
    if rc:
        raise ValueError("bad decode arguments")
    return out


def prefill(t: int, c_k, c_v, w_up_k, w_up_v, mu_k, mu_v, q, scale: float) -> np.ndarray:
    """Causal pass-2 prefill at loop t for one (sequence, head); q [N][d] -> out [N][d]."""
    w_up_k, w_up_v = _f64(w_up_k), _f64(w_up_v)
    T, d, r_k = w_up_k.shape
    r_v = w_up_v.shape[2]
    c_k = _f64(c_k).reshape(-1, r_k)
    c_v = _f64(c_v).reshape(-1, r_v)
    N = c_k.shape[0]
    mu_k = None if mu_k is None else _f64(mu_k).reshape(T * d)
    mu_v = None if mu_v is None else _f64(mu_v).reshape(T * d)
    q = _f64(q).reshape(N, d)
    out = np.zeros((N, d), dtype=np.float64)
    rc = _load().lla_oracle_prefill(T, d, r_k, r_v, t, N, _ptr(c_k), _ptr(c_v), _ptr(w_up_k),
                                    _ptr(w_up_v), _ptr(mu_k), _ptr(mu_v), _ptr(q), scale,
                                    _ptr(out))
    if rc:
        raise ValueError("bad prefill arguments")
    return out


# ---------------------------------------------------------------- rotary positions (Sec. 3)

ROPE_HALF, ROPE_ADJACENT = 0, 1  # pair j = (x[j], x[j + d/2])  or  (x[2j], x[2j + 1])


def rope(x, pos: int, base: float = 10000.0, pairing: int = ROPE_HALF) -> np.ndarray:
    """RoFormer rotation of x [d] at integer position pos: pair j turned by pos * base^(-2j/d)."""
    x = _f64(x)
    d = x.shape[-1]
    assert x.ndim == 1 and d % 2 == 0
    y = np.zeros(d, dtype=np.float64)
    _load().lla_oracle_rope(d, pairing, base, pos, _ptr(x), _ptr(y))
    return y


def decode_rope(t: int, c_k, c_v, w_up_k, w_up_v, mu_k, mu_v, q, cur_k, cur_v, scale: float,
                base: float = 10000.0, pairing: int = ROPE_HALF, pos0: int = 0) -> np.ndarray:
    """``decode`` with RoPE after reconstruction: cached token i at position pos0 + i, the
    current token (and the query) at pos0 + L in pass 1 and pos0 + L - 1 in pass 2."""
    w_up_k, w_up_v = _f64(w_up_k), _f64(w_up_v)
    T, d, r_k = w_up_k.shape
    r_v = w_up_v.shape[2]
    c_k = _f64(c_k).reshape(-1, r_k)
    c_v = _f64(c_v).reshape(-1, r_v)
    L = c_k.shape[0]
    mu_k = None if mu_k is None else _f64(mu_k).reshape(T * d)
    mu_v = None if mu_v is None else _f64(mu_v).reshape(T * d)
    q = _f64(q).reshape(d)
    cur_k = None if cur_k is None else _f64(cur_k).reshape(d)
    cur_v = None if cur_v is None else _f64(cur_v).reshape(d)
    out = np.zeros(d, dtype=np.float64)
    rc = _load().lla_oracle_decode_rope(T, d, r_k, r_v, t, L, _ptr(c_k), _ptr(c_v),
                                        _ptr(w_up_k), _ptr(w_up_v), _ptr(mu_k), _ptr(mu_v),
                                        _ptr(q), _ptr(cur_k), _ptr(cur_v), scale, pairing, base,
                                        pos0, _ptr(out))
    if rc:
        raise ValueError("bad decode arguments")
    return out


def prefill_rope(t: int, c_k, c_v, w_up_k, w_up_v, mu_k, mu_v, q, scale: float,
                 base: float = 10000.0, pairing: int = ROPE_HALF, pos0: int = 0) -> np.ndarray:
    """``prefill`` with RoPE after reconstruction: prompt token i at position pos0 + i."""
    w_up_k, w_up_v = _f64(w_up_k), _f64(w_up_v)
    T, d, r_k = w_up_k.shape
    r_v = w_up_v.shape[2]
    c_k = _f64(c_k).reshape(-1, r_k)
    c_v = _f64(c_v).reshape(-1, r_v)
    N = c_k.shape[0]
    mu_k = None if mu_k is None else _f64(mu_k).reshape(T * d)
    mu_v = None if mu_v is None else _f64(mu_v).reshape(T * d)
    q = _f64(q).reshape(N, d)
    out = np.zeros((N, d), dtype=np.float64)
    rc = _load().lla_oracle_prefill_rope(T, d, r_k, r_v, t, N, _ptr(c_k), _ptr(c_v),
                                         _ptr(w_up_k), _ptr(w_up_v), _ptr(mu_k), _ptr(mu_v),
                                         _ptr(q), scale, pairing, base, pos0, _ptr(out))
    if rc:
        raise ValueError("bad prefill arguments")
    return out


# ---------------------------------------------------------------- decoupled rotary branch

def decode_decoupled(t: int, c_k, c_v, k_rope, w_up_k, w_up_v, mu_k, mu_v, q, q_rope, cur_k,
                     cur_v, cur_k_rope, scale: float, base: float = 10000.0,
                     pairing: int = ROPE_HALF, pos0: int = 0) -> np.ndarray:
    """One decode call for one (sequence, head) at loop t with the decoupled rotary branch:
    s_i = scale (q . khat_t,i + rot(q^R, P) . rot(k^R_i, p_i)).  k_rope [L][d_rope] (one rotary
    key per token, every loop), q_rope [d_rope]; cur_k_rope [d_rope] with cur_k / cur_v in
    pass 1, None in pass 2.  Other arguments as ``decode``."""
    w_up_k, w_up_v = _f64(w_up_k), _f64(w_up_v)
    T, d, r_k = w_up_k.shape
    r_v = w_up_v.shape[2]
    c_k = _f64(c_k).reshape(-1, r_k)
    c_v = _f64(c_v).reshape(-1, r_v)
    L = c_k.shape[0]
    q_rope = _f64(q_rope).reshape(-1)
    d_rope = q_rope.shape[0]
    k_rope = _f64(k_rope).reshape(L, d_rope)
    mu_k = None if mu_k is None else _f64(mu_k).reshape(T * d)
    mu_v = None if mu_v is None else _f64(mu_v).reshape(T * d)
    q = _f64(q).reshape(d)
    cur_k = None if cur_k is None else _f64(cur_k).reshape(d)
    cur_v = None if cur_v is None else _f64(cur_v).reshape(d)
    cur_k_rope = None if cur_k_rope is None else _f64(cur_k_rope).reshape(d_rope)
    out = np.zeros(d, dtype=np.float64)
    rc = _load().lla_oracle_decode_decoupled(
        T, d, d_rope, r_k, r_v, t, L, _ptr(c_k), _ptr(c_v), _ptr(k_rope), _ptr(w_up_k),
        _ptr(w_up_v), _ptr(mu_k), _ptr(mu_v), _ptr(q), _ptr(q_rope), _ptr(cur_k), _ptr(cur_v),
        _ptr(cur_k_rope), scale, pairing, base, pos0, _ptr(out))
    if rc:
        raise ValueError("bad decode arguments")
    return out


# ---------------------------------------------------------------- LLA-2D (Sec. 3)

def ratio_2d(T: int, H: int, d_head: int, r_k: int, r_v: int) -> float:
    """rho_2D = 2 T H d / (r_k + r_v): one latent pair per (token, layer)."""
    return _load().lla_oracle_ratio_2d(T, H, d_head, r_k, r_v)


def encode_2d(x, mu, w_down) -> np.ndarray:
    """LLA-2D encode.  x [T][N][H][d], mu [T*H*d] or None, w_down [T*H*d][r] -> c [N][r]."""
    x, w_down = _f64(x), _f64(w_down)
    T, N, H, d = x.shape
    r = w_down.shape[1]
    assert w_down.shape[0] == T * H * d
    mu = None if mu is None else _f64(mu).reshape(T * H * d)
    c = np.zeros((N, r), dtype=np.float64)
    _load().lla_oracle_encode_2d(T, H, d, r, N, _ptr(x), _ptr(mu), _ptr(w_down), _ptr(c))
    return c


def _decode_2d_args(w_up_k, w_up_v, mu_k, mu_v):
    w_up_k, w_up_v = _f64(w_up_k), _f64(w_up_v)
    T, H, d, r_k = w_up_k.shape
    r_v = w_up_v.shape[3]
    assert w_up_v.shape[:3] == (T, H, d)
    mu_k = None if mu_k is None else _f64(mu_k).reshape(T * H * d)
    mu_v = None if mu_v is None else _f64(mu_v).reshape(T * H * d)
    return w_up_k, w_up_v, mu_k, mu_v, T, H, d, r_k, r_v


def decode_2d(t: int, c_k, c_v, w_up_k, w_up_v, mu_k, mu_v, q, cur_k, cur_v,
              scale: float, heads: Optional[Sequence[int]] = None,
              n_threads: int = 0) -> np.ndarray:
    """One LLA-2D decode call for one sequence at loop t.

    c_k [L][r_k], c_v [L][r_v] (one latent per token for all heads); w_up_k [T][H][d][r_k];
    w_up_v [T][H][d][r_v]; mu_* [T*H*d] or None; q [H][d]; cur_k / cur_v [H][d] (pass 1) or
    None (pass 2).  Returns out [len(heads)][d] for the listed heads (default: all).
    """
    w_up_k, w_up_v, mu_k, mu_v, T, H, d, r_k, r_v = _decode_2d_args(w_up_k, w_up_v, mu_k, mu_v)
    c_k = _f64(c_k).reshape(-1, r_k)
    c_v = _f64(c_v).reshape(-1, r_v)
    L = c_k.shape[0]
    q = _f64(q).reshape(H, d)
    cur_k = None if cur_k is None else _f64(cur_k).reshape(H, d)
    cur_v = None if cur_v is None else _f64(cur_v).reshape(H, d)
    heads = list(range(H)) if heads is None else list(heads)
    out = np.zeros((len(heads), d), dtype=np.float64)
    arr = (_Decode2dItem * len(heads))()
    for k, h in enumerate(heads):
        it = arr[k]
        it.t, it.h, it.L = t, h, L
        it.c_k, it.c_v, it.w_up_k, it.w_up_v = _ptr(c_k), _ptr(c_v), _ptr(w_up_k), _ptr(w_up_v)
        it.mu_k, it.mu_v = _ptr(mu_k), _ptr(mu_v)
        it.q = q[h].ctypes.data
        it.cur_k = None if cur_k is None else cur_k[h].ctypes.data
        it.cur_v = None if cur_v is None else cur_v[h].ctypes.data
        it.out = out[k].ctypes.data
    rc = _load().lla_oracle_decode_2d_batch(T, H, d, r_k, r_v, scale, len(heads),
                                            ctypes.cast(arr, ctypes.c_void_p), n_threads)
    if rc:
        raise ValueError("bad decode arguments")
    return out


# ---------------------------------------------------------------- batched drivers (OpenMP)

class _DecodeItem(ctypes.Structure):
    _fields_ = [("t", ctypes.c_int32), ("rope", ctypes.c_int32), ("L", ctypes.c_int64),
                ("rope_base", ctypes.c_double)] + [
        (n, ctypes.c_void_p) for n in
        ("c_k", "c_v", "w_up_k", "w_up_v", "mu_k", "mu_v", "q", "cur_k", "cur_v", "out")]


class _Decode2dItem(ctypes.Structure):
    _fields_ = [("t", ctypes.c_int32), ("h", ctypes.c_int32), ("L", ctypes.c_int64)] + [
        (n, ctypes.c_void_p) for n in
        ("c_k", "c_v", "w_up_k", "w_up_v", "mu_k", "mu_v", "q", "cur_k", "cur_v", "out")]


class _EncodeItem(ctypes.Structure):
    _fields_ = [("r", ctypes.c_int32), ("pad_", ctypes.c_int32)] + [
        (n, ctypes.c_void_p) for n in ("x", "mu", "w_down", "c")]


def max_threads() -> int:
    return _load().lla_oracle_max_threads()


def decode_batch(T: int, d: int, r_k: int, r_v: int, scale: float, items: Sequence[dict],
                 n_threads: int = 0) -> list:
    """Runs independent decode problems side by side.  Each item is a dict with keys
    t, c_k, c_v, w_up_k, w_up_v, mu_k, mu_v, q, cur_k, cur_v (arrays as in ``decode``) and an
    optional ``rope`` = (pairing, base), which makes the item a ``decode_rope`` problem with
    pos0 = 0.  Returns the list of outputs [d]."""
    keep, outs = [], []
    arr = (_DecodeItem * len(items))()
    for k, it in enumerate(items):
        fields = {}
        for name in ("c_k", "c_v", "w_up_k", "w_up_v", "mu_k", "mu_v", "q", "cur_k", "cur_v"):
            v = it.get(name)
            if v is not None:
                v = _f64(v)
                keep.append(v)
            fields[name] = _ptr(v)
        out = np.zeros(d, dtype=np.float64)
        outs.append(out)
        arr[k].t = it["t"]
        if it.get("rope") is not None:
            arr[k].rope = int(it["rope"][0]) + 1
            arr[k].rope_base = float(it["rope"][1])
        arr[k].L = _f64(it["c_k"]).size // r_k
        for name, v in fields.items():
            setattr(arr[k], name, v)
        arr[k].out = _ptr(out)
    rc = _load().lla_oracle_decode_batch(T, d, r_k, r_v, scale, len(items),
                                         ctypes.cast(arr, ctypes.c_void_p), n_threads)
    if rc:
        raise ValueError("bad decode arguments in batch")
    return outs


def encode_batch(T: int, d: int, items: Sequence[dict], n_threads: int = 0) -> list:
    """Runs independent encode problems side by side.  Each item: x [T][N][d], mu, w_down."""
    keep, outs = [], []
    arr = (_EncodeItem * len(items))()
    N = None
    for k, it in enumerate(items):
        x = _f64(it["x"])
        w = _f64(it["w_down"])
        mu = None if it.get("mu") is None else _f64(it["mu"])
        keep += [x, w, mu]
        N = x.shape[1]
        c = np.zeros((N, w.shape[1]), dtype=np.float64)
        outs.append(c)
        arr[k].r = w.shape[1]
        arr[k].x, arr[k].mu, arr[k].w_down, arr[k].c = _ptr(x), _ptr(mu), _ptr(w), _ptr(c)
    _load().lla_oracle_encode_batch(T, d, N or 0, len(items), ctypes.cast(arr, ctypes.c_void_p),
                                    n_threads)
    return outs


__all__ = ["ratio", "teacher_cache_bytes_per_token", "latent_cache_bytes_per_token", "encode",
           "reconstruct", "attention", "decode", "prefill", "rope", "decode_rope",
           "prefill_rope", "ROPE_HALF", "ROPE_ADJACENT", "decode_decoupled", "ratio_2d",
           "encode_2d", "decode_2d",
           "decode_batch", "encode_batch",
           "max_threads", "build_oracle", "library_path"]
