"""Host-side checks of the C ABI (no GPU): the library loads, exports every entry point that
include/lla.h declares, and rejects bad arguments synchronously, before touching CUDA."""
import ctypes
import os
import re

import pytest

from helpers import ensure_library

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "lla.h")

OK, INVALID, UNSUPPORTED, CUDA_ERR, TIMEOUT, DEVCHECK, WORKSPACE = range(7)
FAKE = 0x10000  # a non-NULL, 16-byte aligned "device pointer" that validation never touches


@pytest.fixture(scope="module")
def lib():
    ensure_library()
    from paper_2607_15456_gb300 import lla
    return lla


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    text = re.sub(r"typedef[^;]*;", "", text)  # callback types, structs and enums
    return sorted(set(re.findall(r"\b(lla_[a-z_0-9]+)\s*\(", text)))


def test_header_declares_the_entry_points():
    names = declared_functions()
    for must in ("lla_encode", "lla_decode_attn", "lla_prefill_attn", "lla_decode_workspace_size",
                 "lla_dense_decode_attn", "lla_get_device_error", "lla_status_string"):
        assert must in names


def test_library_exports_every_declared_symbol(lib):
    so = lib.library()
    missing = [n for n in declared_functions() if not hasattr(so, n)]
    assert not missing, missing


def test_binding_has_every_declared_entry_point(lib):
    """The Python binding carries the C names: one callable per declared function."""
    missing = [n for n in declared_functions() if not callable(getattr(lib, n, None))]
    assert not missing, missing


def test_wait_limit_is_a_host_setting(lib):
    """The pipeline wait limit is kept on the host (no GPU call): 0 means the 2 s default."""
    assert lib.lla_get_wait_limit_ns() == 2_000_000_000
    lib.lla_set_wait_limit_ns(12345)
    try:
        assert lib.lla_get_wait_limit_ns() == 12345
    finally:
        lib.lla_set_wait_limit_ns(0)
    assert lib.lla_get_wait_limit_ns() == 2_000_000_000


def test_status_strings_and_version(lib):
    assert lib.lla_version() >= 100
    assert lib.lla_status_string(0) == "ok"
    assert lib.lla_status_string(6) == "workspace too small"


def test_block_bytes_follow_the_documented_layout(lib):
    for T, H, d, rk, rv, st, es in ((4, 16, 128, 96, 160, "bf16", 2), (4, 16, 128, 18, 30, "bf16", 2),
                                    (4, 4, 128, 96, 160, "fp32", 4)):
        g = lib.Geometry(T, H, d, rk, rv, st)
        assert lib.lla_cache_block_bytes(g) == H * 64 * (rk + rv) * es


def _g(lib, **kw):
    base = dict(T=4, H=16, d=128, r_k=96, r_v=160, storage="bf16")
    base.update(kw)
    return lib.Geometry(**base).c()


def _codec(lib, **kw):
    c = lib.lla_codec(FAKE, FAKE, FAKE, FAKE, None, None)
    for k, v in kw.items():
        setattr(c, k, v)
    return c


def _cache(lib, pool=FAKE, table=FAKE, nb=10, mb=4):
    return lib.lla_cache(pool, nb, table, mb)


@pytest.mark.parametrize("bad", [dict(T=0), dict(T=17), dict(H=0), dict(d=12), dict(d=512),
                                 dict(r_k=1), dict(r_v=513), dict(r_k=95), dict(storage="x")])
def test_bad_geometry_is_rejected(lib, bad):
    kw = dict(T=4, H=16, d=128, r_k=96, r_v=160, storage="bf16")
    kw.update(bad)
    g = lib.Geometry(**{k: v for k, v in kw.items() if k != "storage"}).c()
    if "storage" in bad:
        g.storage = 7
    so = lib.library()
    out = ctypes.c_size_t()
    assert so.lla_cache_block_bytes(ctypes.byref(g), ctypes.byref(out)) == INVALID


def test_block_size_other_than_64_is_unsupported(lib):
    g = _g(lib)
    g.block_size = 32
    out = ctypes.c_size_t()
    assert lib.library().lla_cache_block_bytes(ctypes.byref(g), ctypes.byref(out)) == UNSUPPORTED


def _decode(lib, g=None, codec=None, cache=None, lens=FAKE, B=4, max_ctx=128, loop=0, q=FAKE,
            ck=FAKE, cv=FAKE, io=0, out=FAKE, ws=FAKE, ws_bytes=1 << 20):
    so = lib.library()
    g = g or _g(lib)
    codec = codec or _codec(lib)
    cache = cache or _cache(lib)
    return so.lla_decode_attn(ctypes.byref(g), ctypes.byref(codec), ctypes.byref(cache), lens, B,
                              max_ctx, loop, q, ck, cv, io, out, ws, ws_bytes, None)


def test_decode_argument_checks(lib):
    assert _decode(lib, ck=None) == INVALID                      # cur_k without cur_v
    assert _decode(lib, loop=4) == INVALID                       # loop outside [0, T)
    assert _decode(lib, loop=-1) == INVALID
    assert _decode(lib, B=-1) == INVALID
    assert _decode(lib, B=1025) == INVALID                       # above LLA_MAX_BATCH
    assert _decode(lib, max_ctx=4 * 64 + 1) == INVALID           # beyond the table capacity
    assert _decode(lib, q=None) == INVALID
    assert _decode(lib, lens=None) == INVALID
    assert _decode(lib, out=None) == INVALID
    assert _decode(lib, ws=None) == INVALID
    assert _decode(lib, io=3) == INVALID
    assert _decode(lib, codec=_codec(lib, w_up_k=None)) == INVALID
    assert _decode(lib, codec=_codec(lib, w_up_v=FAKE + 2)) == INVALID   # misaligned bf16 pairs
    assert _decode(lib, cache=_cache(lib, pool=FAKE + 8)) == INVALID     # pool not 16-B aligned
    assert _decode(lib, cache=_cache(lib, table=None)) == INVALID
    assert _decode(lib, cache=_cache(lib, nb=0)) == INVALID
    # an empty batch is a valid no-op that never touches the device
    assert _decode(lib, B=0, lens=None, q=None, out=None, ws=None) == OK


def test_decode_rejects_geometries_without_a_kernel_shape(lib):
    # fp32 latents with r_k + r_v = 1024 do not leave room for two pipeline stages
    g = _g(lib, r_k=512, r_v=512, storage="fp32")
    assert _decode(lib, g=g) == UNSUPPORTED


def test_encode_argument_checks(lib):
    so = lib.library()
    g, cache = _g(lib), _cache(lib)

    def enc(codec=None, xk=FAKE, xv=FAKE, slots=FAKE, N=8, xd=0):
        codec = codec or _codec(lib)
        return so.lla_encode(ctypes.byref(g), ctypes.byref(codec), ctypes.byref(cache), xk, xv,
                             xd, slots, N, None)

    assert enc(codec=_codec(lib, w_down_k=None)) == INVALID
    assert enc(xk=None) == INVALID
    assert enc(slots=None) == INVALID
    assert enc(N=-1) == INVALID
    assert enc(xd=5) == INVALID
    assert enc(N=0, xk=None, xv=None, slots=None) == OK


def test_dense_comparator_needs_r_equal_d(lib):
    so = lib.library()
    g, cache = _g(lib), _cache(lib)  # r_k = 96 != d
    assert so.lla_dense_decode_attn(ctypes.byref(g), ctypes.byref(cache), FAKE, 4, 64, FAKE, None,
                                    None, 0, FAKE, FAKE, 1 << 20, None) == INVALID
    assert so.lla_dense_store(ctypes.byref(g), ctypes.byref(cache), FAKE, FAKE, 0, FAKE, 4,
                              None) == INVALID


def test_prefill_argument_checks(lib):
    so = lib.library()
    g, codec, cache = _g(lib), _codec(lib), _cache(lib)

    def pre(cu=FAKE, B=2, max_len=64, loop=0, q=FAKE, out=FAKE):
        return so.lla_prefill_attn(ctypes.byref(g), ctypes.byref(codec), ctypes.byref(cache), cu,
                                   B, max_len, loop, q, 0, out, None)

    assert pre(cu=None) == INVALID
    assert pre(loop=4) == INVALID
    assert pre(max_len=10**6) == INVALID
    assert pre(B=0, cu=None, q=None, out=None) == OK


def test_workspace_init_rejects_null(lib):
    assert lib.library().lla_decode_workspace_init(None, 16, None) == INVALID


def test_encode_layers_argument_checks(lib):
    so = lib.library()
    g = _g(lib)
    L = 2
    codecs = (lib.lla_codec * L)(*[_codec(lib) for _ in range(L)])
    caches = (lib.lla_cache * L)(*[_cache(lib) for _ in range(L)])
    ptrs = (ctypes.c_void_p * L)(FAKE, FAKE)

    def enc(L=2, codecs=codecs, caches=caches, xk=ptrs, xv=ptrs, slots=FAKE, N=8, xd=0):
        return so.lla_encode_layers(ctypes.byref(g), L, codecs, caches, xk, xv, xd, slots, N, None)

    assert enc(L=0, codecs=None, caches=None, xk=None, xv=None, slots=None) == OK  # no layers
    assert enc(N=0) == OK
    assert enc(L=65) == UNSUPPORTED
    assert enc(L=-1) == INVALID
    assert enc(codecs=None) == INVALID
    assert enc(xk=None) == INVALID
    assert enc(slots=None) == INVALID
    assert enc(xd=5) == INVALID
    bad = (ctypes.c_void_p * L)(FAKE, FAKE + 8)  # layer 1's input not 16-byte aligned
    assert enc(xv=bad) == INVALID
    nocodec = (lib.lla_codec * L)(_codec(lib), _codec(lib, w_down_v=None))
    assert enc(codecs=nocodec) == INVALID


def _decode_rope(lib, rope=None, g=None, codec=None, cache=None, lens=FAKE, B=4, max_ctx=128,
                 loop=0, q=FAKE, ck=FAKE, cv=FAKE, io=0, out=FAKE, ws=FAKE, ws_bytes=1 << 20,
                 no_rope=False):
    so = lib.library()
    g = g or _g(lib)
    codec = codec or _codec(lib)
    cache = cache or _cache(lib)
    rope = rope or lib.lla_rope(10000.0, lib.LLA_ROPE_HALF)
    return so.lla_decode_attn_rope(ctypes.byref(g), ctypes.byref(codec), ctypes.byref(cache),
                                   None if no_rope else ctypes.byref(rope), lens, B, max_ctx,
                                   loop, q, ck, cv, io, out, ws, ws_bytes, None)


def test_decode_rope_argument_checks(lib):
    assert _decode_rope(lib, no_rope=True) == INVALID
    assert _decode_rope(lib, rope=lib.lla_rope(1.0, 0)) == INVALID        # base must exceed 1
    assert _decode_rope(lib, rope=lib.lla_rope(float("nan"), 0)) == INVALID
    assert _decode_rope(lib, rope=lib.lla_rope(10000.0, 2)) == INVALID    # unknown pairing
    assert _decode_rope(lib, q=FAKE + 8) == INVALID                       # q not 16-B aligned
    assert _decode_rope(lib, out=FAKE + 4) == INVALID
    assert _decode_rope(lib, ck=None) == INVALID                          # cur_k without cur_v
    assert _decode_rope(lib, loop=4) == INVALID
    assert _decode_rope(lib, ws=None) == INVALID
    # shapes without a tensor-core key rebuild
    assert _decode_rope(lib, g=_g(lib, r_k=18, r_v=30)) == UNSUPPORTED    # 4-byte K granules
    assert _decode_rope(lib, g=_g(lib, storage="fp32")) == UNSUPPORTED
    assert _decode_rope(lib, g=_g(lib, d=64)) == UNSUPPORTED
    assert _decode_rope(lib, B=0, lens=None, q=None, out=None, ws=None) == OK
    assert _decode_rope(lib, rope=lib.lla_rope(500000.0, lib.LLA_ROPE_ADJACENT), B=0, lens=None,
                        q=None, out=None, ws=None) == OK


def test_prefill_rope_argument_checks(lib):
    so = lib.library()
    g, codec, cache = _g(lib), _codec(lib), _cache(lib)
    rope = lib.lla_rope(10000.0, lib.LLA_ROPE_HALF)
    size = ctypes.c_size_t()
    assert so.lla_prefill_rope_workspace_size(ctypes.byref(g), 4, 128, ctypes.byref(size)) == OK
    assert size.value == 4 * 2 * 16 * 64 * 128 * 2 + 4 * 128 * 16 * 128 * 2
    g72 = _g(lib, r_k=72, r_v=120)
    assert so.lla_prefill_rope_workspace_size(ctypes.byref(g72), 4, 128, ctypes.byref(size)) == UNSUPPORTED

    def call(rope_=rope, g_=g, B=4, max_len=128, loop=0, q=FAKE, io=0, out=FAKE, ws=FAKE,
             cu=FAKE):
        return so.lla_prefill_attn_rope(ctypes.byref(g_), ctypes.byref(codec), ctypes.byref(cache),
                                        None if rope_ is None else ctypes.byref(rope_), cu, B,
                                        max_len, loop, q, io, out, ws, 1 << 30, None)
    assert call(rope_=None) == INVALID
    assert call(rope_=lib.lla_rope(0.5, 0)) == INVALID
    assert call(rope_=lib.lla_rope(10000.0, 7)) == INVALID
    assert call(loop=4) == INVALID
    assert call(q=FAKE + 4) == INVALID
    assert call(ws=None) == INVALID
    assert call(max_len=4 * 64 + 1) == INVALID
    assert call(g_=g72) == UNSUPPORTED
    assert call(g_=_g(lib, storage="fp32")) == UNSUPPORTED
    assert call(B=0, q=None, out=None, ws=None, cu=None) == OK


def test_decode_loops_argument_checks(lib):
    so = lib.library()

    def call(g=None, B=4, max_ctx=128, q=FAKE, ck=FAKE, cv=FAKE, io=0, out=FAKE, ws=FAKE,
             lens=FAKE):
        g = g or _g(lib)
        codec, cache = _codec(lib), _cache(lib)
        return so.lla_decode_attn_loops(ctypes.byref(g), ctypes.byref(codec), ctypes.byref(cache),
                                        lens, B, max_ctx, q, ck, cv, io, out, ws, 1 << 20, None)
    assert call(ck=None) == INVALID
    assert call(B=-1) == INVALID
    assert call(q=None) == INVALID
    assert call(max_ctx=4 * 64 + 1) == INVALID
    assert call(g=_g(lib, T=5)) == UNSUPPORTED          # more loops than query slots
    assert call(g=_g(lib, r_k=18, r_v=30)) == UNSUPPORTED
    assert call(g=_g(lib, storage="fp32")) == UNSUPPORTED
    assert call(B=0, q=None, ck=None, cv=None, out=None, ws=None, lens=None) == OK


def test_2d_block_bytes_and_workspace_shapes(lib):
    so = lib.library()
    n = ctypes.c_size_t(0)
    g = _g(lib, r_k=288, r_v=480)
    assert so.lla_cache_2d_block_bytes(ctypes.byref(g), ctypes.byref(n)) == OK
    assert n.value == 64 * (288 + 480) * 2  # one page of 64 tokens for all heads
    for bad in (_g(lib, r_k=72, r_v=120), _g(lib, d=64), _g(lib, H=17, r_k=288, r_v=480),
                _g(lib, r_k=288, r_v=480, storage="fp32")):
        assert so.lla_decode_2d_workspace_size(ctypes.byref(bad), 4, ctypes.byref(n)) == UNSUPPORTED
    assert so.lla_decode_2d_workspace_size(ctypes.byref(g), -1, ctypes.byref(n)) == INVALID
    # rho_2D = 5.33: 2D latents wider than the per-head limit of 512, up to T H d
    wide = _g(lib, r_k=1152, r_v=1920)
    assert so.lla_cache_2d_block_bytes(ctypes.byref(wide), ctypes.byref(n)) == OK
    assert n.value == 64 * (1152 + 1920) * 2
    assert so.lla_cache_block_bytes(ctypes.byref(wide), ctypes.byref(n)) == INVALID  # per-head: <= 512
    too_wide = _g(lib, T=1, H=4, r_k=1152, r_v=1920)  # T H d = 512
    assert so.lla_cache_2d_block_bytes(ctypes.byref(too_wide), ctypes.byref(n)) == INVALID


def test_decode_2d_argument_checks(lib):
    so = lib.library()

    def call(g=None, B=4, max_ctx=128, loop=0, q=FAKE, ck=FAKE, cv=FAKE, io=0, out=FAKE, ws=FAKE,
             lens=FAKE, codec=None):
        g = g or _g(lib, r_k=288, r_v=480)
        codec, cache = codec or _codec(lib), _cache(lib)
        return so.lla_decode_attn_2d(ctypes.byref(g), ctypes.byref(codec), ctypes.byref(cache),
                                     lens, B, max_ctx, loop, q, ck, cv, io, out, ws, 1 << 20, None)
    assert call(ck=None) == INVALID
    assert call(B=-1) == INVALID
    assert call(B=1025) == INVALID
    assert call(loop=4) == INVALID
    assert call(q=None) == INVALID
    assert call(max_ctx=4 * 64 + 1) == INVALID
    assert call(codec=_codec(lib, w_up_v=None)) == INVALID
    assert call(codec=_codec(lib, w_up_k=FAKE + 8)) == INVALID
    assert call(g=_g(lib, r_k=72, r_v=120)) == UNSUPPORTED
    assert call(g=_g(lib, H=32, r_k=288, r_v=480)) == UNSUPPORTED
    assert call(g=_g(lib, r_k=288, r_v=480, storage="fp32")) == UNSUPPORTED
    assert call(B=0, q=None, ck=None, cv=None, out=None, ws=None, lens=None) == OK


def test_encode_2d_argument_checks(lib):
    so = lib.library()

    def call(g=None, N=8, xk=FAKE, xv=FAKE, slots=FAKE, xdt=0, codec=None):
        g = g or _g(lib, r_k=288, r_v=480)
        codec, cache = codec or _codec(lib), _cache(lib)
        return so.lla_encode_2d(ctypes.byref(g), ctypes.byref(codec), ctypes.byref(cache), xk, xv,
                                xdt, slots, N, None)
    assert call(N=-1) == INVALID
    assert call(xk=None) == INVALID
    assert call(slots=None) == INVALID
    assert call(xdt=7) == INVALID
    assert call(xv=FAKE + 4) == INVALID
    assert call(codec=_codec(lib, w_down_k=None)) == INVALID
    assert call(g=_g(lib, H=4096, d=128)) == UNSUPPORTED  # H d past the stack the encode takes
    assert call(N=0, xk=None, xv=None, slots=None) == OK


def test_decoupled_argument_checks(lib):
    so = lib.library()
    n = ctypes.c_size_t(0)
    assert so.lla_rope_plane_bytes(64, ctypes.byref(n)) == OK and n.value == 64 * 64 * 2
    assert so.lla_rope_plane_bytes(40, ctypes.byref(n)) == INVALID
    g = _g(lib)
    for bad in (_g(lib, r_k=72, r_v=120), _g(lib, d=64), _g(lib, storage="fp32")):
        assert so.lla_decode_decoupled_workspace_size(ctypes.byref(bad), 64, 4, ctypes.byref(n)) == UNSUPPORTED
    assert so.lla_decode_decoupled_workspace_size(ctypes.byref(g), 48, 4, ctypes.byref(n)) == UNSUPPORTED

    def call(g=None, B=4, max_ctx=128, loop=0, q=FAKE, qr=FAKE, ck=FAKE, cv=FAKE, ckr=FAKE, io=0,
             out=FAKE, ws=FAKE, lens=FAKE, rope_pool=FAKE, d_rope=64, rope=None):
        g = g or _g(lib)
        codec, cache = _codec(lib), _cache(lib)
        rope = rope or lib.lla_rope(10000.0, 0)
        return so.lla_decode_attn_decoupled(ctypes.byref(g), ctypes.byref(codec), ctypes.byref(cache),
                                            rope_pool, d_rope, ctypes.byref(rope), lens, B, max_ctx, loop,
                                            q, qr, ck, cv, ckr, io, out, ws, 1 << 20, None)
    assert call(ckr=None) == INVALID          # pass 1 needs the current rotary key
    assert call(ck=None, cv=None) == INVALID  # pass 2 takes none
    assert call(qr=None) == INVALID
    assert call(rope_pool=None) == INVALID
    assert call(rope=lib.lla_rope(1.0, 0)) == INVALID
    assert call(rope=lib.lla_rope(10000.0, 5)) == INVALID
    assert call(loop=4) == INVALID
    assert call(max_ctx=4 * 64 + 1) == INVALID
    assert call(d_rope=48) == UNSUPPORTED
    assert call(g=_g(lib, r_k=128, r_v=128)) == UNSUPPORTED
    assert call(B=0, q=None, qr=None, ck=None, cv=None, ckr=None, out=None, ws=None, lens=None) == OK

    def enc(d_rope=64, N=8, k=FAKE, pos=FAKE, slots=FAKE, pool=FAKE, xdt=0, rope=None):
        rope = rope or lib.lla_rope(10000.0, 1)
        return so.lla_encode_rope_keys(d_rope, ctypes.byref(rope), pool, 10, k, xdt, pos, slots, N, None)
    assert enc(d_rope=40) == INVALID
    assert enc(pos=None) == INVALID
    assert enc(pool=FAKE + 8) == INVALID
    assert enc(N=-1) == INVALID
    assert enc(rope=lib.lla_rope(0.5, 0)) == INVALID
    assert enc(N=0, k=None, pos=None, slots=None) == OK


def test_binding_rejects_host_tensors_before_any_launch(lib):
    """A host tensor's address handed to a kernel would be an illegal device address: the binding
    refuses it while marshalling."""
    import torch
    with pytest.raises(ValueError, match="CUDA tensors"):
        lib._ptr(torch.zeros(4))
    with pytest.raises(ValueError, match="contiguous"):
        lib._ptr(torch.zeros(4, 4).t())
    assert lib._ptr(None) is None and lib._ptr(FAKE) == FAKE


def test_two_pass_prefill_order_and_checks(lib):
    """lla_prefill_two_pass with empty prompts (N = 0, B = 0: nothing reaches the GPU): every
    layer's capture in layer order, then the queries loop by loop and layer by layer; a callback's
    status stops it and is returned; missing callbacks and bad dtypes are rejected."""
    so = lib.library()
    D, T = 3, 4
    g = _g(lib, T=T)
    cds = (lib.lla_codec * D)(*[lib.lla_codec(FAKE, FAKE, FAKE, FAKE, None, None) for _ in range(D)])
    chs = (lib.lla_cache * D)(*[lib.lla_cache(FAKE, 10, FAKE, 4) for _ in range(D)])
    order = []

    def cap(layer, pk, pv, stream, user):
        order.append(("c", layer))
        pk[0] = pv[0] = FAKE
        return 0

    def qry(layer, loop, pq, po, stream, user):
        order.append(("q", layer, loop))
        pq[0] = po[0] = FAKE
        return 0

    c, q = lib.CAPTURE_FN(cap), lib.QUERY_FN(qry)

    def call(capture=c, query=q, xdt=0, iodt=0, D=D):
        return so.lla_prefill_two_pass(ctypes.byref(g), D, cds, chs, xdt, FAKE, 0, FAKE, 0, 0, iodt, None,
                                       capture, query, None, None, 0, None)

    assert call() == OK
    assert order == [("c", l) for l in range(D)] + [("q", l, t) for t in range(T) for l in range(D)]
    assert call(xdt=7) == INVALID
    assert call(iodt=7) == INVALID
    assert call(capture=lib.CAPTURE_FN()) == INVALID
    assert call(D=0, capture=lib.CAPTURE_FN(), query=lib.QUERY_FN()) == OK

    def failing(layer, pk, pv, stream, user):
        order.append(("c", layer))
        pk[0] = pv[0] = FAKE
        return UNSUPPORTED if layer == 1 else OK

    order.clear()
    assert call(capture=lib.CAPTURE_FN(failing)) == UNSUPPORTED
    assert order == [("c", 0), ("c", 1)]
