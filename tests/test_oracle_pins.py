"""Pins the CPU oracle to what the paper and the mathematics fix (no GPU needed).

Each test names the passage it follows.  None of them re-types the oracle's own code:
they check it against printed values (tests/golden), closed forms, library routines that
compute the textbook definition (torch SDPA in float64, numpy SVD), an independently
written absorbed formulation (App. J), hand-expanded tiny cases and invariances.
"""
import json
import math
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle

GOLD = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _gold(name):
    with open(os.path.join(GOLD, name)) as f:
        return json.load(f)


def _rng(seed):
    return np.random.default_rng(seed)


def _orthogonal(n, seed):
    q, r = np.linalg.qr(_rng(seed).standard_normal((n, n)))
    return q * np.sign(np.diag(r))


def _sdpa(q, K, V, scale, causal=False):
    """torch's float64 scaled-dot-product attention (textbook softmax attention)."""
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a, dtype=np.float64))
    qq = t(q).reshape(1, 1, -1, K.shape[1])
    out = F.scaled_dot_product_attention(qq, t(K)[None, None], t(V)[None, None],
                                         is_causal=causal, scale=scale)
    return out[0, 0].numpy()


def _random_codec(T, d, r_k, r_v, seed, with_mu=True):
    g = _rng(seed)
    return dict(
        w_up_k=g.standard_normal((T, d, r_k)) / math.sqrt(r_k),
        w_up_v=g.standard_normal((T, d, r_v)) / math.sqrt(r_v),
        mu_k=g.standard_normal(T * d) if with_mu else None,
        mu_v=g.standard_normal(T * d) if with_mu else None,
    )


# ------------------------------------------------------------------ Eq. ratio (Sec. 3)

@pytest.mark.parametrize("table", ["tier4", "huginn", "isocache"])
def test_ratio_matches_printed_values(table):
    g = _gold("ratios.json")[table]
    for r_k, r_v, printed in g["rows"]:
        rho = oracle.ratio(g["T"], g["d_head"], r_k, r_v)
        # printed to two decimals (Huginn: integers, exact)
        tol = 1e-12 if table == "huginn" else 0.005 + 1e-12
        assert abs(rho - printed) <= tol, (r_k, r_v, rho, printed)


def test_cache_bytes_match_table_memory():
    g = _gold("cache_bytes.json")
    for row in g["per_token_kib"]:
        teacher = oracle.teacher_cache_bytes_per_token(4, 16, 128, row["D"], 2) / 1024
        lla4 = oracle.latent_cache_bytes_per_token(16, row["D"], 96, 160, 2) / 1024
        lla21 = oracle.latent_cache_bytes_per_token(16, row["D"], 18, 30, 2) / 1024
        assert (teacher, lla4, lla21) == (row["teacher"], row["lla4"], row["lla21"])
        # the ratio of the two cache sizes is Eq. ratio exactly
        assert teacher / lla4 == oracle.ratio(4, 128, 96, 160)
        assert abs(teacher / lla21 - oracle.ratio(4, 128, 18, 30)) < 1e-12
    m = g["at_1m_context_gib"]
    gib = lambda b: b * m["tokens"] / 2**30
    assert gib(oracle.teacher_cache_bytes_per_token(4, 16, 128, m["D"], 2)) == m["teacher"]
    assert gib(oracle.latent_cache_bytes_per_token(16, m["D"], 96, 160, 2)) == m["lla4"]
    assert gib(oracle.latent_cache_bytes_per_token(16, m["D"], 18, 30, 2)) == m["lla21"]


# ------------------------------------------------------------------ Eqs. encode / decode

def test_full_rank_orthogonal_codec_is_lossless():
    """r = T d with W_down = Q orthogonal and W_up,t = the loop-t row block of Q:
    Eq. decode(Eq. encode(x)) = x for every loop (Sec. 3)."""
    T, d, N = 4, 128, 24
    g = _rng(1)
    Q = _orthogonal(T * d, 2)
    x = g.standard_normal((T, N, d))
    mu = g.standard_normal(T * d)
    c = oracle.encode(x, mu, Q)
    assert c.shape == (N, T * d)
    for t in range(T):
        xhat = oracle.reconstruct(c, Q[t * d:(t + 1) * d, :], mu[t * d:(t + 1) * d])
        np.testing.assert_allclose(xhat, x[t], rtol=0, atol=1e-12)


def test_encode_matches_stacked_projection_definition():
    """Eq. encode with the stacking of the "Teacher cache" paragraph: the latent of token n
    is the centred stacked vector [x_1; ...; x_T] times W_down (numpy matmul)."""
    T, d, N, r = 4, 16, 9, 7
    g = _rng(3)
    x = g.standard_normal((T, N, d))
    mu = g.standard_normal(T * d)
    w = g.standard_normal((T * d, r))
    stacked = np.concatenate([x[t] for t in range(T)], axis=1)  # [N][T d]
    np.testing.assert_allclose(oracle.encode(x, mu, w), (stacked - mu) @ w, rtol=1e-13,
                               atol=1e-12)
    np.testing.assert_allclose(oracle.encode(x, None, w), stacked @ w, rtol=1e-13, atol=1e-12)


def test_svd_initialised_codec_meets_eckart_young():
    """SVD initialisation (Sec. 3, "Initialization and conversion"; App. A): centre per loop,
    W_down = top-r right singular vectors of the stacked-loop matrix, W_up,t = its loop
    slices.  The total squared reconstruction error is then the sum of the trailing
    squared singular values."""
    T, d, N, r = 4, 16, 300, 10
    g = _rng(4)
    spectrum = np.exp(-np.arange(T * d) / 6.0)
    X = (g.standard_normal((N, T * d)) * spectrum) @ _orthogonal(T * d, 5)
    mu = X.mean(axis=0)
    _, S, Vt = np.linalg.svd(X - mu, full_matrices=False)
    w_down = Vt[:r].T  # [T d][r]
    x = np.stack([X[:, t * d:(t + 1) * d] for t in range(T)])  # [T][N][d]
    c = oracle.encode(x, mu, w_down)
    err = 0.0
    for t in range(T):
        xhat = oracle.reconstruct(c, w_down[t * d:(t + 1) * d, :], mu[t * d:(t + 1) * d])
        err += np.sum((x[t] - xhat) ** 2)
    expect = np.sum(S[r:] ** 2)
    assert abs(err - expect) <= 1e-10 * expect


# ------------------------------------------------------------------ attention

def test_attention_matches_torch_sdpa():
    g = _rng(6)
    d, L = 128, 37
    q, K, V = g.standard_normal(d), g.standard_normal((L, d)), g.standard_normal((L, d))
    scale = 1 / math.sqrt(d)
    np.testing.assert_allclose(oracle.attention(q, K, V, scale), _sdpa(q, K, V, scale)[0],
                               rtol=0, atol=1e-13)


def test_attention_large_scores_are_stable():
    """Softmax with max subtraction: huge equal scores still give the mean."""
    d = 4
    q = np.full(d, 1e3)
    K = np.ones((3, d))
    V = np.arange(12.0).reshape(3, d)
    np.testing.assert_allclose(oracle.attention(q, K, V, 1.0), V.mean(axis=0), atol=1e-12)


def test_decode_tiny_case_expanded_by_hand():
    """T=2, d=2, r_k=r_v=1, L=2 at loop t=1, with mu; softmax expanded with math.exp."""
    w_up_k = np.array([[[1.0], [0.0]], [[2.0], [0.0]]])    # [T][d][r_k]
    w_up_v = np.array([[[5.0], [5.0]], [[1.0], [2.0]]])    # [T][d][r_v]
    mu_k = None
    mu_v = np.array([7.0, 7.0, 10.0, 0.0])                 # loop-1 slice = [10, 0]
    c_k = np.array([[1.0], [2.0]])
    c_v = np.array([[1.0], [-1.0]])
    q = np.array([1.0, 3.0])
    # loop 1: Khat = [2 c_k, 0] -> s = [2, 4];  Vhat = [c_v + 10, 2 c_v]
    v0, v1 = np.array([11.0, 2.0]), np.array([9.0, -2.0])
    e2, e4 = math.exp(2.0), math.exp(4.0)
    expect2 = (e2 * v0 + e4 * v1) / (e2 + e4)
    out2 = oracle.decode(1, c_k, c_v, w_up_k, w_up_v, mu_k, mu_v, q, None, None, 1.0)
    np.testing.assert_allclose(out2, expect2, rtol=0, atol=1e-14)
    # pass 1: exact current key [0.5, 0.5] (score 2) and value [3, -3]
    cur_k, cur_v = np.array([0.5, 0.5]), np.array([3.0, -3.0])
    expect1 = (e2 * v0 + e4 * v1 + e2 * cur_v) / (e2 + e4 + e2)
    out1 = oracle.decode(1, c_k, c_v, w_up_k, w_up_v, mu_k, mu_v, q, cur_k, cur_v, 1.0)
    np.testing.assert_allclose(out1, expect1, rtol=0, atol=1e-14)


def _absorbed(t, c_k, c_v, cod, q, cur_k, cur_v, scale):
    """App. J "Absorbed attention", written independently of the oracle: the K up-projection
    moves to the query (q~ = W_up,t^T q) and the V up-projection leaves the softmax sum."""
    d = q.shape[0]
    Wk, Wv = cod["w_up_k"][t], cod["w_up_v"][t]
    mk = np.zeros(d) if cod["mu_k"] is None else cod["mu_k"][t * d:(t + 1) * d]
    mv = np.zeros(d) if cod["mu_v"] is None else cod["mu_v"][t * d:(t + 1) * d]
    q_lat = Wk.T @ q
    s = scale * (c_k @ q_lat + q @ mk)
    if cur_k is not None:
        s = np.append(s, scale * (q @ cur_k))
    p = np.exp(s - s.max())
    L = c_k.shape[0]
    o_lat = p[:L] @ c_v
    o = Wv @ o_lat + p[:L].sum() * mv
    if cur_k is not None:
        o = o + p[L] * cur_v
    return o / p.sum()


@pytest.mark.parametrize("pass1", [False, True])
@pytest.mark.parametrize("with_mu", [False, True])
def test_decode_equals_absorbed_formulation(pass1, with_mu):
    T, d, r_k, r_v, L = 4, 128, 96, 160, 70
    g = _rng(7)
    cod = _random_codec(T, d, r_k, r_v, 8, with_mu)
    c_k, c_v = g.standard_normal((L, r_k)), g.standard_normal((L, r_v))
    q = g.standard_normal(d)
    cur_k = g.standard_normal(d) if pass1 else None
    cur_v = g.standard_normal(d) if pass1 else None
    scale = 1 / math.sqrt(d)
    for t in range(T):
        out = oracle.decode(t, c_k, c_v, cod["w_up_k"], cod["w_up_v"], cod["mu_k"],
                            cod["mu_v"], q, cur_k, cur_v, scale)
        ref = _absorbed(t, c_k, c_v, cod, q, cur_k, cur_v, scale)
        np.testing.assert_allclose(out, ref, rtol=0, atol=1e-12)


@pytest.mark.parametrize("pass1", [False, True])
def test_full_rank_decode_equals_uncompressed_attention(pass1):
    """With the lossless full-rank codec, LLA decode is exactly uncompressed loop-t attention
    (Sec. 3 "Teacher cache"), computed here by torch SDPA on the raw per-loop K/V."""
    T, d, L = 4, 128, 33
    g = _rng(9)
    Qk, Qv = _orthogonal(T * d, 10), _orthogonal(T * d, 11)
    xk, xv = g.standard_normal((T, L + 1, d)), g.standard_normal((T, L + 1, d))
    mu_k, mu_v = g.standard_normal(T * d), g.standard_normal(T * d)
    n_cached = L if pass1 else L + 1
    c_k = oracle.encode(xk[:, :n_cached], mu_k, Qk)
    c_v = oracle.encode(xv[:, :n_cached], mu_v, Qv)
    w_up_k = np.stack([Qk[t * d:(t + 1) * d] for t in range(T)])
    w_up_v = np.stack([Qv[t * d:(t + 1) * d] for t in range(T)])
    scale = 1 / math.sqrt(d)
    for t in range(T):
        q = g.standard_normal(d)
        cur_k = xk[t, L] if pass1 else None
        cur_v = xv[t, L] if pass1 else None
        out = oracle.decode(t, c_k, c_v, w_up_k, w_up_v, mu_k, mu_v, q, cur_k, cur_v, scale)
        ref = _sdpa(q, xk[t], xv[t], scale)[0]
        np.testing.assert_allclose(out, ref, rtol=0, atol=1e-12)


def test_decode_special_cases():
    T, d, r_k, r_v = 4, 128, 96, 160
    g = _rng(12)
    cod = _random_codec(T, d, r_k, r_v, 13)
    scale = 1 / math.sqrt(d)
    t = 2
    # one cached token, pass 2: the output is that token's reconstructed value
    c_k, c_v = g.standard_normal((1, r_k)), g.standard_normal((1, r_v))
    q = g.standard_normal(d)
    out = oracle.decode(t, c_k, c_v, cod["w_up_k"], cod["w_up_v"], cod["mu_k"], cod["mu_v"],
                        q, None, None, scale)
    vhat = oracle.reconstruct(c_v, cod["w_up_v"][t], cod["mu_v"][t * d:(t + 1) * d])[0]
    np.testing.assert_allclose(out, vhat, rtol=0, atol=1e-12)
    # zero query: uniform weights, the mean of the reconstructed values
    L = 50
    c_k, c_v = g.standard_normal((L, r_k)), g.standard_normal((L, r_v))
    out = oracle.decode(t, c_k, c_v, cod["w_up_k"], cod["w_up_v"], cod["mu_k"], cod["mu_v"],
                        np.zeros(d), None, None, scale)
    vhat = oracle.reconstruct(c_v, cod["w_up_v"][t], cod["mu_v"][t * d:(t + 1) * d])
    np.testing.assert_allclose(out, vhat.mean(axis=0), rtol=0, atol=1e-12)
    # pass 1 with an empty cache: the current token's own value
    cur_k, cur_v = g.standard_normal(d), g.standard_normal(d)
    out = oracle.decode(t, np.zeros((0, r_k)), np.zeros((0, r_v)), cod["w_up_k"],
                        cod["w_up_v"], cod["mu_k"], cod["mu_v"], q, cur_k, cur_v, scale)
    np.testing.assert_array_equal(out, cur_v)
    # pass 2 with an empty cache is not defined
    with pytest.raises(ValueError):
        oracle.decode(t, np.zeros((0, r_k)), np.zeros((0, r_v)), cod["w_up_k"],
                      cod["w_up_v"], None, None, q, None, None, scale)


def test_mu_shift_invariances():
    """Shifting mu^K by delta moves every reconstructed key by delta_t: pass-2 scores all
    shift by one constant and the output is unchanged; pass 1's exact current key does
    not move, so there the output changes.  Shifting mu^V by delta moves every
    reconstructed value by delta_t: the pass-2 output moves by delta_t exactly, the pass-1
    output by (1 - a_cur) delta_t."""
    T, d, r_k, r_v, L = 4, 128, 96, 160, 40
    g = _rng(14)
    cod = _random_codec(T, d, r_k, r_v, 15)
    c_k, c_v = g.standard_normal((L, r_k)), g.standard_normal((L, r_v))
    q, cur_k, cur_v = g.standard_normal(d), g.standard_normal(d), g.standard_normal(d)
    delta = g.standard_normal(T * d)
    scale = 1 / math.sqrt(d)
    t = 1
    dec = lambda mk, mv, ck, cv: oracle.decode(t, c_k, c_v, cod["w_up_k"], cod["w_up_v"], mk,
                                               mv, q, ck, cv, scale)
    base2 = dec(cod["mu_k"], cod["mu_v"], None, None)
    np.testing.assert_allclose(dec(cod["mu_k"] + delta, cod["mu_v"], None, None), base2,
                               rtol=0, atol=1e-12)
    base1 = dec(cod["mu_k"], cod["mu_v"], cur_k, cur_v)
    assert np.abs(dec(cod["mu_k"] + 3 * delta, cod["mu_v"], cur_k, cur_v) - base1).max() > 1e-3
    dt = delta[t * d:(t + 1) * d]
    np.testing.assert_allclose(dec(cod["mu_k"], cod["mu_v"] + delta, None, None), base2 + dt,
                               rtol=0, atol=1e-12)
    # pass-1 weight of the current token, from the definition of the softmax
    Khat = oracle.reconstruct(c_k, cod["w_up_k"][t], cod["mu_k"][t * d:(t + 1) * d])
    s = scale * np.append(Khat @ q, q @ cur_k)
    a_cur = np.exp(s[-1] - s.max()) / np.exp(s - s.max()).sum()
    np.testing.assert_allclose(dec(cod["mu_k"], cod["mu_v"] + delta, cur_k, cur_v),
                               base1 + (1 - a_cur) * dt, rtol=0, atol=1e-12)


# ------------------------------------------------------------------ prefill

def test_prefill_matches_causal_sdpa_and_decode():
    T, d, r_k, r_v, N = 4, 128, 96, 160, 45
    g = _rng(16)
    cod = _random_codec(T, d, r_k, r_v, 17)
    c_k, c_v = g.standard_normal((N, r_k)), g.standard_normal((N, r_v))
    q = g.standard_normal((N, d))
    scale = 1 / math.sqrt(d)
    t = 3
    out = oracle.prefill(t, c_k, c_v, cod["w_up_k"], cod["w_up_v"], cod["mu_k"], cod["mu_v"],
                         q, scale)
    K = oracle.reconstruct(c_k, cod["w_up_k"][t], cod["mu_k"][t * d:(t + 1) * d])
    V = oracle.reconstruct(c_v, cod["w_up_v"][t], cod["mu_v"][t * d:(t + 1) * d])
    np.testing.assert_allclose(out, _sdpa(q, K, V, scale, causal=True), rtol=0, atol=1e-12)
    for i in (0, 1, 17, N - 1):
        row = oracle.decode(t, c_k[:i + 1], c_v[:i + 1], cod["w_up_k"], cod["w_up_v"],
                            cod["mu_k"], cod["mu_v"], q[i], None, None, scale)
        np.testing.assert_allclose(out[i], row, rtol=0, atol=1e-12)


# ------------------------------------------------------------------ batched drivers

def test_batched_drivers_equal_single_calls():
    T, d, r_k, r_v = 4, 32, 12, 20
    g = _rng(18)
    cod = _random_codec(T, d, r_k, r_v, 19)
    scale = 0.3
    items = []
    for k in range(9):
        L = int(g.integers(0, 20))
        pass1 = L == 0 or k % 2 == 0
        items.append(dict(t=k % T, c_k=g.standard_normal((L, r_k)),
                          c_v=g.standard_normal((L, r_v)), q=g.standard_normal(d),
                          cur_k=g.standard_normal(d) if pass1 else None,
                          cur_v=g.standard_normal(d) if pass1 else None, **cod))
    outs = oracle.decode_batch(T, d, r_k, r_v, scale, items, n_threads=3)
    for it, o in zip(items, outs):
        ref = oracle.decode(it["t"], it["c_k"], it["c_v"], cod["w_up_k"], cod["w_up_v"],
                            cod["mu_k"], cod["mu_v"], it["q"], it["cur_k"], it["cur_v"], scale)
        np.testing.assert_array_equal(o, ref)
    enc_items = [dict(x=g.standard_normal((T, 5, d)), mu=g.standard_normal(T * d),
                      w_down=g.standard_normal((T * d, r))) for r in (3, 8)]
    for it, c in zip(enc_items, oracle.encode_batch(T, d, enc_items, n_threads=2)):
        np.testing.assert_array_equal(c, oracle.encode(it["x"], it["mu"], it["w_down"]))


# ------------------------------------------------------------------ RoPE after reconstruction
# Sec. 3 "RoPE and reconstruction": the codec holds pre-RoPE keys and the rotation (RoFormer)
# is applied to each reconstructed key at its token's position.

def _rot_complex(x, pos, base, pairing):
    """RoFormer's complex form: pair j as a complex number, multiplied by exp(i pos theta_j),
    theta_j = base^(-2j/d)."""
    d = x.shape[-1]
    h = d // 2
    theta = base ** (-2.0 * np.arange(h) / d)
    z = (x[:h] + 1j * x[h:]) if pairing == 0 else (x[0::2] + 1j * x[1::2])
    z = z * np.exp(1j * pos * theta)
    y = np.empty(d)
    if pairing == 0:
        y[:h], y[h:] = z.real, z.imag
    else:
        y[0::2], y[1::2] = z.real, z.imag
    return y


@pytest.mark.parametrize("pairing", [oracle.ROPE_HALF, oracle.ROPE_ADJACENT])
def test_rope_closed_form_pair_scores(pairing):
    """Unit vectors of one pair: rot(e_a, P) . rot(e_a, p) = cos((P - p) theta_j) and
    rot(e_a, P) . rot(e_b, p) = sin((P - p) theta_j); at d = 128 and base 10^4 the pair j = 32
    turns at theta = 0.01 and j = 0 at theta = 1."""
    d = 128
    for j, theta in ((0, 1.0), (32, 0.01), (63, 10000.0 ** (-126 / 128))):
        a, b = (j, j + 64) if pairing == oracle.ROPE_HALF else (2 * j, 2 * j + 1)
        ea, eb = np.zeros(d), np.zeros(d)
        ea[a], eb[b] = 1.0, 1.0
        for P, p in ((5, 2), (4097, 0), (30000, 29999), (7, 7)):
            qa = oracle.rope(ea, P, 10000.0, pairing)
            assert qa @ oracle.rope(ea, p, 10000.0, pairing) == pytest.approx(
                math.cos((P - p) * theta), abs=1e-12)
            assert qa @ oracle.rope(eb, p, 10000.0, pairing) == pytest.approx(
                math.sin((P - p) * theta), abs=1e-12)


@pytest.mark.parametrize("pairing", [oracle.ROPE_HALF, oracle.ROPE_ADJACENT])
def test_rope_is_a_rotation(pairing):
    """Complex multiplication form, norm preservation, rot(x, 0) = x, and
    rot(rot(x, a), b) = rot(x, a + b)."""
    g = _rng(40)
    for d, base in ((128, 10000.0), (64, 500000.0), (8, 10.0)):
        x = g.standard_normal(d)
        for pos in (0, 1, 17, 4095, 32767):
            y = oracle.rope(x, pos, base, pairing)
            # the angle pos * theta_j carries one rounding of theta_j, scaled by pos
            np.testing.assert_allclose(y, _rot_complex(x, pos, base, pairing), rtol=0,
                                       atol=1e-13 * (1 + pos))
            assert np.linalg.norm(y) == pytest.approx(np.linalg.norm(x), rel=1e-14)
        np.testing.assert_array_equal(oracle.rope(x, 0, base, pairing), x)
        np.testing.assert_allclose(
            oracle.rope(oracle.rope(x, 300, base, pairing), 1234, base, pairing),
            oracle.rope(x, 1534, base, pairing), rtol=0, atol=1e-12)


@pytest.mark.parametrize("pairing", [oracle.ROPE_HALF, oracle.ROPE_ADJACENT])
def test_rope_decode_tiny_case_expanded_by_hand(pairing):
    """T = 1, d = 4, identity codec (Khat = c_k, Vhat = c_v), base 10^4: the two pairs turn at
    theta = 1 and theta = 0.01.  Two keys at positions 0 and 1, the query at position 1 (pass 2
    with L = 2, or pass 1 with one cached token and the current one)."""
    e = np.eye(4)
    if pairing == oracle.ROPE_HALF:  # pairs (0, 2) and (1, 3)
        a0, b0, a1 = 0, 2, 1
    else:                            # pairs (0, 1) and (2, 3)
        a0, b0, a1 = 0, 1, 2
    q = e[a0] + e[a1]
    k0 = e[b0] + e[a1]   # position 0: distance 1 from the query
    k1 = e[a0]           # position 1: same position as the query, plain dot product 1
    v0, v1 = np.array([1.0, 2.0, 3.0, 4.0]), np.array([-1.0, 0.0, 5.0, 2.0])
    scale = 0.7
    s0 = scale * (math.sin(1.0) + math.cos(0.01))
    s1 = scale * 1.0
    expect = (math.exp(s0) * v0 + math.exp(s1) * v1) / (math.exp(s0) + math.exp(s1))
    w = np.eye(4)[None]
    out2 = oracle.decode_rope(0, np.stack([k0, k1]), np.stack([v0, v1]), w, w, None, None, q,
                              None, None, scale, 10000.0, pairing)
    np.testing.assert_allclose(out2, expect, rtol=0, atol=1e-14)
    out1 = oracle.decode_rope(0, k0[None], v0[None], w, w, None, None, q, k1, v1, scale,
                              10000.0, pairing)
    np.testing.assert_allclose(out1, expect, rtol=0, atol=1e-14)


def _relative_form(t, c_k, c_v, cod, q, cur_k, cur_v, scale, base, pairing):
    """The same attention written through relative positions, independently of the oracle:
    rot(q, P) . rot(k_i, p_i) = rot(q, P - p_i) . k_i, with Khat and Vhat by Eq. decode in numpy."""
    d = q.shape[0]
    L = c_k.shape[0]
    mk = np.zeros(d) if cod["mu_k"] is None else cod["mu_k"][t * d:(t + 1) * d]
    mv = np.zeros(d) if cod["mu_v"] is None else cod["mu_v"][t * d:(t + 1) * d]
    K = c_k @ cod["w_up_k"][t].T + mk
    V = c_v @ cod["w_up_v"][t].T + mv
    if cur_k is not None:
        K, V = np.vstack([K, cur_k]), np.vstack([V, cur_v])
    P = K.shape[0] - 1
    s = np.array([scale * (_rot_complex(q, P - i, base, pairing) @ K[i]) for i in range(P + 1)])
    p = np.exp(s - s.max())
    return (p @ V) / p.sum()


@pytest.mark.parametrize("pass1", [False, True])
@pytest.mark.parametrize("pairing", [oracle.ROPE_HALF, oracle.ROPE_ADJACENT])
def test_rope_decode_equals_relative_position_form(pass1, pairing):
    T, d, r_k, r_v, L = 4, 128, 96, 160, 150
    g = _rng(41)
    cod = _random_codec(T, d, r_k, r_v, 42)
    c_k, c_v = g.standard_normal((L, r_k)), g.standard_normal((L, r_v))
    q = g.standard_normal(d)
    cur_k = g.standard_normal(d) if pass1 else None
    cur_v = g.standard_normal(d) if pass1 else None
    scale = 1 / math.sqrt(d)
    for t in (0, 3):
        out = oracle.decode_rope(t, c_k, c_v, cod["w_up_k"], cod["w_up_v"], cod["mu_k"],
                                 cod["mu_v"], q, cur_k, cur_v, scale, 10000.0, pairing)
        ref = _relative_form(t, c_k, c_v, cod, q, cur_k, cur_v, scale, 10000.0, pairing)
        np.testing.assert_allclose(out, ref, rtol=0, atol=1e-12)


@pytest.mark.parametrize("pass1", [False, True])
def test_rope_decode_depends_on_relative_positions_only(pass1):
    """Moving every position by the same offset leaves the output unchanged; a different
    rotation base changes it."""
    T, d, r_k, r_v, L = 2, 128, 96, 160, 60
    g = _rng(43)
    cod = _random_codec(T, d, r_k, r_v, 44)
    c_k, c_v = g.standard_normal((L, r_k)), g.standard_normal((L, r_v))
    q = 3 * g.standard_normal(d)
    cur_k = g.standard_normal(d) if pass1 else None
    cur_v = g.standard_normal(d) if pass1 else None
    dec = lambda pos0, base: oracle.decode_rope(1, c_k, c_v, cod["w_up_k"], cod["w_up_v"],
                                                cod["mu_k"], cod["mu_v"], q, cur_k, cur_v,
                                                0.125, base, oracle.ROPE_HALF, pos0)
    base_out = dec(0, 10000.0)
    for pos0 in (1, 1000, 123457):
        np.testing.assert_allclose(dec(pos0, 10000.0), base_out, rtol=0, atol=1e-11)
    assert np.abs(dec(0, 500000.0) - base_out).max() > 1e-3


@pytest.mark.parametrize("pass1", [False, True])
def test_rope_full_rank_decode_equals_uncompressed_attention(pass1):
    """Lossless full-rank codec: LLA decode with RoPE is exactly RoPE attention over the raw
    loop-t keys and values (torch SDPA over keys and query rotated in complex form)."""
    T, d, L = 2, 128, 25
    g = _rng(45)
    Qk, Qv = _orthogonal(T * d, 46), _orthogonal(T * d, 47)
    xk, xv = g.standard_normal((T, L + 1, d)), g.standard_normal((T, L + 1, d))
    mu_k, mu_v = g.standard_normal(T * d), g.standard_normal(T * d)
    n_cached = L if pass1 else L + 1
    c_k = oracle.encode(xk[:, :n_cached], mu_k, Qk)
    c_v = oracle.encode(xv[:, :n_cached], mu_v, Qv)
    w_up_k = np.stack([Qk[t * d:(t + 1) * d] for t in range(T)])
    w_up_v = np.stack([Qv[t * d:(t + 1) * d] for t in range(T)])
    scale = 1 / math.sqrt(d)
    for t in range(T):
        q = g.standard_normal(d)
        out = oracle.decode_rope(t, c_k, c_v, w_up_k, w_up_v, mu_k, mu_v, q,
                                 xk[t, L] if pass1 else None, xv[t, L] if pass1 else None,
                                 scale, 10000.0, oracle.ROPE_HALF)
        Kr = np.stack([_rot_complex(xk[t, i], i, 10000.0, 0) for i in range(L + 1)])
        ref = _sdpa(_rot_complex(q, L, 10000.0, 0), Kr, xv[t], scale)[0]
        np.testing.assert_allclose(out, ref, rtol=0, atol=1e-12)


@pytest.mark.parametrize("pairing", [oracle.ROPE_HALF, oracle.ROPE_ADJACENT])
def test_rope_prefill_matches_causal_sdpa_and_decode(pairing):
    T, d, r_k, r_v, N = 4, 128, 96, 160, 40
    g = _rng(48)
    cod = _random_codec(T, d, r_k, r_v, 49)
    c_k, c_v = g.standard_normal((N, r_k)), g.standard_normal((N, r_v))
    q = g.standard_normal((N, d))
    scale = 1 / math.sqrt(d)
    t = 2
    out = oracle.prefill_rope(t, c_k, c_v, cod["w_up_k"], cod["w_up_v"], cod["mu_k"],
                              cod["mu_v"], q, scale, 10000.0, pairing)
    K = c_k @ cod["w_up_k"][t].T + cod["mu_k"][t * d:(t + 1) * d]
    V = c_v @ cod["w_up_v"][t].T + cod["mu_v"][t * d:(t + 1) * d]
    Kr = np.stack([_rot_complex(K[i], i, 10000.0, pairing) for i in range(N)])
    Qr = np.stack([_rot_complex(q[i], i, 10000.0, pairing) for i in range(N)])
    np.testing.assert_allclose(out, _sdpa(Qr, Kr, V, scale, causal=True), rtol=0, atol=1e-12)
    for i in (0, 1, 23, N - 1):
        row = oracle.decode_rope(t, c_k[:i + 1], c_v[:i + 1], cod["w_up_k"], cod["w_up_v"],
                                 cod["mu_k"], cod["mu_v"], q[i], None, None, scale, 10000.0,
                                 pairing)
        np.testing.assert_allclose(out[i], row, rtol=0, atol=1e-12)


def test_rope_batched_driver_equals_single_calls():
    T, d, r_k, r_v = 2, 32, 16, 24
    g = _rng(50)
    cod = _random_codec(T, d, r_k, r_v, 51)
    items = []
    for k in range(6):
        L = int(g.integers(1, 30))
        pass1 = k % 2 == 0
        items.append(dict(t=k % T, c_k=g.standard_normal((L, r_k)),
                          c_v=g.standard_normal((L, r_v)), q=g.standard_normal(d),
                          cur_k=g.standard_normal(d) if pass1 else None,
                          cur_v=g.standard_normal(d) if pass1 else None,
                          rope=(k % 2, 10000.0 if k < 3 else 1e6), **cod))
    outs = oracle.decode_batch(T, d, r_k, r_v, 0.2, items, n_threads=2)
    for it, o in zip(items, outs):
        ref = oracle.decode_rope(it["t"], it["c_k"], it["c_v"], cod["w_up_k"], cod["w_up_v"],
                                 cod["mu_k"], cod["mu_v"], it["q"], it["cur_k"], it["cur_v"],
                                 0.2, it["rope"][1], it["rope"][0])
        np.testing.assert_array_equal(o, ref)


# ------------------------------------------------------------------ LLA-2D (Sec. 3)

def test_ratio_2d_matches_printed_values():
    """Table isocache prints LLA-2D at rho = 5.33 and 21.33 at the per-head rows' cache budget;
    rho_2D = 2 T H d / (r_k + r_v), a factor H above per-head LLA at fixed ranks (App. J "Per-
    head LLA versus LLA-2D at inference")."""
    g = _gold("ratios.json")["isocache_2d"]
    T, H, d = g["T"], g["H"], g["d_head"]
    for r_k, r_v, printed in g["rows"]:
        rho = oracle.ratio_2d(T, H, d, r_k, r_v)
        assert abs(rho - printed) <= 0.005 + 1e-12, (r_k, r_v, rho, printed)
        # matched budget: the 2D latent per token and layer is as large as the H per-head ones
        assert oracle.latent_cache_bytes_per_token(1, 1, r_k, r_v, 2) == \
            oracle.latent_cache_bytes_per_token(H, 1, r_k // H, r_v // H, 2)
        assert rho == oracle.ratio(T, d, r_k // H, r_v // H)
    assert oracle.ratio_2d(4, 16, 128, 96, 160) == 16 * oracle.ratio(4, 128, 96, 160)


def test_encode_2d_matches_loop_major_stack():
    """The 2D stack runs over loops and heads (loop-major, then head): the latent of token n is
    the centred [x_{1,1}; ...; x_{1,H}; ...; x_{T,H}] times W_down (numpy matmul)."""
    T, H, d, N, r = 3, 2, 8, 5, 7
    g = _rng(60)
    x = g.standard_normal((T, N, H, d))
    mu = g.standard_normal(T * H * d)
    w = g.standard_normal((T * H * d, r))
    stacked = np.concatenate([x[t, :, h] for t in range(T) for h in range(H)], axis=1)
    np.testing.assert_allclose(oracle.encode_2d(x, mu, w), (stacked - mu) @ w, rtol=1e-13,
                               atol=1e-12)
    np.testing.assert_allclose(oracle.encode_2d(x, None, w), stacked @ w, rtol=1e-13,
                               atol=1e-12)


@pytest.mark.parametrize("pass1", [False, True])
def test_full_rank_2d_decode_equals_uncompressed_attention(pass1):
    """r = T H d with W_down = Q orthogonal and W_up,t,h = the (t, h) row block of Q: every
    head's keys and values come back exactly, so LLA-2D decode is uncompressed loop-t attention
    of that head (torch SDPA on the raw K/V)."""
    T, H, d, L = 2, 3, 8, 11
    g = _rng(61)
    S = T * H * d
    Qk, Qv = _orthogonal(S, 62), _orthogonal(S, 63)
    xk, xv = g.standard_normal((T, L + 1, H, d)), g.standard_normal((T, L + 1, H, d))
    mu_k, mu_v = g.standard_normal(S), g.standard_normal(S)
    n_cached = L if pass1 else L + 1
    c_k = oracle.encode_2d(xk[:, :n_cached], mu_k, Qk)
    c_v = oracle.encode_2d(xv[:, :n_cached], mu_v, Qv)
    blk = lambda Q, t, h: Q[(t * H + h) * d:(t * H + h + 1) * d]
    w_up_k = np.stack([np.stack([blk(Qk, t, h) for h in range(H)]) for t in range(T)])
    w_up_v = np.stack([np.stack([blk(Qv, t, h) for h in range(H)]) for t in range(T)])
    scale = 1 / math.sqrt(d)
    for t in range(T):
        q = g.standard_normal((H, d))
        cur_k = xk[t, L] if pass1 else None
        cur_v = xv[t, L] if pass1 else None
        out = oracle.decode_2d(t, c_k, c_v, w_up_k, w_up_v, mu_k, mu_v, q, cur_k, cur_v, scale)
        for h in range(H):
            ref = _sdpa(q[h], xk[t, :, h], xv[t, :, h], scale)[0]
            np.testing.assert_allclose(out[h], ref, rtol=0, atol=1e-12)


def _block_2d_codec(T, H, d, r_k, r_v, seed):
    """H per-head codecs arranged as one 2D codec: latent columns h r .. (h+1) r - 1 belong to
    head h, W_up,t,h is zero outside them."""
    per = [_random_codec(T, d, r_k, r_v, seed + h) for h in range(H)]
    g = _rng(seed + 100)
    down = {}
    two = {}
    for ax, r in (("k", r_k), ("v", r_v)):
        wd = [g.standard_normal((T * d, r)) / math.sqrt(T * d) for _ in range(H)]
        W = np.zeros((T * H * d, H * r))
        up = np.zeros((T, H, d, H * r))
        mu = np.zeros(T * H * d)
        for h in range(H):
            for t in range(T):
                rows = slice((t * H + h) * d, (t * H + h + 1) * d)
                W[rows, h * r:(h + 1) * r] = wd[h][t * d:(t + 1) * d]
                up[t, h, :, h * r:(h + 1) * r] = per[h]["w_up_" + ax][t]
                mu[rows] = per[h]["mu_" + ax][t * d:(t + 1) * d]
        down[ax] = wd
        two.update({"w_down_" + ax: W, "w_up_" + ax: up, "mu_" + ax: mu})
    return per, down, two


@pytest.mark.parametrize("pass1", [False, True])
def test_block_diagonal_2d_codec_equals_per_head_lla(pass1):
    """A 2D codec that keeps each head in its own block of the latent is H per-head codecs side
    by side (Sec. 3: per-head LLA is LLA-2D without the cross-head coupling): its encode is the
    per-head latents concatenated and its decode is per-head decode, head by head."""
    T, H, d, r_k, r_v, L = 3, 2, 16, 5, 7, 9
    g = _rng(64)
    per, down, two = _block_2d_codec(T, H, d, r_k, r_v, 65)
    xk, xv = g.standard_normal((T, L, H, d)), g.standard_normal((T, L, H, d))
    c_k = oracle.encode_2d(xk, two["mu_k"], two["w_down_k"])
    c_v = oracle.encode_2d(xv, two["mu_v"], two["w_down_v"])
    for h in range(H):
        np.testing.assert_allclose(c_k[:, h * r_k:(h + 1) * r_k],
                                   oracle.encode(xk[:, :, h], per[h]["mu_k"], down["k"][h]),
                                   rtol=0, atol=1e-12)
        np.testing.assert_allclose(c_v[:, h * r_v:(h + 1) * r_v],
                                   oracle.encode(xv[:, :, h], per[h]["mu_v"], down["v"][h]),
                                   rtol=0, atol=1e-12)
    scale = 1 / math.sqrt(d)
    q = g.standard_normal((H, d))
    cur_k = g.standard_normal((H, d)) if pass1 else None
    cur_v = g.standard_normal((H, d)) if pass1 else None
    for t in range(T):
        out = oracle.decode_2d(t, c_k, c_v, two["w_up_k"], two["w_up_v"], two["mu_k"],
                               two["mu_v"], q, cur_k, cur_v, scale)
        for h in range(H):
            ref = oracle.decode(t, c_k[:, h * r_k:(h + 1) * r_k], c_v[:, h * r_v:(h + 1) * r_v],
                                per[h]["w_up_k"], per[h]["w_up_v"], per[h]["mu_k"],
                                per[h]["mu_v"], q[h], None if cur_k is None else cur_k[h],
                                None if cur_v is None else cur_v[h], scale)
            np.testing.assert_allclose(out[h], ref, rtol=0, atol=1e-12)


def test_svd_initialised_2d_codec_meets_eckart_young():
    """SVD initialisation of the 2D codec over the (loop, head) stack: the squared
    reconstruction error summed over every loop and head is the sum of the trailing squared
    singular values of the stacked matrix."""
    T, H, d, N, r = 2, 3, 8, 200, 9
    g = _rng(66)
    S = T * H * d
    spectrum = np.exp(-np.arange(S) / 5.0)
    X = (g.standard_normal((N, S)) * spectrum) @ _orthogonal(S, 67)
    mu = X.mean(axis=0)
    _, sv, Vt = np.linalg.svd(X - mu, full_matrices=False)
    w_down = Vt[:r].T
    x = np.stack([np.stack([X[:, (t * H + h) * d:(t * H + h + 1) * d] for h in range(H)], axis=1)
                  for t in range(T)])  # [T][N][H][d]
    c = oracle.encode_2d(x, mu, w_down)
    err = 0.0
    for t in range(T):
        for h in range(H):
            rows = slice((t * H + h) * d, (t * H + h + 1) * d)
            xhat = oracle.reconstruct(c, w_down[rows], mu[rows])
            err += np.sum((x[t, :, h] - xhat) ** 2)
    expect = np.sum(sv[r:] ** 2)
    assert abs(err - expect) <= 1e-10 * expect


def _absorbed_2d(t, h, c_k, c_v, up_k, up_v, mu_k, mu_v, q, cur_k, cur_v, scale):
    """App. J "Absorbed attention" for head h of a 2D codec, written independently of the
    oracle: q~ = W_up,t,h^T q against the shared latent, the value sum kept in latent space."""
    H, d = up_k.shape[1], q.shape[0]
    sl = slice((t * H + h) * d, (t * H + h + 1) * d)
    s = scale * (c_k @ (up_k[t, h].T @ q) + (0.0 if mu_k is None else q @ mu_k[sl]))
    if cur_k is not None:
        s = np.append(s, scale * (q @ cur_k))
    p = np.exp(s - s.max())
    L = c_k.shape[0]
    o = up_v[t, h] @ (p[:L] @ c_v) + (0.0 if mu_v is None else p[:L].sum() * mu_v[sl])
    if cur_k is not None:
        o = o + p[L] * cur_v
    return o / p.sum()


@pytest.mark.parametrize("pass1", [False, True])
def test_decode_2d_equals_absorbed_formulation(pass1):
    T, H, d, r_k, r_v, L = 4, 4, 32, 24, 40, 37
    g = _rng(68)
    up_k = g.standard_normal((T, H, d, r_k)) / math.sqrt(r_k)
    up_v = g.standard_normal((T, H, d, r_v)) / math.sqrt(r_v)
    mu_k, mu_v = g.standard_normal(T * H * d), g.standard_normal(T * H * d)
    c_k, c_v = g.standard_normal((L, r_k)), g.standard_normal((L, r_v))
    q = g.standard_normal((H, d))
    cur_k = g.standard_normal((H, d)) if pass1 else None
    cur_v = g.standard_normal((H, d)) if pass1 else None
    scale = 1 / math.sqrt(d)
    for t in range(T):
        out = oracle.decode_2d(t, c_k, c_v, up_k, up_v, mu_k, mu_v, q, cur_k, cur_v, scale)
        for h in range(H):
            ref = _absorbed_2d(t, h, c_k, c_v, up_k, up_v, mu_k, mu_v, q[h],
                               None if cur_k is None else cur_k[h],
                               None if cur_v is None else cur_v[h], scale)
            np.testing.assert_allclose(out[h], ref, rtol=0, atol=1e-12)


def test_decode_2d_special_cases():
    """One cached token in pass 2 returns its rebuilt value; pass 1 with an empty cache returns
    the current value; a zero query averages the rebuilt values (uniform softmax)."""
    T, H, d, r_k, r_v = 2, 3, 8, 6, 10
    g = _rng(69)
    up_k = g.standard_normal((T, H, d, r_k))
    up_v = g.standard_normal((T, H, d, r_v))
    mu_v = g.standard_normal(T * H * d)
    c_k, c_v = g.standard_normal((5, r_k)), g.standard_normal((5, r_v))
    q = g.standard_normal((H, d))
    for t in range(T):
        one = oracle.decode_2d(t, c_k[:1], c_v[:1], up_k, up_v, None, mu_v, q, None, None, 0.3)
        zero = oracle.decode_2d(t, c_k, c_v, up_k, up_v, None, mu_v, np.zeros((H, d)), None,
                                None, 0.3)
        cv = g.standard_normal((H, d))
        empty = oracle.decode_2d(t, c_k[:0], c_v[:0], up_k, up_v, None, mu_v, q,
                                 g.standard_normal((H, d)), cv, 0.3)
        for h in range(H):
            sl = slice((t * H + h) * d, (t * H + h + 1) * d)
            np.testing.assert_allclose(one[h], up_v[t, h] @ c_v[0] + mu_v[sl], rtol=0, atol=1e-12)
            np.testing.assert_allclose(zero[h], up_v[t, h] @ c_v.mean(axis=0) + mu_v[sl],
                                       rtol=0, atol=1e-12)
        np.testing.assert_allclose(empty, cv, rtol=0, atol=0)


# ------------------------------------------------------------------ decoupled rotary branch (App. J)

@pytest.mark.parametrize("pass1", [False, True])
@pytest.mark.parametrize("pairing", [oracle.ROPE_HALF, oracle.ROPE_ADJACENT])
def test_decoupled_full_rank_equals_sdpa_on_joined_keys(pass1, pairing):
    """Lossless full-rank codec: the decoupled decode is softmax attention whose keys are the raw
    loop-t key joined with the token's rotary key turned at its position, and whose query is q
    joined with the rotary query turned at the current position (torch SDPA, complex-form
    rotation); the values are the raw loop-t values."""
    T, d, dr, L, base = 2, 32, 16, 19, 500.0
    g = _rng(90)
    Qk, Qv = _orthogonal(T * d, 91), _orthogonal(T * d, 92)
    xk, xv = g.standard_normal((T, L + 1, d)), g.standard_normal((T, L + 1, d))
    kr = g.standard_normal((L + 1, dr))  # one rotary key per token, every loop
    mu_k, mu_v = g.standard_normal(T * d), g.standard_normal(T * d)
    n_cached = L if pass1 else L + 1
    c_k = oracle.encode(xk[:, :n_cached], mu_k, Qk)
    c_v = oracle.encode(xv[:, :n_cached], mu_v, Qv)
    w_up_k = np.stack([Qk[t * d:(t + 1) * d] for t in range(T)])
    w_up_v = np.stack([Qv[t * d:(t + 1) * d] for t in range(T)])
    scale = 1 / math.sqrt(d + dr)
    pos0 = 7
    for t in range(T):
        q, qr = g.standard_normal(d), g.standard_normal(dr)
        out = oracle.decode_decoupled(t, c_k, c_v, kr[:n_cached], w_up_k, w_up_v, mu_k, mu_v, q, qr,
                                      xk[t, L] if pass1 else None, xv[t, L] if pass1 else None,
                                      kr[L] if pass1 else None, scale, base, pairing, pos0)
        J = np.stack([np.concatenate([xk[t, i], _rot_complex(kr[i], pos0 + i, base, pairing)])
                      for i in range(L + 1)])
        qj = np.concatenate([q, _rot_complex(qr, pos0 + L, base, pairing)])
        ref = _sdpa(qj, J, xv[t], scale)[0]
        np.testing.assert_allclose(out, ref, rtol=0, atol=1e-12)


def test_decoupled_without_rotary_parts_is_the_nope_decode():
    """Zero rotary keys and query leave only the content path: the plain LLA decode (pinned
    above), in both passes and at every loop."""
    T, d, dr, r_k, r_v, L = 4, 32, 8, 12, 20, 23
    g = _rng(93)
    cod = _random_codec(T, d, r_k, r_v, 94)
    c_k, c_v = g.standard_normal((L, r_k)), g.standard_normal((L, r_v))
    q = g.standard_normal(d)
    ck, cv = g.standard_normal(d), g.standard_normal(d)
    for t in range(T):
        for pass1 in (False, True):
            a = oracle.decode_decoupled(t, c_k, c_v, np.zeros((L, dr)), cod["w_up_k"], cod["w_up_v"],
                                        cod["mu_k"], cod["mu_v"], q, np.zeros(dr),
                                        ck if pass1 else None, cv if pass1 else None,
                                        np.zeros(dr) if pass1 else None, 0.2)
            b = oracle.decode(t, c_k, c_v, cod["w_up_k"], cod["w_up_v"], cod["mu_k"], cod["mu_v"], q,
                              ck if pass1 else None, cv if pass1 else None, 0.2)
            np.testing.assert_allclose(a, b, rtol=0, atol=1e-13)


@pytest.mark.parametrize("pass1", [False, True])
def test_decoupled_absorbed_form_and_relative_positions(pass1):
    """App. J absorbed form written independently: the content score moves W_up,t^K to the query
    (q~ = W_up,t^K^T q, plus q . mu^K_t) and the rotary score is rot(q^R, P - p) . k^R (RoFormer's
    relative form, complex multiplication); shifting every position leaves the output unchanged."""
    T, d, dr, r_k, r_v, L, base = 4, 64, 32, 24, 40, 30, 10000.0
    g = _rng(95)
    cod = _random_codec(T, d, r_k, r_v, 96)
    c_k, c_v = g.standard_normal((L, r_k)), g.standard_normal((L, r_v))
    kr = g.standard_normal((L, dr))
    q, qr = g.standard_normal(d), g.standard_normal(dr)
    ck = g.standard_normal(d) if pass1 else None
    cv = g.standard_normal(d) if pass1 else None
    ckr = g.standard_normal(dr) if pass1 else None
    scale = 1 / math.sqrt(d + dr)
    for t in range(T):
        out = oracle.decode_decoupled(t, c_k, c_v, kr, cod["w_up_k"], cod["w_up_v"], cod["mu_k"],
                                      cod["mu_v"], q, qr, ck, cv, ckr, scale, base, 0, 11)
        shifted = oracle.decode_decoupled(t, c_k, c_v, kr, cod["w_up_k"], cod["w_up_v"], cod["mu_k"],
                                          cod["mu_v"], q, qr, ck, cv, ckr, scale, base, 0, 5011)
        np.testing.assert_allclose(out, shifted, rtol=0, atol=1e-10)
        Wk, Wv = cod["w_up_k"][t], cod["w_up_v"][t]
        mk, mv = cod["mu_k"][t * d:(t + 1) * d], cod["mu_v"][t * d:(t + 1) * d]
        P = L if pass1 else L - 1  # the current token's index
        s = scale * (c_k @ (Wk.T @ q) + q @ mk +
                     np.array([_rot_complex(qr, P - i, base, 0) @ kr[i] for i in range(L)]))
        if pass1:
            s = np.append(s, scale * (q @ ck + qr @ ckr))
        p = np.exp(s - s.max())
        o = Wv @ (p[:L] @ c_v) + p[:L].sum() * mv
        if pass1:
            o = o + p[L] * cv
        np.testing.assert_allclose(out, o / p.sum(), rtol=0, atol=1e-12)
