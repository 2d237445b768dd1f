/*
 * lla_oracle.c -- plain, slow CPU float64 oracle for Looped Latent Attention (LLA).
 *
 * TEST INFRASTRUCTURE ONLY.  The tests, the smoke check and the CPU-baseline leg of the
 * benchmark are the only callers.  The CUDA library never calls, links or includes this
 * file, and this file knows nothing about the CUDA library (no paged layout, no absorbed
 * form, no tiling).
 *
 * What it computes, in the paper's notation (Sec. 3, "Looped Latent Attention"):
 *   stacked loop vector   x = [x_1; ...; x_T] in R^{T d}          ("Teacher cache")
 *   encode                c = (x - mu) W_down,  W_down in R^{Td x r}      (Eq. encode)
 *   per-loop decode       xhat_t = c W_up,t^T + mu_t,  W_up,t in R^{d x r} (Eq. decode)
 *   compression ratio     rho = 2 T d / (r_k + r_v)                       (Eq. ratio)
 * and softmax attention over the explicitly reconstructed keys and values:
 *   s_i = scale * q . Khat_t[i],  a = softmax(s),  o = sum_i a_i Vhat_t[i].
 *
 * Rotary positions (RoFormer) are applied after reconstruction when asked for (Sec. 3 "RoPE
 * and reconstruction"): the codec works on pre-RoPE keys, and each reconstructed key is rotated
 * at its token's position before the dot product with the rotated query.
 *
 * Decode follows the two-pass cached reconstruction decoder (App. A, "Decoding and
 * caching"): in pass 1 the current token's stacked vector is not complete yet, so at loop t
 * it attends with its own exact loop-t key and value; in pass 2 the current token has been
 * encoded and is read back through Eq. decode like every other cached token.
 *
 * Everything is double precision with plain loops in the order the equations are written.
 * Inputs that the GPU side stores in bf16 are passed here already widened (exactly) to
 * double.  No fused or reordered arithmetic beyond what the equations state; OpenMP only
 * runs independent (sequence, head, loop) problems side by side.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* Eq. ratio: rho = 2 T H d / ((r_k + r_v) H) = 2 T d / (r_k + r_v). */
double lla_oracle_ratio(int T, int d_head, int r_k, int r_v)
{
    return 2.0 * (double)T * (double)d_head / (double)(r_k + r_v);
}

/* "Teacher cache": 2 T H d scalars per token per layer (K and V of every loop and head). */
double lla_oracle_teacher_cache_bytes_per_token(int T, int H, int d_head, int D, int elem_bytes)
{
    return 2.0 * T * H * (double)d_head * D * elem_bytes;
}

/* Eq. ratio, numerator of the compressed side: (r_k + r_v) H scalars per token per layer. */
double lla_oracle_latent_cache_bytes_per_token(int H, int D, int r_k, int r_v, int elem_bytes)
{
    return (double)(r_k + r_v) * H * D * elem_bytes;
}

/*
 * Eq. encode for N tokens of one (layer, head, axis).
 *   x      [T][N][d]   x[t][n] is the loop-t vector of token n (loops counted from 0)
 *   mu     [T*d]       calibration mean of the stacked vector, or NULL for mu = 0
 *   w_down [T*d][r]
 *   c      [N][r]      output latents
 */
void lla_oracle_encode(int T, int d, int r, int64_t N, const double *x, const double *mu,
                       const double *w_down, double *c)
{
    const int Td = T * d;
    double *xs = (double *)malloc(sizeof(double) * (size_t)Td);
    for (int64_t n = 0; n < N; ++n) {
        /* stack the loop vectors: x = [x_1; ...; x_T] */
        for (int t = 0; t < T; ++t)
            for (int e = 0; e < d; ++e)
                xs[t * d + e] = x[((int64_t)t * N + n) * d + e];
        /* centre: x - mu */
        if (mu)
            for (int k = 0; k < Td; ++k)
                xs[k] = xs[k] - mu[k];
        /* project: c = (x - mu) W_down */
        for (int j = 0; j < r; ++j) {
            double acc = 0.0;
            for (int k = 0; k < Td; ++k)
                acc += xs[k] * w_down[(int64_t)k * r + j];
            c[n * r + j] = acc;
        }
    }
    free(xs);
}

/*
 * Eq. decode for N latents at one loop t.
 *   c      [N][r]
 *   w_up_t [d][r]   W_up,t
 *   mu_t   [d]      loop-t slice of mu, or NULL
 *   xhat   [N][d]   xhat_t = c W_up,t^T + mu_t
 */
void lla_oracle_reconstruct(int d, int r, int64_t N, const double *c, const double *w_up_t,
                            const double *mu_t, double *xhat)
{
    for (int64_t n = 0; n < N; ++n) {
        for (int e = 0; e < d; ++e) {
            double acc = 0.0;
            for (int j = 0; j < r; ++j)
                acc += c[n * r + j] * w_up_t[(int64_t)e * r + j];
            xhat[n * d + e] = acc + (mu_t ? mu_t[e] : 0.0);
        }
    }
}

/*
 * Plain softmax attention of one query over L >= 1 keys and values.
 *   s_i = scale * q . K[i];  a_i = exp(s_i - max s) / sum_j exp(s_j - max s);  o = sum_i a_i V[i]
 * Returns 0, or -1 when L < 1.
 */
int lla_oracle_attention(int d, int64_t L, const double *q, const double *K, const double *V,
                         double scale, double *o)
{
    if (L < 1)
        return -1;
    double *s = (double *)malloc(sizeof(double) * (size_t)L);
    double m = -INFINITY;
    for (int64_t i = 0; i < L; ++i) {
        double dot = 0.0;
        for (int e = 0; e < d; ++e)
            dot += q[e] * K[i * d + e];
        s[i] = scale * dot;
        if (s[i] > m)
            m = s[i];
    }
    double z = 0.0;
    for (int64_t i = 0; i < L; ++i) {
        s[i] = exp(s[i] - m);
        z += s[i];
    }
    for (int64_t i = 0; i < L; ++i)
        s[i] = s[i] / z; /* a_i */
    for (int e = 0; e < d; ++e) {
        double acc = 0.0;
        for (int64_t i = 0; i < L; ++i)
            acc += s[i] * V[i * d + e];
        o[e] = acc;
    }
    free(s);
    return 0;
}

/*
 * The keys and values one loop-t query attends to: Khat_t and Vhat_t of the L cached tokens
 * by Eq. decode, in rows 0 .. L-1 of K and V [L + 1][d]; in pass 1 (cur_k, cur_v not NULL) the
 * current token's exact loop-t key and value as row L.
 */
static void loop_keys_values(int d, int r_k, int r_v, int t, int64_t L, const double *c_k,
                             const double *c_v, const double *w_up_k, const double *w_up_v,
                             const double *mu_k, const double *mu_v, const double *cur_k,
                             const double *cur_v, double *K, double *V)
{
    lla_oracle_reconstruct(d, r_k, L, c_k, w_up_k + (int64_t)t * d * r_k,
                           mu_k ? mu_k + (int64_t)t * d : NULL, K);
    lla_oracle_reconstruct(d, r_v, L, c_v, w_up_v + (int64_t)t * d * r_v,
                           mu_v ? mu_v + (int64_t)t * d : NULL, V);
    if (cur_k) {
        memcpy(K + L * d, cur_k, sizeof(double) * (size_t)d);
        memcpy(V + L * d, cur_v, sizeof(double) * (size_t)d);
    }
}

/*
 * One decode call for one (sequence, head) at loop t (0-based) of one layer.
 *   c_k [L][r_k], c_v [L][r_v]       latents of the L cached tokens
 *   w_up_k [T][d][r_k], w_up_v [T][d][r_v]
 *   mu_k, mu_v [T*d] or NULL
 *   q [d]                            loop-t query of the current token
 *   cur_k, cur_v [d] or NULL         pass 1: the current token's exact loop-t key/value
 *                                    pass 2 (NULL): the current token is one of the L cached
 *   out [d]
 * Returns 0, or -1 on bad arguments (pass 2 needs L >= 1).
 */
int lla_oracle_decode(int T, int d, int r_k, int r_v, int t, int64_t L, const double *c_k,
                      const double *c_v, const double *w_up_k, const double *w_up_v,
                      const double *mu_k, const double *mu_v, const double *q,
                      const double *cur_k, const double *cur_v, double scale, double *out)
{
    if (t < 0 || t >= T || L < 0)
        return -1;
    if ((cur_k == NULL) != (cur_v == NULL))
        return -1;
    const int pass1 = cur_k != NULL;
    if (!pass1 && L < 1)
        return -1;
    const int64_t n = L + (pass1 ? 1 : 0);
    double *K = (double *)malloc(sizeof(double) * (size_t)(n * d));
    double *V = (double *)malloc(sizeof(double) * (size_t)(n * d));
    /* Eq. decode, loop t, for every cached token; pass 1: the current token joins with its
       exact loop-t key and value */
    loop_keys_values(d, r_k, r_v, t, L, c_k, c_v, w_up_k, w_up_v, mu_k, mu_v, cur_k, cur_v, K, V);
    int rc = lla_oracle_attention(d, n, q, K, V, scale, out);
    free(K);
    free(V);
    return rc;
}

/*
 * Causal prefill at loop t for one (sequence, head): the N prompt tokens are all cached as
 * latents (pass 2 of the two-pass prefill, App. A and App. J "Eviction and long-context
 * prefill"); query i attends to keys j <= i through Eq. decode.
 *   q [N][d], out [N][d]
 */
int lla_oracle_prefill(int T, int d, int r_k, int r_v, int t, int64_t N, const double *c_k,
                       const double *c_v, const double *w_up_k, const double *w_up_v,
                       const double *mu_k, const double *mu_v, const double *q, double scale,
                       double *out)
{
    if (t < 0 || t >= T || N < 0)
        return -1;
    double *K = (double *)malloc(sizeof(double) * (size_t)(N * d + 1));
    double *V = (double *)malloc(sizeof(double) * (size_t)(N * d + 1));
    loop_keys_values(d, r_k, r_v, t, N, c_k, c_v, w_up_k, w_up_v, mu_k, mu_v, NULL, NULL, K, V);
    int rc = 0;
    for (int64_t i = 0; i < N && rc == 0; ++i)
        rc = lla_oracle_attention(d, i + 1, q + i * d, K, V, scale, out + i * d);
    free(K);
    free(V);
    return rc;
}

/*
 * Rotary position embedding (RoFormer; Sec. 3 "RoPE and reconstruction") of one d-vector at
 * integer position pos.  Pair j (j = 0 .. d/2 - 1) of x is turned by the angle
 * pos * theta_j with theta_j = base^(-2j/d):
 *   pairing 0 ("rotate half"):     pair j = (x[j], x[j + d/2])
 *   pairing 1 (adjacent elements): pair j = (x[2j], x[2j + 1])
 *   y[a] = x[a] cos(pos theta_j) - x[b] sin(pos theta_j)
 *   y[b] = x[a] sin(pos theta_j) + x[b] cos(pos theta_j)
 * y must not alias x.
 */
void lla_oracle_rope(int d, int pairing, double base, int64_t pos, const double *x, double *y)
{
    const int h = d / 2;
    for (int j = 0; j < h; ++j) {
        const int a = pairing ? 2 * j : j;
        const int b = pairing ? 2 * j + 1 : j + h;
        const double theta = pow(base, -2.0 * j / d);
        const double ang = (double)pos * theta;
        const double c = cos(ang), s = sin(ang);
        y[a] = x[a] * c - x[b] * s;
        y[b] = x[a] * s + x[b] * c;
    }
}

/*
 * lla_oracle_decode with rotary positions applied after reconstruction (Sec. 3 "RoPE and
 * reconstruction": the latent holds the pre-RoPE key; a token keeps its position at every
 * loop).  Cached token i sits at position pos0 + i; in pass 1 the current token's exact key
 * sits at pos0 + L.  The query belongs to the current token, the last key of the attended set:
 * position pos0 + L in pass 1 and pos0 + L - 1 in pass 2.  Values carry no rotation.
 */
int lla_oracle_decode_rope(int T, int d, int r_k, int r_v, int t, int64_t L, const double *c_k,
                           const double *c_v, const double *w_up_k, const double *w_up_v,
                           const double *mu_k, const double *mu_v, const double *q,
                           const double *cur_k, const double *cur_v, double scale, int pairing,
                           double base, int64_t pos0, double *out)
{
    if (t < 0 || t >= T || L < 0 || d < 2 || d % 2 != 0 || base <= 0.0)
        return -1;
    if ((cur_k == NULL) != (cur_v == NULL))
        return -1;
    const int pass1 = cur_k != NULL;
    if (!pass1 && L < 1)
        return -1;
    const int64_t n = L + (pass1 ? 1 : 0);
    double *K = (double *)malloc(sizeof(double) * (size_t)(n * d));
    double *Kr = (double *)malloc(sizeof(double) * (size_t)(n * d));
    double *V = (double *)malloc(sizeof(double) * (size_t)(n * d));
    double *qr = (double *)malloc(sizeof(double) * (size_t)d);
    loop_keys_values(d, r_k, r_v, t, L, c_k, c_v, w_up_k, w_up_v, mu_k, mu_v, cur_k, cur_v, K, V);
    /* RoPE after reconstruction: every key at its own position, the query at the last one */
    for (int64_t i = 0; i < n; ++i)
        lla_oracle_rope(d, pairing, base, pos0 + i, K + i * d, Kr + i * d);
    lla_oracle_rope(d, pairing, base, pos0 + n - 1, q, qr);
    int rc = lla_oracle_attention(d, n, qr, Kr, V, scale, out);
    free(K);
    free(Kr);
    free(V);
    free(qr);
    return rc;
}

/*
 * lla_oracle_prefill with rotary positions after reconstruction: prompt token i (query and
 * key) at position pos0 + i.
 */
int lla_oracle_prefill_rope(int T, int d, int r_k, int r_v, int t, int64_t N, const double *c_k,
                            const double *c_v, const double *w_up_k, const double *w_up_v,
                            const double *mu_k, const double *mu_v, const double *q,
                            double scale, int pairing, double base, int64_t pos0, double *out)
{
    if (t < 0 || t >= T || N < 0 || d < 2 || d % 2 != 0 || base <= 0.0)
        return -1;
    double *K = (double *)malloc(sizeof(double) * (size_t)(N * d + 1));
    double *Kr = (double *)malloc(sizeof(double) * (size_t)(N * d + 1));
    double *V = (double *)malloc(sizeof(double) * (size_t)(N * d + 1));
    double *qr = (double *)malloc(sizeof(double) * (size_t)d);
    loop_keys_values(d, r_k, r_v, t, N, c_k, c_v, w_up_k, w_up_v, mu_k, mu_v, NULL, NULL, K, V);
    for (int64_t i = 0; i < N; ++i)
        lla_oracle_rope(d, pairing, base, pos0 + i, K + i * d, Kr + i * d);
    int rc = 0;
    for (int64_t i = 0; i < N && rc == 0; ++i) {
        lla_oracle_rope(d, pairing, base, pos0 + i, q + i * d, qr);
        rc = lla_oracle_attention(d, i + 1, qr, Kr, V, scale, out + i * d);
    }
    free(K);
    free(Kr);
    free(V);
    free(qr);
    return rc;
}

/*
 * Decoupled rotary branch (App. J "Absorbed attention": an MLA-style NoPE content path plus a
 * small explicit rotary branch shared across recurrence steps for each token; DeepSeek-V2).
 * Loop t's key of cached token i is the pair (khat_t,i, k^R_i): the content key khat_t,i of
 * Eq. decode (no rotation) and a rotary key k^R_i of d_rope dims, one per token for every loop,
 * rotated at the token's position.  The query is the pair (q, q^R), q^R rotated at the current
 * token's position.  The score adds the two dot products under one scale:
 *   s_i = scale (q . khat_t,i + rot(q^R, P) . rot(k^R_i, p_i))
 * and the value is Eq. decode's vhat_t,i.  Cached token i sits at position pos0 + i; the
 * current token (the query) at pos0 + L in pass 1, where it attends with its exact loop-t key
 * and value and its own rotary key, and at pos0 + L - 1 in pass 2.
 *   k_rope [L][d_rope]      pre-rotation rotary keys of the cached tokens
 *   q_rope [d_rope]         pre-rotation rotary query
 *   cur_k_rope [d_rope]     pass 1: the current token's rotary key (NULL in pass 2)
 * Other arguments as lla_oracle_decode.
 */
int lla_oracle_decode_decoupled(int T, int d, int d_rope, int r_k, int r_v, int t, int64_t L,
                                const double *c_k, const double *c_v, const double *k_rope,
                                const double *w_up_k, const double *w_up_v, const double *mu_k,
                                const double *mu_v, const double *q, const double *q_rope,
                                const double *cur_k, const double *cur_v,
                                const double *cur_k_rope, double scale, int pairing, double base,
                                int64_t pos0, double *out)
{
    if (t < 0 || t >= T || L < 0 || d_rope < 2 || d_rope % 2 != 0 || base <= 0.0)
        return -1;
    if ((cur_k == NULL) != (cur_v == NULL) || (cur_k == NULL) != (cur_k_rope == NULL))
        return -1;
    const int pass1 = cur_k != NULL;
    if (!pass1 && L < 1)
        return -1;
    const int64_t n = L + (pass1 ? 1 : 0);
    const int w = d + d_rope; /* width of a joined key [khat; rot(k^R)] */
    double *K = (double *)malloc(sizeof(double) * (size_t)(n * d));
    double *V = (double *)malloc(sizeof(double) * (size_t)(n * d));
    double *J = (double *)malloc(sizeof(double) * (size_t)(n * w));
    double *qj = (double *)malloc(sizeof(double) * (size_t)w);
    /* content keys and values of loop t (Eq. decode; pass 1 appends the exact current pair) */
    loop_keys_values(d, r_k, r_v, t, L, c_k, c_v, w_up_k, w_up_v, mu_k, mu_v, cur_k, cur_v, K, V);
    /* joined keys: the content key, then the rotary key turned at the token's position */
    for (int64_t i = 0; i < n; ++i) {
        memcpy(J + i * w, K + i * d, sizeof(double) * (size_t)d);
        const double *kr = i < L ? k_rope + i * d_rope : cur_k_rope;
        lla_oracle_rope(d_rope, pairing, base, pos0 + i, kr, J + i * w + d);
    }
    /* joined query: content query, then the rotary query at the current token's position */
    memcpy(qj, q, sizeof(double) * (size_t)d);
    lla_oracle_rope(d_rope, pairing, base, pos0 + n - 1, q_rope, qj + d);
    /* softmax over the joined dot products, values of width d */
    double *sj = (double *)malloc(sizeof(double) * (size_t)n);
    double m = -INFINITY;
    for (int64_t i = 0; i < n; ++i) {
        double dot = 0.0;
        for (int e = 0; e < w; ++e)
            dot += qj[e] * J[i * w + e];
        sj[i] = dot * scale;
        if (sj[i] > m)
            m = sj[i];
    }
    double z = 0.0;
    for (int64_t i = 0; i < n; ++i) {
        sj[i] = exp(sj[i] - m);
        z += sj[i];
    }
    for (int e = 0; e < d; ++e) {
        double acc = 0.0;
        for (int64_t i = 0; i < n; ++i)
            acc += sj[i] * V[i * d + e];
        out[e] = acc / z;
    }
    free(sj);
    free(K);
    free(V);
    free(J);
    free(qj);
    return 0;
}

/*
 * LLA-2D (Sec. 3, "The LLA-2D variant (loop x head)"): one latent per (token, layer) that
 * covers every head.  The stacked vector runs over loops and heads, loop-major,
 *   x = [x_{1,1}; ...; x_{1,H}; x_{2,1}; ...; x_{T,H}] in R^{T H d},
 * is encoded as c = (x - mu) W_down with W_down in R^{THd x r}, and head h at loop t is rebuilt
 * as xhat_{t,h} = c W_up,t,h^T + mu_{t,h} with W_up,t,h in R^{d x r}, mu_{t,h} the (t, h) slice
 * of mu.  The cache then holds (r_k + r_v) scalars per token and layer (Sec. 3 and App. J "Per-
 * head LLA versus LLA-2D at inference"): rho_2D = 2 T H d / (r_k + r_v).
 */
double lla_oracle_ratio_2d(int T, int H, int d_head, int r_k, int r_v)
{
    return 2.0 * (double)T * (double)H * (double)d_head / (double)(r_k + r_v);
}

/*
 * LLA-2D encode of N tokens of one (layer, axis).
 *   x      [T][N][H][d]  x[t][n][h] is the loop-t vector of head h of token n
 *   mu     [T*H*d]       mean of the stacked vector, or NULL
 *   w_down [T*H*d][r]
 *   c      [N][r]
 */
void lla_oracle_encode_2d(int T, int H, int d, int r, int64_t N, const double *x,
                          const double *mu, const double *w_down, double *c)
{
    const int S = T * H * d;
    double *xs = (double *)malloc(sizeof(double) * (size_t)S);
    for (int64_t n = 0; n < N; ++n) {
        /* stack over loops, then heads: entry (t, h, e) at (t H + h) d + e */
        for (int t = 0; t < T; ++t)
            for (int h = 0; h < H; ++h)
                for (int e = 0; e < d; ++e)
                    xs[((int64_t)t * H + h) * d + e] = x[(((int64_t)t * N + n) * H + h) * d + e];
        if (mu) /* centre: x - mu */
            for (int k = 0; k < S; ++k)
                xs[k] -= mu[k];
        for (int j = 0; j < r; ++j) {
            double acc = 0.0;
            for (int k = 0; k < S; ++k)
                acc += xs[k] * w_down[(int64_t)k * r + j];
            c[n * r + j] = acc;
        }
    }
    free(xs);
}

/*
 * One LLA-2D decode call for one (sequence, head h) at loop t: every cached token's key and
 * value of head h are rebuilt from the shared latent with the (t, h) up-projection, then plain
 * softmax attention as in lla_oracle_decode (pass 1 appends the current token's exact loop-t
 * key and value of head h).
 *   c_k [L][r_k], c_v [L][r_v]            the sequence's latents (shared by all heads)
 *   w_up_k [T][H][d][r_k], w_up_v [T][H][d][r_v]
 *   mu_k, mu_v [T*H*d] or NULL
 *   q, cur_k, cur_v, out [d]              head h's vectors (cur_* NULL: pass 2)
 */
int lla_oracle_decode_2d_head(int T, int H, int d, int r_k, int r_v, int t, int h, int64_t L,
                              const double *c_k, const double *c_v, const double *w_up_k,
                              const double *w_up_v, const double *mu_k, const double *mu_v,
                              const double *q, const double *cur_k, const double *cur_v,
                              double scale, double *out)
{
    if (t < 0 || t >= T || h < 0 || h >= H || L < 0)
        return -1;
    if ((cur_k == NULL) != (cur_v == NULL))
        return -1;
    const int pass1 = cur_k != NULL;
    if (!pass1 && L < 1)
        return -1;
    const int64_t th = (int64_t)t * H + h; /* slice (t, h) of the up-projections and of mu */
    const int64_t n = L + (pass1 ? 1 : 0);
    double *K = (double *)malloc(sizeof(double) * (size_t)(n * d));
    double *V = (double *)malloc(sizeof(double) * (size_t)(n * d));
    lla_oracle_reconstruct(d, r_k, L, c_k, w_up_k + th * d * r_k, mu_k ? mu_k + th * d : NULL, K);
    lla_oracle_reconstruct(d, r_v, L, c_v, w_up_v + th * d * r_v, mu_v ? mu_v + th * d : NULL, V);
    if (pass1) /* the current token's exact loop-t key and value of head h */
        for (int e = 0; e < d; ++e) {
            K[L * d + e] = cur_k[e];
            V[L * d + e] = cur_v[e];
        }
    int rc = lla_oracle_attention(d, n, q, K, V, scale, out);
    free(K);
    free(V);
    return rc;
}

/* One (sequence, head) problem for lla_oracle_decode_2d_batch. */
typedef struct {
    int32_t t, h;
    int64_t L;
    const double *c_k, *c_v, *w_up_k, *w_up_v, *mu_k, *mu_v;
    const double *q, *cur_k, *cur_v;
    double *out;
} lla_oracle_decode_2d_item;

int lla_oracle_decode_2d_batch(int T, int H, int d, int r_k, int r_v, double scale,
                               int64_t n_items, const lla_oracle_decode_2d_item *items,
                               int n_threads)
{
    int err = 0;
#ifdef _OPENMP
    if (n_threads <= 0)
        n_threads = omp_get_max_threads();
#pragma omp parallel for schedule(dynamic, 1) num_threads(n_threads)
#endif
    for (int64_t i = 0; i < n_items; ++i) {
        const lla_oracle_decode_2d_item *it = &items[i];
        int rc = lla_oracle_decode_2d_head(T, H, d, r_k, r_v, it->t, it->h, it->L, it->c_k,
                                           it->c_v, it->w_up_k, it->w_up_v, it->mu_k, it->mu_v,
                                           it->q, it->cur_k, it->cur_v, scale, it->out);
        if (rc != 0) {
#ifdef _OPENMP
#pragma omp critical
#endif
            err = rc;
        }
    }
    return err;
}

/* One independent decode problem for lla_oracle_decode_batch. */
typedef struct {
    int32_t t;
    int32_t rope; /* 0: no rotary positions; 1: RoPE, rotate-half pairs; 2: RoPE, adjacent pairs */
    int64_t L;
    double rope_base;
    const double *c_k, *c_v, *w_up_k, *w_up_v, *mu_k, *mu_v;
    const double *q, *cur_k, *cur_v;
    double *out;
} lla_oracle_decode_item;

/* Runs n_items independent decode problems, n_threads at a time (<= 0: the OpenMP default).
 * Returns 0, or the first nonzero item status. */
int lla_oracle_decode_batch(int T, int d, int r_k, int r_v, double scale, int64_t n_items,
                            const lla_oracle_decode_item *items, int n_threads)
{
    int err = 0;
#ifdef _OPENMP
    if (n_threads <= 0)
        n_threads = omp_get_max_threads();
#pragma omp parallel for schedule(dynamic, 1) num_threads(n_threads)
#endif
    for (int64_t i = 0; i < n_items; ++i) {
        const lla_oracle_decode_item *it = &items[i];
        int rc = it->rope
                     ? lla_oracle_decode_rope(T, d, r_k, r_v, it->t, it->L, it->c_k, it->c_v,
                                              it->w_up_k, it->w_up_v, it->mu_k, it->mu_v, it->q,
                                              it->cur_k, it->cur_v, scale, it->rope - 1,
                                              it->rope_base, 0, it->out)
                     : lla_oracle_decode(T, d, r_k, r_v, it->t, it->L, it->c_k, it->c_v,
                                         it->w_up_k, it->w_up_v, it->mu_k, it->mu_v, it->q,
                                         it->cur_k, it->cur_v, scale, it->out);
        if (rc != 0) {
#ifdef _OPENMP
#pragma omp critical
#endif
            err = rc;
        }
    }
    return err;
}

/* One (head, axis) encode problem for lla_oracle_encode_batch. */
typedef struct {
    int32_t r;
    int32_t pad_;
    const double *x, *mu, *w_down;
    double *c;
} lla_oracle_encode_item;

int lla_oracle_encode_batch(int T, int d, int64_t N, int64_t n_items,
                            const lla_oracle_encode_item *items, int n_threads)
{
#ifdef _OPENMP
    if (n_threads <= 0)
        n_threads = omp_get_max_threads();
#pragma omp parallel for schedule(dynamic, 1) num_threads(n_threads)
#endif
    for (int64_t i = 0; i < n_items; ++i)
        lla_oracle_encode(T, d, items[i].r, N, items[i].x, items[i].mu, items[i].w_down,
                          items[i].c);
    return 0;
}

/* Threads an unrestricted batch call would use. */
int lla_oracle_max_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}
