/*
 * lla.h -- C ABI of liblla: the hot path of Looped Latent Attention (LLA) on GB300 (sm_103a).
 *
 * A looped transformer runs its D-layer stack T times, and every loop writes its own key and
 * value per layer, head and token ("Teacher cache", Sec. 3).  LLA stores instead one latent
 * pair per (token, layer, head): c = (x - mu) W_down over the stacked loop vector
 * x = [x_1; ...; x_T] (Eq. encode), and rebuilds loop t on demand as
 * xhat_t = c W_up,t^T + mu_t (Eq. decode).  This library implements:
 *
 *   lla_encode           Eq. encode for newly completed tokens, written into a paged cache
 *   lla_decode_attn      one decode call (one layer, one loop) over the paged latent cache,
 *                        for a batch of sequences of different lengths (App. A, "Decoding and
 *                        caching": pass 1 and pass 2 of the cached reconstruction decoder)
 *   lla_decode_attn_rope the same with rotary positions applied after reconstruction (Sec. 3,
 *                        "RoPE and reconstruction"), keys rebuilt on the tensor cores
 *   lla_prefill_attn_rope  causal prefill with rotary positions after reconstruction
 *   lla_decode_attn_loops  the decode calls of all T loops in one pass over the latents
 *   lla_prefill_attn     causal pass-2 prefill attention over the latents of a prompt
 *   lla_prefill_two_pass the two-pass prefill of a batch of prompts through all layers, streamed
 *                        layer by layer (encode, then the loop-major re-forward's attention)
 *   lla_encode_2d, lla_decode_attn_2d
 *                        the LLA-2D variant: one latent per (token, layer) for every head
 *   lla_encode_rope_keys, lla_decode_attn_decoupled
 *                        per-head LLA with a decoupled rotary branch (one rotary key per token)
 *   lla_dense_*          the uncompressed loop-t KV decode in the same kernel style (the
 *                        "teacher" column of Table absorbed_latency, App. J), for comparison
 *
 * Attention reads the latents directly (App. J, "Absorbed attention"): the score is bilinear,
 * q . (W_up,t c) = (W_up,t^T q) . c, and the value path satisfies
 * sum_i a_i W_up,t c_i = W_up,t sum_i a_i c_i.  Reconstructed keys and values are never
 * written to memory.
 *
 * Conventions that hold for every call:
 *   - All pointers named "device" are CUDA device pointers of the current device.  The caller
 *     owns every buffer (weights, cache pool, tables, workspace, inputs, outputs).  No call
 *     allocates memory.
 *   - Work is enqueued on `stream` (a cudaStream_t passed as void*, NULL = legacy default
 *     stream) and is asynchronous.  Argument checks that need no device data are synchronous
 *     and return LLA_ERR_INVALID_ARG or LLA_ERR_UNSUPPORTED before anything is enqueued.
 *   - Checks that need device data (block ids, context lengths) and bounded waits inside the
 *     kernels never fault or hang: a failed check sets a sticky per-device error word, the
 *     affected outputs are undefined, and the host reads the word with lla_get_device_error.
 *   - No call throws; every call returns an lla_status.
 *
 * Cache layout (one layer).  Tokens are grouped in blocks of LLA_BLOCK_TOKENS = 64.  With es =
 * element size of `storage` (2 for bf16, 4 for fp32):
 *   pool      [num_blocks][H][K-plane | V-plane]          (one "head page" per block and head)
 *   K-plane   64 x r_k latents in granules of gk bytes, gk = 16 if (r_k*es) % 16 == 0 else 4:
 *             the byte offset of element (token i, column j) is
 *             ((j*es) / gk) * (64*gk) + i*gk + (j*es) % gk
 *   V-plane   64 x r_v latents, row-major: element (i, j) at byte offset (i*r_v + j)*es
 *   head page = 64*(r_k + r_v)*es bytes; block = H head pages.
 * Token p of sequence b lives in block block_table[b*max_blocks_per_seq + p/64], row p%64.
 * A slot is block_id*64 + row.  The pool must be 16-byte aligned.
 */
#ifndef LLA_H_
#define LLA_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define LLA_BLOCK_TOKENS 64
#define LLA_MAX_BATCH 1024

typedef enum {
    LLA_OK = 0,
    LLA_ERR_INVALID_ARG = 1,  /* a NULL pointer, a bad size or a bad alignment */
    LLA_ERR_UNSUPPORTED = 2,  /* a valid geometry this build has no kernel for */
    LLA_ERR_CUDA = 3,         /* a CUDA runtime call failed (launch, attribute, memcpy) */
    LLA_ERR_TIMEOUT = 4,      /* device error word: a bounded wait inside a kernel expired */
    LLA_ERR_DEVICE_CHECK = 5, /* device error word: a block id or length was out of range */
    LLA_ERR_WORKSPACE = 6     /* the workspace is smaller than the *_workspace_size answer */
} lla_status;

typedef enum { LLA_BF16 = 0, LLA_F32 = 1 } lla_dtype;

/* Bits of the device error word. */
#define LLA_DEVERR_BLOCK_ID 0x1u    /* a block id outside [0, num_blocks) */
#define LLA_DEVERR_CONTEXT 0x2u     /* a context length < 0, > max_ctx or > table capacity */
#define LLA_DEVERR_EMPTY_PASS2 0x4u /* pass 2 with an empty sequence (nothing to attend to) */
#define LLA_DEVERR_TIMEOUT 0x8u     /* a bounded wait expired */
#define LLA_DEVERR_SLOT 0x10u       /* an encode slot outside the pool */

/* Every wait of a kernel on its own pipeline (an mbarrier phase) gives up after this much global
 * time, sets LLA_DEVERR_TIMEOUT and lets the launch finish with undefined outputs. */
#define LLA_DEFAULT_WAIT_LIMIT_NS 2000000000ull

/* Shape of the codec and the cache (Sec. 3; App. A "Models"). */
typedef struct {
    int32_t T;          /* loops (recurrence steps), 1..16 */
    int32_t H;          /* attention heads, >= 1 */
    int32_t d;          /* head width d_head: a multiple of 8, 8..256 */
    int32_t r_k, r_v;   /* latent ranks, 2..512 (LLA-2D entry points: 2..2048 and at most T H d);
                           even for bf16 storage */
    int32_t block_size; /* tokens per cache block: must be LLA_BLOCK_TOKENS */
    lla_dtype storage;  /* dtype of the latents and of the codec weights */
    float scale;        /* softmax scale applied to q . k (e.g. 1/sqrt(d)) */
} lla_geometry;

/* Codec of one layer (Eqs. encode and decode), for all H heads; device pointers. */
typedef struct {
    const void *w_down_k; /* [H][T*d][r_k] storage dtype: W_down of the K axis (16-B aligned) */
    const void *w_down_v; /* [H][T*d][r_v] storage dtype (16-B aligned) */
    const void *w_up_k;   /* [H][T][d][r_k] storage dtype: W_up,t of the K axis (16-B aligned) */
    const void *w_up_v;   /* [H][T][d][r_v] storage dtype (16-B aligned) */
    const float *mu_k;    /* [H][T*d] fp32 calibration mean, or NULL for mu = 0 */
    const float *mu_v;    /* [H][T*d] fp32, or NULL */
} lla_codec;

/* Paged cache of one layer; device pointers. */
typedef struct {
    void *pool;                 /* [num_blocks][H][head page], layout above, 16-byte aligned */
    int64_t num_blocks;
    const int32_t *block_table; /* [B][max_blocks_per_seq] block ids (unused by lla_encode) */
    int32_t max_blocks_per_seq;
} lla_cache;

/* Static description of a status. */
const char *lla_status_string(lla_status status);

/* Library version, major*10000 + minor*100 + patch. */
int32_t lla_version(void);

/* Bytes of one cache block (H head pages) for geometry `g`.  Host only. */
lla_status lla_cache_block_bytes(const lla_geometry *g, size_t *bytes);

/*
 * Eq. encode (Sec. 3) for N newly completed tokens of one layer, written into the cache.
 *   x_k, x_v      device [T][N][H][d] in x_dtype, 16-byte aligned: the pre-RoPE loop-t keys /
 *                 values of each token (Sec. 3 "RoPE and reconstruction"; App. A "LLA codec
 *                 and conversion")
 *   slot_mapping  device [N] int64: destination slot of each token; a negative slot skips
 *                 the token.  A slot beyond the pool sets LLA_DEVERR_SLOT.
 * Latents are computed with fp32 accumulation and rounded to `storage` (round to nearest
 * even for bf16).  N may be 0.
 */
lla_status lla_encode(const lla_geometry *g, const lla_codec *codec, const lla_cache *cache,
                      const void *x_k, const void *x_v, lla_dtype x_dtype,
                      const int64_t *slot_mapping, int32_t N, void *stream);

/*
 * lla_encode for L layers in one call (one launch for a decode batch): the completed tokens of
 * a step are encoded in every layer at once, instead of one launch per layer.  The paper has no
 * counterpart; this is a scheduling convenience over Eq. encode (Sec. 3).
 *   codecs, caches  host arrays of L structs: layer l's codec and cache (same geometry)
 *   x_k, x_v        host arrays of L device pointers: layer l's [T][N][H][d] inputs in x_dtype,
 *                   16-byte aligned
 *   slot_mapping    device [N] int64, the same slots in every layer (one page table)
 * L <= 64 (LLA_ERR_UNSUPPORTED beyond); L = 0 or N = 0 is a valid no-op.  Results are those of
 * L lla_encode calls.
 */
lla_status lla_encode_layers(const lla_geometry *g, int32_t L, const lla_codec *codecs,
                             const lla_cache *caches, const void *const *x_k,
                             const void *const *x_v, lla_dtype x_dtype,
                             const int64_t *slot_mapping, int32_t N, void *stream);

/* Workspace bytes lla_decode_attn needs for a batch of B sequences on the current device. */
lla_status lla_decode_workspace_size(const lla_geometry *g, int32_t B, size_t *bytes);

/* Zero-fills a decode workspace (needed once before first use and after a device error). */
lla_status lla_decode_workspace_init(void *workspace, size_t workspace_bytes, void *stream);

/*
 * One decode call: layer given by `codec` and `cache`, loop `loop` (0-based), B sequences.
 * App. A "Decoding and caching" (two-pass cached reconstruction decoder) and App. J
 * "Absorbed attention".
 *   context_lens  device [B] int32: tokens of sequence b already in the cache (0..max_ctx)
 *   max_ctx       host upper bound of every context length (<= 64*max_blocks_per_seq)
 *   q             device [B][H][d] io_dtype: the loop-t query of the current token
 *   cur_k, cur_v  device [B][H][d] io_dtype, pass 1: the current token's exact loop-t key and
 *                 value, attended beside the cached tokens (its stacked vector is not complete
 *                 before loop T).  Both NULL selects pass 2: the current token was encoded
 *                 and is one of the context_lens cached tokens (then every length must be >= 1).
 *   out           device [B][H][d] io_dtype: softmax(scale q.Khat_t) Vhat_t, Khat/Vhat by Eq.
 *                 decode, without materialising them
 *   workspace     device, >= lla_decode_workspace_size bytes, zero-filled before first use;
 *                 every completed call leaves it zero-filled again.  Calls that share a
 *                 workspace must be ordered (one stream).
 * B may be 0.  B <= LLA_MAX_BATCH.
 */
lla_status lla_decode_attn(const lla_geometry *g, const lla_codec *codec, const lla_cache *cache,
                           const int32_t *context_lens, int32_t B, int32_t max_ctx, int32_t loop,
                           const void *q, const void *cur_k, const void *cur_v,
                           lla_dtype io_dtype, void *out, void *workspace,
                           size_t workspace_bytes, void *stream);

/* Workspace bytes lla_decode_attn_loops needs for a batch of B sequences on the current device. */
lla_status lla_decode_loops_workspace_size(const lla_geometry *g, int32_t B, size_t *bytes);

/*
 * The decode calls of all T loops of one layer in one pass over the latents: T queries of each
 * (sequence, head) against the shared latent (the latent of a token is one code for every loop,
 * Sec. 3 Eq. encode; App. J absorbed attention per loop).  For loops computed in parallel or
 * speculatively, or a verification of several loop outputs; the layer's latents are read once
 * instead of T times.  The result of loop t equals lla_decode_attn at loop t.
 *   q, cur_k, cur_v, out  device [T][B][H][d] io_dtype (loop-major): loop t's query, pass-1 exact
 *                         current key and value (both NULL: pass 2), and output
 *   workspace             >= lla_decode_loops_workspace_size bytes; needs no initialisation (the
 *                         call writes every workspace byte it reads) and holds no state between
 *                         calls, so calls on one stream may share it
 * Other arguments and the error behaviour are those of lla_decode_attn.  Storage LLA_BF16, d = 128,
 * 1 <= T <= 4 and (r_k, r_v) one of (96, 160), (128, 128), (72, 120), (192, 320);
 * LLA_ERR_UNSUPPORTED otherwise.  Three kernels on the stream (q~ absorption; the page stream on
 * the tensor cores, q~ and p as sums of three bf16 parts; the merge and output projection).
 */
lla_status lla_decode_attn_loops(const lla_geometry *g, const lla_codec *codec,
                                 const lla_cache *cache, const int32_t *context_lens, int32_t B,
                                 int32_t max_ctx, const void *q, const void *cur_k,
                                 const void *cur_v, lla_dtype io_dtype, void *out, void *workspace,
                                 size_t workspace_bytes, void *stream);

/* Rotary position embedding (RoFormer) applied after reconstruction (Sec. 3 "RoPE and
 * reconstruction"): pair j of a d-vector at position p is turned by the angle p * base^(-2j/d). */
typedef enum {
    LLA_ROPE_HALF = 0,     /* pair j = (x[j], x[j + d/2])  ("rotate half") */
    LLA_ROPE_ADJACENT = 1  /* pair j = (x[2j], x[2j + 1]) */
} lla_rope_pairing;

typedef struct {
    double base;              /* rotation base, > 1 (10000 in RoFormer) */
    lla_rope_pairing pairing;
} lla_rope;

/*
 * lla_decode_attn with rotary positions applied after reconstruction: the full-RoPE decoder
 * (Sec. 3 "RoPE and reconstruction"; App. A "Decoding and caching").  The latents hold pre-RoPE
 * keys.  Cached key i of sequence b (its index in the sequence) is rebuilt by Eq. decode and
 * rotated at position i; the query, and in pass 1 the current token's exact key, at the current
 * token's position: context_lens[b] in pass 1, context_lens[b] - 1 in pass 2.  Values are not
 * rotated.
 *   rope          host pointer to the rotation (read during the call)
 *   q, cur_k      pre-RoPE: the call rotates them
 * Every other argument, the workspace (lla_decode_workspace_size) and the error behaviour are
 * those of lla_decode_attn.  Keys are rebuilt on the tensor cores: storage must be LLA_BF16,
 * d = 128 and (r_k, r_v) one of (96, 160), (128, 128), (192, 320), (72, 120), else
 * LLA_ERR_UNSUPPORTED.  q, cur_k, cur_v and out must be 16-byte aligned.  For (96, 160),
 * (128, 128) and (72, 120) the latent value sum also runs on the tensor cores (p as three bf16
 * parts) and a second kernel on the stream merges the split runs; (192, 320) is one kernel.
 */
lla_status lla_decode_attn_rope(const lla_geometry *g, const lla_codec *codec,
                                const lla_cache *cache, const lla_rope *rope,
                                const int32_t *context_lens, int32_t B, int32_t max_ctx,
                                int32_t loop, const void *q, const void *cur_k, const void *cur_v,
                                lla_dtype io_dtype, void *out, void *workspace,
                                size_t workspace_bytes, void *stream);

/* Workspace bytes lla_prefill_attn_rope needs for B prompts of at most max_len tokens. */
lla_status lla_prefill_rope_workspace_size(const lla_geometry *g, int32_t B, int32_t max_len,
                                           size_t *bytes);

/*
 * lla_prefill_attn with rotary positions applied after reconstruction (Sec. 3 "RoPE and
 * reconstruction"; App. A two-pass prefill, whose pass 2 attends over the rebuilt, rotated
 * keys).  Prompt token i (query and key) sits at position i of its prompt.  Two launches on
 * `stream`: every key of the prompts is rebuilt by Eq. decode and rotated, and every query
 * rotated and scaled, into the workspace (bf16); then the causal tensor-core attention over them,
 * with values in latent space as in lla_prefill_attn.
 *   rope        host pointer to the rotation (read during the call)
 *   q           pre-RoPE, 16-byte aligned
 *   workspace   device, >= lla_prefill_rope_workspace_size bytes; overwritten (no zero fill
 *               needed); calls that share it must be ordered
 * Other arguments and the error behaviour are those of lla_prefill_attn; a prompt whose tokens
 * reach past row B * max_len of q sets LLA_DEVERR_CONTEXT.  Storage LLA_BF16, d = 128 and
 * (r_k, r_v) one of (96, 160), (192, 320), (128, 128); LLA_ERR_UNSUPPORTED otherwise.
 */
lla_status lla_prefill_attn_rope(const lla_geometry *g, const lla_codec *codec,
                                 const lla_cache *cache, const lla_rope *rope,
                                 const int32_t *cu_seqlens, int32_t B, int32_t max_len,
                                 int32_t loop, const void *q, lla_dtype io_dtype, void *out,
                                 void *workspace, size_t workspace_bytes, void *stream);

/*
 * LLA-2D (Sec. 3, "The LLA-2D variant (loop x head)"; App. J "Per-head LLA versus LLA-2D at
 * inference").  One latent pair per (token, layer) serves all H heads.  A token's stacked
 * vector runs over loops and heads, loop-major: x = [x_{1,1}; ...; x_{1,H}; x_{2,1}; ...;
 * x_{T,H}] in R^{T H d}; c = (x - mu) W_down; head h at loop t is rebuilt as
 * xhat_{t,h} = c W_up,t,h^T + mu_{t,h}.  rho_2D = 2 T H d / (r_k + r_v).
 *
 * The geometry is an lla_geometry whose r_k, r_v are the 2D ranks; the codec is an lla_codec with
 *   w_down_k, w_down_v   [T*H*d][r_k | r_v] storage dtype (rows ordered (t, h, e)), 16-B aligned
 *   w_up_k, w_up_v       [T][H][d][r_k | r_v] storage dtype, 16-B aligned
 *   mu_k, mu_v           [T*H*d] fp32 or NULL
 * and the cache an lla_cache with ONE page per block: pool [num_blocks][K-plane | V-plane], the
 * planes laid out as in the per-head cache (the K-plane granule-interleaved, the V-plane
 * row-major), lla_cache_2d_block_bytes bytes per block.
 */

/* Bytes of one LLA-2D cache block (one page of 64 tokens).  Host only. */
lla_status lla_cache_2d_block_bytes(const lla_geometry *g, size_t *bytes);

/*
 * LLA-2D encode of N newly completed tokens of one layer into the cache.
 *   x_k, x_v      device [T][N][H][d] in x_dtype, 16-byte aligned (pre-RoPE keys / values)
 *   slot_mapping  device [N] int64 (negative: skip the token; past the pool: LLA_DEVERR_SLOT)
 * fp32 accumulation, latents rounded to `storage`.  H * d <= 16384 (LLA_ERR_UNSUPPORTED beyond).
 */
lla_status lla_encode_2d(const lla_geometry *g, const lla_codec *codec, const lla_cache *cache,
                         const void *x_k, const void *x_v, lla_dtype x_dtype,
                         const int64_t *slot_mapping, int32_t N, void *stream);

/* Workspace bytes lla_decode_attn_2d needs for B sequences on the current device
 * (LLA_ERR_UNSUPPORTED for a shape with no kernel). */
lla_status lla_decode_2d_workspace_size(const lla_geometry *g, int32_t B, size_t *bytes);

/*
 * One LLA-2D decode call (one layer, loop `loop`, B sequences, all heads), App. A two-pass
 * decoder with App. J absorbed attention per head against the shared latent:
 *   q~_h = W_up,t,h^K^T q_h,  s_hi = scale (q~_h . c_k,i + q_h . mu^K_{t,h}),
 *   o_h = (W_up,t,h^V sum_i p_hi c_v,i + (sum_i p_hi) mu^V_{t,h} + p_h,cur v_cur,h) / sum p.
 *   q, cur_k, cur_v, out  device [B][H][d] io_dtype (cur_k = cur_v = NULL: pass 2)
 *   workspace             device, >= lla_decode_2d_workspace_size bytes; overwritten (no zero
 *                         fill needed); calls that share it must be ordered (one stream)
 * Other arguments and the error behaviour are those of lla_decode_attn.  Three launches on
 * `stream`.  Storage LLA_BF16, d = 128, H <= 16, (r_k, r_v) one of (96, 160), (128, 128),
 * (288, 480), (1152, 1920) (rho_2D = 5.33: its 384 KB pages stream through the attention kernel in
 * column chunks of the K-plane and row chunks of the V-plane); LLA_ERR_UNSUPPORTED otherwise.
 */
lla_status lla_decode_attn_2d(const lla_geometry *g, const lla_codec *codec, const lla_cache *cache,
                              const int32_t *context_lens, int32_t B, int32_t max_ctx,
                              int32_t loop, const void *q, const void *cur_k, const void *cur_v,
                              lla_dtype io_dtype, void *out, void *workspace,
                              size_t workspace_bytes, void *stream);

/*
 * Decoupled rotary branch (App. J "Absorbed attention": an MLA-style NoPE content path plus a
 * small explicit rotary branch shared across recurrence steps for each token, as in DeepSeek-V2).
 * Loop t's key of cached token i is its content key khat_t,i (Eq. decode, not rotated) joined
 * with one rotary key k^R_i of d_rope dims per token and layer, shared by every loop and head and
 * turned at the token's position; the query of head h is q_h joined with its rotary query q^R_h
 * turned at the current token's position:
 *   s_i = scale (q_h . khat_t,i + rot(q^R_h, P) . rot(k^R_i, p_i)),  o = softmax(s) Vhat_t.
 * The rotary keys live in rotary planes, one per cache block: [num_blocks][64 x d_rope] bf16 in
 * the granule layout of a K-plane (element (row i, column j) at (j/8)*1024 + i*16 + (j%8)*2),
 * lla_rope_plane_bytes bytes each, addressed through the cache's block table.
 */

/* Bytes of one rotary plane (64 tokens x d_rope, bf16); d_rope a multiple of 16 in 16..96. */
lla_status lla_rope_plane_bytes(int32_t d_rope, size_t *bytes);

/*
 * Writes the rotary keys of N tokens, each turned at its position, into the rotary planes.
 *   rope_pool     device [num_blocks][rotary plane], 16-byte aligned
 *   k_rope        device [N][d_rope] x_dtype: pre-rotation rotary keys
 *   positions     device [N] int32: the token's position in its sequence (< 0 sets
 *                 LLA_DEVERR_CONTEXT and skips the token)
 *   slot_mapping  device [N] int64: block * 64 + row (negative: skip; past the pool:
 *                 LLA_DEVERR_SLOT)
 */
lla_status lla_encode_rope_keys(int32_t d_rope, const lla_rope *rope, void *rope_pool, int64_t num_blocks,
                                const void *k_rope, lla_dtype x_dtype, const int32_t *positions,
                                const int64_t *slot_mapping, int32_t N, void *stream);

/* Workspace bytes lla_decode_attn_decoupled needs for B sequences on the current device
 * (LLA_ERR_UNSUPPORTED for a shape with no kernel). */
lla_status lla_decode_decoupled_workspace_size(const lla_geometry *g, int32_t d_rope, int32_t B,
                                               size_t *bytes);

/*
 * One decode call of per-head LLA (the codec and cache of lla_decode_attn) with the decoupled
 * rotary branch.  Cached token i of sequence b sits at position i; the current token at
 * context_lens[b] in pass 1 and context_lens[b] - 1 in pass 2.
 *   rope_pool    device rotary planes written by lla_encode_rope_keys (same block table)
 *   q_rope       device [B][H][d_rope] io_dtype: pre-rotation rotary queries
 *   cur_k_rope   device [B][d_rope] io_dtype, pass 1 (with cur_k, cur_v): the current token's
 *                pre-rotation rotary key; NULL in pass 2
 *   workspace    >= lla_decode_decoupled_workspace_size bytes, zero-filled once before the first
 *                call (lla_decode_workspace_init); as for lla_decode_attn, its split-KV counters
 *                return to zero after every call
 * Other arguments and the error behaviour are those of lla_decode_attn; one launch on `stream`
 * (the absorbed decode kernel with the block's rotary plane streamed beside each head page).
 * Storage LLA_BF16, d = 128, (r_k, r_v) = (96, 160), d_rope 32, 64 or 96; LLA_ERR_UNSUPPORTED
 * otherwise.
 */
lla_status lla_decode_attn_decoupled(const lla_geometry *g, const lla_codec *codec, const lla_cache *cache,
                                     const void *rope_pool, int32_t d_rope, const lla_rope *rope,
                                     const int32_t *context_lens, int32_t B, int32_t max_ctx, int32_t loop,
                                     const void *q, const void *q_rope, const void *cur_k, const void *cur_v,
                                     const void *cur_k_rope, lla_dtype io_dtype, void *out, void *workspace,
                                     size_t workspace_bytes, void *stream);

/*
 * lla_decode_attn for callers that cannot allocate device memory (for example a plug-in inside a
 * host application that owns all device memory and offers it no allocator, or a latency-critical
 * loop that cannot afford cudaMalloc's device-wide synchronisation).  Same arguments and result
 * as lla_decode_attn, without the workspace: the scratch lives in a 1 MiB device array of this
 * library, held on every GPU that loads it until the process exits.  The paper has no
 * counterpart; this is a deployment convenience.
 *   - Returns LLA_ERR_WORKSPACE (and enqueues nothing) when lla_decode_workspace_size for this
 *     geometry and B exceeds 1 MiB.
 *   - Every call shares the array and clears the arrival counters in the part it uses
 *     (cudaMemsetAsync on `stream`); the rest keeps the last call's bytes, which are always
 *     overwritten before they are read.  Calls that can overlap on the GPU race on the array:
 *     order them on one stream.
 *   - The first call on a device looks up the array's address with that device current and
 *     keeps it; make that first call before any stream capture.  After cudaDeviceReset the kept
 *     address is stale: do not call this entry point on that device again.
 *   - Allocates nothing (no cudaMalloc, no cudaFree).
 */
lla_status lla_decode_attn_noalloc(const lla_geometry *g, const lla_codec *codec,
                                   const lla_cache *cache, const int32_t *context_lens, int32_t B,
                                   int32_t max_ctx, int32_t loop, const void *q, const void *cur_k,
                                   const void *cur_v, lla_dtype io_dtype, void *out, void *stream);

/*
 * Causal pass-2 prefill attention at loop `loop` over latents already written by lla_encode
 * (App. A "Decoding and caching": the capacity decoder's two-pass prefill; App. J).
 *   cu_seqlens  device [B+1] int32 prefix sums of prompt lengths (cu_seqlens[0] = 0); the
 *               prompt of sequence b occupies cache positions 0..len_b-1 of block-table row b
 *   max_len     host upper bound of every prompt length (<= 64*max_blocks_per_seq)
 *   q, out      device [cu_seqlens[B]][H][d] io_dtype; query i of sequence b attends to
 *               cache positions 0..i of that sequence
 */
lla_status lla_prefill_attn(const lla_geometry *g, const lla_codec *codec, const lla_cache *cache,
                            const int32_t *cu_seqlens, int32_t B, int32_t max_len, int32_t loop,
                            const void *q, lla_dtype io_dtype, void *out, void *stream);

/*
 * Callbacks of lla_prefill_two_pass, called on the calling host thread in the order given there.
 * Each enqueues its own work on `stream` (the stream passed to lla_prefill_two_pass) and returns
 * LLA_OK, or another status to stop the prefill (lla_prefill_two_pass then returns it).
 *   lla_capture_fn  sets *x_k, *x_v to device [T][N][H][d] arrays (x_dtype, 16-byte aligned) with
 *                   layer `layer`'s pass-1 pre-RoPE keys and values of the N prompt tokens, stacked
 *                   over the loops as Eq. encode takes them.
 *   lla_query_fn    sets *q to device [N][H][d] pass-2 queries (io_dtype) of layer `layer` at loop
 *                   `loop` and *out to where their attention output goes (same shape).
 */
typedef lla_status (*lla_capture_fn)(int32_t layer, const void **x_k, const void **x_v, void *stream,
                                     void *user);
typedef lla_status (*lla_query_fn)(int32_t layer, int32_t loop, const void **q, void **out, void *stream,
                                   void *user);

/*
 * The capacity decoder's two-pass prefill of B prompts through all D layers, streamed layer by
 * layer (App. A "Decoding and caching"; App. J "Eviction and long-context prefill").  Host
 * orchestration of this library's kernels on `stream`, in this order:
 *   phase 1, for l = 0 .. D-1:  capture(l); lla_encode of the N tokens into caches[l]
 *   phase 2, for t = 0 .. T-1, for l = 0 .. D-1:  query(l, t); causal attention at loop t over
 *            caches[l] (lla_prefill_attn, or lla_prefill_attn_rope when rope is not NULL)
 * Only one layer's capture is needed at a time: the arrays capture(l) handed over may be reused
 * or freed, in stream order, once capture(l + 1) has been called (the last once the call has
 * returned).  With rope, the rebuilt keys of one (layer, loop) occupy the workspace and the next
 * overwrites them.
 *   codecs, caches  host arrays of D per-layer codecs and caches (their block tables give the
 *                   positions attention reads, slot_mapping the slots encode writes: the caller
 *                   keeps them consistent, token i of prompt b at row i of its pages)
 *   slot_mapping    device [N] int64, N = cu_seqlens[B] prompt tokens in prompt order
 *   cu_seqlens, B, max_len   as lla_prefill_attn
 *   rope            NULL (positions-free content path) or the rotation of lla_prefill_attn_rope
 *   workspace       with rope: >= lla_prefill_rope_workspace_size(g, B, max_len) bytes (device);
 *                   else unused (may be NULL)
 * Returns the first non-OK status of a callback or of a call it makes (the work enqueued before
 * it stays enqueued); the error behaviour of each step is that of its call.
 */
lla_status lla_prefill_two_pass(const lla_geometry *g, int32_t D, const lla_codec *codecs,
                                const lla_cache *caches, lla_dtype x_dtype,
                                const int64_t *slot_mapping, int32_t N, const int32_t *cu_seqlens,
                                int32_t B, int32_t max_len, lla_dtype io_dtype, const lla_rope *rope,
                                lla_capture_fn capture, lla_query_fn query, void *user,
                                void *workspace, size_t workspace_bytes, void *stream);

/*
 * Comparator: the uncompressed loop-indexed cache ("Teacher cache", Sec. 3) decoded by the same
 * kernel without the codec.  `g` must have r_k = r_v = d; `cache` then holds the plain loop-t
 * keys and values of one layer in the layout above (K-plane = keys, V-plane = values).
 */
lla_status lla_dense_store(const lla_geometry *g, const lla_cache *cache, const void *k,
                           const void *v, lla_dtype x_dtype, const int64_t *slot_mapping,
                           int32_t N, void *stream); /* k, v device [N][H][d] */
lla_status lla_dense_decode_attn(const lla_geometry *g, const lla_cache *cache,
                                 const int32_t *context_lens, int32_t B, int32_t max_ctx,
                                 const void *q, const void *cur_k, const void *cur_v,
                                 lla_dtype io_dtype, void *out, void *workspace,
                                 size_t workspace_bytes, void *stream);

/*
 * Reads the sticky device error word of the current device after synchronising `stream`.
 * *word receives the LLA_DEVERR_* bits; the status is LLA_OK when it is 0, LLA_ERR_TIMEOUT
 * when the timeout bit is set, LLA_ERR_DEVICE_CHECK otherwise.
 */
lla_status lla_get_device_error(void *stream, uint32_t *word);

/* Clears the device error word of the current device (enqueued on `stream`). */
lla_status lla_clear_device_error(void *stream);

/*
 * Limit of each pipeline wait (a host helper; the paper has no counterpart) in
 * the lla_decode_attn and lla_dense_decode_attn launches enqueued after this call, process-wide;
 * 0 restores LLA_DEFAULT_WAIT_LIMIT_NS.  A wait that runs out sets LLA_DEVERR_TIMEOUT and the
 * launch ends with undefined outputs: its producer issues no further copy and waits, with the
 * default limit, for the copies it has in flight, and every other wait of that CTA returns at
 * once.  The split-KV arrival counters still return to zero, so the workspace stays usable.
 * Meant for watchdogs and for tests of the timeout path; a limit below the time a page takes to
 * arrive makes every launch fail.  lla_get_wait_limit_ns returns the limit in force.
 */
lla_status lla_set_wait_limit_ns(uint64_t nanoseconds);
uint64_t lla_get_wait_limit_ns(void);

#ifdef __cplusplus
}
#endif

#endif /* LLA_H_ */
