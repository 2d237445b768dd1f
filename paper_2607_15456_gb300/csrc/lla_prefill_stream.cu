// lla_prefill_stream.cu -- lla_prefill_two_pass: the capacity decoder's two-pass prefill of a
// batch of prompts through all D layers, streamed layer by layer (App. A "Decoding and caching":
// pass 1 captures the teacher's pre-RoPE per-loop K/V, the codec turns them into latents, pass 2
// re-forwards attending over the reconstruction; App. J "Eviction and long-context prefill": long
// prompts fit only when each layer's captures are released as soon as that layer is encoded).
//
// Host orchestration only: every step is one of the library's kernels (lla_encode,
// lla_prefill_attn, lla_prefill_attn_rope), enqueued in order on the caller's stream.  The
// model itself (projections, MLP, norms) belongs to the caller and enters through two callbacks:
//   capture(l)   hands over layer l's stacked pass-1 keys and values [T][N][H][d];
//   query(l, t)  hands over the pass-2 queries of layer l at loop t and where their attention
//                output goes (the caller's model between attention calls runs inside it).
// Phase 1 walks the layers: capture(l), then Eq. encode of all N prompt tokens into layer l's
// paged cache.  Only one layer's capture is ever needed at a time: it may be reused or freed, in
// stream order, as soon as capture(l + 1) is called.  Phase 2 is the re-forward in the model's
// order, loop by loop and within a loop layer by layer: query(l, t), then causal attention over
// layer l's latents.  With rotary positions the rebuilt, rotated keys of one (layer, loop) live in
// the workspace and are overwritten by the next, so full-width reconstructions of only one layer
// exist at any time.
#include <cuda_runtime.h>

#include "lla_internal.h"

extern "C" lla_status lla_prefill_two_pass(
    const lla_geometry *g, int32_t D, const lla_codec *codecs, const lla_cache *caches,
    lla_dtype x_dtype, const int64_t *slot_mapping, int32_t N, const int32_t *cu_seqlens,
    int32_t B, int32_t max_len, lla_dtype io_dtype, const lla_rope *rope, lla_capture_fn capture,
    lla_query_fn query, void *user, void *workspace, size_t workspace_bytes, void *stream) {
    if (!g || D < 0 || N < 0 || B < 0 || max_len < 0) return LLA_ERR_INVALID_ARG;
    if (D > 0 && (!codecs || !caches || !capture || !query)) return LLA_ERR_INVALID_ARG;
    if (x_dtype != LLA_BF16 && x_dtype != LLA_F32) return LLA_ERR_INVALID_ARG;
    if (io_dtype != LLA_BF16 && io_dtype != LLA_F32) return LLA_ERR_INVALID_ARG;
    if (rope) {
        size_t need = 0;
        const lla_status st = lla_prefill_rope_workspace_size(g, B, max_len, &need);
        if (st != LLA_OK) return st;
        if (B > 0 && max_len > 0 && workspace_bytes < need) return LLA_ERR_WORKSPACE;
    }
    // phase 1: pass-1 captures into latents, one layer at a time
    for (int32_t l = 0; l < D; ++l) {
        const void *x_k = nullptr, *x_v = nullptr;
        lla_status st = capture(l, &x_k, &x_v, stream, user);
        if (st != LLA_OK) return st;
        st = lla_encode(g, &codecs[l], &caches[l], x_k, x_v, x_dtype, slot_mapping, N, stream);
        if (st != LLA_OK) return st;
    }
    // phase 2: the re-forward, loop-major as the looped model runs, attending over the latents
    for (int32_t t = 0; t < (D > 0 ? g->T : 0); ++t) {
        for (int32_t l = 0; l < D; ++l) {
            const void *q = nullptr;
            void *out = nullptr;
            lla_status st = query(l, t, &q, &out, stream, user);
            if (st != LLA_OK) return st;
            st = rope ? lla_prefill_attn_rope(g, &codecs[l], &caches[l], rope, cu_seqlens, B, max_len, t,
                                              q, io_dtype, out, workspace, workspace_bytes, stream)
                      : lla_prefill_attn(g, &codecs[l], &caches[l], cu_seqlens, B, max_len, t, q,
                                         io_dtype, out, stream);
            if (st != LLA_OK) return st;
        }
    }
    return LLA_OK;
}
