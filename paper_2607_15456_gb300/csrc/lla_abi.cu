// lla_abi.cu -- the extern "C" entry points of liblla: argument checks, the per-device error
// word, and dispatch to the kernel files.  Checks that need no device data run before anything
// is enqueued; nothing here allocates device memory.
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include <algorithm>
#include <atomic>

#include "lla_internal.h"

namespace lla {

namespace {

__device__ unsigned g_error_word;  // sticky LLA_DEVERR_* bits of this device

constexpr int kMaxDevices = 64;

bool aligned(const void *p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

int elem_size(lla_dtype t) { return t == LLA_BF16 ? 2 : 4; }

bool valid_dtype(lla_dtype t) { return t == LLA_BF16 || t == LLA_F32; }

// max_rank: 512 for the per-head cache; the LLA-2D entry points take latents as wide as the H
// per-head latents together (kMaxRank2D, and at most T H d, the width of the stacked vector)
constexpr int kMaxRank = 512, kMaxRank2D = 2048;
lla_status check_geometry(const lla_geometry *g, int max_rank = kMaxRank) {
    if (!g) return LLA_ERR_INVALID_ARG;
    if (g->T < 1 || g->T > 16 || g->H < 1 || g->H > 4096) return LLA_ERR_INVALID_ARG;
    if (g->d < 8 || g->d > 256 || (g->d % 8) != 0) return LLA_ERR_INVALID_ARG;
    if (g->r_k < 2 || g->r_v < 2 || g->r_k > max_rank || g->r_v > max_rank) return LLA_ERR_INVALID_ARG;
    if (max_rank > kMaxRank && (static_cast<int64_t>(g->r_k) > static_cast<int64_t>(g->T) * g->H * g->d ||
                                static_cast<int64_t>(g->r_v) > static_cast<int64_t>(g->T) * g->H * g->d))
        return LLA_ERR_INVALID_ARG;
    if ((g->r_k % 2) != 0 || (g->r_v % 2) != 0) return LLA_ERR_INVALID_ARG;
    if (g->block_size != LLA_BLOCK_TOKENS) return LLA_ERR_UNSUPPORTED;
    if (!valid_dtype(g->storage)) return LLA_ERR_INVALID_ARG;
    if (!isfinite(g->scale)) return LLA_ERR_INVALID_ARG;
    return LLA_OK;
}

lla_status check_cache(const lla_cache *c, bool need_table) {
    if (!c || !c->pool || c->num_blocks < 1) return LLA_ERR_INVALID_ARG;
    if (!aligned(c->pool, 16)) return LLA_ERR_INVALID_ARG;
    if (need_table && (!c->block_table || c->max_blocks_per_seq < 1)) return LLA_ERR_INVALID_ARG;
    return LLA_OK;
}

}  // namespace

// Per-device caches below are filled on first use; host threads may race to fill one, so each
// entry is atomic (both racers store the same value).
unsigned *device_error_word(lla_status *st) {
    static std::atomic<unsigned *> addr[kMaxDevices];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
        *st = LLA_ERR_CUDA;
        return nullptr;
    }
    unsigned *a = addr[dev].load(std::memory_order_acquire);
    if (!a) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_error_word) != cudaSuccess) {
            *st = LLA_ERR_CUDA;
            return nullptr;
        }
        a = static_cast<unsigned *>(p);
        addr[dev].store(a, std::memory_order_release);
    }
    *st = LLA_OK;
    return a;
}

int num_sms() {
    static std::atomic<int> cached[kMaxDevices];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return 0;
    int n = cached[dev].load(std::memory_order_relaxed);
    if (!n) {
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
        cached[dev].store(n, std::memory_order_relaxed);
    }
    return n;
}

namespace {
std::atomic<uint64_t> g_wait_limit_ns{0};  // 0: LLA_DEFAULT_WAIT_LIMIT_NS
}  // namespace

uint64_t pipeline_wait_limit_ns() { return g_wait_limit_ns.load(std::memory_order_relaxed); }

}  // namespace lla

using namespace lla;

extern "C" {

const char *lla_status_string(lla_status s) {
    switch (s) {
        case LLA_OK: return "ok";
        case LLA_ERR_INVALID_ARG: return "invalid argument";
        case LLA_ERR_UNSUPPORTED: return "unsupported geometry";
        case LLA_ERR_CUDA: return "CUDA runtime error";
        case LLA_ERR_TIMEOUT: return "device wait timed out";
        case LLA_ERR_DEVICE_CHECK: return "device-side check failed";
        case LLA_ERR_WORKSPACE: return "workspace too small";
    }
    return "unknown status";
}

int32_t lla_version(void) { return 100; /* 0.1.0 */ }

lla_status lla_cache_block_bytes(const lla_geometry *g, size_t *bytes) {
    lla_status st = check_geometry(g);
    if (st != LLA_OK) return st;
    if (!bytes) return LLA_ERR_INVALID_ARG;
    *bytes = head_page_bytes(g->r_k, g->r_v, elem_size(g->storage)) * g->H;
    return LLA_OK;
}

lla_status lla_encode(const lla_geometry *g, const lla_codec *codec, const lla_cache *cache,
                      const void *x_k, const void *x_v, lla_dtype x_dtype,
                      const int64_t *slot_mapping, int32_t N, void *stream) {
    lla_status st = check_geometry(g);
    if (st != LLA_OK) return st;
    if (!codec || !codec->w_down_k || !codec->w_down_v) return LLA_ERR_INVALID_ARG;
    if ((st = check_cache(cache, false)) != LLA_OK) return st;
    if (!valid_dtype(x_dtype) || N < 0) return LLA_ERR_INVALID_ARG;
    if (N > 0 && (!x_k || !x_v || !slot_mapping)) return LLA_ERR_INVALID_ARG;
    if (!aligned(codec->w_down_k, 16) || !aligned(codec->w_down_v, 16)) return LLA_ERR_INVALID_ARG;
    if (N > 0 && (!aligned(x_k, 16) || !aligned(x_v, 16))) return LLA_ERR_INVALID_ARG;
    if (N == 0) return LLA_OK;
    EncodeArgs a = {};
    a.T = g->T; a.H = g->H; a.d = g->d; a.r_k = g->r_k; a.r_v = g->r_v;
    a.storage_bf16 = g->storage == LLA_BF16;
    a.x_bf16 = x_dtype == LLA_BF16;
    a.w_down_k = codec->w_down_k; a.w_down_v = codec->w_down_v;
    a.mu_k = codec->mu_k; a.mu_v = codec->mu_v;
    a.x_k = x_k; a.x_v = x_v;
    a.pool = cache->pool; a.num_blocks = cache->num_blocks;
    a.slot_mapping = slot_mapping; a.N = N;
    a.dense = 0;
    return launch_encode(a, static_cast<cudaStream_t>(stream));
}

lla_status lla_encode_layers(const lla_geometry *g, int32_t L, const lla_codec *codecs,
                             const lla_cache *caches, const void *const *x_k,
                             const void *const *x_v, lla_dtype x_dtype,
                             const int64_t *slot_mapping, int32_t N, void *stream) {
    lla_status st = check_geometry(g);
    if (st != LLA_OK) return st;
    if (L < 0 || !valid_dtype(x_dtype) || N < 0) return LLA_ERR_INVALID_ARG;
    if (L == 0 || N == 0) return LLA_OK;
    if (L > kMaxEncodeLayers) return LLA_ERR_UNSUPPORTED;
    if (!codecs || !caches || !x_k || !x_v || !slot_mapping) return LLA_ERR_INVALID_ARG;
    EncodeArgs a[kMaxEncodeLayers];
    for (int l = 0; l < L; ++l) {
        const lla_codec *codec = &codecs[l];
        if (!codec->w_down_k || !codec->w_down_v) return LLA_ERR_INVALID_ARG;
        if ((st = check_cache(&caches[l], false)) != LLA_OK) return st;
        if (!x_k[l] || !x_v[l]) return LLA_ERR_INVALID_ARG;
        if (!aligned(codec->w_down_k, 16) || !aligned(codec->w_down_v, 16)) return LLA_ERR_INVALID_ARG;
        if (!aligned(x_k[l], 16) || !aligned(x_v[l], 16)) return LLA_ERR_INVALID_ARG;
        a[l] = EncodeArgs{};
        a[l].T = g->T; a[l].H = g->H; a[l].d = g->d; a[l].r_k = g->r_k; a[l].r_v = g->r_v;
        a[l].storage_bf16 = g->storage == LLA_BF16;
        a[l].x_bf16 = x_dtype == LLA_BF16;
        a[l].w_down_k = codec->w_down_k; a[l].w_down_v = codec->w_down_v;
        a[l].mu_k = codec->mu_k; a[l].mu_v = codec->mu_v;
        a[l].x_k = x_k[l]; a[l].x_v = x_v[l];
        a[l].pool = caches[l].pool; a[l].num_blocks = caches[l].num_blocks;
        a[l].slot_mapping = slot_mapping; a[l].N = N;
        a[l].dense = 0;
    }
    return launch_encode_layers(a, L, static_cast<cudaStream_t>(stream));
}

lla_status lla_decode_workspace_size(const lla_geometry *g, int32_t B, size_t *bytes) {
    lla_status st = check_geometry(g);
    if (st != LLA_OK) return st;
    if (!bytes || B < 0 || B > LLA_MAX_BATCH) return LLA_ERR_INVALID_ARG;
    const int sms = num_sms();
    if (sms <= 0) return LLA_ERR_CUDA;
    // one CTA per SM; the full-RoPE decode on the tensor cores keeps a slot per (unit, CTA) run
    size_t n = decode_workspace_bytes(g->r_v, B, g->H, sms);
    if (decode_rope_tc_supported(elem_size(g->storage), g->d, g->r_k, g->r_v))
        n = std::max(n, decode_rope_tc_workspace_bytes(g->r_v, B, g->H, sms));
    *bytes = n;
    return LLA_OK;
}

lla_status lla_decode_workspace_init(void *workspace, size_t workspace_bytes, void *stream) {
    if (!workspace || workspace_bytes == 0) return LLA_ERR_INVALID_ARG;
    if (cudaMemsetAsync(workspace, 0, workspace_bytes, static_cast<cudaStream_t>(stream)) !=
        cudaSuccess)
        return LLA_ERR_CUDA;
    return LLA_OK;
}

namespace {

lla_status decode_common(const lla_geometry *g, const lla_codec *codec, const lla_cache *cache,
                         const int32_t *context_lens, int32_t B, int32_t max_ctx, int32_t loop,
                         const void *q, const void *cur_k, const void *cur_v, lla_dtype io_dtype,
                         void *out, void *workspace, size_t workspace_bytes, void *stream,
                         bool absorbed, const lla_rope *rope = nullptr, bool loops = false) {
    lla_status st = check_geometry(g);
    if (st != LLA_OK) return st;
    if ((st = check_cache(cache, true)) != LLA_OK) return st;
    const int es = elem_size(g->storage);
    if (absorbed) {
        if (!codec || !codec->w_up_k || !codec->w_up_v) return LLA_ERR_INVALID_ARG;
        if (!aligned(codec->w_up_k, 16) || !aligned(codec->w_up_v, 16)) return LLA_ERR_INVALID_ARG;
        if (loop < 0 || loop >= g->T) return LLA_ERR_INVALID_ARG;
    } else if (g->r_k != g->d || g->r_v != g->d) {
        return LLA_ERR_INVALID_ARG;
    }
    if (B < 0 || B > LLA_MAX_BATCH || !valid_dtype(io_dtype)) return LLA_ERR_INVALID_ARG;
    if (max_ctx < 0 || static_cast<int64_t>(max_ctx) >
                           static_cast<int64_t>(cache->max_blocks_per_seq) * LLA_BLOCK_TOKENS)
        return LLA_ERR_INVALID_ARG;
    // a sequence's pages of all heads are counted in 32 bits inside the kernel
    if (static_cast<int64_t>(g->H) * ((static_cast<int64_t>(max_ctx) + LLA_BLOCK_TOKENS - 1) / LLA_BLOCK_TOKENS) >=
        (int64_t(1) << 31))
        return LLA_ERR_UNSUPPORTED;
    if ((cur_k == nullptr) != (cur_v == nullptr)) return LLA_ERR_INVALID_ARG;
    if (B > 0 && (!context_lens || !q || !out)) return LLA_ERR_INVALID_ARG;
    if (rope) {
        if (!(rope->base > 1.0) || !(rope->base < 1e300)) return LLA_ERR_INVALID_ARG;
        if (rope->pairing != LLA_ROPE_HALF && rope->pairing != LLA_ROPE_ADJACENT)
            return LLA_ERR_INVALID_ARG;
        if ((q && !aligned(q, 16)) || (cur_k && !aligned(cur_k, 16)) ||
            (cur_v && !aligned(cur_v, 16)) || (out && !aligned(out, 16)))
            return LLA_ERR_INVALID_ARG;
        if ((st = decode_rope_fits(g->r_k, g->r_v, es, g->d, B)) != LLA_OK) return st;
    } else if (loops) {
        if ((st = decode_loops_fits(g->r_k, g->r_v, es, g->d, g->T, B)) != LLA_OK) return st;
    } else if ((st = decode_fits(g->r_k, g->r_v, es, g->d)) != LLA_OK) {
        return st;
    }
    if (B == 0) return LLA_OK;
    if (!workspace) return LLA_ERR_INVALID_ARG;
    DecodeArgs a = {};
    a.T = g->T; a.H = g->H; a.d = g->d; a.r_k = g->r_k; a.r_v = g->r_v;
    a.loop = absorbed ? loop : 0;
    a.absorbed = absorbed ? 1 : 0;
    a.storage_bf16 = g->storage == LLA_BF16;
    a.io_bf16 = io_dtype == LLA_BF16;
    a.scale = g->scale;
    if (absorbed) {
        a.w_up_k = codec->w_up_k; a.w_up_v = codec->w_up_v;
        a.mu_k = codec->mu_k; a.mu_v = codec->mu_v;
    }
    a.pool = cache->pool; a.num_blocks = cache->num_blocks;
    a.block_table = cache->block_table; a.max_blocks = cache->max_blocks_per_seq;
    a.context_lens = context_lens; a.B = B; a.max_ctx = max_ctx;
    a.q = q; a.cur_k = cur_k; a.cur_v = cur_v; a.out = out;
    a.workspace = workspace; a.workspace_bytes = workspace_bytes;
    if (rope)
        return launch_decode_rope(a, rope->base, rope->pairing == LLA_ROPE_ADJACENT ? 1 : 0,
                                  static_cast<cudaStream_t>(stream));
    if (loops) return launch_decode_loops(a, static_cast<cudaStream_t>(stream));
    return launch_decode(a, static_cast<cudaStream_t>(stream));
}

}  // namespace

lla_status lla_decode_attn(const lla_geometry *g, const lla_codec *codec, const lla_cache *cache,
                           const int32_t *context_lens, int32_t B, int32_t max_ctx, int32_t loop,
                           const void *q, const void *cur_k, const void *cur_v,
                           lla_dtype io_dtype, void *out, void *workspace,
                           size_t workspace_bytes, void *stream) {
    return decode_common(g, codec, cache, context_lens, B, max_ctx, loop, q, cur_k, cur_v,
                         io_dtype, out, workspace, workspace_bytes, stream, true);
}

lla_status lla_decode_attn_rope(const lla_geometry *g, const lla_codec *codec,
                                const lla_cache *cache, const lla_rope *rope,
                                const int32_t *context_lens, int32_t B, int32_t max_ctx,
                                int32_t loop, const void *q, const void *cur_k, const void *cur_v,
                                lla_dtype io_dtype, void *out, void *workspace,
                                size_t workspace_bytes, void *stream) {
    if (!rope) return LLA_ERR_INVALID_ARG;
    return decode_common(g, codec, cache, context_lens, B, max_ctx, loop, q, cur_k, cur_v,
                         io_dtype, out, workspace, workspace_bytes, stream, true, rope);
}

lla_status lla_decode_loops_workspace_size(const lla_geometry *g, int32_t B, size_t *bytes) {
    lla_status st = check_geometry(g);
    if (st != LLA_OK) return st;
    if (!bytes || B < 0 || B > LLA_MAX_BATCH) return LLA_ERR_INVALID_ARG;
    const int grid = num_sms();
    if (grid <= 0) return LLA_ERR_CUDA;
    *bytes = decode_loops_workspace_bytes(g->r_k, g->r_v, B, g->H, grid);
    return LLA_OK;
}

lla_status lla_decode_attn_loops(const lla_geometry *g, const lla_codec *codec,
                                 const lla_cache *cache, const int32_t *context_lens, int32_t B,
                                 int32_t max_ctx, const void *q, const void *cur_k,
                                 const void *cur_v, lla_dtype io_dtype, void *out, void *workspace,
                                 size_t workspace_bytes, void *stream) {
    return decode_common(g, codec, cache, context_lens, B, max_ctx, 0, q, cur_k, cur_v, io_dtype,
                         out, workspace, workspace_bytes, stream, true, nullptr, true);
}

lla_status lla_cache_2d_block_bytes(const lla_geometry *g, size_t *bytes) {
    lla_status st = check_geometry(g, kMaxRank2D);
    if (st != LLA_OK) return st;
    if (!bytes) return LLA_ERR_INVALID_ARG;
    *bytes = head_page_bytes(g->r_k, g->r_v, elem_size(g->storage));  // one page per block
    return LLA_OK;
}

lla_status lla_encode_2d(const lla_geometry *g, const lla_codec *codec, const lla_cache *cache,
                         const void *x_k, const void *x_v, lla_dtype x_dtype,
                         const int64_t *slot_mapping, int32_t N, void *stream) {
    lla_status st = check_geometry(g, kMaxRank2D);
    if (st != LLA_OK) return st;
    if (!codec || !codec->w_down_k || !codec->w_down_v) return LLA_ERR_INVALID_ARG;
    if ((st = check_cache(cache, false)) != LLA_OK) return st;
    if (!valid_dtype(x_dtype) || N < 0) return LLA_ERR_INVALID_ARG;
    if (N > 0 && (!x_k || !x_v || !slot_mapping)) return LLA_ERR_INVALID_ARG;
    if (!aligned(codec->w_down_k, 16) || !aligned(codec->w_down_v, 16)) return LLA_ERR_INVALID_ARG;
    if (N > 0 && (!aligned(x_k, 16) || !aligned(x_v, 16))) return LLA_ERR_INVALID_ARG;
    if (static_cast<int64_t>(g->H) * g->d > 16384) return LLA_ERR_UNSUPPORTED;
    if (N == 0) return LLA_OK;
    // The 2D stack [x_{1,1}; ...; x_{1,H}; ...; x_{T,H}] of a token is the per-head stack of one
    // head of width H d: x [T][N][H][d] read as [T][N][1][H d], W_down [T H d][r], mu [T H d],
    // and one page per block.
    EncodeArgs a = {};
    a.T = g->T; a.H = 1; a.d = g->H * g->d; a.r_k = g->r_k; a.r_v = g->r_v;
    a.storage_bf16 = g->storage == LLA_BF16;
    a.x_bf16 = x_dtype == LLA_BF16;
    a.w_down_k = codec->w_down_k; a.w_down_v = codec->w_down_v;
    a.mu_k = codec->mu_k; a.mu_v = codec->mu_v;
    a.x_k = x_k; a.x_v = x_v;
    a.pool = cache->pool; a.num_blocks = cache->num_blocks;
    a.slot_mapping = slot_mapping; a.N = N;
    a.dense = 0;
    return launch_encode(a, static_cast<cudaStream_t>(stream));
}

lla_status lla_decode_2d_workspace_size(const lla_geometry *g, int32_t B, size_t *bytes) {
    lla_status st = check_geometry(g, kMaxRank2D);
    if (st != LLA_OK) return st;
    if (!bytes || B < 0 || B > LLA_MAX_BATCH) return LLA_ERR_INVALID_ARG;
    if (!decode_2d_supported(elem_size(g->storage), g->d, g->H, g->r_k, g->r_v))
        return LLA_ERR_UNSUPPORTED;
    const size_t n = decode_2d_workspace_bytes(g->r_k, g->r_v, B);
    if (n == 0) return LLA_ERR_CUDA;
    *bytes = n;
    return LLA_OK;
}

lla_status lla_decode_attn_2d(const lla_geometry *g, const lla_codec *codec, const lla_cache *cache,
                              const int32_t *context_lens, int32_t B, int32_t max_ctx,
                              int32_t loop, const void *q, const void *cur_k, const void *cur_v,
                              lla_dtype io_dtype, void *out, void *workspace,
                              size_t workspace_bytes, void *stream) {
    lla_status st = check_geometry(g, kMaxRank2D);
    if (st != LLA_OK) return st;
    if ((st = check_cache(cache, true)) != LLA_OK) return st;
    if (!codec || !codec->w_up_k || !codec->w_up_v) return LLA_ERR_INVALID_ARG;
    if (!aligned(codec->w_up_k, 16) || !aligned(codec->w_up_v, 16)) return LLA_ERR_INVALID_ARG;
    if (loop < 0 || loop >= g->T) return LLA_ERR_INVALID_ARG;
    if (B < 0 || B > LLA_MAX_BATCH || !valid_dtype(io_dtype)) return LLA_ERR_INVALID_ARG;
    if (max_ctx < 0 || static_cast<int64_t>(max_ctx) >
                           static_cast<int64_t>(cache->max_blocks_per_seq) * LLA_BLOCK_TOKENS)
        return LLA_ERR_INVALID_ARG;
    // the batch's pages are counted in 32 bits inside the kernels
    if (static_cast<int64_t>(B) * ((static_cast<int64_t>(max_ctx) + LLA_BLOCK_TOKENS - 1) / LLA_BLOCK_TOKENS) >=
        (int64_t(1) << 31))
        return LLA_ERR_UNSUPPORTED;
    if ((cur_k == nullptr) != (cur_v == nullptr)) return LLA_ERR_INVALID_ARG;
    if (B > 0 && (!context_lens || !q || !out)) return LLA_ERR_INVALID_ARG;
    if (!decode_2d_supported(elem_size(g->storage), g->d, g->H, g->r_k, g->r_v))
        return LLA_ERR_UNSUPPORTED;
    if (B == 0) return LLA_OK;
    if (!workspace) return LLA_ERR_INVALID_ARG;
    DecodeArgs a = {};
    a.T = g->T; a.H = g->H; a.d = g->d; a.r_k = g->r_k; a.r_v = g->r_v;
    a.loop = loop;
    a.absorbed = 1;
    a.storage_bf16 = 1;
    a.io_bf16 = io_dtype == LLA_BF16;
    a.scale = g->scale;
    a.w_up_k = codec->w_up_k; a.w_up_v = codec->w_up_v;
    a.mu_k = codec->mu_k; a.mu_v = codec->mu_v;
    a.pool = cache->pool; a.num_blocks = cache->num_blocks;
    a.block_table = cache->block_table; a.max_blocks = cache->max_blocks_per_seq;
    a.context_lens = context_lens; a.B = B; a.max_ctx = max_ctx;
    a.q = q; a.cur_k = cur_k; a.cur_v = cur_v; a.out = out;
    a.workspace = workspace; a.workspace_bytes = workspace_bytes;
    return launch_decode_2d(a, static_cast<cudaStream_t>(stream));
}

lla_status lla_rope_plane_bytes(int32_t d_rope, size_t *bytes) {
    if (!bytes || d_rope < 16 || d_rope > 96 || d_rope % 16 != 0) return LLA_ERR_INVALID_ARG;
    *bytes = static_cast<size_t>(LLA_BLOCK_TOKENS) * d_rope * 2;
    return LLA_OK;
}

namespace {
bool valid_rope(const lla_rope *rope) {
    return rope && rope->base > 1.0 && rope->base < 1e300 &&
           (rope->pairing == LLA_ROPE_HALF || rope->pairing == LLA_ROPE_ADJACENT);
}
}  // namespace

lla_status lla_encode_rope_keys(int32_t d_rope, const lla_rope *rope, void *rope_pool, int64_t num_blocks,
                                const void *k_rope, lla_dtype x_dtype, const int32_t *positions,
                                const int64_t *slot_mapping, int32_t N, void *stream) {
    if (d_rope < 16 || d_rope > 96 || d_rope % 16 != 0 || !valid_rope(rope)) return LLA_ERR_INVALID_ARG;
    if (!rope_pool || num_blocks < 1 || !aligned(rope_pool, 16) || !valid_dtype(x_dtype) || N < 0)
        return LLA_ERR_INVALID_ARG;
    if (N > 0 && (!k_rope || !positions || !slot_mapping)) return LLA_ERR_INVALID_ARG;
    return launch_rope_key_store(d_rope, rope->base, rope->pairing == LLA_ROPE_ADJACENT ? 1 : 0, rope_pool,
                                 num_blocks, k_rope, x_dtype == LLA_BF16, positions, slot_mapping, N,
                                 static_cast<cudaStream_t>(stream));
}

lla_status lla_decode_decoupled_workspace_size(const lla_geometry *g, int32_t d_rope, int32_t B,
                                               size_t *bytes) {
    lla_status st = check_geometry(g);
    if (st != LLA_OK) return st;
    if (!bytes || B < 0 || B > LLA_MAX_BATCH) return LLA_ERR_INVALID_ARG;
    if (!decode_decoupled_supported(elem_size(g->storage), g->d, g->H, g->r_k, g->r_v, d_rope))
        return LLA_ERR_UNSUPPORTED;
    const size_t n = decode_decoupled_workspace_bytes(g->r_k, g->r_v, d_rope, B, g->H);
    if (n == 0) return LLA_ERR_CUDA;
    *bytes = n;
    return LLA_OK;
}

lla_status lla_decode_attn_decoupled(const lla_geometry *g, const lla_codec *codec, const lla_cache *cache,
                                     const void *rope_pool, int32_t d_rope, const lla_rope *rope,
                                     const int32_t *context_lens, int32_t B, int32_t max_ctx, int32_t loop,
                                     const void *q, const void *q_rope, const void *cur_k, const void *cur_v,
                                     const void *cur_k_rope, lla_dtype io_dtype, void *out, void *workspace,
                                     size_t workspace_bytes, void *stream) {
    lla_status st = check_geometry(g);
    if (st != LLA_OK) return st;
    if ((st = check_cache(cache, true)) != LLA_OK) return st;
    if (!codec || !codec->w_up_k || !codec->w_up_v) return LLA_ERR_INVALID_ARG;
    if (!aligned(codec->w_up_k, 16) || !aligned(codec->w_up_v, 16)) return LLA_ERR_INVALID_ARG;
    if (loop < 0 || loop >= g->T) return LLA_ERR_INVALID_ARG;
    if (!valid_rope(rope) || !rope_pool || !aligned(rope_pool, 16)) return LLA_ERR_INVALID_ARG;
    if (B < 0 || B > LLA_MAX_BATCH || !valid_dtype(io_dtype)) return LLA_ERR_INVALID_ARG;
    if (max_ctx < 0 || static_cast<int64_t>(max_ctx) >
                           static_cast<int64_t>(cache->max_blocks_per_seq) * LLA_BLOCK_TOKENS)
        return LLA_ERR_INVALID_ARG;
    if ((cur_k == nullptr) != (cur_v == nullptr) || (cur_k == nullptr) != (cur_k_rope == nullptr))
        return LLA_ERR_INVALID_ARG;
    if (B > 0 && (!context_lens || !q || !q_rope || !out)) return LLA_ERR_INVALID_ARG;
    if (!decode_decoupled_supported(elem_size(g->storage), g->d, g->H, g->r_k, g->r_v, d_rope))
        return LLA_ERR_UNSUPPORTED;
    // the pages of every (sequence, head) are counted in 32 bits inside the kernels
    if (static_cast<int64_t>(B) * g->H *
            ((static_cast<int64_t>(max_ctx) + LLA_BLOCK_TOKENS - 1) / LLA_BLOCK_TOKENS) >= (int64_t(1) << 31))
        return LLA_ERR_UNSUPPORTED;
    if (B == 0) return LLA_OK;
    if (!workspace) return LLA_ERR_INVALID_ARG;
    DecodeArgs a = {};
    a.T = g->T; a.H = g->H; a.d = g->d; a.r_k = g->r_k; a.r_v = g->r_v;
    a.loop = loop;
    a.absorbed = 1;
    a.storage_bf16 = 1;
    a.io_bf16 = io_dtype == LLA_BF16;
    a.scale = g->scale;
    a.w_up_k = codec->w_up_k; a.w_up_v = codec->w_up_v;
    a.mu_k = codec->mu_k; a.mu_v = codec->mu_v;
    a.pool = cache->pool; a.num_blocks = cache->num_blocks;
    a.block_table = cache->block_table; a.max_blocks = cache->max_blocks_per_seq;
    a.context_lens = context_lens; a.B = B; a.max_ctx = max_ctx;
    a.q = q; a.cur_k = cur_k; a.cur_v = cur_v; a.out = out;
    a.workspace = workspace; a.workspace_bytes = workspace_bytes;
    return launch_decode_decoupled(a, rope_pool, d_rope, rope->base, rope->pairing == LLA_ROPE_ADJACENT ? 1 : 0,
                                   q_rope, cur_k_rope, static_cast<cudaStream_t>(stream));
}

lla_status lla_dense_decode_attn(const lla_geometry *g, const lla_cache *cache,
                                 const int32_t *context_lens, int32_t B, int32_t max_ctx,
                                 const void *q, const void *cur_k, const void *cur_v,
                                 lla_dtype io_dtype, void *out, void *workspace,
                                 size_t workspace_bytes, void *stream) {
    return decode_common(g, nullptr, cache, context_lens, B, max_ctx, 0, q, cur_k, cur_v,
                         io_dtype, out, workspace, workspace_bytes, stream, false);
}

lla_status lla_dense_store(const lla_geometry *g, const lla_cache *cache, const void *k,
                           const void *v, lla_dtype x_dtype, const int64_t *slot_mapping,
                           int32_t N, void *stream) {
    lla_status st = check_geometry(g);
    if (st != LLA_OK) return st;
    if (g->r_k != g->d || g->r_v != g->d) return LLA_ERR_INVALID_ARG;
    if ((st = check_cache(cache, false)) != LLA_OK) return st;
    if (!valid_dtype(x_dtype) || N < 0) return LLA_ERR_INVALID_ARG;
    if (N > 0 && (!k || !v || !slot_mapping)) return LLA_ERR_INVALID_ARG;
    if (N == 0) return LLA_OK;
    EncodeArgs a = {};
    a.T = 1; a.H = g->H; a.d = g->d; a.r_k = g->d; a.r_v = g->d;
    a.storage_bf16 = g->storage == LLA_BF16;
    a.x_bf16 = x_dtype == LLA_BF16;
    a.x_k = k; a.x_v = v;
    a.pool = cache->pool; a.num_blocks = cache->num_blocks;
    a.slot_mapping = slot_mapping; a.N = N;
    a.dense = 1;
    return launch_encode(a, static_cast<cudaStream_t>(stream));
}

lla_status lla_prefill_attn(const lla_geometry *g, const lla_codec *codec, const lla_cache *cache,
                            const int32_t *cu_seqlens, int32_t B, int32_t max_len, int32_t loop,
                            const void *q, lla_dtype io_dtype, void *out, void *stream) {
    lla_status st = check_geometry(g);
    if (st != LLA_OK) return st;
    if ((st = check_cache(cache, true)) != LLA_OK) return st;
    if (!codec || !codec->w_up_k || !codec->w_up_v) return LLA_ERR_INVALID_ARG;
    if (!aligned(codec->w_up_k, 16) || !aligned(codec->w_up_v, 16)) return LLA_ERR_INVALID_ARG;
    if ((q && !aligned(q, 16)) || (out && !aligned(out, 16))) return LLA_ERR_INVALID_ARG;
    if (loop < 0 || loop >= g->T || B < 0 || B > LLA_MAX_BATCH || !valid_dtype(io_dtype))
        return LLA_ERR_INVALID_ARG;
    if (max_len < 0 || static_cast<int64_t>(max_len) >
                           static_cast<int64_t>(cache->max_blocks_per_seq) * LLA_BLOCK_TOKENS)
        return LLA_ERR_INVALID_ARG;
    if (B > 0 && (!cu_seqlens || !q || !out)) return LLA_ERR_INVALID_ARG;
    if (B == 0 || max_len == 0) return LLA_OK;
    PrefillArgs a = {};
    a.T = g->T; a.H = g->H; a.d = g->d; a.r_k = g->r_k; a.r_v = g->r_v; a.loop = loop;
    a.storage_bf16 = g->storage == LLA_BF16;
    a.io_bf16 = io_dtype == LLA_BF16;
    a.scale = g->scale;
    a.w_up_k = codec->w_up_k; a.w_up_v = codec->w_up_v;
    a.mu_k = codec->mu_k; a.mu_v = codec->mu_v;
    a.pool = cache->pool; a.num_blocks = cache->num_blocks;
    a.block_table = cache->block_table; a.max_blocks = cache->max_blocks_per_seq;
    a.cu_seqlens = cu_seqlens; a.B = B; a.max_len = max_len;
    a.q = q; a.out = out;
    return launch_prefill(a, static_cast<cudaStream_t>(stream));
}

lla_status lla_prefill_rope_workspace_size(const lla_geometry *g, int32_t B, int32_t max_len,
                                           size_t *bytes) {
    lla_status st = check_geometry(g);
    if (st != LLA_OK) return st;
    if (!bytes || B < 0 || B > LLA_MAX_BATCH || max_len < 0) return LLA_ERR_INVALID_ARG;
    if (!prefill_rope_supported(elem_size(g->storage), g->d, g->r_k, g->r_v)) return LLA_ERR_UNSUPPORTED;
    *bytes = prefill_rope_workspace_bytes(B, max_len, g->H);
    return LLA_OK;
}

lla_status lla_prefill_attn_rope(const lla_geometry *g, const lla_codec *codec,
                                 const lla_cache *cache, const lla_rope *rope,
                                 const int32_t *cu_seqlens, int32_t B, int32_t max_len,
                                 int32_t loop, const void *q, lla_dtype io_dtype, void *out,
                                 void *workspace, size_t workspace_bytes, void *stream) {
    lla_status st = check_geometry(g);
    if (st != LLA_OK) return st;
    if ((st = check_cache(cache, true)) != LLA_OK) return st;
    if (!rope || !(rope->base > 1.0) || !(rope->base < 1e300)) return LLA_ERR_INVALID_ARG;
    if (rope->pairing != LLA_ROPE_HALF && rope->pairing != LLA_ROPE_ADJACENT) return LLA_ERR_INVALID_ARG;
    if (!codec || !codec->w_up_k || !codec->w_up_v) return LLA_ERR_INVALID_ARG;
    if (!aligned(codec->w_up_k, 16) || !aligned(codec->w_up_v, 16)) return LLA_ERR_INVALID_ARG;
    if ((q && !aligned(q, 16)) || (out && !aligned(out, 16))) return LLA_ERR_INVALID_ARG;
    if (loop < 0 || loop >= g->T || B < 0 || B > LLA_MAX_BATCH || !valid_dtype(io_dtype))
        return LLA_ERR_INVALID_ARG;
    if (max_len < 0 || static_cast<int64_t>(max_len) >
                           static_cast<int64_t>(cache->max_blocks_per_seq) * LLA_BLOCK_TOKENS)
        return LLA_ERR_INVALID_ARG;
    if (B > 0 && (!cu_seqlens || !q || !out)) return LLA_ERR_INVALID_ARG;
    if (!prefill_rope_supported(elem_size(g->storage), g->d, g->r_k, g->r_v)) return LLA_ERR_UNSUPPORTED;
    if (B == 0 || max_len == 0) return LLA_OK;
    if (!workspace || !aligned(workspace, 16)) return LLA_ERR_INVALID_ARG;
    PrefillArgs a = {};
    a.T = g->T; a.H = g->H; a.d = g->d; a.r_k = g->r_k; a.r_v = g->r_v; a.loop = loop;
    a.storage_bf16 = g->storage == LLA_BF16;
    a.io_bf16 = io_dtype == LLA_BF16;
    a.scale = g->scale;
    a.w_up_k = codec->w_up_k; a.w_up_v = codec->w_up_v;
    a.mu_k = codec->mu_k; a.mu_v = codec->mu_v;
    a.pool = cache->pool; a.num_blocks = cache->num_blocks;
    a.block_table = cache->block_table; a.max_blocks = cache->max_blocks_per_seq;
    a.cu_seqlens = cu_seqlens; a.B = B; a.max_len = max_len;
    a.q = q; a.out = out;
    return launch_prefill_rope(a, rope->base, rope->pairing == LLA_ROPE_ADJACENT ? 1 : 0, workspace,
                               workspace_bytes, static_cast<cudaStream_t>(stream));
}

lla_status lla_get_device_error(void *stream, uint32_t *word) {
    if (!word) return LLA_ERR_INVALID_ARG;
    lla_status st = LLA_OK;
    unsigned *addr = device_error_word(&st);
    if (st != LLA_OK) return st;
    unsigned host = 0;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (cudaMemcpyAsync(&host, addr, sizeof(unsigned), cudaMemcpyDeviceToHost, s) != cudaSuccess)
        return LLA_ERR_CUDA;
    if (cudaStreamSynchronize(s) != cudaSuccess) return LLA_ERR_CUDA;
    *word = host;
    if (host == 0) return LLA_OK;
    return (host & LLA_DEVERR_TIMEOUT) ? LLA_ERR_TIMEOUT : LLA_ERR_DEVICE_CHECK;
}

lla_status lla_set_wait_limit_ns(uint64_t nanoseconds) {
    g_wait_limit_ns.store(nanoseconds, std::memory_order_relaxed);
    return LLA_OK;
}

uint64_t lla_get_wait_limit_ns(void) {
    const uint64_t v = g_wait_limit_ns.load(std::memory_order_relaxed);
    return v ? v : LLA_DEFAULT_WAIT_LIMIT_NS;
}

lla_status lla_clear_device_error(void *stream) {
    lla_status st = LLA_OK;
    unsigned *addr = device_error_word(&st);
    if (st != LLA_OK) return st;
    if (cudaMemsetAsync(addr, 0, sizeof(unsigned), static_cast<cudaStream_t>(stream)) != cudaSuccess)
        return LLA_ERR_CUDA;
    return LLA_OK;
}

}  // extern "C"
