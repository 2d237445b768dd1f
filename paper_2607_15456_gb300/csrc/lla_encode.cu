// lla_encode.cu -- Eq. encode (Sec. 3) for newly completed tokens, written into the paged cache,
// and the plain K/V page store of the uncompressed comparator.
//
// Encode, per (token n, head h, axis a in {K, V}):
//   x = [x_1; ...; x_T] (stacked loop vectors),  c = (x - mu) W_down   (fp32 accumulation)
// rounded to the storage dtype (round to nearest even for bf16) and scattered to the token's
// slot: the K latent into the granule-interleaved K-plane, the V latent into the row-major
// V-plane of its block's head page.
//
// One CTA takes (a tile of up to 16 tokens, a tile of 32 latent columns of one axis, one head).
// Everything the CTA reads is in flight at once: its W_down columns move into shared memory with
// cp.async in chunks of the T*d reduction axis (double-buffered when T*d is long), and the tile's
// stacked loop vectors are loaded four 16-byte words per thread before any is used, then centred
// (x - mu) into shared memory as fp32.  At a decode step (N = batch) a launch therefore costs
// about one memory round trip.  256 threads are 16 column pairs x 4 groups of 4 tokens x 4
// slices of the reduction axis; the 4 partial sums per output meet in shared memory.
#include <cuda_runtime.h>

#include "lla_device.cuh"
#include "lla_internal.h"

namespace lla {
namespace {

constexpr int kThreads = 256;
constexpr int kColTile = 32;          // latent columns per CTA
constexpr int kPairs = kColTile / 2;  // column pairs per CTA
constexpr int kMaxTileTokens = 16;
constexpr int kTokGroups = kMaxTileTokens / 4;          // groups of 4 tokens
constexpr int kKSlices = kThreads / (kPairs * kTokGroups);  // slices of the reduction axis
constexpr int kXsBudget = 96 * 1024;  // shared bytes for the staged token tile
constexpr int kWBuf = 32 * 1024;      // one chunk of W_down columns (two are in flight)
constexpr int kXBatch = 4;            // 16-byte words of x in flight per thread

struct EncParams {
    int T, H, d, r_k, r_v, x_bf16;
    const void *w_down_k, *w_down_v;
    const float *mu_k, *mu_v;
    const void *x_k, *x_v;
    char *pool;
    int64_t num_blocks, block_bytes;
    int head_page_bytes, kplane_bytes;
    const int64_t *slot_mapping;
    int N, tile, ctiles_k;
    int nbuf;  // W_down chunk buffers: 1 when T*d fits one chunk, else 2
    unsigned *err;
};

template <int ES>
__device__ __forceinline__ float2 load_pair(const void *base, int64_t i) {
    if constexpr (ES == 2) return bf2_to_f2(reinterpret_cast<const uint32_t *>(base)[i >> 1]);
    else return reinterpret_cast<const float2 *>(base)[i >> 1];
}

template <int ES>
__device__ __forceinline__ void store_latent(char *dst, float v) {
    if constexpr (ES == 2) *reinterpret_cast<__nv_bfloat16 *>(dst) = __float2bfloat16_rn(v);
    else *reinterpret_cast<float *>(dst) = v;
}

// Rows of W_down per shared-memory chunk.
template <int ES>
__host__ __device__ constexpr int chunk_rows() { return kWBuf / (kColTile * ES); }

// Starts the copy of rows [k0, k0 + rows) x columns [col0, col0 + ncol) of W (row length r)
// into wb ([rows][kColTile] storage dtype).  16-byte copies when every row segment is 16-byte
// aligned, 4-byte copies otherwise (r x es not a multiple of 16).
template <int ES>
__device__ __forceinline__ void stage_w(char *wb, const char *W, int r, int col0, int ncol, int k0,
                                        int rows, int tid) {
    const bool wide = (r * ES) % 16 == 0 && (ncol * ES) % 16 == 0;
    const int unit = wide ? 16 : 4;
    const int per_row = ncol * ES / unit;
    const int total = rows * per_row;
    for (int i = tid; i < total; i += kThreads) {
        const int k = i / per_row, c = i - k * per_row;
        const char *src = W + (static_cast<int64_t>(k0 + k) * r + col0) * ES + c * unit;
        char *dst = wb + k * (kColTile * ES) + c * unit;
        if (wide) cp_async16(dst, src);
        else cp_async4(dst, src);
    }
    cp_async_commit();
}

template <int ES>
__device__ __forceinline__ void encode_body(const EncParams &p, const int h) {
    extern __shared__ __align__(16) float smem_f[];
    constexpr int KC = chunk_rows<ES>();
    const int Td = p.T * p.d;
    float *xs = smem_f;                                       // [tile][Td] centred stacked vectors
    char *wbuf = reinterpret_cast<char *>(xs + p.tile * Td);  // [2][KC][kColTile] W_down chunks
    float *red = reinterpret_cast<float *>(wbuf + p.nbuf * kWBuf);  // [kKSlices][tile][kColTile]
    const int ct = blockIdx.y;
    const int axis = ct < p.ctiles_k ? 0 : 1;
    const int col0 = (axis ? ct - p.ctiles_k : ct) * kColTile;
    const int n0 = blockIdx.x * p.tile;
    const int nt = min(p.tile, p.N - n0);
    const int r = axis ? p.r_v : p.r_k;
    const int ncol = min(kColTile, r - col0);
    const char *W = static_cast<const char *>(axis ? p.w_down_v : p.w_down_k) +
                    static_cast<int64_t>(h) * Td * r * ES;
    const float *mu = axis ? p.mu_v : p.mu_k;
    const char *x = static_cast<const char *>(axis ? p.x_v : p.x_k);
    const int tid = threadIdx.x;
    const int nch = (Td + KC - 1) / KC;

    pdl_wait();
    stage_w<ES>(wbuf, W, r, col0, ncol, 0, min(KC, Td), tid);
    if (nch > 1) stage_w<ES>(wbuf + kWBuf, W, r, col0, ncol, KC, min(KC, Td - KC), tid);

    // stack the loop vectors of the tile's tokens and centre them: x - mu.  Rows (n, t) of d
    // elements are contiguous in x; kXBatch 16-byte words per thread are loaded before use.
    {
        const int xes = p.x_bf16 ? 2 : 4;
        const int wpr = p.d * xes / 16;  // 16-byte words per row (d is a multiple of 8)
        const int epw = 16 / xes;        // elements per word
        const int total = nt * p.T * wpr;
        for (int base = 0; base < total; base += kThreads * kXBatch) {
            uint4 v[kXBatch];
#pragma unroll
            for (int b = 0; b < kXBatch; ++b) {
                const int i = base + b * kThreads + tid;
                if (i < total) {
                    const int row = i / wpr, c = i - row * wpr;
                    const int n = row / p.T, t = row - n * p.T;
                    const int64_t off =
                        ((static_cast<int64_t>(t) * p.N + n0 + n) * p.H + h) * p.d * xes + c * 16;
                    v[b] = *reinterpret_cast<const uint4 *>(x + off);
                }
            }
#pragma unroll
            for (int b = 0; b < kXBatch; ++b) {
                const int i = base + b * kThreads + tid;
                if (i < total) {
                    const int row = i / wpr, c = i - row * wpr;
                    const int n = row / p.T, t = row - n * p.T;
                    const int k0 = t * p.d + c * epw;
                    float f[8];
                    if (p.x_bf16) {
                        const float2 a = bf2_to_f2(v[b].x), bb = bf2_to_f2(v[b].y),
                                     cc = bf2_to_f2(v[b].z), e = bf2_to_f2(v[b].w);
                        f[0] = a.x; f[1] = a.y; f[2] = bb.x; f[3] = bb.y;
                        f[4] = cc.x; f[5] = cc.y; f[6] = e.x; f[7] = e.y;
                    } else {
                        f[0] = __uint_as_float(v[b].x); f[1] = __uint_as_float(v[b].y);
                        f[2] = __uint_as_float(v[b].z); f[3] = __uint_as_float(v[b].w);
                        f[4] = f[5] = f[6] = f[7] = 0.f;
                    }
#pragma unroll
                    for (int q = 0; q < 8; ++q) {
                        if (q < epw) {
                            float val = f[q];
                            if (mu) val -= mu[static_cast<int64_t>(h) * Td + k0 + q];
                            xs[n * Td + k0 + q] = val;
                        }
                    }
                }
            }
        }
    }

    // c = (x - mu) W_down.  Thread = (column pair jp, group of 4 tokens tg, reduction slice
    // ks); slice ks takes the row quads q = ks, ks + 4, ... of each chunk, so a thread reads a
    // float4 of x per token and one W pair per row.
    const int jp = tid % kPairs, tg = (tid / kPairs) % kTokGroups, ks = tid / (kPairs * kTokGroups);
    const bool active = 2 * jp < ncol && 4 * tg < nt;
    float2 acc[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) acc[i] = make_float2(0.f, 0.f);
    for (int ch = 0; ch < nch; ++ch) {
        if (ch + 1 < nch) cp_async_wait_but_one();
        else cp_async_wait_all();
        __syncthreads();  // chunk ch (and, the first time, the token tile) is visible
        const char *wb = wbuf + (ch & 1) * kWBuf;
        const int kc0 = ch * KC;
        const int quads = min(KC, Td - kc0) / 4;  // T*d and KC are multiples of 8
        if (active) {
            const float *x0 = xs + (4 * tg) * Td + kc0;
#pragma unroll 2
            for (int q = ks; q < quads; q += kKSlices) {
                float4 xv[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) xv[i] = *reinterpret_cast<const float4 *>(x0 + i * Td + 4 * q);
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const float2 w = load_pair<ES>(wb, static_cast<int64_t>(4 * q + u) * kColTile + 2 * jp);
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const float xe = u == 0 ? xv[i].x : u == 1 ? xv[i].y : u == 2 ? xv[i].z : xv[i].w;
                        acc[i].x = fmaf(xe, w.x, acc[i].x);
                        acc[i].y = fmaf(xe, w.y, acc[i].y);
                    }
                }
            }
        }
        if (ch + 2 < nch) {
            __syncthreads();  // every thread is done with this buffer
            stage_w<ES>(wbuf + (ch & 1) * kWBuf, W, r, col0, ncol, (ch + 2) * KC,
                        min(KC, Td - (ch + 2) * KC), tid);
        }
    }
    pdl_trigger();  // the next kernel in the stream may start its launch
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int n = 4 * tg + i;
        if (n < nt) {
            red[(ks * p.tile + n) * kColTile + 2 * jp] = acc[i].x;
            red[(ks * p.tile + n) * kColTile + 2 * jp + 1] = acc[i].y;
        }
    }
    __syncthreads();

    // sum the slices, round to the storage dtype and scatter to each token's slot
    const int gk = granule_bytes(p.r_k, ES);
    for (int o = tid; o < nt * kColTile; o += kThreads) {
        const int i = o / kColTile, c = o % kColTile;
        const int j = col0 + c;
        if (c >= ncol) continue;
        float v = 0.f;
        for (int s2 = 0; s2 < kKSlices; ++s2) v += red[(s2 * p.tile + i) * kColTile + c];
        const int64_t slot = p.slot_mapping[n0 + i];
        if (slot < 0) continue;
        const int64_t blk = slot / kBlockTokens;
        const int row = static_cast<int>(slot % kBlockTokens);
        if (blk >= p.num_blocks) {
            atomicOr(p.err, LLA_DEVERR_SLOT);
            continue;
        }
        char *page = p.pool + blk * p.block_bytes + static_cast<int64_t>(h) * p.head_page_bytes;
        if (axis == 0)
            store_latent<ES>(page + kplane_offset(row, j, ES, gk), v);
        else
            store_latent<ES>(page + p.kplane_bytes + (static_cast<int64_t>(row) * p.r_v + j) * ES, v);
    }
}

template <int ES>
__global__ void __launch_bounds__(kThreads) encode_kernel(const EncParams p) {
    encode_body<ES>(p, blockIdx.z);
}

// Several layers in one launch: blockIdx.z = layer * H + head; each layer's pointers come from
// a table in the kernel parameters.
struct EncLayer {
    const void *w_down_k, *w_down_v;
    const float *mu_k, *mu_v;
    const void *x_k, *x_v;
    char *pool;
    int64_t num_blocks;
};
struct EncLayers {
    EncLayer l[kMaxEncodeLayers];
};

template <int ES>
__global__ void __launch_bounds__(kThreads) encode_layers_kernel(const EncParams p0,
                                                                  const __grid_constant__ EncLayers t) {
    const int layer = blockIdx.z / p0.H;
    EncParams p = p0;
    const EncLayer &e = t.l[layer];
    p.w_down_k = e.w_down_k;
    p.w_down_v = e.w_down_v;
    p.mu_k = e.mu_k;
    p.mu_v = e.mu_v;
    p.x_k = e.x_k;
    p.x_v = e.x_v;
    p.pool = e.pool;
    p.num_blocks = e.num_blocks;
    encode_body<ES>(p, blockIdx.z - layer * p0.H);
}

// Plain K/V store for the uncompressed comparator: k, v [N][H][d] -> K-plane / V-plane of the
// token's slot (r_k = r_v = d).
template <int ES>
__global__ void dense_store_kernel(const EncParams p) {
    const int n = blockIdx.x, h = blockIdx.y;
    pdl_wait();
    const int64_t slot = p.slot_mapping[n];
    if (slot < 0) return;
    const int64_t blk = slot / kBlockTokens;
    const int row = static_cast<int>(slot % kBlockTokens);
    if (blk >= p.num_blocks) {
        if (threadIdx.x == 0) atomicOr(p.err, LLA_DEVERR_SLOT);
        return;
    }
    char *page = p.pool + blk * p.block_bytes + static_cast<int64_t>(h) * p.head_page_bytes;
    const int gk = granule_bytes(p.d, ES);
    const int64_t src = (static_cast<int64_t>(n) * p.H + h) * p.d;
    for (int e = threadIdx.x; e < p.d; e += blockDim.x) {
        store_latent<ES>(page + kplane_offset(row, e, ES, gk), load_elem(p.x_k, src + e, p.x_bf16));
        store_latent<ES>(page + p.kplane_bytes + (static_cast<int64_t>(row) * p.d + e) * ES,
                         load_elem(p.x_v, src + e, p.x_bf16));
    }
}

template <typename K>
lla_status launch(K kern, dim3 grid, dim3 block, int smem, cudaStream_t stream, const EncParams &p) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (cudaLaunchKernelEx(&cfg, kern, p) != cudaSuccess) return LLA_ERR_CUDA;
    return LLA_OK;
}

template <int ES>
lla_status set_smem_layers() {
    static DeviceOnce configured;
    return raise_smem_limit(encode_layers_kernel<ES>, kXsBudget + 2 * kWBuf + kKSlices * kMaxTileTokens * kColTile * 4,
                            configured);
}

template <int ES>
lla_status set_smem() {
    static DeviceOnce configured;
    return raise_smem_limit(encode_kernel<ES>, kXsBudget + 2 * kWBuf + kKSlices * kMaxTileTokens * kColTile * 4,
                            configured);
}

}  // namespace

lla_status launch_encode_layers(const EncodeArgs *a, int L, cudaStream_t stream) {
    if (L <= 0 || a[0].N == 0) return LLA_OK;
    const EncodeArgs &a0 = a[0];
    // prompts take the tensor-core kernel layer by layer; decode batches share one launch
    if (encode_tc_supported(a0) || a0.dense || L > kMaxEncodeLayers) {
        for (int l = 0; l < L; ++l) {
            const lla_status st = launch_encode(a[l], stream);
            if (st != LLA_OK) return st;
        }
        return LLA_OK;
    }
    const int es = a0.storage_bf16 ? 2 : 4;
    lla_status st = LLA_OK;
    unsigned *err = device_error_word(&st);
    if (st != LLA_OK) return st;
    EncParams p = {};
    p.T = a0.T; p.H = a0.H; p.d = a0.d; p.r_k = a0.r_k; p.r_v = a0.r_v; p.x_bf16 = a0.x_bf16;
    p.head_page_bytes = static_cast<int>(head_page_bytes(a0.r_k, a0.r_v, es));
    p.block_bytes = static_cast<int64_t>(p.head_page_bytes) * a0.H;
    p.kplane_bytes = LLA_BLOCK_TOKENS * a0.r_k * es;
    p.slot_mapping = a0.slot_mapping;
    p.N = a0.N;
    p.err = err;
    EncLayers t = {};
    for (int l = 0; l < L; ++l)
        t.l[l] = EncLayer{a[l].w_down_k, a[l].w_down_v, a[l].mu_k, a[l].mu_v, a[l].x_k, a[l].x_v,
                          static_cast<char *>(a[l].pool), a[l].num_blocks};
    const int Td = a0.T * a0.d;
    int tile = kXsBudget / (Td * 4);
    if (tile > kMaxTileTokens) tile = kMaxTileTokens;
    if (tile < 1) return LLA_ERR_UNSUPPORTED;
    p.tile = tile;
    p.ctiles_k = (a0.r_k + kColTile - 1) / kColTile;
    p.nbuf = Td > (es == 2 ? chunk_rows<2>() : chunk_rows<4>()) ? 2 : 1;
    const int ctiles_v = (a0.r_v + kColTile - 1) / kColTile;
    const int smem = (tile * Td + kKSlices * tile * kColTile) * 4 + p.nbuf * kWBuf;
    st = es == 2 ? set_smem_layers<2>() : set_smem_layers<4>();
    if (st != LLA_OK) return st;
    if (static_cast<int64_t>(a0.H) * L > 65535) return LLA_ERR_UNSUPPORTED;
    const dim3 grid((a0.N + tile - 1) / tile, p.ctiles_k + ctiles_v, a0.H * L), block(kThreads);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    const cudaError_t e = es == 2 ? cudaLaunchKernelEx(&cfg, encode_layers_kernel<2>, p, t)
                                  : cudaLaunchKernelEx(&cfg, encode_layers_kernel<4>, p, t);
    return e == cudaSuccess ? LLA_OK : LLA_ERR_CUDA;
}

lla_status launch_encode(const EncodeArgs &a, cudaStream_t stream) {
    if (a.N == 0) return LLA_OK;
    if (encode_tc_supported(a)) return launch_encode_tc(a, stream);
    const int es = a.storage_bf16 ? 2 : 4;
    lla_status st = LLA_OK;
    unsigned *err = device_error_word(&st);
    if (st != LLA_OK) return st;
    EncParams p = {};
    p.T = a.T; p.H = a.H; p.d = a.d; p.r_k = a.r_k; p.r_v = a.r_v; p.x_bf16 = a.x_bf16;
    p.w_down_k = a.w_down_k; p.w_down_v = a.w_down_v; p.mu_k = a.mu_k; p.mu_v = a.mu_v;
    p.x_k = a.x_k; p.x_v = a.x_v;
    p.pool = static_cast<char *>(a.pool);
    p.num_blocks = a.num_blocks;
    p.head_page_bytes = static_cast<int>(head_page_bytes(a.r_k, a.r_v, es));
    p.block_bytes = static_cast<int64_t>(p.head_page_bytes) * a.H;
    p.kplane_bytes = LLA_BLOCK_TOKENS * a.r_k * es;
    p.slot_mapping = a.slot_mapping;
    p.N = a.N;
    p.err = err;
    if (a.dense) {
        const dim3 grid(a.N, a.H), block(128);
        return es == 2 ? launch(dense_store_kernel<2>, grid, block, 0, stream, p)
                       : launch(dense_store_kernel<4>, grid, block, 0, stream, p);
    }
    const int Td = a.T * a.d;
    int tile = kXsBudget / (Td * 4);
    if (tile > kMaxTileTokens) tile = kMaxTileTokens;
    if (tile < 1) return LLA_ERR_UNSUPPORTED;
    p.tile = tile;
    p.ctiles_k = (a.r_k + kColTile - 1) / kColTile;
    p.nbuf = Td > (es == 2 ? chunk_rows<2>() : chunk_rows<4>()) ? 2 : 1;
    const int ctiles_v = (a.r_v + kColTile - 1) / kColTile;
    const int smem = (tile * Td + kKSlices * tile * kColTile) * 4 + p.nbuf * kWBuf;
    st = es == 2 ? set_smem<2>() : set_smem<4>();
    if (st != LLA_OK) return st;
    if (a.H > 65535) return LLA_ERR_UNSUPPORTED;
    const dim3 grid((a.N + tile - 1) / tile, p.ctiles_k + ctiles_v, a.H), block(kThreads);
    return es == 2 ? launch(encode_kernel<2>, grid, block, smem, stream, p)
                   : launch(encode_kernel<4>, grid, block, smem, stream, p);
}

}  // namespace lla
