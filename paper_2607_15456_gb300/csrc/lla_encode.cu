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
// The tile's centred stacked vectors are staged in shared memory (fp32); 256 threads are 16
// column pairs x 16 slices of the T*d reduction axis, each streaming its slice of W_down with
// several loads in flight, and the 16 partial sums per output meet in shared memory.  At a decode
// step (N = batch) this spreads the weight-bound work over H x (r_k + r_v)/32 CTAs.
#include <cuda_runtime.h>

#include "lla_device.cuh"
#include "lla_internal.h"

namespace lla {
namespace {

constexpr int kThreads = 256;
constexpr int kColTile = 32;          // latent columns per CTA
constexpr int kPairs = kColTile / 2;  // column pairs per CTA
constexpr int kSlices = kThreads / kPairs;  // slices of the reduction axis
constexpr int kMaxTileTokens = 16;
constexpr int kXsBudget = 96 * 1024;  // shared bytes for the staged token tile

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

template <int ES>
__global__ void __launch_bounds__(kThreads) encode_kernel(const EncParams p) {
    extern __shared__ __align__(16) float smem_f[];
    const int Td = p.T * p.d;
    float *xs = smem_f;                          // [tile][Td] centred stacked vectors
    float *red = smem_f + p.tile * Td;           // [kSlices][tile][kColTile] partial sums
    const int ct = blockIdx.y;
    const int axis = ct < p.ctiles_k ? 0 : 1;
    const int col0 = (axis ? ct - p.ctiles_k : ct) * kColTile;
    const int h = blockIdx.z;
    const int n0 = blockIdx.x * p.tile;
    const int nt = min(p.tile, p.N - n0);
    const int r = axis ? p.r_v : p.r_k;
    const void *W = axis ? p.w_down_v : p.w_down_k;
    const float *mu = axis ? p.mu_v : p.mu_k;
    const void *x = axis ? p.x_v : p.x_k;
    const int tid = threadIdx.x;

    pdl_wait();
    // stack the loop vectors of the tile's tokens and centre them: x - mu
    for (int idx = tid; idx < nt * Td; idx += kThreads) {
        const int n = idx / Td, k = idx - n * Td;
        const int t = k / p.d, e = k - t * p.d;
        const int64_t src = ((static_cast<int64_t>(t) * p.N + n0 + n) * p.H + h) * p.d + e;
        float v = load_elem(x, src, p.x_bf16);
        if (mu) v -= mu[static_cast<int64_t>(h) * Td + k];
        xs[n * Td + k] = v;
    }
    __syncthreads();

    // c = (x - mu) W_down over this thread's slice of the reduction axis
    const int jp = tid % kPairs, sl = tid / kPairs;
    const int col = col0 + 2 * jp;
    const bool active = col < r;
    float2 acc[kMaxTileTokens];
#pragma unroll
    for (int i = 0; i < kMaxTileTokens; ++i) acc[i] = make_float2(0.f, 0.f);
    if (active) {
        const int64_t wbase = static_cast<int64_t>(h) * Td * r + col;
        int k = sl;
        for (; k + 3 * kSlices < Td; k += 4 * kSlices) {
            float2 w[4];
#pragma unroll
            for (int u = 0; u < 4; ++u)
                w[u] = load_pair<ES>(W, wbase + static_cast<int64_t>(k + u * kSlices) * r);
#pragma unroll
            for (int u = 0; u < 4; ++u) {
#pragma unroll
                for (int i = 0; i < kMaxTileTokens; ++i) {
                    if (i < nt) {
                        const float xv = xs[i * Td + k + u * kSlices];
                        acc[i].x = fmaf(xv, w[u].x, acc[i].x);
                        acc[i].y = fmaf(xv, w[u].y, acc[i].y);
                    }
                }
            }
        }
        for (; k < Td; k += kSlices) {
            const float2 w = load_pair<ES>(W, wbase + static_cast<int64_t>(k) * r);
#pragma unroll
            for (int i = 0; i < kMaxTileTokens; ++i) {
                if (i < nt) {
                    const float xv = xs[i * Td + k];
                    acc[i].x = fmaf(xv, w.x, acc[i].x);
                    acc[i].y = fmaf(xv, w.y, acc[i].y);
                }
            }
        }
    }
#pragma unroll
    for (int i = 0; i < kMaxTileTokens; ++i) {
        if (i < nt) {
            red[(sl * p.tile + i) * kColTile + 2 * jp] = acc[i].x;
            red[(sl * p.tile + i) * kColTile + 2 * jp + 1] = acc[i].y;
        }
    }
    __syncthreads();

    // sum the slices, round to the storage dtype and scatter to each token's slot
    const int gk = granule_bytes(p.r_k, ES);
    for (int o = tid; o < nt * kColTile; o += kThreads) {
        const int i = o / kColTile, c = o % kColTile;
        const int j = col0 + c;
        if (j >= r) continue;
        float v = 0.f;
        for (int s2 = 0; s2 < kSlices; ++s2) v += red[(s2 * p.tile + i) * kColTile + c];
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
lla_status set_smem(int dev) {
    static bool configured[64] = {};
    if (dev < 64 && configured[dev]) return LLA_OK;
    if (cudaFuncSetAttribute(encode_kernel<ES>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             kXsBudget + kSlices * kMaxTileTokens * kColTile * 4) != cudaSuccess)
        return LLA_ERR_CUDA;
    if (dev < 64) configured[dev] = true;
    return LLA_OK;
}

}  // namespace

lla_status launch_encode(const EncodeArgs &a, cudaStream_t stream) {
    if (a.N == 0) return LLA_OK;
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
    const int ctiles_v = (a.r_v + kColTile - 1) / kColTile;
    const int smem = (tile * Td + kSlices * tile * kColTile) * 4;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return LLA_ERR_CUDA;
    st = es == 2 ? set_smem<2>(dev) : set_smem<4>(dev);
    if (st != LLA_OK) return st;
    if (a.H > 65535) return LLA_ERR_UNSUPPORTED;
    const dim3 grid((a.N + tile - 1) / tile, p.ctiles_k + ctiles_v, a.H), block(kThreads);
    return es == 2 ? launch(encode_kernel<2>, grid, block, smem, stream, p)
                   : launch(encode_kernel<4>, grid, block, smem, stream, p);
}

}  // namespace lla
