// lla_encode_tc.cu -- Eq. encode (Sec. 3) of a prompt on tcgen05 tensor cores.
//
// Per (tile of 128 tokens, head h, group of up to 192 latent columns of axis a):
//   C[128 x R] = X[128 x T*d] W_down[T*d x R] - mu W_down,
// with X the stacked loop vectors of the tile's tokens (row n, column t*d + e = x_t[n][h][e]).
// bf16 operands, fp32 accumulation in TMEM, latents rounded to bf16 and scattered to each
// token's slot.  Warp roles:
//   warp 0     producer: per slab of 64 reduction rows, TMA tensor loads with 128-byte swizzle of
//              the x tile (one box of 128 tokens x 64 elements: a K-major operand) and of W_down
//              (one box of 64 rows x 64 columns per 64 latent columns: an MN-major operand),
//              into a ring of stages
//   warp 1     MMA issuer and TMEM owner: 4 MMAs (K = 16) per slab, M = 128, N = R
// Column groups keep a CTA at about 100 KB of shared memory and 256 TMEM columns, so two CTAs
// share an SM and one's epilogue overlaps the other's stream (ranks above 192 split in equal
// groups: 320 = 2 x 160).
//   warps 2-5  the bias mu W_down of the tile's columns (CUDA cores, overlapping the stream),
//              then one token row per thread: TMEM -> bias -> bf16 -> the paged cache.
// Tokens past N read as zeros (tensor-map fill) and are not stored.
#include <cuda_runtime.h>

#include "lla_device.cuh"
#include "lla_internal.h"
#include "lla_tcgen05.cuh"
#include "lla_tmap.h"

namespace lla {
namespace {

constexpr int kEM = 128;  // tokens per tile
constexpr int kES = 64;   // reduction rows per slab
constexpr int kEThreads = 192;

template <int R>
struct EF {
    static constexpr int ATOMS = (R + 63) / 64;         // 64-column atoms of W_down per slab
    static constexpr int ASLAB = kEM * kES * 2;         // x slab (16 KB)
    static constexpr int BATOM = kES * 128;             // one W_down atom column (8 KB)
    static constexpr int BSLAB = ATOMS * BATOM;
    static constexpr int STAGE = ASLAB + BSLAB;
    static constexpr int ST0 = (100 * 1024) / STAGE;    // two CTAs per SM
    static constexpr int ST = ST0 > 4 ? 4 : (ST0 < 2 ? 2 : ST0);
    static constexpr int oBias = ST * STAGE;
    static constexpr int oBar = oBias + R * 4;
    static constexpr int SMEM = 1024 + oBar + (2 * ST + 2) * 8 + 16;  // + alignment slack
    static constexpr uint32_t TM_COLS = 256;
    static_assert(R % 32 == 0 && R <= 256, "column group");
    static_assert(SMEM <= 113 * 1024, "two CTAs per SM");
};

struct ETParams {
    int T, H, d, N, axis;  // axis 0: K latents (granule-interleaved plane), 1: V (row-major)
    int r;                 // rank of the axis (row length of W_down and of the V-plane)
    int r_k, r_v;
    const float *mu;
    const void *w_down;     // [H][T*d][r] bf16 (for the bias)
    char *pool;
    int64_t num_blocks, block_bytes;
    int head_page_bytes, kplane_bytes;
    const int64_t *slot_mapping;
    unsigned *err;
};

template <int R>
__global__ void __launch_bounds__(kEThreads, 1)
    encode_tc_kernel(const __grid_constant__ CUtensorMap tx, const __grid_constant__ CUtensorMap tw,
                     const ETParams p) {
    using F = EF<R>;
    extern __shared__ __align__(1024) char sm_raw[];
    // 128-byte swizzle atoms need a 1024-byte aligned base
    char *sm = reinterpret_cast<char *>((reinterpret_cast<uintptr_t>(sm_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    float *bias = reinterpret_cast<float *>(sm + F::oBias);
    uint64_t *full = reinterpret_cast<uint64_t *>(sm + F::oBar);
    uint64_t *empty = full + F::ST;
    uint64_t *accfull = empty + F::ST;
    volatile int *abort_flag = reinterpret_cast<volatile int *>(accfull + 1);
    uint32_t *tslot = reinterpret_cast<uint32_t *>(accfull + 2);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int n0 = blockIdx.x * kEM, h = blockIdx.y;
    const int col0 = blockIdx.z * R;  // this CTA's column group
    const int Td = p.T * p.d;
    const int NS = Td / kES;

    if (tid == 0) {
        for (int s = 0; s < F::ST; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        mbar_init(accfull, 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 1) tmem_alloc(tslot, F::TM_COLS);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tslot;
    pdl_wait();  // x, slots and the pool may come from the previous kernel

    if (warp == 0) {
        // ------------------------------------------------------------------------- producer
        for (int s = 0; s < NS; ++s) {
            const int st = s % F::ST;
            const uint32_t ph = (s / F::ST) & 1;
            mbar_wait(&empty[st], ph ^ 1u, abort_flag, p.err);
            if (lane == 0) mbar_arrive_expect_tx(&full[st], F::STAGE);
            __syncwarp();
            char *a = sm + st * F::STAGE;
            char *b = a + F::ASLAB;
            const int k0 = s * kES, t = k0 / p.d, e0 = k0 - t * p.d;
            if (lane == 0) tma_load_4d(a, &tx, e0, h, n0, t, &full[st]);
            if (lane < F::ATOMS) tma_load_3d(b + lane * F::BATOM, &tw, col0 + lane * 64, k0, h, &full[st]);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            const uint32_t base = smem_addr(sm);
            constexpr uint32_t id0 = umma_idesc_bf16(128, R, 0, 1);
#pragma unroll 1
            for (int s = 0; s < NS; ++s) {
                const int st = s % F::ST;
                mbar_wait(&full[st], (s / F::ST) & 1, abort_flag, p.err);
                tc_fence_after();
                const uint32_t a = base + st * F::STAGE, b = a + F::ASLAB;
#pragma unroll
                for (int ks = 0; ks < kES / 16; ++ks) {
                    umma_bf16(tmem, umma_desc_sw128_k(a + ks * 32), umma_desc_sw128_mn(b + ks * 2048, F::BATOM),
                              id0, s > 0 || ks > 0);
                }
                umma_commit(&empty[st]);
            }
            umma_commit(accfull);
        }
        __syncwarp();
    } else {
        // --------------------------------------------------------------------------- epilogue
        const int et = tid - 64;  // 0..127
        const char *W = static_cast<const char *>(p.w_down) + static_cast<int64_t>(h) * Td * p.r * 2;
        for (int c = et; c < R; c += 128) {
            float acc = 0.f;
            if (p.mu) {
                const float *mu = p.mu + static_cast<int64_t>(h) * Td;
#pragma unroll 8
                for (int k = 0; k < Td; ++k)
                    acc = fmaf(mu[k], bf_to_f(reinterpret_cast<const uint16_t *>(W)[static_cast<int64_t>(k) * p.r + col0 + c]), acc);
            }
            bias[c] = acc;
        }
        named_bar_sync(1, 128);
        const int quarter = warp & 3;
        const int row = quarter * 32 + lane;
        const int n = n0 + row;
        const uint32_t tl = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
        char *dst = nullptr;
        if (n < p.N) {
            const int64_t slot = p.slot_mapping[n];
            if (slot >= 0) {
                const int64_t blk = slot / kBlockTokens;
                const int r_in = static_cast<int>(slot % kBlockTokens);
                if (blk >= p.num_blocks) {
                    atomicOr(p.err, LLA_DEVERR_SLOT);
                } else {
                    char *page = p.pool + blk * p.block_bytes + static_cast<int64_t>(h) * p.head_page_bytes;
                    dst = p.axis == 0 ? page + r_in * 16 : page + p.kplane_bytes + static_cast<int64_t>(r_in) * p.r * 2;
                }
            }
        }
        mbar_wait(accfull, 0, abort_flag, p.err);
        tc_fence_after();
#pragma unroll 1
        for (int c0 = 0; c0 < R; c0 += 32) {
            float v[32];
            tmem_ld32(tl + c0, v);  // warp-collective: every lane loads, valid rows store
            if (dst) {
#pragma unroll
                for (int k = 0; k < 32; k += 8) {
                    if (c0 + k < R) {
                        const int c = c0 + k, j = col0 + c;  // column within the group, within the axis
                        const uint4 w = make_uint4(pack_bf16(v[k] - bias[c], v[k + 1] - bias[c + 1]),
                                                   pack_bf16(v[k + 2] - bias[c + 2], v[k + 3] - bias[c + 3]),
                                                   pack_bf16(v[k + 4] - bias[c + 4], v[k + 5] - bias[c + 5]),
                                                   pack_bf16(v[k + 6] - bias[c + 6], v[k + 7] - bias[c + 7]));
                        // K-plane: granule j/8 of 16 bytes at (j/8) * 64 * 16 + row * 16
                        char *o = p.axis == 0 ? dst + (j / 8) * (kBlockTokens * 16) : dst + j * 2;
                        *reinterpret_cast<uint4 *>(o) = w;
                    }
                }
            }
        }
    }
    pdl_trigger();
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, F::TM_COLS);
    }
}

template <int R>
lla_status launch_axis(const EncodeArgs &a, int axis, int groups, cudaStream_t stream, unsigned *err) {
    const int Td = a.T * a.d;
    const int r = axis ? a.r_v : a.r_k;
    CUtensorMap tx, tw;
    const void *x = axis ? a.x_v : a.x_k;
    const void *w = axis ? a.w_down_v : a.w_down_k;
    {
        const uint64_t dims[4] = {static_cast<uint64_t>(a.d), static_cast<uint64_t>(a.H),
                                  static_cast<uint64_t>(a.N), static_cast<uint64_t>(a.T)};
        const uint64_t strides[3] = {static_cast<uint64_t>(a.d) * 2, static_cast<uint64_t>(a.H) * a.d * 2,
                                     static_cast<uint64_t>(a.N) * a.H * a.d * 2};
        const uint32_t box[4] = {kES, 1, kEM, 1};
        if (!encode_tmap_bf16(&tx, x, 4, dims, strides, box, true)) return LLA_ERR_CUDA;
    }
    {
        const uint64_t dims[3] = {static_cast<uint64_t>(r), static_cast<uint64_t>(Td), static_cast<uint64_t>(a.H)};
        const uint64_t strides[2] = {static_cast<uint64_t>(r) * 2, static_cast<uint64_t>(Td) * r * 2};
        const uint32_t box[3] = {64, kES, 1};
        if (!encode_tmap_bf16(&tw, w, 3, dims, strides, box, true)) return LLA_ERR_CUDA;
    }
    ETParams p = {};
    p.T = a.T; p.H = a.H; p.d = a.d; p.N = a.N; p.axis = axis; p.r = r;
    p.r_k = a.r_k; p.r_v = a.r_v;
    p.mu = axis ? a.mu_v : a.mu_k;
    p.w_down = w;
    p.pool = static_cast<char *>(a.pool);
    p.num_blocks = a.num_blocks;
    p.head_page_bytes = static_cast<int>(head_page_bytes(a.r_k, a.r_v, 2));
    p.block_bytes = static_cast<int64_t>(p.head_page_bytes) * a.H;
    p.kplane_bytes = LLA_BLOCK_TOKENS * a.r_k * 2;
    p.slot_mapping = a.slot_mapping;
    p.err = err;
    static bool configured[64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return LLA_ERR_CUDA;
    if (dev < 64 && !configured[dev]) {
        if (cudaFuncSetAttribute(encode_tc_kernel<R>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 EF<R>::SMEM) != cudaSuccess)
            return LLA_ERR_CUDA;
        configured[dev] = true;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((a.N + kEM - 1) / kEM, a.H, groups);
    cfg.blockDim = dim3(kEThreads);
    cfg.dynamicSmemBytes = EF<R>::SMEM;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (cudaLaunchKernelEx(&cfg, encode_tc_kernel<R>, tx, tw, p) != cudaSuccess) return LLA_ERR_CUDA;
    return LLA_OK;
}

using AxisLauncher = lla_status (*)(const EncodeArgs &, int, int, cudaStream_t, unsigned *);

// Column groups of an axis of rank r: equal groups of at most 192 columns (a multiple of 32).
struct Groups {
    AxisLauncher launch;
    int n;
};
Groups axis_groups(int r) {
    const int n = (r + 191) / 192;
    if (r % n != 0) return Groups{nullptr, 0};
    switch (r / n) {
        case 96: return Groups{launch_axis<96>, n};
        case 128: return Groups{launch_axis<128>, n};
        case 160: return Groups{launch_axis<160>, n};
        case 192: return Groups{launch_axis<192>, n};
        default: return Groups{nullptr, 0};
    }
}

}  // namespace

bool encode_tc_supported(const EncodeArgs &a) {
    return a.storage_bf16 && a.x_bf16 && !a.dense && a.d % kES == 0 && a.N >= kEM &&
           a.H <= 65535 && axis_groups(a.r_k).launch && axis_groups(a.r_v).launch;
}

lla_status launch_encode_tc(const EncodeArgs &a, cudaStream_t stream) {
    lla_status st = LLA_OK;
    unsigned *err = device_error_word(&st);
    if (st != LLA_OK) return st;
    const Groups gk = axis_groups(a.r_k), gv = axis_groups(a.r_v);
    if ((st = gk.launch(a, 0, gk.n, stream, err)) != LLA_OK) return st;
    return gv.launch(a, 1, gv.n, stream, err);
}

}  // namespace lla
