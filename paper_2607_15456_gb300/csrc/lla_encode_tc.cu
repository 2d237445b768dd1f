// lla_encode_tc.cu -- Eq. encode (Sec. 3) of a prompt on tcgen05 tensor cores, both axes in one
// persistent launch.
//
// A unit is (head h, tile of 128 tokens, column group g of one axis):
//   C[128 x R] = X[128 x T*d] W_down[T*d x R] - mu W_down,
// with X the stacked loop vectors of the tile's tokens (row n, column t*d + e = x_t[n][h][e]).
// An axis of rank r is cut into equal column groups of at most 192 columns (320 = 2 x 160).
// Units are numbered head-major, then tile, then group (K groups first): one CTA per SM takes an
// equal contiguous range of them, so the groups of a tile follow one another on the same SM and
// the second read of a tile's x_v hits L2, and a CTA meets few heads (the bias mu W_down is
// computed once per head it meets).  bf16 operands, fp32 accumulation in TMEM, latents rounded
// to bf16 and scattered to each token's slot.  Warp roles:
//   warp 0     x producer: per slab of 64 reduction rows, a TMA tensor load with 128-byte swizzle
//              of the x tile (one box of 128 tokens x 64 elements: a K-major operand) into its
//              own ring, which runs on across units
//   warp 6     W producer: the slab's W_down (boxes of 64 rows x 64 columns: an MN-major
//              operand) into a second ring; the two rings let the x stream from HBM run ahead
//              of the W_down stream from L2 (one shared ring of 40 KB stages gave x only 16 of
//              every 40 bytes in flight)
//   warp 1     MMA issuer and TMEM owner: 4 MMAs (K = 16) per slab, M = 128, N = R, into one of
//              two accumulator slots, so a unit's epilogue overlaps the next unit's products
//   warps 2-5  epilogue: one token row per thread, TMEM -> bias -> bf16 -> the paged cache (V-plane
//              rows pass through a per-warp staging buffer, so a store writes 8 rows of 64 bytes)
// Tokens past N read as zeros (tensor-map fill) and are not stored.
#include <cuda_runtime.h>

#include "lla_device.cuh"
#include "lla_internal.h"
#include "lla_tcgen05.cuh"
#include "lla_tmap.h"

namespace lla {
namespace {

constexpr int kEM = 128;             // tokens per tile
constexpr int kES = 64;              // reduction rows per slab
constexpr int kEThreads = 224;
constexpr int kMaxGroup = 192;       // columns of a group
constexpr int kMaxGroups = 6;        // groups of both axes (ranks up to 512: at most 3 each)
constexpr int kASlab = kEM * kES * 2;   // x slab (16 KB)
constexpr int kBAtom = kES * 128;       // one W_down atom of 64 columns (8 KB)
constexpr int kWStage = 3 * kBAtom;          // 24 KB
constexpr int kXStages = 5;                 // x slabs in flight (from HBM)
constexpr int kWStages = 5;                 // W_down slabs in flight (from L2)
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kSlotCols = 256;  // accumulator slot s at column s * 256
constexpr int oW = kXStages * kASlab;
constexpr int oBias = oW + kWStages * kWStage;
constexpr int oStg = oBias + kMaxGroups * kMaxGroup * 4;   // V-plane store staging: 4 warps x 32 rows x 80 B
constexpr int oBar = oStg + 4 * 32 * 80;
constexpr int kNumBars = 2 * kXStages + 2 * kWStages + 4 + 1;
constexpr int kSmem = 1024 + oBar + kNumBars * 8 + 16;  // + alignment slack, abort flag, TMEM slot
static_assert(kSmem <= 227 * 1024, "shared memory");

struct ETParams {
    int T, H, d, N;
    int r_k, r_v;
    int nk, nv;      // column groups of each axis
    int gk, gv;      // columns per group of each axis
    int tiles;       // ceil(N / 128)
    int64_t units;   // H * tiles * (nk + nv)
    const float *mu_k, *mu_v;           // [H][T*d] or NULL
    const void *w_down_k, *w_down_v;    // [H][T*d][r] bf16 (for the bias)
    char *pool;
    int64_t num_blocks, block_bytes;
    int head_page_bytes, kplane_bytes;
    const int64_t *slot_mapping;
    unsigned *err;
};

struct Unit {
    int h, n0, axis, col0, R;
};

__device__ __forceinline__ Unit unit_of(const ETParams &p, int64_t u) {
    const int G = p.nk + p.nv;
    const int64_t per_head = static_cast<int64_t>(p.tiles) * G;
    Unit U;
    U.h = static_cast<int>(u / per_head);
    const int rem = static_cast<int>(u - U.h * per_head);
    const int tile = rem / G, g = rem - tile * G;
    U.n0 = tile * kEM;
    U.axis = g < p.nk ? 0 : 1;
    const int ga = U.axis ? g - p.nk : g;
    U.R = U.axis ? p.gv : p.gk;
    U.col0 = ga * U.R;
    return U;
}

__global__ void __launch_bounds__(kEThreads, 1)
    encode_tc_kernel(const __grid_constant__ CUtensorMap txk, const __grid_constant__ CUtensorMap txv,
                     const __grid_constant__ CUtensorMap twk, const __grid_constant__ CUtensorMap twv,
                     const ETParams p) {
    extern __shared__ __align__(1024) char sm_raw[];
    // 128-byte swizzle atoms need a 1024-byte aligned base
    char *sm = reinterpret_cast<char *>((reinterpret_cast<uintptr_t>(sm_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    float *bias = reinterpret_cast<float *>(sm + oBias);  // [group][192] of the current head
    uint64_t *full = reinterpret_cast<uint64_t *>(sm + oBar);
    uint64_t *empty = full + kXStages;
    uint64_t *wfull = empty + kXStages;
    uint64_t *wempty = wfull + kWStages;
    uint64_t *accfull = wempty + kWStages;  // [2]
    uint64_t *accempty = accfull + 2;     // [2]
    uint64_t *done = accempty + 2;
    volatile int *abort_flag = reinterpret_cast<volatile int *>(done + 1);
    uint32_t *tslot = reinterpret_cast<uint32_t *>(done + 1) + 1;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int64_t u0 = static_cast<int64_t>(blockIdx.x) * p.units / gridDim.x;
    const int64_t u1 = static_cast<int64_t>(blockIdx.x + 1) * p.units / gridDim.x;
    const int Td = p.T * p.d;
    const int NS = Td / kES;

    if (tid == 0) {
        for (int s = 0; s < kXStages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int s = 0; s < kWStages; ++s) {
            mbar_init(&wfull[s], 1);
            mbar_init(&wempty[s], 1);
        }
        for (int s = 0; s < 2; ++s) {
            mbar_init(&accfull[s], 1);
            mbar_init(&accempty[s], 4);  // one arrival per epilogue warp
        }
        mbar_init(done, 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 1) tmem_alloc(tslot, kTmemCols);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tslot;
    pdl_wait();  // x, slots and the pool may come from the previous kernel

    if (warp == 0 || warp == 6) {
        // ------------------------------------------------------------ producers: x (0), W (6)
        const bool isx = warp == 0;
        const int NST = isx ? kXStages : kWStages;
        uint64_t *F = isx ? full : wfull;
        uint64_t *E = isx ? empty : wempty;
        int q = 0;  // slabs issued
        bool stop = false;
        for (int64_t u = u0; u < u1 && !stop; ++u) {
            const Unit U = unit_of(p, u);
            const int atoms = (U.R + 63) / 64;
            const CUtensorMap *tx = U.axis ? &txv : &txk;
            const CUtensorMap *tw = U.axis ? &twv : &twk;
            for (int s = 0; s < NS; ++s) {
                const int st = q % NST;
                const uint32_t ph = (q / NST) & 1;
                int halt = 0;
                if (lane == 0) {
                    halt = !mbar_wait(&E[st], ph ^ 1u, abort_flag, p.err) || *abort_flag;
                    if (!halt) mbar_arrive_expect_tx(&F[st], isx ? kASlab : atoms * kBAtom);
                }
                if (__shfl_sync(0xffffffffu, halt, 0)) {
                    stop = true;
                    break;
                }
                __syncwarp();
                const int k0 = s * kES, t = k0 / p.d, e0 = k0 - t * p.d;
                if (isx) {
                    if (lane == 0) tma_load_4d(sm + st * kASlab, tx, e0, U.h, U.n0, t, &F[st]);
                } else {
                    if (lane < atoms) tma_load_3d(sm + oW + st * kWStage + lane * kBAtom, tw, U.col0 + lane * 64, k0, U.h, &F[st]);
                }
                ++q;
            }
        }
        if (lane == 0 && *abort_flag) {
            volatile int never = 0;
            for (int j = q > NST ? q - NST : 0; j < q; ++j)
                mbar_wait(&F[j % NST], (j / NST) & 1, &never, p.err);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            const uint32_t base = smem_addr(sm);
            int q = 0, j = 0;
            for (int64_t u = u0; u < u1; ++u, ++j) {
                const Unit U = unit_of(p, u);
                const uint32_t idesc = umma_idesc_bf16(128, U.R, 0, 1);
                const int slot = j & 1;
                // the epilogue has read this slot's previous unit (j - 2)
                if (!mbar_wait(&accempty[slot], ((j >> 1) & 1) ^ 1u, abort_flag, p.err)) break;
                tc_fence_after();
                const uint32_t d = tmem + slot * kSlotCols;
                bool ok = true;
#pragma unroll 1
                for (int s = 0; s < NS; ++s, ++q) {
                    const int st = q % kXStages, sw = q % kWStages;
                    if (!mbar_wait(&full[st], (q / kXStages) & 1, abort_flag, p.err) ||
                        !mbar_wait(&wfull[sw], (q / kWStages) & 1, abort_flag, p.err)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t a = base + st * kASlab, b = base + oW + sw * kWStage;
#pragma unroll
                    for (int ks = 0; ks < kES / 16; ++ks)
                        umma_bf16(d, umma_desc_sw128_k(a + ks * 32), umma_desc_sw128_mn(b + ks * 2048, kBAtom),
                                  idesc, s > 0 || ks > 0);
                    umma_commit(&empty[st]);
                    umma_commit(&wempty[sw]);
                }
                if (!ok) break;
                umma_commit(&accfull[slot]);
            }
            // every product has completed before TMEM is released
            umma_commit(done);
            volatile int never = 0;
            mbar_wait(done, 0, &never, p.err);
        }
        __syncwarp();
    } else if (warp <= 5) {
        // --------------------------------------------------------------------------- epilogue
        const int et = tid - 64;  // 0..127
        const int quarter = warp & 3;
        const int row = quarter * 32 + lane;
        int bias_head = -1;
        int j = 0;
        for (int64_t u = u0; u < u1; ++u, ++j) {
            const Unit U = unit_of(p, u);
            const int slot = j & 1;
            const int g = (U.axis ? p.nk : 0) + U.col0 / U.R;
            if ((p.mu_k || p.mu_v) && U.h != bias_head) {
                // mu W_down of every group of this head, eight columns per thread at a time
                named_bar_sync(1, 128);  // the previous head's biases are no longer read
                for (int ax = 0; ax < 2; ++ax) {
                    const float *mu = ax ? p.mu_v : p.mu_k;
                    const int r = ax ? p.r_v : p.r_k, R = ax ? p.gv : p.gk, gbase = ax ? p.nk : 0;
                    const uint16_t *W = static_cast<const uint16_t *>(ax ? p.w_down_v : p.w_down_k) +
                                        static_cast<int64_t>(U.h) * Td * r;
                    for (int c8 = et; c8 < r / 8; c8 += 128) {
                        float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
                        if (mu) {
                            const float *m = mu + static_cast<int64_t>(U.h) * Td;
#pragma unroll 4
                            for (int k = 0; k < Td; ++k) {
                                const uint4 w = *reinterpret_cast<const uint4 *>(W + static_cast<int64_t>(k) * r + c8 * 8);
                                const float mk = m[k];
                                const float2 w0 = bf2_to_f2(w.x), w1 = bf2_to_f2(w.y), w2 = bf2_to_f2(w.z), w3 = bf2_to_f2(w.w);
                                acc[0] = fmaf(mk, w0.x, acc[0]); acc[1] = fmaf(mk, w0.y, acc[1]);
                                acc[2] = fmaf(mk, w1.x, acc[2]); acc[3] = fmaf(mk, w1.y, acc[3]);
                                acc[4] = fmaf(mk, w2.x, acc[4]); acc[5] = fmaf(mk, w2.y, acc[5]);
                                acc[6] = fmaf(mk, w3.x, acc[6]); acc[7] = fmaf(mk, w3.y, acc[7]);
                            }
                        }
                        for (int i = 0; i < 8; ++i) {
                            const int c = c8 * 8 + i;
                            bias[(gbase + c / R) * kMaxGroup + c % R] = acc[i];
                        }
                    }
                }
                named_bar_sync(1, 128);
                bias_head = U.h;
            }
            const float *bs = bias + g * kMaxGroup;
            const bool use_bias = (U.axis ? p.mu_v : p.mu_k) != nullptr;
            const int n = U.n0 + row;
            char *dst = nullptr;
            if (n < p.N) {
                const int64_t slot_id = p.slot_mapping[n];
                if (slot_id >= 0) {
                    const int64_t blk = slot_id / kBlockTokens;
                    const int r_in = static_cast<int>(slot_id % kBlockTokens);
                    if (blk >= p.num_blocks) {
                        if (g == 0) atomicOr(p.err, LLA_DEVERR_SLOT);
                    } else {
                        char *page = p.pool + blk * p.block_bytes + static_cast<int64_t>(U.h) * p.head_page_bytes;
                        dst = U.axis == 0 ? page + r_in * 16
                                          : page + p.kplane_bytes + static_cast<int64_t>(r_in) * p.r_v * 2;
                    }
                }
            }
            mbar_wait(&accfull[slot], (j >> 1) & 1, abort_flag, p.err);
            tc_fence_after();
            const uint32_t tl = tmem + slot * kSlotCols + (static_cast<uint32_t>(quarter * 32) << 16);
            char *stg = sm + oStg + quarter * (32 * 80);
#pragma unroll 1
            for (int c0 = 0; c0 < U.R; c0 += 32) {
                float v[32];
                tmem_ld32(tl + c0, v);  // warp-collective: every lane loads, valid rows store
                if (U.axis == 1) {
                    // V-plane rows are r_v * 2 bytes apart: stage the warp's 32 rows x 64 bytes and
                    // store 8 rows of 64 contiguous bytes per instruction
#pragma unroll
                    for (int k = 0; k < 32; k += 8) {
                        const int c = c0 + k;
                        float b8[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
                        if (use_bias) {
#pragma unroll
                            for (int i = 0; i < 8; ++i) b8[i] = bs[c + i];
                        }
                        *reinterpret_cast<uint4 *>(stg + lane * 80 + (k / 8) * 16) =
                            make_uint4(pack_bf16(v[k] - b8[0], v[k + 1] - b8[1]), pack_bf16(v[k + 2] - b8[2], v[k + 3] - b8[3]),
                                       pack_bf16(v[k + 4] - b8[4], v[k + 5] - b8[5]), pack_bf16(v[k + 6] - b8[6], v[k + 7] - b8[7]));
                    }
                    __syncwarp();
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const int rr = 8 * i + (lane >> 2), cc = lane & 3;
                        char *d = reinterpret_cast<char *>(__shfl_sync(0xffffffffu, reinterpret_cast<unsigned long long>(dst), rr));
                        const uint4 val = *reinterpret_cast<const uint4 *>(stg + rr * 80 + cc * 16);
                        if (d) *reinterpret_cast<uint4 *>(d + (U.col0 + c0 + cc * 8) * 2) = val;
                    }
                    __syncwarp();
                } else if (dst) {
#pragma unroll
                    for (int k = 0; k < 32; k += 8) {
                        const int c = c0 + k, jc = U.col0 + c;  // column in the group, in the axis
                        float b8[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
                        if (use_bias) {
#pragma unroll
                            for (int i = 0; i < 8; ++i) b8[i] = bs[c + i];
                        }
                        const uint4 w = make_uint4(pack_bf16(v[k] - b8[0], v[k + 1] - b8[1]),
                                                   pack_bf16(v[k + 2] - b8[2], v[k + 3] - b8[3]),
                                                   pack_bf16(v[k + 4] - b8[4], v[k + 5] - b8[5]),
                                                   pack_bf16(v[k + 6] - b8[6], v[k + 7] - b8[7]));
                        // K-plane: granule jc/8 of 16 bytes at (jc/8) * 64 * 16 + row * 16
                        char *o = U.axis == 0 ? dst + (jc / 8) * (kBlockTokens * 16) : dst + jc * 2;
                        *reinterpret_cast<uint4 *>(o) = w;
                    }
                }
            }
            // this slot may take unit j + 2
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&accempty[slot]);
        }
    }
    pdl_trigger();
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

bool make_maps(const EncodeArgs &a, int axis, CUtensorMap *tx, CUtensorMap *tw) {
    const int Td = a.T * a.d;
    const int r = axis ? a.r_v : a.r_k;
    const void *x = axis ? a.x_v : a.x_k;
    const void *w = axis ? a.w_down_v : a.w_down_k;
    {
        const uint64_t dims[4] = {static_cast<uint64_t>(a.d), static_cast<uint64_t>(a.H),
                                  static_cast<uint64_t>(a.N), static_cast<uint64_t>(a.T)};
        const uint64_t strides[3] = {static_cast<uint64_t>(a.d) * 2, static_cast<uint64_t>(a.H) * a.d * 2,
                                     static_cast<uint64_t>(a.N) * a.H * a.d * 2};
        const uint32_t box[4] = {kES, 1, kEM, 1};
        if (!encode_tmap_bf16(tx, x, 4, dims, strides, box, true)) return false;
    }
    const uint64_t dims[3] = {static_cast<uint64_t>(r), static_cast<uint64_t>(Td), static_cast<uint64_t>(a.H)};
    const uint64_t strides[2] = {static_cast<uint64_t>(r) * 2, static_cast<uint64_t>(Td) * r * 2};
    const uint32_t box[3] = {64, kES, 1};
    return encode_tmap_bf16(tw, w, 3, dims, strides, box, true);
}

// Column groups of an axis of rank r: n equal groups of at most 192 columns, each a multiple of
// 32 (0 groups when r has no such split).
int axis_groups(int r, int *width) {
    const int n = (r + kMaxGroup - 1) / kMaxGroup;
    if (r % n != 0 || (r / n) % 32 != 0) return 0;
    *width = r / n;
    return n;
}

}  // namespace

bool encode_tc_supported(const EncodeArgs &a) {
    int w = 0;
    return a.storage_bf16 && a.x_bf16 && !a.dense && a.d % kES == 0 && a.N >= kEM &&
           (a.T * a.d) % kES == 0 && axis_groups(a.r_k, &w) && axis_groups(a.r_v, &w) &&
           axis_groups(a.r_k, &w) + axis_groups(a.r_v, &w) <= kMaxGroups;
}

lla_status launch_encode_tc(const EncodeArgs &a, cudaStream_t stream) {
    lla_status st = LLA_OK;
    unsigned *err = device_error_word(&st);
    if (st != LLA_OK) return st;
    ETParams p = {};
    p.T = a.T; p.H = a.H; p.d = a.d; p.N = a.N; p.r_k = a.r_k; p.r_v = a.r_v;
    p.nk = axis_groups(a.r_k, &p.gk);
    p.nv = axis_groups(a.r_v, &p.gv);
    p.tiles = (a.N + kEM - 1) / kEM;
    p.units = static_cast<int64_t>(a.H) * p.tiles * (p.nk + p.nv);
    p.mu_k = a.mu_k; p.mu_v = a.mu_v;
    p.w_down_k = a.w_down_k; p.w_down_v = a.w_down_v;
    p.pool = static_cast<char *>(a.pool);
    p.num_blocks = a.num_blocks;
    p.head_page_bytes = static_cast<int>(head_page_bytes(a.r_k, a.r_v, 2));
    p.block_bytes = static_cast<int64_t>(p.head_page_bytes) * a.H;
    p.kplane_bytes = LLA_BLOCK_TOKENS * a.r_k * 2;
    p.slot_mapping = a.slot_mapping;
    p.err = err;
    CUtensorMap txk, txv, twk, twv;
    if (!make_maps(a, 0, &txk, &twk) || !make_maps(a, 1, &txv, &twv)) return LLA_ERR_CUDA;
    static DeviceOnce configured;
    if (raise_smem_limit(encode_tc_kernel, kSmem, configured) != LLA_OK) return LLA_ERR_CUDA;
    const int sms = num_sms();
    if (sms <= 0) return LLA_ERR_CUDA;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(p.units < sms ? p.units : sms));
    cfg.blockDim = dim3(kEThreads);
    cfg.dynamicSmemBytes = kSmem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (cudaLaunchKernelEx(&cfg, encode_tc_kernel, txk, txv, twk, twv, p) != cudaSuccess) return LLA_ERR_CUDA;
    return LLA_OK;
}

}  // namespace lla
