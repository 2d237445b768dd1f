// lla_decode_rope_tc.cu -- decode with rotary positions applied after reconstruction (Sec. 3
// "RoPE and reconstruction"; App. A "Decoding and caching"), keys rebuilt and latent values summed
// on the tensor cores.
//
// The codec holds pre-RoPE keys.  Cached key i of a sequence sits at position p_i = i; the query
// (and, in pass 1, the current token's exact key) at P = L in pass 1 and P = L - 1 in pass 2.
// RoPE (RoFormer) turns pair j of a vector at position p by p theta_j, theta_j = base^(-2j/d):
//   s_i = scale rot(q, P) . rot(khat_i, p_i) = scale rot(q, P - p_i) . khat_i,
//   khat_i = W_up,t^K c_k,i + mu^K_t                                           (Eq. decode)
//   o = (W_up,t^V sum_i p_i c_v,i + (sum_i p_i) mu^V_t + p_cur v_cur) / (sum_i p_i + p_cur).
// The rotation depends on i, so the key up-projection cannot move onto the query: each page's keys
// are rebuilt by an MMA.  Values carry no rotation and stay in latent space.
//
// Units are (sequence, head) pairs; their pages, in unit order, are cut into equal ranges, one per
// CTA (lla_units.cuh), and a CTA takes its range as runs (its part of one unit).  Per CTA, 15 warps:
//   warp 0       producer: per run, W_up,t^K of the run's head into the A slot once the previous
//                run's key products have read it (TMA boxes of 8 columns x 128 rows, the
//                no-swizzle K-major operand layout; the columns past r_k read as zero); per page,
//                the K-plane by one bulk copy and the V-plane by TMA boxes with 128-byte swizzle
//   warp 1       key issuer and TMEM owner: Khat^T (128 x 64) = W_up,t^K C_k^T per page into one of
//                four 64-column accumulators (lane = key dimension, column = token)
//   warp 2       value issuer: O^T (r_v x 16) += C_v^T P^T, with p as three bf16 parts (rows 0-2
//                of P^T, 24 significant bits); M = 128 latent rows per chunk, M = 64 for a last
//                chunk of at most 64 rows (one V box fewer per stage)
//   warps 3-6    rotation group 0 (even pages of the CTA), warps 7-10 group 1 (odd pages): lane m
//                of a warp's TMEM quarter multiplies (khat_m,i + mu_m) by element m of
//                rot(q, P - p_i), a sinusoid in i that starts from an exact phase per page (64-bit
//                fixed-point turns) and steps through the tokens by a second-order recurrence, and
//                the warp sums its 32 dimensions per token through a TMEM transpose and shuffles
//   warps 11-14  softmax: the four quarter sums of each token, the online softmax with a lazily
//                rescaled O^T, P^T; per run, q and mu^K for the rotation groups, and the partial
//                (O^T, maximum, sum) to the run's workspace slot
// rope_finish_kernel: per (head, up to 8 sequences), merges the runs of each unit, zeroes their
// workspace slots, adds the pass-1 current token (its score q . k_cur: both sit at position P) and
// applies W_up,t^V.  Two launches on the caller's stream, chained by programmatic dependent launch.
// Storage bf16, d = 128.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>

#include "lla_device.cuh"
#include "lla_internal.h"
#include "lla_tcgen05.cuh"
#include "lla_tmap.h"
#include "lla_units.cuh"

namespace lla {
namespace {

constexpr int kPT = 64;            // tokens per page
constexpr int kD = 128;            // head width
constexpr int kPairs = kD / 2;
constexpr int kNO = 16;            // O^T columns (p parts in rows 0-2 of P^T, the rest zero)
constexpr int kPParts = 3;
constexpr int kNAcc = 4;           // key accumulators
constexpr int kNRed = 4;           // partial-score slots
constexpr int kMaxSt = 6;
constexpr int kThreads = 480;
constexpr int kWKey = 1, kWVal = 2, kWRot = 3, kWSmx = 11;
constexpr int kBarSmx = 2;         // named barrier of the softmax warps
constexpr float kRescaleLog2 = 8.f;
constexpr int kSmemCap = 227 * 1024;
constexpr int kFinishSeqs = 8;
constexpr int kMaxGrid = 1024;

template <int RK, int RV>
struct ZR {
    static constexpr int RKX = (RK + 15) / 16 * 16;     // key contraction, zero-padded
    static constexpr int NG = RKX / 8;                  // 16-byte granules of a W_up row
    static constexpr int NCH = (RV + 127) / 128;        // 128-row chunks of O^T
    // a last chunk of at most 64 latent rows is one box and an M = 64 product
    static constexpr bool HALF = RV % 128 != 0 && RV % 128 <= 64;
    static constexpr int NBOX = (RV + 63) / 64;         // TMA boxes a V-plane loads
    static constexpr int BOX = kPT * 128;
    static constexpr int KPLANE = kPT * RK * 2;         // bytes of a K-plane copy
    static constexpr int KPAGE = kPT * RKX * 2;         // K stage: the copy, then zero granules
    static constexpr int VPAGE = (HALF ? 2 * NCH - 1 : 2 * NCH) * BOX;
    static constexpr int VBYTES = NBOX * BOX;
    static constexpr int ASLOT = 128 * RKX * 2;         // granule g of W_up row m at g*2048 + m*16
    static constexpr int PBUF = kPT * kNO * 2;
    static constexpr int RED = kNRed * 4 * kPT * 4;     // [slot][quarter][token] partial scores
    static constexpr int QSLOT = (2 * kD + 4) * 4;      // q (scaled), mu^K, query position
    static constexpr int MISC = 64 * 4;                 // softmax maxima and sums
    static constexpr int PREF = (LLA_MAX_BATCH + 1 + 3) / 4 * 16;  // page prefix of the sequences
    static constexpr int NBAR = 56;
    static constexpr int FIXED = ASLOT + 2 * PBUF + RED + 2 * QSLOT + MISC + PREF + NBAR * 8;
    static constexpr int ST0 = (kSmemCap - 1024 - FIXED) / (KPAGE + VPAGE);
    static constexpr int ST = ST0 > kMaxSt ? kMaxSt : ST0;
    static constexpr int oV = 0;
    static constexpr int oK = oV + ST * VPAGE;
    static constexpr int oA = oK + ST * KPAGE;
    static constexpr int oP = oA + ASLOT;
    static constexpr int oRed = oP + 2 * PBUF;
    static constexpr int oQ = oRed + RED;
    static constexpr int oMisc = oQ + 2 * QSLOT;
    static constexpr int oPref = oMisc + MISC;
    static constexpr int oBar = oPref + PREF;
    static constexpr int SMEM = 1024 + oBar + NBAR * 8;
    static constexpr uint32_t TM_O = kNAcc * 64, TM_COLS = 512;
    static constexpr uint32_t IDESC_K = umma_idesc_bf16(128, 64, 0, 0);
    static constexpr uint32_t IDESC_O = umma_idesc_bf16(128, kNO, 1, 0);
    static constexpr uint32_t IDESC_O64 = umma_idesc_bf16(64, kNO, 1, 0);
    // a run partial: O^T ([RV]), the run maximum at RV and its sum at RV + 16
    static constexpr int PSTRIDE = RV + 32;
    static constexpr int PO_M = RV, PO_L = RV + 16;
    static_assert(RK % 8 == 0 && RV % 8 == 0 && NCH <= 2, "ranks in 16-byte granules");
    static_assert(ST >= 2, "pipeline depth");
    static_assert(SMEM <= kSmemCap, "shared memory");
    static_assert(oA % 128 == 0 && oP % 16 == 0 && oBar % 8 == 0, "alignment");
    static_assert(TM_O + NCH * kNO <= TM_COLS, "TMEM columns");
};

// barrier indices
enum {
    bKfull = 0 /* [6] */, bKempty = 6, bVfull = 12, bVempty = 18, bAfull = 24, bAfree = 26,
    bTfull = 28 /* [4] */, bTfree = 32, bSfull = 36 /* [4] */, bSfree = 40, bPfull = 44 /* [2] */,
    bPfree = 46, bOfree = 48, bQready = 49 /* [2] */, bQfree = 51, bAbort = 53, bTslot = 54
};

struct RTParams {
    int B, H, T, loop, io_bf16, pass1, max_ctx, max_blocks, pairing;
    float scale_log2;
    const char *pool;
    int64_t num_blocks, page_bytes;
    const int32_t *block_table, *context_lens;
    const void *q;          // [B][H][d]
    const float *mu_k;      // [H][T*d] or NULL
    float *part;            // [B H + grid][PSTRIDE]: run (unit u, CTA c) at slot u + c
    unsigned *err;
    unsigned long long phi[kPairs];
    float c1[kPairs], s1[kPairs], c32[kPairs], s32[kPairs], s2[kPairs], h2[kPairs];
};

struct RFParams {
    int B, H, T, loop, io_bf16, grid, spb, max_ctx, max_blocks, pass1;
    float scale_log2;
    const int32_t *context_lens;
    const void *w_up_v;     // [H][T][d][r_v] bf16
    const float *mu_v;      // [H][T*d] or NULL
    const void *q, *cur_k, *cur_v;
    void *out;
    float *part;
};

// PB[b] = pages of the sequences before b (PB[B]: all), block-wide; an invalid length counts as
// an empty sequence (flagged when `flag`, with an empty pass-2 sequence).
__device__ void seq_prefix(const int32_t *lens, int B, int max_ctx, int max_blocks, int pass1, bool flag,
                           unsigned *err, int *PB) {
    __shared__ int wsum[32];
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, nt = blockDim.x;
    const int per = (B + nt - 1) / nt;
    const int limit = min(max_ctx, max_blocks * kPT);
    auto pages = [&](int b, bool f) {
        const int L = lens[b];
        if (L < 0 || L > limit) {
            if (f) atomicOr(err, LLA_DEVERR_CONTEXT);
            return 0;
        }
        if (f && !pass1 && L == 0) atomicOr(err, LLA_DEVERR_EMPTY_PASS2);
        return (L + kPT - 1) / kPT;
    };
    int tot = 0;
    for (int b = tid * per; b < min(B, (tid + 1) * per); ++b) tot += pages(b, flag);
    int x = tot;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) wsum[warp] = x;
    __syncthreads();
    int pre = 0;
    for (int w = 0; w < warp; ++w) pre += wsum[w];
    int ex = pre + x - tot;
    for (int b = tid * per; b < min(B, (tid + 1) * per); ++b) {
        PB[b] = ex;
        ex += pages(b, false);
    }
    if (tid == nt - 1) PB[B] = pre + x;
    __syncthreads();
}

// The runs of a CTA holding global pages [g0, g1): unit u = b H + h owns the pages
// [H PB[b] + h P_b, + P_b) (P_b: the pages of sequence b).
struct Runs {
    const int *PB;
    int H, B, g0, g1, u;
    __device__ Runs(const int *pb, int h, int b, int lo, int hi) : PB(pb), H(h), B(b), g0(lo), g1(hi), u(b * h) {
        if (g0 < g1) {
            int lo2 = 0, hi2 = B - 1;  // the last sequence whose first page is at or before g0
            while (lo2 < hi2) {
                const int mid = (lo2 + hi2 + 1) >> 1;
                if (H * PB[mid] <= g0) lo2 = mid;
                else hi2 = mid - 1;
            }
            const int P = PB[lo2 + 1] - PB[lo2];
            u = lo2 * H + (P > 0 ? (g0 - H * PB[lo2]) / P : 0);
        }
    }
    // the next run: sequence b, head h, pages [pa, pe) of the unit's own numbering
    __device__ bool next(int &b, int &h, int &pa, int &pe) {
        while (u < B * H) {
            const int bb = u / H, hh = u - bb * H;
            const int P = PB[bb + 1] - PB[bb];
            const int s0 = H * PB[bb] + hh * P;
            if (s0 >= g1) return false;
            ++u;
            const int a = max(g0, s0) - s0, e = min(g1, s0 + P) - s0;
            if (e > a) {
                b = bb;
                h = hh;
                pa = a;
                pe = e;
                return true;
            }
        }
        return false;
    }
};

template <int RK, int RV>
__global__ void __launch_bounds__(kThreads, 1)
    rope_tc_kernel(const __grid_constant__ CUtensorMap tv, const __grid_constant__ CUtensorMap tw,
                   const __grid_constant__ RTParams p) {
    using Z = ZR<RK, RV>;
    extern __shared__ __align__(1024) char sm_raw[];
    char *sm = reinterpret_cast<char *>((reinterpret_cast<uintptr_t>(sm_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    uint64_t *bar = reinterpret_cast<uint64_t *>(sm + Z::oBar);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(bar + bAbort);
    uint32_t *tslot = reinterpret_cast<uint32_t *>(bar + bTslot);
    float *red = reinterpret_cast<float *>(sm + Z::oRed);
    float *misc = reinterpret_cast<float *>(sm + Z::oMisc);  // [2][4] maxima, [4] sums
    int *PB = reinterpret_cast<int *>(sm + Z::oPref);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int G = gridDim.x, c = blockIdx.x;

    if (tid == 0) {
        for (int s = 0; s < Z::ST; ++s) {
            mbar_init(&bar[bKfull + s], 1);
            mbar_init(&bar[bKempty + s], 1);
            mbar_init(&bar[bVfull + s], 1);
            mbar_init(&bar[bVempty + s], 1);
        }
        mbar_init(&bar[bAfull], 1);
        mbar_init(&bar[bAfree], 1);
        for (int s = 0; s < 2; ++s) {
            mbar_init(&bar[bPfull + s], 128);
            mbar_init(&bar[bPfree + s], 1);
            mbar_init(&bar[bQready + s], 128);
            mbar_init(&bar[bQfree + s], 256);
        }
        for (int s = 0; s < kNAcc; ++s) {
            mbar_init(&bar[bTfull + s], 1);
            mbar_init(&bar[bTfree + s], 4);
        }
        for (int s = 0; s < kNRed; ++s) {
            mbar_init(&bar[bSfull + s], 128);
            mbar_init(&bar[bSfree + s], 128);
        }
        mbar_init(&bar[bOfree], 128);
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == kWKey) tmem_alloc(tslot, Z::TM_COLS);
    // operand bytes that no copy writes stay zero: the V boxes past r_v of a last chunk, the K
    // granules past r_k, and the P^T rows past the three p parts
    if constexpr (Z::VPAGE > Z::VBYTES) {
        for (int s = 0; s < Z::ST; ++s)
            for (int a = Z::NBOX; a < Z::VPAGE / Z::BOX; ++a)
                for (int i = tid; i < Z::BOX / 16; i += kThreads)
                    reinterpret_cast<uint4 *>(sm + Z::oV + s * Z::VPAGE + a * Z::BOX)[i] = make_uint4(0, 0, 0, 0);
    }
    if constexpr (Z::KPAGE > Z::KPLANE) {
        for (int s = 0; s < Z::ST; ++s)
            for (int i = tid; i < (Z::KPAGE - Z::KPLANE) / 16; i += kThreads)
                reinterpret_cast<uint4 *>(sm + Z::oK + s * Z::KPAGE + Z::KPLANE)[i] = make_uint4(0, 0, 0, 0);
    }
    for (int i = tid; i < 2 * Z::PBUF / 16; i += kThreads)
        reinterpret_cast<uint4 *>(sm + Z::oP)[i] = make_uint4(0, 0, 0, 0);
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tslot;
    pdl_wait();  // inputs may come from the previous kernel; the workspace is free after it
    seq_prefix(p.context_lens, p.B, p.max_ctx, p.max_blocks, p.pass1, c == 0, p.err, PB);
    const int NP = p.H * PB[p.B];
    const int g0 = page_lo(c, NP, G), g1 = page_lo(c + 1, NP, G);
    Runs runs(PB, p.H, p.B, g0, g1);
    int rb, rh, pa, pe;

    if (warp == 0) {
        // ------------------------------------------------------------------------- producer
        if (lane == 0) {
            // after a failed wait (or once the abort flag is up) no further copy is issued; the
            // last rounds issued on each barrier are awaited below
            const uint64_t pol = policy_evict_first();
            int itk = 0, itv = 0, ita = 0;
            bool stop = false;
            while (!stop && runs.next(rb, rh, pa, pe)) {
                // W_up,t^K of head rh ([H][T][d][r_k]) once the previous run's key products have
                // read the slot (the key accumulators keep the rotation groups busy meanwhile)
                if (!mbar_wait(&bar[bAfree], (ita & 1) ^ 1u, abort_flag, p.err) || *abort_flag) break;
                mbar_arrive_expect_tx(&bar[bAfull], Z::ASLOT);
                const int wrow = rh * p.T + p.loop;
#pragma unroll 1
                for (int g = 0; g < Z::NG; ++g) tma_load_3d(sm + Z::oA + g * 2048, &tw, 8 * g, 0, wrow, &bar[bAfull]);
                ++ita;
                const int32_t *bt = p.block_table + static_cast<int64_t>(rb) * p.max_blocks;
                for (int pg = pa; pg < pe; ++pg) {
                    const int st = itk % Z::ST;
                    const uint32_t ph = (itk / Z::ST) & 1;
                    int32_t blk = bt[pg];
                    if (blk < 0 || blk >= p.num_blocks) {
                        atomicOr(p.err, LLA_DEVERR_BLOCK_ID);
                        blk = 0;
                    }
                    const int64_t page = static_cast<int64_t>(blk) * p.H + rh;
                    if (!mbar_wait(&bar[bKempty + st], ph ^ 1u, abort_flag, p.err) || *abort_flag) {
                        stop = true;
                        break;
                    }
                    mbar_arrive_expect_tx(&bar[bKfull + st], Z::KPLANE);
                    bulk_g2s(sm + Z::oK + st * Z::KPAGE, p.pool + page * p.page_bytes, Z::KPLANE, &bar[bKfull + st], pol);
                    ++itk;
                    if (!mbar_wait(&bar[bVempty + st], ph ^ 1u, abort_flag, p.err) || *abort_flag) {
                        stop = true;
                        break;
                    }
                    mbar_arrive_expect_tx(&bar[bVfull + st], Z::VBYTES);
                    char *vs = sm + Z::oV + st * Z::VPAGE;
#pragma unroll
                    for (int a = 0; a < Z::NBOX; ++a)
                        tma_load_3d(vs + a * Z::BOX, &tv, a * 64, 0, static_cast<int>(page), &bar[bVfull + st]);
                    ++itv;
                }
            }
            // every copy has landed before the CTA can exit, even after an abort
            volatile int never = 0;
            for (int j = max(0, itk - Z::ST); j < itk; ++j)
                mbar_wait(&bar[bKfull + j % Z::ST], (j / Z::ST) & 1, &never, p.err);
            for (int j = max(0, itv - Z::ST); j < itv; ++j)
                mbar_wait(&bar[bVfull + j % Z::ST], (j / Z::ST) & 1, &never, p.err);
            if (ita > 0) mbar_wait(&bar[bAfull], (ita - 1) & 1, &never, p.err);
        }
        __syncwarp();
    } else if (warp == kWKey) {
        // --------------------------------------------------------------------- key issuer
        if (lane == 0) {
            const uint32_t base = smem_addr(sm);
            int it = 0, r = 0;
            const uint64_t da = umma_desc(base + Z::oA, 2048, 128);
            while (runs.next(rb, rh, pa, pe)) {
                mbar_wait(&bar[bAfull], r & 1, abort_flag, p.err);
                for (int k = pa; k < pe; ++k, ++it) {
                    const int b = it % kNAcc, st = it % Z::ST;
                    mbar_wait(&bar[bKfull + st], (it / Z::ST) & 1, abort_flag, p.err);
                    if (it >= kNAcc) mbar_wait(&bar[bTfree + b], ((it / kNAcc) - 1) & 1, abort_flag, p.err);
                    tc_fence_after();
                    const uint64_t dk = umma_desc(base + Z::oK + st * Z::KPAGE, kPT * 16, 128);
#pragma unroll
                    for (int ks = 0; ks < Z::RKX / 16; ++ks)
                        umma_bf16(tmem + b * 64, da + ks * (4096 >> 4), dk + ks * (2048 >> 4), Z::IDESC_K, ks > 0);
                    umma_commit(&bar[bTfull + b]);
                    umma_commit(&bar[bKempty + st]);  // the K-plane has been read
                }
                umma_commit(&bar[bAfree]);
                ++r;
            }
            // every key product has completed before TMEM is released, even after an abort (when
            // the rotation groups stop waiting for them): the last commit on each accumulator
            volatile int never = 0;
            for (int j = max(0, it - kNAcc); j < it; ++j)
                mbar_wait(&bar[bTfull + j % kNAcc], (j / kNAcc) & 1, &never, p.err);
        }
        __syncwarp();
    } else if (warp == kWVal) {
        // ------------------------------------------------------------------- value issuer
        if (lane == 0) {
            const uint32_t base = smem_addr(sm);
            const uint64_t dp0 = umma_desc(base + Z::oP, kNO * 16, 128);
            const uint64_t dv0 = umma_desc_sw128_mn(base + Z::oV, Z::BOX);
            int it = 0, r = 0;
            while (runs.next(rb, rh, pa, pe)) {
                for (int k = pa; k < pe; ++k, ++it) {
                    // O^T += C_v^T P^T for page it (the first page of run r zeroes O^T, once the
                    // softmax warps have read run r - 1's)
                    const int s = it & 1, st = it % Z::ST;
                    mbar_wait(&bar[bPfull + s], (it >> 1) & 1, abort_flag, p.err);
                    mbar_wait(&bar[bVfull + st], (it / Z::ST) & 1, abort_flag, p.err);
                    if (k == pa && r > 0) mbar_wait(&bar[bOfree], (r - 1) & 1, abort_flag, p.err);
                    tc_fence_after();
                    const uint64_t dv = dv0 + static_cast<uint64_t>((st * Z::VPAGE) >> 4);
                    const uint64_t dp = dp0 + static_cast<uint64_t>((s * Z::PBUF) >> 4);
#pragma unroll
                    for (int ch = 0; ch < Z::NCH; ++ch)
#pragma unroll
                        for (int ks = 0; ks < kPT / 16; ++ks)
                            umma_bf16(tmem + Z::TM_O + ch * kNO, dv + ((ch * 2 * Z::BOX + ks * 2048) >> 4),
                                      dp + ks * ((2 * kNO * 16) >> 4),
                                      Z::HALF && ch == Z::NCH - 1 ? Z::IDESC_O64 : Z::IDESC_O, k > pa || ks > 0);
                    umma_commit(&bar[bVempty + st]);
                    umma_commit(&bar[bPfree + s]);  // also: O^T holds pages up to it
                }
                ++r;
            }
            // every product has completed before TMEM is released, even after an abort
            if (it > 0) {
                volatile int never = 0;
                mbar_wait(&bar[bPfree + ((it - 1) & 1)], ((it - 1) >> 1) & 1, &never, p.err);
            }
        }
        __syncwarp();
    } else if (warp < kWSmx) {
        // ---------------------------------------------------------------- rotation groups
        const int grp = (warp - kWRot) >> 2, quarter = warp & 3;
        const int m = 32 * quarter + lane;  // key dimension = TMEM lane
        const int j = p.pairing ? (m >> 1) : (m & (kPairs - 1));
        const bool upper = p.pairing ? (m & 1) : (m >= kPairs);
        const int ia = p.pairing ? 2 * j : j, ib = p.pairing ? 2 * j + 1 : j + kPairs;
        const unsigned long long phi = p.phi[j];
        const float c1 = p.c1[j], s1 = p.s1[j], c32 = p.c32[j], s32 = p.s32[j];
        const float s2 = p.s2[j], h2 = p.h2[j];
        const float2 nlam = make_float2(-2.f * h2, -2.f * h2);  // -(2 - 2 cos 2 theta_j)
        const uint32_t tlane = tmem + (static_cast<uint32_t>(32 * quarter) << 16);
        int it = 0, r = 0;
        while (runs.next(rb, rh, pa, pe)) {
            const int qs = r & 1;
            mbar_wait(&bar[bQready + qs], (r >> 1) & 1, abort_flag, p.err);
            const float *qv = reinterpret_cast<const float *>(sm + Z::oQ + qs * Z::QSLOT);
            // element m of rot(q, Delta) = Re(G e^{i Delta theta_j}) (q scaled to log2 units)
            const float qa = qv[ia], qb = qv[ib];
            const float Gr = upper ? qb : qa, Gi = upper ? -qa : qb;
            const float mu = qv[kD + m];
            const float2 mu2 = make_float2(mu, mu);
            const int P = reinterpret_cast<const int *>(qv + 2 * kD)[0];  // the query's position
            for (int k = pa; k < pe; ++k, ++it) {
                if ((it & 1) != grp) continue;
                // exact phase of the page's first token: Delta0 theta_j in turns, mod 1
                const int delta0 = P - k * kPT;  // >= 0: the page holds a cached token
                const unsigned long long turns = static_cast<unsigned long long>(delta0) * phi;
                const float tf = __uint2float_rn(static_cast<uint32_t>(turns >> 32)) * 2.3283064365386963e-10f;
                float sa, ca;
                sincospif(2.f * tf, &sa, &ca);
                const float zr = Gr * ca - Gi * sa, zi = Gr * sa + Gi * ca;
                // x_i = Re(z e^{-i i theta}) for the page's tokens i, in four chains that step two
                // tokens at a time (even and odd tokens of each half, packed in pairs):
                // dd = x_i - x_{i-2};  dd' = dd - (2 - 2 cos 2 theta) x;  x' = x + dd'
                float2 X[2], DD[2];
#pragma unroll
                for (int hv = 0; hv < 2; ++hv) {
                    const float er = hv ? fmaf(zr, c32, zi * s32) : zr;
                    const float ei = hv ? fmaf(zi, c32, -zr * s32) : zi;
                    const float orr = fmaf(er, c1, ei * s1), oi = fmaf(ei, c1, -er * s1);
                    X[hv] = make_float2(er, orr);
                    DD[hv] = make_float2(fmaf(er, h2, ei * s2), fmaf(orr, h2, oi * s2));
                }
                const int b = it % kNAcc;
                uint32_t v0[32], v1[32];  // this dimension of tokens 0..31 and 32..63
                mbar_wait(&bar[bTfull + b], (it / kNAcc) & 1, abort_flag, p.err);
                tc_fence_after();
                const uint32_t tcol = tlane + b * 64;
                tmem_ld32_nowait(tcol, v0);
                tmem_ld32_nowait(tcol + 32, v1);
                tmem_wait_ld(v0);
                tmem_wait_ld(v1);
#pragma unroll
                for (int t = 0; t < 16; ++t) {
                    float2 a0 = make_float2(__uint_as_float(v0[2 * t]), __uint_as_float(v0[2 * t + 1]));
                    float2 a1 = make_float2(__uint_as_float(v1[2 * t]), __uint_as_float(v1[2 * t + 1]));
                    a0 = __fmul2_rn(__fadd2_rn(a0, mu2), X[0]);
                    a1 = __fmul2_rn(__fadd2_rn(a1, mu2), X[1]);
                    v0[2 * t] = __float_as_uint(a0.x);
                    v0[2 * t + 1] = __float_as_uint(a0.y);
                    v1[2 * t] = __float_as_uint(a1.x);
                    v1[2 * t + 1] = __float_as_uint(a1.y);
                    DD[0] = __ffma2_rn(nlam, X[0], DD[0]);
                    DD[1] = __ffma2_rn(nlam, X[1], DD[1]);
                    X[0] = __fadd2_rn(X[0], DD[0]);
                    X[1] = __fadd2_rn(X[1], DD[1]);
                }
                // sum over the warp's 32 dimensions of each token: the terms go back to TMEM and
                // return in the 16x256b layout (4 dimensions x 16 tokens per thread), are summed
                // over the 4 dimensions, then over the 8 threads of each token group by shuffles
                tmem_st32u_nowait(tcol, v0);
                tmem_st32u_nowait(tcol + 32, v1);
                tmem_wait_st();
                tmem_ld16x256_x8_nowait(tcol, v0);
                tmem_ld16x256_x8_nowait(tcol + (static_cast<uint32_t>(16) << 16), v1);
                tmem_wait_ld(v0);
                tmem_wait_ld(v1);
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&bar[bTfree + b]);  // the accumulator may take page it + 4
                float S[16];  // S[2k + e]: token 8k + 2(lane % 4) + e, summed over 4 dimensions
#pragma unroll
                for (int k8 = 0; k8 < 8; ++k8) {
                    const float2 x0 = __fadd2_rn(
                        make_float2(__uint_as_float(v0[4 * k8]), __uint_as_float(v0[4 * k8 + 1])),
                        make_float2(__uint_as_float(v0[4 * k8 + 2]), __uint_as_float(v0[4 * k8 + 3])));
                    const float2 x1 = __fadd2_rn(
                        make_float2(__uint_as_float(v1[4 * k8]), __uint_as_float(v1[4 * k8 + 1])),
                        make_float2(__uint_as_float(v1[4 * k8 + 2]), __uint_as_float(v1[4 * k8 + 3])));
                    const float2 sum = __fadd2_rn(x0, x1);
                    S[2 * k8] = sum.x;
                    S[2 * k8 + 1] = sum.y;
                }
                // lanes differing in bits 4, 3, 2 hold the same tokens: halve the token set per
                // level, keeping the half that the lane's bit selects
#pragma unroll
                for (int lv = 0; lv < 3; ++lv) {
                    const int half = 8 >> lv, bit = 16 >> lv;
                    const bool up = lane & bit;
#pragma unroll
                    for (int i = 0; i < half; ++i) {
                        const float lo = S[i], hi = S[i + half];
                        const float keep = up ? hi : lo, send = up ? lo : hi;
                        S[i] = keep + __shfl_xor_sync(0xffffffffu, send, bit);
                    }
                }
                // this lane holds the warp's sums for tokens 2 lane and 2 lane + 1
                const int slot = it % kNRed;
                mbar_wait(&bar[bSfree + slot], ((it / kNRed) & 1) ^ 1u, abort_flag, p.err);
                *reinterpret_cast<float2 *>(red + (slot * 4 + quarter) * kPT + 2 * lane) = make_float2(S[0], S[1]);
                mbar_arrive(&bar[bSfull + slot]);
            }
            mbar_arrive(&bar[bQfree + qs]);
            ++r;
        }
        tc_fence_before();
    } else {
        // ------------------------------------------------------------------ softmax warps
        const int st_tid = tid - kWSmx * 32, quarter = warp & 3;
        const uint32_t tlo = tmem + (static_cast<uint32_t>(32 * quarter) << 16) + Z::TM_O;
        const int t = st_tid;  // the token of this thread (st_tid < 64)
        // q (scaled into the exp2 domain), mu^K and the query's position of a run, for the
        // rotation groups, staged one run ahead so that they never wait for these loads
        auto stage = [&](int qs, int b_, int h_) {
            float *qv = reinterpret_cast<float *>(sm + Z::oQ + qs * Z::QSLOT);
            const int64_t row = (static_cast<int64_t>(b_) * p.H + h_) * kD;
            qv[st_tid] = load_elem(p.q, row + st_tid, p.io_bf16) * p.scale_log2;
            qv[kD + st_tid] = p.mu_k ? p.mu_k[(static_cast<int64_t>(h_) * p.T + p.loop) * kD + st_tid] : 0.f;
            if (st_tid == 0) {
                const int Lq = p.context_lens[b_];  // the run has pages, so Lq >= 1
                reinterpret_cast<int *>(qv + 2 * kD)[0] = p.pass1 ? Lq : Lq - 1;
            }
            mbar_arrive(&bar[bQready + qs]);
        };
        Runs ahead = runs;  // one run ahead of `runs`
        int ab, ah, apa, ape;
        if (ahead.next(ab, ah, apa, ape)) stage(0, ab, ah);
        int it = 0, r = 0;
        while (runs.next(rb, rh, pa, pe)) {
            const int L = p.context_lens[rb];  // valid: the unit has pages
            if (ahead.next(ab, ah, apa, ape)) {
                // run r + 1 into the slot of run r - 1, once both rotation groups have left it
                const int qs1 = (r + 1) & 1;
                if (r >= 1) mbar_wait(&bar[bQfree + qs1], ((r - 1) >> 1) & 1, abort_flag, p.err);
                stage(qs1, ab, ah);
            }
            float m_run = -INFINITY, acc = 0.f;
            const int nps = pe - pa;
            for (int k = 0; k < nps; ++k, ++it) {
                const int slot = it % kNRed, s = it & 1, st = it % Z::ST;
                const int tok0 = (pa + k) * kPT;
                mbar_wait(&bar[bSfull + slot], (it / kNRed) & 1, abort_flag, p.err);
                float x = -INFINITY;
                if (t < kPT) {
                    const float *rs = red + slot * 4 * kPT + t;
                    const float sc = (rs[0] + rs[kPT]) + (rs[2 * kPT] + rs[3 * kPT]);
                    x = tok0 + t < L ? sc : -INFINITY;
                }
                mbar_arrive(&bar[bSfree + slot]);  // the partial scores are read
                const float mx = warp_max(x);
                if (lane == 0) misc[s * 4 + (warp - kWSmx)] = mx;
                named_bar_sync(kBarSmx, 128);
                const float pm = fmaxf(fmaxf(misc[s * 4], misc[s * 4 + 1]), fmaxf(misc[s * 4 + 2], misc[s * 4 + 3]));
                const float mn = fmaxf(m_run, pm);
                if (mn > m_run + kRescaleLog2) {  // also the first page; uniform over the warps
                    const float f = ex2_approx(m_run - mn);
                    acc *= f;
                    m_run = mn;
                    if (k > 0) {
                        // O^T holds pages up to it - 1 of this run: scale its p columns by f
                        mbar_wait(&bar[bPfree + ((it - 1) & 1)], ((it - 1) >> 1) & 1, abort_flag, p.err);
                        tc_fence_after();
#pragma unroll
                        for (int ch = 0; ch < Z::NCH; ++ch) {
                            float o[kNO];
                            tmem_ld16(tlo + ch * kNO, o);
#pragma unroll
                            for (int e = 0; e < kPParts; ++e) o[e] *= f;
                            tmem_st16(tlo + ch * kNO, o);
                        }
                    }
                }
                const float pv = t < kPT ? ex2_approx(x - m_run) : 0.f;
                acc += pv;
                if (it >= 2) mbar_wait(&bar[bPfree + s], ((it - 2) >> 1) & 1, abort_flag, p.err);
                if (t < kPT) {
                    // P^T as a K-major operand: row e = bf16 part e of p, tokens 8g .. 8g + 7 at
                    // g*256 + row*16
                    char *pp = sm + Z::oP + s * Z::PBUF + (t >> 3) * (kNO * 16) + (t & 7) * 2;
                    float rest = pv;
#pragma unroll
                    for (int e = 0; e < kPParts; ++e) {
                        const __nv_bfloat16 part = __float2bfloat16_rn(rest);
                        rest -= __bfloat162float(part);
                        *reinterpret_cast<uint16_t *>(pp + e * 16) = __bfloat16_as_ushort(part);
                    }
                }
                if (k == nps - 1 && tok0 + kPT > L) {
                    // V rows past the sequence hold no latents: zero them (0 * NaN would poison O)
                    mbar_wait(&bar[bVfull + st], (it / Z::ST) & 1, abort_flag, p.err);
                    char *vs = sm + Z::oV + st * Z::VPAGE;
                    const int nv = L - tok0;
                    const int nz = (kPT - nv) * Z::NBOX * 8;
                    for (int w = st_tid; w < nz; w += 128) {
                        const int cc = w & 7, r2 = w >> 3;
                        const int a = r2 % Z::NBOX, row = nv + r2 / Z::NBOX;
                        *reinterpret_cast<uint4 *>(vs + a * Z::BOX + row * 128 + cc * 16) = make_uint4(0, 0, 0, 0);
                    }
                }
                fence_proxy_async_smem();
                tc_fence_before();
                mbar_arrive(&bar[bPfull + s]);
            }
            // the run's partial: O^T (complete once the last page's product has released its P
            // buffer), the run maximum and sum
            mbar_wait(&bar[bPfree + ((it - 1) & 1)], ((it - 1) >> 1) & 1, abort_flag, p.err);
            tc_fence_after();
            const float ls = warp_sum(acc);
            if (lane == 0) misc[8 + (warp - kWSmx)] = ls;
            float *dst = p.part + (static_cast<int64_t>(rb) * p.H + rh + c) * Z::PSTRIDE;
#pragma unroll
            for (int ch = 0; ch < Z::NCH; ++ch) {
                float o[kNO];
                tmem_ld16(tlo + ch * kNO, o);
                // an M = 128 chunk: row 32 quarter + lane; an M = 64 one: row 16 quarter + lane
                // in lanes 0-15 of each quarter
                const bool half = Z::HALF && ch == Z::NCH - 1;
                const int jj = ch * 128 + (half ? (lane < 16 ? 16 * quarter + lane : RV) : 32 * quarter + lane);
                if (jj < RV) dst[jj] = (o[0] + o[1]) + o[2];
            }
            tc_fence_before();
            mbar_arrive(&bar[bOfree]);
            named_bar_sync(kBarSmx, 128);  // the run sums are visible
            if (st_tid == 0) {
                dst[Z::PO_M] = m_run;
                dst[Z::PO_L] = (misc[8] + misc[9]) + (misc[10] + misc[11]);
            }
            named_bar_sync(kBarSmx, 128);  // misc is free for the next run
            ++r;
        }
    }
    pdl_trigger();
    tc_fence_before();
    __syncthreads();
    if (warp == kWKey) {
        tc_fence_after();
        tmem_dealloc(tmem, Z::TM_COLS);
    }
}

// Grid (H, ceil(B / spb)), 128 threads (thread e = output element e of head h).  spb (at most 8)
// sequences share one pass over W_up,t^V of head h.  Everything that is an input of the call (the
// weights, the context lengths, q, k_cur and v_cur) is read before the wait on the attention
// kernel, which launches this one ahead of its end.  The runs of a unit are merged by one warp, or
// by two or four that split its columns when the CTA has fewer than three units; the merged slots
// are then zeroed (each slot belongs to one unit, so to this CTA alone).
template <int RV>
__global__ void __launch_bounds__(128, 1) rope_finish_kernel(const RFParams p) {
    constexpr int PS = RV + 32, PO_M = RV, PO_L = RV + 16;
    constexpr bool kPre = RV <= 160;
    constexpr int NW = kPre ? RV / 8 : 1;
    constexpr int NJ = (RV + 31) / 32;
    __shared__ __align__(16) float ob[kFinishSeqs][RV];
    __shared__ float wts[4][kMaxGrid], wls[4][kMaxGrid];  // per warp: run weights and sums
    __shared__ float coef[kFinishSeqs][3], scs[kFinishSeqs];
    __shared__ int PB[LLA_MAX_BATCH + 1];
    const int h = blockIdx.x, b0 = blockIdx.y * p.spb, tid = threadIdx.x;
    const int warp = tid >> 5, lane = tid & 31;
    const int nb = min(p.spb, p.B - b0);
    const int64_t th = static_cast<int64_t>(h) * p.T + p.loop;
    const int e = tid;
    const uint4 *W = reinterpret_cast<const uint4 *>(static_cast<const uint16_t *>(p.w_up_v) + (th * kD + e) * RV);
    uint4 wr[NW];
    if constexpr (kPre) {
#pragma unroll
        for (int j8 = 0; j8 < NW; ++j8) wr[j8] = W[j8];
    }
    const float muv = p.mu_v ? p.mu_v[th * kD + e] : 0.f;
    // the call's own inputs (not outputs of the attention kernel) before the wait on it: the page
    // prefix of the sequences, each unit's current-token score and value element e
    seq_prefix(p.context_lens, p.B, p.max_ctx, p.max_blocks, p.pass1, false, nullptr, PB);
    float cv[kFinishSeqs];
#pragma unroll
    for (int bi = 0; bi < kFinishSeqs; ++bi)
        cv[bi] = p.cur_v && bi < nb ? load_elem(p.cur_v, (static_cast<int64_t>(b0 + bi) * p.H + h) * kD + e, p.io_bf16) : 0.f;
    if (p.cur_k) {
        for (int bi = warp; bi < nb; bi += 4) {
            const int64_t row = (static_cast<int64_t>(b0 + bi) * p.H + h) * kD;
            float qk = 0.f;
#pragma unroll
            for (int i = 0; i < kD / 32; ++i)
                qk = fmaf(load_elem(p.q, row + lane + 32 * i, p.io_bf16), load_elem(p.cur_k, row + lane + 32 * i, p.io_bf16), qk);
            qk = warp_sum(qk);
            if (lane == 0) scs[bi] = qk * p.scale_log2;
        }
    }
    __syncthreads();
    pdl_wait();
    const int NP = p.H * PB[p.B];
    const int G = nb == 1 ? 4 : nb == 2 ? 2 : 1;
    const int grp = warp / G, sub = warp - grp * G;
    float *wt = wts[warp];
    float *wl = wls[warp];
    for (int bi = grp; bi < kFinishSeqs; bi += 4 / G) {
        if (bi >= nb) {
            for (int j = lane + 32 * sub; j < RV; j += 32 * G) ob[bi][j] = 0.f;
            continue;
        }
        const int b = b0 + bi;
        const int64_t u = static_cast<int64_t>(b) * p.H + h;
        const int P = PB[b + 1] - PB[b];
        const int s0 = p.H * PB[b] + h * P, s1 = s0 + P;
        float M = -INFINITY, l = 0.f;
        float acc[NJ];
#pragma unroll
        for (int q = 0; q < NJ; ++q) acc[q] = 0.f;
        if (s1 > s0) {
            const int c0 = cta_of(s0, NP, p.grid), c1 = cta_of(s1 - 1, NP, p.grid);
            const int nr = c1 - c0 + 1;
            const float *pu = p.part + (u + c0) * PS;
            // the run maxima and sums in one round of loads
            float mm = -INFINITY;
            for (int i = lane; i < nr; i += 32) {
                const bool has = page_lo(c0 + i + 1, NP, p.grid) > page_lo(c0 + i, NP, p.grid);
                wt[i] = has ? pu[static_cast<int64_t>(i) * PS + PO_M] : -INFINITY;
                wl[i] = has ? pu[static_cast<int64_t>(i) * PS + PO_L] : 0.f;
                mm = fmaxf(mm, wt[i]);
            }
            M = warp_max(mm);
            float ls = 0.f;
            for (int i = lane; i < nr; i += 32) {
                const float w8 = wt[i] == -INFINITY ? 0.f : ex2_approx(wt[i] - M);
                ls = fmaf(w8, wl[i], ls);
                wt[i] = w8;
            }
            l = warp_sum(ls);
            __syncwarp();
#pragma unroll 4
            for (int i = 0; i < nr; ++i) {
                const float w8 = wt[i];
                if (w8 > 0.f) {
                    const float *pr = pu + static_cast<int64_t>(i) * PS;
#pragma unroll
                    for (int q = 0; q < NJ; ++q) {
                        const int j = lane + 32 * (sub + G * q);
                        if (j < RV) acc[q] = fmaf(w8, pr[j], acc[q]);
                    }
                }
            }
            __syncwarp();
        }
#pragma unroll
        for (int q = 0; q < NJ; ++q) {
            const int j = lane + 32 * (sub + G * q);
            if (j < RV) ob[bi][j] = acc[q];
        }
        if (sub == 0 && lane == 0) {
            const float sc = p.cur_k ? scs[bi] : -INFINITY;
            const float Mx = fmaxf(M, sc);
            const float al = M == -INFINITY ? 0.f : ex2_approx(M - Mx);
            const float pc = p.cur_k ? ex2_approx(sc - Mx) : 0.f;
            const float den = al * l + pc;
            const float inv = den > 0.f ? 1.f / den : 0.f;
            coef[bi][0] = al * inv;
            coef[bi][1] = al * l * inv;
            coef[bi][2] = pc * inv;
        }
    }
    __syncthreads();  // every partial has been read
    float acc[kFinishSeqs];
#pragma unroll
    for (int bi = 0; bi < kFinishSeqs; ++bi) acc[bi] = 0.f;
    auto step = [&](int j8, const uint4 w4) {
        const float2 w0 = bf2_to_f2(w4.x), w1 = bf2_to_f2(w4.y), w2 = bf2_to_f2(w4.z), w3 = bf2_to_f2(w4.w);
#pragma unroll
        for (int bi = 0; bi < kFinishSeqs; ++bi) {
            const float4 o0 = *reinterpret_cast<const float4 *>(&ob[bi][j8 * 8]);
            const float4 o1 = *reinterpret_cast<const float4 *>(&ob[bi][j8 * 8 + 4]);
            float a = acc[bi];
            a = fmaf(w0.x, o0.x, a); a = fmaf(w0.y, o0.y, a); a = fmaf(w1.x, o0.z, a); a = fmaf(w1.y, o0.w, a);
            a = fmaf(w2.x, o1.x, a); a = fmaf(w2.y, o1.y, a); a = fmaf(w3.x, o1.z, a); a = fmaf(w3.y, o1.w, a);
            acc[bi] = a;
        }
    };
    if constexpr (kPre) {
#pragma unroll
        for (int j8 = 0; j8 < NW; ++j8) step(j8, wr[j8]);
    } else {
#pragma unroll 4
        for (int j8 = 0; j8 < RV / 8; ++j8) step(j8, W[j8]);
    }
#pragma unroll
    for (int bi = 0; bi < kFinishSeqs; ++bi) {
        if (bi >= nb) break;
        const int64_t idx = (static_cast<int64_t>(b0 + bi) * p.H + h) * kD + e;
        float v = acc[bi] * coef[bi][0] + coef[bi][1] * muv;
        if (p.cur_v) v = fmaf(coef[bi][2], cv[bi], v);
        store_elem(p.out, idx, v, p.io_bf16);
    }
    // the merged slots return to zero
    for (int bi = 0; bi < nb; ++bi) {
        const int b = b0 + bi;
        const int P = PB[b + 1] - PB[b];
        if (P == 0) continue;
        const int s0 = p.H * PB[b] + h * P;
        const int c0 = cta_of(s0, NP, p.grid), c1 = cta_of(s0 + P - 1, NP, p.grid);
        float *pu = p.part + (static_cast<int64_t>(b) * p.H + h + c0) * PS;
        for (int i = 0; i <= c1 - c0; ++i) {
            if (page_lo(c0 + i + 1, NP, p.grid) <= page_lo(c0 + i, NP, p.grid)) continue;  // no run
            for (int jj = tid; jj < PS; jj += 128) pu[static_cast<int64_t>(i) * PS + jj] = 0.f;
        }
    }
    __syncthreads();
    pdl_trigger();
}

template <int RK, int RV>
lla_status launch_tc(const DecodeArgs &a, const RopeTables &tab, int pairing, cudaStream_t stream) {
    using Z = ZR<RK, RV>;
    lla_status st = LLA_OK;
    unsigned *err = device_error_word(&st);
    if (st != LLA_OK) return st;
    const int grid = num_sms();
    if (grid <= 0 || grid > kMaxGrid) return LLA_ERR_UNSUPPORTED;
    if (static_cast<int64_t>(a.num_blocks) * a.H >= (int64_t(1) << 31)) return LLA_ERR_UNSUPPORTED;
    if (static_cast<int64_t>(a.B) * a.H * ((static_cast<int64_t>(a.max_ctx) + kPT - 1) / kPT) >= (int64_t(1) << 31))
        return LLA_ERR_UNSUPPORTED;  // the units' pages are numbered in 32 bits
    if (a.workspace_bytes < decode_rope_tc_workspace_bytes(RV, a.B, a.H, grid)) return LLA_ERR_WORKSPACE;
    static DeviceOnce configured;
    if (raise_smem_limit(rope_tc_kernel<RK, RV>, Z::SMEM, configured) != LLA_OK) return LLA_ERR_CUDA;
    const int64_t page_bytes = static_cast<int64_t>(head_page_bytes(RK, RV, 2));
    // the V-planes of every head page: [num_blocks * H][64 tokens][r_v] bf16
    CUtensorMap tv, tw;
    {
        const uint64_t dims[3] = {static_cast<uint64_t>(RV), static_cast<uint64_t>(kPT),
                                  static_cast<uint64_t>(a.num_blocks) * a.H};
        const uint64_t strides[2] = {static_cast<uint64_t>(RV) * 2, static_cast<uint64_t>(page_bytes)};
        const uint32_t box[3] = {64, kPT, 1};
        if (!encode_tmap_bf16(&tv, static_cast<const char *>(a.pool) + kPT * RK * 2, 3, dims, strides, box, true))
            return LLA_ERR_CUDA;
    }
    {
        // W_up^K: [H * T][d rows][r_k]; a box is 8 columns of the 128 rows of one (head, loop)
        const uint64_t dims[3] = {static_cast<uint64_t>(RK), static_cast<uint64_t>(kD),
                                  static_cast<uint64_t>(a.H) * a.T};
        const uint64_t strides[2] = {static_cast<uint64_t>(RK) * 2, static_cast<uint64_t>(kD) * RK * 2};
        const uint32_t box[3] = {8, kD, 1};
        if (!encode_tmap_bf16(&tw, a.w_up_k, 3, dims, strides, box, false)) return LLA_ERR_CUDA;
    }
    RTParams rp = {};
    rp.B = a.B; rp.H = a.H; rp.T = a.T; rp.loop = a.loop; rp.io_bf16 = a.io_bf16;
    rp.pass1 = a.cur_k != nullptr; rp.max_ctx = a.max_ctx; rp.max_blocks = a.max_blocks;
    rp.pairing = pairing;
    rp.scale_log2 = a.scale * 1.4426950408889634f;
    rp.pool = static_cast<const char *>(a.pool);
    rp.num_blocks = a.num_blocks; rp.page_bytes = page_bytes;
    rp.block_table = a.block_table; rp.context_lens = a.context_lens;
    rp.q = a.q; rp.mu_k = a.mu_k;
    rp.part = static_cast<float *>(a.workspace);
    rp.err = err;
    for (int j = 0; j < kPairs; ++j) {
        rp.phi[j] = tab.phi[j];
        rp.c1[j] = tab.c1[j]; rp.s1[j] = tab.s1[j]; rp.c32[j] = tab.c32[j]; rp.s32[j] = tab.s32[j];
        rp.s2[j] = tab.s2[j]; rp.h2[j] = tab.h2[j];
    }
    if ((st = launch_ex(rope_tc_kernel<RK, RV>, dim3(grid), kThreads, Z::SMEM, stream, tv, tw, rp)) != LLA_OK)
        return st;
    RFParams fp = {};
    fp.B = a.B; fp.H = a.H; fp.T = a.T; fp.loop = a.loop; fp.io_bf16 = a.io_bf16; fp.grid = grid;
    fp.max_ctx = a.max_ctx; fp.max_blocks = a.max_blocks; fp.pass1 = rp.pass1;
    fp.scale_log2 = rp.scale_log2;
    fp.context_lens = a.context_lens;
    fp.w_up_v = a.w_up_v; fp.mu_v = a.mu_v;
    fp.q = a.q; fp.cur_k = a.cur_k; fp.cur_v = a.cur_v; fp.out = a.out;
    fp.part = rp.part;
    // about two finish CTAs per SM: fewer sequences per CTA for small batches
    const int64_t want = static_cast<int64_t>(a.B) * a.H;
    fp.spb = static_cast<int>(std::min<int64_t>(kFinishSeqs, std::max<int64_t>(1, (want + 2 * grid - 1) / (2 * grid))));
    return launch_ex(rope_finish_kernel<RV>, dim3(a.H, (a.B + fp.spb - 1) / fp.spb), 128, 0, stream, fp);
}

}  // namespace

bool decode_rope_tc_supported(int es, int d, int r_k, int r_v) {
    return es == 2 && d == kD &&
           ((r_k == 96 && r_v == 160) || (r_k == 128 && r_v == 128) || (r_k == 72 && r_v == 120));
}

size_t decode_rope_tc_workspace_bytes(int r_v, int B, int H, int grid) {
    const size_t n = (static_cast<size_t>(B) * H + grid) * (r_v + 32) * sizeof(float);
    return (n + 255) & ~static_cast<size_t>(255);
}

lla_status launch_decode_rope_tc(const DecodeArgs &a, const RopeTables &t, int pairing, cudaStream_t stream) {
    if (a.B == 0) return LLA_OK;
    if (a.r_k == 96 && a.r_v == 160) return launch_tc<96, 160>(a, t, pairing, stream);
    if (a.r_k == 128 && a.r_v == 128) return launch_tc<128, 128>(a, t, pairing, stream);
    if (a.r_k == 72 && a.r_v == 120) return launch_tc<72, 120>(a, t, pairing, stream);
    return LLA_ERR_UNSUPPORTED;
}

}  // namespace lla
