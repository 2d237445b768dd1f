// lla_prefill.cu -- causal pass-2 prefill attention over latents (App. A, two-pass prefill;
// App. J absorbed attention).
//
// For a prompt of L tokens whose latents are all in the cache, query i at loop t attends to
// keys 0..i:
//   q~_i = W_up,t^K^T q_i                       (the constant q_i . mu^K_t cancels in softmax)
//   s_ij = scale * q~_i . c_k,j,   p_i = softmax_j<=i(s_i)
//   o_i  = W_up,t^V (sum_j p_ij c_v,j) + mu^V_t
//
// Tensor-core path (bf16 storage, d = 128, r_k and r_v multiples of 32): one CTA per
// (128-query tile, sequence, head) and four warp roles.
//   warp 0      K producer: W_up,t^K into shared memory (cp.async), then per page of 64 keys
//               the K-plane (one bulk copy: its granule-interleaved layout is already the
//               core-matrix layout of a K-major MMA operand), and W_up,t^V for the epilogue;
//               the V-plane of each page comes as one TMA tensor load with 128-byte swizzle per
//               64 latent columns (an MN-major operand)
//   warp 2      V producer (one thread), decoupled from the K-planes so that neither ring
//               waits on the other
//   warp 1      Q~ and S issuer (one thread) and TMEM owner:
//                 Q~ = Q W_up,t^K             M=128, N=r_k, K=d
//                 S_j = Q~ C_k,j^T            M=128, N=64,  K=r_k   (double-buffered in TMEM)
//   warp 3      PV and output issuer (one thread), so that neither MMA stream waits behind the
//               other's barriers:
//                 O += P_j C_v,j              M=128, N=r_v (split at 256), K=64
//                 out = (O/l) W_up,t^V^T      M=128, N=d,   K=r_v
//   warps 4-11  two threads per query row, each with 32 keys of every page (warps w and w + 4
//               share TMEM lanes): Q and Q~ into bf16 operands, causal mask on diagonal pages,
//               online softmax in the exp2 domain with the row maximum exchanged through shared
//               memory, P into a bf16 operand, O rescaled in TMEM only when a row maximum grows
//               by more than 2^8, V rows past the prompt zeroed on its last page, then the
//               epilogue.
// Accumulators are fp32 in TMEM; operands are bf16 (q~ carries scale * log2 e).
//
// CUDA-core path (fp32 storage, other ranks, d != 128): one CTA per (query, sequence, head),
// fp32 throughout.
#include <cuda_runtime.h>

#include "lla_device.cuh"
#include "lla_internal.h"
#include "lla_tcgen05.cuh"
#include "lla_tmap.h"

namespace lla {
namespace {

constexpr int kBM = 128;         // queries per tile
constexpr int kPT = 64;          // keys per page
constexpr int kSWarps = 8;       // softmax warps: two threads per query row
constexpr int kSWarp0 = 4;       // K producer, S issuer, V producer, PV issuer, then softmax
constexpr int kPThreads = (kSWarp0 + kSWarps) * 32;
constexpr int kSThreads = kSWarps * 32;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kRescaleLog2 = 8.f;  // rescale O only when a row maximum grows by more

struct PParams {
    int T, H, loop, io_bf16;
    float scale_log2;
    const void *w_up_k, *w_up_v;
    const float *mu_v;
    const char *pool;
    int64_t num_blocks, block_bytes;
    int head_page_bytes;
    const int32_t *block_table;
    int max_blocks;
    const int32_t *cu_seqlens;
    int B, max_len;
    const void *q;
    void *out;
    unsigned *err;
    // rotary positions after reconstruction: keys rebuilt and rotated, [B][kpps][H] pages of
    // 64 keys x d in the K-plane layout, and queries rotated and scaled, [Ntok][H][d], bf16
    const char *krot;
    const void *qrot;
    int kpps;
    int64_t qrows;  // rows of the rotated-query buffer (B * max_len)
};

// Shared-memory plan of the tensor-core kernel for ranks (RK, RV); d = 128.  Offsets are
// multiples of 1024 bytes from a 1024-byte aligned base (128-byte swizzle atoms).  With ROPE
// the scores are formed from rebuilt, rotated keys of width d instead of latents of width RK.
template <int RK, int RV, bool ROPE = false>
struct PF {
    static constexpr int D = 128;
    static constexpr int RS = ROPE ? D : RK;         // contraction width of the scores
    static constexpr int NKC = RK / 8;               // 16-byte chunks of a K row
    static constexpr int NVC = RV / 8;               // 16-byte chunks of a V row
    static constexpr int VATOMS = (RV + 63) / 64;    // 64-column atoms of a V page (TMA boxes)
    static constexpr int N0 = RV > 256 ? 256 : RV;   // PV MMA split on atom boundaries
    static constexpr int N1 = RV - N0;
    static constexpr int KPAGE = kPT * RS * 2;
    static constexpr int VPAGE = VATOMS * kPT * 128;
    static constexpr int QT = kBM * RS * 2;          // q~ (or rotated q) operand
    static constexpr int PB = kBM * kPT * 2;         // P operand (one of two)
    static constexpr int QA = kBM * D * 2;           // q operand (prologue)
    static constexpr int WK = D * RK * 2;            // W_up,t^K operand (prologue)
    static constexpr int WV = D * RV * 2;            // W_up,t^V operand (epilogue)
    static constexpr int OA = kBM * RV * 2;          // O / l operand (epilogue)
    // K and V pipeline stages: as deep as shared memory allows (up to 4), V at least 2 deep
    static constexpr int BUDGET = 220 * 1024 - QT - 2 * PB;
    static constexpr int STV = (BUDGET - 2 * KPAGE) / VPAGE >= 4 ? 4 : (BUDGET - 2 * KPAGE) / VPAGE >= 3 ? 3 : 2;
    static constexpr int STK0 = (BUDGET - STV * VPAGE) / KPAGE;
    static constexpr int STK = STK0 > 4 ? 4 : STK0;
    static constexpr int oQT = 0;
    static constexpr int oK = oQT + QT;
    static constexpr int oV = oK + STK * KPAGE;
    static constexpr int oP = oV + STV * VPAGE;
    static constexpr int oEnd = oP + 2 * PB;
    // the prologue operands alias the V ring and P; the epilogue operands alias K, V and P
    static constexpr int oQA = oV, oWK = oV + QA;
    static constexpr int oOA = oK, oWV = oK + OA;
    static constexpr int oX = oEnd;                   // [2 pages][2 halves][128 rows] maxima
    static constexpr int oL = oX + 2 * 2 * kBM * 4;   // [2 halves][128 rows] row sums
    static constexpr int oBar = oL + 2 * kBM * 4;
    static constexpr int NBAR = 40;
    static constexpr int SMEM = 1024 + oBar + NBAR * 8 + 16;
    // TMEM columns: S double buffer [0, 128), O [128, 128 + RV); q~ and out reuse [0, ...)
    static constexpr uint32_t TM_S = 0, TM_O = 128, TM_COLS = 512;
    static_assert(RK % 32 == 0 && RV % 32 == 0 && RK <= 256 && 128 + RV <= 512, "ranks");
    static_assert(N0 % 16 == 0 && N1 % 16 == 0 && N1 <= 256, "PV split");
    static_assert(STK >= 2 && STV >= 2, "pipeline depth");
    static_assert(oK % 1024 == 0 && oV % 1024 == 0 && oP % 1024 == 0 && VPAGE % 1024 == 0, "align");
    static_assert(oWK + WK <= oEnd && oWV + WV <= oEnd, "aliased operands fit");
    static_assert(SMEM <= 227 * 1024, "shared memory");
};

// barrier indices
enum {
    kBSetup = 0, kBQt, kBQs, kBOa, kBWv, kBOut, kBUnused, kBOfin,
    kBSfull = 8 /* [2] */, kBSfree = 10, kBPfull = 12, kBPfree = 14,
    kBOa2 = 16, kBOut1 = 17,
    kBKfull = 18 /* [4] */, kBKempty = 22, kBVfull = 26, kBVempty = 30,
    kBAbort = 34  // slot used as the CTA's abort flag
};

template <int RK, int RV, bool ROPE>
__global__ void __launch_bounds__(kPThreads, 1)
    prefill_tc_kernel(const __grid_constant__ CUtensorMap tv, const PParams p) {
    using F = PF<RK, RV, ROPE>;
    constexpr int D = F::D;
    extern __shared__ __align__(1024) char sm_raw[];
    char *sm = reinterpret_cast<char *>((reinterpret_cast<uintptr_t>(sm_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    uint64_t *bar = reinterpret_cast<uint64_t *>(sm + F::oBar);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(bar + kBAbort);
    uint32_t *tslot = reinterpret_cast<uint32_t *>(bar + F::NBAR);
    float *xmax = reinterpret_cast<float *>(sm + F::oX);
    float *xsum = reinterpret_cast<float *>(sm + F::oL);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

    const int nqt = (p.max_len + kBM - 1) / kBM;
    const int qt = nqt - 1 - static_cast<int>(blockIdx.x);  // longest causal ranges first
    const int b = blockIdx.y, h = blockIdx.z;
    pdl_wait();
    const int q0 = p.cu_seqlens[b];
    const int L = p.cu_seqlens[b + 1] - q0;
    if (L > p.max_len || L < 0 || (ROPE && static_cast<int64_t>(q0) + L > p.qrows)) {
        if (tid == 0 && qt == nqt - 1) atomicOr(p.err, LLA_DEVERR_CONTEXT);
        return;
    }
    const int i0 = qt * kBM;
    if (i0 >= L) return;  // uniform over the CTA, before any barrier or TMEM use
    const int iend = min(L, i0 + kBM);
    const int NP = (iend - 1) / kPT + 1;  // pages 0..NP-1 hold every key of the tile
    const int64_t wofs = (static_cast<int64_t>(h) * p.T + p.loop) * D;
    const int32_t *bt = p.block_table + static_cast<int64_t>(b) * p.max_blocks;

    if (tid == 0) {
        mbar_init(&bar[kBSetup], 32 + kSThreads);
        mbar_init(&bar[kBQt], 1);
        mbar_init(&bar[kBQs], kSThreads);
        mbar_init(&bar[kBOa], kSThreads);
        mbar_init(&bar[kBOa2], kSThreads);
        mbar_init(&bar[kBWv], 32);
        mbar_init(&bar[kBOut1], 1);
        mbar_init(&bar[kBOut], 1);
        mbar_init(&bar[kBOfin], 1);
        for (int s = 0; s < F::STK; ++s) {
            mbar_init(&bar[kBKfull + s], 1);
            mbar_init(&bar[kBKempty + s], 1);
        }
        for (int s = 0; s < F::STV; ++s) {
            mbar_init(&bar[kBVfull + s], 1);
            mbar_init(&bar[kBVempty + s], 1);
        }
        for (int s = 0; s < 2; ++s) {
            mbar_init(&bar[kBSfull + s], 1);
            mbar_init(&bar[kBSfree + s], kSThreads);
            mbar_init(&bar[kBPfull + s], kSThreads);
            mbar_init(&bar[kBPfree + s], 1);
        }
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 1) tmem_alloc(tslot, F::TM_COLS);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tslot;

    if (warp == 0) {
        // ------------------------------------------------------------------------- producer
        if constexpr (!ROPE) {
            const char *wk = static_cast<const char *>(p.w_up_k) + wofs * RK * 2;
            // W_up,t^K [d][r_k] as an MN-major operand: (row e, column chunk g) at g*(d*16) + e*16
            for (int i = lane; i < D * F::NKC; i += 32) {
                const int e = i / F::NKC, g = i - e * F::NKC;
                cp_async16(sm + F::oWK + g * (D * 16) + e * 16, wk + (static_cast<int64_t>(e) * RK + g * 8) * 2);
            }
            cp_async_commit();
            cp_async_wait_all();
            fence_proxy_async_smem();
        }
        mbar_arrive(&bar[kBSetup]);
        if (lane == 0) {  // K-planes: one bulk copy per page
            const uint64_t pol = policy_evict_first();
            int nk = 0;  // copies issued
            for (int j = 0; j < NP; ++j) {
                const int s = j % F::STK;
                const uint32_t ph = (j / F::STK) & 1;
                int32_t blk = bt[j];
                if (blk < 0 || blk >= p.num_blocks) {
                    atomicOr(p.err, LLA_DEVERR_BLOCK_ID);
                    blk = 0;
                }
                const int64_t hp = static_cast<int64_t>(blk) * p.H + h;  // head page index
                // the latent K-plane of the page, or its rebuilt and rotated keys
                const char *src = ROPE ? p.krot + ((static_cast<int64_t>(b) * p.kpps + j) * p.H + h) * F::KPAGE
                                       : p.pool + hp * p.head_page_bytes;
                if (!mbar_wait(&bar[kBKempty + s], ph ^ 1u, abort_flag, p.err) || *abort_flag) break;
                mbar_arrive_expect_tx(&bar[kBKfull + s], F::KPAGE);
                bulk_g2s(sm + F::oK + s * F::KPAGE, src, F::KPAGE, &bar[kBKfull + s], pol);
                ++nk;
            }
            // every copy has landed before the ring is reused or the CTA exits, even after an
            // abort (no copy is issued once a wait has failed)
            volatile int never = 0;
            for (int j = max(0, nk - F::STK); j < nk; ++j)
                mbar_wait(&bar[kBKfull + j % F::STK], (j / F::STK) & 1, &never, p.err);
        }
        __syncwarp();
        // epilogue operand W_up,t^V [d][r_v] (K-major): (row e, chunk c) at c*(d*16) + e*16,
        // into the K ring once every MMA of the loop has completed
        mbar_wait(&bar[kBOfin], 0, abort_flag, p.err);
        const char *wv = static_cast<const char *>(p.w_up_v) + wofs * RV * 2;
        for (int i = lane; i < D * F::NVC; i += 32) {
            const int e = i / F::NVC, c = i - e * F::NVC;
            cp_async16(sm + F::oWV + c * (D * 16) + e * 16, wv + (static_cast<int64_t>(e) * RV + c * 8) * 2);
        }
        cp_async_commit();
        cp_async_wait_all();
        fence_proxy_async_smem();
        mbar_arrive(&bar[kBWv]);
    } else if (warp == 2) {
        // ---------------------------------------------------------------------- V producer
        if (lane == 0) {  // V-planes: one TMA tensor load with 128-byte swizzle per 64 columns
            // the V ring aliases the prologue operands: wait until Q~ has been computed
            mbar_wait(&bar[kBQt], 0, abort_flag, p.err);
            int nv = 0;  // copies issued
            for (int j = 0; j < NP; ++j) {
                const int s = j % F::STV;
                const uint32_t ph = (j / F::STV) & 1;
                int32_t blk = bt[j];
                if (blk < 0 || blk >= p.num_blocks) blk = 0;  // flagged by the K producer
                const int64_t hp = static_cast<int64_t>(blk) * p.H + h;
                if (!mbar_wait(&bar[kBVempty + s], ph ^ 1u, abort_flag, p.err) || *abort_flag) break;
                mbar_arrive_expect_tx(&bar[kBVfull + s], F::VPAGE);
                char *vs = sm + F::oV + s * F::VPAGE;
#pragma unroll
                for (int a = 0; a < F::VATOMS; ++a)
                    tma_load_3d(vs + a * (kPT * 128), &tv, a * 64, 0, static_cast<int>(hp), &bar[kBVfull + s]);
                ++nv;
            }
            volatile int never = 0;  // as for the K ring
            for (int j = max(0, nv - F::STV); j < nv; ++j)
                mbar_wait(&bar[kBVfull + j % F::STV], (j / F::STV) & 1, &never, p.err);
        }
        __syncwarp();
    } else if (warp == 1) {
        // -------------------------------------------------------------- Q~ and S MMA issuer
        if (lane == 0) {
            const uint32_t base = smem_addr(sm);
            mbar_wait(&bar[kBSetup], 0, abort_flag, p.err);
            tc_fence_after();
            if constexpr (ROPE) {
                mbar_arrive(&bar[kBQt]);  // the rotated queries come ready from global memory
            } else {
                constexpr uint32_t idq = umma_idesc_bf16(128, RK, 0, 1);
                const uint64_t dqa = umma_desc(base + F::oQA, 2048, 128);
                const uint64_t dwk = umma_desc(base + F::oWK, 128, 2048);
#pragma unroll
                for (int ks = 0; ks < D / 16; ++ks)
                    umma_bf16(tmem + 0, dqa + ks * (4096 >> 4), dwk + ks * (256 >> 4), idq, ks > 0);
                umma_commit(&bar[kBQt]);
            }
            mbar_wait(&bar[kBQs], 0, abort_flag, p.err);
            tc_fence_after();
            constexpr uint32_t ids = umma_idesc_bf16(128, kPT, 0, 0);
            // descriptors are built once; a byte offset moves the start-address field by offset/16
            const uint64_t dq = umma_desc(base + F::oQT, 2048, 128);
            const uint64_t dk0 = umma_desc(base + F::oK, 1024, 128);
#pragma unroll 1
            for (int j = 0; j < NP; ++j) {
                const int s = j & 1, sk = j % F::STK;
                mbar_wait(&bar[kBKfull + sk], (j / F::STK) & 1, abort_flag, p.err);
                if (j >= 2) mbar_wait(&bar[kBSfree + s], ((j - 2) >> 1) & 1, abort_flag, p.err);
                tc_fence_after();
                const uint64_t dk = dk0 + static_cast<uint64_t>(sk * (F::KPAGE >> 4));
                const uint32_t ds = tmem + F::TM_S + s * kPT;
#pragma unroll
                for (int ks = 0; ks < F::RS / 16; ++ks)
                    umma_bf16(ds, dq + ks * (4096 >> 4), dk + ks * (2048 >> 4), ids, ks > 0);
                umma_commit(&bar[kBSfull + s]);
                umma_commit(&bar[kBKempty + sk]);
            }
            // every product of this thread has completed before TMEM is released, even after an
            // abort (when the softmax warps stop waiting for them): a commit tracks all earlier
            // products of its thread, so the last one suffices
            volatile int never = 0;
            if (NP > 0)
                mbar_wait(&bar[kBSfull + ((NP - 1) & 1)], ((NP - 1) >> 1) & 1, &never, p.err);
            else if constexpr (!ROPE)
                mbar_wait(&bar[kBQt], 0, &never, p.err);
        }
        __syncwarp();
    } else if (warp == 3) {
        // ----------------------------------------------------------- PV and output MMA issuer
        if (lane == 0) {
            const uint32_t base = smem_addr(sm);
            constexpr uint32_t idv0 = umma_idesc_bf16(128, F::N0, 0, 1);
            constexpr uint32_t idv1 = umma_idesc_bf16(128, F::N1 > 0 ? F::N1 : 16, 0, 1);
            const uint64_t dp0 = umma_desc(base + F::oP, 2048, 128);
            const uint64_t dv0 = umma_desc_sw128_mn(base + F::oV, kPT * 128);
#pragma unroll 1
            for (int jj = 0; jj < NP; ++jj) {
                const int s = jj & 1, sv = jj % F::STV;
                mbar_wait(&bar[kBPfull + s], (jj >> 1) & 1, abort_flag, p.err);
                mbar_wait(&bar[kBVfull + sv], (jj / F::STV) & 1, abort_flag, p.err);
                tc_fence_after();
                const uint64_t dp = dp0 + static_cast<uint64_t>(s * (F::PB >> 4));
                const uint64_t dv = dv0 + static_cast<uint64_t>(sv * (F::VPAGE >> 4));
                const bool acc = jj > 0;
#pragma unroll
                for (int ks = 0; ks < kPT / 16; ++ks) {
                    umma_bf16(tmem + F::TM_O, dp + ks * (4096 >> 4), dv + ks * (2048 >> 4), idv0, acc || ks > 0);
                    if constexpr (F::N1 > 0)
                        umma_bf16(tmem + F::TM_O + F::N0, dp + ks * (4096 >> 4),
                                  dv + ((F::N0 / 64) * (kPT * 128) >> 4) + ks * (2048 >> 4), idv1,
                                  acc || ks > 0);
                }
                umma_commit(&bar[kBVempty + sv]);
                umma_commit(&bar[kBPfree + s]);
            }
            umma_commit(&bar[kBOfin]);  // every PV MMA (and, before them, every S MMA) has completed
            // out = (O / l) W_up,t^V^T, with O / l = hi + lo as two bf16 operands in turn, so
            // that the projection sees O / l to about 16 significant bits
            mbar_wait(&bar[kBWv], 0, abort_flag, p.err);
            constexpr uint32_t ido = umma_idesc_bf16(128, D, 0, 0);
            const uint64_t doa = umma_desc(base + F::oOA, 2048, 128);
            const uint64_t dwv = umma_desc(base + F::oWV, 2048, 128);
#pragma unroll 1
            for (int part = 0; part < 2; ++part) {
                mbar_wait(&bar[part ? kBOa2 : kBOa], 0, abort_flag, p.err);
                tc_fence_after();
#pragma unroll 1
                for (int ks = 0; ks < RV / 16; ++ks)
                    umma_bf16(tmem + 0, doa + ks * (4096 >> 4), dwv + ks * (4096 >> 4), ido, part > 0 || ks > 0);
                umma_commit(&bar[part ? kBOut : kBOut1]);
            }
            volatile int never = 0;  // as for the S^T issuer: the last commit of this thread
            mbar_wait(&bar[kBOut], 0, &never, p.err);
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------------ softmax and epilogue
        // warps 4..11: quarter (TMEM lanes) = warp % 4, half = which 32 keys of a page (and which
        // half of every other row-wise job) this thread owns; warps w and w + 4 share rows
        const int quarter = warp & 3;
        const int half = (warp - kSWarp0) >> 2;
        const int row = quarter * 32 + lane;
        const int pair_bar = 2 + quarter;  // named barrier of the two warps of this quarter
        const uint32_t tl = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
        const int qi = i0 + row;
        const bool valid_row = qi < L;
        const int64_t qrow = (static_cast<int64_t>(q0) + qi) * p.H + h;
        if constexpr (ROPE) {
            // the rotated, scaled q row (this half's 64 elements) -> the score operand directly
            char *qt_ = sm + F::oQT + row * 16;
            const uint4 *src = reinterpret_cast<const uint4 *>(static_cast<const char *>(p.qrot) + qrow * D * 2);
            const int c0 = half * (D / 16);
#pragma unroll
            for (int c = c0; c < c0 + D / 16; ++c)
                *reinterpret_cast<uint4 *>(qt_ + c * 2048) = valid_row ? src[c] : make_uint4(0, 0, 0, 0);
            fence_proxy_async_smem();
            mbar_arrive(&bar[kBSetup]);
            mbar_wait(&bar[kBQt], 0, abort_flag, p.err);
            mbar_arrive(&bar[kBQs]);
        } else {
        // q row (this half's 64 elements) -> bf16 K-major operand: chunk c at c*2048 + row*16
        {
            char *qa = sm + F::oQA + row * 16;
            const int c0 = half * (D / 16);
            if (p.io_bf16) {
                const uint4 *src = reinterpret_cast<const uint4 *>(static_cast<const char *>(p.q) + qrow * D * 2);
#pragma unroll
                for (int c = c0; c < c0 + D / 16; ++c)
                    *reinterpret_cast<uint4 *>(qa + c * 2048) = valid_row ? src[c] : make_uint4(0, 0, 0, 0);
            } else {
                const float4 *src = reinterpret_cast<const float4 *>(static_cast<const char *>(p.q) + qrow * D * 4);
#pragma unroll
                for (int c = c0; c < c0 + D / 16; ++c) {
                    float4 a = make_float4(0.f, 0.f, 0.f, 0.f), b2 = a;
                    if (valid_row) {
                        a = src[2 * c];
                        b2 = src[2 * c + 1];
                    }
                    *reinterpret_cast<uint4 *>(qa + c * 2048) =
                        make_uint4(pack_bf16x2(a.x, a.y), pack_bf16x2(a.z, a.w), pack_bf16x2(b2.x, b2.y),
                                   pack_bf16x2(b2.z, b2.w));
                }
            }
        }
        fence_proxy_async_smem();
        mbar_arrive(&bar[kBSetup]);
        // q~ (scaled into the exp2 domain) -> bf16 K-major operand; this half's RK/2 columns
        mbar_wait(&bar[kBQt], 0, abort_flag, p.err);
        tc_fence_after();
#pragma unroll 1
        for (int c0 = half * (RK / 2); c0 < (half + 1) * (RK / 2); c0 += 16) {
            float v[16];
            tmem_ld16(tl + c0, v);
            char *qt_ = sm + F::oQT + row * 16;
            const float sc = p.scale_log2;
#pragma unroll
            for (int k = 0; k < 16; k += 8)
                *reinterpret_cast<uint4 *>(qt_ + ((c0 + k) / 8) * 2048) =
                    make_uint4(pack_bf16x2(v[k] * sc, v[k + 1] * sc), pack_bf16x2(v[k + 2] * sc, v[k + 3] * sc),
                               pack_bf16x2(v[k + 4] * sc, v[k + 5] * sc), pack_bf16x2(v[k + 6] * sc, v[k + 7] * sc));
        }
        fence_proxy_async_smem();
        tc_fence_before();
        mbar_arrive(&bar[kBQs]);
        }

        const int lim = min(qi, L - 1);  // keys 0..lim are visible to this row
        const int kofs = half * 32;      // this thread's keys within a page
        float m = -INFINITY, l = 0.f;
#pragma unroll 1
        for (int j = 0; j < NP; ++j) {
            const int s = j & 1;
            const int kb = j * kPT;
            mbar_wait(&bar[kBSfull + s], (j >> 1) & 1, abort_flag, p.err);
            tc_fence_after();
            float x[32];
            tmem_ld32(tl + F::TM_S + s * kPT + kofs, x);
            tc_fence_before();
            mbar_arrive(&bar[kBSfree + s]);
            if (kb + kPT - 1 > i0) {  // a page on the diagonal (or past the prompt): mask
                const int nv = lim - (kb + kofs);  // keys c <= nv are visible
#pragma unroll
                for (int c = 0; c < 32; ++c) x[c] = c <= nv ? x[c] : -INFINITY;
            }
            float mx;
            {  // tree maximum: 5 dependent steps instead of 32
                float t[16];
#pragma unroll
                for (int c = 0; c < 16; ++c) t[c] = fmaxf(x[c], x[c + 16]);
#pragma unroll
                for (int w = 8; w >= 1; w >>= 1)
#pragma unroll
                    for (int c = 0; c < w; ++c) t[c] = fmaxf(t[c], t[c + w]);
                mx = t[0];
            }
            // the row maximum over both halves
            xmax[(s * 2 + half) * kBM + row] = mx;
            named_bar_sync(pair_bar, 64);
            mx = fmaxf(mx, xmax[(s * 2 + (half ^ 1)) * kBM + row]);
            const float m_new = fmaxf(m, mx);
            const bool need = m_new > m + kRescaleLog2;  // also the first finite maximum
            const float factor = need ? ex2_approx(m - m_new) : 1.f;
            if (need) {
                l *= factor;
                m = m_new;
            }
            if (__any_sync(0xffffffffu, need && j > 0)) {
                // O holds pages 0..j-1: wait for the last of them, then rescale this half.  The
                // product of page j - 1 releases P buffer (j - 1) & 1; the one of page j - 3 had
                // released it before this row wrote page j - 1, so the parity test cannot pass a
                // phase early (a barrier committed once per page could be two phases behind)
                mbar_wait(&bar[kBPfree + ((j - 1) & 1)], ((j - 1) >> 1) & 1, abort_flag, p.err);
                tc_fence_after();
#pragma unroll 1
                for (int c0 = half * (RV / 2); c0 < (half + 1) * (RV / 2); c0 += 16) {
                    float v[16];
                    tmem_ld16(tl + F::TM_O + c0, v);
#pragma unroll
                    for (int c = 0; c < 16; ++c) v[c] *= factor;
                    tmem_st16(tl + F::TM_O + c0, v);
                }
            }
            if (j >= 2) mbar_wait(&bar[kBPfree + s], ((j - 2) >> 1) & 1, abort_flag, p.err);
            char *pr = sm + F::oP + s * F::PB + row * 16 + (kofs / 8) * 2048;
#pragma unroll
            for (int c = 0; c < 32; ++c) x[c] = ex2_approx(x[c] - m);
#pragma unroll
            for (int c = 0; c < 32; c += 8)
                *reinterpret_cast<uint4 *>(pr + (c / 8) * 2048) =
                    make_uint4(pack_bf16x2(x[c], x[c + 1]), pack_bf16x2(x[c + 2], x[c + 3]),
                               pack_bf16x2(x[c + 4], x[c + 5]), pack_bf16x2(x[c + 6], x[c + 7]));
            {  // tree sum of this half's probabilities
                float t[16];
#pragma unroll
                for (int c = 0; c < 16; ++c) t[c] = x[c] + x[c + 16];
#pragma unroll
                for (int w = 8; w >= 1; w >>= 1)
#pragma unroll
                    for (int c = 0; c < w; ++c) t[c] += t[c + w];
                l += t[0];
            }
            if (j == NP - 1 && kb + kPT > L) {
                // last page of the prompt: V rows past it hold no latents; zero them before the
                // PV product reads them (0 * NaN would poison the sum)
                const int sv = j % F::STV;
                mbar_wait(&bar[kBVfull + sv], (j / F::STV) & 1, abort_flag, p.err);
                char *vs = sm + F::oV + sv * F::VPAGE;
                const int valid = L - kb;
                const int nz = (kPT - valid) * F::VATOMS * 8;  // 16-byte words to clear
                for (int w = tid - kSWarp0 * 32; w < nz; w += kSThreads) {
                    const int c = w & 7, r2 = w >> 3;
                    const int a = r2 % F::VATOMS, i = valid + r2 / F::VATOMS;
                    *reinterpret_cast<uint4 *>(vs + a * (kPT * 128) + i * 128 + c * 16) = make_uint4(0, 0, 0, 0);
                }
            }
            fence_proxy_async_smem();
            tc_fence_before();
            mbar_arrive(&bar[kBPfull + s]);
        }
        // the row sum over both halves
        xsum[half * kBM + row] = l;
        named_bar_sync(pair_bar, 64);
        l += xsum[(half ^ 1) * kBM + row];
        // epilogue: O / l -> two bf16 K-major operands in turn (hi, then lo = O/l - hi) in one
        // buffer that aliases the K ring; O stays in TMEM between the two
        mbar_wait(&bar[kBOfin], 0, abort_flag, p.err);
        tc_fence_after();
        const float inv = l > 0.f ? 1.f / l : 0.f;
#pragma unroll 1
        for (int part = 0; part < 2; ++part) {
            if (part) {
                mbar_wait(&bar[kBOut1], 0, abort_flag, p.err);  // the hi product has read the buffer
                tc_fence_after();
            }
#pragma unroll 1
            for (int c0 = half * (RV / 2); c0 < (half + 1) * (RV / 2); c0 += 16) {
                float v[16];
                tmem_ld16(tl + F::TM_O + c0, v);
#pragma unroll
                for (int k = 0; k < 16; ++k) {
                    const float xv = v[k] * inv;
                    const float hi = __bfloat162float(__float2bfloat16_rn(xv));
                    v[k] = part ? xv - hi : hi;
                }
                char *oa = sm + F::oOA + row * 16;
#pragma unroll
                for (int k = 0; k < 16; k += 8)
                    *reinterpret_cast<uint4 *>(oa + ((c0 + k) / 8) * 2048) =
                        make_uint4(pack_bf16x2(v[k], v[k + 1]), pack_bf16x2(v[k + 2], v[k + 3]),
                                   pack_bf16x2(v[k + 4], v[k + 5]), pack_bf16x2(v[k + 6], v[k + 7]));
            }
            fence_proxy_async_smem();
            tc_fence_before();
            mbar_arrive(&bar[part ? kBOa2 : kBOa]);
        }
        mbar_wait(&bar[kBOut], 0, abort_flag, p.err);
        tc_fence_after();
        const float *muv = p.mu_v ? p.mu_v + wofs : nullptr;
#pragma unroll 1
        for (int c0 = half * (D / 2); c0 < (half + 1) * (D / 2); c0 += 32) {
            float v[32];
            tmem_ld32(tl + c0, v);
            if (muv) {
#pragma unroll
                for (int c = 0; c < 32; ++c) v[c] += muv[c0 + c];
            }
            if (valid_row) {
                char *dst = static_cast<char *>(p.out) + (qrow * D + c0) * (p.io_bf16 ? 2 : 4);
                if (p.io_bf16) {
#pragma unroll
                    for (int k = 0; k < 32; k += 8)
                        *reinterpret_cast<uint4 *>(dst + k * 2) =
                            make_uint4(pack_bf16x2(v[k], v[k + 1]), pack_bf16x2(v[k + 2], v[k + 3]),
                                       pack_bf16x2(v[k + 4], v[k + 5]), pack_bf16x2(v[k + 6], v[k + 7]));
                } else {
#pragma unroll
                    for (int k = 0; k < 32; k += 4)
                        *reinterpret_cast<float4 *>(dst + k * 4) = make_float4(v[k], v[k + 1], v[k + 2], v[k + 3]);
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

// ------------------------------------------------------------------------- CUDA-core path

struct GParams {
    int T, H, d, r_k, r_v, loop, storage_bf16, io_bf16;
    float scale_log2;
    const void *w_up_k, *w_up_v;
    const float *mu_v;
    const char *pool;
    int64_t num_blocks, block_bytes;
    int head_page_bytes, kplane_bytes;
    const int32_t *block_table;
    int max_blocks;
    const int32_t *cu_seqlens;
    int max_len;
    const void *q;
    void *out;
    unsigned *err;
};

constexpr int kGThreads = 128;
constexpr int kGKeys = 128;  // keys per step

// One CTA per (query, sequence, head), fp32 accumulation.  Shared memory: q [d], q~ [r_k],
// o~ [r_v], p [kGKeys], reduction scratch.
__global__ void __launch_bounds__(kGThreads) prefill_generic_kernel(const GParams p) {
    extern __shared__ __align__(16) float gs[];
    const int qi = blockIdx.x, b = blockIdx.y, h = blockIdx.z, tid = threadIdx.x;
    pdl_wait();
    const int q0 = p.cu_seqlens[b];
    const int L = p.cu_seqlens[b + 1] - q0;
    if (L > p.max_len || L < 0) {
        if (tid == 0 && qi == 0) atomicOr(p.err, LLA_DEVERR_CONTEXT);
        return;
    }
    if (qi >= L) return;
    const int es = p.storage_bf16 ? 2 : 4;
    float *qv = gs, *qt = qv + p.d, *ov = qt + p.r_k, *pv = ov + p.r_v, *red = pv + kGKeys;
    const int64_t qrow = (static_cast<int64_t>(q0) + qi) * p.H + h;
    const int64_t wofs = (static_cast<int64_t>(h) * p.T + p.loop) * p.d;
    for (int e = tid; e < p.d; e += kGThreads) qv[e] = load_elem(p.q, qrow * p.d + e, p.io_bf16);
    for (int j = tid; j < p.r_v; j += kGThreads) ov[j] = 0.f;
    __syncthreads();
    for (int j = tid; j < p.r_k; j += kGThreads) {  // q~ = W_up,t^K^T q
        float acc = 0.f;
        for (int e = 0; e < p.d; ++e)
            acc = fmaf(load_elem(p.w_up_k, (wofs + e) * p.r_k + j, p.storage_bf16), qv[e], acc);
        qt[j] = acc * p.scale_log2;
    }
    __syncthreads();
    const int gk = granule_bytes(p.r_k, es);
    const int32_t *bt = p.block_table + static_cast<int64_t>(b) * p.max_blocks;
    float m = -INFINITY, l = 0.f;
    for (int k0 = 0; k0 <= qi; k0 += kGKeys) {
        const int kj = k0 + tid;
        float s = -INFINITY;
        if (kj <= qi) {
            int32_t blk = bt[kj / kPT];
            if (blk < 0 || blk >= p.num_blocks) {
                atomicOr(p.err, LLA_DEVERR_BLOCK_ID);
                blk = 0;
            }
            const char *page = p.pool + blk * p.block_bytes + static_cast<int64_t>(h) * p.head_page_bytes;
            float acc = 0.f;
            for (int j = 0; j < p.r_k; ++j) {
                const char *e = page + kplane_offset(kj % kPT, j, es, gk);
                acc = fmaf(qt[j], es == 2 ? bf_to_f(*reinterpret_cast<const uint16_t *>(e))
                                          : *reinterpret_cast<const float *>(e), acc);
            }
            s = acc;
        }
        // block maximum
        float mx = warp_max(s);
        if ((tid & 31) == 0) red[tid >> 5] = mx;
        __syncthreads();
        mx = red[0];
        for (int w = 1; w < kGThreads / 32; ++w) mx = fmaxf(mx, red[w]);
        const float m_new = fmaxf(m, mx);
        const float alpha = exp2f(m - m_new);
        const float pj = kj <= qi ? exp2f(s - m_new) : 0.f;
        pv[tid] = pj;
        float ps = warp_sum(pj);
        __syncthreads();  // every thread has read red[] for the maximum
        if ((tid & 31) == 0) red[tid >> 5] = ps;
        __syncthreads();
        float psum = 0.f;
        for (int w = 0; w < kGThreads / 32; ++w) psum += red[w];
        l = l * alpha + psum;
        m = m_new;
        const int nk = min(kGKeys, qi + 1 - k0);
        for (int j = tid; j < p.r_v; j += kGThreads) {
            float acc = ov[j] * alpha;
            for (int t = 0; t < nk; ++t) {
                const int kk = k0 + t;
                int32_t blk = bt[kk / kPT];
                if (blk < 0 || blk >= p.num_blocks) blk = 0;
                const char *e = p.pool + blk * p.block_bytes + static_cast<int64_t>(h) * p.head_page_bytes +
                                p.kplane_bytes + (static_cast<int64_t>(kk % kPT) * p.r_v + j) * es;
                acc = fmaf(pv[t], es == 2 ? bf_to_f(*reinterpret_cast<const uint16_t *>(e))
                                          : *reinterpret_cast<const float *>(e), acc);
            }
            ov[j] = acc;
        }
        __syncthreads();
    }
    const float inv = 1.f / l;
    for (int e = tid; e < p.d; e += kGThreads) {
        float acc = 0.f;
        for (int j = 0; j < p.r_v; ++j)
            acc = fmaf(load_elem(p.w_up_v, (wofs + e) * p.r_v + j, p.storage_bf16), ov[j], acc);
        float o = acc * inv;
        if (p.mu_v) o += p.mu_v[wofs + e];
        store_elem(p.out, qrow * p.d + e, o, p.io_bf16);
    }
    pdl_trigger();
}

// ------------------------------------------------- rotary positions: rebuild and rotate keys
//
// Sec. 3 "RoPE and reconstruction": keys are rebuilt by Eq. decode and rotated at their
// positions before attention.  One CTA per (sequence, page of 64 prompt tokens, group of heads)
// loops over its heads: Khat (64 tokens x d) = C_k W_up,t^K^T + mu^K_t on tcgen05 (M = 64 tokens, N = d,
// K = r_k, plus one K step for mu^K_t), then each token's pairs are rotated in registers and
// written as a bf16 page in the K-plane layout (granule g of 8 dimensions at g*1024 + token*16),
// and the page's queries are rotated and scaled by scale * log2 e into a bf16 copy of q.

// 32 consecutive elements (bf16 or fp32, 16-byte aligned) as floats, loads issued together.
__device__ __forceinline__ void load32(const void *src, int is_bf16, float (&v)[32]) {
    if (is_bf16) {
        uint4 u[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) u[i] = reinterpret_cast<const uint4 *>(src)[i];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float2 a = bf2_to_f2(u[i].x), b = bf2_to_f2(u[i].y), c = bf2_to_f2(u[i].z), d = bf2_to_f2(u[i].w);
            v[8 * i] = a.x; v[8 * i + 1] = a.y; v[8 * i + 2] = b.x; v[8 * i + 3] = b.y;
            v[8 * i + 4] = c.x; v[8 * i + 5] = c.y; v[8 * i + 6] = d.x; v[8 * i + 7] = d.y;
        }
    } else {
        float4 f[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) f[i] = reinterpret_cast<const float4 *>(src)[i];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            v[4 * i] = f[i].x; v[4 * i + 1] = f[i].y; v[4 * i + 2] = f[i].z; v[4 * i + 3] = f[i].w;
        }
    }
}

// 32 floats as bf16 (round to nearest even) with 16-byte stores.
__device__ __forceinline__ void store32_bf16(void *dst, const float (&v)[32]) {
#pragma unroll
    for (int i = 0; i < 4; ++i)
        reinterpret_cast<uint4 *>(dst)[i] =
            make_uint4(pack_bf16x2(v[8 * i], v[8 * i + 1]), pack_bf16x2(v[8 * i + 2], v[8 * i + 3]),
                       pack_bf16x2(v[8 * i + 4], v[8 * i + 5]), pack_bf16x2(v[8 * i + 6], v[8 * i + 7]));
}

struct RParams {
    int T, H, loop, io_bf16, kpps, pairing;
    float scale_log2;
    const void *w_up_k;
    const float *mu_k;
    const char *pool;
    int64_t num_blocks;
    int head_page_bytes;
    const int32_t *block_table;
    int max_blocks;
    const int32_t *cu_seqlens;
    int max_len;
    const void *q;
    char *krot;
    void *qrot;
    int64_t qrows;  // rows of the rotated-query buffer: B * max_len
    unsigned *err;
    unsigned long long phi[64];  // theta_j / (2 pi) * 2^64
};

template <int RK>
struct RB {
    static constexpr int D = 128;
    static constexpr int NG = RK / 8;                 // 16-byte granules of a latent row
    static constexpr int oTab = 0;                    // [64 tokens][65] (cos, sin) per pair
    static constexpr int TAB = 64 * 65 * 8;
    static constexpr int oB = (TAB + 1023) & ~1023;   // (mu_hi, mu_lo) granule, then W_up,t^K
    static constexpr int oW = oB + D * 16;
    static constexpr int oA = oW + NG * D * 16;       // the page's K-plane, then ones and zeros
    static constexpr int oOnes = oA + NG * 64 * 16;
    static constexpr int oBar = oOnes + 2 * 64 * 16;
    static constexpr int SMEM = oBar + 16 + 1024;     // + alignment slack
    static constexpr uint32_t IDESC = umma_idesc_bf16(64, D, 0, 0);
    static_assert(RK % 16 == 0, "K steps");
};

template <int RK>
__global__ void __launch_bounds__(128) rope_rebuild_kernel(const __grid_constant__ RParams p) {
    using Z = RB<RK>;
    constexpr int D = Z::D;
    extern __shared__ __align__(1024) char rb_raw[];
    char *sm = reinterpret_cast<char *>((reinterpret_cast<uintptr_t>(rb_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    float2 *tab = reinterpret_cast<float2 *>(sm + Z::oTab);
    uint64_t *bar = reinterpret_cast<uint64_t *>(sm + Z::oBar);
    uint32_t *tslot = reinterpret_cast<uint32_t *>(bar + 1);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int pg = blockIdx.x, b = blockIdx.y;
    const int hpg = (p.H + gridDim.z - 1) / gridDim.z;  // heads of this CTA: [h0, h1)
    const int h0 = blockIdx.z * hpg, h1 = min(p.H, h0 + hpg);
    pdl_wait();
    const int q0 = p.cu_seqlens[b];
    const int L = p.cu_seqlens[b + 1] - q0;
    if (L > p.max_len || L < 0 || static_cast<int64_t>(q0) + L > p.qrows) {
        if (tid == 0 && pg == 0) atomicOr(p.err, LLA_DEVERR_CONTEXT);
        return;
    }
    if (pg * kPT >= L || h0 >= h1) return;  // uniform, before any barrier
    const int nvalid = min(kPT, L - pg * kPT);
    int32_t blk = p.block_table[static_cast<int64_t>(b) * p.max_blocks + pg];
    if (blk < 0 || blk >= p.num_blocks) {
        if (tid == 0) atomicOr(p.err, LLA_DEVERR_BLOCK_ID);
        blk = 0;
    }
    if (tid == 0) {
        mbar_init(bar, 1);
        fence_mbar_init();
    }
    if (warp == 0) tmem_alloc(tslot, 128);
    // rotation of each token of the page at each pair's frequency, from exact turns
    for (int i = tid; i < 64 * 64; i += 128) {
        const int r = i >> 6, j = i & 63;
        const unsigned long long turns = static_cast<unsigned long long>(pg * kPT + r) * p.phi[j];
        const float tf = __uint2float_rn(static_cast<uint32_t>(turns >> 32)) * 2.3283064365386963e-10f;
        float sa, ca;
        sincospif(2.f * tf, &sa, &ca);
        tab[r * 65 + j] = make_float2(ca, sa);
    }
    // A of the mu step: a (1, 1) pair per token, then a zero granule
    for (int i = tid; i < 128; i += 128)
        reinterpret_cast<uint4 *>(sm + Z::oOnes)[i] = i < 64 ? make_uint4(0x3f803f80u, 0u, 0u, 0u) : make_uint4(0u, 0u, 0u, 0u);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tslot;
    const uint32_t base = smem_addr(sm);
    // epilogue geometry (16x256b fragments of the M = 64 accumulator): warp w holds tokens
    // 16w + lane/4 and 16w + lane/4 + 8; columns 8k + 2c and 8k + 2c + 1, c = lane % 4
    const int c = lane & 3;
    const int tok0 = 16 * warp + (lane >> 2);
    const uint32_t tq = tmem + (static_cast<uint32_t>(32 * warp) << 16);
    // W_up,t^K of head h (B: row e = dimension, K-major) and the page's K-plane of head h (A, as
    // stored), by cp.async; the (mu_hi, mu_lo) granule of head h before W
    auto stage = [&](int h) {
        const int64_t hl = (static_cast<int64_t>(h) * p.T + p.loop) * D;
        const char *W = static_cast<const char *>(p.w_up_k) + hl * RK * 2;
        for (int i = tid; i < D * Z::NG; i += 128) {
            const int e = i / Z::NG, g = i - e * Z::NG;
            cp_async16(sm + Z::oW + g * (D * 16) + e * 16, W + (static_cast<int64_t>(e) * RK + g * 8) * 2);
        }
        const char *K = p.pool + (static_cast<int64_t>(blk) * p.H + h) * p.head_page_bytes;
        for (int i = tid; i < Z::NG * 64; i += 128) cp_async16(sm + Z::oA + i * 16, K + i * 16);
        cp_async_commit();
        const float mu = p.mu_k ? p.mu_k[hl + tid] : 0.f;
        const __nv_bfloat16 hi = __float2bfloat16_rn(mu);
        const __nv_bfloat16 lo = __float2bfloat16_rn(mu - __bfloat162float(hi));
        *reinterpret_cast<uint4 *>(sm + Z::oB + tid * 16) =
            make_uint4(static_cast<uint32_t>(__bfloat16_as_ushort(hi)) |
                           (static_cast<uint32_t>(__bfloat16_as_ushort(lo)) << 16),
                       0u, 0u, 0u);
    };
    stage(h0);
    for (int h = h0; h < h1; ++h) {
        cp_async_wait_all();
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();
        if (tid == 0) {
            tc_fence_after();
#pragma unroll
            for (int st = 0; st < RK / 16; ++st)
                umma_bf16(tmem, umma_desc(base + Z::oA + st * 2048, 1024, 128),
                          umma_desc(base + Z::oW + st * 4096, 2048, 128), Z::IDESC, st > 0);
            // mu: the ones pair of every token against (mu_hi, mu_lo) of every dimension; the
            // second granules are zeros (A) and W_up,t^K (B, finite)
            umma_bf16(tmem, umma_desc(base + Z::oOnes, 1024, 128), umma_desc(base + Z::oB, 2048, 128),
                      Z::IDESC, true);
            umma_commit(bar);
        }
        {
            volatile int never = 0;
            mbar_wait(bar, (h - h0) & 1, &never, p.err);
        }
        tc_fence_after();
        // the MMA has read its operands: the next head's travel while this one's epilogue runs
        if (h + 1 < h1) stage(h + 1);
        uint32_t r0[32], r1[32];  // dimensions 0..63 (k = 0..7) and 64..127 (k = 8..15)
        tmem_ld16x256_x8_nowait(tq, r0);
        tmem_ld16x256_x8_nowait(tq + 64, r1);
        tmem_wait_ld(r0);
        tmem_wait_ld(r1);
        // rotate each token's pairs and write the page: dims (8k + 2c, +1) of token t at
        // granule k, byte 4c
        char *kout = p.krot + ((static_cast<int64_t>(b) * p.kpps + pg) * p.H + h) * (kPT * D * 2);
#pragma unroll
        for (int u = 0; u < 2; ++u) {
            const int t = tok0 + 8 * u;
            const float2 *tr = tab + t * 65;
            const bool ok = t < nvalid;
            float y[32];  // y[2k + e]: dimension 8k + 2c + e
            if (p.pairing == 0) {  // pairs (j, j + 64): k and k + 8
#pragma unroll
                for (int k = 0; k < 8; ++k)
#pragma unroll
                    for (int e = 0; e < 2; ++e) {
                        const float xa = __uint_as_float(r0[4 * k + 2 * u + e]);
                        const float xb = __uint_as_float(r1[4 * k + 2 * u + e]);
                        const float2 cs = tr[8 * k + 2 * c + e];
                        y[2 * k + e] = xa * cs.x - xb * cs.y;
                        y[2 * (k + 8) + e] = xa * cs.y + xb * cs.x;
                    }
            } else {  // pairs (2j, 2j + 1), j = 4k + c
#pragma unroll
                for (int k = 0; k < 16; ++k) {
                    const uint32_t *rr = k < 8 ? r0 : r1;
                    const int kk = k & 7;
                    const float xa = __uint_as_float(rr[4 * kk + 2 * u]);
                    const float xb = __uint_as_float(rr[4 * kk + 2 * u + 1]);
                    const float2 cs = tr[4 * k + c];
                    y[2 * k] = xa * cs.x - xb * cs.y;
                    y[2 * k + 1] = xa * cs.y + xb * cs.x;
                }
            }
#pragma unroll
            for (int k = 0; k < 16; ++k)
                *reinterpret_cast<uint32_t *>(kout + k * 1024 + t * 16 + c * 4) =
                    ok ? pack_bf16x2(y[2 * k], y[2 * k + 1]) : 0u;
        }
        // the page's queries of head h: rotated at their positions, scaled into the exp2 domain;
        // thread (r, hf) rotates pairs 32 hf .. 32 hf + 31 of query r
        {
            const int r = tid >> 1, hf = tid & 1;
            if (r < nvalid) {
                const int64_t qrow = (static_cast<int64_t>(q0) + pg * kPT + r) * p.H + h;
                const float2 *tr = tab + r * 65 + 32 * hf;
                const int es = p.io_bf16 ? 2 : 4;
                const char *qs = static_cast<const char *>(p.q) + qrow * D * es;
                char *qo = static_cast<char *>(p.qrot) + qrow * D * 2;
                float xa[32], xb[32];
                if (p.pairing == 0) {  // pairs (j, j + 64): two runs of 32
                    load32(qs + 32 * hf * es, p.io_bf16, xa);
                    load32(qs + (64 + 32 * hf) * es, p.io_bf16, xb);
#pragma unroll
                    for (int i = 0; i < 32; ++i) {
                        const float2 cs = tr[i];
                        const float a = xa[i], bb = xb[i];
                        xa[i] = (a * cs.x - bb * cs.y) * p.scale_log2;
                        xb[i] = (a * cs.y + bb * cs.x) * p.scale_log2;
                    }
                    store32_bf16(qo + 32 * hf * 2, xa);
                    store32_bf16(qo + (64 + 32 * hf) * 2, xb);
                } else {  // pairs (2j, 2j + 1): one run of 64
                    load32(qs + 64 * hf * es, p.io_bf16, xa);
                    load32(qs + (64 * hf + 32) * es, p.io_bf16, xb);
#pragma unroll
                    for (int i = 0; i < 32; ++i) {
                        const float2 cs = tr[i];
                        float *pr = i < 16 ? xa + 2 * i : xb + 2 * (i - 16);
                        const float a = pr[0], bb = pr[1];
                        pr[0] = (a * cs.x - bb * cs.y) * p.scale_log2;
                        pr[1] = (a * cs.y + bb * cs.x) * p.scale_log2;
                    }
                    store32_bf16(qo + 64 * hf * 2, xa);
                    store32_bf16(qo + (64 * hf + 32) * 2, xb);
                }
            }
        }
        tc_fence_before();
        __syncthreads();  // the operands and the accumulator may take the next head
        tc_fence_after();
    }
    pdl_trigger();
    if (warp == 0) tmem_dealloc(tmem, 128);
}

template <typename K, typename P>
lla_status launch_pf(K kern, dim3 grid, int threads, int smem, cudaStream_t stream, const P &prm) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = dim3(threads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (cudaLaunchKernelEx(&cfg, kern, prm) != cudaSuccess) return LLA_ERR_CUDA;
    return LLA_OK;
}

template <int RK, int RV, bool ROPE = false>
lla_status launch_tc(const PParams &prm, int nqt, int B, int H, cudaStream_t stream) {
    static DeviceOnce configured;
    if (raise_smem_limit(prefill_tc_kernel<RK, RV, ROPE>, PF<RK, RV, ROPE>::SMEM, configured) != LLA_OK) return LLA_ERR_CUDA;
    // the V-planes of every head page: [pages][64 tokens][r_v] bf16, one page = one head page
    CUtensorMap tv;
    const uint64_t dims[3] = {static_cast<uint64_t>(RV), static_cast<uint64_t>(kPT),
                              static_cast<uint64_t>(prm.num_blocks) * prm.H};
    const uint64_t strides[2] = {static_cast<uint64_t>(RV) * 2, static_cast<uint64_t>(prm.head_page_bytes)};
    const uint32_t box[3] = {64, kPT, 1};
    if (!encode_tmap_bf16(&tv, prm.pool + kPT * RK * 2, 3, dims, strides, box, true)) return LLA_ERR_CUDA;
    cudaLaunchConfig_t cfg = {};
    // x fastest: the tiles of one (sequence, head), longest first, run together and share its
    // pages in L2 (ordering the longest tiles of every head first was slower: 1.90 -> 2.17 ms)
    cfg.gridDim = dim3(nqt, B, H);
    cfg.blockDim = dim3(kPThreads);
    cfg.dynamicSmemBytes = PF<RK, RV, ROPE>::SMEM;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (cudaLaunchKernelEx(&cfg, prefill_tc_kernel<RK, RV, ROPE>, tv, prm) != cudaSuccess) return LLA_ERR_CUDA;
    return LLA_OK;
}

}  // namespace

lla_status launch_prefill(const PrefillArgs &a, cudaStream_t stream) {
    lla_status st = LLA_OK;
    unsigned *err = device_error_word(&st);
    if (st != LLA_OK) return st;
    const int es = a.storage_bf16 ? 2 : 4;
    const int hpb = static_cast<int>(head_page_bytes(a.r_k, a.r_v, es));
    if (a.B > 65535 || a.H > 65535) return LLA_ERR_UNSUPPORTED;
    // the tensor-core kernel addresses head pages with a 32-bit TMA coordinate
    if (a.storage_bf16 && a.d == 128 && a.num_blocks * a.H < (int64_t(1) << 31)) {
        PParams p = {};
        p.T = a.T; p.H = a.H; p.loop = a.loop; p.io_bf16 = a.io_bf16;
        p.scale_log2 = a.scale * kLog2e;
        p.w_up_k = a.w_up_k; p.w_up_v = a.w_up_v; p.mu_v = a.mu_v;
        p.pool = static_cast<const char *>(a.pool);
        p.num_blocks = a.num_blocks;
        p.head_page_bytes = hpb;
        p.block_bytes = static_cast<int64_t>(hpb) * a.H;
        p.block_table = a.block_table; p.max_blocks = a.max_blocks;
        p.cu_seqlens = a.cu_seqlens; p.B = a.B; p.max_len = a.max_len;
        p.q = a.q; p.out = a.out; p.err = err;
        const int nqt = (a.max_len + kBM - 1) / kBM;
#define LLA_PF(K, V) \
        if (a.r_k == K && a.r_v == V) return launch_tc<K, V>(p, nqt, a.B, a.H, stream);
        LLA_PF(96, 160)
        LLA_PF(192, 320)
        LLA_PF(128, 128)
#undef LLA_PF
    }
    GParams g = {};
    g.T = a.T; g.H = a.H; g.d = a.d; g.r_k = a.r_k; g.r_v = a.r_v; g.loop = a.loop;
    g.storage_bf16 = a.storage_bf16; g.io_bf16 = a.io_bf16;
    g.scale_log2 = a.scale * kLog2e;
    g.w_up_k = a.w_up_k; g.w_up_v = a.w_up_v; g.mu_v = a.mu_v;
    g.pool = static_cast<const char *>(a.pool);
    g.num_blocks = a.num_blocks;
    g.head_page_bytes = hpb;
    g.block_bytes = static_cast<int64_t>(hpb) * a.H;
    g.kplane_bytes = kPT * a.r_k * es;
    g.block_table = a.block_table; g.max_blocks = a.max_blocks;
    g.cu_seqlens = a.cu_seqlens; g.max_len = a.max_len;
    g.q = a.q; g.out = a.out; g.err = err;
    const int smem = (a.d + a.r_k + a.r_v + kGKeys + 32) * 4;
    return launch_pf(prefill_generic_kernel, dim3(a.max_len, a.B, a.H), kGThreads, smem, stream, g);
}


size_t prefill_rope_workspace_bytes(int B, int max_len, int H) {
    const size_t kpps = (static_cast<size_t>(max_len) + kPT - 1) / kPT;
    const size_t krot = static_cast<size_t>(B) * kpps * H * kPT * 128 * 2;
    const size_t qrot = static_cast<size_t>(B) * max_len * H * 128 * 2;
    return krot + qrot;
}

bool prefill_rope_supported(int es, int d, int r_k, int r_v) {
    return es == 2 && d == 128 &&
           ((r_k == 96 && r_v == 160) || (r_k == 192 && r_v == 320) || (r_k == 128 && r_v == 128));
}

namespace {
template <int RK>
lla_status launch_rebuild(const RParams &rp, int kpps, int B, cudaStream_t stream) {
    static DeviceOnce configured;
    if (raise_smem_limit(rope_rebuild_kernel<RK>, RB<RK>::SMEM, configured) != LLA_OK) return LLA_ERR_CUDA;
    // heads split over a few CTAs per page, so that more CTAs hide each other's load latency
    const int groups = rp.H >= 8 ? 4 : 1;
    return launch_pf(rope_rebuild_kernel<RK>, dim3(kpps, B, groups), 128, RB<RK>::SMEM, stream, rp);
}
}  // namespace

lla_status launch_prefill_rope(const PrefillArgs &a, double base, int pairing, void *workspace,
                               size_t workspace_bytes, cudaStream_t stream) {
    const int es = a.storage_bf16 ? 2 : 4;
    if (!prefill_rope_supported(es, a.d, a.r_k, a.r_v)) return LLA_ERR_UNSUPPORTED;
    if (a.B > 65535 || a.H > 65535 || a.num_blocks * a.H >= (int64_t(1) << 31)) return LLA_ERR_UNSUPPORTED;
    if (workspace_bytes < prefill_rope_workspace_bytes(a.B, a.max_len, a.H)) return LLA_ERR_WORKSPACE;
    lla_status st = LLA_OK;
    unsigned *err = device_error_word(&st);
    if (st != LLA_OK) return st;
    const int hpb = static_cast<int>(head_page_bytes(a.r_k, a.r_v, es));
    const int kpps = (a.max_len + kPT - 1) / kPT;
    char *krot = static_cast<char *>(workspace);
    void *qrot = krot + static_cast<size_t>(a.B) * kpps * a.H * kPT * 128 * 2;

    RParams r = {};
    r.T = a.T; r.H = a.H; r.loop = a.loop; r.io_bf16 = a.io_bf16; r.kpps = kpps; r.pairing = pairing;
    r.scale_log2 = a.scale * kLog2e;
    r.w_up_k = a.w_up_k; r.mu_k = a.mu_k;
    r.pool = static_cast<const char *>(a.pool); r.num_blocks = a.num_blocks;
    r.head_page_bytes = hpb;
    r.block_table = a.block_table; r.max_blocks = a.max_blocks;
    r.cu_seqlens = a.cu_seqlens; r.max_len = a.max_len;
    r.q = a.q; r.krot = krot; r.qrot = qrot; r.err = err;
    r.qrows = static_cast<int64_t>(a.B) * a.max_len;
    const double two_pi = 6.283185307179586476925286766559;
    for (int j = 0; j < 64; ++j)
        r.phi[j] = static_cast<unsigned long long>(ldexp(pow(base, -2.0 * j / a.d) / two_pi, 64));
    lla_status rs = LLA_ERR_UNSUPPORTED;
    if (a.r_k == 96) rs = launch_rebuild<96>(r, kpps, a.B, stream);
    else if (a.r_k == 192) rs = launch_rebuild<192>(r, kpps, a.B, stream);
    else if (a.r_k == 128) rs = launch_rebuild<128>(r, kpps, a.B, stream);
    if (rs != LLA_OK) return rs;

    PParams p = {};
    p.T = a.T; p.H = a.H; p.loop = a.loop; p.io_bf16 = a.io_bf16;
    p.scale_log2 = a.scale * kLog2e;
    p.w_up_k = a.w_up_k; p.w_up_v = a.w_up_v; p.mu_v = a.mu_v;
    p.pool = static_cast<const char *>(a.pool);
    p.num_blocks = a.num_blocks;
    p.head_page_bytes = hpb;
    p.block_bytes = static_cast<int64_t>(hpb) * a.H;
    p.block_table = a.block_table; p.max_blocks = a.max_blocks;
    p.cu_seqlens = a.cu_seqlens; p.B = a.B; p.max_len = a.max_len;
    p.q = a.q; p.out = a.out; p.err = err;
    p.krot = krot; p.qrot = qrot; p.kpps = kpps;
    p.qrows = static_cast<int64_t>(a.B) * a.max_len;
    const int nqt = (a.max_len + kBM - 1) / kBM;
    if (a.r_k == 96) return launch_tc<96, 160, true>(p, nqt, a.B, a.H, stream);
    if (a.r_k == 192) return launch_tc<192, 320, true>(p, nqt, a.B, a.H, stream);
    return launch_tc<128, 128, true>(p, nqt, a.B, a.H, stream);
}

}  // namespace lla
