// lla_decode_2d.cu -- decode over a latent page that several queries share, on the tensor cores:
//   * the LLA-2D cache (Sec. 3, "The LLA-2D variant (loop x head)"; App. J "Absorbed attention"
//     and "Per-head LLA versus LLA-2D at inference"): one latent pair per (token, layer) serves
//     every head, so the H queries of a sequence read the same page;
//   * the T loops of a per-head cache (Sec. 3, Eq. encode: one stacked code per (token, layer,
//     head) serves every loop), so the T loop queries of a (sequence, head) read the same page.
// A unit is what owns a page stream (a sequence for LLA-2D, a (sequence, head) pair for the
// loops) and a query is one of its NQ readers (a head, a loop).  Query n of a unit rebuilds its
// key and value as c W_up,n^T + mu_n.  Absorbed query by query (App. J), each page of 64 tokens
// is a small dense contraction:
//   q~_n = W_up,n^K^T q_n,  beta_n = q_n . mu^K_n                            (absorb kernel)
//   S^T [64 x 2NQ]  = C_k [64 x r_k] [Q~_hi; Q~_lo]^T     s_n,i = scale (q~_n . c_k,i + beta_n)
//   O^T [r_v x 16] += C_v^T [r_v x 64] P^T                online softmax over tokens per query
//   o_n = (W_up,n^V o~_n + l_n mu^V_n + p_cur v_cur,n) / (l_n + p_cur)      (finish kernel)
// Three launches on the caller's stream, chained by programmatic dependent launch:
//   absorb2d_kernel   q~ (fp32, scaled into the exp2 domain) and beta of every (unit, query),
//                     the page prefix sums of the units and the length checks
//   attn2d_kernel     one CTA per SM.  The units' pages, in unit order, are split evenly over
//                     the CTAs; a CTA takes its pages as runs (its part of one unit) and writes
//                     per run the partial (maximum, sum, O^T) of every query.
//                       warp 0     producer: the K-plane of a page by one bulk copy, its V-plane
//                                  by TMA boxes of 64 columns with 128-byte swizzle
//                       warp 1     S^T issuer and TMEM owner: M = 64 tokens, N = the q~ parts
//                                  of the NQ queries (q~ as a bf16 high part and remainders, so
//                                  that the scores see q~ to 16 or 24 significant bits), K = r_k
//                                  (a rank that is not a multiple of 16 padded with zero
//                                  columns); it runs up to two pages ahead of the softmax
//                       warp 6     O^T issuer: M = 128 latent rows per chunk, N = 16 (the p
//                                  parts of the queries, padded with zero rows of P^T), K = 64
//                                  tokens; the swizzled V-plane is an MN-major A operand.  Two
//                                  issuing threads, because an MMA takes its issuing thread tens
//                                  of cycles
//                       warps 2-5  per page: the scores of 16 tokens per warp, the maxima over
//                                  the page per query, P^T as a bf16 operand, the lazy O^T
//                                  rescale; per run: the partial out to the workspace
//   finish2d_kernel   per (query slice, up to 8 units, and for small batches or wide latents a
//                     quarter of the output rows): merges the runs of each unit, adds the pass-1
//                     current token, and applies W_up,n^V once for those units
//   attn2d_big_kernel replaces attn2d_kernel for latents wider than a page stage ((1152, 1920)):
//                     pages stream as K-plane column chunks and V-plane row chunks
// Storage bf16, d = 128; accumulators fp32 in TMEM.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstring>

#include "lla_device.cuh"
#include "lla_internal.h"
#include "lla_tcgen05.cuh"
#include "lla_tmap.h"
#include "lla_units.cuh"

namespace lla {
namespace {

constexpr int kPT = 64;          // tokens per page
constexpr int kD = 128;          // head width
constexpr int kNQ = 16;          // O^T columns: the queries of a unit, padded
constexpr int kT2 = 224;         // threads of the attention kernel
constexpr int kSm0 = 64;         // first softmax thread
constexpr int kPvWarp = 6;       // issuer of the O^T products
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kRescaleLog2 = 8.f;  // rescale O^T only when a query's maximum grows by more
constexpr int kSmemCap = 227 * 1024;
constexpr int kFinishSeqs = 8;   // most units per finish CTA (4 for latents wider than 512)
constexpr int kMaxGrid = 256;    // attention CTAs (the runs of one unit fit one finish CTA)

__host__ __device__ constexpr int finish_seqs(int rv) { return rv > 512 ? 4 : kFinishSeqs; }
// Row slices of the output projection per finish CTA, for latents wider than 160: the d output
// rows of a head split over 4 CTAs, so that each reads a quarter of W_up,t,h^V (four threads per
// row reading it in 64-byte runs) for all of its sequences, instead of every CTA reading all of
// it.  Latents wider than 512 always take them; narrower ones only when the batch leaves SMs
// idle (a large batch keeps its finish to one wave of CTAs).
__host__ __device__ constexpr int finish_slices(int rv) { return rv > 160 ? 4 : 1; }

// Shared-memory plan of the attention kernel for ranks (RK, RV) and NQ query slots per unit
// (16: the heads of an LLA-2D sequence; 4: the loops of a per-head (sequence, head)).  Offsets
// from a 1024-byte aligned base (128-byte swizzle atoms of the V stages).
template <int RK, int RV, int NQ>
struct Z2 {
    static constexpr int RKX = (RK + 15) / 16 * 16;     // score contraction, zero-padded
    // q~ and p as sums of bf16 parts, each the rounding of what the earlier parts leave: with
    // 16 query slots q~ in two parts (about 16 significant bits) and p in one; with 4 slots the
    // MMA's padding columns carry three parts of each (24 bits, the precision of fp32)
    static constexpr int QS = NQ == 4 ? 3 : 2;
    static constexpr int PSPL = NQ == 4 ? 3 : 1;
    static constexpr int NS = (QS * NQ + 7) / 8 * 8;    // score MMA N: the q~ parts, padded
    static constexpr int NQM = NQ;                      // queries of a unit in the workspace
    static constexpr int NCH = (RV + 127) / 128;        // 128-row chunks of O^T
    static constexpr int NBOX = (RV + 63) / 64;         // TMA boxes a V-plane loads
    static constexpr int BOX = kPT * 128;               // one box: 64 rows x 128 bytes
    static constexpr int KPLANE = kPT * RK * 2;         // bytes of a K-plane copy
    static constexpr int KPAGE = kPT * RKX * 2;         // K stage: the copy, then zero granules
    static constexpr int VPAGE = NCH * 2 * BOX;         // two boxes per chunk, loaded or zero
    static constexpr int VBYTES = NBOX * BOX;
    static constexpr int QB = NS * RKX * 2;             // [Q~_hi; Q~_lo] operand
    static constexpr int PBUF = kPT * kNQ * 2;          // P^T operand (one of two)
    static constexpr int RED = 1024;                    // maxima, sums, beta
    static constexpr int NBAR = 32;
    static constexpr int FIXED = QB + 2 * PBUF + RED + NBAR * 8;
    static constexpr int ST0 = (kSmemCap - 1024 - FIXED) / (KPAGE + VPAGE);
    static constexpr int ST = ST0 > 4 ? 4 : ST0;
    static constexpr int oV = 0;
    static constexpr int oK = oV + ST * VPAGE;
    static constexpr int oQ = oK + ST * KPAGE;
    static constexpr int oP = oQ + QB;
    static constexpr int oRed = oP + 2 * PBUF;
    static constexpr int oBar = oRed + RED;
    static constexpr int SMEM = 1024 + oBar + NBAR * 8;
    // TMEM columns: S^T double buffer [0, 2 NS), O^T chunks [2 NS, 2 NS + 16 NCH)
    static constexpr uint32_t TM_S = 0, TM_O = 2 * NS, TM_COLS = 128;
    static constexpr uint32_t IDESC_S = umma_idesc_bf16(64, NS, 0, 0);
    static constexpr uint32_t IDESC_O = umma_idesc_bf16(128, kNQ, 1, 0);
    // a run partial: O^T of each query ([NQM][RV]), then 16 maxima and 16 sums
    static constexpr int PSTRIDE = NQM * RV + 2 * kNQ;
    static constexpr int PO_M = NQM * RV, PO_L = NQM * RV + kNQ;
    static_assert(NQ == 4 || NQ == 16, "query slots");
    static_assert(PSPL * NQ <= kNQ, "p parts in the O^T columns");
    static_assert(RK % 8 == 0 && RV % 8 == 0 && NCH <= 4, "ranks in 16-byte granules");
    static_assert(ST >= 2, "pipeline depth");
    static_assert(SMEM <= kSmemCap, "shared memory");
    static_assert(TM_O + NCH * kNQ <= TM_COLS, "TMEM columns");
};

// barrier indices
enum {
    bKfull = 0 /* [4] */, bKempty = 4, bVfull = 8, bVempty = 12,
    bSfull = 16 /* [2] */, bSfree = 18, bPfull = 20, bPfree = 22,
    bOfree = 25, bQready = 26, bQfree = 27, bAbort = 28, bTslot = 29
};

// Unit u of the batch: sequence u / hu, head u % hu of a per-head cache (hu = H for the loops,
// 1 for LLA-2D, whose one page per block serves every head).  Query n of unit u:
//   LLA-2D  head n of sequence u at loop `loop`: weights [T][H][d][r] at (loop, n), io row (u H + n)
//   loops   loop n of (sequence b, head h):      weights [H][T][d][r] at (h, n),
//                                                io row ((n B + b) H + h)
// (mu alike: [T*H*d] rows (t, h, e) for LLA-2D, [H][T*d] for the per-head codec).
struct A2Params {
    int T, H, loop, io_bf16, pass1, B, max_ctx, max_blocks;
    int loops;           // 0: LLA-2D, 1: the loops of a per-head cache
    int hu;              // units per sequence
    float scale_log2;
    const void *w_up_k;  // LLA-2D [T][H][d][r_k], per-head [H][T][d][r_k]
    const float *mu_k;   // LLA-2D [T*H*d], per-head [H][T*d], or NULL
    const void *q;       // io rows of d
    const int32_t *context_lens;
    float *qt;           // [units][NQM][RKX]: q~ * scale * log2 e, zero past r_k
    float *beta;         // [units][NQM]: beta * scale * log2 e
    int *pstart;         // [units + 1]: first global page of each unit
    unsigned *err;
};

struct T2Params {
    int nq;   // queries of a unit
    int U;    // units
    int hu;   // units per sequence
    const char *pool;
    int64_t num_blocks, page_bytes;
    const int32_t *block_table;
    int max_blocks;
    const int32_t *context_lens;
    const float *qt;
    const float *beta;
    const int *pstart;
    float *part;  // [U + grid][PSTRIDE]: run (unit u, CTA c) at slot u + c
    unsigned *err;
};

struct F2Params {
    int T, H, loop, io_bf16, B, grid;
    int loops, hu, U;
    int spb;  // units per CTA (1 .. 8)
    float scale_log2;
    const void *w_up_v;  // LLA-2D [T][H][d][r_v], per-head [H][T][d][r_v], bf16
    const float *mu_v;   // LLA-2D [T*H*d], per-head [H][T*d], or NULL
    const void *q, *cur_k, *cur_v;
    void *out;
    const int *pstart;
    const float *part;
};

// ------------------------------------------------------------------------- absorb kernel

// One CTA: the page prefix sums of the units with the length checks (once per sequence); an
// invalid length counts as an empty sequence.
__device__ void page_prefix(const A2Params &p) {
    __shared__ int wsum[8];
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int U = p.B * p.hu;
    const int per = (U + 255) / 256;  // units of this thread: [tid per, (tid + 1) per)
    const int limit = min(p.max_ctx, p.max_blocks * kPT);
    auto pages = [&](int u, bool flag) {
        const int L = p.context_lens[u / p.hu];
        flag = flag && u % p.hu == 0;
        if (L < 0 || L > limit) {
            if (flag) atomicOr(p.err, LLA_DEVERR_CONTEXT);
            return 0;
        }
        if (flag && !p.pass1 && L == 0) atomicOr(p.err, LLA_DEVERR_EMPTY_PASS2);
        return (L + kPT - 1) / kPT;
    };
    int tot = 0;
    for (int u = tid * per; u < min(U, (tid + 1) * per); ++u) tot += pages(u, true);
    int x = tot;  // inclusive scan over the warp
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
    for (int u = tid * per; u < min(U, (tid + 1) * per); ++u) {
        p.pstart[u] = ex;
        ex += pages(u, false);
    }
    if (tid == blockDim.x - 1) p.pstart[U] = pre + x;
}

// Grid (weight slices, RKX / 32, ceil(B / 16)), 256 threads = 32 columns x 8 slices of 16 rows:
// q~ of 32 columns of one weight slice for 16 sequences, every weight load of a thread in flight
// at once; beta by the CTAs of the first column chunk.  Slice w is (loop, head w) for LLA-2D and
// (loop w / H, head w % H) for the loops (th: its row block of d in W_up and mu); columns
// r_k .. RKX - 1 of q~ are written as zeros.
template <int RK, int NQ>
__global__ void __launch_bounds__(256) absorb2d_kernel(const A2Params p) {
    constexpr int RKX = (RK + 15) / 16 * 16;
    __shared__ float qs[16][kD];
    __shared__ float red[8][16][33];
    const int w = blockIdx.x, j0 = blockIdx.y * 32, b0 = blockIdx.z * 16, tid = threadIdx.x;
    const int warp = tid >> 5, lane = tid & 31;
    const int nb = min(16, p.B - b0);
    const int t = p.loops ? w / p.H : p.loop, h = p.loops ? w - t * p.H : w;
    const int64_t th = p.loops ? static_cast<int64_t>(h) * p.T + t : static_cast<int64_t>(t) * p.H + h;
    const int n = p.loops ? t : h;  // the query of (sequence b, slice w) within its unit
    auto unit = [&](int b) { return p.loops ? b * p.H + h : b; };
    auto iorow = [&](int b) { return ((p.loops ? static_cast<int64_t>(t) * p.B : 0) + b) * p.H + h; };
    const int col = j0 + lane;
    // this thread's 16 weights (column j0 + lane, rows 16 warp .. 16 warp + 15): inputs of the
    // call, loaded before the wait on the previous kernel
    const uint16_t *W = static_cast<const uint16_t *>(p.w_up_k) + th * kD * RK + col;
    float wv[16];
#pragma unroll
    for (int u = 0; u < 16; ++u) wv[u] = col < RK ? bf_to_f(W[(warp * 16 + u) * RK]) : 0.f;
    pdl_wait();  // the queries may come from the previous kernel; the workspace is free after it
    if (blockIdx.x == 0 && blockIdx.y == 0 && blockIdx.z == 0) page_prefix(p);
    for (int i = tid; i < 16 * kD; i += 256) {
        const int bi = i >> 7, e = i & (kD - 1);
        qs[bi][e] = bi < nb ? load_elem(p.q, iorow(b0 + bi) * kD + e, p.io_bf16) : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int bi = 0; bi < 16; ++bi) {
        float a = 0.f;
#pragma unroll
        for (int u = 0; u < 16; ++u) a = fmaf(wv[u], qs[bi][warp * 16 + u], a);
        red[warp][bi][lane] = a;
    }
    __syncthreads();
    for (int o = tid; o < 16 * 32; o += 256) {
        const int bi = o >> 5, c = o & 31;
        float a = 0.f;
#pragma unroll
        for (int sl = 0; sl < 8; ++sl) a += red[sl][bi][c];
        if (bi < nb && j0 + c < RKX)
            p.qt[(static_cast<int64_t>(unit(b0 + bi)) * NQ + n) * RKX + j0 + c] = j0 + c < RK ? a * p.scale_log2 : 0.f;
    }
    if (blockIdx.y == 0) {
        // beta_n = q_n . mu^K_n: warp w takes sequences w and w + 8
        for (int bi = warp; bi < nb; bi += 8) {
            float s = 0.f;
            if (p.mu_k)
                for (int e = lane; e < kD; e += 32) s = fmaf(qs[bi][e], p.mu_k[th * kD + e], s);
            s = warp_sum(s);
            if (lane == 0) p.beta[static_cast<int64_t>(unit(b0 + bi)) * NQ + n] = s * p.scale_log2;
        }
    }
    // (triggering the attention kernel's launch right after the wait, so that its set-up could
    // overlap this kernel where their CTAs fit one SM, gained 2 % at rho = 4 and lost 10 % on the
    // Ouro-2.6B batch)
    __syncthreads();
    pdl_trigger();
}

// ------------------------------------------------------------------------- attention kernel

// First unit with pages at or after global page g0: the last u with pstart[u] <= g0.
__device__ __forceinline__ int first_unit(const int *pstart, int U, int g0) {
    int lo = 0, hi = U - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (pstart[mid] <= g0) lo = mid;
        else hi = mid - 1;
    }
    return lo;
}

template <int N>
__device__ __forceinline__ void tmem_ld_cols(uint32_t taddr, float (&v)[N]) {
    static_assert(N == 16 || N == 32, "score columns");
    if constexpr (N == 16) tmem_ld16(taddr, v);
    else tmem_ld32(taddr, v);
}

// The K bf16 parts of v: part 0 = bf16(v), part k = bf16 of what parts 0 .. k-1 leave (each
// difference is exact in fp32).
template <int K>
__device__ __forceinline__ void bf16_parts(float v, float (&part)[K]) {
#pragma unroll
    for (int k = 0; k < K; ++k) {
        part[k] = __bfloat162float(__float2bfloat16_rn(v));
        v -= part[k];
    }
}

template <int RK, int RV, int NQ>
__global__ void __launch_bounds__(kT2, 1)
    attn2d_kernel(const __grid_constant__ CUtensorMap tv, const T2Params p) {
    using Z = Z2<RK, RV, NQ>;
    extern __shared__ __align__(1024) char sm_raw[];
    char *sm = reinterpret_cast<char *>((reinterpret_cast<uintptr_t>(sm_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    uint64_t *bar = reinterpret_cast<uint64_t *>(sm + Z::oBar);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(bar + bAbort);
    uint32_t *tslot = reinterpret_cast<uint32_t *>(bar + bTslot);
    float *red = reinterpret_cast<float *>(sm + Z::oRed);  // [2 pages][4 warps][16] maxima
    float *lsum = red + 128;                                // [4 warps][16] run sums
    float *betas = lsum + 64;                               // [16]
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int G = gridDim.x, c = blockIdx.x;

    if (tid == 0) {
        for (int s = 0; s < Z::ST; ++s) {
            mbar_init(&bar[bKfull + s], 1);
            mbar_init(&bar[bKempty + s], 1);
            mbar_init(&bar[bVfull + s], 1);
            mbar_init(&bar[bVempty + s], 1);
        }
        for (int s = 0; s < 2; ++s) {
            mbar_init(&bar[bSfull + s], 1);
            mbar_init(&bar[bSfree + s], 128);
            mbar_init(&bar[bPfull + s], 128);
            mbar_init(&bar[bPfree + s], 1);
        }
        mbar_init(&bar[bOfree], 128);
        mbar_init(&bar[bQready], 128);
        mbar_init(&bar[bQfree], 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 1) tmem_alloc(tslot, Z::TM_COLS);
    // operand bytes that no copy writes stay zero: the V boxes past r_v of a last chunk, the K
    // granules past r_k (against zero q~ columns), and the P^T rows of absent queries
    if constexpr (Z::NCH * 2 > Z::NBOX) {
        for (int s = 0; s < Z::ST; ++s)
            for (int a = Z::NBOX; a < Z::NCH * 2; ++a)
                for (int i = tid; i < Z::BOX / 16; i += kT2)
                    reinterpret_cast<uint4 *>(sm + Z::oV + s * Z::VPAGE + a * Z::BOX)[i] = make_uint4(0, 0, 0, 0);
    }
    if constexpr (Z::KPAGE > Z::KPLANE) {
        for (int s = 0; s < Z::ST; ++s)
            for (int i = tid; i < (Z::KPAGE - Z::KPLANE) / 16; i += kT2)
                reinterpret_cast<uint4 *>(sm + Z::oK + s * Z::KPAGE + Z::KPLANE)[i] = make_uint4(0, 0, 0, 0);
    }
    if constexpr (Z::PSPL * NQ < kNQ) {
        for (int i = tid; i < 2 * Z::PBUF / 16; i += kT2)
            reinterpret_cast<uint4 *>(sm + Z::oP)[i] = make_uint4(0, 0, 0, 0);
    }
    if constexpr (Z::QS * NQ < Z::NS) {  // the padding rows of the q~ operand
        for (int i = tid; i < Z::QB / 16; i += kT2)
            reinterpret_cast<uint4 *>(sm + Z::oQ)[i] = make_uint4(0, 0, 0, 0);
    }
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tslot;
    pdl_wait();  // q~, beta and the page prefix sums come from the absorb kernel

    const int NP = p.pstart[p.U];
    const int g0 = page_lo(c, NP, G), g1 = page_lo(c + 1, NP, G);
    const int ufirst = g0 < g1 ? first_unit(p.pstart, p.U, g0) : p.U;

    if (warp == 0) {
        // ------------------------------------------------------------------------- producer
        if (lane == 0) {
            // after a failed wait (or once the abort flag is up) no further copy is issued, so no
            // full barrier receives a second arrival in one phase; itk / itv count the K and V
            // rounds issued, and the last ST of each are awaited below
            const uint64_t pol = policy_evict_first();
            int itk = 0, itv = 0;
            bool stop = false;
            for (int u = ufirst; u < p.U && !stop; ++u) {
                const int s0 = p.pstart[u], s1 = p.pstart[u + 1];
                if (s0 >= g1) break;
                const int pa = max(g0, s0) - s0, pe = min(g1, s1) - s0;
                const int b = u / p.hu, hh = u - b * p.hu;
                const int32_t *bt = p.block_table + static_cast<int64_t>(b) * p.max_blocks;
                for (int pg = pa; pg < pe; ++pg) {
                    const int it = itk;
                    const int st = it % Z::ST;
                    const uint32_t ph = (it / Z::ST) & 1;
                    int32_t blk = bt[pg];
                    if (blk < 0 || blk >= p.num_blocks) {
                        atomicOr(p.err, LLA_DEVERR_BLOCK_ID);
                        blk = 0;
                    }
                    const int64_t page = static_cast<int64_t>(blk) * p.hu + hh;
                    if (!mbar_wait(&bar[bKempty + st], ph ^ 1u, abort_flag, p.err) || *abort_flag) {
                        stop = true;
                        break;
                    }
                    mbar_arrive_expect_tx(&bar[bKfull + st], Z::KPLANE);
                    char *ks = sm + Z::oK + st * Z::KPAGE;
                    bulk_g2s(ks, p.pool + page * p.page_bytes, Z::KPLANE, &bar[bKfull + st], pol);
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
        }
        __syncwarp();
    } else if (warp == 1) {
        // ---------------------------------------------------------------- S^T issuer
        // (an MMA takes its issuing thread tens of cycles: the score and value products of a
        // page are issued by two threads, each committing only its own products)
        if (lane == 0) {
            const uint32_t base = smem_addr(sm);
            const uint64_t dq = umma_desc(base + Z::oQ, Z::NS * 16, 128);
            const uint64_t dk0 = umma_desc(base + Z::oK, kPT * 16, 128);
            int it = 0, r = 0;
            for (int u = ufirst; u < p.U; ++u) {
                const int s0 = p.pstart[u], s1 = p.pstart[u + 1];
                if (s0 >= g1) break;
                const int n = min(g1, s1) - max(g0, s0);
                if (n <= 0) continue;
                mbar_wait(&bar[bQready], r & 1, abort_flag, p.err);
                tc_fence_after();
                for (int k = 0; k < n; ++k, ++it) {
                    const int s = it & 1, st = it % Z::ST;
                    mbar_wait(&bar[bKfull + st], (it / Z::ST) & 1, abort_flag, p.err);
                    if (it >= 2) mbar_wait(&bar[bSfree + s], ((it - 2) >> 1) & 1, abort_flag, p.err);
                    tc_fence_after();
                    const uint64_t dk = dk0 + static_cast<uint64_t>((st * Z::KPAGE) >> 4);
#pragma unroll
                    for (int ks = 0; ks < Z::RKX / 16; ++ks)
                        umma_bf16(tmem + Z::TM_S + s * Z::NS, dk + ks * ((2 * kPT * 16) >> 4),
                                  dq + ks * ((2 * Z::NS * 16) >> 4), Z::IDESC_S, ks > 0);
                    umma_commit(&bar[bSfull + s]);
                    umma_commit(&bar[bKempty + st]);
                    if (k == n - 1) umma_commit(&bar[bQfree]);
                }
                ++r;
            }
            // every product has completed before TMEM is released, even after an abort (when the
            // softmax warps stop waiting for them): the last commit on each S^T buffer
            volatile int never = 0;
            for (int j = max(0, it - 2); j < it; ++j)
                mbar_wait(&bar[bSfull + (j & 1)], (j >> 1) & 1, &never, p.err);
        }
        __syncwarp();
    } else if (warp == kPvWarp) {
        // ---------------------------------------------------------------- O^T issuer
        if (lane == 0) {
            const uint32_t base = smem_addr(sm);
            const uint64_t dp0 = umma_desc(base + Z::oP, kNQ * 16, 128);
            const uint64_t dv0 = umma_desc_sw128_mn(base + Z::oV, Z::BOX);
            int it = 0, r = 0;
            for (int u = ufirst; u < p.U; ++u) {
                const int s0 = p.pstart[u], s1 = p.pstart[u + 1];
                if (s0 >= g1) break;
                const int n = min(g1, s1) - max(g0, s0);
                if (n <= 0) continue;
                for (int k = 0; k < n; ++k, ++it) {
                    // O^T += C_v^T P^T for page it (the first page of run r zeroes O^T, once the
                    // softmax warps have read run r - 1's)
                    const int s = it & 1, st = it % Z::ST;
                    mbar_wait(&bar[bPfull + s], (it >> 1) & 1, abort_flag, p.err);
                    mbar_wait(&bar[bVfull + st], (it / Z::ST) & 1, abort_flag, p.err);
                    if (k == 0 && r > 0) mbar_wait(&bar[bOfree], (r - 1) & 1, abort_flag, p.err);
                    tc_fence_after();
                    const uint64_t dv = dv0 + static_cast<uint64_t>((st * Z::VPAGE) >> 4);
                    const uint64_t dp = dp0 + static_cast<uint64_t>((s * Z::PBUF) >> 4);
#pragma unroll
                    for (int ch = 0; ch < Z::NCH; ++ch)
#pragma unroll
                        for (int ks = 0; ks < kPT / 16; ++ks)
                            umma_bf16(tmem + Z::TM_O + ch * kNQ, dv + ((ch * 2 * Z::BOX + ks * 2048) >> 4),
                                      dp + ks * ((2 * kNQ * 16) >> 4), Z::IDESC_O, k > 0 || ks > 0);
                    umma_commit(&bar[bVempty + st]);
                    umma_commit(&bar[bPfree + s]);  // also: O^T holds pages up to it
                }
                ++r;
            }
            // every product has completed before TMEM is released, even after an abort (the last
            // product's completion on its P buffer; the one before on the other buffer had
            // completed before the softmax released the last page)
            if (it > 0) {
                volatile int never = 0;
                mbar_wait(&bar[bPfree + ((it - 1) & 1)], ((it - 1) >> 1) & 1, &never, p.err);
            }
        }
        __syncwarp();
    } else {
        // --------------------------------------------------------------- softmax warps 2-5
        const int q4 = warp & 3;  // TMEM lane quarter
        const uint32_t tl = tmem + (static_cast<uint32_t>(32 * q4) << 16);
        const int st_tid = tid - kSm0;
        const int tok = 16 * q4 + lane;  // the token of this lane in the M = 64 layout (lane < 16)
        int it = 0, r = 0;
        for (int u = ufirst; u < p.U; ++u) {
            const int s0 = p.pstart[u], s1 = p.pstart[u + 1];
            if (s0 >= g1) break;
            const int pa = max(g0, s0) - s0, pe = min(g1, s1) - s0;
            if (pe <= pa) continue;
            const int L = p.context_lens[u / p.hu];
            // q~ of the unit as a K-major operand of NS rows: row k NQ + n = bf16 part k of q~_n,
            // granule g of row n at g*(NS * 16) + n*16 (rows past QS NQ stay zero); and beta
            if (r > 0) mbar_wait(&bar[bQfree], (r - 1) & 1, abort_flag, p.err);
            {
                const float4 *src = reinterpret_cast<const float4 *>(p.qt + static_cast<int64_t>(u) * Z::NQM * Z::RKX);
                for (int i = st_tid; i < NQ * (Z::RKX / 8); i += 128) {
                    const int n = i / (Z::RKX / 8), g = i - n * (Z::RKX / 8);
                    float pt[Z::QS][8];
#pragma unroll
                    for (int k = 0; k < Z::QS; ++k)
#pragma unroll
                        for (int e = 0; e < 8; ++e) pt[k][e] = 0.f;
                    if (n < p.nq) {
                        const float4 a = src[2 * i], c4 = src[2 * i + 1];
                        const float v[8] = {a.x, a.y, a.z, a.w, c4.x, c4.y, c4.z, c4.w};
#pragma unroll
                        for (int e = 0; e < 8; ++e) {
                            float pe[Z::QS];
                            bf16_parts(v[e], pe);
#pragma unroll
                            for (int k = 0; k < Z::QS; ++k) pt[k][e] = pe[k];
                        }
                    }
                    char *dq = sm + Z::oQ + g * (Z::NS * 16);
#pragma unroll
                    for (int k = 0; k < Z::QS; ++k)
                        *reinterpret_cast<uint4 *>(dq + (k * NQ + n) * 16) =
                            make_uint4(pack_bf16x2(pt[k][0], pt[k][1]), pack_bf16x2(pt[k][2], pt[k][3]),
                                       pack_bf16x2(pt[k][4], pt[k][5]), pack_bf16x2(pt[k][6], pt[k][7]));
                }
                if (st_tid < NQ) betas[st_tid] = st_tid < p.nq ? p.beta[static_cast<int64_t>(u) * Z::NQM + st_tid] : 0.f;
            }
            fence_proxy_async_smem();
            mbar_arrive(&bar[bQready]);
            named_bar_sync(1, 128);  // beta is visible
            float m[NQ], acc[NQ];
#pragma unroll
            for (int n = 0; n < NQ; ++n) {
                m[n] = -INFINITY;
                acc[n] = 0.f;
            }
            const int nps = pe - pa;
            for (int k = 0; k < nps; ++k, ++it) {
                const int s = it & 1, st = it % Z::ST;
                const int tok0 = (pa + k) * kPT;
                mbar_wait(&bar[bSfull + s], (it >> 1) & 1, abort_flag, p.err);
                tc_fence_after();
                float x2[Z::NS], x[NQ];
                tmem_ld_cols(tl + Z::TM_S + s * Z::NS, x2);
                tc_fence_before();
                mbar_arrive(&bar[bSfree + s]);
                const bool valid = lane < 16 && tok0 + tok < L;
#pragma unroll
                for (int n = 0; n < NQ; ++n) {
                    float sn = x2[n];
#pragma unroll
                    for (int k = 1; k < Z::QS; ++k) sn += x2[k * NQ + n];
                    x[n] = valid ? sn + betas[n] : -INFINITY;
                }
                // per-query maxima over the page: 16 tokens per warp, then the 4 warps
                float mx[NQ];
#pragma unroll
                for (int n = 0; n < NQ; ++n) mx[n] = x[n];
#pragma unroll
                for (int o = 8; o >= 1; o >>= 1)
#pragma unroll
                    for (int n = 0; n < NQ; ++n) mx[n] = fmaxf(mx[n], __shfl_xor_sync(0xffffffffu, mx[n], o));
                float *rp = red + s * 64;
                if (lane == 0) {
#pragma unroll
                    for (int n = 0; n < NQ; n += 4)
                        *reinterpret_cast<float4 *>(rp + q4 * 16 + n) = make_float4(mx[n], mx[n + 1], mx[n + 2], mx[n + 3]);
                }
                named_bar_sync(1, 128);
                bool any = false;
                float f[NQ];
#pragma unroll
                for (int n = 0; n < NQ; n += 4) {
                    float4 a = *reinterpret_cast<const float4 *>(rp + n);
#pragma unroll
                    for (int w = 1; w < 4; ++w) {
                        const float4 bb = *reinterpret_cast<const float4 *>(rp + w * 16 + n);
                        a = make_float4(fmaxf(a.x, bb.x), fmaxf(a.y, bb.y), fmaxf(a.z, bb.z), fmaxf(a.w, bb.w));
                    }
                    const float pm[4] = {a.x, a.y, a.z, a.w};
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const float mn = fmaxf(m[n + e], pm[e]);
                        const bool need = mn > m[n + e] + kRescaleLog2;  // also the first page
                        f[n + e] = need ? ex2_approx(m[n + e] - mn) : 1.f;
                        if (need) {
                            acc[n + e] *= f[n + e];
                            m[n + e] = mn;
                            any = true;
                        }
                    }
                }
                if (any && k > 0) {
                    // O^T holds pages up to it - 1 of this run (the product of page it - 1 has
                    // released its P buffer; the one of page it - 2 had released the other before
                    // this warp wrote page it - 1, so the parity test cannot pass a phase early):
                    // scale query n's columns by f[n]
                    mbar_wait(&bar[bPfree + ((it - 1) & 1)], ((it - 1) >> 1) & 1, abort_flag, p.err);
                    tc_fence_after();
#pragma unroll
                    for (int ch = 0; ch < Z::NCH; ++ch) {
                        float o[kNQ];
                        tmem_ld16(tl + Z::TM_O + ch * kNQ, o);
#pragma unroll
                        for (int k = 0; k < Z::PSPL; ++k)
#pragma unroll
                            for (int n = 0; n < NQ; ++n) o[k * NQ + n] *= f[n];
                        tmem_st16(tl + Z::TM_O + ch * kNQ, o);
                    }
                }
                float pv[NQ];
#pragma unroll
                for (int n = 0; n < NQ; ++n) {
                    pv[n] = ex2_approx(x[n] - m[n]);
                    acc[n] += pv[n];
                }
                if (it >= 2) mbar_wait(&bar[bPfree + s], ((it - 2) >> 1) & 1, abort_flag, p.err);
                if (lane < 16) {
                    // P^T as a K-major operand: row k NQ + n = bf16 part k of query n's p, tokens
                    // 8g .. 8g + 7 at g*256 + row*16
                    char *pp = sm + Z::oP + s * Z::PBUF + (tok >> 3) * (kNQ * 16) + (tok & 7) * 2;
#pragma unroll
                    for (int n = 0; n < NQ; ++n) {
                        float pe[Z::PSPL];
                        bf16_parts(pv[n], pe);
#pragma unroll
                        for (int k = 0; k < Z::PSPL; ++k)
                            *reinterpret_cast<uint16_t *>(pp + (k * NQ + n) * 16) =
                                __bfloat16_as_ushort(__float2bfloat16_rn(pe[k]));
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
            // the run's partial: maxima, sums over its tokens, and O^T (complete once the last
            // page's product has released its P buffer)
            mbar_wait(&bar[bPfree + ((it - 1) & 1)], ((it - 1) >> 1) & 1, abort_flag, p.err);
            tc_fence_after();
#pragma unroll
            for (int o = 8; o >= 1; o >>= 1)
#pragma unroll
                for (int n = 0; n < NQ; ++n) acc[n] += __shfl_xor_sync(0xffffffffu, acc[n], o);
            if (lane == 0) {
#pragma unroll
                for (int n = 0; n < NQ; n += 4)
                    *reinterpret_cast<float4 *>(lsum + q4 * 16 + n) = make_float4(acc[n], acc[n + 1], acc[n + 2], acc[n + 3]);
            }
            float *dst = p.part + static_cast<int64_t>(u + c) * Z::PSTRIDE;
#pragma unroll
            for (int ch = 0; ch < Z::NCH; ++ch) {
                float o[kNQ];
                tmem_ld16(tl + Z::TM_O + ch * kNQ, o);
                const int j = ch * 128 + 32 * q4 + lane;
                if (j < RV) {
#pragma unroll
                    for (int n = 0; n < NQ; ++n) {
                        float on = o[n];
#pragma unroll
                        for (int k = 1; k < Z::PSPL; ++k) on += o[k * NQ + n];
                        if (n < p.nq) dst[n * RV + j] = on;
                    }
                }
            }
            tc_fence_before();
            mbar_arrive(&bar[bOfree]);
            named_bar_sync(1, 128);  // the run sums are visible
            if (st_tid < NQ) {
                float mine = 0.f;
#pragma unroll
                for (int n = 0; n < NQ; ++n)
                    if (st_tid == n) mine = m[n];
                dst[Z::PO_M + st_tid] = mine;
                dst[Z::PO_L + st_tid] = (lsum[st_tid] + lsum[16 + st_tid]) + (lsum[32 + st_tid] + lsum[48 + st_tid]);
            }
            named_bar_sync(1, 128);  // lsum and red are free for the next run
            ++r;
        }
    }
    pdl_trigger();
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, Z::TM_COLS);
    }
}

// ---------------------------------------------------------------- attention, large latents

// LLA-2D latents too wide for a whole page per pipeline stage ((1152, 1920): a 384 KB page).  A
// page streams through two rings: its K-plane as KC column chunks (each a contiguous run of
// granules, one bulk copy), accumulated into S^T chunk by chunk, and its V-plane as 128-row
// chunks (two 64-column TMA boxes each), each feeding one 16-column O^T accumulator.  Warps:
//   0     K producer                    1     S^T issuer and TMEM owner
//   2-5   softmax (as attn2d_kernel)    6     O^T issuer
//   7     V producer: it also zeroes, once a chunk of a run's partial last page has landed, the
//         rows past the sequence (0 * NaN would poison O^T), and only then hands the chunk to the
//         O^T issuer; the hand-over trails the copies by VST - 1 chunks
template <int RK, int RV>
struct ZB {
    static constexpr int NS = 2 * kNQ;
    static constexpr int RKC = 288;                    // K chunk columns
    static constexpr int KC = RK / RKC;
    static constexpr int KCB = kPT * RKC * 2;          // bytes of a K chunk (36 KB)
    static constexpr int VC = RV / 128;                // 128-row V chunks
    static constexpr int BOX = kPT * 128;
    static constexpr int VCB = 2 * BOX;                // bytes of a V chunk (16 KB)
    static constexpr int KST = 2, VST = 4;
    static constexpr int QB = NS * RK * 2;             // [Q~_hi; Q~_lo] operand (72 KB)
    static constexpr int PBUF = kPT * kNQ * 2;
    static constexpr int RED = 1024;
    static constexpr int NBAR = 42;
    static constexpr int oV = 0;                       // 1024-byte aligned (128-byte swizzle)
    static constexpr int oK = oV + VST * VCB;
    static constexpr int oQ = oK + KST * KCB;
    static constexpr int oP = oQ + QB;
    static constexpr int oRed = oP + 2 * PBUF;
    static constexpr int oBar = oRed + RED;
    static constexpr int SMEM = 1024 + oBar + NBAR * 8;
    static constexpr uint32_t TM_S = 0, TM_O = 2 * NS, TM_COLS = 512;
    static constexpr uint32_t IDESC_S = umma_idesc_bf16(64, NS, 0, 0);
    static constexpr uint32_t IDESC_O = umma_idesc_bf16(128, kNQ, 1, 0);
    static constexpr int PSTRIDE = kNQ * RV + 2 * kNQ;
    static constexpr int PO_M = kNQ * RV, PO_L = kNQ * RV + kNQ;
    static_assert(RK % RKC == 0 && RV % 128 == 0, "chunks");
    static_assert(SMEM <= kSmemCap, "shared memory");
    static_assert(TM_O + VC * kNQ <= TM_COLS, "TMEM columns");
    static_assert(VST >= 2 && KST >= 2 && VST <= 8, "ring depths");
};

// barrier indices of the large-latent kernel
enum {
    cKfull = 0 /* [2] */, cKempty = 2, cVfull = 4 /* [8] */, cVok = 12, cVempty = 20,
    cSfull = 28 /* [2] */, cSfree = 30, cPfull = 32, cPfree = 34, cOfree = 36, cQready = 37,
    cQfree = 38, cAbort = 39, cTslot = 40
};

template <int RK, int RV>
__global__ void __launch_bounds__(256, 1)
    attn2d_big_kernel(const __grid_constant__ CUtensorMap tv, const T2Params p) {
    using Z = ZB<RK, RV>;
    extern __shared__ __align__(1024) char sm_raw[];
    char *sm = reinterpret_cast<char *>((reinterpret_cast<uintptr_t>(sm_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    uint64_t *bar = reinterpret_cast<uint64_t *>(sm + Z::oBar);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(bar + cAbort);
    uint32_t *tslot = reinterpret_cast<uint32_t *>(bar + cTslot);
    float *red = reinterpret_cast<float *>(sm + Z::oRed);  // [2 pages][4 warps][16] maxima
    float *lsum = red + 128;                                // [4 warps][16] run sums
    float *betas = lsum + 64;                               // [16]
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int G = gridDim.x, c = blockIdx.x;

    if (tid == 0) {
        for (int s = 0; s < Z::KST; ++s) {
            mbar_init(&bar[cKfull + s], 1);
            mbar_init(&bar[cKempty + s], 1);
        }
        for (int s = 0; s < Z::VST; ++s) {
            mbar_init(&bar[cVfull + s], 1);
            mbar_init(&bar[cVok + s], 1);
            mbar_init(&bar[cVempty + s], 1);
        }
        for (int s = 0; s < 2; ++s) {
            mbar_init(&bar[cSfull + s], 1);
            mbar_init(&bar[cSfree + s], 128);
            mbar_init(&bar[cPfull + s], 128);
            mbar_init(&bar[cPfree + s], 1);
        }
        mbar_init(&bar[cOfree], 128);
        mbar_init(&bar[cQready], 128);
        mbar_init(&bar[cQfree], 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 1) tmem_alloc(tslot, Z::TM_COLS);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tslot;
    pdl_wait();  // q~, beta and the page prefix sums come from the absorb kernel

    const int NP = p.pstart[p.U];
    const int g0 = page_lo(c, NP, G), g1 = page_lo(c + 1, NP, G);
    const int ufirst = g0 < g1 ? first_unit(p.pstart, p.U, g0) : p.U;

    if (warp == 0) {
        // ----------------------------------------------------------------------- K producer
        if (lane == 0) {
            const uint64_t pol = policy_evict_first();
            int itk = 0;
            bool stop = false;
            for (int u = ufirst; u < p.U && !stop; ++u) {
                const int s0 = p.pstart[u], s1 = p.pstart[u + 1];
                if (s0 >= g1) break;
                const int pa = max(g0, s0) - s0, pe = min(g1, s1) - s0;
                const int32_t *bt = p.block_table + static_cast<int64_t>(u) * p.max_blocks;
                for (int pg = pa; pg < pe && !stop; ++pg) {
                    int32_t blk = bt[pg];
                    if (blk < 0 || blk >= p.num_blocks) {
                        atomicOr(p.err, LLA_DEVERR_BLOCK_ID);
                        blk = 0;
                    }
                    const char *src = p.pool + static_cast<int64_t>(blk) * p.page_bytes;
                    for (int kc = 0; kc < Z::KC; ++kc) {
                        const int st = itk % Z::KST;
                        if (!mbar_wait(&bar[cKempty + st], ((itk / Z::KST) & 1) ^ 1u, abort_flag, p.err) || *abort_flag) {
                            stop = true;
                            break;
                        }
                        mbar_arrive_expect_tx(&bar[cKfull + st], Z::KCB);
                        bulk_g2s(sm + Z::oK + st * Z::KCB, src + kc * Z::KCB, Z::KCB, &bar[cKfull + st], pol);
                        ++itk;
                    }
                }
            }
            volatile int never = 0;
            for (int j = max(0, itk - Z::KST); j < itk; ++j)
                mbar_wait(&bar[cKfull + j % Z::KST], (j / Z::KST) & 1, &never, p.err);
        }
        __syncwarp();
    } else if (warp == 7) {
        // ---------------------------------------------------------- V producer and hand-over
        int itv = 0, handed = 0;
        int nvs[Z::VST];  // per stage: valid rows of its chunk (64: nothing to zero)
#pragma unroll
        for (int i = 0; i < Z::VST; ++i) nvs[i] = kPT;
        // chunk j has landed: zero its rows past the sequence, then pass it to the O^T issuer
        auto hand_over = [&](int j) {
            const int st = j % Z::VST;
            volatile int never = 0;
            mbar_wait(&bar[cVfull + st], (j / Z::VST) & 1, &never, p.err);
            int nv = kPT;
#pragma unroll
            for (int i = 0; i < Z::VST; ++i)
                if (i == st) nv = nvs[i];
            if (nv < kPT) {
                char *vs = sm + Z::oV + st * Z::VCB;
                for (int w = lane; w < (kPT - nv) * 2 * 8; w += 32) {
                    const int cc = w & 7, r2 = w >> 3;
                    const int a = r2 & 1, row = nv + (r2 >> 1);
                    *reinterpret_cast<uint4 *>(vs + a * Z::BOX + row * 128 + cc * 16) = make_uint4(0, 0, 0, 0);
                }
                fence_proxy_async_smem();
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&bar[cVok + st]);
        };
        bool stop = false;
        for (int u = ufirst; u < p.U && !stop; ++u) {
            const int s0 = p.pstart[u], s1 = p.pstart[u + 1];
            if (s0 >= g1) break;
            const int pa = max(g0, s0) - s0, pe = min(g1, s1) - s0;
            const int L = p.context_lens[u];
            const int32_t *bt = p.block_table + static_cast<int64_t>(u) * p.max_blocks;
            for (int pg = pa; pg < pe && !stop; ++pg) {
                int32_t blk = bt[pg];
                if (blk < 0 || blk >= p.num_blocks) blk = 0;  // flagged by the K producer
                const int nv = min(kPT, L - pg * kPT);
                for (int vc = 0; vc < Z::VC; ++vc) {
                    const int st = itv % Z::VST;
                    bool ok = true;
                    if (lane == 0)
                        ok = mbar_wait(&bar[cVempty + st], ((itv / Z::VST) & 1) ^ 1u, abort_flag, p.err) && !*abort_flag;
                    ok = __shfl_sync(0xffffffffu, ok, 0);
                    if (!ok) {
                        stop = true;
                        break;
                    }
#pragma unroll
                    for (int i = 0; i < Z::VST; ++i)
                        if (i == st) nvs[i] = nv;
                    if (lane == 0) {
                        mbar_arrive_expect_tx(&bar[cVfull + st], Z::VCB);
                        char *vs = sm + Z::oV + st * Z::VCB;
                        tma_load_3d(vs, &tv, (2 * vc) * 64, 0, blk, &bar[cVfull + st]);
                        tma_load_3d(vs + Z::BOX, &tv, (2 * vc + 1) * 64, 0, blk, &bar[cVfull + st]);
                    }
                    ++itv;
                    if (itv - handed >= Z::VST) hand_over(handed++);
                }
            }
        }
        while (handed < itv) hand_over(handed++);  // also drains every copy after an abort
    } else if (warp == 1) {
        // ----------------------------------------------------------------------- S^T issuer
        if (lane == 0) {
            const uint32_t base = smem_addr(sm);
            const uint64_t dq = umma_desc(base + Z::oQ, Z::NS * 16, 128);
            int it = 0, itk = 0, r = 0;
            for (int u = ufirst; u < p.U; ++u) {
                const int s0 = p.pstart[u], s1 = p.pstart[u + 1];
                if (s0 >= g1) break;
                const int n = min(g1, s1) - max(g0, s0);
                if (n <= 0) continue;
                mbar_wait(&bar[cQready], r & 1, abort_flag, p.err);
                tc_fence_after();
                for (int k = 0; k < n; ++k, ++it) {
                    const int s = it & 1;
                    if (it >= 2) mbar_wait(&bar[cSfree + s], ((it - 2) >> 1) & 1, abort_flag, p.err);
                    for (int kc = 0; kc < Z::KC; ++kc, ++itk) {
                        const int st = itk % Z::KST;
                        mbar_wait(&bar[cKfull + st], (itk / Z::KST) & 1, abort_flag, p.err);
                        tc_fence_after();
                        const uint64_t dk = umma_desc(base + Z::oK + st * Z::KCB, kPT * 16, 128);
#pragma unroll 6
                        for (int ks = 0; ks < Z::RKC / 16; ++ks)
                            umma_bf16(tmem + Z::TM_S + s * Z::NS, dk + ks * ((2 * kPT * 16) >> 4),
                                      dq + (kc * (Z::RKC / 8) + 2 * ks) * ((Z::NS * 16) >> 4), Z::IDESC_S,
                                      kc > 0 || ks > 0);
                        umma_commit(&bar[cKempty + st]);
                    }
                    umma_commit(&bar[cSfull + s]);
                    if (k == n - 1) umma_commit(&bar[cQfree]);
                }
                ++r;
            }
            // every product has completed before TMEM is released, even after an abort: the last
            // commit on each S^T buffer
            volatile int never = 0;
            for (int j = max(0, it - 2); j < it; ++j)
                mbar_wait(&bar[cSfull + (j & 1)], (j >> 1) & 1, &never, p.err);
        }
        __syncwarp();
    } else if (warp == 6) {
        // ----------------------------------------------------------------------- O^T issuer
        if (lane == 0) {
            const uint32_t base = smem_addr(sm);
            const uint64_t dp0 = umma_desc(base + Z::oP, kNQ * 16, 128);
            int it = 0, itv = 0, r = 0;
            for (int u = ufirst; u < p.U; ++u) {
                const int s0 = p.pstart[u], s1 = p.pstart[u + 1];
                if (s0 >= g1) break;
                const int n = min(g1, s1) - max(g0, s0);
                if (n <= 0) continue;
                for (int k = 0; k < n; ++k, ++it) {
                    const int s = it & 1;
                    mbar_wait(&bar[cPfull + s], (it >> 1) & 1, abort_flag, p.err);
                    if (k == 0 && r > 0) mbar_wait(&bar[cOfree], (r - 1) & 1, abort_flag, p.err);
                    const uint64_t dp = dp0 + static_cast<uint64_t>((s * Z::PBUF) >> 4);
                    for (int vc = 0; vc < Z::VC; ++vc, ++itv) {
                        const int st = itv % Z::VST;
                        mbar_wait(&bar[cVok + st], (itv / Z::VST) & 1, abort_flag, p.err);
                        tc_fence_after();
                        const uint64_t dv = umma_desc_sw128_mn(base + Z::oV + st * Z::VCB, Z::BOX);
#pragma unroll
                        for (int ks = 0; ks < kPT / 16; ++ks)
                            umma_bf16(tmem + Z::TM_O + vc * kNQ, dv + ((ks * 2048) >> 4),
                                      dp + ks * ((2 * kNQ * 16) >> 4), Z::IDESC_O, k > 0 || ks > 0);
                        umma_commit(&bar[cVempty + st]);
                    }
                    umma_commit(&bar[cPfree + s]);  // also: O^T holds pages up to it
                }
                ++r;
            }
            if (it > 0) {
                volatile int never = 0;
                mbar_wait(&bar[cPfree + ((it - 1) & 1)], ((it - 1) >> 1) & 1, &never, p.err);
            }
        }
        __syncwarp();
    } else {
        // --------------------------------------------------------------- softmax warps 2-5
        const int q4 = warp & 3;
        const uint32_t tl = tmem + (static_cast<uint32_t>(32 * q4) << 16);
        const int st_tid = tid - kSm0;
        const int tok = 16 * q4 + lane;
        int it = 0, r = 0;
        for (int u = ufirst; u < p.U; ++u) {
            const int s0 = p.pstart[u], s1 = p.pstart[u + 1];
            if (s0 >= g1) break;
            const int pa = max(g0, s0) - s0, pe = min(g1, s1) - s0;
            if (pe <= pa) continue;
            const int L = p.context_lens[u];
            if (r > 0) mbar_wait(&bar[cQfree], (r - 1) & 1, abort_flag, p.err);
            {
                const float4 *src = reinterpret_cast<const float4 *>(p.qt + static_cast<int64_t>(u) * kNQ * RK);
                for (int i = st_tid; i < kNQ * (RK / 8); i += 128) {
                    const int n = i / (RK / 8), g = i - n * (RK / 8);
                    uint4 hi = make_uint4(0, 0, 0, 0), lo = hi;
                    if (n < p.nq) {
                        const float4 a = src[2 * i], c4 = src[2 * i + 1];
                        const float v[8] = {a.x, a.y, a.z, a.w, c4.x, c4.y, c4.z, c4.w};
                        float r8[8];
#pragma unroll
                        for (int e = 0; e < 8; ++e) r8[e] = v[e] - __bfloat162float(__float2bfloat16_rn(v[e]));
                        hi = make_uint4(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]),
                                        pack_bf16x2(v[4], v[5]), pack_bf16x2(v[6], v[7]));
                        lo = make_uint4(pack_bf16x2(r8[0], r8[1]), pack_bf16x2(r8[2], r8[3]),
                                        pack_bf16x2(r8[4], r8[5]), pack_bf16x2(r8[6], r8[7]));
                    }
                    char *dq = sm + Z::oQ + g * (Z::NS * 16);
                    *reinterpret_cast<uint4 *>(dq + n * 16) = hi;
                    *reinterpret_cast<uint4 *>(dq + (kNQ + n) * 16) = lo;
                }
                if (st_tid < kNQ) betas[st_tid] = st_tid < p.nq ? p.beta[static_cast<int64_t>(u) * kNQ + st_tid] : 0.f;
            }
            fence_proxy_async_smem();
            mbar_arrive(&bar[cQready]);
            named_bar_sync(1, 128);
            float m[kNQ], acc[kNQ];
#pragma unroll
            for (int n = 0; n < kNQ; ++n) {
                m[n] = -INFINITY;
                acc[n] = 0.f;
            }
            const int nps = pe - pa;
            for (int k = 0; k < nps; ++k, ++it) {
                const int s = it & 1;
                const int tok0 = (pa + k) * kPT;
                mbar_wait(&bar[cSfull + s], (it >> 1) & 1, abort_flag, p.err);
                tc_fence_after();
                float x2[Z::NS], x[kNQ];
                tmem_ld32(tl + Z::TM_S + s * Z::NS, x2);
                tc_fence_before();
                mbar_arrive(&bar[cSfree + s]);
                const bool valid = lane < 16 && tok0 + tok < L;
#pragma unroll
                for (int n = 0; n < kNQ; ++n) x[n] = valid ? (x2[n] + x2[kNQ + n]) + betas[n] : -INFINITY;
                float mx[kNQ];
#pragma unroll
                for (int n = 0; n < kNQ; ++n) mx[n] = x[n];
#pragma unroll
                for (int o = 8; o >= 1; o >>= 1)
#pragma unroll
                    for (int n = 0; n < kNQ; ++n) mx[n] = fmaxf(mx[n], __shfl_xor_sync(0xffffffffu, mx[n], o));
                float *rp = red + s * 64;
                if (lane == 0) {
#pragma unroll
                    for (int n = 0; n < kNQ; n += 4)
                        *reinterpret_cast<float4 *>(rp + q4 * 16 + n) = make_float4(mx[n], mx[n + 1], mx[n + 2], mx[n + 3]);
                }
                named_bar_sync(1, 128);
                bool any = false;
                float f[kNQ];
#pragma unroll
                for (int n = 0; n < kNQ; n += 4) {
                    float4 a = *reinterpret_cast<const float4 *>(rp + n);
#pragma unroll
                    for (int w = 1; w < 4; ++w) {
                        const float4 bb = *reinterpret_cast<const float4 *>(rp + w * 16 + n);
                        a = make_float4(fmaxf(a.x, bb.x), fmaxf(a.y, bb.y), fmaxf(a.z, bb.z), fmaxf(a.w, bb.w));
                    }
                    const float pm[4] = {a.x, a.y, a.z, a.w};
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const float mn = fmaxf(m[n + e], pm[e]);
                        const bool need = mn > m[n + e] + kRescaleLog2;
                        f[n + e] = need ? ex2_approx(m[n + e] - mn) : 1.f;
                        if (need) {
                            acc[n + e] *= f[n + e];
                            m[n + e] = mn;
                            any = true;
                        }
                    }
                }
                if (any && k > 0) {
                    mbar_wait(&bar[cPfree + ((it - 1) & 1)], ((it - 1) >> 1) & 1, abort_flag, p.err);
                    tc_fence_after();
#pragma unroll 1
                    for (int ch = 0; ch < Z::VC; ++ch) {
                        float o[kNQ];
                        tmem_ld16(tl + Z::TM_O + ch * kNQ, o);
#pragma unroll
                        for (int n = 0; n < kNQ; ++n) o[n] *= f[n];
                        tmem_st16(tl + Z::TM_O + ch * kNQ, o);
                    }
                }
                float pv[kNQ];
#pragma unroll
                for (int n = 0; n < kNQ; ++n) {
                    pv[n] = ex2_approx(x[n] - m[n]);
                    acc[n] += pv[n];
                }
                if (it >= 2) mbar_wait(&bar[cPfree + s], ((it - 2) >> 1) & 1, abort_flag, p.err);
                if (lane < 16) {
                    char *pp = sm + Z::oP + s * Z::PBUF + (tok >> 3) * (kNQ * 16) + (tok & 7) * 2;
#pragma unroll
                    for (int n = 0; n < kNQ; ++n)
                        *reinterpret_cast<uint16_t *>(pp + n * 16) = __bfloat16_as_ushort(__float2bfloat16_rn(pv[n]));
                }
                fence_proxy_async_smem();
                tc_fence_before();
                mbar_arrive(&bar[cPfull + s]);
            }
            mbar_wait(&bar[cPfree + ((it - 1) & 1)], ((it - 1) >> 1) & 1, abort_flag, p.err);
            tc_fence_after();
#pragma unroll
            for (int o = 8; o >= 1; o >>= 1)
#pragma unroll
                for (int n = 0; n < kNQ; ++n) acc[n] += __shfl_xor_sync(0xffffffffu, acc[n], o);
            if (lane == 0) {
#pragma unroll
                for (int n = 0; n < kNQ; n += 4)
                    *reinterpret_cast<float4 *>(lsum + q4 * 16 + n) = make_float4(acc[n], acc[n + 1], acc[n + 2], acc[n + 3]);
            }
            float *dst = p.part + static_cast<int64_t>(u + c) * Z::PSTRIDE;
#pragma unroll 1
            for (int ch = 0; ch < Z::VC; ++ch) {
                float o[kNQ];
                tmem_ld16(tl + Z::TM_O + ch * kNQ, o);
                const int j = ch * 128 + 32 * q4 + lane;
#pragma unroll
                for (int n = 0; n < kNQ; ++n)
                    if (n < p.nq) dst[n * RV + j] = o[n];
            }
            tc_fence_before();
            mbar_arrive(&bar[cOfree]);
            named_bar_sync(1, 128);
            if (st_tid < kNQ) {
                float mine = 0.f;
#pragma unroll
                for (int n = 0; n < kNQ; ++n)
                    if (st_tid == n) mine = m[n];
                dst[Z::PO_M + st_tid] = mine;
                dst[Z::PO_L + st_tid] = (lsum[st_tid] + lsum[16 + st_tid]) + (lsum[32 + st_tid] + lsum[48 + st_tid]);
            }
            named_bar_sync(1, 128);
            ++r;
        }
    }
    pdl_trigger();
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, Z::TM_COLS);
    }
}

// ------------------------------------------------------------------------- finish kernel

// Grid (weight slices, ceil(B / spb), row slices), 128 threads (thread e = output element e,
// or, with four row slices, threads 4r .. 4r + 3 = row r of the CTA's 32).  spb (at most 8)
// sequences share one pass over the slice's W_up^V; small batches take fewer per CTA to use more
// SMs.  Slice w and sequence b give unit and query as in the absorb kernel.  The runs of a unit
// are merged by one warp, or by two or four that split its columns when the CTA has fewer than
// three units (no block barrier between units: each is a chain of dependent loads), then all
// threads apply W_up^V; a thread's weights, when they fit 80 registers (latents up to 640 wide),
// are loaded before the wait on the attention kernel.
template <int RV, int NQM, int RS>
__global__ void __launch_bounds__(128, 1) finish2d_kernel(const F2Params p) {
    constexpr int PS = NQM * RV + 2 * kNQ;
    constexpr int PO_M = NQM * RV, PO_L = NQM * RV + kNQ;
    constexpr int SPB = finish_seqs(RV);
    static_assert(RS == 1 || RS == 4, "row slices");
    static_assert(RS == 1 || (RV / 8) % RS == 0, "row slices read whole 16-byte units");
    constexpr bool kPre = RV / 8 / RS <= 20;  // the thread's weights fit 80 registers
    constexpr int NW = kPre ? RV / 8 / RS : 1;
    __shared__ __align__(16) float ob[SPB][RV];
    __shared__ float wts[4][kMaxGrid], wls[4][kMaxGrid];  // per warp: run weights and sums
    __shared__ float coef[SPB][3], scs[SPB];
    const int w = blockIdx.x, b0 = blockIdx.y * p.spb, tid = threadIdx.x;
    const int warp = tid >> 5, lane = tid & 31;
    const int nb = min(p.spb, p.B - b0);
    const int t = p.loops ? w / p.H : p.loop, h = p.loops ? w - t * p.H : w;
    const int64_t th = p.loops ? static_cast<int64_t>(h) * p.T + t : static_cast<int64_t>(t) * p.H + h;
    const int qn = p.loops ? t : h;  // the query of (b, w) within its unit
    auto iorow = [&](int b) { return ((p.loops ? static_cast<int64_t>(t) * p.B : 0) + b) * p.H + h; };
    // this thread's row e of W_up^V and mu^V (inputs of the call, not of earlier kernels); with
    // row slices, four threads per row (part q4 of its 16-byte units)
    const int e = RS == 1 ? tid : static_cast<int>(blockIdx.z) * (kD / RS) + (tid >> 2);
    const int q4 = RS == 1 ? 0 : (tid & 3);
    const uint4 *W = reinterpret_cast<const uint4 *>(static_cast<const uint16_t *>(p.w_up_v) + (th * kD + e) * RV);
    uint4 wr[NW];
    if constexpr (kPre) {
#pragma unroll
        for (int j = 0; j < NW; ++j) wr[j] = W[q4 + RS * j];
    }
    const float muv = p.mu_v ? p.mu_v[th * kD + e] : 0.f;
    // the call's own inputs (not outputs of the earlier kernels) before the wait: each unit's
    // current-token score and value element e
    float cv[SPB];
#pragma unroll
    for (int bi = 0; bi < SPB; ++bi)
        cv[bi] = p.cur_v && bi < nb ? load_elem(p.cur_v, iorow(b0 + bi) * kD + e, p.io_bf16) : 0.f;
    if (p.cur_k) {
        for (int bi = warp; bi < nb; bi += 4) {
            const int64_t row = iorow(b0 + bi) * kD;
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
    const int NP = p.pstart[p.U];
    // G warps per unit (all four for one unit, two each for two): warp `sub` of a group takes
    // the columns j = lane + 32 (sub + G q)
    const int G = nb == 1 ? 4 : nb == 2 ? 2 : 1;
    const int grp = warp / G, sub = warp - grp * G;
    constexpr int NJ = (RV + 31) / 32;
    constexpr int KR = NJ <= 16 ? 4 : NJ <= 32 ? 2 : 1;  // runs whose loads are in flight together
    float *wt = wts[warp];
    float *wl = wls[warp];
    for (int bi = grp; bi < SPB; bi += 4 / G) {
        if (bi >= nb) {
            for (int j = lane + 32 * sub; j < RV; j += 32 * G) ob[bi][j] = 0.f;
            continue;
        }
        const int b = b0 + bi;
        const int u = p.loops ? b * p.H + h : b;
        const int s0 = p.pstart[u], s1 = p.pstart[u + 1];
        float M = -INFINITY, l = 0.f;
        float acc[NJ];
#pragma unroll
        for (int q = 0; q < NJ; ++q) acc[q] = 0.f;
        if (s1 > s0) {
            // the runs of unit u: the CTAs c0 .. c1 that hold pages (a CTA between them may hold
            // none and writes nothing), partials at slots u + c
            const int c0 = cta_of(s0, NP, p.grid), c1 = cta_of(s1 - 1, NP, p.grid);
            const int nr = c1 - c0 + 1;
            const float *pu = p.part + static_cast<int64_t>(u + c0) * PS;
            // the run maxima and sums in one round of loads
            float mm = -INFINITY;
            for (int i = lane; i < nr; i += 32) {
                const bool has = page_lo(c0 + i + 1, NP, p.grid) > page_lo(c0 + i, NP, p.grid);
                wt[i] = has ? pu[static_cast<int64_t>(i) * PS + PO_M + qn] : -INFINITY;
                wl[i] = has ? pu[static_cast<int64_t>(i) * PS + PO_L + qn] : 0.f;
                mm = fmaxf(mm, wt[i]);
            }
            M = warp_max(mm);
            float ls = 0.f;
            for (int i = lane; i < nr; i += 32) {
                const float w8 = wt[i] == -INFINITY ? 0.f : ex2_approx(wt[i] - M);  // no run: 0
                ls = fmaf(w8, wl[i], ls);
                wt[i] = w8;
            }
            l = warp_sum(ls);
            __syncwarp();
            // the column loads of KR runs in flight at once, then their sums: a slot between the
            // unit's first and last CTA that holds no run (weight 0) is read, inside the
            // workspace, but its values are never used
            for (int i0 = 0; i0 < nr; i0 += KR) {
                float v[KR][NJ];
#pragma unroll
                for (int k = 0; k < KR; ++k) {
                    const float *pr = pu + static_cast<int64_t>(min(i0 + k, nr - 1)) * PS + qn * RV;
#pragma unroll
                    for (int q = 0; q < NJ; ++q) {
                        const int j = lane + 32 * (sub + G * q);
                        v[k][q] = j < RV ? pr[j] : 0.f;
                    }
                }
#pragma unroll
                for (int k = 0; k < KR; ++k) {
                    const float w8 = i0 + k < nr ? wt[i0 + k] : 0.f;
                    if (w8 > 0.f) {  // warp-uniform
#pragma unroll
                        for (int q = 0; q < NJ; ++q) acc[q] = fmaf(w8, v[k][q], acc[q]);
                    }
                }
            }
            __syncwarp();  // wt is free for the warp's next unit
        }
#pragma unroll
        for (int q = 0; q < NJ; ++q) {
            const int j = lane + 32 * (sub + G * q);
            if (j < RV) ob[bi][j] = acc[q];
        }
        if (sub == 0) {
            const float sc = p.cur_k ? scs[bi] : -INFINITY;
            if (lane == 0) {
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
    }
    __syncthreads();
    // out_b[e] = coef0 (W_up^V o~_b)[e] + coef1 mu^V[e] + coef2 v_cur,b[e]
    float acc[SPB];
#pragma unroll
    for (int bi = 0; bi < SPB; ++bi) acc[bi] = 0.f;
    auto step = [&](int j8, const uint4 w4) {
        const float2 w0 = bf2_to_f2(w4.x), w1 = bf2_to_f2(w4.y), w2 = bf2_to_f2(w4.z), w3 = bf2_to_f2(w4.w);
#pragma unroll
        for (int bi = 0; bi < SPB; ++bi) {
            const float4 o0 = *reinterpret_cast<const float4 *>(&ob[bi][j8 * 8]);
            const float4 o1 = *reinterpret_cast<const float4 *>(&ob[bi][j8 * 8 + 4]);
            float a = acc[bi];
            a = fmaf(w0.x, o0.x, a); a = fmaf(w0.y, o0.y, a); a = fmaf(w1.x, o0.z, a); a = fmaf(w1.y, o0.w, a);
            a = fmaf(w2.x, o1.x, a); a = fmaf(w2.y, o1.y, a); a = fmaf(w3.x, o1.z, a); a = fmaf(w3.y, o1.w, a);
            acc[bi] = a;
        }
    };
    // with row slices, a quarter of the row's 16-byte units (threads 4r .. 4r + 3 read 64
    // consecutive bytes), then the four partial sums of the row
    if constexpr (kPre) {
#pragma unroll
        for (int j = 0; j < NW; ++j) step(q4 + RS * j, wr[j]);  // fully unrolled: wr stays in registers
    } else {
#pragma unroll 12
        for (int j8 = q4; j8 < RV / 8; j8 += RS) step(j8, W[j8]);
    }
    if constexpr (RS > 1) {
#pragma unroll
        for (int bi = 0; bi < SPB; ++bi) {
            acc[bi] += __shfl_xor_sync(0xffffffffu, acc[bi], 1);
            acc[bi] += __shfl_xor_sync(0xffffffffu, acc[bi], 2);
        }
    }
#pragma unroll
    for (int bi = 0; bi < SPB; ++bi) {
        if (bi >= nb || q4 != 0) break;
        const int64_t idx = iorow(b0 + bi) * kD + e;
        float v = acc[bi] * coef[bi][0] + coef[bi][1] * muv;
        if (p.cur_v) v = fmaf(coef[bi][2], cv[bi], v);
        store_elem(p.out, idx, v, p.io_bf16);
    }
    __syncthreads();
    pdl_trigger();
}

// ------------------------------------------------------------------------- host side

struct WS2 {
    size_t part, qt, beta, pstart, total;
};

inline size_t al256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

// Workspace of U units: run partials, q~ rows, beta, page prefix sums.
WS2 ws2_layout(int rkx, int r_v, int nqm, int U, int grid) {
    WS2 w;
    w.part = 0;
    w.qt = al256(static_cast<size_t>(U + grid) * (nqm * r_v + 2 * kNQ) * sizeof(float));
    w.beta = w.qt + al256(static_cast<size_t>(U) * nqm * rkx * sizeof(float));
    w.pstart = w.beta + al256(static_cast<size_t>(U) * nqm * sizeof(float));
    w.total = w.pstart + al256(static_cast<size_t>(U + 1) * sizeof(int));
    return w;
}

// The three launches for NQ query slots per unit; loops: the T loops of each (sequence, head)
// of a per-head cache (hu = H units per sequence), else the H heads of each LLA-2D sequence.
template <int RK, int RV, int NQ>
lla_status launch_units(const DecodeArgs &a, bool loops, cudaStream_t stream) {
    using Z = Z2<RK, RV, NQ>;
    lla_status st = LLA_OK;
    unsigned *err = device_error_word(&st);
    if (st != LLA_OK) return st;
    const int grid = num_sms();
    if (grid <= 0 || grid > kMaxGrid) return LLA_ERR_UNSUPPORTED;
    const int hu = loops ? a.H : 1;
    const int nq = loops ? a.T : a.H;
    const int nw = loops ? a.T * a.H : a.H;  // weight slices
    if (nq < 1 || nq > NQ) return LLA_ERR_UNSUPPORTED;
    if (static_cast<int64_t>(a.num_blocks) * hu >= (int64_t(1) << 31)) return LLA_ERR_UNSUPPORTED;  // TMA coordinate
    const int U = a.B * hu;
    // the units' pages are numbered in 32 bits
    if (static_cast<int64_t>(U) * ((static_cast<int64_t>(a.max_ctx) + kPT - 1) / kPT) >= (int64_t(1) << 31))
        return LLA_ERR_UNSUPPORTED;
    const WS2 w = ws2_layout(Z::RKX, RV, Z::NQM, U, grid);
    if (a.workspace_bytes < w.total) return LLA_ERR_WORKSPACE;
    char *ws = static_cast<char *>(a.workspace);
    static DeviceOnce configured;
    if (raise_smem_limit(attn2d_kernel<RK, RV, NQ>, Z::SMEM, configured) != LLA_OK) return LLA_ERR_CUDA;
    const int64_t page_bytes = static_cast<int64_t>(head_page_bytes(RK, RV, 2));
    // the V-planes of every page: [num_blocks * hu][64 tokens][r_v] bf16
    CUtensorMap tv;
    const uint64_t dims[3] = {static_cast<uint64_t>(RV), static_cast<uint64_t>(kPT),
                              static_cast<uint64_t>(a.num_blocks) * hu};
    const uint64_t strides[2] = {static_cast<uint64_t>(RV) * 2, static_cast<uint64_t>(page_bytes)};
    const uint32_t box[3] = {64, kPT, 1};
    if (!encode_tmap_bf16(&tv, static_cast<const char *>(a.pool) + kPT * RK * 2, 3, dims, strides, box, true))
        return LLA_ERR_CUDA;

    A2Params ap = {};
    ap.T = a.T; ap.H = a.H; ap.loop = a.loop; ap.io_bf16 = a.io_bf16; ap.pass1 = a.cur_k != nullptr;
    ap.B = a.B; ap.max_ctx = a.max_ctx; ap.max_blocks = a.max_blocks;
    ap.loops = loops ? 1 : 0; ap.hu = hu;
    ap.scale_log2 = a.scale * kLog2e;
    ap.w_up_k = a.w_up_k; ap.mu_k = a.mu_k; ap.q = a.q; ap.context_lens = a.context_lens;
    ap.qt = reinterpret_cast<float *>(ws + w.qt);
    ap.beta = reinterpret_cast<float *>(ws + w.beta);
    ap.pstart = reinterpret_cast<int *>(ws + w.pstart);
    ap.err = err;
    if ((st = launch_ex(absorb2d_kernel<RK, NQ>, dim3(nw, Z::RKX / 32 + (Z::RKX % 32 ? 1 : 0), (a.B + 15) / 16), 256, 0,
                        stream, ap)) != LLA_OK)
        return st;

    T2Params tp = {};
    tp.nq = nq; tp.U = U; tp.hu = hu;
    tp.pool = static_cast<const char *>(a.pool);
    tp.num_blocks = a.num_blocks; tp.page_bytes = page_bytes;
    tp.block_table = a.block_table; tp.max_blocks = a.max_blocks;
    tp.context_lens = a.context_lens;
    tp.qt = ap.qt; tp.beta = ap.beta; tp.pstart = ap.pstart;
    tp.part = reinterpret_cast<float *>(ws + w.part);
    tp.err = err;
    if ((st = launch_ex(attn2d_kernel<RK, RV, NQ>, dim3(grid), kT2, Z::SMEM, stream, tv, tp)) != LLA_OK)
        return st;

    F2Params fp = {};
    fp.T = a.T; fp.H = a.H; fp.loop = a.loop; fp.io_bf16 = a.io_bf16; fp.B = a.B; fp.grid = grid;
    fp.loops = ap.loops; fp.hu = hu; fp.U = U;
    fp.scale_log2 = ap.scale_log2;
    fp.w_up_v = a.w_up_v; fp.mu_v = a.mu_v;
    fp.q = a.q; fp.cur_k = a.cur_k; fp.cur_v = a.cur_v; fp.out = a.out;
    fp.pstart = ap.pstart; fp.part = tp.part;
    // about two finish CTAs per SM: fewer sequences per CTA for small batches, and row slices
    // when even one sequence per CTA leaves SMs idle
    const int64_t units = static_cast<int64_t>(a.B) * nw;
    const int rs = units <= 2 * grid ? finish_slices(RV) : 1;
    const int64_t want = units * rs;
    fp.spb = static_cast<int>(std::min<int64_t>(finish_seqs(RV), std::max<int64_t>(1, (want + 2 * grid - 1) / (2 * grid))));
    const dim3 fg(nw, (a.B + fp.spb - 1) / fp.spb, rs);
    if constexpr (finish_slices(RV) > 1) {
        if (rs > 1) return launch_ex(finish2d_kernel<RV, Z::NQM, finish_slices(RV)>, fg, 128, 0, stream, fp);
    }
    return launch_ex(finish2d_kernel<RV, Z::NQM, 1>, fg, 128, 0, stream, fp);
}

// ------------------------------------------------------------------------- rotary keys

struct RKParams {
    int N, d_rope, pairing, x_bf16;
    char *pool;
    int64_t num_blocks;
    const void *k;  // [N][d_rope]
    const int32_t *positions;
    const int64_t *slots;
    unsigned long long phi[48];
    unsigned *err;
};

// One thread per (token, pair): k^R of token n turned at positions[n] (pair j by
// positions[n] theta_j), written as bf16 at row slot % 64 of block slot / 64 in the granule
// layout of a K-plane (granule g of row i at g*1024 + i*16).
__global__ void __launch_bounds__(256) rope_key_store_kernel(const RKParams p) {
    const int hp = p.d_rope / 2;
    const int64_t i = static_cast<int64_t>(blockIdx.x) * 256 + threadIdx.x;
    pdl_wait();
    if (i < static_cast<int64_t>(p.N) * hp) {
        const int n = static_cast<int>(i / hp), j = static_cast<int>(i - static_cast<int64_t>(n) * hp);
        const int64_t slot = p.slots[n];
        const int pos = p.positions[n];
        if (slot >= 0) {
            const int64_t blk = slot / kPT;
            const int row = static_cast<int>(slot - blk * kPT);
            if (blk >= p.num_blocks) {
                atomicOr(p.err, LLA_DEVERR_SLOT);
            } else if (pos < 0) {
                atomicOr(p.err, LLA_DEVERR_CONTEXT);
            } else {
                float sn, cs;
                turn_sincos(pos, p.phi[j], &sn, &cs);
                const int a = p.pairing ? 2 * j : j, c = p.pairing ? 2 * j + 1 : j + hp;
                const float x = load_elem(p.k, static_cast<int64_t>(n) * p.d_rope + a, p.x_bf16);
                const float y = load_elem(p.k, static_cast<int64_t>(n) * p.d_rope + c, p.x_bf16);
                char *plane = p.pool + blk * (static_cast<int64_t>(kPT) * p.d_rope * 2);
                *reinterpret_cast<__nv_bfloat16 *>(plane + (a >> 3) * (kPT * 16) + row * 16 + (a & 7) * 2) =
                    __float2bfloat16_rn(x * cs - y * sn);
                *reinterpret_cast<__nv_bfloat16 *>(plane + (c >> 3) * (kPT * 16) + row * 16 + (c & 7) * 2) =
                    __float2bfloat16_rn(x * sn + y * cs);
            }
        }
    }
    pdl_trigger();
}

}  // namespace

// theta_j = base^(-2j/d_rope) in 64-bit fixed-point turns (theta_j <= 1 rad < 1 turn).
void rotary_phases(int d_rope, double base, unsigned long long *phi) {
    const double two_pi = 6.283185307179586476925286766559;
    for (int j = 0; j < d_rope / 2; ++j)
        phi[j] = static_cast<unsigned long long>(ldexp(pow(base, -2.0 * j / d_rope) / two_pi, 64));
}

bool decode_2d_supported(int es, int d, int H, int r_k, int r_v) {
    return es == 2 && d == kD && H >= 1 && H <= kNQ &&
           ((r_k == 96 && r_v == 160) || (r_k == 128 && r_v == 128) || (r_k == 288 && r_v == 480) ||
            (r_k == 1152 && r_v == 1920));
}

size_t decode_2d_workspace_bytes(int r_k, int r_v, int B) {
    const int grid = num_sms();
    if (grid <= 0) return 0;
    return ws2_layout(r_k, r_v, kNQ, B, grid).total;
}

lla_status launch_rope_key_store(int d_rope, double base, int pairing, void *rope_pool, int64_t num_blocks,
                                 const void *k, int x_bf16, const int32_t *positions, const int64_t *slots,
                                 int N, cudaStream_t stream) {
    if (N == 0) return LLA_OK;
    lla_status st = LLA_OK;
    unsigned *err = device_error_word(&st);
    if (st != LLA_OK) return st;
    RKParams rp = {};
    rp.N = N; rp.d_rope = d_rope; rp.pairing = pairing; rp.x_bf16 = x_bf16;
    rp.pool = static_cast<char *>(rope_pool); rp.num_blocks = num_blocks;
    rp.k = k; rp.positions = positions; rp.slots = slots; rp.err = err;
    rotary_phases(d_rope, base, rp.phi);
    const int64_t total = static_cast<int64_t>(N) * (d_rope / 2);
    if ((total + 255) / 256 > 0x7fffffff) return LLA_ERR_UNSUPPORTED;
    return launch_ex(rope_key_store_kernel, dim3(static_cast<unsigned>((total + 255) / 256)), 256, 0, stream, rp);
}

namespace {

// LLA-2D with latents too wide for whole-page stages: the absorb and finish kernels of
// launch_units around attn2d_big_kernel.
template <int RK, int RV>
lla_status launch_big(const DecodeArgs &a, cudaStream_t stream) {
    using Z = ZB<RK, RV>;
    lla_status st = LLA_OK;
    unsigned *err = device_error_word(&st);
    if (st != LLA_OK) return st;
    const int grid = num_sms();
    if (grid <= 0 || grid > kMaxGrid) return LLA_ERR_UNSUPPORTED;
    if (a.H < 1 || a.H > kNQ) return LLA_ERR_UNSUPPORTED;
    if (static_cast<int64_t>(a.B) * ((static_cast<int64_t>(a.max_ctx) + kPT - 1) / kPT) >= (int64_t(1) << 31))
        return LLA_ERR_UNSUPPORTED;
    const WS2 w = ws2_layout(RK, RV, kNQ, a.B, grid);
    if (a.workspace_bytes < w.total) return LLA_ERR_WORKSPACE;
    char *ws = static_cast<char *>(a.workspace);
    static DeviceOnce configured;
    if (raise_smem_limit(attn2d_big_kernel<RK, RV>, Z::SMEM, configured) != LLA_OK) return LLA_ERR_CUDA;
    const int64_t page_bytes = static_cast<int64_t>(head_page_bytes(RK, RV, 2));
    CUtensorMap tv;
    const uint64_t dims[3] = {static_cast<uint64_t>(RV), static_cast<uint64_t>(kPT), static_cast<uint64_t>(a.num_blocks)};
    const uint64_t strides[2] = {static_cast<uint64_t>(RV) * 2, static_cast<uint64_t>(page_bytes)};
    const uint32_t box[3] = {64, kPT, 1};
    if (!encode_tmap_bf16(&tv, static_cast<const char *>(a.pool) + kPT * RK * 2, 3, dims, strides, box, true))
        return LLA_ERR_CUDA;

    A2Params ap = {};
    ap.T = a.T; ap.H = a.H; ap.loop = a.loop; ap.io_bf16 = a.io_bf16; ap.pass1 = a.cur_k != nullptr;
    ap.B = a.B; ap.max_ctx = a.max_ctx; ap.max_blocks = a.max_blocks;
    ap.loops = 0; ap.hu = 1;
    ap.scale_log2 = a.scale * kLog2e;
    ap.w_up_k = a.w_up_k; ap.mu_k = a.mu_k; ap.q = a.q; ap.context_lens = a.context_lens;
    ap.qt = reinterpret_cast<float *>(ws + w.qt);
    ap.beta = reinterpret_cast<float *>(ws + w.beta);
    ap.pstart = reinterpret_cast<int *>(ws + w.pstart);
    ap.err = err;
    if ((st = launch_ex(absorb2d_kernel<RK, kNQ>, dim3(a.H, RK / 32, (a.B + 15) / 16), 256, 0, stream, ap)) != LLA_OK)
        return st;
    T2Params tp = {};
    tp.nq = a.H; tp.U = a.B; tp.hu = 1;
    tp.pool = static_cast<const char *>(a.pool);
    tp.num_blocks = a.num_blocks; tp.page_bytes = page_bytes;
    tp.block_table = a.block_table; tp.max_blocks = a.max_blocks;
    tp.context_lens = a.context_lens;
    tp.qt = ap.qt; tp.beta = ap.beta; tp.pstart = ap.pstart;
    tp.part = reinterpret_cast<float *>(ws + w.part);
    tp.err = err;
    if ((st = launch_ex(attn2d_big_kernel<RK, RV>, dim3(grid), 256, Z::SMEM, stream, tv, tp)) != LLA_OK)
        return st;
    F2Params fp = {};
    fp.T = a.T; fp.H = a.H; fp.loop = a.loop; fp.io_bf16 = a.io_bf16; fp.B = a.B; fp.grid = grid;
    fp.loops = 0; fp.hu = 1; fp.U = a.B;
    fp.scale_log2 = ap.scale_log2;
    fp.w_up_v = a.w_up_v; fp.mu_v = a.mu_v;
    fp.q = a.q; fp.cur_k = a.cur_k; fp.cur_v = a.cur_v; fp.out = a.out;
    fp.pstart = ap.pstart; fp.part = tp.part;
    // each CTA takes a quarter of a head's output rows for up to four sequences
    fp.spb = std::min(finish_seqs(RV), a.B);
    return launch_ex(finish2d_kernel<RV, kNQ, finish_slices(RV)>, dim3(a.H, (a.B + fp.spb - 1) / fp.spb, finish_slices(RV)), 128, 0,
                     stream, fp);
}

}  // namespace

lla_status launch_decode_2d(const DecodeArgs &a, cudaStream_t stream) {
    if (a.B == 0) return LLA_OK;
    if (a.num_blocks >= (int64_t(1) << 31)) return LLA_ERR_UNSUPPORTED;  // 32-bit TMA coordinate
#define LLA_2D(K, V) \
    if (a.r_k == K && a.r_v == V) return launch_units<K, V, kNQ>(a, false, stream);
    LLA_2D(96, 160)
    LLA_2D(128, 128)
    LLA_2D(288, 480)
#undef LLA_2D
    if (a.r_k == 1152 && a.r_v == 1920) return launch_big<1152, 1920>(a, stream);
    return LLA_ERR_UNSUPPORTED;
}

// The T loops of a per-head cache: up to 4 loops per (sequence, head) unit.
constexpr int kLoopSlots = 4;

lla_status decode_loops_fits(int r_k, int r_v, int es, int d, int T, int B) {
    (void)B;
    if (es != 2 || d != kD || T < 1 || T > kLoopSlots) return LLA_ERR_UNSUPPORTED;
    if ((r_k == 96 && r_v == 160) || (r_k == 128 && r_v == 128) || (r_k == 72 && r_v == 120) ||
        (r_k == 192 && r_v == 320))
        return LLA_OK;
    return LLA_ERR_UNSUPPORTED;
}

size_t decode_loops_workspace_bytes(int r_k, int r_v, int B, int H, int grid) {
    return ws2_layout((r_k + 15) / 16 * 16, r_v, kLoopSlots, B * H, grid).total;
}

lla_status launch_decode_loops(const DecodeArgs &a, cudaStream_t stream) {
    if (a.B == 0) return LLA_OK;
#define LLA_LOOPS(K, V) \
    if (a.r_k == K && a.r_v == V) return launch_units<K, V, kLoopSlots>(a, true, stream);
    LLA_LOOPS(96, 160)
    LLA_LOOPS(128, 128)
    LLA_LOOPS(72, 120)
    LLA_LOOPS(192, 320)
#undef LLA_LOOPS
    return LLA_ERR_UNSUPPORTED;
}

}  // namespace lla
