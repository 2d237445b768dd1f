// lla_decode_rope.cu -- decode with rotary positions applied after reconstruction: the full-RoPE
// decoder of Looped Latent Attention (Sec. 3 "RoPE and reconstruction"; App. A "Decoding and
// caching").
//
// The codec holds pre-RoPE keys.  Cached key i of a sequence sits at position p_i = i; the query
// (and, in pass 1, the current token's exact key) at P = L in pass 1 and P = L - 1 in pass 2.
// RoPE (RoFormer) turns pair j of a vector at position p by p theta_j, theta_j = base^(-2j/d):
//   s_i = scale rot(q, P) . rot(khat_i, p_i) = scale rot(q, P - p_i) . khat_i,
//   khat_i = W_up,t^K c_k,i + mu^K_t                                           (Eq. decode)
// The rotation depends on i, so the key up-projection cannot move onto the query as in the
// absorbed kernel; each page's keys are rebuilt on the tensor cores instead.  Values carry no
// rotation, so the value side stays in latent space as in lla_decode.cu:
//   o = (W_up,t^V sum_i p_i c_v,i + (sum_i p_i) mu^V_t + p_cur v_cur) / (sum_i p_i + p_cur).
//
// This kernel serves (r_k, r_v) = (192, 320), whose 64 KB head pages and 48 KB W_up rows leave
// no room for the tensor-core value path of lla_decode_rope_tc.cu (which serves the other shapes).
//
// GB300 mapping (one CTA per SM; the persistent split of (sequence, head, page) units over the
// CTAs, the TMA ring, the split-KV merge and the output projection are shared with lla_decode.cu
// through lla_decode_common.cuh):
//   * producer warp: TMA bulk copies of whole head pages (K-plane + V-plane) into the ring.
//   * MMA warp: per page, Khat^T (d x 64) = W_up,t^K (d x r_k) . C_k^T with tcgen05.mma.  A is
//     W_up,t^K, staged once per run as no-swizzle K-major core matrices; B is the page's K-plane
//     exactly as it sits in the ring (its granule-interleaved layout is a no-swizzle K-major
//     operand with the 64 tokens along N); one more K step adds mu^K_t as a (mu_hi, mu_lo) pair
//     of bf16 columns against a pair of ones.  D lands in TMEM (lane = key dimension, column =
//     token), in two buffers so that a page's MMA overlaps the previous page's epilogue.
//   * four epilogue warps (one per TMEM lane quarter): lane m multiplies its 64 columns by
//     element m of rot(q, P - p_i).  Along a page that element is a sinusoid in i; it starts from
//     a phase computed exactly per page (64-bit fixed-point turns) and steps through the tokens
//     with a second-order recurrence (two flops per token).  The 128 products of a token are
//     summed through a shared-memory transpose, then the online softmax runs as in the absorbed
//     kernel.
//   * four value warps: sum_i p_i c_v,i from the V-plane (shared with lla_decode.cu).
//   * four management warps: per run, W_up,t^K and mu^K_t into an A slot and q into a query
//     slot; the merge of split runs and W_up,t^V, mu^V_t, 1/l (shared with lla_decode.cu).
#include <string.h>

// one head page per pipeline step at every rank shape this kernel takes
#define LLA_DECODE_STEP_BYTES (32 * 1024)
#include "lla_decode_common.cuh"
#include "lla_tcgen05.cuh"

namespace lla {
namespace {

constexpr int kRopeD = 128;                        // head width of the tensor-core path
constexpr int kRopePairs = kRopeD / 2;
constexpr int kMmaWarp = kAsyncThreads / 32;       // warp 13, after the management warps
constexpr int kRopeThreads = kAsyncThreads + 32;   // 448
constexpr int kRopeWst = 20 * 1024;                // staging buffer of W_up,t^V rows
constexpr int kBarTmem = 5;                        // epilogue warps + MMA warp, before dealloc

// Launch parameters: the decode parameters plus, per rotation pair j, the phase step theta_j as
// 64-bit fixed-point turns (theta_j / 2 pi * 2^64), cos / sin of theta_j and of 32 theta_j, and
// sin 2 theta_j and 1 - cos 2 theta_j, all computed on the host in double precision.
struct RopeParams {
    Params p;
    unsigned long long phi[kRopePairs];
    float c1[kRopePairs], s1[kRopePairs], c32[kRopePairs], s32[kRopePairs];
    float s2[kRopePairs], h2[kRopePairs];
    int pairing;  // 0: pair j = (j, j + d/2); 1: pair j = (2j, 2j + 1)
};

template <int RK, int RV>
struct RopeShape {
    using F = Fast<2, RK, RV>;
    // MMAs of K = 16 per page: a rank that is not a multiple of 16 (72) takes one more step whose
    // upper half multiplies zero columns of A (its B half lies past the K-plane, in the first
    // 1 KB of the V-plane: rows below the token's own, so written for every valid token)
    static constexpr int KSTEPS = (RK + 15) / 16;
    static constexpr int KPAD = KSTEPS * 16;
    // TMEM columns: three 64-column accumulators (the MMA runs up to two pages ahead of the
    // epilogue), then two A slots of W_up,t^K (two bf16 per column) followed by the mu step's
    // (mu_hi, mu_lo, 0, ...) in 8 more columns
    static constexpr int NACC = 3;
    static constexpr int A_BASE = NACC * 64;
    static constexpr int A_COLS = KPAD / 2 + 8;
    static constexpr int A_STRIDE = A_COLS <= 64 ? 64 : A_COLS <= 96 ? 96 : 128;
    static constexpr int TMEM_COLS = A_BASE + 2 * A_STRIDE <= 256 ? 256 : 512;
    static constexpr uint32_t IDESC = umma_idesc_bf16(kRopeD, 64, 0, 0);
    static_assert(RK % 8 == 0 && (RK % 32 == 0 || RK % 32 == 8), "W_up,t^K rows in 16- and 8-column TMEM stores");
    static_assert(A_COLS <= A_STRIDE, "A slot");
    static_assert(F::PPS == 1 && F::TT == 64, "one page per pipeline step");
    static_assert(F::S_WARPS == 4 && F::V_WARPS == 4, "four epilogue and four value warps");
};

struct RopeLayout {
    int ones, red, bars, tmem, total;
};

template <int RK, int RV>
__host__ __device__ inline RopeLayout rope_layout(int stages, int stage_bytes, int B) {
    RopeLayout L;
    int o = (async_layout<2, RK, RV, kRopeD, kRopeWst>(stages, stage_bytes, B).total + 127) & ~127;
    L.ones = o;  o += 2 * 64 * 16;                // B operand of the mu step: (1, 1, 0...) and zeros
    L.red = o;   o += 2 * 4 * 64 * 4;             // per-warp partial scores, two page slots
    L.bars = o;  o += 10 * 8;                     // aful[2], afree[2], tfull[3], tfree[3]
    L.tmem = o;  o += 16;
    L.total = o;
    return L;
}

template <int RK, int RV>
__global__ void __launch_bounds__(kRopeThreads, 1) decode_rope_kernel(const __grid_constant__ RopeParams rp) {
    using Z = RopeShape<RK, RV>;
    using F = typename Z::F;
    constexpr int ES = 2, D = kRopeD;
    const Params &p = rp.p;
    extern __shared__ __align__(128) char smem[];
    const ASmem a = carve_async<ES, RK, RV, D, kRopeWst>(smem, p);
    const Smem &s = a.s;
    const RopeLayout RL = rope_layout<RK, RV>(p.stages, p.stage_bytes, p.B);
    char *ones = smem + RL.ones;
    float *red4 = reinterpret_cast<float *>(smem + RL.red);
    uint64_t *aful = reinterpret_cast<uint64_t *>(smem + RL.bars);
    uint64_t *afree = aful + 2, *tfull = aful + 4, *tfree = aful + 7;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(smem + RL.tmem);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const bool pass1 = p.cur_k != nullptr;

    // set-up that reads no input runs before the previous kernel in the stream has finished
    if (tid == 0) {
        for (int i = 0; i < kQSlots; ++i) mbar_init(&a.qready[i], kMThreads);
        for (int i = 0; i < 2; ++i) {
            mbar_init(&a.stfull[i], F::V_THREADS);  // the value warps hold a run's state
            mbar_init(&a.stfree[i], kMThreads);
            mbar_init(&aful[i], 1);
            mbar_init(&afree[i], 1);
        }
        for (int i = 0; i < Z::NACC; ++i) {
            mbar_init(&tfull[i], 1);
            mbar_init(&tfree[i], 4);
        }
    }
    if (warp == kMmaWarp) {
        tmem_alloc(tmem_slot, Z::TMEM_COLS);
        // the B operand of the mu step: a (1, 1) pair per token, then a zero granule
        uint4 *o4 = reinterpret_cast<uint4 *>(ones);
        for (int i = lane; i < 128; i += 32)
            o4[i] = i < 64 ? make_uint4(0x3f803f80u, 0u, 0u, 0u) : make_uint4(0u, 0u, 0u, 0u);
        fence_proxy_async_smem();
        tc_fence_before();
    }
    pdl_wait();  // inputs may come from the previous kernel in the stream
    // empty: one arrival per page from the MMA warp's commit and one from each value warp;
    // pfull: the epilogue threads (a page's partial scores); pempty: the value threads
    Range rg = prologue(p, s, kComputeThreads / 2, F::V_THREADS, 1 + F::V_WARPS);
    order_runs(p, s, rg);
    pdl_trigger();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;

    if (warp == kComputeWarps) {
        if (rg.A0 < rg.A1) named_bar_sync(kBarStart, kMThreads + 32);
        producer(p, s, rg);
        return;
    }

    if (warp == kMmaWarp) {
        // ------------------------------------------------------------------------- MMA warp
        int it = 0, stage = 0, r = 0;
        uint32_t ph = 0;
        const bool has_mu = p.mu_k != nullptr;
        const uint64_t ones_desc = umma_desc(smem_addr(ones), 1024, 128);
        for (int pass = 0; pass < 3; ++pass)
        for (int64_t u = rg.lo[pass]; u < rg.hi[pass]; ++r) {
            const Run R = locate_run(p, s, u, rg.hi[pass]);
            const int as = r & 1;
            const uint32_t acol = tmem_base + Z::A_BASE + as * Z::A_STRIDE;
            if (lane == 0) mbar_wait(&aful[as], (r >> 1) & 1, s.abort_flag, p.err);
            for (int k = 0; k < R.npages; ++k, ++it) {
                const int b = it % Z::NACC;
                if (lane == 0) {
                    mbar_wait(&s.full[stage], ph, s.abort_flag, p.err);
                    if (it >= Z::NACC)
                        mbar_wait(&tfree[b], ((it - Z::NACC) / Z::NACC) & 1, s.abort_flag, p.err);
                    tc_fence_after();
                    const uint32_t d = tmem_base + b * 64;
                    const uint32_t bbase = smem_addr(s.ring + stage * p.stage_bytes);
#pragma unroll
                    for (int st = 0; st < Z::KSTEPS; ++st)
                        umma_bf16_ts(d, acol + st * 8, umma_desc(bbase + st * 2048, 1024, 128),
                                     Z::IDESC, st > 0);
                    if (has_mu) umma_bf16_ts(d, acol + Z::KPAD / 2, ones_desc, Z::IDESC, true);
                    umma_commit(&tfull[b]);
                    umma_commit(&s.empty[stage]);  // the K-plane has been read
                    if (k == R.npages - 1) umma_commit(&afree[as]);
                }
                __syncwarp();
                if (++stage == p.stages) {
                    stage = 0;
                    ph ^= 1u;
                }
            }
            u = R.run_end;
        }
        // every MMA has completed before TMEM is released, even after an abort
        if (lane == 0 && it > 0) {
            volatile int never = 0;
            mbar_wait(&tfull[(it - 1) % Z::NACC], ((it - 1) / Z::NACC) & 1, &never, p.err);
        }
        named_bar_sync(kBarTmem, 128 + 32);  // the epilogue warps have read every buffer
        tc_fence_after();
        tmem_dealloc(tmem_base, Z::TMEM_COLS);
        return;
    }

    if (tid >= kMBase) {
        // ------------------------------------------------------------------ management warps
        const int mt = tid - kMBase;
        auto finish = [&](const Run &R, int64_t u, int k) {
            m_finish<ES, RK, RV, D, F::TT, F::NTG, kRopeWst>(p, a, R, u, rg, k & 1, (k >> 1) & 1,
                                                            k % kQSlots, mt);
        };
        // this thread's row of W_up,t^K is TMEM lane `row` (the warp's lane quarter)
        const int row = 32 * (warp & 3) + lane;
        const uint32_t tlane = tmem_base + (static_cast<uint32_t>(32 * (warp & 3)) << 16);
        int r = 0;
        Run q0{}, q1{};
        int64_t u0 = 0, u1 = 0;
        for (int pass = 0; pass < 3; ++pass)
        for (int64_t u = rg.lo[pass]; u < rg.hi[pass];) {
            const Run R = locate_run(p, s, u, rg.hi[pass]);
            const int slot = r % kQSlots, as = r & 1;
            if (r == 0) named_bar_arrive(kBarStart, kMThreads + 32);  // the ring may start
            // W_up,t^K of head R.h and mu^K_t into A slot `as` once run r - 2's MMAs have read it
            const int64_t hl = (static_cast<int64_t>(R.h) * p.T + p.loop) * D;
            const uint4 *W4 = reinterpret_cast<const uint4 *>(
                static_cast<const char *>(p.w_up_k) + (hl + row) * (RK * ES));
            uint32_t wv[RK / 2];
#pragma unroll
            for (int g = 0; g < RK / 8; ++g) {
                const uint4 w = W4[g];
                wv[4 * g] = w.x;
                wv[4 * g + 1] = w.y;
                wv[4 * g + 2] = w.z;
                wv[4 * g + 3] = w.w;
            }
            const float mu = p.mu_k ? p.mu_k[hl + row] : 0.f;
            const __nv_bfloat16 hi = __float2bfloat16_rn(mu);
            const __nv_bfloat16 lo = __float2bfloat16_rn(mu - __bfloat162float(hi));
            uint32_t mv[8] = {static_cast<uint32_t>(__bfloat16_as_ushort(hi)) |
                                  (static_cast<uint32_t>(__bfloat16_as_ushort(lo)) << 16),
                              0u, 0u, 0u, 0u, 0u, 0u, 0u};
            if (r >= 2) mbar_wait(&afree[as], ((r - 2) >> 1) & 1, s.abort_flag, p.err);
            tc_fence_after();
            const uint32_t acol = tlane + Z::A_BASE + as * Z::A_STRIDE;
#pragma unroll
            for (int c = 0; c < RK / 32; ++c) {
                uint32_t part[16];
#pragma unroll
                for (int i = 0; i < 16; ++i) part[i] = wv[16 * c + i];
                tmem_st16u(acol + 16 * c, part);
            }
            if constexpr (RK % 32 == 8) {  // the last 8 K elements, then the zero pad of the step
                const uint32_t tail[8] = {wv[RK / 2 - 4], wv[RK / 2 - 3], wv[RK / 2 - 2], wv[RK / 2 - 1], 0u, 0u, 0u, 0u};
                tmem_st8u(acol + (RK / 32) * 16, tail);
            }
            tmem_st8u(acol + Z::KPAD / 2, mv);
            tmem_wait_st();
            tc_fence_before();
            m_sync();
            if (mt == 0) mbar_arrive(&aful[as]);
            m_setup<ES, RK, RV, D, false, kRopeWst>(p, a, R.b, R.h, slot, mt, false);
            mbar_arrive(&a.qready[slot]);
            if (r >= 2) finish(q0, u0, r - 2);
            q0 = q1;
            u0 = u1;
            q1 = R;
            u1 = u;
            ++r;
            u = R.run_end;
        }
        if (r >= 2) finish(q0, u0, r - 2);
        if (r >= 1) finish(q1, u1, r - 1);
        for (int b = 0; b < p.B; ++b) {  // no cached token: pass 1 attends to the current token
            if (s.lens[b] != 0) continue;
            for (int h = 0; h < p.H; ++h) {
                if ((b * p.H + h) % gridDim.x != blockIdx.x) continue;
                const int64_t orow = (static_cast<int64_t>(b) * p.H + h) * D;
                if (!pass1 && mt == 0) atomicOr(p.err, LLA_DEVERR_EMPTY_PASS2);
                for (int e = mt; e < D; e += kMThreads)
                    store_elem(p.out, orow + e, pass1 ? load_elem(p.cur_v, orow + e, p.io_bf16) : 0.f,
                               p.io_bf16);
            }
        }
        cp_async_wait_all();
        return;
    }

    if (warp < F::S_WARPS) {
        // ------------------------------------------------------------------- epilogue warps
        // lane m = key dimension m; its rotation pair j and its role in the pair
        const int m = tid;
        const int j = rp.pairing ? (m >> 1) : (m & (kRopePairs - 1));
        const bool upper = rp.pairing ? (m & 1) : (m >= kRopePairs);
        const int ia = rp.pairing ? 2 * j : j, ib = rp.pairing ? 2 * j + 1 : j + kRopePairs;
        const unsigned long long phi = rp.phi[j];
        const float c1 = rp.c1[j], s1 = rp.s1[j], c32 = rp.c32[j], s32 = rp.s32[j];
        const float s2 = rp.s2[j], h2 = rp.h2[j];
        const float2 nlam = make_float2(-2.f * h2, -2.f * h2);  // -(2 - 2 cos 2 theta_j)
        const uint32_t tlane = tmem_base + (static_cast<uint32_t>(32 * warp) << 16);
        int it = 0, r = 0;
        for (int pass = 0; pass < 3; ++pass)
        for (int64_t u = rg.lo[pass]; u < rg.hi[pass]; ++r) {
            const Run R = locate_run(p, s, u, rg.hi[pass]);
            const int qslot = r % kQSlots;
            mbar_wait(&a.qready[qslot], (r / kQSlots) & 1, s.abort_flag, p.err);
            // element m of rot(q, Delta) = Re(G e^{i Delta theta_j}), scaled to log2 units
            float Gr, Gi;
            {
                const float *qv = a.qlat + qslot * a.qslot;
                const float qa = qv[ia], qb = qv[ib];
                Gr = (upper ? qb : qa) * p.scale_log2;
                Gi = (upper ? -qa : qb) * p.scale_log2;
            }
            const int P = pass1 ? R.Lb : R.Lb - 1;  // the query's position
            for (int k = 0; k < R.npages; ++k, ++it) {
                const int b = it % Z::NACC, slot = it & 1;
                const int pg = R.pg0 + k;
                // exact phase of the page's first token: Delta0 theta_j in turns, mod 1
                const int delta0 = P - pg * kBlockTokens;  // >= 0: the page holds a cached token
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
                    // the half's first token: z e^{-i 32 hv theta}; the odd chain one token later
                    const float er = hv ? fmaf(zr, c32, zi * s32) : zr;
                    const float ei = hv ? fmaf(zi, c32, -zr * s32) : zi;
                    const float orr = fmaf(er, c1, ei * s1), oi = fmaf(ei, c1, -er * s1);
                    X[hv] = make_float2(er, orr);
                    DD[hv] = make_float2(fmaf(er, h2, ei * s2), fmaf(orr, h2, oi * s2));
                }
                uint32_t v0[32], v1[32];  // this dimension of tokens 0..31 and 32..63
                mbar_wait(&tfull[b], (it / Z::NACC) & 1, s.abort_flag, p.err);
                tc_fence_after();
                const uint32_t tcol = tlane + b * 64;
                tmem_ld32_nowait(tcol, v0);
                tmem_ld32_nowait(tcol + 32, v1);
                tmem_wait_ld(v0);
                tmem_wait_ld(v1);
                // this dimension's score terms in place
#pragma unroll
                for (int t = 0; t < 16; ++t) {
                    float2 a0 = make_float2(__uint_as_float(v0[2 * t]), __uint_as_float(v0[2 * t + 1]));
                    float2 a1 = make_float2(__uint_as_float(v1[2 * t]), __uint_as_float(v1[2 * t + 1]));
                    a0 = __fmul2_rn(a0, X[0]);
                    a1 = __fmul2_rn(a1, X[1]);
                    v0[2 * t] = __float_as_uint(a0.x);
                    v0[2 * t + 1] = __float_as_uint(a0.y);
                    v1[2 * t] = __float_as_uint(a1.x);
                    v1[2 * t + 1] = __float_as_uint(a1.y);
                    DD[0] = __ffma2_rn(nlam, X[0], DD[0]);
                    DD[1] = __ffma2_rn(nlam, X[1], DD[1]);
                    X[0] = __fadd2_rn(X[0], DD[0]);
                    X[1] = __fadd2_rn(X[1], DD[1]);
                }
                // sum over the 128 dimensions of each token: the terms go back to TMEM and return
                // in the 16x256b layout (4 dimensions x 16 tokens per thread), are summed over
                // the 4 dimensions, then over the 8 threads of each token group by shuffles
                tmem_st32u_nowait(tcol, v0);
                tmem_st32u_nowait(tcol + 32, v1);
                tmem_wait_st();
                tmem_ld16x256_x8_nowait(tcol, v0);                                  // dims +0, +8
                tmem_ld16x256_x8_nowait(tcol + (static_cast<uint32_t>(16) << 16), v1);  // +16, +24
                tmem_wait_ld(v0);
                tmem_wait_ld(v1);
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&tfree[b]);  // the buffer may take page it + NACC
                float S[16];  // S[2k + e]: token 8k + 2(lane % 4) + e, summed over 4 dimensions
#pragma unroll
                for (int k8 = 0; k8 < 8; ++k8) {
                    const float2 a = __fadd2_rn(
                        make_float2(__uint_as_float(v0[4 * k8]), __uint_as_float(v0[4 * k8 + 1])),
                        make_float2(__uint_as_float(v0[4 * k8 + 2]), __uint_as_float(v0[4 * k8 + 3])));
                    const float2 c = __fadd2_rn(
                        make_float2(__uint_as_float(v1[4 * k8]), __uint_as_float(v1[4 * k8 + 1])),
                        make_float2(__uint_as_float(v1[4 * k8 + 2]), __uint_as_float(v1[4 * k8 + 3])));
                    const float2 sum = __fadd2_rn(a, c);
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
                mbar_wait(&s.pempty[slot], ((it >> 1) & 1) ^ 1u, s.abort_flag, p.err);
                *reinterpret_cast<float2 *>(red4 + slot * 256 + warp * 64 + 2 * lane) =
                    make_float2(S[0], S[1]);
                mbar_arrive(&s.pfull[slot]);
            }
            u = R.run_end;
        }
        tc_fence_before();
        named_bar_arrive(kBarTmem, 128 + 32);
        return;
    }

    // --------------------------------------------------------------------------- value warps
    // Per page: the online softmax over the page's scores (threads vt < 64, one token each),
    // then sum_i p_i c_v,i from the V-plane.
    const int vt = tid - F::S_THREADS, vwarp = warp - F::S_WARPS;
    const int vc = vt % F::VC, tg = vt / F::VC;
    const bool vwork = tg < F::NTG;
    constexpr int AV = F::UPT * F::VE;
    int it = 0, stage = 0, r = 0;
    uint32_t ph = 0;
    for (int pass = 0; pass < 3; ++pass)
    for (int64_t u = rg.lo[pass]; u < rg.hi[pass]; ++r) {
        const Run R = locate_run(p, s, u, rg.hi[pass]);
        const int rslot = r & 1;
        float m_run = -INFINITY, l_part = 0.f;
        float accv[AV];
#pragma unroll
        for (int e = 0; e < AV; ++e) accv[e] = 0.f;
        for (int k = 0; k < R.npages; ++k, ++it) {
            const int slot = it & 1;
            const uint32_t pph = (it >> 1) & 1;
            const char *sb = s.ring + stage * p.stage_bytes;
            const int nvalid = min(kBlockTokens, R.Lb - (R.pg0 + k) * kBlockTokens);
            float *wmax = s.misc + kAWmax + slot * 8;
            float *pring = s.psm + slot * kComputeThreads;
            mbar_wait(&s.pfull[slot], pph, s.abort_flag, p.err);
            float xs = -INFINITY;
            if (vt < kBlockTokens) {
                const float *rs = red4 + slot * 256;
                const float sc = (rs[vt] + rs[64 + vt]) + (rs[128 + vt] + rs[192 + vt]);
                xs = vt < nvalid ? sc : -INFINITY;
                const float lm = warp_max(xs);
                if (lane == 0) wmax[vwarp] = lm;
            }
            mbar_arrive(&s.pempty[slot]);  // the partial scores are read
            named_bar_sync(kBarTok, F::V_THREADS);
            if (vt < kBlockTokens) {
                const float m_new = fmaxf(m_run, fmaxf(wmax[0], wmax[1]));
                const float alpha = exp2f(m_run - m_new);
                m_run = m_new;
                const float pv = vt < nvalid ? exp2f(xs - m_new) : 0.f;
                pring[vt] = pv;
                l_part = fmaf(l_part, alpha, pv);
                if (vt == 0) s.misc[kAPAlpha + slot] = alpha;
            }
            named_bar_sync(kBarTok, F::V_THREADS);
            mbar_wait(&s.full[stage], ph, s.abort_flag, p.err);
            if (vwork) value_step<ES, RK, RV>(accv, sb, pring, s.misc[kAPAlpha + slot], nvalid, vc, tg);
            __syncwarp();
            if (lane == 0) mbar_arrive(&s.empty[stage]);  // V-plane read
            if (++stage == p.stages) {
                stage = 0;
                ph ^= 1u;
            }
        }
        if (r >= 2) mbar_wait(&a.stfree[rslot], ((r - 2) >> 1) & 1, s.abort_flag, p.err);
        if (vt < kBlockTokens) a.lred[rslot * kLredSlot + vt] = l_part;
        if (vt == 0) s.misc[kAM + rslot] = m_run;
        if (vwork) value_store<ES, RK, RV>(a.red + rslot * a.redslot, accv, vc, tg);
        mbar_arrive(&a.stfull[rslot]);
        u = R.run_end;
    }
}

template <int RK, int RV>
lla_status launch_rope(const RopeParams &prm, int grid, int smem, cudaStream_t stream) {
    static DeviceOnce configured;
    return launch_kernel(decode_rope_kernel<RK, RV>, configured, prm, grid, smem, stream,
                         kRopeThreads);
}

template <int RK, int RV>
int rope_layout_bytes(int stages, int stage_bytes, int B) {
    return rope_layout<RK, RV>(stages, stage_bytes, B).total;
}

using RopeLauncher = lla_status (*)(const RopeParams &, int, int, cudaStream_t);
using RopeLayoutFn = int (*)(int, int, int);
struct RopeEntry {
    RopeLauncher launch;
    RopeLayoutFn layout;
};
RopeEntry rope_entry(int es, int d, int r_k, int r_v) {
    if (es != 2 || d != kRopeD) return RopeEntry{nullptr, nullptr};
    // the other shapes run on the tensor-core value path (lla_decode_rope_tc.cu)
    if (r_k == 192 && r_v == 320) return RopeEntry{launch_rope<192, 320>, rope_layout_bytes<192, 320>};
    return RopeEntry{nullptr, nullptr};
}

// Ring stages that fit beside the fixed layout (head pages of stage_bytes each).
int rope_stages(const RopeEntry &e, int stage_bytes, int B) {
    const int fixed = e.layout(0, stage_bytes, B);
    int stages = (kSmemLimit - fixed) / (stage_bytes + 16);
    return stages > kMaxStages ? kMaxStages : stages;
}

}  // namespace

lla_status decode_rope_fits(int r_k, int r_v, int es, int d, int B) {
    if (decode_rope_tc_supported(es, d, r_k, r_v)) return LLA_OK;
    const RopeEntry e = rope_entry(es, d, r_k, r_v);
    if (!e.launch) return LLA_ERR_UNSUPPORTED;
    const int hpb = static_cast<int>(head_page_bytes(r_k, r_v, es));
    return rope_stages(e, hpb, B) >= 2 ? LLA_OK : LLA_ERR_UNSUPPORTED;
}

void rope_tables(double base, int d, RopeTables *t) {
    const double two_pi = 6.283185307179586476925286766559;
    for (int j = 0; j < kRopePairs; ++j) {
        const double theta = pow(base, -2.0 * j / d);
        const double turns = theta / two_pi;  // < 1: theta_j <= 1
        t->phi[j] = static_cast<unsigned long long>(ldexp(turns, 64));
        t->c1[j] = static_cast<float>(cos(theta));
        t->s1[j] = static_cast<float>(sin(theta));
        t->c32[j] = static_cast<float>(cos(32.0 * theta));
        t->s32[j] = static_cast<float>(sin(32.0 * theta));
        t->s2[j] = static_cast<float>(sin(2.0 * theta));
        const double sh = sin(theta);
        t->h2[j] = static_cast<float>(2.0 * sh * sh);  // 1 - cos 2 theta, without cancellation
    }
}

lla_status launch_decode_rope(const DecodeArgs &a, double base, int pairing, cudaStream_t stream) {
    const int es = a.storage_bf16 ? 2 : 4;
    // the rotation tables of this base (kept for the next call with the same base and width)
    struct TableCache {
        double base = 0.0;
        int d = 0;
        RopeTables t;
    };
    static thread_local TableCache cache;
    if (!(cache.base == base && cache.d == a.d)) {
        rope_tables(base, a.d, &cache.t);
        cache.base = base;
        cache.d = a.d;
    }
    const RopeTables &t = cache.t;
    if (decode_rope_tc_supported(es, a.d, a.r_k, a.r_v)) return launch_decode_rope_tc(a, t, pairing, stream);
    const RopeEntry e = rope_entry(es, a.d, a.r_k, a.r_v);
    if (!e.launch) return LLA_ERR_UNSUPPORTED;
    const int hpb = static_cast<int>(head_page_bytes(a.r_k, a.r_v, es));
    const int stages = rope_stages(e, hpb, a.B);
    if (stages < 2) return LLA_ERR_UNSUPPORTED;
    const int smem = e.layout(stages, hpb, a.B);
    const int grid = num_sms();
    if (grid <= 0) return LLA_ERR_CUDA;
    if (a.workspace_bytes < decode_workspace_bytes(a.r_v, a.B, a.H, grid)) return LLA_ERR_WORKSPACE;
    lla_status st = LLA_OK;
    unsigned *err = device_error_word(&st);
    if (st != LLA_OK) return st;

    RopeParams rp = {};
    Params &p = rp.p;
    p.T = a.T; p.H = a.H; p.d = a.d; p.r_k = a.r_k; p.r_v = a.r_v; p.loop = a.loop;
    p.absorbed = 1; p.io_bf16 = a.io_bf16;
    p.scale_log2 = a.scale * 1.4426950408889634f;
    p.w_up_k = a.w_up_k; p.w_up_v = a.w_up_v; p.mu_k = a.mu_k; p.mu_v = a.mu_v;
    p.pool = static_cast<const char *>(a.pool);
    p.num_blocks = a.num_blocks;
    p.block_bytes = static_cast<int64_t>(hpb) * a.H;
    p.head_page_bytes = hpb;
    p.kplane_bytes = kBlockTokens * a.r_k * es;
    p.block_table = a.block_table; p.max_blocks = a.max_blocks;
    p.context_lens = a.context_lens; p.B = a.B; p.max_ctx = a.max_ctx;
    p.q = a.q; p.cur_k = a.cur_k; p.cur_v = a.cur_v; p.out = a.out;
    const size_t part = static_cast<size_t>(grid) * 2 * (a.r_v + 2) * sizeof(float);
    const size_t part_al = (part + 255) & ~static_cast<size_t>(255);
    p.partials = static_cast<float *>(a.workspace);
    p.counters = reinterpret_cast<int *>(static_cast<char *>(a.workspace) + part_al);
    p.pps = 1; p.stages = stages; p.stage_bytes = hpb;
    p.err = err;
    memcpy(rp.phi, t.phi, sizeof(rp.phi));
    memcpy(rp.c1, t.c1, sizeof(rp.c1));
    memcpy(rp.s1, t.s1, sizeof(rp.s1));
    memcpy(rp.c32, t.c32, sizeof(rp.c32));
    memcpy(rp.s32, t.s32, sizeof(rp.s32));
    memcpy(rp.s2, t.s2, sizeof(rp.s2));
    memcpy(rp.h2, t.h2, sizeof(rp.h2));
    rp.pairing = pairing;
    return e.launch(rp, grid, smem, stream);
}

}  // namespace lla
