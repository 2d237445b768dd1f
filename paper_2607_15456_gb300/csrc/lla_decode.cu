// lla_decode.cu -- one decode call of Looped Latent Attention over the paged latent cache
// (App. A "Decoding and caching", App. J "Absorbed attention"), and the same kernel without the
// codec for the uncompressed loop-t comparator ("Teacher cache", Sec. 3).
//
// What one launch computes, for every sequence b and head h at loop t:
//   q~ = W_up,t^K^T q,  beta = q . mu^K_t                       (key up-projection on the query)
//   s_i = scale (q~ . c_k,i + beta)          for the cached tokens i < L_b
//   s_cur = scale q . k_cur                  (pass 1 only: the current token's exact key)
//   o = (W_up,t^V sum_i p_i c_v,i + (sum_i p_i) mu^V_t + p_cur v_cur) / (sum_i p_i + p_cur)
// with p = exp(s - max s): the softmax over the reconstructed keys and values of Eq. decode,
// without ever forming them.
//
// GB300 mapping (HBM-bound: about one flop per byte of latent):
//   * Work units are (sequence, head, 64-token page).  All units of the batch are split into
//     equal contiguous ranges, one per CTA, one CTA per SM (persistent "stream-K" split), so a
//     batch of mixed lengths keeps every SM streaming until the end.
//   * One producer warp walks the CTA's range and moves each page's K-plane and V-plane (one
//     contiguous head page) into a shared-memory ring with the TMA bulk-copy engine
//     (cp.async.bulk + mbarrier transaction counts), evict-first in L2.
//   * Eight consumer warps compute scores from the K-plane (granule-interleaved so that
//     consecutive lanes read consecutive 16-byte words), an exact online softmax (warp-shuffle
//     max, exp2), and accumulate sum_i p_i c_v,i in latent space from the V-plane.
//   * A range that covers a (sequence, head) completely finishes it in place; ranges that split
//     one write (m, l, o_latent) partials, and the last CTA to arrive (atomic counter) merges
//     them by log-sum-exp, adds the current token and applies W_up,t^V, mu^V_t and 1/l.
#include <cuda_runtime.h>
#include <math.h>

#include "lla_device.cuh"
#include "lla_internal.h"

namespace lla {
namespace {

constexpr int kComputeWarps = 8;
constexpr int kComputeThreads = kComputeWarps * 32;
constexpr int kThreads = kComputeThreads + 32;  // + one producer warp
constexpr int kMaxStages = 8;
constexpr int kSmemLimit = 227 * 1024;
constexpr int kStepTargetBytes = 32 * 1024;
constexpr int kBarAll = 1;   // named barrier over the 256 consumer threads
constexpr int kBarTok = 2;   // named barrier over the score-owning threads

struct Params {
    int T, H, d, r_k, r_v, loop, absorbed, io_bf16;
    float scale_log2;
    const void *w_up_k, *w_up_v;
    const float *mu_k, *mu_v;
    const char *pool;
    int64_t num_blocks, block_bytes;
    int head_page_bytes, kplane_bytes;
    const int32_t *block_table;
    int max_blocks;
    const int32_t *context_lens;
    int B, max_ctx;
    const void *q, *cur_k, *cur_v;
    void *out;
    float *partials;  // [gridDim.x][2][r_v + 2]
    int *counters;    // [B * H]
    int pps, stages, stage_bytes;
    unsigned *err;
};

struct Layout {
    int ring, full, empty, prefix, lens, qlat, qfull, spart, psm, tmp, red, lred, ovec, misc,
        total;
};

__host__ __device__ inline int up16(int x) { return (x + 15) & ~15; }

__host__ __device__ inline Layout make_layout(int stages, int stage_bytes, int B, int r_k, int r_v,
                                              int d) {
    Layout L;
    int o = 0;
    L.ring = o;
    o += stages * stage_bytes;
    L.full = o;
    o += stages * 8;
    L.empty = o;
    o += stages * 8;
    L.prefix = o;
    o += up16((B + 1) * 8);
    L.lens = o;
    o += up16(B * 4);
    L.qlat = o;
    o += up16((r_k > d ? r_k : d) * 4);
    L.qfull = o;
    o += up16(d * 4);
    L.spart = o;
    o += kComputeThreads * 4;
    L.psm = o;
    o += kComputeThreads * 4;
    L.tmp = o;
    o += 2 * kComputeThreads * 4;
    L.red = o;
    o += 8 * kComputeThreads * 4;
    L.lred = o;
    o += kComputeThreads * 4;
    L.ovec = o;
    o += up16((r_v > d ? r_v : d) * 4);
    L.misc = o;
    o += 32 * 4;
    L.total = o;
    return L;
}

// misc slots
constexpr int kMiscAlpha = 0, kMiscM = 1, kMiscL = 2, kMiscBeta = 3, kMiscScur = 4,
              kMiscWmax = 8, kMiscAbort = 16, kMiscLast = 17;

template <int ES, int GB>
__device__ __forceinline__ void load_gran(const char *p, float (&v)[GB / ES]) {
    if constexpr (GB == 16) {
        const uint4 u = *reinterpret_cast<const uint4 *>(p);
        if constexpr (ES == 2) {
            float2 a = bf2_to_f2(u.x), b = bf2_to_f2(u.y), c = bf2_to_f2(u.z), e = bf2_to_f2(u.w);
            v[0] = a.x; v[1] = a.y; v[2] = b.x; v[3] = b.y;
            v[4] = c.x; v[5] = c.y; v[6] = e.x; v[7] = e.y;
        } else {
            v[0] = __uint_as_float(u.x); v[1] = __uint_as_float(u.y);
            v[2] = __uint_as_float(u.z); v[3] = __uint_as_float(u.w);
        }
    } else {
        const uint32_t u = *reinterpret_cast<const uint32_t *>(p);
        if constexpr (ES == 2) {
            const float2 a = bf2_to_f2(u);
            v[0] = a.x; v[1] = a.y;
        } else {
            v[0] = __uint_as_float(u);
        }
    }
}

// Two consecutive elements (even index) of a storage-dtype array.
template <int ES>
__device__ __forceinline__ float2 load_pair(const void *base, int64_t i) {
    if constexpr (ES == 2) return bf2_to_f2(reinterpret_cast<const uint32_t *>(base)[i >> 1]);
    else return reinterpret_cast<const float2 *>(base)[i >> 1];
}

__device__ __forceinline__ int seq_of_unit(const int64_t *prefix, int B, int64_t u) {
    int lo = 0, hi = B - 1;
    while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (prefix[mid + 1] > u) hi = mid;
        else lo = mid + 1;
    }
    return lo;
}

// CTA owning unit u when U units are split into Geff equal contiguous ranges.
__device__ __forceinline__ int owner_of(int64_t u, int64_t U, int Geff) {
    return static_cast<int>(((u + 1) * Geff - 1) / U);
}

__device__ __forceinline__ int64_t range_start(int c, int64_t U, int Geff) {
    return static_cast<int64_t>(c) * U / Geff;
}

// Query set-up of one (sequence, head): q in d-space, q~ = W_up,t^K^T q (or q itself for the
// dense comparator) and beta = q . mu^K_t.  All consumer threads.
template <int ES>
__device__ void setup_query(const Params &p, int b, int h, float *qfull, float *qlat, float *tmp,
                            float *misc) {
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int64_t qoff = (static_cast<int64_t>(b) * p.H + h) * p.d;
    for (int e = tid; e < p.d; e += kComputeThreads) qfull[e] = load_elem(p.q, qoff + e, p.io_bf16);
    named_bar_sync(kBarAll, kComputeThreads);
    if (p.absorbed) {
        const int njp = p.r_k >> 1;
        const int neg = kComputeThreads / njp;
        const int jp = tid % njp, eg = tid / njp;
        if (eg < neg) {
            const int64_t w0 = (static_cast<int64_t>(h) * p.T + p.loop) * p.d * p.r_k;
            float a0 = 0.f, a1 = 0.f;
            for (int e = eg; e < p.d; e += neg) {
                const float2 w = load_pair<ES>(p.w_up_k, w0 + static_cast<int64_t>(e) * p.r_k + 2 * jp);
                const float qe = qfull[e];
                a0 = fmaf(w.x, qe, a0);
                a1 = fmaf(w.y, qe, a1);
            }
            tmp[eg * p.r_k + 2 * jp] = a0;
            tmp[eg * p.r_k + 2 * jp + 1] = a1;
        }
        if (warp == kComputeWarps - 1) {
            float bsum = 0.f;
            if (p.mu_k) {
                const float *mu = p.mu_k + (static_cast<int64_t>(h) * p.T + p.loop) * p.d;
                for (int e = lane; e < p.d; e += 32) bsum = fmaf(qfull[e], mu[e], bsum);
            }
            bsum = warp_sum(bsum);
            // written after the partial sums of this warp; read after the next barrier
            if (lane == 0) misc[kMiscBeta] = bsum;
        }
        named_bar_sync(kBarAll, kComputeThreads);
        for (int j = tid; j < p.r_k; j += kComputeThreads) {
            float s = 0.f;
            for (int g = 0; g < neg; ++g) s += tmp[g * p.r_k + j];
            qlat[j] = s;
        }
    } else {
        for (int e = tid; e < p.d; e += kComputeThreads) qlat[e] = qfull[e];
        if (tid == 0) misc[kMiscBeta] = 0.f;
    }
    named_bar_sync(kBarAll, kComputeThreads);
}

// Final output of one (sequence, head) from its cached softmax state: maximum m (log2 units),
// mass l and latent value sum ovec (all relative to m).  All consumer threads.
template <int ES>
__device__ void finish_output(const Params &p, int b, int h, float m, float l, const float *ovec,
                              const float *qfull, float *misc) {
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const bool pass1 = p.cur_k != nullptr;
    const int64_t row = (static_cast<int64_t>(b) * p.H + h) * p.d;
    if (pass1 && warp == 0) {
        float s = 0.f;
        for (int e = lane; e < p.d; e += 32) s = fmaf(qfull[e], load_elem(p.cur_k, row + e, p.io_bf16), s);
        s = warp_sum(s);
        if (lane == 0) misc[kMiscScur] = s * p.scale_log2;
    }
    named_bar_sync(kBarAll, kComputeThreads);
    float M = m, pc = 0.f;
    if (pass1) {
        const float sc = misc[kMiscScur];
        M = fmaxf(m, sc);
        pc = exp2f(sc - M);
    }
    const float wl = exp2f(m - M);
    const float lc = l * wl;  // cached softmax mass
    const float inv = 1.f / (lc + pc);
    if (p.absorbed) {
        const int64_t w0 = (static_cast<int64_t>(h) * p.T + p.loop) * p.d * p.r_v;
        const float *mu = p.mu_v ? p.mu_v + (static_cast<int64_t>(h) * p.T + p.loop) * p.d : nullptr;
        const int njp = p.r_v >> 1;
        for (int e = warp; e < p.d; e += kComputeWarps) {
            float acc = 0.f;
            for (int jp = lane; jp < njp; jp += 32) {
                const float2 w = load_pair<ES>(p.w_up_v, w0 + static_cast<int64_t>(e) * p.r_v + 2 * jp);
                acc = fmaf(w.x, ovec[2 * jp], acc);
                acc = fmaf(w.y, ovec[2 * jp + 1], acc);
            }
            acc = warp_sum(acc);
            if (lane == 0) {
                float o = acc * wl;
                if (mu) o = fmaf(lc, mu[e], o);
                if (pass1) o = fmaf(pc, load_elem(p.cur_v, row + e, p.io_bf16), o);
                store_elem(p.out, row + e, o * inv, p.io_bf16);
            }
        }
    } else {
        for (int e = tid; e < p.d; e += kComputeThreads) {
            float o = ovec[e] * wl;
            if (pass1) o = fmaf(pc, load_elem(p.cur_v, row + e, p.io_bf16), o);
            store_elem(p.out, row + e, o * inv, p.io_bf16);
        }
    }
    named_bar_sync(kBarAll, kComputeThreads);
}

template <int ES, int GK, int VB>
__global__ void __launch_bounds__(kThreads, 1) decode_kernel(const Params p) {
    extern __shared__ __align__(128) char smem[];
    const Layout L = make_layout(p.stages, p.stage_bytes, p.B, p.r_k, p.r_v, p.d);
    char *ring = smem + L.ring;
    uint64_t *full = reinterpret_cast<uint64_t *>(smem + L.full);
    uint64_t *empty = reinterpret_cast<uint64_t *>(smem + L.empty);
    int64_t *prefix = reinterpret_cast<int64_t *>(smem + L.prefix);
    int *lens = reinterpret_cast<int *>(smem + L.lens);
    float *qlat = reinterpret_cast<float *>(smem + L.qlat);
    float *qfull = reinterpret_cast<float *>(smem + L.qfull);
    float *spart = reinterpret_cast<float *>(smem + L.spart);
    float *psm = reinterpret_cast<float *>(smem + L.psm);
    float *tmp = reinterpret_cast<float *>(smem + L.tmp);
    float *red = reinterpret_cast<float *>(smem + L.red);
    float *lred = reinterpret_cast<float *>(smem + L.lred);
    float *ovec = reinterpret_cast<float *>(smem + L.ovec);
    float *misc = reinterpret_cast<float *>(smem + L.misc);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(misc + kMiscAbort);
    int *last_flag = reinterpret_cast<int *>(misc + kMiscLast);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int c = blockIdx.x;
    const int hpb = p.head_page_bytes;

    // Inputs may come from the previous kernel in the stream.
    pdl_wait();

    if (tid == 0) {
        for (int s = 0; s < p.stages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], kComputeWarps);
        }
        *abort_flag = 0;
        fence_mbar_init();
    }
    // Units per sequence (H heads x pages), exclusive prefix; lengths checked on the device.
    if (warp == 0) {
        const int cap = min(p.max_ctx, p.max_blocks * kBlockTokens);
        int64_t run = 0;
        for (int b0 = 0; b0 < p.B; b0 += 32) {
            const int b = b0 + lane;
            int np = 0;
            if (b < p.B) {
                int Lb = p.context_lens[b];
                if (Lb < 0 || Lb > cap) {
                    if (c == 0) atomicOr(p.err, LLA_DEVERR_CONTEXT);
                    Lb = max(0, min(Lb, cap));
                }
                lens[b] = Lb;
                np = (Lb + kBlockTokens - 1) / kBlockTokens;
            }
            int v = np;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int n = __shfl_up_sync(0xffffffffu, v, o);
                if (lane >= o) v += n;
            }
            if (b < p.B) prefix[b] = run + static_cast<int64_t>(v - np) * p.H;
            run += static_cast<int64_t>(__shfl_sync(0xffffffffu, v, 31)) * p.H;
        }
        if (lane == 0) prefix[p.B] = run;
    }
    __syncthreads();
    pdl_trigger();

    const int64_t U = prefix[p.B];
    const int Geff = static_cast<int>(U < gridDim.x ? U : gridDim.x);
    int64_t A0 = 0, A1 = 0;
    if (c < Geff) {
        A0 = range_start(c, U, Geff);
        A1 = range_start(c + 1, U, Geff);
    }

    if (warp == kComputeWarps) {
        // ------------------------------------------------------------------ producer warp
        if (lane == 0) {
            const uint64_t pol = policy_evict_first();
            int it = 0;
            for (int64_t u = A0; u < A1;) {
                const int b = seq_of_unit(prefix, p.B, u);
                const int np = static_cast<int>((prefix[b + 1] - prefix[b]) / p.H);
                const int64_t off = u - prefix[b];
                const int h = static_cast<int>(off / np);
                const int pg0 = static_cast<int>(off % np);
                const int64_t seg_end = prefix[b] + static_cast<int64_t>(h + 1) * np;
                const int64_t run_end = seg_end < A1 ? seg_end : A1;
                const int npages = static_cast<int>(run_end - u);
                const int32_t *bt = p.block_table + static_cast<int64_t>(b) * p.max_blocks + pg0;
                for (int k = 0; k < npages; k += p.pps, ++it) {
                    const int stage = it % p.stages;
                    const uint32_t ph = (it / p.stages) & 1;
                    mbar_wait(&empty[stage], ph ^ 1u, abort_flag, p.err);
                    const int n = min(p.pps, npages - k);
                    int32_t blk[4];
                    uint32_t bytes = 0;
                    for (int i = 0; i < n; ++i) {
                        blk[i] = bt[k + i];
                        if (blk[i] < 0 || blk[i] >= p.num_blocks) {
                            atomicOr(p.err, LLA_DEVERR_BLOCK_ID);
                            blk[i] = -1;
                        } else {
                            bytes += hpb;
                        }
                    }
                    mbar_arrive_expect_tx(&full[stage], bytes);
                    char *dst = ring + stage * p.stage_bytes;
                    for (int i = 0; i < n; ++i)
                        if (blk[i] >= 0)
                            bulk_g2s(dst + i * hpb, p.pool + blk[i] * p.block_bytes + static_cast<int64_t>(h) * hpb,
                                     hpb, &full[stage], pol);
                }
                u = run_end;
            }
            if (*abort_flag) {
                // let the copies still in flight land before the CTA exits
                volatile int never = 0;
                const int first = it > p.stages ? it - p.stages : 0;
                for (int j = first; j < it; ++j)
                    mbar_wait(&full[j % p.stages], (j / p.stages) & 1, &never, p.err);
            }
        }
        return;
    }

    // ---------------------------------------------------------------------- consumer warps
    constexpr int KE = GK / ES;  // elements per K granule
    constexpr int VE = VB / ES;  // elements per V unit
    const int TOK = p.pps * kBlockTokens;
    const int SPLIT = kComputeThreads / TOK;
    const int NGK = p.r_k * ES / GK;
    const int NVU = p.r_v * ES / VB;
    const int NTG = kComputeThreads / NVU;
    const int vu = tid % NVU, tg = tid / NVU;
    const bool vthread = tg < NTG;
    const bool pass1 = p.cur_k != nullptr;

    int it = 0;
    for (int64_t u = A0; u < A1;) {
        const int b = seq_of_unit(prefix, p.B, u);
        const int Lb = lens[b];
        const int np = static_cast<int>((prefix[b + 1] - prefix[b]) / p.H);
        const int64_t off = u - prefix[b];
        const int h = static_cast<int>(off / np);
        const int pg0 = static_cast<int>(off % np);
        const int64_t seg_start = prefix[b] + static_cast<int64_t>(h) * np;
        const int64_t seg_end = seg_start + np;
        const int64_t run_end = seg_end < A1 ? seg_end : A1;
        const int npages = static_cast<int>(run_end - u);

        setup_query<ES>(p, b, h, qfull, qlat, tmp, misc);
        const float beta = misc[kMiscBeta];

        float m_run = -INFINITY, l_part = 0.f;
        float accv[VE];
#pragma unroll
        for (int k = 0; k < VE; ++k) accv[k] = 0.f;

        for (int k = 0; k < npages; k += p.pps, ++it) {
            const int stage = it % p.stages;
            const uint32_t ph = (it / p.stages) & 1;
            mbar_wait(&full[stage], ph, abort_flag, p.err);
            const char *sb = ring + stage * p.stage_bytes;
            const int n = min(p.pps, npages - k);
            const int tok0 = (pg0 + k) * kBlockTokens;  // sequence position of the step's row 0
            const int nvalid = min(n * kBlockTokens, Lb - tok0);

            // scores: partial dot products of q~ with the K-plane rows
            {
                const int tk = tid % TOK, sp = tid / TOK;
                const int pi = tk >> 6, ti = tk & 63;
                float acc = 0.f;
                if (tk < nvalid) {
                    const char *kp = sb + pi * hpb + ti * GK;
                    for (int g = sp; g < NGK; g += SPLIT) {
                        float v[KE];
                        load_gran<ES, GK>(kp + g * (kBlockTokens * GK), v);
                        const float *qq = qlat + g * KE;
#pragma unroll
                        for (int e = 0; e < KE; ++e) acc = fmaf(v[e], qq[e], acc);
                    }
                }
                spart[sp * TOK + tk] = acc;
            }
            named_bar_sync(kBarAll, kComputeThreads);
            // online softmax over the step's tokens (threads that own a token)
            if (tid < TOK) {
                float s = 0.f;
                for (int sp = 0; sp < SPLIT; ++sp) s += spart[sp * TOK + tid];
                const bool valid = tid < nvalid;
                const float x = valid ? (s + beta) * p.scale_log2 : -INFINITY;
                const float wm = warp_max(x);
                if (lane == 0) misc[kMiscWmax + warp] = wm;
                named_bar_sync(kBarTok, TOK);
                float ms = misc[kMiscWmax];
                for (int w = 1; w < (TOK >> 5); ++w) ms = fmaxf(ms, misc[kMiscWmax + w]);
                const float m_new = fmaxf(m_run, ms);
                const float alpha = exp2f(m_run - m_new);
                const float pv = valid ? exp2f(x - m_new) : 0.f;
                l_part = fmaf(l_part, alpha, pv);
                psm[tid] = pv;
                if (tid == 0) misc[kMiscAlpha] = alpha;
                m_run = m_new;
            }
            named_bar_sync(kBarAll, kComputeThreads);
            // latent value accumulation: sum_i p_i c_v,i
            if (vthread) {
                const float alpha = misc[kMiscAlpha];
#pragma unroll
                for (int e = 0; e < VE; ++e) accv[e] *= alpha;
                const char *vp = sb + p.kplane_bytes + vu * VB;
                for (int tk = tg; tk < nvalid; tk += NTG) {
                    const float pv = psm[tk];
                    float v[VE];
                    load_gran<ES, VB>(vp + (tk >> 6) * hpb + (tk & 63) * (p.r_v * ES), v);
#pragma unroll
                    for (int e = 0; e < VE; ++e) accv[e] = fmaf(pv, v[e], accv[e]);
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&empty[stage]);
        }

        // reduce the run's softmax state across threads
        if (tid < TOK) lred[tid] = l_part;
        if (vthread) {
#pragma unroll
            for (int e = 0; e < VE; ++e) red[tg * p.r_v + vu * VE + e] = accv[e];
        }
        if (tid == 0) misc[kMiscM] = m_run;
        named_bar_sync(kBarAll, kComputeThreads);
        for (int j = tid; j < p.r_v; j += kComputeThreads) {
            float s = 0.f;
            for (int g = 0; g < NTG; ++g) s += red[g * p.r_v + j];
            ovec[j] = s;
        }
        if (warp == 0) {
            float s = 0.f;
            for (int i = lane; i < TOK; i += 32) s += lred[i];
            s = warp_sum(s);
            if (lane == 0) misc[kMiscL] = s;
        }
        named_bar_sync(kBarAll, kComputeThreads);

        if (u == seg_start && run_end == seg_end) {
            finish_output<ES>(p, b, h, misc[kMiscM], misc[kMiscL], ovec, qfull, misc);
        } else {
            // partial of a (sequence, head) split across CTAs: slot 0 if this is the CTA's first
            // run, slot 1 if its last
            const int slot = (seg_start <= A0) ? 0 : 1;
            float *rec = p.partials + (static_cast<int64_t>(c) * 2 + slot) * (p.r_v + 2);
            if (tid == 0) {
                rec[0] = misc[kMiscM];
                rec[1] = misc[kMiscL];
            }
            for (int j = tid; j < p.r_v; j += kComputeThreads) rec[2 + j] = ovec[j];
            __threadfence();
            named_bar_sync(kBarAll, kComputeThreads);
            const int c_first = owner_of(seg_start, U, Geff);
            const int c_last = owner_of(seg_end - 1, U, Geff);
            if (tid == 0) {
                const int prev = atomicAdd(&p.counters[b * p.H + h], 1);
                *last_flag = (prev == c_last - c_first);
            }
            named_bar_sync(kBarAll, kComputeThreads);
            if (*last_flag) {
                __threadfence();
                float M = -INFINITY;
                for (int cc = c_first; cc <= c_last; ++cc) {
                    const int sl = (seg_start <= range_start(cc, U, Geff)) ? 0 : 1;
                    M = fmaxf(M, __ldcg(p.partials + (static_cast<int64_t>(cc) * 2 + sl) * (p.r_v + 2)));
                }
                float lsum = 0.f;
                for (int cc = c_first; cc <= c_last; ++cc) {
                    const int sl = (seg_start <= range_start(cc, U, Geff)) ? 0 : 1;
                    const float *r = p.partials + (static_cast<int64_t>(cc) * 2 + sl) * (p.r_v + 2);
                    lsum += __ldcg(r + 1) * exp2f(__ldcg(r) - M);
                }
                named_bar_sync(kBarAll, kComputeThreads);  // ovec is rewritten below
                for (int j = tid; j < p.r_v; j += kComputeThreads) {
                    float s = 0.f;
                    for (int cc = c_first; cc <= c_last; ++cc) {
                        const int sl = (seg_start <= range_start(cc, U, Geff)) ? 0 : 1;
                        const float *r = p.partials + (static_cast<int64_t>(cc) * 2 + sl) * (p.r_v + 2);
                        s = fmaf(__ldcg(r + 2 + j), exp2f(__ldcg(r) - M), s);
                    }
                    ovec[j] = s;
                }
                named_bar_sync(kBarAll, kComputeThreads);
                finish_output<ES>(p, b, h, M, lsum, ovec, qfull, misc);
                if (tid == 0) atomicExch(&p.counters[b * p.H + h], 0);
            }
        }
        u = run_end;
    }

    // sequences with no cached token: pass 1 attends to the current token only
    for (int b = 0; b < p.B; ++b) {
        if (lens[b] != 0) continue;
        for (int h = 0; h < p.H; ++h) {
            if ((b * p.H + h) % gridDim.x != c) continue;
            const int64_t row = (static_cast<int64_t>(b) * p.H + h) * p.d;
            if (!pass1 && tid == 0) atomicOr(p.err, LLA_DEVERR_EMPTY_PASS2);
            for (int e = tid; e < p.d; e += kComputeThreads)
                store_elem(p.out, row + e, pass1 ? load_elem(p.cur_v, row + e, p.io_bf16) : 0.f,
                           p.io_bf16);
        }
    }
}

template <int ES, int GK, int VB>
lla_status launch_t(const Params &prm, int grid, int smem, cudaStream_t stream) {
    auto kern = decode_kernel<ES, GK, VB>;
    static bool configured[64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return LLA_ERR_CUDA;
    if (dev < 64 && !configured[dev]) {
        if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemLimit) !=
            cudaSuccess)
            return LLA_ERR_CUDA;
        configured[dev] = true;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kThreads);
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

}  // namespace

size_t decode_workspace_bytes(int r_v, int B, int H, int grid) {
    const size_t part = static_cast<size_t>(grid) * 2 * (r_v + 2) * sizeof(float);
    const size_t part_al = (part + 255) & ~static_cast<size_t>(255);
    return part_al + static_cast<size_t>(B) * H * sizeof(int);
}

lla_status decode_fits(int r_k, int r_v, int es, int d) {
    const int hpb = static_cast<int>(head_page_bytes(r_k, r_v, es));
    int pps = 1;
    if (4 * hpb <= kStepTargetBytes) pps = 4;
    else if (2 * hpb <= kStepTargetBytes) pps = 2;
    const Layout base = make_layout(0, pps * hpb, LLA_MAX_BATCH, r_k, r_v, d);
    if ((kSmemLimit - base.total) / (pps * hpb) < 2) return LLA_ERR_UNSUPPORTED;
    if (r_v * es / granule_bytes(r_v, es) > kComputeThreads) return LLA_ERR_UNSUPPORTED;
    return LLA_OK;
}

lla_status launch_decode(const DecodeArgs &a, cudaStream_t stream) {
    const int es = a.storage_bf16 ? 2 : 4;
    const int hpb = static_cast<int>(head_page_bytes(a.r_k, a.r_v, es));
    int pps = 1;
    if (4 * hpb <= kStepTargetBytes) pps = 4;
    else if (2 * hpb <= kStepTargetBytes) pps = 2;
    const int stage_bytes = pps * hpb;
    const Layout base = make_layout(0, stage_bytes, a.B, a.r_k, a.r_v, a.d);
    int stages = (kSmemLimit - base.total) / stage_bytes;
    if (stages > kMaxStages) stages = kMaxStages;
    if (stages < 2) return LLA_ERR_UNSUPPORTED;
    const int smem = make_layout(stages, stage_bytes, a.B, a.r_k, a.r_v, a.d).total;
    const int grid = num_sms();
    if (grid <= 0) return LLA_ERR_CUDA;
    if (a.workspace_bytes < decode_workspace_bytes(a.r_v, a.B, a.H, grid)) return LLA_ERR_WORKSPACE;
    lla_status st = LLA_OK;
    unsigned *err = device_error_word(&st);
    if (st != LLA_OK) return st;

    Params p = {};
    p.T = a.T; p.H = a.H; p.d = a.d; p.r_k = a.r_k; p.r_v = a.r_v; p.loop = a.loop;
    p.absorbed = a.absorbed; p.io_bf16 = a.io_bf16;
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
    p.pps = pps; p.stages = stages; p.stage_bytes = stage_bytes;
    p.err = err;

    const int gk = granule_bytes(a.r_k, es), vb = granule_bytes(a.r_v, es);
    if (es == 2) {
        if (gk == 16 && vb == 16) return launch_t<2, 16, 16>(p, grid, smem, stream);
        if (gk == 16 && vb == 4) return launch_t<2, 16, 4>(p, grid, smem, stream);
        if (gk == 4 && vb == 16) return launch_t<2, 4, 16>(p, grid, smem, stream);
        return launch_t<2, 4, 4>(p, grid, smem, stream);
    }
    if (gk == 16 && vb == 16) return launch_t<4, 16, 16>(p, grid, smem, stream);
    if (gk == 16 && vb == 4) return launch_t<4, 16, 4>(p, grid, smem, stream);
    if (gk == 4 && vb == 16) return launch_t<4, 4, 16>(p, grid, smem, stream);
    return launch_t<4, 4, 4>(p, grid, smem, stream);
}

}  // namespace lla
