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
//     max, exp2), and accumulate sum_i p_i c_v,i in latent space from the V-plane.  For the rank
//     shapes of the Ouro workloads a shape-specialised kernel splits them into score warps
//     (one token per thread, q~ held in registers, softmax) and value warps, which run one or
//     two steps apart through a two-slot ring of softmax weights in shared memory; any other
//     shape runs the generic kernel, where all eight warps take each phase in turn.
//   * A range that covers a (sequence, head) completely finishes it in place; ranges that split
//     one write (m, l, o_latent) partials, and the last CTA to arrive (atomic counter) merges
//     them by log-sum-exp, adds the current token and applies W_up,t^V, mu^V_t and 1/l.
#include "lla_decode_async.cuh"

namespace lla {
namespace {

// ------------------------------------------------------------------ generic kernel (any shape)

template <int ES, int GK, int VB>
__global__ void __launch_bounds__(kThreads, 1) decode_kernel(const Params p) {
    extern __shared__ __align__(128) char smem[];
    const Smem s = carve(smem, p);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int hpb = p.head_page_bytes;

    pdl_wait();  // inputs may come from the previous kernel in the stream
    Range rg = prologue(p, s, 1, 1);
    order_runs(p, s, rg);
    pdl_trigger();

    if (warp == kComputeWarps) {
        producer(p, s, rg);
        return;
    }

    constexpr int KE = GK / ES;  // elements per K granule
    constexpr int VE = VB / ES;  // elements per V unit
    const int TOK = p.pps * kBlockTokens;
    const int SPLIT = kComputeThreads / TOK;
    const int NGK = p.r_k * ES / GK;
    const int NVU = p.r_v * ES / VB;
    const int NTG = kComputeThreads / NVU;
    const int vu = tid % NVU, tg = tid / NVU;
    const bool vthread = tg < NTG;

    int stage = 0;
    uint32_t ph = 0;
    for (int pass = 0; pass < 3; ++pass)
    for (int64_t u = rg.lo[pass]; u < rg.hi[pass];) {
        const Run R = locate_run(p, s, u, rg.hi[pass]);
        setup_query<ES>(p, s, R.b, R.h);
        const float beta = s.misc[kMiscBeta];

        float m_run = -INFINITY, l_part = 0.f;
        float accv[VE];
#pragma unroll
        for (int k = 0; k < VE; ++k) accv[k] = 0.f;

        for (int k = 0; k < R.npages; k += p.pps) {
            mbar_wait(&s.full[stage], ph, s.abort_flag, p.err, wait_limit(p));
            const char *sb = s.ring + stage * p.stage_bytes;
            const int n = min(p.pps, R.npages - k);
            const int tok0 = (R.pg0 + k) * kBlockTokens;  // sequence position of row 0
            const int nvalid = min(n * kBlockTokens, R.Lb - tok0);

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
                        const float *qq = s.qlat + g * KE;
#pragma unroll
                        for (int e = 0; e < KE; ++e) acc = fmaf(v[e], qq[e], acc);
                    }
                }
                s.spart[sp * TOK + tk] = acc;
            }
            named_bar_sync(kBarAll, kComputeThreads);
            // online softmax over the step's tokens (threads that own a token)
            if (tid < TOK) {
                float sc = 0.f;
                for (int sp = 0; sp < SPLIT; ++sp) sc += s.spart[sp * TOK + tid];
                const bool valid = tid < nvalid;
                const float x = valid ? (sc + beta) * p.scale_log2 : -INFINITY;
                const float wm = warp_max(x);
                if (lane == 0) s.misc[kMiscWmax + warp] = wm;
                named_bar_sync(kBarTok, TOK);
                float ms = s.misc[kMiscWmax];
                for (int w = 1; w < (TOK >> 5); ++w) ms = fmaxf(ms, s.misc[kMiscWmax + w]);
                const float m_new = fmaxf(m_run, ms);
                const float alpha = exp2f(m_run - m_new);
                const float pv = valid ? exp2f(x - m_new) : 0.f;
                l_part = fmaf(l_part, alpha, pv);
                s.psm[tid] = pv;
                if (tid == 0) s.misc[kMiscAlpha] = alpha;
                m_run = m_new;
            }
            named_bar_sync(kBarAll, kComputeThreads);
            // latent value accumulation: sum_i p_i c_v,i
            if (vthread) {
                const float alpha = s.misc[kMiscAlpha];
#pragma unroll
                for (int e = 0; e < VE; ++e) accv[e] *= alpha;
                const char *vp = sb + p.kplane_bytes + vu * VB;
                for (int tk = tg; tk < nvalid; tk += NTG) {
                    const float pv = s.psm[tk];
                    float v[VE];
                    load_gran<ES, VB>(vp + (tk >> 6) * hpb + (tk & 63) * (p.r_v * ES), v);
#pragma unroll
                    for (int e = 0; e < VE; ++e) accv[e] = fmaf(pv, v[e], accv[e]);
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&s.empty[stage]);
            if (++stage == p.stages) {
                stage = 0;
                ph ^= 1u;
            }
        }

        // reduce the run's softmax state across threads
        if (tid < TOK) s.lred[tid] = l_part;
        if (vthread) {
#pragma unroll
            for (int e = 0; e < VE; ++e) s.red[tg * p.r_v + vu * VE + e] = accv[e];
        }
        if (tid == 0) s.misc[kMiscM] = m_run;
        named_bar_sync(kBarAll, kComputeThreads);
        for (int j = tid; j < p.r_v; j += kComputeThreads) {
            float acc = 0.f;
            for (int g = 0; g < NTG; ++g) acc += s.red[g * p.r_v + j];
            s.ovec[j] = acc;
        }
        if (warp == 0) {
            float acc = 0.f;
            for (int i = lane; i < TOK; i += 32) acc += s.lred[i];
            acc = warp_sum(acc);
            if (lane == 0) s.misc[kMiscL] = acc;
        }
        named_bar_sync(kBarAll, kComputeThreads);
        finish_run<GenericFinish<ES>>(p, s, R, u, rg);
        u = R.run_end;
    }
    empty_sequences(p, s);
}

template <int ES, int GK, int VB>
lla_status launch_generic(const Params &prm, int grid, int smem, cudaStream_t stream) {
    static DeviceOnce configured;
    return launch_kernel(decode_kernel<ES, GK, VB>, configured, prm, grid, smem, stream);
}

template <int ES, int RK, int RV>
lla_status launch_fast(const Params &prm, int grid, int smem, cudaStream_t stream) {
    static DeviceOnce configured;
    return launch_kernel(decode_async_kernel<ES, RK, RV, 128, 0>, configured, prm, grid, smem, stream,
                         kAsyncThreads);
}

template <int ES, int RK, int RV>
int fast_layout_bytes(int stages, int stage_bytes, int B) {
    return async_layout<ES, RK, RV, 128>(stages, stage_bytes, B).total;
}


// Shape-specialised kernel for (es, r_k, r_v): its launcher and shared-memory layout size
// (both null when the shape has none).
using FastLauncher = lla_status (*)(const Params &, int, int, cudaStream_t);
using FastLayout = int (*)(int, int, int);
struct FastEntry {
    FastLauncher launch;
    FastLayout layout;
};
FastEntry fast_entry(int es, int r_k, int r_v) {
#define LLA_FAST(E, K, V) \
    if (es == E && r_k == K && r_v == V) return FastEntry{launch_fast<E, K, V>, fast_layout_bytes<E, K, V>};
    LLA_FAST(2, 96, 160)
    LLA_FAST(2, 192, 320)
    LLA_FAST(2, 72, 120)
    LLA_FAST(2, 18, 30)
    LLA_FAST(2, 128, 128)
    LLA_FAST(4, 96, 160)
    LLA_FAST(4, 72, 120)
    LLA_FAST(4, 18, 30)
    LLA_FAST(4, 128, 128)
#undef LLA_FAST
    return FastEntry{nullptr, nullptr};
}

}  // namespace

size_t decode_counters_offset(int r_v, int grid) {
    const size_t part = static_cast<size_t>(grid) * 2 * (r_v + 2) * sizeof(float);
    return (part + 255) & ~static_cast<size_t>(255);
}

size_t decode_workspace_bytes(int r_v, int B, int H, int grid) {
    return decode_counters_offset(r_v, grid) + static_cast<size_t>(B) * H * sizeof(int);
}

lla_status decode_fits(int r_k, int r_v, int es, int d) {
    const int hpb = static_cast<int>(head_page_bytes(r_k, r_v, es));
    const int pps = pages_per_step(hpb);
    int fixed = make_layout(0, pps * hpb, LLA_MAX_BATCH, r_k, r_v, d).total;
    const FastEntry fe = d == 128 ? fast_entry(es, r_k, r_v) : FastEntry{nullptr, nullptr};
    if (fe.layout) fixed = fe.layout(0, pps * hpb, LLA_MAX_BATCH);
    if ((kSmemLimit - fixed) / (pps * hpb + 16) < 2) return LLA_ERR_UNSUPPORTED;
    if (r_v * es / granule_bytes(r_v, es) > kComputeThreads) return LLA_ERR_UNSUPPORTED;
    return LLA_OK;
}

lla_status launch_decode(const DecodeArgs &a, cudaStream_t stream) {
    const int es = a.storage_bf16 ? 2 : 4;
    const int hpb = static_cast<int>(head_page_bytes(a.r_k, a.r_v, es));
    const int pps = pages_per_step(hpb);
    const int stage_bytes = pps * hpb;
    const FastEntry fe = a.d == 128 ? fast_entry(es, a.r_k, a.r_v) : FastEntry{nullptr, nullptr};
    const int fixed = fe.launch ? fe.layout(0, stage_bytes, a.B)
                                : make_layout(0, stage_bytes, a.B, a.r_k, a.r_v, a.d).total;
    int stages = (kSmemLimit - fixed) / (stage_bytes + 16);  // + its full and empty barriers
    if (stages > kMaxStages) stages = kMaxStages;
    if (stages < 2) return LLA_ERR_UNSUPPORTED;
    const int smem = fe.launch ? fe.layout(stages, stage_bytes, a.B)
                               : make_layout(stages, stage_bytes, a.B, a.r_k, a.r_v, a.d).total;
    const int grid = num_sms();  // one CTA per SM
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
    p.partials = static_cast<float *>(a.workspace);
    p.counters = reinterpret_cast<int *>(static_cast<char *>(a.workspace) +
                                         decode_counters_offset(a.r_v, grid));
    p.pps = pps; p.stages = stages; p.stage_bytes = stage_bytes;
    p.err = err;
    p.wait_ns = pipeline_wait_limit_ns();

    if (fe.launch) return fe.launch(p, grid, smem, stream);

    const int gk = granule_bytes(a.r_k, es), vb = granule_bytes(a.r_v, es);
    if (es == 2) {
        if (gk == 16 && vb == 16) return launch_generic<2, 16, 16>(p, grid, smem, stream);
        if (gk == 16 && vb == 4) return launch_generic<2, 16, 4>(p, grid, smem, stream);
        if (gk == 4 && vb == 16) return launch_generic<2, 4, 16>(p, grid, smem, stream);
        return launch_generic<2, 4, 4>(p, grid, smem, stream);
    }
    if (gk == 16 && vb == 16) return launch_generic<4, 16, 16>(p, grid, smem, stream);
    if (gk == 16 && vb == 4) return launch_generic<4, 16, 4>(p, grid, smem, stream);
    if (gk == 4 && vb == 16) return launch_generic<4, 4, 16>(p, grid, smem, stream);
    return launch_generic<4, 4, 4>(p, grid, smem, stream);
}

}  // namespace lla
