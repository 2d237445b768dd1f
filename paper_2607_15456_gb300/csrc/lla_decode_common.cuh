// lla_decode_common.cuh -- pieces shared by the decode kernels over the paged latent cache
// (App. A "Decoding and caching"): launch parameters, the persistent stream-K split of
// (sequence, head, page) units over the CTAs, the producer warp's TMA ring, the management
// warps' query set-up, split-KV merge and output projection (App. J "Absorbed attention").
// Included by lla_decode.cu (absorbed attention and the dense comparator) and by
// lla_decode_rope.cu (rotary positions after reconstruction); everything here has internal
// linkage.
#pragma once

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
// Most data per pipeline step (whole head pages).  A file whose kernel takes one head page per
// step defines LLA_DECODE_STEP_BYTES as 32 KB before including this header.
#ifndef LLA_DECODE_STEP_BYTES
#define LLA_DECODE_STEP_BYTES (48 * 1024)
#endif
constexpr int kStepTargetBytes = LLA_DECODE_STEP_BYTES;
constexpr int kBarAll = 1;  // named barrier over the 256 consumer threads
constexpr int kBarTok = 2;  // named barrier over the score threads

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
    uint64_t wait_ns;  // limit of each pipeline wait; 0 = kWaitLimitNs
};

__device__ __forceinline__ uint64_t wait_limit(const Params &p) {
    return p.wait_ns ? p.wait_ns : kWaitLimitNs;
}

struct Layout {
    int ring, full, empty, pfull, pempty, prefix, lens, qlat, qfull, spart, psm, tmp, red, lred,
        ovec, misc, total;
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
    L.pfull = o;
    o += 2 * 8;
    L.pempty = o;
    o += 2 * 8;
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
    o += 2 * kComputeThreads * 4;
    L.tmp = o;
    o += 2 * kComputeThreads * 4;
    L.red = o;
    o += 8 * kComputeThreads * 4;
    L.lred = o;
    o += kComputeThreads * 4;
    L.ovec = o;
    o += up16((r_v > d ? r_v : d) * 4);
    L.misc = o;
    o += 64 * 4;
    L.total = o;
    return L;
}

// misc slots
constexpr int kMiscAlpha = 0, kMiscM = 1, kMiscL = 2, kMiscBeta = 3, kMiscScur = 4,
              kMiscWmax = 16 /* [2][8] */, kMiscAbort = 32, kMiscLast = 33;

struct Smem {
    char *ring;
    uint64_t *full, *empty, *pfull, *pempty;
    int64_t *prefix;
    int *lens;
    float *qlat, *qfull, *spart, *psm, *tmp, *red, *lred, *ovec, *misc;
    volatile int *abort_flag;
    int *last_flag;
};

__device__ __forceinline__ Smem carve(char *smem, const Params &p) {
    const Layout L = make_layout(p.stages, p.stage_bytes, p.B, p.r_k, p.r_v, p.d);
    Smem s;
    s.ring = smem + L.ring;
    s.full = reinterpret_cast<uint64_t *>(smem + L.full);
    s.empty = reinterpret_cast<uint64_t *>(smem + L.empty);
    s.pfull = reinterpret_cast<uint64_t *>(smem + L.pfull);
    s.pempty = reinterpret_cast<uint64_t *>(smem + L.pempty);
    s.prefix = reinterpret_cast<int64_t *>(smem + L.prefix);
    s.lens = reinterpret_cast<int *>(smem + L.lens);
    s.qlat = reinterpret_cast<float *>(smem + L.qlat);
    s.qfull = reinterpret_cast<float *>(smem + L.qfull);
    s.spart = reinterpret_cast<float *>(smem + L.spart);
    s.psm = reinterpret_cast<float *>(smem + L.psm);
    s.tmp = reinterpret_cast<float *>(smem + L.tmp);
    s.red = reinterpret_cast<float *>(smem + L.red);
    s.lred = reinterpret_cast<float *>(smem + L.lred);
    s.ovec = reinterpret_cast<float *>(smem + L.ovec);
    s.misc = reinterpret_cast<float *>(smem + L.misc);
    s.abort_flag = reinterpret_cast<volatile int *>(s.misc + kMiscAbort);
    s.last_flag = reinterpret_cast<int *>(s.misc + kMiscLast);
    return s;
}

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

struct Range {
    int64_t U, A0, A1;
    int Geff;
    // the order in which the CTA walks its runs: [lo[0], hi[0]), [lo[1], hi[1]), [lo[2], hi[2])
    int64_t lo[3], hi[3];
};

// Barrier set-up and the per-sequence unit prefix (H heads x pages), with device-side length
// checks.  All threads of the CTA; ends with __syncthreads.
__device__ Range prologue(const Params &p, const Smem &s, uint32_t pfull_count,
                          uint32_t pempty_count, uint32_t empty_count = kComputeWarps) {
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    if (tid == 0) {
        for (int i = 0; i < p.stages; ++i) {
            mbar_init(&s.full[i], 1);
            mbar_init(&s.empty[i], empty_count);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&s.pfull[i], pfull_count);
            mbar_init(&s.pempty[i], pempty_count);
        }
        *s.abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 0) {
        const int cap = min(p.max_ctx, p.max_blocks * kBlockTokens);
        int64_t run = 0;
        for (int b0 = 0; b0 < p.B; b0 += 32) {
            const int b = b0 + lane;
            int np = 0;
            if (b < p.B) {
                int Lb = p.context_lens[b];
                if (Lb < 0 || Lb > cap) {
                    if (blockIdx.x == 0) atomicOr(p.err, LLA_DEVERR_CONTEXT);
                    Lb = max(0, min(Lb, cap));
                }
                s.lens[b] = Lb;
                np = (Lb + kBlockTokens - 1) / kBlockTokens;
            }
            int v = np;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int n = __shfl_up_sync(0xffffffffu, v, o);
                if (lane >= o) v += n;
            }
            if (b < p.B) s.prefix[b] = run + static_cast<int64_t>(v - np) * p.H;
            run += static_cast<int64_t>(__shfl_sync(0xffffffffu, v, 31)) * p.H;
        }
        if (lane == 0) s.prefix[p.B] = run;
    }
    __syncthreads();
    Range r;
    r.U = s.prefix[p.B];
    r.Geff = static_cast<int>(r.U < gridDim.x ? r.U : gridDim.x);
    r.A0 = r.A1 = 0;
    if (static_cast<int>(blockIdx.x) < r.Geff) {
        r.A0 = range_start(blockIdx.x, r.U, r.Geff);
        r.A1 = range_start(blockIdx.x + 1, r.U, r.Geff);
    }
    r.lo[0] = r.A0;
    r.hi[0] = r.A1;
    r.lo[1] = r.hi[1] = r.lo[2] = r.hi[2] = 0;
    return r;
}

// One run: the part of a (sequence, head) inside this CTA's range.
struct Run {
    int b, h, Lb, pg0, npages;
    int64_t seg_start, seg_end, run_end;
};

__device__ __forceinline__ Run locate_run(const Params &p, const Smem &s, int64_t u, int64_t A1) {
    Run R;
    R.b = seq_of_unit(s.prefix, p.B, u);
    R.Lb = s.lens[R.b];
    // 32-bit arithmetic only: a 64-bit division is a called subroutine, cold in the instruction
    // cache at run boundaries while the streaming loops run
    const int np = (R.Lb + kBlockTokens - 1) / kBlockTokens;  // pages of the sequence
    const int off = static_cast<int>(u - s.prefix[R.b]);      // < H * np
    R.h = off / np;
    R.pg0 = off - R.h * np;
    R.seg_start = s.prefix[R.b] + static_cast<int64_t>(R.h) * np;
    R.seg_end = R.seg_start + np;
    R.run_end = R.seg_end < A1 ? R.seg_end : A1;
    R.npages = static_cast<int>(R.run_end - u);
    return R;
}

// Split runs first: a CTA streams its first run, then its last run when that is the start of a
// (sequence, head) the next CTA finishes, then the runs between them.  Both split runs are
// then merged while the CTA still streams, and it ends on a whole (sequence, head) that it
// finishes in place, so the launch does not end on a merge; a short first run is followed by
// a run whose query set-up is already done.
__device__ __forceinline__ void order_runs(const Params &p, const Smem &s, Range &r) {
    if (r.A1 <= r.A0) return;
    const Run T = locate_run(p, s, r.A1 - 1, r.A1);
    const int64_t ts = T.seg_start > r.A0 ? T.seg_start : r.A0;  // start of the last run
    if (ts == r.A0 || r.A1 == T.seg_end) return;                  // one run, or the last is whole
    const Run Hd = locate_run(p, s, r.A0, r.A1);
    const int64_t he = Hd.run_end;                                // end of the first run
    if (he >= ts) return;                                         // two runs: already in order
    r.lo[0] = r.A0;
    r.hi[0] = he;
    r.lo[1] = ts;
    r.hi[1] = r.A1;
    r.lo[2] = he;
    r.hi[2] = ts;
}

// Producer: the whole warp walks the CTA's range.  Block ids are fetched 32 pages at a time
// (one per lane) so the copies of consecutive steps are issued back to back instead of each
// waiting for its own block-table load.  Lane 0 issues a one-page step's bulk copy; when a step
// holds several small pages, lanes 0 .. n-1 issue one copy each in the same instruction (issued
// one after another from one lane, the copies of 6 KB pages paced the whole kernel).
//
// After a failed wait (or once another thread raised the abort flag) no further copy is issued:
// a new round on a stage whose previous copies have not landed would arrive twice on one phase
// of its full barrier.  Every round issued before that found its stage released by all consumer
// warps with the flag still down, so its previous round had landed; the last `stages` issued
// rounds are then awaited with the full limit, so no copy outlives the CTA.
// With a rotary pool (the decoupled rotary branch, one page per step) the block's rotary plane of
// `rope_bytes` lands right after the head page, on the same barrier.
__device__ void producer(const Params &p, const Smem &s, const Range &rg, const char *rope_pool = nullptr,
                         int rope_bytes = 0) {
    const int lane = threadIdx.x & 31;
    const int hpb = p.head_page_bytes;
    const uint64_t pol = policy_evict_first();
    int it = 0, st = 0;  // it: rounds issued
    uint32_t sph = 0;
    bool stop = false;
    for (int pass = 0; pass < 3 && !stop; ++pass)
    for (int64_t u = rg.lo[pass]; u < rg.hi[pass] && !stop;) {
        const Run R = locate_run(p, s, u, rg.hi[pass]);
        const int32_t *bt = p.block_table + static_cast<int64_t>(R.b) * p.max_blocks + R.pg0;
        for (int k0 = 0; k0 < R.npages && !stop; k0 += 32) {
            const int32_t blk_lane = (k0 + lane < R.npages) ? bt[k0 + lane] : -1;
            const int kend = min(R.npages, k0 + 32);
            for (int k = k0; k < kend; k += p.pps) {
                const int stage = st;
                const uint32_t ph = sph;
                int halt = 0;
                if (p.pps == 1) {
                    const int32_t b0 = __shfl_sync(0xffffffffu, blk_lane, (k - k0) & 31);
                    if (lane == 0) {
                        halt = !mbar_wait(&s.empty[stage], ph ^ 1u, s.abort_flag, p.err, wait_limit(p)) ||
                               *s.abort_flag;
                        if (!halt) {
                            const bool ok = b0 >= 0 && b0 < p.num_blocks;
                            if (!ok) atomicOr(p.err, LLA_DEVERR_BLOCK_ID);
                            mbar_arrive_expect_tx(&s.full[stage], ok ? hpb + rope_bytes : 0);
                            if (ok) {
                                char *dst = s.ring + stage * p.stage_bytes;
                                bulk_g2s(dst, p.pool + b0 * p.block_bytes + static_cast<int64_t>(R.h) * hpb, hpb,
                                         &s.full[stage], pol);
                                if (rope_pool)  // shared by the block's heads: read again from L2
                                    bulk_g2s(dst + hpb, rope_pool + static_cast<int64_t>(b0) * rope_bytes,
                                             rope_bytes, &s.full[stage], pol);
                            }
                        }
                    }
                    if (__shfl_sync(0xffffffffu, halt, 0)) {
                        stop = true;
                        break;
                    }
                } else {
                    // several pages per step: lanes 0 .. n-1 issue one bulk copy each, together
                    if (lane == 0)
                        halt = !mbar_wait(&s.empty[stage], ph ^ 1u, s.abort_flag, p.err, wait_limit(p)) ||
                               *s.abort_flag;
                    if (__shfl_sync(0xffffffffu, halt, 0)) {
                        stop = true;
                        break;
                    }
                    const int n = min(p.pps, R.npages - k);
                    const int32_t mine = __shfl_sync(0xffffffffu, blk_lane, (k - k0 + lane) & 31);
                    const bool valid = lane < n && mine >= 0 && mine < p.num_blocks;
                    if (lane < n && !valid) atomicOr(p.err, LLA_DEVERR_BLOCK_ID);
                    const unsigned vm = __ballot_sync(0xffffffffu, valid);
                    if (lane == 0) mbar_arrive_expect_tx(&s.full[stage], __popc(vm) * hpb);
                    __syncwarp();
                    if (valid)
                        bulk_g2s(s.ring + stage * p.stage_bytes + lane * hpb,
                                 p.pool + mine * p.block_bytes + static_cast<int64_t>(R.h) * hpb, hpb,
                                 &s.full[stage], pol);
                }
                ++it;
                if (++st == p.stages) {
                    st = 0;
                    sph ^= 1u;
                }
            }
        }
        u = R.run_end;
    }
    if (lane == 0 && *s.abort_flag) {
        // let the copies still in flight land before the CTA exits (full limit, whatever the
        // pipeline's limit was)
        volatile int never = 0;
        const int first = it > p.stages ? it - p.stages : 0;
        for (int j = first; j < it; ++j)
            mbar_wait(&s.full[j % p.stages], (j / p.stages) & 1, &never, p.err);
    }
}

// Query set-up of one (sequence, head): q in d-space, q~ = W_up,t^K^T q (or q itself for the
// dense comparator) and beta = q . mu^K_t.  All consumer threads.
template <int ES>
__device__ void setup_query(const Params &p, const Smem &s, int b, int h) {
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int64_t qoff = (static_cast<int64_t>(b) * p.H + h) * p.d;
    for (int e = tid; e < p.d; e += kComputeThreads) s.qfull[e] = load_elem(p.q, qoff + e, p.io_bf16);
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
                const float qe = s.qfull[e];
                a0 = fmaf(w.x, qe, a0);
                a1 = fmaf(w.y, qe, a1);
            }
            s.tmp[eg * p.r_k + 2 * jp] = a0;
            s.tmp[eg * p.r_k + 2 * jp + 1] = a1;
        }
        if (warp == kComputeWarps - 1) {
            float bsum = 0.f;
            if (p.mu_k) {
                const float *mu = p.mu_k + (static_cast<int64_t>(h) * p.T + p.loop) * p.d;
                for (int e = lane; e < p.d; e += 32) bsum = fmaf(s.qfull[e], mu[e], bsum);
            }
            bsum = warp_sum(bsum);
            if (lane == 0) s.misc[kMiscBeta] = bsum;
        }
        named_bar_sync(kBarAll, kComputeThreads);
        for (int j = tid; j < p.r_k; j += kComputeThreads) {
            float acc = 0.f;
            for (int g = 0; g < neg; ++g) acc += s.tmp[g * p.r_k + j];
            s.qlat[j] = acc;
        }
    } else {
        for (int e = tid; e < p.d; e += kComputeThreads) s.qlat[e] = s.qfull[e];
        if (tid == 0) s.misc[kMiscBeta] = 0.f;
    }
    named_bar_sync(kBarAll, kComputeThreads);
}

// Final output of one (sequence, head) from its cached softmax state: maximum m (log2 units),
// mass l and latent value sum ovec (all relative to m).  All consumer threads.
template <int ES>
__device__ void finish_output(const Params &p, const Smem &s, int b, int h, float m, float l) {
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const bool pass1 = p.cur_k != nullptr;
    const int64_t row = (static_cast<int64_t>(b) * p.H + h) * p.d;
    if (pass1 && warp == 0) {
        float acc = 0.f;
        for (int e = lane; e < p.d; e += 32)
            acc = fmaf(s.qfull[e], load_elem(p.cur_k, row + e, p.io_bf16), acc);
        acc = warp_sum(acc);
        if (lane == 0) s.misc[kMiscScur] = acc * p.scale_log2;
    }
    named_bar_sync(kBarAll, kComputeThreads);
    float M = m, pc = 0.f;
    if (pass1) {
        const float sc = s.misc[kMiscScur];
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
                acc = fmaf(w.x, s.ovec[2 * jp], acc);
                acc = fmaf(w.y, s.ovec[2 * jp + 1], acc);
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
            float o = s.ovec[e] * wl;
            if (pass1) o = fmaf(pc, load_elem(p.cur_v, row + e, p.io_bf16), o);
            store_elem(p.out, row + e, o * inv, p.io_bf16);
        }
    }
    named_bar_sync(kBarAll, kComputeThreads);
}

// After a run, with misc[kMiscM], misc[kMiscL] and ovec holding its softmax state: finish the
// (sequence, head) in place when the run covers it, else leave a partial and, if this CTA is
// the last to arrive, merge all partials by log-sum-exp and finish.  All consumer threads.
template <class Finish>
__device__ void finish_run(const Params &p, const Smem &s, const Run &R, int64_t u,
                           const Range &rg) {
    const int tid = threadIdx.x;
    if (u == R.seg_start && R.run_end == R.seg_end) {
        Finish::run(p, s, R.b, R.h, s.misc[kMiscM], s.misc[kMiscL]);
        return;
    }
    // partial of a (sequence, head) split across CTAs: slot 0 if this is the CTA's first run,
    // slot 1 if its last
    const int c = blockIdx.x;
    const int slot = (R.seg_start <= rg.A0) ? 0 : 1;
    float *rec = p.partials + (static_cast<int64_t>(c) * 2 + slot) * (p.r_v + 2);
    if (tid == 0) {
        rec[0] = s.misc[kMiscM];
        rec[1] = s.misc[kMiscL];
    }
    for (int j = tid; j < p.r_v; j += kComputeThreads) rec[2 + j] = s.ovec[j];
    __threadfence();
    named_bar_sync(kBarAll, kComputeThreads);
    const int c_first = owner_of(R.seg_start, rg.U, rg.Geff);
    const int c_last = owner_of(R.seg_end - 1, rg.U, rg.Geff);
    int *counter = &p.counters[R.b * p.H + R.h];
    if (tid == 0) {
        const int prev = atomicAdd(counter, 1);
        *s.last_flag = (prev == c_last - c_first);
    }
    named_bar_sync(kBarAll, kComputeThreads);
    if (!*s.last_flag) return;
    __threadfence();
    auto record = [&](int cc) {
        const int sl = (R.seg_start <= range_start(cc, rg.U, rg.Geff)) ? 0 : 1;
        return p.partials + (static_cast<int64_t>(cc) * 2 + sl) * (p.r_v + 2);
    };
    // every part's (m, l) into shared memory (tmp: 2 x 256 floats), then the maximum
    const int nparts = c_last - c_first + 1;
    float M = -INFINITY, lsum = 0.f;
    for (int c0 = 0; c0 < nparts; c0 += kComputeThreads) {
        const int np = min(kComputeThreads, nparts - c0);
        if (tid < np) {
            const float *r = record(c_first + c0 + tid);
            s.tmp[tid] = __ldcg(r);
            s.tmp[kComputeThreads + tid] = __ldcg(r + 1);
        }
        named_bar_sync(kBarAll, kComputeThreads);
        float Mc = M;
        for (int i = 0; i < np; ++i) Mc = fmaxf(Mc, s.tmp[i]);
        lsum *= exp2f(M - Mc);
        for (int i = 0; i < np; ++i) lsum = fmaf(s.tmp[kComputeThreads + i], exp2f(s.tmp[i] - Mc), lsum);
        M = Mc;
        named_bar_sync(kBarAll, kComputeThreads);
    }
    for (int j = tid; j < p.r_v; j += kComputeThreads) {
        float acc = 0.f;
#pragma unroll 4
        for (int cc = c_first; cc <= c_last; ++cc) {
            const float *r = record(cc);
            acc = fmaf(__ldcg(r + 2 + j), exp2f(__ldcg(r) - M), acc);
        }
        s.ovec[j] = acc;
    }
    named_bar_sync(kBarAll, kComputeThreads);
    Finish::run(p, s, R.b, R.h, M, lsum);
    if (tid == 0) atomicExch(counter, 0);
}

// Finisher of the generic kernel.
template <int ES>
struct GenericFinish {
    __device__ static void run(const Params &p, const Smem &s, int b, int h, float m, float l) {
        finish_output<ES>(p, s, b, h, m, l);
    }
};

// Sequences with no cached token: pass 1 attends to the current token only.  Consumers.
__device__ void empty_sequences(const Params &p, const Smem &s) {
    const int tid = threadIdx.x;
    const bool pass1 = p.cur_k != nullptr;
    for (int b = 0; b < p.B; ++b) {
        if (s.lens[b] != 0) continue;
        for (int h = 0; h < p.H; ++h) {
            if ((b * p.H + h) % gridDim.x != blockIdx.x) continue;
            const int64_t row = (static_cast<int64_t>(b) * p.H + h) * p.d;
            if (!pass1 && tid == 0) atomicOr(p.err, LLA_DEVERR_EMPTY_PASS2);
            for (int e = tid; e < p.d; e += kComputeThreads)
                store_elem(p.out, row + e, pass1 ? load_elem(p.cur_v, row + e, p.io_bf16) : 0.f,
                           p.io_bf16);
        }
    }
}

// --------------------------------------------- shape-specialised kernel (Ouro rank shapes)

template <int ES, int RK, int RV>
struct Fast {
    static constexpr int HPB = kBlockTokens * (RK + RV) * ES;  // head page bytes
    static constexpr int PPS = (4 * HPB <= kStepTargetBytes) ? 4 : (2 * HPB <= kStepTargetBytes) ? 2 : 1;
    static constexpr int TOK = PPS * kBlockTokens;             // tokens per pipeline step
    static constexpr int GK = ((RK * ES) % 16 == 0) ? 16 : 4;  // K granule bytes
    static constexpr int KE = GK / ES;                         // elements per K granule
    static constexpr int NGK = RK * ES / GK;                   // K granules per token
    // Score threads: TT threads per k-split, each owning TPT tokens; KSPLIT groups share a
    // token's granules so that the score role has up to four warps.
    static constexpr int TPT = TOK > 128 ? TOK / 128 : 1;
    static constexpr int TT = TOK / TPT;
    static constexpr int KSPLIT = (TT <= 64 && NGK > 6) ? 2 : 1;
    static constexpr int NGT = (NGK + KSPLIT - 1) / KSPLIT;    // granules per k-split
    static constexpr int S_THREADS = TT * KSPLIT;
    static constexpr int S_WARPS = S_THREADS / 32;
    static constexpr int V_WARPS = kComputeWarps - S_WARPS;
    static constexpr int V_THREADS = V_WARPS * 32;
    static constexpr int VB = ((RV * ES) % 16 == 0) ? 16 : 4;  // V unit bytes
    static constexpr int VE = VB / ES;                         // elements per V unit
    static constexpr int VU = RV * ES / VB;                    // V units per row
    static constexpr int UPT = (VU % 2 == 0 && VU / 2 >= 8) ? 2 : 1;  // units per value thread
    static constexpr int VC = VU / UPT;                        // value threads per token row
    static constexpr int NTG = V_THREADS / VC;                 // token groups of value threads
    static constexpr int ROWB = RV * ES;                       // V-plane row bytes
    static constexpr int KPLANE = kBlockTokens * RK * ES;      // K-plane bytes
    static_assert(S_THREADS % 32 == 0 && S_WARPS >= 1 && V_WARPS >= 1, "role split");
    static_assert(NTG >= 1 && TT * TPT == TOK, "every token has a score thread");
    static_assert(KE % 4 == 0 || KE <= 2, "q~ vector loads");
    static_assert(TT % 32 == 0, "score-owning threads are whole warps");
};

// KE consecutive floats of q~ from shared memory (16-byte aligned at every granule start).
template <int KE>
__device__ __forceinline__ void load_qvec(const float *q, float (&v)[KE]) {
    if constexpr (KE % 4 == 0) {
#pragma unroll
        for (int i = 0; i < KE; i += 4) {
            const float4 t = *reinterpret_cast<const float4 *>(q + i);
            v[i] = t.x; v[i + 1] = t.y; v[i + 2] = t.z; v[i + 3] = t.w;
        }
    } else if constexpr (KE == 2) {
        const float2 t = *reinterpret_cast<const float2 *>(q);
        v[0] = t.x; v[1] = t.y;
    } else {
#pragma unroll
        for (int i = 0; i < KE; ++i) v[i] = q[i];
    }
}

// Value warps, one pipeline step: rescale this thread's latent value sums by the step's alpha,
// then add p_i c_v,i for the step's valid tokens from the V-planes of the stage at `sb`.  The
// thread owns the units vc, vc + VC, ... (UPT units of VE columns, spread over the row so that
// the eight threads of a shared-memory phase read neighbouring units) and the token rows
// tg, tg + NTG, ... of each page.
template <int ES, int RK, int RV>
__device__ __forceinline__ void value_step(float (&accv)[Fast<ES, RK, RV>::UPT * Fast<ES, RK, RV>::VE],
                                           const char *sb, const float *pring, float alpha,
                                           int nvalid, int vc, int tg) {
    using F = Fast<ES, RK, RV>;
    constexpr int AV = F::UPT * F::VE;
#pragma unroll
    for (int e = 0; e < AV; ++e) accv[e] *= alpha;
    const char *vbase = sb + F::KPLANE + vc * F::VB + tg * F::ROWB;
    if constexpr (kBlockTokens % F::NTG == 0 && F::VE % 2 == 0) {
        // A full step (the common case): every thread owns RPT rows of each page, known at
        // compile time, so the loads of G rows go out together and two accumulator sets halve
        // the dependent chains (the loop below ran latency-bound on 4-byte units).
        if (nvalid == F::TOK) {
            constexpr int RPT = kBlockTokens / F::NTG;
            constexpr int G = RPT >= 4 ? 4 : RPT;  // rows whose loads go out together
            float acc2[AV];
#pragma unroll
            for (int e = 0; e < AV; ++e) acc2[e] = 0.f;
#pragma unroll
            for (int pi = 0; pi < F::PPS; ++pi) {
                const char *vp = vbase + pi * F::HPB;
                const float *pp = pring + pi * kBlockTokens + tg;
#pragma unroll
                for (int i0 = 0; i0 < RPT; i0 += G) {
                    float pv[G];
                    float v[G][F::UPT][F::VE];
#pragma unroll
                    for (int i = 0; i < G; ++i) {
                        pv[i] = pp[(i0 + i) * F::NTG];
#pragma unroll
                        for (int uu = 0; uu < F::UPT; ++uu)
                            load_gran<ES, F::VB>(vp + (i0 + i) * (F::NTG * F::ROWB) + uu * (F::VC * F::VB), v[i][uu]);
                    }
#pragma unroll
                    for (int i = 0; i < G; ++i) {
                        float *acc = (i & 1) ? acc2 : accv;
                        const float2 p2 = make_float2(pv[i], pv[i]);
#pragma unroll
                        for (int uu = 0; uu < F::UPT; ++uu)
#pragma unroll
                            for (int e = 0; e < F::VE; e += 2) {
                                const float2 r = __ffma2_rn(p2, make_float2(v[i][uu][e], v[i][uu][e + 1]),
                                                            make_float2(acc[uu * F::VE + e], acc[uu * F::VE + e + 1]));
                                acc[uu * F::VE + e] = r.x;
                                acc[uu * F::VE + e + 1] = r.y;
                            }
                    }
                }
            }
#pragma unroll
            for (int e = 0; e < AV; ++e) accv[e] += acc2[e];
            return;
        }
    }
#pragma unroll
    for (int pi = 0; pi < F::PPS; ++pi) {
        // rows tg, tg + NTG, ... of page pi that hold valid tokens
        const int rows = min(kBlockTokens, nvalid - pi * kBlockTokens);
        const int cnt = rows > tg ? (rows - tg + F::NTG - 1) / F::NTG : 0;
        const char *vp = vbase + pi * F::HPB;
        const float *pp = pring + pi * kBlockTokens + tg;
#pragma unroll 4
        for (int i = 0; i < cnt; ++i) {
            const float pv = pp[i * F::NTG];
            const char *rowp = vp + i * (F::NTG * F::ROWB);
#pragma unroll
            for (int uu = 0; uu < F::UPT; ++uu) {
                float v[F::VE];
                load_gran<ES, F::VB>(rowp + uu * (F::VC * F::VB), v);
                if constexpr (F::VE % 2 == 0) {
                    const float2 p2 = make_float2(pv, pv);
#pragma unroll
                    for (int e = 0; e < F::VE; e += 2) {
                        const float2 r = __ffma2_rn(p2, make_float2(v[e], v[e + 1]),
                                                    make_float2(accv[uu * F::VE + e],
                                                                accv[uu * F::VE + e + 1]));
                        accv[uu * F::VE + e] = r.x;
                        accv[uu * F::VE + e + 1] = r.y;
                    }
                } else {
#pragma unroll
                    for (int e = 0; e < F::VE; ++e)
                        accv[uu * F::VE + e] = fmaf(pv, v[e], accv[uu * F::VE + e]);
                }
            }
        }
    }
}

// Value warps at a run's end: this thread's latent value sums into its token group's row of the
// run's state (red [NTG][RV]), at the columns of the units it owns.
template <int ES, int RK, int RV>
__device__ __forceinline__ void value_store(float *red, const float (&accv)[Fast<ES, RK, RV>::UPT * Fast<ES, RK, RV>::VE],
                                            int vc, int tg) {
    using F = Fast<ES, RK, RV>;
#pragma unroll
    for (int uu = 0; uu < F::UPT; ++uu)
#pragma unroll
        for (int e = 0; e < F::VE; ++e)
            red[tg * RV + (vc + uu * F::VC) * F::VE + e] = accv[uu * F::VE + e];
}

// ------------------------------------------------------------------------------------------
// Shape-specialised kernel with asynchronous run boundaries.
//
// Warp roles (one CTA per SM):
//   warps 0..S_WARPS-1     score warps: q~ . c_k for the step's tokens, online softmax
//   warps S_WARPS..7       value warps: sum_i p_i c_v,i
//   warp 8                 producer: TMA bulk copies of head pages into the ring
//   warps 9..12            management warps: for run r+1 they load q and W_up,t^K and form
//                          q~ while the other warps stream run r; for run r-1 they reduce the
//                          left-behind softmax state, write or merge the split partials and
//                          apply W_up,t^V.  Their global round trips never stall the stream.
// Hand-offs: qready[r % 3] (management -> score warps: q~ of run r is ready), stfull[r % 2]
// (score + value warps -> management: the run's softmax state is written) and stfree[r % 2]
// (management -> score and value warps: that state has been read).  The management warps set
// up run r, then finish run r - 2; three query slots keep a set-up from overwriting what a
// pending finish still reads, and the stfree wait keeps run r from overwriting the state of run
// r - 2 before its finish has read it.  W_up,t rows reach the management warps through a shared
// staging buffer filled with cp.async, so no register holds them while they are in flight.
// ------------------------------------------------------------------------------------------

constexpr int kMWarps = 4;
constexpr int kQSlots = 3;  // query slots: set-ups run two runs ahead of finishes
constexpr int kLredSlot = 128;  // row sums of one run (one per score thread of a k-split)
constexpr int kMThreads = kMWarps * 32;
constexpr int kMBase = kComputeThreads + 32;       // first management thread
constexpr int kAsyncThreads = kMBase + kMThreads;  // 416
constexpr int kBarM = 3;                           // named barrier of the management warps
constexpr int kBarStart = 4;                       // producer waits for the first set-up's loads
constexpr int kWstMax = 40 * 1024;                 // staging buffer for W_up,t rows (upper bound)

struct AsyncLayout {
    int ring, full, empty, pfull, pempty, qready, stfull, stfree, prefix, lens, qlat, qfull, spart,
        psm, lred, red, ovec, mred, mtmp, xtra, misc, wst, total;
};

// Shared-memory sizes of the asynchronous kernel for one rank shape (floats per slot); WL
// bounds the staging buffer of W_up,t rows.
template <int ES, int RK, int RV, int D, int WL = kWstMax>
struct AsyncSizes {
    using F = Fast<ES, RK, RV>;
    static constexpr int QSLOT = ((RK > D ? RK : D) + 3) & ~3;  // q~ or q, one run
    static constexpr int REDSLOT = F::NTG * RV;                 // value partials, one run
    static constexpr int MRED = (kMThreads / (RK / 2)) * RK;    // q~ partial sums
    // staging buffer: the larger of W_up,t^K and W_up,t^V, at most WL
    static constexpr int WMAT = D * (RK > RV ? RK : RV) * ES;
    static constexpr int WST = WMAT < WL ? WMAT : WL;
};

__host__ __device__ inline AsyncLayout make_async_layout(int stages, int stage_bytes, int B,
                                                         int qslot, int redslot, int mred, int rv,
                                                         int xslot, int wst) {
    AsyncLayout L;
    int o = 0;
    L.ring = o;   o += stages * stage_bytes;
    L.full = o;   o += stages * 8;
    L.empty = o;  o += stages * 8;
    L.pfull = o;  o += 16;
    L.pempty = o; o += 16;
    L.qready = o; o += 32;  // [kQSlots]
    L.stfull = o; o += 16;
    L.stfree = o; o += 16;
    L.prefix = o; o += up16((B + 1) * 8);
    L.lens = o;   o += up16(B * 4);
    L.qlat = o;   o += up16(kQSlots * qslot * 4);
    L.qfull = o;  o += up16(qslot * 4);  // q of the set-up in progress
    L.spart = o;  o += kComputeThreads * 4;
    L.psm = o;    o += 2 * kComputeThreads * 4;
    L.lred = o;   o += 2 * kLredSlot * 4;
    L.red = o;    o += up16(2 * redslot * 4);
    L.ovec = o;   o += up16(rv * 4);
    L.mred = o;   o += up16(mred * 4);
    L.mtmp = o;   o += 2 * kMThreads * 4;
    L.xtra = o;   o += up16(kQSlots * xslot * 4);
    L.misc = o;   o += 64 * 4;
    L.wst = o;    o += up16(wst);
    L.total = o;
    return L;
}

template <int ES, int RK, int RV, int D, int WL = kWstMax>
__host__ __device__ inline AsyncLayout async_layout(int stages, int stage_bytes, int B) {
    using Z = AsyncSizes<ES, RK, RV, D, WL>;
    return make_async_layout(stages, stage_bytes, B, Z::QSLOT, Z::REDSLOT, Z::MRED, RV, 2 * D, Z::WST);
}

// misc slots of the asynchronous kernel
constexpr int kAM = 0 /* [2] run maximum by state slot */, kAPAlpha = 5 /* [2] */,
              kAWmax = 16 /* [2][8] */, kAAbort = 32, kALast = 33,
              kAPart = 40 /* [3 query slots][4 warps][q.k_cur, q.mu^K] */;

struct ASmem {
    Smem s;  // fields shared with the generic helpers (ring, barriers, prefix, lens, abort flag)
    uint64_t *qready, *stfull, *stfree;
    float *qlat, *qfull, *lred, *red, *mred, *mtmp;
    float *xtra;  // [kQSlots][v_cur (D), mu^V_t (D)] by query slot
    char *wst;
    int qslot, redslot;  // floats per slot
};

template <int ES, int RK, int RV, int D, int WL = kWstMax>
__device__ __forceinline__ ASmem carve_async(char *smem, const Params &p) {
    const AsyncLayout L = async_layout<ES, RK, RV, D, WL>(p.stages, p.stage_bytes, p.B);
    ASmem a;
    a.s.ring = smem + L.ring;
    a.s.full = reinterpret_cast<uint64_t *>(smem + L.full);
    a.s.empty = reinterpret_cast<uint64_t *>(smem + L.empty);
    a.s.pfull = reinterpret_cast<uint64_t *>(smem + L.pfull);
    a.s.pempty = reinterpret_cast<uint64_t *>(smem + L.pempty);
    a.s.prefix = reinterpret_cast<int64_t *>(smem + L.prefix);
    a.s.lens = reinterpret_cast<int *>(smem + L.lens);
    a.s.qlat = nullptr;
    a.s.qfull = nullptr;
    a.s.spart = reinterpret_cast<float *>(smem + L.spart);
    a.s.psm = reinterpret_cast<float *>(smem + L.psm);
    a.s.tmp = nullptr;
    a.s.red = nullptr;
    a.s.lred = nullptr;
    a.s.ovec = reinterpret_cast<float *>(smem + L.ovec);
    a.s.misc = reinterpret_cast<float *>(smem + L.misc);
    a.s.abort_flag = reinterpret_cast<volatile int *>(a.s.misc + kAAbort);
    a.s.last_flag = reinterpret_cast<int *>(a.s.misc + kALast);
    a.qready = reinterpret_cast<uint64_t *>(smem + L.qready);
    a.stfull = reinterpret_cast<uint64_t *>(smem + L.stfull);
    a.stfree = reinterpret_cast<uint64_t *>(smem + L.stfree);
    a.qlat = reinterpret_cast<float *>(smem + L.qlat);
    a.qfull = reinterpret_cast<float *>(smem + L.qfull);
    a.lred = reinterpret_cast<float *>(smem + L.lred);
    a.red = reinterpret_cast<float *>(smem + L.red);
    a.mred = reinterpret_cast<float *>(smem + L.mred);
    a.mtmp = reinterpret_cast<float *>(smem + L.mtmp);
    a.xtra = reinterpret_cast<float *>(smem + L.xtra);
    a.wst = smem + L.wst;
    a.qslot = AsyncSizes<ES, RK, RV, D, WL>::QSLOT;
    a.redslot = AsyncSizes<ES, RK, RV, D, WL>::REDSLOT;
    return a;
}

__device__ __forceinline__ void m_sync() { named_bar_sync(kBarM, kMThreads); }

// Passes through the staging buffer for a D x R matrix of W_up,t: the smallest power of two
// that makes one pass fit.
template <int ES, int R, int D, int WST>
struct WPasses {
    static constexpr int BYTES = D * R * ES;
    static constexpr int N = BYTES <= WST ? 1 : BYTES <= 2 * WST ? 2 : BYTES <= 4 * WST ? 4 : 8;
    static constexpr int ROWS = D / N;                // rows per pass
    static constexpr int PASS_BYTES = ROWS * R * ES;  // multiple of 16 since D = 128
    static_assert(D % N == 0 && PASS_BYTES <= WST && PASS_BYTES % 16 == 0, "staging passes");
};

// Starts the copy of rows [pass*ROWS, (pass+1)*ROWS) of W into the staging buffer.
template <int ES, int R, int D, int WST>
__device__ __forceinline__ void m_stage_rows(const ASmem &a, const char *W, int pass, int mt) {
    using P = WPasses<ES, R, D, WST>;
    const char *src = W + static_cast<int64_t>(pass) * P::PASS_BYTES;
    for (int i = mt; i < P::PASS_BYTES / 16; i += kMThreads) cp_async16(a.wst + i * 16, src + i * 16);
    cp_async_commit();
}

// Chunk geometry of W_up,t^V in the staging buffer: rows cut into CB-byte chunks, stored chunk
// by chunk (chunk c of row e of a pass at (c * ROWS + e) * CB), so that threads owning
// consecutive rows read consecutive chunks.
template <int ES, int RV, int D, int WST>
struct VStage {
    using P = WPasses<ES, RV, D, WST>;
    static constexpr int CB = (RV * ES) % 16 == 0 ? 16 : 4;  // chunk bytes
    static constexpr int CPR = RV * ES / CB;                 // chunks per row
    static constexpr int EPC = CB / ES;                      // elements per chunk
    static constexpr int TPR = kMThreads / P::ROWS;          // threads per row
    static_assert(kMThreads % P::ROWS == 0 && (RV * ES) % 4 == 0, "row ownership");
};

// Starts the copy of pass `pass` of W_up,t^V into the staging buffer, chunk-major.
template <int ES, int RV, int D, int WST>
__device__ __forceinline__ void m_stage_v(const ASmem &a, const char *W, int pass, int mt) {
    using V = VStage<ES, RV, D, WST>;
    const char *src = W + static_cast<int64_t>(pass) * V::P::PASS_BYTES;
    for (int i = mt; i < V::P::ROWS * V::CPR; i += kMThreads) {
        const int e = i / V::CPR, c = i - e * V::CPR;
        char *dst = a.wst + (c * V::P::ROWS + e) * V::CB;
        if constexpr (V::CB == 16) cp_async16(dst, src + i * 16);
        else cp_async4(dst, src + i * 4);
    }
    cp_async_commit();
}

// Management: everything a run needs that does not depend on its results, into slot `slot`:
// q, q~ = W_up,t^K^T q, and the per-warp partial sums of beta = q . mu^K_t and of q . k_cur;
// v_cur and mu^V_t for its output.  All of its global loads go out together, so the set-up costs
// one round trip plus the W_up,t^K passes, and the run's finish needs none of them.  With
// ABSORB_K false (keys rebuilt from the latents elsewhere) the slot receives q itself and
// beta's partials are zero.
template <int ES, int RK, int RV, int D, bool ABSORB_K = true, int WL = kWstMax>
__device__ void m_setup(const Params &p, const ASmem &a, int b, int h, int slot, int mt,
                        bool release_producer) {
    static_assert(D <= kMThreads, "one management thread per element of q");
    constexpr int WST = AsyncSizes<ES, RK, RV, D, WL>::WST;
    const bool absorb_k = ABSORB_K && p.absorbed;
    float *qfull = a.qfull;
    float *qlat = a.qlat + slot * a.qslot;
    float *xtra = a.xtra + slot * 2 * D;
    const int mwarp = mt >> 5, lane = mt & 31;
    const int64_t qoff = (static_cast<int64_t>(b) * p.H + h) * D;
    const int64_t hl = (static_cast<int64_t>(h) * p.T + p.loop) * D;
    const bool pass1 = p.cur_k != nullptr;
    cp_async_wait_all();  // nothing of an earlier use of the staging buffer is still in flight
    m_sync();
    using P = WPasses<ES, RK, D, WST>;
    const char *W = static_cast<const char *>(p.w_up_k) + hl * RK * ES;
    if (absorb_k) m_stage_rows<ES, RK, D, WST>(a, W, 0, mt);
    // the first set-up's loads go out before the producer fills the ring, not queued behind it
    if (release_producer) named_bar_arrive(kBarStart, kMThreads + 32);
    float qv = 0.f, ck = 0.f, cv = 0.f, muk = 0.f, muv = 0.f;
    if (mt < D) {
        qv = load_elem(p.q, qoff + mt, p.io_bf16);
        if (pass1) {
            ck = load_elem(p.cur_k, qoff + mt, p.io_bf16);
            cv = load_elem(p.cur_v, qoff + mt, p.io_bf16);
        }
        if (absorb_k && p.mu_k) muk = p.mu_k[hl + mt];
        if (p.absorbed && p.mu_v) muv = p.mu_v[hl + mt];
        qfull[mt] = qv;
        xtra[mt] = cv;
        xtra[D + mt] = muv;
    }
    const float ps = warp_sum(qv * ck), pb = warp_sum(qv * muk);
    if (lane == 0) {
        a.s.misc[kAPart + slot * 8 + mwarp * 2] = ps;
        a.s.misc[kAPart + slot * 8 + mwarp * 2 + 1] = pb;
    }
    if (!absorb_k) {
        if (mt < D) qlat[mt] = qv;
        return;
    }
    constexpr int CPR = RK / 2;          // pairs per row of W
    constexpr int RG = kMThreads / CPR;  // row groups
    static_assert(RG >= 1 && RG * RK <= 2048, "partial sums fit the management buffer");
    const int cg = mt % CPR, rg = mt / CPR;
    float acc0 = 0.f, acc1 = 0.f;
#pragma unroll 1
    for (int pass = 0; pass < P::N; ++pass) {
        cp_async_wait_all();
        m_sync();  // the pass (and qfull) is in shared memory for every thread
        if (rg < RG) {
            for (int el = rg; el < P::ROWS; el += RG) {
                const float2 w = load_pair<ES>(a.wst, static_cast<int64_t>(el) * RK + cg * 2);
                const float qe = qfull[pass * P::ROWS + el];
                acc0 = fmaf(w.x, qe, acc0);
                acc1 = fmaf(w.y, qe, acc1);
            }
        }
        if (pass + 1 < P::N) {
            m_sync();  // the buffer is read before the next pass overwrites it
            m_stage_rows<ES, RK, D, WST>(a, W, pass + 1, mt);
        }
    }
    if (rg < RG) {
        a.mred[rg * RK + cg * 2] = acc0;
        a.mred[rg * RK + cg * 2 + 1] = acc1;
    }
    m_sync();
    for (int j = mt; j < RK; j += kMThreads) {
        float acc = 0.f;
#pragma unroll 4
        for (int g = 0; g < RG; ++g) acc += a.mred[g * RK + j];
        qlat[j] = acc;
    }
}

// Sum of the management warps' partials k (0: q . k_cur, 1: q . mu^K_t) of a slot.
__device__ __forceinline__ float m_part(const ASmem &a, int slot, int k) {
    const float *pp = a.s.misc + kAPart + slot * 8 + k;
    return (pp[0] + pp[2]) + (pp[4] + pp[6]);
}

// Management: output of one (sequence, head) from its softmax state (m, l, a.s.ovec).
// o = (W_up,t^V ovec wl + lc mu^V_t + p_cur v_cur) / (lc + p_cur).  The first pass of W_up,t^V
// is already in flight in the staging buffer.  Each row of the pass has TPR threads (one when
// the pass holds all D rows); their chunk reads are conflict-free, ovec reads are broadcasts
// and the output stores coalesce.
template <int ES, int RK, int RV, int D, int WL = kWstMax>
__device__ void m_output(const Params &p, const ASmem &a, int b, int h, float m, float l, int slot,
                         int mt) {
    static_assert(D <= kMThreads, "one management thread per output element");
    constexpr int WST = AsyncSizes<ES, RK, RV, D, WL>::WST;
    using V = VStage<ES, RV, D, WST>;
    using P = typename V::P;
    const float *vcur = a.xtra + slot * 2 * D, *muv = vcur + D;
    const bool pass1 = p.cur_k != nullptr;
    const int64_t orow = (static_cast<int64_t>(b) * p.H + h) * D;
    float M = m, pc = 0.f;
    if (pass1) {
        const float sc = m_part(a, slot, 0) * p.scale_log2;
        M = fmaxf(m, sc);
        pc = exp2f(sc - M);
    }
    const float wl = exp2f(m - M);
    const float lc = l * wl;
    const float inv = 1.f / (lc + pc);
    if (!p.absorbed) {
        for (int e = mt; e < D; e += kMThreads) {
            const float o = fmaf(pc, vcur[e], a.s.ovec[e] * wl);
            store_elem(p.out, orow + e, o * inv, p.io_bf16);
        }
        m_sync();
        return;
    }
    const char *W = static_cast<const char *>(p.w_up_v) +
                    (static_cast<int64_t>(h) * p.T + p.loop) * D * RV * ES;
    const int er = mt % P::ROWS, sub = mt / P::ROWS;
#pragma unroll 1
    for (int pass = 0; pass < P::N; ++pass) {
        cp_async_wait_all();
        m_sync();
        float acc0 = 0.f, acc1 = 0.f;
#pragma unroll 4
        for (int c = sub; c < V::CPR; c += V::TPR) {
            float w[V::EPC];
            load_gran<ES, V::CB>(a.wst + (c * P::ROWS + er) * V::CB, w);
            const float *ov = a.s.ovec + c * V::EPC;
#pragma unroll
            for (int k = 0; k < V::EPC; ++k) {
                if (k & 1) acc1 = fmaf(w[k], ov[k], acc1);
                else acc0 = fmaf(w[k], ov[k], acc0);
            }
        }
        float acc = acc0 + acc1;
        if constexpr (V::TPR > 1) {
            a.mtmp[mt] = acc;
            m_sync();
            if (sub == 0) {
#pragma unroll
                for (int t = 1; t < V::TPR; ++t) acc += a.mtmp[er + t * P::ROWS];
            }
        }
        if (sub == 0) {
            const int e = pass * P::ROWS + er;
            float o = fmaf(lc, muv[e], acc * wl);
            o = fmaf(pc, vcur[e], o);
            store_elem(p.out, orow + e, o * inv, p.io_bf16);
        }
        m_sync();  // the buffer (and mtmp) is read before the next pass or set-up overwrites it
        if (pass + 1 < P::N) m_stage_v<ES, RV, D, WST>(a, W, pass + 1, mt);
    }
}

__device__ __forceinline__ int atom_add_acq_rel_gpu(int *addr, int v) {
    int old;
    asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], %2;" : "=r"(old) : "l"(addr), "r"(v) : "memory");
    return old;
}

// Management: the run that left its state in slot `slot` -- reduce it, then finish the
// (sequence, head) in place, or write a partial and merge all of them if this CTA is the last
// to arrive.  One acquire-release atomic both publishes this CTA's partial and tells the last
// CTA that every other partial is visible.  With RELEASE false the state slot stays taken (a
// later finish reads more of it and releases it).
template <int ES, int RK, int RV, int D, int TT, int NTG, int WL = kWstMax, bool RELEASE = true>
__device__ void m_finish(const Params &p, const ASmem &a, const Run &R, int64_t u, const Range &rg,
                         int slot, uint32_t parity, int qs, int mt) {
    constexpr int WST = AsyncSizes<ES, RK, RV, D, WL>::WST;
    // The output's first pass of W_up,t^V travels while the run still streams.  Earlier uses of
    // the staging buffer (a set-up's reads, a finish that returned with its copies in flight)
    // are over before it is written again.
    if (p.absorbed) {
        cp_async_wait_all();
        m_sync();
        m_stage_v<ES, RV, D, WST>(a, static_cast<const char *>(p.w_up_v) +
                                         (static_cast<int64_t>(R.h) * p.T + p.loop) * D * RV * ES,
                                  0, mt);
    }
    mbar_wait(&a.stfull[slot], parity, a.s.abort_flag, p.err, wait_limit(p));
    const float *red = a.red + slot * a.redslot;
    const float *lred = a.lred + slot * kLredSlot;
    for (int j = mt; j < RV; j += kMThreads) {  // fixed order: bitwise-reproducible sums
        float acc = 0.f;
#pragma unroll 4
        for (int g = 0; g < NTG; ++g) acc += red[g * RV + j];
        a.s.ovec[j] = acc;
    }
    float l = 0.f;
    for (int i = 0; i < TT; ++i) l += lred[i];
    const float m = a.s.misc[kAM + slot];
    m_sync();
    if constexpr (RELEASE) mbar_arrive(&a.stfree[slot]);  // the slot may take a later run's state
    if (u == R.seg_start && R.run_end == R.seg_end) {
        m_output<ES, RK, RV, D, WL>(p, a, R.b, R.h, m, l, qs, mt);
        return;
    }
    const int c = blockIdx.x;
    const int pslot = (R.seg_start <= rg.A0) ? 0 : 1;
    float *rec = p.partials + (static_cast<int64_t>(c) * 2 + pslot) * (RV + 2);
    if (mt == 0) {
        rec[0] = m;
        rec[1] = l;
    }
    for (int j = mt; j < RV; j += kMThreads) rec[2 + j] = a.s.ovec[j];
    m_sync();
    const int c_first = owner_of(R.seg_start, rg.U, rg.Geff);
    const int c_last = owner_of(R.seg_end - 1, rg.U, rg.Geff);
    int *counter = &p.counters[R.b * p.H + R.h];
    if (mt == 0) {
        const int prev = atom_add_acq_rel_gpu(counter, 1);
        *a.s.last_flag = (prev == c_last - c_first);
    }
    m_sync();
    if (!*a.s.last_flag) return;
    auto record = [&](int cc) {
        const int sl = (R.seg_start <= range_start(cc, rg.U, rg.Geff)) ? 0 : 1;
        return p.partials + (static_cast<int64_t>(cc) * 2 + sl) * (RV + 2);
    };
    const int nparts = c_last - c_first + 1;
    constexpr int kQuick = 8;  // parts merged with every load issued in one round trip
    float M = -INFINITY, lsum = 0.f;
    if (nparts <= kQuick) {
        constexpr int JPT = (RV + kMThreads - 1) / kMThreads;  // columns per thread
        float pm[kQuick], pl[kQuick], po[kQuick][JPT];
#pragma unroll
        for (int k = 0; k < kQuick; ++k) {
            if (k < nparts) {
                const float *r = record(c_first + k);
                pm[k] = __ldcg(r);
                pl[k] = __ldcg(r + 1);
#pragma unroll
                for (int q = 0; q < JPT; ++q) {
                    const int j = mt + q * kMThreads;
                    po[k][q] = j < RV ? __ldcg(r + 2 + j) : 0.f;
                }
            }
        }
#pragma unroll
        for (int k = 0; k < kQuick; ++k)
            if (k < nparts) M = fmaxf(M, pm[k]);
        float acc[JPT];
#pragma unroll
        for (int q = 0; q < JPT; ++q) acc[q] = 0.f;
#pragma unroll
        for (int k = 0; k < kQuick; ++k) {
            if (k < nparts) {
                const float w = exp2f(pm[k] - M);
                lsum = fmaf(pl[k], w, lsum);
#pragma unroll
                for (int q = 0; q < JPT; ++q) acc[q] = fmaf(po[k][q], w, acc[q]);
            }
        }
#pragma unroll
        for (int q = 0; q < JPT; ++q) {
            const int j = mt + q * kMThreads;
            if (j < RV) a.s.ovec[j] = acc[q];
        }
    } else {
        for (int c0 = 0; c0 < nparts; c0 += kMThreads) {
            const int np = min(kMThreads, nparts - c0);
            if (mt < np) {
                const float *r = record(c_first + c0 + mt);
                a.mtmp[mt] = __ldcg(r);
                a.mtmp[kMThreads + mt] = __ldcg(r + 1);
            }
            m_sync();
            float Mc = M;
            for (int i = 0; i < np; ++i) Mc = fmaxf(Mc, a.mtmp[i]);
            lsum *= exp2f(M - Mc);
            for (int i = 0; i < np; ++i) lsum = fmaf(a.mtmp[kMThreads + i], exp2f(a.mtmp[i] - Mc), lsum);
            M = Mc;
            m_sync();
        }
        for (int j = mt; j < RV; j += kMThreads) {
            float acc = 0.f;
#pragma unroll 4
            for (int cc = c_first; cc <= c_last; ++cc) {
                const float *r = record(cc);
                acc = fmaf(__ldcg(r + 2 + j), exp2f(__ldcg(r) - M), acc);
            }
            a.s.ovec[j] = acc;
        }
    }
    m_sync();
    m_output<ES, RK, RV, D, WL>(p, a, R.b, R.h, M, lsum, qs, mt);
    if (mt == 0) atomicExch(counter, 0);
}

template <typename Kern, typename Prm>
lla_status launch_kernel(Kern kern, DeviceOnce &configured, const Prm &prm, int grid, int smem,
                         cudaStream_t stream, int threads = kThreads) {
    if (raise_smem_limit(kern, kSmemLimit, configured) != LLA_OK) return LLA_ERR_CUDA;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
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

// Pages per pipeline step: small head pages are grouped so one step moves about 32 KiB.
int pages_per_step(int hpb) {
    if (4 * hpb <= kStepTargetBytes) return 4;
    if (2 * hpb <= kStepTargetBytes) return 2;
    return 1;
}

}  // namespace
}  // namespace lla
