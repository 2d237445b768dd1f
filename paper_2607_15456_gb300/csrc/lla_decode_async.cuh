// lla_decode_async.cuh -- the shape-specialised decode kernel with asynchronous run boundaries
// (App. A "Decoding and caching", App. J "Absorbed attention"), shared by lla_decode.cu (the
// absorbed decode and the dense comparator) and lla_decode_decoupled.cu (the same kernel with the
// decoupled rotary branch of App. J: one rotary key per token, shared by every head and loop,
// scored against the query's rotary part turned at the current position).  Everything here has
// internal linkage.
#pragma once

#include "lla_decode_common.cuh"

namespace lla {
namespace {

constexpr int kMaxRopePairs = 48;  // d_rope <= 96

// Launch parameters of the rotary branch: the decode parameters, the rotary planes (one per
// block, [64 x d_rope] bf16 in the K-plane's granule layout), the rotary query q^R [B][H][d_rope]
// and, in pass 1, the current token's rotary key [B][d_rope], and theta_j of every pair in 64-bit
// fixed-point turns (theta_j / 2 pi * 2^64).
struct DecParams {
    Params p;
    const char *rope_pool;
    const void *q_rope, *cur_k_rope;
    int pairing;  // 0: pair j = (j, j + d_rope/2); 1: (2j, 2j + 1)
    unsigned long long phi[kMaxRopePairs];
};

template <int DR>
struct KParamsOf {
    using type = DecParams;
};
template <>
struct KParamsOf<0> {
    using type = Params;
};
__device__ __forceinline__ const Params &base_params(const Params &p) { return p; }
__device__ __forceinline__ const Params &base_params(const DecParams &d) { return d.p; }

// Byte offset of the rotary query slots ([kQSlots][d_rope] floats) after the shared layout.
template <int ES, int RK, int RV, int D>
__host__ __device__ inline int rotary_query_offset(int stages, int stage_bytes, int B) {
    return (async_layout<ES, RK, RV, D>(stages, stage_bytes, B).total + 15) & ~15;
}

// Management warps, after m_setup of a run: rot(q^R, P) into the run's rotary query slot, with P
// the current token's position (its context length in pass 1, one less in pass 2), and in pass 1
// q^R . k^R_cur added to the partial of q . k_cur (both sit at P, so the rotation cancels).
template <int DR>
__device__ void m_rotary(const DecParams &d, const ASmem &a, int b, int h, int slot, int mt, float *rq) {
    const Params &p = d.p;
    const bool pass1 = p.cur_k != nullptr;
    const int L = a.s.lens[b];
    const long long P = max(0, pass1 ? L : L - 1);
    const int64_t src = (static_cast<int64_t>(b) * p.H + h) * DR;
    float *dst = rq + slot * DR;
    for (int j = mt; j < DR / 2; j += kMThreads) {
        float sn, cs;
        turn_sincos(P, d.phi[j], &sn, &cs);
        const int ia = d.pairing ? 2 * j : j, ic = d.pairing ? 2 * j + 1 : j + DR / 2;
        const float x = load_elem(d.q_rope, src + ia, p.io_bf16);
        const float y = load_elem(d.q_rope, src + ic, p.io_bf16);
        dst[ia] = x * cs - y * sn;
        dst[ic] = x * sn + y * cs;
    }
    if (pass1) {
        float part = 0.f;
        for (int e = mt; e < DR; e += kMThreads)
            part = fmaf(load_elem(d.q_rope, src + e, p.io_bf16),
                        load_elem(d.cur_k_rope, static_cast<int64_t>(b) * DR + e, p.io_bf16), part);
        part = warp_sum(part);
        // the same lane wrote this warp's q . k_cur partial in m_setup
        if ((mt & 31) == 0) a.s.misc[kAPart + slot * 8 + (mt >> 5) * 2] += part;
    }
}

template <int ES, int RK, int RV, int D, int DR>
__global__ void __launch_bounds__(kAsyncThreads, 1)
    decode_async_kernel(const __grid_constant__ typename KParamsOf<DR>::type kprm) {
    using F = Fast<ES, RK, RV>;
    static_assert(DR == 0 || (F::PPS == 1 && DR % 16 == 0 && ES == 2), "rotary branch: one page per step");
    const Params &p = base_params(kprm);
    extern __shared__ __align__(128) char smem[];
    const ASmem a = carve_async<ES, RK, RV, D>(smem, p);
    // rotary branch: rot(q^R, P) of each query slot, after the shared layout
    float *rq = reinterpret_cast<float *>(smem + rotary_query_offset<ES, RK, RV, D>(p.stages, p.stage_bytes, p.B));
    const Smem &s = a.s;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

    pdl_wait();  // inputs may come from the previous kernel in the stream
    if (tid == 0) {
        for (int i = 0; i < kQSlots; ++i) mbar_init(&a.qready[i], kMThreads);
        for (int i = 0; i < 2; ++i) {
            mbar_init(&a.stfull[i], kComputeThreads);
            mbar_init(&a.stfree[i], kMThreads);
        }
    }
    Range rg = prologue(p, s, F::S_THREADS, F::V_THREADS);  // fences the inits above too
    order_runs(p, s, rg);
    pdl_trigger();

    if (warp == kComputeWarps) {
        if (rg.A0 < rg.A1) named_bar_sync(kBarStart, kMThreads + 32);
        if constexpr (DR > 0) producer(p, s, rg, kprm.rope_pool, kBlockTokens * DR * 2);
        else producer(p, s, rg);
        return;
    }

    if (tid >= kMBase) {
        // ---------------------------------------------------------------- management warps
        const int mt = tid - kMBase;
        // set-ups run two runs ahead of finishes: set-up(r), then finish(r - 2), so that a short
        // run is never followed by a wait for the next run's q~ behind a merge
        auto finish = [&](const Run &R, int64_t u, int k) {
            m_finish<ES, RK, RV, D, F::TT, F::NTG>(p, a, R, u, rg, k & 1, (k >> 1) & 1, k % kQSlots, mt);
        };
        int r = 0;
        Run q0{}, q1{};  // runs r - 2 and r - 1, awaiting their finish
        int64_t u0 = 0, u1 = 0;
        for (int pass = 0; pass < 3; ++pass)
        for (int64_t u = rg.lo[pass]; u < rg.hi[pass];) {
            const Run R = locate_run(p, s, u, rg.hi[pass]);
            const int slot = r % kQSlots;
            m_setup<ES, RK, RV, D>(p, a, R.b, R.h, slot, mt, r == 0);
            if constexpr (DR > 0) m_rotary<DR>(kprm, a, R.b, R.h, slot, mt, rq);
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
        // sequences with no cached token: pass 1 attends to the current token only
        const bool pass1 = p.cur_k != nullptr;
        for (int b = 0; b < p.B; ++b) {
            if (s.lens[b] != 0) continue;
            for (int h = 0; h < p.H; ++h) {
                if ((b * p.H + h) % gridDim.x != blockIdx.x) continue;
                const int64_t row = (static_cast<int64_t>(b) * p.H + h) * D;
                if (!pass1 && mt == 0) atomicOr(p.err, LLA_DEVERR_EMPTY_PASS2);
                for (int e = mt; e < D; e += kMThreads)
                    store_elem(p.out, row + e, pass1 ? load_elem(p.cur_v, row + e, p.io_bf16) : 0.f,
                               p.io_bf16);
            }
        }
        cp_async_wait_all();  // no copy into shared memory outlives the CTA
        return;
    }

    // ------------------------------------------------------------------ score and value warps
    const bool is_s = warp < F::S_WARPS;
    const int ks = tid / F::TT, tt = tid % F::TT;  // score threads
    const int vt = tid - F::S_THREADS;              // value threads
    const int vc = vt % F::VC, tg = vt / F::VC;
    const bool vwork = !is_s && tg < F::NTG;
    constexpr int AV = F::UPT * F::VE;

    int it = 0, stage = 0, r = 0;
    uint32_t ph = 0;
    for (int pass = 0; pass < 3; ++pass)
    for (int64_t u = rg.lo[pass]; u < rg.hi[pass]; ++r) {
        const Run R = locate_run(p, s, u, rg.hi[pass]);
        const int rslot = r & 1;         // state slot
        const int qslot = r % kQSlots;   // query slot
        float beta = 0.f;
        const float *qq = a.qlat + qslot * a.qslot + ks * F::NGT * F::KE;
        // q~ of this thread's granules stays in registers for the whole run when it is small
        // enough (up to 48 floats); else it is re-read from shared memory (a broadcast) per token
        constexpr bool kQreg = F::NGT * F::KE <= 48;
        float qr[kQreg ? F::NGT * F::KE : 1];
        if (is_s) {
            mbar_wait(&a.qready[qslot], (r / kQSlots) & 1, s.abort_flag, p.err, wait_limit(p));
            beta = m_part(a, qslot, 1);
            if constexpr (kQreg) {
#pragma unroll
                for (int g = 0; g < F::NGT; ++g) {
                    if (F::NGK % F::KSPLIT != 0 && ks * F::NGT + g >= F::NGK) break;
                    float t[F::KE];
                    load_qvec<F::KE>(qq + g * F::KE, t);
#pragma unroll
                    for (int e = 0; e < F::KE; ++e) qr[g * F::KE + e] = t[e];
                }
            }
        }
        float m_run = -INFINITY, l_part = 0.f;
        float accv[AV];
#pragma unroll
        for (int e = 0; e < AV; ++e) accv[e] = 0.f;

        for (int k = 0; k < R.npages; k += F::PPS, ++it) {
            const int slot = it & 1;
            const uint32_t pph = (it >> 1) & 1;
            const char *sb = s.ring + stage * p.stage_bytes;
            const int n = min(F::PPS, R.npages - k);
            const int tok0 = (R.pg0 + k) * kBlockTokens;
            const int nvalid = min(n * kBlockTokens, R.Lb - tok0);
            float *pring = s.psm + slot * kComputeThreads;

            if (is_s) {
                mbar_wait(&s.full[stage], ph, s.abort_flag, p.err, wait_limit(p));
                float sc[F::TPT];
#pragma unroll
                for (int i = 0; i < F::TPT; ++i) {
                    const int tok = tt + i * F::TT;
                    float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
                    if (tok < nvalid) {
                        const char *kp = sb + (tok >> 6) * F::HPB + (tok & 63) * F::GK +
                                         ks * F::NGT * (kBlockTokens * F::GK);
#pragma unroll
                        for (int g = 0; g < F::NGT; ++g) {
                            if (F::NGK % F::KSPLIT != 0 && ks * F::NGT + g >= F::NGK) break;
                            float v[F::KE], qv[F::KE];
                            load_gran<ES, F::GK>(kp + g * (kBlockTokens * F::GK), v);
                            if constexpr (kQreg) {
#pragma unroll
                                for (int e = 0; e < F::KE; ++e) qv[e] = qr[g * F::KE + e];
                            } else {
                                load_qvec<F::KE>(qq + g * F::KE, qv);  // broadcast read
                            }
#pragma unroll
                            for (int e = 0; e < F::KE; ++e) {
                                if ((e & 3) == 0) a0 = fmaf(v[e], qv[e], a0);
                                else if ((e & 3) == 1) a1 = fmaf(v[e], qv[e], a1);
                                else if ((e & 3) == 2) a2 = fmaf(v[e], qv[e], a2);
                                else a3 = fmaf(v[e], qv[e], a3);
                            }
                        }
                        if constexpr (DR > 0) {
                            // the rotary key of the token (plane after the head page, same granule
                            // layout) against rot(q^R, P); the k-splits share its granules too
                            constexpr int NGR = DR / 8, NGRT = (NGR + F::KSPLIT - 1) / F::KSPLIT;
                            const char *rpp = sb + F::HPB + (tok & 63) * 16 + ks * NGRT * (kBlockTokens * 16);
                            const float *rqq = rq + qslot * DR + ks * NGRT * 8;
#pragma unroll
                            for (int g = 0; g < NGRT; ++g) {
                                if (NGR % F::KSPLIT != 0 && ks * NGRT + g >= NGR) break;
                                float v[8], qv[8];
                                load_gran<2, 16>(rpp + g * (kBlockTokens * 16), v);
                                load_qvec<8>(rqq + g * 8, qv);
#pragma unroll
                                for (int e = 0; e < 8; e += 4) {
                                    a0 = fmaf(v[e], qv[e], a0);
                                    a1 = fmaf(v[e + 1], qv[e + 1], a1);
                                    a2 = fmaf(v[e + 2], qv[e + 2], a2);
                                    a3 = fmaf(v[e + 3], qv[e + 3], a3);
                                }
                            }
                        }
                    }
                    sc[i] = (a0 + a1) + (a2 + a3);
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(&s.empty[stage]);  // K-plane read
                if constexpr (F::KSPLIT == 2) {
                    if (ks == 1) {
#pragma unroll
                        for (int i = 0; i < F::TPT; ++i) s.spart[tt + i * F::TT] = sc[i];
                    }
                    named_bar_sync(kBarTok, F::S_THREADS);
                    if (ks == 0) {
#pragma unroll
                        for (int i = 0; i < F::TPT; ++i) sc[i] += s.spart[tt + i * F::TT];
                    }
                }
                float x[F::TPT];
                float lm = -INFINITY;
#pragma unroll
                for (int i = 0; i < F::TPT; ++i) {
                    const bool valid = tt + i * F::TT < nvalid;
                    x[i] = valid ? (sc[i] + beta) * p.scale_log2 : -INFINITY;
                    lm = fmaxf(lm, x[i]);
                }
                float *wmax = s.misc + kAWmax + slot * 8;
                if (ks == 0) {
                    lm = warp_max(lm);
                    if (lane == 0) wmax[warp] = lm;
                }
                named_bar_sync(kBarTok, F::S_THREADS);
                float ms = wmax[0];
#pragma unroll
                for (int w = 1; w < F::TT / 32; ++w) ms = fmaxf(ms, wmax[w]);
                const float m_new = fmaxf(m_run, ms);
                const float alpha = exp2f(m_run - m_new);
                m_run = m_new;
                if (ks == 0) {
                    mbar_wait(&s.pempty[slot], pph ^ 1u, s.abort_flag, p.err, wait_limit(p));
                    float lsum = 0.f;
#pragma unroll
                    for (int i = 0; i < F::TPT; ++i) {
                        const float pv = (tt + i * F::TT < nvalid) ? exp2f(x[i] - m_new) : 0.f;
                        pring[tt + i * F::TT] = pv;
                        lsum += pv;
                    }
                    l_part = fmaf(l_part, alpha, lsum);
                    if (tid == 0) s.misc[kAPAlpha + slot] = alpha;
                }
                mbar_arrive(&s.pfull[slot]);
            } else {
                mbar_wait(&s.full[stage], ph, s.abort_flag, p.err, wait_limit(p));
                mbar_wait(&s.pfull[slot], pph, s.abort_flag, p.err, wait_limit(p));
                if (vwork) value_step<ES, RK, RV>(accv, sb, pring, s.misc[kAPAlpha + slot], nvalid, vc, tg);
                mbar_arrive(&s.pempty[slot]);
                __syncwarp();
                if (lane == 0) mbar_arrive(&s.empty[stage]);  // V-plane read
            }
            if (++stage == p.stages) {
                stage = 0;
                ph ^= 1u;
            }
        }

        // leave the run's softmax state in slot rslot for the management warps, once the run
        // that used the slot before (r - 2) has been read
        if (r >= 2) mbar_wait(&a.stfree[rslot], ((r - 2) >> 1) & 1, s.abort_flag, p.err, wait_limit(p));
        if (is_s && ks == 0) a.lred[rslot * kLredSlot + tt] = l_part;
        if (tid == 0) s.misc[kAM + rslot] = m_run;
        if (vwork) value_store<ES, RK, RV>(a.red + rslot * a.redslot, accv, vc, tg);
        mbar_arrive(&a.stfull[rslot]);
        u = R.run_end;
    }
}


}  // namespace
}  // namespace lla
