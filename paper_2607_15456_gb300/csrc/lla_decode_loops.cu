// lla_decode_loops.cu -- the decode calls of all T loops of a layer in one pass over the latents:
// several queries against a shared latent.
//
// The latent of a (token, layer, head) is one stacked code for every loop (Sec. 3, Eq. encode),
// and the loop-t key and value come from it through loop-t up-projections (Eq. decode).  Attention
// at loop t absorbs them (App. J): q~_t = W_up,t^K^T q_t, s_t,i = scale (q~_t . c_k,i + q_t .
// mu^K_t), o_t = (W_up,t^V sum_i p_t,i c_v,i + l_t mu^V_t + p_t,cur v_t,cur) / (l_t + p_t,cur).
// When the T loop queries of a step are available together (loops computed in parallel or
// speculatively, or a verification of several loop outputs), their T decode calls read the same
// latents: this kernel streams each latent page once and forms all T scores, softmaxes and latent
// value sums from it, so a layer's latent bytes cross HBM once instead of T times.  Each loop's
// result is that of lla_decode_attn at that loop.
//
// GB300 mapping: the warp roles, the persistent split of (sequence, head, page) units, the TMA ring
// and the split-KV merge are those of the absorbed kernel (lla_decode_common.cuh); the score warps
// form T dot products per token (q~_t read as shared-memory broadcasts), the online softmax keeps T
// states, the value warps keep T latent sums (one 16-byte unit of 8 latents per thread, so that a
// run's state stays small), and the management warps set up and finish the T loops of a run one
// after the other through per-loop views of the run state.
// one head page per pipeline step at every rank shape this kernel takes
#define LLA_DECODE_STEP_BYTES (32 * 1024)
#include "lla_decode_common.cuh"

namespace lla {
namespace {

constexpr int kLoopsWst = 40 * 1024;  // staging buffer of W_up,t rows (one pass each)
constexpr int kNQ = 4;                // loops per call

template <int RK, int RV>
struct LoopShape {
    using F = Fast<2, RK, RV>;               // score-role geometry of the absorbed kernel
    static constexpr int D = 128;
    static constexpr int VB = 16, VE = 8;    // one 16-byte unit of 8 latents per value thread
    static constexpr int VC = RV * 2 / VB;   // value threads per V row
    static constexpr int NTG = F::V_THREADS / VC;  // token groups of value threads
    static constexpr int REDSLOT = NTG * RV;       // value partials of one run and loop
    static constexpr int QSLOT = AsyncSizes<2, RK, RV, D, kLoopsWst>::QSLOT;
    static constexpr int MRED = AsyncSizes<2, RK, RV, D, kLoopsWst>::MRED;
    static constexpr int WST = AsyncSizes<2, RK, RV, D, kLoopsWst>::WST;
    static_assert(F::PPS == 1 && F::TT == 64 && F::KSPLIT == 2, "one page per step, two k-splits");
    static_assert((RV * 2) % VB == 0 && NTG >= 1, "value units");
};

struct LoopLayout {
    int ring, full, empty, pfull, pempty, qready, stfull, stfree, prefix, lens, qfull, psm, ovec,
        mred, mtmp, misc, wst, qlat, spart, lred, red, xtra, miscl, total;
};

template <int RK, int RV>
__host__ __device__ inline LoopLayout loop_layout(int stages, int stage_bytes, int B) {
    using Z = LoopShape<RK, RV>;
    LoopLayout L;
    int o = 0;
    L.ring = o;   o += stages * stage_bytes;
    L.full = o;   o += stages * 8;
    L.empty = o;  o += stages * 8;
    L.pfull = o;  o += 16;
    L.pempty = o; o += 16;
    L.qready = o; o += 32;
    L.stfull = o; o += 16;
    L.stfree = o; o += 16;
    L.prefix = o; o += up16((B + 1) * 8);
    L.lens = o;   o += up16(B * 4);
    L.qfull = o;  o += up16(Z::QSLOT * 4);
    L.psm = o;    o += 2 * kNQ * 64 * 4;             // [2 page slots][loop][token]
    L.ovec = o;   o += up16(RV * 4);
    L.mred = o;   o += up16(Z::MRED * 4);
    L.mtmp = o;   o += 2 * kMThreads * 4;
    L.misc = o;   o += 64 * 4;
    L.wst = o;    o += up16(Z::WST);
    L.qlat = o;   o += kNQ * kQSlots * Z::QSLOT * 4; // [loop][query slot][q~]
    L.spart = o;  o += kNQ * 64 * 4;                 // [loop][token] second k-split
    L.lred = o;   o += kNQ * 2 * kLredSlot * 4;      // [loop][state slot][score thread]
    L.red = o;    o += up16(kNQ * 2 * Z::REDSLOT * 4);  // [loop][state slot][token group][RV]
    L.xtra = o;   o += kNQ * kQSlots * 2 * Z::D * 4; // [loop][query slot][v_cur, mu^V_t]
    L.miscl = o;  o += kNQ * 64 * 4;                 // [loop][misc slots]
    L.total = o;
    return L;
}

// The shared view of the state, then the view of loop t: its q~ slots, run-state slots, v_cur and
// mu^V_t, and misc slots (run maxima, beta and q . k_cur partials, softmax alphas and maxima).
struct LoopSmem {
    ASmem a;
    float *qlat, *spart, *lred, *red, *xtra, *miscl;
};

template <int RK, int RV>
__device__ __forceinline__ LoopSmem carve_loops(char *smem, const Params &p) {
    using Z = LoopShape<RK, RV>;
    const LoopLayout L = loop_layout<RK, RV>(p.stages, p.stage_bytes, p.B);
    LoopSmem l;
    ASmem &a = l.a;
    a.s.ring = smem + L.ring;
    a.s.full = reinterpret_cast<uint64_t *>(smem + L.full);
    a.s.empty = reinterpret_cast<uint64_t *>(smem + L.empty);
    a.s.pfull = reinterpret_cast<uint64_t *>(smem + L.pfull);
    a.s.pempty = reinterpret_cast<uint64_t *>(smem + L.pempty);
    a.s.prefix = reinterpret_cast<int64_t *>(smem + L.prefix);
    a.s.lens = reinterpret_cast<int *>(smem + L.lens);
    a.s.qlat = a.s.qfull = a.s.spart = a.s.tmp = a.s.red = a.s.lred = nullptr;
    a.s.psm = reinterpret_cast<float *>(smem + L.psm);
    a.s.ovec = reinterpret_cast<float *>(smem + L.ovec);
    a.s.misc = reinterpret_cast<float *>(smem + L.misc);
    a.s.abort_flag = reinterpret_cast<volatile int *>(a.s.misc + kAAbort);
    a.s.last_flag = reinterpret_cast<int *>(a.s.misc + kALast);
    a.qready = reinterpret_cast<uint64_t *>(smem + L.qready);
    a.stfull = reinterpret_cast<uint64_t *>(smem + L.stfull);
    a.stfree = reinterpret_cast<uint64_t *>(smem + L.stfree);
    a.qfull = reinterpret_cast<float *>(smem + L.qfull);
    a.mred = reinterpret_cast<float *>(smem + L.mred);
    a.mtmp = reinterpret_cast<float *>(smem + L.mtmp);
    a.wst = smem + L.wst;
    a.qslot = Z::QSLOT;
    a.redslot = Z::REDSLOT;
    a.qlat = a.lred = a.red = a.xtra = nullptr;
    l.qlat = reinterpret_cast<float *>(smem + L.qlat);
    l.spart = reinterpret_cast<float *>(smem + L.spart);
    l.lred = reinterpret_cast<float *>(smem + L.lred);
    l.red = reinterpret_cast<float *>(smem + L.red);
    l.xtra = reinterpret_cast<float *>(smem + L.xtra);
    l.miscl = reinterpret_cast<float *>(smem + L.miscl);
    return l;
}

template <int RK, int RV>
__device__ __forceinline__ ASmem loop_view(const LoopSmem &l, int t) {
    using Z = LoopShape<RK, RV>;
    ASmem a = l.a;
    a.qlat = l.qlat + t * kQSlots * Z::QSLOT;
    a.lred = l.lred + t * 2 * kLredSlot;
    a.red = l.red + t * 2 * Z::REDSLOT;
    a.xtra = l.xtra + t * kQSlots * 2 * Z::D;
    a.s.misc = l.miscl + t * 64;  // the abort and last flags stay those of the shared misc slots
    return a;
}

// The decode arguments of loop t: its inputs, outputs and split-KV records.
__device__ __forceinline__ Params loop_params(const Params &p, int t, int grid) {
    Params q = p;
    const int64_t n = static_cast<int64_t>(p.B) * p.H * p.d;
    const int es = p.io_bf16 ? 2 : 4;
    q.loop = t;
    q.q = static_cast<const char *>(p.q) + t * n * es;
    if (p.cur_k) {
        q.cur_k = static_cast<const char *>(p.cur_k) + t * n * es;
        q.cur_v = static_cast<const char *>(p.cur_v) + t * n * es;
    }
    q.out = static_cast<char *>(p.out) + t * n * es;
    q.partials = p.partials + static_cast<int64_t>(t) * grid * 2 * (p.r_v + 2);
    q.counters = p.counters + static_cast<int64_t>(t) * p.B * p.H;
    return q;
}

template <int RK, int RV>
__global__ void __launch_bounds__(kAsyncThreads, 1) decode_loops_kernel(const Params p) {
    using Z = LoopShape<RK, RV>;
    using F = typename Z::F;
    constexpr int ES = 2, D = Z::D;
    extern __shared__ __align__(128) char smem[];
    const LoopSmem l = carve_loops<RK, RV>(smem, p);
    const ASmem &a = l.a;
    const Smem &s = a.s;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

    if (tid == 0) {
        for (int i = 0; i < kQSlots; ++i) mbar_init(&a.qready[i], kMThreads);
        for (int i = 0; i < 2; ++i) {
            mbar_init(&a.stfull[i], kComputeThreads);
            mbar_init(&a.stfree[i], kMThreads);
        }
    }
    pdl_wait();  // inputs may come from the previous kernel in the stream
    Range rg = prologue(p, s, F::S_THREADS, F::V_THREADS);  // fences the inits above too
    order_runs(p, s, rg);
    pdl_trigger();

    if (warp == kComputeWarps) {
        if (rg.A0 < rg.A1) named_bar_sync(kBarStart, kMThreads + 32);
        producer(p, s, rg);
        return;
    }

    if (tid >= kMBase) {
        // ---------------------------------------------------------------- management warps
        const int mt = tid - kMBase;
        auto finish = [&](const Run &R, int64_t u, int k) {
            for (int t = 0; t < kNQ; ++t) {
                const Params pt = loop_params(p, t, gridDim.x);
                const ASmem at = loop_view<RK, RV>(l, t);
                // the state slot is released once the last loop has read it
                if (t + 1 < kNQ)
                    m_finish<ES, RK, RV, D, F::TT, Z::NTG, kLoopsWst, false>(pt, at, R, u, rg, k & 1,
                                                                          (k >> 1) & 1, k % kQSlots, mt);
                else
                    m_finish<ES, RK, RV, D, F::TT, Z::NTG, kLoopsWst, true>(pt, at, R, u, rg, k & 1,
                                                                         (k >> 1) & 1, k % kQSlots, mt);
            }
        };
        int r = 0;
        Run q0{}, q1{};
        int64_t u0 = 0, u1 = 0;
        for (int pass = 0; pass < 3; ++pass)
        for (int64_t u = rg.lo[pass]; u < rg.hi[pass];) {
            const Run R = locate_run(p, s, u, rg.hi[pass]);
            const int slot = r % kQSlots;
            for (int t = 0; t < kNQ; ++t)
                m_setup<ES, RK, RV, D, true, kLoopsWst>(loop_params(p, t, gridDim.x), loop_view<RK, RV>(l, t),
                                                        R.b, R.h, slot, mt, r == 0 && t == 0);
            m_sync();  // the last set-up's q~ is complete before the score warps read it
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
        const bool pass1 = p.cur_k != nullptr;
        for (int b = 0; b < p.B; ++b) {  // no cached token: pass 1 attends to the current token
            if (s.lens[b] != 0) continue;
            for (int h = 0; h < p.H; ++h) {
                if ((b * p.H + h) % gridDim.x != blockIdx.x) continue;
                if (!pass1 && mt == 0) atomicOr(p.err, LLA_DEVERR_EMPTY_PASS2);
                for (int t = 0; t < kNQ; ++t) {
                    const Params pt = loop_params(p, t, gridDim.x);
                    const int64_t row = (static_cast<int64_t>(b) * p.H + h) * D;
                    for (int e = mt; e < D; e += kMThreads)
                        store_elem(pt.out, row + e, pass1 ? load_elem(pt.cur_v, row + e, p.io_bf16) : 0.f,
                                   p.io_bf16);
                }
            }
        }
        cp_async_wait_all();
        return;
    }

    // ------------------------------------------------------------------ score and value warps
    const bool is_s = warp < F::S_WARPS;
    const int ks = tid / F::TT, tt = tid % F::TT;  // score threads: k-split, token
    const int vt = tid - F::S_THREADS;              // value threads: unit vc of row group tg
    const int vc = vt % Z::VC, tg = vt / Z::VC;
    const bool vwork = !is_s && tg < Z::NTG;

    int it = 0, stage = 0, r = 0;
    uint32_t ph = 0;
    for (int pass = 0; pass < 3; ++pass)
    for (int64_t u = rg.lo[pass]; u < rg.hi[pass]; ++r) {
        const Run R = locate_run(p, s, u, rg.hi[pass]);
        const int rslot = r & 1, qslot = r % kQSlots;
        float beta[kNQ];
        if (is_s) {
            mbar_wait(&a.qready[qslot], (r / kQSlots) & 1, s.abort_flag, p.err);
#pragma unroll
            for (int t = 0; t < kNQ; ++t) beta[t] = m_part(loop_view<RK, RV>(l, t), qslot, 1);
        }
        float m_run[kNQ], l_part[kNQ];
        float accv[kNQ][Z::VE];
#pragma unroll
        for (int t = 0; t < kNQ; ++t) {
            m_run[t] = -INFINITY;
            l_part[t] = 0.f;
#pragma unroll
            for (int e = 0; e < Z::VE; ++e) accv[t][e] = 0.f;
        }

        for (int k = 0; k < R.npages; ++k, ++it) {
            const int slot = it & 1;
            const uint32_t pph = (it >> 1) & 1;
            const char *sb = s.ring + stage * p.stage_bytes;
            const int nvalid = min(kBlockTokens, R.Lb - (R.pg0 + k) * kBlockTokens);
            float *pring = s.psm + slot * kNQ * 64;  // [loop][token]

            if (is_s) {
                mbar_wait(&s.full[stage], ph, s.abort_flag, p.err);
                float sc[kNQ];
                {
                    float2 acc[kNQ];  // even and odd latent columns, packed
#pragma unroll
                    for (int t = 0; t < kNQ; ++t) acc[t] = make_float2(0.f, 0.f);
                    if (tt < nvalid) {
                        const char *kp = sb + tt * F::GK + ks * F::NGT * (kBlockTokens * F::GK);
#pragma unroll
                        for (int g = 0; g < F::NGT; ++g) {
                            if (F::NGK % F::KSPLIT != 0 && ks * F::NGT + g >= F::NGK) break;
                            float v[F::KE];
                            load_gran<ES, F::GK>(kp + g * (kBlockTokens * F::GK), v);
#pragma unroll
                            for (int t = 0; t < kNQ; ++t) {
                                float qv[F::KE];  // broadcast read of q~_t
                                load_qvec<F::KE>(l.qlat + (t * kQSlots + qslot) * Z::QSLOT +
                                                     (ks * F::NGT + g) * F::KE, qv);
#pragma unroll
                                for (int e = 0; e < F::KE; e += 2)
                                    acc[t] = __ffma2_rn(make_float2(v[e], v[e + 1]),
                                                        make_float2(qv[e], qv[e + 1]), acc[t]);
                            }
                        }
                    }
#pragma unroll
                    for (int t = 0; t < kNQ; ++t) sc[t] = acc[t].x + acc[t].y;
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(&s.empty[stage]);  // K-plane read
                if (ks == 1) {
#pragma unroll
                    for (int t = 0; t < kNQ; ++t) l.spart[t * 64 + tt] = sc[t];
                }
                named_bar_sync(kBarTok, F::S_THREADS);
                const bool valid = tt < nvalid;
                float x[kNQ];
                if (ks == 0) {
                    float lm[kNQ];
#pragma unroll
                    for (int t = 0; t < kNQ; ++t) {
                        x[t] = valid ? (sc[t] + l.spart[t * 64 + tt] + beta[t]) * p.scale_log2 : -INFINITY;
                        lm[t] = x[t];
                    }
#pragma unroll
                    for (int o = 16; o > 0; o >>= 1)  // the T warp maxima, interleaved
#pragma unroll
                        for (int t = 0; t < kNQ; ++t) lm[t] = fmaxf(lm[t], __shfl_xor_sync(0xffffffffu, lm[t], o));
                    if (lane == 0) {
#pragma unroll
                        for (int t = 0; t < kNQ; ++t) l.miscl[t * 64 + kAWmax + slot * 8 + warp] = lm[t];
                    }
                }
                named_bar_sync(kBarTok, F::S_THREADS);
                float alpha[kNQ];
#pragma unroll
                for (int t = 0; t < kNQ; ++t) {
                    const float *wm = l.miscl + t * 64 + kAWmax + slot * 8;
                    const float m_new = fmaxf(m_run[t], fmaxf(wm[0], wm[1]));
                    alpha[t] = exp2f(m_run[t] - m_new);
                    m_run[t] = m_new;
                }
                if (ks == 0) {
                    mbar_wait(&s.pempty[slot], pph ^ 1u, s.abort_flag, p.err);
#pragma unroll
                    for (int t = 0; t < kNQ; ++t) {
                        const float pv = valid ? exp2f(x[t] - m_run[t]) : 0.f;
                        pring[t * 64 + tt] = pv;
                        l_part[t] = fmaf(l_part[t], alpha[t], pv);
                        if (tid == 0) l.miscl[t * 64 + kAPAlpha + slot] = alpha[t];
                    }
                }
                mbar_arrive(&s.pfull[slot]);
            } else {
                mbar_wait(&s.full[stage], ph, s.abort_flag, p.err);
                mbar_wait(&s.pfull[slot], pph, s.abort_flag, p.err);
                if (vwork) {
#pragma unroll
                    for (int t = 0; t < kNQ; ++t) {
                        const float al = l.miscl[t * 64 + kAPAlpha + slot];
#pragma unroll
                        for (int e = 0; e < Z::VE; ++e) accv[t][e] *= al;
                    }
                    const char *vp = sb + F::KPLANE + tg * F::ROWB + vc * Z::VB;
                    const int cnt = nvalid > tg ? (nvalid - tg + Z::NTG - 1) / Z::NTG : 0;
#pragma unroll 4
                    for (int i = 0; i < cnt; ++i) {
                        const int row = tg + i * Z::NTG;
                        float v[Z::VE];
                        load_gran<ES, Z::VB>(vp + i * (Z::NTG * F::ROWB), v);
#pragma unroll
                        for (int t = 0; t < kNQ; ++t) {
                            const float pv = pring[t * 64 + row];
                            const float2 p2 = make_float2(pv, pv);
#pragma unroll
                            for (int e = 0; e < Z::VE; e += 2) {
                                const float2 rr = __ffma2_rn(p2, make_float2(v[e], v[e + 1]),
                                                             make_float2(accv[t][e], accv[t][e + 1]));
                                accv[t][e] = rr.x;
                                accv[t][e + 1] = rr.y;
                            }
                        }
                    }
                }
                mbar_arrive(&s.pempty[slot]);
                __syncwarp();
                if (lane == 0) mbar_arrive(&s.empty[stage]);  // V-plane read
            }
            if (++stage == p.stages) {
                stage = 0;
                ph ^= 1u;
            }
        }

        // leave the run's T softmax states in slot rslot for the management warps, once the run
        // that used the slot before (r - 2) has been read
        if (r >= 2) mbar_wait(&a.stfree[rslot], ((r - 2) >> 1) & 1, s.abort_flag, p.err);
#pragma unroll
        for (int t = 0; t < kNQ; ++t) {
            if (is_s && ks == 0) l.lred[(t * 2 + rslot) * kLredSlot + tt] = l_part[t];
            if (tid == 0) l.miscl[t * 64 + kAM + rslot] = m_run[t];
            if (vwork) {
                float *red = l.red + (t * 2 + rslot) * Z::REDSLOT + tg * RV + vc * Z::VE;
#pragma unroll
                for (int e = 0; e < Z::VE; ++e) red[e] = accv[t][e];
            }
        }
        mbar_arrive(&a.stfull[rslot]);
        u = R.run_end;
    }
}

template <int RK, int RV>
lla_status launch_loops(const Params &prm, int grid, int smem, cudaStream_t stream) {
    static bool configured[64] = {};
    return launch_kernel(decode_loops_kernel<RK, RV>, configured, prm, grid, smem, stream, kAsyncThreads);
}

template <int RK, int RV>
int loops_layout_bytes(int stages, int stage_bytes, int B) {
    return loop_layout<RK, RV>(stages, stage_bytes, B).total;
}

struct LoopsEntry {
    lla_status (*launch)(const Params &, int, int, cudaStream_t);
    int (*layout)(int, int, int);
};
LoopsEntry loops_entry(int es, int d, int T, int r_k, int r_v) {
    if (es != 2 || d != 128 || T != kNQ) return LoopsEntry{nullptr, nullptr};
    if (r_k == 96 && r_v == 160) return LoopsEntry{launch_loops<96, 160>, loops_layout_bytes<96, 160>};
    if (r_k == 128 && r_v == 128) return LoopsEntry{launch_loops<128, 128>, loops_layout_bytes<128, 128>};
    if (r_k == 72 && r_v == 120) return LoopsEntry{launch_loops<72, 120>, loops_layout_bytes<72, 120>};
    return LoopsEntry{nullptr, nullptr};
}

int loops_stages(const LoopsEntry &e, int stage_bytes, int B) {
    const int fixed = e.layout(0, stage_bytes, B);
    const int stages = (kSmemLimit - fixed) / (stage_bytes + 16);
    return stages > kMaxStages ? kMaxStages : stages;
}

}  // namespace

lla_status decode_loops_fits(int r_k, int r_v, int es, int d, int T, int B) {
    const LoopsEntry e = loops_entry(es, d, T, r_k, r_v);
    if (!e.launch) return LLA_ERR_UNSUPPORTED;
    const int hpb = static_cast<int>(head_page_bytes(r_k, r_v, es));
    return loops_stages(e, hpb, B) >= 2 ? LLA_OK : LLA_ERR_UNSUPPORTED;
}

size_t decode_loops_workspace_bytes(int r_v, int B, int H, int T, int grid) {
    const size_t part = static_cast<size_t>(T) * grid * 2 * (r_v + 2) * sizeof(float);
    const size_t part_al = (part + 255) & ~static_cast<size_t>(255);
    return part_al + static_cast<size_t>(T) * B * H * sizeof(int);
}

lla_status launch_decode_loops(const DecodeArgs &a, cudaStream_t stream) {
    const int es = a.storage_bf16 ? 2 : 4;
    const LoopsEntry e = loops_entry(es, a.d, a.T, a.r_k, a.r_v);
    if (!e.launch) return LLA_ERR_UNSUPPORTED;
    const int hpb = static_cast<int>(head_page_bytes(a.r_k, a.r_v, es));
    const int stages = loops_stages(e, hpb, a.B);
    if (stages < 2) return LLA_ERR_UNSUPPORTED;
    const int smem = e.layout(stages, hpb, a.B);
    const int grid = num_sms();
    if (grid <= 0) return LLA_ERR_CUDA;
    if (a.workspace_bytes < decode_loops_workspace_bytes(a.r_v, a.B, a.H, a.T, grid)) return LLA_ERR_WORKSPACE;
    lla_status st = LLA_OK;
    unsigned *err = device_error_word(&st);
    if (st != LLA_OK) return st;

    Params p = {};
    p.T = a.T; p.H = a.H; p.d = a.d; p.r_k = a.r_k; p.r_v = a.r_v; p.loop = 0;
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
    const size_t part = static_cast<size_t>(a.T) * grid * 2 * (a.r_v + 2) * sizeof(float);
    const size_t part_al = (part + 255) & ~static_cast<size_t>(255);
    p.partials = static_cast<float *>(a.workspace);
    p.counters = reinterpret_cast<int *>(static_cast<char *>(a.workspace) + part_al);
    p.pps = 1; p.stages = stages; p.stage_bytes = hpb;
    p.err = err;
    return e.launch(p, grid, smem, stream);
}

}  // namespace lla
