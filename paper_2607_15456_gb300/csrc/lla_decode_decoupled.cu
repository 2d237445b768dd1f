// lla_decode_decoupled.cu -- per-head LLA decode with the decoupled rotary branch (App. J
// "Absorbed attention": an MLA-style content path on the latents plus a small explicit rotary
// branch shared across recurrence steps; d_rope in Table decoupled_char).
//
// Score of cached token i at loop t, with P the current token's position:
//   s_i = scale (q~ . c_k,i + beta + rot(q^R, P) . k^R_i),   k^R_i stored turned at position i,
// and of the pass-1 current token s_cur = scale (q . k_cur + q^R . k^R_cur).  Values as in the
// absorbed decode.  This is the absorbed decode kernel (lla_decode_async.cuh) with one more
// operand per page: the block's rotary plane, one per block and layer, shared by every head,
// copied into the ring right after the head page; the score warps extend each token's dot
// product over its d_rope rotary dimensions, and the management warps turn q^R at P.
#include "lla_decode_async.cuh"

namespace lla {
namespace {

template <int DR>
lla_status launch_dec(const DecParams &dp, int grid, int smem, cudaStream_t stream) {
    static DeviceOnce configured;
    return launch_kernel(decode_async_kernel<2, 96, 160, 128, DR>, configured, dp, grid, smem, stream,
                         kAsyncThreads);
}

template <int DR>
int dec_layout_bytes(int stages, int stage_bytes, int B) {
    return rotary_query_offset<2, 96, 160, 128>(stages, stage_bytes, B) + kQSlots * DR * 4;
}

}  // namespace

bool decode_decoupled_supported(int es, int d, int H, int r_k, int r_v, int d_rope) {
    return es == 2 && d == 128 && H >= 1 && r_k == 96 && r_v == 160 &&
           (d_rope == 32 || d_rope == 64 || d_rope == 96);
}

size_t decode_decoupled_workspace_bytes(int r_k, int r_v, int d_rope, int B, int H) {
    (void)r_k;
    (void)d_rope;
    const int grid = num_sms();
    if (grid <= 0) return 0;
    return decode_workspace_bytes(r_v, B, H, grid);
}

lla_status launch_decode_decoupled(const DecodeArgs &a, const void *rope_pool, int d_rope, double base,
                                   int pairing, const void *q_rope, const void *cur_k_rope,
                                   cudaStream_t stream) {
    if (!decode_decoupled_supported(a.storage_bf16 ? 2 : 4, a.d, a.H, a.r_k, a.r_v, d_rope))
        return LLA_ERR_UNSUPPORTED;
    using Lay = int (*)(int, int, int);
    using Launch = lla_status (*)(const DecParams &, int, int, cudaStream_t);
    Lay lay = d_rope == 32 ? dec_layout_bytes<32> : d_rope == 64 ? dec_layout_bytes<64> : dec_layout_bytes<96>;
    Launch go = d_rope == 32 ? launch_dec<32> : d_rope == 64 ? launch_dec<64> : launch_dec<96>;
    const int hpb = static_cast<int>(head_page_bytes(a.r_k, a.r_v, 2));
    const int stage_bytes = hpb + LLA_BLOCK_TOKENS * d_rope * 2;  // head page, then the rotary plane
    int stages = (kSmemLimit - lay(0, stage_bytes, a.B)) / (stage_bytes + 16);
    if (stages > kMaxStages) stages = kMaxStages;
    if (stages < 2) return LLA_ERR_UNSUPPORTED;
    const int smem = lay(stages, stage_bytes, a.B);
    const int grid = num_sms();
    if (grid <= 0) return LLA_ERR_CUDA;
    if (a.workspace_bytes < decode_workspace_bytes(a.r_v, a.B, a.H, grid)) return LLA_ERR_WORKSPACE;
    lla_status st = LLA_OK;
    unsigned *err = device_error_word(&st);
    if (st != LLA_OK) return st;

    DecParams dp = {};
    Params &p = dp.p;
    p.T = a.T; p.H = a.H; p.d = a.d; p.r_k = a.r_k; p.r_v = a.r_v; p.loop = a.loop;
    p.absorbed = 1; p.io_bf16 = a.io_bf16;
    p.scale_log2 = a.scale * 1.4426950408889634f;
    p.w_up_k = a.w_up_k; p.w_up_v = a.w_up_v; p.mu_k = a.mu_k; p.mu_v = a.mu_v;
    p.pool = static_cast<const char *>(a.pool);
    p.num_blocks = a.num_blocks;
    p.block_bytes = static_cast<int64_t>(hpb) * a.H;
    p.head_page_bytes = hpb;
    p.kplane_bytes = kBlockTokens * a.r_k * 2;
    p.block_table = a.block_table; p.max_blocks = a.max_blocks;
    p.context_lens = a.context_lens; p.B = a.B; p.max_ctx = a.max_ctx;
    p.q = a.q; p.cur_k = a.cur_k; p.cur_v = a.cur_v; p.out = a.out;
    p.partials = static_cast<float *>(a.workspace);
    p.counters = reinterpret_cast<int *>(static_cast<char *>(a.workspace) + decode_counters_offset(a.r_v, grid));
    p.pps = 1; p.stages = stages; p.stage_bytes = stage_bytes;
    p.err = err;
    p.wait_ns = 0;
    dp.rope_pool = static_cast<const char *>(rope_pool);
    dp.q_rope = q_rope;
    dp.cur_k_rope = cur_k_rope;
    dp.pairing = pairing;
    rotary_phases(d_rope, base, dp.phi);
    return go(dp, grid, smem, stream);
}

}  // namespace lla
