// lla_internal.h -- host-side interface between the C ABI (lla_abi.cu) and the kernel files.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include <atomic>

#include "../../include/lla.h"

namespace lla {

// Everything one decode launch needs (one layer, one loop, B sequences).
struct DecodeArgs {
    int T, H, d, r_k, r_v, loop;
    int absorbed;  // 1: latent cache with codec; 0: dense comparator (r_k = r_v = d, no codec)
    int storage_bf16, io_bf16;
    float scale;
    const void *w_up_k, *w_up_v;  // [H][T][d][r] storage dtype (absorbed only)
    const float *mu_k, *mu_v;     // [H][T*d] or NULL
    const void *pool;
    int64_t num_blocks;
    const int32_t *block_table;
    int max_blocks;
    const int32_t *context_lens;
    int B, max_ctx;
    const void *q, *cur_k, *cur_v;
    void *out;
    void *workspace;
    size_t workspace_bytes;
};

struct EncodeArgs {
    int T, H, d, r_k, r_v;
    int storage_bf16, x_bf16;
    const void *w_down_k, *w_down_v;  // [H][T*d][r]
    const float *mu_k, *mu_v;         // [H][T*d] or NULL
    const void *x_k, *x_v;            // [T][N][H][d]
    void *pool;
    int64_t num_blocks;
    const int64_t *slot_mapping;
    int N;
    int dense;  // 1: store x_k / x_v ([N][H][d]) as plain K/V pages (r_k = r_v = d, T = 1)
};

struct PrefillArgs {
    int T, H, d, r_k, r_v, loop;
    int storage_bf16, io_bf16;
    float scale;
    const void *w_up_k, *w_up_v;
    const float *mu_k, *mu_v;
    const void *pool;
    int64_t num_blocks;
    const int32_t *block_table;
    int max_blocks;
    const int32_t *cu_seqlens;
    int B, max_len;
    const void *q;
    void *out;
};

// Per-device address of the sticky error word (owned by lla_abi.cu).
unsigned *device_error_word(lla_status *st);

// Bytes of one head page (K-plane + V-plane) and of one block.
inline size_t head_page_bytes(int r_k, int r_v, int es) {
    return static_cast<size_t>(LLA_BLOCK_TOKENS) * (r_k + r_v) * es;
}

// Decode: workspace bytes for `grid` CTAs and B sequences (split-KV partial records, then the
// B*H arrival counters from decode_counters_offset on, the only part that must start at zero);
// launch.
size_t decode_counters_offset(int r_v, int grid);
size_t decode_workspace_bytes(int r_v, int B, int H, int grid);
lla_status decode_fits(int r_k, int r_v, int es, int d);  // UNSUPPORTED if no kernel shape fits
lla_status launch_decode(const DecodeArgs &a, cudaStream_t stream);
// Decode with rotary positions after reconstruction (tensor-core key rebuild): UNSUPPORTED
// unless a kernel shape exists and fits for B sequences; the launch takes the rotation base and
// pairing (0: (j, j + d/2), 1: (2j, 2j + 1)).
lla_status decode_rope_fits(int r_k, int r_v, int es, int d, int B);
// The decode calls of all T loops in one pass over the latents (q, cur_k, cur_v, out are
// [T][B][H][d]; the shared-latent tensor-core kernels of lla_decode_2d.cu with one unit per
// (sequence, head)): UNSUPPORTED unless a kernel shape exists; its workspace size.
lla_status decode_loops_fits(int r_k, int r_v, int es, int d, int T, int B);
size_t decode_loops_workspace_bytes(int r_k, int r_v, int B, int H, int grid);
lla_status launch_decode_loops(const DecodeArgs &a, cudaStream_t stream);
lla_status launch_decode_rope(const DecodeArgs &a, double base, int pairing, cudaStream_t stream);
// Per rotation pair j of a 128-wide head: theta_j = base^(-2j/128) as 64-bit fixed-point turns,
// and cos / sin of theta_j and of 32 theta_j, sin 2 theta_j and 1 - cos 2 theta_j (computed in
// double precision; the last without cancellation).
struct RopeTables {
    unsigned long long phi[64];
    float c1[64], s1[64], c32[64], s32[64], s2[64], h2[64];
};
void rope_tables(double base, int d, RopeTables *t);
// The full-RoPE decode with the latent value sum on the tensor cores (units of one (sequence,
// head) each, a separate merge kernel): the shapes with a kernel, its workspace, launch.  Its
// workspace slots return to zero when a call completes.
bool decode_rope_tc_supported(int es, int d, int r_k, int r_v);
size_t decode_rope_tc_workspace_bytes(int r_v, int B, int H, int grid);
lla_status launch_decode_rope_tc(const DecodeArgs &a, const RopeTables &t, int pairing, cudaStream_t stream);

lla_status launch_encode(const EncodeArgs &a, cudaStream_t stream);
// The same encode for L layers (one launch for decode batches).
constexpr int kMaxEncodeLayers = 64;
lla_status launch_encode_layers(const EncodeArgs *a, int L, cudaStream_t stream);
// Tensor-core encode for prompts (bf16 x and storage, N >= 128, instantiated ranks).
bool encode_tc_supported(const EncodeArgs &a);
lla_status launch_encode_tc(const EncodeArgs &a, cudaStream_t stream);
lla_status launch_prefill(const PrefillArgs &a, cudaStream_t stream);
// Prefill with rotary positions after reconstruction: keys rebuilt and rotated into the
// workspace, then the tensor-core attention over them (bf16 storage, d = 128, the prefill ranks).
size_t prefill_rope_workspace_bytes(int B, int max_len, int H);
bool prefill_rope_supported(int es, int d, int r_k, int r_v);
lla_status launch_prefill_rope(const PrefillArgs &a, double base, int pairing, void *workspace,
                               size_t workspace_bytes, cudaStream_t stream);

// LLA-2D decode (one latent per token and layer; w_up_* [T][H][d][r], mu_* [T*H*d]): the
// shapes with a kernel, the workspace for B sequences (0 if the device is unknown), launch.
bool decode_2d_supported(int es, int d, int H, int r_k, int r_v);
size_t decode_2d_workspace_bytes(int r_k, int r_v, int B);
lla_status launch_decode_2d(const DecodeArgs &a, cudaStream_t stream);
// theta_j = base^(-2j/d_rope) of each rotation pair in 64-bit fixed-point turns.
void rotary_phases(int d_rope, double base, unsigned long long *phi);
// Per-head LLA decode with the decoupled rotary branch (App. J) on the absorbed decode kernel: the
// shapes with a kernel, the workspace for B sequences of H heads (the absorbed decode's: zeroed
// once, its counters return to zero), launch (rope_pool [num_blocks][64 x d_rope] rotary planes,
// q_rope [B][H][d_rope], cur_k_rope [B][d_rope] in pass 1); and the rotary-key store.
bool decode_decoupled_supported(int es, int d, int H, int r_k, int r_v, int d_rope);
size_t decode_decoupled_workspace_bytes(int r_k, int r_v, int d_rope, int B, int H);
lla_status launch_decode_decoupled(const DecodeArgs &a, const void *rope_pool, int d_rope, double base,
                                   int pairing, const void *q_rope, const void *cur_k_rope,
                                   cudaStream_t stream);
lla_status launch_rope_key_store(int d_rope, double base, int pairing, void *rope_pool, int64_t num_blocks,
                                 const void *k, int x_bf16, const int32_t *positions, const int64_t *slots,
                                 int N, cudaStream_t stream);

int num_sms();  // SM count of the current device (cached), 0 on failure

// Per-device flags of a one-time kernel set-up.  Host threads that race on a first call both
// make the same set-up call; each flag is atomic.
struct DeviceOnce {
    std::atomic<bool> done[64];
};

// Raises the dynamic shared-memory limit of `kern` to `bytes` on the current device, once per
// device (a flag in `once`).
template <typename K>
inline lla_status raise_smem_limit(K kern, int bytes, DeviceOnce &once) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return LLA_ERR_CUDA;
    const bool cached = dev >= 0 && dev < 64;
    if (cached && once.done[dev].load(std::memory_order_acquire)) return LLA_OK;
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes) != cudaSuccess)
        return LLA_ERR_CUDA;
    if (cached) once.done[dev].store(true, std::memory_order_release);
    return LLA_OK;
}

// The limit of each pipeline wait in lla_decode_attn / lla_dense_decode_attn launches, as set by
// lla_set_wait_limit_ns (0: the kernels' own 2 s).
uint64_t pipeline_wait_limit_ns();

}  // namespace lla
