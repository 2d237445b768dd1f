// lla_noalloc.cu -- lla_decode_attn_noalloc: the decode call with its scratch memory held in a
// fixed device array of this library instead of a workspace the caller allocates.
//
// Who needs it: callers that cannot allocate device memory, for example a plug-in running inside
// a host application that owns all device memory through its own pool and gives the plug-in no
// allocator, or a latency-critical loop where cudaMalloc (which can synchronise the whole device)
// is not acceptable.  Such callers still pass their inputs and outputs; only the decode scratch
// (the split-KV partial records and the per-(sequence, head) arrival counters) moves here.
//
// Rules of use:
//   * The array is kScratchBytes = 1 MiB.  It exists on every GPU that loads the library and is
//     held there until the process exits.  A call whose scratch need (the answer of
//     lla_decode_workspace_size for the same geometry and batch) is larger returns
//     LLA_ERR_WORKSPACE and enqueues nothing.
//   * All calls on a device share the one array, and it keeps whatever the last call left in it.
//     Calls that can overlap on the GPU (unordered streams, several host threads) race on it and
//     produce wrong results: order them on one stream.
//   * The first call on a device looks up the array's device address with cudaGetSymbolAddress,
//     with that device current, and keeps it for later calls.  Make that first call before any
//     stream capture.  The kept address belongs to the device's current context: after
//     cudaDeviceReset it is stale, and the library must not be called on that device again.
//   * Every call clears the arrival counters (the B*H integers at the end of its part of the
//     array, cudaMemsetAsync on the caller's stream), because they must start at zero.  The
//     split-KV partial records before them are always written before they are read, so stale
//     bytes there from an earlier call are never seen.  The clear is enqueued before
//     lla_decode_attn checks its remaining arguments, so a call rejected there leaves only the
//     clear of this library-owned array behind.
//   * Nothing here calls cudaMalloc, cudaFree or any allocating library routine.
#include <cuda_runtime.h>

#include <atomic>

#include "lla_internal.h"

namespace {

constexpr size_t kScratchBytes = size_t(1) << 20;
constexpr int kMaxDevices = 64;

// Host code must not take this name's address as a device pointer: on the host it is only a
// stand-in symbol.  scratch_address() returns the real device address.
static __device__ __align__(256) unsigned char g_decode_scratch[kScratchBytes];

// Host threads may make their first calls at the same time: every entry is atomic, and two
// threads that both look the address up store the same value.
std::atomic<void *> g_scratch_addr[kMaxDevices];

lla_status scratch_address(void **out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return LLA_ERR_CUDA;
    void *p = g_scratch_addr[dev].load(std::memory_order_acquire);
    if (!p) {
        if (cudaGetSymbolAddress(&p, g_decode_scratch) != cudaSuccess || !p) return LLA_ERR_CUDA;
        g_scratch_addr[dev].store(p, std::memory_order_release);
    }
    *out = p;
    return LLA_OK;
}

}  // namespace

extern "C" lla_status lla_decode_attn_noalloc(const lla_geometry *g, const lla_codec *codec,
                                              const lla_cache *cache, const int32_t *context_lens,
                                              int32_t B, int32_t max_ctx, int32_t loop,
                                              const void *q, const void *cur_k, const void *cur_v,
                                              lla_dtype io_dtype, void *out, void *stream) {
    size_t need = 0;
    lla_status st = lla_decode_workspace_size(g, B, &need);
    if (st != LLA_OK) return st;
    if (need > kScratchBytes) return LLA_ERR_WORKSPACE;
    void *scratch = nullptr;
    if ((st = scratch_address(&scratch)) != LLA_OK) return st;
    const int sms = lla::num_sms();
    if (sms <= 0) return LLA_ERR_CUDA;
    const size_t counters = lla::decode_counters_offset(g->r_v, sms);  // the counters start here
    if (B > 0 && need > counters &&
        cudaMemsetAsync(static_cast<char *>(scratch) + counters, 0, need - counters,
                        static_cast<cudaStream_t>(stream)) != cudaSuccess)
        return LLA_ERR_CUDA;
    return lla_decode_attn(g, codec, cache, context_lens, B, max_ctx, loop, q, cur_k, cur_v,
                           io_dtype, out, scratch, kScratchBytes, stream);
}
