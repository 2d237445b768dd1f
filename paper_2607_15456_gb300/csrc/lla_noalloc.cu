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
//     with that device current.  Make that first call before any stream capture.
//   * Every call clears the part of the array it uses (cudaMemsetAsync on the caller's stream),
//     because the arrival counters must start at zero.  That clear is enqueued before
//     lla_decode_attn checks its remaining arguments, so a call rejected there leaves only the
//     clear of this library-owned array behind.
//   * Nothing here calls cudaMalloc, cudaFree or any allocating library routine.
#include <cuda_runtime.h>

#include "lla_internal.h"

namespace {

constexpr size_t kScratchBytes = size_t(1) << 20;
constexpr int kMaxDevices = 64;

// Host code must not take this name's address as a device pointer: on the host it is only a
// stand-in symbol.  scratch_address() returns the real device address.
static __device__ __align__(256) unsigned char g_decode_scratch[kScratchBytes];

lla_status scratch_address(void **out) {
    static void *addr[kMaxDevices] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return LLA_ERR_CUDA;
    if (!addr[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_decode_scratch) != cudaSuccess || !p) return LLA_ERR_CUDA;
        addr[dev] = p;
    }
    *out = addr[dev];
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
    if (B > 0 && cudaMemsetAsync(scratch, 0, need, static_cast<cudaStream_t>(stream)) != cudaSuccess)
        return LLA_ERR_CUDA;
    return lla_decode_attn(g, codec, cache, context_lens, B, max_ctx, loop, q, cur_k, cur_v,
                           io_dtype, out, scratch, kScratchBytes, stream);
}
