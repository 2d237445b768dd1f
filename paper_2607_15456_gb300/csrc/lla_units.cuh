// lla_units.cuh -- the page split shared by the tensor-core decode kernels (lla_decode_2d.cu,
// lla_decode_rope_tc.cu): the units of a batch (a sequence, or a (sequence, head) pair) own
// consecutive ranges of a global page numbering, which is cut into equal page ranges, one per
// CTA; a CTA takes its range as runs (its part of one unit).
#pragma once

#include <cuda_runtime.h>

#include <stdint.h>

#include "lla_device.cuh"
#include "lla_internal.h"

namespace lla {
namespace {

// CTA c of `grid` holds the global pages [page_lo(c), page_lo(c + 1)) of the np pages; with
// fewer pages than CTAs some CTAs hold none.
__host__ __device__ __forceinline__ int page_lo(int c, int np, int grid) {
    return static_cast<int>(static_cast<int64_t>(c) * np / grid);
}

// The CTA that holds global page g (the last c with page_lo(c) <= g).
__host__ __device__ __forceinline__ int cta_of(int g, int np, int grid) {
    return static_cast<int>((static_cast<int64_t>(g + 1) * grid + np - 1) / np) - 1;
}

// A launch on `stream` that may start before the previous kernel in the stream has finished
// (programmatic dependent launch: the kernel waits for it with pdl_wait).
template <typename K, typename... Args>
lla_status launch_ex(K kern, dim3 grid, int threads, int smem, cudaStream_t stream, Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = dim3(threads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (cudaLaunchKernelEx(&cfg, kern, args...) != cudaSuccess) return LLA_ERR_CUDA;
    return LLA_OK;
}

}  // namespace
}  // namespace lla
