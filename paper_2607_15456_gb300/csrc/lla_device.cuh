// lla_device.cuh -- device helpers shared by the liblla kernels (sm_103a, inline PTX).
//
// mbarrier waits are bounded: a wait that has not completed within its limit (kWaitLimitNs of
// global time unless the launch passes a shorter one) sets LLA_DEVERR_TIMEOUT in the error word
// and reports failure, so no kernel here can spin forever.  Callers keep going after a failed
// wait (with undefined results) so that every CTA still reaches every barrier and exits; a
// producer stops issuing copies once a wait has failed and waits, with the full limit, for the
// copies it has in flight before its CTA exits.
#pragma once

#include <cuda_bf16.h>
#include <stdint.h>

#include "../../include/lla.h"

namespace lla {

constexpr int kBlockTokens = LLA_BLOCK_TOKENS;
constexpr uint64_t kWaitLimitNs = LLA_DEFAULT_WAIT_LIMIT_NS;  // 2 s of global time per wait

__device__ __forceinline__ uint64_t global_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__device__ __forceinline__ uint32_t smem_addr(const void *p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count));
}

__device__ __forceinline__ void fence_mbar_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t *bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)),
                 "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t *bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}

// Tests phase `parity` of `bar`; while it is incomplete the thread is suspended by the hardware
// for up to kSuspendNs (it does not spin and take issue slots from other warps).
constexpr uint32_t kSuspendNs = 1000000;  // 1 ms

__device__ __forceinline__ bool mbar_try_wait(uint64_t *bar, uint32_t parity,
                                              uint32_t suspend_ns = kSuspendNs) {
    uint32_t done;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(done)
        : "r"(smem_addr(bar)), "r"(parity), "r"(suspend_ns)
        : "memory");
    return done != 0;
}

// Non-blocking test of phase `parity` of `bar` (no suspension when the phase is incomplete).
__device__ __forceinline__ bool mbar_test_wait(uint64_t *bar, uint32_t parity) {
    uint32_t done;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(done)
        : "r"(smem_addr(bar)), "r"(parity)
        : "memory");
    return done != 0;
}

// Bounded wait on phase `parity` of `bar`.  Returns false (and flags the error word) when the
// wait expired after `limit_ns` of global time, or at once when `abort_flag` (shared) was
// already raised by another thread.  The flag is written before the caller's next arrival on
// any barrier, so a thread that completes a phase those arrivals end sees it raised.
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t parity, volatile int *abort_flag,
                                          unsigned *err, uint64_t limit_ns = kWaitLimitNs) {
    if (mbar_test_wait(bar, parity)) return true;  // already complete: no suspension
    if (*abort_flag) return false;
    const uint32_t hint = limit_ns < kSuspendNs ? static_cast<uint32_t>(limit_ns) : kSuspendNs;
    if (mbar_try_wait(bar, parity, hint)) return true;
    const uint64_t t0 = global_ns();
    for (;;) {
        if (mbar_try_wait(bar, parity, hint)) return true;
        if (*abort_flag) return false;
        if (global_ns() - t0 > limit_ns) {
            *abort_flag = 1;
            atomicOr(err, LLA_DEVERR_TIMEOUT);
            return false;
        }
    }
}

// One bulk copy (TMA engine, no tensor map): `bytes` (multiple of 16) from global `src`
// (16-byte aligned) to shared `dst` (16-byte aligned), completing on `bar`.
__device__ __forceinline__ void bulk_g2s(void *dst, const void *src, uint32_t bytes, uint64_t *bar,
                                         uint64_t policy) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
        " [%0], [%1], %2, [%3], %4;" ::"r"(smem_addr(dst)),
        "l"(src), "r"(bytes), "r"(smem_addr(bar)), "l"(policy)
        : "memory");
}

// 16-byte asynchronous copy global -> shared (no register holds the data in flight).
__device__ __forceinline__ void cp_async16(void *smem_dst, const void *gsrc) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_addr(smem_dst)), "l"(gsrc)
                 : "memory");
}
__device__ __forceinline__ void cp_async4(void *smem_dst, const void *gsrc) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(smem_addr(smem_dst)), "l"(gsrc) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all() {
    asm volatile("cp.async.wait_group 0;" ::: "memory");
}
// all but the most recent group of copies have landed
__device__ __forceinline__ void cp_async_wait_but_one() {
    asm volatile("cp.async.wait_group 1;" ::: "memory");
}

__device__ __forceinline__ uint64_t policy_evict_first() {
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
    return p;
}

__device__ __forceinline__ void named_bar_sync(int id, int nthreads) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}

__device__ __forceinline__ void named_bar_arrive(int id, int nthreads) {
    asm volatile("bar.arrive %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}

// Programmatic dependent launch: wait for the previous grid in the stream to complete (or to
// trigger), and allow the next grid to be scheduled.  Both are no-ops without the attribute.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// bf16 pair (low element in the low half) to two floats; exact.
__device__ __forceinline__ float2 bf2_to_f2(uint32_t u) {
    return make_float2(__uint_as_float(u << 16), __uint_as_float(u & 0xffff0000u));
}

__device__ __forceinline__ float bf_to_f(uint16_t u) {
    return __uint_as_float(static_cast<uint32_t>(u) << 16);
}

// Loads element i of an array of `dtype` (LLA_BF16 / LLA_F32) as float.
__device__ __forceinline__ float load_elem(const void *base, int64_t i, int is_bf16) {
    if (is_bf16) return bf_to_f(reinterpret_cast<const uint16_t *>(base)[i]);
    return reinterpret_cast<const float *>(base)[i];
}

__device__ __forceinline__ void store_elem(void *base, int64_t i, float v, int is_bf16) {
    if (is_bf16)
        reinterpret_cast<__nv_bfloat16 *>(base)[i] = __float2bfloat16_rn(v);
    else
        reinterpret_cast<float *>(base)[i] = v;
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// (cos, sin) of pos turns of phi / 2^64 (phi = theta / 2 pi in 64-bit fixed point): the product
// wraps modulo one turn exactly, and 32 bits of the fraction reach sincospif.
__device__ __forceinline__ void turn_sincos(long long pos, unsigned long long phi, float *sn, float *cs) {
    const unsigned long long turns = static_cast<unsigned long long>(pos) * phi;
    const float tf = __uint2float_rn(static_cast<uint32_t>(turns >> 32)) * 2.3283064365386963e-10f;
    sincospif(2.f * tf, sn, cs);
}

// Byte offset of element (row i, column j) inside a K-plane (see lla.h).
__host__ __device__ __forceinline__ int64_t kplane_offset(int i, int j, int es, int gk) {
    const int byte = j * es;
    return static_cast<int64_t>(byte / gk) * (kBlockTokens * gk) + i * gk + (byte % gk);
}

__host__ __device__ __forceinline__ int granule_bytes(int r, int es) {
    return ((r * es) % 16 == 0) ? 16 : 4;
}

}  // namespace lla
