// bc_tma.cuh -- the shared-memory pipeline primitives of the streaming kernels (sm_103a):
// 1-D TMA bulk copies (cp.async.bulk, global -> shared) completing on mbarriers with a
// transaction count, and mbarrier waits bounded in time.
//
// A stage's mbarrier is initialised with one arrival; the producer thread arms it with
// mbarrier.arrive.expect_tx (the bytes the stage will receive) and issues the bulk copies,
// whose completion decrements the transaction count; the phase flips when both are done.
// Waiters spin on mbarrier.try_wait.parity with a limit of kTmaWaitNs by %globaltimer (and
// an iteration backstop), so a completion that never comes ends in a reported failure,
// never in a hung device.
#pragma once

#include <cuda_runtime.h>

#include <atomic>
#include <cstdint>

namespace bc {

constexpr uint64_t kTmaWaitNs = 1000000000ull;   // about one second

__device__ __forceinline__ uint32_t smem_u32(const void *p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t global_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count)
                 : "memory");
}

// Make the initialised barriers visible to the async proxy (the bulk copies).
__device__ __forceinline__ void mbar_init_fence() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t *bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
                 "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t *bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
        " selp.u32 %0, 1, 0, p;\n}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

// Wait for the given phase parity; false if the time limit (or, as a backstop, an
// iteration count) passed first.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t *bar, uint32_t parity) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = global_ns();
    for (uint32_t spins = 0; !mbar_try_wait(bar, parity); ++spins)
        if (global_ns() - t0 > kTmaWaitNs || spins > (1u << 26)) return false;
    return true;
}

// Copy `bytes` (a multiple of 16; both addresses 16-byte aligned) from global to shared
// memory, completing on `bar`.
__device__ __forceinline__ void bulk_copy_to_shared(void *dst, const void *src, uint32_t bytes,
                                                    uint64_t *bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
        ::"r"(smem_u32(dst)), "l"(src), "r"(bytes), "r"(smem_u32(bar))
        : "memory");
}

// Order this thread's earlier shared-memory accesses before later async-proxy operations
// on shared memory (a bulk store issued after the data landed).
__device__ __forceinline__ void fence_proxy_async_shared() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Copy `bytes` (a multiple of 16; both addresses 16-byte aligned) from shared to global
// memory as part of the current bulk async-group.
__device__ __forceinline__ void bulk_store_from_shared(void *dst, const void *src,
                                                       uint32_t bytes) {
    asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;"
                 ::"l"(dst), "r"(smem_u32(src)), "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ void bulk_commit_group() {
    asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}

// Wait until at most N of this thread's bulk groups still read their shared-memory source.
template <int N>
__device__ __forceinline__ void bulk_wait_group_read() {
    asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(N) : "memory");
}

// Wait until every bulk group of this thread has completed (its writes are performed).
__device__ __forceinline__ void bulk_wait_group_all() {
    asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
}

// Host side: raise a pipeline kernel's dynamic shared-memory limit to `bytes`, once per
// device (host threads may race here; they set the same value).
template <class KernelPtr>
int ensure_smem_attribute(KernelPtr kern, std::atomic<bool> (&done)[64], int bytes) {
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev >= 0 && dev < 64 && done[dev].load(std::memory_order_acquire)) return cudaSuccess;
    const int err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (err != cudaSuccess) {
        cudaGetLastError();  // reported once, by return value, not again to later calls
        return err;
    }
    if (dev >= 0 && dev < 64) done[dev].store(true, std::memory_order_release);
    return cudaSuccess;
}

}  // namespace bc
