// Bulk-copy (TMA) and mbarrier helpers for sm_103a, inline PTX.
//
// 1-D bulk copies (cp.async.bulk) move contiguous global byte ranges into
// shared memory and signal an mbarrier with the byte count.  Every wait is
// bounded: on timeout the kernel records an error code in g_pipo_error (read by
// the host after the step) instead of spinning forever.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace pipo {

// Device error word: 0 = fine; kErrWaitTimeout when a bounded wait gave up.
// One copy per translation unit (the kernels are compiled in several); the
// host reads and clears every unit's copy after a step (take_unit_error).
static __device__ unsigned int g_pipo_error;
// First wait that gave up: {site code, linear block index, iteration, parity}
// (the site codes name the wait: 11-15 projection GEMM producer-empty,
// producer-drain, MMA-full, epilogue-accumulator, converter-full; 21-23 attention
// producer-empty, producer-drain, consumer-full; 24-26 prefill attention; 27 the
// staged single-sequence attention;
// 90 the wait self-test).
static __device__ unsigned int g_pipo_error_info[4];
constexpr unsigned kErrWaitTimeout = 1u;
constexpr unsigned long long kWaitNs = 2000000000ull;  // give up after 2 s of waiting

// Host: read and clear this translation unit's error word and wait record.
static inline cudaError_t take_unit_error(unsigned* code, unsigned info[4]) {
    cudaError_t e = cudaMemcpyFromSymbol(code, g_pipo_error, sizeof(unsigned));
    if (e != cudaSuccess || *code == 0) return e;
    e = cudaMemcpyFromSymbol(info, g_pipo_error_info, 4 * sizeof(unsigned));
    if (e != cudaSuccess) return e;
    const unsigned zero[4] = {0, 0, 0, 0};
    e = cudaMemcpyToSymbol(g_pipo_error, zero, sizeof(unsigned));
    if (e == cudaSuccess) e = cudaMemcpyToSymbol(g_pipo_error_info, zero, sizeof(zero));
    return e;
}

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

// make barrier initialisation visible to the async (bulk-copy) proxy
__device__ __forceinline__ void mbar_init_fence() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void fence_proxy_async() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

// global -> shared bulk copy of `bytes` (multiple of 16, both addresses
// 16-byte aligned), completing on `bar`
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
            smem_u32(dst)),
        "l"(src), "r"(bytes), "r"(smem_u32(bar))
        : "memory");
}

// start fetching a tensor map (kernel parameter) into the TMA descriptor cache
__device__ __forceinline__ void prefetch_tmap(const CUtensorMap* tm) {
    asm volatile("prefetch.tensormap [%0];" ::"l"(tm) : "memory");
}

// 2-D tiled tensor copy (TMA) of the box at element coordinates (x, y) of the
// tensor map into shared memory, completing on `bar`
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* tm, int x, int y, uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
            smem_u32(dst)),
        "l"(tm), "r"(x), "r"(y), "r"(smem_u32(bar))
        : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

__device__ __forceinline__ unsigned long long global_ns() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Bounded wait for phase `parity` of `bar`: false (and the error word set)
// once limit_ns of wall time (kWaitNs unless given) have passed without the
// phase completing; the first wait to give up records `site`, its block and
// `iter` for the host.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, unsigned site = 0, unsigned iter = 0,
                                          unsigned long long limit_ns = kWaitNs) {
    if (mbar_try_wait(bar, parity)) return true;
    const unsigned long long t0 = global_ns();
    for (;;) {
        for (int i = 0; i < 64; ++i)
            if (mbar_try_wait(bar, parity)) return true;
        if (global_ns() - t0 > limit_ns) break;
    }
    atomicOr(&g_pipo_error, kErrWaitTimeout);
    if (atomicCAS(&g_pipo_error_info[0], 0u, site ? site : 99u) == 0u) {
        g_pipo_error_info[1] = blockIdx.x + gridDim.x * (blockIdx.y + gridDim.y * blockIdx.z);
        g_pipo_error_info[2] = iter;
        g_pipo_error_info[3] = parity;
    }
    return false;
}

}  // namespace pipo
