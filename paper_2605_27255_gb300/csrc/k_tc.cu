// tcgen05 tensor-core projection kernels (a translation unit of its own).
#include "kernel_tables.h"
#include "tcgen05_gemm.cuh"

namespace pipo {

namespace {

template <int BH, bool DEEP>
void* tc_fn() { return reinterpret_cast<void*>(&gemm_tc_kernel<BH, tc_stages(BH, DEEP)>); }

template <bool DEEP>
void* pick_tc_v(int bh) {
    switch (bh) {
        case 16: return tc_fn<16, DEEP>();
        case 32: return tc_fn<32, DEEP>();
        case 64: return tc_fn<64, DEEP>();
        default: return tc_fn<128, DEEP>();
    }
}

template <int BH, bool DEEP>
void* tcf_fn() { return reinterpret_cast<void*>(&gemm_tcf_kernel<BH, tcf_stages(BH, DEEP)>); }

template <bool DEEP>
void* pick_tcf_v(int bh) {
    switch (bh) {
        case 16: return tcf_fn<16, DEEP>();
        case 32: return tcf_fn<32, DEEP>();
        case 64: return tcf_fn<64, DEEP>();
        default: return tcf_fn<128, DEEP>();
    }
}

}  // namespace

// fused (activation split inside the GEMM) or fed by prep_bf16_kernel; deep
// (one CTA per SM) or not
void* k_pick_tcv(int bh, bool deep, bool fused) {
    if (fused) return deep ? pick_tcf_v<true>(bh) : pick_tcf_v<false>(bh);
    return deep ? pick_tc_v<true>(bh) : pick_tc_v<false>(bh);
}

void* k_pick_prep_bf16() { return reinterpret_cast<void*>(&prep_bf16_kernel<__nv_bfloat16>); }

cudaError_t k_take_error_tc(unsigned* code, unsigned* info) { return take_unit_error(code, info); }

// Self-test of the bounded wait (site 90): thread 0 waits, with a limit of
// limit_ns, on an mbarrier of one arrival that it completes itself only when
// `signal` is set.  Unsignalled, the wait must give up after limit_ns, set
// the error word, record the site and return: the kernel always ends.
__global__ void wait_selftest_kernel(int signal, unsigned long long limit_ns) {
    __shared__ __align__(8) uint64_t bar;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        mbar_init_fence();
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        if (signal) mbar_arrive(&bar);
        mbar_wait(&bar, 0, 90, 0, limit_ns);
    }
}

void* k_pick_wait_selftest() { return reinterpret_cast<void*>(&wait_selftest_kernel); }

#ifdef PIPO_TRACE
cudaError_t k_trace_set_tc(unsigned long long* buf) { return set_unit_trace(buf); }
#endif

}  // namespace pipo
