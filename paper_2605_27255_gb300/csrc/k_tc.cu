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

}  // namespace pipo
