// Kernel entry points of the library's kernel translation units, as untyped
// launch handles for cudaLaunchKernelExC and the function-attribute and
// occupancy queries of the host code (pipo_capi.cu).  The kernels are
// compiled in several units so that the build runs them in parallel; each
// unit keeps its own device error word, read and cleared through its
// take_error function.
#pragma once

#include <cuda_runtime.h>

namespace pipo {

// k_gemv_bf16.cu / k_gemv_f32.cu: the CUDA-core GEMVs of one weight type
void* k_pick_gemv_bf16(int nb, bool two);           // gemv_kernel<bf16, nb, two>
void* k_pick_gemv_f32(int nb, bool two);
void* k_pick_stream_bf16(int nb, int ru, bool rows);  // gemv_rows_kernel (rows) / gemv_stream_kernel
void* k_pick_stream_f32(int nb, int ru, bool rows);

// k_tc.cu: the tcgen05 projections
void* k_pick_tcv(int bh, bool deep, bool fused);    // gemm_tcf_kernel (fused) / gemm_tc_kernel
void* k_pick_prep_bf16();                           // prep_bf16_kernel<bf16>
cudaError_t k_take_error_tc(unsigned* code, unsigned* info);
void* k_pick_wait_selftest();                       // wait_selftest_kernel (reports through k_take_error_tc)

// k_attn.cu: attention and RoPE / append kernels
void* k_pick_attn_decode(bool bf, int DH, int G);   // attn_decode_kernel
void* k_pick_attn_cluster(bool bf, int DH, int G);  // attn_cluster_kernel
void* k_pick_attn_flat(bool bf, int DH, int G);     // attn_cluster_kernel, unclustered (global merge)
void* k_pick_attn_mma(int G, bool deep);            // attn_mma_kernel (deep: the kMmaDeepStages ring)
void* k_pick_attn_mma_flat(int G);                  // attn_mma_kernel, unclustered (global merge)
void* k_pick_attn_prefill(int G);                   // attn_prefill_kernel
void* k_pick_rope_append(bool bf, int DH);          // rope_append_kernel
void* k_pick_append_rows(bool bf, int DH);          // append_rows_kernel
cudaError_t k_take_error_attn(unsigned* code, unsigned* info);

#ifdef PIPO_TRACE
// measurement build only: point each unit's timeline buffer at `buf` (or nullptr)
cudaError_t k_trace_set_gemv_bf16(unsigned long long* buf);
cudaError_t k_trace_set_gemv_f32(unsigned long long* buf);
cudaError_t k_trace_set_tc(unsigned long long* buf);
cudaError_t k_trace_set_attn(unsigned long long* buf);
#endif

}  // namespace pipo
