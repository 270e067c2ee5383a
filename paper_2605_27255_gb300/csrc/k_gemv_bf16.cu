// CUDA-core GEMV kernels for bf16 weights (a translation unit of its own).
#include "k_gemv_impl.cuh"

namespace pipo {

void* k_pick_gemv_bf16(int nb, bool two) { return pick_gemv_t<__nv_bfloat16>(nb, two); }
void* k_pick_stream_bf16(int nb, int ru, bool rows) { return pick_stream_t<__nv_bfloat16>(nb, ru, rows); }

#ifdef PIPO_TRACE
cudaError_t k_trace_set_gemv_bf16(unsigned long long* buf) { return set_unit_trace(buf); }
#endif

}  // namespace pipo
