// CUDA-core GEMV kernels for fp32 weights (a translation unit of its own).
#include "k_gemv_impl.cuh"

namespace pipo {

void* k_pick_gemv_f32(int nb, bool two) { return pick_gemv_t<float>(nb, two); }
void* k_pick_stream_f32(int nb, int ru, bool rows) { return pick_stream_t<float>(nb, ru, rows); }

#ifdef PIPO_TRACE
cudaError_t k_trace_set_gemv_f32(unsigned long long* buf) { return set_unit_trace(buf); }
#endif

}  // namespace pipo
