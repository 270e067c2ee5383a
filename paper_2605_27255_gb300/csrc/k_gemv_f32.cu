// CUDA-core GEMV kernels for fp32 weights (a translation unit of its own).
#include "k_gemv_impl.cuh"

namespace pipo {

void* k_pick_gemv_f32(int nb, bool two) { return pick_gemv_t<float>(nb, two); }
void* k_pick_tma_f32(int nb, int ru) { return pick_tma_t<float>(nb, ru); }
void* k_pick_stream_f32(int nb, int ru, bool rows) { return pick_stream_t<float>(nb, ru, rows); }
cudaError_t k_take_error_gemv_f32(unsigned* code, unsigned* info) { return take_unit_error(code, info); }

}  // namespace pipo
