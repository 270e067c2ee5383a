// The persistent step kernel (a translation unit of its own).
#include "kernel_tables.h"
#include "megakernel.cuh"

namespace pipo {

namespace {

template <typename T, int NB, int DH, int G>
void* mk_fn() { return reinterpret_cast<void*>(&step_kernel<T, NB, DH, G>); }

}  // namespace

void* k_pick_step_kernel(bool bf, int nb, int DH, int G) {
    using bf16 = __nv_bfloat16;
    if (bf && DH == 128 && G == 4)
        return nb == 1 ? mk_fn<bf16, 1, 128, 4>() : nb == 2 ? mk_fn<bf16, 2, 128, 4>() : mk_fn<bf16, 4, 128, 4>();
    if (!bf && DH == 64 && G == 2)
        return nb == 1 ? mk_fn<float, 1, 64, 2>() : nb == 2 ? mk_fn<float, 2, 64, 2>() : mk_fn<float, 4, 64, 2>();
    return nullptr;
}

cudaError_t k_take_error_mk(unsigned* code, unsigned* info) { return take_unit_error(code, info); }

}  // namespace pipo
