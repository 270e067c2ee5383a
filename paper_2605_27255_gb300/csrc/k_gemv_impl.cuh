// Launch handles of the CUDA-core GEMV kernels of one weight type T (included
// by k_gemv_bf16.cu and k_gemv_f32.cu).
#pragma once

#include "gemv_stream.cuh"
#include "kernel_tables.h"
#include "kernels.cuh"

namespace pipo {

constexpr int kStreamDepth = 4;  // chunks per register batch (two batches in flight)

template <typename T, int NB, bool TWO>
void* gemv_fn() { return reinterpret_cast<void*>(&gemv_kernel<T, NB, TWO>); }

template <typename T>
void* pick_gemv_t(int nb, bool two) {
    switch (nb) {
        case 1: return two ? gemv_fn<T, 1, true>() : gemv_fn<T, 1, false>();
        case 2: return two ? gemv_fn<T, 2, true>() : gemv_fn<T, 2, false>();
        case 4: return two ? gemv_fn<T, 4, true>() : gemv_fn<T, 4, false>();
        default: return two ? gemv_fn<T, 8, true>() : gemv_fn<T, 8, false>();
    }
}

template <typename T, int NB, int RU>
void* stream_fn(bool rows) {
    return rows ? reinterpret_cast<void*>(&gemv_rows_kernel<T, NB, RU, kStreamDepth>)
                : reinterpret_cast<void*>(&gemv_stream_kernel<T, NB, RU, kStreamDepth>);
}

// rows: every weight row is a whole number of 512-byte chunks (fast kernel)
template <typename T>
void* pick_stream_t(int nb, int ru, bool rows) {
    switch (nb) {
        case 1: return ru == 2 ? stream_fn<T, 1, 2>(rows) : stream_fn<T, 1, 1>(rows);
        case 2: return ru == 2 ? stream_fn<T, 2, 2>(rows) : stream_fn<T, 2, 1>(rows);
        default: return ru == 2 ? stream_fn<T, 4, 2>(rows) : stream_fn<T, 4, 1>(rows);
    }
}

}  // namespace pipo
