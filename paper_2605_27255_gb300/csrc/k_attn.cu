// Attention kernels and the RoPE / KV append kernels (a translation unit of
// its own).
#include "attn_cluster.cuh"
#include "attn_mma.cuh"
#include "attn_prefill.cuh"
#include "kernel_tables.h"
#include "kernels.cuh"

namespace pipo {

namespace {

using bf16 = __nv_bfloat16;

template <typename T, int DH, int G>
void* attn_fn() { return reinterpret_cast<void*>(&attn_decode_kernel<T, DH, G>); }

template <typename T, int DH>
void* attn_pick_g(int G) {
    switch (G) {
        case 1: return attn_fn<T, DH, 1>();
        case 2: return attn_fn<T, DH, 2>();
        case 4: return attn_fn<T, DH, 4>();
        case 8: return attn_fn<T, DH, 8>();
        default: return nullptr;
    }
}

template <typename T, int DH, int G, bool FLAT>
void* attnc_fn() { return reinterpret_cast<void*>(&attn_cluster_kernel<T, DH, G, FLAT>); }

template <typename T, int DH, bool FLAT = false>
void* attnc_pick_g(int G) {
    switch (G) {
        case 1: return attnc_fn<T, DH, 1, FLAT>();
        case 2: return attnc_fn<T, DH, 2, FLAT>();
        case 4: return attnc_fn<T, DH, 4, FLAT>();
        case 8: return attnc_fn<T, DH, 8, FLAT>();
        default: return nullptr;
    }
}

}  // namespace

// the unclustered split-KV attention (with rope_append_kernel before it)
void* k_pick_attn_decode(bool bf, int DH, int G) {
    if (DH == 64) return bf ? attn_pick_g<bf16, 64>(G) : attn_pick_g<float, 64>(G);
    if (DH == 128) return bf ? attn_pick_g<bf16, 128>(G) : attn_pick_g<float, 128>(G);
    return nullptr;
}

// one kernel for every cluster size (read from the cluster at run time)
void* k_pick_attn_cluster(bool bf, int DH, int G) {
    if (DH == 64) return bf ? attnc_pick_g<bf16, 64>(G) : attnc_pick_g<float, 64>(G);
    if (DH == 128) return bf ? attnc_pick_g<bf16, 128>(G) : attnc_pick_g<float, 128>(G);
    return nullptr;
}

// the same attention without a cluster: any split count, merged through global scratch
void* k_pick_attn_flat(bool bf, int DH, int G) {
    if (DH == 64) return bf ? attnc_pick_g<bf16, 64, true>(G) : attnc_pick_g<float, 64, true>(G);
    if (DH == 128) return bf ? attnc_pick_g<bf16, 128, true>(G) : attnc_pick_g<float, 128, true>(G);
    return nullptr;
}

// tensor-core attention (bf16 cache, d_h = 128, 1, 2 or 4 query heads per
// kv head); deep: the kMmaDeepStages ring
void* k_pick_attn_mma(int G, bool deep) {
    switch (G) {
        case 1: return deep ? reinterpret_cast<void*>(&attn_mma_kernel<1, false, kMmaDeepStages>)
                            : reinterpret_cast<void*>(&attn_mma_kernel<1>);
        case 2: return deep ? reinterpret_cast<void*>(&attn_mma_kernel<2, false, kMmaDeepStages>)
                            : reinterpret_cast<void*>(&attn_mma_kernel<2>);
        case 4: return deep ? reinterpret_cast<void*>(&attn_mma_kernel<4, false, kMmaDeepStages>)
                            : reinterpret_cast<void*>(&attn_mma_kernel<4>);
        default: return nullptr;
    }
}

// the same without clusters, split partials merged through global memory
void* k_pick_attn_mma_flat(int G) {
    switch (G) {
        case 1: return reinterpret_cast<void*>(&attn_mma_kernel<1, true>);
        case 2: return reinterpret_cast<void*>(&attn_mma_kernel<2, true>);
        case 4: return reinterpret_cast<void*>(&attn_mma_kernel<4, true>);
        default: return nullptr;
    }
}

// causal tile attention of prefill chunks (same cache and head constraints)
void* k_pick_attn_prefill(int G) {
    switch (G) {
        case 1: return reinterpret_cast<void*>(&attn_prefill_kernel<1>);
        case 2: return reinterpret_cast<void*>(&attn_prefill_kernel<2>);
        case 4: return reinterpret_cast<void*>(&attn_prefill_kernel<4>);
        default: return nullptr;
    }
}

void* k_pick_rope_append(bool bf, int DH) {
    if (DH == 64) return bf ? (void*)&rope_append_kernel<bf16, 64> : (void*)&rope_append_kernel<float, 64>;
    if (DH == 128) return bf ? (void*)&rope_append_kernel<bf16, 128> : (void*)&rope_append_kernel<float, 128>;
    return nullptr;
}

void* k_pick_append_rows(bool bf, int DH) {
    if (DH == 64) return bf ? (void*)&append_rows_kernel<bf16, 64> : (void*)&append_rows_kernel<float, 64>;
    if (DH == 128) return bf ? (void*)&append_rows_kernel<bf16, 128> : (void*)&append_rows_kernel<float, 128>;
    return nullptr;
}

cudaError_t k_take_error_attn(unsigned* code, unsigned* info) { return take_unit_error(code, info); }

#ifdef PIPO_TRACE
cudaError_t k_trace_set_attn(unsigned long long* buf) { return set_unit_trace(buf); }
#endif

}  // namespace pipo
