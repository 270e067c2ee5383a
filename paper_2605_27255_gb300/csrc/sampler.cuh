// The paper's evaluation sampler on the GPU (Sec. 4: temperature, top-k,
// top-p, repetition penalty), run after an LM-head launch has written the
// head's fp32 logits.  One CTA per sequence:
//   1. every thread scans a strided share of the V logits, applies the
//      repetition penalty to ids present in the sequence's token history
//      (a bitmap: l / r if l > 0, else l * r) and the temperature, and keeps
//      its own best kSampMaxK (value, id) pairs in registers (sorted by value,
//      ties to the lower id);
//   2. each warp merges its 32 lanes' lists into the warp's best k;
//   3. warp 0 merges the warp lists into the best k;
//   4. thread 0 takes the shortest prefix of those k whose softmax mass
//      reaches p and picks the first id whose cumulative renormalised mass
//      exceeds u * (prefix mass), u being this position's uniform draw.
// The pick is written as the head's packed argmax key (the MTP input gather
// and the acceptance read the token from there), and the backbone head's
// pick joins the history bitmap before the draft head samples.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "kernels.cuh"

namespace pipo {

constexpr int kSampMaxK = 32;                // top-k supported on the GPU: 1 .. 32
constexpr int kSampThreads = 256;
constexpr int kSampWarps = kSampThreads / 32;

// (v, id) ranks before (w, jd): larger value first, then the lower id
__device__ __forceinline__ bool samp_before(float v, int id, float w, int jd) {
    return v > w || (v == w && id < jd);
}

struct SampParams {
    const float* logits;      // [B][ld] fp32 logits of this head
    int ld;
    int V;
    const uint32_t* presence; // [B][W] history bitmap
    uint32_t* presence_add;   // backbone head: add the pick to the bitmap (else nullptr)
    int W;
    float inv_T, top_p, rep;
    int top_k;                // 1 .. kSampMaxK
    const float* u;           // [n_u][u_rows][2] draws
    const int32_t* u_step;    // index of this position's draws (mod n_u)
    int n_u, u_rows, head;    // head 0: backbone, 1: draft
    unsigned long long* am;   // [B] packed argmax keys: the pick is written here
};

__global__ void __launch_bounds__(kSampThreads) sample_kernel(SampParams p) {
    __shared__ float wv[kSampWarps][kSampMaxK];
    __shared__ int wi[kSampWarps][kSampMaxK];
    __shared__ float fv[kSampMaxK];
    __shared__ int fi[kSampMaxK];
    pdl_launch();
    pdl_wait();
    const int b = blockIdx.x, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int k = p.top_k < p.V ? p.top_k : p.V;
    const float* lg = p.logits + (size_t)b * p.ld;
    const uint32_t* pres = p.presence + (size_t)b * p.W;

    // 1. per-thread best kSampMaxK, sorted (compile-time indices: registers)
    float vals[kSampMaxK];
    int ids[kSampMaxK];
#pragma unroll
    for (int j = 0; j < kSampMaxK; ++j) { vals[j] = -INFINITY; ids[j] = 0x7fffffff; }
    for (int i = threadIdx.x; i < p.V; i += kSampThreads) {
        float l = lg[i];
        if ((pres[i >> 5] >> (i & 31)) & 1u) l = l > 0.f ? l / p.rep : l * p.rep;
        const float v = l * p.inv_T;
        if (!samp_before(v, i, vals[kSampMaxK - 1], ids[kSampMaxK - 1])) continue;
        vals[kSampMaxK - 1] = v;
        ids[kSampMaxK - 1] = i;
#pragma unroll
        for (int j = kSampMaxK - 1; j > 0; --j) {
            if (samp_before(vals[j], ids[j], vals[j - 1], ids[j - 1])) {
                const float tv = vals[j]; vals[j] = vals[j - 1]; vals[j - 1] = tv;
                const int ti = ids[j]; ids[j] = ids[j - 1]; ids[j - 1] = ti;
            }
        }
    }

    // 2. warp merge: k rounds of a warp-wide best over the lanes' list heads
    for (int r = 0; r < k; ++r) {
        float bv = vals[0];
        int bi = ids[0];
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) {
            const float ov = __shfl_xor_sync(0xffffffffu, bv, off);
            const int oi = __shfl_xor_sync(0xffffffffu, bi, off);
            if (samp_before(ov, oi, bv, bi)) { bv = ov; bi = oi; }
        }
        if (ids[0] == bi && vals[0] == bv) {  // the owner (ids are unique) drops its head
#pragma unroll
            for (int j = 0; j < kSampMaxK - 1; ++j) { vals[j] = vals[j + 1]; ids[j] = ids[j + 1]; }
            vals[kSampMaxK - 1] = -INFINITY;
            ids[kSampMaxK - 1] = 0x7fffffff;
        }
        if (lane == 0) { wv[warp][r] = bv; wi[warp][r] = bi; }
    }
    __syncthreads();

    // 3. warp 0 merges the warp lists (lane w < kSampWarps reads list w)
    if (warp == 0) {
        int pos = 0;
        for (int r = 0; r < k; ++r) {
            float bv = -INFINITY;
            int bi = 0x7fffffff;
            if (lane < kSampWarps && pos < k) { bv = wv[lane][pos]; bi = wi[lane][pos]; }
            const float mv = bv;
            const int mi = bi;
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) {
                const float ov = __shfl_xor_sync(0xffffffffu, bv, off);
                const int oi = __shfl_xor_sync(0xffffffffu, bi, off);
                if (samp_before(ov, oi, bv, bi)) { bv = ov; bi = oi; }
            }
            if (lane < kSampWarps && pos < k && mi == bi && mv == bv) ++pos;
            if (lane == 0) { fv[r] = bv; fi[r] = bi; }
        }
    }
    __syncthreads();

    // 4. nucleus and the draw
    if (threadIdx.x == 0) {
        float e[kSampMaxK];
        float Z = 0.f;
        for (int i = 0; i < k; ++i) { e[i] = expf(fv[i] - fv[0]); Z += e[i]; }
        int np = k;
        float cum = 0.f;
        for (int i = 0; i < k; ++i) {
            cum += e[i];
            if (cum / Z >= p.top_p) { np = i + 1; break; }
        }
        float Zp = 0.f;
        for (int i = 0; i < np; ++i) Zp += e[i];
        const int t = *p.u_step % p.n_u;
        const float u = p.u[((size_t)t * p.u_rows + b) * 2 + p.head];
        const float target = u * Zp;
        int pick = fi[np - 1];
        cum = 0.f;
        for (int i = 0; i < np; ++i) {
            if (cum + e[i] > target) { pick = fi[i]; break; }
            cum += e[i];
        }
        p.am[b] = argmax_key(0.f, pick);
        if (p.presence_add) atomicOr(p.presence_add + (size_t)b * p.W + (pick >> 5), 1u << (pick & 31));
    }
}

}  // namespace pipo
