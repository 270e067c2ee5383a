// Weight-streaming GEMV for small batches (B <= 4 per pass) on sm_103a.
//
// y[b, u] = epi( sum_k W[u*RU + r, k] * xin[b, k] ),  r < RU (RU = 2 pairs the
// gate and up rows of SwiGLU, interleaved at upload).
//
// Work split: CTA c owns a contiguous range of units (balanced to +-1 unit);
// inside the CTA the flat range of 512-byte chunks (32 lanes x 16 bytes) is
// split evenly over the warps, across unit boundaries, so every warp streams
// the same number of bytes.  Each lane keeps two batches of kU 128-bit loads
// (one in flight while the other is consumed): with 16 warps one CTA per SM
// holds 32-64 KB of weights in flight.
// A unit that lies inside one warp's range is finished by that warp; a unit
// split between warps is finished after a block barrier by the warp holding
// its last chunk, adding the partials in warp order: the result does not
// depend on timing (deterministic), and no split-K atomics are used.
//
// Programmatic dependent launch: the first 2*kU chunks are loaded before
// griddepcontrol.wait, so weight streaming overlaps the previous kernel's tail.
#pragma once

#include "kernels.cuh"
#include "tma.cuh"

namespace pipo {

#ifndef PIPO_STREAM_THREADS
#define PIPO_STREAM_THREADS 768
#endif
#ifndef PIPO_STREAM_CTAS_PER_SM
#define PIPO_STREAM_CTAS_PER_SM 1
#endif
constexpr int kStreamThreads = PIPO_STREAM_THREADS;
constexpr int kStreamCtasPerSm = PIPO_STREAM_CTAS_PER_SM;  // CTAs per SM of one GEMV launch
constexpr int kStreamWarps = kStreamThreads / 32;

template <typename T> struct Chunk16;  // 16 bytes of weights
template <> struct Chunk16<__nv_bfloat16> {
    static constexpr int kElems = 8;
    __device__ __forceinline__ static void to_float(const uint4& v, float* f) {
        f[0] = bf_lo(v.x); f[1] = bf_hi(v.x); f[2] = bf_lo(v.y); f[3] = bf_hi(v.y);
        f[4] = bf_lo(v.z); f[5] = bf_hi(v.z); f[6] = bf_lo(v.w); f[7] = bf_hi(v.w);
    }
};
template <> struct Chunk16<float> {
    static constexpr int kElems = 4;
    __device__ __forceinline__ static void to_float(const uint4& v, float* f) {
        f[0] = __uint_as_float(v.x); f[1] = __uint_as_float(v.y); f[2] = __uint_as_float(v.z); f[3] = __uint_as_float(v.w);
    }
};

// Stage the (gathered, normalised) input of sequences [b0, b0+nb) in smem.
template <typename T, int NB>
__device__ __forceinline__ void stage_input(const GemvParams& p, float* xs, int b0, int nb) {
    __shared__ float rstd_s[NB][2];
    const int K = p.K;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int bb = 0; bb < NB; ++bb) {
        const int b = b0 + bb;
        int koff = 0;
        for (int s = 0; s < p.nseg; ++s) {
            const Seg& sg = p.seg[s];
            int tok = 0;
            if (!sg.src && bb < nb) tok = sg.tok_am ? argmax_row(sg.tok_am[b]) : sg.tok[(size_t)b * sg.tok_ld];
            for (int k = threadIdx.x; k < sg.K; k += blockDim.x) {
                float v = 0.f;
                if (bb < nb) {
                    if (sg.src) v = sg.src[(size_t)b * sg.ld + k];
                    else v = (tok < 0) ? ldw<T>(sg.pad, k) : ldw<T>(sg.table, (size_t)tok * sg.K + k);
                }
                xs[bb * K + koff + k] = v;
            }
            koff += sg.K;
        }
    }
    __syncthreads();
    const bool any_norm = p.seg[0].gamma || (p.nseg > 1 && p.seg[1].gamma);
    if (!any_norm) return;
    const int ngrp = p.joint_norm ? 1 : p.nseg;
    for (int q = warp; q < NB * ngrp; q += blockDim.x / 32) {
        const int bb = q / ngrp, s = q % ngrp;
        const int k0 = (s == 0) ? 0 : p.seg[0].K;
        const int len = p.joint_norm ? K : p.seg[s].K;
        float ss = 0.f;
        for (int k = lane; k < len; k += 32) {
            const float v = xs[bb * K + k0 + k];
            ss += v * v;
        }
        ss = warp_sum(ss);
        if (lane == 0) rstd_s[bb][s] = 1.0f / sqrtf(ss / (float)len + p.eps);
    }
    __syncthreads();
    for (int bb = 0; bb < NB; ++bb)
        for (int k = threadIdx.x; k < K; k += blockDim.x) {
            const int s = (p.joint_norm || k < p.seg[0].K) ? 0 : 1;
            const Seg& sg = p.seg[s];
            if (!sg.gamma) continue;
            const int kk = (p.joint_norm || s == 0) ? k : k - p.seg[0].K;
            xs[bb * K + k] *= rstd_s[bb][s] * ldw<T>(sg.gamma, kk);
        }
    __syncthreads();
}

// Epilogue of one finished unit u with sums a[r][bb] (lane-uniform).
template <typename T, int RU, int NB>
__device__ __forceinline__ void unit_epilogue(const GemvParams& p, int u, const float (&a)[RU][NB], int b0, int nb,
                                              float (&best_v)[NB], int (&best_r)[NB],
                                              const float* ypre = nullptr) {
    const int lane = threadIdx.x & 31;
    if (p.epi == EPI_ARGMAX) {
#pragma unroll
        for (int bb = 0; bb < NB; ++bb)
            if (a[0][bb] > best_v[bb] || (a[0][bb] == best_v[bb] && u < best_r[bb])) {
                best_v[bb] = a[0][bb];
                best_r[bb] = u;
            }
        if (p.dbg) {
#pragma unroll
            for (int bb = 0; bb < NB; ++bb)
                if (bb == lane && bb < nb) p.dbg[(size_t)(b0 + bb) * p.ld_dbg + u] = a[0][bb];
        }
        return;
    }
#pragma unroll
    for (int bb = 0; bb < NB; ++bb) {
        if (bb != lane || bb >= nb) continue;
        float* yp = p.y + (size_t)(b0 + bb) * p.ldy + u;
        const float s = a[0][bb];
        switch (p.epi) {
            case EPI_STORE: *yp = s; break;
            case EPI_BIAS: *yp = s + ldw<T>(p.bias, u); break;
            case EPI_SILU: *yp = silu(s); break;
            case EPI_RESADD: *yp = (ypre ? ypre[bb] : *yp) + s; break;
            case EPI_SWIGLU: *yp = silu(s) * a[RU - 1][bb]; break;
            default: break;
        }
    }
}

template <typename T, int NB, int RU, int kU>
__global__ void __launch_bounds__(kStreamThreads) gemv_stream_kernel(GemvParams p) {
    extern __shared__ float4 smem4[];
    float* xs = reinterpret_cast<float*>(smem4);  // [NB][K]
    __shared__ int head_unit[kStreamWarps], tail_unit[kStreamWarps], head_fin[kStreamWarps];
    __shared__ float head_val[kStreamWarps][RU][NB], tail_val[kStreamWarps][RU][NB];
    __shared__ float red_v[kStreamWarps][NB];
    __shared__ int red_r[kStreamWarps][NB];
    constexpr int EPC = Chunk16<T>::kElems;  // elements per lane per chunk

    pdl_launch();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int K = p.K;
    const int row_bytes = K * (int)sizeof(T);
    const int cpr = (row_bytes + 511) / 512;  // chunks per row
    const int cpu = cpr * RU;                 // chunks per unit
    const int G = gridDim.x;
    const int u0 = (int)((long long)blockIdx.x * p.N / G);
    const int u1 = (int)((long long)(blockIdx.x + 1) * p.N / G);
    const int C = (u1 - u0) * cpu;            // chunks of this CTA (< 2^31)
    const int c0 = (int)((long long)warp * C / kStreamWarps);
    const int c1 = (int)((long long)(warp + 1) * C / kStreamWarps);
    const char* Wb = static_cast<const char*>(p.W) + (size_t)u0 * RU * row_bytes + lane * 16;
    const char* Wb0 = static_cast<const char*>(p.W) + (lane * 16) % row_bytes;  // always a valid address
    const int lane_off = lane * 16;

    for (int b0 = 0; b0 < p.B; b0 += NB) {
        const int nb = min(NB, p.B - b0);
        // Two register batches of kU chunks: one is consumed while the other's
        // loads are in flight.  Loads past the warp's range are skipped; a lane
        // past a ragged row end reads a valid address instead (never used), so
        // no select waits on a load result.
        int lc = c0, lrow = c0 / cpr, lj = c0 - (c0 / cpr) * cpr;
        uint4 bufA[kU], bufB[kU];
        auto load_batch = [&](uint4 (&buf)[kU]) {
#pragma unroll
            for (int u = 0; u < kU; ++u) {
                if (lc < c1) {
                    const bool ok = lj * 512 + lane_off < row_bytes;
                    buf[u] = ldg_stream(ok ? Wb + (size_t)lrow * row_bytes + lj * 512 : Wb0);
                }
                ++lc;
                if (++lj == cpr) { lj = 0; ++lrow; }
            }
        };
        load_batch(bufA);
        load_batch(bufB);
        if (b0 == 0) {
            pdl_wait();
            if (p.zero_ptr && blockIdx.x == 0)
                for (int i = threadIdx.x; i < p.zero_n; i += blockDim.x) p.zero_ptr[i] = 0ull;
        }
        __syncthreads();
        stage_input<T, NB>(p, xs, b0, nb);

        float best_v[NB];
        int best_r[NB];
#pragma unroll
        for (int bb = 0; bb < NB; ++bb) { best_v[bb] = -INFINITY; best_r[bb] = 0x7fffffff; }
        float acc[RU][NB];
#pragma unroll
        for (int r = 0; r < RU; ++r)
#pragma unroll
            for (int bb = 0; bb < NB; ++bb) acc[r][bb] = 0.f;
        if (lane == 0) { head_fin[warp] = 0; head_unit[warp] = -1; tail_unit[warp] = -1; }

        // consume cursor (cc = chunk, crow/cj = row and chunk in row)
        int cc = c0, crow = c0 / cpr, cj = c0 - (c0 / cpr) * cpr;
        int cur_unit = (c0 < c1) ? crow / RU : -1;
        auto consume_batch = [&](const uint4 (&buf)[kU]) {
#pragma unroll
            for (int u = 0; u < kU; ++u) {
                if (cc < c1) {
                    const int unit = crow / RU;
                    if (unit != cur_unit) {
                        // flush the finished unit cur_unit
                        float a[RU][NB];
#pragma unroll
                        for (int r = 0; r < RU; ++r)
#pragma unroll
                            for (int bb = 0; bb < NB; ++bb) { a[r][bb] = warp_sum(acc[r][bb]); acc[r][bb] = 0.f; }
                        if (cur_unit * cpu >= c0) {
                            unit_epilogue<T, RU, NB>(p, u0 + cur_unit, a, b0, nb, best_v, best_r);
                        } else if (lane == 0) {
                            head_unit[warp] = cur_unit;
                            head_fin[warp] = 1;
#pragma unroll
                            for (int r = 0; r < RU; ++r)
#pragma unroll
                                for (int bb = 0; bb < NB; ++bb) head_val[warp][r][bb] = a[r][bb];
                        }
                        cur_unit = unit;
                    }
                    const int r = crow - unit * RU;
                    const int k = cj * (512 / (int)sizeof(T)) + lane * EPC;
                    if (k < K) {
                        float w[EPC];
                        Chunk16<T>::to_float(buf[u], w);
#pragma unroll
                        for (int bb = 0; bb < NB; ++bb) {
                            const float* xp = xs + bb * K + k;
                            float s = 0.f;
#pragma unroll
                            for (int e = 0; e < EPC; e += 4) {
                                const float4 xv = *reinterpret_cast<const float4*>(xp + e);
                                s += w[e] * xv.x + w[e + 1] * xv.y + w[e + 2] * xv.z + w[e + 3] * xv.w;
                            }
#pragma unroll
                            for (int rr = 0; rr < RU; ++rr)
                                if (rr == r) acc[rr][bb] += s;
                        }
                    }
                    ++cc;
                    if (++cj == cpr) { cj = 0; ++crow; }
                }
            }
        };
        while (cc < c1) {
            consume_batch(bufA);
            load_batch(bufA);
            if (cc >= c1) break;
            consume_batch(bufB);
            load_batch(bufB);
        }
        // the warp's last unit
        if (c0 < c1) {
            float a[RU][NB];
#pragma unroll
            for (int r = 0; r < RU; ++r)
#pragma unroll
                for (int bb = 0; bb < NB; ++bb) a[r][bb] = warp_sum(acc[r][bb]);
            const bool started_here = cur_unit * cpu >= c0;
            const bool ends_here = (cur_unit + 1) * cpu <= c1;
            if (started_here && ends_here) {
                unit_epilogue<T, RU, NB>(p, u0 + cur_unit, a, b0, nb, best_v, best_r);
            } else if (lane == 0) {
                if (started_here) {
                    tail_unit[warp] = cur_unit;
#pragma unroll
                    for (int r = 0; r < RU; ++r)
#pragma unroll
                        for (int bb = 0; bb < NB; ++bb) tail_val[warp][r][bb] = a[r][bb];
                } else {
                    head_unit[warp] = cur_unit;
                    head_fin[warp] = ends_here ? 1 : 0;
#pragma unroll
                    for (int r = 0; r < RU; ++r)
#pragma unroll
                        for (int bb = 0; bb < NB; ++bb) head_val[warp][r][bb] = a[r][bb];
                }
            }
        }
        __syncthreads();
        // units split between warps: the warp holding the last chunk adds the
        // partials in warp order (start warp's tail, middle warps, its own)
        if (head_fin[warp] && head_unit[warp] >= 0) {
            const int unit = head_unit[warp];
            int ws = warp - 1;
            while (ws >= 0 && tail_unit[ws] != unit) --ws;
            float a[RU][NB];
#pragma unroll
            for (int r = 0; r < RU; ++r)
#pragma unroll
                for (int bb = 0; bb < NB; ++bb) {
                    float s = (ws >= 0) ? tail_val[ws][r][bb] : 0.f;
                    for (int v = (ws >= 0 ? ws + 1 : 0); v <= warp; ++v)
                        if (head_unit[v] == unit) s += head_val[v][r][bb];
                    a[r][bb] = s;
                }
            unit_epilogue<T, RU, NB>(p, u0 + unit, a, b0, nb, best_v, best_r);
        }
        if (p.epi == EPI_ARGMAX) {
            if (lane == 0)
#pragma unroll
                for (int bb = 0; bb < NB; ++bb) { red_v[warp][bb] = best_v[bb]; red_r[warp][bb] = best_r[bb]; }
            __syncthreads();
            if (threadIdx.x < nb) {
                const int bb = threadIdx.x;
                float bv = -INFINITY;
                int br = 0x7fffffff;
                for (int w = 0; w < kStreamWarps; ++w)
                    if (red_r[w][bb] != 0x7fffffff && (red_v[w][bb] > bv || (red_v[w][bb] == bv && red_r[w][bb] < br))) {
                        bv = red_v[w][bb];
                        br = red_r[w][bb];
                    }
                if (br != 0x7fffffff) atomicMax(p.am + b0 + bb, argmax_key(bv, br));
            }
        }
        __syncthreads();
    }
}

// Fast path for rows of a whole number of 512-byte chunks (every model shape
// of the benchmark).  The CTA's weights are one contiguous byte range, so the
// load address of a warp's chunk f is base + 512 f: loads need no row
// arithmetic, and the row bookkeeping (warp reduction, epilogue) runs once per
// row.  x is staged in a bank-conflict-free layout: for 16-bit weights the two
// float4 halves of each lane's 8 elements live in two separate K/2 planes.
template <typename T>
__device__ __forceinline__ int xs_index(int k, int K) {
    if (sizeof(T) == 2) return (k & 4) * (K / 8) + (k >> 3) * 4 + (k & 3);  // plane (k&4)/4, group k/8
    return k;
}

template <typename T, int NB>
__device__ __forceinline__ void stage_input_split(const GemvParams& p, float* xs, int b0, int nb) {
    // stage in natural order into the split layout: element k of sequence bb at
    // xs[bb*K + xs_index(k)]
    __shared__ float rstd_s[NB][2];
    const int K = p.K;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int bb = 0; bb < NB; ++bb) {
        const int b = b0 + bb;
        int koff = 0;
        for (int s = 0; s < p.nseg; ++s) {
            const Seg& sg = p.seg[s];
            int tok = 0;
            if (!sg.src && bb < nb) tok = sg.tok_am ? argmax_row(sg.tok_am[b]) : sg.tok[(size_t)b * sg.tok_ld];
            for (int k = threadIdx.x; k < sg.K; k += blockDim.x) {
                float v = 0.f;
                if (bb < nb) {
                    if (sg.src) v = sg.src[(size_t)b * sg.ld + k];
                    else v = (tok < 0) ? ldw<T>(sg.pad, k) : ldw<T>(sg.table, (size_t)tok * sg.K + k);
                }
                xs[bb * K + xs_index<T>(koff + k, K)] = v;
            }
            koff += sg.K;
        }
    }
    __syncthreads();
    const bool any_norm = p.seg[0].gamma || (p.nseg > 1 && p.seg[1].gamma);
    if (!any_norm) return;
    const int ngrp = p.joint_norm ? 1 : p.nseg;
    for (int q = warp; q < NB * ngrp; q += blockDim.x / 32) {
        const int bb = q / ngrp, s = q % ngrp;
        const int k0 = (s == 0) ? 0 : p.seg[0].K;
        const int len = p.joint_norm ? K : p.seg[s].K;
        float ss = 0.f;
        for (int k = lane; k < len; k += 32) {
            const float v = xs[bb * K + xs_index<T>(k0 + k, K)];
            ss += v * v;
        }
        ss = warp_sum(ss);
        if (lane == 0) rstd_s[bb][s] = 1.0f / sqrtf(ss / (float)len + p.eps);
    }
    __syncthreads();
    for (int bb = 0; bb < NB; ++bb)
        for (int k = threadIdx.x; k < K; k += blockDim.x) {
            const int s = (p.joint_norm || k < p.seg[0].K) ? 0 : 1;
            const Seg& sg = p.seg[s];
            if (!sg.gamma) continue;
            const int kk = (p.joint_norm || s == 0) ? k : k - p.seg[0].K;
            xs[bb * K + xs_index<T>(k, K)] *= rstd_s[bb][s] * ldw<T>(sg.gamma, kk);
        }
    __syncthreads();
}

// 4 consecutive elements of a weight-typed vector as floats (16- or 8-byte load)
template <typename T>
__device__ __forceinline__ float4 ld4(const void* base, size_t i) {
    if (sizeof(T) == 4) return *reinterpret_cast<const float4*>(static_cast<const float*>(base) + i);
    const uint2 u = *reinterpret_cast<const uint2*>(static_cast<const __nv_bfloat16*>(base) + i);
    return make_float4(bf_lo(u.x), bf_hi(u.x), bf_lo(u.y), bf_hi(u.y));
}

// Fast staging of the GEMV input in the split layout of gemv_rows: every
// thread owns up to kMaxQ float4 groups of the K inputs, issues all their loads
// (activation or gathered embedding, and the RMSNorm gain) at once, reduces the
// sums of squares over the block, and stores the scaled values: one global
// round trip per sequence instead of one per loop iteration.
template <typename T, int NB, int kThreadsPerBlock>
__device__ __forceinline__ void stage_input_fast(const GemvParams& p, float* xs, int b0, int nb) {
    constexpr int kMaxQ = 4096 / kThreadsPerBlock;  // K <= 16384 inputs
    __shared__ float red_ss[32][2];
    __shared__ float rstd_s[2];
    __shared__ int tok_s[NB][2];
    const int K = p.K, K4 = K / 4, K0q = p.seg[0].K / 4;
    const int tid = threadIdx.x, nt = blockDim.x, warp = tid >> 5, lane = tid & 31;
    const bool norm0 = p.seg[0].gamma != nullptr, norm1 = p.nseg > 1 && p.seg[1].gamma != nullptr;
    // gathered rows: token ids first (one round trip for all sequences)
    if (tid < NB * 2) {
        const int bb = tid >> 1, s = tid & 1;
        int t = 0;
        if (bb < nb && s < p.nseg && !p.seg[s].src) {
            const Seg& sg = p.seg[s];
            t = sg.tok_am ? argmax_row(sg.tok_am[b0 + bb]) : sg.tok[(size_t)(b0 + bb) * sg.tok_ld];
        }
        tok_s[bb][s] = t;
    }
    // gains (shared by every sequence)
    float4 gm[kMaxQ];
#pragma unroll
    for (int i = 0; i < kMaxQ; ++i) {
        const int q = tid + i * nt;
        gm[i] = make_float4(1.f, 1.f, 1.f, 1.f);
        if (q < K4) {
            if (p.joint_norm) {
                if (norm0) gm[i] = ld4<T>(p.seg[0].gamma, (size_t)q * 4);
            } else if (q < K0q) {
                if (norm0) gm[i] = ld4<T>(p.seg[0].gamma, (size_t)q * 4);
            } else if (norm1) {
                gm[i] = ld4<T>(p.seg[1].gamma, (size_t)(q - K0q) * 4);
            }
        }
    }
    __syncthreads();
    for (int bb = 0; bb < NB; ++bb) {
        const int b = b0 + bb;
        float4 v[kMaxQ];
        float ss0 = 0.f, ss1 = 0.f;
#pragma unroll
        for (int i = 0; i < kMaxQ; ++i) {
            const int q = tid + i * nt;
            v[i] = make_float4(0.f, 0.f, 0.f, 0.f);
            if (q < K4 && bb < nb) {
                const int s = q < K0q ? 0 : 1;
                const Seg& sg = p.seg[s];
                const int qq = s == 0 ? q : q - K0q;
                if (sg.src) {
                    v[i] = *reinterpret_cast<const float4*>(sg.src + (size_t)b * sg.ld + (size_t)qq * 4);
                } else {
                    const int t = tok_s[bb][s];
                    v[i] = t < 0 ? ld4<T>(sg.pad, (size_t)qq * 4) : ld4<T>(sg.table, (size_t)t * sg.K + (size_t)qq * 4);
                }
            }
        }
#pragma unroll
        for (int i = 0; i < kMaxQ; ++i) {
            const int q = tid + i * nt;
            const float sq = v[i].x * v[i].x + v[i].y * v[i].y + v[i].z * v[i].z + v[i].w * v[i].w;
            if (p.joint_norm || q < K0q) ss0 += sq; else ss1 += sq;
        }
        if (norm0 || norm1) {
            ss0 = warp_sum(ss0);
            ss1 = warp_sum(ss1);
            if (lane == 0) { red_ss[warp][0] = ss0; red_ss[warp][1] = ss1; }
            __syncthreads();
            if (tid < 2) {
                float t = 0.f;
                for (int w = 0; w < nt / 32; ++w) t += red_ss[w][tid];
                const int len = p.joint_norm ? (tid == 0 ? K : 1) : (tid == 0 ? p.seg[0].K : (p.nseg > 1 ? p.seg[1].K : 1));
                rstd_s[tid] = 1.0f / sqrtf(t / (float)len + p.eps);
            }
            __syncthreads();
        }
        const float r0 = norm0 ? rstd_s[0] : 1.f;
        const float r1 = norm1 ? rstd_s[1] : 1.f;
#pragma unroll
        for (int i = 0; i < kMaxQ; ++i) {
            const int q = tid + i * nt;
            if (q < K4) {
                const float r = (p.joint_norm || q < K0q) ? r0 : r1;
                float4 o = v[i];
                if (norm0 || norm1) {
                    o.x *= r * gm[i].x; o.y *= r * gm[i].y; o.z *= r * gm[i].z; o.w *= r * gm[i].w;
                }
                const int idx = sizeof(T) == 2 ? (q & 1) * (K / 2) + (q >> 1) * 4 : q * 4;
                *reinterpret_cast<float4*>(xs + bb * K + idx) = o;
            }
        }
    }
    __syncthreads();
}

__device__ __forceinline__ void cp_async16(void* smem_dst, const void* gsrc, int src_bytes) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_u32(smem_dst)), "l"(gsrc), "r"(src_bytes)
                 : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
    asm volatile("cp.async.commit_group;\n cp.async.wait_group 0;" ::: "memory");
}

// Register-light staging for the register-ring GEMV: activations and RMSNorm
// gains travel global -> shared with cp.async (no registers held), gathered
// embedding rows (compressor and MTP inputs only) through registers; then one
// block reduction for the norms and one scaling pass in shared memory.
// gsm: K elements of type T for the gains.  Same split layout as stage_input_fast.
// yres (EPI_RESADD, or nullptr): [units][NB] receives y of units [u0, u0 +
// units) of sequences b0 .. b0 + nb - 1, loaded while the input copies fly.
template <typename T, int NB>
__device__ __forceinline__ void stage_input_async(const GemvParams& p, float* xs, T* gsm, int b0, int nb,
                                                  float (*yres)[NB] = nullptr, int u0 = 0, int units = 0) {
    __shared__ float red_ss[32][NB][2];
    __shared__ float rstd_s[NB][2];
    const int K = p.K, K0q = p.seg[0].K / 4;
    const int tid = threadIdx.x, nt = blockDim.x, warp = tid >> 5, lane = tid & 31;
    const bool norm0 = p.seg[0].gamma != nullptr, norm1 = p.nseg > 1 && p.seg[1].gamma != nullptr;
    auto xidx = [&](int q) { return sizeof(T) == 2 ? (q & 1) * (K / 2) + (q >> 1) * 4 : q * 4; };
    // the residual values first: their loads fly with the input copies below
    float yv = 0.f;
    if (yres && tid < units * nb) yv = __ldcg(p.y + (size_t)(b0 + tid % nb) * p.ldy + u0 + tid / nb);
    // gains: raw bytes of each normalised segment into gsm (element k at gsm[k])
    {
        int koff = 0;
        for (int s = 0; s < p.nseg; ++s) {
            const Seg& sg = p.seg[s];
            const int len = p.joint_norm ? K : sg.K;
            const void* gp = sg.gamma;
            if (gp && !(p.joint_norm && s > 0)) {
                const int n16 = len * (int)sizeof(T) / 16;
                for (int i = tid; i < n16; i += nt)
                    cp_async16(reinterpret_cast<char*>(gsm + koff) + 16 * i, static_cast<const char*>(gp) + 16 * i, 16);
            }
            koff += sg.K;
        }
    }
    // activations: 16-byte pieces straight into the split layout (zero-filled past nb)
    for (int bb = 0; bb < NB; ++bb) {
        int qoff = 0;
        for (int s = 0; s < p.nseg; ++s) {
            const Seg& sg = p.seg[s];
            const int nq = sg.K / 4;
            if (sg.src) {
                const float* row = sg.src + (size_t)(b0 + min(bb, nb - 1)) * sg.ld;
                for (int q = tid; q < nq; q += nt)
                    cp_async16(xs + bb * K + xidx(qoff + q), row + 4 * q, bb < nb ? 16 : 0);
            } else {
                const int t = bb < nb ? (sg.tok_am ? argmax_row(sg.tok_am[b0 + bb]) : sg.tok[(size_t)(b0 + bb) * sg.tok_ld])
                                      : 0;
                for (int q = tid; q < nq; q += nt) {
                    float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
                    if (bb < nb) v = t < 0 ? ld4<T>(sg.pad, (size_t)q * 4) : ld4<T>(sg.table, (size_t)t * sg.K + (size_t)q * 4);
                    *reinterpret_cast<float4*>(xs + bb * K + xidx(qoff + q)) = v;
                }
            }
            qoff += nq;
        }
    }
    if (yres && tid < units * nb) yres[tid / nb][tid % nb] = yv;  // units * nb <= the block's threads
    cp_async_wait_all();
    __syncthreads();
    if (!norm0 && !norm1) return;
    // sums of squares per sequence and norm group
    const int K4 = K / 4;
    float ss[NB][2];
#pragma unroll
    for (int bb = 0; bb < NB; ++bb) { ss[bb][0] = 0.f; ss[bb][1] = 0.f; }
    for (int q = tid; q < K4; q += nt) {
        const int gsel = (p.joint_norm || q < K0q) ? 0 : 1;
#pragma unroll
        for (int bb = 0; bb < NB; ++bb) {
            const float4 v = *reinterpret_cast<const float4*>(xs + bb * K + xidx(q));
            const float sq = v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
            if (gsel == 0) ss[bb][0] += sq; else ss[bb][1] += sq;
        }
    }
#pragma unroll
    for (int bb = 0; bb < NB; ++bb) {
        const float a = warp_sum(ss[bb][0]), c = warp_sum(ss[bb][1]);
        if (lane == 0) { red_ss[warp][bb][0] = a; red_ss[warp][bb][1] = c; }
    }
    __syncthreads();
    if (tid < NB * 2) {
        const int bb = tid >> 1, g = tid & 1;
        float t = 0.f;
        for (int w = 0; w < nt / 32; ++w) t += red_ss[w][bb][g];
        const int len = p.joint_norm ? K : (g == 0 ? p.seg[0].K : (p.nseg > 1 ? p.seg[1].K : 1));
        rstd_s[bb][g] = 1.0f / sqrtf(t / (float)len + p.eps);
    }
    __syncthreads();
    for (int q = tid; q < K4; q += nt) {
        const int gsel = (p.joint_norm || q < K0q) ? 0 : 1;
        if (!(gsel == 0 ? norm0 : norm1)) continue;
        const float4 gm = ld4<T>(gsm, (size_t)q * 4);
#pragma unroll
        for (int bb = 0; bb < NB; ++bb) {
            float4* xp = reinterpret_cast<float4*>(xs + bb * K + xidx(q));
            const float r = rstd_s[bb][gsel];
            float4 v = *xp;
            v.x *= r * gm.x; v.y *= r * gm.y; v.z *= r * gm.z; v.w *= r * gm.w;
            *xp = v;
        }
    }
    __syncthreads();
}

template <typename T, int NB, int RU, int kU>
__global__ void __launch_bounds__(kStreamThreads) gemv_rows_kernel(GemvParams p) {
    extern __shared__ float4 smem4[];
    float* xs = reinterpret_cast<float*>(smem4);  // [NB][K], split layout
    __shared__ int head_unit[kStreamWarps], tail_unit[kStreamWarps], head_fin[kStreamWarps];
    __shared__ float head_val[kStreamWarps][RU][NB], tail_val[kStreamWarps][RU][NB];
    __shared__ float red_v[kStreamWarps][NB];
    __shared__ int red_r[kStreamWarps][NB];
    // EPI_RESADD: the CTA's residual values, loaded with the input after the
    // dependency wait, so that finishing a row does not wait for a load
    constexpr int kYpreUnits = 64;
    __shared__ float ypre_s[kYpreUnits][NB];
    constexpr int EPC = Chunk16<T>::kElems;

    pdl_launch();
    PIPO_TR(const TraceT0 tr0 = trace_begin(); unsigned long long tr1 = 0;
            __shared__ unsigned long long tr_lo, tr_hi;
            if (threadIdx.x == 0) { tr_lo = ~0ull; tr_hi = 0ull; })
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int K = p.K;
    const int cpr = K * (int)sizeof(T) / 512;  // exact
    const int cpu = cpr * RU;
    const int G = gridDim.x;
    const int u0 = (int)((long long)blockIdx.x * p.N / G);
    const int u1 = (int)((long long)(blockIdx.x + 1) * p.N / G);
    const int C = (u1 - u0) * cpu;
    const int c0 = (int)((long long)warp * C / kStreamWarps);
    const int c1 = (int)((long long)(warp + 1) * C / kStreamWarps);
    const char* wbase = static_cast<const char*>(p.W) + (size_t)u0 * cpu * 512 + lane * 16;

    for (int b0 = 0; b0 < p.B; b0 += NB) {
        const int nb = min(NB, p.B - b0);
        const char* wp = wbase + (size_t)c0 * 512;  // next chunk to load
        int lc = c0;
        uint4 bufA[kU], bufB[kU];
        auto load_batch = [&](uint4 (&buf)[kU]) {
#pragma unroll
            for (int u = 0; u < kU; ++u)
                if (lc + u < c1) buf[u] = ldg_stream(wp + u * 512);
            wp += kU * 512;
            lc += kU;
        };
        load_batch(bufA);
        load_batch(bufB);
        // with this warp's first weight loads in flight
        if (b0 == 0 && p.pf_k && threadIdx.x == 0) l2_warm_pages(p);
        if (b0 == 0) {
            pdl_wait();
            PIPO_TR(tr1 = trace_now();)
            if (p.zero_ptr && blockIdx.x == 0)
                for (int i = threadIdx.x; i < p.zero_n; i += blockDim.x) p.zero_ptr[i] = 0ull;
        }
        const bool ypre_on = p.epi == EPI_RESADD && u1 - u0 <= kYpreUnits;
        __syncthreads();
        stage_input_async<T, NB>(p, xs, reinterpret_cast<T*>(xs + NB * K), b0, nb, ypre_on ? ypre_s : nullptr, u0,
                                 u1 - u0);

        float best_v[NB];
        int best_r[NB];
#pragma unroll
        for (int bb = 0; bb < NB; ++bb) { best_v[bb] = -INFINITY; best_r[bb] = 0x7fffffff; }
        float acc[NB], part[RU][NB];  // running row sum; finished rows of the current unit
#pragma unroll
        for (int bb = 0; bb < NB; ++bb) {
            acc[bb] = 0.f;
#pragma unroll
            for (int r = 0; r < RU; ++r) part[r][bb] = 0.f;
        }
        if (lane == 0) { head_fin[warp] = 0; head_unit[warp] = -1; tail_unit[warp] = -1; }

        int cc = c0;
        int crow = c0 / cpr, cj = c0 - crow * cpr;
        // x float4 index of this lane at chunk j: plane 0 at j*32 + lane, plane 1 at + K/8
        int xi = cj * 32 + lane;
        const float4* xs4 = reinterpret_cast<const float4*>(xs);
        const int plane = K / 8;  // float4s per plane (16-bit weights)
        auto consume_batch = [&](const uint4 (&buf)[kU]) {
#pragma unroll
            for (int u = 0; u < kU; ++u) {
                if (cc < c1) {
                    float w[EPC];
                    Chunk16<T>::to_float(buf[u], w);
#pragma unroll
                    for (int bb = 0; bb < NB; ++bb) {
                        const float4 xa = xs4[bb * (K / 4) + xi];
                        float sum = w[0] * xa.x + w[1] * xa.y + w[2] * xa.z + w[3] * xa.w;
                        if (EPC == 8) {
                            const float4 xb = xs4[bb * (K / 4) + plane + xi];
                            sum += w[4 % EPC] * xb.x + w[5 % EPC] * xb.y + w[6 % EPC] * xb.z + w[7 % EPC] * xb.w;
                        }
                        acc[bb] += sum;
                    }
                    ++cc;
                    xi += 32;
                    if (++cj == cpr) {
                        // row crow finished: its partial is this warp's whole
                        // contribution to that row
                        const int r = crow % RU;
#pragma unroll
                        for (int bb = 0; bb < NB; ++bb) {
                            const float t = warp_sum(acc[bb]);
                            acc[bb] = 0.f;
#pragma unroll
                            for (int rr = 0; rr < RU; ++rr)
                                if (rr == r) part[rr][bb] = t;
                        }
                        if (r == RU - 1) {
                            const int unit = crow / RU;
                            if (unit * cpu >= c0) {
                                unit_epilogue<T, RU, NB>(p, u0 + unit, part, b0, nb, best_v, best_r, ypre_on ? ypre_s[unit] : nullptr);
                            } else if (lane == 0) {
                                head_unit[warp] = unit;
                                head_fin[warp] = 1;
#pragma unroll
                                for (int rr = 0; rr < RU; ++rr)
#pragma unroll
                                    for (int bb = 0; bb < NB; ++bb) head_val[warp][rr][bb] = part[rr][bb];
                            }
#pragma unroll
                            for (int rr = 0; rr < RU; ++rr)
#pragma unroll
                                for (int bb = 0; bb < NB; ++bb) part[rr][bb] = 0.f;
                        }
                        cj = 0;
                        xi = lane;
                        ++crow;
                    }
                }
            }
        };
        while (cc < c1) {
            consume_batch(bufA);
            load_batch(bufA);
            if (cc >= c1) break;
            consume_batch(bufB);
            load_batch(bufB);
        }
        PIPO_TR(if (lane == 0) { const unsigned long long te = trace_now(); atomicMin(&tr_lo, te); atomicMax(&tr_hi, te); })
        // the range ended inside a unit: record the partial (rows done + running row)
        if (c0 < c1 && (c1 % cpu) != 0) {
            const int unit = (c1 - 1) / cpu;
            const int r = crow % RU;  // row in progress (cj > 0) or next row
            float a[RU][NB];
#pragma unroll
            for (int bb = 0; bb < NB; ++bb) {
                const float t = warp_sum(acc[bb]);
#pragma unroll
                for (int rr = 0; rr < RU; ++rr) a[rr][bb] = part[rr][bb] + ((rr == r && cj > 0) ? t : 0.f);
            }
            if (lane == 0) {
                if (unit * cpu >= c0) {
                    tail_unit[warp] = unit;
#pragma unroll
                    for (int rr = 0; rr < RU; ++rr)
#pragma unroll
                        for (int bb = 0; bb < NB; ++bb) tail_val[warp][rr][bb] = a[rr][bb];
                } else {
                    head_unit[warp] = unit;
                    head_fin[warp] = 0;
#pragma unroll
                    for (int rr = 0; rr < RU; ++rr)
#pragma unroll
                        for (int bb = 0; bb < NB; ++bb) head_val[warp][rr][bb] = a[rr][bb];
                }
            }
        }
        __syncthreads();
        if (head_fin[warp] && head_unit[warp] >= 0) {
            const int unit = head_unit[warp];
            int ws = warp - 1;
            while (ws >= 0 && tail_unit[ws] != unit) --ws;
            float a[RU][NB];
#pragma unroll
            for (int r = 0; r < RU; ++r)
#pragma unroll
                for (int bb = 0; bb < NB; ++bb) {
                    float sum = (ws >= 0) ? tail_val[ws][r][bb] : 0.f;
                    for (int v = (ws >= 0 ? ws + 1 : 0); v <= warp; ++v)
                        if (head_unit[v] == unit) sum += head_val[v][r][bb];
                    a[r][bb] = sum;
                }
            unit_epilogue<T, RU, NB>(p, u0 + unit, a, b0, nb, best_v, best_r, ypre_on ? ypre_s[unit] : nullptr);
        }
        if (p.epi == EPI_ARGMAX) {
            if (lane == 0)
#pragma unroll
                for (int bb = 0; bb < NB; ++bb) { red_v[warp][bb] = best_v[bb]; red_r[warp][bb] = best_r[bb]; }
            __syncthreads();
            if (threadIdx.x < nb) {
                const int bb = threadIdx.x;
                float bv = -INFINITY;
                int br = 0x7fffffff;
                for (int w = 0; w < kStreamWarps; ++w)
                    if (red_r[w][bb] != 0x7fffffff && (red_v[w][bb] > bv || (red_v[w][bb] == bv && red_r[w][bb] < br))) {
                        bv = red_v[w][bb];
                        br = red_r[w][bb];
                    }
                if (br != 0x7fffffff) atomicMax(p.am + b0 + bb, argmax_key(bv, br));
            }
        }
        __syncthreads();
    }
    PIPO_TR(if (threadIdx.x == 0) trace_put(TR_GEMV, tr0, tr0.clk, tr1, tr_lo, tr_hi);)
}

// ---------------------------------------------------------------------------
// Per-warp accumulation over a contiguous range [c0, c1) of 512-byte chunks of
// whole-chunk rows (shared by the register-ring and the bulk-copy kernels).
template <typename T, int NB, int RU>
struct WarpRows {
    static constexpr int EPC = Chunk16<T>::kElems;
    const GemvParams* p;
    int K, cpr, cpu, u0, c0, c1, b0, nb, lane, warp;
    int cc, crow, cj, xi, plane;
    const float4* xs4;
    float acc[NB], part[RU][NB];
    float best_v[NB];
    int best_r[NB];

    __device__ __forceinline__ void init(const GemvParams* pp, const float* xs, int cpr_, int u0_, int c0_, int c1_,
                                         int b0_, int nb_) {
        p = pp;
        K = pp->K;
        cpr = cpr_;
        cpu = cpr_ * RU;
        u0 = u0_;
        c0 = c0_;
        c1 = c1_;
        b0 = b0_;
        nb = nb_;
        lane = threadIdx.x & 31;
        warp = threadIdx.x >> 5;
        cc = c0;
        crow = c0 / cpr;
        cj = c0 - crow * cpr;
        xi = cj * 32 + lane;
        plane = K / 8;
        xs4 = reinterpret_cast<const float4*>(xs);
#pragma unroll
        for (int bb = 0; bb < NB; ++bb) {
            acc[bb] = 0.f;
            best_v[bb] = -INFINITY;
            best_r[bb] = 0x7fffffff;
#pragma unroll
            for (int r = 0; r < RU; ++r) part[r][bb] = 0.f;
        }
    }

    // consume the next chunk cc of the range (its 16 bytes for this lane)
    template <int NW>
    __device__ __forceinline__ void chunk(const uint4& wv, int (&head_unit)[NW], int (&head_fin)[NW],
                                          float (&head_val)[NW][RU][NB]) {
        float w[EPC];
        Chunk16<T>::to_float(wv, w);
#pragma unroll
        for (int bb = 0; bb < NB; ++bb) {
            const float4 xa = xs4[bb * (K / 4) + xi];
            float sum = w[0] * xa.x + w[1] * xa.y + w[2] * xa.z + w[3] * xa.w;
            if (EPC == 8) {
                const float4 xb = xs4[bb * (K / 4) + plane + xi];
                sum += w[4 % EPC] * xb.x + w[5 % EPC] * xb.y + w[6 % EPC] * xb.z + w[7 % EPC] * xb.w;
            }
            acc[bb] += sum;
        }
        ++cc;
        xi += 32;
        if (++cj == cpr) {
            const int r = crow % RU;
#pragma unroll
            for (int bb = 0; bb < NB; ++bb) {
                const float t = warp_sum(acc[bb]);
                acc[bb] = 0.f;
#pragma unroll
                for (int rr = 0; rr < RU; ++rr)
                    if (rr == r) part[rr][bb] = t;
            }
            if (r == RU - 1) {
                const int unit = crow / RU;
                if (unit * cpu >= c0) {
                    unit_epilogue<T, RU, NB>(*p, u0 + unit, part, b0, nb, best_v, best_r);
                } else if (lane == 0) {
                    head_unit[warp] = unit;
                    head_fin[warp] = 1;
#pragma unroll
                    for (int rr = 0; rr < RU; ++rr)
#pragma unroll
                        for (int bb = 0; bb < NB; ++bb) head_val[warp][rr][bb] = part[rr][bb];
                }
#pragma unroll
                for (int rr = 0; rr < RU; ++rr)
#pragma unroll
                    for (int bb = 0; bb < NB; ++bb) part[rr][bb] = 0.f;
            }
            cj = 0;
            xi = lane;
            ++crow;
        }
    }

    // the range ended inside a unit: record this warp's partial of it
    template <int NW>
    __device__ __forceinline__ void finish(int (&head_unit)[NW], int (&head_fin)[NW], int (&tail_unit)[NW],
                                           float (&head_val)[NW][RU][NB], float (&tail_val)[NW][RU][NB]) {
        if (!(c0 < c1 && (c1 % cpu) != 0)) return;
        const int unit = (c1 - 1) / cpu;
        const int r = crow % RU;
        float a[RU][NB];
#pragma unroll
        for (int bb = 0; bb < NB; ++bb) {
            const float t = warp_sum(acc[bb]);
#pragma unroll
            for (int rr = 0; rr < RU; ++rr) a[rr][bb] = part[rr][bb] + ((rr == r && cj > 0) ? t : 0.f);
        }
        if (lane != 0) return;
        if (unit * cpu >= c0) {
            tail_unit[warp] = unit;
#pragma unroll
            for (int rr = 0; rr < RU; ++rr)
#pragma unroll
                for (int bb = 0; bb < NB; ++bb) tail_val[warp][rr][bb] = a[rr][bb];
        } else {
            head_unit[warp] = unit;
            head_fin[warp] = 0;
#pragma unroll
            for (int rr = 0; rr < RU; ++rr)
#pragma unroll
                for (int bb = 0; bb < NB; ++bb) head_val[warp][rr][bb] = a[rr][bb];
        }
    }
};

// After a block barrier: units split between warps are finished by the warp
// holding their last chunk (partials added in warp order); then the argmax
// reduction of the block.
template <typename T, int NB, int RU, int NW>
__device__ __forceinline__ void finish_block(const GemvParams& p, WarpRows<T, NB, RU>& wr, int (&head_unit)[NW],
                                             int (&head_fin)[NW], int (&tail_unit)[NW], float (&head_val)[NW][RU][NB],
                                             float (&tail_val)[NW][RU][NB], float (&red_v)[NW][NB],
                                             int (&red_r)[NW][NB]) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (head_fin[warp] && head_unit[warp] >= 0) {
        const int unit = head_unit[warp];
        int ws = warp - 1;
        while (ws >= 0 && tail_unit[ws] != unit) --ws;
        float a[RU][NB];
#pragma unroll
        for (int r = 0; r < RU; ++r)
#pragma unroll
            for (int bb = 0; bb < NB; ++bb) {
                float sum = (ws >= 0) ? tail_val[ws][r][bb] : 0.f;
                for (int v = (ws >= 0 ? ws + 1 : 0); v <= warp; ++v)
                    if (head_unit[v] == unit) sum += head_val[v][r][bb];
                a[r][bb] = sum;
            }
        unit_epilogue<T, RU, NB>(p, wr.u0 + unit, a, wr.b0, wr.nb, wr.best_v, wr.best_r);
    }
    if (p.epi == EPI_ARGMAX) {
        if (lane == 0)
#pragma unroll
            for (int bb = 0; bb < NB; ++bb) { red_v[warp][bb] = wr.best_v[bb]; red_r[warp][bb] = wr.best_r[bb]; }
        __syncthreads();
        if (threadIdx.x < wr.nb) {
            const int bb = threadIdx.x;
            float bv = -INFINITY;
            int br = 0x7fffffff;
            for (int w = 0; w < NW; ++w)
                if (red_r[w][bb] != 0x7fffffff && (red_v[w][bb] > bv || (red_v[w][bb] == bv && red_r[w][bb] < br))) {
                    bv = red_v[w][bb];
                    br = red_r[w][bb];
                }
            if (br != 0x7fffffff) atomicMax(p.am + wr.b0 + bb, argmax_key(bv, br));
        }
    }
}

}  // namespace pipo
