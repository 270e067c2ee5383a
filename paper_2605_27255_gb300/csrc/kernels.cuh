// Device kernels of the PIPO pair-decode step (sm_103a).
//
// Every weight matrix is streamed from HBM once per step; activations stay in
// fp32; weights, embeddings and the KV cache are bf16 (or fp32 for fp32
// models).  The step is a chain of these kernels replayed as one CUDA graph.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace pipo {

constexpr int kThreads = 256;  // GEMV block
constexpr int kWarps = kThreads / 32;

enum Epi : int {
    EPI_STORE = 0,   // y = W x
    EPI_BIAS = 1,    // y = W x + bias
    EPI_SILU = 2,    // y = SiLU(W x)
    EPI_RESADD = 3,  // y += W x            (residual stream; split-K: fixed-order sum)
    EPI_SWIGLU = 4,  // y = SiLU(W_2r x) * (W_2r+1 x)   (gate and up rows interleaved)
    EPI_ARGMAX = 5,  // packed (logit, -row) max per sequence; optional logits
};

// One input segment of a GEMV: either fp32 activations or an embedding-row
// gather, optionally RMS-normalised (y = x / sqrt(mean(x^2) + eps) * gamma).
struct Seg {
    const float* src;                  // [B, ld] activations, or nullptr (gather)
    int ld;
    const void* table;                 // gather table [*, K] (weight type)
    const void* pad;                   // [K] row used for token id < 0 (PAD)
    const int32_t* tok;                // token of sequence b: tok[b * tok_ld]
    int tok_ld;
    const unsigned long long* tok_am;  // or: packed argmax of sequence b
    const void* gamma;                 // [K] gain or nullptr (no norm)
    int K;
};

struct GemvParams {
    Seg seg[2];
    int nseg;
    int joint_norm;      // one RMSNorm over the concatenation (gain in seg[0].gamma, length K)
    const void* W;       // [rows, K]
    int N;               // output rows
    int K;               // input length (sum of the segments)
    int epi;
    float* y;
    int ldy;
    const void* bias;
    unsigned long long* am;  // EPI_ARGMAX target [B]
    float* dbg;              // EPI_ARGMAX logits [B, ld_dbg] or nullptr
    int ld_dbg;
    int B;
    int splitk;
    float eps;
    unsigned long long* zero_ptr;  // zeroed by block 0 before anything else (or nullptr)
    int zero_n;
    float* part;         // EPI_RESADD with splitk > 1: partials [splitk][B][N]
    unsigned* rowcnt;    // arrival counters per (batch group, row), [ceil(B/NB)][N] (zero between launches)
    // L2 warm-up of the next attention's cached pages (streaming GEMV, a
    // decode step's QKV projection; pf_k == nullptr: none).  Before its
    // dependency wait the kernel prefetches into L2 the key and value pages
    // that hold entries 0 .. pf_npos[b] - 1 of sequences b < pf_nseq: page
    // block blk of a layer is pf_bytes contiguous bytes at pf_k / pf_v +
    // blk * pf_bytes (every kv head), blk = pf_table[b * pf_bps + page].
    const void* pf_k;
    const void* pf_v;
    const int32_t* pf_table;
    const int32_t* pf_npos;
    int pf_bps, pf_page, pf_nseq;
    unsigned pf_bytes;
};

// ---------------------------------------------------------------- loads

// 128-bit streaming load of read-only weights.  volatile keeps the issue
// point where the code puts it (ahead of the compute that consumes an older
// load), so the register ring really holds several loads in flight.
__device__ __forceinline__ uint4 ldg_stream(const void* p) {
    uint4 r;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
        : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
        : "l"(p));
    return r;
}

// Bulk prefetch of [ptr, ptr + bytes) into L2 (16-byte aligned, bytes a
// multiple of 16); no data reaches the SM.
__device__ __forceinline__ void prefetch_l2_bulk(const void* ptr, unsigned bytes) {
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(ptr), "r"(bytes) : "memory");
}

// GemvParams::pf_*: the pages are spread over the CTAs of the grid, one bulk
// prefetch per page of keys or values.  The cached lengths and page tables
// change only between steps (graph launches), so they are read before the
// dependency wait; the entries prefetched were written by earlier steps.
__device__ __forceinline__ void l2_warm_pages(const GemvParams& p) {
    int i0 = 0;  // items of the sequences before b
    for (int b = 0; b < p.pf_nseq; ++b) {
        const int items = 2 * ((p.pf_npos[b] + p.pf_page - 1) / p.pf_page);
        for (int i = ((int)blockIdx.x - i0 % (int)gridDim.x + (int)gridDim.x) % (int)gridDim.x; i < items;
             i += gridDim.x) {
            const int blk = p.pf_table[(size_t)b * p.pf_bps + (i >> 1)];
            const char* base = static_cast<const char*>((i & 1) ? p.pf_v : p.pf_k);
            prefetch_l2_bulk(base + (size_t)blk * p.pf_bytes, p.pf_bytes);
        }
        i0 += items;
    }
}

// 128-bit load of cache data written by earlier kernels (L1 bypassed).
__device__ __forceinline__ uint4 ldg_cg(const void* p) {
    uint4 r;
    asm volatile("ld.global.cg.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
                 : "l"(p));
    return r;
}

__device__ __forceinline__ float bf_lo(uint32_t u) { return __uint_as_float(u << 16); }
__device__ __forceinline__ float bf_hi(uint32_t u) { return __uint_as_float(u & 0xffff0000u); }

template <typename T> struct W8;  // 8 consecutive weights

template <> struct W8<__nv_bfloat16> {
    uint4 v;
    __device__ __forceinline__ void load(const __nv_bfloat16* p) { v = ldg_stream(p); }
    __device__ __forceinline__ void unpack(float (&f)[8]) const {
        f[0] = bf_lo(v.x); f[1] = bf_hi(v.x); f[2] = bf_lo(v.y); f[3] = bf_hi(v.y);
        f[4] = bf_lo(v.z); f[5] = bf_hi(v.z); f[6] = bf_lo(v.w); f[7] = bf_hi(v.w);
    }
};

template <> struct W8<float> {
    uint4 a, b;
    __device__ __forceinline__ void load(const float* p) { a = ldg_stream(p); b = ldg_stream(p + 4); }
    __device__ __forceinline__ void unpack(float (&f)[8]) const {
        f[0] = __uint_as_float(a.x); f[1] = __uint_as_float(a.y); f[2] = __uint_as_float(a.z); f[3] = __uint_as_float(a.w);
        f[4] = __uint_as_float(b.x); f[5] = __uint_as_float(b.y); f[6] = __uint_as_float(b.z); f[7] = __uint_as_float(b.w);
    }
};

__device__ __forceinline__ float to_f(float v) { return v; }
__device__ __forceinline__ float to_f(__nv_bfloat16 v) { return __bfloat162float(v); }
template <typename T> __device__ __forceinline__ float ldw(const void* p, size_t i) {
    return to_f(static_cast<const T*>(p)[i]);
}
template <typename T> __device__ __forceinline__ T from_f(float v);
template <> __device__ __forceinline__ float from_f<float>(float v) { return v; }
template <> __device__ __forceinline__ __nv_bfloat16 from_f<__nv_bfloat16>(float v) { return __float2bfloat16_rn(v); }

__device__ __forceinline__ float silu(float x) { return x / (1.0f + expf(-x)); }

// Packed argmax key: higher logit first, then lower row.
__device__ __forceinline__ unsigned long long argmax_key(float v, int row) {
    uint32_t u = __float_as_uint(v);
    uint32_t o = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
    return ((unsigned long long)o << 32) | (unsigned long long)(0xFFFFFFFFu - (uint32_t)row);
}
__device__ __forceinline__ int argmax_row(unsigned long long k) {
    return (int)(0xFFFFFFFFu - (uint32_t)(k & 0xFFFFFFFFull));
}

// Programmatic dependent launch: let the next kernel of the stream start its
// independent prologue, and wait for the previous kernel's results.  Both are
// no-ops for a kernel launched without the programmatic-serialization attribute.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_launch() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// ---------------------------------------------------------------- timeline
//
// Built only with -DPIPO_TRACE (a measurement build; the default build has
// none of it): one record per CTA of the projection and attention kernels,
// {kind | sm << 8 | CTAs of the grid << 16 | linear block << 32, entry time,
// time past the dependency wait, two kernel-specific phase times, exit time}
// (%globaltimer, ns), appended to a device buffer [count, capacity, records]
// whose address each translation unit holds (set by the host, see
// pipo_trace_setup).  The records show, under graph replay with programmatic
// dependent launch, when each CTA started, waited and finished.
enum TraceKind : unsigned { TR_GEMV = 1, TR_TCF = 2, TR_TC = 3, TR_ATTN_MMA = 4, TR_ATTN_CL = 5, TR_ATTN_FLAT = 6,
                       TR_TCF_EPI = 7, TR_ATTN_MMA_EPI = 8, TR_ATTN_CL_EPI = 11 };
#ifdef PIPO_TRACE
constexpr int kTraceWords = 6;
// Phase times are SM cycles (clock64: no memory path, unlike %globaltimer
// reads, which queue behind outstanding loads) placed on the global clock
// through one (%globaltimer, clock64) pair read at entry, at the 2070 MHz SM
// clock the benchmark runs at.
constexpr double kTraceNsPerClk = 1.0 / 2.07;
static __device__ unsigned long long* g_trace_buf;
struct TraceT0 {
    unsigned long long gt, clk;
};
__device__ __forceinline__ unsigned long long trace_now() { return (unsigned long long)clock64(); }
// read by thread 0 only (which writes the records): the others get zeros
__device__ __forceinline__ TraceT0 trace_begin() {
    TraceT0 b{0ull, 0ull};
    if (threadIdx.x == 0) {
        asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(b.gt));
        b.clk = trace_now();
    }
    return b;
}
__device__ __forceinline__ unsigned long long trace_ns(const TraceT0& b, unsigned long long c) {
    return c ? b.gt + (unsigned long long)((double)(long long)(c - b.clk) * kTraceNsPerClk) : 0ull;
}
__device__ __forceinline__ void trace_put(unsigned kind, const TraceT0& base, unsigned long long t0,
                                          unsigned long long t1, unsigned long long t2, unsigned long long t3,
                                          unsigned long long t4 = 0) {
    if (!t4) t4 = trace_now();  // exit: before the slot atomic and its latency
    unsigned long long* b = g_trace_buf;
    if (!b) return;
    const unsigned long long i = atomicAdd(b, 1ull);
    if (i >= b[1]) return;
    unsigned sm;
    asm volatile("mov.u32 %0, %%smid;" : "=r"(sm));
    const unsigned long long nblk = (unsigned long long)gridDim.x * gridDim.y * gridDim.z;
    const unsigned long long blk = blockIdx.x + (unsigned long long)gridDim.x * (blockIdx.y + (unsigned long long)gridDim.y * blockIdx.z);
    unsigned long long* r = b + 2 + i * kTraceWords;
    r[0] = kind | ((unsigned long long)(sm & 0xffu) << 8) | ((nblk & 0xffffull) << 16) | (blk << 32);
    r[1] = trace_ns(base, t0);
    r[2] = trace_ns(base, t1);
    r[3] = trace_ns(base, t2);
    r[4] = trace_ns(base, t3);
    r[5] = trace_ns(base, t4);
}
static inline cudaError_t set_unit_trace(unsigned long long* buf) {
    return cudaMemcpyToSymbol(g_trace_buf, &buf, sizeof(buf));
}
#define PIPO_TR(...) __VA_ARGS__
#else
#define PIPO_TR(...)
#endif

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// ---------------------------------------------------------------- GEMV
//
// y[b, r] = epi( sum_k W[r, k] * xin[b, k] ),  xin = staged (gathered,
// normalised) input in shared memory, NB sequences at a time.  A warp owns one
// (row, K-slice) task at a time and streams its weights with 128-bit
// non-allocating loads, kU chunks in flight per lane.
template <typename T, int NB, bool TWO>
__global__ void __launch_bounds__(kThreads) gemv_kernel(GemvParams p) {
    extern __shared__ float4 smem4[];
    float* xs = reinterpret_cast<float*>(smem4);  // [NB][K]
    __shared__ float rstd_s[NB][2];
    constexpr int kU = 8;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int K = p.K;
    const T* W = static_cast<const T*>(p.W);

    pdl_launch();
    pdl_wait();
    if (p.zero_ptr && blockIdx.x == 0)
        for (int i = threadIdx.x; i < p.zero_n; i += blockDim.x) p.zero_ptr[i] = 0ull;

    const int S = p.splitk;
    const int Ks = ((K + S * 8 - 1) / (S * 8)) * 8;
    const int tasks = p.N * S;

    for (int b0 = 0; b0 < p.B; b0 += NB) {
        const int nb = min(NB, p.B - b0);
        __syncthreads();
        // ---- stage inputs
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
        // ---- RMSNorm of each segment (or of the concatenation): one warp per sum
        const bool any_norm = p.seg[0].gamma || (p.nseg > 1 && p.seg[1].gamma);
        if (any_norm) {
            const int ngrp = p.joint_norm ? 1 : p.nseg;
            for (int q = warp; q < NB * ngrp; q += kWarps) {
                const int bb = q / ngrp, s = q % ngrp;
                const int k0 = (s == 0) ? 0 : p.seg[0].K;
                const int len = p.joint_norm ? K : p.seg[s].K;
                float ss = 0.f;
                for (int k = lane; k < len; k += 32) {
                    float v = xs[bb * K + k0 + k];
                    ss += v * v;
                }
                ss = warp_sum(ss);
                if (lane == 0) rstd_s[bb][s] = 1.0f / sqrtf(ss / (float)len + p.eps);
            }
            __syncthreads();
            for (int bb = 0; bb < NB; ++bb) {
                for (int k = threadIdx.x; k < K; k += blockDim.x) {
                    int s = (p.joint_norm || k < p.seg[0].K) ? 0 : 1;
                    const Seg& sg = p.seg[s];
                    if (!sg.gamma) continue;
                    int kk = (p.joint_norm || s == 0) ? k : k - p.seg[0].K;
                    xs[bb * K + k] *= rstd_s[bb][s] * ldw<T>(sg.gamma, kk);
                }
            }
            __syncthreads();
        }

        // ---- rows
        float best_v[NB];
        int best_r[NB];
#pragma unroll
        for (int bb = 0; bb < NB; ++bb) { best_v[bb] = -INFINITY; best_r[bb] = 0x7fffffff; }

        for (int t = blockIdx.x * kWarps + warp; t < tasks; t += gridDim.x * kWarps) {
            const int r = t / S, s = t % S;
            const int k0 = s * Ks, k1 = min(K, k0 + Ks);
            float acc0[NB], acc1[NB];
#pragma unroll
            for (int bb = 0; bb < NB; ++bb) { acc0[bb] = 0.f; acc1[bb] = 0.f; }
            // SwiGLU: gate row 2r and up row 2r+1 (interleaved at upload)
            const T* w0 = W + (size_t)(TWO ? 2 * r : r) * K;
            const T* w1 = W + (size_t)(2 * r + 1) * K;
            for (int kb = k0 + lane * 8; kb < k1; kb += 256 * kU) {
                W8<T> wa[kU], wb[kU];
#pragma unroll
                for (int u = 0; u < kU; ++u) {
                    const int k = kb + u * 256;
                    if (k < k1) {
                        wa[u].load(w0 + k);
                        if (TWO) wb[u].load(w1 + k);
                    }
                }
#pragma unroll
                for (int u = 0; u < kU; ++u) {
                    const int k = kb + u * 256;
                    if (k < k1) {
                        float fa[8], fb[8];
                        wa[u].unpack(fa);
                        if (TWO) wb[u].unpack(fb);
#pragma unroll
                        for (int bb = 0; bb < NB; ++bb) {
                            const float4 x0 = *reinterpret_cast<const float4*>(xs + bb * K + k);
                            const float4 x1 = *reinterpret_cast<const float4*>(xs + bb * K + k + 4);
                            acc0[bb] += fa[0] * x0.x + fa[1] * x0.y + fa[2] * x0.z + fa[3] * x0.w +
                                        fa[4] * x1.x + fa[5] * x1.y + fa[6] * x1.z + fa[7] * x1.w;
                            if (TWO)
                                acc1[bb] += fb[0] * x0.x + fb[1] * x0.y + fb[2] * x0.z + fb[3] * x0.w +
                                            fb[4] * x1.x + fb[5] * x1.y + fb[6] * x1.z + fb[7] * x1.w;
                        }
                    }
                }
            }
#pragma unroll
            for (int bb = 0; bb < NB; ++bb) {
                acc0[bb] = warp_sum(acc0[bb]);
                if (TWO) acc1[bb] = warp_sum(acc1[bb]);
            }
            if (p.epi == EPI_ARGMAX) {
#pragma unroll
                for (int bb = 0; bb < NB; ++bb)
                    if (acc0[bb] > best_v[bb] || (acc0[bb] == best_v[bb] && r < best_r[bb])) {
                        best_v[bb] = acc0[bb];
                        best_r[bb] = r;
                    }
                if (p.dbg && lane < nb) {
#pragma unroll
                    for (int bb = 0; bb < NB; ++bb)
                        if (bb == lane) p.dbg[(size_t)(b0 + bb) * p.ld_dbg + r] = acc0[bb];
                }
                continue;
            }
            if (lane < nb) {
#pragma unroll
                for (int bb = 0; bb < NB; ++bb) {
                    if (bb != lane) continue;
                    float* yp = p.y + (size_t)(b0 + bb) * p.ldy + r;
                    const float a = acc0[bb];
                    switch (p.epi) {
                        case EPI_STORE: *yp = a; break;
                        case EPI_BIAS: *yp = a + ldw<T>(p.bias, r); break;
                        case EPI_SILU: *yp = silu(a); break;
                        case EPI_RESADD:
                            if (S == 1) *yp += a;
                            break;
                        case EPI_SWIGLU: *yp = silu(a) * acc1[bb]; break;
                        default: break;
                    }
                }
            }
            // split-K residual add: every slice stores its partial; the last
            // slice of the row to arrive adds them in slice order (deterministic).
            // CTAs reach the batch groups at different times: one counter per
            // (group, row).
            if (p.epi == EPI_RESADD && S > 1 && lane == 0) {
                for (int bb = 0; bb < nb; ++bb) p.part[((size_t)s * p.B + b0 + bb) * p.N + r] = acc0[bb];
                __threadfence();
                unsigned* cnt = p.rowcnt + (size_t)(b0 / NB) * p.N + r;
                const unsigned prev = atomicAdd(cnt, 1u);
                if (prev == (unsigned)S - 1) {
                    __threadfence();
                    for (int bb = 0; bb < nb; ++bb) {
                        float sum = 0.f;
                        for (int ss = 0; ss < S; ++ss) sum += __ldcg(p.part + ((size_t)ss * p.B + b0 + bb) * p.N + r);
                        p.y[(size_t)(b0 + bb) * p.ldy + r] += sum;
                    }
                    *cnt = 0u;
                }
            }
        }
        if (p.epi == EPI_ARGMAX && lane < nb) {
#pragma unroll
            for (int bb = 0; bb < NB; ++bb)
                if (bb == lane && best_r[bb] != 0x7fffffff)
                    atomicMax(p.am + b0 + bb, argmax_key(best_v[bb], best_r[bb]));
        }
    }
}

// ---------------------------------------------------------------- attention

struct KVView {
    void* K;                  // layer base: [blocks][n_kv][page][d_h]
    void* V;
    const int32_t* table;     // [B][blocks_per_seq]
    int blocks_per_seq;
    int page;
    int n_kv;
};

template <typename T, int DH>
__device__ __forceinline__ size_t kv_off(const KVView& kv, int b, int pos, int g) {
    const int blk = kv.table[(size_t)b * kv.blocks_per_seq + pos / kv.page];
    return (((size_t)blk * kv.n_kv + g) * kv.page + (pos % kv.page)) * DH;
}

// Prefill chunk: RoPE on the keys of every row and the append of its key and
// value, before the chunk's attention reads them (row r is sequence r % nseq
// at position n_pos[r % nseq] + r / nseq).  Rotate-half with the fp32
// cos/sin table the attention kernels use ([max_ctx][d_h/2][2]), rounded to
// the cache type.  grid (rows, n_kv), DH/2 threads.
template <typename T, int DH>
__global__ void append_rows_kernel(const float* __restrict__ qkv, int ld_qkv, int n_q, KVView kv,
                                   const int32_t* __restrict__ n_pos, int nseq, const float* __restrict__ rope) {
    pdl_launch();
    pdl_wait();
    const int row = blockIdx.x, g = blockIdx.y, i = threadIdx.x;
    const int b = row % nseq;
    const int pos = n_pos[b] + row / nseq;
    const float* k = qkv + (size_t)row * ld_qkv + (size_t)(n_q + g) * DH;
    const float* v = qkv + (size_t)row * ld_qkv + (size_t)(n_q + kv.n_kv + g) * DH;
    const float c = rope[((size_t)pos * (DH / 2) + i) * 2], s = rope[((size_t)pos * (DH / 2) + i) * 2 + 1];
    const float a = k[i], bb = k[i + DH / 2];
    const size_t off = kv_off<T, DH>(kv, b, pos, g);
    T* K = static_cast<T*>(kv.K) + off;
    T* V = static_cast<T*>(kv.V) + off;
    K[i] = from_f<T>(a * c - bb * s);
    K[i + DH / 2] = from_f<T>(bb * c + a * s);
    V[i] = from_f<T>(v[i]);
    V[i + DH / 2] = from_f<T>(v[i + DH / 2]);
}

// RoPE on q and k (rotate-half, angle = pos * theta^(-2i/d) in double), then
// the new k and v appended at entry pos = n[b].  grid (B, n_q + 2 n_kv), DH/2 threads.
template <typename T, int DH>
__global__ void rope_append_kernel(const float* __restrict__ qkv, int ld_qkv, float* __restrict__ q_out,
                                   KVView kv, const int32_t* __restrict__ n_pos, int n_q, double theta) {
    pdl_launch();
    pdl_wait();
    const int b = blockIdx.x, h = blockIdx.y, i = threadIdx.x;
    const int pos = n_pos[b];
    const float* src = qkv + (size_t)b * ld_qkv + (size_t)h * DH;
    const int n_kv = kv.n_kv;
    if (h >= n_q + n_kv) {  // value head: copy into the cache
        const int g = h - n_q - n_kv;
        T* dst = static_cast<T*>(kv.V) + kv_off<T, DH>(kv, b, pos, g);
        dst[i] = from_f<T>(src[i]);
        dst[i + DH / 2] = from_f<T>(src[i + DH / 2]);
        return;
    }
    double sn, cs;
    sincos((double)pos * pow(theta, -2.0 * (double)i / (double)DH), &sn, &cs);
    const float c = (float)cs, s = (float)sn;
    const float a = src[i], bb = src[i + DH / 2];
    const float ra = a * c - bb * s, rb = bb * c + a * s;
    if (h < n_q) {
        q_out[(size_t)b * n_q * DH + (size_t)h * DH + i] = ra;
        q_out[(size_t)b * n_q * DH + (size_t)h * DH + i + DH / 2] = rb;
    } else {
        const int g = h - n_q;
        T* dst = static_cast<T*>(kv.K) + kv_off<T, DH>(kv, b, pos, g);
        dst[i] = from_f<T>(ra);
        dst[i + DH / 2] = from_f<T>(rb);
    }
}

// Split-KV flash decode.  grid (S, n_kv, B), 128 threads (4 warps).  CTA
// (s, g, b) attends the G = n_q/n_kv query heads of group g over its slice
// of entries [0, n[b]] and writes (m, l, o) partials; the last CTA of (b, g)
// to finish merges the S partials (log-sum-exp) into out[b, h*DH + t].
template <typename T, int DH, int G>
__global__ void __launch_bounds__(128) attn_decode_kernel(const float* __restrict__ q, KVView kv,
                                                          const int32_t* __restrict__ n_pos, float* __restrict__ out,
                                                          float* __restrict__ part_o, float* __restrict__ part_ml,
                                                          unsigned int* __restrict__ counters, int S, float scale) {
    constexpr int EPL = DH / 32;  // elements per lane
    pdl_launch();
    pdl_wait();
    const int s = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int n_kv = kv.n_kv, n_q = n_kv * G;
    const int len = n_pos[b] + 1;
    const int chunk = (len + S - 1) / S;
    const int j0 = s * chunk, j1 = min(len, j0 + chunk);

    float qr[G][EPL];
#pragma unroll
    for (int hh = 0; hh < G; ++hh)
#pragma unroll
        for (int e = 0; e < EPL; ++e)
            qr[hh][e] = q[(size_t)b * n_q * DH + (size_t)(g * G + hh) * DH + lane * EPL + e] * scale;

    float m[G], l[G], o[G][EPL];
#pragma unroll
    for (int hh = 0; hh < G; ++hh) {
        m[hh] = -INFINITY; l[hh] = 0.f;
#pragma unroll
        for (int e = 0; e < EPL; ++e) o[hh][e] = 0.f;
    }
    const T* Kb = static_cast<const T*>(kv.K);
    const T* Vb = static_cast<const T*>(kv.V);
    for (int j = j0 + warp; j < j1; j += 4) {
        const size_t off = kv_off<T, DH>(kv, b, j, g) + lane * EPL;
        float kk[EPL], vv[EPL];
#pragma unroll
        for (int e = 0; e < EPL; ++e) { kk[e] = to_f(Kb[off + e]); vv[e] = to_f(Vb[off + e]); }
#pragma unroll
        for (int hh = 0; hh < G; ++hh) {
            float d = 0.f;
#pragma unroll
            for (int e = 0; e < EPL; ++e) d += qr[hh][e] * kk[e];
            d = warp_sum(d);
            const float mn = fmaxf(m[hh], d);
            const float corr = expf(m[hh] - mn);
            const float pj = expf(d - mn);
            l[hh] = l[hh] * corr + pj;
#pragma unroll
            for (int e = 0; e < EPL; ++e) o[hh][e] = o[hh][e] * corr + pj * vv[e];
            m[hh] = mn;
        }
    }
    // merge the 4 warps
    __shared__ float sm_m[4][G], sm_l[4][G];
    __shared__ float sm_o[4][G][DH];
#pragma unroll
    for (int hh = 0; hh < G; ++hh) {
        if (lane == 0) { sm_m[warp][hh] = m[hh]; sm_l[warp][hh] = l[hh]; }
#pragma unroll
        for (int e = 0; e < EPL; ++e) sm_o[warp][hh][lane * EPL + e] = o[hh][e];
    }
    __syncthreads();
    for (int idx = threadIdx.x; idx < G * DH; idx += blockDim.x) {
        const int hh = idx / DH, t = idx % DH;
        float M = -INFINITY;
        for (int w = 0; w < 4; ++w) M = fmaxf(M, sm_m[w][hh]);
        float L = 0.f, Ov = 0.f;
        for (int w = 0; w < 4; ++w) {
            const float f = (sm_m[w][hh] == -INFINITY) ? 0.f : expf(sm_m[w][hh] - M);
            L += sm_l[w][hh] * f;
            Ov += sm_o[w][hh][t] * f;
        }
        const int h = g * G + hh;
        const size_t pi = ((size_t)(b * n_q + h) * S + s);
        part_o[pi * DH + t] = Ov;
        if (t == 0) { part_ml[pi * 2] = M; part_ml[pi * 2 + 1] = L; }
    }
    // last CTA of (b, g) merges the S partials
    __shared__ bool last;
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) {
        const unsigned prev = atomicAdd(&counters[b * n_kv + g], 1u);
        last = (prev == (unsigned)S - 1);
    }
    __syncthreads();
    if (!last) return;
    __threadfence();
    for (int idx = threadIdx.x; idx < G * DH; idx += blockDim.x) {
        const int hh = idx / DH, t = idx % DH;
        const int h = g * G + hh;
        const size_t p0 = (size_t)(b * n_q + h) * S;
        float M = -INFINITY;
        for (int ss = 0; ss < S; ++ss) M = fmaxf(M, __ldcg(part_ml + (p0 + ss) * 2));
        float L = 0.f, Ov = 0.f;
        for (int ss = 0; ss < S; ++ss) {
            const float ms = __ldcg(part_ml + (p0 + ss) * 2);
            const float f = (ms == -INFINITY) ? 0.f : expf(ms - M);
            L += __ldcg(part_ml + (p0 + ss) * 2 + 1) * f;
            Ov += __ldcg(part_o + (p0 + ss) * DH + t) * f;
        }
        out[(size_t)b * n_q * DH + (size_t)h * DH + t] = Ov / L;
    }
    if (threadIdx.x == 0) counters[b * n_kv + g] = 0u;
}

// ---------------------------------------------------------------- heads

struct StepState {
    int32_t* pending;      // [B,2]
    int32_t* n_pos;        // [B] entries in the caches
    long long* emitted;    // [B]
    int32_t* out_tokens;   // [B,2]
    int32_t* out_nacc;     // [B]
    const unsigned long long* am_b;
    const unsigned long long* am_d;
    float* dbg_conf;       // [B] or nullptr
    float* dbg_hb;         // [B,H] or nullptr
    float* dbg_hd;
    int32_t* dbg_xb;       // [B]
    int32_t* dbg_xd;
    // sampling in both heads (nullptr when greedy): the token-history bitmap
    // [B][presence_w] gains an accepted draft; the draw index advances
    uint32_t* presence;
    int presence_w;
    int32_t* samp_step;
};

// Confidence c = sigmoid(W2 . t) with t = SiLU(W1 RMSNorm([h_b; h_d])) computed
// by the preceding GEMV; acceptance; next pending pair; counters.  grid B.
template <typename T>
__global__ void accept_kernel(const float* __restrict__ t, const void* W2, int H, float tau, int force,
                              StepState st, const float* hb, const float* hd) {
    pdl_launch();
    pdl_wait();
    const int b = blockIdx.x;
    float acc = 0.f;
    for (int k = threadIdx.x; k < H; k += blockDim.x) acc += ldw<T>(W2, k) * t[(size_t)b * H + k];
    acc = warp_sum(acc);
    __shared__ float red[32];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) red[warp] = acc;
    __syncthreads();
    if (st.dbg_hb)
        for (int k = threadIdx.x; k < H; k += blockDim.x) {
            st.dbg_hb[(size_t)b * H + k] = hb[(size_t)b * H + k];
            st.dbg_hd[(size_t)b * H + k] = hd[(size_t)b * H + k];
        }
    if (threadIdx.x != 0) return;
    float s = 0.f;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) s += red[w];
    const float c = 1.0f / (1.0f + expf(-s));
    const int accept = (force == 1) ? 1 : (force == 2) ? 0 : (c >= tau ? 1 : 0);
    const int xb = argmax_row(st.am_b[b]), xd = argmax_row(st.am_d[b]);
    st.out_tokens[2 * b] = xb;
    st.out_tokens[2 * b + 1] = accept ? xd : -1;
    st.out_nacc[b] = accept;
    st.pending[2 * b] = xb;
    st.pending[2 * b + 1] = accept ? xd : -1;
    st.n_pos[b] += 1;
    st.emitted[b] += 1 + accept;
    if (st.dbg_conf) st.dbg_conf[b] = c;
    if (st.dbg_xb) { st.dbg_xb[b] = xb; st.dbg_xd[b] = xd; }
    if (st.presence && accept) atomicOr(st.presence + (size_t)b * st.presence_w + (xd >> 5), 1u << (xd & 31));
    if (st.samp_step && b == 0) st.samp_step[0] += 1;
}

// The residual term of the residual MLP compressor (App. A.1): x[r] = a + b,
// the two slot embeddings of pair r (E rows, x_pad for PAD = -1); the W2
// projection then adds W2 SiLU(W1 [a;b]).  An id outside [-1, V) (never
// produced: the host validates ids) contributes zeros.  grid rows, any block.
template <typename T>
__global__ void pair_sum_kernel(const void* E, const void* pad, const int32_t* tok, int tok_ld, int V, int H,
                                float* x) {
    pdl_launch();
    pdl_wait();
    const int r = blockIdx.x;
    const int t0 = tok[(size_t)r * tok_ld], t1 = tok[(size_t)r * tok_ld + 1];
    for (int k = threadIdx.x; k < H; k += blockDim.x) {
        const float a = t0 < 0 ? ldw<T>(pad, k) : t0 < V ? ldw<T>(E, (size_t)t0 * H + k) : 0.f;
        const float b = t1 < 0 ? ldw<T>(pad, k) : t1 < V ? ldw<T>(E, (size_t)t1 * H + k) : 0.f;
        x[(size_t)r * H + k] = a + b;
    }
}

// Regular decoding (the paper's baseline, Sec. 4): the backbone input is the
// token's own embedding, x[b] = E[tok[b * ld]], with no compressor.  Also
// zeroes the argmax keys of the step.  An id outside [0, V) (never produced:
// the host validates ids) gives a zero row instead of an out-of-range read.
// grid B, any block size.
template <typename T>
__global__ void embed_kernel(const void* E, const int32_t* tok, int ld, int V, int H, float* x,
                             unsigned long long* zero, int zero_n) {
    pdl_launch();
    pdl_wait();
    const int b = blockIdx.x;
    if (b == 0)
        for (int i = threadIdx.x; i < zero_n; i += blockDim.x) zero[i] = 0ull;
    const int t = tok[(size_t)b * ld];
    const bool ok = t >= 0 && t < V;
    for (int k = threadIdx.x; k < H; k += blockDim.x)
        x[(size_t)b * H + k] = ok ? ldw<T>(E, (size_t)t * H + k) : 0.f;
}

}  // namespace pipo
