// The whole pair-decode step as one persistent kernel (sm_103a).
//
// One CTA per SM, cooperative launch (all CTAs resident).  The step is a list
// of phases (GEMV, attention, acceptance) separated by grid barriers.  Weights
// never depend on activations, so every warp streams its share of ALL weight
// phases through a private ring of bulk-copy (TMA) stages in shared memory:
// while the CTA waits at a barrier, or works on an attention phase, the ring
// already holds the next weight phase's first bytes.  HBM keeps streaming
// across layer boundaries and there is no kernel launch inside the step.
//
// GEMV phases use the same work split as gemv_tma_kernel (CTA: balanced unit
// range; warp: balanced chunk range; deterministic boundary partials).
// Attention phases split each (sequence, kv head) over S CTAs; partials go to
// global scratch and the last CTA of the group merges them in split order.
// All waits are bounded and record an error code instead of hanging.
#pragma once

#include "attn_cluster.cuh"
#include "gemv_stream.cuh"
#include "tma.cuh"

namespace pipo {

#ifndef PIPO_MK_WARPS
#define PIPO_MK_WARPS 16
#endif
constexpr int kMkWarps = PIPO_MK_WARPS;
constexpr int kMkThreads = kMkWarps * 32;
constexpr int kMkStageChunks = 8;  // 4 KB stages
constexpr int kMkStageBytes = kMkStageChunks * 512;
constexpr int kMkStages = 2;       // per warp: 16 warps x 2 x 4 KB = 128 KB ring per SM

constexpr unsigned kErrBarrierTimeout = 2u;

enum PhaseType : int { PH_GEMV = 0, PH_ATTN = 1, PH_ACCEPT = 2, PH_ADVANCE = 3 };

struct AttnPhase {
    const float* qkv;
    int ld_qkv;
    KVView kv;
    const int32_t* n_pos;
    const float* rope;
    float* out;
    float scale;
    float* part_o;      // [B][n_q][S][DH]
    float* part_ml;     // [B][n_q][S][2]
    unsigned* counters; // [B][n_kv], zero between phases
    int S;
    int B;
};

struct AcceptPhase {
    const float* t;
    const void* W2;
    int H;
    float tau;
    int force;
    StepState st;
    const float* hb;
    const float* hd;
    int B;
};

struct Phase {
    int type;
    int ru;  // GEMV rows per unit
    GemvParams g;
    AttnPhase a;
    AcceptPhase c;
};

__device__ __forceinline__ unsigned ld_acquire(const unsigned* p) {
    unsigned v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

// Grid barrier on a counter zeroed before the launch: wait until `target`
// CTAs have arrived.  Bounded: on timeout the error word is set.
__device__ __forceinline__ void grid_sync(unsigned* ctr, unsigned target) {
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        atomicAdd(ctr, 1u);
        int spins = 0;
        while (ld_acquire(ctr) < target) {
            if (++spins > (1 << 24)) {
                atomicOr(&g_pipo_error, kErrBarrierTimeout);
                break;
            }
            __nanosleep(32);
        }
        __threadfence();
    }
    __syncthreads();
}

// Per-warp weight ring: the producer cursor (lane 0) runs ahead through the
// GEMV phases of the step, at most kMkStages stages ahead of the consumer.
struct WarpRing {
    unsigned char* base;
    uint64_t* bars;
    int issued, consumed;  // stage sequence numbers
    int pp, pi;            // producer: phase and stage within it
};

// this warp's chunk range of GEMV phase `ph` in this CTA
__device__ __forceinline__ void gemv_range(const Phase& ph, int esz, int& c0, int& c1, const char*& src) {
    const GemvParams& p = ph.g;
    const int cpr = p.K * esz / 512;
    const int cpu = cpr * ph.ru;
    const int u0 = (int)((long long)blockIdx.x * p.N / gridDim.x);
    const int u1 = (int)((long long)(blockIdx.x + 1) * p.N / gridDim.x);
    const int C = (u1 - u0) * cpu;
    const int warp = threadIdx.x >> 5;
    c0 = (int)((long long)warp * C / kMkWarps);
    c1 = (int)((long long)(warp + 1) * C / kMkWarps);
    src = static_cast<const char*>(p.W) + ((size_t)u0 * cpu + c0) * 512;
}

// lane 0: issue the next weight stage in step order, if any
__device__ __forceinline__ void ring_issue_next(WarpRing& r, const Phase* phases, int nph, int esz) {
    while (r.pp < nph) {
        const Phase& ph = phases[r.pp];
        if (ph.type == PH_GEMV) {
            int c0, c1;
            const char* src;
            gemv_range(ph, esz, c0, c1, src);
            const int nst = (c1 - c0 + kMkStageChunks - 1) / kMkStageChunks;
            if (r.pi < nst) {
                const int first = r.pi * kMkStageChunks;
                const int n = min(kMkStageChunks, (c1 - c0) - first);
                const int slot = r.issued % kMkStages;
                mbar_arrive_expect_tx(r.bars + slot, (uint32_t)n * 512u);
                bulk_g2s(r.base + (size_t)slot * kMkStageBytes, src + (size_t)first * 512, (uint32_t)n * 512u,
                         r.bars + slot);
                ++r.issued;
                ++r.pi;
                return;
            }
        }
        ++r.pp;
        r.pi = 0;
    }
}

template <typename T, int NB, int RU>
__device__ __forceinline__ bool mk_gemv_phase(const Phase& ph, WarpRing& r, const Phase* phases, int nph, float* xs,
                                              int* head_unit, int* tail_unit, int* head_fin, float* hv, float* tv,
                                              float* rv, int* rr) {
    const GemvParams& p = ph.g;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int cpr = p.K * (int)sizeof(T) / 512;
    const int u0 = (int)((long long)blockIdx.x * p.N / gridDim.x);
    int c0, c1;
    const char* src;
    gemv_range(ph, (int)sizeof(T), c0, c1, src);
    const int nst = (c1 - c0 + kMkStageChunks - 1) / kMkStageChunks;
    // shared scratch views with the compile-time shapes of the helpers
    auto& head_u = *reinterpret_cast<int(*)[kMkWarps]>(head_unit);
    auto& tail_u = *reinterpret_cast<int(*)[kMkWarps]>(tail_unit);
    auto& head_f = *reinterpret_cast<int(*)[kMkWarps]>(head_fin);
    auto& head_v = *reinterpret_cast<float(*)[kMkWarps][RU][NB]>(hv);
    auto& tail_v = *reinterpret_cast<float(*)[kMkWarps][RU][NB]>(tv);
    auto& red_v = *reinterpret_cast<float(*)[kMkWarps][NB]>(rv);
    auto& red_r = *reinterpret_cast<int(*)[kMkWarps][NB]>(rr);

    if (p.zero_ptr && blockIdx.x == 0)
        for (int i = threadIdx.x; i < p.zero_n; i += blockDim.x) p.zero_ptr[i] = 0ull;
    if (lane == 0) { head_f[warp] = 0; head_u[warp] = -1; tail_u[warp] = -1; }
    stage_input_fast<T, NB, kMkThreads>(p, xs, 0, min(NB, p.B));

    WarpRows<T, NB, RU> wr;
    wr.init(&p, xs, cpr, u0, c0, c1, 0, min(NB, p.B));
    bool ok = true;
    for (int i = 0; i < nst; ++i) {
        const int slot = r.consumed % kMkStages;
        ok = __all_sync(0xffffffffu, mbar_wait(r.bars + slot, (uint32_t)((r.consumed / kMkStages) & 1), 41, r.consumed));
        if (!ok) break;
        const unsigned char* sp = r.base + (size_t)slot * kMkStageBytes + lane * 16;
        const int n = min(kMkStageChunks, (c1 - c0) - i * kMkStageChunks);
        if (n == kMkStageChunks) {
#pragma unroll
            for (int ch = 0; ch < kMkStageChunks; ++ch)
                wr.chunk(*reinterpret_cast<const uint4*>(sp + ch * 512), head_u, head_f, head_v);
        } else {
            for (int ch = 0; ch < n; ++ch)
                wr.chunk(*reinterpret_cast<const uint4*>(sp + ch * 512), head_u, head_f, head_v);
        }
        ++r.consumed;
        __syncwarp();
        if (lane == 0) {
            fence_proxy_async();  // generic reads of the slot before its async overwrite
            ring_issue_next(r, phases, nph, (int)sizeof(T));
        }
        __syncwarp();
    }
    wr.finish(head_u, head_f, tail_u, head_v, tail_v);
    __syncthreads();
    finish_block<T, NB, RU, kMkWarps>(p, wr, head_u, head_f, tail_u, head_v, tail_v, red_v, red_r);
    return ok;
}

// Attention over one split of one (sequence, kv head) with all warps of the
// CTA; RoPE + append of the new entry as in attn_cluster_kernel.  Writes the
// split's (m, l, o) partial; the last split to finish merges.
template <typename T, int DH, int G>
__device__ __forceinline__ void mk_attn_phase(const AttnPhase& a, float* smem) {
    constexpr int LPE = DH / 8, EPW = 32 / LPE, kU = 2, NW = kMkWarps, STEP = NW * EPW;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int li = lane % LPE, slot = lane / LPE;
    const int n_kv = a.kv.n_kv, n_q = n_kv * G, S = a.S;
    float* wm = smem;                  // [NW][G]
    float* wl = wm + NW * G;           // [NW][G]
    float* wo = wl + NW * G;           // [NW][G][DH]
    __shared__ bool last;
    const T* Kb = static_cast<const T*>(a.kv.K);
    const T* Vb = static_cast<const T*>(a.kv.V);
    const int units = a.B * n_kv * S;
    for (int u = blockIdx.x; u < units; u += gridDim.x) {
        const int b = u / (n_kv * S), g = (u / S) % n_kv, s = u % S;
        const int n = a.n_pos[b], len = n + 1;
        const int chunk = (len + S - 1) / S;
        const int j0 = s * chunk, j1 = min(len, j0 + chunk), jc = min(j1, n);
        const float* qrow = a.qkv + (size_t)b * a.ld_qkv;
        const int jwb = j0 + warp * EPW;
        // first keys/values (independent of q) in flight before q and RoPE
        KV8<T> kk[kU], vv[kU];
#pragma unroll
        for (int uu = 0; uu < kU; ++uu) {
            const int j = jwb + slot + uu * STEP;
            const size_t off = kv_off<T, DH>(a.kv, b, j < jc ? j : 0, g) + li * 8;
            kk[uu].load(Kb + off);
            vv[uu].load(Vb + off);
        }
        float4 rope_cs[4];
        rope_load<DH>(rope_cs, li, n, a.rope);
        float q[G][8];
#pragma unroll
        for (int hh = 0; hh < G; ++hh) {
            const float4* qp = reinterpret_cast<const float4*>(qrow + (size_t)(g * G + hh) * DH + li * 8);
            const float4 x0 = qp[0], x1 = qp[1];
            q[hh][0] = x0.x; q[hh][1] = x0.y; q[hh][2] = x0.z; q[hh][3] = x0.w;
            q[hh][4] = x1.x; q[hh][5] = x1.y; q[hh][6] = x1.z; q[hh][7] = x1.w;
            rope8<DH>(q[hh], li, rope_cs);
#pragma unroll
            for (int e = 0; e < 8; ++e) q[hh][e] *= a.scale;
        }
        float m[G], l[G], o[G][8];
#pragma unroll
        for (int hh = 0; hh < G; ++hh) {
            m[hh] = -INFINITY;
            l[hh] = 0.f;
#pragma unroll
            for (int e = 0; e < 8; ++e) o[hh][e] = 0.f;
        }
        for (int jb = jwb; jb < jc; jb += kU * STEP) {
            if (jb != jwb) {
#pragma unroll
                for (int uu = 0; uu < kU; ++uu) {
                    const int j = jb + slot + uu * STEP;
                    const size_t off = kv_off<T, DH>(a.kv, b, j < jc ? j : 0, g) + li * 8;
                    kk[uu].load(Kb + off);
                    vv[uu].load(Vb + off);
                }
            }
            float sc[kU][G];
#pragma unroll
            for (int uu = 0; uu < kU; ++uu) {
                float kf[8];
                kk[uu].to_float(kf);
#pragma unroll
                for (int hh = 0; hh < G; ++hh) {
                    float d = 0.f;
#pragma unroll
                    for (int e = 0; e < 8; ++e) d += q[hh][e] * kf[e];
#pragma unroll
                    for (int off = LPE / 2; off > 0; off >>= 1) d += __shfl_xor_sync(0xffffffffu, d, off, LPE);
                    sc[uu][hh] = (jb + slot + uu * STEP < jc) ? d : -INFINITY;
                }
            }
#pragma unroll
            for (int hh = 0; hh < G; ++hh) {
                float mx = m[hh];
#pragma unroll
                for (int uu = 0; uu < kU; ++uu) mx = fmaxf(mx, sc[uu][hh]);
                if (mx == -INFINITY) continue;
                const float corr = expf(m[hh] - mx);
                l[hh] *= corr;
#pragma unroll
                for (int e = 0; e < 8; ++e) o[hh][e] *= corr;
                m[hh] = mx;
            }
#pragma unroll
            for (int uu = 0; uu < kU; ++uu) {
                float vf[8];
                vv[uu].to_float(vf);
#pragma unroll
                for (int hh = 0; hh < G; ++hh) {
                    const float pj = (sc[uu][hh] == -INFINITY) ? 0.f : expf(sc[uu][hh] - m[hh]);
                    l[hh] += pj;
#pragma unroll
                    for (int e = 0; e < 8; ++e) o[hh][e] += pj * vf[e];
                }
            }
        }
        if (n >= j0 && n < j1 && warp == 0) {  // the new entry: rotate, round, append, attend
            const float* kp = qrow + (size_t)(n_q + g) * DH + li * 8;
            const float* vp = qrow + (size_t)(n_q + n_kv + g) * DH + li * 8;
            float kf[8], vf[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) { kf[e] = kp[e]; vf[e] = vp[e]; }
            rope8<DH>(kf, li, rope_cs);
            const size_t off = kv_off<T, DH>(a.kv, b, n, g) + li * 8;
            T* Kw = static_cast<T*>(a.kv.K) + off;
            T* Vw = static_cast<T*>(a.kv.V) + off;
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                const T kt = from_f<T>(kf[e]), vt = from_f<T>(vf[e]);
                if (slot == 0) { Kw[e] = kt; Vw[e] = vt; }
                kf[e] = to_f(kt);
                vf[e] = to_f(vt);
            }
#pragma unroll
            for (int hh = 0; hh < G; ++hh) {
                float d = 0.f;
#pragma unroll
                for (int e = 0; e < 8; ++e) d += q[hh][e] * kf[e];
#pragma unroll
                for (int off2 = LPE / 2; off2 > 0; off2 >>= 1) d += __shfl_xor_sync(0xffffffffu, d, off2, LPE);
                if (slot != 0) continue;
                const float mx = fmaxf(m[hh], d);
                const float corr = expf(m[hh] - mx);
                const float pj = expf(d - mx);
                l[hh] = l[hh] * corr + pj;
#pragma unroll
                for (int e = 0; e < 8; ++e) o[hh][e] = o[hh][e] * corr + pj * vf[e];
                m[hh] = mx;
            }
        }
        // merge the lane groups of each warp, then the warps (shared memory)
#pragma unroll
        for (int hh = 0; hh < G; ++hh) {
#pragma unroll
            for (int off = LPE; off < 32; off <<= 1) {
                const float m2 = __shfl_xor_sync(0xffffffffu, m[hh], off);
                const float l2 = __shfl_xor_sync(0xffffffffu, l[hh], off);
                const float mx = fmaxf(m[hh], m2);
                const float f1 = (m[hh] == -INFINITY) ? 0.f : expf(m[hh] - mx);
                const float f2 = (m2 == -INFINITY) ? 0.f : expf(m2 - mx);
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    const float o2 = __shfl_xor_sync(0xffffffffu, o[hh][e], off);
                    o[hh][e] = o[hh][e] * f1 + o2 * f2;
                }
                l[hh] = l[hh] * f1 + l2 * f2;
                m[hh] = mx;
            }
            if (slot == 0) {
#pragma unroll
                for (int e = 0; e < 8; ++e) wo[(warp * G + hh) * DH + li * 8 + e] = o[hh][e];
                if (li == 0) { wm[warp * G + hh] = m[hh]; wl[warp * G + hh] = l[hh]; }
            }
        }
        __syncthreads();
        for (int i = threadIdx.x; i < G * DH; i += blockDim.x) {
            const int hh = i / DH, t = i % DH;
            float M = -INFINITY;
            for (int w = 0; w < NW; ++w) M = fmaxf(M, wm[w * G + hh]);
            float L = 0.f, Ov = 0.f;
            for (int w = 0; w < NW; ++w) {
                const float f = (wm[w * G + hh] == -INFINITY) ? 0.f : expf(wm[w * G + hh] - M);
                L += wl[w * G + hh] * f;
                Ov += wo[(w * G + hh) * DH + t] * f;
            }
            const int h = g * G + hh;
            const size_t pi = (size_t)(b * n_q + h) * S + s;
            a.part_o[pi * DH + t] = Ov;
            if (t == 0) { a.part_ml[pi * 2] = M; a.part_ml[pi * 2 + 1] = L; }
        }
        __threadfence();
        __syncthreads();
        if (threadIdx.x == 0) {
            const unsigned prev = atomicAdd(&a.counters[b * n_kv + g], 1u);
            last = (prev == (unsigned)S - 1);
        }
        __syncthreads();
        if (last) {
            // the S partials of the G heads to shared memory in one parallel pass
            // (they are contiguous: heads g*G .. g*G+G-1 of sequence b), then merge
            __threadfence();
            float* po = smem;                                  // [G][S][DH]
            float* pml = smem + (size_t)G * S * DH;            // [G][S][2]
            const size_t base = (size_t)(b * n_q + g * G) * S;
            const float4* src4 = reinterpret_cast<const float4*>(a.part_o + base * DH);
            for (int i = threadIdx.x; i < G * S * DH / 4; i += blockDim.x)
                reinterpret_cast<float4*>(po)[i] = __ldcg(src4 + i);
            for (int i = threadIdx.x; i < G * S * 2; i += blockDim.x) pml[i] = __ldcg(a.part_ml + base * 2 + i);
            __syncthreads();
            for (int i = threadIdx.x; i < G * DH; i += blockDim.x) {
                const int hh = i / DH, t = i % DH;
                float M = -INFINITY;
                for (int ss = 0; ss < S; ++ss) M = fmaxf(M, pml[(hh * S + ss) * 2]);
                float L = 0.f, Ov = 0.f;
                for (int ss = 0; ss < S; ++ss) {
                    const float ms = pml[(hh * S + ss) * 2];
                    const float f = (ms == -INFINITY) ? 0.f : expf(ms - M);
                    L += pml[(hh * S + ss) * 2 + 1] * f;
                    Ov += po[((size_t)hh * S + ss) * DH + t] * f;
                }
                a.out[(size_t)b * n_q * DH + (size_t)(g * G + hh) * DH + t] = Ov / L;
            }
            if (threadIdx.x == 0) a.counters[b * n_kv + g] = 0u;
        }
        __syncthreads();
    }
}

template <typename T>
__device__ __forceinline__ void mk_accept_phase(const AcceptPhase& c) {
    for (int b = blockIdx.x; b < c.B; b += gridDim.x) {
        float acc = 0.f;
        for (int k = threadIdx.x; k < c.H; k += blockDim.x) acc += ldw<T>(c.W2, k) * c.t[(size_t)b * c.H + k];
        acc = warp_sum(acc);
        __shared__ float red[32];
        const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
        if (lane == 0) red[warp] = acc;
        __syncthreads();
        const StepState& st = c.st;
        if (st.dbg_hb)
            for (int k = threadIdx.x; k < c.H; k += blockDim.x) {
                st.dbg_hb[(size_t)b * c.H + k] = c.hb[(size_t)b * c.H + k];
                st.dbg_hd[(size_t)b * c.H + k] = c.hd[(size_t)b * c.H + k];
            }
        if (threadIdx.x == 0) {
            float s = 0.f;
            for (int w = 0; w < (int)(blockDim.x >> 5); ++w) s += red[w];
            const float conf = 1.0f / (1.0f + expf(-s));
            const int accept = (c.force == 1) ? 1 : (c.force == 2) ? 0 : (conf >= c.tau ? 1 : 0);
            const int xb = argmax_row(st.am_b[b]), xd = argmax_row(st.am_d[b]);
            st.out_tokens[2 * b] = xb;
            st.out_tokens[2 * b + 1] = accept ? xd : -1;
            st.out_nacc[b] = accept;
            st.pending[2 * b] = xb;
            st.pending[2 * b + 1] = accept ? xd : -1;
            st.n_pos[b] += 1;
            st.emitted[b] += 1 + accept;
            if (st.dbg_conf) st.dbg_conf[b] = conf;
            if (st.dbg_xb) { st.dbg_xb[b] = xb; st.dbg_xd[b] = xd; }
        }
        __syncthreads();
    }
}

// smem: [ring: kMkWarps x kMkStages x 4 KB][bars][phase copy][staging area]
__host__ __device__ constexpr size_t mk_stage_offset() {
    return (((size_t)kMkWarps * kMkStages * kMkStageBytes + (size_t)kMkWarps * kMkStages * 8 + 2 * sizeof(Phase)) +
            127) / 128 * 128;
}
template <typename T, int NB, int DH, int G>
__global__ void __launch_bounds__(kMkThreads, 1) step_kernel(const Phase* __restrict__ phases, int nph, unsigned* bar_ctr) {
    extern __shared__ __align__(128) unsigned char smem_raw[];
    __shared__ int head_unit[kMkWarps], tail_unit[kMkWarps], head_fin[kMkWarps];
    __shared__ float head_val[kMkWarps * 2 * NB], tail_val[kMkWarps * 2 * NB];
    __shared__ float red_v[kMkWarps * NB];
    __shared__ int red_r[kMkWarps * NB];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    unsigned char* ring_all = smem_raw;
    uint64_t* bars_all = reinterpret_cast<uint64_t*>(smem_raw + (size_t)kMkWarps * kMkStages * kMkStageBytes);
    Phase* ph_s0 = reinterpret_cast<Phase*>(bars_all + kMkWarps * kMkStages);  // two descriptor buffers
    float* stage = reinterpret_cast<float*>(smem_raw + mk_stage_offset());

    WarpRing r;
    r.base = ring_all + (size_t)warp * kMkStages * kMkStageBytes;
    r.bars = bars_all + warp * kMkStages;
    r.issued = r.consumed = 0;
    r.pp = r.pi = 0;
    if (lane == 0) {
        for (int s = 0; s < kMkStages; ++s) mbar_init(r.bars + s, 1);
        mbar_init_fence();
        for (int s = 0; s < kMkStages; ++s) ring_issue_next(r, phases, nph, (int)sizeof(T));
    }
    __syncwarp();

    // descriptor of phase p in ph_s0[p & 1]; phase p+1's is loaded before the barrier
    auto load_desc = [&](int p) {
        if (p >= nph) return;
        const int* src = reinterpret_cast<const int*>(phases + p);
        int* dst = reinterpret_cast<int*>(ph_s0 + (p & 1));
        for (int i = threadIdx.x; i < (int)(sizeof(Phase) / 4); i += blockDim.x) dst[i] = src[i];
    };
    load_desc(0);
    bool ok = true;
    for (int p = 0; p < nph; ++p) {
        if (p > 0) grid_sync(bar_ctr, (unsigned)p * gridDim.x);
        else __syncthreads();
        const Phase& ph = ph_s0[p & 1];
        if (ph.type == PH_GEMV) {
            if (ph.ru == 2)
                ok &= mk_gemv_phase<T, NB, 2>(ph, r, phases, nph, stage, head_unit, tail_unit, head_fin, head_val,
                                              tail_val, red_v, red_r);
            else
                ok &= mk_gemv_phase<T, NB, 1>(ph, r, phases, nph, stage, head_unit, tail_unit, head_fin, head_val,
                                              tail_val, red_v, red_r);
        } else if (ph.type == PH_ATTN) {
            mk_attn_phase<T, DH, G>(ph.a, stage);
        } else if (ph.type == PH_ACCEPT) {
            mk_accept_phase<T>(ph.c);
        }
        __syncthreads();
        load_desc(p + 1);
    }
    // drain (bounded) any stage still in flight (only after a failed wait)
    if (lane == 0)
        while (r.consumed < r.issued) {
            mbar_wait(r.bars + (r.consumed % kMkStages), (uint32_t)((r.consumed / kMkStages) & 1), 42, r.consumed);
            ++r.consumed;
        }
    (void)ok;
}

}  // namespace pipo
