// Split-KV GQA flash-decode over the paged pair-KV cache, one thread-block
// cluster per (sequence, kv head) (sm_103a).
//
// Grid (CS, n_kv, rows), cluster (CS, 1, 1), 256 threads; CS (1 .. 16) is
// read from the cluster at run time, so one kernel serves every split.  CTA s
// of the cluster attends the G = n_q/n_kv query heads of its kv head over a
// contiguous slice of entries 0..n (n = entries before this step; entry n is
// this step's new key/value).  A decode step has one row per sequence; a
// prefill chunk has one row per (position, sequence), whose entries were
// appended before the launch (AttnParams::no_append).  Fused in:
//   * RoPE of q and of the new k (rotate-half, angle table cos/sin
//     [max_ctx][d_h/2] precomputed in fp64 and stored as fp32);
//   * the KV append: the CTA owning entry n rounds k, v to the cache type,
//     writes them to block table[b][n/64], slot n%64, and attends to them.
// Each lane covers 8 dims of one entry (d_h/8 lanes per entry), keys and
// values are read with 16-byte loads, kU entries in flight per lane group.
// The CS partials (m, l, o) are merged through distributed shared memory:
// each CTA merges a 1/CS slice of the output dims.  No global scratch.
//
// Unclustered form (FLAT): grid (S, n_kv, rows) without a cluster, S read
// from the grid, so a split count is not limited by cluster scheduling (at
// batch 1 about two CTAs per SM instead of one cluster of 8 per kv head).
// Each CTA writes its partial to global scratch, and the last CTA of a
// (row, kv head) to arrive merges the S partials in split order (L2 reads).
//
// Programmatic dependent launch: the first keys/values of the slice are loaded
// before griddepcontrol.wait (the cache entries < n and n itself come from
// earlier steps); q and the new k, v are read after it.
#pragma once

#include <cooperative_groups.h>

#include "kernels.cuh"
#include "tma.cuh"

namespace pipo {

namespace cg = cooperative_groups;

template <typename T> struct KV8;  // 8 consecutive cache elements
template <> struct KV8<__nv_bfloat16> {
    uint4 v;
    __device__ __forceinline__ void load(const __nv_bfloat16* p) { v = ldg_cg(p); }
    __device__ __forceinline__ void load_s(const unsigned char* p) { v = *reinterpret_cast<const uint4*>(p); }
    __device__ __forceinline__ void zero() { v = make_uint4(0, 0, 0, 0); }
    __device__ __forceinline__ void to_float(float (&f)[8]) const {
        f[0] = bf_lo(v.x); f[1] = bf_hi(v.x); f[2] = bf_lo(v.y); f[3] = bf_hi(v.y);
        f[4] = bf_lo(v.z); f[5] = bf_hi(v.z); f[6] = bf_lo(v.w); f[7] = bf_hi(v.w);
    }
};
template <> struct KV8<float> {
    uint4 a, b;
    __device__ __forceinline__ void load(const float* p) {
        a = ldg_cg(p);
        b = ldg_cg(p + 4);
    }
    __device__ __forceinline__ void load_s(const unsigned char* p) {
        a = *reinterpret_cast<const uint4*>(p);
        b = *reinterpret_cast<const uint4*>(p + 16);
    }
    __device__ __forceinline__ void zero() { a = b = make_uint4(0, 0, 0, 0); }
    __device__ __forceinline__ void to_float(float (&f)[8]) const {
        f[0] = __uint_as_float(a.x); f[1] = __uint_as_float(a.y); f[2] = __uint_as_float(a.z); f[3] = __uint_as_float(a.w);
        f[4] = __uint_as_float(b.x); f[5] = __uint_as_float(b.y); f[6] = __uint_as_float(b.z); f[7] = __uint_as_float(b.w);
    }
};

struct AttnParams {
    const float* qkv;       // [rows][(n_q + 2 n_kv) * d_h] projections of this step (not rotated)
    int ld_qkv;
    KVView kv;
    const int32_t* n_pos;   // [nseq] entries before this step
    const float* rope;      // [max_ctx][d_h/2][2] (cos, sin)
    float* out;             // [rows][n_q * d_h]
    float scale;            // 1/sqrt(d_h)
    // Rows (grid z) map to sequences: row r is sequence r % nseq at position
    // n_pos[r % nseq] + r / nseq.  A decode step has one row per sequence
    // (rows == nseq); a prefill chunk has several consecutive positions of
    // every sequence, whose entries an earlier kernel has already appended
    // (no_append = 1): each row then attends to entries 0..n of the cache and
    // writes none.
    int nseq;
    int no_append;
    // unclustered form (attn_cluster_kernel<..., true>): the CTA partials
    // (m, l, o) of row r, query head h, split s at [(r * n_q + h) * S + s],
    // and one arrival counter per (row, kv head), zero between launches
    float* part_o;
    float* part_ml;
    unsigned* counters;
    // staged form (stage_max > 0): the CTA's whole slice of cached keys and
    // values is copied to shared memory (bulk copies, one per page run and
    // tensor) before the dependency wait; stage_max entries fit
    int stage_max;
};

// cos/sin of the 8 rotation pairs of lane slice li at position pos
template <int DH>
__device__ __forceinline__ void rope_load(float4 (&cs)[4], int li, int pos, const float* rope) {
    constexpr int LPE = DH / 8;
    const int i0 = (li % (LPE / 2)) * 8;  // pair index of dim e is i0 + e
    const float4* t = reinterpret_cast<const float4*>(rope + ((size_t)pos * (DH / 2) + i0) * 2);
#pragma unroll
    for (int e = 0; e < 4; ++e) cs[e] = t[e];
}

// rotate-half RoPE of the 8 dims [8*li, 8*li+8) of a d_h vector held as one
// 8-dim slice per lane; partner lane holds the other half (li ^ (LPE/2)).
template <int DH>
__device__ __forceinline__ void rope8(float (&x)[8], int li, const float4 (&cs)[4]) {
    constexpr int LPE = DH / 8;
    float other[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) other[e] = __shfl_xor_sync(0xffffffffu, x[e], LPE / 2, LPE);
    const bool first = li < LPE / 2;
#pragma unroll
    for (int e = 0; e < 8; e += 2) {
        const float4 t = cs[e / 2];  // cos(i0+e), sin(i0+e), cos(i0+e+1), sin(i0+e+1)
        if (first) {
            x[e] = x[e] * t.x - other[e] * t.y;
            x[e + 1] = x[e + 1] * t.z - other[e + 1] * t.w;
        } else {
            x[e] = x[e] * t.x + other[e] * t.y;
            x[e + 1] = x[e + 1] * t.z + other[e + 1] * t.w;
        }
    }
}

// Cluster merge of one output element from the CS (<= 16) partial softmax
// states (m, l, o) of cluster ranks 0..CS-1: every distributed-shared-memory
// load is issued before any is used, then the ranks are combined in order.
__device__ __forceinline__ float cluster_merge_elem(cg::cluster_group& cluster, const float* m_loc,
                                                    const float* l_loc, const float* o_loc, int CS) {
    float mr[16], lr[16], orr[16];
#pragma unroll
    for (int r = 0; r < 16; ++r)
        if (r < CS) {
            mr[r] = *cluster.map_shared_rank(m_loc, r);
            lr[r] = *cluster.map_shared_rank(l_loc, r);
            orr[r] = *cluster.map_shared_rank(o_loc, r);
        }
    float M = -INFINITY;
#pragma unroll
    for (int r = 0; r < 16; ++r)
        if (r < CS) M = fmaxf(M, mr[r]);
    float L = 0.f, Ov = 0.f;
#pragma unroll
    for (int r = 0; r < 16; ++r)
        if (r < CS) {
            const float f = (mr[r] == -INFINITY) ? 0.f : expf(mr[r] - M);
            L += lr[r] * f;
            Ov += orr[r] * f;
        }
    return Ov / L;
}

constexpr int kAttnWarps = 8;
constexpr int kAttnThreads = kAttnWarps * 32;
constexpr int kFlatMaxSplits = 64;  // splits of the unclustered form (its merge stages 2 x G x S floats)

#ifndef PIPO_ATTN_KU
#define PIPO_ATTN_KU 4
#endif

template <typename T, int DH, int G, bool FLAT = false>
__global__ void __launch_bounds__(kAttnThreads) attn_cluster_kernel(AttnParams p) {
    constexpr int LPE = DH / 8;        // lanes per entry
    constexpr int EPW = 32 / LPE;      // entries per warp step
    constexpr int kU = PIPO_ATTN_KU;   // warp steps in flight
    constexpr int NW = kAttnWarps;
    constexpr int STEP = NW * EPW;     // entries per CTA step
    __shared__ float sm_o[G][DH];
    __shared__ float sm_m[G], sm_l[G];
    __shared__ float wm[NW][G], wl[NW][G];
    __shared__ float wo[NW][G][DH];

    __shared__ int last_cta;
    __shared__ __align__(8) uint64_t kv_bar;
    extern __shared__ __align__(128) unsigned char kv_stage[];  // staged form: [stage_max][DH] keys, then values

    pdl_launch();
    PIPO_TR(const TraceT0 tr0 = trace_begin(); unsigned long long tr1 = 0, tr2 = 0, tr3 = 0, trq = 0, trk = 0, trc = 0;)
    const int s = FLAT ? (int)blockIdx.x : (int)cg::this_cluster().block_rank();
    const int CS = FLAT ? (int)gridDim.x : (int)cg::this_cluster().num_blocks();
    const int g = blockIdx.y, row = blockIdx.z;
    const int b = row % p.nseq;        // sequence: its block table and length
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int li = lane % LPE, slot = lane / LPE;
    const int n_kv = p.kv.n_kv, n_q = n_kv * G;
    const int n = p.n_pos[b] + row / p.nseq;  // cached entries before this row's; entry n is its own
    const int len = n + 1;
    const int chunk = (len + CS - 1) / CS;
    const int j0 = s * chunk, j1 = min(len, j0 + chunk);
    const int jc = min(j1, p.no_append ? len : n);  // read from the cache: [j0, jc)
    const T* Kb = static_cast<const T*>(p.kv.K);
    const T* Vb = static_cast<const T*>(p.kv.V);

    // staged form: the whole slice to shared memory, page run by page run
    const bool staged = p.stage_max > 0 && !p.no_append && jc - j0 <= p.stage_max;
    if (staged) {
        if (threadIdx.x == 0) {
            mbar_init(&kv_bar, 1);
            mbar_init_fence();
            const uint32_t eb = (uint32_t)(DH * sizeof(T));  // bytes of one entry (a multiple of 16)
            mbar_arrive_expect_tx(&kv_bar, (uint32_t)(jc > j0 ? jc - j0 : 0) * eb * 2u);
            unsigned char* vs = kv_stage + (size_t)p.stage_max * eb;
            for (int j = j0; j < jc;) {
                const int run = min(jc, (j / p.kv.page + 1) * p.kv.page) - j;  // entries left in this page
                const size_t off = kv_off<T, DH>(p.kv, b, j, g);
                bulk_g2s(kv_stage + (size_t)(j - j0) * eb, static_cast<const T*>(p.kv.K) + off, (uint32_t)run * eb, &kv_bar);
                bulk_g2s(vs + (size_t)(j - j0) * eb, static_cast<const T*>(p.kv.V) + off, (uint32_t)run * eb, &kv_bar);
                j += run;
            }
        }
        __syncthreads();  // the barrier's initialisation, before any other thread waits on it
    }
    // prefetch the first kU warp steps of keys/values (independent of this
    // step, unless the entries were appended by the kernel before)
    if (p.no_append) pdl_wait();
    KV8<T> kr[kU], vr[kU];
    const int jwb = j0 + warp * EPW;  // warp-uniform base; lane group entry = base + slot
    // loads are unconditional: an entry outside the slice reads entry 0 of the
    // sequence instead and is masked out of the softmax (a select on a load
    // result would make the thread wait for it)
    if (!staged) {
#pragma unroll
        for (int u = 0; u < kU; ++u) {
            const int j = jwb + slot + u * STEP;
            const size_t off = kv_off<T, DH>(p.kv, b, j < jc ? j : 0, g) + li * 8;
            kr[u].load(Kb + off);
            vr[u].load(Vb + off);
        }
    }
    float4 rope_cs[4];  // rotation of position n (static table)
    rope_load<DH>(rope_cs, li, n, p.rope);
    pdl_wait();
    PIPO_TR(tr1 = trace_now();)

    // q of the G heads, 8 dims per lane, rotated, pre-scaled
    float q[G][8];
    const float* qrow = p.qkv + (size_t)row * p.ld_qkv;
#pragma unroll
    for (int hh = 0; hh < G; ++hh) {
        const float4* qp = reinterpret_cast<const float4*>(qrow + (size_t)(g * G + hh) * DH + li * 8);
        const float4 a = qp[0], c = qp[1];
        q[hh][0] = a.x; q[hh][1] = a.y; q[hh][2] = a.z; q[hh][3] = a.w;
        q[hh][4] = c.x; q[hh][5] = c.y; q[hh][6] = c.z; q[hh][7] = c.w;
        rope8<DH>(q[hh], li, rope_cs);
#pragma unroll
        for (int e = 0; e < 8; ++e) q[hh][e] *= p.scale;
    }
    PIPO_TR(trq = trace_now() + (q[0][0] == 12345.f ? 1 : 0);)

    float m[G], l[G], o[G][8];
#pragma unroll
    for (int hh = 0; hh < G; ++hh) {
        m[hh] = -INFINITY;
        l[hh] = 0.f;
#pragma unroll
        for (int e = 0; e < 8; ++e) o[hh][e] = 0.f;
    }

    // one block of kU entries per lane group: scores, one max update, sums
    auto consume = [&](KV8<T> (&kk)[kU], KV8<T> (&vv)[kU], int jbase) {
        float sc[kU][G];
#pragma unroll
        for (int u = 0; u < kU; ++u) {
            float kf[8];
            kk[u].to_float(kf);
#pragma unroll
            for (int hh = 0; hh < G; ++hh) {
                float d = 0.f;
#pragma unroll
                for (int e = 0; e < 8; ++e) d += q[hh][e] * kf[e];
#pragma unroll
                for (int off = LPE / 2; off > 0; off >>= 1) d += __shfl_xor_sync(0xffffffffu, d, off, LPE);
                sc[u][hh] = (jbase + u * STEP < jc) ? d : -INFINITY;
            }
        }
#pragma unroll
        for (int hh = 0; hh < G; ++hh) {
            float mx = m[hh];
#pragma unroll
            for (int u = 0; u < kU; ++u) mx = fmaxf(mx, sc[u][hh]);
            if (mx == -INFINITY) continue;
            const float corr = expf(m[hh] - mx);
            l[hh] *= corr;
#pragma unroll
            for (int e = 0; e < 8; ++e) o[hh][e] *= corr;
            m[hh] = mx;
        }
#pragma unroll
        for (int u = 0; u < kU; ++u) {
            float vf[8];
            vv[u].to_float(vf);
#pragma unroll
            for (int hh = 0; hh < G; ++hh) {
                const float pj = (sc[u][hh] == -INFINITY) ? 0.f : expf(sc[u][hh] - m[hh]);
                l[hh] += pj;
#pragma unroll
                for (int e = 0; e < 8; ++e) o[hh][e] += pj * vf[e];
            }
        }
    };

    if (staged) {
        // the slice in shared memory: every lane group takes its entries in turn
        if (jc > j0) mbar_wait(&kv_bar, 0, 27, (unsigned)(jc - j0));
        PIPO_TR(trk = trace_now();)
        const size_t eb = (size_t)DH * sizeof(T);
        const unsigned char* ks = kv_stage + li * 8 * sizeof(T);
        const unsigned char* vs = kv_stage + (size_t)p.stage_max * eb + li * 8 * sizeof(T);
        for (int jb = jwb; jb < jc; jb += kU * STEP) {  // warp-uniform trip count
#pragma unroll
            for (int u = 0; u < kU; ++u) {
                const int j = jb + slot + u * STEP;
                const size_t e = (size_t)((j < jc ? j : j0) - j0) * eb;
                kr[u].load_s(ks + e);
                vr[u].load_s(vs + e);
            }
            consume(kr, vr, jb + slot);
        }
    } else {
        for (int jb = jwb; jb < jc; jb += kU * STEP) {  // warp-uniform trip count
            KV8<T> kn[kU], vn[kU];
#pragma unroll
            for (int u = 0; u < kU; ++u) {
                const int j = jb + slot + (kU + u) * STEP;
                const size_t off = kv_off<T, DH>(p.kv, b, j < jc ? j : 0, g) + li * 8;
                kn[u].load(Kb + off);
                vn[u].load(Vb + off);
            }
            consume(kr, vr, jb + slot);
#pragma unroll
            for (int u = 0; u < kU; ++u) { kr[u] = kn[u]; vr[u] = vn[u]; }
        }
    }

    // the new entry n: rotate k, round k and v to the cache type, append, attend
    // (the whole warp 0 runs it so that the shuffles see full warps; lane
    // group 0 writes the cache and keeps the entry in its softmax state)
    if (!p.no_append && n >= j0 && n < j1 && warp == 0) {
        const float* kp = qrow + (size_t)(n_q + g) * DH + li * 8;
        const float* vp = qrow + (size_t)(n_q + n_kv + g) * DH + li * 8;
        float kf[8], vf[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) { kf[e] = kp[e]; vf[e] = vp[e]; }
        rope8<DH>(kf, li, rope_cs);
        const size_t off = kv_off<T, DH>(p.kv, b, n, g) + li * 8;
        T* Kw = static_cast<T*>(p.kv.K) + off;
        T* Vw = static_cast<T*>(p.kv.V) + off;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const T kt = from_f<T>(kf[e]), vt = from_f<T>(vf[e]);
            if (slot == 0) {
                Kw[e] = kt;
                Vw[e] = vt;
            }
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

    PIPO_TR(tr2 = trace_now();)
    // merge the EPW lane groups of the warp (same dims, different entries)
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
            for (int e = 0; e < 8; ++e) wo[warp][hh][li * 8 + e] = o[hh][e];
            if (li == 0) { wm[warp][hh] = m[hh]; wl[warp][hh] = l[hh]; }
        }
    }
    __syncthreads();
    // merge the warps: CTA partial (m, l, o) in shared memory (FLAT: in the
    // global scratch)
    for (int i = threadIdx.x; i < G * DH; i += blockDim.x) {
        const int hh = i / DH, t = i % DH;
        float M = -INFINITY;
#pragma unroll
        for (int w = 0; w < NW; ++w) M = fmaxf(M, wm[w][hh]);
        float L = 0.f, Ov = 0.f;
#pragma unroll
        for (int w = 0; w < NW; ++w) {
            const float f = (wm[w][hh] == -INFINITY) ? 0.f : expf(wm[w][hh] - M);
            L += wl[w][hh] * f;
            Ov += wo[w][hh][t] * f;
        }
        if constexpr (FLAT) {
            const size_t pi = (size_t)(row * n_q + g * G + hh) * CS + s;
            p.part_o[pi * DH + t] = Ov;
            if (t == 0) { p.part_ml[pi * 2] = M; p.part_ml[pi * 2 + 1] = L; }
        } else {
            sm_o[hh][t] = Ov;
            if (t == 0) { sm_m[hh] = M; sm_l[hh] = L; }
        }
    }
    PIPO_TR(tr3 = trace_now();)
    if constexpr (FLAT) {
        // the last CTA of (row, kv head) to arrive merges the CS partials in split order
        __threadfence();
        __syncthreads();
        if (threadIdx.x == 0) {
            const unsigned prev = atomicAdd(p.counters + row * n_kv + g, 1u);
            last_cta = prev == (unsigned)(CS - 1);
            if (last_cta) p.counters[row * n_kv + g] = 0u;
        }
        __syncthreads();
        PIPO_TR(if (threadIdx.x == 0) trace_put(TR_ATTN_FLAT, tr0, tr0.clk, tr1, tr2, tr3);)
        if (!last_cta) return;
        __threadfence();
        // (m, l) of every split in one round of loads, the split weights per
        // head, then each output summed over the splits with 8 loads in flight
        float* ms = &wo[0][0][0];                 // [G][CS] (the warp partials are no longer needed)
        float* fs = ms + G * kFlatMaxSplits;      // [G][CS]
        for (int i = threadIdx.x; i < G * CS; i += blockDim.x) {
            const int hh = i / CS, r = i % CS;
            ms[hh * CS + r] = __ldcg(p.part_ml + ((size_t)(row * n_q + g * G + hh) * CS + r) * 2);
            fs[hh * CS + r] = __ldcg(p.part_ml + ((size_t)(row * n_q + g * G + hh) * CS + r) * 2 + 1);
        }
        __syncthreads();
        if (threadIdx.x < G) {
            const int hh = threadIdx.x;
            float M = -INFINITY;
            for (int r = 0; r < CS; ++r) M = fmaxf(M, ms[hh * CS + r]);
            float L = 0.f;
            for (int r = 0; r < CS; ++r) {
                const float f = (ms[hh * CS + r] == -INFINITY) ? 0.f : expf(ms[hh * CS + r] - M);
                L += fs[hh * CS + r] * f;
                fs[hh * CS + r] = f;
            }
            sm_l[hh] = L;
        }
        __syncthreads();
        for (int i = threadIdx.x; i < G * DH; i += blockDim.x) {
            const int hh = i / DH, t = i % DH;
            const float* po = p.part_o + (size_t)(row * n_q + g * G + hh) * CS * DH + t;
            float Ov = 0.f;
            for (int r0 = 0; r0 < CS; r0 += 8) {
                float ov[8];
#pragma unroll
                for (int u = 0; u < 8; ++u) ov[u] = __ldcg(po + (size_t)min(r0 + u, CS - 1) * DH);
#pragma unroll
                for (int u = 0; u < 8; ++u)
                    if (r0 + u < CS) Ov += ov[u] * fs[hh * CS + r0 + u];
            }
            p.out[(size_t)row * n_q * DH + (size_t)(g * G + hh) * DH + t] = Ov / sm_l[hh];
        }
        return;
    }
    cg::cluster_group cluster = cg::this_cluster();
    cluster.sync();
    PIPO_TR(trc = trace_now();)
    // cluster merge: CTA s finishes dims [s*G*DH/CS, (s+1)*G*DH/CS) of the G heads
    const int PER = (G * DH + CS - 1) / CS;
    for (int i = s * PER + threadIdx.x; i < min(G * DH, (s + 1) * PER); i += blockDim.x) {
        const int hh = i / DH, t = i % DH;
        p.out[(size_t)row * n_q * DH + (size_t)(g * G + hh) * DH + t] =
            cluster_merge_elem(cluster, &sm_m[hh], &sm_l[hh], &sm_o[hh][t], CS);
    }
    cluster.sync();  // keep every CTA's shared memory alive until all merges read it
    PIPO_TR(if (threadIdx.x == 0) {
        trace_put(TR_ATTN_CL, tr0, tr0.clk, tr1, tr2, tr3);
        trace_put(TR_ATTN_CL_EPI, tr0, tr1, trq, trk, tr2, trc);
    })
}

}  // namespace pipo
