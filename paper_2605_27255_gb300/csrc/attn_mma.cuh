// Split-KV GQA flash-decode on the tensor cores (mma.sync m16n8k16, bf16 in,
// fp32 accumulate) with the keys and values streamed into shared memory by
// bulk asynchronous copies (sm_103a; bf16 cache, d_h = 128).
//
// One thread-block cluster of CS CTAs per (row, kv head), as in
// attn_cluster_kernel (a row is a sequence in a decode step, a (position,
// sequence) of a prefill chunk): CTA s owns a contiguous slice of the entries
// 0..n (in a decode step entry n is the new key/value, which the CTA owning it
// rotates, rounds to bf16, appends and attends to; a prefill chunk's entries
// are in the cache already); the CS partial softmax states are merged through
// distributed shared memory.
//
// Per CTA: a producer thread copies aligned 16-entry groups of the slice into
// a ring of ST stages with TMA tensor copies (each compute warp owns
// ST / kMmaWarps of the stages, see mma_stage): the cache layer is a 2-D
// tensor of rows (block, kv head, slot) x d_h bf16, and a group is four boxes
// of 16 rows x 64 dims (K and V, two halves each) stored with the 128-byte
// swizzle, which keeps the ldmatrix reads free of bank conflicts.  Four
// compute warps take the groups in turn.  For a group:
//   S = Q K^T    A = Q: rows 0..G-1 the bf16 part of the G query heads of
//                this kv head (rotated, pre-scaled by 1/sqrt(d_h)), rows
//                G..2G-1 the bf16 remainder q - bf16(q); B = K from ldmatrix.
//                Score of head h = row h + row h+G (fp32-accurate).
//   online softmax per head on the accumulator fragments;
//   O += P V     A = P in the same hi / lo row split (the accumulator layout
//                of S is the A-fragment layout of P), B = V (ldmatrix.trans).
// About six warp instructions per cached entry, against ~160 for the
// CUDA-core kernels, so the kernel streams the cache at memory rate.
// Entries of a group outside the slice are masked (p = 0; the cache holds
// only finite values).  Every wait is bounded (error word, shared abort flag).
#pragma once

#include "attn_cluster.cuh"
#include "tma.cuh"

namespace pipo {

constexpr int kMmaDH = 128;
constexpr int kMmaRun = 16;                         // entries per group
constexpr int kMmaHalf = kMmaRun * 128;             // one box: 16 rows x 64 dims bf16 (2 KB)
constexpr int kMmaStageBytes = 4 * kMmaHalf;        // K (2 halves) + V (2 halves)
#ifndef PIPO_MMA_STAGES
#define PIPO_MMA_STAGES 10
#endif
#ifndef PIPO_MMA_WARPS
#define PIPO_MMA_WARPS 5
#endif
#ifndef PIPO_MMA_DEEP_STAGES
#define PIPO_MMA_DEEP_STAGES 20
#endif
constexpr int kMmaStages = PIPO_MMA_STAGES;
// the deep ring, for launches whose CTAs each have an SM of their own: a CTA
// whose slice has kMmaDeepStages groups of 16 entries or fewer issues every
// copy at its entry (a shallow ring re-issues a stage only after its first
// group is consumed, one more HBM round trip after the dependency wait)
constexpr int kMmaDeepStages = PIPO_MMA_DEEP_STAGES;
constexpr int kMmaWarps = PIPO_MMA_WARPS;           // compute warps (at least the G heads of a kv head)
constexpr int kMmaThreads = (kMmaWarps + 1) * 32;   // + the producer warp
static_assert(kMmaStages % kMmaWarps == 0 && kMmaDeepStages % kMmaWarps == 0,
              "every compute warp owns the same number of stages");

// Group t (16 cached entries) is consumed by compute warp t % kMmaWarps and
// travels through that warp's own stages in turn.  Each stage then has one
// consumer taking its groups in order, so a consumer never waits on a stage
// whose previous group is still in flight: mbarrier parity waits tell apart
// only the current and the preceding phase, and with one ring shared by all
// warps a fast warp could otherwise meet the parity of a phase two behind
// (copies need not land in the order they were issued).  The k-th group of a
// stage has phase k; the parity of group t is (t / ST) & 1 in a ring of ST
// stages.
template <int ST>
__device__ __forceinline__ int mma_stage(int t) {
    constexpr int spw = ST / kMmaWarps;  // stages of one compute warp
    return (t % kMmaWarps) * spw + (t / kMmaWarps) % spw;
}

// dynamic shared memory: the stage ring, its barriers, and the receive
// buffer of the cluster merge, one slot per CTA of the cluster (CS), each
// [G][DH] partial output then [G] maxima and [G] sums (fp32; G <= 4)
constexpr int kMmaRcvSlot = 4 * 128 + 8;  // floats per slot at G = 4 (smaller G use a prefix)
constexpr size_t mma_attn_smem(int cs = 8, int st = kMmaStages) {
    return 1024 + (size_t)st * kMmaStageBytes + 2 * st * 8 + (size_t)cs * kMmaRcvSlot * 4;
}

// The cluster merge pushes every CTA's partial softmax state into rank 0's
// receive buffer (distributed shared memory stores), and each CTA then
// arrives on rank 0's barrier with release semantics at cluster scope; rank
// 0 waits (acquire, cluster scope, bounded), merges in rank order and writes
// the output.  The other CTAs leave right after their arrival.
__device__ __forceinline__ void cluster_arrive_release() {
    asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait_acquire() {
    asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ void fence_acq_rel_cluster() { asm volatile("fence.acq_rel.cluster;" ::: "memory"); }
// arrive on the mbarrier at the same shared offset in the CTA of cluster rank `rank`
__device__ __forceinline__ void mbar_arrive_remote(uint64_t* bar, int rank) {
    asm volatile(
        "{\n .reg .b32 ra;\n mapa.shared::cluster.u32 ra, %0, %1;\n"
        " mbarrier.arrive.release.cluster.shared::cluster.b64 _, [ra];\n}" ::"r"(smem_u32(bar)),
        "r"(rank)
        : "memory");
}
__device__ __forceinline__ bool mbar_try_wait_cluster(uint64_t* bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n"
        " selp.u32 %0, 1, 0, p;\n}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}
// bounded wait (as mbar_wait) with cluster-scope acquire
__device__ __forceinline__ bool mbar_wait_cluster(uint64_t* bar, uint32_t parity, unsigned site, unsigned iter) {
    if (mbar_try_wait_cluster(bar, parity)) return true;
    const unsigned long long t0 = global_ns();
    for (;;) {
        for (int i = 0; i < 64; ++i)
            if (mbar_try_wait_cluster(bar, parity)) return true;
        if (global_ns() - t0 > kWaitNs) break;
    }
    atomicOr(&g_pipo_error, kErrWaitTimeout);
    if (atomicCAS(&g_pipo_error_info[0], 0u, site) == 0u) {
        g_pipo_error_info[1] = blockIdx.x + gridDim.x * (blockIdx.y + gridDim.y * blockIdx.z);
        g_pipo_error_info[2] = iter;
        g_pipo_error_info[3] = parity;
    }
    return false;
}

// byte offset of 8-dim chunk c (0..15) of row `row` (0..15) of a K or V tile:
// two 64-dim halves of 16 x 128 bytes, 16-byte chunks XOR-swizzled by row % 8
__device__ __forceinline__ uint32_t mma_tile_off(int row, int c) {
    return (uint32_t)((c >> 3) * kMmaHalf + row * 128 + (((c & 7) ^ (row & 7)) << 4));
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo_col, float hi_col) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(lo_col, hi_col);
    return *reinterpret_cast<const uint32_t*>(&h);
}

__device__ __forceinline__ float bf16_rest(float x) { return x - __bfloat162float(__float2bfloat16_rn(x)); }

__device__ __forceinline__ void ldsm_x4(uint32_t (&r)[4], uint32_t addr) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr));
}

__device__ __forceinline__ void ldsm_x4_t(uint32_t (&r)[4], uint32_t addr) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr));
}

// D += A B with A rows 8..15 zero (a1 = a3 = 0)
__device__ __forceinline__ void mma_rows8(float (&d)[4], uint32_t a0, uint32_t a2, uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(0u), "r"(a2), "r"(0u), "r"(b0), "r"(b1));
}

// tmK, tmV: this layer's K and V cache as [blocks * n_kv * page][d_h] bf16,
// boxes of 64 dims x 16 rows, 128-byte swizzle
// FLAT: no cluster; the grid's x dimension splits the entries (S = gridDim.x
// CTAs per (row, kv head)), each CTA writes its partial to the global
// scratch (AttnParams::part_o, part_ml) and the last of a (row, kv head) to
// arrive (AttnParams::counters) merges the S partials in split order: any
// split count, so that long caches fill the GPU evenly.
template <int G, bool FLAT = false, int ST = kMmaStages>
__global__ void __launch_bounds__(kMmaThreads) attn_mma_kernel(AttnParams p, const __grid_constant__ CUtensorMap tmK,
                                                               const __grid_constant__ CUtensorMap tmV) {
    static_assert(G == 1 || G == 2 || G == 4, "2G query rows must fit the 8 live MMA rows");
    static_assert(kMmaWarps >= G && kMmaWarps <= 16 && ST >= kMmaWarps && ST % kMmaWarps == 0,
                  "warps hold the new entry's heads; every warp owns the same number of stages");
    constexpr int DH = kMmaDH;
    constexpr int NW = kMmaWarps;
    constexpr int NP = NW + 1;  // softmax partials: one per compute warp + the new entry
    extern __shared__ __align__(1024) unsigned char am_smem_raw[];
    __shared__ float qs[G][DH];       // rotated, pre-scaled queries (fp32)
    __shared__ float kn_s[DH], vn_s[DH];  // the new entry, rounded to bf16
    __shared__ float wm[NP][G], wl[NP][G];
    __shared__ __align__(16) float wo_new[G][DH];  // the new entry's partial (partial NW); the compute
                                     // warps' partials go to their own first stage
    __shared__ int abort_flag;
    __shared__ __align__(8) uint64_t rcv_bar;  // rank 0: one arrival per CTA of the cluster
    PIPO_TR(__shared__ unsigned long long tr_s[3], tr_m[2], tr_f; const TraceT0 tr0 = trace_begin();)

    unsigned char* ring = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(am_smem_raw) + 1023) & ~(uintptr_t)1023);
    uint64_t* full = reinterpret_cast<uint64_t*>(ring + (size_t)ST * kMmaStageBytes);
    uint64_t* empty = full + ST;
    float* rcv = reinterpret_cast<float*>(empty + ST);  // [CS][kMmaRcvSlot] (rank 0's is used)
    // partial of compute warp w: [G][DH] floats at the start of its first stage
    auto wpart = [&](int w) { return reinterpret_cast<float*>(ring + (size_t)(w * (ST / NW)) * kMmaStageBytes); };

    pdl_launch();
    cg::cluster_group cluster = cg::this_cluster();
    const int s = FLAT ? (int)blockIdx.x : (int)cluster.block_rank();
    const int CS = FLAT ? (int)gridDim.x : (int)cluster.num_blocks();
    __shared__ int last_cta;
    const int g = blockIdx.y, row = blockIdx.z;
    const int b = row % p.nseq;        // sequence: its block table and length
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int n_kv = p.kv.n_kv, n_q = n_kv * G;
    const int n = p.n_pos[b] + row / p.nseq;  // cached entries before this row's; entry n is its own
    const int len = n + 1;
    const int chunk = (len + CS - 1) / CS;
    const int j0 = s * chunk, j1 = min(len, j0 + chunk);
    const int jc = min(j1, p.no_append ? len : n);  // read from the cache: [j0, jc)
    const int grp0 = j0 / kMmaRun;
    const int ngrp = jc > j0 ? (jc - 1) / kMmaRun - grp0 + 1 : 0;
    const bool owns_new = !p.no_append && n >= j0 && n < j1;

    if (threadIdx.x == 0) {
        prefetch_tmap(&tmK);
        prefetch_tmap(&tmV);
        for (int i = 0; i < ST; ++i) {
            mbar_init(full + i, 1);
            mbar_init(empty + i, 1);
        }
        abort_flag = 0;
        mbar_init(&rcv_bar, (uint32_t)CS);
        mbar_init_fence();
    }
    __syncthreads();
    // every thread: the first half of the cluster barrier that orders rank 0's
    // barrier initialisation before the other CTAs' arrivals on it
    if (!FLAT && CS > 1) cluster_arrive_release();

    if (warp == NW) {
        // ---- producer: whole 16-entry groups (earlier steps wrote them, so
        // the copies start before the dependency wait, unless the kernel
        // before appended some of them)
        if (lane == 0) {
            if (p.no_append) pdl_wait();
            int t = 0;
            for (; t < ngrp; ++t) {
                const int st = mma_stage<ST>(t);
                if (t >= ST && (*(volatile int*)&abort_flag ||
                                        !mbar_wait(empty + st, (uint32_t)(((t / ST) & 1) ^ 1), 21, t))) {
                    *(volatile int*)&abort_flag = 1;
                    break;
                }
                const int e = (grp0 + t) * kMmaRun;  // a group never crosses a page
                const int blk = p.kv.table[(size_t)b * p.kv.blocks_per_seq + e / p.kv.page];
                const int trow = (blk * n_kv + g) * p.kv.page + e % p.kv.page;  // row of the cache tensor
                unsigned char* stg = ring + (size_t)st * kMmaStageBytes;
                mbar_arrive_expect_tx(full + st, (uint32_t)kMmaStageBytes);
                tma_load_2d(stg, &tmK, 0, trow, full + st);
                tma_load_2d(stg + kMmaHalf, &tmK, 64, trow, full + st);
                tma_load_2d(stg + 2 * kMmaHalf, &tmV, 0, trow, full + st);
                tma_load_2d(stg + 3 * kMmaHalf, &tmV, 64, trow, full + st);
            }
            // no copy into this CTA's shared memory may still be in flight at exit
            for (int i = max(0, t - ST); i < t; ++i)
                mbar_wait(full + mma_stage<ST>(i), (uint32_t)((i / ST) & 1), 22, i);
        }
        __syncwarp();
    } else {
        const int ct = threadIdx.x;  // 0 .. 32*NW-1
        // ---- prologue: rotated, pre-scaled q of the G heads; the new k, v
        pdl_wait();
        PIPO_TR(if (ct == 0) tr_s[0] = tr_f = trace_now();)
        const float* qrow = p.qkv + (size_t)row * p.ld_qkv;
        const float* rope = p.rope + (size_t)n * DH;  // [DH/2][2] cos, sin at position n
        for (int i = ct; i < (G + 1) * (DH / 2); i += 32 * NW) {
            const int h = i / (DH / 2), pr = i % (DH / 2);
            const float c = rope[2 * pr], sn = rope[2 * pr + 1];
            if (h < G) {
                const float* q = qrow + (size_t)(g * G + h) * DH;
                const float x1 = q[pr], x2 = q[pr + DH / 2];
                qs[h][pr] = (x1 * c - x2 * sn) * p.scale;
                qs[h][pr + DH / 2] = (x2 * c + x1 * sn) * p.scale;
            } else if (owns_new) {
                const float* k = qrow + (size_t)(n_q + g) * DH;
                const float x1 = k[pr], x2 = k[pr + DH / 2];
                kn_s[pr] = __bfloat162float(__float2bfloat16_rn(x1 * c - x2 * sn));
                kn_s[pr + DH / 2] = __bfloat162float(__float2bfloat16_rn(x2 * c + x1 * sn));
            }
        }
        if (owns_new)
            for (int d = ct; d < DH; d += 32 * NW)
                vn_s[d] = __bfloat162float(__float2bfloat16_rn(qrow[(size_t)(n_q + n_kv + g) * DH + d]));
        asm volatile("bar.sync 1, %0;" ::"n"(32 * NW) : "memory");  // compute warps only
        PIPO_TR(if (ct == 0) tr_s[1] = trace_now();)

        // the new entry: append it to the cache and make it partial NW
        if (owns_new) {
            const size_t off = kv_off<__nv_bfloat16, DH>(p.kv, b, n, g);
            __nv_bfloat16* Kw = static_cast<__nv_bfloat16*>(p.kv.K) + off;
            __nv_bfloat16* Vw = static_cast<__nv_bfloat16*>(p.kv.V) + off;
            for (int d = ct; d < DH; d += 32 * NW) {
                Kw[d] = __float2bfloat16_rn(kn_s[d]);
                Vw[d] = __float2bfloat16_rn(vn_s[d]);
            }
        }
        if (warp < G) {
            const int h = warp;
            float dsum = 0.f;
            if (owns_new) {  // uniform over the CTA: the shuffles below see whole warps
                for (int d = lane; d < DH; d += 32) dsum += qs[h][d] * kn_s[d];
                dsum = warp_sum(dsum);
            }
            for (int d = lane; d < DH; d += 32) wo_new[h][d] = owns_new ? vn_s[d] : 0.f;
            if (lane == 0) {
                wm[NW][h] = owns_new ? dsum : -INFINITY;
                wl[NW][h] = owns_new ? 1.f : 0.f;
            }
        }

        // ---- A fragments of Q: row r = lane / 4 (hi part for r < G, remainder for r < 2G)
        const int r = lane >> 2, tq = lane & 3;
        uint32_t qa[DH / 16][2];
#pragma unroll
        for (int kc = 0; kc < DH / 16; ++kc) {
#pragma unroll
            for (int half = 0; half < 2; ++half) {
                const int d0 = kc * 16 + half * 8 + 2 * tq;
                float x0 = 0.f, x1 = 0.f;
                if (r < G) {
                    x0 = qs[r][d0];
                    x1 = qs[r][d0 + 1];
                } else if (r < 2 * G) {
                    x0 = bf16_rest(qs[r - G][d0]);
                    x1 = bf16_rest(qs[r - G][d0 + 1]);
                }
                qa[kc][half] = pack_bf16x2(x0, x1);
            }
        }

        float o[DH / 8][4];
#pragma unroll
        for (int nd = 0; nd < DH / 8; ++nd) o[nd][0] = o[nd][1] = o[nd][2] = o[nd][3] = 0.f;
        float m_run = -INFINITY, l_run = 0.f;
        const int lm = lane >> 3, lr = lane & 7;  // ldmatrix: matrix index, row within it

        for (int t = warp; t < ngrp; t += NW) {
            const int st = mma_stage<ST>(t);
            if (*(volatile int*)&abort_flag || !mbar_wait(full + st, (uint32_t)((t / ST) & 1), 23, t)) {
                *(volatile int*)&abort_flag = 1;
                break;
            }
            PIPO_TR(if (ct == 0 && t == warp) tr_f = trace_now();)
            const uint32_t kS = smem_u32(ring + (size_t)st * kMmaStageBytes);
            const uint32_t vS = kS + 2 * kMmaHalf;
            const int e0 = (grp0 + t) * kMmaRun;
            const int lo = max(j0, e0) - e0, hi = min(jc, e0 + kMmaRun) - e0;  // valid entries [lo, hi)

            // S = Q K^T: two n-tiles of 8 entries, 8 k-chunks of 16 dims
            float sacc[2][4];
#pragma unroll
            for (int nt = 0; nt < 2; ++nt) {
                sacc[nt][0] = sacc[nt][1] = sacc[nt][2] = sacc[nt][3] = 0.f;
#pragma unroll
                for (int kc2 = 0; kc2 < DH / 32; ++kc2) {
                    uint32_t bk[4];
                    ldsm_x4(bk, kS + mma_tile_off(nt * 8 + lr, 4 * kc2 + 2 * (lm >> 1) + (lm & 1)));
                    mma_rows8(sacc[nt], qa[kc2 * 2][0], qa[kc2 * 2][1], bk[0], bk[1]);
                    mma_rows8(sacc[nt], qa[kc2 * 2 + 1][0], qa[kc2 * 2 + 1][1], bk[2], bk[3]);
                }
            }
            // score of (head r mod G, entry nt*8 + 2tq + j): bf16 row + remainder row
            float sv[2][2];
#pragma unroll
            for (int nt = 0; nt < 2; ++nt)
#pragma unroll
                for (int j = 0; j < 2; ++j) {
                    const float v = sacc[nt][j] + __shfl_xor_sync(0xffffffffu, sacc[nt][j], 4 * G);
                    const int e = nt * 8 + 2 * tq + j;
                    sv[nt][j] = (e >= lo && e < hi) ? v : -INFINITY;
                }
            float rmax = fmaxf(fmaxf(sv[0][0], sv[0][1]), fmaxf(sv[1][0], sv[1][1]));
            rmax = fmaxf(rmax, __shfl_xor_sync(0xffffffffu, rmax, 1));
            rmax = fmaxf(rmax, __shfl_xor_sync(0xffffffffu, rmax, 2));
            const float m_new = fmaxf(m_run, rmax);
            const float corr = (m_run == -INFINITY) ? 0.f : expf(m_run - m_new);
            float pv[2][2], rsum = 0.f;
#pragma unroll
            for (int nt = 0; nt < 2; ++nt)
#pragma unroll
                for (int j = 0; j < 2; ++j) {
                    pv[nt][j] = (sv[nt][j] == -INFINITY) ? 0.f : expf(sv[nt][j] - m_new);
                    rsum += pv[nt][j];
                }
            rsum += __shfl_xor_sync(0xffffffffu, rsum, 1);
            rsum += __shfl_xor_sync(0xffffffffu, rsum, 2);
            l_run = l_run * corr + rsum;
            m_run = m_new;
#pragma unroll
            for (int nd = 0; nd < DH / 8; ++nd) {
                o[nd][0] *= corr;
                o[nd][1] *= corr;
            }
            // A fragments of P: k = entry; bf16 part in rows < G, remainder in rows G..2G-1
            uint32_t pa0, pa2;
            if (r < G) {
                pa0 = pack_bf16x2(pv[0][0], pv[0][1]);
                pa2 = pack_bf16x2(pv[1][0], pv[1][1]);
            } else if (r < 2 * G) {
                pa0 = pack_bf16x2(bf16_rest(pv[0][0]), bf16_rest(pv[0][1]));
                pa2 = pack_bf16x2(bf16_rest(pv[1][0]), bf16_rest(pv[1][1]));
            } else {
                pa0 = pa2 = 0u;
            }
            // O += P V: 16 n-tiles of 8 dims
#pragma unroll
            for (int nd2 = 0; nd2 < DH / 16; ++nd2) {
                uint32_t bv[4];
                ldsm_x4_t(bv, vS + mma_tile_off(lr + (lm & 1) * 8, nd2 * 2 + (lm >> 1)));
                mma_rows8(o[nd2 * 2], pa0, pa2, bv[0], bv[1]);
                mma_rows8(o[nd2 * 2 + 1], pa0, pa2, bv[2], bv[3]);
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(empty + st);  // this group's stage is free
        }

        PIPO_TR(if (ct == 0) tr_m[0] = trace_now();)
        // warp partial: O of head r = bf16-part row r + remainder row r + G,
        // into this warp's first stage (its groups are all consumed: no copy
        // lands in its stages any more)
        __syncwarp();
        float* wp = wpart(warp);
#pragma unroll
        for (int nd = 0; nd < DH / 8; ++nd)
#pragma unroll
            for (int j = 0; j < 2; ++j) {
                const float v = o[nd][j] + __shfl_xor_sync(0xffffffffu, o[nd][j], 4 * G);
                if (r < G) wp[r * DH + nd * 8 + 2 * tq + j] = v;
            }
        if (r < G && tq == 0) {
            wm[warp][r] = m_run;
            wl[warp][r] = l_run;
        }
    }
    __syncthreads();
    // merge the partials: this CTA's (m, l, o), then the cluster's at rank 0
    float* slot = nullptr;
    if (!FLAT && CS > 1) {
        cluster_wait_acquire();  // rank 0's receive barrier is initialised
        slot = cluster.map_shared_rank(rcv, 0) + (size_t)s * kMmaRcvSlot;
    }
    // four consecutive output dims per thread (16-byte stores, also into rank 0)
    for (int i4 = threadIdx.x; i4 < G * DH / 4; i4 += blockDim.x) {
        const int hh = (4 * i4) / DH, t = (4 * i4) % DH;
        float M = -INFINITY;
#pragma unroll
        for (int w = 0; w < NP; ++w) M = fmaxf(M, wm[w][hh]);
        float L = 0.f;
        float4 Ov = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int w = 0; w < NP; ++w) {
            const float f = (wm[w][hh] == -INFINITY) ? 0.f : expf(wm[w][hh] - M);
            L += wl[w][hh] * f;
            const float4 v = *reinterpret_cast<const float4*>(w < NW ? wpart(w) + hh * DH + t : &wo_new[hh][t]);
            Ov.x += v.x * f; Ov.y += v.y * f; Ov.z += v.z * f; Ov.w += v.w * f;
        }
        if (FLAT) {
            const size_t pi = (size_t)(row * n_q + g * G + hh) * CS + s;
            __stcg(reinterpret_cast<float4*>(p.part_o + pi * DH + t), Ov);
            if (t == 0) {
                p.part_ml[pi * 2] = M;
                p.part_ml[pi * 2 + 1] = L;
            }
        } else if (CS == 1) {
            const float il = 1.0f / L;
            *reinterpret_cast<float4*>(p.out + (size_t)row * n_q * DH + (size_t)(g * G + hh) * DH + t) =
                make_float4(Ov.x * il, Ov.y * il, Ov.z * il, Ov.w * il);
        } else {
            *reinterpret_cast<float4*>(slot + hh * DH + t) = Ov;
            if (t == 0) {
                slot[G * DH + hh] = M;
                slot[G * DH + G + hh] = L;
            }
        }
    }
    PIPO_TR(if (threadIdx.x == 0) tr_s[2] = trace_now();)
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
        if (!last_cta) return;
        __threadfence();
        // split weights per head in the (now idle) stage ring: ms [G][CS], fs [G][CS]
        float* ms = reinterpret_cast<float*>(ring);
        float* fs = ms + G * CS;
        for (int i = threadIdx.x; i < G * CS; i += blockDim.x) {
            const int hh = i / CS, r2 = i % CS;
            const size_t pi = (size_t)(row * n_q + g * G + hh) * CS + r2;
            ms[i] = __ldcg(p.part_ml + pi * 2);
            fs[i] = __ldcg(p.part_ml + pi * 2 + 1);
        }
        __syncthreads();
        if (threadIdx.x < G) {
            const int hh = threadIdx.x;
            float M = -INFINITY;
            for (int r2 = 0; r2 < CS; ++r2) M = fmaxf(M, ms[hh * CS + r2]);
            float L = 0.f;
            for (int r2 = 0; r2 < CS; ++r2) {
                const float f = (ms[hh * CS + r2] == -INFINITY) ? 0.f : expf(ms[hh * CS + r2] - M);
                L += fs[hh * CS + r2] * f;
                fs[hh * CS + r2] = f;  // weight of split r2
            }
            ms[hh * CS] = 1.0f / L;  // the maxima are no longer needed
        }
        __syncthreads();
        for (int i4 = threadIdx.x; i4 < G * DH / 4; i4 += blockDim.x) {
            const int hh = (4 * i4) / DH, t = (4 * i4) % DH;
            const float* po = p.part_o + (size_t)(row * n_q + g * G + hh) * CS * DH + t;
            float4 Ov = make_float4(0.f, 0.f, 0.f, 0.f);
            for (int r0 = 0; r0 < CS; r0 += 4) {
                float4 ov[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) ov[u] = __ldcg(reinterpret_cast<const float4*>(po + (size_t)min(r0 + u, CS - 1) * DH));
#pragma unroll
                for (int u = 0; u < 4; ++u)
                    if (r0 + u < CS) {
                        const float f = fs[hh * CS + r0 + u];
                        Ov.x += ov[u].x * f; Ov.y += ov[u].y * f; Ov.z += ov[u].z * f; Ov.w += ov[u].w * f;
                    }
            }
            const float il = ms[hh * CS];
            *reinterpret_cast<float4*>(p.out + (size_t)row * n_q * DH + (size_t)(g * G + hh) * DH + t) =
                make_float4(Ov.x * il, Ov.y * il, Ov.z * il, Ov.w * il);
        }
        return;
    }
    if (CS == 1) {
        PIPO_TR(if (threadIdx.x == 0) {
            trace_put(TR_ATTN_MMA, tr0, tr0.clk, tr_s[0], tr_f, tr_s[2]);
            trace_put(TR_ATTN_MMA_EPI, tr0, tr_s[0], tr_s[1], tr_m[0], tr_s[2], tr_s[2]);
        })
        return;
    }
    fence_acq_rel_cluster();  // this thread's stores into rank 0, before the arrival below
    __syncthreads();
    if (threadIdx.x == 0) mbar_arrive_remote(&rcv_bar, 0);
    if (s != 0) {
        PIPO_TR(if (threadIdx.x == 0) {
            trace_put(TR_ATTN_MMA, tr0, tr0.clk, tr_s[0], tr_f, tr_s[2]);
            trace_put(TR_ATTN_MMA_EPI, tr0, tr_s[0], tr_s[1], tr_m[0], tr_s[2], tr_s[2]);
        })
        return;  // rank 0 merges; nothing reads this CTA's shared memory
    }
    const bool got = mbar_wait_cluster(&rcv_bar, 0, 28, (unsigned)CS);
    PIPO_TR(if (threadIdx.x == 0) tr_m[1] = trace_now();)
    if (got) {
        for (int i4 = threadIdx.x; i4 < G * DH / 4; i4 += blockDim.x) {
            const int hh = (4 * i4) / DH, t = (4 * i4) % DH;
            float M = -INFINITY;
            for (int r2 = 0; r2 < CS; ++r2) M = fmaxf(M, rcv[r2 * kMmaRcvSlot + G * DH + hh]);
            float L = 0.f;
            float4 Ov = make_float4(0.f, 0.f, 0.f, 0.f);
            for (int r2 = 0; r2 < CS; ++r2) {
                const float* sl = rcv + r2 * kMmaRcvSlot;
                const float f = (sl[G * DH + hh] == -INFINITY) ? 0.f : expf(sl[G * DH + hh] - M);
                L += sl[G * DH + G + hh] * f;
                const float4 v = *reinterpret_cast<const float4*>(sl + hh * DH + t);
                Ov.x += v.x * f; Ov.y += v.y * f; Ov.z += v.z * f; Ov.w += v.w * f;
            }
            const float il = 1.0f / L;
            *reinterpret_cast<float4*>(p.out + (size_t)row * n_q * DH + (size_t)(g * G + hh) * DH + t) =
                make_float4(Ov.x * il, Ov.y * il, Ov.z * il, Ov.w * il);
        }
    }
    PIPO_TR(if (threadIdx.x == 0) {
        trace_put(TR_ATTN_MMA, tr0, tr0.clk, tr_s[0], tr_f, tr_s[2]);
        trace_put(TR_ATTN_MMA_EPI, tr0, tr_s[0], tr_s[1], tr_m[0], tr_s[2], tr_m[1]);
    })
}

}  // namespace pipo
