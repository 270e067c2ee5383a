// Causal attention of a prefill chunk on the tensor cores (mma.sync
// m16n8k16, bf16 in, fp32 accumulate), each key and value read once per tile
// of query positions (sm_103a; bf16 cache, d_h = 128).
//
// A prefill chunk holds C consecutive positions n0 .. n0+C-1 of every
// sequence (row r = position r / B of sequence r % B, AttnParams's mapping),
// whose keys and values append_rows_kernel has already written.  One CTA per
// (tile of TP positions, kv head, sequence): its 32 query vectors (TP
// positions x the G query heads of the kv head, TP = 32 / G) attend causally
// over the entries 0 .. n0 + (the tile's last position).  A producer thread
// streams 16-entry groups of K and V into a ring of shared-memory stages with
// TMA tensor copies (the layout of attn_mma_kernel); each of the four compute
// warps owns 8 query vectors and consumes every group:
//   S = Q K^T   A rows 0..7: the bf16 part of the 8 rotated, pre-scaled
//               queries; rows 8..15: the bf16 remainder q - bf16(q).  The
//               score of query i is row i + row i+8 (fp32-accurate);
//   causal mask (entry e <= the query's position), online softmax per query;
//   O += P V    A = P in the same hi / lo row split; O of query i = row i +
//               row i+8.
// Against one decode-style CTA per row, the cache bytes a tile reads drop by
// the TP positions that share them.  Every wait is bounded (error word, shared
// abort flag).
#pragma once

#include "attn_mma.cuh"

namespace pipo {

constexpr int kPfWarps = 4;                       // compute warps
constexpr int kPfThreads = (kPfWarps + 1) * 32;   // + the producer warp
constexpr int kPfVec = 8 * kPfWarps;              // query vectors per CTA

constexpr size_t prefill_attn_smem() { return 1024 + (size_t)kMmaStages * kMmaStageBytes + 2 * kMmaStages * 8; }

// D += A B, all 16 rows of A
__device__ __forceinline__ void mma16(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3, uint32_t b0,
                                      uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// grid (ceil(C / TP), n_kv, nseq); C = positions of the chunk per sequence.
// tmK, tmV: this layer's K and V cache as [blocks * n_kv * page][d_h] bf16,
// boxes of 64 dims x 16 rows, 128-byte swizzle.
template <int G>
__global__ void __launch_bounds__(kPfThreads) attn_prefill_kernel(AttnParams p, int C,
                                                                  const __grid_constant__ CUtensorMap tmK,
                                                                  const __grid_constant__ CUtensorMap tmV) {
    static_assert(G == 1 || G == 2 || G == 4, "32 query vectors per CTA");
    constexpr int DH = kMmaDH;
    constexpr int NW = kPfWarps;
    constexpr int TP = kPfVec / G;  // positions per tile
    extern __shared__ __align__(1024) unsigned char pf_smem_raw[];
    __shared__ float qs[kPfVec][DH];  // rotated, pre-scaled queries of the tile (fp32)
    __shared__ int abort_flag;

    unsigned char* ring = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(pf_smem_raw) + 1023) & ~(uintptr_t)1023);
    uint64_t* full = reinterpret_cast<uint64_t*>(ring + (size_t)kMmaStages * kMmaStageBytes);
    uint64_t* empty = full + kMmaStages;

    pdl_launch();
    pdl_wait();  // the chunk's entries come from the kernel before
    const int tile = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int n_kv = p.kv.n_kv, n_q = n_kv * G;
    const int B = p.nseq;
    const int n0 = p.n_pos[b];                     // entries before the chunk
    const int jfirst = tile * TP;                  // first chunk position of the tile
    const int jlast = min(C, jfirst + TP) - 1;     // last one
    const int nent = n0 + jlast + 1;               // entries read: 0 .. n0 + jlast
    const int ngrp = (nent + kMmaRun - 1) / kMmaRun;

    if (threadIdx.x == 0) {
        prefetch_tmap(&tmK);
        prefetch_tmap(&tmV);
        for (int i = 0; i < kMmaStages; ++i) {
            mbar_init(full + i, 1);
            mbar_init(empty + i, NW);  // every compute warp consumes every group
        }
        abort_flag = 0;
        mbar_init_fence();
    }
    __syncthreads();

    if (warp == NW) {
        // ---- producer: whole 16-entry groups (a group never crosses a page)
        if (lane == 0) {
            int t = 0;
            for (; t < ngrp; ++t) {
                const int st = t % kMmaStages;
                if (t >= kMmaStages && (*(volatile int*)&abort_flag ||
                                        !mbar_wait(empty + st, (uint32_t)(((t / kMmaStages) & 1) ^ 1), 24, t))) {
                    *(volatile int*)&abort_flag = 1;
                    break;
                }
                const int e = t * kMmaRun;
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
            for (int i = max(0, t - kMmaStages); i < t; ++i)
                mbar_wait(full + (i % kMmaStages), (uint32_t)((i / kMmaStages) & 1), 25, i);
        }
        __syncwarp();
        return;
    }

    // ---- prologue: the tile's queries, rotated at their positions and pre-scaled
    const int ct = threadIdx.x;  // 0 .. 32*NW-1
    for (int i = ct; i < kPfVec * (DH / 2); i += 32 * NW) {
        const int v = i / (DH / 2), pr = i % (DH / 2);
        const int j = jfirst + v / G, h = v % G;
        float r1 = 0.f, r2 = 0.f;
        if (j < C) {
            const float* q = p.qkv + (size_t)(j * B + b) * p.ld_qkv + (size_t)(g * G + h) * DH;
            const float* rope = p.rope + (size_t)(n0 + j) * DH;  // [DH/2][2] cos, sin
            const float c = rope[2 * pr], sn = rope[2 * pr + 1];
            const float x1 = q[pr], x2 = q[pr + DH / 2];
            r1 = (x1 * c - x2 * sn) * p.scale;
            r2 = (x2 * c + x1 * sn) * p.scale;
        }
        qs[v][pr] = r1;
        qs[v][pr + DH / 2] = r2;
    }
    asm volatile("bar.sync 1, %0;" ::"n"(32 * NW) : "memory");  // compute warps only

    // A fragments of this lane's query (row gq: bf16 part, row gq + 8: remainder)
    const int gq = lane >> 2, tq = lane & 3;
    const int vq = warp * 8 + gq;
    const int jq = jfirst + vq / G;
    const bool qvalid = jq < C;
    const int qpos = n0 + jq;  // the query attends to entries 0 .. qpos
    uint32_t qa[DH / 16][4];
#pragma unroll
    for (int kc = 0; kc < DH / 16; ++kc) {
        const int d0 = kc * 16 + 2 * tq;
        const float x0 = qs[vq][d0], x1 = qs[vq][d0 + 1], x8 = qs[vq][d0 + 8], x9 = qs[vq][d0 + 9];
        qa[kc][0] = pack_bf16x2(x0, x1);
        qa[kc][1] = pack_bf16x2(bf16_rest(x0), bf16_rest(x1));
        qa[kc][2] = pack_bf16x2(x8, x9);
        qa[kc][3] = pack_bf16x2(bf16_rest(x8), bf16_rest(x9));
    }

    float o[DH / 8][4];
#pragma unroll
    for (int nd = 0; nd < DH / 8; ++nd) o[nd][0] = o[nd][1] = o[nd][2] = o[nd][3] = 0.f;
    float m_run = -INFINITY, l_run = 0.f;
    const int lm = lane >> 3, lr = lane & 7;  // ldmatrix: matrix index, row within it
    bool ok = true;

    for (int t = 0; t < ngrp; ++t) {
        const int st = t % kMmaStages;
        if (*(volatile int*)&abort_flag || !mbar_wait(full + st, (uint32_t)((t / kMmaStages) & 1), 26, t)) {
            *(volatile int*)&abort_flag = 1;
            ok = false;
            break;
        }
        const uint32_t kS = smem_u32(ring + (size_t)st * kMmaStageBytes);
        const uint32_t vS = kS + 2 * kMmaHalf;
        const int e0 = t * kMmaRun;

        // S = Q K^T: two n-tiles of 8 entries, 8 k-chunks of 16 dims
        float sacc[2][4];
#pragma unroll
        for (int nt = 0; nt < 2; ++nt) {
            sacc[nt][0] = sacc[nt][1] = sacc[nt][2] = sacc[nt][3] = 0.f;
#pragma unroll
            for (int kc2 = 0; kc2 < DH / 32; ++kc2) {
                uint32_t bk[4];
                ldsm_x4(bk, kS + mma_tile_off(nt * 8 + lr, 4 * kc2 + 2 * (lm >> 1) + (lm & 1)));
                mma16(sacc[nt], qa[kc2 * 2][0], qa[kc2 * 2][1], qa[kc2 * 2][2], qa[kc2 * 2][3], bk[0], bk[1]);
                mma16(sacc[nt], qa[kc2 * 2 + 1][0], qa[kc2 * 2 + 1][1], qa[kc2 * 2 + 1][2], qa[kc2 * 2 + 1][3],
                      bk[2], bk[3]);
            }
        }
        // score of (query vq, entry e0 + nt*8 + 2tq + j): bf16 row + remainder row, causal
        float sv[2][2];
#pragma unroll
        for (int nt = 0; nt < 2; ++nt)
#pragma unroll
            for (int j = 0; j < 2; ++j) {
                const int e = e0 + nt * 8 + 2 * tq + j;
                sv[nt][j] = (qvalid && e <= qpos) ? sacc[nt][j] + sacc[nt][2 + j] : -INFINITY;
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
            o[nd][2] *= corr;
            o[nd][3] *= corr;
        }
        // A fragments of P: k = entry; bf16 part in row gq, remainder in row gq + 8
        const uint32_t pa0 = pack_bf16x2(pv[0][0], pv[0][1]);
        const uint32_t pa1 = pack_bf16x2(bf16_rest(pv[0][0]), bf16_rest(pv[0][1]));
        const uint32_t pa2 = pack_bf16x2(pv[1][0], pv[1][1]);
        const uint32_t pa3 = pack_bf16x2(bf16_rest(pv[1][0]), bf16_rest(pv[1][1]));
        // O += P V: 16 n-tiles of 8 dims
#pragma unroll
        for (int nd2 = 0; nd2 < DH / 16; ++nd2) {
            uint32_t bv[4];
            ldsm_x4_t(bv, vS + mma_tile_off(lr + (lm & 1) * 8, nd2 * 2 + (lm >> 1)));
            mma16(o[nd2 * 2], pa0, pa1, pa2, pa3, bv[0], bv[1]);
            mma16(o[nd2 * 2 + 1], pa0, pa1, pa2, pa3, bv[2], bv[3]);
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(empty + st);  // this warp is done with the stage
    }

    // O of query vq, dims nd*8 + 2tq + j: bf16-part row + remainder row, normalised
    if (ok && qvalid) {
        const float inv = 1.0f / l_run;
        float* out = p.out + (size_t)(jq * B + b) * n_q * DH + (size_t)(g * G + vq % G) * DH;
#pragma unroll
        for (int nd = 0; nd < DH / 8; ++nd) {
            out[nd * 8 + 2 * tq] = (o[nd][0] + o[nd][2]) * inv;
            out[nd * 8 + 2 * tq + 1] = (o[nd][1] + o[nd][3]) * inv;
        }
    }
}

}  // namespace pipo
