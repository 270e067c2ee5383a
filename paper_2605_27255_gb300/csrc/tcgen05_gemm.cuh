// Tensor-core (tcgen05 / TMEM) skinny GEMM for batched projections, sm_103a.
//
// For batches of two sequences and more the weight stream is fed to the
// 5th-generation tensor cores instead of CUDA cores (every weight byte then
// serves the whole batch at once).  Swap-AB: D[rows, B] = W[rows, K] .
// X[B, K]^T, so the 128 weight rows of a tile fill the MMA's M = 128 and the
// batch (padded to a multiple of 16) is its N.  Both operands are K-major bf16
// tiles loaded by TMA tensor copies with 128-byte swizzle into a
// shared-memory ring of ST stages (mbarrier completion; ST sized for two CTAs
// per SM, or for one in the deep variant).  One thread issues the
// copies, one thread issues tcgen05.mma.cta_group::1.kind::f16 (fp32
// accumulation in TMEM), and four warps read the accumulator back with
// tcgen05.ld for the epilogue.  A CTA owns one (128-row tile, K split).  When
// there are fewer tiles than SM slots, K is split over the CTAs of a thread-
// block cluster: each parks its partial tile in its own shared memory, and
// CTA s adds the rows of slice s over the cluster through distributed shared
// memory in split order (deterministic), then applies the epilogue to them.
//
// The activations enter as two bf16 parts, x = hi + lo with hi = bf16(x) and
// lo = bf16(x - hi) (prep_bf16_kernel, after the RMSNorm / gather of the GEMV
// input segments in fp32; or, in gemm_tcf_kernel below, converter warps inside
// the GEMM).  Both parts are B columns of the MMA (N = 2 * BH),
// so the bf16 weights meet an activation accurate to about 2^-17 relative:
// the weight stream is unchanged, only the (idle) tensor-core work doubles.
// The epilogue adds the two accumulator halves.  Every wait is bounded
// (error word + drain, no hang).
#pragma once

#include <cooperative_groups.h>
#include <cuda.h>

#include "kernels.cuh"
#include "tma.cuh"

namespace pipo {

constexpr int kTcM = 128;                   // weight rows per tile (MMA M)
constexpr int kTcBK = 64;                   // bf16 K per stage: 128-byte rows
constexpr int kTcThreads = 128;
constexpr int kTcABytes = kTcM * kTcBK * 2;  // 16 KB per stage
constexpr int kTcMaxSplits = 8;             // portable cluster size

// operand stages per batch width BH: about 100 KB of shared memory (two CTAs
// per SM), or, for grids of at most one CTA per SM, about 200 KB (deep): a
// lone CTA needs the deeper ring to keep enough weight bytes in flight
__host__ __device__ constexpr int tc_stages(int bh, bool deep = false) {
    return deep ? (bh <= 16 ? 10 : bh <= 32 ? 8 : bh <= 64 ? 6 : 4) : (bh <= 16 ? 5 : bh <= 32 ? 4 : bh <= 64 ? 3 : 2);
}

struct TcParams {
    int rows;            // W rows (output units * ru)
    int K;
    int B;               // sequences (batch columns < B are real)
    int ru;              // 1, or 2 (SwiGLU: gate/up rows interleaved)
    int epi;
    float* y;
    int ldy;
    const void* bias;    // bf16 [rows]
    unsigned long long* am;
    float* dbg;
    int ld_dbg;
    int splits;          // K splits per tile = cluster size (1 .. kTcMaxSplits)
};


// Shared-memory matrix descriptor: K-major, 128-byte swizzle (8-row groups of
// 128-byte rows, 1024 B apart), tile base 1024-byte aligned.
__device__ __forceinline__ uint64_t umma_desc_sw128(uint32_t saddr) {
    uint64_t d = 0;
    d |= (uint64_t)((saddr >> 4) & 0x3FFFu);  // start address (16-byte units)
    d |= (uint64_t)1 << 16;                    // leading byte offset (unused for swizzled K-major)
    d |= (uint64_t)(1024 >> 4) << 32;          // stride byte offset between 8-row groups
    d |= (uint64_t)1 << 46;                    // descriptor version
    d |= (uint64_t)2 << 61;                    // 128-byte swizzle
    return d;
}

// Instruction descriptor of kind::f16: D fp32, A and B bf16, both K-major.
__host__ __device__ constexpr uint32_t umma_idesc_bf16(int M, int N) {
    return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

__device__ __forceinline__ void umma_bf16(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(
            d_tmem),
        "l"(a), "l"(b), "r"(idesc), "r"(acc)
        : "memory");
}

// arrive on `bar` once all tcgen05.mma issued before it by this thread complete
__device__ __forceinline__ void umma_commit(uint64_t* bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
                 : "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

__device__ __forceinline__ void tmem_alloc(uint32_t* dst, uint32_t ncols) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(dst)), "r"(ncols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}

// 16 consecutive fp32 columns of this thread's TMEM lane
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float (&v)[16]) {
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
          "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// Epilogue of batch columns [c0, c0+16) of weight row `row` (thread = TMEM
// lane; quad = the warp's TMEM lane quadrant).  All threads of the warp call
// it (the SwiGLU pairing shuffles).
template <int BH>
__device__ __forceinline__ void tc_epilogue16(const TcParams& p, int row, int c0, const float (&v)[16],
                                              float (*red_v)[BH], int (*red_r)[BH], int quad,
                                              const float* ypre = nullptr) {
    const int warp = quad, lane = threadIdx.x & 31;
    const bool in = row < p.rows;
    if (p.epi == EPI_ARGMAX) {
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            const int b = c0 + j;
            float bv = in ? v[j] : -INFINITY;
            int br = in ? row : 0x7fffffff;
            if (p.dbg && in && b < p.B) p.dbg[(size_t)b * p.ld_dbg + row] = v[j];
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) {
                const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
                const int orow = __shfl_xor_sync(0xffffffffu, br, o);
                if (ov > bv || (ov == bv && orow < br)) { bv = ov; br = orow; }
            }
            if (lane == 0) { red_v[warp][b] = bv; red_r[warp][b] = br; }
        }
        return;
    }
    if (p.ru == 2) {  // gate on even rows, up on the odd row after it
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            const float up = __shfl_xor_sync(0xffffffffu, v[j], 1);
            const int b = c0 + j;
            if (in && (row & 1) == 0 && b < p.B) p.y[(size_t)b * p.ldy + (row >> 1)] = silu(v[j]) * up;
        }
        return;
    }
    if (!in) return;
#pragma unroll
    for (int j = 0; j < 16; ++j) {
        const int b = c0 + j;
        if (b >= p.B) continue;
        float* yp = p.y + (size_t)b * p.ldy + row;
        const float a = v[j];
        switch (p.epi) {
            case EPI_STORE: *yp = a; break;
            case EPI_BIAS: *yp = a + __bfloat162float(static_cast<const __nv_bfloat16*>(p.bias)[row]); break;
            case EPI_SILU: *yp = silu(a); break;
            case EPI_RESADD: *yp = (ypre ? ypre[j] : *yp) + a; break;
            default: break;
        }
    }
}

// float index of float4 group c4 of row r in a [128][BH] fp32 tile parked in
// shared memory: groups XOR-swizzled by row (conflict-free row-wise stores)
template <int BH>
__device__ __forceinline__ int tc_park_idx(int r, int c4) {
    constexpr int NC4 = BH / 4;
    return r * BH + ((c4 ^ (r & (NC4 - 1))) << 2);
}

// Split-K epilogue of 4 batch columns [4*c4, 4*c4+4) of tile row rr (and, for
// SwiGLU, its up row rr+1), summed over the cluster in split order, scaled by
// rstd[b] (a per-sequence RMSNorm factor) when rstd is given.
template <int BH>
__device__ __forceinline__ void tc_cluster_epilogue(const TcParams& p, cooperative_groups::cluster_group& cl,
                                                    float* park, int tile, int rr, int c4,
                                                    const float* rstd = nullptr, const float* ypre = nullptr) {
    // every split's distributed-shared-memory load is issued before any is
    // used (a remote load takes several hundred cycles), then the splits are
    // added in split order (deterministic)
    float4 ta[kTcMaxSplits], tu[kTcMaxSplits];
#pragma unroll
    for (int s = 0; s < kTcMaxSplits; ++s) {
        if (s < p.splits) {
            const float* rem = cl.map_shared_rank(park, s);
            ta[s] = *reinterpret_cast<const float4*>(rem + tc_park_idx<BH>(rr, c4));
            if (p.ru == 2) tu[s] = *reinterpret_cast<const float4*>(rem + tc_park_idx<BH>(rr + 1, c4));
        }
    }
    float4 a = make_float4(0.f, 0.f, 0.f, 0.f), u = a;
#pragma unroll
    for (int s = 0; s < kTcMaxSplits; ++s) {
        if (s < p.splits) {
            a.x += ta[s].x; a.y += ta[s].y; a.z += ta[s].z; a.w += ta[s].w;
            if (p.ru == 2) { u.x += tu[s].x; u.y += tu[s].y; u.z += tu[s].z; u.w += tu[s].w; }
        }
    }
    float va[4] = {a.x, a.y, a.z, a.w}, vu[4] = {u.x, u.y, u.z, u.w};
    if (rstd) {
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            va[j] *= rstd[4 * c4 + j];
            vu[j] *= rstd[4 * c4 + j];
        }
    }
    const int row = tile * kTcM + rr;
    if (row >= p.rows) return;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const int b = 4 * c4 + j;
        if (b >= p.B) break;
        if (p.ru == 2) {
            p.y[(size_t)b * p.ldy + (row >> 1)] = silu(va[j]) * vu[j];
            continue;
        }
        float* yp = p.y + (size_t)b * p.ldy + row;
        switch (p.epi) {
            case EPI_STORE: *yp = va[j]; break;
            case EPI_BIAS: *yp = va[j] + __bfloat162float(static_cast<const __nv_bfloat16*>(p.bias)[row]); break;
            case EPI_SILU: *yp = silu(va[j]); break;
            case EPI_RESADD: *yp = (ypre ? ypre[j] : *yp) + va[j]; break;
            case EPI_ARGMAX:
                if (p.dbg) p.dbg[(size_t)b * p.ld_dbg + row] = va[j];
                atomicMax(p.am + b, argmax_key(va[j], row));
                break;
            default: break;
        }
    }
}

// BH: batch columns (a multiple of 16, >= B); the MMA N is 2 * BH (hi | lo).
// ST: operand stages.  Launched with cluster size p.splits when p.splits > 1.
template <int BH, int ST>
__global__ void __launch_bounds__(kTcThreads, 1) gemm_tc_kernel(const __grid_constant__ CUtensorMap tmW,
                                                                const __grid_constant__ CUtensorMap tmX, TcParams p) {
    extern __shared__ __align__(1024) unsigned char tc_smem_raw[];
    constexpr int BN = 2 * BH;
    constexpr int kBBytes = BN * kTcBK * 2;
    constexpr uint32_t kCols = BN <= 32 ? 32u : BN <= 64 ? 64u : BN <= 128 ? 128u : 256u;
    static_assert(kTcM * BH * 4 <= ST * (kTcABytes + kBBytes), "parked tile must fit in the operand stages");
    unsigned char* sm = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(tc_smem_raw) + 1023) & ~(uintptr_t)1023);
    unsigned char* sA = sm;
    unsigned char* sB = sm + ST * kTcABytes;
    uint64_t* full = reinterpret_cast<uint64_t*>(sB + ST * kBBytes);
    uint64_t* empty = full + ST;
    uint64_t* accb = empty + ST;
    __shared__ uint32_t tmem_base;
    __shared__ float red_v[4][BH];
    __shared__ int red_r[4][BH];
    PIPO_TR(__shared__ unsigned long long tr_s[3]; const TraceT0 tr0 = trace_begin();)

    pdl_launch();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int tile = blockIdx.x / p.splits, split = blockIdx.x % p.splits;
    const int nkb = p.K / kTcBK;
    const int kb0 = (int)((long long)split * nkb / p.splits), kb1 = (int)((long long)(split + 1) * nkb / p.splits);
    const int nk = kb1 - kb0;  // >= 1 (splits <= nkb)

    if (threadIdx.x == 64) {
        prefetch_tmap(&tmW);
        prefetch_tmap(&tmX);
    }
    if (warp == 0) tmem_alloc(&tmem_base, kCols);
    if (threadIdx.x == 32) {
        for (int s = 0; s < ST; ++s) {
            mbar_init(full + s, 1);
            mbar_init(empty + s, 1);
        }
        mbar_init(accb, 1);
        mbar_init_fence();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_base;

    if (warp == 0) {
        if (lane == 0) {
            // TMA producer: the weight tiles of the first ST stages need
            // nothing from the previous kernel and go out before the
            // dependency wait (programmatic dependent launch); the
            // activation tiles follow it
            const int pre = min(nk, ST);
            for (int i = 0; i < pre; ++i) {
                mbar_arrive_expect_tx(full + i, (uint32_t)(kTcABytes + kBBytes));
                tma_load_2d(sA + i * kTcABytes, &tmW, (kb0 + i) * kTcBK, tile * kTcM, full + i);
            }
            pdl_wait();
            PIPO_TR(tr_s[0] = trace_now();)
            for (int i = 0; i < pre; ++i) tma_load_2d(sB + i * kBBytes, &tmX, (kb0 + i) * kTcBK, 0, full + i);
            int issued = pre;
            for (int i = pre; i < nk; ++i) {
                const int s = i % ST;
                if (!mbar_wait(empty + s, (uint32_t)(((i / ST) & 1) ^ 1), 11, i)) break;
                mbar_arrive_expect_tx(full + s, (uint32_t)(kTcABytes + kBBytes));
                tma_load_2d(sA + s * kTcABytes, &tmW, (kb0 + i) * kTcBK, tile * kTcM, full + s);
                tma_load_2d(sB + s * kBBytes, &tmX, (kb0 + i) * kTcBK, 0, full + s);
                issued = i + 1;
            }
            // no copy into this CTA's shared memory may still be in flight at exit
            for (int i = max(0, issued - ST); i < issued; ++i) mbar_wait(full + (i % ST), (uint32_t)((i / ST) & 1), 12, i);
        }
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0) {
            // MMA issuer: 4 MMAs of K = 16 per stage, the operand
            // descriptors advanced by 32 bytes inside the swizzled rows
            const uint32_t idesc = umma_idesc_bf16(kTcM, BN);
            for (int i = 0; i < nk; ++i) {
                const int s = i % ST;
                if (!mbar_wait(full + s, (uint32_t)((i / ST) & 1), 13, i)) break;
                tc_fence_after();
                const uint32_t a0 = smem_u32(sA + s * kTcABytes), b0 = smem_u32(sB + s * kBBytes);
#pragma unroll
                for (int k = 0; k < kTcBK / 16; ++k)
                    umma_bf16(tmem, umma_desc_sw128(a0 + k * 32), umma_desc_sw128(b0 + k * 32), idesc,
                              (i > 0 || k > 0) ? 1u : 0u);
                umma_commit(empty + s);  // frees the stage once these MMAs have read it
            }
            umma_commit(accb);
        }
        __syncwarp();
    }

    // epilogue: thread t holds TMEM lane t = weight row tile*128 + t
    mbar_wait(accb, 0, 14, (unsigned)nk);
    PIPO_TR(if (threadIdx.x == 0) tr_s[1] = trace_now();)
    __syncwarp();
    tc_fence_after();
    pdl_wait();
    const int row = tile * kTcM + threadIdx.x;
    const uint32_t lane_addr = tmem + ((uint32_t)(warp * 32) << 16);
    // 16 batch columns: hi part at column c0, lo part at column BH + c0
    auto ld_cols = [&](int c0, float (&v)[16]) {
        float lo[16];
        tmem_ld16(lane_addr + c0, v);
        tmem_ld16(lane_addr + BH + c0, lo);
#pragma unroll
        for (int j = 0; j < 16; ++j) v[j] += lo[j];
    };
    if (p.splits == 1) {
#pragma unroll 1
        for (int c0 = 0; c0 < BH; c0 += 16) {
            float v[16];
            ld_cols(c0, v);
            tc_epilogue16<BH>(p, row, c0, v, red_v, red_r, warp);
        }
        if (p.epi == EPI_ARGMAX) {
            __syncthreads();
            if (threadIdx.x < p.B) {
                const int b = threadIdx.x;
                float bv = -INFINITY;
                int br = 0x7fffffff;
                for (int w = 0; w < 4; ++w)
                    if (red_r[w][b] != 0x7fffffff && (red_v[w][b] > bv || (red_v[w][b] == bv && red_r[w][b] < br))) {
                        bv = red_v[w][b];
                        br = red_r[w][b];
                    }
                if (br != 0x7fffffff) atomicMax(p.am + b, argmax_key(bv, br));
            }
        }
    } else {
        // park this split's partial tile in the (now idle) operand stages
        namespace cg = cooperative_groups;
        cg::cluster_group cl = cg::this_cluster();
        float* park = reinterpret_cast<float*>(sm);
#pragma unroll 1
        for (int c0 = 0; c0 < BH; c0 += 16) {
            float v[16];
            ld_cols(c0, v);
#pragma unroll
            for (int q = 0; q < 4; ++q)
                *reinterpret_cast<float4*>(park + tc_park_idx<BH>(threadIdx.x, c0 / 4 + q)) =
                    make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
        }
        cl.sync();  // every split's partial is parked
        // rows [r0, r1) of the tile are this CTA's: an even count (SwiGLU pairs)
        const int R = (((kTcM + p.splits - 1) / p.splits) + 1) & ~1;
        const int r0 = min(kTcM, split * R), r1 = min(kTcM, r0 + R);
        const int step = p.ru == 2 ? 2 : 1;
        const int items = (r1 - r0) / step * (BH / 4);
        for (int it = threadIdx.x; it < items; it += kTcThreads) {
            const int rr = r0 + (it / (BH / 4)) * step, c4 = it % (BH / 4);
            tc_cluster_epilogue<BH>(p, cl, park, tile, rr, c4);
        }
        cl.sync();  // no CTA leaves while others still read its shared memory
    }
    PIPO_TR(if (threadIdx.x == 0) tr_s[2] = trace_now();)
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tmem, kCols);
    }
    PIPO_TR(if (threadIdx.x == 0) trace_put(TR_TC, tr0, tr0.clk, tr_s[0], tr_s[1], tr_s[2]);)
}

// ---------------------------------------------------------------- fused form
//
// The same projection with the activation split done inside the GEMM: per
// stage the producer thread also copies the raw fp32 activation tile
// [BH rows][64] (TMA, rows past the batch read as zeros) and, for a
// normalised input, the 64 RMSNorm gains; four converter warps turn it into
// the swizzled bf16 hi | lo operand tile (rows b and BH + b) in the stage and
// accumulate sum(x^2) per sequence.  The norm factor rstd[b] =
// 1/sqrt(mean(x^2) + eps) multiplies the accumulator in the epilogue
// (W (g . x) rstd is the projection of the normalised input); with K split
// over a cluster the sums are added over the cluster in split order.  The
// converter warps are also the epilogue warps (TMEM lane quadrants 2, 3, 0, 1).
// Inputs: one activation segment, or two under one joint norm (no gathers,
// no separate norms of two segments: those keep prep_bf16_kernel).
constexpr int kTcfThreads = 192;  // W producer, MMA issuer, 4 converter / epilogue warps

__host__ __device__ constexpr int tcf_stages(int bh, bool deep) {
    return deep ? (bh <= 16 ? 8 : bh <= 32 ? 6 : bh <= 64 ? 4 : 2) : (bh <= 16 ? 4 : bh <= 32 ? 3 : 2);
}
// stage: W tile, bf16 operand tile [2BH][64], raw fp32 tile [BH][64], gains (128 B), 1024-byte aligned
__host__ __device__ constexpr int tcf_stage_bytes(int bh) { return kTcABytes + 512 * bh + 1024; }

struct TcfIn {
    int nseg, K0, norm, klen;  // segments, length of segment 0, norm applied, norm length
    const void* gamma;         // [K] bf16 gains (joint or single segment) when norm
    float eps;
    int B;
    unsigned long long* zero_ptr;  // zeroed by block 0 before anything else (or nullptr)
    int zero_n;
};

template <int BH, int ST>
__global__ void __launch_bounds__(kTcfThreads, 1)
    gemm_tcf_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmX0,
                    const __grid_constant__ CUtensorMap tmX1, TcfIn in, TcParams p) {
    extern __shared__ __align__(1024) unsigned char tcf_smem_raw[];
    constexpr int BN = 2 * BH;
    constexpr int SB = tcf_stage_bytes(BH);
    constexpr int kBOff = kTcABytes, kRawOff = kTcABytes + 256 * BH, kGmOff = kTcABytes + 512 * BH;
    constexpr uint32_t kCols = BN <= 32 ? 32u : BN <= 64 ? 64u : BN <= 128 ? 128u : 256u;
    constexpr int NQ = BH / 16;  // conversion tasks per converter thread per stage
    static_assert(kTcM * BH * 4 <= ST * SB, "parked tile must fit in the stages");
    unsigned char* sm = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(tcf_smem_raw) + 1023) & ~(uintptr_t)1023);
    uint64_t* full_raw = reinterpret_cast<uint64_t*>(sm + (size_t)ST * SB);
    uint64_t* full_mma = full_raw + ST;
    uint64_t* empty = full_mma + ST;
    uint64_t* accb = empty + ST;
    __shared__ uint32_t tmem_base;
    __shared__ float red_v[4][BH];
    __shared__ int red_r[4][BH];
    __shared__ float ss_s[BH], rstd_s[BH];
    // EPI_RESADD: the residual values this thread's epilogue updates, loaded
    // right after the dependency wait so that the epilogue does not wait for them
    float ypre[BH];
    constexpr int kPreItems = (kTcM / 2) * (BH / 4) / 128;  // cluster items per thread (splits >= 2)
    PIPO_TR(__shared__ unsigned long long tr_s[3], tr_e[3]; const TraceT0 tr0 = trace_begin();)

    pdl_launch();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int tile = blockIdx.x / p.splits, split = blockIdx.x % p.splits;
    const int nkb = p.K / kTcBK;
    const int kb0 = (int)((long long)split * nkb / p.splits), kb1 = (int)((long long)(split + 1) * nkb / p.splits);
    const int nk = kb1 - kb0;  // >= 1 (splits <= nkb)
    const uint32_t raw_bytes = (uint32_t)(BH * kTcBK * 4) + (in.norm ? 128u : 0u);

    if (threadIdx.x == 64) {
        prefetch_tmap(&tmW);
        prefetch_tmap(&tmX0);
        if (in.nseg == 2) prefetch_tmap(&tmX1);
    }
    if (warp == 0) tmem_alloc(&tmem_base, kCols);
    if (threadIdx.x == 32) {
        for (int s = 0; s < ST; ++s) {
            mbar_init(full_raw + s, 1);
            mbar_init(full_mma + s, 4);
            mbar_init(empty + s, 1);
        }
        mbar_init(accb, 1);
        mbar_init_fence();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_base;

    if (warp == 0) {
        if (lane == 0) {
            // producer: weights and gains of the first ST stages before the
            // dependency wait, the activation tiles after it
            auto x_tile = [&](int i, unsigned char* stg, uint64_t* bar) {
                const int k = (kb0 + i) * kTcBK;
                if (in.nseg == 2 && k >= in.K0) tma_load_2d(stg + kRawOff, &tmX1, k - in.K0, 0, bar);
                else tma_load_2d(stg + kRawOff, &tmX0, k, 0, bar);
            };
            const int pre = min(nk, ST);
            for (int i = 0; i < pre; ++i) {
                unsigned char* stg = sm + (size_t)i * SB;
                mbar_arrive_expect_tx(full_raw + i, (uint32_t)kTcABytes + raw_bytes);
                tma_load_2d(stg, &tmW, (kb0 + i) * kTcBK, tile * kTcM, full_raw + i);
                if (in.norm)
                    bulk_g2s(stg + kGmOff, static_cast<const __nv_bfloat16*>(in.gamma) + (size_t)(kb0 + i) * kTcBK,
                             128, full_raw + i);
            }
            pdl_wait();
            for (int i = 0; i < pre; ++i) x_tile(i, sm + (size_t)i * SB, full_raw + i);
            int issued = pre;
            for (int i = pre; i < nk; ++i) {
                const int s = i % ST;
                if (!mbar_wait(empty + s, (uint32_t)(((i / ST) & 1) ^ 1), 11, i)) break;
                unsigned char* stg = sm + (size_t)s * SB;
                mbar_arrive_expect_tx(full_raw + s, (uint32_t)kTcABytes + raw_bytes);
                tma_load_2d(stg, &tmW, (kb0 + i) * kTcBK, tile * kTcM, full_raw + s);
                if (in.norm)
                    bulk_g2s(stg + kGmOff, static_cast<const __nv_bfloat16*>(in.gamma) + (size_t)(kb0 + i) * kTcBK,
                             128, full_raw + s);
                x_tile(i, stg, full_raw + s);
                issued = i + 1;
            }
            for (int i = max(0, issued - ST); i < issued; ++i)
                mbar_wait(full_raw + (i % ST), (uint32_t)((i / ST) & 1), 12, i);
        }
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0) {
            // MMA issuer: a stage is ready once the converter warps filled its operand tile
            const uint32_t idesc = umma_idesc_bf16(kTcM, BN);
            for (int i = 0; i < nk; ++i) {
                const int s = i % ST;
                if (!mbar_wait(full_mma + s, (uint32_t)((i / ST) & 1), 13, i)) break;
                tc_fence_after();
                const uint32_t a0 = smem_u32(sm + (size_t)s * SB), b0 = a0 + kBOff;
#pragma unroll
                for (int k = 0; k < kTcBK / 16; ++k)
                    umma_bf16(tmem, umma_desc_sw128(a0 + k * 32), umma_desc_sw128(b0 + k * 32), idesc,
                              (i > 0 || k > 0) ? 1u : 0u);
                umma_commit(empty + s);
            }
            umma_commit(accb);
        }
        __syncwarp();
    } else {
        // converter warps: raw fp32 tile -> bf16 hi | lo operand tile, sum(x^2)
        const int xt = threadIdx.x - 64;  // 0..127
        pdl_wait();
        if (p.epi == EPI_RESADD) {
            if (p.splits == 1) {
                const int row = tile * kTcM + (warp & 3) * 32 + lane;
#pragma unroll
                for (int b = 0; b < BH; ++b)
                    ypre[b] = (row < p.rows && b < p.B) ? __ldcg(p.y + (size_t)b * p.ldy + row) : 0.f;
            } else {
                const int R = (((kTcM + p.splits - 1) / p.splits) + 1) & ~1;
                const int r0 = min(kTcM, split * R), r1 = min(kTcM, r0 + R);
                const int items = (r1 - r0) * (BH / 4);  // RESADD: one row per item
#pragma unroll
                for (int k = 0; k < kPreItems; ++k) {
                    const int it = xt + 128 * k;
                    const int row = tile * kTcM + r0 + it / (BH / 4), c4 = it % (BH / 4);
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        const int b = 4 * c4 + j;
                        ypre[4 * k + j] = (it < items && row < p.rows && b < p.B)
                                              ? __ldcg(p.y + (size_t)b * p.ldy + row) : 0.f;
                    }
                }
            }
        }
        PIPO_TR(if (xt == 0) tr_s[0] = trace_now();)
        if (in.zero_ptr && blockIdx.x == 0)
            for (int i = xt; i < in.zero_n; i += 128) in.zero_ptr[i] = 0ull;
        float ss[NQ];
#pragma unroll
        for (int q = 0; q < NQ; ++q) ss[q] = 0.f;
        for (int i = 0; i < nk; ++i) {
            const int s = i % ST;
            if (!mbar_wait(full_raw + s, (uint32_t)((i / ST) & 1), 15, i)) break;
            unsigned char* stg = sm + (size_t)s * SB;
            const float* raw = reinterpret_cast<const float*>(stg + kRawOff);
            float gm[8];
            const int c = xt & 7;  // 8-element chunk of the 64-wide stage (same for every task)
            if (in.norm) {
                const uint4 g4 = *reinterpret_cast<const uint4*>(stg + kGmOff + c * 16);
                gm[0] = bf_lo(g4.x); gm[1] = bf_hi(g4.x); gm[2] = bf_lo(g4.y); gm[3] = bf_hi(g4.y);
                gm[4] = bf_lo(g4.z); gm[5] = bf_hi(g4.z); gm[6] = bf_lo(g4.w); gm[7] = bf_hi(g4.w);
            }
#pragma unroll
            for (int q = 0; q < NQ; ++q) {
                const int b = (xt >> 3) + 16 * q;
                const float4 r0 = *reinterpret_cast<const float4*>(raw + b * kTcBK + c * 8);
                const float4 r1 = *reinterpret_cast<const float4*>(raw + b * kTcBK + c * 8 + 4);
                float x[8] = {r0.x, r0.y, r0.z, r0.w, r1.x, r1.y, r1.z, r1.w};
                if (b >= in.B) {
#pragma unroll
                    for (int e = 0; e < 8; ++e) x[e] = 0.f;
                }
                if (in.norm) {
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        ss[q] += x[e] * x[e];
                        x[e] *= gm[e];
                    }
                }
                uint32_t hi[4], lo[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const __nv_bfloat162 h = __floats2bfloat162_rn(x[2 * e], x[2 * e + 1]);
                    const float2 hf = __bfloat1622float2(h);
                    const __nv_bfloat162 l = __floats2bfloat162_rn(x[2 * e] - hf.x, x[2 * e + 1] - hf.y);
                    hi[e] = *reinterpret_cast<const uint32_t*>(&h);
                    lo[e] = *reinterpret_cast<const uint32_t*>(&l);
                }
                const int sw = (c ^ (b & 7)) << 4;
                *reinterpret_cast<uint4*>(stg + kBOff + b * 128 + sw) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
                *reinterpret_cast<uint4*>(stg + kBOff + (BH + b) * 128 + sw) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
            }
            fence_proxy_async();  // the generic-proxy stores above, before the MMAs read them
            __syncwarp();
            if (lane == 0) mbar_arrive(full_mma + s);
        }
        // sum(x^2) of sequence b over this CTA's K range
#pragma unroll
        for (int q = 0; q < NQ; ++q) {
            float v = ss[q];
            v += __shfl_xor_sync(0xffffffffu, v, 1);
            v += __shfl_xor_sync(0xffffffffu, v, 2);
            v += __shfl_xor_sync(0xffffffffu, v, 4);
            if ((xt & 7) == 0) ss_s[(xt >> 3) + 16 * q] = v;
        }
        asm volatile("bar.sync 1, 128;" ::: "memory");
        if (p.splits == 1 && xt < BH)
            rstd_s[xt] = in.norm ? 1.0f / sqrtf(ss_s[xt] / (float)in.klen + in.eps) : 1.0f;
        asm volatile("bar.sync 1, 128;" ::: "memory");
    }

    // ---- epilogue: the converter warps hold TMEM lane quadrants 2, 3, 0, 1
    const int quad = warp & 3;
    const int row = tile * kTcM + quad * 32 + lane;
    const uint32_t lane_addr = tmem + ((uint32_t)(quad * 32) << 16);
    const bool epi_warp = warp >= 2;
    if (epi_warp) {
        mbar_wait(accb, 0, 14, (unsigned)nk);
        PIPO_TR(if (threadIdx.x == 64) tr_s[1] = trace_now();)
        __syncwarp();
        tc_fence_after();
    }
    auto ld_cols = [&](int c0, float (&v)[16]) {
        float lo[16];
        tmem_ld16(lane_addr + c0, v);
        tmem_ld16(lane_addr + BH + c0, lo);
#pragma unroll
        for (int j = 0; j < 16; ++j) v[j] += lo[j];
    };
    if (p.splits == 1) {
        if (epi_warp) {
#pragma unroll
            for (int c0 = 0; c0 < BH; c0 += 16) {
                float v[16];
                ld_cols(c0, v);
                PIPO_TR(if (threadIdx.x == 64 && c0 == 0) tr_e[0] = trace_now();)
#pragma unroll
                for (int j = 0; j < 16; ++j) v[j] *= rstd_s[c0 + j];
                tc_epilogue16<BH>(p, row, c0, v, red_v, red_r, quad, p.epi == EPI_RESADD ? ypre + c0 : nullptr);
            }
            PIPO_TR(if (threadIdx.x == 64) { tr_e[1] = trace_now(); tr_e[2] = tr_e[1]; })
            if (p.epi == EPI_ARGMAX) {
                asm volatile("bar.sync 1, 128;" ::: "memory");
                const int b = threadIdx.x - 64;
                if (b < p.B) {
                    float bv = -INFINITY;
                    int br = 0x7fffffff;
                    for (int w = 0; w < 4; ++w)
                        if (red_r[w][b] != 0x7fffffff &&
                            (red_v[w][b] > bv || (red_v[w][b] == bv && red_r[w][b] < br))) {
                            bv = red_v[w][b];
                            br = red_r[w][b];
                        }
                    if (br != 0x7fffffff) atomicMax(p.am + b, argmax_key(bv, br));
                }
            }
        }
    } else {
        namespace cg = cooperative_groups;
        cg::cluster_group cl = cg::this_cluster();
        float* park = reinterpret_cast<float*>(sm);
        if (epi_warp) {
            const int r = quad * 32 + lane;
#pragma unroll 1
            for (int c0 = 0; c0 < BH; c0 += 16) {
                float v[16];
                ld_cols(c0, v);
#pragma unroll
                for (int q = 0; q < 4; ++q)
                    *reinterpret_cast<float4*>(park + tc_park_idx<BH>(r, c0 / 4 + q)) =
                        make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
            }
            PIPO_TR(if (threadIdx.x == 64) tr_e[0] = trace_now();)
        }
        cl.sync();  // every split's partial tile and sum(x^2) are in place
        PIPO_TR(if (threadIdx.x == 64) tr_e[1] = trace_now();)
        if (epi_warp) {
            const int xt = threadIdx.x - 64;
            if (xt < BH) {
                float ts[kTcMaxSplits];  // every remote load first, then the sum in split order
#pragma unroll
                for (int rk = 0; rk < kTcMaxSplits; ++rk)
                    if (rk < p.splits) ts[rk] = *cl.map_shared_rank(&ss_s[xt], rk);
                float t = 0.f;
#pragma unroll
                for (int rk = 0; rk < kTcMaxSplits; ++rk)
                    if (rk < p.splits) t += ts[rk];
                rstd_s[xt] = in.norm ? 1.0f / sqrtf(t / (float)in.klen + in.eps) : 1.0f;
            }
            asm volatile("bar.sync 1, 128;" ::: "memory");
            const int R = (((kTcM + p.splits - 1) / p.splits) + 1) & ~1;
            const int r0 = min(kTcM, split * R), r1 = min(kTcM, r0 + R);
            const int step = p.ru == 2 ? 2 : 1;
            const int items = (r1 - r0) / step * (BH / 4);
#pragma unroll
            for (int k = 0; k < kPreItems; ++k) {
                const int it = xt + 128 * k;
                if (it >= items) break;
                const int rr = r0 + (it / (BH / 4)) * step, c4 = it % (BH / 4);
                tc_cluster_epilogue<BH>(p, cl, park, tile, rr, c4, rstd_s,
                                        p.epi == EPI_RESADD ? ypre + 4 * k : nullptr);
            }
            PIPO_TR(if (threadIdx.x == 64) tr_e[2] = trace_now();)
        }
        cl.sync();  // no CTA leaves while others still read its shared memory
    }
    PIPO_TR(if (threadIdx.x == 64) tr_s[2] = trace_now();)
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tmem, kCols);
    }
    PIPO_TR(if (threadIdx.x == 0) {
        trace_put(TR_TCF, tr0, tr0.clk, tr_s[0], tr_s[1], tr_s[2]);
        trace_put(TR_TCF_EPI, tr0, tr_s[1], tr_e[0], tr_e[1], tr_e[2]);
    })
}

// Activations of the tensor-core GEMM, [2 * BH][K] bf16: row b < B holds
// hi = bf16(x_b) and row BH + b holds lo = bf16(x_b - hi), where x_b is the
// (gathered, RMS-normalised) GEMV input of sequence b; rows of b >= B are
// zero.  grid BH, kPrepThreads threads; one pass: every thread keeps its
// (at most kPrepQ) groups of 4 inputs in registers between the sum of squares
// and the write, and all its loads are in flight together.
constexpr int kPrepThreads = 512;
constexpr int kPrepQ = 8;  // K <= 4 * kPrepQ * kPrepThreads = 16384

template <typename T>
__device__ __forceinline__ float4 ld4_any(const void* p, size_t i) {
    if constexpr (sizeof(T) == 2) {
        const uint2 u = *reinterpret_cast<const uint2*>(static_cast<const __nv_bfloat16*>(p) + i);
        return make_float4(bf_lo(u.x), bf_hi(u.x), bf_lo(u.y), bf_hi(u.y));
    } else {
        return *reinterpret_cast<const float4*>(static_cast<const float*>(p) + i);
    }
}

template <typename T>
__global__ void __launch_bounds__(kPrepThreads) prep_bf16_kernel(GemvParams p, __nv_bfloat16* xb, int BH) {
    __shared__ float red[kPrepThreads / 32][2];
    __shared__ float rstd[2];
    pdl_launch();
    pdl_wait();
    const int b = blockIdx.x, K = p.K, K4 = K / 4, tid = threadIdx.x;
    if (p.zero_ptr && b == 0)  // argmax keys of this step (read by later kernels only)
        for (int i = tid; i < p.zero_n; i += blockDim.x) p.zero_ptr[i] = 0ull;
    uint2* dst = reinterpret_cast<uint2*>(xb + (size_t)b * K);
    uint2* dst_lo = reinterpret_cast<uint2*>(xb + (size_t)(BH + b) * K);
    if (b >= p.B) {
        for (int q = tid; q < K4; q += kPrepThreads) dst[q] = dst_lo[q] = make_uint2(0u, 0u);
        return;
    }
    const int K0q = p.seg[0].K / 4;
    int tok[2] = {0, 0};
#pragma unroll
    for (int s = 0; s < 2; ++s)
        if (s < p.nseg && !p.seg[s].src) {
            const Seg& sg = p.seg[s];
            tok[s] = sg.tok_am ? argmax_row(sg.tok_am[b]) : sg.tok[(size_t)b * sg.tok_ld];
        }
    float4 v[kPrepQ];
    float ss0 = 0.f, ss1 = 0.f;
#pragma unroll
    for (int i = 0; i < kPrepQ; ++i) {
        const int q = tid + i * kPrepThreads;
        v[i] = make_float4(0.f, 0.f, 0.f, 0.f);
        if (q < K4) {
            const int s = q < K0q ? 0 : 1;
            const Seg& sg = p.seg[s];
            const size_t kk = (size_t)(s == 0 ? q : q - K0q) * 4;
            if (sg.src) v[i] = *reinterpret_cast<const float4*>(sg.src + (size_t)b * sg.ld + kk);
            else v[i] = tok[s] < 0 ? ld4_any<T>(sg.pad, kk) : ld4_any<T>(sg.table, (size_t)tok[s] * sg.K + kk);
        }
    }
    const bool norm0 = p.seg[0].gamma != nullptr, norm1 = p.nseg > 1 && p.seg[1].gamma != nullptr;
    if (norm0 || norm1) {
#pragma unroll
        for (int i = 0; i < kPrepQ; ++i) {
            const int q = tid + i * kPrepThreads;
            const float sq = v[i].x * v[i].x + v[i].y * v[i].y + v[i].z * v[i].z + v[i].w * v[i].w;
            if (p.joint_norm || q < K0q) ss0 += sq; else ss1 += sq;
        }
        ss0 = warp_sum(ss0);
        ss1 = warp_sum(ss1);
        if ((tid & 31) == 0) { red[tid >> 5][0] = ss0; red[tid >> 5][1] = ss1; }
        __syncthreads();
        if (tid < 2) {
            float t = 0.f;
            for (int w = 0; w < kPrepThreads / 32; ++w) t += red[w][tid];
            const int len = p.joint_norm ? (tid == 0 ? K : 1) : (tid == 0 ? p.seg[0].K : (p.nseg > 1 ? p.seg[1].K : 1));
            rstd[tid] = 1.0f / sqrtf(t / (float)len + p.eps);
        }
        __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < kPrepQ; ++i) {
        const int q = tid + i * kPrepThreads;
        if (q >= K4) break;
        float4 x = v[i];
        const int g = (p.joint_norm || q < K0q) ? 0 : 1;
        const Seg& sg = p.seg[p.joint_norm ? 0 : g];
        if (sg.gamma) {
            const size_t kk = (size_t)((p.joint_norm || g == 0) ? q : q - K0q) * 4;
            const float4 gm = ld4_any<T>(sg.gamma, kk);
            const float r = rstd[g];
            x.x *= r * gm.x; x.y *= r * gm.y; x.z *= r * gm.z; x.w *= r * gm.w;
        }
        const __nv_bfloat162 h01 = __floats2bfloat162_rn(x.x, x.y), h23 = __floats2bfloat162_rn(x.z, x.w);
        const float2 f01 = __bfloat1622float2(h01), f23 = __bfloat1622float2(h23);
        const __nv_bfloat162 l01 = __floats2bfloat162_rn(x.x - f01.x, x.y - f01.y);
        const __nv_bfloat162 l23 = __floats2bfloat162_rn(x.z - f23.x, x.w - f23.y);
        dst[q] = make_uint2(*reinterpret_cast<const uint32_t*>(&h01), *reinterpret_cast<const uint32_t*>(&h23));
        dst_lo[q] = make_uint2(*reinterpret_cast<const uint32_t*>(&l01), *reinterpret_cast<const uint32_t*>(&l23));
    }
}

}  // namespace pipo
