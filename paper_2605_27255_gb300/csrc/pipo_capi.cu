// C ABI of the PIPO pair-decode library (declared in include/pipo.h).
//
// A context owns the model weights (fused QKV and gate|up layouts), a paged
// KV cache per decoder block (backbone blocks + the MTP block), fp32
// activation buffers and the per-sequence device state (pending pair, KV
// length, emitted count).  A decode step is one captured CUDA graph: no host
// round trip inside the step.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdarg>
#include <cstdio>
#include <cmath>
#include <cstdlib>
#include <cstring>
#include <map>
#include <mutex>
#include <numeric>
#include <random>
#include <string>
#include <type_traits>
#include <vector>

// Kernel headers for their parameter structs and launch constants; the
// kernels themselves are compiled in the k_*.cu units (kernel_tables.h).
#include "attn_cluster.cuh"
#include "attn_mma.cuh"
#include "attn_prefill.cuh"
#include "gemv_stream.cuh"
#include "kernel_tables.h"
#include "kernels.cuh"
#include "pipo.h"
#include "sampler.cuh"
#include "tcgen05_gemm.cuh"

using namespace pipo;
using bf16 = __nv_bfloat16;

namespace pipo {

// Packed argmax keys -> token ids.
__global__ void keys_to_tokens_kernel(const unsigned long long* keys, int32_t* tokens, int B) {
    const int b = blockIdx.x * blockDim.x + threadIdx.x;
    if (b < B) tokens[b] = argmax_row(keys[b]);
}

// Prefill positions before the last: n[b] += by (the positions just run).
__global__ void advance_kernel(int32_t* n_pos, int B, int by) {
    pdl_launch();
    pdl_wait();
    const int b = blockIdx.x * blockDim.x + threadIdx.x;
    if (b < B) n_pos[b] += by;
}


// Regular decoding, end of a step: the LM-head argmax is the output token and
// the next input (slot 1 stays PAD, nothing is drafted), one more cache entry,
// one more emitted token.  grid B, any block size.
__global__ void regular_accept_kernel(StepState st, int H, const float* h) {
    pdl_launch();
    pdl_wait();
    const int b = blockIdx.x;
    if (st.dbg_hb)
        for (int k = threadIdx.x; k < H; k += blockDim.x) st.dbg_hb[(size_t)b * H + k] = h[(size_t)b * H + k];
    if (threadIdx.x != 0) return;
    const int xb = argmax_row(st.am_b[b]);
    st.out_tokens[2 * b] = xb;
    st.out_tokens[2 * b + 1] = -1;
    st.out_nacc[b] = 0;
    st.pending[2 * b] = xb;
    st.pending[2 * b + 1] = -1;
    st.n_pos[b] += 1;
    st.emitted[b] += 1;
    if (st.dbg_xb) st.dbg_xb[b] = xb;
}

}  // namespace pipo

namespace {

// message of the last failure of a call made without a context (pipo_init,
// the pipo_op_* entry points) on this thread: thread-local, so that threads
// failing at once neither race on it nor free a string another one returns
thread_local std::string g_init_error = "no error";

struct BlockW {
    void *attn_norm = nullptr, *Wqkv = nullptr, *Wo = nullptr, *ffn_norm = nullptr, *Wgu = nullptr, *Wdown = nullptr;
};

enum Mode { DECODE = 0, PREFILL_MID = 1, PREFILL_LAST = 2 };

}  // namespace

struct pipo_ctx {
    pipo_config cfg{};
    int dev = 0, sms = 0;
    size_t esz = 4;
    cudaStream_t own_stream = nullptr, stream = nullptr;
    std::vector<void*> allocs;

    void *E = nullptr, *x_pad = nullptr, *comp_W = nullptr, *comp_b = nullptr, *comp_W1 = nullptr, *comp_W2 = nullptr;
    std::vector<BlockW> blocks;
    BlockW mtp;
    void *final_norm = nullptr, *mtp_norm_h = nullptr, *mtp_norm_e = nullptr, *mtp_W_fc = nullptr,
         *mtp_norm_post = nullptr, *conf_norm = nullptr, *conf_W1 = nullptr, *conf_W2 = nullptr;

    // paged KV cache: n_cache_layers x [num_blocks][n_kv][page][d_h]
    void *Kc = nullptr, *Vc = nullptr;
    int n_cache_layers = 0, blocks_per_seq = 0, num_blocks = 0;
    size_t layer_elems = 0;
    int32_t* block_table = nullptr;

    float *x = nullptr, *x2 = nullptr, *qkv = nullptr, *q = nullptr, *attn = nullptr, *act = nullptr, *t = nullptr;
    float *part_o = nullptr, *part_ml = nullptr;
    unsigned* counters = nullptr;
    float* gemv_part = nullptr;     // split-K partials of the residual-add GEMVs
    unsigned* gemv_rowcnt = nullptr;
    unsigned long long* am = nullptr;  // [2][max_batch]
    // tensor-core projections (bf16, batch >= tc_min_b)
    bf16* tc_xb = nullptr;          // [2 * tc_bn_max][tc_kmax] bf16 activations (hi rows, lo rows)
    int tc_kmax = 0, tc_bn_max = 0;
    int act_rows = 0;               // rows of the fp32 activation buffers (>= the batch width BH)
    bool tc_shallow = false;        // this step's projections: two-per-SM ring (room for a co-resident neighbour)
    int tc_min_b = 2;               // measured: a tie with the CUDA-core GEMV at B = 1, far ahead from B = 4
    int attn_mma_min_b = 1;         // smallest batch on the tensor-core attention (PIPO_ATTN_MMA_MIN_BATCH)
    int tc_splits = 0;              // forced K splits (0: automatic)

    int32_t *pending = nullptr, *n_pos = nullptr, *out_tokens = nullptr, *out_nacc = nullptr;
    long long* emitted = nullptr;
    float *dbg_lb = nullptr, *dbg_ld = nullptr, *dbg_conf = nullptr, *dbg_hb = nullptr, *dbg_hd = nullptr;
    int32_t *dbg_xb = nullptr, *dbg_xd = nullptr;
    float* cache_tmp = nullptr;
    size_t cache_tmp_elems = 0;

    int32_t *pf_pairs = nullptr, *pf_mtp = nullptr;
    size_t pf_cap = 0;
    int32_t* multi_out = nullptr;     // pipo_decode_steps: [n][B][3] tokens and acceptances of n steps
    size_t multi_cap = 0;

    float* rope = nullptr;            // [max_ctx][d_h/2][2] cos, sin
    bool pdl = false;                 // programmatic dependent launch (decode graph only)
    bool attn_cs16 = false;           // 16-CTA attention clusters available
    int attn_cs_force = 0;            // (development) fixed attention cluster size
    int attn_cs_target = 0;           // attention CTAs per SM above which clusters shrink (0: per kernel)
    bool attn_v0 = false;             // (development) the unclustered attention path
    bool attn_regs = false;           // register-ring attention instead of the tensor-core one
    int attn_flat = 1;                // register-ring decode attention without clusters (global merge):
                                      // 0 never, 1 from kFlatMinEntries cached entries, 2 always
    std::vector<CUtensorMap> kv_tm;   // tensor-core attention: K and V tensor map of every cache layer
    // per-launch timing (pipo_profile_step): events around every launch
    bool prof = false;
    int prof_kind = 2;
    double prof_bytes = 0.0;
    std::vector<cudaEvent_t> prof_ev;
    std::vector<int> prof_k;
    std::vector<double> prof_b;
    size_t prof_n = 0;
    // one kernel family of the decode step alone (pipo_replay_family)
    int only_family = -1;             // while capturing: launches of other families are not enqueued
    bool launch_prep = false;         // the next launch prepares a projection's operand (family 0)
    double fam_bytes = 0.0;           // algorithmic bytes of the captured family's launches
    int fam_launches = 0;
    cudaGraphExec_t fam_graph = nullptr;
    int fam_graph_family = -1, fam_graph_B = -1;

    // host-side fault injection (PIPO_TEST_FAIL_ALLOC=k): the k-th device
    // allocation of pipo_init reports out-of-memory without calling cudaMalloc
    int fail_alloc_at = 0;
    int n_dalloc = 0;

    int B = 0;
    int rows = 0;                     // activation rows of the enqueue in progress (0: B, one per sequence)
    int max_rows = 0;                 // rows the activation buffers hold: max(max_batch, prefill_rows)
    int prefill_rows = 0;             // rows of a prefill chunk (positions x sequences; 0: one position at a time)
    bool prefill_tile_attn = false;   // chunk attention by tiles of positions (attn_prefill_kernel)
    // sampling in both heads (pipo_set_sampler; greedy when off)
    bool samp_on = false;
    float samp_T = 1.f, samp_p = 1.f, samp_rep = 1.f;
    int samp_k = 1, samp_nu = 0;
    float* samp_u = nullptr;          // [samp_nu][max_batch][2] draws
    int32_t* samp_step = nullptr;     // draw index of the next position
    float* samp_logits = nullptr;     // [2][max_batch][V] logits of both heads
    uint32_t* presence = nullptr;     // [max_batch][presence_w] token-history bitmap
    int presence_w = 0;
    bool prefilled = false;
    bool regular = false;             // the prefill was regular decoding (one token per backbone pass)
    std::vector<int32_t> h_len;
    cudaGraphExec_t graph = nullptr;
    int graph_B = -1;
    double plan_len = -1.0;           // mean cached length the step graph's launch plan was made for
    bool graph_regular = false;       // the captured step is a regular-decoding step
    int launches = 0;
    std::map<long long, int> occ;
    std::string err = "no error";
};

// ------------------------------------------------------------------ helpers
namespace {

pipo_status fail(pipo_ctx* c, pipo_status s, const char* fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    if (c) c->err = buf; else g_init_error = buf;
    return s;
}

#define CK(call)                                                                                  \
    do {                                                                                          \
        cudaError_t e_ = (call);                                                                  \
        if (e_ != cudaSuccess) return fail(ctx, PIPO_ECUDA, "%s: %s", #call, cudaGetErrorString(e_)); \
    } while (0)

template <typename P>
pipo_status dalloc(pipo_ctx* ctx, P** p, size_t bytes) {
    if (ctx->fail_alloc_at > 0 && ++ctx->n_dalloc == ctx->fail_alloc_at)
        return fail(ctx, PIPO_ENOMEM, "cudaMalloc(%zu bytes): injected failure of device allocation %d", bytes,
                    ctx->n_dalloc);
    void* q = nullptr;
    cudaError_t e = cudaMalloc(&q, bytes ? bytes : 16);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return fail(ctx, PIPO_ENOMEM, "cudaMalloc(%zu bytes): %s", bytes, cudaGetErrorString(e));
    }
    ctx->allocs.push_back(q);
    *p = static_cast<P*>(q);
    return PIPO_OK;
}

#define TRY(x)                              \
    do {                                    \
        pipo_status s_ = (x);               \
        if (s_ != PIPO_OK) return s_;       \
    } while (0)

// copy n elements from a host or device source (UVA) into dst + offset
pipo_status put(pipo_ctx* ctx, void* dst, size_t off_elems, const void* src, size_t n_elems) {
    if (!src) return fail(ctx, PIPO_EINVAL, "missing weight tensor");
    CK(cudaMemcpy(static_cast<char*>(dst) + off_elems * ctx->esz, src, n_elems * ctx->esz, cudaMemcpyDefault));
    return PIPO_OK;
}

pipo_status upload(pipo_ctx* ctx, void** dst, const void* src, size_t n) {
    TRY(dalloc(ctx, reinterpret_cast<char**>(dst), n * ctx->esz));
    return put(ctx, *dst, 0, src, n);
}

const void* at(const void* p, size_t off_elems, size_t esz) {
    return p ? static_cast<const char*>(p) + off_elems * esz : nullptr;
}

pipo_status upload_block(pipo_ctx* ctx, BlockW& bw, int l, const void* an, const void* wq, const void* wk,
                         const void* wv, const void* wo, const void* fn, const void* wg, const void* wu,
                         const void* wd) {
    const pipo_config& c = ctx->cfg;
    const size_t H = c.hidden, qd = (size_t)c.n_q_heads * c.head_dim, kd = (size_t)c.n_kv_heads * c.head_dim,
                 F = c.ffn, e = ctx->esz;
    TRY(upload(ctx, &bw.attn_norm, at(an, l * H, e), H));
    TRY(dalloc(ctx, reinterpret_cast<char**>(&bw.Wqkv), (qd + 2 * kd) * H * e));
    TRY(put(ctx, bw.Wqkv, 0, at(wq, l * qd * H, e), qd * H));
    TRY(put(ctx, bw.Wqkv, qd * H, at(wk, l * kd * H, e), kd * H));
    TRY(put(ctx, bw.Wqkv, (qd + kd) * H, at(wv, l * kd * H, e), kd * H));
    TRY(upload(ctx, &bw.Wo, at(wo, l * H * qd, e), H * qd));
    TRY(upload(ctx, &bw.ffn_norm, at(fn, l * H, e), H));
    // gate|up interleaved by row: row 2f = gate_f, row 2f+1 = up_f
    TRY(dalloc(ctx, reinterpret_cast<char**>(&bw.Wgu), 2 * F * H * e));
    if (!wg || !wu) return fail(ctx, PIPO_EINVAL, "missing gate/up weights");
    CK(cudaMemcpy2D(bw.Wgu, 2 * H * e, at(wg, l * F * H, e), H * e, H * e, F, cudaMemcpyDefault));
    CK(cudaMemcpy2D(static_cast<char*>(bw.Wgu) + H * e, 2 * H * e, at(wu, l * F * H, e), H * e, H * e, F,
                    cudaMemcpyDefault));
    TRY(upload(ctx, &bw.Wdown, at(wd, l * H * F, e), H * F));
    return PIPO_OK;
}

int next_pow2_le8(int b) {
    int nb = 1;
    while (nb < b && nb < 8) nb <<= 1;
    return nb;
}

// launch handles of the GEMV kernels of weight type T (k_gemv_*.cu)
template <typename T>
void* pick_gemv(int nb, bool two) {
    return std::is_same<T, bf16>::value ? k_pick_gemv_bf16(nb, two) : k_pick_gemv_f32(nb, two);
}
template <typename T>
void* pick_stream(int nb, int ru, bool rows) {
    return std::is_same<T, bf16>::value ? k_pick_stream_bf16(nb, ru, rows) : k_pick_stream_f32(nb, ru, rows);
}

constexpr size_t kXsBudget = 100 * 1024;      // staged-input bytes per v0 GEMV block
// shared memory of the staged register-ring attention (the CTA's slice of
// cached keys and values); longer slices take the register ring alone
constexpr size_t kAttnStageMax = 160 * 1024;
constexpr size_t kStreamBudget = 200 * 1024;  // staged-input bytes per streaming GEMV block

// Launch with programmatic dependent launch (decode graph) and an optional
// cluster dimension.
pipo_status launch_ex(pipo_ctx* ctx, const void* fn, dim3 grid, dim3 block, size_t smem, void** args,
                      int cluster_x = 1) {
    if (ctx->only_family >= 0) {
        // family capture: keep the launches of one family, in step order
        const int fam = ctx->launch_prep ? 0 : ctx->prof_kind;
        const bool keep = fam == ctx->only_family;
        if (keep) {
            ctx->fam_bytes += ctx->prof_bytes;
            ctx->fam_launches++;
        }
        ctx->prof_kind = 2;
        ctx->prof_bytes = 0.0;
        ctx->launch_prep = false;
        if (!keep) return PIPO_OK;
    }
    cudaLaunchConfig_t lc = {};
    lc.gridDim = grid;
    lc.blockDim = block;
    lc.dynamicSmemBytes = smem;
    lc.stream = ctx->stream;
    cudaLaunchAttribute at[2];
    int na = 0;
    if (ctx->pdl) {
        at[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        at[na].val.programmaticStreamSerializationAllowed = 1;
        ++na;
    }
    if (cluster_x > 1) {
        at[na].id = cudaLaunchAttributeClusterDimension;
        at[na].val.clusterDim.x = cluster_x;
        at[na].val.clusterDim.y = 1;
        at[na].val.clusterDim.z = 1;
        ++na;
    }
    lc.attrs = at;
    lc.numAttrs = na;
    if (ctx->prof) {
        while (ctx->prof_ev.size() < 2 * (ctx->prof_n + 1)) {
            cudaEvent_t e;
            CK(cudaEventCreate(&e));
            ctx->prof_ev.push_back(e);
        }
        CK(cudaEventRecord(ctx->prof_ev[2 * ctx->prof_n], ctx->stream));
    }
    CK(cudaLaunchKernelExC(&lc, fn, args));
    if (ctx->prof) {
        CK(cudaEventRecord(ctx->prof_ev[2 * ctx->prof_n + 1], ctx->stream));
        ctx->prof_k.push_back(ctx->prof_kind);
        ctx->prof_b.push_back(ctx->prof_bytes);
        ctx->prof_n++;
    }
    // the kind and bytes describe one launch: callers set them before it
    ctx->prof_kind = 2;
    ctx->prof_bytes = 0.0;
    ctx->launch_prep = false;
    ctx->launches++;
    return PIPO_OK;
}

size_t g_smem_optin = 0;  // opt-in shared memory per block of the device


// bh: batch columns of the tensor-core GEMM (its MMA N is 2 * bh: hi | lo)
size_t tc_smem(int bh, bool deep = false) {
    const int st = tc_stages(bh, deep);
    return 1024 + (size_t)st * (kTcABytes + (size_t)2 * bh * kTcBK * 2) + (2 * st + 1) * 8;
}

// kernel variants of the tensor-core projection (k_tc.cu): fused (activation
// split inside the GEMM) or fed by prep_bf16_kernel; deep (one CTA per SM) or not
void* pick_tc(int bh, bool deep = false) { return k_pick_tcv(bh, deep, false); }
void* pick_tcv(int bh, bool deep, bool fused) { return k_pick_tcv(bh, deep, fused); }
size_t tcv_smem(int bh, bool deep, bool fused) {
    if (!fused) return tc_smem(bh, deep);
    const int st = tcf_stages(bh, deep);
    return 1024 + (size_t)st * tcf_stage_bytes(bh) + (3 * st + 1) * 8;
}
int tcv_threads(bool fused) { return fused ? kTcfThreads : kTcThreads; }

bool tc_cluster_spread();
void* attnm_pick(int G, bool deep = false);

cudaError_t set_smem_attrs(bool bf) {
    int dev = 0, optin = 0;
    cudaError_t e0 = cudaGetDevice(&dev);
    if (e0 == cudaSuccess) e0 = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    if (e0 != cudaSuccess) return e0;
    g_smem_optin = (size_t)optin;
    for (int nb : {1, 2, 4})
        for (int ru : {1, 2})
            for (bool rows : {false, true}) {
                void* f = bf ? pick_stream<bf16>(nb, ru, rows) : pick_stream<float>(nb, ru, rows);
                cudaError_t e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kStreamBudget);
                if (e != cudaSuccess) return e;
            }
    const int nbs[4] = {1, 2, 4, 8};
    for (int i = 0; i < 4; ++i)
        for (int two = 0; two < 2; ++two) {
            void* f = bf ? pick_gemv<bf16>(nbs[i], two) : pick_gemv<float>(nbs[i], two);
            cudaError_t e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kXsBudget);
            if (e != cudaSuccess) return e;
        }
    for (int dh : {64, 128})
        for (int g : {1, 2, 4, 8})
            for (void* f : {k_pick_attn_cluster(bf, dh, g), k_pick_attn_flat(bf, dh, g)}) {
                if (!f) continue;
                cudaError_t e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kAttnStageMax);
                if (e != cudaSuccess) return e;
            }
    if (bf)
        for (int g : {1, 2, 4})
            for (void* f : {attnm_pick(g), k_pick_attn_mma_flat(g), attnm_pick(g, true)}) {
                const size_t smem = f == attnm_pick(g, true) ? mma_attn_smem(8, kMmaDeepStages) : mma_attn_smem();
                cudaError_t e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
                if (e != cudaSuccess) return e;
            }
    if (bf)
        for (int bn : {16, 32, 64, 128})
            for (bool deep : {false, true})
                for (bool fused : {false, true}) {
                    void* fn = pick_tcv(bn, deep, fused);
                    cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                         (int)tcv_smem(bn, deep, fused));
                    if (e != cudaSuccess) return e;
                    e = cudaFuncSetAttribute(fn, cudaFuncAttributeClusterSchedulingPolicyPreference,
                                             tc_cluster_spread() ? cudaClusterSchedulingPolicySpread
                                                                 : cudaClusterSchedulingPolicyLoadBalancing);
                    if (e != cudaSuccess) return e;
                }
    return cudaSuccess;
}

// ---------------------------------------------------- tensor-core projections
PFN_cuTensorMapEncodeTiled_v12000 g_encode_tiled = nullptr;
std::mutex g_encode_mu;

// the driver's tensor-map encoder, looked up once
pipo_status load_encoder(pipo_ctx* ctx) {
    std::lock_guard<std::mutex> lk(g_encode_mu);
    if (!g_encode_tiled) {
        void* fn = nullptr;
        cudaDriverEntryPointQueryResult q{};
        CK(cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q));
        if (q != cudaDriverEntryPointSuccess || !fn)
            return fail(ctx, PIPO_ECUDA, "cuTensorMapEncodeTiled is not available");
        g_encode_tiled = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    }
    return PIPO_OK;
}

// 2-D bf16 tensor map over a row-major [rows, K] matrix: boxes of 64 x box_rows
// elements, 128-byte swizzle (the layout the tcgen05 descriptors expect).
pipo_status make_tmap(pipo_ctx* ctx, CUtensorMap* tm, const void* base, int K, int rows, int box_rows) {
    TRY(load_encoder(ctx));
    if (reinterpret_cast<uintptr_t>(base) % 16 != 0 || K % kTcBK != 0 || rows < box_rows)
        return fail(ctx, PIPO_EINVAL, "tensor map: base %% 16, K %% 64 and rows >= %d required", box_rows);
    const cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)rows};
    const cuuint64_t strides[1] = {(cuuint64_t)K * 2};
    const cuuint32_t box[2] = {(cuuint32_t)kTcBK, (cuuint32_t)box_rows};
    const cuuint32_t es[2] = {1, 1};
    const CUresult r = g_encode_tiled(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
                                      box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                                      CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(ctx, PIPO_ECUDA, "cuTensorMapEncodeTiled: error %d", (int)r);
    return PIPO_OK;
}

// 2-D fp32 tensor map over activations [rows][ld] (first K columns): boxes of
// 64 x box_rows elements, no swizzle; rows past `rows` read as zeros.
pipo_status make_tmap_x(pipo_ctx* ctx, CUtensorMap* tm, const float* base, int K, int ld, int rows, int box_rows) {
    TRY(load_encoder(ctx));
    if (!base || reinterpret_cast<uintptr_t>(base) % 16 != 0 || K % kTcBK != 0 || ld % 4 != 0 || rows < 1)
        return fail(ctx, PIPO_EINVAL, "activation tensor map: base %% 16, K %% 64, ld %% 4 required");
    const cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)rows};
    const cuuint64_t strides[1] = {(cuuint64_t)ld * 4};
    const cuuint32_t box[2] = {(cuuint32_t)kTcBK, (cuuint32_t)box_rows};
    const cuuint32_t es[2] = {1, 1};
    const CUresult r = g_encode_tiled(tm, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<float*>(base), dims, strides,
                                      box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                                      CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(ctx, PIPO_ECUDA, "cuTensorMapEncodeTiled (activations): error %d", (int)r);
    return PIPO_OK;
}

int tc_bn(int B) { return B <= 16 ? 16 : B <= 32 ? 32 : B <= 64 ? 64 : 128; }

// resident CTAs per SM of the tensor-core GEMM at this BN (shared memory bound)
int tc_ctas_per_sm(int bn, bool deep = false, bool fused = false) {
    const size_t per = tcv_smem(bn, deep, fused) + 48 * (size_t)bn + 1024;  // dynamic + static + reserve
    return std::max(1, (int)(g_smem_optin ? 228 * 1024 / per : 1));
}

// Cluster placement of the tensor-core GEMM: load-balancing (several CTAs of
// a cluster may share an SM) unless PIPO_TC_CLUSTER_SPREAD=1.
bool tc_cluster_spread() {
    static const bool v = [] {
        const char* ev = getenv("PIPO_TC_CLUSTER_SPREAD");
        return ev && ev[0] == '1';
    }();
    return v;
}

// Clusters of `cs` CTAs of the GEMM at batch width bh that can be resident at
// once on the current device (cudaOccupancyMaxActiveClusters; cached).
int tc_max_clusters(int bh, int cs, bool deep, bool fused) {
    static std::mutex mu;
    static std::map<long long, int> cache;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) { cudaGetLastError(); return 0; }
    const long long key =
        ((long long)dev << 20) | ((long long)fused << 17) | ((long long)deep << 16) | ((long long)bh << 8) | cs;
    std::lock_guard<std::mutex> lk(mu);
    auto it = cache.find(key);
    if (it != cache.end()) return it->second;
    cudaLaunchConfig_t lc = {};
    lc.gridDim = dim3(cs);
    lc.blockDim = dim3(tcv_threads(fused));
    lc.dynamicSmemBytes = tcv_smem(bh, deep, fused);
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = cs;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    lc.attrs = at;
    lc.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, pick_tcv(bh, deep, fused), &lc) != cudaSuccess) {
        cudaGetLastError();
        n = 0;
    }
    cache[key] = n;
    return n;
}

// Launch plan of a tensor-core projection: the K splits (the cluster size)
// and the pipeline variant (the two-per-SM ring, or the deep ring of one CTA
// per SM).  Each split has at least kTcMinKb 64-wide K blocks, at most
// kTcMaxSplits, and the clusters must fit in `waves` waves.
constexpr int kTcMinKb = 4;
struct TcPlan {
    int splits;
    bool deep;
};
TcPlan tc_plan(int sms, int bn, int tiles, int nkb, bool fused, bool allow_deep = true) {
    static const int force_deep = [] {
        const char* ev = getenv("PIPO_TC_DEEP");
        return ev ? atoi(ev) : -1;
    }();
    // K splits planned for up to `waves` waves of CTAs on the two-per-SM ring.
    // Measured (GB300, graph replay, ms per step; two waves on the two-per-SM
    // ring / one wave with the deep ring where the tiles fit one per SM /
    // one wave on the two-per-SM ring): 9b-b8 4.30 / 4.52 / 4.61, 4b-b16
    // 2.83 / 2.96 / 3.17, 4b-b4 2.62 / 2.90 / 2.92, 4b-lc 4.49 / 4.76 / 4.77,
    // 4b-b64 5.41 / 5.41 / 5.78; three or four waves, or two with the deep
    // ring, were slower.  More waves let the hardware scheduler even out the
    // SMs' finishing times; the splits of a tile stay one cluster.
    // PIPO_TC_WAVES=1 restores the one-wave plan (deep ring when the tiles
    // fit one per SM), PIPO_TC_DEEP=1 forces the deep ring.
    static const int waves = [] {
        const char* ev = getenv("PIPO_TC_WAVES");
        return ev ? std::max(1, atoi(ev)) : 2;
    }();
    const bool deep = force_deep >= 0 ? force_deep == 1 : (waves == 1 && allow_deep && tiles <= sms);
    const int target = sms * tc_ctas_per_sm(bn, deep, fused);
    if (tiles >= target * waves) return {1, deep};
    static const bool verbose = getenv("PIPO_VERBOSE") != nullptr;
    for (int s = std::min({target * waves / tiles, nkb / kTcMinKb, kTcMaxSplits}); s >= 2; --s) {
        const int mc = tc_max_clusters(bn, s, deep, fused);
        if (verbose)
            fprintf(stderr, "[pipo] tc plan: bh=%d deep=%d tiles=%d nkb=%d s=%d max_clusters=%d\n", bn, (int)deep, tiles,
                    nkb, s, mc);
        if (mc * waves >= tiles) return {s, deep};
    }
    return {1, deep};
}

// The activation split can run inside the GEMM: activation segments only (no
// embedding gathers), at most one RMSNorm (a single segment, or one joint norm
// over both), TMA-addressable rows.
bool tcf_eligible(const GemvParams& p) {
    for (int s = 0; s < p.nseg; ++s) {
        const Seg& sg = p.seg[s];
        if (!sg.src || reinterpret_cast<uintptr_t>(sg.src) % 16 != 0 || sg.ld % 4 != 0 || sg.K % kTcBK != 0) return false;
    }
    if (p.nseg == 2 && !p.joint_norm && (p.seg[0].gamma || p.seg[1].gamma)) return false;
    if (p.zero_ptr && p.epi == EPI_ARGMAX) return false;  // block 0 zeroes keys the other blocks update
    return true;
}

bool tc_prep_forced() {
    const char* ev = getenv("PIPO_TC_PREP");
    return ev && ev[0] == '1';
}

// Widest batch width that runs the fused form.  Measured on the 4B shapes:
// fused ahead at BH 16 (B = 4: 3.08 -> 2.84 ms, B = 16: 3.29 -> 2.86 ms per
// step), behind at BH 64 (5.02 -> 5.33 ms), where the fp32 activation tile
// halves the pipeline depth.  PIPO_TC_FUSED_MAX_BH overrides.
int tc_fused_max_bh() {
    static const int v = [] {
        const char* ev = getenv("PIPO_TC_FUSED_MAX_BH");
        return ev ? atoi(ev) : 32;
    }();
    return v;
}

// Projection on the tensor cores: the fused GEMM, or bf16 activations from
// prep_bf16_kernel and then the tcgen05 GEMM.  Eligible: bf16 weights,
// K % 64 == 0, rows >= 128, B <= 128.  x_rows: rows behind each activation
// pointer (the tensor maps read no further; at least BH for box-sized maps).
pipo_status launch_gemm_tc(pipo_ctx* ctx, const GemvParams& p, bf16* xb, int splits_req, int x_rows) {
    const int ru = p.epi == EPI_SWIGLU ? 2 : 1;
    const int rows = p.N * ru, bn = tc_bn(p.B), tiles = (rows + kTcM - 1) / kTcM, nkb = p.K / kTcBK;
    const bool fused = tcf_eligible(p) && !tc_prep_forced() && x_rows >= bn && bn <= tc_fused_max_bh();
    // PIPO_TC_SWIGLU_SHALLOW=1: the gate/up projection on the two-per-SM ring
    // (in isolation at B = 16: 22.9 us with two K splits against 24.8 us deep)
    static const bool swiglu_shallow = [] {
        const char* ev = getenv("PIPO_TC_SWIGLU_SHALLOW");
        return ev && ev[0] == '1';
    }();
    const bool allow_deep = !ctx->tc_shallow && !(swiglu_shallow && p.epi == EPI_SWIGLU);
    TcPlan plan = tc_plan(ctx->sms, bn, tiles, nkb, fused, allow_deep);
    if (splits_req > 0) plan.splits = std::min({splits_req, nkb, kTcMaxSplits});
    TcParams tp{};
    tp.rows = rows; tp.K = p.K; tp.B = p.B; tp.ru = ru; tp.epi = p.epi;
    tp.y = p.y; tp.ldy = p.ldy; tp.bias = p.bias; tp.am = p.am; tp.dbg = p.dbg; tp.ld_dbg = p.ld_dbg;
    tp.splits = plan.splits;
    if (fused) {
        CUtensorMap tmW, tmX0, tmX1;
        TRY(make_tmap(ctx, &tmW, p.W, p.K, rows, kTcM));
        TRY(make_tmap_x(ctx, &tmX0, p.seg[0].src, p.seg[0].K, p.seg[0].ld, x_rows, bn));
        if (p.nseg == 2) TRY(make_tmap_x(ctx, &tmX1, p.seg[1].src, p.seg[1].K, p.seg[1].ld, x_rows, bn));
        else tmX1 = tmX0;
        TcfIn in{};
        in.nseg = p.nseg;
        in.K0 = p.seg[0].K;
        in.norm = p.seg[0].gamma != nullptr;
        in.klen = p.joint_norm ? p.K : p.seg[0].K;
        in.gamma = p.seg[0].gamma;
        in.eps = p.eps;
        in.B = p.B;
        in.zero_ptr = p.zero_ptr;
        in.zero_n = p.zero_n;
        void* args[] = {&tmW, &tmX0, &tmX1, &in, &tp};
        ctx->prof_kind = 0;
        ctx->prof_bytes = (double)rows * p.K * 2;
        return launch_ex(ctx, pick_tcv(bn, plan.deep, true), dim3(tiles * plan.splits), dim3(kTcfThreads),
                         tcv_smem(bn, plan.deep, true), args, plan.splits);
    }
    const int splits = plan.splits;
    CUtensorMap tmW, tmX;
    TRY(make_tmap(ctx, &tmW, p.W, p.K, rows, kTcM));
    TRY(make_tmap(ctx, &tmX, xb, p.K, 2 * bn, 2 * bn));
    {
        GemvParams pp = p;
        int bh = bn;
        void* args[] = {&pp, &xb, &bh};
        ctx->prof_kind = 2;
        ctx->prof_bytes = 0.0;
        ctx->launch_prep = true;
        TRY(launch_ex(ctx, reinterpret_cast<const void*>(k_pick_prep_bf16()), dim3(bn), dim3(kPrepThreads), 0,
                      args));
    }
    void* args[] = {&tmW, &tmX, &tp};
    ctx->prof_kind = 0;
    ctx->prof_bytes = (double)rows * p.K * 2;
    return launch_ex(ctx, pick_tc(bn, plan.deep), dim3(tiles * splits), dim3(kTcThreads), tc_smem(bn, plan.deep), args,
                     splits);
}

bool tc_eligible(const pipo_ctx* ctx, const GemvParams& p) {
    const int rows = p.N * (p.epi == EPI_SWIGLU ? 2 : 1);
    return ctx->cfg.dtype == 1 && ctx->tc_xb && p.B >= ctx->tc_min_b && p.B <= ctx->tc_bn_max &&
           p.K % kTcBK == 0 && p.K <= ctx->tc_kmax && p.K <= 4 * kPrepQ * kPrepThreads && rows >= kTcM;
}

pipo_status launch_gemv(pipo_ctx* ctx, GemvParams p) {
    const bool bf = ctx->cfg.dtype == 1;
    const bool two = p.epi == EPI_SWIGLU;
    if (tc_eligible(ctx, p))
        return launch_gemm_tc(ctx, p, ctx->tc_xb, ctx->tc_splits, ctx->act_rows);
    ctx->prof_kind = 0;
    ctx->prof_bytes = (double)p.N * (two ? 2 : 1) * p.K * ctx->esz;
    if (p.B <= 4) {
        // streaming kernel: one CTA per SM, chunk-balanced, deterministic
        int nb = std::min(4, next_pow2_le8(std::max(1, p.B)));
        while (nb > 1 && (size_t)nb * p.K * 4 + (size_t)p.K * ctx->esz > kStreamBudget) nb >>= 1;
        if ((size_t)p.K * 4 > kStreamBudget) return fail(ctx, PIPO_EINVAL, "GEMV input length %d too large", p.K);
        const bool rows = ((size_t)p.K * ctx->esz) % 512 == 0;
        const size_t xbytes = (size_t)nb * p.K * 4;
        void* fn = bf ? pick_stream<bf16>(nb, two ? 2 : 1, rows) : pick_stream<float>(nb, two ? 2 : 1, rows);
        void* args[] = {&p};
        // staged input, then (row kernel) the RMSNorm gains in their storage type
        const size_t smem = xbytes + (rows ? (size_t)p.K * ctx->esz + 16 : 0);
        return launch_ex(ctx, fn, dim3(ctx->sms * kStreamCtasPerSm), dim3(kStreamThreads), smem, args);
    }
    int nb = next_pow2_le8(std::max(1, p.B));
    while (nb > 1 && (size_t)nb * p.K * 4 > kXsBudget) nb >>= 1;
    if ((size_t)p.K * 4 > kXsBudget) return fail(ctx, PIPO_EINVAL, "GEMV input length %d too large", p.K);
    const size_t smem = (size_t)nb * p.K * 4;
    void* fn = bf ? pick_gemv<bf16>(nb, two) : pick_gemv<float>(nb, two);
    const long long key = (reinterpret_cast<long long>(fn) << 1) ^ (long long)smem;
    int per_sm;
    auto it = ctx->occ.find(key);
    if (it == ctx->occ.end()) {
        CK(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, kThreads, smem));
        ctx->occ[key] = per_sm;
    } else {
        per_sm = it->second;
    }
    per_sm = std::max(1, per_sm);
    if (p.splitk < 1) p.splitk = 1;
    const long long tasks = (long long)p.N * p.splitk;
    const int grid = (int)std::max(1LL, std::min<long long>((tasks + kWarps - 1) / kWarps, (long long)ctx->sms * per_sm));
    void* args[] = {&p};
    return launch_ex(ctx, fn, dim3(grid), dim3(kThreads), smem, args);
}

Seg act_seg(const float* src, int ld, int K, const void* gamma = nullptr) {
    Seg s{};
    s.src = src; s.ld = ld; s.K = K; s.gamma = gamma;
    return s;
}

GemvParams gemv_base(pipo_ctx* ctx, const void* W, int N, int epi, float* y, int ldy) {
    GemvParams p{};
    p.W = W; p.N = N; p.epi = epi; p.y = y; p.ldy = ldy;
    p.B = ctx->rows > 0 ? ctx->rows : ctx->B; p.splitk = 1; p.eps = ctx->cfg.rms_eps; p.nseg = 1;
    return p;
}

int resadd_splits(pipo_ctx* ctx, int N, int K) {
    const long long target = (long long)ctx->sms * kWarps * 2 * 4;
    int s = (int)std::max(1LL, (target + N - 1) / N);
    s = std::min(s, std::max(1, K / 256));
    return s;
}

int attn_splits(const pipo_ctx* ctx, int B) {
    const pipo_config& c = ctx->cfg;
    int s = (2 * ctx->sms + B * c.n_kv_heads - 1) / (B * c.n_kv_heads);
    s = std::max(1, std::min(s, (c.max_ctx + 15) / 16));
    return s;
}

// attention launch handles (k_attn.cu)
void* attn_pick(bool bf, int DH, int G) { return k_pick_attn_decode(bf, DH, G); }
// one kernel for every cluster size (read from the cluster at run time)
void* attnc_pick(bool bf, int DH, int G) { return k_pick_attn_cluster(bf, DH, G); }
// tensor-core attention (bf16 cache, d_h = 128, 1, 2 or 4 query heads per kv head)
void* attnm_pick(int G, bool deep) { return k_pick_attn_mma(G, deep); }

// Can a 16-CTA cluster of this kernel be scheduled here?  (sets the
// non-portable cluster attribute; any failure selects 8)
bool cluster16_ok(bool bf, int DH, int G) {
    void* fn = attnc_pick(bf, DH, G);
    if (!fn) return false;
    if (cudaFuncSetAttribute(fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    cudaLaunchConfig_t lc = {};
    lc.gridDim = dim3(16, 1, 1);
    lc.blockDim = dim3(kAttnThreads);
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = 16;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    lc.attrs = at;
    lc.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, fn, &lc) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return n > 0;
}

void* rope_pick(bool bf, int DH) { return k_pick_rope_append(bf, DH); }

KVView kv_view(pipo_ctx* ctx, int layer) {
    KVView v;
    v.K = static_cast<char*>(ctx->Kc) + (size_t)layer * ctx->layer_elems * ctx->esz;
    v.V = static_cast<char*>(ctx->Vc) + (size_t)layer * ctx->layer_elems * ctx->esz;
    v.table = ctx->block_table;
    v.blocks_per_seq = ctx->blocks_per_seq;
    v.page = ctx->cfg.page_size;
    v.n_kv = ctx->cfg.n_kv_heads;
    return v;
}

// One shared-memory carveout preference for every kernel of a step
// (PIPO_CARVEOUT=<percent>; default: the driver's choice).  Measured on the
// 4B shapes: a 100 % carveout for all kernels helps the tensor-core attention
// next to the small-batch GEMVs and slows the register-ring attention, while
// the driver's choice with the kernel selection of attn_use_mma is as fast.
cudaError_t set_carveouts(bool bf) {
    int pct = -1;
    if (const char* ev = getenv("PIPO_CARVEOUT")) pct = atoi(ev);
    if (pct < 0) return cudaSuccess;
    std::vector<const void*> fns;
    for (int nb : {1, 2, 4, 8})
        for (int two = 0; two < 2; ++two) fns.push_back(bf ? pick_gemv<bf16>(nb, two) : pick_gemv<float>(nb, two));
    for (int nb : {1, 2, 4})
        for (int ru : {1, 2}) {
            for (bool rows : {false, true})
                fns.push_back(bf ? pick_stream<bf16>(nb, ru, rows) : pick_stream<float>(nb, ru, rows));
        }
    if (bf) {
        for (int bn : {16, 32, 64, 128})
            for (bool deep : {false, true})
                for (bool fused : {false, true}) fns.push_back(pick_tcv(bn, deep, fused));
        fns.push_back(reinterpret_cast<const void*>(k_pick_prep_bf16()));
        for (int g : {1, 2, 4})
            for (bool deep : {false, true}) fns.push_back(attnm_pick(g, deep));
    }
    for (int dh : {64, 128}) {
        for (int g : {1, 2, 4, 8}) {
            fns.push_back(attnc_pick(bf, dh, g));
            fns.push_back(attn_pick(bf, dh, g));
        }
        fns.push_back(rope_pick(bf, dh));
    }
    fns.push_back(bf ? (const void*)&accept_kernel<bf16> : (const void*)&accept_kernel<float>);
    fns.push_back((const void*)&advance_kernel);
    for (const void* f : fns) {
        if (!f) continue;
        const cudaError_t e = cudaFuncSetAttribute(f, cudaFuncAttributePreferredSharedMemoryCarveout, pct);
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

// the tensor-core attention applies: bf16 cache, d_h = 128, G in {1, 2, 4},
// pages of whole 16-entry groups
bool attn_mma_ok(const pipo_ctx* ctx) {
    const pipo_config& c = ctx->cfg;
    const int G = c.n_q_heads / c.n_kv_heads;
    return !ctx->attn_regs && c.dtype == 1 && c.head_dim == kMmaDH && (G == 1 || G == 2 || G == 4) &&
           c.page_size % kMmaRun == 0;
}

// ... and is used: from the batch at which the projections move to the tensor
// cores (measured: below it the register-ring attention is slightly faster
// next to the CUDA-core GEMVs, from B = 4 the tensor-core one by far), with
// the cache tensor maps in place
bool attn_use_mma(const pipo_ctx* ctx, int B) {
    return attn_mma_ok(ctx) && B >= std::min(ctx->tc_min_b, ctx->attn_mma_min_b) &&
           (int)ctx->kv_tm.size() == 2 * ctx->n_cache_layers;
}

// Mean cached length (pairs per sequence) the launch plan is made for.  A
// captured step graph keeps its launches while the caches grow, so the
// length is frozen at its capture: later captures of kernel families and
// pipo_describe_step then see the plan the graph runs.  Without a graph, the
// current mean.
double plan_mean_len(const pipo_ctx* ctx) {
    if (ctx->graph && ctx->plan_len >= 0.0) return ctx->plan_len;
    double sum = 0.0;
    int n = 0;
    for (int b = 0; b < ctx->B && b < (int)ctx->h_len.size(); ++b, ++n) sum += ctx->h_len[b];
    return n > 0 ? sum / n : 0.0;
}

bool attn_mma_deep_on();

// CTAs per (sequence, kv head) of the clustered attention: 8 while the batch
// leaves SMs idle (16 where allowed and still under two per SM), fewer as the
// (sequence, kv head) pairs alone fill the GPU.
int attn_cluster_size(const pipo_ctx* ctx, int B) {
    if (ctx->attn_cs_force) return ctx->attn_cs_force;
    // one sequence on the tensor-core attention: 8-CTA clusters on the deep
    // stage ring when every CTA has an SM of its own, else 4.  4b-b1 (ms per
    // step): 8-CTA deep 2.463, 4-CTA deep 2.571, 4-CTA with 10 stages 2.615
    // (an 8-CTA slice of ~1160 pairs spans 10 or 11 groups of 16: one more
    // than 10 stages hold)
    if (B == 1 && attn_use_mma(ctx, B))
        return attn_mma_deep_on() && (long long)ctx->cfg.n_kv_heads * 8 <= ctx->sms ? 8 : 4;
    const long long pairs = (long long)B * ctx->cfg.n_kv_heads;
    if (ctx->attn_cs16 && pairs * 16 <= 2 * ctx->sms) return 16;
    // measured best: about two tensor-core attention CTAs per SM (they are
    // resident two at a time), one register-ring CTA per SM
    const long long target = ctx->attn_cs_target > 0 ? ctx->attn_cs_target : (attn_use_mma(ctx, B) ? 2 : 1);
    int cs = 8;
    while (cs > 1 && pairs * cs > target * ctx->sms) cs >>= 1;
    return cs;
}

// The register-ring decode attention without clusters (one CTA per SM, split
// partials merged through global memory by the last arrival) against the
// 8-CTA clusters (distributed-shared-memory merge), decided by the mean cached
// length at graph capture.  Measured at 4B B = 1: 1156 entries 2.689 ms
// (unclustered) against 2.660 ms per step; 8212 entries 3.082 against 3.539 ms.
constexpr int kFlatMinEntries = 2048;
bool attn_flat_now(const pipo_ctx* ctx) {
    if (ctx->attn_flat <= 0) return false;
    if (ctx->attn_flat >= 2) return true;
    return plan_mean_len(ctx) >= kFlatMinEntries;
}

// The QKV projection of a decode step on the streaming GEMV prefetches the
// layer's cached key and value pages into L2 before its dependency wait, so
// that the attention's copies, issued when its CTAs find room (as the
// projection's CTAs leave), are served from L2 rather than queued behind the
// weight stream in HBM.  PIPO_ATTN_L2_WARM=0: never.
bool attn_l2_warm() {
    static const bool on = [] {
        const char* ev = getenv("PIPO_ATTN_L2_WARM");
        return ev ? atoi(ev) != 0 : true;
    }();
    return on;
}

// The deep stage ring for the clustered tensor-core attention when each of
// its CTAs has an SM of its own (rows x kv heads x cluster size <= SMs): the
// shared memory it takes then keeps no CTA of this launch from starting, and
// a CTA's slice of up to kMmaDeepStages groups is in flight from its entry.
// 4b-b1 (one sequence, ~1160 cached pairs, 4-CTA clusters, 32 CTAs):
// 2.595 ms per step with 10 stages, 2.563 with 15, 2.551 with 20.
// PIPO_ATTN_MMA_DEEP=0: never.
bool attn_mma_deep_on() {
    static const bool on = [] {
        const char* ev = getenv("PIPO_ATTN_MMA_DEEP");
        return ev ? atoi(ev) != 0 : true;
    }();
    return on;
}
bool attn_mma_deep(const pipo_ctx* ctx, int R, int cs) {
    return attn_mma_deep_on() && (long long)R * ctx->cfg.n_kv_heads * cs <= ctx->sms;
}

// Split count of the unclustered tensor-core attention, or 0 for the
// clustered one: when the (row, kv head) pairs times the largest cluster
// (8) leave SMs without two CTAs and the cached slices stay long (mean
// context at graph capture of kFlatMmaMinEntries and more), S splits fill
// one wave of two CTAs per SM, at most kFlatMaxSplits.  Measured on 4b-lc
// (B = 4, ~15.5 K cached pairs, ms per step): 8-CTA clusters (256 CTAs)
// 4.32; unclustered one wave (S = 9, 288 CTAs) 4.09; two waves (S = 19)
// 4.35; three 4.53 (more waves balance the SMs but leave no room for the
// next kernel's CTAs to start early).  One sequence at ~2180 pairs (9b-b1):
// 3.83 against 3.89 ms with the register-ring attention (unclustered), but
// 3.71 with 8-CTA clusters on the deep ring, which therefore stay while
// that ring holds a CTA's slice.
// PIPO_ATTN_MMA_WAVES sets the waves, PIPO_ATTN_MMA_FLAT=0 / 2: never / also
// for short caches.
constexpr int kFlatMmaMinEntries = 2048;
int attn_mma_flat_splits(const pipo_ctx* ctx, int R) {
    static const int mode = [] {
        const char* ev = getenv("PIPO_ATTN_MMA_FLAT");
        return ev ? atoi(ev) : 1;
    }();
    if (mode <= 0) return 0;
    const long long pairs = (long long)R * ctx->cfg.n_kv_heads;
    if (pairs * 8 >= 2LL * ctx->sms) return 0;
    const double mean = plan_mean_len(ctx);
    if (mode == 1 && mean < kFlatMmaMinEntries) return 0;
    // 8-CTA clusters on the deep ring while it holds a CTA's whole slice (a
    // slice of c entries spans at most c / 16 + 2 groups)
    if (mode == 1 && attn_mma_deep(ctx, R, 8) && mean <= 8.0 * kMmaRun * (kMmaDeepStages - 2)) return 0;
    static const int waves = [] {
        const char* ev = getenv("PIPO_ATTN_MMA_WAVES");
        return ev ? std::max(1, atoi(ev)) : 1;
    }();
    int S = (int)(2LL * waves * ctx->sms / pairs);
    if (S > 0 && mean / S < 512.0) S = (int)(2LL * ctx->sms / pairs);
    return std::max(1, std::min(S, kFlatMaxSplits));
}

// Long attention: the cached K/V bytes of a layer are at least six times the
// QKV weight bytes (cached lengths at graph capture).  Then every projection
// takes the two-per-SM ring, whose shared memory leaves room for a
// neighbouring kernel's CTAs: under programmatic dependent launch the
// attention starts streaming the cache during the QKV projection and each
// projection prefetches its weights during the kernel before it.  Measured on
// 4B (ratio of cache to QKV bytes in brackets): B=4 at ~15.9 K cached pairs
// [8.3] 5.82 -> 4.73 ms per step; B=64 at ~530 pairs [4.4] 5.07 (deep) vs
// 5.38 ms with the QKV and O projections shallow; B=16 [1.1] 2.87 (deep) vs
// 3.08 ms all shallow.  PIPO_TC_SHALLOW_ATTN=0/1 overrides.
bool attn_is_long(const pipo_ctx* ctx) {
    static const int force = [] {
        const char* ev = getenv("PIPO_TC_SHALLOW_ATTN");
        return ev ? atoi(ev) : -1;
    }();
    if (force >= 0) return force == 1;
    const pipo_config& c = ctx->cfg;
    const double ctx_sum = plan_mean_len(ctx) * std::min(ctx->B, (int)ctx->h_len.size());
    const double kv_bytes = ctx_sum * c.n_kv_heads * c.head_dim * 2.0 * ctx->esz;
    const double qkv_bytes = (double)(c.n_q_heads + 2 * c.n_kv_heads) * c.head_dim * c.hidden * ctx->esz;
    return kv_bytes >= 6.0 * qkv_bytes;
}

// Staged form of the register-ring decode attention: when the longest slice
// a CTA can get (the context capacity over `splits`) fits kAttnStageMax, the
// CTA copies its slice of cached keys and values to shared memory before the
// dependency wait and attends from there.  Returns the dynamic shared memory
// and sets *stage_max (0: the register ring alone).  PIPO_ATTN_STAGE=0 turns
// it off.
size_t attn_stage(const pipo_ctx* ctx, int splits, bool chunk, int* stage_max) {
    static const bool off = [] {
        const char* ev = getenv("PIPO_ATTN_STAGE");
        return ev && ev[0] == '0';
    }();
    *stage_max = 0;
    if (off || chunk || splits < 1) return 0;
    const pipo_config& c = ctx->cfg;
    const int entries = (c.max_ctx + splits - 1) / splits + 1;
    const size_t bytes = (size_t)entries * c.head_dim * ctx->esz * 2;
    if (bytes > kAttnStageMax) return 0;
    *stage_max = entries;
    return bytes;
}

// One decoder block on the residual stream xr (pre-norm attention + SwiGLU).
pipo_status enqueue_block(pipo_ctx* ctx, const BlockW& bw, int cache_layer, float* xr) {
    const pipo_config& c = ctx->cfg;
    const int H = c.hidden, DH = c.head_dim, qd = c.n_q_heads * DH, kd = c.n_kv_heads * DH, rows = qd + 2 * kd;
    const bool bf = c.dtype == 1;
    // RMSNorm -> fused QKV projection
    GemvParams p = gemv_base(ctx, bw.Wqkv, rows, EPI_STORE, ctx->qkv, rows);
    p.seg[0] = act_seg(xr, H, H, bw.attn_norm);
    p.K = H;
    KVView kv = kv_view(ctx, cache_layer);
    if (attn_l2_warm() && (ctx->rows <= 0 || ctx->rows == ctx->B)) {
        // a decode step: the streaming GEMV warms L2 with this layer's cached pages
        p.pf_k = kv.K;
        p.pf_v = kv.V;
        p.pf_table = kv.table;
        p.pf_npos = ctx->n_pos;
        p.pf_bps = kv.blocks_per_seq;
        p.pf_page = kv.page;
        p.pf_nseq = ctx->B;
        p.pf_bytes = (unsigned)((size_t)kv.n_kv * kv.page * DH * ctx->esz);
    }
    TRY(launch_gemv(ctx, p));
    if (!ctx->attn_v0) {
        // RoPE + KV append + split-KV attention, one cluster per (row, kv head).
        // A prefill chunk (several positions per sequence) appends all its
        // rows' entries first: its rows read each other's.
        const int R = ctx->rows > 0 ? ctx->rows : ctx->B;
        const bool chunk = R > ctx->B;
        if (chunk) {
            const float* qkv = ctx->qkv;
            int ld = rows, nq = c.n_q_heads, nseq = ctx->B;
            const int32_t* np = ctx->n_pos;
            const float* rope = ctx->rope;
            void* args[] = {(void*)&qkv, &ld, &nq, &kv, (void*)&np, &nseq, (void*)&rope};
            void* fn = k_pick_append_rows(bf, DH);
            TRY(launch_ex(ctx, fn, dim3(R, c.n_kv_heads), dim3(DH / 2), 0, args));
        }
        ctx->prof_kind = 1;
        ctx->prof_bytes = 0.0;
        for (int b = 0; b < ctx->B && b < (int)ctx->h_len.size(); ++b)
            ctx->prof_bytes += (double)(ctx->h_len[b] + 2) * kd * 2 * ctx->esz;
        AttnParams ap{};
        ap.qkv = ctx->qkv;
        ap.ld_qkv = rows;
        ap.kv = kv;
        ap.n_pos = ctx->n_pos;
        ap.rope = ctx->rope;
        ap.out = ctx->attn;
        ap.scale = 1.0f / sqrtf((float)DH);
        ap.nseq = ctx->B;
        ap.no_append = chunk ? 1 : 0;
        void* args[] = {&ap};
        const int cs = attn_cluster_size(ctx, R);
        const int G = c.n_q_heads / c.n_kv_heads;
        if (chunk && ctx->prefill_tile_attn && attn_mma_ok(ctx) && (int)ctx->kv_tm.size() == 2 * ctx->n_cache_layers) {
            // causal tiles: the positions of a tile share every key and value they read
            void* fn = k_pick_attn_prefill(G);
            CK(cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)prefill_attn_smem()));
            int C = R / ctx->B;
            const int TP = kPfVec / G;
            void* pargs[] = {&ap, &C, &ctx->kv_tm[2 * cache_layer], &ctx->kv_tm[2 * cache_layer + 1]};
            TRY(launch_ex(ctx, fn, dim3((C + TP - 1) / TP, c.n_kv_heads, ctx->B), dim3(kPfThreads),
                          prefill_attn_smem(), pargs));
        } else if (attn_use_mma(ctx, R) && !chunk && attn_mma_flat_splits(ctx, R) > 0) {
            // long caches: unclustered splits, one wave of two CTAs per SM
            ap.part_o = ctx->part_o;
            ap.part_ml = ctx->part_ml;
            ap.counters = ctx->counters;
            const int S = attn_mma_flat_splits(ctx, R);
            void* margs[] = {&ap, &ctx->kv_tm[2 * cache_layer], &ctx->kv_tm[2 * cache_layer + 1]};
            TRY(launch_ex(ctx, k_pick_attn_mma_flat(G), dim3(S, c.n_kv_heads, R), dim3(kMmaThreads), mma_attn_smem(1),
                          margs));
        } else if (attn_use_mma(ctx, R) && cs <= 8) {
            void* margs[] = {&ap, &ctx->kv_tm[2 * cache_layer], &ctx->kv_tm[2 * cache_layer + 1]};
            const bool deep = attn_mma_deep(ctx, R, cs);
            const size_t smem = mma_attn_smem(cs, deep ? kMmaDeepStages : kMmaStages);
            static const bool verbose = getenv("PIPO_VERBOSE") != nullptr;
            if (verbose) {
                int per_sm = 0;
                cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, attnm_pick(G, deep), kMmaThreads, smem);
                fprintf(stderr, "[pipo] attention: tensor-core, cluster %d, %zu B shared memory, %d CTAs per SM\n", cs,
                        smem, per_sm);
            }
            TRY(launch_ex(ctx, attnm_pick(G, deep), dim3(cs, c.n_kv_heads, R), dim3(kMmaThreads), smem, margs, cs));
        }
        else if (attn_flat_now(ctx) && !chunk && !ctx->attn_cs_force) {
            // register-ring attention over about two CTAs per SM, no cluster:
            // the split partials merge through the scratch (last arrival)
            ap.part_o = ctx->part_o;
            ap.part_ml = ctx->part_ml;
            ap.counters = ctx->counters;
            // one CTA per SM (the kernel's registers allow one), at least 16 entries per split
            const int S = std::max(1, std::min({ctx->sms / (R * c.n_kv_heads), (c.max_ctx + 15) / 16, kFlatMaxSplits}));
            const size_t smem = attn_stage(ctx, S, chunk, &ap.stage_max);
            TRY(launch_ex(ctx, k_pick_attn_flat(bf, DH, G), dim3(S, c.n_kv_heads, R), dim3(kAttnThreads), smem, args));
        } else {
            const size_t smem = attn_stage(ctx, cs, chunk, &ap.stage_max);
            TRY(launch_ex(ctx, attnc_pick(bf, DH, G), dim3(cs, c.n_kv_heads, R), dim3(kAttnThreads), smem, args,
                          cs));
        }
    } else {
    // RoPE + KV append
    {
        const float* qkv = ctx->qkv;
        int ld = rows;
        float* qo = ctx->q;
        const int32_t* np = ctx->n_pos;
        int nq = c.n_q_heads;
        double theta = c.rope_theta;
        void* args[] = {(void*)&qkv, &ld, &qo, &kv, (void*)&np, &nq, &theta};
        TRY(launch_ex(ctx, rope_pick(bf, DH), dim3(ctx->B, c.n_q_heads + 2 * c.n_kv_heads), dim3(DH / 2), 0, args));
    }
    // split-KV attention
    {
        const int S = attn_splits(ctx, ctx->B);
        const float* qp = ctx->q;
        const int32_t* np = ctx->n_pos;
        float* out = ctx->attn;
        float* po = ctx->part_o;
        float* pml = ctx->part_ml;
        unsigned* cnt = ctx->counters;
        int Sv = S;
        float scale = 1.0f / sqrtf((float)DH);
        void* args[] = {(void*)&qp, &kv, (void*)&np, &out, &po, &pml, &cnt, &Sv, &scale};
        TRY(launch_ex(ctx, attn_pick(bf, DH, c.n_q_heads / c.n_kv_heads), dim3(S, c.n_kv_heads, ctx->B), dim3(128),
                      0, args));
    }
    }
    // O projection + residual
    p = gemv_base(ctx, bw.Wo, H, EPI_RESADD, xr, H);
    p.seg[0] = act_seg(ctx->attn, qd, qd);
    p.K = qd;
    p.splitk = resadd_splits(ctx, H, qd);
    p.part = ctx->gemv_part; p.rowcnt = ctx->gemv_rowcnt;
    TRY(launch_gemv(ctx, p));
    // RMSNorm -> gate|up -> SwiGLU
    p = gemv_base(ctx, bw.Wgu, c.ffn, EPI_SWIGLU, ctx->act, c.ffn);
    p.seg[0] = act_seg(xr, H, H, bw.ffn_norm);
    p.K = H;
    TRY(launch_gemv(ctx, p));
    // down projection + residual
    p = gemv_base(ctx, bw.Wdown, H, EPI_RESADD, xr, H);
    p.seg[0] = act_seg(ctx->act, c.ffn, c.ffn);
    p.K = c.ffn;
    p.splitk = resadd_splits(ctx, H, c.ffn);
    p.part = ctx->gemv_part; p.rowcnt = ctx->gemv_rowcnt;
    TRY(launch_gemv(ctx, p));
    return PIPO_OK;
}

pipo_status enqueue_lm_head(pipo_ctx* ctx, const float* h, const void* gamma, unsigned long long* am, float* dbg) {
    const pipo_config& c = ctx->cfg;
    GemvParams p = gemv_base(ctx, ctx->E, c.vocab, EPI_ARGMAX, nullptr, 0);
    p.seg[0] = act_seg(h, c.hidden, c.hidden, gamma);
    p.K = c.hidden;
    p.am = am;
    p.dbg = dbg;
    p.ld_dbg = c.vocab;
    return launch_gemv(ctx, p);
}

// x = a + b of every row's pair (the residual MLP compressor's residual term).
pipo_status enqueue_pair_sum(pipo_ctx* ctx, const int32_t* pairs, int rows) {
    const pipo_config& c = ctx->cfg;
    const void* E = ctx->E;
    const void* pad = ctx->x_pad;
    int ld = 2, V = c.vocab, H = c.hidden;
    float* x = ctx->x;
    void* args[] = {(void*)&E, (void*)&pad, (void*)&pairs, &ld, &V, &H, &x};
    return launch_ex(ctx, c.dtype == 1 ? (const void*)&pair_sum_kernel<bf16> : (const void*)&pair_sum_kernel<float>,
                     dim3(rows), dim3(256), 0, args);
}

// The evaluation sampler on one head's logits (sample_kernel): the pick
// replaces the head's argmax key; the backbone head's pick joins the history.
pipo_status enqueue_sample(pipo_ctx* ctx, const float* logits, int head, unsigned long long* am) {
    const pipo_config& c = ctx->cfg;
    SampParams sp{};
    sp.logits = logits;
    sp.ld = c.vocab;
    sp.V = c.vocab;
    sp.presence = ctx->presence;
    sp.presence_add = head == 0 ? ctx->presence : nullptr;
    sp.W = ctx->presence_w;
    sp.inv_T = 1.0f / ctx->samp_T;
    sp.top_p = ctx->samp_p;
    sp.rep = ctx->samp_rep;
    sp.top_k = ctx->samp_k;
    sp.u = ctx->samp_u;
    sp.u_step = ctx->samp_step;
    sp.n_u = ctx->samp_nu;
    sp.u_rows = c.max_batch;
    sp.head = head;
    sp.am = am;
    void* args[] = {&sp};
    return launch_ex(ctx, (const void*)&sample_kernel, dim3(ctx->B), dim3(kSampThreads), 0, args);
}

// One pair position of every sequence.  DECODE: the pending pair; PREFILL_*:
// prompt pair j.  PREFILL_MID stops after the MTP block (teacher-forced token).
pipo_status enqueue_position(pipo_ctx* ctx, Mode mode, int j) {
    const pipo_config& c = ctx->cfg;
    ctx->tc_shallow = attn_is_long(ctx);
    const int H = c.hidden, B = ctx->B;
    const bool bf = c.dtype == 1;
    unsigned long long* am_b = ctx->am;
    unsigned long long* am_d = ctx->am + c.max_batch;

    // pair embed + compressor (Eq. 1)
    const int32_t* pairs = (mode == DECODE) ? ctx->pending : ctx->pf_pairs + (size_t)j * B * 2;
    Seg s0{}, s1{};
    s0.table = ctx->E; s0.pad = ctx->x_pad; s0.tok = pairs; s0.tok_ld = 2; s0.K = H;
    s1 = s0; s1.tok = pairs + 1;
    GemvParams p;
    if (c.compressor == 0) {
        p = gemv_base(ctx, ctx->comp_W, H, EPI_BIAS, ctx->x, H);
        p.bias = ctx->comp_b;
    } else {
        p = gemv_base(ctx, ctx->comp_W1, H, EPI_SILU, ctx->t, H);
    }
    p.seg[0] = s0; p.seg[1] = s1; p.nseg = 2; p.K = 2 * H;
    if (mode != PREFILL_MID) { p.zero_ptr = ctx->am; p.zero_n = 2 * c.max_batch; }
    TRY(launch_gemv(ctx, p));
    if (c.compressor == 1) {
        if (c.comp_residual) TRY(enqueue_pair_sum(ctx, pairs, B));
        p = gemv_base(ctx, ctx->comp_W2, H, c.comp_residual ? EPI_RESADD : EPI_STORE, ctx->x, H);
        p.seg[0] = act_seg(ctx->t, H, H);
        p.K = H;
        TRY(launch_gemv(ctx, p));
    }
    // backbone (Eq. 2)
    for (int l = 0; l < c.n_layers; ++l) TRY(enqueue_block(ctx, ctx->blocks[l], l, ctx->x));
    // LM head + argmax (Eq. 3), or + the sampler (the history gains x_b)
    float* lg_b = c.debug ? ctx->dbg_lb : ctx->samp_on ? ctx->samp_logits : nullptr;
    float* lg_d = c.debug ? ctx->dbg_ld : ctx->samp_on ? ctx->samp_logits + (size_t)c.max_batch * c.vocab : nullptr;
    if (mode != PREFILL_MID) {
        TRY(enqueue_lm_head(ctx, ctx->x, ctx->final_norm, am_b, lg_b));
        if (ctx->samp_on) TRY(enqueue_sample(ctx, lg_b, 0, am_b));
    }
    // MTP head input (App. A.2): W_fc [RMSNorm(h_b); RMSNorm(E[x_b])]
    p = gemv_base(ctx, ctx->mtp_W_fc, H, EPI_STORE, ctx->x2, H);
    p.seg[0] = act_seg(ctx->x, H, H, ctx->mtp_norm_h);
    Seg se{};
    se.table = ctx->E; se.pad = ctx->x_pad; se.gamma = ctx->mtp_norm_e; se.K = H;
    if (mode == PREFILL_MID) { se.tok = ctx->pf_mtp + (size_t)j * B; se.tok_ld = 1; }
    else se.tok_am = am_b;
    p.seg[1] = se; p.nseg = 2; p.K = 2 * H;
    TRY(launch_gemv(ctx, p));
    if (c.mtp_block) TRY(enqueue_block(ctx, ctx->mtp, c.n_layers, ctx->x2));
    if (mode == PREFILL_MID) {
        int32_t* np = ctx->n_pos;
        int Bv = B, by = 1;
        void* args[] = {&np, &Bv, &by};
        return launch_ex(ctx, (const void*)&advance_kernel, dim3((B + 127) / 128), dim3(128), 0, args);
    }
    // draft token (Eq. 5)
    TRY(enqueue_lm_head(ctx, ctx->x2, ctx->mtp_norm_post, am_d, lg_d));
    if (ctx->samp_on) TRY(enqueue_sample(ctx, lg_d, 1, am_d));
    // confidence (Eq. 6, App. A.3): t = SiLU(W1 RMSNorm([h_b; h_d]))
    p = gemv_base(ctx, ctx->conf_W1, H, EPI_SILU, ctx->t, H);
    p.seg[0] = act_seg(ctx->x, H, H, ctx->conf_norm);
    p.seg[1] = act_seg(ctx->x2, H, H, nullptr);
    p.nseg = 2; p.K = 2 * H; p.joint_norm = 1;
    TRY(launch_gemv(ctx, p));
    StepState st{};
    st.pending = ctx->pending; st.n_pos = ctx->n_pos; st.emitted = ctx->emitted;
    st.out_tokens = ctx->out_tokens; st.out_nacc = ctx->out_nacc;
    st.am_b = am_b; st.am_d = am_d;
    if (c.debug) {
        st.dbg_conf = ctx->dbg_conf; st.dbg_hb = ctx->dbg_hb; st.dbg_hd = ctx->dbg_hd;
        st.dbg_xb = ctx->dbg_xb; st.dbg_xd = ctx->dbg_xd;
    }
    if (ctx->samp_on) {
        st.presence = ctx->presence; st.presence_w = ctx->presence_w; st.samp_step = ctx->samp_step;
    }
    {
        const float* tp = ctx->t;
        const void* w2 = ctx->conf_W2;
        int Hv = H, force = c.force_mode;
        float tau = c.tau;
        const float* hb = ctx->x;
        const float* hd = ctx->x2;
        void* args[] = {(void*)&tp, (void*)&w2, &Hv, &tau, &force, &st, (void*)&hb, (void*)&hd};
        return launch_ex(ctx, bf ? (const void*)&accept_kernel<bf16> : (const void*)&accept_kernel<float>, dim3(B),
                         dim3(256), 0, args);
    }
}

// One position of regular decoding (the baseline of Sec. 4) for every
// sequence: DECODE embeds the pending token (slot 0), PREFILL_* prompt token
// j; the backbone blocks run at position n on the backbone caches; the
// positions before the last of a prefill stop there, the others run the
// final-norm tied LM head and take its argmax as the next token.  Same
// kernels as the pair step, without the compressor and the two extra heads.
pipo_status enqueue_regular(pipo_ctx* ctx, Mode mode, int j) {
    const pipo_config& c = ctx->cfg;
    ctx->tc_shallow = attn_is_long(ctx);
    const int H = c.hidden, B = ctx->B;
    const bool bf = c.dtype == 1;
    {
        const void* E = ctx->E;
        const int32_t* tok = (mode == DECODE) ? ctx->pending : ctx->pf_pairs + (size_t)j * B;
        int ld = (mode == DECODE) ? 2 : 1, V = c.vocab, Hv = H, zn = 2 * c.max_batch;
        float* x = ctx->x;
        unsigned long long* am = ctx->am;
        void* args[] = {(void*)&E, (void*)&tok, &ld, &V, &Hv, &x, &am, &zn};
        TRY(launch_ex(ctx, bf ? (const void*)&embed_kernel<bf16> : (const void*)&embed_kernel<float>, dim3(B),
                      dim3(256), 0, args));
    }
    for (int l = 0; l < c.n_layers; ++l) TRY(enqueue_block(ctx, ctx->blocks[l], l, ctx->x));
    if (mode == PREFILL_MID) {
        int32_t* np = ctx->n_pos;
        int Bv = B, by = 1;
        void* args[] = {&np, &Bv, &by};
        return launch_ex(ctx, (const void*)&advance_kernel, dim3((B + 127) / 128), dim3(128), 0, args);
    }
    TRY(enqueue_lm_head(ctx, ctx->x, ctx->final_norm, ctx->am, c.debug ? ctx->dbg_lb : nullptr));
    StepState st{};
    st.pending = ctx->pending; st.n_pos = ctx->n_pos; st.emitted = ctx->emitted;
    st.out_tokens = ctx->out_tokens; st.out_nacc = ctx->out_nacc;
    st.am_b = ctx->am; st.am_d = ctx->am;
    if (c.debug) { st.dbg_hb = ctx->dbg_hb; st.dbg_xb = ctx->dbg_xb; }
    int Hv = H;
    const float* h = ctx->x;
    void* args[] = {&st, &Hv, (void*)&h};
    return launch_ex(ctx, (const void*)&regular_accept_kernel, dim3(B), dim3(256), 0, args);
}

// C consecutive prompt positions j0 .. j0+C-1 of every sequence at once, all
// before the prompt's last position (a pair prefill's teacher-forced
// positions, Sec. 3 / App. A.2, or regular decoding's prompt tokens): the
// C x B rows (row r = position j0 + r / B of sequence r % B, the layout of
// the prompt buffers) go through the projections as one batch, so each
// weight streams once per chunk instead of once per position; each block
// appends the chunk's keys and values and then attends row by row over the
// entries up to the row's own.  The heads do not run (the MTP block does,
// teacher-forced, for pairs); the positions advance by C.
pipo_status enqueue_prefill_chunk(pipo_ctx* ctx, bool regular, int j0, int C) {
    const pipo_config& c = ctx->cfg;
    const int H = c.hidden, B = ctx->B, R = C * B;
    if (R > ctx->max_rows || C < 1 || ctx->attn_v0)
        return fail(ctx, PIPO_EINVAL, "prefill chunk of %d rows (at most %d)", R, ctx->max_rows);
    struct RowsGuard {
        pipo_ctx* c;
        ~RowsGuard() { c->rows = 0; }
    } guard{ctx};
    ctx->rows = R;
    ctx->tc_shallow = attn_is_long(ctx);
    const bool bf = c.dtype == 1;
    if (regular) {
        const void* E = ctx->E;
        const int32_t* tok = ctx->pf_pairs + (size_t)j0 * B;
        int ld = 1, V = c.vocab, Hv = H, zn = 0;
        float* x = ctx->x;
        unsigned long long* am = ctx->am;
        void* args[] = {(void*)&E, (void*)&tok, &ld, &V, &Hv, &x, &am, &zn};
        TRY(launch_ex(ctx, bf ? (const void*)&embed_kernel<bf16> : (const void*)&embed_kernel<float>, dim3(R),
                      dim3(256), 0, args));
    } else {
        // pair embed + compressor (Eq. 1) of the chunk's pairs
        Seg s0{}, s1{};
        s0.table = ctx->E; s0.pad = ctx->x_pad; s0.tok = ctx->pf_pairs + (size_t)j0 * B * 2; s0.tok_ld = 2; s0.K = H;
        s1 = s0; s1.tok = s0.tok + 1;
        GemvParams p;
        if (c.compressor == 0) {
            p = gemv_base(ctx, ctx->comp_W, H, EPI_BIAS, ctx->x, H);
            p.bias = ctx->comp_b;
        } else {
            p = gemv_base(ctx, ctx->comp_W1, H, EPI_SILU, ctx->t, H);
        }
        p.seg[0] = s0; p.seg[1] = s1; p.nseg = 2; p.K = 2 * H;
        TRY(launch_gemv(ctx, p));
        if (c.compressor == 1) {
            if (c.comp_residual) TRY(enqueue_pair_sum(ctx, s0.tok, R));
            p = gemv_base(ctx, ctx->comp_W2, H, c.comp_residual ? EPI_RESADD : EPI_STORE, ctx->x, H);
            p.seg[0] = act_seg(ctx->t, H, H);
            p.K = H;
            TRY(launch_gemv(ctx, p));
        }
    }
    for (int l = 0; l < c.n_layers; ++l) TRY(enqueue_block(ctx, ctx->blocks[l], l, ctx->x));
    if (!regular) {
        // MTP head, teacher-forced (App. A.2): W_fc [RMSNorm(h_b); RMSNorm(E[next prompt token])]
        GemvParams p = gemv_base(ctx, ctx->mtp_W_fc, H, EPI_STORE, ctx->x2, H);
        p.seg[0] = act_seg(ctx->x, H, H, ctx->mtp_norm_h);
        Seg se{};
        se.table = ctx->E; se.pad = ctx->x_pad; se.gamma = ctx->mtp_norm_e; se.K = H;
        se.tok = ctx->pf_mtp + (size_t)j0 * B; se.tok_ld = 1;
        p.seg[1] = se; p.nseg = 2; p.K = 2 * H;
        TRY(launch_gemv(ctx, p));
        if (c.mtp_block) TRY(enqueue_block(ctx, ctx->mtp, c.n_layers, ctx->x2));
    }
    int32_t* np = ctx->n_pos;
    int Bv = B, by = C;
    void* args[] = {&np, &Bv, &by};
    return launch_ex(ctx, (const void*)&advance_kernel, dim3((B + 127) / 128), dim3(128), 0, args);
}

// The positions before a prompt's last one in chunks of prefill_rows / B
// positions (when chunks are enabled and hold two or more positions);
// *j receives the first position left for the position-by-position path.
pipo_status enqueue_prefill_chunks(pipo_ctx* ctx, bool regular, int N, int* j) {
    const int B = ctx->B;
    const int cmax = ctx->prefill_rows / B;
    *j = 0;
    if (cmax < 2 || ctx->attn_v0) return PIPO_OK;
    while (N - 1 - *j >= 2) {
        const int C = std::min(cmax, N - 1 - *j);
        TRY(enqueue_prefill_chunk(ctx, regular, *j, C));
        *j += C;
        ctx->h_len.assign(B, *j);
    }
    return PIPO_OK;
}

// The decode step of the context's current mode.
pipo_status enqueue_step(pipo_ctx* ctx) {
    return ctx->regular ? enqueue_regular(ctx, DECODE, 0) : enqueue_position(ctx, DECODE, 0);
}

void drop_graph(pipo_ctx* ctx) {
    if (ctx->graph) cudaGraphExecDestroy(ctx->graph);
    ctx->graph = nullptr;
    ctx->graph_B = -1;
    ctx->plan_len = -1.0;
    if (ctx->fam_graph) cudaGraphExecDestroy(ctx->fam_graph);
    ctx->fam_graph = nullptr;
    ctx->fam_graph_B = -1;
}

pipo_status ensure_graph(pipo_ctx* ctx) {
    if (ctx->graph && ctx->graph_B == ctx->B && ctx->graph_regular == ctx->regular) return PIPO_OK;
    drop_graph(ctx);
    const double plan_len = plan_mean_len(ctx);
    cudaGraph_t g = nullptr;
    CK(cudaStreamBeginCapture(ctx->stream, cudaStreamCaptureModeThreadLocal));
    ctx->launches = 0;
    ctx->pdl = true;
    pipo_status s = enqueue_step(ctx);
    ctx->pdl = false;
    cudaError_t e = cudaStreamEndCapture(ctx->stream, &g);
    if (s != PIPO_OK) {
        if (g) cudaGraphDestroy(g);
        return s;
    }
    if (e != cudaSuccess) return fail(ctx, PIPO_ECUDA, "graph capture: %s", cudaGetErrorString(e));
    e = cudaGraphInstantiate(&ctx->graph, g, 0);
    cudaGraphDestroy(g);
    if (e != cudaSuccess) return fail(ctx, PIPO_ECUDA, "graph instantiate: %s", cudaGetErrorString(e));
    ctx->graph_B = ctx->B;
    ctx->graph_regular = ctx->regular;
    ctx->plan_len = plan_len;
    return PIPO_OK;
}

__global__ void cache_copy_kernel(KVView kv, int b, int n, int dh, float* buf, int to_cache, int bf) {
    const int j = blockIdx.x;
    const int kd = kv.n_kv * dh;
    for (int i = threadIdx.x; i < kd; i += blockDim.x) {
        const int g = i / dh, d = i % dh;
        const int blk = kv.table[(size_t)b * kv.blocks_per_seq + j / kv.page];
        const size_t off = (((size_t)blk * kv.n_kv + g) * kv.page + (j % kv.page)) * dh + d;
        float* bk = buf + (size_t)j * kd + i;
        float* bv = buf + (size_t)n * kd + (size_t)j * kd + i;
        if (bf) {
            bf16* K = static_cast<bf16*>(kv.K);
            bf16* V = static_cast<bf16*>(kv.V);
            if (to_cache) { K[off] = __float2bfloat16_rn(*bk); V[off] = __float2bfloat16_rn(*bv); }
            else { *bk = __bfloat162float(K[off]); *bv = __bfloat162float(V[off]); }
        } else {
            float* K = static_cast<float*>(kv.K);
            float* V = static_cast<float*>(kv.V);
            if (to_cache) { K[off] = *bk; V[off] = *bv; }
            else { *bk = K[off]; *bv = V[off]; }
        }
    }
}

pipo_status ensure_cache_tmp(pipo_ctx* ctx, size_t elems) {
    if (ctx->cache_tmp_elems >= elems) return PIPO_OK;
    if (ctx->cache_tmp) {
        cudaFree(ctx->cache_tmp);
        ctx->allocs.erase(std::find(ctx->allocs.begin(), ctx->allocs.end(), (void*)ctx->cache_tmp));
        ctx->cache_tmp = nullptr;
    }
    TRY(dalloc(ctx, &ctx->cache_tmp, elems * sizeof(float)));
    ctx->cache_tmp_elems = elems;
    return PIPO_OK;
}

// Read and clear the device error words of the kernel units whose kernels
// wait (bounded waits that gave up; the host unit's kernels never wait): the
// tensor-core attention and projections always, the bulk-copy GEMV and the
// step kernel when the context uses them.  The first unit with an error
// names the wait.
pipo_status check_device_error(pipo_ctx* ctx) {
    // the units whose kernels wait on mbarriers: attention and tensor-core projections
    cudaError_t (*units[2])(unsigned*, unsigned*) = {k_take_error_attn, k_take_error_tc};
    const int nu = 2;
    unsigned e = 0, info[4] = {0, 0, 0, 0};
    for (int i = 0; i < nu; ++i) {
        auto take = units[i];
        unsigned ue = 0, ui[4] = {0, 0, 0, 0};
        CK(take(&ue, ui));
        if (ue && !e) {
            e = ue;
            for (int i = 0; i < 4; ++i) info[i] = ui[i];
        }
    }
    if (!e) return PIPO_OK;
    return fail(ctx, PIPO_ECUDA,
                "device wait timed out (code %u; first at wait site %u, block %u, iteration %u, parity %u): "
                "results of this step are invalid",
                e, info[0], info[1], info[2], info[3]);
}

}  // namespace

// ------------------------------------------------------------------ C ABI
extern "C" {

const char* pipo_last_error(const pipo_ctx* ctx) { return ctx ? ctx->err.c_str() : g_init_error.c_str(); }

int32_t pipo_step_launches(const pipo_ctx* ctx) { return ctx ? ctx->launches : 0; }

void pipo_free(pipo_ctx* ctx) {
    if (!ctx) return;
    cudaSetDevice(ctx->dev);
    if (ctx->stream) cudaStreamSynchronize(ctx->stream);
    drop_graph(ctx);
    for (cudaEvent_t e : ctx->prof_ev) cudaEventDestroy(e);
    for (void* p : ctx->allocs) cudaFree(p);
    if (ctx->own_stream) cudaStreamDestroy(ctx->own_stream);
    delete ctx;
}

pipo_status pipo_init(const pipo_config* cfg, const pipo_weights* w, pipo_ctx** out) {
    pipo_ctx* ctx = nullptr;
    if (!cfg || !w || !out) return fail(nullptr, PIPO_EINVAL, "null argument");
    *out = nullptr;
    const pipo_config& c = *cfg;
    if (c.hidden <= 0 || c.hidden % 8 || c.n_layers < 0 || c.n_q_heads <= 0 || c.n_kv_heads <= 0 ||
        c.n_q_heads % c.n_kv_heads || c.ffn <= 0 || c.ffn % 8 || c.vocab <= 0 || c.max_batch <= 0 ||
        c.max_ctx <= 0 || c.page_size <= 0 || (c.dtype != 0 && c.dtype != 1) ||
        (c.compressor != 0 && c.compressor != 1) || (c.mtp_block != 0 && c.mtp_block != 1) ||
        (c.comp_residual != 0 && c.comp_residual != 1) || (c.comp_residual && c.compressor != 1))
        return fail(nullptr, PIPO_EINVAL, "invalid config");
    if (c.head_dim != 64 && c.head_dim != 128) return fail(nullptr, PIPO_EINVAL, "head_dim must be 64 or 128");
    const int G = c.n_q_heads / c.n_kv_heads;
    if (G != 1 && G != 2 && G != 4 && G != 8) return fail(nullptr, PIPO_EINVAL, "n_q/n_kv must be 1, 2, 4 or 8");
    if ((size_t)c.ffn * 4 > kXsBudget || (size_t)2 * c.hidden * 4 > kXsBudget)
        return fail(nullptr, PIPO_EINVAL, "hidden/ffn too large for the staged GEMV input");

    ctx = new pipo_ctx();
    ctx->cfg = c;
    ctx->esz = c.dtype == 1 ? 2 : 4;
    if (const char* ev = getenv("PIPO_TEST_FAIL_ALLOC")) ctx->fail_alloc_at = std::max(0, atoi(ev));
    pipo_status s = [&]() -> pipo_status {
        CK(cudaGetDevice(&ctx->dev));
        CK(cudaDeviceGetAttribute(&ctx->sms, cudaDevAttrMultiProcessorCount, ctx->dev));
        CK(cudaStreamCreateWithFlags(&ctx->own_stream, cudaStreamNonBlocking));
        ctx->stream = ctx->own_stream;
        CK(set_smem_attrs(c.dtype == 1));
        const size_t H = c.hidden, V = c.vocab;
        TRY(upload(ctx, &ctx->E, w->E, V * H));
        TRY(upload(ctx, &ctx->x_pad, w->x_pad, H));
        if (c.compressor == 0) {
            TRY(upload(ctx, &ctx->comp_W, w->comp_W, H * 2 * H));
            TRY(upload(ctx, &ctx->comp_b, w->comp_b, H));
        } else {
            TRY(upload(ctx, &ctx->comp_W1, w->comp_W1, H * 2 * H));
            TRY(upload(ctx, &ctx->comp_W2, w->comp_W2, H * H));
        }
        ctx->blocks.resize(c.n_layers);
        for (int l = 0; l < c.n_layers; ++l)
            TRY(upload_block(ctx, ctx->blocks[l], l, w->attn_norm, w->Wq, w->Wk, w->Wv, w->Wo, w->ffn_norm, w->Wgate,
                             w->Wup, w->Wdown));
        if (c.mtp_block)
            TRY(upload_block(ctx, ctx->mtp, 0, w->m_attn_norm, w->m_Wq, w->m_Wk, w->m_Wv, w->m_Wo, w->m_ffn_norm,
                             w->m_Wgate, w->m_Wup, w->m_Wdown));
        TRY(upload(ctx, &ctx->final_norm, w->final_norm, H));
        TRY(upload(ctx, &ctx->mtp_norm_h, w->mtp_norm_h, H));
        TRY(upload(ctx, &ctx->mtp_norm_e, w->mtp_norm_e, H));
        TRY(upload(ctx, &ctx->mtp_W_fc, w->mtp_W_fc, H * 2 * H));
        TRY(upload(ctx, &ctx->mtp_norm_post, w->mtp_norm_post, H));
        TRY(upload(ctx, &ctx->conf_norm, w->conf_norm, 2 * H));
        TRY(upload(ctx, &ctx->conf_W1, w->conf_W1, H * 2 * H));
        TRY(upload(ctx, &ctx->conf_W2, w->conf_W2, H));

        // paged KV cache
        const int MB = c.max_batch, DH = c.head_dim;
        ctx->n_cache_layers = c.n_layers + (c.mtp_block ? 1 : 0);
        ctx->blocks_per_seq = (c.max_ctx + c.page_size - 1) / c.page_size;
        ctx->num_blocks = MB * ctx->blocks_per_seq;
        ctx->layer_elems = (size_t)ctx->num_blocks * c.n_kv_heads * c.page_size * DH;
        TRY(dalloc(ctx, reinterpret_cast<char**>(&ctx->Kc), std::max<size_t>(1, ctx->n_cache_layers) * ctx->layer_elems * ctx->esz));
        TRY(dalloc(ctx, reinterpret_cast<char**>(&ctx->Vc), std::max<size_t>(1, ctx->n_cache_layers) * ctx->layer_elems * ctx->esz));
        // zeroed: masked lanes of the attention kernel read (and multiply by 0) entry 0
        CK(cudaMemset(ctx->Kc, 0, std::max<size_t>(1, ctx->n_cache_layers) * ctx->layer_elems * ctx->esz));
        CK(cudaMemset(ctx->Vc, 0, std::max<size_t>(1, ctx->n_cache_layers) * ctx->layer_elems * ctx->esz));
        std::vector<int32_t> table(ctx->num_blocks);
        std::iota(table.begin(), table.end(), 0);
        if (c.page_shuffle_seed) {
            std::mt19937 rng(c.page_shuffle_seed);
            std::shuffle(table.begin(), table.end(), rng);
        }
        TRY(dalloc(ctx, &ctx->block_table, table.size() * sizeof(int32_t)));
        CK(cudaMemcpy(ctx->block_table, table.data(), table.size() * sizeof(int32_t), cudaMemcpyHostToDevice));

        // RoPE angle table: angle = pos * theta^(-2i/d_h), cos/sin in double, stored fp32
        {
            std::vector<float> tab((size_t)c.max_ctx * DH);
            for (int pos = 0; pos < c.max_ctx; ++pos)
                for (int i = 0; i < DH / 2; ++i) {
                    const double ang = (double)pos * std::pow((double)c.rope_theta, -2.0 * i / DH);
                    tab[((size_t)pos * (DH / 2) + i) * 2] = (float)std::cos(ang);
                    tab[((size_t)pos * (DH / 2) + i) * 2 + 1] = (float)std::sin(ang);
                }
            TRY(dalloc(ctx, &ctx->rope, tab.size() * 4));
            CK(cudaMemcpy(ctx->rope, tab.data(), tab.size() * 4, cudaMemcpyHostToDevice));
        }
        CK(set_carveouts(c.dtype == 1));
        if (const char* ev = getenv("PIPO_ATTN_V0")) ctx->attn_v0 = ev[0] == '1';
        if (const char* ev = getenv("PIPO_ATTN_IMPL")) ctx->attn_regs = strcmp(ev, "regs") == 0;
        if (const char* ev = getenv("PIPO_ATTN_FLAT")) ctx->attn_flat = atoi(ev);
        if (attn_mma_ok(ctx)) {
            // the cache layers as 2-D tensors [blocks * n_kv * page][d_h] for the tensor-core attention
            const int rows = ctx->num_blocks * c.n_kv_heads * c.page_size;
            ctx->kv_tm.resize(2 * ctx->n_cache_layers);
            for (int l = 0; l < ctx->n_cache_layers; ++l) {
                const KVView v = kv_view(ctx, l);
                TRY(make_tmap(ctx, &ctx->kv_tm[2 * l], v.K, DH, rows, kMmaRun));
                TRY(make_tmap(ctx, &ctx->kv_tm[2 * l + 1], v.V, DH, rows, kMmaRun));
            }
        }
        // 16-CTA clusters measured slower than 8 at 4B B=1 (2.77 vs 2.55 ms per step): opt-in only
        if (const char* ev = getenv("PIPO_ATTN_CS16"))
            ctx->attn_cs16 = ev[0] == '1' && cluster16_ok(c.dtype == 1, c.head_dim, c.n_q_heads / c.n_kv_heads);
        if (const char* ev = getenv("PIPO_ATTN_CS")) {
            const int v = atoi(ev);
            if (v == 1 || v == 2 || v == 4 || v == 8 || (v == 16 && cluster16_ok(c.dtype == 1, c.head_dim,
                                                                               c.n_q_heads / c.n_kv_heads)))
                ctx->attn_cs_force = v;
        }
        if (const char* ev = getenv("PIPO_ATTN_CS_TARGET")) ctx->attn_cs_target = std::max(1, atoi(ev));

        // activations and state
        const int qd = c.n_q_heads * DH, kd = c.n_kv_heads * DH;
        // prefill chunks: PIPO_PREFILL_ROWS=<rows> (positions x sequences per
        // chunk, at most 128; 0 or unset: one position at a time)
        if (const char* ev = getenv("PIPO_PREFILL_ROWS")) ctx->prefill_rows = std::min(128, std::max(0, atoi(ev)));
        if (const char* ev = getenv("PIPO_PREFILL_ATTN")) ctx->prefill_tile_attn = strcmp(ev, "tile") == 0;
        const int MR = std::max(MB, ctx->prefill_rows);
        ctx->max_rows = MR;
        // GEMM inputs get at least as many rows as the tensor-core batch width
        // (their activation tensor maps read box-sized tiles of BH rows)
        ctx->act_rows = c.dtype == 1 ? std::max(MR, tc_bn(std::min(MR, 128))) : MR;
        const size_t AR = (size_t)ctx->act_rows;
        TRY(dalloc(ctx, &ctx->x, AR * H * 4));
        TRY(dalloc(ctx, &ctx->x2, AR * H * 4));
        TRY(dalloc(ctx, &ctx->qkv, (size_t)MR * (qd + 2 * kd) * 4));
        TRY(dalloc(ctx, &ctx->q, (size_t)MB * qd * 4));
        TRY(dalloc(ctx, &ctx->attn, AR * qd * 4));
        TRY(dalloc(ctx, &ctx->act, AR * c.ffn * 4));
        TRY(dalloc(ctx, &ctx->t, AR * H * 4));
        size_t parts = 0;
        for (int b = 1; b <= MB; ++b) parts = std::max(parts, (size_t)b * c.n_q_heads * attn_splits(ctx, b));
        // the unclustered tensor-core attention: rows x n_kv < 2 sms / 8, at most kFlatMaxSplits splits
        parts = std::max(parts, (size_t)(2 * ctx->sms / 8 + 1) * (c.n_q_heads / c.n_kv_heads) * kFlatMaxSplits);
        TRY(dalloc(ctx, &ctx->part_o, parts * DH * 4));
        TRY(dalloc(ctx, &ctx->part_ml, parts * 2 * 4));
        TRY(dalloc(ctx, &ctx->counters, (size_t)MB * c.n_kv_heads * 4));
        CK(cudaMemset(ctx->counters, 0, (size_t)MB * c.n_kv_heads * 4));
        TRY(dalloc(ctx, &ctx->am, (size_t)2 * MB * 8));
        const int smax = std::max(resadd_splits(ctx, H, qd), resadd_splits(ctx, H, c.ffn));
        TRY(dalloc(ctx, &ctx->gemv_part, (size_t)smax * MR * H * 4));
        // one counter per (batch group, row): at most MR groups
        TRY(dalloc(ctx, &ctx->gemv_rowcnt, (size_t)MR * H * 4));
        CK(cudaMemset(ctx->gemv_rowcnt, 0, (size_t)MR * H * 4));
        // tensor-core projections: the bf16 activation tile
        if (const char* ev = getenv("PIPO_TC_MIN_BATCH")) ctx->tc_min_b = std::max(1, atoi(ev));
        if (const char* ev = getenv("PIPO_ATTN_MMA_MIN_BATCH")) ctx->attn_mma_min_b = std::max(1, atoi(ev));
        if (const char* ev = getenv("PIPO_TC_SPLITS")) ctx->tc_splits = std::max(0, atoi(ev));
        if (c.dtype == 1 && MR >= ctx->tc_min_b) {
            ctx->tc_bn_max = tc_bn(std::min(MR, 128));
            ctx->tc_kmax = std::max({2 * (int)H, qd, c.ffn});
            TRY(dalloc(ctx, &ctx->tc_xb, (size_t)2 * ctx->tc_bn_max * ctx->tc_kmax * 2));
        }
        TRY(dalloc(ctx, &ctx->pending, (size_t)MB * 2 * 4));
        TRY(dalloc(ctx, &ctx->n_pos, (size_t)MB * 4));
        TRY(dalloc(ctx, &ctx->out_tokens, (size_t)MB * 2 * 4));
        TRY(dalloc(ctx, &ctx->out_nacc, (size_t)MB * 4));
        TRY(dalloc(ctx, &ctx->emitted, (size_t)MB * 8));
        CK(cudaMemset(ctx->n_pos, 0, (size_t)MB * 4));
        CK(cudaMemset(ctx->emitted, 0, (size_t)MB * 8));
        CK(cudaMemset(ctx->pending, 0, (size_t)MB * 2 * 4));  // a slot never prefilled holds valid ids
        if (c.debug) {
            TRY(dalloc(ctx, &ctx->dbg_lb, (size_t)MB * V * 4));
            TRY(dalloc(ctx, &ctx->dbg_ld, (size_t)MB * V * 4));
            TRY(dalloc(ctx, &ctx->dbg_conf, (size_t)MB * 4));
            TRY(dalloc(ctx, &ctx->dbg_hb, (size_t)MB * H * 4));
            TRY(dalloc(ctx, &ctx->dbg_hd, (size_t)MB * H * 4));
            TRY(dalloc(ctx, &ctx->dbg_xb, (size_t)MB * 4));
            TRY(dalloc(ctx, &ctx->dbg_xd, (size_t)MB * 4));
        }
        CK(cudaDeviceSynchronize());
        return PIPO_OK;
    }();
    ctx->fail_alloc_at = 0;  // the injection covers pipo_init only
    if (s != PIPO_OK) {
        g_init_error = ctx->err;
        pipo_free(ctx);
        return s;
    }
    *out = ctx;
    return PIPO_OK;
}

pipo_status pipo_set_stream(pipo_ctx* ctx, void* stream) {
    if (!ctx) return fail(nullptr, PIPO_EINVAL, "null context");
    CK(cudaSetDevice(ctx->dev));
    CK(cudaStreamSynchronize(ctx->stream));
    ctx->stream = stream ? static_cast<cudaStream_t>(stream) : ctx->own_stream;
    drop_graph(ctx);
    return PIPO_OK;
}

pipo_status pipo_set_threshold(pipo_ctx* ctx, float tau, int32_t force_mode) {
    if (!ctx) return fail(nullptr, PIPO_EINVAL, "null context");
    if (force_mode < 0 || force_mode > 2 || !std::isfinite(tau)) return fail(ctx, PIPO_EINVAL, "bad threshold or force mode");
    if (ctx->cfg.tau != tau || ctx->cfg.force_mode != force_mode) drop_graph(ctx);
    ctx->cfg.tau = tau;
    ctx->cfg.force_mode = force_mode;
    return PIPO_OK;
}

pipo_status pipo_set_sampler(pipo_ctx* ctx, float temperature, int32_t top_k, float top_p, float rep_penalty,
                             const float* h_u, int32_t n_u) {
    if (!ctx) return fail(nullptr, PIPO_EINVAL, "null context");
    const pipo_config& c = ctx->cfg;
    if (!(temperature > 0.f)) {
        if (ctx->samp_on) drop_graph(ctx);
        ctx->samp_on = false;
        return PIPO_OK;
    }
    if (top_k < 1 || top_k > kSampMaxK || !(top_p > 0.f && top_p <= 1.f) || !(rep_penalty > 0.f) ||
        !std::isfinite(temperature) || !std::isfinite(rep_penalty) || !h_u || n_u < 1)
        return fail(ctx, PIPO_EINVAL, "bad sampler settings (top_k in [1, %d], top_p in (0, 1], penalty > 0, "
                                      "draws given)", kSampMaxK);
    const size_t nu = (size_t)n_u * c.max_batch * 2;
    for (size_t i = 0; i < nu; ++i)
        if (!(h_u[i] >= 0.f && h_u[i] < 1.f)) return fail(ctx, PIPO_EINVAL, "draw %zu not in [0, 1)", i);
    CK(cudaSetDevice(ctx->dev));
    CK(cudaStreamSynchronize(ctx->stream));
    // off until the buffers below are in place (a failed call leaves the sampler off)
    if (ctx->samp_on) drop_graph(ctx);
    ctx->samp_on = false;
    if (!ctx->samp_logits) {
        ctx->presence_w = (c.vocab + 31) / 32;
        TRY(dalloc(ctx, &ctx->samp_logits, (size_t)2 * c.max_batch * c.vocab * 4));
        TRY(dalloc(ctx, &ctx->presence, (size_t)c.max_batch * ctx->presence_w * 4));
        TRY(dalloc(ctx, &ctx->samp_step, 4));
        CK(cudaMemset(ctx->presence, 0, (size_t)c.max_batch * ctx->presence_w * 4));
    }
    if (n_u > ctx->samp_nu) {
        if (ctx->samp_u) {
            cudaFree(ctx->samp_u);
            ctx->allocs.erase(std::find(ctx->allocs.begin(), ctx->allocs.end(), (void*)ctx->samp_u));
            ctx->samp_u = nullptr;
        }
        ctx->samp_nu = 0;
        TRY(dalloc(ctx, &ctx->samp_u, nu * 4));
    }
    CK(cudaMemcpy(ctx->samp_u, h_u, nu * 4, cudaMemcpyHostToDevice));
    CK(cudaMemset(ctx->samp_step, 0, 4));
    ctx->samp_nu = n_u;
    ctx->samp_T = temperature;
    ctx->samp_k = top_k;
    ctx->samp_p = top_p;
    ctx->samp_rep = rep_penalty;
    ctx->samp_on = true;
    drop_graph(ctx);
    return PIPO_OK;
}

}  // extern "C"

namespace {

// Device copy of prompt inputs (int32, n elements): pf_pairs (and pf_mtp) grow
// to hold them.
pipo_status ensure_prompt_buffers(pipo_ctx* ctx, size_t n) {
    if (n <= ctx->pf_cap) return PIPO_OK;
    for (void* p : {(void*)ctx->pf_pairs, (void*)ctx->pf_mtp})
        if (p) {
            cudaFree(p);
            ctx->allocs.erase(std::find(ctx->allocs.begin(), ctx->allocs.end(), p));
        }
    ctx->pf_pairs = ctx->pf_mtp = nullptr;
    ctx->pf_cap = 0;
    TRY(dalloc(ctx, &ctx->pf_pairs, n * 4));
    TRY(dalloc(ctx, &ctx->pf_mtp, n * 4));
    ctx->pf_cap = n;
    return PIPO_OK;
}

// Shared checks of both prefills: batch, lengths in [1, stride], ids in
// [0, V).  Returns the lengths' common value of units (pairs: (len + 1) / 2;
// regular decoding: len) in *units.
pipo_status check_prompt(pipo_ctx* ctx, int32_t batch, const int32_t* h_ids, int32_t stride, const int32_t* h_lens,
                         bool pairs, int* units) {
    const pipo_config& c = ctx->cfg;
    if (batch < 1 || batch > c.max_batch || !h_ids || !h_lens || stride < 1)
        return fail(ctx, PIPO_EINVAL, "bad prefill arguments (batch %d, stride %d)", batch, stride);
    int N = -1;
    for (int b = 0; b < batch; ++b) {
        const int len = h_lens[b];
        if (len < 1 || len > stride) return fail(ctx, PIPO_EINVAL, "sequence %d: length %d not in [1, %d]", b, len, stride);
        const int nb = pairs ? (len + 1) / 2 : len;
        if (N >= 0 && nb != N)
            return fail(ctx, PIPO_EINVAL, pairs ? "sequences must give the same number of pairs"
                                                : "sequences must have the same length");
        N = nb;
        for (int i = 0; i < len; ++i) {
            const int32_t t = h_ids[(size_t)b * stride + i];
            if (t < 0 || t >= c.vocab) return fail(ctx, PIPO_EINVAL, "token id %d out of range at (%d, %d)", t, b, i);
        }
    }
    if (N > c.max_ctx) return fail(ctx, PIPO_ECAPACITY, "prompt needs %d entries > max_ctx %d", N, c.max_ctx);
    *units = N;
    return PIPO_OK;
}

}  // namespace

extern "C" {

pipo_status pipo_prefill(pipo_ctx* ctx, int32_t batch, const int32_t* h_ids, int32_t stride, const int32_t* h_lens,
                         int32_t* h_tokens, int32_t* h_n_accepted) {
    if (!ctx) return fail(nullptr, PIPO_EINVAL, "null context");
    drop_graph(ctx);  // the next step's launch plan is made for the new lengths
    if (batch > 1 && batch <= ctx->cfg.max_batch && h_ids && h_lens && stride >= 1) {
        bool ragged = false;
        for (int b = 1; b < batch; ++b) ragged |= (h_lens[b] + 1) / 2 != (h_lens[0] + 1) / 2;
        if (ragged) {
            // different numbers of pairs: every sequence on its own, as a slot
            for (int b = 0; b < batch; ++b) {  // validate all before any runs
                int nb = 0;
                TRY(check_prompt(ctx, 1, h_ids + (size_t)b * stride, stride, h_lens + b, true, &nb));
            }
            ctx->prefilled = false;
            ctx->B = 0;
            ctx->h_len.clear();
            for (int b = 0; b < batch; ++b) {
                const pipo_status st = pipo_prefill_slot(ctx, b, h_ids + (size_t)b * stride, h_lens[b],
                                                         h_tokens ? h_tokens + 2 * b : nullptr,
                                                         h_n_accepted ? h_n_accepted + b : nullptr);
                if (st != PIPO_OK) {
                    // no partial batch: the context is left not prefilled (decode steps return ESTATE)
                    ctx->prefilled = false;
                    ctx->B = 0;
                    ctx->h_len.clear();
                    return st;
                }
            }
            return PIPO_OK;
        }
    }
    int N = 0;
    TRY(check_prompt(ctx, batch, h_ids, stride, h_lens, true, &N));
    CK(cudaSetDevice(ctx->dev));
    // pairs [N][B][2] (PAD = -1 in an odd prompt's last slot), MTP inputs [N][B]
    std::vector<int32_t> pairs((size_t)N * batch * 2), mtp((size_t)N * batch, 0);
    for (int j = 0; j < N; ++j)
        for (int b = 0; b < batch; ++b) {
            const int32_t* t = h_ids + (size_t)b * stride;
            const int len = h_lens[b];
            pairs[((size_t)j * batch + b) * 2] = t[2 * j];
            pairs[((size_t)j * batch + b) * 2 + 1] = (2 * j + 1 < len) ? t[2 * j + 1] : -1;
            if (j + 1 < N) mtp[(size_t)j * batch + b] = t[2 * j + 2];
        }
    TRY(ensure_prompt_buffers(ctx, pairs.size()));
    CK(cudaMemcpyAsync(ctx->pf_pairs, pairs.data(), pairs.size() * 4, cudaMemcpyHostToDevice, ctx->stream));
    CK(cudaMemcpyAsync(ctx->pf_mtp, mtp.data(), mtp.size() * 4, cudaMemcpyHostToDevice, ctx->stream));
    std::vector<uint32_t> bits;
    if (ctx->samp_on) {
        // the sampler's repetition history starts with the prompt
        bits.assign((size_t)batch * ctx->presence_w, 0u);
        for (int b = 0; b < batch; ++b)
            for (int i = 0; i < h_lens[b]; ++i) {
                const int32_t t = h_ids[(size_t)b * stride + i];
                bits[(size_t)b * ctx->presence_w + (t >> 5)] |= 1u << (t & 31);
            }
        CK(cudaMemcpyAsync(ctx->presence, bits.data(), bits.size() * 4, cudaMemcpyHostToDevice, ctx->stream));
    }
    CK(cudaMemsetAsync(ctx->n_pos, 0, (size_t)batch * 4, ctx->stream));
    CK(cudaMemsetAsync(ctx->emitted, 0, (size_t)batch * 8, ctx->stream));
    ctx->B = batch;
    ctx->regular = false;
    ctx->prefilled = false;
    ctx->h_len.assign(batch, 0);
    const int saved = ctx->launches;
    int j = 0;
    TRY(enqueue_prefill_chunks(ctx, false, N, &j));
    for (; j < N; ++j) {
        TRY(enqueue_position(ctx, j + 1 < N ? PREFILL_MID : PREFILL_LAST, j));
        ctx->h_len.assign(batch, j + 1);
    }
    ctx->launches = saved;
    if (h_tokens) CK(cudaMemcpyAsync(h_tokens, ctx->out_tokens, (size_t)batch * 8, cudaMemcpyDeviceToHost, ctx->stream));
    if (h_n_accepted) CK(cudaMemcpyAsync(h_n_accepted, ctx->out_nacc, (size_t)batch * 4, cudaMemcpyDeviceToHost, ctx->stream));
    CK(cudaStreamSynchronize(ctx->stream));
    ctx->h_len.assign(batch, N);
    ctx->prefilled = true;
    return check_device_error(ctx);
}

}  // extern "C"

namespace {

// The per-sequence device state of one slot as a batch of one: every
// per-sequence buffer starts at the slot (the activation and prompt buffers
// are scratch shared by all slots).  Restored on destruction.
struct SlotView {
    pipo_ctx* c;
    int32_t *n_pos, *pending, *out_tokens, *out_nacc, *block_table, *dbg_xb, *dbg_xd;
    long long* emitted;
    float *dbg_lb, *dbg_ld, *dbg_conf, *dbg_hb, *dbg_hd, *samp_u;
    uint32_t* presence;
    SlotView(pipo_ctx* ctx, int s) : c(ctx) {
        const size_t V = ctx->cfg.vocab, H = ctx->cfg.hidden;
        n_pos = ctx->n_pos; pending = ctx->pending; out_tokens = ctx->out_tokens; out_nacc = ctx->out_nacc;
        block_table = ctx->block_table; dbg_xb = ctx->dbg_xb; dbg_xd = ctx->dbg_xd; emitted = ctx->emitted;
        dbg_lb = ctx->dbg_lb; dbg_ld = ctx->dbg_ld; dbg_conf = ctx->dbg_conf; dbg_hb = ctx->dbg_hb;
        dbg_hd = ctx->dbg_hd; samp_u = ctx->samp_u; presence = ctx->presence;
        ctx->n_pos += s; ctx->pending += 2 * s; ctx->out_tokens += 2 * s; ctx->out_nacc += s; ctx->emitted += s;
        ctx->block_table += (size_t)s * ctx->blocks_per_seq;
        if (ctx->dbg_lb) {
            ctx->dbg_lb += s * V; ctx->dbg_ld += s * V; ctx->dbg_conf += s; ctx->dbg_hb += s * H;
            ctx->dbg_hd += s * H; ctx->dbg_xb += s; ctx->dbg_xd += s;
        }
        if (ctx->samp_u) ctx->samp_u += 2 * s;
        if (ctx->presence) ctx->presence += (size_t)s * ctx->presence_w;
    }
    ~SlotView() {
        c->n_pos = n_pos; c->pending = pending; c->out_tokens = out_tokens; c->out_nacc = out_nacc;
        c->block_table = block_table; c->dbg_xb = dbg_xb; c->dbg_xd = dbg_xd; c->emitted = emitted;
        c->dbg_lb = dbg_lb; c->dbg_ld = dbg_ld; c->dbg_conf = dbg_conf; c->dbg_hb = dbg_hb; c->dbg_hd = dbg_hd;
        c->samp_u = samp_u; c->presence = presence;
    }
};

}  // namespace

extern "C" {

pipo_status pipo_prefill_slot(pipo_ctx* ctx, int32_t slot, const int32_t* h_ids, int32_t len, int32_t* h_tokens,
                              int32_t* h_n_accepted) {
    if (!ctx) return fail(nullptr, PIPO_EINVAL, "null context");
    if (slot < 0 || slot >= ctx->cfg.max_batch || !h_ids || len < 1)
        return fail(ctx, PIPO_EINVAL, "bad slot prefill arguments (slot %d of %d, length %d)", slot,
                    ctx->cfg.max_batch, len);
    if (ctx->prefilled && ctx->regular) return fail(ctx, PIPO_ESTATE, "slot prefill after a regular-decoding prefill");
    drop_graph(ctx);  // the next step's launch plan is made for the new lengths
    const bool was = ctx->prefilled;
    const int B_old = was ? ctx->B : 0;
    const std::vector<int32_t> len_old = was ? ctx->h_len : std::vector<int32_t>();
    pipo_status st;
    {
        SlotView view(ctx, slot);
        int32_t one = len;
        st = pipo_prefill(ctx, 1, h_ids, len, &one, h_tokens, h_n_accepted);
    }
    if (st != PIPO_OK) {  // this slot's state is undefined; the other slots are untouched
        ctx->B = B_old;
        ctx->h_len = len_old;
        ctx->prefilled = was;
        if (ctx->B == 0) ctx->prefilled = false;
        return st;
    }
    std::vector<int32_t> lens = len_old;
    lens.resize(std::max(B_old, slot + 1), 0);
    lens[slot] = (len + 1) / 2;
    ctx->B = (int)lens.size();
    ctx->h_len = lens;
    ctx->prefilled = true;
    ctx->regular = false;
    return PIPO_OK;
}

pipo_status pipo_regular_prefill(pipo_ctx* ctx, int32_t batch, const int32_t* h_ids, int32_t stride,
                                 const int32_t* h_lens, int32_t* h_tokens, int32_t* h_n_accepted) {
    if (!ctx) return fail(nullptr, PIPO_EINVAL, "null context");
    drop_graph(ctx);  // the next step's launch plan is made for the new lengths
    int N = 0;
    TRY(check_prompt(ctx, batch, h_ids, stride, h_lens, false, &N));
    CK(cudaSetDevice(ctx->dev));
    // tokens [N][B]
    std::vector<int32_t> toks((size_t)N * batch);
    for (int j = 0; j < N; ++j)
        for (int b = 0; b < batch; ++b) toks[(size_t)j * batch + b] = h_ids[(size_t)b * stride + j];
    TRY(ensure_prompt_buffers(ctx, toks.size()));
    CK(cudaMemcpyAsync(ctx->pf_pairs, toks.data(), toks.size() * 4, cudaMemcpyHostToDevice, ctx->stream));
    CK(cudaMemsetAsync(ctx->n_pos, 0, (size_t)batch * 4, ctx->stream));
    ctx->B = batch;
    ctx->regular = true;
    ctx->prefilled = false;
    ctx->h_len.assign(batch, 0);
    const int saved = ctx->launches;
    int j = 0;
    TRY(enqueue_prefill_chunks(ctx, true, N, &j));
    for (; j < N; ++j) {
        TRY(enqueue_regular(ctx, j + 1 < N ? PREFILL_MID : PREFILL_LAST, j));
        ctx->h_len.assign(batch, j + 1);
    }
    ctx->launches = saved;
    // the prefill's token is the first output, not a decode step's
    CK(cudaMemsetAsync(ctx->emitted, 0, (size_t)batch * 8, ctx->stream));
    if (h_tokens) CK(cudaMemcpyAsync(h_tokens, ctx->out_tokens, (size_t)batch * 8, cudaMemcpyDeviceToHost, ctx->stream));
    if (h_n_accepted) CK(cudaMemcpyAsync(h_n_accepted, ctx->out_nacc, (size_t)batch * 4, cudaMemcpyDeviceToHost, ctx->stream));
    CK(cudaStreamSynchronize(ctx->stream));
    ctx->h_len.assign(batch, N);
    ctx->prefilled = true;
    return check_device_error(ctx);
}

}  // extern "C"

namespace {

// One decode step of the context's mode, enqueued (graph replay).
pipo_status step_async(pipo_ctx* ctx, bool regular, int32_t* d_tokens, int32_t* d_n_accepted) {
    if (!ctx) return fail(nullptr, PIPO_EINVAL, "null context");
    if (!ctx->prefilled) return fail(ctx, PIPO_ESTATE, "decode step before prefill");
    if (ctx->regular != regular)
        return fail(ctx, PIPO_ESTATE, regular ? "regular step after a pair prefill (pipo_prefill)"
                                              : "pair step after a regular-decoding prefill (pipo_regular_prefill)");
    for (int b = 0; b < ctx->B; ++b)
        if (ctx->h_len[b] + 1 > ctx->cfg.max_ctx)
            return fail(ctx, PIPO_ECAPACITY, "sequence %d: KV cache full (%d entries)", b, ctx->h_len[b]);
    CK(cudaSetDevice(ctx->dev));
    TRY(ensure_graph(ctx));
    CK(cudaGraphLaunch(ctx->graph, ctx->stream));
    if (d_tokens) CK(cudaMemcpyAsync(d_tokens, ctx->out_tokens, (size_t)ctx->B * 8, cudaMemcpyDeviceToDevice, ctx->stream));
    if (d_n_accepted) CK(cudaMemcpyAsync(d_n_accepted, ctx->out_nacc, (size_t)ctx->B * 4, cudaMemcpyDeviceToDevice, ctx->stream));
    for (int b = 0; b < ctx->B; ++b) ctx->h_len[b] += 1;
    return PIPO_OK;
}

pipo_status step_sync(pipo_ctx* ctx, bool regular, int32_t* h_tokens, int32_t* h_n_accepted) {
    TRY(step_async(ctx, regular, nullptr, nullptr));
    if (h_tokens) CK(cudaMemcpyAsync(h_tokens, ctx->out_tokens, (size_t)ctx->B * 8, cudaMemcpyDeviceToHost, ctx->stream));
    if (h_n_accepted) CK(cudaMemcpyAsync(h_n_accepted, ctx->out_nacc, (size_t)ctx->B * 4, cudaMemcpyDeviceToHost, ctx->stream));
    CK(cudaStreamSynchronize(ctx->stream));
    return check_device_error(ctx);
}

}  // namespace

extern "C" {

pipo_status pipo_decode_step_async(pipo_ctx* ctx, int32_t* d_tokens, int32_t* d_n_accepted) {
    return step_async(ctx, false, d_tokens, d_n_accepted);
}

pipo_status pipo_decode_step(pipo_ctx* ctx, int32_t* h_tokens, int32_t* h_n_accepted) {
    return step_sync(ctx, false, h_tokens, h_n_accepted);
}

pipo_status pipo_decode_steps(pipo_ctx* ctx, int32_t n_steps, int32_t* h_tokens, int32_t* h_n_accepted) {
    if (!ctx) return fail(nullptr, PIPO_EINVAL, "null context");
    if (n_steps < 1) return fail(ctx, PIPO_EINVAL, "n_steps %d < 1", n_steps);
    if (!ctx->prefilled) return fail(ctx, PIPO_ESTATE, "decode step before prefill");
    for (int b = 0; b < ctx->B; ++b)
        if (ctx->h_len[b] + n_steps > ctx->cfg.max_ctx)
            return fail(ctx, PIPO_ECAPACITY, "sequence %d: %d entries + %d steps > max_ctx", b, ctx->h_len[b], n_steps);
    CK(cudaSetDevice(ctx->dev));
    const size_t B = ctx->B, need = (size_t)n_steps * B * 3;
    if (need > ctx->multi_cap) {
        if (ctx->multi_out) {
            cudaFree(ctx->multi_out);
            ctx->allocs.erase(std::find(ctx->allocs.begin(), ctx->allocs.end(), (void*)ctx->multi_out));
            ctx->multi_out = nullptr;
        }
        ctx->multi_cap = 0;
        TRY(dalloc(ctx, &ctx->multi_out, need * 4));
        ctx->multi_cap = need;
    }
    // per step: tokens [B][2] then acceptances [B], gathered on the device
    for (int i = 0; i < n_steps; ++i) {
        int32_t* o = ctx->multi_out + (size_t)i * B * 3;
        TRY(step_async(ctx, false, o, o + 2 * B));
    }
    std::vector<int32_t> host(need);
    CK(cudaMemcpyAsync(host.data(), ctx->multi_out, need * 4, cudaMemcpyDeviceToHost, ctx->stream));
    CK(cudaStreamSynchronize(ctx->stream));
    for (int i = 0; i < n_steps; ++i) {
        const int32_t* o = host.data() + (size_t)i * B * 3;
        if (h_tokens) std::copy(o, o + 2 * B, h_tokens + (size_t)i * B * 2);
        if (h_n_accepted) std::copy(o + 2 * B, o + 3 * B, h_n_accepted + (size_t)i * B);
    }
    return check_device_error(ctx);
}

pipo_status pipo_regular_step_async(pipo_ctx* ctx, int32_t* d_tokens) {
    return step_async(ctx, true, d_tokens, nullptr);
}

pipo_status pipo_regular_step(pipo_ctx* ctx, int32_t* h_tokens) {
    return step_sync(ctx, true, h_tokens, nullptr);
}

pipo_status pipo_rollback(pipo_ctx* ctx, const int32_t* h_n_pairs) {
    if (!ctx || !h_n_pairs) return fail(ctx, PIPO_EINVAL, "null argument");
    if (!ctx->prefilled) return fail(ctx, PIPO_ESTATE, "rollback before prefill");
    for (int b = 0; b < ctx->B; ++b)
        if (h_n_pairs[b] < 0 || h_n_pairs[b] > ctx->h_len[b])
            return fail(ctx, PIPO_EINVAL, "sequence %d: rollback to %d of %d entries", b, h_n_pairs[b], ctx->h_len[b]);
    CK(cudaSetDevice(ctx->dev));
    CK(cudaMemcpyAsync(ctx->n_pos, h_n_pairs, (size_t)ctx->B * 4, cudaMemcpyHostToDevice, ctx->stream));
    CK(cudaStreamSynchronize(ctx->stream));
    for (int b = 0; b < ctx->B; ++b) ctx->h_len[b] = h_n_pairs[b];
    return PIPO_OK;
}

pipo_status pipo_set_pending(pipo_ctx* ctx, const int32_t* h_pairs) {
    if (!ctx || !h_pairs) return fail(ctx, PIPO_EINVAL, "null argument");
    if (!ctx->prefilled) return fail(ctx, PIPO_ESTATE, "set_pending before prefill");
    for (int b = 0; b < ctx->B; ++b) {
        if (h_pairs[2 * b] < 0 || h_pairs[2 * b] >= ctx->cfg.vocab || h_pairs[2 * b + 1] < -1 ||
            h_pairs[2 * b + 1] >= ctx->cfg.vocab)
            return fail(ctx, PIPO_EINVAL, "sequence %d: pending pair out of range", b);
    }
    CK(cudaSetDevice(ctx->dev));
    CK(cudaMemcpyAsync(ctx->pending, h_pairs, (size_t)ctx->B * 8, cudaMemcpyHostToDevice, ctx->stream));
    CK(cudaStreamSynchronize(ctx->stream));
    return PIPO_OK;
}

pipo_status pipo_get_counters(pipo_ctx* ctx, int32_t* h_kv_len, int64_t* h_emitted) {
    if (!ctx) return fail(nullptr, PIPO_EINVAL, "null context");
    CK(cudaSetDevice(ctx->dev));
    if (h_kv_len) CK(cudaMemcpyAsync(h_kv_len, ctx->n_pos, (size_t)ctx->B * 4, cudaMemcpyDeviceToHost, ctx->stream));
    if (h_emitted) CK(cudaMemcpyAsync(h_emitted, ctx->emitted, (size_t)ctx->B * 8, cudaMemcpyDeviceToHost, ctx->stream));
    CK(cudaStreamSynchronize(ctx->stream));
    return check_device_error(ctx);
}

pipo_status pipo_debug_dump(pipo_ctx* ctx, const pipo_debug* o) {
    if (!ctx || !o) return fail(ctx, PIPO_EINVAL, "null argument");
    if (!ctx->cfg.debug) return fail(ctx, PIPO_ESTATE, "context was created without debug buffers");
    CK(cudaSetDevice(ctx->dev));
    const size_t B = ctx->B, V = ctx->cfg.vocab, H = ctx->cfg.hidden;
    cudaStream_t s = ctx->stream;
    if (o->logits_b) CK(cudaMemcpyAsync(o->logits_b, ctx->dbg_lb, B * V * 4, cudaMemcpyDeviceToHost, s));
    if (o->logits_d) CK(cudaMemcpyAsync(o->logits_d, ctx->dbg_ld, B * V * 4, cudaMemcpyDeviceToHost, s));
    if (o->conf) CK(cudaMemcpyAsync(o->conf, ctx->dbg_conf, B * 4, cudaMemcpyDeviceToHost, s));
    if (o->h_b) CK(cudaMemcpyAsync(o->h_b, ctx->dbg_hb, B * H * 4, cudaMemcpyDeviceToHost, s));
    if (o->h_d) CK(cudaMemcpyAsync(o->h_d, ctx->dbg_hd, B * H * 4, cudaMemcpyDeviceToHost, s));
    if (o->x_b) CK(cudaMemcpyAsync(o->x_b, ctx->dbg_xb, B * 4, cudaMemcpyDeviceToHost, s));
    if (o->x_d) CK(cudaMemcpyAsync(o->x_d, ctx->dbg_xd, B * 4, cudaMemcpyDeviceToHost, s));
    CK(cudaStreamSynchronize(s));
    return PIPO_OK;
}

pipo_status pipo_read_cache(pipo_ctx* ctx, int32_t b, int32_t layer, int32_t n, float* h_K, float* h_V) {
    if (!ctx || !h_K || !h_V) return fail(ctx, PIPO_EINVAL, "null argument");
    if (b < 0 || b >= ctx->cfg.max_batch || layer < 0 || layer >= ctx->n_cache_layers || n < 0 || n > ctx->cfg.max_ctx)
        return fail(ctx, PIPO_EINVAL, "read_cache: bad index");
    if (n == 0) return PIPO_OK;
    CK(cudaSetDevice(ctx->dev));
    const size_t kd = (size_t)ctx->cfg.n_kv_heads * ctx->cfg.head_dim;
    TRY(ensure_cache_tmp(ctx, 2 * kd * n));
    cache_copy_kernel<<<n, 256, 0, ctx->stream>>>(kv_view(ctx, layer), b, n, ctx->cfg.head_dim, ctx->cache_tmp, 0,
                                                   ctx->cfg.dtype == 1);
    CK(cudaGetLastError());
    CK(cudaMemcpyAsync(h_K, ctx->cache_tmp, kd * n * 4, cudaMemcpyDeviceToHost, ctx->stream));
    CK(cudaMemcpyAsync(h_V, ctx->cache_tmp + kd * n, kd * n * 4, cudaMemcpyDeviceToHost, ctx->stream));
    CK(cudaStreamSynchronize(ctx->stream));
    return PIPO_OK;
}

pipo_status pipo_load_cache(pipo_ctx* ctx, int32_t b, int32_t n, const float* h_K, const float* h_V) {
    if (!ctx || !h_K || !h_V) return fail(ctx, PIPO_EINVAL, "null argument");
    if (!ctx->prefilled || b < 0 || b >= ctx->B) return fail(ctx, PIPO_ESTATE, "load_cache needs a prefilled sequence b");
    if (n < 1 || n > ctx->cfg.max_ctx) return fail(ctx, PIPO_ECAPACITY, "load_cache: %d entries", n);
    drop_graph(ctx);  // the next step's launch plan is made for the new length
    CK(cudaSetDevice(ctx->dev));
    const size_t kd = (size_t)ctx->cfg.n_kv_heads * ctx->cfg.head_dim;
    TRY(ensure_cache_tmp(ctx, 2 * kd * n));
    for (int l = 0; l < ctx->n_cache_layers; ++l) {
        CK(cudaMemcpyAsync(ctx->cache_tmp, h_K + (size_t)l * n * kd, kd * n * 4, cudaMemcpyHostToDevice, ctx->stream));
        CK(cudaMemcpyAsync(ctx->cache_tmp + kd * n, h_V + (size_t)l * n * kd, kd * n * 4, cudaMemcpyHostToDevice, ctx->stream));
        cache_copy_kernel<<<n, 256, 0, ctx->stream>>>(kv_view(ctx, l), b, n, ctx->cfg.head_dim, ctx->cache_tmp, 1,
                                                       ctx->cfg.dtype == 1);
        CK(cudaGetLastError());
    }
    std::vector<int32_t> nn(1, n);
    CK(cudaMemcpyAsync(ctx->n_pos + b, nn.data(), 4, cudaMemcpyHostToDevice, ctx->stream));
    CK(cudaStreamSynchronize(ctx->stream));
    ctx->h_len[b] = n;
    return PIPO_OK;
}

namespace {
// launch settings of the kernel-level entry points (owns no memory)
pipo_status op_setup(pipo_ctx& op, int32_t dtype, void* stream) {
    pipo_ctx* ctx = &op;
    int dev = 0;
    CK(cudaGetDevice(&dev));
    if (op.sms == 0 || op.dev != dev || (int)op.esz != (dtype == 1 ? 2 : 4)) {
        op.dev = dev;
        CK(cudaDeviceGetAttribute(&op.sms, cudaDevAttrMultiProcessorCount, dev));
        op.cfg.dtype = dtype;
        op.esz = dtype == 1 ? 2 : 4;
        CK(set_smem_attrs(dtype == 1));
    }
    op.stream = static_cast<cudaStream_t>(stream);
    op.pdl = false;
    return PIPO_OK;
}

pipo_status op_lm_head_impl(pipo_ctx& op, int32_t dtype, const void* d_E, int32_t V, int32_t H, const float* d_h,
                            const void* d_gamma, float eps, int32_t B, int32_t* d_tokens, float* d_logits,
                            unsigned long long* keys, void* stream) {
    pipo_ctx* ctx = &op;
    TRY(op_setup(op, dtype, stream));
    CK(cudaMemsetAsync(keys, 0, (size_t)B * 8, op.stream));
    GemvParams p{};
    p.W = d_E;
    p.N = V;
    p.K = H;
    p.epi = EPI_ARGMAX;
    p.am = keys;
    p.dbg = d_logits;
    p.ld_dbg = V;
    p.B = B;
    p.splitk = 1;
    p.nseg = 1;
    p.eps = eps;
    p.seg[0] = act_seg(d_h, H, H, d_gamma);
    TRY(launch_gemv(ctx, p));
    keys_to_tokens_kernel<<<(B + 127) / 128, 128, 0, op.stream>>>(keys, d_tokens, B);
    CK(cudaGetLastError());
    return PIPO_OK;
}

pipo_status op_gemv_impl(pipo_ctx& op, int32_t dtype, int32_t mode, const void* d_W, int32_t N, int32_t K,
                         const float* d_x, int32_t B, float* d_y, void* stream) {
    pipo_ctx* ctx = &op;
    if (!d_W || !d_x || !d_y || N < 1 || K < 8 || K % 8 || B < 1 || (dtype != 0 && dtype != 1) ||
        (mode != 0 && mode != 1))
        return fail(nullptr, PIPO_EINVAL, "pipo_op_gemv: bad arguments");
    TRY(op_setup(op, dtype, stream));
    GemvParams p{};
    p.W = d_W;
    p.N = N;
    p.K = K;
    p.epi = mode == 1 ? EPI_SWIGLU : EPI_STORE;
    p.y = d_y;
    p.ldy = N;
    p.B = B;
    p.splitk = 1;
    p.nseg = 1;
    p.seg[0] = act_seg(d_x, K, K);
    return launch_gemv(ctx, p);
}
}  // namespace

pipo_status pipo_op_lm_head_argmax(int32_t dtype, const void* d_E, int32_t V, int32_t H, const float* d_h,
                                   const void* d_gamma, float eps, int32_t B, int32_t* d_tokens, float* d_logits,
                                   void* d_scratch, size_t scratch_bytes, void* stream) {
    if (!d_E || !d_h || !d_tokens || !d_scratch || V < 1 || H < 8 || H % 8 || B < 1 || (dtype != 0 && dtype != 1) ||
        !(eps >= 0.f) || reinterpret_cast<uintptr_t>(d_scratch) % 8 != 0)
        return fail(nullptr, PIPO_EINVAL, "pipo_op_lm_head_argmax: bad arguments");
    if (scratch_bytes < (size_t)B * 8)
        return fail(nullptr, PIPO_EINVAL, "pipo_op_lm_head_argmax: scratch needs %zu bytes, got %zu", (size_t)B * 8,
                    scratch_bytes);
    static thread_local pipo_ctx op;
    const pipo_status st = op_lm_head_impl(op, dtype, d_E, V, H, d_h, d_gamma, eps, B, d_tokens, d_logits,
                                           static_cast<unsigned long long*>(d_scratch), stream);
    if (st != PIPO_OK) g_init_error = op.err;
    return st;
}

}  // extern "C"

// ---- LM-head argmax without caller scratch --------------------------------
// For callers that may not allocate device memory.  The packed-key scratch is
// this fixed array: 64 keys, kept on every device that loads the library.  In
// host code its name is only a stand-in for the symbol, never a device
// address: the address is looked up per device with cudaGetSymbolAddress.
namespace {
constexpr int kNoAllocMaxBatch = 64;
constexpr int kNoAllocMaxDevices = 64;
unsigned long long* g_noalloc_keys_addr[kNoAllocMaxDevices] = {};  // per device, set on first use
std::mutex g_noalloc_mu;
}  // namespace
static __device__ __align__(256) unsigned long long g_lm_head_noalloc_keys[kNoAllocMaxBatch];

extern "C" {

pipo_status pipo_op_lm_head_argmax_noalloc(int32_t dtype, const void* d_E, int32_t V, int32_t H, const float* d_h,
                                           const void* d_gamma, float eps, int32_t B, int32_t* d_tokens,
                                           float* d_logits, void* stream) {
    if (!d_E || !d_h || !d_tokens || V < 1 || H < 8 || H % 8 || B < 1 || (dtype != 0 && dtype != 1) || !(eps >= 0.f))
        return fail(nullptr, PIPO_EINVAL, "pipo_op_lm_head_argmax_noalloc: bad arguments");
    if (B > kNoAllocMaxBatch)
        return fail(nullptr, PIPO_EINVAL, "pipo_op_lm_head_argmax_noalloc: %d sequences, at most %d", B,
                    kNoAllocMaxBatch);
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return fail(nullptr, PIPO_ECUDA, "cudaGetDevice: %s", cudaGetErrorString(e));
    if (dev < 0 || dev >= kNoAllocMaxDevices) return fail(nullptr, PIPO_EINVAL, "device ordinal %d unsupported", dev);
    unsigned long long* keys = nullptr;
    {
        std::lock_guard<std::mutex> lk(g_noalloc_mu);
        if (!g_noalloc_keys_addr[dev]) {
            // set-up, once per device, with that device current
            void* addr = nullptr;
            e = cudaGetSymbolAddress(&addr, g_lm_head_noalloc_keys);
            if (e != cudaSuccess)
                return fail(nullptr, PIPO_ECUDA, "cudaGetSymbolAddress(scratch): %s", cudaGetErrorString(e));
            g_noalloc_keys_addr[dev] = static_cast<unsigned long long*>(addr);
        }
        keys = g_noalloc_keys_addr[dev];
    }
    static thread_local pipo_ctx op;
    const pipo_status st = op_lm_head_impl(op, dtype, d_E, V, H, d_h, d_gamma, eps, B, d_tokens, d_logits, keys, stream);
    if (st != PIPO_OK) g_init_error = op.err;
    return st;
}

pipo_status pipo_op_gemv(int32_t dtype, int32_t mode, const void* d_W, int32_t N, int32_t K, const float* d_x,
                         int32_t B, float* d_y, void* stream) {
    static thread_local pipo_ctx op;  // device facts and launch settings only; owns no memory
    const pipo_status st = op_gemv_impl(op, dtype, mode, d_W, N, K, d_x, B, d_y, stream);
    if (st != PIPO_OK) g_init_error = op.err;
    return st;
}

pipo_status pipo_op_gemv_chain(int32_t dtype, int32_t mode, const void* const* d_Ws, int32_t count, int32_t N,
                               int32_t K, const float* d_x, int32_t B, float* d_y, int32_t pdl, void* stream) {
    static thread_local pipo_ctx op;
    pipo_ctx* ctx = &op;
    if (!d_Ws || count < 1 || !d_x || !d_y || N < 1 || K < 8 || K % 8 || B < 1 || (dtype != 0 && dtype != 1) ||
        (mode != 0 && mode != 1))
        return fail(nullptr, PIPO_EINVAL, "pipo_op_gemv_chain: bad arguments");
    for (int i = 0; i < count; ++i)
        if (!d_Ws[i]) return fail(nullptr, PIPO_EINVAL, "pipo_op_gemv_chain: null weight %d", i);
    pipo_status st = op_setup(op, dtype, stream);
    GemvParams p{};
    p.N = N; p.K = K; p.epi = mode == 1 ? EPI_SWIGLU : EPI_STORE; p.y = d_y; p.ldy = N; p.B = B;
    p.splitk = 1; p.nseg = 1; p.seg[0] = act_seg(d_x, K, K);
    for (int i = 0; st == PIPO_OK && i < count; ++i) {
        p.W = d_Ws[i];
        st = launch_gemv(ctx, p);
        op.pdl = pdl != 0;  // every launch after the first waits on the one before in-kernel
    }
    op.pdl = false;
    if (st != PIPO_OK) g_init_error = op.err;
    return st;
}

}  // extern "C"

namespace {
// scratch of pipo_op_gemm_tc: the [2 * BH][K] bf16 activation tile
size_t tc_scratch_bytes(int32_t K, int32_t B) { return (size_t)2 * tc_bn(B) * K * 2; }

bool tc_op_args_ok(int32_t mode, int32_t N, int32_t K, int32_t B, int32_t splits) {
    return (mode == 0 || mode == 1) && N >= 1 && N * (mode == 1 ? 2 : 1) >= kTcM && K >= kTcBK && K % kTcBK == 0 &&
           K <= 4 * kPrepQ * kPrepThreads &&
           B >= 1 && B <= 128 && splits >= 0;
}
}  // namespace

extern "C" {

size_t pipo_op_gemm_tc_scratch(int32_t mode, int32_t N, int32_t K, int32_t B, int32_t splits) {
    if (!tc_op_args_ok(mode, N, K, B, splits)) return 0;
    return tc_scratch_bytes(K, B);
}

pipo_status pipo_op_gemm_tc(int32_t mode, const void* d_W, int32_t N, int32_t K, const float* d_x, int32_t B,
                            float* d_y, int32_t splits, void* d_scratch, size_t scratch_bytes, void* stream) {
    if (!d_W || !d_x || !d_y || !d_scratch || !tc_op_args_ok(mode, N, K, B, splits) ||
        reinterpret_cast<uintptr_t>(d_W) % 16 != 0 || reinterpret_cast<uintptr_t>(d_scratch) % 1024 != 0)
        return fail(nullptr, PIPO_EINVAL, "pipo_op_gemm_tc: bad arguments");
    static thread_local pipo_ctx op;  // device facts and launch settings only; owns no memory
    pipo_ctx* ctx = &op;
    pipo_status st = op_setup(op, 1, stream);
    if (st == PIPO_OK) {
        const size_t need = tc_scratch_bytes(K, B);
        if (scratch_bytes < need) {
            st = fail(ctx, PIPO_EINVAL, "pipo_op_gemm_tc: scratch needs %zu bytes, got %zu", need, scratch_bytes);
        } else {
            GemvParams p{};
            p.W = d_W; p.N = N; p.K = K; p.epi = mode == 1 ? EPI_SWIGLU : EPI_STORE;
            p.y = d_y; p.ldy = N; p.B = B; p.splitk = 1; p.nseg = 1;
            p.seg[0] = act_seg(d_x, K, K);
            st = launch_gemm_tc(ctx, p, static_cast<bf16*>(d_scratch), splits, B);
        }
    }
    if (st != PIPO_OK) g_init_error = op.err;
    return st;
}

pipo_status pipo_op_gemm_tc_norm(int32_t mode, const void* d_W, int32_t N, const float* d_x0, int32_t K0,
                                 const void* d_gamma0, const float* d_x1, int32_t K1, const void* d_gamma1,
                                 int32_t joint, float eps, int32_t B, float* d_y, int32_t splits, void* d_scratch,
                                 size_t scratch_bytes, void* stream) {
    const bool two = d_x1 != nullptr;
    const int32_t K = K0 + (two ? K1 : 0);
    auto a16 = [](const void* q) { return reinterpret_cast<uintptr_t>(q) % 16 == 0; };
    const bool segs_ok = K0 >= kTcBK && K0 % kTcBK == 0 && (two ? (K1 >= kTcBK && K1 % kTcBK == 0) : K1 == 0) &&
                         (!joint || (two && d_gamma0 && !d_gamma1)) && (two || !d_gamma1) && eps >= 0.f;
    if (!d_W || !d_x0 || !d_y || !d_scratch || !segs_ok || !tc_op_args_ok(mode, N, K, B, splits) || !a16(d_W) ||
        !a16(d_x0) || (two && !a16(d_x1)) || !a16(d_gamma0) || !a16(d_gamma1) ||
        reinterpret_cast<uintptr_t>(d_scratch) % 1024 != 0)
        return fail(nullptr, PIPO_EINVAL, "pipo_op_gemm_tc_norm: bad arguments");
    static thread_local pipo_ctx op;  // device facts and launch settings only; owns no memory
    pipo_ctx* ctx = &op;
    pipo_status st = op_setup(op, 1, stream);
    if (st == PIPO_OK) {
        const size_t need = tc_scratch_bytes(K, B);
        if (scratch_bytes < need) {
            st = fail(ctx, PIPO_EINVAL, "pipo_op_gemm_tc_norm: scratch needs %zu bytes, got %zu", need, scratch_bytes);
        } else {
            GemvParams p{};
            p.W = d_W; p.N = N; p.K = K; p.epi = mode == 1 ? EPI_SWIGLU : EPI_STORE;
            p.y = d_y; p.ldy = N; p.B = B; p.splitk = 1; p.eps = eps;
            p.nseg = two ? 2 : 1;
            p.joint_norm = joint ? 1 : 0;
            p.seg[0] = act_seg(d_x0, K0, K0, d_gamma0);
            if (two) p.seg[1] = act_seg(d_x1, K1, K1, d_gamma1);
            st = launch_gemm_tc(ctx, p, static_cast<bf16*>(d_scratch), splits, B);
        }
    }
    if (st != PIPO_OK) g_init_error = op.err;
    return st;
}

pipo_status pipo_replay_family(pipo_ctx* ctx, int32_t family, int32_t n, double* h_bytes, int32_t* h_launches) {
    if (!ctx || family < 0 || family > 1 || n < 0) return fail(ctx, PIPO_EINVAL, "pipo_replay_family: bad arguments");
    if (!ctx->prefilled) return fail(ctx, PIPO_ESTATE, "family replay before prefill");
    if (ctx->regular) return fail(ctx, PIPO_ESTATE, "family replay of a regular-decoding context");
    CK(cudaSetDevice(ctx->dev));
    if (!ctx->fam_graph || ctx->fam_graph_family != family || ctx->fam_graph_B != ctx->B) {
        if (ctx->fam_graph) cudaGraphExecDestroy(ctx->fam_graph);
        ctx->fam_graph = nullptr;
        // the step's launch plan, captured with the other families' launches left out
        const int launches_before = ctx->launches;
        cudaGraph_t g = nullptr;
        CK(cudaStreamBeginCapture(ctx->stream, cudaStreamCaptureModeThreadLocal));
        ctx->only_family = family;
        ctx->fam_bytes = 0.0;
        ctx->fam_launches = 0;
        ctx->pdl = true;
        pipo_status s = enqueue_step(ctx);
        ctx->pdl = false;
        ctx->only_family = -1;
        ctx->launches = launches_before;
        cudaError_t e = cudaStreamEndCapture(ctx->stream, &g);
        if (s != PIPO_OK) {
            if (g) cudaGraphDestroy(g);
            return s;
        }
        if (e != cudaSuccess) return fail(ctx, PIPO_ECUDA, "family capture: %s", cudaGetErrorString(e));
        e = cudaGraphInstantiate(&ctx->fam_graph, g, 0);
        cudaGraphDestroy(g);
        if (e != cudaSuccess) return fail(ctx, PIPO_ECUDA, "family instantiate: %s", cudaGetErrorString(e));
        ctx->fam_graph_family = family;
        ctx->fam_graph_B = ctx->B;
    }
    for (int i = 0; i < n; ++i) CK(cudaGraphLaunch(ctx->fam_graph, ctx->stream));
    if (h_bytes) *h_bytes = ctx->fam_bytes;
    if (h_launches) *h_launches = ctx->fam_launches;
    return PIPO_OK;
}

pipo_status pipo_selftest_wait(int32_t signal, uint64_t limit_ns, uint32_t* h_info) {
    if (limit_ns == 0 || limit_ns > 10000000000ull)
        return fail(nullptr, PIPO_EINVAL, "pipo_selftest_wait: limit must be in (0, 10 s]");
    pipo_ctx* ctx = nullptr;  // failures go to the thread's context-free message
    unsigned code = 0, info[4] = {0, 0, 0, 0};
    CK(k_take_error_tc(&code, info));  // start from a clear error word
    int sig = signal ? 1 : 0;
    unsigned long long lim = limit_ns;
    void* args[] = {&sig, &lim};
    CK(cudaLaunchKernel(k_pick_wait_selftest(), dim3(1), dim3(32), args, 0, nullptr));
    CK(cudaStreamSynchronize(nullptr));
    code = 0;
    info[0] = info[1] = info[2] = info[3] = 0;
    CK(k_take_error_tc(&code, info));
    if (h_info) for (int i = 0; i < 4; ++i) h_info[i] = info[i];
    if (code)
        return fail(nullptr, PIPO_ECUDA, "device wait timed out (code %u; first at wait site %u, block %u)", code,
                    info[0], info[1]);
    return PIPO_OK;
}

#ifdef PIPO_TRACE
// Measurement build only (not part of the header): one timeline buffer of
// `cap` CTA records for the whole process, shared by every kernel unit.
// pipo_trace_setup(0) detaches and frees it.  pipo_trace_fetch copies the
// record count and up to cap records (6 words each) to h_out and resets the
// count.
namespace {
unsigned long long* g_trace_dev = nullptr;
size_t g_trace_cap = 0;
}  // namespace

PIPO_API pipo_status pipo_trace_setup(size_t cap) {
    pipo_ctx* ctx = nullptr;
    unsigned long long* buf = nullptr;
    if (cap) {
        CK(cudaMalloc(&buf, (2 + kTraceWords * cap) * sizeof(unsigned long long)));
        const unsigned long long head[2] = {0ull, (unsigned long long)cap};
        CK(cudaMemset(buf, 0, (2 + kTraceWords * cap) * sizeof(unsigned long long)));
        CK(cudaMemcpy(buf, head, sizeof(head), cudaMemcpyHostToDevice));
    }
    CK(k_trace_set_gemv_bf16(buf));
    CK(k_trace_set_gemv_f32(buf));
    CK(k_trace_set_tc(buf));
    CK(k_trace_set_attn(buf));
    CK(cudaDeviceSynchronize());
    if (g_trace_dev) CK(cudaFree(g_trace_dev));
    g_trace_dev = buf;
    g_trace_cap = cap;
    return PIPO_OK;
}

PIPO_API pipo_status pipo_trace_fetch(unsigned long long* h_out, size_t cap, unsigned long long* h_n) {
    pipo_ctx* ctx = nullptr;
    if (!g_trace_dev) return fail(nullptr, PIPO_ESTATE, "pipo_trace_fetch: no trace buffer");
    CK(cudaDeviceSynchronize());
    unsigned long long n = 0;
    CK(cudaMemcpy(&n, g_trace_dev, sizeof(n), cudaMemcpyDeviceToHost));
    *h_n = n;
    const size_t m = std::min<size_t>(std::min<size_t>(n, cap), g_trace_cap);
    if (m) CK(cudaMemcpy(h_out, g_trace_dev + 2, m * kTraceWords * sizeof(unsigned long long), cudaMemcpyDeviceToHost));
    CK(cudaMemset(g_trace_dev, 0, sizeof(unsigned long long)));
    CK(cudaDeviceSynchronize());
    return PIPO_OK;
}
#endif

pipo_status pipo_describe_step(const pipo_ctx* ctx, char* h_buf, size_t cap) {
    if (!ctx || !h_buf || cap == 0) return fail(nullptr, PIPO_EINVAL, "pipo_describe_step: bad arguments");
    const pipo_config& c = ctx->cfg;
    const int B = ctx->prefilled ? ctx->B : c.max_batch;
    const int H = c.hidden, qd = c.n_q_heads * c.head_dim, kd = c.n_kv_heads * c.head_dim;
    // the projections of a decoder block: (rows, K)
    const int shp[4][2] = {{qd + 2 * kd, H}, {H, qd}, {2 * c.ffn, H}, {H, c.ffn}};
    int n_tc = 0;
    for (auto& sh : shp) {
        GemvParams p{};
        p.N = sh[0];
        p.K = sh[1];
        p.B = B;
        p.epi = EPI_STORE;
        n_tc += tc_eligible(ctx, p) ? 1 : 0;
    }
    std::string proj;
    const std::string cuda_core = B <= 4 ? "gemv_rows_kernel" : "gemv_kernel";
    const bool fused = !tc_prep_forced() && tc_bn(B) <= tc_fused_max_bh();
    const std::string tck = fused ? "gemm_tcf_kernel<" + std::to_string(tc_bn(B)) + ">"
                                  : "gemm_tc_kernel<" + std::to_string(tc_bn(B)) + ">+prep_bf16_kernel";
    if (n_tc == 4) proj = tck + " (tcgen05)";
    else if (n_tc > 0) proj = tck + " (tcgen05; " + std::to_string(4 - n_tc) + " of 4 block projections on " +
                              cuda_core + ")";
    else proj = cuda_core;
    const int cs = attn_cluster_size(ctx, B);
    const int mma_flat = ctx->attn_v0 || !attn_use_mma(ctx, B) ? 0 : attn_mma_flat_splits(ctx, B);
    const bool mma = attn_use_mma(ctx, B) && (cs <= 8 || mma_flat > 0);
    const bool flat = !ctx->attn_v0 && !mma && attn_flat_now(ctx) && !ctx->attn_cs_force;
    std::string d = "B=" + std::to_string(B) + " projections=" + proj + " attention=" +
                    (ctx->attn_v0 ? std::string("attn_decode_kernel") : mma ? "attn_mma_kernel" : "attn_cluster_kernel") +
                    (mma_flat > 0 ? " unclustered splits=" + std::to_string(mma_flat)
                     : flat ? " unclustered splits=" +
                                  std::to_string(std::max(1, std::min({ctx->sms / (B * c.n_kv_heads),
                                                                       (c.max_ctx + 15) / 16, kFlatMaxSplits})))
                            : " cluster=" + std::to_string(cs) +
                                  (mma && attn_mma_deep(ctx, B, cs) ? " stages=" + std::to_string(kMmaDeepStages)
                                                                      : std::string()));
    // decoding mode, heads and prefill arrangement
    d += ctx->regular ? " mode=regular" : " mode=pair";
    d += ctx->samp_on ? " heads=sampled" : " heads=argmax";
    if (ctx->prefill_rows >= 2)
        d += " prefill=chunks of " + std::to_string(ctx->prefill_rows) + " rows (" +
             (ctx->prefill_tile_attn && attn_mma_ok(ctx) ? "attn_prefill_kernel" : "per-row attention") + ")";
    snprintf(h_buf, cap, "%s", d.c_str());
    return PIPO_OK;
}

pipo_status pipo_profile_step(pipo_ctx* ctx, int32_t cap, int32_t* h_kind, double* h_bytes, float* h_ms,
                              int32_t* h_n) {
    if (!ctx || !h_n || cap < 0) return fail(ctx, PIPO_EINVAL, "null argument");
    if (!ctx->prefilled) return fail(ctx, PIPO_ESTATE, "profile step before prefill");
    for (int b = 0; b < ctx->B; ++b)
        if (ctx->h_len[b] + 1 > ctx->cfg.max_ctx)
            return fail(ctx, PIPO_ECAPACITY, "sequence %d: KV cache full (%d entries)", b, ctx->h_len[b]);
    CK(cudaSetDevice(ctx->dev));
    CK(cudaStreamSynchronize(ctx->stream));
    ctx->prof = true;
    ctx->prof_n = 0;
    ctx->prof_k.clear();
    ctx->prof_b.clear();
    const int saved = ctx->launches;
    const bool pdl = ctx->pdl;
    ctx->pdl = false;
    pipo_status s = enqueue_step(ctx);
    ctx->pdl = pdl;
    ctx->prof = false;
    ctx->launches = saved;
    if (s != PIPO_OK) return s;
    CK(cudaStreamSynchronize(ctx->stream));
    for (int b = 0; b < ctx->B; ++b) ctx->h_len[b] += 1;
    *h_n = (int32_t)ctx->prof_n;
    for (size_t i = 0; i < ctx->prof_n && (int)i < cap; ++i) {
        float ms = 0.f;
        CK(cudaEventElapsedTime(&ms, ctx->prof_ev[2 * i], ctx->prof_ev[2 * i + 1]));
        if (h_kind) h_kind[i] = ctx->prof_k[i];
        if (h_bytes) h_bytes[i] = ctx->prof_b[i];
        if (h_ms) h_ms[i] = ms;
    }
    return check_device_error(ctx);
}

}  // extern "C"
