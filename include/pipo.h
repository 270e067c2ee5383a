/*
 * pipo.h -- C ABI of the GB300 (sm_103a) PIPO pair-decode library.
 *
 * PIPO ("Pair-In, Pair-Out") decodes two tokens per backbone pass:
 *   Eq. 1  z^i = f([x^{2i}; x^{2i+1}])           pair-in compressor
 *   Eq. 2  h_b^i = Backbone(z^{<=i})              one decoder pass per pair
 *   Eq. 3  x_b = argmax LMHead(h_b^i)             LM head tied to E (App. B.2)
 *   Eq. 4  h_d^i = MTPHead(h_b^i, x_b)            App. A.2
 *   Eq. 5  x_d = argmax LMHead(h_d^i)
 *   Eq. 6  c^i = g([h_b^i; h_d^i])                confidence head, App. A.3
 *   Sec. 3.1-3.2: the next pair is (x_b, x_d) when c >= tau, else (x_b, PAD).
 *
 * Conventions for every entry point:
 *   - returns a pipo_status; never aborts the process; on failure the context
 *     keeps its previous state and pipo_last_error() describes the failure;
 *   - pointers named h_* or documented as "host" are host memory owned by the
 *     caller, read or written before the call returns; "device" pointers are
 *     device memory on the context's GPU, owned by the caller;
 *   - token ids are int32 in [0, vocab); -1 marks the PAD slot of a pair;
 *   - matrices are row-major [out, in] (a Linear layer's weight layout).
 *
 * Ownership: pipo_init copies the weights; the caller may free its buffers
 * afterwards.  The context owns every device buffer it allocates and frees
 * them in pipo_free.
 */
#ifndef PIPO_H
#define PIPO_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define PIPO_API __attribute__((visibility("default")))
#else
#define PIPO_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    PIPO_OK = 0,
    PIPO_EINVAL = 1,     /* bad argument (null pointer, id out of range, shape) */
    PIPO_ENOMEM = 2,     /* device allocation failed */
    PIPO_ECAPACITY = 3,  /* a KV cache would exceed max_ctx entries */
    PIPO_ECUDA = 4,      /* a CUDA runtime call failed */
    PIPO_ESTATE = 5      /* call out of order (e.g. a step before prefill) */
} pipo_status;

typedef struct pipo_ctx pipo_ctx; /* opaque */

/* Model dimensions and run-time switches. */
typedef struct {
    int32_t hidden;      /* H */
    int32_t n_layers;    /* L backbone blocks */
    int32_t n_q_heads;
    int32_t n_kv_heads;  /* GQA: n_q_heads % n_kv_heads == 0 */
    int32_t head_dim;    /* 64 or 128 */
    int32_t ffn;         /* SwiGLU inner size F */
    int32_t vocab;       /* V */
    int32_t compressor;  /* 0: Linear W[a;b]+b;  1: MLP W2 SiLU(W1[a;b]) (App. A.1) */
    int32_t mtp_block;   /* 1: W_fc then one decoder block (App. A.2); 0: W_fc only */
    int32_t dtype;       /* 0: fp32 weights and KV;  1: bf16 weights and KV */
    float rope_theta;    /* rotate-half RoPE base; position = pair index */
    float rms_eps;       /* RMSNorm epsilon (inside the root) */
    int32_t max_batch;   /* sequences decoded together */
    int32_t max_ctx;     /* KV entries (pairs) per sequence, prompt included */
    int32_t page_size;   /* entries per KV block; 64 */
    float tau;           /* acceptance threshold tau_c (c >= tau accepts) */
    int32_t force_mode;  /* 0: confidence rule; 1: accept every draft; 2: reject every draft */
    int32_t debug;       /* 1: keep logits and head states for pipo_debug_dump */
    uint32_t page_shuffle_seed; /* 0: blocks in order; else a seeded permutation of
                                   the physical block pool (layout must not matter) */
    int32_t comp_residual; /* 1: the MLP compressor adds a + b, z = a + b + W2 SiLU(W1[a;b])
                              (its residual form, App. A.1); requires compressor = 1 */
} pipo_config;

/* Weights: one pointer per tensor, element type per pipo_config.dtype
 * (float, or bf16 bit patterns as uint16).  Stacked tensors hold the L
 * backbone blocks back to back.  `location`: 0 host, 1 device memory.
 * Unused tensors (the other compressor variant, the MTP block when
 * mtp_block == 0) may be NULL. */
typedef struct {
    int32_t location;
    const void *E;          /* [V, H] token embedding, tied LM head */
    const void *x_pad;      /* [H]    PAD embedding */
    const void *comp_W;     /* [H, 2H] Linear compressor */
    const void *comp_b;     /* [H] */
    const void *comp_W1;    /* [H, 2H] MLP compressor */
    const void *comp_W2;    /* [H, H] */
    const void *attn_norm;  /* [L, H] */
    const void *Wq;         /* [L, n_q*d_h, H] */
    const void *Wk;         /* [L, n_kv*d_h, H] */
    const void *Wv;         /* [L, n_kv*d_h, H] */
    const void *Wo;         /* [L, H, n_q*d_h] */
    const void *ffn_norm;   /* [L, H] */
    const void *Wgate;      /* [L, F, H] */
    const void *Wup;        /* [L, F, H] */
    const void *Wdown;      /* [L, H, F] */
    const void *final_norm; /* [H] */
    const void *mtp_norm_h; /* [H]  norm of h_b at the MTP input */
    const void *mtp_norm_e; /* [H]  norm of E[x_b] at the MTP input */
    const void *mtp_W_fc;   /* [H, 2H] */
    const void *m_attn_norm, *m_Wq, *m_Wk, *m_Wv, *m_Wo, *m_ffn_norm, *m_Wgate, *m_Wup, *m_Wdown; /* one block */
    const void *mtp_norm_post; /* [H] norm before the LM head on h_d */
    const void *conf_norm;  /* [2H] one RMSNorm over [h_b; h_d] */
    const void *conf_W1;    /* [H, 2H] */
    const void *conf_W2;    /* [1, H] */
} pipo_weights;

/* Head states of the last step (debug contexts only); host buffers. */
typedef struct {
    float *logits_b;   /* [B, V] backbone LM-head logits, or NULL */
    float *logits_d;   /* [B, V] MTP LM-head logits, or NULL */
    float *conf;       /* [B] confidence c, or NULL */
    float *h_b;        /* [B, H] last backbone block output, or NULL */
    float *h_d;        /* [B, H] MTP block output, or NULL */
    int32_t *x_b;      /* [B] backbone argmax, or NULL */
    int32_t *x_d;      /* [B] draft argmax (whether accepted or not), or NULL */
} pipo_debug;

/* Create a context on the current CUDA device for one PIPO model: the latent
 * compressor (Sec. 3.2 Eq. 1, App. A.1), the backbone decoder blocks (Eq. 2),
 * the tied LM head (Eq. 3, App. B.2), the MTP head (Eq. 4-5, App. A.2) and
 * the confidence head (Eq. 6, App. A.3), with the shapes in cfg.  Validates
 * the config, copies the weights to device memory (fused QKV and gate|up
 * layouts), allocates the paged KV caches (backbone layers and the MTP
 * layer) for max_batch x max_ctx entries.  *out receives the context.
 * EINVAL for inconsistent shapes or a missing weight tensor, ENOMEM when
 * device memory runs out (everything allocated so far is freed and *out is
 * left NULL).  For tests of that path, the environment variable
 * PIPO_TEST_FAIL_ALLOC=k makes the k-th device allocation of this call
 * report out-of-memory without allocating. */
PIPO_API pipo_status pipo_init(const pipo_config *cfg, const pipo_weights *w, pipo_ctx **out);

/* Prefill B sequences (B <= max_batch) from host token ids h_ids, row b at
 * h_ids + b*stride, h_lens[b] tokens (1 <= len <= stride).  Tokens are paired
 * (t_{2j}, t_{2j+1}); an odd length ends in (t_last, PAD) (App. B.2).  Runs
 * the backbone over the N latents, fills both caches, and runs the heads on
 * the last latent: h_tokens[B,2] / h_n_accepted[B] (host, may be NULL) get
 * the first pair output, which also becomes the pending pair.  Resets the
 * emitted counters.  ECAPACITY when N > max_ctx.  Sequences that yield
 * different numbers of pairs are prefilled one after another, each as
 * pipo_prefill_slot does (all are validated first).  On any failure the
 * context is left not prefilled (a decode step returns ESTATE until the next
 * successful prefill). */
PIPO_API pipo_status pipo_prefill(pipo_ctx *ctx, int32_t batch, const int32_t *h_ids, int32_t stride,
                         const int32_t *h_lens, int32_t *h_tokens, int32_t *h_n_accepted);

/* Continuous batching: prefill one slot (sequence `slot` < max_batch) from
 * the host prompt h_ids[0, len) while every other slot keeps its state (its
 * cache, length, pending pair and counters), e.g. a request joining a batch
 * that is decoding.  The prompt is paired as in pipo_prefill; (len + 1) / 2
 * <= max_ctx entries.  Outputs (host, may be NULL): h_tokens[2] and
 * h_n_accepted[1] of the slot's first pair.  The decode steps then run slots
 * 0 .. max(slot, previous batch - 1); a slot that was never prefilled decodes
 * from token 0 on an empty cache (its outputs mean nothing).  Slots of one
 * batch may hold prompts of different lengths.  ESTATE after a
 * regular-decoding prefill; EINVAL for a bad slot, length or id;
 * ECAPACITY as pipo_prefill.  On failure the slot's state is undefined and
 * the other slots are unchanged. */
PIPO_API pipo_status pipo_prefill_slot(pipo_ctx *ctx, int32_t slot, const int32_t *h_ids, int32_t len,
                                       int32_t *h_tokens, int32_t *h_n_accepted);

/* One pair-decode step of every prefilled sequence: compress the pending
 * pair, one backbone pass, both heads, the confidence rule, next pair, KV
 * append.  Host outputs (may be NULL): h_tokens[B,2] = (x_b, x_d or -1 when
 * the draft was rejected), h_n_accepted[B] in {0,1}.  Synchronous.
 * ESTATE before a prefill; ECAPACITY when a cache is full. */
PIPO_API pipo_status pipo_decode_step(pipo_ctx *ctx, int32_t *h_tokens, int32_t *h_n_accepted);

/* The same step, enqueued on the context stream without a host sync;
 * d_tokens[B,2] / d_n_accepted[B] are device buffers (may be NULL).  The
 * step is a captured CUDA graph replayed per call.  Its launch plan (kernel
 * forms, attention splits) is made for the mean cached length at capture
 * and kept while the caches grow; a prefill, a cache load or a change of
 * batch, stream, threshold or sampler drops the graph, and the next step
 * captures a new one. */
PIPO_API pipo_status pipo_decode_step_async(pipo_ctx *ctx, int32_t *d_tokens, int32_t *d_n_accepted);

/* n_steps pair-decode steps in one call (graph replays back to back, one
 * host synchronisation at the end): h_tokens[n_steps][B][2] and
 * h_n_accepted[n_steps][B] (host, may be NULL) receive every step's
 * outputs.  ESTATE before a prefill or in regular mode; ECAPACITY when a
 * cache would exceed max_ctx within the n steps (nothing runs then). */
PIPO_API pipo_status pipo_decode_steps(pipo_ctx *ctx, int32_t n_steps, int32_t *h_tokens,
                                       int32_t *h_n_accepted);

/* Regular decoding, the baseline the paper measures PIPO against (Sec. 4,
 * "Regular"; its TPOT comparison): the same backbone, one token per pass.
 * The input of a pass is the token's embedding E[t] (no compressor), its
 * position is the token index, the cache holds one entry per token (backbone
 * caches only), and the final-norm tied LM head's argmax (Eq. 3) is the next
 * token; the MTP and confidence heads do not run.
 *
 * pipo_regular_prefill: arguments as pipo_prefill, but every sequence must
 * have the same length N (EINVAL otherwise) and the prompt takes N cache
 * entries (ECAPACITY when N > max_ctx).  Each prompt token runs the backbone
 * at its own position; the last one also runs the LM head.  Outputs (may be
 * NULL): h_tokens[B,2] = (first generated token, -1), h_n_accepted[B] = 0.
 * Resets the emitted counters to 0.  Puts the context in regular mode until
 * the next pipo_prefill.
 *
 * pipo_regular_step: one pass for every sequence, from the pending token
 * (slot 0 of the pending pair; pipo_set_pending overwrites it).  h_tokens
 * [B,2] = (token, -1) (may be NULL).  Synchronous; ESTATE before a regular
 * prefill or after a pair prefill, ECAPACITY when a cache is full.
 * pipo_decode_step returns ESTATE in regular mode.
 *
 * pipo_regular_step_async: the same step enqueued on the context stream (a
 * captured CUDA graph); d_tokens[B,2] is a device buffer (may be NULL). */
PIPO_API pipo_status pipo_regular_prefill(pipo_ctx *ctx, int32_t batch, const int32_t *h_ids, int32_t stride,
                                          const int32_t *h_lens, int32_t *h_tokens, int32_t *h_n_accepted);
PIPO_API pipo_status pipo_regular_step(pipo_ctx *ctx, int32_t *h_tokens);
PIPO_API pipo_status pipo_regular_step_async(pipo_ctx *ctx, int32_t *d_tokens);

/* Truncate both KV caches of sequence b to h_n_pairs[b] entries (host,
 * [B], each <= the current length).  Test and bookkeeping primitive: PIPO
 * itself never caches a rejected draft (Sec. 3.1), so decoding never calls it.
 * The pending pair is left as is (set it with pipo_set_pending). */
PIPO_API pipo_status pipo_rollback(pipo_ctx *ctx, const int32_t *h_n_pairs);

/* Acceptance threshold tau_c of the confidence rule (Sec. 3.1-3.2: the draft
 * is kept when c >= tau_c) and the force mode: 0 the rule; 1 accept every
 * draft, which is the "MTP without verification" baseline of App. C.2; 2
 * reject every draft (one token per pair, Sec. 3.1).  Takes effect from the
 * next step.  EINVAL for a mode outside 0..2 or a tau that is not finite. */
PIPO_API pipo_status pipo_set_threshold(pipo_ctx *ctx, float tau, int32_t force_mode);

/* The paper's evaluation sampler in both heads (Sec. 4; its settings:
 * temperature 1, top_k 20, top_p 0.95, repetition penalty 1.5) in place of
 * the greedy argmax.  Per head and sequence: a logit l of an id already in the
 * sequence's tokens so far (the prompt, then every emitted token) becomes
 * l / rep_penalty if l > 0, else l * rep_penalty; divide by temperature; keep
 * the top_k largest (ties to the lower id); keep the shortest prefix whose
 * softmax mass reaches top_p; pick the first id whose cumulative renormalised
 * mass exceeds u times the prefix mass.  x_b is drawn first and joins the
 * history before x_d is drawn; an accepted x_d joins it after the decision;
 * the MTP input takes the drawn x_b.
 *
 * h_u: host [n_u][max_batch][2] uniform draws in [0, 1) (slot 0 for x_b,
 * slot 1 for x_d); the k-th position that runs the heads (the prefill's last
 * position, then each decode step) takes row k mod n_u.  Copied; the caller
 * keeps ownership.  Resets the draw index to 0.  Call before pipo_prefill
 * (the history is seeded from the prompt there).  temperature <= 0 turns the
 * sampler off (greedy; the other arguments are ignored).  EINVAL: top_k not
 * in [1, 32], top_p not in (0, 1], rep_penalty <= 0, a draw outside [0, 1),
 * or no draws.  Regular decoding stays greedy. */
PIPO_API pipo_status pipo_set_sampler(pipo_ctx *ctx, float temperature, int32_t top_k, float top_p,
                                      float rep_penalty, const float *h_u, int32_t n_u);

/* Test hook for forced replay: overwrite the pending pairs, host [B,2]
 * (slot 1 may be -1 = PAD). */
PIPO_API pipo_status pipo_set_pending(pipo_ctx *ctx, const int32_t *h_pairs);

/* Host copies of the per-sequence counters: kv entries [B] and tokens
 * emitted since the prefill [B] (either may be NULL). */
PIPO_API pipo_status pipo_get_counters(pipo_ctx *ctx, int32_t *h_kv_len, int64_t *h_emitted);

/* Head states of the last step or prefill, for parity checks of Eq. 3-6:
 * the LM-head logits of both heads (Eq. 3 and Eq. 5), the confidence c
 * (Eq. 6), h_b and h_d (the block outputs the heads read, App. A.2-A.3) and
 * both argmax tokens.  Requires cfg.debug = 1 (ESTATE otherwise); host
 * buffers in *out, any of them NULL to skip. */
PIPO_API pipo_status pipo_debug_dump(pipo_ctx *ctx, const pipo_debug *out);

/* Host fp32 copy of cache entries [0, n) of sequence b, layer l (l == L is
 * the MTP layer): h_K, h_V [n, n_kv*d_h]. */
PIPO_API pipo_status pipo_read_cache(pipo_ctx *ctx, int32_t b, int32_t layer, int32_t n, float *h_K, float *h_V);

/* Write n entries into every cache layer of sequence b and set its length
 * to n: host fp32 [L+1, n, n_kv*d_h] (rounded to the cache type).  For
 * timing runs that need a long context without a long prefill. */
PIPO_API pipo_status pipo_load_cache(pipo_ctx *ctx, int32_t b, int32_t n, const float *h_K, const float *h_V);

/* Use a caller-owned CUDA stream (cudaStream_t) for all later work; NULL
 * restores the context's own stream.  Drops the captured step graph. */
PIPO_API pipo_status pipo_set_stream(pipo_ctx *ctx, void *stream);

/* ---- kernel-level entry points (device buffers, no context) ------------
 * They run one kernel of the decode path on caller-owned device memory, on
 * `stream` (a cudaStream_t; NULL = the legacy default stream), without a
 * host sync.  Used to time and test kernels in isolation. */

/* Weight-streaming GEMV of the backbone projections (Eq. 2 blocks):
 *   mode 0: y[b*N + r] = sum_k W[r*K + k] * x[b*K + k]             (W: [N, K])
 *   mode 1: y[b*N + r] = SiLU(W[2r,:] . x[b,:]) * (W[2r+1,:] . x[b,:])
 *           (SwiGLU with gate and up rows interleaved; W: [2N, K])
 * dtype 0: W fp32, 1: W bf16; x [B, K] and y [B, N] fp32.  K must be a
 * multiple of 8 and B*K*4 <= 200 KB per 4 sequences.  EINVAL otherwise. */
PIPO_API pipo_status pipo_op_gemv(int32_t dtype, int32_t mode, const void *d_W, int32_t N, int32_t K,
                                  const float *d_x, int32_t B, float *d_y, void *stream);

/* Measurement op: `count` GEMVs of the pipo_op_gemv form back to back on
 * `stream`, weights d_Ws[i] (device pointers, [N or 2N, K] each), the same
 * input and output; with pdl != 0 every launch after the first carries the
 * programmatic-dependent-launch attribute (its weight prologue overlaps the
 * launch before, its input and output wait for it), as in a decode step.
 * Captured in a CUDA graph, the time per launch against one GEMV of the
 * summed weights gives the fixed cost of a launch.  EINVAL as pipo_op_gemv
 * or for a NULL weight. */
PIPO_API pipo_status pipo_op_gemv_chain(int32_t dtype, int32_t mode, const void *const *d_Ws, int32_t count,
                                        int32_t N, int32_t K, const float *d_x, int32_t B, float *d_y, int32_t pdl,
                                        void *stream);

/* Tensor-core form of the same projections (Eq. 2 blocks) for batches that
 * make them dense contractions: tcgen05 MMAs with fp32 accumulation in TMEM.
 * Each fp32 activation enters as two bf16 parts, hi = bf16(x) and
 * lo = bf16(x - hi), multiplied by the same bf16 weights (about 2^-17
 * relative representation error; the weight traffic is that of one pass):
 *   mode 0: y[b*N + r] = sum_k W[r*K + k] * x[b*K + k]              (W: [N, K])
 *   mode 1: SwiGLU as in pipo_op_gemv (W: [2N, K], gate/up rows interleaved).
 * W bf16, 16-byte aligned; x [B, K] and y [B, N] fp32.  K a multiple of 64
 * and at most 16384, N (mode 1: 2N) >= 128, 1 <= B <= 128.  splits: K splits per 128-row tile,
 * at most 8 (0 = automatic; larger values are clamped); the splits of a tile
 * are one thread-block cluster and add their partials in split order
 * (deterministic).
 * d_scratch: 1024-byte-aligned device memory of at least
 * pipo_op_gemm_tc_scratch(mode, N, K, B, splits) bytes, overwritten.
 * EINVAL for bad shapes, alignment or a short scratch buffer. */
PIPO_API pipo_status pipo_op_gemm_tc(int32_t mode, const void *d_W, int32_t N, int32_t K, const float *d_x,
                                     int32_t B, float *d_y, int32_t splits, void *d_scratch, size_t scratch_bytes,
                                     void *stream);

/* Scratch bytes pipo_op_gemm_tc needs on the current device (0 for
 * arguments it rejects or when no device is usable). */
PIPO_API size_t pipo_op_gemm_tc_scratch(int32_t mode, int32_t N, int32_t K, int32_t B, int32_t splits);

/* The tensor-core projection of RMS-normalised inputs, as the decode step
 * applies it: to RMSNorm(x; gamma) in the blocks (Eq. 2, pre-norm), to
 * [RMSNorm(h_b); RMSNorm(E[x_b])] with two gains at the MTP input (App. A.2)
 * and to RMSNorm([h_b; h_d]) with one gain over 2H in the confidence head
 * (App. A.3).  The input of sequence b is the concatenation of
 *   segment 0: x0[b*K0 .. b*K0 + K0)   and, when d_x1 != NULL,
 *   segment 1: x1[b*K1 .. b*K1 + K1)   (K = K0 + K1; else K1 must be 0),
 * normalised as follows (r(v) = v / sqrt(mean(v^2) + eps)):
 *   joint = 0: each segment with a non-NULL gain becomes gamma_s * r(segment),
 *              a segment with a NULL gain enters unchanged;
 *   joint = 1: both segments together become gamma0 * r(concatenation),
 *              gamma0 of length K, d_gamma1 NULL.
 * Then y = W . input as pipo_op_gemm_tc (mode 0 plain, mode 1 SwiGLU).
 * Gains bf16, W bf16; x0, x1, y fp32; W, x0, x1 and the gains 16-byte
 * aligned; K0 and K1 multiples of 64; N, B, splits and the scratch
 * (pipo_op_gemm_tc_scratch(mode, N, K0 + K1, B, splits) bytes, 1024-byte
 * aligned) as pipo_op_gemm_tc.  B <= 32 with one segment or one joint norm
 * runs the converter warps inside the GEMM when B is 16 or 32; every other
 * case prepares the bf16 operand in a separate pass first.  EINVAL for bad
 * shapes, alignment, gain combinations or a short scratch buffer. */
PIPO_API pipo_status pipo_op_gemm_tc_norm(int32_t mode, const void *d_W, int32_t N, const float *d_x0, int32_t K0,
                                          const void *d_gamma0, const float *d_x1, int32_t K1, const void *d_gamma1,
                                          int32_t joint, float eps, int32_t B, float *d_y, int32_t splits,
                                          void *d_scratch, size_t scratch_bytes, void *stream);

/* Fused LM head + argmax over the tied embedding (Eq. 3 and Eq. 5, App. B.2):
 *   d_tokens[b] = argmax_v  E[v,:] . RMSNorm(h[b,:]; gamma)
 * with the lowest v winning ties; the logits are never stored unless
 * d_logits [B, V] fp32 is given.  dtype 0: E and gamma fp32, 1: bf16;
 * E [V, H]; d_h [B, H] fp32; d_gamma [H] or NULL (no norm); eps inside the
 * root.  d_scratch: at least 8*B bytes of 8-byte-aligned device memory for the
 * packed (logit, row) keys, overwritten (contents unspecified on return).
 * Enqueued on `stream`.  EINVAL for bad shapes or a short scratch buffer. */
PIPO_API pipo_status pipo_op_lm_head_argmax(int32_t dtype, const void *d_E, int32_t V, int32_t H, const float *d_h,
                                            const void *d_gamma, float eps, int32_t B, int32_t *d_tokens,
                                            float *d_logits, void *d_scratch, size_t scratch_bytes, void *stream);

/* The same fused LM head + argmax as pipo_op_lm_head_argmax, for callers
 * that cannot allocate device memory: for example a host program that hands
 * every byte of the GPU to its own pool at start-up and allows no other
 * allocation, or a latency-critical loop in which a cudaMalloc (which can
 * synchronize the device) is not acceptable.  The paper has no counterpart:
 * it is a deployment variant of this library.  It allocates nothing; its
 * scratch is a fixed array of 64 packed keys (512 bytes) that the library
 * keeps in device memory on every GPU that loads it, for the life of the
 * process.  Hence B <= 64 (EINVAL otherwise).  The first call on each device
 * looks up that array's device address (cudaGetSymbolAddress) with the device
 * current; make that first call before any stream capture.  Every call on a
 * device shares the one array and zeroes it first, so calls that overlap on
 * the GPU (other streams, or other host threads) race and must be
 * serialized by the caller.  The looked-up address is kept for the life of
 * the process: after cudaDeviceReset (or anything else that destroys the
 * device's primary context) the entry point must not be called again on that
 * device.  Arguments otherwise as pipo_op_lm_head_argmax. */
PIPO_API pipo_status pipo_op_lm_head_argmax_noalloc(int32_t dtype, const void *d_E, int32_t V, int32_t H,
                                                    const float *d_h, const void *d_gamma, float eps, int32_t B,
                                                    int32_t *d_tokens, float *d_logits, void *stream);

/* Kernel timing of one decode step run eagerly (no graph) on the context
 * stream, with CUDA events recorded around every launch.  For launch i in step
 * order: h_kind[i] (0 weight-streaming GEMV, 1 attention, 2 other), h_bytes[i]
 * the algorithmic bytes it must move (weights it streams; for attention the
 * KV entries it reads plus the one it writes), h_ms[i] its event-timed
 * duration.  *h_n receives the launch count (at most cap are written).
 * Advances the decode state exactly like pipo_decode_step. */
PIPO_API pipo_status pipo_profile_step(pipo_ctx *ctx, int32_t cap, int32_t *h_kind, double *h_bytes, float *h_ms,
                                       int32_t *h_n);

/* Roofline timing of one kernel family inside the decode step: enqueues, on
 * the context stream, n replays of a CUDA graph holding only that family's
 * launches of one pair-decode step (Sec. 3.2 Eq. 1-6), with the step's launch
 * plan, in step order and with the step's programmatic dependent launch
 * between consecutive launches.  family 0: the weight-streaming projections
 * (every projection of Eq. 1-6 and both LM-head passes, Eq. 3 and Eq. 5,
 * with the operand preparation some of them need); family 1: the attention
 * launches (Eq. 2).  Time the replays with events on the context stream.
 * With a captured step graph the family takes that graph's launch plan.
 * The decoding state does not change: pending pairs, cache lengths,
 * counters and every live cache entry stay as they were (an attention
 * replay writes only the entry one past each sequence's cached length, which
 * the next step overwrites before reading it); the activation buffers are
 * left with meaningless values.  *h_bytes receives the algorithmic bytes
 * one replay moves (weights streamed; for attention the cached entries read
 * and the one written), *h_launches its launch count (either may be NULL).
 * The graph is captured on the first call for a family and batch (n = 0
 * captures without replaying).  EINVAL for a bad family or n < 0; ESTATE
 * before a prefill or on a regular-decoding context.  A measurement aid of
 * this library; the paper has no counterpart. */
PIPO_API pipo_status pipo_replay_family(pipo_ctx *ctx, int32_t family, int32_t n, double *h_bytes,
                                        int32_t *h_launches);

/* Self-test of the bounded device waits that every kernel of this library
 * uses (mbarrier waits give up after a time limit instead of spinning
 * forever, set a device error word and record the wait site; the host then
 * reports PIPO_ECUDA).  Launches one block on the legacy default stream of the
 * current device whose thread 0 waits, with a limit of limit_ns
 * nanoseconds, on an mbarrier that only it can complete: signal != 0
 * completes it first (PIPO_OK expected), signal == 0 never does, so the
 * wait gives up after limit_ns and the call returns PIPO_ECUDA.
 * h_info[4] (host, may be NULL) receives the wait record {site (90 for this
 * test), block, iteration, parity}, zeros when nothing timed out.  Reads and
 * clears the error word of the tensor-core unit, so run it while no other
 * work of this library is in flight on the device.  EINVAL for a limit of
 * 0 or above 10 s.  A reliability aid of this library; the paper has no
 * counterpart. */
PIPO_API pipo_status pipo_selftest_wait(int32_t signal, uint64_t limit_ns, uint32_t *h_info);

/* Which kernels the next decode step launches for the projections and the
 * attention, and the attention cluster size, as one NUL-terminated line of
 * at most cap bytes in h_buf, e.g. "B=16 projections=gemm_tc_kernel<16>+
 * prep_bf16_kernel (tcgen05) attention=attn_mma_kernel cluster=2
 * mode=pair heads=argmax", followed by the prefill arrangement when chunks
 * are enabled.  Batch B
 * is the prefilled batch (before a prefill: cfg.max_batch).  A report of
 * this library's kernel choices; the paper has no counterpart.  EINVAL for
 * a NULL context or buffer or cap == 0. */
PIPO_API pipo_status pipo_describe_step(const pipo_ctx *ctx, char *h_buf, size_t cap);

/* Number of kernel launches one decode step enqueues (for launch accounting). */
PIPO_API int32_t pipo_step_launches(const pipo_ctx *ctx);

/* Message of the last failure on this context; with ctx NULL, of the last
 * failed call made without a context (pipo_init, the pipo_op_* entry points)
 * on the calling thread.  Never NULL; the string stays valid until the next
 * failing call on the same context (ctx NULL: on the same thread). */
PIPO_API const char *pipo_last_error(const pipo_ctx *ctx);

/* Release every device buffer and the context; NULL is a no-op. */
PIPO_API void pipo_free(pipo_ctx *ctx);

#ifdef __cplusplus
}
#endif
#endif /* PIPO_H */
