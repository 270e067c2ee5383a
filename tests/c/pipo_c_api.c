/*
 * A C99 program that uses only include/pipo.h: a small fp32 PIPO model
 * (the Tiny dimensions: H 256, 2 blocks, 4 query / 2 kv heads of 64, F 1024,
 * V 4096, Linear compressor, MTP block) with pseudo-random weights, a step
 * before any prefill (ESTATE), a prefill of an odd 11-token prompt (6
 * pairs, the last one ending in PAD), 8 decode steps with their outputs
 * checked for range and consistency, the counters, and pipo_free.
 *
 * Exit status: 0 all checks passed, 1 a check failed, 2 no context could be
 * created (e.g. no CUDA device): pipo_init returned a status and a message.
 */
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>

#include "pipo.h"

enum { H = 256, L = 2, NQ = 4, NKV = 2, DH = 64, F = 1024, V = 4096 };

static uint64_t rng_state = 88172645463325252ull;

/* xorshift64: uniform in [-0.035, 0.035) (standard deviation about 0.02) */
static float rnd(void) {
    rng_state ^= rng_state << 13;
    rng_state ^= rng_state >> 7;
    rng_state ^= rng_state << 17;
    return ((float)(rng_state >> 40) / 16777216.0f - 0.5f) * 0.07f;
}

static float *tensor(size_t n, int gain) {
    float *p = (float *)malloc(n * sizeof(float));
    if (!p) exit(1);
    for (size_t i = 0; i < n; i++) p[i] = gain ? 1.0f : rnd();
    return p;
}

#define CHECK(cond, ...)                     \
    do {                                     \
        if (!(cond)) {                       \
            fprintf(stderr, "FAIL: " __VA_ARGS__); \
            fprintf(stderr, "\n");           \
            return 1;                        \
        }                                    \
    } while (0)

int main(void) {
    const size_t qd = (size_t)NQ * DH, kd = (size_t)NKV * DH;
    pipo_config c = {0};
    c.hidden = H; c.n_layers = L; c.n_q_heads = NQ; c.n_kv_heads = NKV; c.head_dim = DH; c.ffn = F;
    c.vocab = V; c.compressor = 0; c.mtp_block = 1; c.dtype = 0; c.rope_theta = 1.0e4f; c.rms_eps = 1.0e-6f;
    c.max_batch = 1; c.max_ctx = 64; c.page_size = 64; c.tau = 0.5f; c.force_mode = 0; c.debug = 0;
    c.page_shuffle_seed = 0; c.comp_residual = 0;

    pipo_weights w = {0};
    w.location = 0;
    w.E = tensor((size_t)V * H, 0);
    w.x_pad = tensor(H, 0);
    w.comp_W = tensor((size_t)H * 2 * H, 0);
    w.comp_b = tensor(H, 0);
    w.attn_norm = tensor((size_t)L * H, 1);
    w.Wq = tensor((size_t)L * qd * H, 0);
    w.Wk = tensor((size_t)L * kd * H, 0);
    w.Wv = tensor((size_t)L * kd * H, 0);
    w.Wo = tensor((size_t)L * H * qd, 0);
    w.ffn_norm = tensor((size_t)L * H, 1);
    w.Wgate = tensor((size_t)L * F * H, 0);
    w.Wup = tensor((size_t)L * F * H, 0);
    w.Wdown = tensor((size_t)L * H * F, 0);
    w.final_norm = tensor(H, 1);
    w.mtp_norm_h = tensor(H, 1);
    w.mtp_norm_e = tensor(H, 1);
    w.mtp_W_fc = tensor((size_t)H * 2 * H, 0);
    w.m_attn_norm = tensor(H, 1);
    w.m_Wq = tensor(qd * H, 0);
    w.m_Wk = tensor(kd * H, 0);
    w.m_Wv = tensor(kd * H, 0);
    w.m_Wo = tensor((size_t)H * qd, 0);
    w.m_ffn_norm = tensor(H, 1);
    w.m_Wgate = tensor((size_t)F * H, 0);
    w.m_Wup = tensor((size_t)F * H, 0);
    w.m_Wdown = tensor((size_t)H * F, 0);
    w.mtp_norm_post = tensor(H, 1);
    w.conf_norm = tensor(2 * H, 1);
    w.conf_W1 = tensor((size_t)H * 2 * H, 0);
    w.conf_W2 = tensor(H, 0);

    pipo_ctx *ctx = NULL;
    pipo_status st = pipo_init(&c, &w, &ctx);
    if (st != PIPO_OK) {
        printf("pipo_init: status %d: %s\n", (int)st, pipo_last_error(NULL));
        return 2;
    }
    /* the weights were copied: the host buffers may go */
    free((void *)w.E);
    free((void *)w.Wgate);
    free((void *)w.Wup);

    int32_t tok[2] = {0, 0}, nacc = 0;
    CHECK(pipo_decode_step(ctx, tok, &nacc) == PIPO_ESTATE, "a step before the prefill must be ESTATE");

    int32_t ids[11], len = 11;
    for (int i = 0; i < 11; i++) ids[i] = (i * 37 + 5) % V;
    st = pipo_prefill(ctx, 1, ids, 11, &len, tok, &nacc);
    CHECK(st == PIPO_OK, "pipo_prefill: %d %s", (int)st, pipo_last_error(ctx));
    for (int step = 0; step <= 8; step++) {
        if (step > 0) {
            st = pipo_decode_step(ctx, tok, &nacc);
            CHECK(st == PIPO_OK, "pipo_decode_step: %d %s", (int)st, pipo_last_error(ctx));
        }
        CHECK(tok[0] >= 0 && tok[0] < V, "x_b out of range: %d", tok[0]);
        CHECK(nacc == 0 || nacc == 1, "n_accepted not 0/1: %d", nacc);
        CHECK(nacc ? (tok[1] >= 0 && tok[1] < V) : tok[1] == -1, "slot 1 %d does not match n_accepted %d",
              tok[1], nacc);
        printf("position %d: %d %d\n", step, tok[0], tok[1]);
    }
    int32_t kv = 0;
    int64_t emitted = 0;
    CHECK(pipo_get_counters(ctx, &kv, &emitted) == PIPO_OK, "pipo_get_counters");
    CHECK(kv == 6 + 8, "cache entries %d, expected 14", kv);
    CHECK(emitted >= 9 && emitted <= 18, "emitted %lld", (long long)emitted);
    pipo_free(ctx);
    printf("ok\n");
    return 0;
}
