/*
 * PIPO oracle: a plain, slow, fp64 CPU implementation of the PIPO pair step.
 *
 * TEST INFRASTRUCTURE ONLY.  The CUDA library never links, includes or calls
 * this file; only the test-suite, the package smoke check and the CPU-baseline
 * leg of the benchmark load it.  It shares no code with the GPU path.
 *
 * What it computes (per sequence; notation of paper Sec. 3):
 *   Eq. 1      z^i   = f_theta([x^{2i}; x^{2i+1}])          compressor
 *              Linear variant  W [a;b] + b,  MLP variant  W2 SiLU(W1 [a;b])
 *              (App. A.1, Table "Compressor variants"); optionally the MLP
 *              with the residual a + b added (comp_residual), the form whose
 *              zeroed branch gives a + b
 *   Eq. 2      h_b^i = Backbone(z^{<=i})                     decoder stack
 *   Eq. 3      p_b   = LMHead(h_b^i)                          tied to E (App. B.2)
 *   Eq. 4      h_d^i = MTPHead(h_b^i, x^{2i+2})
 *              = Layer(W_fc [RMSNorm(h_b^i); RMSNorm(x^{2i+2})])   (App. A.2)
 *   Eq. 5      p_d   = LMHead(h_d^i)  (after the MTP post-norm, App. B.2)
 *   Eq. 6      c^i   = sigma(W2 SiLU(W1 RMSNorm([h_b^i; h_d^i])))   (App. A.3)
 *   Sec. 3.1 / 3.2 acceptance: next pair (x^{2i+2}, x^{2i+3}) if c >= tau,
 *              else (x^{2i+2}, x^pad).
 *
 * Readings where the paper is silent (each also listed in the design notes):
 *   decoder block = pre-norm RMSNorm -> GQA attention with rotate-half RoPE at
 *   position = pair index -> residual -> RMSNorm -> SwiGLU -> residual, no
 *   biases; RMSNorm y = x / sqrt(mean(x^2) + eps) * gamma; h_b and h_d are the
 *   block outputs before any final norm; the LM head applies the final norm;
 *   argmax ties go to the lowest index; c >= tau accepts; the MTP layer keeps
 *   its own KV cache with one entry per pair step, teacher-forced at prefill
 *   with the first token of the following pair; an odd prompt ends in a pair
 *   whose second slot is PAD (App. B.2).
 *
 * Precision: all arithmetic in double.  Weights are read in their storage type
 * (fp32 or bf16) and widened exactly.  With kv_bf16 set, keys (after RoPE)
 * and values are rounded to bf16 when stored, as a bf16 cache stores them.
 *
 * Also: regular decoding of the same backbone (one token per pass, no
 * compressor or heads beyond the LM head), the baseline the paper compares
 * PIPO with (orc_regular_prefill / orc_regular_step); and the paper's
 * evaluation sampler in both heads (orc_set_sampler, orc_step_u,
 * orc_prefill_u: temperature, top-k, top-p, repetition penalty over the
 * sequence's tokens so far, the uniform draws passed in).
 *
 * Parity of every function here is pinned by the not-gpu tests (closed forms,
 * special cases, brute-force recompute, invariants).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORC_PAD (-1)

typedef struct {
    int H, L, n_q, n_kv, d_h, F, V;
    int compressor; /* 0 linear, 1 mlp */
    int mtp_block;  /* 1: W_fc then one decoder block; 0: W_fc only */
    int wdtype;     /* 0 fp32, 1 bf16 (uint16 bit patterns) */
    int kv_bf16;    /* round cached K,V to bf16 */
    double rope_theta, eps;
    int max_ctx;    /* cache entries per sequence */
    int comp_residual; /* 1: the MLP compressor adds a + b (the residual form of App. A.1) */
} orc_config;

/* Host pointers; element type per wdtype; matrices row-major [out, in]. */
typedef struct {
    const void *E, *x_pad;
    const void *comp_W, *comp_b, *comp_W1, *comp_W2;
    const void *attn_norm, *Wq, *Wk, *Wv, *Wo, *ffn_norm, *Wgate, *Wup, *Wdown; /* stacked [L,...] */
    const void *final_norm;
    const void *mtp_norm_h, *mtp_norm_e, *mtp_W_fc;
    const void *m_attn_norm, *m_Wq, *m_Wk, *m_Wv, *m_Wo, *m_ffn_norm, *m_Wgate, *m_Wup, *m_Wdown;
    const void *mtp_norm_post;
    const void *conf_norm, *conf_W1, *conf_W2;
} orc_weights;

/* ------------------------------------------------------------------ */
/* element access                                                      */

static double wget(const void *p, size_t i, int dt) {
    if (dt == 0) return (double)((const float *)p)[i];
    uint32_t bits = ((uint32_t)((const uint16_t *)p)[i]) << 16;
    float f;
    memcpy(&f, &bits, 4);
    return (double)f;
}

/* round a double to the nearest bf16 value (ties to even), returned as double */
double orc_round_bf16(double d) {
    if (d == 0.0 || !isfinite(d)) return d;
    int e;
    double m = frexp(d, &e);          /* d = m * 2^e, 0.5 <= |m| < 1 */
    double r = nearbyint(ldexp(m, 8)); /* 8 significant bits */
    return ldexp(r, e - 8);
}

/* ------------------------------------------------------------------ */
/* primitives                                                          */

/* RMSNorm: y = x / sqrt(mean(x^2) + eps) * gamma */
void orc_rmsnorm(const double *x, int n, const void *gamma, size_t goff, int dt,
                 double eps, double *y) {
    double ss = 0.0;
    for (int i = 0; i < n; i++) ss += x[i] * x[i];
    double r = 1.0 / sqrt(ss / n + eps);
    for (int i = 0; i < n; i++) y[i] = x[i] * r * wget(gamma, goff + i, dt);
}

/* y[n] = sum_k W[off + n*K + k] * x[k], n < N */
void orc_matvec(const void *W, size_t off, int dt, int N, int K, const double *x, double *y) {
#pragma omp parallel for schedule(static)
    for (int n = 0; n < N; n++) {
        double acc = 0.0;
        size_t row = off + (size_t)n * K;
        for (int k = 0; k < K; k++) acc += wget(W, row + k, dt) * x[k];
        y[n] = acc;
    }
}

double orc_silu(double x) { return x / (1.0 + exp(-x)); }
double orc_sigmoid(double x) { return 1.0 / (1.0 + exp(-x)); }

/* Rotate-half RoPE on n_heads vectors of size d at position pos:
 * for i < d/2, (v_i, v_{i+d/2}) is rotated by angle pos * theta^(-2i/d). */
void orc_rope(double *v, int n_heads, int d, int pos, double theta) {
    int half = d / 2;
    for (int i = 0; i < half; i++) {
        double ang = (double)pos * pow(theta, -2.0 * i / d);
        double c = cos(ang), s = sin(ang);
        for (int h = 0; h < n_heads; h++) {
            double *u = v + (size_t)h * d;
            double a = u[i], b = u[i + half];
            u[i] = a * c - b * s;
            u[i + half] = b * c + a * s;
        }
    }
}

/* GQA attention of one position: for query head h, group g = h / (n_q/n_kv);
 * out_h = sum_j softmax_j(q_h . k_{j,g} / sqrt(d)) v_{j,g}, j < n.
 * K and V: [n][n_kv*d]. */
void orc_attend(const double *q, const double *K, const double *V, int n,
                int n_q, int n_kv, int d, double *out) {
    int grp = n_q / n_kv;
    double scale = 1.0 / sqrt((double)d);
#pragma omp parallel for schedule(static)
    for (int h = 0; h < n_q; h++) {
        int g = h / grp;
        const double *qh = q + (size_t)h * d;
        double *s = (double *)malloc(sizeof(double) * (n > 0 ? n : 1));
        double m = -INFINITY;
        for (int j = 0; j < n; j++) {
            const double *kj = K + (size_t)j * n_kv * d + (size_t)g * d;
            double dot = 0.0;
            for (int t = 0; t < d; t++) dot += qh[t] * kj[t];
            s[j] = dot * scale;
            if (s[j] > m) m = s[j];
        }
        double den = 0.0;
        for (int j = 0; j < n; j++) { s[j] = exp(s[j] - m); den += s[j]; }
        double *oh = out + (size_t)h * d;
        for (int t = 0; t < d; t++) oh[t] = 0.0;
        for (int j = 0; j < n; j++) {
            const double *vj = V + (size_t)j * n_kv * d + (size_t)g * d;
            double p = s[j] / den;
            for (int t = 0; t < d; t++) oh[t] += p * vj[t];
        }
        free(s);
    }
}

/* argmax with the lowest index winning ties; *margin = top1 - top2 */
int orc_argmax(const double *x, int n, double *margin) {
    int best = 0;
    for (int i = 1; i < n; i++) if (x[i] > x[best]) best = i;
    double second = -INFINITY;
    for (int i = 0; i < n; i++) if (i != best && x[i] > second) second = x[i];
    if (margin) *margin = (n > 1) ? x[best] - second : INFINITY;
    return best;
}

/* The paper's evaluation sampler as a primitive (temperature, top-k, top-p,
 * repetition penalty; its settings: T = 1, k = 20, p = 0.95, penalty 1.5).
 * The random draw u in [0, 1) is an input.  Steps, in this order:
 *   1. repetition penalty r over the distinct ids of hist[0, n_hist): a logit
 *      l becomes l / r if l > 0, else l * r;
 *   2. temperature T: l / T;
 *   3. top-k: the k largest (k <= 0 or k >= V keeps all), in descending logit
 *      order with ties to the lower id;
 *   4. top-p: the shortest prefix of that order whose softmax mass reaches p;
 *   5. the first id of that prefix whose cumulative renormalised mass exceeds u.
 * k == 1 is greedy (the argmax with ties to the lower id). */
typedef struct {
    double v;
    int id;
} orc_scored;

static int scored_desc(const void *a, const void *b) {
    const orc_scored *x = (const orc_scored *)a, *y = (const orc_scored *)b;
    if (x->v > y->v) return -1;
    if (x->v < y->v) return 1;
    return (x->id > y->id) - (x->id < y->id);
}

/* The same draw, also returning in *margin (if not NULL) how far the decision
 * is from changing: the smallest of
 *   - the logit gaps (after penalty and temperature) between the picked id
 *     and its neighbours in the order (a swap would move the pick),
 *   - the gap at the top-k boundary when the nucleus takes all k ids,
 *   - the distance of the top-p cut from p (p < 1),
 *   - the distance of u from the ends of the picked id's interval of
 *     cumulative renormalised mass.
 * Logit gaps and masses mix units; a caller compares the margin with a
 * threshold above both its logit and its mass errors.  For k == 1 the margin
 * is the top-1 / top-2 logit gap, as for the argmax. */
int orc_sample_ex(const double *logits, int V, const int32_t *hist, int n_hist, double temperature, int top_k,
                  double top_p, double rep_penalty, double u, double *margin) {
    orc_scored *sc = (orc_scored *)malloc(sizeof(orc_scored) * V);
    unsigned char *seen = (unsigned char *)calloc(V, 1);
    for (int i = 0; i < n_hist; i++)
        if (hist[i] >= 0 && hist[i] < V) seen[hist[i]] = 1;
    for (int i = 0; i < V; i++) {
        double l = logits[i];
        if (seen[i]) l = (l > 0.0) ? l / rep_penalty : l * rep_penalty;
        sc[i].v = l / temperature;
        sc[i].id = i;
    }
    qsort(sc, V, sizeof(orc_scored), scored_desc);
    int keep = (top_k <= 0 || top_k > V) ? V : top_k;
    double *e = (double *)malloc(sizeof(double) * keep);
    double Z = 0.0;
    for (int i = 0; i < keep; i++) { e[i] = exp(sc[i].v - sc[0].v); Z += e[i]; }
    int np = keep;
    double cum = 0.0;
    for (int i = 0; i < keep; i++) {
        cum += e[i];
        if (cum / Z >= top_p) { np = i + 1; break; }
    }
    double Zp = 0.0;
    for (int i = 0; i < np; i++) Zp += e[i];
    const double target = u * Zp;
    int k = np - 1;  /* position of the pick in the order */
    cum = 0.0;
    for (int i = 0; i < np; i++) {
        if (cum + e[i] > target) { k = i; break; }
        cum += e[i];
    }
    double below = 0.0;  /* mass before position k */
    for (int i = 0; i < k; i++) below += e[i];
    int pick = sc[k].id;
    if (margin) {
        double m = INFINITY;
        if (k > 0) m = fmin(m, sc[k - 1].v - sc[k].v);
        if (k + 1 < V) m = fmin(m, sc[k].v - sc[k + 1].v);
        if (np == keep && keep < V) m = fmin(m, sc[keep - 1].v - sc[keep].v);
        if (top_p < 1.0) {
            double c = 0.0;
            for (int i = 0; i < np; i++) c += e[i];
            m = fmin(m, c / Z - top_p);
            if (np >= 2) m = fmin(m, top_p - (c - e[np - 1]) / Z);
        }
        if (k > 0) m = fmin(m, u - below / Zp);                  /* interior interval ends only */
        if (k < np - 1) m = fmin(m, (below + e[k]) / Zp - u);
        *margin = m;
    }
    free(sc); free(seen); free(e);
    return pick;
}

int orc_sample(const double *logits, int V, const int32_t *hist, int n_hist, double temperature, int top_k,
               double top_p, double rep_penalty, double u) {
    return orc_sample_ex(logits, V, hist, n_hist, temperature, top_k, top_p, rep_penalty, u, NULL);
}

/* ------------------------------------------------------------------ */
/* model pieces                                                        */

typedef struct {
    const void *attn_norm, *Wq, *Wk, *Wv, *Wo, *ffn_norm, *Wgate, *Wup, *Wdown;
    int idx; /* layer index inside the stacked tensors */
} blockw;

static blockw backbone_layer(const orc_weights *w, int l) {
    blockw b = {w->attn_norm, w->Wq, w->Wk, w->Wv, w->Wo, w->ffn_norm, w->Wgate, w->Wup, w->Wdown, l};
    return b;
}
static blockw mtp_layer(const orc_weights *w) {
    blockw b = {w->m_attn_norm, w->m_Wq, w->m_Wk, w->m_Wv, w->m_Wo, w->m_ffn_norm, w->m_Wgate, w->m_Wup, w->m_Wdown, 0};
    return b;
}

/* embedding of one slot: a row of E, or x^pad for the PAD slot */
static void embed(const orc_config *c, const orc_weights *w, int tok, double *x) {
    for (int i = 0; i < c->H; i++)
        x[i] = (tok == ORC_PAD) ? wget(w->x_pad, i, c->wdtype)
                                : wget(w->E, (size_t)tok * c->H + i, c->wdtype);
}

/* Eq. 1 with the App. A.1 variants: z = f([emb(t0); emb(t1)]) */
void orc_compress(const orc_config *c, const orc_weights *w, int t0, int t1, double *z) {
    int H = c->H, dt = c->wdtype;
    double *ab = (double *)malloc(sizeof(double) * 2 * H);
    embed(c, w, t0, ab);
    embed(c, w, t1, ab + H);
    if (c->compressor == 0) {
        orc_matvec(w->comp_W, 0, dt, H, 2 * H, ab, z);
        for (int i = 0; i < H; i++) z[i] += wget(w->comp_b, i, dt);
    } else {
        double *t = (double *)malloc(sizeof(double) * H);
        orc_matvec(w->comp_W1, 0, dt, H, 2 * H, ab, t);
        for (int i = 0; i < H; i++) t[i] = orc_silu(t[i]);
        orc_matvec(w->comp_W2, 0, dt, H, H, t, z);
        if (c->comp_residual)
            for (int i = 0; i < H; i++) z[i] += ab[i] + ab[H + i];
        free(t);
    }
    free(ab);
}

/* q, k, v of one position: RMSNorm then the three projections, RoPE on q, k.
 * k and v are rounded to bf16 when the cache stores bf16. */
static void block_qkv(const orc_config *c, blockw b, const double *x, int pos,
                      double *q, double *k, double *v) {
    int H = c->H, dt = c->wdtype, qd = c->n_q * c->d_h, kd = c->n_kv * c->d_h;
    double *y = (double *)malloc(sizeof(double) * H);
    orc_rmsnorm(x, H, b.attn_norm, (size_t)b.idx * H, dt, c->eps, y);
    orc_matvec(b.Wq, (size_t)b.idx * qd * H, dt, qd, H, y, q);
    orc_matvec(b.Wk, (size_t)b.idx * kd * H, dt, kd, H, y, k);
    orc_matvec(b.Wv, (size_t)b.idx * kd * H, dt, kd, H, y, v);
    orc_rope(q, c->n_q, c->d_h, pos, c->rope_theta);
    orc_rope(k, c->n_kv, c->d_h, pos, c->rope_theta);
    if (c->kv_bf16)
        for (int i = 0; i < kd; i++) { k[i] = orc_round_bf16(k[i]); v[i] = orc_round_bf16(v[i]); }
    free(y);
}

/* the rest of the block once the attention output a is known:
 * x += Wo a; x += Wdown(SiLU(Wgate y) * Wup y), y = RMSNorm(x) */
static void block_tail(const orc_config *c, blockw b, double *x, const double *a) {
    int H = c->H, F = c->F, dt = c->wdtype, qd = c->n_q * c->d_h;
    double *o = (double *)malloc(sizeof(double) * H);
    double *y = (double *)malloc(sizeof(double) * H);
    double *g = (double *)malloc(sizeof(double) * F);
    double *u = (double *)malloc(sizeof(double) * F);
    orc_matvec(b.Wo, (size_t)b.idx * H * qd, dt, H, qd, a, o);
    for (int i = 0; i < H; i++) x[i] += o[i];
    orc_rmsnorm(x, H, b.ffn_norm, (size_t)b.idx * H, dt, c->eps, y);
    orc_matvec(b.Wgate, (size_t)b.idx * F * H, dt, F, H, y, g);
    orc_matvec(b.Wup, (size_t)b.idx * F * H, dt, F, H, y, u);
    for (int i = 0; i < F; i++) g[i] = orc_silu(g[i]) * u[i];
    orc_matvec(b.Wdown, (size_t)b.idx * H * F, dt, H, F, g, o);
    for (int i = 0; i < H; i++) x[i] += o[i];
    free(o); free(y); free(g); free(u);
}

/* Final-norm LM head over the tied embedding: logits = E RMSNorm(h; gamma) */
static void lm_head(const orc_config *c, const orc_weights *w, const double *h,
                    const void *gamma, double *logits) {
    double *y = (double *)malloc(sizeof(double) * c->H);
    orc_rmsnorm(h, c->H, gamma, 0, c->wdtype, c->eps, y);
    orc_matvec(w->E, 0, c->wdtype, c->V, c->H, y, logits);
    free(y);
}

/* App. A.2 input of the MTP layer: u = W_fc [RMSNorm(h_b); RMSNorm(E[tok])] */
static void mtp_input(const orc_config *c, const orc_weights *w, const double *hb, int tok, double *u) {
    int H = c->H, dt = c->wdtype;
    double *cat = (double *)malloc(sizeof(double) * 2 * H);
    double *e = (double *)malloc(sizeof(double) * H);
    orc_rmsnorm(hb, H, w->mtp_norm_h, 0, dt, c->eps, cat);
    embed(c, w, tok, e);
    orc_rmsnorm(e, H, w->mtp_norm_e, 0, dt, c->eps, cat + H);
    orc_matvec(w->mtp_W_fc, 0, dt, H, 2 * H, cat, u);
    free(cat); free(e);
}

/* App. A.3: c = sigma(W2 SiLU(W1 RMSNorm([h_b; h_d]))) with one norm over 2H */
double orc_confidence(const orc_config *c, const orc_weights *w, const double *hb, const double *hd) {
    int H = c->H, dt = c->wdtype;
    double *cat = (double *)malloc(sizeof(double) * 2 * H);
    double *y = (double *)malloc(sizeof(double) * 2 * H);
    double *t = (double *)malloc(sizeof(double) * H);
    memcpy(cat, hb, sizeof(double) * H);
    memcpy(cat + H, hd, sizeof(double) * H);
    orc_rmsnorm(cat, 2 * H, w->conf_norm, 0, dt, c->eps, y);
    orc_matvec(w->conf_W1, 0, dt, H, 2 * H, y, t);
    double s = 0.0;
    for (int i = 0; i < H; i++) s += wget(w->conf_W2, i, dt) * orc_silu(t[i]);
    free(cat); free(y); free(t);
    return orc_sigmoid(s);
}

/* ------------------------------------------------------------------ */
/* stateful, KV-cached decoding                                        */

typedef struct {
    int p0, p1;        /* pending pair; p1 may be PAD */
    int n;             /* cache entries = pairs consumed */
    long emitted;      /* tokens emitted by decode steps */
    double **K, **Vc;  /* L+1 caches of [max_ctx][n_kv*d_h]; index L = MTP layer */
    int32_t *hist;     /* the sequence's tokens so far: the prompt, then every emitted token */
    int n_hist, cap_hist;
} orc_seq;

/* Sampling in both heads (the paper's evaluation setting, Sec. 4): off
 * (greedy argmax) unless set. */
typedef struct {
    int on;
    double temperature, top_p, rep_penalty;
    int top_k;
} orc_sampler;

typedef struct {
    orc_config c;
    orc_weights w;
    int B;
    orc_seq *s;
    orc_sampler sp;
} orc_state;

static void hist_push(orc_seq *s, int tok) {
    if (s->n_hist == s->cap_hist) {
        s->cap_hist = s->cap_hist ? 2 * s->cap_hist : 256;
        s->hist = (int32_t *)realloc(s->hist, sizeof(int32_t) * s->cap_hist);
    }
    s->hist[s->n_hist++] = tok;
}

/* per-sequence, per-step results */
typedef struct {
    int32_t *tokens;   /* [B,2]; slot 1 = -1 when the draft is rejected */
    int32_t *n_acc;    /* [B] */
    double *logits_b;  /* [B,V] or NULL */
    double *logits_d;  /* [B,V] or NULL */
    double *conf;      /* [B] or NULL */
    double *h_b, *h_d; /* [B,H] or NULL */
    double *margin_b, *margin_d; /* [B] or NULL */
    int32_t *x_b, *x_d; /* [B] or NULL: both argmaxes, whatever the decision */
} orc_out;

orc_state *orc_new(const orc_config *c, const orc_weights *w, int B) {
    orc_state *st = (orc_state *)calloc(1, sizeof(orc_state));
    st->c = *c;
    st->w = *w;
    st->B = B;
    st->s = (orc_seq *)calloc(B > 0 ? B : 1, sizeof(orc_seq));
    size_t per = (size_t)c->max_ctx * c->n_kv * c->d_h;
    int nl = c->L + (c->mtp_block ? 1 : 0);
    for (int b = 0; b < B; b++) {
        st->s[b].K = (double **)calloc(c->L + 1, sizeof(double *));
        st->s[b].Vc = (double **)calloc(c->L + 1, sizeof(double *));
        for (int l = 0; l < nl; l++) {
            st->s[b].K[l] = (double *)calloc(per, sizeof(double));
            st->s[b].Vc[l] = (double *)calloc(per, sizeof(double));
            if (!st->s[b].K[l] || !st->s[b].Vc[l]) return NULL;
        }
        st->s[b].p0 = 0;
        st->s[b].p1 = ORC_PAD;
    }
    return st;
}

void orc_free(orc_state *st) {
    if (!st) return;
    for (int b = 0; b < st->B; b++) {
        for (int l = 0; l <= st->c.L; l++) { free(st->s[b].K[l]); free(st->s[b].Vc[l]); }
        free(st->s[b].K); free(st->s[b].Vc);
        free(st->s[b].hist);
    }
    free(st->s);
    free(st);
}

/* one decoder block at position pos with a KV cache: append, then attend
 * over entries 0..pos (pos = entries before the append). */
static void block_cached(const orc_config *c, blockw b, double *x, int pos, double *Kc, double *Vc) {
    int kd = c->n_kv * c->d_h, qd = c->n_q * c->d_h;
    double *q = (double *)malloc(sizeof(double) * qd);
    double *a = (double *)malloc(sizeof(double) * qd);
    block_qkv(c, b, x, pos, q, Kc + (size_t)pos * kd, Vc + (size_t)pos * kd);
    orc_attend(q, Kc, Vc, pos + 1, c->n_q, c->n_kv, c->d_h, a);
    block_tail(c, b, x, a);
    free(q); free(a);
}

/* backbone pass of one latent at position n of sequence s: returns h_b in x */
static void backbone_at(orc_state *st, orc_seq *s, double *x) {
    for (int l = 0; l < st->c.L; l++)
        block_cached(&st->c, backbone_layer(&st->w, l), x, s->n, s->K[l], s->Vc[l]);
}

/* MTP head at position n: h_d from h_b and the token fed to the MTP input */
static void mtp_at(orc_state *st, orc_seq *s, const double *hb, int tok, double *hd) {
    mtp_input(&st->c, &st->w, hb, tok, hd);
    if (st->c.mtp_block)
        block_cached(&st->c, mtp_layer(&st->w), hd, s->n, s->K[st->c.L], s->Vc[st->c.L]);
}

/* Heads and acceptance of one position: LM head -> x_b, MTP -> x_d,
 * confidence, the acceptance rule, next pair, n += 1.  With the sampler on,
 * x_b is drawn from the backbone head with the draw u2[0] and the sequence's
 * tokens so far as the repetition history, and x_d from the draft head with
 * u2[1] and that history followed by x_b (x_b precedes x_d in the output);
 * the MTP input takes the drawn x_b.  The history then keeps x_b, and x_d
 * when it is accepted. */
static void heads_and_accept(orc_state *st, int b, double *hb, double tau, int force, const double *u2,
                             orc_out *o) {
    const orc_config *c = &st->c;
    const orc_sampler *sp = &st->sp;
    orc_seq *s = &st->s[b];
    int H = c->H, V = c->V;
    double *lb = (double *)malloc(sizeof(double) * V);
    double *ld = (double *)malloc(sizeof(double) * V);
    double *hd = (double *)malloc(sizeof(double) * H);
    double mb, md;
    lm_head(c, &st->w, hb, st->w.final_norm, lb);
    int xb = sp->on ? orc_sample_ex(lb, V, s->hist, s->n_hist, sp->temperature, sp->top_k, sp->top_p,
                                    sp->rep_penalty, u2[0], &mb)
                    : orc_argmax(lb, V, &mb);
    hist_push(s, xb);
    mtp_at(st, s, hb, xb, hd);
    lm_head(c, &st->w, hd, st->w.mtp_norm_post, ld);
    int xd = sp->on ? orc_sample_ex(ld, V, s->hist, s->n_hist, sp->temperature, sp->top_k, sp->top_p,
                                    sp->rep_penalty, u2[1], &md)
                    : orc_argmax(ld, V, &md);
    double conf = orc_confidence(c, &st->w, hb, hd);
    int acc = (force == 1) ? 1 : (force == 2) ? 0 : (conf >= tau);
    if (acc) hist_push(s, xd);
    s->p0 = xb;
    s->p1 = acc ? xd : ORC_PAD;
    s->n += 1;
    s->emitted += 1 + acc;
    if (o) {
        if (o->tokens) { o->tokens[2 * b] = xb; o->tokens[2 * b + 1] = acc ? xd : -1; }
        if (o->n_acc) o->n_acc[b] = acc;
        if (o->logits_b) memcpy(o->logits_b + (size_t)b * V, lb, sizeof(double) * V);
        if (o->logits_d) memcpy(o->logits_d + (size_t)b * V, ld, sizeof(double) * V);
        if (o->conf) o->conf[b] = conf;
        if (o->h_b) memcpy(o->h_b + (size_t)b * H, hb, sizeof(double) * H);
        if (o->h_d) memcpy(o->h_d + (size_t)b * H, hd, sizeof(double) * H);
        if (o->margin_b) o->margin_b[b] = mb;
        if (o->margin_d) o->margin_d[b] = md;
        if (o->x_b) o->x_b[b] = xb;
        if (o->x_d) o->x_d[b] = xd;
    }
    free(lb); free(ld); free(hd);
}

/* error codes shared with the Python wrapper */
#define ORC_OK 0
#define ORC_EINVAL 1
#define ORC_ECAPACITY 3

/* Sampling in both heads: temperature T, top-k, top-p, repetition penalty
 * (orc_sample_ex); T <= 0 turns it off (greedy argmax). */
int orc_set_sampler(orc_state *st, double temperature, int top_k, double top_p, double rep_penalty) {
    if (temperature <= 0.0) { st->sp.on = 0; return ORC_OK; }
    if (!(top_p > 0.0 && top_p <= 1.0) || !(rep_penalty > 0.0)) return ORC_EINVAL;
    st->sp.on = 1;
    st->sp.temperature = temperature;
    st->sp.top_k = top_k;
    st->sp.top_p = top_p;
    st->sp.rep_penalty = rep_penalty;
    return ORC_OK;
}

/* One pair-decode step for every sequence (Sec. 3.1-3.2). force: 0 use the
 * confidence rule, 1 accept every draft, 2 reject every draft.  u: the draws
 * [B][2] of both heads when the sampler is on (else unused, may be NULL). */
int orc_step_u(orc_state *st, double tau, int force, const double *u, orc_out *o) {
    const orc_config *c = &st->c;
    if (st->sp.on && !u) return ORC_EINVAL;
    for (int b = 0; b < st->B; b++) if (st->s[b].n >= c->max_ctx) return ORC_ECAPACITY;
    double *x = (double *)malloc(sizeof(double) * c->H);
    for (int b = 0; b < st->B; b++) {
        orc_seq *s = &st->s[b];
        orc_compress(c, &st->w, s->p0, s->p1, x);
        backbone_at(st, s, x);
        heads_and_accept(st, b, x, tau, force, u ? u + 2 * b : NULL, o);
    }
    free(x);
    return ORC_OK;
}

int orc_step(orc_state *st, double tau, int force, orc_out *o) { return orc_step_u(st, tau, force, NULL, o); }

/* Prefill: prompt of len_b tokens per sequence (row stride `stride`), paired
 * as (t_{2j}, t_{2j+1}); an odd length ends in (t_last, PAD) (App. B.2).
 * Every latent runs the backbone causally; the MTP cache entry of position
 * j < N-1 is fed the first token of pair j+1; the last position runs the
 * heads and the acceptance rule, which sets the first pending pair. */
int orc_prefill_u(orc_state *st, const int32_t *ids, const int32_t *lens, int stride,
                  double tau, int force, const double *u, orc_out *o) {
    const orc_config *c = &st->c;
    if (st->sp.on && !u) return ORC_EINVAL;
    for (int b = 0; b < st->B; b++) {
        int len = lens[b];
        int N = (len + 1) / 2;
        if (len < 1 || len > stride || N > c->max_ctx) return N > c->max_ctx ? ORC_ECAPACITY : ORC_EINVAL;
        for (int t = 0; t < len; t++) if (ids[(size_t)b * stride + t] < 0 || ids[(size_t)b * stride + t] >= c->V) return ORC_EINVAL;
    }
    double *x = (double *)malloc(sizeof(double) * c->H);
    double *hd = (double *)malloc(sizeof(double) * c->H);
    for (int b = 0; b < st->B; b++) {
        orc_seq *s = &st->s[b];
        const int32_t *t = ids + (size_t)b * stride;
        int len = lens[b], N = (len + 1) / 2;
        s->n = 0;
        s->emitted = 0;
        s->n_hist = 0;
        for (int i = 0; i < len; i++) hist_push(s, t[i]);
        for (int j = 0; j < N; j++) {
            int t0 = t[2 * j], t1 = (2 * j + 1 < len) ? t[2 * j + 1] : ORC_PAD;
            orc_compress(c, &st->w, t0, t1, x);
            backbone_at(st, s, x);
            if (j < N - 1) {
                mtp_at(st, s, x, t[2 * j + 2], hd);
                s->n += 1;
            } else {
                heads_and_accept(st, b, x, tau, force, u ? u + 2 * b : NULL, o);
            }
        }
    }
    free(x); free(hd);
    return ORC_OK;
}

int orc_prefill(orc_state *st, const int32_t *ids, const int32_t *lens, int stride,
                double tau, int force, orc_out *o) {
    return orc_prefill_u(st, ids, lens, stride, tau, force, NULL, o);
}

/* Introspection for the tests: the token history of sequence b (the prompt,
 * then every emitted token); copies at most cap ids, returns the length. */
int orc_get_hist(const orc_state *st, int b, int32_t *out, int cap) {
    const orc_seq *s = &st->s[b];
    for (int i = 0; i < s->n_hist && i < cap; i++) out[i] = s->hist[i];
    return s->n_hist;
}

/* ------------------------------------------------------------------ */
/* regular decoding: the same backbone without pairs                  */
/*
 * The baseline the paper measures PIPO against (Sec. 4, "Regular"): one
 * token per backbone pass, the input is the token's embedding E[t] (no
 * compressor), the position is the token index and the cache holds one entry
 * per token; the final-norm tied LM head and greedy argmax give the next
 * token.  No MTP head, no confidence head.  Uses the backbone caches of the
 * state; the pending token is p0 (p1 unused), n counts the tokens consumed.
 */
static void regular_head(orc_state *st, int b, double *h, orc_out *o) {
    const orc_config *c = &st->c;
    orc_seq *s = &st->s[b];
    int H = c->H, V = c->V;
    double *lg = (double *)malloc(sizeof(double) * V);
    double m;
    lm_head(c, &st->w, h, st->w.final_norm, lg);
    int x = orc_argmax(lg, V, &m);
    hist_push(s, x);
    s->p0 = x;
    s->p1 = ORC_PAD;
    s->n += 1;
    s->emitted += 1;
    if (o) {
        if (o->tokens) { o->tokens[2 * b] = x; o->tokens[2 * b + 1] = -1; }
        if (o->n_acc) o->n_acc[b] = 0;
        if (o->logits_b) memcpy(o->logits_b + (size_t)b * V, lg, sizeof(double) * V);
        if (o->h_b) memcpy(o->h_b + (size_t)b * H, h, sizeof(double) * H);
        if (o->margin_b) o->margin_b[b] = m;
        if (o->x_b) o->x_b[b] = x;
    }
    free(lg);
}

/* Prefill of regular decoding: every prompt token runs the backbone at its
 * own position; the last one also runs the LM head, whose argmax becomes the
 * pending token. */
int orc_regular_prefill(orc_state *st, const int32_t *ids, const int32_t *lens, int stride, orc_out *o) {
    const orc_config *c = &st->c;
    for (int b = 0; b < st->B; b++) {
        int len = lens[b];
        if (len < 1 || len > stride) return ORC_EINVAL;
        if (len > c->max_ctx) return ORC_ECAPACITY;
        for (int t = 0; t < len; t++) if (ids[(size_t)b * stride + t] < 0 || ids[(size_t)b * stride + t] >= c->V) return ORC_EINVAL;
    }
    double *x = (double *)malloc(sizeof(double) * c->H);
    for (int b = 0; b < st->B; b++) {
        orc_seq *s = &st->s[b];
        const int32_t *t = ids + (size_t)b * stride;
        s->n = 0;
        s->emitted = 0;
        s->n_hist = 0;
        for (int j = 0; j < lens[b]; j++) hist_push(s, t[j]);
        for (int j = 0; j < lens[b]; j++) {
            embed(c, &st->w, t[j], x);
            backbone_at(st, s, x);
            if (j < lens[b] - 1) s->n += 1;
            else regular_head(st, b, x, o);
        }
        s->emitted = 0;  /* the prefill's token is the first output, not a decode step's */
    }
    free(x);
    return ORC_OK;
}

/* One regular decode step for every sequence: embed the pending token, one
 * backbone pass at position n, LM head, argmax. */
int orc_regular_step(orc_state *st, orc_out *o) {
    const orc_config *c = &st->c;
    for (int b = 0; b < st->B; b++) if (st->s[b].n >= c->max_ctx) return ORC_ECAPACITY;
    double *x = (double *)malloc(sizeof(double) * c->H);
    for (int b = 0; b < st->B; b++) {
        orc_seq *s = &st->s[b];
        embed(c, &st->w, s->p0, x);
        backbone_at(st, s, x);
        regular_head(st, b, x, o);
    }
    free(x);
    return ORC_OK;
}

/* Test hook: overwrite the pending pairs ([B,2], -1 = PAD in slot 1). */
int orc_set_pending(orc_state *st, const int32_t *pairs) {
    for (int b = 0; b < st->B; b++) {
        st->s[b].p0 = pairs[2 * b];
        st->s[b].p1 = pairs[2 * b + 1] < 0 ? ORC_PAD : pairs[2 * b + 1];
    }
    return ORC_OK;
}

/* Truncate both caches of each sequence to n[b] entries (n[b] <= current);
 * entries beyond are zeroed, so the state equals one that never appended. */
int orc_rollback(orc_state *st, const int32_t *n) {
    const orc_config *c = &st->c;
    size_t kd = (size_t)c->n_kv * c->d_h;
    int nl = c->L + (c->mtp_block ? 1 : 0);
    for (int b = 0; b < st->B; b++) if (n[b] < 0 || n[b] > st->s[b].n) return ORC_EINVAL;
    for (int b = 0; b < st->B; b++) {
        orc_seq *s = &st->s[b];
        for (int l = 0; l < nl; l++) {
            memset(s->K[l] + (size_t)n[b] * kd, 0, sizeof(double) * kd * (s->n - n[b]));
            memset(s->Vc[l] + (size_t)n[b] * kd, 0, sizeof(double) * kd * (s->n - n[b]));
        }
        s->n = n[b];
    }
    return ORC_OK;
}

/* Introspection for the tests: pending pair, n, emitted; cache rows. */
void orc_get_seq(const orc_state *st, int b, int32_t *p0, int32_t *p1, int32_t *n, int64_t *emitted) {
    *p0 = st->s[b].p0; *p1 = st->s[b].p1; *n = st->s[b].n; *emitted = st->s[b].emitted;
}
/* copies entries [0, n) of cache layer l of sequence b: [n][n_kv*d_h] */
void orc_get_cache(const orc_state *st, int b, int l, int n, double *K, double *V) {
    size_t kd = (size_t)st->c.n_kv * st->c.d_h;
    memcpy(K, st->s[b].K[l], sizeof(double) * kd * n);
    memcpy(V, st->s[b].Vc[l], sizeof(double) * kd * n);
}
/* Timing helper: load n entries of every cache layer of sequence b from
 * fp32 arrays [L+1][n][n_kv*d_h] and set the length to n. */
int orc_set_cache(orc_state *st, int b, int n, const float *K, const float *V) {
    const orc_config *c = &st->c;
    size_t kd = (size_t)c->n_kv * c->d_h;
    if (n > c->max_ctx) return ORC_ECAPACITY;
    int nl = c->L + (c->mtp_block ? 1 : 0);
    for (int l = 0; l < nl; l++)
        for (size_t i = 0; i < kd * n; i++) {
            st->s[b].K[l][i] = K[(size_t)l * n * kd + i];
            st->s[b].Vc[l][i] = V[(size_t)l * n * kd + i];
        }
    st->s[b].n = n;
    return ORC_OK;
}

/* ------------------------------------------------------------------ */
/* brute-force twin: no cache, whole sequence recomputed layer by layer  */

/* Given pairs P_0..P_n of one sequence ([n+1][2], -1 = PAD) and the tokens
 * fed to the MTP input at positions 0..n-1 (mtp_tok[n] is ignored: the last
 * position uses its own argmax), recompute everything from scratch with a
 * causal mask and return the results of the last position in slot 0 of o. */
int orc_bruteforce(const orc_config *c, const orc_weights *w, int n1, const int32_t *pairs,
                   const int32_t *mtp_tok, double tau, int force, orc_out *o) {
    int H = c->H, V = c->V, qd = c->n_q * c->d_h, kd = c->n_kv * c->d_h;
    double *X = (double *)malloc(sizeof(double) * (size_t)n1 * H);
    double *Q = (double *)malloc(sizeof(double) * (size_t)n1 * qd);
    double *K = (double *)malloc(sizeof(double) * (size_t)n1 * kd);
    double *Vv = (double *)malloc(sizeof(double) * (size_t)n1 * kd);
    double *A = (double *)malloc(sizeof(double) * qd);
    double *U = (double *)malloc(sizeof(double) * (size_t)n1 * H);
    for (int j = 0; j < n1; j++)
        orc_compress(c, w, pairs[2 * j], pairs[2 * j + 1] < 0 ? ORC_PAD : pairs[2 * j + 1], X + (size_t)j * H);
    int nblocks = c->L;
    for (int l = 0; l < nblocks; l++) {
        blockw bw = backbone_layer(w, l);
        for (int j = 0; j < n1; j++)
            block_qkv(c, bw, X + (size_t)j * H, j, Q + (size_t)j * qd, K + (size_t)j * kd, Vv + (size_t)j * kd);
        for (int j = 0; j < n1; j++) {
            orc_attend(Q + (size_t)j * qd, K, Vv, j + 1, c->n_q, c->n_kv, c->d_h, A);
            block_tail(c, bw, X + (size_t)j * H, A);
        }
    }
    double *hb = X + (size_t)(n1 - 1) * H;
    double *lb = (double *)malloc(sizeof(double) * V);
    double *ld = (double *)malloc(sizeof(double) * V);
    double mb, md;
    lm_head(c, w, hb, w->final_norm, lb);
    int xb = orc_argmax(lb, V, &mb);
    for (int j = 0; j < n1; j++)
        mtp_input(c, w, X + (size_t)j * H, j == n1 - 1 ? xb : mtp_tok[j], U + (size_t)j * H);
    if (c->mtp_block) {
        blockw bw = mtp_layer(w);
        for (int j = 0; j < n1; j++)
            block_qkv(c, bw, U + (size_t)j * H, j, Q + (size_t)j * qd, K + (size_t)j * kd, Vv + (size_t)j * kd);
        for (int j = 0; j < n1; j++) {
            orc_attend(Q + (size_t)j * qd, K, Vv, j + 1, c->n_q, c->n_kv, c->d_h, A);
            block_tail(c, bw, U + (size_t)j * H, A);
        }
    }
    double *hd = U + (size_t)(n1 - 1) * H;
    lm_head(c, w, hd, w->mtp_norm_post, ld);
    int xd = orc_argmax(ld, V, &md);
    double conf = orc_confidence(c, w, hb, hd);
    int acc = (force == 1) ? 1 : (force == 2) ? 0 : (conf >= tau);
    if (o->tokens) { o->tokens[0] = xb; o->tokens[1] = acc ? xd : -1; }
    if (o->n_acc) o->n_acc[0] = acc;
    if (o->logits_b) memcpy(o->logits_b, lb, sizeof(double) * V);
    if (o->logits_d) memcpy(o->logits_d, ld, sizeof(double) * V);
    if (o->conf) o->conf[0] = conf;
    if (o->h_b) memcpy(o->h_b, hb, sizeof(double) * H);
    if (o->h_d) memcpy(o->h_d, hd, sizeof(double) * H);
    if (o->margin_b) o->margin_b[0] = mb;
    if (o->margin_d) o->margin_d[0] = md;
    if (o->x_b) o->x_b[0] = xb;
    if (o->x_d) o->x_d[0] = xd;
    free(X); free(Q); free(K); free(Vv); free(A); free(U); free(lb); free(ld);
    return ORC_OK;
}
