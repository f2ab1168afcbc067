/*
 * KV-PRM verify-token scoring -- CPU ORACLE.  TEST INFRASTRUCTURE ONLY.
 *
 * Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline leg may
 * load this file's library.  The CUDA scoring library never links, calls or
 * falls back to it, and the two share no code.
 *
 * What it computes (one candidate trajectory b with a cached length L_b; all
 * arithmetic in IEEE double, sums taken in plain index order):
 *
 *   Scoring, Sec. 4.1 Eq. (score): one verify token v is forwarded through the
 *   scorer's N_L layers against the existing per-layer cache (K, V), and the
 *   reward is s = P(+) = softmax([z_-, z_+]) taken at the "+" entry, where z_-
 *   and z_+ are the logits of the judgment tokens (App. B.2).  Only those two
 *   rows of the output head are needed: P(+) = 1 / (1 + exp(z_- - z_+)).
 *
 *   The verify token is appended at the end of the sequence (Sec. 1), so it
 *   sits at position p = L_b and, like any causal decoder token, also attends
 *   to its own key/value (softmax over L_b + 1 entries).  Its own k/v are not
 *   written into the cache.
 *
 *   Attention read-out, App. A.3: head_i = softmax(q_i^T K / sqrt(d_k)) V.
 *   Grouped-query heads: query head h reads kv head floor(h / G), G = n_q/n_kv.
 *
 *   Per layer (pre-norm decoder block; the cost of Eq. (cost_kv) is this
 *   block's attention term c_attn*d*L plus its feed-forward term c_ffn*d^2):
 *     x   = RMSNorm(h) * g_attn                     eps = rms_eps
 *     q,k,v = W_qkv x                               rows: [q heads | k heads | v heads]
 *     q,k = RoPE(q, k; p = L_b)                     rotate-half pairs (i, i + hd/2),
 *                                                   angle p * base^(-2i/hd)
 *     o_h = softmax over {cache of b} U {self} of q_h.k_j / sqrt(hd), times v_j
 *     h  += W_o o
 *     x   = RMSNorm(h) * g_mlp
 *     h  += W_down (SiLU(W_gate x) * (W_up x))      W_gate_up rows: [gate | up]
 *   then x = RMSNorm(h) * g_final, z_+ = w_plus . x, z_- = w_minus . x.
 *
 *   Depth-k readout (Sec. 3, definition of R_k; Sec. 5 "more verify tokens"): with
 *   depth = k > 1, k verify tokens follow the trajectory at positions
 *   L_b .. L_b + k - 1 and run causally among themselves: token t attends to the
 *   cache and to tokens 0 .. t; the reward is read at the last one.  Internally
 *   candidate b is k rows b k + t.
 *
 *   Per-head q/k norm (reading of the paper's Qwen3 scorers, Sec. 5 "Setup"):
 *   with qk_norm set, each query head's and each key head's projection is
 *   RMS-normalised over its head_dim entries, with that layer's gain vector
 *   g_q or g_k [head_dim] (shared by all heads) and the same eps, before RoPE.
 *
 *   Scorer adapter, Sec. 4.1 (f_{theta + Delta theta}, a LoRA adapter) and App.
 *   B.1 (rank r = 256, alpha = 32): when lora_rank > 0 each of the four
 *   projections y = W x above becomes y = W x + s B (A x) with its own factors
 *   A [r][in] and B [out][r] and s = lora_scale (alpha / r); A x is a
 *   projection input like x (rounded to bf16 in mirror mode).  With
 *   lora_rank = 0 the weights are the merged scorer's.
 *
 * Precision.  The paper trains and serves in bf16 (App. B.1), so weights and
 * cached K/V are bf16 values.  "exact" mode (mirror = 0) computes everything
 * else exactly (double) on those bf16 inputs; it is the reference the CUDA
 * library is compared with.  "mirror" mode (mirror = 1) additionally rounds to
 * bf16 (nearest, ties to even) every activation a bf16 inference stack would
 * round: each projection input (x after each norm, the attention output o,
 * the SiLU(gate)*up product, the final x), the rotated q and the self k/v.  It
 * measures how far such a stack drifts from the exact value; it is not used
 * as a reference because two correct bf16 stacks that round from different
 * intermediate precisions disagree by whole bf16 ulps, and those differences
 * compound from layer to layer.
 *
 * Inputs arrive through provider callbacks (weights one matrix at a time, the
 * logical per-candidate K/V one layer at a time), so full-size workloads need
 * no host copy of the whole model or cache.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* weight kinds, as asked of the weight provider */
enum { K_EMBED = 0, K_FINAL_NORM, K_W_PLUS, K_W_MINUS, K_ATTN_NORM, K_W_QKV, K_W_O, K_MLP_NORM, K_W_GATE_UP, K_W_DOWN,
       K_LORA_A_QKV, K_LORA_B_QKV, K_LORA_A_O, K_LORA_B_O, K_LORA_A_GATE_UP, K_LORA_B_GATE_UP, K_LORA_A_DOWN,
       K_LORA_B_DOWN, K_Q_NORM, K_K_NORM };

typedef int (*oracle_weight_fn)(void* user, int kind, int layer, uint16_t* out, int64_t n);
typedef int (*oracle_kv_fn)(void* user, int layer, int cand, uint16_t* K, uint16_t* V, int64_t L);

typedef struct {
    int n_layers, d_model, n_q_heads, n_kv_heads, head_dim, d_ff;
    double rope_base, rms_eps;
    int mirror;   /* 1: bf16 rounding at the precision contract's points; 0: exact */
    int nthreads;
    int lora_rank;       /* 0: no adapter */
    double lora_scale;   /* s in y = W x + s B (A x) */
    int depth;           /* verify tokens per candidate (depth-k readout); 0 or 1: one */
    int qk_norm;         /* 1: per-head RMSNorm of q and k before RoPE (gains K_Q_NORM, K_K_NORM) */
} oracle_cfg;

/* ------------------------------------------------------------------ numbers */
static inline double bf16_to_f64(uint16_t b) {
    uint32_t u = (uint32_t)b << 16;
    float f;
    memcpy(&f, &u, 4);
    return (double)f;
}

/* Round a double to the nearest bf16 value (ties to even): 8 significant bits,
 * exponent range of IEEE binary32, subnormal quantum 2^-133. */
double oracle_bf16_round(double x) {
    if (x == 0.0 || !isfinite(x)) return x;
    int e;
    frexp(x, &e);                       /* x = m * 2^e, 0.5 <= |m| < 1 */
    int qe = e - 8;
    if (qe < -133) qe = -133;
    double r = ldexp(nearbyint(ldexp(x, -qe)), qe);
    if (fabs(r) >= 0x1p128) return copysign(INFINITY, x);
    return r;
}

static inline double rnd(const oracle_cfg* c, double x) { return c->mirror ? oracle_bf16_round(x) : x; }

/* ------------------------------------------------------------ parallel for */
typedef void (*idx_fn)(void* ctx, int64_t i);
typedef struct { idx_fn fn; void* ctx; int64_t n; int t, nt; } pf_job;
static void* pf_run(void* p) {
    pf_job* j = (pf_job*)p;
    for (int64_t i = j->t; i < j->n; i += j->nt) j->fn(j->ctx, i);
    return NULL;
}
static void par_for(int64_t n, int nthreads, idx_fn fn, void* ctx) {
    if (nthreads > 128) nthreads = 128;
    if (nthreads <= 1 || n <= 1) {
        for (int64_t i = 0; i < n; ++i) fn(ctx, i);
        return;
    }
    if (nthreads > n) nthreads = (int)n;
    pthread_t th[128];
    pf_job jobs[128];
    int ok[128];
    for (int t = 0; t < nthreads; ++t) {
        jobs[t] = (pf_job){ fn, ctx, n, t, nthreads };
        ok[t] = pthread_create(&th[t], NULL, pf_run, &jobs[t]) == 0;
        if (!ok[t]) pf_run(&jobs[t]);
    }
    for (int t = 0; t < nthreads; ++t)
        if (ok[t]) pthread_join(th[t], NULL);
}

/* --------------------------------------------------------------- primitives */

/* RMSNorm: out = h / sqrt(mean(h^2) + eps) * g. */
void oracle_rmsnorm(const double* h, const uint16_t* g, int d, double eps, double* out) {
    double ss = 0.0;
    for (int i = 0; i < d; ++i) ss += h[i] * h[i];
    double r = 1.0 / sqrt(ss / d + eps);
    for (int i = 0; i < d; ++i) out[i] = h[i] * r * bf16_to_f64(g[i]);
}

/* Rotary embedding, rotate-half convention: for i < hd/2 the pair
 * (x_i, x_{i+hd/2}) is rotated by the angle pos * base^(-2i/hd). */
void oracle_rope(double* x, int hd, double pos, double base) {
    int half = hd / 2;
    for (int i = 0; i < half; ++i) {
        double ang = pos * pow(base, -2.0 * i / hd);
        double c = cos(ang), s = sin(ang);
        double a = x[i], b = x[i + half];
        x[i] = a * c - b * s;
        x[i + half] = b * c + a * s;
    }
}

/* Attention read-out of one query head (App. A.3) over the L cached entries and
 * n_self verify-token entries (their own keys/values, the last one being the
 * token's own; one entry except in a depth-k readout):
 *   s_j = q . K_j / sqrt(hd) for j < L,   s_{L+t} = q . k_self[t] / sqrt(hd)
 *   w = softmax(s),  o = sum_j w_j V_j + sum_t w_{L+t} v_self[t].
 * K and V are bf16 rows with `stride` elements between consecutive tokens;
 * self entry t starts at k_self + t * self_stride (likewise v_self).  If
 * `weights` is non-NULL it receives the L + n_self softmax weights. */
void oracle_attend_multi(const double* q, const uint16_t* K, const uint16_t* V, int64_t L, int64_t stride,
                         const double* k_self, const double* v_self, int64_t self_stride, int n_self, int hd,
                         double* o, double* weights) {
    double scale = 1.0 / sqrt((double)hd);
    const int64_t N = L + n_self;
    double* s = (double*)malloc(sizeof(double) * (size_t)N);
    for (int64_t j = 0; j < L; ++j) {
        double acc = 0.0;
        for (int d = 0; d < hd; ++d) acc += q[d] * bf16_to_f64(K[j * stride + d]);
        s[j] = acc * scale;
    }
    for (int t = 0; t < n_self; ++t) {
        double acc = 0.0;
        for (int d = 0; d < hd; ++d) acc += q[d] * k_self[t * self_stride + d];
        s[L + t] = acc * scale;
    }
#if ORACLE_MUTANT == 1 /* planted mistake: the verify token ignores itself */
    if (L > 0) s[N - 1] = -INFINITY;
#endif
    double m = s[0];
    for (int64_t j = 1; j < N; ++j)
        if (s[j] > m) m = s[j];
    double l = 0.0;
    for (int64_t j = 0; j < N; ++j) {
        s[j] = exp(s[j] - m);
        l += s[j];
    }
    for (int d = 0; d < hd; ++d) o[d] = 0.0;
    for (int64_t j = 0; j < L; ++j) {
        double w = s[j] / l;
        for (int d = 0; d < hd; ++d) o[d] += w * bf16_to_f64(V[j * stride + d]);
    }
    for (int t = 0; t < n_self; ++t) {
        double w = s[L + t] / l;
        for (int d = 0; d < hd; ++d) o[d] += w * v_self[t * self_stride + d];
    }
    if (weights)
        for (int64_t j = 0; j < N; ++j) weights[j] = s[j] / l;
    free(s);
}

/* The single-verify-token read-out: the token's own key/value as the last entry. */
void oracle_attend(const double* q, const uint16_t* K, const uint16_t* V, int64_t L, int64_t stride,
                   const double* k_self, const double* v_self, int hd, double* o, double* weights) {
    oracle_attend_multi(q, K, V, L, stride, k_self, v_self, 0, 1, hd, o, weights);
}

/* Reward head (Eq. score): P(+) = softmax([z_-, z_+]) at "+" = 1/(1+exp(z_- - z_+)). */
double oracle_reward(const double* x, const uint16_t* w_plus, const uint16_t* w_minus, int d) {
    double zp = 0.0, zm = 0.0;
    for (int i = 0; i < d; ++i) {
        zp += bf16_to_f64(w_plus[i]) * x[i];
        zm += bf16_to_f64(w_minus[i]) * x[i];
    }
#if ORACLE_MUTANT == 7 /* planted mistake: the "-" entry is read as P(+) */
    return 1.0 / (1.0 + exp(zp - zm));
#else
    return 1.0 / (1.0 + exp(zm - zp));
#endif
}

/* ------------------------------------------------------------- projections */
/* y[i][r] (+)= sum_c W[r][c] * x[i][c] for n candidates; W is bf16 [rows][cols]. */
typedef struct {
    const uint16_t* W; int rows, cols; const double* x; double* y; int n; int accumulate; int transposed;
} proj_ctx;
static void proj_row(void* p, int64_t r) {
    const proj_ctx* c = (const proj_ctx*)p;
    for (int i = 0; i < c->n; ++i) {
        const double* xi = c->x + (int64_t)i * c->cols;
        double acc = 0.0;
        for (int k = 0; k < c->cols; ++k) {
            int64_t idx = c->transposed ? (int64_t)k * c->rows + r : r * (int64_t)c->cols + k;
            acc += bf16_to_f64(c->W[idx]) * xi[k];
        }
        double* yi = c->y + (int64_t)i * c->rows + r;
        *yi = c->accumulate ? *yi + acc : acc;
    }
}
static void project(const oracle_cfg* cfg, const uint16_t* W, int rows, int cols, const double* x, double* y, int n,
                    int accumulate, int transposed) {
    proj_ctx c = { W, rows, cols, x, y, n, accumulate, transposed };
    par_for(rows, cfg->nthreads, proj_row, &c);
}

/* The adapter term of one projection: y[i][r] += s * sum_j B[r][j] t[i][j], t = A x (t and tmp are
 * scratch of n * lora_rank and n * rows doubles). */
static void lora_add(const oracle_cfg* cfg, const uint16_t* A, const uint16_t* B, int rows, int cols,
                     const double* x, double* y, int n, double* t, double* tmp) {
    const int r = cfg->lora_rank;
    project(cfg, A, r, cols, x, t, n, 0, 0);
    for (int64_t e = 0; e < (int64_t)n * r; ++e) t[e] = rnd(cfg, t[e]);
    project(cfg, B, rows, r, t, tmp, n, 0, 0);
#if ORACLE_MUTANT == 15 /* planted mistake: adapter scale left out */
    const double s = 1.0;
#else
    const double s = cfg->lora_scale;
#endif
    for (int64_t e = 0; e < (int64_t)n * rows; ++e)
#if ORACLE_MUTANT == 16 /* planted mistake: adapter term subtracted */
        y[e] -= s * tmp[e];
#else
        y[e] += s * tmp[e];
#endif
}

/* ------------------------------------------------------------- attention */
typedef struct {
    const oracle_cfg* cfg;
    const double* q;        /* [rows][nq][hd]   rotated (and rounded in mirror mode) */
    const double* kself;    /* [rows][nkv][hd] */
    const double* vself;    /* [rows][nkv][hd] */
    uint16_t* const* K;     /* per candidate [L][nkv][hd] */
    uint16_t* const* V;
    const int64_t* lens;    /* per candidate */
    int depth;              /* rows per candidate (verify tokens) */
    double* o;              /* [rows][nq][hd] */
} attn_ctx;
static void attn_item(void* p, int64_t it) {
    const attn_ctx* c = (const attn_ctx*)p;
    const oracle_cfg* cfg = c->cfg;
    int nq = cfg->n_q_heads, nkv = cfg->n_kv_heads, hd = cfg->head_dim, G = nq / nkv;
    int row = (int)(it / nq), h = (int)(it % nq);
    int i = row / c->depth, t = row % c->depth;   /* candidate, verify token */
#if ORACLE_MUTANT == 3 /* planted mistake: interleaved instead of contiguous head groups */
    int g = h % nkv;
#elif ORACLE_MUTANT == 12 /* planted mistake: every query head reads kv head 0 */
    int g = 0;
    (void)G;
#else
    int g = h / G;
#endif
    const double* q = c->q + ((int64_t)row * nq + h) * hd;
    double qs[1024];
#if ORACLE_MUTANT == 4 /* planted mistake: scores not divided by sqrt(hd) */
    for (int d = 0; d < hd; ++d) qs[d] = q[d] * sqrt((double)hd);
#else
    for (int d = 0; d < hd; ++d) qs[d] = q[d];
#endif
    /* token t sees the candidate's verify tokens 0 .. t (causal) */
    const int64_t first = (int64_t)i * c->depth;
#if ORACLE_MUTANT == 17 /* planted mistake: every verify token also sees the ones after it */
    const int n_self = c->depth;
    (void)t;
#else
    const int n_self = t + 1;
#endif
    oracle_attend_multi(qs, c->K[i] + (int64_t)g * hd, c->V[i] + (int64_t)g * hd, c->lens[i], (int64_t)nkv * hd,
                        c->kself + (first * nkv + g) * hd, c->vself + (first * nkv + g) * hd, (int64_t)nkv * hd,
                        n_self, hd, c->o + ((int64_t)row * nq + h) * hd, NULL);
}

/* ------------------------------------------------------------------ scorer */
/*
 * Score n candidates.  cand_ids[i] is passed to the kv provider; lens[i] is its
 * cached length L.  With depth D > 1 the per-row outputs below have n D rows
 * (candidate i's tokens are rows i D .. i D + D - 1) and h_out is each
 * candidate's last row.  Outputs: p_plus[n]; if non-NULL, attn_out[N_L][n][nq*hd]
 * (each layer's attention output o before rounding), h_out[n][d] (final
 * residual stream), qkv_out[N_L][n][(nq+2nkv)*hd] (each layer's rotated q,
 * self k and self v as the attention consumes them) and
 * h_layers_out[N_L][n][d] (residual stream after each layer).  Returns 0, or a negative code when a provider fails or
 * memory runs out.
 */
int oracle_score(const oracle_cfg* cfg, oracle_weight_fn wfn, void* wuser, oracle_kv_fn kvfn, void* kvuser, int n,
                 const int32_t* cand_ids, const int64_t* lens, double* p_plus, double* attn_out, double* h_out,
                 double* qkv_out, double* h_layers_out) {
    const int NL = cfg->n_layers, d = cfg->d_model, nq = cfg->n_q_heads, nkv = cfg->n_kv_heads, hd = cfg->head_dim;
    const int ff = cfg->d_ff, qkv_rows = (nq + 2 * nkv) * hd;
    if (hd > 1024 || hd % 2 || nq % nkv) return -1;
    int rc = 0;
    /* rows: candidate i's verify tokens are rows i D .. i D + D - 1 (one row each without depth-k) */
    const int D = cfg->depth > 1 ? cfg->depth : 1;
    const int nr = n * D;
    uint16_t *embed = malloc(2 * (size_t)d), *gfin = malloc(2 * (size_t)d), *wp = malloc(2 * (size_t)d),
             *wm = malloc(2 * (size_t)d), *gattn = malloc(2 * (size_t)d), *gmlp = malloc(2 * (size_t)d);
    uint16_t *Wqkv = malloc(2 * (size_t)qkv_rows * d), *Wo = malloc(2 * (size_t)d * nq * hd),
             *Wgu = malloc(2 * (size_t)2 * ff * d), *Wd = malloc(2 * (size_t)d * ff);
    double *h = calloc((size_t)nr * d, 8), *x = calloc((size_t)nr * d, 8), *qkv = calloc((size_t)nr * qkv_rows, 8);
    double *q = calloc((size_t)nr * nq * hd, 8), *ks = calloc((size_t)nr * nkv * hd, 8),
           *vs = calloc((size_t)nr * nkv * hd, 8), *o = calloc((size_t)nr * nq * hd, 8);
    double *gu = calloc((size_t)nr * 2 * ff, 8), *a = calloc((size_t)nr * ff, 8);
    uint16_t** K = calloc((size_t)n, sizeof(uint16_t*));
    uint16_t** V = calloc((size_t)n, sizeof(uint16_t*));
    uint16_t *gq = malloc(2 * (size_t)hd), *gk = malloc(2 * (size_t)hd);   /* q/k norm gains */
    /* adapter factors of the four projections (A [r][in], B [out][r]) and scratch */
    const int r = cfg->lora_rank;
    const int64_t in_of[4] = { d, (int64_t)nq * hd, d, ff }, out_of[4] = { qkv_rows, d, 2 * (int64_t)ff, d };
    uint16_t* LA[4] = { NULL, NULL, NULL, NULL };
    uint16_t* LB[4] = { NULL, NULL, NULL, NULL };
    double *lt = NULL, *ltmp = NULL;
    if (r < 0) { rc = -1; goto done; }
    if (r > 0) {
        int64_t most = qkv_rows > 2 * (int64_t)ff ? qkv_rows : 2 * (int64_t)ff;
        if (d > most) most = d;
        for (int j = 0; j < 4; ++j) {
            LA[j] = malloc(2 * (size_t)r * in_of[j]);
            LB[j] = malloc(2 * (size_t)out_of[j] * r);
            if (!LA[j] || !LB[j]) { rc = -2; goto done; }
        }
        lt = calloc((size_t)nr * r, 8);
        ltmp = calloc((size_t)nr * most, 8);
        if (!lt || !ltmp) { rc = -2; goto done; }
    }
    if (!embed || !gfin || !wp || !wm || !gattn || !gmlp || !Wqkv || !Wo || !Wgu || !Wd || !h || !x || !qkv || !q ||
        !ks || !vs || !o || !gu || !a || !K || !V || !gq || !gk) {
        rc = -2;
        goto done;
    }
    for (int i = 0; i < n; ++i) {
        size_t sz = 2 * (size_t)(lens[i] > 0 ? lens[i] : 1) * nkv * hd;
        K[i] = malloc(sz);
        V[i] = malloc(sz);
        if (!K[i] || !V[i]) { rc = -2; goto done; }
    }
    if (wfn(wuser, K_EMBED, 0, embed, d) || wfn(wuser, K_FINAL_NORM, 0, gfin, d) || wfn(wuser, K_W_PLUS, 0, wp, d) ||
        wfn(wuser, K_W_MINUS, 0, wm, d)) { rc = -3; goto done; }

    /* the verify token's embedding starts every row's residual stream */
    for (int i = 0; i < nr; ++i)
        for (int c = 0; c < d; ++c) h[(int64_t)i * d + c] = bf16_to_f64(embed[c]);

    for (int l = 0; l < NL; ++l) {
        if (wfn(wuser, K_ATTN_NORM, l, gattn, d) || wfn(wuser, K_W_QKV, l, Wqkv, (int64_t)qkv_rows * d) ||
            wfn(wuser, K_W_O, l, Wo, (int64_t)d * nq * hd) || wfn(wuser, K_MLP_NORM, l, gmlp, d) ||
            wfn(wuser, K_W_GATE_UP, l, Wgu, (int64_t)2 * ff * d) || wfn(wuser, K_W_DOWN, l, Wd, (int64_t)d * ff)) {
            rc = -3;
            goto done;
        }
        if (cfg->qk_norm && (wfn(wuser, K_Q_NORM, l, gq, hd) || wfn(wuser, K_K_NORM, l, gk, hd))) {
            rc = -3;
            goto done;
        }
        for (int j = 0; j < 4 && r > 0; ++j)
            if (wfn(wuser, K_LORA_A_QKV + 2 * j, l, LA[j], (int64_t)r * in_of[j]) ||
                wfn(wuser, K_LORA_B_QKV + 2 * j, l, LB[j], out_of[j] * r)) {
                rc = -3;
                goto done;
            }
        for (int i = 0; i < n; ++i)
            if (lens[i] > 0 && kvfn(kvuser, l, cand_ids[i], K[i], V[i], lens[i])) { rc = -4; goto done; }

        /* attention block */
        for (int i = 0; i < nr; ++i) {
            double* xi = x + (int64_t)i * d;
#if ORACLE_MUTANT == 9 /* planted mistake: eps left out of the norm */
            oracle_rmsnorm(h + (int64_t)i * d, gattn, d, 0.0, xi);
#else
            oracle_rmsnorm(h + (int64_t)i * d, gattn, d, cfg->rms_eps, xi);
#endif
            for (int c = 0; c < d; ++c) xi[c] = rnd(cfg, xi[c]);
        }
        project(cfg, Wqkv, qkv_rows, d, x, qkv, nr, 0, 0);
        if (r > 0) lora_add(cfg, LA[0], LB[0], qkv_rows, d, x, qkv, nr, lt, ltmp);
        for (int i = 0; i < nr; ++i) {
            const double* qr = qkv + (int64_t)i * qkv_rows;
            /* verify token t of candidate i / D sits at position L + t */
#if ORACLE_MUTANT == 8 /* planted mistake: verify token placed on the last cached position */
            double pos = (double)lens[i / D] - 1.0 + (double)(i % D);
#else
            double pos = (double)lens[i / D] + (double)(i % D);
#endif
            for (int hh = 0; hh < nq; ++hh) {
                double* qh = q + ((int64_t)i * nq + hh) * hd;
                memcpy(qh, qr + (int64_t)hh * hd, 8 * (size_t)hd);
#if ORACLE_MUTANT == 18 /* planted mistake: q/k norm applied after RoPE */
                oracle_rope(qh, hd, pos, cfg->rope_base);
                if (cfg->qk_norm) oracle_rmsnorm(qh, gq, hd, cfg->rms_eps, qh);
#else
                if (cfg->qk_norm) oracle_rmsnorm(qh, gq, hd, cfg->rms_eps, qh);
#if ORACLE_MUTANT == 2 /* planted mistake: rotation in the wrong direction */
                oracle_rope(qh, hd, -pos, cfg->rope_base);
#else
                oracle_rope(qh, hd, pos, cfg->rope_base);
#endif
#endif
                for (int c = 0; c < hd; ++c) qh[c] = rnd(cfg, qh[c]);
            }
            for (int g = 0; g < nkv; ++g) {
                double* kh = ks + ((int64_t)i * nkv + g) * hd;
                double* vh = vs + ((int64_t)i * nkv + g) * hd;
                memcpy(kh, qr + (int64_t)(nq + g) * hd, 8 * (size_t)hd);
                memcpy(vh, qr + (int64_t)(nq + nkv + g) * hd, 8 * (size_t)hd);
#if ORACLE_MUTANT == 19 /* planted mistake: the key norm takes the query norm's gain */
                if (cfg->qk_norm) oracle_rmsnorm(kh, gq, hd, cfg->rms_eps, kh);
#elif ORACLE_MUTANT == 18
                (void)0;
#else
                if (cfg->qk_norm) oracle_rmsnorm(kh, gk, hd, cfg->rms_eps, kh);
#endif
                oracle_rope(kh, hd, pos, cfg->rope_base);
#if ORACLE_MUTANT == 18
                if (cfg->qk_norm) oracle_rmsnorm(kh, gk, hd, cfg->rms_eps, kh);
#endif
                for (int c = 0; c < hd; ++c) {
                    kh[c] = rnd(cfg, kh[c]);
                    vh[c] = rnd(cfg, vh[c]);
                }
            }
        }
        if (qkv_out)
            for (int i = 0; i < nr; ++i) {
                double* dst = qkv_out + ((int64_t)l * nr + i) * qkv_rows;
                memcpy(dst, q + (int64_t)i * nq * hd, 8 * (size_t)nq * hd);
                memcpy(dst + (int64_t)nq * hd, ks + (int64_t)i * nkv * hd, 8 * (size_t)nkv * hd);
                memcpy(dst + (int64_t)(nq + nkv) * hd, vs + (int64_t)i * nkv * hd, 8 * (size_t)nkv * hd);
            }
        attn_ctx ac = { cfg, q, ks, vs, K, V, lens, D, o };
        par_for((int64_t)nr * nq, cfg->nthreads, attn_item, &ac);
        if (attn_out) memcpy(attn_out + (int64_t)l * nr * nq * hd, o, 8 * (size_t)nr * nq * hd);
        for (int64_t e = 0; e < (int64_t)nr * nq * hd; ++e) o[e] = rnd(cfg, o[e]);
#if ORACLE_MUTANT == 5 /* planted mistake: output projection applied transposed */
        project(cfg, Wo, d, nq * hd, o, h, nr, 1, 1);
#else
        project(cfg, Wo, d, nq * hd, o, h, nr, 1, 0);
#endif
        if (r > 0) lora_add(cfg, LA[1], LB[1], d, nq * hd, o, h, nr, lt, ltmp);

        /* feed-forward block */
        for (int i = 0; i < nr; ++i) {
            double* xi = x + (int64_t)i * d;
            oracle_rmsnorm(h + (int64_t)i * d, gmlp, d, cfg->rms_eps, xi);
            for (int c = 0; c < d; ++c) xi[c] = rnd(cfg, xi[c]);
        }
        project(cfg, Wgu, 2 * ff, d, x, gu, nr, 0, 0);
        if (r > 0) lora_add(cfg, LA[2], LB[2], 2 * ff, d, x, gu, nr, lt, ltmp);
        for (int i = 0; i < nr; ++i)
            for (int j = 0; j < ff; ++j) {
                double gt = gu[(int64_t)i * 2 * ff + j], up = gu[(int64_t)i * 2 * ff + ff + j];
#if ORACLE_MUTANT == 10 /* planted mistake: gate not passed through SiLU */
                double act = gt * up;
#elif ORACLE_MUTANT == 14 /* planted mistake: gate and up exchanged */
                double act = up / (1.0 + exp(-up)) * gt;
#else
                double act = gt / (1.0 + exp(-gt)) * up;
#endif
                a[(int64_t)i * ff + j] = rnd(cfg, act);
            }
#if ORACLE_MUTANT == 6 /* planted mistake: feed-forward output replaces the residual stream */
        project(cfg, Wd, d, ff, a, h, nr, 0, 0);
#else
        project(cfg, Wd, d, ff, a, h, nr, 1, 0);
#endif
        if (r > 0) lora_add(cfg, LA[3], LB[3], d, ff, a, h, nr, lt, ltmp);
        if (h_layers_out) memcpy(h_layers_out + (int64_t)l * nr * d, h, 8 * (size_t)nr * d);
    }

    /* reward head on the final-normed stream of each candidate's last verify token */
    for (int i = 0; i < n; ++i) {
        const int64_t row = (int64_t)i * D + D - 1;
        double* xi = x + row * d;
        oracle_rmsnorm(h + row * d, gfin, d, cfg->rms_eps, xi);
        for (int c = 0; c < d; ++c) xi[c] = rnd(cfg, xi[c]);
        p_plus[i] = oracle_reward(xi, wp, wm, d);
        if (h_out) memcpy(h_out + (int64_t)i * d, h + row * d, 8 * (size_t)d);
    }

done:
    if (K)
        for (int i = 0; i < n; ++i) free(K[i]);
    if (V)
        for (int i = 0; i < n; ++i) free(V[i]);
    free(K); free(V);
    free(gq); free(gk);
    free(embed); free(gfin); free(wp); free(wm); free(gattn); free(gmlp);
    free(Wqkv); free(Wo); free(Wgu); free(Wd);
    for (int j = 0; j < 4; ++j) { free(LA[j]); free(LB[j]); }
    free(lt); free(ltmp);
    free(h); free(x); free(qkv); free(q); free(ks); free(vs); free(o); free(gu); free(a);
    return rc;
}

/* ----------------------------------------------- dense in-memory providers */
/* Weights held in caller arrays: top[kind] for kinds 0..3, layer[kind-4][l] otherwise. */
typedef struct {
    const uint16_t* top[4];
    const uint16_t* const* layer[16];   /* kinds 4 .. 19 (adapter factors and q/k norm gains may be NULL when unused) */
} oracle_dense_weights;

int oracle_dense_weight_provider(void* user, int kind, int layer, uint16_t* out, int64_t n) {
    const oracle_dense_weights* w = (const oracle_dense_weights*)user;
    if (kind < 0 || kind > K_K_NORM) return -1;
    if (kind >= 4 && !w->layer[kind - 4]) return -1;
    const uint16_t* src = kind < 4 ? w->top[kind] : w->layer[kind - 4][layer];
    if (!src) return -1;
    memcpy(out, src, 2 * (size_t)n);
    return 0;
}

/* Logical K/V held in caller arrays: K[l * n_cand + cand] -> [L][nkv][hd]. */
typedef struct {
    int n_cand;
    int64_t per_token;              /* nkv * hd */
    const uint16_t* const* K;
    const uint16_t* const* V;
    const int64_t* lens;
} oracle_dense_kv;

int oracle_dense_kv_provider(void* user, int layer, int cand, uint16_t* K, uint16_t* V, int64_t L) {
    const oracle_dense_kv* c = (const oracle_dense_kv*)user;
    if (cand < 0 || cand >= c->n_cand || c->lens[cand] != L) return -1;
    int64_t slot = (int64_t)layer * c->n_cand + cand;
    memcpy(K, c->K[slot], 2 * (size_t)(L * c->per_token));
    memcpy(V, c->V[slot], 2 * (size_t)(L * c->per_token));
    return 0;
}
