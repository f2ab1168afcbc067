/*
 * kvsynth host generator: seeded synthetic inputs for KV-PRM scoring.
 *
 * Every value is a bf16 bit pattern looked up in a 65,536-entry quantile
 * table with the top 16 bits of one SplitMix64 output (Steele, Lea & Flood,
 * "Fast splittable pseudorandom number generators", OOPSLA 2014):
 *     key(seed, tid)  = mix64(seed ^ tid * GAMMA)
 *     draw(key, n)    = mix64(key + (n + 1) * GAMMA)      (n-th stream output)
 *     value           = table[draw >> 48]
 * The element index n of a cached key/value is derived from the token's
 * logical identity (segment, offset), never from the physical page it lands
 * in, so a paged pool and a logical (unpaged) view of the same cache hold the
 * same bits.  The device twin of this file is synth_fill.cu; both follow the
 * same published definition and are checked bit-for-bit against each other.
 *
 * This module holds none of the scoring method's arithmetic.  It also
 * provides the weight and key/value provider callbacks that the oracle
 * consumes through function pointers.
 */
#include <stdint.h>
#include <stddef.h>
#include <string.h>
#include <pthread.h>

#define GAMMA 0x9E3779B97F4A7C15ULL

static inline uint64_t mix64(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}
static inline uint64_t stream_key(uint64_t seed, uint64_t tid) { return mix64(seed ^ (tid * GAMMA)); }
static inline uint64_t draw(uint64_t key, uint64_t n) { return mix64(key + (n + 1) * GAMMA); }

/* Tensor ids.  Weights: ((kind + 1) << 16) | layer.  Cached K/V of layer l:
 * KV_TID_BASE + 2*l + (0 for K, 1 for V). */
#define KV_TID_BASE 0x4B560000ULL
uint64_t synth_weight_tid(int kind, int layer) { return ((uint64_t)(kind + 1) << 16) | (uint64_t)layer; }
uint64_t synth_kv_tid(int layer, int is_v) { return KV_TID_BASE + 2ULL * (uint64_t)layer + (uint64_t)is_v; }

/* Element index of cached K/V value (segment, offset, kv head, dim). */
static inline uint64_t kv_index(int32_t seg, int32_t off, int head, int dim, int n_kv, int hd) {
    uint64_t tok = ((uint64_t)(uint32_t)seg << 24) | (uint64_t)(uint32_t)off;
    return (tok * (uint64_t)n_kv + (uint64_t)head) * (uint64_t)hd + (uint64_t)dim;
}

/* ---- tiny parallel-for over [0, n) ---------------------------------------- */
typedef void (*range_fn)(void* ctx, int64_t lo, int64_t hi);
typedef struct { range_fn fn; void* ctx; int64_t lo, hi; } range_job;
static void* range_run(void* p) { range_job* j = (range_job*)p; j->fn(j->ctx, j->lo, j->hi); return NULL; }
static void par_range(int64_t n, int nthreads, range_fn fn, void* ctx) {
    if (nthreads < 1) nthreads = 1;
    if (nthreads > 64) nthreads = 64;
    if (n < 65536 || nthreads == 1) { fn(ctx, 0, n); return; }
    pthread_t th[64]; range_job jobs[64]; int started[64];
    for (int t = 0; t < nthreads; ++t) {
        jobs[t].fn = fn; jobs[t].ctx = ctx;
        jobs[t].lo = n * t / nthreads; jobs[t].hi = n * (t + 1) / nthreads;
        started[t] = pthread_create(&th[t], NULL, range_run, &jobs[t]) == 0;
        if (!started[t]) range_run(&jobs[t]);
    }
    for (int t = 0; t < nthreads; ++t) if (started[t]) pthread_join(th[t], NULL);
}

/* ---- flat tensor fill ---------------------------------------------------- */
typedef struct { uint16_t* out; uint64_t key; const uint16_t* table; } fill_ctx;
static void fill_range(void* p, int64_t lo, int64_t hi) {
    fill_ctx* c = (fill_ctx*)p;
    for (int64_t i = lo; i < hi; ++i) c->out[i] = c->table[draw(c->key, (uint64_t)i) >> 48];
}
/* out[i] = table[draw(key(seed, tid), i) >> 48] for i in [0, n). */
void synth_fill(uint16_t* out, int64_t n, uint64_t seed, uint64_t tid, const uint16_t* table, int nthreads) {
    fill_ctx c = { out, stream_key(seed, tid), table };
    par_range(n, nthreads, fill_range, &c);
}

/* ---- logical K/V of one sequence: [L][n_kv][hd] for K and for V ------------ */
typedef struct {
    uint16_t *K, *V; const int32_t *seg, *off; int n_kv, hd; uint64_t kk, kv; const uint16_t* table;
} kvlog_ctx;
static void kvlog_range(void* p, int64_t lo, int64_t hi) {
    kvlog_ctx* c = (kvlog_ctx*)p;
    for (int64_t t = lo; t < hi; ++t)
        for (int h = 0; h < c->n_kv; ++h)
            for (int d = 0; d < c->hd; ++d) {
                uint64_t n = kv_index(c->seg[t], c->off[t], h, d, c->n_kv, c->hd);
                int64_t o = (t * c->n_kv + h) * (int64_t)c->hd + d;
                if (c->K) c->K[o] = c->table[draw(c->kk, n) >> 48];
                if (c->V) c->V[o] = c->table[draw(c->kv, n) >> 48];
            }
}
void synth_kv_logical(uint16_t* K, uint16_t* V, int64_t L, const int32_t* seg, const int32_t* off,
                      int n_kv, int hd, int layer, uint64_t seed, const uint16_t* table, int nthreads) {
    kvlog_ctx c = { K, V, seg, off, n_kv, hd, stream_key(seed, synth_kv_tid(layer, 0)),
                    stream_key(seed, synth_kv_tid(layer, 1)), table };
    par_range(L, L * n_kv * hd >= 65536 ? nthreads : 1, kvlog_range, &c);
}

/* ---- one layer of the paged pool: [n_pages][2][n_kv][P][hd] -------------- */
typedef struct {
    uint16_t* pool; const int32_t *pseg, *poff; int P, n_kv, hd; uint64_t kk, kv; const uint16_t* table;
} kvpool_ctx;
static void kvpool_range(void* p, int64_t lo, int64_t hi) {
    kvpool_ctx* c = (kvpool_ctx*)p;
    for (int64_t pg = lo; pg < hi; ++pg)
        for (int w = 0; w < 2; ++w)
            for (int h = 0; h < c->n_kv; ++h)
                for (int s = 0; s < c->P; ++s) {
                    int32_t seg = c->pseg[pg * c->P + s], off = c->poff[pg * c->P + s];
                    uint16_t* dst = c->pool + (((pg * 2 + w) * c->n_kv + h) * (int64_t)c->P + s) * c->hd;
                    for (int d = 0; d < c->hd; ++d)
                        dst[d] = seg < 0 ? 0 : c->table[draw(w ? c->kv : c->kk, kv_index(seg, off, h, d, c->n_kv, c->hd)) >> 48];
                }
}
void synth_kv_pool_layer(uint16_t* pool_layer, int64_t n_pages, const int32_t* page_seg, const int32_t* page_off,
                         int page_size, int n_kv, int hd, int layer, uint64_t seed, const uint16_t* table,
                         int nthreads) {
    kvpool_ctx c = { pool_layer, page_seg, page_off, page_size, n_kv, hd,
                     stream_key(seed, synth_kv_tid(layer, 0)), stream_key(seed, synth_kv_tid(layer, 1)), table };
    par_range(n_pages, n_pages * 2 * n_kv * page_size * hd >= 65536 ? nthreads : 1, kvpool_range, &c);
}

/* ---- providers consumed by the oracle through function pointers ---------- */
/* Weight kinds, in the order the oracle asks for them:
 *   0 embed_verify [d], 1 final_norm [d], 2 w_plus [d], 3 w_minus [d],
 *   4 attn_norm [d], 5 w_qkv [(nq+2nkv)hd][d], 6 w_o [d][nq hd],
 *   7 mlp_norm [d], 8 w_gate_up [2ff][d], 9 w_down [d][ff],
 *   10 .. 17 low-rank adapter factors, 18 q_norm [hd], 19 k_norm [hd]        */
typedef struct {
    uint64_t seed;
    const uint16_t* table_w;   /* weights: bf16(0.02 * quantile) */
    const uint16_t* table_g;   /* norm gains: bf16(1 + gain_std * quantile) */
    const uint16_t* table_kv;  /* cached K/V: bf16(quantile) */
    int nthreads;
    int n_kv, hd;
    /* per candidate logical token identities */
    int n_cand;
    const int64_t* cand_len;
    const int32_t* const* cand_seg;
    const int32_t* const* cand_off;
    const uint16_t* table_qkv; /* W_qkv when non-NULL (a wider draw for peaked attention), else table_w */
} synth_model;

int synth_weight_provider(void* user, int kind, int layer, uint16_t* out, int64_t n) {
    const synth_model* m = (const synth_model*)user;
    int is_gain = (kind == 1 || kind == 4 || kind == 7 || kind == 18 || kind == 19);
    int lay = (kind >= 4) ? layer : 0;
    const uint16_t* table = is_gain ? m->table_g : ((kind == 5 && m->table_qkv) ? m->table_qkv : m->table_w);
    synth_fill(out, n, m->seed, synth_weight_tid(kind, lay), table, m->nthreads);
    return 0;
}

int synth_kv_provider(void* user, int layer, int cand, uint16_t* K, uint16_t* V, int64_t L) {
    const synth_model* m = (const synth_model*)user;
    if (cand < 0 || cand >= m->n_cand || L != m->cand_len[cand]) return -1;
    synth_kv_logical(K, V, L, m->cand_seg[cand], m->cand_off[cand], m->n_kv, m->hd, layer, m->seed, m->table_kv,
                     m->nthreads);
    return 0;
}
