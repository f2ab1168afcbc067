/*
 * kvprm.h -- C ABI of the GB300 (sm_103a) KV-PRM verify-token scoring library.
 *
 * KV-PRM (Sec. 4.1, Eq. score) scores a candidate trajectory by forwarding one
 * "verify" token through the scorer's layers; at every layer its query attends
 * over the generator's existing per-layer key/value cache of that candidate
 * (the attention read-out of App. A.3, k = 1 query in the depth-k read-out of
 * Def. 1), and a two-logit head over the judgment tokens "+"/"-" (App. B.2)
 * gives the reward s = P(+) = softmax([z_-, z_+]) at "+".  The cost per call is
 * N_L * (c_attn d L + c_ffn d^2) (Eq. cost_kv): the cache is read once and the
 * scorer's weights are streamed once per call, for all candidates together.
 *
 * Conventions (all entry points):
 *  - Return 0 (KVPRM_OK) or a positive KVPRM_E* code; no entry point aborts.
 *    kvprm_last_error() describes the last failure on a context.  All
 *    argument checks run on the host before anything is enqueued.
 *  - "device" pointers are CUDA device (or managed) memory on the device that
 *    was current when the context was created; "host" pointers are ordinary
 *    host memory.  Tensors are dense, row-major, 16-byte aligned.
 *  - bf16 = IEEE bfloat16 bit patterns (uint16 storage).
 *  - A context is used by one host thread at a time.  Work is enqueued on the
 *    caller's CUDA stream (NULL = legacy default stream).
 *  - The library never writes the caller's weights or key/value pages.
 */
#ifndef KVPRM_H
#define KVPRM_H

#include <stdint.h>

#if defined(__GNUC__)
#define KVPRM_API __attribute__((visibility("default")))
#else
#define KVPRM_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

enum {
  KVPRM_OK = 0,
  KVPRM_EINVAL = 1,       /* malformed argument (null pointer, bad shape, misalignment) */
  KVPRM_ECAPACITY = 2,    /* more candidates, or a longer cache, than the context was created for */
  KVPRM_EINDEX = 3,       /* a block-table entry outside [0, n_pages) */
  KVPRM_ECUDA = 4,        /* a CUDA runtime/driver call failed */
  KVPRM_ENOMEM = 5,       /* device or pinned-host allocation failed */
  KVPRM_ETIMEOUT = 6,     /* a bounded in-kernel wait gave up (blocking calls, kvprm_check_device) */
  KVPRM_EUNSUPPORTED = 7  /* a shape the library does not implement */
};

/* Scorer shape and context capacity.
 *  n_layers N_L, d_model d, n_q_heads, n_kv_heads (GQA: query head h reads kv
 *  head floor(h / G), G = n_q_heads / n_kv_heads, 1 <= G <= 16), head_dim in
 *  {64, 128}, d_ff (SiLU-gated MLP width), page_size must be 16.
 *  rope_base: rotary base (rotate-half pairs (i, i + hd/2), angle
 *  p * base^(-2i/hd), the verify token at position p = L_b).  rms_eps: RMSNorm
 *  epsilon.  qk_norm: 0 (default) or 1 -- each query head's and key head's
 *  projection is RMS-normalised over its head_dim entries (eps = rms_eps) with
 *  the layer's gain vector before RoPE, as in the paper's Qwen3 scorers (Sec. 5
 *  "Setup"); the gains are kvprm_weights.q_norm / k_norm.  max_candidates in
 *  [1, 256]; max_blocks_per_seq = the row length of every block table passed
 *  to this context.
 *  d_model, n_q_heads*head_dim and d_ff must be multiples of 64. */
typedef struct {
  int32_t n_layers, d_model, n_q_heads, n_kv_heads, head_dim, d_ff, page_size;
  float rope_base, rms_eps;
  int32_t qk_norm;
  int32_t max_candidates, max_blocks_per_seq;
} kvprm_config;

/* Scorer weights: device bf16, row-major [out][in], borrowed (must outlive the
 * context; not copied).  Per-layer members are HOST arrays of N_L device
 * pointers (the arrays themselves are read during kvprm_create only).
 *  embed_verify [d]     the verify token's embedding row
 *  final_norm   [d]     final RMSNorm gain
 *  w_plus, w_minus [d]  output-head rows of the "+" and "-" judgment tokens
 *  attn_norm[l] [d]     pre-attention RMSNorm gain
 *  w_qkv[l]     [(n_q + 2 n_kv) hd][d]   rows: q heads, then k heads, then v heads
 *  w_o[l]       [d][n_q hd]
 *  mlp_norm[l]  [d]     pre-MLP RMSNorm gain
 *  w_gate_up[l] [2 d_ff][d]              rows: gate, then up
 *  w_down[l]    [d][d_ff]
 *  q_norm[l], k_norm[l] [head_dim]  per-head q / k RMSNorm gains (shared by the
 *               heads of a layer); read only when cfg.qk_norm is set, else the
 *               two members may be NULL                                     */
typedef struct {
  const void* embed_verify;
  const void* final_norm;
  const void* w_plus;
  const void* w_minus;
  const void* const* attn_norm;
  const void* const* w_qkv;
  const void* const* w_o;
  const void* const* mlp_norm;
  const void* const* w_gate_up;
  const void* const* w_down;
  const void* const* q_norm;
  const void* const* k_norm;
} kvprm_weights;

typedef struct kvprm_ctx kvprm_ctx;

/* Create a scoring context: validates the shape, borrows the weights, builds
 * the weight tensor maps and allocates the device workspace (sized for
 * max_candidates x max_blocks_per_seq) on the current device.  On failure
 * *out is NULL and the return code says why (details are not retrievable
 * without a context).  Sec. 4.1 "Architecture". */
KVPRM_API int kvprm_create(const kvprm_config* cfg, const kvprm_weights* weights, kvprm_ctx** out);

/* How a context schedules the attention of each call (fixed at kvprm_create;
 * every choice gives the same result up to fp32 rounding order):
 *  - calls whose candidates all have about the same number of pages (longest
 *    <= 5/4 of the shortest), share no page and have group <= 8 use the
 *    fused-combine plan when it leaves <= 64 pages per CTA: one thread-block
 *    cluster per (candidate, kv head), whose CTAs merge their partial states
 *    through distributed shared memory, so no combine launch follows
 *    (KVPRM_PLAN_FUSE below; environment KVPRM_NO_FUSED_COMBINE=1 turns it off);
 *  - otherwise the persistent plan (kvprm_plan_attention): pages referenced by
 *    several candidates are scored once per group; with head_dim 128, groups of
 *    >= 6 candidates go to a tensor-core launch on a share of the SMs that runs
 *    beside the private pages' launch (a second stream forked and joined inside
 *    the call; share mode 3), smaller groups to the persistent kernel.
 *    Environment: KVPRM_NO_SHARING=1 (every page per candidate),
 *    KVPRM_NO_TC_SHARING=1 (shared groups on the persistent kernel),
 *    KVPRM_TC_SERIAL=1 (the two launches one after the other, all SMs each).
 * KVPRM_NO_GRAPH=1 and KVPRM_NO_PDL=1 switch off graph capture and programmatic
 * dependent launch (for debugging). */

/* Depth-k readout (Sec. 3, Definition "Depth-k Readout": k query vectors
 * against the cache; Sec. 5, "more verify tokens"): every scoring call then
 * appends k verify tokens to each candidate, at positions L_b .. L_b + k - 1,
 * run causally among themselves (token t attends to the cache and to tokens
 * 0 .. t), and reads P(+) at the last one.  Candidate b becomes k rows of the
 * batch that share its pages (each page is still read once per candidate), so
 * n_candidates * k <= max_candidates.  Debug captures (kvprm_debug_attn_out,
 * ...) then hold n_candidates * k rows, candidate b's tokens at rows b k + t.
 * kvprm_attention is not affected.
 *  depth  1 .. 8 (1, the default: one verify token).
 * Errors: KVPRM_EINVAL (depth out of range; nothing changes).  Takes effect for
 * the next scoring call. */
KVPRM_API int kvprm_set_readout_depth(kvprm_ctx* ctx, int32_t depth);

/* Scorer adapter kept apart from the base weights (Sec. 4.1: the scorer is
 * f_{theta + Delta theta}, the base model with a LoRA adapter; App. B.1: rank
 * r = 256, alpha = 32): every projection y = W x of every layer becomes
 * y = W x + scale * B (A x), so one copy of the base weights serves both the
 * generator and the scorer.  Factors are device bf16, row-major, borrowed like
 * the weights (must outlive the context or the next kvprm_set_lora); each
 * member is a HOST array of N_L device pointers, read during this call only:
 *  a_qkv[l] [r][d]        b_qkv[l]     [(n_q + 2 n_kv) hd][r]
 *  a_o[l]   [r][n_q hd]   b_o[l]       [d][r]
 *  a_gate_up[l] [r][d]    b_gate_up[l] [2 d_ff][r]  rows: gate, then up
 *  a_down[l] [r][d_ff]    b_down[l]    [d][r]
 * A per-module adapter on q, k and v (or gate and up) is this form with the
 * modules' A stacked and B block-diagonal.  Each projection then takes two
 * launches: t = scale * (A x), kept at fp32 precision as a bf16 hi/lo pair,
 * then W x + B t as one K loop over the columns of W followed by those of B.
 *  rank   a multiple of 64 in [64, 1024], or 0 to go back to the merged
 *         weights alone (lora is then ignored and may be NULL).
 *  scale  alpha / r in the usual LoRA parameterisation.
 * Errors: KVPRM_EINVAL (bad rank, NULL or unaligned factor; nothing changes),
 * KVPRM_ENOMEM.  Takes effect for the next scoring call (the captured graph
 * is rebuilt). */
typedef struct {
  const void* const* a_qkv;
  const void* const* b_qkv;
  const void* const* a_o;
  const void* const* b_o;
  const void* const* a_gate_up;
  const void* const* b_gate_up;
  const void* const* a_down;
  const void* const* b_down;
} kvprm_lora;
KVPRM_API int kvprm_set_lora(kvprm_ctx* ctx, int32_t rank, float scale, const kvprm_lora* lora);

/* Free the workspace.  Waits for work the context enqueued.  NULL is a no-op. */
KVPRM_API void kvprm_destroy(kvprm_ctx* ctx);

/* Human-readable description of the last failure on ctx ("" if none).  The
 * string is owned by the context and valid until the next call on it. */
KVPRM_API const char* kvprm_last_error(const kvprm_ctx* ctx);

/* Score n_candidates trajectories against their paged caches (Sec. 4.1 Eq.
 * score; the verify token is appended after each candidate's cache, Sec. 1).
 *  kv_pages     device bf16 [N_L][n_pages][2][n_kv_heads][16][head_dim]:
 *               per layer and physical page, the 16 cached keys (index 0) and
 *               values (index 1) of every kv head.  Keys are post-RoPE.
 *  n_pages      physical pages per layer in kv_pages.
 *  block_table  host int32 [n_candidates][max_blocks_per_seq]: logical page j
 *               of candidate b (positions 16j .. 16j+15) is physical page
 *               block_table[b][j].  Candidates may share pages (beam / MCTS
 *               siblings).  Entries j >= ceil(seq_lens[b] / 16) are ignored.
 *  seq_lens     host int32 [n_candidates]: cached length L_b in
 *               [0, 16 * max_blocks_per_seq].  L_b = 0 is legal (the verify
 *               token then attends to itself only).
 *  n_candidates 0 .. max_candidates (0 is a no-op).
 *  rewards      host float [n_candidates]: P(+) per candidate.
 *  stream       cudaStream_t or NULL.
 * Blocking: returns after rewards are written.  The verify token's own k/v are
 * kept in the workspace, never written into kv_pages. */
KVPRM_API int kvprm_score(kvprm_ctx* ctx, const void* kv_pages, int64_t n_pages, const int32_t* block_table,
                const int32_t* seq_lens, int32_t n_candidates, float* rewards, void* stream);

/* As kvprm_score, but stream-ordered: d_rewards is device float [n_candidates]
 * and the call returns once the work is enqueued.  block_table and seq_lens are
 * host arrays; they are copied before the call returns. */
KVPRM_API int kvprm_score_async(kvprm_ctx* ctx, const void* kv_pages, int64_t n_pages, const int32_t* block_table,
                      const int32_t* seq_lens, int32_t n_candidates, float* d_rewards, void* stream);

/* As kvprm_score, but with the cache in HOST memory: h_kv_pages has the
 * kv_pages layout above.  The pages are copied, layer by layer, into a
 * library-owned device pool (grown on demand) after the work already on
 * `stream`, and each layer's attention waits only for its own layer, so the
 * copy of later layers overlaps the scoring of earlier ones; rewards is a host
 * array.  Blocking.  Pinned host memory (page-locked by cudaHostAlloc or
 * cudaHostRegister; first and last byte checked) at a 16-byte aligned address
 * is read by a copy kernel (64 CTAs of 128 threads, 64 MB per launch) that
 * shares SMs with the scoring kernels and holds the host link at its full
 * rate; any other host memory goes through the copy engine (cudaMemcpyAsync).
 * While the copy runs, the forward's kernels are launched without
 * programmatic dependent launch. */
KVPRM_API int kvprm_score_host(kvprm_ctx* ctx, const void* h_kv_pages, int64_t n_pages, const int32_t* block_table,
                     const int32_t* seq_lens, int32_t n_candidates, float* rewards, void* stream);

/* Paged GQA attention read-out alone (App. A.3 with the self entry; the inner
 * step of kvprm_score), for callers that already hold the verify token's
 * rotated query and its own key/value:
 *  kv_layer  device bf16 [n_pages][2][n_kv_heads][16][head_dim] (one layer)
 *  q         device float [n_candidates][n_q_heads][head_dim]
 *  k_self, v_self  device float [n_candidates][n_kv_heads][head_dim]
 *  out       device float [n_candidates][n_q_heads][head_dim]
 * block_table / seq_lens as in kvprm_score.  Stream-ordered. */
KVPRM_API int kvprm_attention(kvprm_ctx* ctx, const void* kv_layer, int64_t n_pages, const int32_t* block_table,
                    const int32_t* seq_lens, int32_t n_candidates, const void* q, const void* k_self,
                    const void* v_self, float* out, void* stream);

/* One projection of the verify-token forward alone (the c_ffn d^2 term of
 * Eq. cost_kv), batched over candidates: Y[n][M] = X[n][K] * W[M][K]^T with
 * bf16 inputs and fp32 accumulation, using the context's split-K GEMM and
 * workspace.  W device bf16 [M][K] (16-byte aligned, K a multiple of 8),
 * X device bf16 [n][K], Y device float [n][M]; 1 <= n <= max_candidates and
 * M * n must fit the context's partial buffer (any M, K of the context's
 * scorer shape does).  Stream-ordered. */
KVPRM_API int kvprm_projection(kvprm_ctx* ctx, const void* W, int32_t M, int32_t K, const void* X, int32_t n,
                               float* Y, void* stream);

/* Final residual stream h (float [n_candidates][d_model], before the final
 * RMSNorm) of the last kvprm_score* call, copied to device memory d_out
 * (stream-ordered on the last call's stream). */
KVPRM_API int kvprm_debug_hidden(kvprm_ctx* ctx, float* d_out);

/* The paged attention read-out (as kvprm_attention) for callers that cannot
 * allocate device memory -- e.g. a serving runtime that reserves all GPU memory
 * up front and forbids allocations afterwards, or code running inside another
 * framework's memory-managed region.  The paper has no counterpart; this is a
 * deployment variant.  It needs no context and calls no cudaMalloc / cudaFree
 * or allocating routine: its scratch is one static device array of
 * KVPRM_NOALLOC_SCRATCH_BYTES that every GPU loading this library holds until
 * the process exits.
 *  kv_layer     device bf16 [n_pages][2][n_kv_heads][16][head_dim] (one layer)
 *  block_table  host int32 [n_candidates][max_blocks_per_seq]; seq_lens host int32
 *               [n_candidates] (validated and copied into the scratch array)
 *  q            device float [n_candidates][n_q_heads][head_dim]
 *  k_self, v_self  device float [n_candidates][n_kv_heads][head_dim]
 *  out          device float [n_candidates][n_q_heads][head_dim]
 * Stream-ordered.  Returns KVPRM_ECAPACITY when the block table, query and
 * split partials would not fit in the array even with one split per sequence
 * (roughly n_candidates * n_q_heads * head_dim * 18 B plus the tables), and
 * the other codes as kvprm_attention (no detailed message: there is no
 * context).  The first call on a device, made with that device current, looks
 * up the array's address (cudaGetSymbolAddress) and configures the kernels:
 * make it before any stream capture.  All calls share the array, which keeps
 * the last call's contents; calls that overlap on the GPU race with each other
 * and must be serialised by the caller.  An in-kernel bounded-wait timeout is
 * recorded in the array but not reported by this entry point.
 * The attention schedule is built on the host for each call and uploaded from
 * pageable host memory, so the call blocks the host until the driver has
 * staged those bytes.  A stream that is being captured into a CUDA graph is
 * refused with KVPRM_EUNSUPPORTED (a graph would replay that one call's
 * schedule from a host buffer that later calls overwrite). */
#define KVPRM_NOALLOC_SCRATCH_BYTES (32u << 20)
KVPRM_API int kvprm_attention_noalloc(const void* kv_layer, int64_t n_pages, const int32_t* block_table,
                                      int32_t max_blocks_per_seq, const int32_t* seq_lens, int32_t n_candidates,
                                      int32_t n_q_heads, int32_t n_kv_heads, int32_t head_dim, const float* q,
                                      const float* k_self, const float* v_self, float* out, void* stream);

/* Debug capture.  flags bit 0: keep every layer's attention output (the
 * combine result o, float, before its bf16 rounding) of each later
 * kvprm_score* call.  kvprm_debug_attn_out copies the last call's capture to
 * device float [N_L][n_candidates][n_q_heads * head_dim] (stream-ordered on
 * the last call's stream).  Bit 1: keep every layer's rotated q, self k and
 * self v (float); bit 2: keep the residual stream after every layer (float).
 * kvprm_debug_layers copies them: which = 1 q [N_L][n][n_q*hd], 2 k_self
 * [N_L][n][n_kv*hd], 3 v_self (same), 4 h [N_L][n][d_model].  Bit 4: the
 * tensor-core attention of shared pages rescales its running state on every
 * new row maximum instead of only beyond a margin of 2^8 (same result up to
 * rounding; exercises the rescale path).  Bit 5: the tensor-core attention
 * accumulates a wait profile; which = 5 copies uint64 [1024 + n_SM * 16]:
 * first CTA 0's event log of the last launch, [8][128] SM-clock stamps -- per
 * chunk 0 S issued, 1 O issued, 2 S seen by the softmax, 3 P written, 4
 * values requested, 5 keys requested; per segment 6 Q loaded, 7 O written
 * out ([7][127] holds the CTA's start) -- then [n_SM][16] SM-clock cycles per
 * CTA, summed over every launch since the flag was set: 0 the MMA issuer
 * waiting for keys, 1 for the S buffer (the O MMAs four chunks back), 2 for
 * P, 3 for values; 4 the softmax waiting for S, 5 for the previous O before a
 * rescale; 6 the loader waiting for a free key stage, 7 for a free value
 * stage; 8 reading S, 9 computing and storing P, 10 a segment's O read-out,
 * 11 loading Q; 12 chunks scored; 13 the CTA's lifetime.  Bit 6: the combine
 * of one verify token per candidate takes its flat form (one warp per query
 * head, every slot's partial loaded in one round) at every batch size, not
 * only when the (candidate, kv head) pairs outnumber the SMs (same result up
 * to rounding; exercises the flat form). */
KVPRM_API int kvprm_set_debug(kvprm_ctx* ctx, int flags);
KVPRM_API int kvprm_debug_attn_out(kvprm_ctx* ctx, float* d_out);
KVPRM_API int kvprm_debug_layers(kvprm_ctx* ctx, int which, void* d_out);

/* Page resolution of the last kvprm_score* call (the block-table walk the
 * attention kernel performs): phys_row[j] = block_table[b][j / 16] * 16 + j % 16
 * for j < seq_lens[b], computed on the device; phys_row is host int64 [L_b].
 * Blocking. */
KVPRM_API int kvprm_resolve(kvprm_ctx* ctx, int32_t b, int64_t* phys_row);

/* The paged-attention schedule a scoring call builds (host only; no context,
 * no GPU).  The paper's read-out (App. A.3) is split here into segments: a
 * segment is a run of physical pages of one kv head scored for one candidate
 * (kind 0) or, when pages are shared by several candidates (a beam prefix or
 * MCTS ancestors), for up to 8 of them at once (kind 1).  Segments are cut so
 * that each of n_ctas CTAs gets an equal share of the estimated cost; each
 * segment writes partial softmax states ("slots") that are merged per
 * (candidate, kv head) with the verify token's own entry.
 * Inputs: block_table host int32 [n_candidates][max_blocks_per_seq], seq_lens
 * host int32 [n_candidates], group = n_q_heads / n_kv_heads, n_ctas >= 1,
 * share: 0 no sharing, 1 shared segments (kind 1) on the persistent CTAs, 2
 * shared pages scored on the tensor cores (kind 2): tiles of up to
 * 128 / group candidates whose 4-page chunks are cut into equal ranges, one
 * per CTA of a separate launch (at most n_ctas of them); 3 (what scoring
 * contexts with head_dim 128 use) as 2, with the n_ctas SMs split between the
 * two launches so that the later one, estimated under a cost model (a
 * tensor-core CTA: 29 units per chunk plus 180; a private page 4, a shared
 * page 2 per candidate), ends soonest (n_ctas + n_tc_ctas <= the given
 * n_ctas), so that they run side by side.  Shared tiles of different groups
 * with the same candidates form one run over all their pages.  Kind-2 segments follow
 * the persistent CTAs' segments (segs[cta_seg[n_ctas]] on), and tensor-core
 * CTA k scores segments segs[tc_cta[k]] .. segs[tc_cta[k + 1] - 1].
 * Outputs go to caller-owned arrays with the capacities given (elements); the
 * counts are always written:
 *  segs       [n_segs][8] int32: kind, kv head, candidate (kind 0) or offset
 *             into cands (kinds 1, 2), candidates, offset into pages, pages,
 *             valid tokens of the last page, slot (kind 0) or offset into slots
 *  cta_seg    [n_ctas + 1] first segment of each persistent CTA
 *  pages      physical page ids referenced by segments
 *  cands      candidates of kind-1 and kind-2 segments; slots: their partial
 *             slots -- a kind-1 segment of n candidates has (8 / n) * n, slot w
 *             written by the warp that scores candidate w % n on every
 *             (8 / n)-th page of each stage (all 8 warps busy for n <= 4); a
 *             kind-2 segment one per candidate
 *  slot_base, nslots  [n_candidates][n_kv_heads] first slot and slot count
 *  tc_cta     [n_tc_ctas + 1] first segment (index into segs) of each
 *             tensor-core CTA
 * Returns KVPRM_EINVAL for bad arguments and KVPRM_ECAPACITY if an array is
 * too small (counts still reflect the full plan). */
typedef struct {
  int32_t n_segs, n_ctas, n_pages, n_cands, n_slot_refs, n_slots; /* out */
  int32_t* segs;
  int64_t segs_cap; /* segments (8 ints each) */
  int32_t* cta_seg;
  int64_t cta_cap;
  int32_t* pages;
  int64_t pages_cap;
  int32_t* cands;
  int64_t cands_cap;
  int32_t* slots;
  int64_t slots_cap;
  int32_t* slot_base; /* [n_candidates * n_kv_heads] */
  int32_t* nslots;    /* [n_candidates * n_kv_heads] */
  int32_t n_tc_ctas;  /* out */
  int32_t* tc_cta;
  int64_t tc_cta_cap;
  int32_t fuse_cs;    /* out: 0, or the cluster size of a fused-combine plan */
} kvprm_attn_plan;
/* share | KVPRM_PLAN_FUSE: first try the fused-combine plan (what scoring
 * contexts do): when every candidate has about the same number of pages (the
 * longest at most 5/4 of the shortest), no page is referenced twice and
 * group <= 8, (candidate, kv head) pair p = b * n_kv_heads + g is scored by the
 * fuse_cs CTAs fuse_cs * p .. fuse_cs * p + fuse_cs - 1 (one thread-block
 * cluster; fuse_cs a power of two <= 8 with pairs * fuse_cs <= n_ctas, at most
 * 64 pages per CTA), rank r taking pages [r L / fuse_cs, (r + 1) L / fuse_cs) of
 * the candidate's L and partial slot fuse_cs * p + r; rank 0 merges the
 * pair's slots in the same launch, so no combine launch follows. */
#define KVPRM_PLAN_FUSE 16
KVPRM_API int kvprm_plan_attention(const int32_t* block_table, int32_t max_blocks_per_seq, const int32_t* seq_lens,
                                   int32_t n_candidates, int32_t n_kv_heads, int32_t group, int32_t n_ctas,
                                   int32_t share, kvprm_attn_plan* plan);

/* The launch plan a scoring context uses for one projection GEMM y = W x (W [M][K] bf16, x a bf16
 * hi/lo pair when has_lo, batch padded to n_pad, a multiple of 16), computed on the host only (no
 * device call), so that its invariants can be checked without a GPU.  gate_up: W holds the gate rows
 * then the up rows (M = d_ff pairs, 64 of each per tile).
 *  m_tiles       128-row tiles (gate/up: 64-pair tiles)
 *  k_tiles       64-wide K tiles; kt_per_split per rank of a split-K cluster
 *  cluster       CTAs per thread-block cluster (split-K ranks)
 *  tiles_per_cta m-tiles each CTA takes (1, or 2 for large batches)
 *  stages        shared-memory ring stages; tmem_cols tensor-memory columns; smem_bytes per CTA
 *  threads       threads per CTA: 256 for n_pad >= 64 (the large-batch kernel image), else 128
 * Errors: KVPRM_EINVAL (M, K or num_sms < 1, n_pad not a positive multiple of 16, out NULL). */
typedef struct {
  int32_t m_tiles, k_tiles, kt_per_split, cluster, tiles_per_cta, stages, tmem_cols;
  int64_t smem_bytes;
  int32_t threads;
} kvprm_projection_plan;
KVPRM_API int kvprm_plan_projection(int32_t M, int32_t K, int32_t n_pad, int32_t num_sms, int32_t has_lo,
                                    int32_t gate_up, kvprm_projection_plan* out);

/* Device-side status: returns KVPRM_OK, or KVPRM_ETIMEOUT if an in-kernel
 * bounded wait gave up since the last check (the flag is then cleared).
 * Synchronises the context's last stream. */
KVPRM_API int kvprm_check_device(kvprm_ctx* ctx);

/* KV Steering (Sec. 6 "Discussion on Broader Applications"; App. C, Algorithm
 * "KV Steering at agent handoff"): KV-PRM's score is differentiable in the
 * cache, so the cache can be refined by gradient steps on l = -log P(+).
 *
 * kvprm_score_grad scores the candidates as kvprm_score does (rewards, host
 * float [n_candidates], P(+)) and writes the gradient of the batch's loss
 * sum_b -log P(+)_b with respect to every cached key and value:
 *  d_grad  device float, the kv_pages layout [N_L][n_pages][2][n_kv_heads][16]
 *          [head_dim] (16-byte aligned): for every page some candidate's block
 *          table references, in every layer, dl/dK and dl/dV of its 16 slots
 *          (slots past a candidate's length in its last page: 0; a page several
 *          candidates read holds the sum of their gradients).  Pages no
 *          candidate references are not written.
 * The backward pass runs the verify-token forward with its intermediates
 * kept, then the chain rule in reverse: each projection's transposed product
 * on the forward's tensor-core GEMM, the attention read-out's backward over
 * the pages (w_j = softmax weight, ds_j = w_j (do . V_j - do . o),
 * dK_j += ds_j q / sqrt(hd), dV_j += w_j do), RoPE and RMSNorm backward.  The
 * first call on a context builds library-owned transposed copies of the four
 * projection matrices of every layer (as much device memory as the weights)
 * and buffers for the intermediates (sized for max_candidates).
 * Scope: merged weights (no kvprm_set_lora adapter), readout depth 1, qk_norm
 * 0; otherwise KVPRM_EUNSUPPORTED.  Other errors as kvprm_score, KVPRM_ENOMEM.
 * Blocking.  The caller's pages are only read.
 *
 * kvprm_steer runs `steps` steps of the algorithm on a caller-owned copy of the
 * cache, kv_pages (device bf16, kvprm_score's layout, READ AND WRITTEN): each
 * step takes the gradient at the current pages and sets every referenced
 * page's keys and values to RNE_bf16(kv - eta * grad) (the cache stays bf16,
 * the paper's precision); a page several candidates read takes their summed
 * gradient once.  p_first / p_last (host float [n_candidates], may be NULL):
 * P(+) before the first step and after the last.  Uses a library-owned fp32
 * gradient buffer of the pool's size.  Same scope and errors as
 * kvprm_score_grad; steps >= 0 (0 scores only).  Blocking. */
KVPRM_API int kvprm_score_grad(kvprm_ctx* ctx, const void* kv_pages, int64_t n_pages, const int32_t* block_table,
                               const int32_t* seq_lens, int32_t n_candidates, float* d_grad, float* rewards,
                               void* stream);
KVPRM_API int kvprm_steer(kvprm_ctx* ctx, void* kv_pages, int64_t n_pages, const int32_t* block_table,
                          const int32_t* seq_lens, int32_t n_candidates, float eta, int32_t steps, float* p_first,
                          float* p_last, void* stream);

/* Failure-detection test hooks (no counterpart in the paper: they let tests
 * drive the error paths on the host, without faulting or hanging a GPU).
 *  kvprm_debug_set_alloc_limit: from now on the library may allocate at most
 *    `bytes` more device and pinned-host memory, process-wide (every allocation
 *    lowers the remainder; -1 removes the limit).  An allocation beyond it fails
 *    as if the device were full: kvprm_create, kvprm_score_host (growing its
 *    device pool) and kvprm_set_lora return KVPRM_ENOMEM and leave an existing
 *    context as it was.
 *  kvprm_debug_inject_error: where = 1 makes the next scoring call on ctx
 *    report a failed launch of its forward (KVPRM_ECUDA, nothing of the forward
 *    enqueued) as a CUDA error would; where = 0 cancels it.  Later calls run
 *    normally.
 *  kvprm_debug_wait_probe: enqueues on `stream` one thread that waits, bounded
 *    by limit_us (1 .. 2e6 microseconds), for a device flag that nothing sets,
 *    with the same give-up protocol as every in-kernel wait: when the limit
 *    passes it records its site (code 9) in the context's device error word and
 *    returns, so the next kvprm_check_device (or blocking call) returns
 *    KVPRM_ETIMEOUT and clears the word; the context stays usable.
 * Errors: KVPRM_EINVAL (NULL context, bad argument), KVPRM_ECUDA. */
KVPRM_API int kvprm_debug_set_alloc_limit(int64_t bytes);
KVPRM_API int kvprm_debug_inject_error(kvprm_ctx* ctx, int32_t where);
KVPRM_API int kvprm_debug_wait_probe(kvprm_ctx* ctx, int32_t limit_us, void* stream);

/* Per-kernel-class timing of kvprm_score* calls, measured with CUDA events on
 * the scoring stream while enabled (one event pair per launch; programmatic
 * launch overlap is switched off meanwhile, so each launch is timed alone).
 * Classes: 0..3 the QKV, O, gate/up and down projections, 4 paged attention
 * (split-K, CUDA cores), 5 attention combine, 6 fused norm / RoPE / SiLU /
 * head kernels, 7 paged attention of shared pages on the tensor cores, 8 the
 * scorer adapter's A x products (kvprm_set_lora).
 * Profiled calls synchronise the stream.  kvprm_get_profile returns per class
 * the launch count and total milliseconds since profiling was enabled. */
enum {
  KVPRM_PROF_GEMM_QKV = 0,
  KVPRM_PROF_GEMM_O = 1,
  KVPRM_PROF_GEMM_GATE_UP = 2,
  KVPRM_PROF_GEMM_DOWN = 3,
  KVPRM_PROF_ATTN = 4,
  KVPRM_PROF_COMBINE = 5,
  KVPRM_PROF_FUSED = 6,
  KVPRM_PROF_ATTN_TC = 7,
  KVPRM_PROF_LORA = 8,
  KVPRM_PROF_N = 9
};
KVPRM_API int kvprm_set_profile(kvprm_ctx* ctx, int enable);

/* Device timeline of the last kvprm_score* call, recorded by the kernels
 * themselves with the GPU global timer while enabled (two atomics per CTA;
 * launch overlap is kept).  kvprm_get_trace synchronises and fills, per launch
 * in issue order, its class (as for profiling), the start of its first CTA and
 * the end of its last CTA in microseconds from the first start; returns the
 * number of records written, or a negative KVPRM_E* code. */
KVPRM_API int kvprm_set_trace(kvprm_ctx* ctx, int enable);
KVPRM_API int kvprm_get_trace(kvprm_ctx* ctx, int32_t max_records, int32_t* cls, double* start_us, double* end_us);
/* As kvprm_get_trace, plus the critical path inside each projection launch:
 * events_us [max_records][8] (may be NULL) holds, per launch, the time at
 * which the LAST CTA passed each milestone -- 0 the preceding kernel had
 * completed (programmatic-launch wait returned), 1 the first weight and
 * activation tiles landed, 2 all MMAs completed, 3 the accumulators were
 * parked in shared memory cluster-wide, 4 the split-K reduction over the
 * cluster was done, 5 the RMSNorm factors were ready, 6 the epilogue was
 * written, 7 the cluster released.  Attention launches record 0 the query
 * was ready, 1 the consumer warps had scored every page, 2 the private runs
 * were merged into their partial slots; combine launches 0 the partials were
 * ready, 1 the outputs were written.  -1 where a launch has no such
 * milestone. */
KVPRM_API int kvprm_get_trace_events(kvprm_ctx* ctx, int32_t max_records, int32_t* cls, double* start_us,
                                     double* end_us, double* events_us);
KVPRM_API int kvprm_get_profile(kvprm_ctx* ctx, int64_t* launches, double* total_ms);

#ifdef __cplusplus
}
#endif

#endif /* KVPRM_H */
