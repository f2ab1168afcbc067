// Kernel launchers of the scoring library (internal).
#pragma once

#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <vector>

namespace kvprm {

// Launch trace record (ptx.cuh: trace_begin / trace_end / trace_event): u64
// [0] earliest CTA start, [1] ~latest CTA end, [2 + e] ~time the last CTA
// passed milestone e of the kernel.
constexpr int kTraceEvents = 8;
constexpr int kTraceStride = 2 + kTraceEvents;

// ---------------------------------------------------------------- projection GEMM
struct GemmPlan {
  bool has_lo = true;    // activation given as a bf16 (hi, lo) pair
  bool gate_up = false;  // tiles of 64 gate rows + the matching 64 up rows
  int m_tiles = 0, k_tiles = 0, kt_per_split = 0, splits = 0, stages = 0, cluster = 1;
  // m-tiles per CTA: 2 for a gate/up projection without split K whose one-tile CTAs would need two
  // waves (large batches); the CTA's stage then holds both weight tiles and one activation tile
  int mt = 1;
  // threads per CTA: 256 on the large-batch image (n_pad >= 64), else 128
  int threads = 128;
  uint32_t tmem_cols = 32;
  size_t smem_bytes = 0;
};
// What the cluster does with the reduced tile (see gemm_tc.cu).
struct GemmEpilogue {
  enum Mode : int { PLAIN = 0, QKV = 1, RESID = 2, SILU = 3, LOWRANK = 4 };
  int mode = PLAIN;
  int M = 0;             // rows of the full output (PLAIN, RESID: row stride of out / h)
  int n_valid = 0;       // candidates
  float* out = nullptr;  // PLAIN: [n][M]
  float* h = nullptr;    // RESID: [n][M], updated in place
  float* sumsq = nullptr;  // RESID: [m_tiles][n] sum of squares of the new h per tile
  // RESID: when set, also x = h ⊙ gain (the next RMSNorm's input before its
  // per-candidate scale) as a bf16 hi/lo pair [n][M] for the next projection
  const __nv_bfloat16* gain_next = nullptr;
  __nv_bfloat16* x_hi = nullptr;
  __nv_bfloat16* x_lo = nullptr;
  // RESID: when set, the new h is also written here ([n][M]; kept for a backward pass)
  float* h_copy = nullptr;
  // SILU: when set, the gate and up pre-activations (after the RMSNorm factor) as [n][2 ff]: gate
  // columns, then up (kept for a backward pass)
  float* gu_save = nullptr;
  // QKV, SILU: when set, the input was h ⊙ gain and the accumulator is scaled
  // per candidate by the RMSNorm factor 1/sqrt(sum_t rs_sumsq[t][n] / rs_d + rs_eps)
  const float* rs_sumsq = nullptr;
  int rs_tiles = 0, rs_d = 0;
  float rs_eps = 0.f;
  const float2* rope = nullptr;  // QKV: [n][hd/2] (cos, sin)
  int n_q = 0, n_kv = 0, hd = 0;
  float* q = nullptr;
  __nv_bfloat16* q_hi = nullptr;
  __nv_bfloat16* q_lo = nullptr;
  float* kself = nullptr;
  float* vself = nullptr;
  // QKV with the per-head q/k RMSNorm (when qn_gain is set): each q and k head's rows are scaled by
  // 1/sqrt(mean over the head of y^2 + rs_eps) and the gain [hd] (q heads qn_gain, k heads kn_gain)
  // before RoPE; y is the projection after the column's RMSNorm factor
  const __nv_bfloat16* qn_gain = nullptr;
  const __nv_bfloat16* kn_gain = nullptr;
  int ff = 0;            // SILU: output width; up rows start at row ff of W
  __nv_bfloat16* a_hi = nullptr;
  __nv_bfloat16* a_lo = nullptr;
  // LOWRANK: t = lr_scale * (A x) as a bf16 hi/lo pair [n][M] (M = the adapter's rank), the extra K
  // columns of the projection that follows (GemmLowRank)
  float lr_scale = 0.f;
  __nv_bfloat16* t_hi = nullptr;
  __nv_bfloat16* t_lo = nullptr;
  // let the next kernel in the stream launch only once this one's partials are parked (after its
  // first cluster barrier) instead of at entry: a next kernel whose CTAs fit beside this one's on
  // an SM otherwise slows that barrier by ~2.5 us (measured for the O projection before gate/up)
  bool late_trigger = false;
};
GemmPlan plan_gemm(int M, int K, int n_pad, int num_sms, bool has_lo, bool gate_up);
// A scorer adapter's term of a projection, y = W x + B t with t = s A x already computed (LOWRANK):
// after its k_main K tiles of W and x the projection streams B [out][r] against t [n][r] as further
// K tiles (the plan counts both: plan_gemm(M, 64 k_main + r, ...)).
struct GemmLowRank {
  const CUtensorMap* b = nullptr;      // B, box of the projection's weight tile
  const CUtensorMap* t_hi = nullptr;   // t hi / lo, box of its activation tile
  const CUtensorMap* t_lo = nullptr;
  int k_main = 0;
};
cudaError_t gemm_configure();
cudaError_t launch_gemm(const GemmPlan& p, const CUtensorMap* tmW, const CUtensorMap* tmX, const CUtensorMap* tmXlo,
                        const GemmEpilogue& ep, int n_pad, int* err, cudaStream_t stream, bool pdl,
                        unsigned long long* ts = nullptr, const GemmLowRank* lr = nullptr);

// ---------------------------------------------------------------- paged attention
struct AttnShape {
  int n_q, n_kv, hd, group;     // group = n_q / n_kv
  int max_blocks;               // block-table row length
  int64_t layer_pages;          // pages per layer of the pool (n_pages)
};
// Tensor map of a paged KV pool [layers][n_pages][2][n_kv][16][hd] (bf16) whose
// box is one page of one kv head, K and V together: 5-D (column within a
// 64-column sub-tile, token, sub-tile, kv head, 2 * (layer * n_pages + page) +
// {0: K, 1: V}) with the 128-byte swizzle, landing in shared memory as
// [K, V][sub-tile][token][64 columns].  page_units = layers * n_pages.
CUresult encode_pool_map(PFN_cuTensorMapEncodeTiled_v12000 encode, CUtensorMap* map, const void* pool,
                         int64_t page_units, int n_kv, int hd);
// One segment of attention work (see attention.cu): a run of physical pages of
// one kv head, scored for one candidate (kind 0) or for up to 8 candidates that
// all reference those pages (kind 1).
struct AttnSeg {
  int32_t kind;
  int32_t g;           // kv head
  int32_t cand;        // kind 0: the candidate; kind 1: offset into AttnWork::cands
  int32_t n_cands;     // kind 1: candidates (<= 8)
  int32_t page_off;    // offset into AttnWork::pages
  int32_t n_pages;     // 0: an empty cache (self entry only)
  int32_t last_valid;  // valid tokens in the segment's last page (1..16)
  int32_t slot;        // kind 0: the partial slot; kind 1: offset into AttnWork::slots
};
struct AttnWork {             // device arrays
  const AttnSeg* segs;
  const int32_t* cta_seg;     // [n_ctas + 1] first segment of each CTA
  const int32_t* pages;       // physical page ids
  const int32_t* cands;       // candidates of shared segments
  const int32_t* slots;       // their partial slots
  const int32_t* slot_base;   // [B][n_kv] first partial slot of each (candidate, kv head)
  const int32_t* nslots;      // [B][n_kv] number of partial slots
  int n_ctas;
  int tc_seg0, n_tc;          // tensor-core segments (kind 2)
  const int32_t* tc_cta;      // [n_tc_ctas + 1] first tensor-core segment of each CTA of attn_tc_kernel
  int n_tc_ctas;
  int fuse_cs;                // > 0: CTAs fuse_cs p .. fuse_cs p + fuse_cs - 1 (one cluster) score pair p and
                              // its rank 0 merges the pair's slots (no combine launch)
};
struct AttnWorkHost {
  std::vector<AttnSeg> segs;
  std::vector<int32_t> cta_seg, pages, cands, slots, slot_base, nslots;
  int n_slots = 0, n_ctas = 0;
  int tc_seg0 = 0, n_tc = 0;   // tensor-core segments (kind 2): segs[tc_seg0, tc_seg0 + n_tc)
  int n_tc_ctas = 0;
  std::vector<int32_t> tc_cta;   // [n_tc_ctas + 1] first segment (index into segs) of each tensor-core CTA
  bool tc_concurrent = false;    // the two attention launches have disjoint SMs and may run at once
  int fuse_cs = 0;               // see AttnWork::fuse_cs
};
// share: 0 every page scored per candidate; 1 shared pages scored once per run
// of <= 8 candidates by the persistent kernel; 2 shared pages scored on the
// tensor cores (head_dim 128 only), tiles of <= 128 / group candidates, each
// launch planned over all n_ctas SMs; 3 as 2, with the SMs split between the
// tensor-core and the private launch so that the later of the two (estimated
// under a cost model) ends soonest, and the two run concurrently.
bool build_attn_work(const int32_t* bt, const int32_t* sl, int n, int max_blocks, int n_kv, int group, int n_ctas,
                     size_t slot_limit, int share, AttnWorkHost& w);
// The plan with the combine fused into the attention launch, for calls where
// every candidate has about the same number of pages, no page is shared and
// group <= 8: (candidate, kv head) pair p = b n_kv + g is scored by the fuse_cs
// CTAs of cluster p, one equal page range and one partial slot each, and the
// cluster's rank 0 merges the slots once all are written.  Returns false (and
// leaves w untouched) when the call does not qualify or the plan would leave
// more than kFuseMaxPages pages per CTA (then the persistent plan is better).
constexpr int kFuseMaxPages = 64;
bool build_attn_work_fused(const int32_t* bt, const int32_t* sl, int n, int max_blocks, int n_kv, int group,
                           int n_ctas, size_t slot_limit, AttnWorkHost& w);
// partial slots a context sized for max_candidates provides (the planner falls
// back to private runs, which always fit, when sharing needs more)
size_t attn_slot_capacity(int max_candidates, int n_kv, int num_sms);
// The same pool with a box of one 64-column sub-tile of one page, K or V
// (2 KB): the tensor-core attention lays a 4-page chunk's tokens contiguously.
CUresult encode_pool_map_tc(PFN_cuTensorMapEncodeTiled_v12000 encode, CUtensorMap* map, const void* pool,
                            int64_t page_units, int n_kv, int hd);
size_t attention_smem_bytes(int hd);
cudaError_t attention_configure();
// Inputs and outputs of the combine (attn_combine_kernel).
struct AttnMerge {
  const float* q;       // [B][n_q][hd] rotated query (fp32)
  const float* kself;   // [B][n_kv][hd]
  const float* vself;   // [B][n_kv][hd]
  __nv_bfloat16* o_hi;  // [B][n_q][hd] attention output as a bf16 pair
  __nv_bfloat16* o_lo;
  float* out_f32;       // optional fp32 copy
  float* dbg;           // optional fp32 copy
  // depth-k readout: row b is verify token b % depth of its candidate and also attends to the
  // candidate's earlier tokens (rows b - b % depth .. b - 1); 1: each row its own entry only
  int depth = 1;
  // optional [B][n_q]: the natural log of each row's softmax normaliser, log sum_j exp(q.k_j / sqrt(hd))
  // over the cache and the self entries (kept for a backward pass)
  float* lse = nullptr;
};
constexpr int kMaxReadoutDepth = 8;
// q_hi / q_lo: bf16 pair of the rotated query [B][n_q][hd]; partial slot s of
// query row r of its group at part_o[(s * group + r) * hd] (values) and
// part_ml[(s * group + r) * 2] (max in log2 units, sum).  One CTA per entry of
// wk.cta_seg.  With wk.fuse_cs > 0 the launch is made of clusters of fuse_cs
// CTAs and also does the combine (mg: its inputs and outputs).
cudaError_t launch_attention(const AttnShape& s, const AttnWork& wk, const CUtensorMap* tm_pool, int layer,
                             const __nv_bfloat16* q_hi, const __nv_bfloat16* q_lo, float* part_o, float* part_ml,
                             const AttnMerge& mg, int* err, cudaStream_t stream, bool pdl,
                             unsigned long long* ts = nullptr);
// The kind-2 segments (wk.tc_seg0 .., wk.n_tc of them; head_dim 128): shared
// pages scored on the tensor cores, one CTA per segment.  Writes the same
// partial slots as launch_attention.  margin: the running row maximum moves
// only when a chunk's scores exceed it by more than this (log2 units; 8 in
// production, 0 to rescale on every new maximum).
// Debug profile of the tensor-core attention (flag 32): an event log of CTA 0
// ([8][128] clock64 stamps) followed by [n_SM][16] per-CTA accumulators.
constexpr int kTcEventLog = 8 * 128;
cudaError_t launch_attention_tc(const AttnShape& s, const AttnWork& wk, const CUtensorMap* tm_pool_tc, int layer,
                                const __nv_bfloat16* q_hi, const __nv_bfloat16* q_lo, float* part_o, float* part_ml,
                                float margin, int* err, cudaStream_t stream, bool pdl,
                                unsigned long long* ts = nullptr, unsigned long long* prof = nullptr);
// Merge every (candidate, kv head)'s slots (wk.slot_base / wk.nslots) of the
// n candidates with the self entry into the attention output.  A single verify
// token per candidate takes the flat form when its (candidate, kv head) pairs
// outnumber one wave of the general form (or always, with force_flat).
cudaError_t launch_attn_combine(const AttnShape& s, const AttnWork& wk, int n, const float* part_o,
                                const float* part_ml, const AttnMerge& mg, cudaStream_t stream, bool pdl,
                                unsigned long long* ts = nullptr, bool force_flat = false);
cudaError_t launch_resolve(const int32_t* bt, const int32_t* seq_lens, int max_blocks, int b, int64_t* out,
                           cudaStream_t stream);

// ---------------------------------------------------------------- fused small kernels
struct ModelDims {
  int d, n_q, n_kv, hd, ff, qkv_rows;
  float eps;
};
// rows b: verify token b % depth of candidate b / depth, at position seq_lens[b] + b % depth
cudaError_t launch_rope_table(const int32_t* seq_lens, int n_rows, int hd, double base, int depth, float2* table,
                              cudaStream_t stream, bool pdl, unsigned long long* ts = nullptr);
// Activations handed to a projection are stored as a bf16 (hi, lo) pair.
struct HiLo {
  __nv_bfloat16* hi;
  __nv_bfloat16* lo;
};
cudaError_t launch_embed_norm(const ModelDims& m, const __nv_bfloat16* e_v, const __nv_bfloat16* gain,
                              int n_cand, float* h, float* sumsq, HiLo x, cudaStream_t stream, bool pdl,
                              unsigned long long* ts = nullptr);
// rewards = P(+) from the final RMSNorm of h and the two head rows
// rewards[b] from row b depth + depth - 1 (each candidate's last verify token)
cudaError_t launch_head(const ModelDims& m, const float* h, const float* sumsq, int m_tiles, int n_rows, int depth,
                        const __nv_bfloat16* gain, const __nv_bfloat16* w_plus, const __nv_bfloat16* w_minus,
                        float* rewards, cudaStream_t stream, bool pdl, unsigned long long* ts = nullptr);
cudaError_t launch_split_hilo(const float* in, int64_t count, HiLo out, cudaStream_t stream);
// ---------------------------------------------------------------- backward pass (KV Steering, grad.cu)
constexpr int kMaxGroup = 16;   // query heads per kv head
cudaError_t launch_transpose(const __nv_bfloat16* in, __nv_bfloat16* out, int rows, int cols, cudaStream_t st);
// d(-log P(+))/dh at the final residual stream h [n][d]; dh fp32 and optionally as hi/lo
cudaError_t launch_head_back(const float* h, const float* p_plus, const __nv_bfloat16* gain,
                             const __nv_bfloat16* w_plus, const __nv_bfloat16* w_minus, int n, int d, float eps,
                             float* dh, __nv_bfloat16* dh_hi, __nv_bfloat16* dh_lo, cudaStream_t st);
// out = dres + RMSNorm backward at h (fp32 [n][d], or h_bf16: one bf16 row for every row) of dy
cudaError_t launch_rms_back(const float* h, const __nv_bfloat16* h_bf16, const __nv_bfloat16* gain, const float* dy,
                            const float* dres, int n, int d, float eps, float* out, __nv_bfloat16* o_hi,
                            __nv_bfloat16* o_lo, cudaStream_t st);
cudaError_t launch_silu_back(const float* da, const float* gu, int n, int ff, __nv_bfloat16* o_hi,
                             __nv_bfloat16* o_lo, cudaStream_t st);
// The attention read-out's backward of one layer.  units: int4 {b, g, j0, j1} (candidate b's logical
// pages j0 .. j1 - 1 of kv head g); shared[page] != 0 for pages several candidates read (their
// gradient accumulates atomically and must be zeroed first).
struct AttnBackArgs {
  int n, n_q, n_kv, hd;
  const float *q, *kself, *vself, *o, *dout, *lse;   // forward saves [n][...] and d(out) [n][n_q hd]
  float *D, *dq, *dks, *dvs;                         // [n][n_q], [n][n_q hd], [n][n_kv hd] x 2
  const int4* units;
  int n_units;
  const int32_t* seq_lens;
  const int32_t* block_table;
  int max_blocks;
  const __nv_bfloat16* pool_layer;                   // [n_pages][2][n_kv][16][hd]
  const uint8_t* shared;
  float* grad_layer;                                 // same layout, fp32
  int* err;                                          // device error word (a bounded wait that gave up)
  // the pool's tensor map (the forward's, one box per page) and this layer's first page unit; with
  // group <= 8 the backward then runs on the tensor cores, else (or when NULL) on the CUDA cores
  const CUtensorMap* tm_pool = nullptr;
  int64_t layer_page0 = 0;
};
// units hold at most this many pages (the pages kernel stages them all in shared memory)
constexpr int kBackUnitPagesMax = 8;
cudaError_t grad_configure();
cudaError_t launch_attn_back(const AttnBackArgs& a, cudaStream_t st);
cudaError_t launch_rope_back(const float* dq, const float* dks, const float* dvs, const float2* rope, int n, int n_q,
                             int n_kv, int hd, __nv_bfloat16* o_hi, __nv_bfloat16* o_lo, cudaStream_t st);
cudaError_t launch_zero_pages(float* grad, const int32_t* pages, int n_list, int n_layers, int64_t n_pages,
                              int64_t page_elems, cudaStream_t st);
cudaError_t launch_steer_update(__nv_bfloat16* kv, const float* grad, const int32_t* pages, int n_list, int n_layers,
                                int64_t n_pages, int64_t page_elems, float eta, cudaStream_t st);

// One thread waits (bounded by limit_ns, see flag_wait) for *flag to become nonzero; on timeout it
// records kDevProbeTimeout in *err.  The failure-detection test hook behind kvprm_debug_wait_probe.
cudaError_t launch_wait_probe(const int* flag, int* err, unsigned long long limit_ns, cudaStream_t stream);


}  // namespace kvprm
