// Kernel launchers of the scoring library (internal).
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <vector>

namespace kvprm {

// ---------------------------------------------------------------- projection GEMM
struct GemmPlan {
  bool has_lo = true;    // activation given as a bf16 (hi, lo) pair
  bool gate_up = false;  // tiles of 64 gate rows + the matching 64 up rows
  int m_tiles = 0, k_tiles = 0, kt_per_split = 0, splits = 0, stages = 0, cluster = 1;
  uint32_t tmem_cols = 32;
  size_t smem_bytes = 0;
};
// What the cluster does with the reduced tile (see gemm_tc.cu).
struct GemmEpilogue {
  enum Mode : int { PLAIN = 0, QKV = 1, RESID = 2, SILU = 3 };
  int mode = PLAIN;
  int M = 0;             // rows of the full output (PLAIN, RESID: row stride of out / h)
  int n_valid = 0;       // candidates
  float* out = nullptr;  // PLAIN: [n][M]
  float* h = nullptr;    // RESID: [n][M], updated in place
  float* sumsq = nullptr;  // RESID: [m_tiles][n] sum of squares of the new h per tile
  const float2* rope = nullptr;  // QKV: [n][hd/2] (cos, sin)
  int n_q = 0, n_kv = 0, hd = 0;
  float* q = nullptr;
  __nv_bfloat16* q_hi = nullptr;
  __nv_bfloat16* q_lo = nullptr;
  float* kself = nullptr;
  float* vself = nullptr;
  int ff = 0;            // SILU: output width; up rows start at row ff of W
  __nv_bfloat16* a_hi = nullptr;
  __nv_bfloat16* a_lo = nullptr;
};
GemmPlan plan_gemm(int M, int K, int n_pad, int num_sms, bool has_lo, bool gate_up);
cudaError_t gemm_configure();
cudaError_t launch_gemm(const GemmPlan& p, const CUtensorMap* tmW, const CUtensorMap* tmX, const CUtensorMap* tmXlo,
                        const GemmEpilogue& ep, int n_pad, int* err, cudaStream_t stream, bool pdl,
                        unsigned long long* ts = nullptr);

// ---------------------------------------------------------------- paged attention
struct AttnShape {
  int n_q, n_kv, hd, group;     // group = n_q / n_kv
  int max_blocks;               // block-table row length
  int64_t layer_rows;           // rows (of hd elements) per layer in the pool map: n_pages * 2 * n_kv * 16
};
// One unit of attention work (see attention.cu): a run of physical pages of one
// candidate (kind 0) or pages shared by up to 8 candidates (kind 1).
struct AttnItem {
  int32_t kind;
  int32_t cand;        // kind 0: the candidate; kind 1: offset into AttnWork::cands
  int32_t n_cands;     // kind 1: candidates (<= 8)
  int32_t page_off;    // offset into AttnWork::pages
  int32_t n_pages;     // 0: an empty cache (self entry only)
  int32_t last_valid;  // valid tokens in the item's last page (1..16)
  int32_t slot;        // kind 0: the candidate's partial slot; kind 1: offset into AttnWork::slots
  int32_t pad;
};
struct AttnWork {            // device arrays
  const AttnItem* items;
  const int32_t* pages;      // physical page ids
  const int32_t* cands;      // candidates of shared items
  const int32_t* slots;      // their partial slots
  const int32_t* nslots;     // [B] partial slots of each candidate
  int n_items;
};
struct AttnWorkHost {
  std::vector<AttnItem> items;
  std::vector<int32_t> pages, cands, slots, nslots;
  int max_item_pages = 0;
};
bool build_attn_work(const int32_t* bt, const int32_t* sl, int n, int max_blocks, int n_kv, int hd, int num_sms,
                     int slot_cap, bool share, AttnWorkHost& w);
size_t attention_smem_bytes(int hd, int max_item_pages);
cudaError_t attention_configure();
// Inputs and outputs of the split merge done by the last CTA of each (candidate, kv head).
struct AttnMerge {
  const float* q;       // [B][n_q][hd] rotated query (fp32)
  const float* kself;   // [B][n_kv][hd]
  const float* vself;   // [B][n_kv][hd]
  int* counter;         // [B][n_kv] arrival counters, zero between calls
  __nv_bfloat16* o_hi;  // [B][n_q][hd] attention output as a bf16 pair
  __nv_bfloat16* o_lo;
  float* out_f32;       // optional fp32 copy
  float* dbg;           // optional fp32 copy
};
// q_hi / q_lo: bf16 pair of the rotated query [B][n_q][hd]; partial slots
// [B][n_q][stride][hd] (values) and [B][n_q][stride][2] (max in log2 units, sum)
cudaError_t launch_attention(const AttnShape& s, const AttnWork& wk, int max_item_pages, const CUtensorMap* tm_pool,
                             int layer, const __nv_bfloat16* q_hi, const __nv_bfloat16* q_lo, int stride,
                             float* part_o, float* part_ml, const AttnMerge& mg, int* err, cudaStream_t stream,
                             bool pdl, unsigned long long* ts = nullptr);
cudaError_t launch_resolve(const int32_t* bt, const int32_t* seq_lens, int max_blocks, int b, int64_t* out,
                           cudaStream_t stream);

// ---------------------------------------------------------------- fused small kernels
struct ModelDims {
  int d, n_q, n_kv, hd, ff, qkv_rows;
  float eps;
};
cudaError_t launch_rope_table(const int32_t* seq_lens, int n_cand, int hd, double base, float2* table,
                              cudaStream_t stream, bool pdl, unsigned long long* ts = nullptr);
// Activations handed to a projection are stored as a bf16 (hi, lo) pair.
struct HiLo {
  __nv_bfloat16* hi;
  __nv_bfloat16* lo;
};
cudaError_t launch_embed_norm(const ModelDims& m, const __nv_bfloat16* e_v, const __nv_bfloat16* gain,
                              int n_cand, float* h, float* sumsq, HiLo x, cudaStream_t stream, bool pdl,
                              unsigned long long* ts = nullptr);
// x = h * r * gain as a hi/lo pair, r = 1/sqrt(sum of the m_tiles partial sums of squares / d + eps)
cudaError_t launch_norm(const ModelDims& m, const float* h, const float* sumsq, int m_tiles, int n_cand,
                        const __nv_bfloat16* gain, HiLo x, cudaStream_t stream, bool pdl,
                        unsigned long long* ts = nullptr);
// rewards = P(+) from the final RMSNorm of h and the two head rows
cudaError_t launch_head(const ModelDims& m, const float* h, const float* sumsq, int m_tiles, int n_cand,
                        const __nv_bfloat16* gain, const __nv_bfloat16* w_plus, const __nv_bfloat16* w_minus,
                        float* rewards, cudaStream_t stream, bool pdl, unsigned long long* ts = nullptr);
cudaError_t launch_split_hilo(const float* in, int64_t count, HiLo out, cudaStream_t stream);


}  // namespace kvprm
