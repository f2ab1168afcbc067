// Kernel launchers of the scoring library (internal).
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

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
struct AttnPlan {
  int n_split = 1;              // splits of the page range per (candidate, kv head)
  int pages_per_split = 1;
  size_t smem_bytes = 0;
};
AttnPlan plan_attention(const AttnShape& s, int n_cand, int max_pages, int num_sms, int split_cap);
cudaError_t attention_configure();
// part_o [B][n_q][n_split][hd] (unnormalised), part_ml [B][n_q][n_split][2] (max in log2 units, sum)
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
// q_hi / q_lo: bf16 pair of the rotated query [B][n_q][hd]
cudaError_t launch_attn_split(const AttnShape& s, const AttnPlan& p, const CUtensorMap* tm_pool, int layer,
                              const int32_t* bt, const int32_t* seq_lens, const __nv_bfloat16* q_hi,
                              const __nv_bfloat16* q_lo, int n_cand, float* part_o, float* part_ml,
                              const AttnMerge& mg, int* err, cudaStream_t stream, bool pdl,
                              unsigned long long* ts = nullptr);
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
