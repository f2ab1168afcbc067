// Kernel launchers of the scoring library (internal).
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace kvprm {

// ---------------------------------------------------------------- projection GEMM
struct GemmPlan {
  bool has_lo = true;   // activation given as a bf16 (hi, lo) pair
  int m_tiles = 0, k_tiles = 0, kt_per_split = 0, splits = 0, stages = 0;
  uint32_t tmem_cols = 32;
  size_t smem_bytes = 0;
};
GemmPlan plan_gemm(int M, int K, int n_pad, int num_sms, bool has_lo);
cudaError_t gemm_configure();
cudaError_t launch_gemm(const GemmPlan& p, const CUtensorMap* tmW, const CUtensorMap* tmX, const CUtensorMap* tmXlo,
                        float* part, int M, int n_valid, int n_pad, int* err, cudaStream_t stream, bool pdl);

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
// q_hi / q_lo: bf16 pair of the rotated query [B][n_q][hd]
cudaError_t launch_attn_split(const AttnShape& s, const AttnPlan& p, const CUtensorMap* tm_pool, int layer,
                              const int32_t* bt, const int32_t* seq_lens, const __nv_bfloat16* q_hi,
                              const __nv_bfloat16* q_lo, int n_cand, float* part_o, float* part_ml, int* err,
                              cudaStream_t stream, bool pdl);
// o = merge(splits, self entry) -> (o_hi, o_lo) bf16 pair [n_pad rows][n_q*hd], optionally fp32 copies
cudaError_t launch_attn_combine(const AttnShape& s, const AttnPlan& p, const int32_t* seq_lens, const float* q,
                                const float* kself, const float* vself, const float* part_o, const float* part_ml,
                                int n_cand, __nv_bfloat16* o_hi, __nv_bfloat16* o_lo, float* out_f32, float* dbg,
                                cudaStream_t stream, bool pdl);
cudaError_t launch_resolve(const int32_t* bt, const int32_t* seq_lens, int max_blocks, int b, int64_t* out,
                           cudaStream_t stream);

// ---------------------------------------------------------------- fused small kernels
struct ModelDims {
  int d, n_q, n_kv, hd, ff, qkv_rows;
  float eps;
};
cudaError_t launch_rope_table(const int32_t* seq_lens, int n_cand, int hd, double base, float2* table,
                              cudaStream_t stream, bool pdl);
// Activations handed to a projection are stored as a bf16 (hi, lo) pair.
struct HiLo {
  __nv_bfloat16* hi;
  __nv_bfloat16* lo;
};
cudaError_t launch_embed_norm(const ModelDims& m, const __nv_bfloat16* e_v, const __nv_bfloat16* gain,
                              int n_cand, float* h, HiLo x, cudaStream_t stream, bool pdl);
// q (fp32 and hi/lo pair) and the self k / v (fp32), RoPE applied to q and k
cudaError_t launch_qkv_post(const ModelDims& m, const float* part, int splits, int n_cand, const float2* rope,
                            float* q, HiLo qp, float* kself, float* vself, cudaStream_t stream, bool pdl);
// h += sum_s part; then either x = RMSNorm(h) * gain as a hi/lo pair (w_plus == nullptr)
// or rewards = P(+) from the final norm and the two head rows.
cudaError_t launch_resid_norm(const ModelDims& m, const float* part, int splits, int n_cand, float* h,
                              const __nv_bfloat16* gain, HiLo x, const __nv_bfloat16* w_plus,
                              const __nv_bfloat16* w_minus, float* rewards, cudaStream_t stream, bool pdl);
cudaError_t launch_split_sum(const float* part, int splits, int64_t count, float* out, cudaStream_t stream);
cudaError_t launch_silu_mul(const ModelDims& m, const float* part, int splits, int n_cand, HiLo a,
                            cudaStream_t stream, bool pdl);
cudaError_t launch_split_hilo(const float* in, int64_t count, HiLo out, cudaStream_t stream);

}  // namespace kvprm
