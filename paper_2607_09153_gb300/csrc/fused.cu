// Small kernels around the projections of the verify-token forward (Sec. 4.1;
// the c_ffn d^2 and c_attn d L terms of Eq. cost_kv live in the GEMMs and the
// attention, these are the O(d) glue).  All arithmetic is fp32; an activation
// that feeds a tensor-core contraction is stored as a bf16 (hi, lo) pair,
// hi = bf16(x), lo = bf16(x - hi), so no bf16 rounding of the activation
// itself enters the result.
//   rope_table   cos/sin of p * base^(-2i/hd) at p = L_b (fp64 angles)
//   embed_norm   h = e_v ; per-tile sums of squares of h ; x = h ⊙ g (the
//                RMSNorm's per-candidate factor 1/sqrt(mean(h^2) + eps) is
//                applied by the QKV epilogue, as between all projections)
//   head         x = RMSNorm(h) * g_final with mean(h^2) from the per-tile
//                sums of squares the last residual epilogue wrote (summed in
//                tile order: deterministic);
//                P(+) = 1/(1 + exp(w_minus.x - w_plus.x)) (Eq. score, App. B.2)
#include <cuda_bf16.h>

#include "kernels.h"
#include "ptx.cuh"

namespace kvprm {

namespace {

__device__ __forceinline__ void store_hilo(HiLo o, int64_t i, float x) {
  const __nv_bfloat16 hi = __float2bfloat16_rn(x);
  o.hi[i] = hi;
  o.lo[i] = __float2bfloat16_rn(x - __bfloat162float(hi));
}

// Sum over the block; every thread gets the total.  `red` has >= 32 floats.
__device__ __forceinline__ float block_sum(float v, float* red) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31, nw = (blockDim.x + 31) >> 5;
  __syncthreads();
  if (l == 0) red[w] = v;
  __syncthreads();
  float t = 0.f;
  for (int i = 0; i < nw; ++i) t += red[i];
  return t;
}

// 1/sqrt(mean(h^2) + eps) of candidate b from the per-tile sums of squares,
// summed in tile order by one thread and broadcast through shared memory.
__device__ __forceinline__ float row_rscale(const float* __restrict__ sumsq, int m_tiles, int n_cand, int b, int d,
                                            float eps, float* slot) {
  if (threadIdx.x == 0) {
    float s = 0.f;
    for (int t = 0; t < m_tiles; ++t) s += sumsq[static_cast<int64_t>(t) * n_cand + b];
    *slot = 1.0f / sqrtf(s / d + eps);
  }
  __syncthreads();
  return *slot;
}

__global__ void rope_table_kernel(const int32_t* __restrict__ seq_lens, int hd, double base, int depth,
                                  float2* __restrict__ tab, unsigned long long* ts) {
  trace_begin(ts);
  grid_dep_launch();
  grid_dep_wait();
  const int b = blockIdx.x, i = threadIdx.x;
  if (i < hd / 2) {
    // row b is verify token b % depth of its candidate: position L + b % depth
    const double ang = static_cast<double>(seq_lens[b] + b % depth) * pow(base, -2.0 * i / hd);
    tab[b * (hd / 2) + i] = make_float2(static_cast<float>(cos(ang)), static_cast<float>(sin(ang)));
  }
  trace_end(ts);
}

// One CTA per candidate: h = e_v, its per-tile sums of squares, and x.
__global__ void embed_norm_kernel(const __nv_bfloat16* __restrict__ e_v, const __nv_bfloat16* __restrict__ gain,
                                  int d, int n_cand, float* __restrict__ h, float* __restrict__ sumsq, HiLo x,
                                  unsigned long long* ts) {
  trace_begin(ts);
  grid_dep_launch();
  grid_dep_wait();
  const int b = blockIdx.x;
  // per-tile sums of squares of h, as the residual GEMM epilogue writes them
  const int m_tiles = (d + 127) / 128;
  if (threadIdx.x < m_tiles) {
    float t = 0.f;
    for (int c = threadIdx.x * 128; c < min(d, threadIdx.x * 128 + 128); ++c) {
      const float v = __bfloat162float(e_v[c]);
      t += v * v;
    }
    sumsq[static_cast<int64_t>(threadIdx.x) * n_cand + b] = t;
  }
  // h = e_v, and the QKV projection's input h ⊙ g before the RMSNorm's
  // per-candidate factor, which its epilogue applies from the tile sums
  for (int c = threadIdx.x; c < d; c += blockDim.x) {
    const float v = __bfloat162float(e_v[c]);
    h[static_cast<int64_t>(b) * d + c] = v;
    store_hilo(x, static_cast<int64_t>(b) * d + c, v * __bfloat162float(gain[c]));
  }
  trace_end(ts);
}

// One CTA per candidate: the reward of its last row (its last verify token; one row per candidate
// except in a depth-k readout).
__global__ void head_kernel(const float* __restrict__ h, const float* __restrict__ sumsq, int m_tiles, int n_rows,
                            int depth, int d, float eps, const __nv_bfloat16* __restrict__ gain,
                            const __nv_bfloat16* __restrict__ w_plus, const __nv_bfloat16* __restrict__ w_minus,
                            float* __restrict__ rewards, unsigned long long* ts) {
  trace_begin(ts);
  __shared__ float red[32];
  __shared__ float slot;
  grid_dep_launch();
  grid_dep_wait();
  const int b = blockIdx.x, row = b * depth + depth - 1;
  const float r = row_rscale(sumsq, m_tiles, n_rows, row, d, eps, &slot);
  float zp = 0.f, zm = 0.f;
  for (int c = threadIdx.x; c < d; c += blockDim.x) {
    const float xf = h[static_cast<int64_t>(row) * d + c] * r * __bfloat162float(gain[c]);
    zp += xf * __bfloat162float(w_plus[c]);
    zm += xf * __bfloat162float(w_minus[c]);
  }
  zp = block_sum(zp, red);
  zm = block_sum(zm, red);
  if (threadIdx.x == 0) rewards[b] = 1.0f / (1.0f + expf(zm - zp));
  trace_end(ts);
}

__global__ void split_hilo_kernel(const float* __restrict__ in, int64_t count, HiLo out) {
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < count;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x)
    store_hilo(out, i, in[i]);
}

cudaLaunchConfig_t make_cfg(dim3 grid, dim3 block, cudaStream_t st, cudaLaunchAttribute* attr, bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = 0;
  cfg.stream = st;
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cfg;
}

}  // namespace

cudaError_t launch_rope_table(const int32_t* seq_lens, int n_rows, int hd, double base, int depth, float2* table,
                              cudaStream_t stream, bool pdl, unsigned long long* ts) {
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = make_cfg(dim3(n_rows), dim3(64), stream, attr, pdl);
  return cudaLaunchKernelEx(&cfg, rope_table_kernel, seq_lens, hd, base, depth, table, ts);
}

cudaError_t launch_embed_norm(const ModelDims& m, const __nv_bfloat16* e_v, const __nv_bfloat16* gain, int n_cand,
                              float* h, float* sumsq, HiLo x, cudaStream_t stream, bool pdl,
                              unsigned long long* ts) {
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = make_cfg(dim3(n_cand), dim3(256), stream, attr, pdl);
  return cudaLaunchKernelEx(&cfg, embed_norm_kernel, e_v, gain, m.d, n_cand, h, sumsq, x, ts);
}

cudaError_t launch_head(const ModelDims& m, const float* h, const float* sumsq, int m_tiles, int n_rows, int depth,
                        const __nv_bfloat16* gain, const __nv_bfloat16* w_plus, const __nv_bfloat16* w_minus,
                        float* rewards, cudaStream_t stream, bool pdl, unsigned long long* ts) {
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = make_cfg(dim3(n_rows / depth), dim3(256), stream, attr, pdl);
  return cudaLaunchKernelEx(&cfg, head_kernel, h, sumsq, m_tiles, n_rows, depth, m.d, m.eps, gain, w_plus, w_minus,
                            rewards, ts);
}

__global__ void wait_probe_kernel(const int* flag, int* err, unsigned long long limit_ns) {
  if (threadIdx.x == 0) flag_wait(flag, err, limit_ns, kDevProbeTimeout);
}

cudaError_t launch_wait_probe(const int* flag, int* err, unsigned long long limit_ns, cudaStream_t stream) {
  if (limit_ns > kWaitTimeoutNs) limit_ns = kWaitTimeoutNs;
  wait_probe_kernel<<<1, 32, 0, stream>>>(flag, err, limit_ns);
  return cudaGetLastError();
}

cudaError_t launch_split_hilo(const float* in, int64_t count, HiLo out, cudaStream_t stream) {
  int64_t blocks = (count + 255) / 256;
  if (blocks > 152 * 8) blocks = 152 * 8;
  if (blocks < 1) blocks = 1;
  split_hilo_kernel<<<static_cast<unsigned>(blocks), 256, 0, stream>>>(in, count, out);
  return cudaGetLastError();
}

}  // namespace kvprm
