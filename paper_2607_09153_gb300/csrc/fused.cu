// Small fused kernels around the projections, each reducing the GEMM's split-K
// partials in a fixed order (deterministic) and applying the next step of the
// decoder block for the verify token (Sec. 4.1; cost term c_ffn d^2 of Eq.
// cost_kv is in the GEMMs, these are the O(d) glue).  All arithmetic is fp32;
// an activation that feeds a tensor-core contraction is stored as a bf16
// (hi, lo) pair, hi = bf16(x), lo = bf16(x - hi), so no bf16 rounding of the
// activation itself enters the result.
//   rope_table   cos/sin of p * base^(-2i/hd) at p = L_b (fp64 angles)
//   embed_norm   h = e_v ; x = RMSNorm(h) * g
//   qkv_post     q, k, v = sum of splits ; RoPE(q, k)
//   resid_norm   h += sum of splits ; x = RMSNorm(h) * g, or, after the last
//                layer, x = RMSNorm(h) * g_final and
//                P(+) = 1 / (1 + exp(w_minus.x - w_plus.x))   (Eq. score)
//   silu_mul     a = SiLU(gate) * up
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

__global__ void rope_table_kernel(const int32_t* __restrict__ seq_lens, int hd, double base, float2* __restrict__ tab) {
  grid_dep_wait();
  const int b = blockIdx.x, i = threadIdx.x;
  if (i < hd / 2) {
    const double ang = static_cast<double>(seq_lens[b]) * pow(base, -2.0 * i / hd);
    tab[b * (hd / 2) + i] = make_float2(static_cast<float>(cos(ang)), static_cast<float>(sin(ang)));
  }
  grid_dep_launch();
}

__global__ void embed_norm_kernel(const __nv_bfloat16* __restrict__ e_v, const __nv_bfloat16* __restrict__ gain,
                                  int d, float eps, float* __restrict__ h, HiLo x) {
  __shared__ float red[32];
  grid_dep_wait();
  const int b = blockIdx.x;
  float ss = 0.f;
  for (int c = threadIdx.x; c < d; c += blockDim.x) {
    const float v = __bfloat162float(e_v[c]);
    h[static_cast<int64_t>(b) * d + c] = v;
    ss += v * v;
  }
  const float r = 1.0f / sqrtf(block_sum(ss, red) / d + eps);
  for (int c = threadIdx.x; c < d; c += blockDim.x)
    store_hilo(x, static_cast<int64_t>(b) * d + c, __bfloat162float(e_v[c]) * r * __bfloat162float(gain[c]));
  grid_dep_launch();
}

__global__ void qkv_post_kernel(const float* __restrict__ part, int splits, int n_cand, int M, int n_q, int n_kv,
                                int hd, const float2* __restrict__ rope, float* __restrict__ q, HiLo qp,
                                float* __restrict__ kself, float* __restrict__ vself) {
  grid_dep_wait();
  const int hs = blockIdx.x, b = blockIdx.y, i = threadIdx.x, half = hd / 2;
  if (i < half) {
    const int64_t base = static_cast<int64_t>(b) * M + static_cast<int64_t>(hs) * hd;
    const int64_t sstride = static_cast<int64_t>(n_cand) * M;
    float a = 0.f, c = 0.f;
    for (int s = 0; s < splits; ++s) {
      a += part[s * sstride + base + i];
      c += part[s * sstride + base + i + half];
    }
    if (hs < n_q + n_kv) {   // rotate-half RoPE for q and k at p = L_b
      const float2 cs = rope[b * half + i];
      const float a2 = a * cs.x - c * cs.y;
      const float c2 = c * cs.x + a * cs.y;
      a = a2;
      c = c2;
    }
    if (hs < n_q) {
      const int64_t o = (static_cast<int64_t>(b) * n_q + hs) * hd;
      q[o + i] = a;
      q[o + i + half] = c;
      store_hilo(qp, o + i, a);
      store_hilo(qp, o + i + half, c);
    } else {
      float* dst = hs < n_q + n_kv ? kself + (static_cast<int64_t>(b) * n_kv + (hs - n_q)) * hd
                                   : vself + (static_cast<int64_t>(b) * n_kv + (hs - n_q - n_kv)) * hd;
      dst[i] = a;
      dst[i + half] = c;
    }
  }
  grid_dep_launch();
}

__global__ void resid_norm_kernel(const float* __restrict__ part, int splits, int n_cand, int d, float eps,
                                  float* __restrict__ h, const __nv_bfloat16* __restrict__ gain, HiLo x,
                                  const __nv_bfloat16* __restrict__ w_plus,
                                  const __nv_bfloat16* __restrict__ w_minus, float* __restrict__ rewards) {
  __shared__ float red[32];
  grid_dep_wait();
  const int b = blockIdx.x;
  float* hb = h + static_cast<int64_t>(b) * d;
  const int64_t sstride = static_cast<int64_t>(n_cand) * d;
  float ss = 0.f;
  for (int c = threadIdx.x; c < d; c += blockDim.x) {
    float v = hb[c];
    for (int s = 0; s < splits; ++s) v += part[s * sstride + static_cast<int64_t>(b) * d + c];
    hb[c] = v;
    ss += v * v;
  }
  const float r = 1.0f / sqrtf(block_sum(ss, red) / d + eps);
  if (w_plus == nullptr) {
    for (int c = threadIdx.x; c < d; c += blockDim.x)
      store_hilo(x, static_cast<int64_t>(b) * d + c, hb[c] * r * __bfloat162float(gain[c]));
  } else {
    float zp = 0.f, zm = 0.f;
    for (int c = threadIdx.x; c < d; c += blockDim.x) {
      const float xf = hb[c] * r * __bfloat162float(gain[c]);
      zp += xf * __bfloat162float(w_plus[c]);
      zm += xf * __bfloat162float(w_minus[c]);
    }
    zp = block_sum(zp, red);
    zm = block_sum(zm, red);
    if (threadIdx.x == 0) rewards[b] = 1.0f / (1.0f + expf(zm - zp));
  }
  grid_dep_launch();
}

__global__ void silu_mul_kernel(const float* __restrict__ part, int splits, int n_cand, int ff, HiLo a) {
  grid_dep_wait();
  const int64_t total = static_cast<int64_t>(n_cand) * ff;
  const int64_t sstride = total * 2;
  for (int64_t idx = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; idx < total;
       idx += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t b = idx / ff, j = idx - b * ff;
    float g = 0.f, u = 0.f;
    for (int s = 0; s < splits; ++s) {
      g += part[s * sstride + b * 2 * ff + j];
      u += part[s * sstride + b * 2 * ff + ff + j];
    }
    store_hilo(a, idx, g / (1.0f + expf(-g)) * u);
  }
  grid_dep_launch();
}

__global__ void split_sum_kernel(const float* __restrict__ part, int splits, int64_t count, float* __restrict__ out) {
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < count;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    float v = 0.f;
    for (int s = 0; s < splits; ++s) v += part[s * count + i];
    out[i] = v;
  }
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

cudaError_t launch_rope_table(const int32_t* seq_lens, int n_cand, int hd, double base, float2* table,
                              cudaStream_t stream, bool pdl) {
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = make_cfg(dim3(n_cand), dim3(64), stream, attr, pdl);
  return cudaLaunchKernelEx(&cfg, rope_table_kernel, seq_lens, hd, base, table);
}

cudaError_t launch_embed_norm(const ModelDims& m, const __nv_bfloat16* e_v, const __nv_bfloat16* gain, int n_cand,
                              float* h, HiLo x, cudaStream_t stream, bool pdl) {
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = make_cfg(dim3(n_cand), dim3(256), stream, attr, pdl);
  return cudaLaunchKernelEx(&cfg, embed_norm_kernel, e_v, gain, m.d, m.eps, h, x);
}

cudaError_t launch_qkv_post(const ModelDims& m, const float* part, int splits, int n_cand, const float2* rope,
                            float* q, HiLo qp, float* kself, float* vself, cudaStream_t stream, bool pdl) {
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = make_cfg(dim3(m.n_q + 2 * m.n_kv, n_cand), dim3(64), stream, attr, pdl);
  return cudaLaunchKernelEx(&cfg, qkv_post_kernel, part, splits, n_cand, m.qkv_rows, m.n_q, m.n_kv, m.hd, rope, q,
                            qp, kself, vself);
}

cudaError_t launch_resid_norm(const ModelDims& m, const float* part, int splits, int n_cand, float* h,
                              const __nv_bfloat16* gain, HiLo x, const __nv_bfloat16* w_plus,
                              const __nv_bfloat16* w_minus, float* rewards, cudaStream_t stream, bool pdl) {
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = make_cfg(dim3(n_cand), dim3(512), stream, attr, pdl);
  return cudaLaunchKernelEx(&cfg, resid_norm_kernel, part, splits, n_cand, m.d, m.eps, h, gain, x, w_plus, w_minus,
                            rewards);
}

cudaError_t launch_split_hilo(const float* in, int64_t count, HiLo out, cudaStream_t stream) {
  int64_t blocks = (count + 255) / 256;
  if (blocks > 152 * 8) blocks = 152 * 8;
  if (blocks < 1) blocks = 1;
  split_hilo_kernel<<<static_cast<unsigned>(blocks), 256, 0, stream>>>(in, count, out);
  return cudaGetLastError();
}

cudaError_t launch_split_sum(const float* part, int splits, int64_t count, float* out, cudaStream_t stream) {
  int64_t blocks = (count + 255) / 256;
  if (blocks > 152 * 8) blocks = 152 * 8;
  if (blocks < 1) blocks = 1;
  split_sum_kernel<<<static_cast<unsigned>(blocks), 256, 0, stream>>>(part, splits, count, out);
  return cudaGetLastError();
}

cudaError_t launch_silu_mul(const ModelDims& m, const float* part, int splits, int n_cand, HiLo a,
                            cudaStream_t stream, bool pdl) {
  cudaLaunchAttribute attr[1];
  const int64_t total = static_cast<int64_t>(n_cand) * m.ff;
  int64_t blocks = (total + 255) / 256;
  if (blocks > 152 * 8) blocks = 152 * 8;
  cudaLaunchConfig_t cfg = make_cfg(dim3(static_cast<unsigned>(blocks)), dim3(256), stream, attr, pdl);
  return cudaLaunchKernelEx(&cfg, silu_mul_kernel, part, splits, n_cand, m.ff, a);
}

}  // namespace kvprm
