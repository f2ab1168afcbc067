// Backward pass of the verify-token forward, for KV Steering (Sec. 6; App. C, Algorithm "KV Steering
// at agent handoff"): the gradient of l = sum_b -log P(+)_b with respect to every cached key and
// value.  The projections' transposed products run on the forward's tensor-core GEMM against
// transposed weight copies (kvprm_api.cu); this file holds the rest:
//   transpose       W [rows][cols] -> W^T (bf16), once per context
//   head_back       dh = d(-log P)/dh at the final RMSNorm: dx = (1 - P)(w_- - w_+)
//   rms_back        dh = dres + r g dy - h r^3 (sum_i g_i dy_i h_i) / d,  r = (mean h^2 + eps)^-1/2
//   silu_back       du = da t SiLU'(u),  dt = da SiLU(u)
//   attn_back_pre   per (candidate, kv head): D_h = do_h . o_h and the self entry's terms
//   attn_back_pages per run of cached pages: w_j = exp(q.K_j / sqrt(hd) - lse), ds_j = w_j (do.V_j - D),
//                   dK_j = sum_h ds_j q_h / sqrt(hd), dV_j = sum_h w_j do_h, dq_h += ds_j K_j / sqrt(hd)
//   rope_back       the rotation by the negative angle, and [dq; dk; dv] as the next GEMM's input
//   zero_pages      clears the gradient of pages several candidates read (they are accumulated)
//   steer_update    kv <- RNE_bf16(kv - eta grad) on the pages the block tables reference
// Every product runs in fp32; a gradient that feeds a tensor-core contraction is stored as a bf16
// (hi, lo) pair like the forward's activations.
#include <cuda_bf16.h>

#include <utility>

#include "kernels.h"
#include "ptx.cuh"

namespace kvprm {

namespace {

typedef __nv_bfloat16 bf16;

__device__ __forceinline__ void put_hilo(bf16* hi, bf16* lo, int64_t i, float x) {
  const bf16 h = __float2bfloat16_rn(x);
  hi[i] = h;
  lo[i] = __float2bfloat16_rn(x - __bfloat162float(h));
}

// two block-wide sums at once (blockDim.x a multiple of 32, <= 1024); every thread gets both
__device__ __forceinline__ float2 block_sum2(float a, float b, float2* red) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    a += __shfl_xor_sync(0xffffffffu, a, off);
    b += __shfl_xor_sync(0xffffffffu, b, off);
  }
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31, nw = blockDim.x >> 5;
  __syncthreads();
  if (l == 0) red[w] = make_float2(a, b);
  __syncthreads();
  float2 t = make_float2(0.f, 0.f);
  for (int i = 0; i < nw; ++i) {
    t.x += red[i].x;
    t.y += red[i].y;
  }
  return t;
}

__global__ void transpose_kernel(const bf16* __restrict__ in, bf16* __restrict__ out, int rows, int cols) {
  __shared__ bf16 tile[32][34];
  const int c0 = blockIdx.x * 32, r0 = blockIdx.y * 32;
  for (int j = threadIdx.y; j < 32; j += blockDim.y) {
    const int r = r0 + j, c = c0 + threadIdx.x;
    if (r < rows && c < cols) tile[j][threadIdx.x] = in[static_cast<int64_t>(r) * cols + c];
  }
  __syncthreads();
  for (int j = threadIdx.y; j < 32; j += blockDim.y) {
    const int c = c0 + j, r = r0 + threadIdx.x;
    if (c < cols && r < rows) out[static_cast<int64_t>(c) * rows + r] = tile[threadIdx.x][j];
  }
}

// One CTA per row: the loss gradient at the final residual stream h.
__global__ void head_back_kernel(const float* __restrict__ h, const float* __restrict__ p_plus,
                                 const bf16* __restrict__ gain, const bf16* __restrict__ w_plus,
                                 const bf16* __restrict__ w_minus, int d, float eps, float* __restrict__ dh,
                                 bf16* __restrict__ dh_hi, bf16* __restrict__ dh_lo) {
  __shared__ float2 red[32];
  grid_dep_launch();
  grid_dep_wait();   // every input is written by earlier kernels of the stream
  const int b = blockIdx.x;
  const float* hb = h + static_cast<int64_t>(b) * d;
  const float q = 1.f - p_plus[b];   // d(-log P)/dz_- = 1 - P = -d(-log P)/dz_+
  float ss = 0.f, sd = 0.f;
  for (int i = threadIdx.x; i < d; i += blockDim.x) {
    const float hv = hb[i];
    const float gdy = __bfloat162float(gain[i]) * q * (__bfloat162float(w_minus[i]) - __bfloat162float(w_plus[i]));
    ss += hv * hv;
    sd += gdy * hv;
  }
  const float2 t = block_sum2(ss, sd, red);
  const float r = rsqrtf(t.x / d + eps);
  const float c = r * r * r * t.y / d;
  for (int i = threadIdx.x; i < d; i += blockDim.x) {
    const float gdy = __bfloat162float(gain[i]) * q * (__bfloat162float(w_minus[i]) - __bfloat162float(w_plus[i]));
    const float v = r * gdy - hb[i] * c;
    dh[static_cast<int64_t>(b) * d + i] = v;
    if (dh_hi) put_hilo(dh_hi, dh_lo, static_cast<int64_t>(b) * d + i, v);
  }
}

// One CTA per row: dh = dres + RMSNorm backward of (h, gain) applied to dy (may run in place:
// dres == out).  h_bf16 (when set) is one bf16 row shared by every row (the embedding of layer 0).
__global__ void rms_back_kernel(const float* __restrict__ h, const bf16* __restrict__ h_bf16,
                                const bf16* __restrict__ gain, const float* __restrict__ dy, const float* dres, int d,
                                float eps, float* out, bf16* __restrict__ o_hi, bf16* __restrict__ o_lo) {
  __shared__ float2 red[32];
  grid_dep_launch();
  grid_dep_wait();
  const int b = blockIdx.x;
  const int64_t row = static_cast<int64_t>(b) * d;
  float ss = 0.f, sd = 0.f;
  for (int i = threadIdx.x; i < d; i += blockDim.x) {
    const float hv = h_bf16 ? __bfloat162float(h_bf16[i]) : h[row + i];
    ss += hv * hv;
    sd += __bfloat162float(gain[i]) * dy[row + i] * hv;
  }
  const float2 t = block_sum2(ss, sd, red);
  const float r = rsqrtf(t.x / d + eps);
  const float c = r * r * r * t.y / d;
  for (int i = threadIdx.x; i < d; i += blockDim.x) {
    const float hv = h_bf16 ? __bfloat162float(h_bf16[i]) : h[row + i];
    const float v = dres[row + i] + r * __bfloat162float(gain[i]) * dy[row + i] - hv * c;
    out[row + i] = v;
    if (o_hi) put_hilo(o_hi, o_lo, row + i, v);
  }
}

// da [n][ff], gu [n][2 ff] (gate then up pre-activations) -> [du; dt] [n][2 ff] as hi/lo
__global__ void silu_back_kernel(const float* __restrict__ da, const float* __restrict__ gu, int n, int ff,
                                 bf16* __restrict__ o_hi, bf16* __restrict__ o_lo) {
  grid_dep_launch();
  grid_dep_wait();
  const int64_t total = static_cast<int64_t>(n) * ff;
  for (int64_t e = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; e < total;
       e += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t b = e / ff, j = e - b * ff;
    const float u = gu[b * 2 * ff + j], t = gu[b * 2 * ff + ff + j];
    const float sg = 1.f / (1.f + expf(-u));
    const float a = da[e];
    put_hilo(o_hi, o_lo, b * 2 * ff + j, a * t * sg * (1.f + u * (1.f - sg)));
    put_hilo(o_hi, o_lo, b * 2 * ff + ff + j, a * u * sg);
  }
}

// One CTA of 128 threads per (row b, kv head g): D_h = do_h . o_h for the G query heads, and the
// verify token's own entry: w_s = exp(q_h . k_s / sqrt(hd) - lse_h), ds_s = w_s (do_h . v_s - D_h),
// dk_s = sum_h ds_s q_h / sqrt(hd), dv_s = sum_h w_s do_h, dq_h = ds_s k_s / sqrt(hd) (the pages add on).
__global__ void attn_back_pre_kernel(const float* __restrict__ q, const float* __restrict__ ks,
                                     const float* __restrict__ vs, const float* __restrict__ o,
                                     const float* __restrict__ dout, const float* __restrict__ lse, int n_q, int n_kv,
                                     int hd, float* __restrict__ D, float* __restrict__ dq, float* __restrict__ dks,
                                     float* __restrict__ dvs) {
  __shared__ float s_w[kMaxGroup], s_ds[kMaxGroup];
  grid_dep_launch();
  grid_dep_wait();
  const int b = blockIdx.x / n_kv, g = blockIdx.x % n_kv, G = n_q / n_kv;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const float scale = rsqrtf(static_cast<float>(hd));
  const int64_t hk = (static_cast<int64_t>(b) * n_kv + g) * hd;
  for (int r = warp; r < G; r += blockDim.x >> 5) {
    const int64_t hq = (static_cast<int64_t>(b) * n_q + g * G + r) * hd;
    float dd = 0.f, sq = 0.f, dp = 0.f;
    for (int e = lane; e < hd; e += 32) {
      dd += dout[hq + e] * o[hq + e];
      sq += q[hq + e] * ks[hk + e];
      dp += dout[hq + e] * vs[hk + e];
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      dd += __shfl_xor_sync(0xffffffffu, dd, off);
      sq += __shfl_xor_sync(0xffffffffu, sq, off);
      dp += __shfl_xor_sync(0xffffffffu, dp, off);
    }
    if (lane == 0) {
      const int64_t row = static_cast<int64_t>(b) * n_q + g * G + r;
      const float w = expf(sq * scale - lse[row]);
      D[row] = dd;
      s_w[r] = w;
      s_ds[r] = w * (dp - dd);
    }
  }
  __syncthreads();
  for (int e = threadIdx.x; e < hd; e += blockDim.x) {
    float ak = 0.f, av = 0.f;
    for (int r = 0; r < G; ++r) {
      const int64_t hq = (static_cast<int64_t>(b) * n_q + g * G + r) * hd;
      ak += s_ds[r] * q[hq + e];
      av += s_w[r] * dout[hq + e];
      dq[hq + e] = s_ds[r] * ks[hk + e] * scale;
    }
    dks[hk + e] = ak * scale;
    dvs[hk + e] = av;
  }
}

// One CTA of 4 warps per unit {b, g, j0, j1}: candidate b's logical pages j0 .. j1 - 1 (at most
// kBackUnitPages) of kv head g.  Thread 0 bulk-copies the unit's K and V blocks (16 x HD bf16 each,
// contiguous in the pool) into shared memory at once, so every byte of the unit is in flight before
// any is used.  Warp w then takes tokens w, w + 4, .. of each page; each lane holds HD / 32
// consecutive elements of the token's key and value, of the G query rows and of their output
// gradients, so every dot product is a lane-local sum and one warp reduction.  dK and dV of a page
// only this candidate reads are stored; of a page several read (shared[page] != 0) they are added
// with atomics (zero_pages cleared them).  dq is summed over the CTA's warps (in the shared memory
// the pages occupied), then added atomically.
constexpr int kBackUnitPages = kBackUnitPagesMax;

template <int HD>
constexpr size_t back_pages_smem() {
  return static_cast<size_t>(kBackUnitPages) * 2 * 16 * HD * 2 + 16;   // the pages' K and V, the barrier
}

template <int HD, int GMAX>
__global__ void __launch_bounds__(128) attn_back_pages_kernel(
    const int4* __restrict__ units, const int32_t* __restrict__ seq_lens, const int32_t* __restrict__ block_table,
    int max_blocks, const bf16* __restrict__ pool_layer, const uint8_t* __restrict__ shared, const float* __restrict__ q,
    const float* __restrict__ dout, const float* __restrict__ lse, const float* __restrict__ D, int n_q, int n_kv,
    float* __restrict__ grad_layer, float* __restrict__ dq, int* err) {
  constexpr int kPer = HD / 32;   // 4 (hd 128) or 2 (hd 64)
  constexpr uint32_t kBlock = 16 * HD * 2;   // one page's K (or V) of one kv head, bytes
  extern __shared__ __align__(16) uint8_t smem[];
  bf16* s_kv = reinterpret_cast<bf16*>(smem);   // [page][K, V][16][HD]
  uint64_t* bar = reinterpret_cast<uint64_t*>(smem + static_cast<size_t>(kBackUnitPages) * 2 * kBlock);
  grid_dep_launch();
  grid_dep_wait();
  const int4 u = units[blockIdx.x];
  const int b = u.x, g = u.y, j0 = u.z, j1 = u.w;
  const int npg = j1 - j0;   // 1 .. kBackUnitPages
  const int G = n_q / n_kv;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const float scale = rsqrtf(static_cast<float>(HD));
  const int L = seq_lens[b];
  const int64_t page_elems = static_cast<int64_t>(2) * n_kv * 16 * HD;   // one page of one layer
  if (threadIdx.x == 0) {
    mbar_init(bar, 1);
    fence_mbar_init();
    mbar_arrive_expect_tx(bar, static_cast<uint32_t>(npg) * 2 * kBlock);
    for (int i = 0; i < npg; ++i) {
      const int32_t p = block_table[static_cast<int64_t>(b) * max_blocks + j0 + i];
      const bf16* kp = pool_layer + p * page_elems + static_cast<int64_t>(g) * 16 * HD;
      bulk_load(s_kv + (2 * i) * 16 * HD, kp, kBlock, bar);
      bulk_load(s_kv + (2 * i + 1) * 16 * HD, kp + static_cast<int64_t>(n_kv) * 16 * HD, kBlock, bar);
    }
  }
  float qr[GMAX][kPer], dr[GMAX][kPer], acc[GMAX][kPer];
  float lse_r[GMAX], D_r[GMAX];
#pragma unroll
  for (int r = 0; r < GMAX; ++r) {
    if (r < G) {
      const int64_t row = static_cast<int64_t>(b) * n_q + g * G + r;
#pragma unroll
      for (int k = 0; k < kPer; ++k) {
        qr[r][k] = q[row * HD + lane * kPer + k];
        dr[r][k] = dout[row * HD + lane * kPer + k];
        acc[r][k] = 0.f;
      }
      lse_r[r] = lse[row];
      D_r[r] = D[row];
    }
  }
  __syncthreads();   // the barrier is initialised
  if (!mbar_wait(bar, 0, err)) {
    // gave up (the error word is set): wait, bounded again, for the copies still landing in this
    // CTA's shared memory before leaving
    mbar_wait(bar, 0, err);
    return;
  }
  for (int i = 0; i < npg; ++i) {
    const int j = j0 + i;
    const int32_t p = block_table[static_cast<int64_t>(b) * max_blocks + j];
    const int valid = min(16, L - 16 * j);
    const bf16* ks = s_kv + (2 * i) * 16 * HD;
    const bf16* vs = ks + 16 * HD;
    float* gk = grad_layer + p * page_elems + static_cast<int64_t>(g) * 16 * HD;
    float* gv = gk + static_cast<int64_t>(n_kv) * 16 * HD;
    const bool sh = shared[p] != 0;
    for (int t = warp; t < 16; t += 4) {
      float kf[kPer], vf[kPer];
      if constexpr (kPer == 4) {
        const uint2 kb = *reinterpret_cast<const uint2*>(ks + t * HD + lane * 4);
        const uint2 vb = *reinterpret_cast<const uint2*>(vs + t * HD + lane * 4);
        const float2 k01 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&kb.x));
        const float2 k23 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&kb.y));
        const float2 v01 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&vb.x));
        const float2 v23 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&vb.y));
        kf[0] = k01.x; kf[1] = k01.y; kf[2] = k23.x; kf[3] = k23.y;
        vf[0] = v01.x; vf[1] = v01.y; vf[2] = v23.x; vf[3] = v23.y;
      } else {
        const uint32_t kb = *reinterpret_cast<const uint32_t*>(ks + t * HD + lane * 2);
        const uint32_t vb = *reinterpret_cast<const uint32_t*>(vs + t * HD + lane * 2);
        const float2 k01 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&kb));
        const float2 v01 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&vb));
        kf[0] = k01.x; kf[1] = k01.y;
        vf[0] = v01.x; vf[1] = v01.y;
      }
      float dk[kPer], dv[kPer];
#pragma unroll
      for (int k = 0; k < kPer; ++k) dk[k] = dv[k] = 0.f;
      if (t < valid) {
        // the G heads' two dot products, reduced over the warp together
        float sv[GMAX], pv[GMAX];
#pragma unroll
        for (int r = 0; r < GMAX; ++r) {
          sv[r] = 0.f;
          pv[r] = 0.f;
          if (r < G) {
#pragma unroll
            for (int k = 0; k < kPer; ++k) {
              sv[r] += qr[r][k] * kf[k];
              pv[r] += dr[r][k] * vf[k];
            }
          }
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1)
#pragma unroll
          for (int r = 0; r < GMAX; ++r)
            if (r < G) {
              sv[r] += __shfl_xor_sync(0xffffffffu, sv[r], off);
              pv[r] += __shfl_xor_sync(0xffffffffu, pv[r], off);
            }
#pragma unroll
        for (int r = 0; r < GMAX; ++r) {
          if (r >= G) break;
          const float w = expf(sv[r] * scale - lse_r[r]);
          const float ds = w * (pv[r] - D_r[r]);
#pragma unroll
          for (int k = 0; k < kPer; ++k) {
            dk[k] += ds * scale * qr[r][k];
            dv[k] += w * dr[r][k];
            acc[r][k] += ds * scale * kf[k];
          }
        }
      }
      float* gkt = gk + t * HD + lane * kPer;
      float* gvt = gv + t * HD + lane * kPer;
      if constexpr (kPer == 4) {
        const float4 k4 = make_float4(dk[0], dk[1], dk[2], dk[3]);
        const float4 v4 = make_float4(dv[0], dv[1], dv[2], dv[3]);
        if (sh) {
          atomicAdd(reinterpret_cast<float4*>(gkt), k4);
          atomicAdd(reinterpret_cast<float4*>(gvt), v4);
        } else {
          *reinterpret_cast<float4*>(gkt) = k4;
          *reinterpret_cast<float4*>(gvt) = v4;
        }
      } else {
        if (sh) {
#pragma unroll
          for (int k = 0; k < kPer; ++k) {
            atomicAdd(gkt + k, dk[k]);
            atomicAdd(gvt + k, dv[k]);
          }
        } else {
          *reinterpret_cast<float2*>(gkt) = make_float2(dk[0], dk[1]);
          *reinterpret_cast<float2*>(gvt) = make_float2(dv[0], dv[1]);
        }
      }
    }
  }
  // dq: the four warps' sums (in the shared memory the pages occupied), then one atomic add each
  __syncthreads();
  float* s_dq = reinterpret_cast<float*>(smem);   // [4][GMAX][HD] <= the page buffer
#pragma unroll
  for (int r = 0; r < GMAX; ++r)
    if (r < G)
#pragma unroll
      for (int k = 0; k < kPer; ++k) s_dq[(warp * GMAX + r) * HD + lane * kPer + k] = acc[r][k];
  __syncthreads();
  for (int i = threadIdx.x; i < G * HD; i += blockDim.x) {
    const int r = i / HD, e = i - r * HD;
    const float v = s_dq[(0 * GMAX + r) * HD + e] + s_dq[(1 * GMAX + r) * HD + e] + s_dq[(2 * GMAX + r) * HD + e] +
                    s_dq[(3 * GMAX + r) * HD + e];
    atomicAdd(dq + (static_cast<int64_t>(b) * n_q + g * G + r) * HD + e, v);
  }
}

// ---------------------------------------------------------------- attention backward on the tensor cores
// The same unit of work (candidate b, kv head g, up to kBackUnitPages pages) for G <= 8 query heads
// per kv head.  Thread 0 loads the unit's pages with the forward's tensor map (one 128-byte-swizzled
// box per page: K then V), so each page's keys and values are addressed exactly as in the forward.
// Each warp takes pages w, w + 4 and per page of 16 tokens computes, with mma.m16n8k16 (bf16 in,
// fp32 accumulate) -- every fp32 operand entering as a bf16 (hi, lo) pair so that the products keep
// ~16 bits:
//   S  = Q K^T and dP = dO V^T   A = q (or dO) with the hi parts in rows 0..7 and the lo parts in
//                                rows 8..15 of the same heads (their sum is the product), B = K or V
//                                from shared memory (ldmatrix);
//   w = exp(S / sqrt(hd) - lse), ds = w (dP - D) / sqrt(hd)     in registers, row = head;
//   dq += ds K                   A = ds (hi rows 0..7, lo rows 8..15), B = K through ldmatrix.trans;
//   dV = w^T dO, dK = ds^T Q     contractions over the heads: w and ds go through movmatrix (an 8x8
//                                transpose in registers) into A fragments whose k columns 0..7 hold
//                                the heads' hi parts and 8..15 their lo parts; B holds [dO_hi; dO_hi]
//                                for one MMA and [dO_lo; 0] for a second, so the sum is
//                                w_hi dO_hi + w_lo dO_hi + w_hi dO_lo (the lo x lo term, ~2^-16 of the
//                                product, is left out);
// then stores the page's dK and dV rows (or adds them atomically on a shared page).
template <int HD>
struct BackTcSmem {
  static constexpr uint32_t kBlock = (HD / 64) * 16 * 128;   // one page's K (or V) of one kv head
  static constexpr uint32_t kPage = 2 * kBlock;
  static constexpr uint32_t kPages = 0;                      // [pages][K, V], as the forward's box lands
  static constexpr int kLd = HD + 8;                          // padded row of the B matrices (elements)
  static constexpr uint32_t kB = kPages + kBackUnitPages * kPage;   // [4][16][kLd] bf16: Q hh, Q l0, dO hh, dO l0
  static constexpr uint32_t kBar = kB + 4 * 16 * kLd * 2;
  static constexpr size_t kBytes = kBar + 16 + 1024;          // + alignment slack
};

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~static_cast<uintptr_t>(1023));
}

__device__ __forceinline__ uint32_t movmatrix_trans(uint32_t a) {
  uint32_t d;
  asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(d) : "r"(a));
  return d;
}

__device__ __forceinline__ float bf16_hi(float x) { return __bfloat162float(__float2bfloat16_rn(x)); }

template <int HD>
__global__ void __launch_bounds__(128) attn_back_tc_kernel(
    const __grid_constant__ CUtensorMap tm_pool, int64_t layer_page0, const int4* __restrict__ units,
    const int32_t* __restrict__ seq_lens, const int32_t* __restrict__ block_table, int max_blocks,
    const uint8_t* __restrict__ shared, const float* __restrict__ q, const float* __restrict__ dout,
    const float* __restrict__ lse, const float* __restrict__ D, int n_q, int n_kv, float* __restrict__ grad_layer,
    float* __restrict__ dq, int* err) {
  using SM = BackTcSmem<HD>;
  constexpr int KS = HD / 16;   // 16-wide steps over the head dimension
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = align1024(smem_raw);
  uint64_t* bar = reinterpret_cast<uint64_t*>(base + SM::kBar);
  bf16* Bq_hh = reinterpret_cast<bf16*>(base + SM::kB);   // rows 0..7 q_hi of the heads, rows 8..15 q_hi again
  bf16* Bq_l0 = Bq_hh + 16 * SM::kLd;                     // rows 0..7 q_lo, rows 8..15 zero
  bf16* Bd_hh = Bq_l0 + 16 * SM::kLd;                     // the same for dO
  bf16* Bd_l0 = Bd_hh + 16 * SM::kLd;
  const int4 u = units[blockIdx.x];
  const int b = u.x, g = u.y, j0 = u.z, npg = u.w - u.z;
  const int G = n_q / n_kv;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, gid = lane >> 2, tig = lane & 3;
  const float scale = rsqrtf(static_cast<float>(HD));
  const int L = seq_lens[b];
  const int64_t page_elems = static_cast<int64_t>(2) * n_kv * 16 * HD;
  const int64_t row0 = static_cast<int64_t>(b) * n_q + static_cast<int64_t>(g) * G;   // the group's first row
  if (threadIdx.x == 0) {
    mbar_init(bar, 1);
    fence_mbar_init();
    tma_prefetch_desc(&tm_pool);
    mbar_arrive_expect_tx(bar, static_cast<uint32_t>(npg) * SM::kPage);
    const uint64_t pol = policy_evict_first();
    for (int i = 0; i < npg; ++i) {
      const int32_t p = block_table[static_cast<int64_t>(b) * max_blocks + j0 + i];
      tma_load_5d(base + SM::kPages + i * SM::kPage, &tm_pool, bar, 0, 0, 0, g,
                  static_cast<int32_t>(2 * (layer_page0 + p)), pol);
    }
  }
  // the pages (an input of the whole pass) are in flight; q, dO, lse and D may be written by the
  // kernels just before this one
  grid_dep_launch();
  grid_dep_wait();
  // the B matrices of dV and dK: [16 k rows][HD] bf16, k = head (hi parts twice, or lo parts then zeros)
  for (int i = threadIdx.x; i < 16 * HD; i += blockDim.x) {
    const int k = i / HD, e = i - k * HD, h = k & 7;
    const bool ok = h < G;
    const float qv = ok ? q[(row0 + h) * HD + e] : 0.f, dv = ok ? dout[(row0 + h) * HD + e] : 0.f;
    const float qh = bf16_hi(qv), dh = bf16_hi(dv);
    Bq_hh[k * SM::kLd + e] = __float2bfloat16_rn(qh);
    Bd_hh[k * SM::kLd + e] = __float2bfloat16_rn(dh);
    Bq_l0[k * SM::kLd + e] = __float2bfloat16_rn(k < 8 ? qv - qh : 0.f);
    Bd_l0[k * SM::kLd + e] = __float2bfloat16_rn(k < 8 ? dv - dh : 0.f);
  }
  // A fragments of q and dO for S and dP: row gid the hi part, row gid + 8 the lo part of head gid
  uint32_t qa[KS][4], da[KS][4];
  {
    const bool ok = gid < G;
    const float* qr = q + (row0 + gid) * HD;
    const float* dr = dout + (row0 + gid) * HD;
#pragma unroll
    for (int ks = 0; ks < KS; ++ks) {
      const int c = ks * 16 + tig * 2;
      float qv[4], dv[4];
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        const int cc = c + (t & 1) + 8 * (t >> 1);
        qv[t] = ok ? qr[cc] : 0.f;
        dv[t] = ok ? dr[cc] : 0.f;
      }
      qa[ks][0] = pack_bf16(qv[0], qv[1]);
      qa[ks][1] = pack_bf16(qv[0] - bf16_hi(qv[0]), qv[1] - bf16_hi(qv[1]));
      qa[ks][2] = pack_bf16(qv[2], qv[3]);
      qa[ks][3] = pack_bf16(qv[2] - bf16_hi(qv[2]), qv[3] - bf16_hi(qv[3]));
      da[ks][0] = pack_bf16(dv[0], dv[1]);
      da[ks][1] = pack_bf16(dv[0] - bf16_hi(dv[0]), dv[1] - bf16_hi(dv[1]));
      da[ks][2] = pack_bf16(dv[2], dv[3]);
      da[ks][3] = pack_bf16(dv[2] - bf16_hi(dv[2]), dv[3] - bf16_hi(dv[3]));
    }
  }
  const float lse_g = gid < G ? lse[row0 + gid] : 0.f;
  const float D_g = gid < G ? D[row0 + gid] : 0.f;
  float dqa[HD / 8][4];
#pragma unroll
  for (int n = 0; n < HD / 8; ++n) dqa[n][0] = dqa[n][1] = dqa[n][2] = dqa[n][3] = 0.f;
  __syncthreads();   // the barrier is initialised and the B matrices are written
  if (!__all_sync(0xffffffffu, mbar_wait(bar, 0, err))) {
    // gave up (the error word is set): wait, bounded again, for the copies still landing in this
    // CTA's shared memory before leaving
    mbar_wait(bar, 0, err);
    return;
  }
  const int mi = lane >> 3;
  for (int i = warp; i < npg; i += 4) {
    const int j = j0 + i;
    const int32_t p = block_table[static_cast<int64_t>(b) * max_blocks + j];
    const int valid = min(16, L - 16 * j);
    const uint32_t kbase = smem_u32(base + SM::kPages + i * SM::kPage), vbase = kbase + SM::kBlock;
    // S = Q K^T and dP = dO V^T over the page's 16 tokens (two n-tiles of 8)
    float s0[4] = {0.f, 0.f, 0.f, 0.f}, s1[4] = {0.f, 0.f, 0.f, 0.f};
    float p0[4] = {0.f, 0.f, 0.f, 0.f}, p1[4] = {0.f, 0.f, 0.f, 0.f};
    {
      const int tok = (mi >> 1) * 8 + (lane & 7);
#pragma unroll
      for (int ks = 0; ks < KS; ++ks) {
        const int hdc = ks * 16 + (mi & 1) * 8;
        const uint32_t off = (hdc >> 6) * 2048 + tok * 128 + ((((hdc & 63) >> 3) ^ (tok & 7)) << 4);
        uint32_t kb[4], vb[4];
        ldsm_x4(kbase + off, kb[0], kb[1], kb[2], kb[3]);
        ldsm_x4(vbase + off, vb[0], vb[1], vb[2], vb[3]);
        mma_bf16_16816(s0, qa[ks][0], qa[ks][1], qa[ks][2], qa[ks][3], kb[0], kb[1]);
        mma_bf16_16816(s1, qa[ks][0], qa[ks][1], qa[ks][2], qa[ks][3], kb[2], kb[3]);
        mma_bf16_16816(p0, da[ks][0], da[ks][1], da[ks][2], da[ks][3], vb[0], vb[1]);
        mma_bf16_16816(p1, da[ks][0], da[ks][1], da[ks][2], da[ks][3], vb[2], vb[3]);
      }
    }
    // head gid, tokens tig*2, tig*2 + 1, 8 + tig*2, 9 + tig*2: the hi and lo rows summed
    const float x[4] = {s0[0] + s0[2], s0[1] + s0[3], s1[0] + s1[2], s1[1] + s1[3]};
    const float dp[4] = {p0[0] + p0[2], p0[1] + p0[3], p1[0] + p1[2], p1[1] + p1[3]};
    float w[4], ds[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int t = (e & 1) + tig * 2 + 8 * (e >> 1);
      w[e] = (gid < G && t < valid) ? expf(x[e] * scale - lse_g) : 0.f;
      ds[e] = w[e] * (dp[e] - D_g) * scale;
    }
    float wl[4], dl[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      wl[e] = w[e] - bf16_hi(w[e]);
      dl[e] = ds[e] - bf16_hi(ds[e]);
    }
    // dq += ds K (K as the k x n operand through ldmatrix.trans, as V in the forward's P V)
    {
      const uint32_t a0 = pack_bf16(ds[0], ds[1]), a1 = pack_bf16(dl[0], dl[1]);
      const uint32_t a2 = pack_bf16(ds[2], ds[3]), a3 = pack_bf16(dl[2], dl[3]);
      const int tok = (mi & 1) * 8 + (lane & 7);
#pragma unroll
      for (int j2 = 0; j2 < HD / 16; ++j2) {
        const int hdc = j2 * 16 + (mi >> 1) * 8;
        uint32_t kb[4];
        ldsm_x4_t(kbase + (hdc >> 6) * 2048 + tok * 128 + ((((hdc & 63) >> 3) ^ (tok & 7)) << 4), kb[0], kb[1],
                  kb[2], kb[3]);
        mma_bf16_16816(dqa[2 * j2], a0, a1, a2, a3, kb[0], kb[1]);
        mma_bf16_16816(dqa[2 * j2 + 1], a0, a1, a2, a3, kb[2], kb[3]);
      }
    }
    // w^T and ds^T as A fragments: rows = tokens, k 0..7 = the heads' hi parts, 8..15 their lo parts
    const uint32_t wt0 = movmatrix_trans(pack_bf16(w[0], w[1])), wt1 = movmatrix_trans(pack_bf16(w[2], w[3]));
    const uint32_t wt2 = movmatrix_trans(pack_bf16(wl[0], wl[1])), wt3 = movmatrix_trans(pack_bf16(wl[2], wl[3]));
    const uint32_t st0 = movmatrix_trans(pack_bf16(ds[0], ds[1])), st1 = movmatrix_trans(pack_bf16(ds[2], ds[3]));
    const uint32_t st2 = movmatrix_trans(pack_bf16(dl[0], dl[1])), st3 = movmatrix_trans(pack_bf16(dl[2], dl[3]));
    float* gk = grad_layer + p * page_elems + static_cast<int64_t>(g) * 16 * HD;
    float* gv = gk + static_cast<int64_t>(n_kv) * 16 * HD;
    const bool sh = shared[p] != 0;
    auto put = [&](float* dst, float a, float c) {
      if (sh)
        atomicAdd(reinterpret_cast<float2*>(dst), make_float2(a, c));
      else
        *reinterpret_cast<float2*>(dst) = make_float2(a, c);
    };
    {
      const int krow = (mi & 1) * 8 + (lane & 7);
#pragma unroll
      for (int j2 = 0; j2 < HD / 16; ++j2) {
        const int col = j2 * 16 + (mi >> 1) * 8;
        uint32_t dh[4], dlo[4], qh[4], ql[4];
        ldsm_x4_t(smem_u32(Bd_hh + krow * SM::kLd + col), dh[0], dh[1], dh[2], dh[3]);
        ldsm_x4_t(smem_u32(Bd_l0 + krow * SM::kLd + col), dlo[0], dlo[1], dlo[2], dlo[3]);
        ldsm_x4_t(smem_u32(Bq_hh + krow * SM::kLd + col), qh[0], qh[1], qh[2], qh[3]);
        ldsm_x4_t(smem_u32(Bq_l0 + krow * SM::kLd + col), ql[0], ql[1], ql[2], ql[3]);
        float v0[4] = {0.f, 0.f, 0.f, 0.f}, v1[4] = {0.f, 0.f, 0.f, 0.f};
        float k0[4] = {0.f, 0.f, 0.f, 0.f}, k1[4] = {0.f, 0.f, 0.f, 0.f};
        mma_bf16_16816(v0, wt0, wt1, wt2, wt3, dh[0], dh[1]);
        mma_bf16_16816(v0, wt0, wt1, wt2, wt3, dlo[0], dlo[1]);
        mma_bf16_16816(v1, wt0, wt1, wt2, wt3, dh[2], dh[3]);
        mma_bf16_16816(v1, wt0, wt1, wt2, wt3, dlo[2], dlo[3]);
        mma_bf16_16816(k0, st0, st1, st2, st3, qh[0], qh[1]);
        mma_bf16_16816(k0, st0, st1, st2, st3, ql[0], ql[1]);
        mma_bf16_16816(k1, st0, st1, st2, st3, qh[2], qh[3]);
        mma_bf16_16816(k1, st0, st1, st2, st3, ql[2], ql[3]);
        // C rows: token gid (elements 0, 1) and gid + 8 (2, 3); columns of the two n-tiles
        const int c0 = j2 * 16 + tig * 2, c1 = c0 + 8;
        put(gv + gid * HD + c0, v0[0], v0[1]);
        put(gv + (gid + 8) * HD + c0, v0[2], v0[3]);
        put(gv + gid * HD + c1, v1[0], v1[1]);
        put(gv + (gid + 8) * HD + c1, v1[2], v1[3]);
        put(gk + gid * HD + c0, k0[0], k0[1]);
        put(gk + (gid + 8) * HD + c0, k0[2], k0[3]);
        put(gk + gid * HD + c1, k1[0], k1[1]);
        put(gk + (gid + 8) * HD + c1, k1[2], k1[3]);
      }
    }
  }
  // dq: rows gid (hi) and gid + 8 (lo) of head gid summed, the four warps' parts through shared
  // memory (the page buffer, no longer read), then one atomic add per element
  __syncthreads();
  float* s_dq = reinterpret_cast<float*>(base);   // [4][8][HD] <= the page buffer
#pragma unroll
  for (int n = 0; n < HD / 8; ++n) {
    const int c = n * 8 + tig * 2;
    s_dq[(warp * 8 + gid) * HD + c] = dqa[n][0] + dqa[n][2];
    s_dq[(warp * 8 + gid) * HD + c + 1] = dqa[n][1] + dqa[n][3];
  }
  __syncthreads();
  for (int i2 = threadIdx.x; i2 < G * HD; i2 += blockDim.x) {
    const int r = i2 / HD, e = i2 - r * HD;
    const float v = s_dq[(0 * 8 + r) * HD + e] + s_dq[(1 * 8 + r) * HD + e] + s_dq[(2 * 8 + r) * HD + e] +
                    s_dq[(3 * 8 + r) * HD + e];
    atomicAdd(dq + (row0 + r) * HD + e, v);
  }
}

// One CTA per row: [dq; dk; dv] before RoPE (the rotation by the negative angle of position L_b)
// as the bf16 hi/lo input of the W_qkv^T product, [n][(n_q + 2 n_kv) hd].
__global__ void rope_back_kernel(const float* __restrict__ dq, const float* __restrict__ dks,
                                 const float* __restrict__ dvs, const float2* __restrict__ rope, int n_q, int n_kv,
                                 int hd, bf16* __restrict__ o_hi, bf16* __restrict__ o_lo) {
  grid_dep_launch();
  grid_dep_wait();
  const int b = blockIdx.x, half = hd / 2;
  const int rows = (n_q + 2 * n_kv) * hd;
  const int64_t ob = static_cast<int64_t>(b) * rows;
  for (int e = threadIdx.x; e < (n_q + n_kv) * half; e += blockDim.x) {
    const int head = e / half, i = e - head * half;
    const float* src = head < n_q ? dq + (static_cast<int64_t>(b) * n_q + head) * hd
                                  : dks + (static_cast<int64_t>(b) * n_kv + head - n_q) * hd;
    const float2 cs = rope[static_cast<int64_t>(b) * half + i];
    const float da = src[i], db = src[i + half];
    put_hilo(o_hi, o_lo, ob + head * hd + i, da * cs.x + db * cs.y);
    put_hilo(o_hi, o_lo, ob + head * hd + i + half, db * cs.x - da * cs.y);
  }
  for (int e = threadIdx.x; e < n_kv * hd; e += blockDim.x)
    put_hilo(o_hi, o_lo, ob + (n_q + n_kv) * hd + e, dvs[static_cast<int64_t>(b) * n_kv * hd + e]);
}

// Zero every layer's gradient of the listed pages.
__global__ void zero_pages_kernel(float* __restrict__ grad, const int32_t* __restrict__ pages, int n_list,
                                  int n_layers, int64_t n_pages, int64_t page_elems) {
  grid_dep_launch();
  grid_dep_wait();
  const int64_t per = page_elems / 4;
  const int64_t total = static_cast<int64_t>(n_list) * n_layers * per;
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < total;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t e = i % per, rest = i / per;
    const int64_t l = rest % n_layers, k = rest / n_layers;
    float4* dst = reinterpret_cast<float4*>(grad + (l * n_pages + pages[k]) * page_elems) + e;
    *dst = make_float4(0.f, 0.f, 0.f, 0.f);
  }
}

// kv <- RNE_bf16(kv - eta grad) for every layer of the listed pages.
__global__ void steer_update_kernel(bf16* __restrict__ kv, const float* __restrict__ grad,
                                    const int32_t* __restrict__ pages, int n_list, int n_layers, int64_t n_pages,
                                    int64_t page_elems, float eta) {
  grid_dep_launch();
  grid_dep_wait();
  const int64_t per = page_elems / 4;
  const int64_t total = static_cast<int64_t>(n_list) * n_layers * per;
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < total;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t e = i % per, rest = i / per;
    const int64_t l = rest % n_layers, k = rest / n_layers;
    const int64_t base = (l * n_pages + pages[k]) * page_elems + 4 * e;
    const float4 gr = *reinterpret_cast<const float4*>(grad + base);
    uint2 raw = *reinterpret_cast<const uint2*>(kv + base);
    const float2 a = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&raw.x));
    const float2 c = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&raw.y));
    const __nv_bfloat162 na = __floats2bfloat162_rn(a.x - eta * gr.x, a.y - eta * gr.y);
    const __nv_bfloat162 nc = __floats2bfloat162_rn(c.x - eta * gr.z, c.y - eta * gr.w);
    raw.x = *reinterpret_cast<const uint32_t*>(&na);
    raw.y = *reinterpret_cast<const uint32_t*>(&nc);
    *reinterpret_cast<uint2*>(kv + base) = raw;
  }
}

// Launch with programmatic dependent launch: the kernel may start while the previous one in the
// stream drains; every kernel here waits (griddepcontrol.wait) before touching what that one writes.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, std::forward<Args>(args)...);
}

unsigned grid_1d(int64_t total, int threads) {
  int64_t b = (total + threads - 1) / threads;
  if (b > 152 * 16) b = 152 * 16;
  return static_cast<unsigned>(b < 1 ? 1 : b);
}

}  // namespace

cudaError_t launch_transpose(const __nv_bfloat16* in, __nv_bfloat16* out, int rows, int cols, cudaStream_t st) {
  const dim3 grid((cols + 31) / 32, (rows + 31) / 32);
  if (grid.y > 65535u) return cudaErrorInvalidValue;
  transpose_kernel<<<grid, dim3(32, 8), 0, st>>>(in, out, rows, cols);
  return cudaGetLastError();
}

cudaError_t launch_head_back(const float* h, const float* p_plus, const __nv_bfloat16* gain,
                             const __nv_bfloat16* w_plus, const __nv_bfloat16* w_minus, int n, int d, float eps,
                             float* dh, __nv_bfloat16* dh_hi, __nv_bfloat16* dh_lo, cudaStream_t st) {
  return launch_pdl(head_back_kernel, dim3(n), dim3(256), 0, st, h, p_plus, gain, w_plus, w_minus, d, eps, dh, dh_hi,
                    dh_lo);
}

cudaError_t launch_rms_back(const float* h, const __nv_bfloat16* h_bf16, const __nv_bfloat16* gain, const float* dy,
                            const float* dres, int n, int d, float eps, float* out, __nv_bfloat16* o_hi,
                            __nv_bfloat16* o_lo, cudaStream_t st) {
  return launch_pdl(rms_back_kernel, dim3(n), dim3(256), 0, st, h, h_bf16, gain, dy, dres, d, eps, out, o_hi, o_lo);
}

cudaError_t launch_silu_back(const float* da, const float* gu, int n, int ff, __nv_bfloat16* o_hi,
                             __nv_bfloat16* o_lo, cudaStream_t st) {
  return launch_pdl(silu_back_kernel, dim3(grid_1d(static_cast<int64_t>(n) * ff, 256)), dim3(256), 0, st, da, gu, n,
                    ff, o_hi, o_lo);
}

cudaError_t launch_attn_back(const AttnBackArgs& a, cudaStream_t st) {
  if (a.n_q / a.n_kv > kMaxGroup || (a.hd != 64 && a.hd != 128)) return cudaErrorInvalidValue;
  cudaError_t e = launch_pdl(attn_back_pre_kernel, dim3(a.n * a.n_kv), dim3(128), 0, st, a.q, a.kself, a.vself, a.o,
                             a.dout, a.lse, a.n_q, a.n_kv, a.hd, a.D, a.dq, a.dks, a.dvs);
  if (e != cudaSuccess || a.n_units == 0) return e;
  const int G = a.n_q / a.n_kv;
  if (G <= 8 && a.tm_pool) {   // the tensor-core backward
    if (a.hd == 128)
      return launch_pdl(attn_back_tc_kernel<128>, dim3(a.n_units), dim3(128), BackTcSmem<128>::kBytes, st, *a.tm_pool,
                        a.layer_page0, a.units, a.seq_lens, a.block_table, a.max_blocks, a.shared, a.q, a.dout, a.lse,
                        a.D, a.n_q, a.n_kv, a.grad_layer, a.dq, a.err);
    return launch_pdl(attn_back_tc_kernel<64>, dim3(a.n_units), dim3(128), BackTcSmem<64>::kBytes, st, *a.tm_pool,
                      a.layer_page0, a.units, a.seq_lens, a.block_table, a.max_blocks, a.shared, a.q, a.dout, a.lse,
                      a.D, a.n_q, a.n_kv, a.grad_layer, a.dq, a.err);
  }
  const size_t smem = a.hd == 128 ? back_pages_smem<128>() : back_pages_smem<64>();
  cudaError_t le = cudaSuccess;
  auto go = [&](auto kern) {
    le = launch_pdl(kern, dim3(a.n_units), dim3(128), smem, st, a.units, a.seq_lens, a.block_table, a.max_blocks,
                    a.pool_layer, a.shared, a.q, a.dout, a.lse, a.D, a.n_q, a.n_kv, a.grad_layer, a.dq, a.err);
  };
  if (a.hd == 128) {
    if (G <= 4)
      go(attn_back_pages_kernel<128, 4>);
    else if (G <= 8)
      go(attn_back_pages_kernel<128, 8>);
    else
      go(attn_back_pages_kernel<128, 16>);
  } else {
    if (G <= 4)
      go(attn_back_pages_kernel<64, 4>);
    else if (G <= 8)
      go(attn_back_pages_kernel<64, 8>);
    else
      go(attn_back_pages_kernel<64, 16>);
  }
  return le;
}

cudaError_t grad_configure() {
  cudaError_t e = cudaSuccess;
  auto set = [&](auto kern, size_t bytes) {
    if (e == cudaSuccess) e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(bytes));
  };
  set(attn_back_pages_kernel<128, 4>, back_pages_smem<128>());
  set(attn_back_pages_kernel<128, 8>, back_pages_smem<128>());
  set(attn_back_pages_kernel<128, 16>, back_pages_smem<128>());
  set(attn_back_pages_kernel<64, 4>, back_pages_smem<64>());
  set(attn_back_pages_kernel<64, 8>, back_pages_smem<64>());
  set(attn_back_pages_kernel<64, 16>, back_pages_smem<64>());
  set(attn_back_tc_kernel<128>, BackTcSmem<128>::kBytes);
  set(attn_back_tc_kernel<64>, BackTcSmem<64>::kBytes);
  return e;
}

cudaError_t launch_rope_back(const float* dq, const float* dks, const float* dvs, const float2* rope, int n, int n_q,
                             int n_kv, int hd, __nv_bfloat16* o_hi, __nv_bfloat16* o_lo, cudaStream_t st) {
  return launch_pdl(rope_back_kernel, dim3(n), dim3(256), 0, st, dq, dks, dvs, rope, n_q, n_kv, hd, o_hi, o_lo);
}

cudaError_t launch_zero_pages(float* grad, const int32_t* pages, int n_list, int n_layers, int64_t n_pages,
                              int64_t page_elems, cudaStream_t st) {
  if (n_list == 0) return cudaSuccess;
  return launch_pdl(zero_pages_kernel, dim3(grid_1d(static_cast<int64_t>(n_list) * n_layers * (page_elems / 4), 256)),
                    dim3(256), 0, st, grad, pages, n_list, n_layers, n_pages, page_elems);
}

cudaError_t launch_steer_update(__nv_bfloat16* kv, const float* grad, const int32_t* pages, int n_list, int n_layers,
                                int64_t n_pages, int64_t page_elems, float eta, cudaStream_t st) {
  if (n_list == 0) return cudaSuccess;
  return launch_pdl(steer_update_kernel, dim3(grid_1d(static_cast<int64_t>(n_list) * n_layers * (page_elems / 4), 256)),
                    dim3(256), 0, st, kv, grad, pages, n_list, n_layers, n_pages, page_elems, eta);
}

}  // namespace kvprm
