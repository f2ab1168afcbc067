// Paged GQA decode attention for the verify token (App. A.3 read-out,
// head = softmax(q^T K / sqrt(d_k)) V, one query per head, k = 1 of Def. 1),
// split-K over the cache ("flash decoding") plus a combine kernel that merges
// the splits together with the verify token's own key/value.
//
// Split kernel, one CTA per (split, kv head, candidate), 5 warps:
//  - warp 4 (producer) copies the CTA's block-table slice to shared memory and
//    streams K and V pages with TMA (tiled, 128-byte swizzle) into a 3-stage
//    ring, 4 pages (64 tokens) per stage, one mbarrier pair per slot;
//  - warps 0..3 (consumers) each take one page of a stage: S = Q K^T on the
//    tensor cores (mma.m16n8k16), an online softmax in fp32 registers with
//    quad shuffles, then O += P V.  The query and the probabilities enter the
//    bf16 MMAs as (hi, lo) pairs so both keep ~16 bits: with G <= 8 query
//    heads per group the hi parts fill MMA rows 0..7 and the lo parts rows
//    8..15 of the same instruction (their results are summed), so the split
//    costs no extra MMAs; with 8 < G <= 16 hi and lo take one MMA each;
//  - the four warps' (m, l, O) are merged in shared memory and written as one
//    unnormalised split partial;
//  - the last CTA of a (candidate, kv head) to finish (an atomic arrival
//    counter, no waiting) merges that group's splits together with the verify
//    token's own entry and writes the attention output as a bf16 (hi, lo)
//    pair for the O projection.
// All scores are kept in log2 units (scaled by log2(e) / sqrt(hd)).
#include <cuda_bf16.h>

#include "kernels.h"
#include "ptx.cuh"

namespace kvprm {

namespace {

constexpr int kPagesPerStage = 4;
constexpr int kStages = 3;
constexpr int kConsumerWarps = 4;
constexpr int kThreads = (kConsumerWarps + 1) * 32;
constexpr float kLog2e = 1.4426950408889634f;

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~static_cast<uintptr_t>(1023));
}

// Physical page of logical page `j` of candidate `b` (the block-table walk;
// also used by the resolve entry point so indexing can be checked bit-exactly).
__device__ __forceinline__ int32_t phys_page(const int32_t* __restrict__ bt, int b, int max_blocks, int j) {
  return bt[static_cast<int64_t>(b) * max_blocks + j];
}

// Merge the ns split partials of every query head of group g of candidate b
// with the verify token's own entry s_self = q . k_self / sqrt(hd):
//   M = max(m_i, s_self), o = (sum_i 2^(m_i - M) o_i + 2^(s_self - M) v_self)
//                             / (sum_i 2^(m_i - M) l_i + 2^(s_self - M)),
// summed in split order.  One warp per head (5 warps, heads strided).
template <int HD>
__device__ __forceinline__ void merge_group(int b, int g, int n_q, int n_kv, int group, int ns, int n_split,
                                            const float* __restrict__ part_o, const float* __restrict__ part_ml,
                                            const AttnMerge& mg) {
  constexpr int kPer = HD / 32;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t hk = static_cast<int64_t>(b) * n_kv + g;
  for (int r = warp; r < group; r += kThreads / 32) {
    const int64_t hq = static_cast<int64_t>(b) * n_q + static_cast<int64_t>(g) * group + r;
    float qv[kPer], vv[kPer];
    float dot = 0.f;
#pragma unroll
    for (int j = 0; j < kPer; ++j) {
      const int d = lane + 32 * j;
      qv[j] = mg.q[hq * HD + d];
      dot += qv[j] * mg.kself[hk * HD + d];
      vv[j] = mg.vself[hk * HD + d];
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) dot += __shfl_xor_sync(0xffffffffu, dot, off);
    const float s_self = dot * (kLog2e * rsqrtf(static_cast<float>(HD)));
    const float mi = lane < ns ? __ldcg(part_ml + (hq * n_split + lane) * 2) : -INFINITY;
    const float li = lane < ns ? __ldcg(part_ml + (hq * n_split + lane) * 2 + 1) : 0.f;
    float M = fmaxf(mi, s_self);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
    const float wi = lane < ns ? exp2f(mi - M) : 0.f;
    const float wself = exp2f(s_self - M);
    float lsum = wself;
    for (int i = 0; i < ns; ++i) lsum += __shfl_sync(0xffffffffu, wi * li, i);
    const float inv = 1.0f / lsum;
    float acc[kPer];
#pragma unroll
    for (int j = 0; j < kPer; ++j) acc[j] = wself * vv[j];
    const float* po = part_o + hq * n_split * HD + lane;
    for (int i = 0; i < ns; ++i) {
      const float w = __shfl_sync(0xffffffffu, wi, i);
#pragma unroll
      for (int j = 0; j < kPer; ++j) acc[j] += w * __ldcg(po + i * HD + 32 * j);
    }
#pragma unroll
    for (int j = 0; j < kPer; ++j) {
      const int d = lane + 32 * j;
      const float out = acc[j] * inv;
      const __nv_bfloat16 hi = __float2bfloat16_rn(out);
      mg.o_hi[hq * HD + d] = hi;
      mg.o_lo[hq * HD + d] = __float2bfloat16_rn(out - __bfloat162float(hi));
      if (mg.out_f32) mg.out_f32[hq * HD + d] = out;
      if (mg.dbg) mg.dbg[hq * HD + d] = out;
    }
  }
}

template <int HD, bool TWO_ROWS>
__global__ void __launch_bounds__(kThreads) attn_split_kernel(
    const __grid_constant__ CUtensorMap tm_pool, int64_t layer_row0, const int32_t* __restrict__ bt,
    const int32_t* __restrict__ seq_lens, const __nv_bfloat16* __restrict__ q_hi,
    const __nv_bfloat16* __restrict__ q_lo, int n_q, int n_kv, int group, int max_blocks, int pages_per_split,
    int n_split, float* __restrict__ part_o, float* __restrict__ part_ml, AttnMerge mg, int* err,
    unsigned long long* ts) {
  trace_begin(ts);
  constexpr int kSub = HD / 64;                       // 64-column sub-tiles per row
  constexpr uint32_t kBlockBytes = kSub * 16 * 128;   // one K (or V) page of one kv head
  constexpr uint32_t kPageBytes = 2 * kBlockBytes;
  constexpr uint32_t kStageBytes = kPagesPerStage * kPageBytes;

  extern __shared__ uint8_t smem_raw[];
  uint8_t* ring = align1024(smem_raw);
  uint64_t* full = reinterpret_cast<uint64_t*>(ring + kStages * kStageBytes);
  uint64_t* empty = full + kStages;
  int32_t* bt_s = reinterpret_cast<int32_t*>(empty + kStages);

  const int split = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
  const int L = seq_lens[b];
  const int n_pages_b = (L + 15) >> 4;
  const int p0 = split * pages_per_split;
  const int p1 = min(n_pages_b, p0 + pages_per_split);
  if (p0 >= p1) {
    grid_dep_wait();
    if (n_pages_b == 0 && split == 0) merge_group<HD>(b, g, n_q, n_kv, group, 0, n_split, part_o, part_ml, mg);
    trace_end(ts);
    return;
  }
  const int np = p1 - p0;
  const int n_stages = (np + kPagesPerStage - 1) / kPagesPerStage;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], kConsumerWarps);
    }
    fence_mbar_init();
  }
  if (warp == kConsumerWarps) {
    for (int i = lane; i < np; i += 32) bt_s[i] = phys_page(bt, b, max_blocks, p0 + i);
  }
  __syncthreads();
  grid_dep_launch();   // the next kernel may start; it waits for this grid before reading its output

  const int gid = lane >> 2, tig = lane & 3;
  float m_run[2] = {-INFINITY, -INFINITY};
  float l_run[2] = {0.f, 0.f};
  float o[HD / 8][4];
#pragma unroll
  for (int n = 0; n < HD / 8; ++n) o[n][0] = o[n][1] = o[n][2] = o[n][3] = 0.f;

  if (warp == kConsumerWarps) {
    // ------------------------------------------------ producer
    if (lane == 0) {
      tma_prefetch_desc(&tm_pool);
      const uint64_t pol = policy_evict_first();
      for (int u = 0; u < n_stages; ++u) {
        const int slot = u % kStages;
        const uint32_t use = static_cast<uint32_t>(u / kStages);
        if (u >= kStages && !mbar_wait(&empty[slot], (use & 1u) ^ 1u, err)) break;
        const int npg = min(kPagesPerStage, np - u * kPagesPerStage);
        mbar_arrive_expect_tx(&full[slot], static_cast<uint32_t>(npg) * kPageBytes);
        uint8_t* st = ring + slot * kStageBytes;
        for (int pi = 0; pi < npg; ++pi) {
          const int64_t phys = bt_s[u * kPagesPerStage + pi];
          const int32_t row_k = static_cast<int32_t>(layer_row0 + (phys * 2 * n_kv + g) * 16);
          const int32_t row_v = row_k + n_kv * 16;
#pragma unroll
          for (int sub = 0; sub < kSub; ++sub) {
            tma_load_2d(st + pi * kPageBytes + sub * 2048, &tm_pool, &full[slot], sub * 64, row_k, pol);
            tma_load_2d(st + pi * kPageBytes + kBlockBytes + sub * 2048, &tm_pool, &full[slot], sub * 64, row_v,
                        pol);
          }
        }
      }
    }
  } else {
    // ------------------------------------------------ consumers
    grid_dep_wait();   // q is written by the preceding kernel
    const int64_t q0 = (static_cast<int64_t>(b) * n_q + static_cast<int64_t>(g) * group) * HD;
    const __nv_bfloat16* qh = q_hi + q0;
    const __nv_bfloat16* ql = q_lo + q0;
    auto ldq = [&](const __nv_bfloat16* base, int row, int col) -> uint32_t {
      return row < group ? *reinterpret_cast<const uint32_t*>(base + row * HD + col) : 0u;
    };
    // A fragments of Q.  Packed (G <= 8): rows 0..7 = hi, rows 8..15 = lo of
    // the same heads.  Two-row (G > 8): a hi and a lo fragment over 16 heads.
    uint32_t qa0[HD / 16], qa1[HD / 16], qa2[HD / 16], qa3[HD / 16];
    uint32_t qb0[HD / 16], qb1[HD / 16], qb2[HD / 16], qb3[HD / 16];
#pragma unroll
    for (int ks = 0; ks < HD / 16; ++ks) {
      const int c = ks * 16 + tig * 2;
      if (!TWO_ROWS) {
        qa0[ks] = ldq(qh, gid, c);
        qa1[ks] = ldq(ql, gid, c);
        qa2[ks] = ldq(qh, gid, c + 8);
        qa3[ks] = ldq(ql, gid, c + 8);
        qb0[ks] = qb1[ks] = qb2[ks] = qb3[ks] = 0u;
      } else {
        qa0[ks] = ldq(qh, gid, c);
        qa1[ks] = ldq(qh, gid + 8, c);
        qa2[ks] = ldq(qh, gid, c + 8);
        qa3[ks] = ldq(qh, gid + 8, c + 8);
        qb0[ks] = ldq(ql, gid, c);
        qb1[ks] = ldq(ql, gid + 8, c);
        qb2[ks] = ldq(ql, gid, c + 8);
        qb3[ks] = ldq(ql, gid + 8, c + 8);
      }
    }
    const float sl2 = kLog2e * rsqrtf(static_cast<float>(HD));

    for (int u = 0; u < n_stages; ++u) {
      const int slot = u % kStages;
      const uint32_t use = static_cast<uint32_t>(u / kStages);
      if (!__all_sync(0xffffffffu, mbar_wait(&full[slot], use & 1u, err))) break;
      const int pg = u * kPagesPerStage + warp;
      if (pg < np) {
        const int valid = min(16, L - (p0 + pg) * 16);
        const uint32_t kbase = smem_u32(ring + slot * kStageBytes + pg % kPagesPerStage * kPageBytes);
        const uint32_t vbase = kbase + kBlockBytes;
        // S = Q K^T for the page's 16 tokens (two n-tiles of 8 tokens)
        float s0[4] = {0.f, 0.f, 0.f, 0.f}, s1[4] = {0.f, 0.f, 0.f, 0.f};
        {
          const int mi = lane >> 3, r = lane & 7;
          const int tok = (mi >> 1) * 8 + r;
#pragma unroll
          for (int ks = 0; ks < HD / 16; ++ks) {
            const int hdc = ks * 16 + (mi & 1) * 8;
            const uint32_t addr = kbase + (hdc >> 6) * 2048 + tok * 128 + ((((hdc & 63) >> 3) ^ (tok & 7)) << 4);
            uint32_t b0, b1, b2, b3;
            ldsm_x4(addr, b0, b1, b2, b3);
            mma_bf16_16816(s0, qa0[ks], qa1[ks], qa2[ks], qa3[ks], b0, b1);
            mma_bf16_16816(s1, qa0[ks], qa1[ks], qa2[ks], qa3[ks], b2, b3);
            if (TWO_ROWS) {
              mma_bf16_16816(s0, qb0[ks], qb1[ks], qb2[ks], qb3[ks], b0, b1);
              mma_bf16_16816(s1, qb0[ks], qb1[ks], qb2[ks], qb3[ks], b2, b3);
            }
          }
        }
        const int t0 = tig * 2, t1 = tig * 2 + 1, t2 = 8 + tig * 2, t3 = 9 + tig * 2;
        // per-thread scores of its row(s): x[r][token slot]
        float x[2][4];
        if (!TWO_ROWS) {   // hi (row gid) + lo (row gid + 8) parts of the same head
          x[0][0] = s0[0] + s0[2];
          x[0][1] = s0[1] + s0[3];
          x[0][2] = s1[0] + s1[2];
          x[0][3] = s1[1] + s1[3];
        } else {
          x[0][0] = s0[0];
          x[0][1] = s0[1];
          x[0][2] = s1[0];
          x[0][3] = s1[1];
          x[1][0] = s0[2];
          x[1][1] = s0[3];
          x[1][2] = s1[2];
          x[1][3] = s1[3];
        }
        uint32_t ph[4], pl[4];   // A fragments of P: hi / lo
#pragma unroll
        for (int r = 0; r < (TWO_ROWS ? 2 : 1); ++r) {
          x[r][0] = t0 < valid ? x[r][0] * sl2 : -INFINITY;
          x[r][1] = t1 < valid ? x[r][1] * sl2 : -INFINITY;
          x[r][2] = t2 < valid ? x[r][2] * sl2 : -INFINITY;
          x[r][3] = t3 < valid ? x[r][3] * sl2 : -INFINITY;
          float mx = fmaxf(fmaxf(x[r][0], x[r][1]), fmaxf(x[r][2], x[r][3]));
          mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
          mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
          const float m_new = fmaxf(m_run[r], mx);
          const float alpha = exp2f(m_run[r] - m_new);
          float p[4];
#pragma unroll
          for (int i2 = 0; i2 < 4; ++i2) p[i2] = exp2f(x[r][i2] - m_new);
          l_run[r] = l_run[r] * alpha + ((p[0] + p[1]) + (p[2] + p[3]));
          m_run[r] = m_new;
          float hi[4], lo[4];
#pragma unroll
          for (int i2 = 0; i2 < 4; ++i2) {
            hi[i2] = __bfloat162float(__float2bfloat16_rn(p[i2]));
            lo[i2] = p[i2] - hi[i2];
          }
          if (!TWO_ROWS) {
            // one head per thread row: both MMA row halves rescale together
#pragma unroll
            for (int n = 0; n < HD / 8; ++n) {
              o[n][0] *= alpha;
              o[n][1] *= alpha;
              o[n][2] *= alpha;
              o[n][3] *= alpha;
            }
            ph[0] = pack_bf16(hi[0], hi[1]);   // row gid: P_hi
            ph[1] = pack_bf16(lo[0], lo[1]);   // row gid + 8: P_lo
            ph[2] = pack_bf16(hi[2], hi[3]);
            ph[3] = pack_bf16(lo[2], lo[3]);
          } else {
#pragma unroll
            for (int n = 0; n < HD / 8; ++n) {
              o[n][2 * r] *= alpha;
              o[n][2 * r + 1] *= alpha;
            }
            ph[r] = pack_bf16(hi[0], hi[1]);
            ph[r + 2] = pack_bf16(hi[2], hi[3]);
            pl[r] = pack_bf16(lo[0], lo[1]);
            pl[r + 2] = pack_bf16(lo[2], lo[3]);
          }
        }
        // O += P V  (V^T fragments through ldmatrix.trans)
        {
          const int mi = lane >> 3;
          const int tok = (mi & 1) * 8 + (lane & 7);
#pragma unroll
          for (int j2 = 0; j2 < HD / 16; ++j2) {
            const int hdc = j2 * 16 + (mi >> 1) * 8;
            const uint32_t addr = vbase + (hdc >> 6) * 2048 + tok * 128 + ((((hdc & 63) >> 3) ^ (tok & 7)) << 4);
            uint32_t b0, b1, b2, b3;
            ldsm_x4_t(addr, b0, b1, b2, b3);
            mma_bf16_16816(o[2 * j2], ph[0], ph[1], ph[2], ph[3], b0, b1);
            mma_bf16_16816(o[2 * j2 + 1], ph[0], ph[1], ph[2], ph[3], b2, b3);
            if (TWO_ROWS) {
              mma_bf16_16816(o[2 * j2], pl[0], pl[1], pl[2], pl[3], b0, b1);
              mma_bf16_16816(o[2 * j2 + 1], pl[0], pl[1], pl[2], pl[3], b2, b3);
            }
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty[slot]);
    }
    if (!TWO_ROWS) {   // fold the lo-part rows onto their heads
#pragma unroll
      for (int n = 0; n < HD / 8; ++n) {
        o[n][0] += o[n][2];
        o[n][1] += o[n][3];
      }
    }
    // quad-reduce the row sums
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      l_run[r] += __shfl_xor_sync(0xffffffffu, l_run[r], 1);
      l_run[r] += __shfl_xor_sync(0xffffffffu, l_run[r], 2);
    }
  }
  // all stages consumed (every issued copy was waited for): reuse the ring for the merge
  __syncthreads();
  if (warp < kConsumerWarps) {
    float* mo = reinterpret_cast<float*>(ring);                 // [4][16][HD]
    float* mm = mo + kConsumerWarps * 16 * HD;                  // [4][16]
    float* ml = mm + kConsumerWarps * 16;                       // [4][16]
#pragma unroll
    for (int r = 0; r < (TWO_ROWS ? 2 : 1); ++r) {
      const int row = gid + 8 * r;
      if (row < group) {
#pragma unroll
        for (int n = 0; n < HD / 8; ++n) {
          mo[(warp * 16 + row) * HD + n * 8 + tig * 2] = o[n][2 * r];
          mo[(warp * 16 + row) * HD + n * 8 + tig * 2 + 1] = o[n][2 * r + 1];
        }
        if (tig == 0) {
          mm[warp * 16 + row] = m_run[r];
          ml[warp * 16 + row] = l_run[r];
        }
      }
    }
  }
  __syncthreads();
  grid_dep_wait();
  {
    const float* mo = reinterpret_cast<const float*>(ring);
    const float* mm = mo + kConsumerWarps * 16 * HD;
    const float* ml = mm + kConsumerWarps * 16;
    for (int idx = threadIdx.x; idx < group * HD; idx += kThreads) {
      const int row = idx / HD, d = idx - row * HD;
      float M = -INFINITY;
#pragma unroll
      for (int w = 0; w < kConsumerWarps; ++w) M = fmaxf(M, mm[w * 16 + row]);
      float acc = 0.f, lsum = 0.f;
#pragma unroll
      for (int w = 0; w < kConsumerWarps; ++w) {
        const float mw = mm[w * 16 + row];
        const float f = (mw == -INFINITY) ? 0.f : exp2f(mw - M);
        acc += f * mo[(w * 16 + row) * HD + d];
        lsum += f * ml[w * 16 + row];
      }
      const int64_t hq = static_cast<int64_t>(b) * n_q + static_cast<int64_t>(g) * group + row;
      part_o[(hq * n_split + split) * HD + d] = acc;
      if (d == 0) {
        part_ml[(hq * n_split + split) * 2 + 0] = M;
        part_ml[(hq * n_split + split) * 2 + 1] = lsum;
      }
    }
  }
  // the last split of this (candidate, kv head) to arrive merges all of them
  __shared__ int s_last;
  __threadfence();
  __syncthreads();
  const int ns_b = (n_pages_b + pages_per_split - 1) / pages_per_split;
  if (threadIdx.x == 0) s_last = atomicAdd(&mg.counter[b * n_kv + g], 1) == ns_b - 1;
  __syncthreads();
  if (s_last) {
    __threadfence();
    merge_group<HD>(b, g, n_q, n_kv, group, ns_b, n_split, part_o, part_ml, mg);
    if (threadIdx.x == 0) mg.counter[b * n_kv + g] = 0;   // ready for the next layer
  }
  trace_end(ts);
}

__global__ void resolve_kernel(const int32_t* __restrict__ bt, const int32_t* __restrict__ seq_lens, int max_blocks,
                               int b, int64_t* __restrict__ out) {
  const int L = seq_lens[b];
  for (int j = blockIdx.x * blockDim.x + threadIdx.x; j < L; j += gridDim.x * blockDim.x)
    out[j] = static_cast<int64_t>(phys_page(bt, b, max_blocks, j >> 4)) * 16 + (j & 15);
}

template <typename K>
cudaError_t set_smem(K kernel) {
  return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
}

}  // namespace

AttnPlan plan_attention(const AttnShape& s, int n_cand, int max_pages, int num_sms, int split_cap) {
  AttnPlan p;
  const int pairs = n_cand * s.n_kv;
  const int target = 2 * num_sms;   // one wave at two CTAs per SM: every CTA can prefetch before q is ready
  int ns = target / (pairs > 0 ? pairs : 1);
  if (ns < 1) ns = 1;
  if (ns > split_cap) ns = split_cap;
  if (max_pages < 1) max_pages = 1;
  if (ns > max_pages) ns = max_pages;
  p.pages_per_split = (max_pages + ns - 1) / ns;
  p.n_split = (max_pages + p.pages_per_split - 1) / p.pages_per_split;
  const size_t stage = static_cast<size_t>(kPagesPerStage) * 2 * (s.hd / 64) * 2048;
  p.smem_bytes = kStages * stage + 1024 + 2 * kStages * 8 + static_cast<size_t>(p.pages_per_split) * 4 + 64;
  return p;
}

cudaError_t attention_configure() {
  cudaError_t e;
  if ((e = set_smem(attn_split_kernel<64, false>)) != cudaSuccess) return e;
  if ((e = set_smem(attn_split_kernel<64, true>)) != cudaSuccess) return e;
  if ((e = set_smem(attn_split_kernel<128, false>)) != cudaSuccess) return e;
  return set_smem(attn_split_kernel<128, true>);
}

static cudaLaunchConfig_t make_cfg(dim3 grid, dim3 block, size_t smem, cudaStream_t st, cudaLaunchAttribute* attr,
                                   bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cfg;
}

cudaError_t launch_attn_split(const AttnShape& s, const AttnPlan& p, const CUtensorMap* tm_pool, int layer,
                              const int32_t* bt, const int32_t* seq_lens, const __nv_bfloat16* q_hi,
                              const __nv_bfloat16* q_lo, int n_cand, float* part_o, float* part_ml,
                              const AttnMerge& mg, int* err, cudaStream_t stream, bool pdl, unsigned long long* ts) {
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg =
      make_cfg(dim3(p.n_split, s.n_kv, n_cand), dim3(kThreads), p.smem_bytes, stream, attr, pdl);
  const int64_t row0 = static_cast<int64_t>(layer) * s.layer_rows;
  const bool two = s.group > 8;
  if (s.hd == 128) {
    if (two)
      return cudaLaunchKernelEx(&cfg, attn_split_kernel<128, true>, *tm_pool, row0, bt, seq_lens, q_hi, q_lo, s.n_q, s.n_kv,
                                s.group, s.max_blocks, p.pages_per_split, p.n_split, part_o, part_ml, mg, err, ts);
    return cudaLaunchKernelEx(&cfg, attn_split_kernel<128, false>, *tm_pool, row0, bt, seq_lens, q_hi, q_lo, s.n_q, s.n_kv,
                              s.group, s.max_blocks, p.pages_per_split, p.n_split, part_o, part_ml, mg, err, ts);
  }
  if (two)
    return cudaLaunchKernelEx(&cfg, attn_split_kernel<64, true>, *tm_pool, row0, bt, seq_lens, q_hi, q_lo, s.n_q, s.n_kv,
                              s.group, s.max_blocks, p.pages_per_split, p.n_split, part_o, part_ml, mg, err, ts);
  return cudaLaunchKernelEx(&cfg, attn_split_kernel<64, false>, *tm_pool, row0, bt, seq_lens, q_hi, q_lo, s.n_q, s.n_kv,
                            s.group, s.max_blocks, p.pages_per_split, p.n_split, part_o, part_ml, mg, err, ts);
}

cudaError_t launch_resolve(const int32_t* bt, const int32_t* seq_lens, int max_blocks, int b, int64_t* out,
                           cudaStream_t stream) {
  resolve_kernel<<<64, 256, 0, stream>>>(bt, seq_lens, max_blocks, b, out);
  return cudaGetLastError();
}

}  // namespace kvprm
