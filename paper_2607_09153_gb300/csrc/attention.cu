// Paged GQA decode attention for the verify token (App. A.3 read-out,
// head = softmax(q^T K / sqrt(d_k)) V, one query per head, k = 1 of Def. 1),
// split over the cache ("flash decoding"), with the splits merged together
// with the verify token's own key/value.
//
// The work is a list of items built on the host from the block tables
// (build_attn_work), one CTA per (item, kv head), 9 warps:
//  - warp 8 (producer) copies the item's physical page ids to shared memory
//    and streams K and V pages with TMA (tiled, 128-byte swizzle) into a
//    3-stage ring of 8 pages (128 tokens) per stage -- starting before the
//    query is ready, since the cache does not depend on it;
//  - a *private* item holds pages of one candidate: consumer warp w scores
//    page w of every stage, and the eight warps' (m, l, O) are merged in
//    shared memory into one partial;
//  - a *shared* item holds pages that several candidates reference (a beam
//    prefix, an MCTS ancestor): each page is loaded once and consumer warp w
//    scores it for candidate w (up to 8), writing its own partial.  Attention
//    is invariant to the order of the keys, so shared pages need not sit at
//    the same positions in the candidates' sequences;
//  - per page and warp: S = Q K^T on the tensor cores (mma.m16n8k16), an
//    online softmax in fp32 registers with quad shuffles, then O += P V.  The
//    query and the probabilities enter the bf16 MMAs as (hi, lo) pairs so both
//    keep ~16 bits: with G <= 8 query heads per group the hi parts fill MMA
//    rows 0..7 and the lo parts rows 8..15 of the same instruction (summed
//    afterwards), so the split costs no extra MMAs; with 8 < G <= 16 hi and lo
//    take one MMA each;
//  - every partial lands in a slot of its candidate; the last arrival per
//    (candidate, kv head) (an atomic counter, no waiting) merges the slots with
//    the self entry and writes the attention output as a bf16 (hi, lo) pair
//    for the O projection.
// All scores are kept in log2 units (scaled by log2(e) / sqrt(hd)).
#include <cuda_bf16.h>

#include <algorithm>
#include <unordered_map>
#include <vector>

#include "kernels.h"
#include "ptx.cuh"

namespace kvprm {

namespace {

constexpr int kPagesPerStage = 8;
constexpr int kStages = 3;
constexpr int kConsumerWarps = 8;
constexpr int kThreads = (kConsumerWarps + 1) * 32;
constexpr float kLog2e = 1.4426950408889634f;

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~static_cast<uintptr_t>(1023));
}

// Physical page of logical page `j` of candidate `b` (the block-table walk
// used by the resolve entry point, so indexing can be checked bit-exactly).
__device__ __forceinline__ int32_t phys_page(const int32_t* __restrict__ bt, int b, int max_blocks, int j) {
  return bt[static_cast<int64_t>(b) * max_blocks + j];
}

// Merge the ns partial slots of every query head of group g of candidate b
// with the verify token's own entry s_self = q . k_self / sqrt(hd):
//   M = max(m_i, s_self), o = (sum_i 2^(m_i - M) o_i + 2^(s_self - M) v_self)
//                             / (sum_i 2^(m_i - M) l_i + 2^(s_self - M)),
// summed in slot order.  Warps w0, w0 + nw, ... take one head each.
template <int HD>
__device__ __forceinline__ void merge_group(int b, int g, int n_q, int n_kv, int group, int ns, int stride,
                                            const float* __restrict__ part_o, const float* __restrict__ part_ml,
                                            const AttnMerge& mg, int w0, int nw) {
  constexpr int kPer = HD / 32;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t hk = static_cast<int64_t>(b) * n_kv + g;
  for (int r = warp - w0; r < group; r += nw) {
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
    const float mi = lane < ns ? __ldcg(part_ml + (hq * stride + lane) * 2) : -INFINITY;
    const float li = lane < ns ? __ldcg(part_ml + (hq * stride + lane) * 2 + 1) : 0.f;
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
    const float* po = part_o + hq * stride * HD + lane;
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

// A fragments of one warp's query rows.
template <int HD>
struct WarpQ {
  uint32_t a0[HD / 16], a1[HD / 16], a2[HD / 16], a3[HD / 16];   // packed: rows hi / lo; two-row: hi
  uint32_t b0[HD / 16], b1[HD / 16], b2[HD / 16], b3[HD / 16];   // two-row: lo
};

template <int HD, bool TWO_ROWS>
__device__ __forceinline__ void load_q(WarpQ<HD>& q, const __nv_bfloat16* __restrict__ qh,
                                       const __nv_bfloat16* __restrict__ ql, int group, int lane) {
  const int gid = lane >> 2, tig = lane & 3;
  auto ldq = [&](const __nv_bfloat16* base, int row, int col) -> uint32_t {
    return row < group ? *reinterpret_cast<const uint32_t*>(base + row * HD + col) : 0u;
  };
#pragma unroll
  for (int ks = 0; ks < HD / 16; ++ks) {
    const int c = ks * 16 + tig * 2;
    if (!TWO_ROWS) {   // rows 0..7 = hi, rows 8..15 = lo of the same heads
      q.a0[ks] = ldq(qh, gid, c);
      q.a1[ks] = ldq(ql, gid, c);
      q.a2[ks] = ldq(qh, gid, c + 8);
      q.a3[ks] = ldq(ql, gid, c + 8);
      q.b0[ks] = q.b1[ks] = q.b2[ks] = q.b3[ks] = 0u;
    } else {           // a hi and a lo fragment over 16 heads
      q.a0[ks] = ldq(qh, gid, c);
      q.a1[ks] = ldq(qh, gid + 8, c);
      q.a2[ks] = ldq(qh, gid, c + 8);
      q.a3[ks] = ldq(qh, gid + 8, c + 8);
      q.b0[ks] = ldq(ql, gid, c);
      q.b1[ks] = ldq(ql, gid + 8, c);
      q.b2[ks] = ldq(ql, gid, c + 8);
      q.b3[ks] = ldq(ql, gid + 8, c + 8);
    }
  }
}

// Score one page (16 tokens, `valid` of them real) for one warp's query rows
// and fold it into the online softmax state.
template <int HD, bool TWO_ROWS>
__device__ __forceinline__ void process_page(const WarpQ<HD>& q, uint32_t kbase, uint32_t vbase, int valid, int lane,
                                             float (&m_run)[2], float (&l_run)[2], float (&o)[HD / 8][4]) {
  const int tig = lane & 3;
  const float sl2 = kLog2e * rsqrtf(static_cast<float>(HD));
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
      mma_bf16_16816(s0, q.a0[ks], q.a1[ks], q.a2[ks], q.a3[ks], b0, b1);
      mma_bf16_16816(s1, q.a0[ks], q.a1[ks], q.a2[ks], q.a3[ks], b2, b3);
      if (TWO_ROWS) {
        mma_bf16_16816(s0, q.b0[ks], q.b1[ks], q.b2[ks], q.b3[ks], b0, b1);
        mma_bf16_16816(s1, q.b0[ks], q.b1[ks], q.b2[ks], q.b3[ks], b2, b3);
      }
    }
  }
  const int t0 = tig * 2, t1 = tig * 2 + 1, t2 = 8 + tig * 2, t3 = 9 + tig * 2;
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
    if (!TWO_ROWS) {   // one head per thread row: both MMA row halves rescale together
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

template <int HD, bool TWO_ROWS>
__global__ void __launch_bounds__(kThreads, 1) attn_kernel(
    const __grid_constant__ CUtensorMap tm_pool, int64_t layer_row0, AttnWork wk,
    const __nv_bfloat16* __restrict__ q_hi, const __nv_bfloat16* __restrict__ q_lo, int n_q, int n_kv, int group,
    int stride, float* __restrict__ part_o, float* __restrict__ part_ml, AttnMerge mg, int* err,
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
  // no static shared memory: the dynamic request alone reaches the 227 KiB limit
  int* s_last_p = reinterpret_cast<int*>(empty + kStages);   // 16 B: merge decision of this CTA
  int32_t* pages_s = s_last_p + 4;

  const AttnItem it = wk.items[blockIdx.x];
  const int g = blockIdx.y;
  const bool shared = it.kind == 1;
  const int np = it.n_pages;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int gid = lane >> 2, tig = lane & 3;

  if (np == 0) {   // a candidate with an empty cache: the verify token attends to itself only
    grid_dep_launch();
    grid_dep_wait();
    merge_group<HD>(it.cand, g, n_q, n_kv, group, 0, stride, part_o, part_ml, mg, 0, kThreads / 32);
    trace_end(ts);
    return;
  }
  const int n_stages = (np + kPagesPerStage - 1) / kPagesPerStage;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], kConsumerWarps);
    }
    fence_mbar_init();
  }
  if (warp == kConsumerWarps)
    for (int i = lane; i < np; i += 32) pages_s[i] = wk.pages[it.page_off + i];
  __syncthreads();
  grid_dep_launch();   // the next kernel may start; it waits for this grid before reading its output

  float m_run[2] = {-INFINITY, -INFINITY};
  float l_run[2] = {0.f, 0.f};
  float o[HD / 8][4];
#pragma unroll
  for (int n = 0; n < HD / 8; ++n) o[n][0] = o[n][1] = o[n][2] = o[n][3] = 0.f;
  int cand = shared ? -1 : it.cand;   // the candidate this warp scores

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
          const int64_t phys = pages_s[u * kPagesPerStage + pi];
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
    if (shared) cand = warp < it.n_cands ? wk.cands[it.cand + warp] : -1;
    grid_dep_wait();   // q is written by the preceding kernel
    WarpQ<HD> q;
    if (cand >= 0) {
      const int64_t q0 = (static_cast<int64_t>(cand) * n_q + static_cast<int64_t>(g) * group) * HD;
      load_q<HD, TWO_ROWS>(q, q_hi + q0, q_lo + q0, group, lane);
    }
    for (int u = 0; u < n_stages; ++u) {
      const int slot = u % kStages;
      const uint32_t use = static_cast<uint32_t>(u / kStages);
      if (!__all_sync(0xffffffffu, mbar_wait(&full[slot], use & 1u, err))) break;
      const uint32_t sbase = smem_u32(ring + slot * kStageBytes);
      const int npg = min(kPagesPerStage, np - u * kPagesPerStage);
      if (!shared) {   // page `warp` of this stage
        if (warp < npg) {
          const int pg = u * kPagesPerStage + warp;
          const int valid = pg == np - 1 ? it.last_valid : 16;
          const uint32_t kb = sbase + warp * kPageBytes;
          process_page<HD, TWO_ROWS>(q, kb, kb + kBlockBytes, valid, lane, m_run, l_run, o);
        }
      } else if (cand >= 0) {   // every page of this stage, for this warp's candidate
        for (int pi = 0; pi < npg; ++pi) {
          const int pg = u * kPagesPerStage + pi;
          const int valid = pg == np - 1 ? it.last_valid : 16;
          const uint32_t kb = sbase + pi * kPageBytes;
          process_page<HD, TWO_ROWS>(q, kb, kb + kBlockBytes, valid, lane, m_run, l_run, o);
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
#pragma unroll
    for (int r = 0; r < 2; ++r) {   // quad-reduce the row sums
      l_run[r] += __shfl_xor_sync(0xffffffffu, l_run[r], 1);
      l_run[r] += __shfl_xor_sync(0xffffffffu, l_run[r], 2);
    }
  }
  // all stages consumed (every issued copy was waited for)
  __syncthreads();
  grid_dep_wait();

  if (shared) {
    // each consumer warp owns one candidate's partial
    if (warp < kConsumerWarps && cand >= 0) {
      const int slot_id = wk.slots[it.slot + warp];
#pragma unroll
      for (int r = 0; r < (TWO_ROWS ? 2 : 1); ++r) {
        const int row = gid + 8 * r;
        if (row < group) {
          const int64_t hq = static_cast<int64_t>(cand) * n_q + static_cast<int64_t>(g) * group + row;
          float* dst = part_o + (hq * stride + slot_id) * HD;
#pragma unroll
          for (int n = 0; n < HD / 8; ++n) {
            dst[n * 8 + tig * 2] = o[n][2 * r];
            dst[n * 8 + tig * 2 + 1] = o[n][2 * r + 1];
          }
          if (tig == 0) {
            part_ml[(hq * stride + slot_id) * 2 + 0] = m_run[r];
            part_ml[(hq * stride + slot_id) * 2 + 1] = l_run[r];
          }
        }
      }
      __threadfence();
      __syncwarp();
      int last = 0;
      if (lane == 0) last = atomicAdd(&mg.counter[cand * n_kv + g], 1) == wk.nslots[cand] - 1;
      last = __shfl_sync(0xffffffffu, last, 0);
      if (last) {
        __threadfence();
        merge_group<HD>(cand, g, n_q, n_kv, group, wk.nslots[cand], stride, part_o, part_ml, mg, warp, 1);
        if (lane == 0) mg.counter[cand * n_kv + g] = 0;   // ready for the next layer
      }
    }
  } else {
    // merge the eight warps' states through shared memory into one partial
    float* mo = reinterpret_cast<float*>(ring);                 // [8][16][HD]
    float* mm = mo + kConsumerWarps * 16 * HD;                  // [8][16]
    float* ml = mm + kConsumerWarps * 16;                       // [8][16]
    if (warp < kConsumerWarps) {
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
      const int64_t hq = static_cast<int64_t>(cand) * n_q + static_cast<int64_t>(g) * group + row;
      part_o[(hq * stride + it.slot) * HD + d] = acc;
      if (d == 0) {
        part_ml[(hq * stride + it.slot) * 2 + 0] = M;
        part_ml[(hq * stride + it.slot) * 2 + 1] = lsum;
      }
    }
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) *s_last_p = atomicAdd(&mg.counter[cand * n_kv + g], 1) == wk.nslots[cand] - 1;
    __syncthreads();
    if (*s_last_p) {
      __threadfence();
      merge_group<HD>(cand, g, n_q, n_kv, group, wk.nslots[cand], stride, part_o, part_ml, mg, 0, kThreads / 32);
      if (threadIdx.x == 0) mg.counter[cand * n_kv + g] = 0;   // ready for the next layer
    }
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
  return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024);
}

uint64_t hash_list(const int32_t* v, int n) {
  uint64_t h = 1469598103934665603ull;
  for (int i = 0; i < n; ++i) {
    h ^= static_cast<uint32_t>(v[i]);
    h *= 1099511628211ull;
  }
  return h ^ static_cast<uint64_t>(n);
}

}  // namespace

size_t attention_smem_bytes(int hd, int max_item_pages) {
  const size_t stage = static_cast<size_t>(kPagesPerStage) * 2 * (hd / 64) * 2048;
  return kStages * stage + 1024 + 2 * kStages * 8 + 16 + static_cast<size_t>(max_item_pages) * 4 + 64;
}

int attention_max_item_pages(int hd) {
  const size_t fixed = attention_smem_bytes(hd, 0);
  return static_cast<int>((227 * 1024 - fixed) / 4);
}

// Host planner: split each candidate's private pages into items, and group the
// full pages that several candidates reference (each exactly once) by their
// exact candidate set into shared items of up to kConsumerWarps candidates.
// Items are sized so that about two waves of CTAs (one per SM) cover the work,
// counting a shared page as kConsumerWarps times the per-CTA work of a private
// one (every warp scores every page of a shared item).  Returns false when some
// candidate would need more than slot_cap partial slots at any item size.
bool build_attn_work(const int32_t* bt, const int32_t* sl, int n, int max_blocks, int n_kv, int hd, int num_sms,
                     int slot_cap, bool share, AttnWorkHost& w) {
  const int max_pages_item = attention_max_item_pages(hd);
  std::vector<int> np(n);
  int64_t total_refs = 0;
  for (int b = 0; b < n; ++b) {
    np[b] = (sl[b] + 15) / 16;
    total_refs += np[b];
  }
  // ---- shared pages: full pages referenced once each by >= 2 candidates
  std::vector<uint8_t> is_shared(static_cast<size_t>(n) * max_blocks, 0);
  std::vector<std::vector<int32_t>> group_cands, group_pages;
  if (share && total_refs > 0) {
    std::unordered_map<int32_t, std::vector<int32_t>> refs;   // page -> candidates (full refs)
    refs.reserve(static_cast<size_t>(total_refs));
    bool any_dup = false;
    for (int b = 0; b < n; ++b) {
      const int nfull = sl[b] / 16;
      for (int j = 0; j < nfull; ++j) {
        auto& v = refs[bt[static_cast<int64_t>(b) * max_blocks + j]];
        v.push_back(b);
        if (v.size() > 1) any_dup = true;
      }
    }
    if (any_dup) {
      std::unordered_map<uint64_t, int> gidx;
      std::unordered_map<int32_t, char> in_group;
      for (auto& kv : refs) {
        const std::vector<int32_t>& c = kv.second;
        if (c.size() < 2) continue;
        bool once = true;   // a candidate listing the page twice keeps it private
        for (size_t i = 1; i < c.size(); ++i)
          if (c[i] == c[i - 1]) once = false;   // candidates were appended in increasing order
        if (!once) continue;
        const uint64_t h = hash_list(c.data(), static_cast<int>(c.size()));
        auto itg = gidx.find(h);
        int gi;
        if (itg != gidx.end()) {
          if (group_cands[itg->second] != c) continue;   // hash collision: keep it private
          gi = itg->second;
        } else {
          gi = static_cast<int>(group_cands.size());
          gidx.emplace(h, gi);
          group_cands.push_back(c);
          group_pages.emplace_back();
        }
        group_pages[gi].push_back(kv.first);
        in_group[kv.first] = 1;
      }
      for (int b = 0; b < n; ++b) {
        const int nfull = sl[b] / 16;
        for (int j = 0; j < nfull; ++j)
          if (in_group.count(bt[static_cast<int64_t>(b) * max_blocks + j]))
            is_shared[static_cast<size_t>(b) * max_blocks + j] = 1;
      }
      for (auto& pgs : group_pages) std::sort(pgs.begin(), pgs.end());   // deterministic item contents
      // deterministic group order (the hash map's iteration order is not)
      std::vector<int> order(group_cands.size());
      for (size_t i = 0; i < order.size(); ++i) order[i] = static_cast<int>(i);
      std::sort(order.begin(), order.end(), [&](int a, int b2) {
        return group_pages[a].front() < group_pages[b2].front();
      });
      std::vector<std::vector<int32_t>> gc, gp;
      for (int i : order) {
        gc.push_back(std::move(group_cands[i]));
        gp.push_back(std::move(group_pages[i]));
      }
      group_cands.swap(gc);
      group_pages.swap(gp);
    }
  }
  // ---- cost model and item sizes
  int64_t priv_pages = 0, shared_units = 0;
  for (int b = 0; b < n; ++b)
    for (int j = 0; j < np[b]; ++j) priv_pages += is_shared[static_cast<size_t>(b) * max_blocks + j] ? 0 : 1;
  for (size_t gi = 0; gi < group_cands.size(); ++gi) {
    const int64_t chunks = (static_cast<int64_t>(group_cands[gi].size()) + kConsumerWarps - 1) / kConsumerWarps;
    shared_units += chunks * static_cast<int64_t>(group_pages[gi].size()) * kConsumerWarps;
  }
  const int64_t total = (priv_pages + shared_units) * n_kv;
  const int64_t target_ctas = 2LL * num_sms;
  int64_t unit = total / (target_ctas > 0 ? target_ctas : 1);   // private pages per item
  if (unit < kPagesPerStage) unit = kPagesPerStage;
  for (int attempt = 0; attempt < 20; ++attempt, unit *= 2) {
    w.items.clear();
    w.pages.clear();
    w.cands.clear();
    w.slots.clear();
    w.nslots.assign(n, 0);
    const int64_t priv_split =
        std::min<int64_t>(max_pages_item, (unit + kPagesPerStage - 1) / kPagesPerStage * kPagesPerStage);
    const int64_t shared_split = std::min<int64_t>(max_pages_item, std::max<int64_t>(1, unit / kConsumerWarps));
    bool ok = true;
    // shared items first: they are the longest per CTA
    for (size_t gi = 0; gi < group_cands.size() && ok; ++gi) {
      const auto& c = group_cands[gi];
      const auto& pg = group_pages[gi];
      for (size_t c0 = 0; c0 < c.size(); c0 += kConsumerWarps) {
        const int nc = static_cast<int>(std::min<size_t>(kConsumerWarps, c.size() - c0));
        for (size_t p0 = 0; p0 < pg.size(); p0 += static_cast<size_t>(shared_split)) {
          const int npg = static_cast<int>(std::min<size_t>(static_cast<size_t>(shared_split), pg.size() - p0));
          AttnItem it{};
          it.kind = 1;
          it.cand = static_cast<int32_t>(w.cands.size());
          it.n_cands = nc;
          it.page_off = static_cast<int32_t>(w.pages.size());
          it.n_pages = npg;
          it.last_valid = 16;
          it.slot = static_cast<int32_t>(w.slots.size());
          for (int k = 0; k < nc; ++k) {
            const int b = c[c0 + k];
            w.cands.push_back(b);
            w.slots.push_back(w.nslots[b]++);
            if (w.nslots[b] > slot_cap) ok = false;
          }
          w.pages.insert(w.pages.end(), pg.begin() + p0, pg.begin() + p0 + npg);
          w.items.push_back(it);
        }
      }
    }
    for (int b = 0; b < n && ok; ++b) {
      std::vector<int32_t> priv;
      for (int j = 0; j < np[b]; ++j)
        if (!is_shared[static_cast<size_t>(b) * max_blocks + j])
          priv.push_back(bt[static_cast<int64_t>(b) * max_blocks + j]);
      const int last_valid_b = np[b] > 0 ? sl[b] - 16 * (np[b] - 1) : 16;
      const bool last_private = np[b] > 0 && !is_shared[static_cast<size_t>(b) * max_blocks + np[b] - 1];
      if (priv.empty()) {
        if (np[b] == 0) {   // empty cache: an item with no pages merges the self entry alone
          AttnItem it{};
          it.kind = 0;
          it.cand = b;
          it.n_cands = 1;
          it.page_off = static_cast<int32_t>(w.pages.size());
          it.n_pages = 0;
          it.last_valid = 16;
          it.slot = 0;
          w.items.push_back(it);
        }
        continue;
      }
      for (size_t p0 = 0; p0 < priv.size(); p0 += static_cast<size_t>(priv_split)) {
        const int npg = static_cast<int>(std::min<size_t>(static_cast<size_t>(priv_split), priv.size() - p0));
        const bool ends = p0 + npg == priv.size();
        AttnItem it{};
        it.kind = 0;
        it.cand = b;
        it.n_cands = 1;
        it.page_off = static_cast<int32_t>(w.pages.size());
        it.n_pages = npg;
        it.last_valid = (ends && last_private) ? last_valid_b : 16;
        it.slot = w.nslots[b]++;
        if (w.nslots[b] > slot_cap) ok = false;
        w.pages.insert(w.pages.end(), priv.begin() + p0, priv.begin() + p0 + npg);
        w.items.push_back(it);
      }
    }
    if (ok) {
      w.max_item_pages = 0;
      for (const auto& it : w.items) w.max_item_pages = std::max(w.max_item_pages, it.n_pages);
      return true;
    }
  }
  return false;
}

cudaError_t attention_configure() {
  cudaError_t e;
  if ((e = set_smem(attn_kernel<64, false>)) != cudaSuccess) return e;
  if ((e = set_smem(attn_kernel<64, true>)) != cudaSuccess) return e;
  if ((e = set_smem(attn_kernel<128, false>)) != cudaSuccess) return e;
  return set_smem(attn_kernel<128, true>);
}

cudaError_t launch_attention(const AttnShape& s, const AttnWork& wk, int max_item_pages, const CUtensorMap* tm_pool,
                             int layer, const __nv_bfloat16* q_hi, const __nv_bfloat16* q_lo, int stride,
                             float* part_o, float* part_ml, const AttnMerge& mg, int* err, cudaStream_t stream,
                             bool pdl, unsigned long long* ts) {
  if (wk.n_items == 0) return cudaSuccess;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(wk.n_items, s.n_kv, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = attention_smem_bytes(s.hd, max_item_pages);
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  const int64_t row0 = static_cast<int64_t>(layer) * s.layer_rows;
  const bool two = s.group > 8;
  if (s.hd == 128) {
    if (two)
      return cudaLaunchKernelEx(&cfg, attn_kernel<128, true>, *tm_pool, row0, wk, q_hi, q_lo, s.n_q, s.n_kv, s.group,
                                stride, part_o, part_ml, mg, err, ts);
    return cudaLaunchKernelEx(&cfg, attn_kernel<128, false>, *tm_pool, row0, wk, q_hi, q_lo, s.n_q, s.n_kv, s.group,
                              stride, part_o, part_ml, mg, err, ts);
  }
  if (two)
    return cudaLaunchKernelEx(&cfg, attn_kernel<64, true>, *tm_pool, row0, wk, q_hi, q_lo, s.n_q, s.n_kv, s.group,
                              stride, part_o, part_ml, mg, err, ts);
  return cudaLaunchKernelEx(&cfg, attn_kernel<64, false>, *tm_pool, row0, wk, q_hi, q_lo, s.n_q, s.n_kv, s.group,
                            stride, part_o, part_ml, mg, err, ts);
}

cudaError_t launch_resolve(const int32_t* bt, const int32_t* seq_lens, int max_blocks, int b, int64_t* out,
                           cudaStream_t stream) {
  resolve_kernel<<<64, 256, 0, stream>>>(bt, seq_lens, max_blocks, b, out);
  return cudaGetLastError();
}

}  // namespace kvprm
