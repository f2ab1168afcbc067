// Paged GQA decode attention for the verify token (App. A.3 read-out,
// head = softmax(q^T K / sqrt(d_k)) V, one query per head, k = 1 of Def. 1),
// split over the cache ("flash decoding"), with the splits merged together
// with the verify token's own key/value.
//
// Persistent layout: one CTA per SM (9 warps) works through a host-built
// schedule (build_attn_work).  The schedule lays every (run of pages, kv head)
// end to end on a cost axis and cuts the axis into equal CTA ranges, so every
// SM streams the same number of bytes whatever the mix of lengths; a run cut
// by a range boundary simply yields one more partial.
//  - warp 8 (producer) streams the K and V pages of the CTA's segments, one
//    after the other, with TMA (one 5-D box per page and kv head: K and V,
//    128-byte swizzle) through a 3-stage ring of 8 pages (128 tokens) per
//    stage -- starting before the query is ready, since the cache does not
//    depend on it -- and never drains the ring between segments;
//  - a *private* segment holds pages of one candidate: consumer warp w scores
//    page w of every stage;
//  - a *shared* segment holds pages that several candidates reference (a beam
//    prefix, an MCTS ancestor): each page is loaded once and consumer warp w
//    scores it for candidate w (up to 8).  Attention is invariant to the order
//    of the keys, so shared pages need not sit at the same positions in the
//    candidates' sequences;
//  - per page and warp: S = Q K^T on the tensor cores (mma.m16n8k16), an
//    online softmax in fp32 registers with quad shuffles, then O += P V.  The
//    query and the probabilities enter the bf16 MMAs as (hi, lo) pairs so both
//    keep ~16 bits: with G <= 8 query heads per group the hi parts fill MMA
//    rows 0..7 and the lo parts rows 8..15 of the same instruction (summed
//    afterwards), so the split costs no extra MMAs; with 8 < G <= 16 hi and lo
//    take one MMA each;
//  - at the end of a private segment the consumer warps hand their (m, l, O)
//    to warp 9 (the merger) through shared memory and go straight on to the
//    next segment; the merger folds them into the segment's partial slot.  In
//    a shared segment each warp writes its own candidate's slot.  No barrier,
//    fence or atomic is involved;
//  - a second small kernel (attn_combine_kernel) merges each (candidate, kv
//    head)'s slots with the verify token's own entry and writes the attention
//    output as a bf16 (hi, lo) pair for the O projection.
// All scores are kept in log2 units (scaled by log2(e) / sqrt(hd)).
#include <cuda_bf16.h>

#include <algorithm>
#include <climits>
#include <unordered_map>
#include <vector>

#include "attn_core.cuh"
#include "kernels.h"
#include "ptx.cuh"

namespace kvprm {

namespace {

using namespace ac;

constexpr int kPagesPerStage = 8;
constexpr int kStages = 3;
constexpr int kConsumerWarps = 8;
constexpr int kProducerWarp = kConsumerWarps;       // warp 8: TMA
constexpr int kMergerWarp = kConsumerWarps + 1;     // warp 9: folds private segments' warp states
constexpr int kThreads = (kConsumerWarps + 2) * 32;

// Schedule costs per page and kv head.  A private page is read by one warp
// while the other seven read the rest of its stage, so a private stage costs
// the time to stream it (measured ~0.19 us per page per SM at full HBM rate).
// A shared page is scored by one warp per candidate, and those warps compete
// for the same SM pipelines: measured ~0.1 us per page and candidate, i.e. about
// half a private page per candidate.
constexpr int64_t kPrivateCost = 4;
constexpr int64_t kSharedCostPerCand = 2;
// A shared run of n candidates is scored by (8 / n) warps per candidate, each taking every
// (8 / n)-th page of a stage and writing its own partial slot: warp w scores candidate w % n,
// pages p with p % (8 / n) == w / n, into slot w of the segment.  (n <= 4 keeps every warp busy.)
__host__ __device__ constexpr int shared_reps(int n_cands) { return kConsumerWarps / n_cands; }
// The tensor-core launch, in the same units, when it runs beside the private pages' launch: a CTA
// costs kTcChunkCost per 64-token chunk plus kTcCtaCost once (the first query load and pages'
// latency, the last output read-out).  Fitted to the SM split that measured fastest on the beam
// (86 of 152 SMs, 12 chunks per CTA) and MCTS (16 SMs, ~115 chunks per CTA) workloads: ~1.2 us per
// chunk and ~8 us per CTA against ~0.045 us per unit on the private side (a sweep of 24-32 units
// per chunk and 150-210 per CTA moved the MCTS attention by a few percent, 26 fastest; beam alike).
constexpr int64_t kTcChunkCost = 26;
constexpr int64_t kTcCtaCost = 180;
// pages shared by fewer candidates go to the persistent kernel as kind-1 runs: 2 units per page
// and candidate there against kTcChunkCost / 4 per page on the tensor cores, whatever the tile's rows
constexpr size_t kTcMinCands = 6;
// Tensor-core scoring of shared pages (attn_tc_kernel): query rows per tile
// and pages per 64-token chunk.
constexpr int kTcRows = 128;
constexpr int kTcChunkPages = 4;

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~static_cast<uintptr_t>(1023));
}

// Physical page of logical page `j` of candidate `b` (the block-table walk
// used by the resolve entry point, so indexing can be checked bit-exactly).
__device__ __forceinline__ int32_t phys_page(const int32_t* __restrict__ bt, int b, int max_blocks, int j) {
  return bt[static_cast<int64_t>(b) * max_blocks + j];
}

// Shared-memory layout of the kernel (offsets from the 1024-aligned base).
template <int HD>
struct AttnSmem {
  static constexpr uint32_t kBlockBytes = (HD / 64) * 16 * 128;   // one K (or V) page of one kv head
  static constexpr uint32_t kPageBytes = 2 * kBlockBytes;
  static constexpr uint32_t kStageBytes = kPagesPerStage * kPageBytes;
  static constexpr uint32_t kRing = 0;
  static constexpr uint32_t kMergeO = kStages * kStageBytes;                  // [8 warps][8 rows][HD] fp32
  static constexpr uint32_t kMergeM = kMergeO + kConsumerWarps * 8 * HD * 4;  // [8][8] running max
  static constexpr uint32_t kMergeL = kMergeM + kConsumerWarps * 8 * 4;       // [8][8] running sum
  static constexpr uint32_t kBars = kMergeL + kConsumerWarps * 8 * 4;   // full[kStages], empty[kStages], seg_full, seg_free
  static constexpr uint32_t kSelf = kBars + (2 * kStages + 2) * 8;   // fused combine: [8] own logits,
  static constexpr uint32_t kEnd = kSelf + (8 + HD) * 4;                // then v_self [HD]
  static constexpr size_t kDynamic = kEnd + 1024;   // + alignment slack
};
static_assert(AttnSmem<128>::kDynamic <= 227 * 1024, "attention shared memory exceeds the per-block limit");

template <int HD, bool TWO_ROWS>
__global__ void __launch_bounds__(kThreads, 1) attn_kernel(
    const __grid_constant__ CUtensorMap tm_pool, int64_t layer_page0, AttnWork wk,
    const __nv_bfloat16* __restrict__ q_hi, const __nv_bfloat16* __restrict__ q_lo, int n_q, int n_kv, int group,
    float* __restrict__ part_o, float* __restrict__ part_ml, AttnMerge mg, int* err, unsigned long long* ts) {
  using SM = AttnSmem<HD>;
  trace_begin(ts);

  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = align1024(smem_raw);
  uint8_t* ring = base + SM::kRing;
  float* mo = reinterpret_cast<float*>(base + SM::kMergeO);
  float* mm = reinterpret_cast<float*>(base + SM::kMergeM);
  float* ml = reinterpret_cast<float*>(base + SM::kMergeL);
  uint64_t* full = reinterpret_cast<uint64_t*>(base + SM::kBars);
  uint64_t* empty = full + kStages;
  uint64_t* seg_full = empty + kStages;   // the 8 consumer warps' states of a private segment are in mo / mm / ml
  uint64_t* seg_free = seg_full + 1;      // the merger has read them

  const int seg0 = wk.cta_seg[blockIdx.x], seg1 = wk.cta_seg[blockIdx.x + 1];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], kConsumerWarps);
    }
    mbar_init(seg_full, kConsumerWarps);
    mbar_init(seg_free, 1);
    fence_mbar_init();
  }
  __syncthreads();
  grid_dep_launch();   // the next kernel may start; it waits for this grid before reading its output

  if (warp == kProducerWarp) {
    // ------------------------------------------------ producer
    // One TMA box per page: K and V of kv head g (coordinates: column 0,
    // token 0, sub-tile 0, head g, 2 * (layer * n_pages + page)).
    if (lane == 0) {
      tma_prefetch_desc(&tm_pool);
      const uint64_t pol = policy_evict_first();
      uint32_t u = 0;   // stage sequence number over all segments
      bool ok = true;
      for (int si = seg0; si < seg1 && ok; ++si) {
        const AttnSeg sg = wk.segs[si];
        const int32_t* pg = wk.pages + sg.page_off;
        for (int p0 = 0; p0 < sg.n_pages; p0 += kPagesPerStage, ++u) {
          const int slot = static_cast<int>(u % kStages);
          if (u >= static_cast<uint32_t>(kStages) &&
              !mbar_wait(&empty[slot], ((u / kStages) & 1u) ^ 1u, err)) {
            ok = false;
            break;
          }
          const int npg = min(kPagesPerStage, sg.n_pages - p0);
          mbar_arrive_expect_tx(&full[slot], static_cast<uint32_t>(npg) * SM::kPageBytes);
          uint8_t* stg = ring + slot * SM::kStageBytes;
          for (int pi = 0; pi < npg; ++pi) {
            const int64_t phys = __ldg(pg + p0 + pi);
            tma_load_5d(stg + pi * SM::kPageBytes, &tm_pool, &full[slot], 0, 0, 0, sg.g,
                        static_cast<int32_t>(2 * (layer_page0 + phys)), pol);
          }
        }
      }
      // Every copy issued above has landed once the consumers released the
      // last stages (each slot's latest phase); a lost arrival times out.
      if (ok)
        for (uint32_t v = u > static_cast<uint32_t>(kStages) ? u - kStages : 0; v < u; ++v)
          if (!mbar_wait(&empty[v % kStages], (v / kStages) & 1u, err)) break;
    }
  } else if (warp < kConsumerWarps) {
    // ------------------------------------------------ consumers
    // Every warp waits for every stage before releasing it, busy or not, so
    // no warp can arrive for a slot's next use early.
    grid_dep_wait();   // q is written by the preceding kernel
    if (warp == 0 && lane == 0) trace_event(ts, 0);   // the query is ready
    if (!TWO_ROWS && wk.fuse_cs > 0) {
      // fused combine, before the pages: the verify token's own logit of head `warp`
      // (q . k_self / sqrt(hd), log2 units) and the pair's v_self, into shared memory
      const int pr = blockIdx.x / wk.fuse_cs, b = pr / n_kv, g = pr - b * n_kv;
      const float* kr = mg.kself + (static_cast<int64_t>(b) * n_kv + g) * HD;
      float* s_self = reinterpret_cast<float*>(base + SM::kSelf);
      if (warp < group) {
        const float* qr = mg.q + (static_cast<int64_t>(b) * n_q + g * group + warp) * HD;
        float dot = 0.f;
#pragma unroll
        for (int j = 0; j < HD / 32; ++j) dot += __ldcg(qr + lane + 32 * j) * __ldcg(kr + lane + 32 * j);
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) dot += __shfl_xor_sync(0xffffffffu, dot, off);
        if (lane == 0) s_self[warp] = dot * (kLog2e * rsqrtf(static_cast<float>(HD)));
      }
      for (int d = threadIdx.x; d < HD; d += kConsumerWarps * 32)
        s_self[8 + d] = __ldcg(mg.vself + (static_cast<int64_t>(b) * n_kv + g) * HD + d);
    }
    bool ok = true;
    uint32_t u = 0, n_priv = 0;
    for (int si = seg0; si < seg1; ++si) {
      const AttnSeg sg = wk.segs[si];
      const bool shared = sg.kind == 1;
      // the candidate this warp scores in this segment, -1 if none (and, in a shared run, which of the
      // candidate's replica warps it is)
      const int reps = shared ? shared_reps(sg.n_cands) : 1;
      const int cand = shared ? (warp < reps * sg.n_cands ? wk.cands[sg.cand + warp % sg.n_cands] : -1)
                              : (warp < sg.n_pages ? sg.cand : -1);
      const int part = shared ? warp / sg.n_cands : 0;
      WarpQ<HD> q;
      if (cand >= 0) {
        const int64_t q0 = (static_cast<int64_t>(cand) * n_q + static_cast<int64_t>(sg.g) * group) * HD;
        load_q<HD, TWO_ROWS>(q, q_hi + q0, q_lo + q0, group, lane);
      }
      WarpState<HD> st;
      st.reset();
      for (int p0 = 0; p0 < sg.n_pages; p0 += kPagesPerStage, ++u) {
        const int slot = static_cast<int>(u % kStages);
        if (ok) ok = __all_sync(0xffffffffu, mbar_wait(&full[slot], (u / kStages) & 1u, err));
        if (ok && cand >= 0) {
          const uint32_t sbase = smem_u32(ring + slot * SM::kStageBytes);
          const int npg = min(kPagesPerStage, sg.n_pages - p0);
          if (!shared) {   // page `warp` of this stage
            if (warp < npg) {
              const int valid = p0 + warp == sg.n_pages - 1 ? sg.last_valid : 16;
              const uint32_t kb = sbase + warp * SM::kPageBytes;
              process_page<HD, TWO_ROWS>(q, kb, kb + SM::kBlockBytes, valid, lane, st);
            }
          } else {         // this replica's pages of this stage, for this warp's candidate
            int pi = part;
            if (!TWO_ROWS)   // two pages at a time: their dependent steps overlap
              for (; pi + reps < npg; pi += 2 * reps) {
                const int va = p0 + pi == sg.n_pages - 1 ? sg.last_valid : 16;
                const int vb = p0 + pi + reps == sg.n_pages - 1 ? sg.last_valid : 16;
                const uint32_t ka = sbase + pi * SM::kPageBytes, kb = sbase + (pi + reps) * SM::kPageBytes;
                process_page_pair<HD>(q, ka, ka + SM::kBlockBytes, va, kb, kb + SM::kBlockBytes, vb, lane, st);
              }
            for (; pi < npg; pi += reps) {
              const int valid = p0 + pi == sg.n_pages - 1 ? sg.last_valid : 16;
              const uint32_t kb = sbase + pi * SM::kPageBytes;
              process_page<HD, TWO_ROWS>(q, kb, kb + SM::kBlockBytes, valid, lane, st);
            }
          }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty[slot]);
      }
      if (cand >= 0 && ok) finish_state<HD, TWO_ROWS>(st);
      if (!shared && !TWO_ROWS) {
        // hand the warp's state to the merger warp (one slot per private
        // segment); wait only until it has read the previous segment's states
        if (n_priv > 0) ok = __all_sync(0xffffffffu, mbar_wait(seg_free, (n_priv - 1) & 1u, err)) && ok;
        stash_state<HD>(st, cand >= 0 && ok, warp, group, lane, mo, mm, ml);
        __syncwarp();
        if (lane == 0) mbar_arrive(seg_full);
        ++n_priv;
      } else if (cand >= 0 && ok) {
        // this warp's own partial slot
        const int slot_id = shared ? wk.slots[sg.slot + warp] : sg.slot + warp;
        store_state_slot<HD, TWO_ROWS>(st, slot_id, group, lane, part_o, part_ml);
      }
    }
    if (lane == 0) trace_event(ts, 1);   // this warp has scored every page of its CTA
    if (!TWO_ROWS && wk.fuse_cs > 0) {
      // fused combine (one private run per CTA): once every consumer warp has stashed its state and
      // read its last stage, warp r folds query row r of the eight states into the idle ring
      named_bar_sync(3, kConsumerWarps * 32);
      if (warp < group) {
        float* st_o = reinterpret_cast<float*>(ring);
        merge_row<HD>(warp, mo, mm, ml, lane, st_o + warp * HD, st_o + 8 * HD + 2 * warp);
      }
    }

  } else if (warp == kMergerWarp && !TWO_ROWS) {
    // ------------------------------------------------ merger
    // For every private segment, in order: fold the eight consumer warps'
    // (m, l, O) into the segment's partial slot,
    //   M = max_w m_w, L = sum_w 2^(m_w - M) l_w, O = sum_w 2^(m_w - M) O_w.
    uint32_t k = 0;
    bool ok = true;
    for (int si = wk.fuse_cs > 0 ? seg1 : seg0; si < seg1; ++si) {   // fused plans: the consumers merge
      const AttnSeg sg = wk.segs[si];
      if (sg.kind != 0) continue;
      if (ok) ok = __all_sync(0xffffffffu, mbar_wait(seg_full, k & 1u, err));
      if (ok) merge_warp_states<HD>(group, mo, mm, ml, sg.slot, lane, part_o, part_ml);
      __syncwarp();
      if (lane == 0) mbar_arrive(seg_free);
      ++k;
    }
    if (lane == 0) trace_event(ts, 2);   // every private run of this CTA is merged
  }
  if (!TWO_ROWS && wk.fuse_cs > 0) {   // fused plans have group <= 8
    // The cluster scored one (candidate, kv head); every rank left its (M, L, O) per query row at
    // the start of its ring and the verify token's own logits in kSelf.  Rank k then produces
    // head-dimension slice k of every row, reading the ranks' states through distributed shared
    // memory and merging them with the verify token's own entry:
    //   M* = max(s_self, M_j), o = (2^(s_self - M*) v_self + sum_j 2^(M_j - M*) O_j)
    //                              / (2^(s_self - M*) + sum_j 2^(M_j - M*) L_j).
    // The second cluster barrier keeps every rank's shared memory until all have read it.  The
    // consumer warps produce the outputs (they wrote the logits and v_self, after the
    // grid-dependency wait).
    constexpr int kMergeThreads = kConsumerWarps * 32;
    constexpr int kOut = (8 * HD + kMergeThreads - 1) / kMergeThreads;
    const int cs = wk.fuse_cs, pr = blockIdx.x / cs, b = pr / n_kv, g = pr - b * n_kv;
    const int slice = HD / cs, d0 = static_cast<int>(cluster_rank()) * slice;
    const bool mine = warp < kConsumerWarps;
    const int64_t hq0 = static_cast<int64_t>(b) * n_q + static_cast<int64_t>(g) * group;
    __syncwarp();
    cluster_sync();
    if (mine) {
      const float* st_o = reinterpret_cast<const float*>(ring);
      const float* st_ml = st_o + 8 * HD;
      const float* s_self = reinterpret_cast<const float*>(base + SM::kSelf);
#pragma unroll
      for (int i = 0; i < kOut; ++i) {
        const int idx = threadIdx.x + i * kMergeThreads;
        if (idx >= group * slice) break;
        const int r = idx / slice, d = d0 + idx - r * slice;
        const float ss = s_self[r];
        float Mk[8], Lk[8], Ok[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          if (k >= cs) break;
          Mk[k] = ld_cluster(st_ml + 2 * r, k);
          Lk[k] = ld_cluster(st_ml + 2 * r + 1, k);
          Ok[k] = ld_cluster(st_o + r * HD + d, k);
        }
        float Mt = ss;
#pragma unroll
        for (int k = 0; k < 8; ++k)
          if (k < cs) Mt = fmaxf(Mt, Mk[k]);
        const float ws = exp2f(ss - Mt);
        float num = ws * s_self[8 + d], den = ws;
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          if (k >= cs || Mk[k] == -INFINITY) continue;   // a rank with no pages
          const float f = exp2f(Mk[k] - Mt);
          num += f * Ok[k];
          den += f * Lk[k];
        }
        const float out = num / den;
        const int64_t o = (hq0 + r) * HD + d;
        const __nv_bfloat16 hi = __float2bfloat16_rn(out);
        mg.o_hi[o] = hi;
        mg.o_lo[o] = __float2bfloat16_rn(out - __bfloat162float(hi));
        if (mg.out_f32) mg.out_f32[o] = out;
        if (mg.dbg) mg.dbg[o] = out;
        if (mg.lse && d == 0) mg.lse[hq0 + r] = Mt * kLn2 + logf(den);   // scores are in log2 units
      }
      if (threadIdx.x == 0) trace_event(ts, 3);   // this rank's outputs are written
    }
    __syncwarp();
    cluster_sync();
  }
  trace_end(ts);
}

// The combine: one CTA of W warps per (candidate, kv head) running combine_group (DEEP: a depth-k
// readout's causal verify-token entries).
template <int HD, int ROWS, int W, bool DEEP>
__global__ void __launch_bounds__(W * 32) attn_combine_kernel(
    const int32_t* __restrict__ slot_base, const int32_t* __restrict__ nslots, int n_q, int n_kv, int group,
    const float* __restrict__ part_o, const float* __restrict__ part_ml, AttnMerge mg, unsigned long long* ts) {
  trace_begin(ts);
  grid_dep_launch();
  extern __shared__ __align__(16) uint8_t csm[];
  const int cg = blockIdx.x, b = cg / n_kv, g = cg - b * n_kv;
  const int first = slot_base[cg], ns = nslots[cg];   // host-uploaded before the call: no wait needed
  grid_dep_wait();   // the partials (and q, k_self, v_self) are written by earlier kernels
  if (threadIdx.x == 0) trace_event(ts, 0);
  combine_group<HD, ROWS, W, DEEP>(threadIdx.x, b, g, first, ns, n_q, n_kv, group, part_o, part_ml, mg, csm,
                                   [] { __syncthreads(); });
  if (threadIdx.x == 0) trace_event(ts, 1);
  trace_end(ts);
}

// The combine of a single verify token per candidate, flat: one CTA per (candidate, kv head) and
// one warp per query head of the group, lane i holding head-dim elements i + 32 j.  A round issues
// every load it uses (up to kFlatSlots partial slots' (m, l) and O values; in the first round also
// q, k_self and v_self) before using any, so it costs one memory round trip; the slots then merge
// into the running (M, L, acc) started from the verify token's own entry.  No shared memory and no
// CTA barrier, so CTAs are short and many fit on an SM.
constexpr int kFlatSlots = 8;

template <int HD>
__global__ void __launch_bounds__(512) attn_combine_flat_kernel(
    const int32_t* __restrict__ slot_base, const int32_t* __restrict__ nslots, int n_q, int n_kv, int group,
    const float* __restrict__ part_o, const float* __restrict__ part_ml, AttnMerge mg, unsigned long long* ts) {
  constexpr int kPer = HD / 32;
  trace_begin(ts);
  grid_dep_launch();
  const int cg = blockIdx.x, b = cg / n_kv, g = cg - b * n_kv;
  const int r = static_cast<int>(threadIdx.x >> 5), lane = static_cast<int>(threadIdx.x & 31);
  const int first = slot_base[cg], ns = nslots[cg];   // host-uploaded before the call: no wait needed
  const int64_t hq = static_cast<int64_t>(b) * n_q + static_cast<int64_t>(g) * group + r;
  const int64_t hk = static_cast<int64_t>(b) * n_kv + g;
  grid_dep_wait();   // the partials (and q, k_self, v_self) are written by earlier kernels
  if (threadIdx.x == 0) trace_event(ts, 0);
  float2 ml[kFlatSlots];
  float o[kFlatSlots][kPer];
  auto load_round = [&](int s0) {
#pragma unroll
    for (int k = 0; k < kFlatSlots; ++k) {
      const bool in = s0 + k < ns;
      const int64_t pr = (static_cast<int64_t>(first) + (in ? s0 + k : 0)) * group + r;
      ml[k] = in ? __ldcg(reinterpret_cast<const float2*>(part_ml) + pr) : make_float2(-INFINITY, 0.f);
#pragma unroll
      for (int j = 0; j < kPer; ++j) o[k][j] = in ? __ldcg(part_o + pr * HD + lane + 32 * j) : 0.f;
    }
  };
  float qd[kPer], kd[kPer], acc[kPer];
#pragma unroll
  for (int j = 0; j < kPer; ++j) {
    qd[j] = __ldcg(mg.q + hq * HD + lane + 32 * j);
    kd[j] = __ldcg(mg.kself + hk * HD + lane + 32 * j);
    acc[j] = __ldcg(mg.vself + hk * HD + lane + 32 * j);
  }
  load_round(0);
  // the verify token's own entry: score q . k_self (log2 units), weight 1 at M = that score
  float dot = 0.f;
#pragma unroll
  for (int j = 0; j < kPer; ++j) dot += qd[j] * kd[j];
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) dot += __shfl_xor_sync(0xffffffffu, dot, off);
  float M = dot * (kLog2e * rsqrtf(static_cast<float>(HD))), L = 1.f;
  for (int s0 = 0;; s0 += kFlatSlots) {
#pragma unroll
    for (int k = 0; k < kFlatSlots; ++k) {
      if (ml[k].x == -INFINITY) continue;   // past the last slot, or a slot with no token (warp-uniform)
      const float Mn = fmaxf(M, ml[k].x);
      const float sc = exp2f(M - Mn), w = exp2f(ml[k].x - Mn);
      L = L * sc + w * ml[k].y;
#pragma unroll
      for (int j = 0; j < kPer; ++j) acc[j] = acc[j] * sc + w * o[k][j];
      M = Mn;
    }
    if (s0 + kFlatSlots >= ns) break;
    load_round(s0 + kFlatSlots);
  }
  const float inv = 1.f / L;
#pragma unroll
  for (int j = 0; j < kPer; ++j) {
    const float out = acc[j] * inv;
    const int64_t oi = hq * HD + lane + 32 * j;
    const __nv_bfloat16 hi = __float2bfloat16_rn(out);
    mg.o_hi[oi] = hi;
    mg.o_lo[oi] = __float2bfloat16_rn(out - __bfloat162float(hi));
    if (mg.out_f32) mg.out_f32[oi] = out;
    if (mg.dbg) mg.dbg[oi] = out;
  }
  if (mg.lse && lane == 0) mg.lse[hq] = M * kLn2 + logf(L);   // scores are in log2 units
  if (threadIdx.x == 0) trace_event(ts, 1);
  trace_end(ts);
}

// ---------------------------------------------------------------- shared pages on the tensor cores
// attn_tc_kernel: persistent CTAs, each scoring its range of kind-2 segments
// (wk.tc_cta).  A segment is a tile of <= 128 / G candidates that all
// reference its pages, for one kv head; the tile's query rows (candidate,
// head) are the M = 128 side of tcgen05 MMAs whose A operands live in tensor
// memory:
//   S = Q K^T   per 64-token chunk (4 pages): A = Q as bf16 hi and lo (two
//               MMAs, so S sees the fp32 query), B = the chunk's keys in
//               shared memory; S in TMEM, two 64-column buffers;
//   softmax     one thread per query row reads its S row; the running
//               maximum m only moves when a chunk's scores exceed it by more
//               than `margin` (log2 units; then the row's O is rescaled in
//               TMEM), so P = 2^(s - m) stays below 2^margin and rescales are
//               rare; P goes back as bf16 hi and lo (truncations by bit mask,
//               |P - hi - lo| < 2^-14 P) over the S buffer it came from;
//   O += P V    A = P (hi, lo) from TMEM, B = the chunk's values in shared
//               memory as TMA left them (token rows of 128 bytes): an
//               MN-major operand, so nothing is transposed; O in TMEM (128
//               columns).
// Warp 0 streams K with TMA (one 2 KB box per page and 64-column sub-tile,
// so a chunk's 64 tokens land contiguously; a segment's missing tail pages
// are read at an out-of-range page and arrive as zeros) through a 6-stage
// ring released by the S MMAs that read it; warp 10 streams V the same way
// through a ring released by the O MMAs, so neither waits for the other.
// Warp 1 issues the S MMAs (up to four chunks ahead: four S/P buffers) and
// warp 11 the O MMAs, so neither stream waits behind the other's bookkeeping;
// warps 2..9 run the softmax, two threads per query row (each 32 of
// a chunk's 64 columns; the half maxima meet in shared memory) and, at each
// segment's end, write every live row's (m, l, O) into its candidate's
// partial slot.
struct TcSmem {
  static constexpr int kStages = 6;
  static constexpr uint32_t kKVTile = 2 * 64 * 128;          // [2 sub-tiles][64 tokens][128 B] = 16 KB
  static constexpr uint32_t kK = 0;                          // key stages
  static constexpr uint32_t kV = kK + kStages * kKVTile;     // value stages
  static constexpr uint32_t kBars = kV + kStages * kKVTile;
  static constexpr uint32_t kXch = kBars + 512;               // softmax exchange: half maxima [2][128], l [128]
  static constexpr uint32_t kEnd = kXch + 3 * 128 * 4;
  static constexpr size_t kDynamic = kEnd + 1024;
};
static_assert(TcSmem::kDynamic <= 227 * 1024, "tensor-core attention shared memory exceeds the per-block limit");
constexpr int kTcThreads = 384;   // warp 0 key TMA, 1 S MMAs, 2..9 softmax (two threads per row), 10 value TMA,
                                  // 11 O MMAs
constexpr uint32_t kTcTmemCols = 512;
// TMEM columns: four S/P buffers at 0, 64, 128, 192; O at 256..383; Q hi at 384..447, Q lo at 448..511.
// With four S buffers the MMA warp issues S two chunks ahead of the softmax without waiting for
// the O MMAs that read the P it overwrites (those completed two chunks earlier).
constexpr int kTcSBufs = 4;
constexpr uint32_t kColO = 256, kColQhi = 384, kColQlo = 448;

__global__ void __launch_bounds__(kTcThreads, 1) attn_tc_kernel(
    const __grid_constant__ CUtensorMap tm_pool_tc, int64_t layer_page0, AttnWork wk,
    const __nv_bfloat16* __restrict__ q_hi, const __nv_bfloat16* __restrict__ q_lo, int n_q, int group,
    float* __restrict__ part_o, float* __restrict__ part_ml, float margin, int* err, unsigned long long* ts,
    unsigned long long* prof) {
  using SM = TcSmem;
  trace_begin(ts);
  // optional wait profile (SM clock cycles per CTA, accumulated with reductions so that the
  // measured warps never wait on a load) and CTA 0's per-chunk event log: see kvprm_set_debug, flag 32
  unsigned long long* pr = prof ? prof + kTcEventLog + static_cast<int64_t>(blockIdx.x) * 16 : nullptr;
  unsigned long long* ev = (prof && blockIdx.x == 0) ? prof : nullptr;
  auto tic = [&]() -> long long { return pr ? clock64() : 0; };
  auto toc = [&](int slot, long long t0) {
    if (pr) atomicAdd(pr + slot, static_cast<unsigned long long>(clock64() - t0));
  };
  auto event = [&](int kind, uint32_t i) {
    if (ev && i < 128) ev[kind * 128 + i] = static_cast<unsigned long long>(clock64());
  };
  const long long t_start = tic();
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = align1024(smem_raw);
  uint64_t* k_full = reinterpret_cast<uint64_t*>(base + SM::kBars);    // [6] keys landed
  uint64_t* k_empty = k_full + SM::kStages;                           // [6] the S MMAs read the keys
  uint64_t* v_full = k_empty + SM::kStages;                           // [6] values landed
  uint64_t* v_empty = v_full + SM::kStages;                           // [6] the O MMAs read the values
  uint64_t* s_full = v_empty + SM::kStages;                           // [4] S in TMEM
  uint64_t* p_full = s_full + kTcSBufs;                               // [4] P in TMEM
  uint64_t* pv_done = p_full + kTcSBufs;                              // [4] the O MMAs of a chunk completed
  uint64_t* q_ready = pv_done + kTcSBufs;                             // Q of the current segment in TMEM
  uint64_t* o_free = q_ready + 1;                                     // O of the previous segment read out
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(o_free + 1);
  const int seg0 = wk.tc_cta[blockIdx.x], seg1 = wk.tc_cta[blockIdx.x + 1];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  auto chunks = [](const AttnSeg& sg) { return (sg.n_pages + kTcChunkPages - 1) / kTcChunkPages; };

  if (threadIdx.x == 0) {
    for (int s = 0; s < SM::kStages; ++s) {
      mbar_init(&k_full[s], 1);
      mbar_init(&k_empty[s], 1);
      mbar_init(&v_full[s], 1);
      mbar_init(&v_empty[s], 1);
    }
    for (int b = 0; b < kTcSBufs; ++b) {
      mbar_init(&s_full[b], 1);
      mbar_init(&p_full[b], 8);
      mbar_init(&pv_done[b], 1);
    }
    mbar_init(q_ready, 8);
    mbar_init(o_free, 8);
    fence_mbar_init();
    tma_prefetch_desc(&tm_pool_tc);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, kTcTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  grid_dep_launch();

  if (warp == 0 || warp == 10) {
    // ------------------------------------------------ loaders: warp 0 the keys, warp 10 the values
    // (the cache does not depend on q; each ring runs ahead of its own consumer)
    if (lane == 0) {
      const bool keys = warp == 0;
      const uint64_t pol = policy_evict_normal();   // the group's other tiles read the same pages
      // one ring (keys or values): wait for the stage, then all four pages of the chunk, a page
      // past the segment's end at unit -1 (out of range: TMA writes zeros and counts the bytes)
      auto load = [&](uint64_t* full, uint64_t* empty, uint32_t off, int slot, uint32_t u, const int32_t* pg, int npg,
                      int g, int kv) -> bool {
        const int st = static_cast<int>(u % SM::kStages);
        const long long t0 = tic();
        if (u >= static_cast<uint32_t>(SM::kStages) && !mbar_wait(&empty[st], ((u / SM::kStages) - 1) & 1u, err))
          return false;
        toc(slot, t0);
        mbar_arrive_expect_tx(&full[st], SM::kKVTile);
        uint8_t* dst = base + off + st * SM::kKVTile;
#pragma unroll
        for (int i = 0; i < kTcChunkPages; ++i) {
          const int32_t unit = i < npg ? static_cast<int32_t>(2 * (layer_page0 + __ldg(pg + i))) + kv : -1;
#pragma unroll
          for (int sub = 0; sub < 2; ++sub)
            tma_load_5d(dst + sub * 8192 + i * 2048, &tm_pool_tc, &full[st], 0, 0, sub, g, unit, pol);
        }
        return true;
      };
      uint64_t* full = keys ? k_full : v_full;
      uint64_t* empty = keys ? k_empty : v_empty;
      uint32_t u = 0;
      bool ok = true;
      for (int si = seg0; si < seg1 && ok; ++si) {
        const AttnSeg sg = wk.segs[si];
        const int32_t* pg = wk.pages + sg.page_off;
        for (int c = 0; c < chunks(sg) && ok; ++c, ++u) {
          const int npg = min(kTcChunkPages, sg.n_pages - c * kTcChunkPages);
          event(keys ? 5 : 4, u);
          ok = load(full, empty, keys ? SM::kK : SM::kV, keys ? 6 : 7, u, pg + c * kTcChunkPages, npg, sg.g,
                    keys ? 0 : 1);
        }
      }
      for (uint32_t v = u > static_cast<uint32_t>(SM::kStages) ? u - SM::kStages : 0; v < u; ++v)   // all landed
        if (!mbar_wait(&full[v % SM::kStages], (v / SM::kStages) & 1u, err)) break;
    }
  } else if (warp == 1 || warp == 11) {
    // ------------------------------------------------ MMA issuers: warp 1 the S MMAs, warp 11 the O MMAs
    // (each the whole warp; one elected lane issues, and its commits track only its own MMAs)
    // O MMAs take V as an MN-major B operand (instruction descriptor bit 16)
    const uint32_t id_s = idesc_bf16_f32(128, 64), id_o = idesc_bf16_f32(128, 128) | (1u << 16);
    auto wait_all = [&](uint64_t* bar, uint32_t parity) { return __all_sync(0xffffffffu, mbar_wait(bar, parity, err)); };
    auto issue_s = [&](uint32_t v) -> bool {
      const int st = static_cast<int>(v % SM::kStages);
      const uint32_t b = v % kTcSBufs;
      long long t0 = tic();
      if (!wait_all(&k_full[st], (v / SM::kStages) & 1u)) return false;
      if (lane == 0) toc(0, t0);
      t0 = tic();
      if (v >= kTcSBufs && !wait_all(&pv_done[b], ((v / kTcSBufs) - 1) & 1u)) return false;   // P of v - 4 consumed
      if (lane == 0) toc(1, t0);
      tc_fence_after();
      // keys: two 64-column sub-tiles of 8 KB; K step kk at sub-tile kk / 4, 32 bytes per step inside it
      const uint64_t k0 = desc_sw128(smem_u32(base + SM::kK + st * SM::kKVTile));
      const uint32_t d = tmem + b * 64;
#pragma unroll
      for (int kk = 0; kk < 8; ++kk) {
        const uint64_t kdesc = k0 + (((kk >> 2) * 8192 + (kk & 3) * 32) >> 4);
        umma_bf16_ta_w(d, tmem + kColQhi + kk * 8, kdesc, id_s, kk > 0 ? 1u : 0u);
        umma_bf16_ta_w(d, tmem + kColQlo + kk * 8, kdesc, id_s, 1u);
      }
      umma_commit_w(&s_full[b]);
      umma_commit_w(&k_empty[st]);
      if (lane == 0) event(0, v);
      return true;
    };
    auto issue_o = [&](uint32_t v, bool first) -> bool {
      const int st = static_cast<int>(v % SM::kStages);
      const uint32_t b = v % kTcSBufs;
      long long t0 = tic();
      if (!wait_all(&p_full[b], (v / kTcSBufs) & 1u)) return false;
      if (lane == 0) toc(2, t0);
      t0 = tic();
      if (!wait_all(&v_full[st], (v / SM::kStages) & 1u)) return false;
      if (lane == 0) toc(3, t0);
      tc_fence_after();
      // values: N = head dim over the two 64-column sub-tiles (8 KB apart), K = tokens in groups
      // of 8 rows (1 KB apart); K step kk starts 16 rows (2 KB) further
      const uint64_t v0 = desc_sw128_mn(smem_u32(base + SM::kV + st * SM::kKVTile), 8192);
      const uint32_t p = tmem + b * 64;
      const uint32_t acc0 = first ? 0u : 1u;
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {   // the chunk's 64 tokens in steps of 16
        umma_bf16_ta_w(tmem + kColO, p + kk * 8, v0 + 128 * kk, id_o, kk > 0 ? 1u : acc0);
        umma_bf16_ta_w(tmem + kColO, p + 32 + kk * 8, v0 + 128 * kk, id_o, 1u);
      }
      umma_commit_w(&pv_done[b]);
      umma_commit_w(&v_empty[st]);
      if (lane == 0) event(1, v);
      return true;
    };
    uint32_t u = 0, k = 0;
    bool ok = true;
    for (int si = seg0; si < seg1 && ok; ++si, ++k) {
      const int nch = chunks(wk.segs[si]);
      if (warp == 1) {   // S of a segment once its Q is in TMEM; up to four chunks ahead of O
        ok = wait_all(q_ready, k & 1u);
        for (int c = 0; c < nch && ok; ++c, ++u) ok = issue_s(u);
      } else {           // O of a segment once the previous segment's O is read out
        ok = k == 0 || wait_all(o_free, (k - 1) & 1u);
        for (int c = 0; c < nch && ok; ++c, ++u) ok = issue_o(u, c == 0);
      }
    }
  } else if (warp < 10) {
    // ------------------------------------------------ softmax: two threads per query row (columns 0..31 / 32..63)
    const int w4 = warp & 3;              // TMEM lane quadrant of this warp
    const int hsel = (warp - 2) >> 2;     // which half of the chunk's columns (and of Q, O) this thread owns
    const int r = w4 * 32 + lane;
    const uint32_t trow = tmem + (static_cast<uint32_t>(w4 * 32) << 16);
    float* s_hmax = reinterpret_cast<float*>(base + SM::kXch);   // [2 halves][128 rows]
    float* s_l = s_hmax + 256;                                   // [128 rows]
    const float sl2 = kLog2e * rsqrtf(128.f);
    grid_dep_wait();   // q is written by the preceding kernel
    if (threadIdx.x == 64) trace_event(ts, 0);
    // this thread's query row of segment `sg` (half 0 the hi part, half 1 the lo part), or null
    // for a row past the tile's candidates
    auto q_row = [&](const AttnSeg& sg) -> const __nv_bfloat16* {
      const int ci = r / group, hr = r - ci * group;
      if (ci >= sg.n_cands) return nullptr;
      return (hsel ? q_lo : q_hi) +
             (static_cast<int64_t>(wk.cands[sg.cand + ci]) * n_q + static_cast<int64_t>(sg.g) * group + hr) * 128;
    };
    // Q of segment `sg` into TMEM, then the arrival that lets the S MMAs of the segment start (the
    // caller has seen every S MMA that read the previous segment's Q complete)
    auto q_in = [&](const AttnSeg& sg, uint32_t k) {
      const long long tq = tic();
      const __nv_bfloat16* src = q_row(sg);
      uint4 w[16];
#pragma unroll
      for (int e = 0; e < 16; ++e) w[e] = src ? *reinterpret_cast<const uint4*>(src + e * 8) : make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
      for (int j = 0; j < 4; ++j) {   // 32 head-dim elements = 16 columns per store
        float v[16];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          v[4 * e] = __uint_as_float(w[4 * j + e].x);
          v[4 * e + 1] = __uint_as_float(w[4 * j + e].y);
          v[4 * e + 2] = __uint_as_float(w[4 * j + e].z);
          v[4 * e + 3] = __uint_as_float(w[4 * j + e].w);
        }
        tmem_st16(trow + (hsel ? kColQlo : kColQhi) + j * 16, v);
      }
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(q_ready);
      if (lane == 0 && warp == 2) {
        toc(11, tq);
        event(6, k);
      }
    };
    uint32_t u = 0, k = 0;
    bool ok = true;
    if (seg0 < seg1) q_in(wk.segs[seg0], 0);
    for (int si = seg0; si < seg1; ++si, ++k) {
      const AttnSeg sg = wk.segs[si];
      const int nch = chunks(sg);
      const int ci = r / group, hr = r - ci * group;
      const bool live = ci < sg.n_cands;
      float m = -INFINITY, l = 0.f;
      for (int c = 0; c < nch; ++c, ++u) {
        if (c == nch - 1 && si + 1 < seg1) {   // the next segment's query row on its way to L1
          const __nv_bfloat16* nq = q_row(wk.segs[si + 1]);
          if (nq) {
            prefetch_l1(nq);
            prefetch_l1(nq + 64);
          }
        }
        const uint32_t b = u % kTcSBufs;
        long long t0 = tic();
        if (ok) ok = __all_sync(0xffffffffu, mbar_wait(&s_full[b], (u / kTcSBufs) & 1u, err));
        // tokens of my 32 that exist (none after a timeout: x is then never read)
        const int valid = ok ? min(kTcChunkPages, sg.n_pages - c * kTcChunkPages) * 16 - 32 * hsel : 0;
        tc_fence_after();
        if (lane == 0 && warp == 2) {
          toc(4, t0);
          event(2, u);
        }
        t0 = tic();
        float x[32];
        if (ok) {
          float v0[16], v1[16];
          tmem_ld16_nowait(trow + b * 64 + hsel * 32, v0);
          tmem_ld16_nowait(trow + b * 64 + hsel * 32 + 16, v1);
          tmem_wait_ld();
          tmem_hold(v0);
          tmem_hold(v1);
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            x[j] = v0[j];
            x[16 + j] = v1[j];
          }
        }
        if (lane == 0 && warp == 2) toc(8, t0);
        t0 = tic();
        float hm = -INFINITY;   // my half's maximum of the raw scores, then in log2 units
        if (valid >= 32) {
#pragma unroll
          for (int j = 0; j < 32; ++j) hm = fmaxf(hm, x[j]);
        } else {
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            x[j] = j < valid ? x[j] : -INFINITY;
            hm = fmaxf(hm, x[j]);
          }
        }
        hm *= sl2;
        s_hmax[hsel * 128 + r] = hm;
        tc_fence_before();   // my S loads are done before the other half may write P over them
        named_bar_sync(1, 256);
        const float mx = fmaxf(hm, s_hmax[(hsel ^ 1) * 128 + r]);
        named_bar_sync(1, 256);   // both halves have read before the next chunk overwrites
        tc_fence_after();
        const bool grow = mx > m + margin;   // else keep the stale maximum: 2^(s - m) <= 2^margin
        if (c > 0 && ok && __any_sync(0xffffffffu, grow)) {   // move my half of O to the new maximum
          const uint32_t pb = (u - 1) % kTcSBufs;
          const long long tr = tic();
          ok = __all_sync(0xffffffffu, mbar_wait(&pv_done[pb], ((u - 1) / kTcSBufs) & 1u, err));
          if (lane == 0 && warp == 2) toc(5, tr);
          tc_fence_after();
          const float alpha = grow ? exp2f(m - mx) : 1.f;
          if (ok) {
#pragma unroll 1
            for (int c0 = 0; c0 < 64; c0 += 16) {
              float v[16];
              tmem_ld16(trow + kColO + hsel * 64 + c0, v);
#pragma unroll
              for (int j = 0; j < 16; ++j) v[j] *= alpha;
              tmem_st16(trow + kColO + hsel * 64 + c0, v);
            }
            tmem_wait_st();
          }
        }
        if (grow) {
          l *= exp2f(m - mx);
          m = mx;
        }
        // P = 2^(s - m) for my 32 tokens as bf16 hi (columns hsel*16 ..) and lo (32 + hsel*16 ..):
        // hi = p truncated to bf16, lo = (p - hi) truncated, by bit masks: |p - hi - lo| < 2^-14 p
        float hv[16], lv[16];
        const float nm = -m;
#pragma unroll
        for (int e = 0; e < 16; ++e) {
          const float p0 = ex2_ftz(fmaf(x[2 * e], sl2, nm)), p1 = ex2_ftz(fmaf(x[2 * e + 1], sl2, nm));
          l += p0 + p1;
          const uint32_t h0 = __float_as_uint(p0) & 0xFFFF0000u, h1 = __float_as_uint(p1) & 0xFFFF0000u;
          const uint32_t l0 = __float_as_uint(p0 - __uint_as_float(h0));
          const uint32_t l1 = __float_as_uint(p1 - __uint_as_float(h1));
          hv[e] = __uint_as_float(__byte_perm(h0, h1, 0x7632));   // upper halves: (h0, h1)
          lv[e] = __uint_as_float(__byte_perm(l0, l1, 0x7632));
        }
        tmem_st16(trow + b * 64 + hsel * 16, hv);
        tmem_st16(trow + b * 64 + 32 + hsel * 16, lv);
        tmem_wait_st();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&p_full[b]);
        if (lane == 0 && warp == 2) {
          toc(9, t0);
          if (pr) atomicAdd(pr + 12, 1ull);
          event(3, u);
        }
      }
      if (threadIdx.x == 64 && si == seg1 - 1) trace_event(ts, 1);
      // every S MMA of this segment has completed (its last S was read above): the next segment's Q
      // goes into TMEM now, so that its S MMAs run while this segment's O is read out
      if (si + 1 < seg1) q_in(wk.segs[si + 1], k + 1);
      // the segment's partial slots: (m, l) and the unnormalised O of every live row, my half of O
      const uint32_t lb = (u - 1) % kTcSBufs;
      const long long to = tic();
      if (ok) ok = __all_sync(0xffffffffu, mbar_wait(&pv_done[lb], ((u - 1) / kTcSBufs) & 1u, err));
      tc_fence_after();
      if (hsel) s_l[r] = l;
      named_bar_sync(1, 256);
      if (ok) {
        const int slot = live ? wk.slots[sg.slot + ci] : 0;
        float* dst = part_o + (static_cast<int64_t>(slot) * group + hr) * 128 + hsel * 64;
        float v[4][16];
#pragma unroll
        for (int q = 0; q < 4; ++q) tmem_ld16_nowait(trow + kColO + hsel * 64 + q * 16, v[q]);
        tmem_wait_ld();
#pragma unroll
        for (int q = 0; q < 4; ++q) tmem_hold(v[q]);
        if (live) {
#pragma unroll
          for (int q = 0; q < 4; ++q)
#pragma unroll
            for (int j = 0; j < 16; j += 4)
              *reinterpret_cast<float4*>(dst + q * 16 + j) = make_float4(v[q][j], v[q][j + 1], v[q][j + 2], v[q][j + 3]);
          if (!hsel)
            *reinterpret_cast<float2*>(part_ml + (static_cast<int64_t>(slot) * group + hr) * 2) = make_float2(m, l + s_l[r]);
        }
      }
      named_bar_sync(1, 256);   // s_l is read before the next segment writes it
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(o_free);
      if (lane == 0 && warp == 2) {
        toc(10, to);
        event(7, k);
      }
    }
    if (threadIdx.x == 64) trace_event(ts, 2);
  }
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTcTmemCols);
  }
  if (threadIdx.x == 0) {
    toc(13, t_start);
    if (ev) ev[7 * 128 + 127] = static_cast<unsigned long long>(t_start);
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
cudaError_t set_smem(K kernel, size_t bytes) {
  return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(bytes));
}

uint64_t hash_list(const int32_t* v, int n) {
  uint64_t h = 1469598103934665603ull;
  for (int i = 0; i < n; ++i) {
    h ^= static_cast<uint32_t>(v[i]);
    h *= 1099511628211ull;
  }
  return h;
}

// A run of pages scored together: one candidate's private pages, or pages
// shared by one chunk (<= 8) of a candidate set.
struct Run {
  int kind;
  int cand;        // kind 0: candidate; kind 1: offset into cands
  int n_cands;
  int page_off;    // offset into pages
  int n_pages;
  int last_valid;
  int64_t cost;    // per page and kv head
};

}  // namespace

CUresult encode_pool_map(PFN_cuTensorMapEncodeTiled_v12000 encode, CUtensorMap* map, const void* pool,
                         int64_t page_units, int n_kv, int hd) {
  const cuuint64_t row = static_cast<cuuint64_t>(hd) * 2;   // bytes per token row
  cuuint64_t dims[5] = {64, 16, static_cast<cuuint64_t>(hd / 64), static_cast<cuuint64_t>(n_kv),
                        static_cast<cuuint64_t>(page_units) * 2};
  cuuint64_t strides[4] = {row, 128, 16 * row, static_cast<cuuint64_t>(n_kv) * 16 * row};
  cuuint32_t box[5] = {64, 16, static_cast<cuuint32_t>(hd / 64), 1, 2};
  cuuint32_t estr[5] = {1, 1, 1, 1, 1};
  return encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, const_cast<void*>(pool), dims, strides, box, estr,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
}

size_t attention_smem_bytes(int hd) {
  return hd == 128 ? AttnSmem<128>::kDynamic : AttnSmem<64>::kDynamic;
}

size_t attn_slot_capacity(int max_candidates, int n_kv, int num_sms) {
  // private runs: at most B * n_kv + n_ctas segments of at most 8 slots each
  return static_cast<size_t>(kConsumerWarps) * 2 * (static_cast<size_t>(max_candidates) * n_kv + num_sms);
}

// Host planner.
//  1. Shared pages: full pages that >= 2 candidates reference, each exactly
//     once, grouped by their exact candidate set; each set is cut into chunks
//     of <= 8 candidates (share = 1: scored by the persistent kernel, one
//     warp per candidate) or of <= 128 / G candidates (share = 2: one
//     tensor-core tile of up to 128 query rows, see attn_tc_kernel), one run
//     per chunk, except that chunks of the same kind with the same candidates
//     (from different sets) share one run over all their pages.  Every other
//     page of a candidate goes to its private run.
//  2. The (run, kv head) pairs are laid end to end on a cost axis (a page
//     costs kPrivateCost, or kSharedCostPerCand per candidate) and each page goes to the CTA whose
//     equal share of the axis holds the page's midpoint; the pages of a pair
//     that fall to one CTA form a segment.  A private segment adds one
//     partial slot (with G > 8 one per warp that gets a page, page i going
//     to warp i mod 8); a shared segment adds one per candidate.
//     Tensor-core runs (kind 2) stay off that axis: their (run, kv head)
//     pairs' 4-page chunks are laid end to end and cut into equal ranges, one
//     per CTA of the tensor-core launch (at most n_ctas); the chunks of a pair
//     falling to one CTA form a segment, stored after the persistent CTAs'
//     segments, with one slot per candidate.
//  3. The slots of each (candidate, kv head) are numbered consecutively from
//     slot_base.
// Falls back to private runs when sharing would need more than slot_limit
// slots; returns false if even those do not fit.
bool build_attn_work(const int32_t* bt, const int32_t* sl, int n, int max_blocks, int n_kv, int group, int n_ctas,
                     size_t slot_limit, int share, AttnWorkHost& w) {
  w.tc_seg0 = 0;
  w.n_tc = 0;
  w.n_tc_ctas = 0;
  w.tc_concurrent = false;
  w.tc_cta.clear();
  w.segs.clear();
  w.cta_seg.clear();
  w.pages.clear();
  w.cands.clear();
  w.slots.clear();
  w.slot_base.assign(static_cast<size_t>(n) * n_kv, 0);
  w.nslots.assign(static_cast<size_t>(n) * n_kv, 0);
  w.n_slots = 0;
  w.n_ctas = 0;
  if (n <= 0) {
    w.cta_seg.push_back(0);
    return true;
  }
  std::vector<int> np(n);
  int64_t total_refs = 0;
  for (int b = 0; b < n; ++b) {
    np[b] = (sl[b] + 15) / 16;
    total_refs += np[b];
  }
  // ---- 1. runs
  std::vector<uint8_t> is_shared(static_cast<size_t>(n) * max_blocks, 0);
  std::vector<Run> runs;
  if (share && total_refs > 0) {
    // Every full page's referencing candidates, in increasing candidate order.  Page ids up to a few
    // times the number of references index dense arrays (counts, offsets, one list of all
    // references: no allocation per page); sparser ids go through a hash map.
    int32_t max_page = -1, min_page = 0;
    int64_t full_refs = 0;
    for (int b = 0; b < n; ++b) {
      const int nfull = sl[b] / 16;
      full_refs += nfull;
      for (int j = 0; j < nfull; ++j) {
        const int32_t pg = bt[static_cast<int64_t>(b) * max_blocks + j];
        max_page = std::max(max_page, pg);
        min_page = std::min(min_page, pg);
      }
    }
    const bool dense = min_page >= 0 && static_cast<int64_t>(max_page) + 1 <= 8 * full_refs + 65536;
    std::vector<int32_t> ref_off, ref_list;                            // dense: CSR over page ids
    std::unordered_map<int32_t, std::vector<int32_t>> refs;           // sparse
    bool any_dup = false;
    if (dense) {
      ref_off.assign(static_cast<size_t>(max_page) + 2, 0);
      for (int b = 0; b < n; ++b)
        for (int j = 0, nfull = sl[b] / 16; j < nfull; ++j) ++ref_off[bt[static_cast<int64_t>(b) * max_blocks + j] + 1];
      for (size_t pg = 1; pg < ref_off.size(); ++pg) {
        any_dup = any_dup || ref_off[pg] > 1;
        ref_off[pg] += ref_off[pg - 1];
      }
      ref_list.resize(static_cast<size_t>(full_refs));
      std::vector<int32_t> fill(ref_off.begin(), ref_off.end() - 1);
      for (int b = 0; b < n; ++b)
        for (int j = 0, nfull = sl[b] / 16; j < nfull; ++j) ref_list[fill[bt[static_cast<int64_t>(b) * max_blocks + j]]++] = b;
    } else {
      refs.reserve(static_cast<size_t>(total_refs));
      for (int b = 0; b < n; ++b) {
        const int nfull = sl[b] / 16;
        for (int j = 0; j < nfull; ++j) {
          auto& v = refs[bt[static_cast<int64_t>(b) * max_blocks + j]];
          v.push_back(b);
          if (v.size() > 1) any_dup = true;
        }
      }
    }
    if (any_dup) {
      std::vector<std::vector<int32_t>> group_cands, group_pages;
      std::unordered_map<uint64_t, int> gidx;
      std::vector<uint8_t> in_group_dense(dense ? static_cast<size_t>(max_page) + 1 : 0, 0);
      std::unordered_map<int32_t, char> in_group;
      // a page referenced (in full) by the candidates c[0 .. len), in increasing order
      auto consider = [&](int32_t page, const int32_t* c, size_t len) {
        if (len < 2) return;
        for (size_t i = 1; i < len; ++i)
          if (c[i] == c[i - 1]) return;   // a candidate listing the page twice keeps it private
        const uint64_t h = hash_list(c, static_cast<int>(len));
        auto itg = gidx.find(h);
        int gi;
        if (itg != gidx.end()) {
          const std::vector<int32_t>& g = group_cands[itg->second];
          if (g.size() != len || !std::equal(g.begin(), g.end(), c)) return;   // hash collision: private
          gi = itg->second;
        } else {
          gi = static_cast<int>(group_cands.size());
          gidx.emplace(h, gi);
          group_cands.emplace_back(c, c + len);
          group_pages.emplace_back();
        }
        group_pages[gi].push_back(page);
        if (dense)
          in_group_dense[page] = 1;
        else
          in_group[page] = 1;
      };
      if (dense) {
        for (int32_t pg = 0; pg <= max_page; ++pg)
          consider(pg, ref_list.data() + ref_off[pg], static_cast<size_t>(ref_off[pg + 1] - ref_off[pg]));
      } else {
        for (auto& kv : refs) consider(kv.first, kv.second.data(), kv.second.size());
      }
      for (int b = 0; b < n; ++b) {
        const int nfull = sl[b] / 16;
        for (int j = 0; j < nfull; ++j) {
          const int32_t pg = bt[static_cast<int64_t>(b) * max_blocks + j];
          if (dense ? in_group_dense[pg] != 0 : in_group.count(pg) != 0) is_shared[static_cast<size_t>(b) * max_blocks + j] = 1;
        }
      }
      for (auto& pgs : group_pages) std::sort(pgs.begin(), pgs.end());   // deterministic contents
      std::vector<int> order(group_cands.size());   // deterministic group order
      for (size_t i = 0; i < order.size(); ++i) order[i] = static_cast<int>(i);
      std::sort(order.begin(), order.end(),
                [&](int a, int b2) { return group_pages[a].front() < group_pages[b2].front(); });
      // Runs: each group's candidates cut into tiles; tiles of the same kind with the same candidate
      // list (an MCTS tile of 16 leaves under a depth-1 edge and the depth-2 edge above those same
      // leaves) become one run over both groups' pages, so that its query rows are loaded and its
      // partials written once.  Attention is invariant to the order of the keys.
      struct Tile {
        int kind;
        std::vector<int32_t> cands;
        std::vector<int> groups;
      };
      std::vector<Tile> tiles;
      std::unordered_map<uint64_t, std::vector<int>> tile_idx;   // hash of (kind, candidates) -> tiles
      for (int gi : order) {
        const auto& c = group_cands[gi];
        // tensor-core tiles: as few as possible, with the candidates spread evenly over them
        const bool tc = share >= 2 && c.size() >= kTcMinCands;
        const size_t per = tc ? static_cast<size_t>(kTcRows / group) : static_cast<size_t>(kConsumerWarps);
        const size_t n_chunks = (c.size() + per - 1) / per;
        for (size_t k = 0, c0 = 0; k < n_chunks; ++k) {
          const size_t c1 = tc ? c.size() * (k + 1) / n_chunks : std::min(c.size(), c0 + per);
          const int kind = tc ? 2 : 1;
          const uint64_t h = hash_list(c.data() + c0, static_cast<int>(c1 - c0)) * 3 + static_cast<uint64_t>(kind);
          int ti = -1;
          for (int t : tile_idx[h])
            if (tiles[t].kind == kind && tiles[t].cands.size() == c1 - c0 &&
                std::equal(tiles[t].cands.begin(), tiles[t].cands.end(), c.begin() + c0))
              ti = t;
          if (ti < 0) {
            ti = static_cast<int>(tiles.size());
            tiles.push_back(Tile{kind, std::vector<int32_t>(c.begin() + c0, c.begin() + c1), {}});
            tile_idx[h].push_back(ti);
          }
          tiles[ti].groups.push_back(gi);
          c0 = c1;
        }
      }
      std::vector<int> group_off(group_cands.size(), -1);   // a single group's pages, stored once
      for (const Tile& t : tiles) {
        Run r;
        r.kind = t.kind;
        r.cand = static_cast<int>(w.cands.size());
        r.n_cands = static_cast<int>(t.cands.size());
        if (t.groups.size() == 1) {
          const int gi = t.groups[0];
          if (group_off[gi] < 0) {
            group_off[gi] = static_cast<int>(w.pages.size());
            w.pages.insert(w.pages.end(), group_pages[gi].begin(), group_pages[gi].end());
          }
          r.page_off = group_off[gi];
          r.n_pages = static_cast<int>(group_pages[gi].size());
        } else {
          r.page_off = static_cast<int>(w.pages.size());
          for (int gi : t.groups) w.pages.insert(w.pages.end(), group_pages[gi].begin(), group_pages[gi].end());
          r.n_pages = static_cast<int>(w.pages.size()) - r.page_off;
        }
        r.last_valid = 16;
        r.cost = kSharedCostPerCand * r.n_cands;
        w.cands.insert(w.cands.end(), t.cands.begin(), t.cands.end());
        runs.push_back(r);
      }
    }
  }
  for (int b = 0; b < n; ++b) {
    Run r;
    r.kind = 0;
    r.cand = b;
    r.n_cands = 1;
    r.page_off = static_cast<int>(w.pages.size());
    r.last_valid = 16;
    for (int j = 0; j < np[b]; ++j)
      if (!is_shared[static_cast<size_t>(b) * max_blocks + j]) {
        w.pages.push_back(bt[static_cast<int64_t>(b) * max_blocks + j]);
        if (j == np[b] - 1) r.last_valid = sl[b] - 16 * (np[b] - 1);
      }
    r.n_pages = static_cast<int>(w.pages.size()) - r.page_off;
    if (r.n_pages == 0) continue;   // an empty cache, or every page shared
    r.cost = kPrivateCost;
    runs.push_back(r);
  }
  // ---- 2. cut the cost axis into C equal ranges (at least a stage of work each)
  int64_t total = 0, tc_chunks = 0;
  for (const Run& r : runs) {
    if (r.kind == 2)
      tc_chunks += static_cast<int64_t>((r.n_pages + kTcChunkPages - 1) / kTcChunkPages) * n_kv;
    else
      total += static_cast<int64_t>(r.n_pages) * r.cost * n_kv;
  }
  // SMs for the private launch: all of them, or (share 3, both kinds of work) the split that makes
  // the later of the two launches end soonest when they run side by side
  int priv_ctas = n_ctas, tc_ctas = n_ctas;
  if (share == 3 && total > 0 && tc_chunks > 0 && n_ctas >= 2) {
    int64_t best = INT64_MAX;
    for (int x = 1; x < n_ctas; ++x) {
      const int64_t t_tc = (tc_chunks + x - 1) / x * kTcChunkCost + kTcCtaCost;
      const int64_t t_pr = (total + (n_ctas - x) - 1) / (n_ctas - x);
      const int64_t t = std::max(t_tc, t_pr);
      if (t < best) {
        best = t;
        tc_ctas = x;
      }
    }
    priv_ctas = n_ctas - tc_ctas;
    w.tc_concurrent = true;
  }
  const int C = total == 0 ? 0
                           : static_cast<int>(std::max<int64_t>(
                                 1, std::min<int64_t>(priv_ctas, total / (kPagesPerStage * kPrivateCost))));
  // The (run, kv head) pairs in axis order: the pairs of shared runs (bound by their MMAs: a warp
  // per candidate scores every page) interleaved with the private pairs (bound by HBM) in proportion
  // to their cost, so that every CTA's range mixes both kinds and its ring fetches the private pages
  // of a later segment while its warps score the shared pages of the current one.
  std::vector<std::pair<int, int>> pairs;
  {
    std::vector<std::pair<int, int>> sh, pv;
    int64_t c_sh = 0, c_pv = 0;
    for (size_t ri = 0; ri < runs.size(); ++ri) {
      const Run& r = runs[ri];
      if (r.kind == 2) continue;
      for (int g = 0; g < n_kv; ++g) (r.kind == 1 ? sh : pv).emplace_back(static_cast<int>(ri), g);
      (r.kind == 1 ? c_sh : c_pv) += static_cast<int64_t>(r.n_pages) * r.cost * n_kv;
    }
    auto cost_of = [&](const std::pair<int, int>& pr) {
      return static_cast<int64_t>(runs[pr.first].n_pages) * runs[pr.first].cost;
    };
    size_t a = 0, b = 0;
    int64_t d_sh = 0, d_pv = 0;   // cost laid so far of each kind
    while (a < sh.size() || b < pv.size()) {
      // the kind whose laid fraction of its own total is smaller goes next
      const bool take_sh = b >= pv.size() || (a < sh.size() && d_sh * c_pv <= d_pv * c_sh);
      if (take_sh) {
        d_sh += cost_of(sh[a]);
        pairs.push_back(sh[a++]);
      } else {
        d_pv += cost_of(pv[b]);
        pairs.push_back(pv[b++]);
      }
    }
  }
  std::vector<int> seg_cta;
  int64_t pos = 0;   // cost position of the current pair's first unit
  for (const auto& pr : pairs) {
    const Run& r = runs[pr.first];
    {
      const int g = pr.second;
      const int units = r.n_pages;
      const int64_t c = r.cost;
      int i = 0;
      while (i < units) {
        // CTA of unit i: floor((2 pos + (2 i + 1) c) C / (2 total))
        const int k = static_cast<int>(((2 * pos + (2 * static_cast<int64_t>(i) + 1) * c) * C) / (2 * total));
        // first unit of a later CTA: the smallest e with (2 pos + (2 e + 1) c) C >= 2 total (k + 1)
        const int64_t num = 2 * total * (k + 1) - (2 * pos + c) * C;
        int64_t e = num <= 0 ? 0 : (num + 2 * c * C - 1) / (2 * c * C);
        e = std::min<int64_t>(std::max<int64_t>(e, i + 1), units);
        AttnSeg s;
        s.kind = r.kind;
        s.g = g;
        s.cand = r.cand;
        s.n_cands = r.n_cands;
        s.page_off = r.page_off + i;
        s.n_pages = static_cast<int>(e - i);
        s.last_valid = e == units ? r.last_valid : 16;
        if (r.kind == 0) {   // one slot (the merger's), or one per warp that gets a page when G > 8
          int32_t& ns = w.nslots[static_cast<size_t>(r.cand) * n_kv + g];
          s.slot = ns;
          ns += group > 8 ? std::min(s.n_pages, kConsumerWarps) : 1;
        } else {
          s.slot = static_cast<int>(w.slots.size());   // slot w of the segment: warp w (shared_reps)
          for (int w2 = 0; w2 < shared_reps(r.n_cands) * r.n_cands; ++w2)
            w.slots.push_back(w.nslots[static_cast<size_t>(w.cands[r.cand + w2 % r.n_cands]) * n_kv + g]++);
        }
        w.segs.push_back(s);
        seg_cta.push_back(k);
        i = static_cast<int>(e);
      }
      pos += static_cast<int64_t>(units) * c;
    }
  }
  // tensor-core work: the (run, kv head) pairs' 4-page chunks laid end to end
  // and cut into equal ranges, one per CTA of the tensor-core launch; a pair's
  // chunks falling to one CTA form a segment (one slot per candidate)
  w.tc_seg0 = static_cast<int>(w.segs.size());
  w.tc_cta.clear();
  w.n_tc_ctas = 0;
  if (tc_chunks > 0) {
    const int64_t T = tc_chunks;
    const int Ct = static_cast<int>(std::min<int64_t>(tc_ctas, T));
    std::vector<int> tc_seg_cta;
    int64_t at = 0;   // chunk position of the current pair's first chunk
    for (const Run& r : runs) {
      if (r.kind != 2) continue;
      const int nch = (r.n_pages + kTcChunkPages - 1) / kTcChunkPages;
      for (int g = 0; g < n_kv; ++g) {
        for (int i = 0; i < nch;) {
          const int k = static_cast<int>((at + i) * Ct / T);                 // CTA of chunk i
          const int64_t next = ((k + 1) * T + Ct - 1) / Ct;                  // first chunk of CTA k + 1
          const int e = static_cast<int>(std::min<int64_t>(nch, std::max<int64_t>(i + 1, next - at)));
          AttnSeg sg;
          sg.kind = 2;
          sg.g = g;
          sg.cand = r.cand;
          sg.n_cands = r.n_cands;
          sg.page_off = r.page_off + i * kTcChunkPages;
          sg.n_pages = std::min(r.n_pages, e * kTcChunkPages) - i * kTcChunkPages;
          sg.last_valid = 16;
          sg.slot = static_cast<int>(w.slots.size());
          for (int k2 = 0; k2 < r.n_cands; ++k2)
            w.slots.push_back(w.nslots[static_cast<size_t>(w.cands[r.cand + k2]) * n_kv + g]++);
          w.segs.push_back(sg);
          tc_seg_cta.push_back(k);
          i = e;
        }
        at += nch;
      }
    }
    w.n_tc_ctas = Ct;
    w.tc_cta.assign(Ct + 1, 0);
    for (int k : tc_seg_cta) w.tc_cta[k + 1]++;
    for (int k = 0; k < Ct; ++k) w.tc_cta[k + 1] += w.tc_cta[k];
    for (int32_t& v : w.tc_cta) v += w.tc_seg0;   // indices into segs
  }
  w.n_tc = static_cast<int>(w.segs.size()) - w.tc_seg0;
  // ---- 3. slot numbering
  size_t next = 0;
  for (size_t cg = 0; cg < w.nslots.size(); ++cg) {
    w.slot_base[cg] = static_cast<int32_t>(next);
    next += static_cast<size_t>(w.nslots[cg]);
  }
  if (next > slot_limit) {
    if (share) return build_attn_work(bt, sl, n, max_blocks, n_kv, group, n_ctas, slot_limit, 0, w);
    return false;
  }
  w.n_slots = static_cast<int>(next);
  for (AttnSeg& s : w.segs) {
    if (s.kind == 0)
      s.slot += w.slot_base[static_cast<size_t>(s.cand) * n_kv + s.g];
    else   // kind 1: shared_reps(n) * n slots, slot w for candidate w % n; kind 2: one per candidate
      for (int k2 = 0; k2 < (s.kind == 1 ? shared_reps(s.n_cands) : 1) * s.n_cands; ++k2)
        w.slots[s.slot + k2] += w.slot_base[static_cast<size_t>(w.cands[s.cand + k2 % s.n_cands]) * n_kv + s.g];
  }
  w.n_ctas = C;
  w.cta_seg.assign(C + 1, 0);
  for (int k : seg_cta) w.cta_seg[k + 1]++;
  for (int k = 0; k < C; ++k) w.cta_seg[k + 1] += w.cta_seg[k];
  return true;
}

bool build_attn_work_fused(const int32_t* bt, const int32_t* sl, int n, int max_blocks, int n_kv, int group,
                           int n_ctas, size_t slot_limit, AttnWorkHost& w) {
  if (n <= 0 || group > 8 || n_kv < 1) return false;
  int lo = INT32_MAX, hi = 0;
  for (int b = 0; b < n; ++b) {
    const int np = (sl[b] + 15) / 16;
    lo = std::min(lo, np);
    hi = std::max(hi, np);
  }
  if (lo < 1 || 4 * hi > 5 * lo) return false;   // equal ranges need about equal lengths
  const int64_t pairs = static_cast<int64_t>(n) * n_kv;
  int cs = 0;
  for (int c = 8; c >= 1; c >>= 1)
    if (pairs * c <= n_ctas && c <= lo) {
      cs = c;
      break;
    }
  if (cs == 0 || (hi + cs - 1) / cs > kFuseMaxPages) return false;
  if (static_cast<size_t>(pairs) * cs > slot_limit) return false;
  {   // a page referenced twice (sharing, or a repeat) is left to the persistent plan
    int32_t pmin = 0, pmax = -1;
    int64_t refs = 0;
    for (int b = 0; b < n; ++b)
      for (int j = 0, np = (sl[b] + 15) / 16; j < np; ++j, ++refs) {
        pmin = std::min(pmin, bt[static_cast<int64_t>(b) * max_blocks + j]);
        pmax = std::max(pmax, bt[static_cast<int64_t>(b) * max_blocks + j]);
      }
    if (pmin >= 0 && static_cast<int64_t>(pmax) + 1 <= 8 * refs + 65536) {   // dense page ids: a flag each
      std::vector<uint8_t> seen(static_cast<size_t>(pmax) + 1, 0);
      for (int b = 0; b < n; ++b)
        for (int j = 0, np = (sl[b] + 15) / 16; j < np; ++j) {
          uint8_t& f = seen[bt[static_cast<int64_t>(b) * max_blocks + j]];
          if (f) return false;
          f = 1;
        }
    } else {
      std::unordered_map<int32_t, char> seen;
      seen.reserve(static_cast<size_t>(refs));
      for (int b = 0; b < n; ++b)
        for (int j = 0, np = (sl[b] + 15) / 16; j < np; ++j)
          if (!seen.emplace(bt[static_cast<int64_t>(b) * max_blocks + j], 1).second) return false;
    }
  }
  w = AttnWorkHost();
  w.fuse_cs = cs;
  w.slot_base.assign(static_cast<size_t>(pairs), 0);
  w.nslots.assign(static_cast<size_t>(pairs), cs);
  w.cta_seg.reserve(static_cast<size_t>(pairs) * cs + 1);
  w.cta_seg.push_back(0);
  for (int b = 0; b < n; ++b) {
    const int np = (sl[b] + 15) / 16;
    const int page_off = static_cast<int>(w.pages.size());
    for (int j = 0; j < np; ++j) w.pages.push_back(bt[static_cast<int64_t>(b) * max_blocks + j]);
    for (int g = 0; g < n_kv; ++g) {
      const int pr = b * n_kv + g;
      w.slot_base[pr] = pr * cs;
      for (int r = 0; r < cs; ++r) {   // rank r: pages [r np / cs, (r + 1) np / cs)
        const int p0 = r * np / cs, p1 = (r + 1) * np / cs;
        AttnSeg sg;
        sg.kind = 0;
        sg.g = g;
        sg.cand = b;
        sg.n_cands = 1;
        sg.page_off = page_off + p0;
        sg.n_pages = p1 - p0;
        sg.last_valid = p1 == np ? sl[b] - 16 * (np - 1) : 16;
        sg.slot = pr * cs + r;
        w.segs.push_back(sg);
        w.cta_seg.push_back(static_cast<int32_t>(w.segs.size()));
      }
    }
  }
  w.n_ctas = static_cast<int>(pairs * cs);
  w.n_slots = static_cast<int>(pairs * cs);
  w.tc_seg0 = static_cast<int>(w.segs.size());
  return true;
}

cudaError_t attention_configure() {
  cudaError_t e;
#define KVPRM_COMBINE_SMEM(HD_, R_, W_)                                                                           \
  if ((e = set_smem(attn_combine_kernel<HD_, R_, W_, false>, CombineShape<HD_, R_, W_>::kBytes)) != cudaSuccess) \
    return e;                                                                                                    \
  if ((e = set_smem(attn_combine_kernel<HD_, R_, W_, true>, CombineShape<HD_, R_, W_>::kBytes)) != cudaSuccess)  \
    return e;
  KVPRM_COMBINE_SMEM(64, 8, 8)
  KVPRM_COMBINE_SMEM(64, 16, 8)
  KVPRM_COMBINE_SMEM(128, 8, 8)
  KVPRM_COMBINE_SMEM(128, 16, 8)
  KVPRM_COMBINE_SMEM(64, 8, 4)
  KVPRM_COMBINE_SMEM(64, 16, 4)
  KVPRM_COMBINE_SMEM(128, 8, 4)
  KVPRM_COMBINE_SMEM(128, 16, 4)
#undef KVPRM_COMBINE_SMEM
  if ((e = set_smem(attn_kernel<64, false>, AttnSmem<64>::kDynamic)) != cudaSuccess) return e;
  if ((e = set_smem(attn_kernel<64, true>, AttnSmem<64>::kDynamic)) != cudaSuccess) return e;
  if ((e = set_smem(attn_kernel<128, false>, AttnSmem<128>::kDynamic)) != cudaSuccess) return e;
  if ((e = set_smem(attn_tc_kernel, TcSmem::kDynamic)) != cudaSuccess) return e;
  return set_smem(attn_kernel<128, true>, AttnSmem<128>::kDynamic);
}

cudaError_t launch_attention(const AttnShape& s, const AttnWork& wk, const CUtensorMap* tm_pool, int layer,
                             const __nv_bfloat16* q_hi, const __nv_bfloat16* q_lo, float* part_o, float* part_ml,
                             const AttnMerge& mg, int* err, cudaStream_t stream, bool pdl, unsigned long long* ts) {
  if (wk.n_ctas == 0) return cudaSuccess;
  if (wk.fuse_cs > 0 && (wk.n_ctas % wk.fuse_cs != 0 || wk.fuse_cs > 8)) return cudaErrorInvalidValue;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(wk.n_ctas, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = attention_smem_bytes(s.hd);
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  int na = 0;
  if (pdl) {
    attr[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[na].val.programmaticStreamSerializationAllowed = 1;
    ++na;
  }
  if (wk.fuse_cs > 0) {
    attr[na].id = cudaLaunchAttributeClusterDimension;
    attr[na].val.clusterDim.x = static_cast<unsigned>(wk.fuse_cs);
    attr[na].val.clusterDim.y = 1;
    attr[na].val.clusterDim.z = 1;
    ++na;
  }
  cfg.attrs = attr;
  cfg.numAttrs = na;
  const int64_t page0 = static_cast<int64_t>(layer) * s.layer_pages;
  const bool two = s.group > 8;
  if (s.hd == 128) {
    if (two)
      return cudaLaunchKernelEx(&cfg, attn_kernel<128, true>, *tm_pool, page0, wk, q_hi, q_lo, s.n_q, s.n_kv, s.group,
                                part_o, part_ml, mg, err, ts);
    return cudaLaunchKernelEx(&cfg, attn_kernel<128, false>, *tm_pool, page0, wk, q_hi, q_lo, s.n_q, s.n_kv, s.group,
                              part_o, part_ml, mg, err, ts);
  }
  if (two)
    return cudaLaunchKernelEx(&cfg, attn_kernel<64, true>, *tm_pool, page0, wk, q_hi, q_lo, s.n_q, s.n_kv, s.group,
                              part_o, part_ml, mg, err, ts);
  return cudaLaunchKernelEx(&cfg, attn_kernel<64, false>, *tm_pool, page0, wk, q_hi, q_lo, s.n_q, s.n_kv, s.group,
                            part_o, part_ml, mg, err, ts);
}

CUresult encode_pool_map_tc(PFN_cuTensorMapEncodeTiled_v12000 encode, CUtensorMap* map, const void* pool,
                            int64_t page_units, int n_kv, int hd) {
  const cuuint64_t row = static_cast<cuuint64_t>(hd) * 2;   // bytes per token row
  cuuint64_t dims[5] = {64, 16, static_cast<cuuint64_t>(hd / 64), static_cast<cuuint64_t>(n_kv),
                        static_cast<cuuint64_t>(page_units) * 2};
  cuuint64_t strides[4] = {row, 128, 16 * row, static_cast<cuuint64_t>(n_kv) * 16 * row};
  cuuint32_t box[5] = {64, 16, 1, 1, 1};
  cuuint32_t estr[5] = {1, 1, 1, 1, 1};
  return encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, const_cast<void*>(pool), dims, strides, box, estr,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
}

cudaError_t launch_attention_tc(const AttnShape& s, const AttnWork& wk, const CUtensorMap* tm_pool_tc, int layer,
                                const __nv_bfloat16* q_hi, const __nv_bfloat16* q_lo, float* part_o, float* part_ml,
                                float margin, int* err, cudaStream_t stream, bool pdl, unsigned long long* ts,
                                unsigned long long* prof) {
  if (wk.n_tc == 0 || wk.n_tc_ctas == 0) return cudaSuccess;
  if (s.hd != 128) return cudaErrorInvalidValue;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(wk.n_tc_ctas, 1, 1);
  cfg.blockDim = dim3(kTcThreads, 1, 1);
  cfg.dynamicSmemBytes = TcSmem::kDynamic;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  const int64_t page0 = static_cast<int64_t>(layer) * s.layer_pages;
  return cudaLaunchKernelEx(&cfg, attn_tc_kernel, *tm_pool_tc, page0, wk, q_hi, q_lo, s.n_q, s.group, part_o, part_ml,
                            margin, err, ts, prof);
}

cudaError_t launch_attn_combine(const AttnShape& s, const AttnWork& wk, int n, const float* part_o,
                                const float* part_ml, const AttnMerge& mg, cudaStream_t stream, bool pdl,
                                unsigned long long* ts, bool force_flat) {
  if (n == 0) return cudaSuccess;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(n) * s.n_kv, 1, 1);

  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  const bool two = s.group > 8;
  // 8 warps per (candidate, kv head) while the launch fits one wave (<= 6 CTAs of 256 threads per SM),
  // else 4 (half the shared memory and threads: one wave up to ~12 per SM)
  static int sms = 0;
  if (sms == 0) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) !=
                                                 cudaSuccess)
      sms = 1;
  }
  const int64_t pairs = static_cast<int64_t>(n) * s.n_kv;
  const bool narrow = pairs > 6 * static_cast<int64_t>(sms);
  // A single verify token per candidate with more (candidate, kv head) pairs than SMs: the flat
  // combine, one memory round trip per warp (beam's 256 pairs: 17.09k -> 17.30k scores/s; MCTS's
  // 1,024, where the general form's 4-warp CTAs took two waves of several round trips: ~1 %); fewer
  // pairs keep the general form (long 8B's 64: the flat form 0.6 % slower).
  if (mg.depth == 1 && (pairs > sms || force_flat)) {
    cfg.dynamicSmemBytes = 0;
    cfg.blockDim = dim3(32 * static_cast<unsigned>(s.group), 1, 1);
    if (s.hd == 128)
      return cudaLaunchKernelEx(&cfg, attn_combine_flat_kernel<128>, wk.slot_base, wk.nslots, s.n_q, s.n_kv, s.group,
                                part_o, part_ml, mg, ts);
    return cudaLaunchKernelEx(&cfg, attn_combine_flat_kernel<64>, wk.slot_base, wk.nslots, s.n_q, s.n_kv, s.group,
                              part_o, part_ml, mg, ts);
  }
#define KVPRM_COMBINE_W(HD_, R_, W_)                                                                               \
  do {                                                                                                           \
    cfg.dynamicSmemBytes = CombineShape<HD_, R_, W_>::kBytes;                                                    \
    cfg.blockDim = dim3(32 * W_, 1, 1);                                                                          \
    if (mg.depth > 1)                                                                                            \
      return cudaLaunchKernelEx(&cfg, attn_combine_kernel<HD_, R_, W_, true>, wk.slot_base, wk.nslots, s.n_q,    \
                                s.n_kv, s.group, part_o, part_ml, mg, ts);                                       \
    return cudaLaunchKernelEx(&cfg, attn_combine_kernel<HD_, R_, W_, false>, wk.slot_base, wk.nslots, s.n_q,     \
                              s.n_kv, s.group, part_o, part_ml, mg, ts);                                         \
  } while (0)
#define KVPRM_COMBINE(HD_, R_)             \
  do {                                     \
    if (narrow) KVPRM_COMBINE_W(HD_, R_, 4); \
    KVPRM_COMBINE_W(HD_, R_, 8);           \
  } while (0)
  if (s.hd == 128) {
    if (two) KVPRM_COMBINE(128, 16);
    KVPRM_COMBINE(128, 8);
  }
  if (two) KVPRM_COMBINE(64, 16);
  KVPRM_COMBINE(64, 8);
#undef KVPRM_COMBINE
#undef KVPRM_COMBINE_W
}

cudaError_t launch_resolve(const int32_t* bt, const int32_t* seq_lens, int max_blocks, int b, int64_t* out,
                           cudaStream_t stream) {
  resolve_kernel<<<64, 256, 0, stream>>>(bt, seq_lens, max_blocks, b, out);
  return cudaGetLastError();
}

}  // namespace kvprm
