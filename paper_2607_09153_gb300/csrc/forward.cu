// The verify-token forward of every layer (Sec. 4.1; the per-layer cost
// c_attn d L + c_ffn d^2 of Eq. cost_kv) as ONE persistent kernel: one CTA per
// SM runs every layer's QKV projection, paged attention, combine, O projection,
// gate/up projection and down projection.
//
// Why one kernel: the work is a stream of bytes (each layer's weights once, the
// candidates' cached K/V once) with a chain of small data dependencies between
// the steps.  Separate launches drain the memory pipe at every step boundary;
// here the bytes never wait for the dependencies.  Each CTA runs a static
// program, identical for every layer:
//   QKV pieces -> attention segments -> (combine) -> O pieces -> gate/up pieces
//   -> down pieces
// and its warps split the roles:
//   warp 0  producer: walks the whole program (all layers) and streams every
//           weight tile (TMA 2-D, 128 rows x 64 K, 16 KB) and every K/V page
//           (TMA 5-D, K and V of one kv head) into one ring of 16 KB slots.
//           It waits only for free slots, never for activations, so it runs
//           ahead across step and layer boundaries.
//   warp 1  MMA issuer: tcgen05.mma (kind::f16, M = 128 weight rows, N = the
//           candidate batch padded to 16, K = 16) of each piece into one of two
//           TMEM accumulators; the activation enters as a bf16 (hi, lo) pair,
//           two MMAs per K step, so the contraction sees the fp32 activation.
//   warp 2  activation loader: the piece's activation tiles (TMA, L2-resident)
//           once the step that writes them has completed everywhere.
//   warp 3  merger: folds the eight attention warps' states of a private run.
//   warps 4..11  math: attention (mma.sync, online softmax; attn_core.cuh),
//           the combine, and the projection epilogues: drain the TMEM
//           accumulator and add it into the tile's fp32 accumulator in L2
//           (red.add.v4); the last piece of a tile to arrive (an atomic per
//           tile) reads the sum, clears it and applies the step's epilogue:
//             QKV    RMSNorm factor, RoPE -> q (fp32 and hi/lo), self k, self v
//             O      h += y, per-tile sum of squares, x = h ⊙ g_mlp (hi/lo)
//             gate/up  RMSNorm factor, a = SiLU(gate) * up (hi/lo)
//             down   h += y, per-tile sum of squares, x = h ⊙ g_attn(next)
// Steps hand over through monotonic counters in global memory (release:
// fence + atomic add; acquire: ld.acquire polling), zeroed per call:
//   QKV(l) loads x      after done[down] = l * T_down
//   attention(l)        after done[QKV] = (l + 1) * T_qkv
//   combine(l)          after every CTA finished attention(l)
//   O(l) loads o        after every CTA finished combine(l)
//   gate/up(l) loads x  after done[O] = (l + 1) * T_o
//   down(l) loads a     after done[gate/up] = (l + 1) * T_gu
// The program order of every CTA lists a step's ring items after those of the
// steps it depends on, so no wait can close a cycle; every wait is bounded.
#include <cuda_bf16.h>

#include <algorithm>

#include "attn_core.cuh"
#include "kernels.h"
#include "ptx.cuh"

namespace kvprm {

namespace {

using namespace ac;

constexpr int kThreads = 384;
constexpr int kWarpProducer = 0, kWarpMma = 1, kWarpX = 2, kWarpMerger = 3, kWarpMath0 = 4;
constexpr int kMathThreads = 256;
constexpr uint32_t kSlot = 16384;
constexpr int kMaxSlots = 16, kMaxXStages = 8;
constexpr uint32_t kResidentBytes = 65536;   // activation slice of a resident step
constexpr int kBarMath = 1;   // named barrier: the 8 math warps
constexpr int kBarAttn = 2;   // named barrier: merger + math warps
constexpr int kPhases = 6;    // trace: QKV, attention, combine, O, gate/up, down
constexpr int kProbeEvents = 48;
constexpr uint32_t kMaxSmem = 232448;   // 227 KB per CTA (opt-in)
// codes a timed-out wait records in the error word (the first one wins)
enum : int {
  kSiteProdAttn = 10, kSiteProdW, kSiteMmaAcc = 20, kSiteMmaW, kSiteMmaX, kSiteXEmpty = 30, kSiteXDep = 31,
  kSiteMerger = 40, kSiteDrain = 50, kSiteQ, kSiteAttnDone, kSiteAttnFull, kSiteSegFree
};

// misc area (after the ring and the aux area)
constexpr uint32_t kMiscBars = 0;                          // mbarriers, 64 x 8 B
constexpr uint32_t kMiscRel = 512;                         // attention release counters per slot [16]
constexpr uint32_t kMiscTmem = kMiscRel + 4 * kMaxSlots;   // TMEM base
constexpr uint32_t kMiscFlag = kMiscTmem + 4;              // last-arriver flag / wait result
constexpr uint32_t kMiscCnt = kMiscFlag + 12;              // ring slots per step of this CTA [8]
constexpr uint32_t kMiscRs = 640;                          // RMSNorm factor per candidate [256]
constexpr uint32_t kMiscSq = kMiscRs + 4 * 256;            // sum-of-squares partials [256][4]
constexpr uint32_t kMiscBytes = kMiscSq + 4 * 256 * 4;

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~static_cast<uintptr_t>(1023));
}
__device__ __forceinline__ void store_hilo(__nv_bfloat16* hi, __nv_bfloat16* lo, int64_t i, float x) {
  const __nv_bfloat16 h = __float2bfloat16_rn(x);
  hi[i] = h;
  lo[i] = __float2bfloat16_rn(x - __bfloat162float(h));
}
__device__ __forceinline__ void trace_phase(const FwdArgs& a, int l, int ph, int mt) {
  if (a.phase_ts && mt == 0) atomicMax(a.phase_ts + 1 + l * kPhases + ph, static_cast<unsigned long long>(global_timer_ns()));
}
__device__ __forceinline__ void red_add_v4(float* p, float a0, float a1, float a2, float a3) {
  asm volatile("red.global.add.v4.f32 [%0], {%1, %2, %3, %4};" ::"l"(p), "f"(a0), "f"(a1), "f"(a2), "f"(a3)
               : "memory");
}
// Optional event timeline of each CTA: probe[cta][layer][event] (global timer,
// ns).  Events 3 k + {0, 1, 2} for projection kind k: its activations became
// ready (loader), its last MMA was committed, its drains and epilogues ended;
// 12..15: the query became ready, attention ended, the combine could start, the
// combine ended.
__device__ __forceinline__ void probe(const FwdArgs& a, int l, int ev) {
  if (a.probe) a.probe[(static_cast<int64_t>(blockIdx.x) * a.n_layers + l) * kProbeEvents + ev] = global_timer_ns();
}
// Events 16.. hold durations (ns) summed over the step: 16 + k the MMA issuer's
// waits for weight slots of projection k, 20 + k its waits for activation
// stages, 24 + k the drains' release fences, 28 + k tile arrival (atomic and
// flag broadcast).
__device__ __forceinline__ void probe_set(const FwdArgs& a, int l, int ev, uint64_t ns) {
  if (a.probe) a.probe[(static_cast<int64_t>(blockIdx.x) * a.n_layers + l) * kProbeEvents + ev] = ns;
}
// step `ph` of the program (0 QKV, 1 attention, 2 O, 3 gate/up, 4 down) -> projection kind
__device__ __forceinline__ int kind_of(int ph) { return ph == 0 ? FWD_QKV : ph - 1; }

// RMSNorm factor 1/sqrt(mean(h^2) + eps) of every candidate from the per-tile
// sums of squares, into s_rs; math threads only.  The loads are spread over
// all threads (thread (r, c) sums tiles r, r + R, ... of candidate c) and the R
// partial sums are added in a fixed order, so every caller gets the same value.
__device__ __forceinline__ void rms_factors(const FwdArgs& a, int mt, float* s_rs, float* s_part) {
  const int n = a.n, R = kMathThreads / n;   // n <= 256
  if (mt < R * n) {
    const int c = mt % n, r = mt / n;
    float s = 0.f;
#pragma unroll 4
    for (int t = r; t < a.d_tiles; t += R) s += __ldcg(a.sumsq + static_cast<int64_t>(t) * n + c);
    s_part[r * n + c] = s;
  }
  named_bar_sync(kBarMath, kMathThreads);
  for (int c = mt; c < n; c += kMathThreads) {
    float s = 0.f;
    for (int r = 0; r < R; ++r) s += s_part[r * n + c];
    s_rs[c] = 1.0f / sqrtf(s / a.d + a.eps);
  }
  named_bar_sync(kBarMath, kMathThreads);
}

// The epilogue of projection tile `t` (layer l), run by the 256 math threads
// of the CTA whose piece completed the tile.  Every piece of the tile has added
// its partial product into the tile accumulator acc[t][128 rows][n_pad] (vector
// reductions in L2); the epilogue reads each 4-column chunk once, clears it for
// the next step, and writes the step's outputs.  Only the chunks below
// round_up(n, 8) are ever touched (the drain skips the rest).
__device__ void finalize_tile(const FwdArgs& a, int kind, int t, int l, int mt, float* s_rs, float* s_sq) {
  const int n = a.n, np = a.n_pad;
  const int nz = min(np, (n + 7) & ~7);
  float* accT = a.acc + static_cast<int64_t>(t) * 128 * np;
  auto take4 = [&](int row, int c) -> float4 {
    float4* p = reinterpret_cast<float4*>(accT + row * np + c);
    const float4 v = __ldcg(p);
    __stcg(p, make_float4(0.f, 0.f, 0.f, 0.f));
    return v;
  };
  auto at = [](const float4& v, int j) { return j == 0 ? v.x : (j == 1 ? v.y : (j == 2 ? v.z : v.w)); };
  if (kind == FWD_QKV) {
    rms_factors(a, mt, s_rs, s_sq);
    const int hd = a.hd, half = hd / 2;
    for (int idx = mt; idx < 64 * (nz / 4); idx += kMathThreads) {
      const int pr = idx & 63, c4 = (idx >> 6) * 4;
      const int row_a = (pr / half) * hd + (pr % half);   // first row of the rotate-half pair, within the tile
      const int row_b = row_a + half;
      const int grow = t * 128 + row_a;                   // row of W_qkv
      const int head = grow / hd, i = grow % hd;
      const float4 va = take4(row_a, c4), vb = take4(row_b, c4);
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int c = c4 + j;
        if (c >= n) break;
        float ya = at(va, j) * s_rs[c], yb = at(vb, j) * s_rs[c];
        if (head < a.n_q + a.n_kv) {
          const float2 cs = a.rope[c * half + i];
          const float ra = ya * cs.x - yb * cs.y;
          const float rb = yb * cs.x + ya * cs.y;
          ya = ra;
          yb = rb;
        }
        if (head < a.n_q) {
          const int64_t o = (static_cast<int64_t>(c) * a.n_q + head) * hd + i;
          a.q[o] = ya;
          a.q[o + half] = yb;
          store_hilo(a.q_hi, a.q_lo, o, ya);
          store_hilo(a.q_hi, a.q_lo, o + half, yb);
          if (a.dbg_q) {
            float* dq = a.dbg_q + static_cast<int64_t>(l) * n * a.n_q * hd;
            dq[o] = ya;
            dq[o + half] = yb;
          }
        } else if (head < a.n_q + 2 * a.n_kv) {
          const bool is_k = head < a.n_q + a.n_kv;
          const int kvh = is_k ? head - a.n_q : head - a.n_q - a.n_kv;
          const int64_t o = (static_cast<int64_t>(c) * a.n_kv + kvh) * hd + i;
          float* dst = is_k ? a.kself : a.vself;
          dst[o] = ya;
          dst[o + half] = yb;
          float* dd = is_k ? a.dbg_k : a.dbg_v;
          if (dd) {
            dd += static_cast<int64_t>(l) * n * a.n_kv * hd;
            dd[o] = ya;
            dd[o + half] = yb;
          }
        }
      }
    }
  } else if (kind == FWD_GU) {
    rms_factors(a, mt, s_rs, s_sq);
    for (int idx = mt; idx < 64 * (nz / 4); idx += kMathThreads) {
      const int r = idx & 63, c4 = (idx >> 6) * 4;
      const int j0 = t * 64 + r;
      const float4 g4 = take4(r, c4), u4 = take4(64 + r, c4);
      if (j0 < a.ff) {
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const int c = c4 + j;
          if (c >= n) break;
          const float g = at(g4, j) * s_rs[c], u = at(u4, j) * s_rs[c];
          store_hilo(a.a_hi, a.a_lo, static_cast<int64_t>(c) * a.ff + j0, g / (1.0f + expf(-g)) * u);
        }
      }
    }
  } else {   // O, down: residual
    const __nv_bfloat16* gn = kind == FWD_O ? a.mlp_norm[l] : (l + 1 < a.n_layers ? a.attn_norm[l + 1] : nullptr);
    const int row = mt & 127, hsel = mt >> 7, wq = (mt >> 5) & 3, lane = mt & 31;
    const int gm = t * 128 + row;
    const bool in = gm < a.d;
    const float gv = (gn && in) ? __bfloat162float(gn[gm]) : 0.f;
    // chunks c0 = 4 hsel + 8 k: this thread's row, two chunks per round
    for (int c0 = hsel * 4; c0 < nz; c0 += 16) {
      const bool two = c0 + 8 < nz;
      const float4 v0 = take4(row, c0);
      const float4 v1 = two ? take4(row, c0 + 8) : make_float4(0.f, 0.f, 0.f, 0.f);
      float hv[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int c = c0 + (j < 4 ? j : 4 + j);
        hv[j] = (in && c < n) ? __ldcg(a.h + static_cast<int64_t>(c) * a.d + gm) : 0.f;
      }
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int c = c0 + (j < 4 ? j : 4 + j);
        if (c >= n) continue;
        if (in) {
          hv[j] += j < 4 ? at(v0, j) : at(v1, j - 4);
          const int64_t o = static_cast<int64_t>(c) * a.d + gm;
          a.h[o] = hv[j];
          if (gn) store_hilo(a.x_hi, a.x_lo, o, hv[j] * gv);
          if (kind == FWD_DOWN && a.dbg_h) a.dbg_h[static_cast<int64_t>(l) * n * a.d + o] = hv[j];
        }
        float sq = hv[j] * hv[j];
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, off);
        if (lane == 0) s_sq[c * 4 + wq] = sq;
      }
    }
    named_bar_sync(kBarMath, kMathThreads);
    for (int c = mt; c < n; c += kMathThreads)
      a.sumsq[static_cast<int64_t>(t) * n + c] = (s_sq[c * 4] + s_sq[c * 4 + 1]) + (s_sq[c * 4 + 2] + s_sq[c * 4 + 3]);
  }
}

template <int HD, bool TWO_ROWS>
__global__ void __launch_bounds__(kThreads, 1) forward_kernel(const __grid_constant__ FwdMaps maps,
                                                              const __grid_constant__ FwdArgs a,
                                                              unsigned long long* ts) {
  constexpr uint32_t kBlock = (HD / 64) * 16 * 128;   // one K (or V) page of one kv head
  constexpr uint32_t kPage = 2 * kBlock;
  constexpr int kPPS = static_cast<int>(kSlot / kPage);   // pages per ring slot
  constexpr int kStagePages = 8;                          // attention stage: one page per math warp
  constexpr int kRows = TWO_ROWS ? 16 : 8;
  trace_begin(ts);
  if (a.phase_ts && threadIdx.x == 0) atomicMin(a.phase_ts, static_cast<unsigned long long>(global_timer_ns()));

  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = align1024(smem_raw);
  uint8_t* ring = base;
  uint8_t* aux = base + a.aux_off;
  uint8_t* misc = base + a.misc_off;
  const int S = a.ring_slots, SX = a.x_stages;
  uint64_t* full_w = reinterpret_cast<uint64_t*>(misc + kMiscBars);
  uint64_t* empty_w = full_w + kMaxSlots;
  uint64_t* full_x = empty_w + kMaxSlots;
  uint64_t* empty_x = full_x + kMaxXStages;
  uint64_t* acc_full = empty_x + kMaxXStages;
  uint64_t* acc_empty = acc_full + 2;
  uint64_t* seg_full = acc_empty + 2;
  uint64_t* seg_free = seg_full + 1;
  uint64_t* xr_full = seg_free + 1;   // resident activation slice loaded (one phase per step with pieces)
  uint64_t* xr_free = xr_full + 1;    // the MMAs reading it have completed
  int* attn_rel = reinterpret_cast<int*>(misc + kMiscRel);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(misc + kMiscTmem);
  volatile int* s_flag = reinterpret_cast<volatile int*>(misc + kMiscFlag);
  int* s_cnt = reinterpret_cast<int*>(misc + kMiscCnt);
  float* s_rs = reinterpret_cast<float*>(misc + kMiscRs);
  float* s_sq = reinterpret_cast<float*>(misc + kMiscSq);
  // attention hand-off to the merger (aliases the activation ring, see below)
  float* mo = reinterpret_cast<float*>(aux);
  float* mm = mo + kStateWarps * 8 * HD;
  float* mlv = mm + kStateWarps * 8;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int cta = blockIdx.x, P = gridDim.x;
  const int seg0 = cta < a.wk.n_ctas ? a.wk.cta_seg[cta] : 0;
  const int seg1 = cta < a.wk.n_ctas ? a.wk.cta_seg[cta + 1] : 0;
  int* const cnt_done = a.counters + a.done_off;
  int* const cnt_attn = a.counters + a.attn_done_off;
  int* const cnt_comb = a.counters + a.comb_done_off;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kMaxSlots; ++s) {
      mbar_init(&full_w[s], 1);
      mbar_init(&empty_w[s], 1);
      attn_rel[s] = 0;
    }
    for (int s = 0; s < kMaxXStages; ++s) {
      mbar_init(&full_x[s], 1);
      mbar_init(&empty_x[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], kMathThreads / 32);
    }
    mbar_init(seg_full, kStateWarps);
    mbar_init(seg_free, 1);
    mbar_init(xr_full, 1);
    mbar_init(xr_free, 1);
    fence_mbar_init();
    // ring slots of each step of this CTA's program (the same every layer)
    for (int ph = 0; ph < 5; ++ph) {
      int c = 0;
      if (ph == 1) {
        for (int si = seg0; si < seg1; ++si) c += (a.wk.segs[si].n_pages + kPPS - 1) / kPPS;
      } else {
        const FwdGemmDev& G = a.gemm[kind_of(ph)];
        for (int p = G.cta_piece[cta]; p < G.cta_piece[cta + 1]; ++p) c += G.pieces[p].kt1 - G.pieces[p].kt0;
      }
      s_cnt[ph] = c;
    }
    tma_prefetch_desc(&maps.pool);
  }
  if (warp == kWarpMma) {
    tmem_alloc(tmem_slot, a.tmem_cols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const int L = a.n_layers;

  if (warp == kWarpProducer) {
    // ================================================================ producer
    if (lane == 0) {
      const uint64_t pol = policy_evict_first();
      uint32_t u = 0;
      bool ok = true;
      for (int l = 0; l < L && ok; ++l) {
        for (int ph = 0; ph < 5 && ok; ++ph) {
          if (ph == 1) {
            for (int si = seg0; si < seg1 && ok; ++si) {
              const AttnSeg sg = a.wk.segs[si];
              const int32_t* pg = a.wk.pages + sg.page_off;
              for (int p0 = 0; p0 < sg.n_pages; p0 += kPPS, ++u) {
                const int s = static_cast<int>(u % S);
                if (u >= static_cast<uint32_t>(S) && !mbar_wait(&empty_w[s], ((u / S) - 1) & 1u, a.err, kSiteProdAttn)) {
                  ok = false;
                  break;
                }
                const int cnt = min(kPPS, sg.n_pages - p0);
                mbar_arrive_expect_tx(&full_w[s], static_cast<uint32_t>(cnt) * kPage);
                for (int i = 0; i < cnt; ++i) {
                  const int64_t phys = __ldg(pg + p0 + i);
                  tma_load_5d(ring + s * kSlot + i * kPage, &maps.pool, &full_w[s], 0, 0, 0, sg.g,
                              static_cast<int32_t>(2 * (static_cast<int64_t>(l) * a.layer_pages + phys)), pol);
                }
              }
            }
          } else {
            const int kind = kind_of(ph);
            const FwdGemmDev& G = a.gemm[kind];
            const CUtensorMap* wm = a.wmaps + l * FWD_KINDS + kind;
            for (int p = G.cta_piece[cta]; p < G.cta_piece[cta + 1] && ok; ++p) {
              const FwdPiece pc = G.pieces[p];
              for (int kt = pc.kt0; kt < pc.kt1; ++kt, ++u) {
                const int s = static_cast<int>(u % S);
                if (u >= static_cast<uint32_t>(S) && !mbar_wait(&empty_w[s], ((u / S) - 1) & 1u, a.err, kSiteProdW)) {
                  ok = false;
                  break;
                }
                mbar_arrive_expect_tx(&full_w[s], kSlot);
                uint8_t* dst = ring + s * kSlot;
                if (kind == FWD_GU) {   // 64 gate rows, then the matching 64 up rows
                  tma_load_2d(dst, wm, &full_w[s], kt * 64, pc.tile * 64, pol);
                  tma_load_2d(dst + kSlot / 2, wm, &full_w[s], kt * 64, a.ff + pc.tile * 64, pol);
                } else {
                  tma_load_2d(dst, wm, &full_w[s], kt * 64, pc.tile * 128, pol);
                }
              }
            }
            if (G.cta_piece[cta] < G.cta_piece[cta + 1]) probe(a, l, 44 + kind);
          }
        }
      }
      // every copy issued has landed before the CTA may exit
      for (uint32_t v = u > static_cast<uint32_t>(S) ? u - S : 0; v < u; ++v)
        if (!mbar_wait(&full_w[v % S], (v / S) & 1u, a.err)) break;
    }
  } else if (warp == kWarpMma) {
    // ================================================================ MMA issuer
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16_f32(128, a.n_pad);
      const uint32_t xhalf = a.x_bytes / 2;
      uint32_t u = 0, xu = 0, au = 0, xp = 0;
      bool ok = true;
      for (int l = 0; l < L && ok; ++l) {
        for (int ph = 0; ph < 5 && ok; ++ph) {
          if (ph == 1) {
            u += s_cnt[1];
            continue;
          }
          const FwdGemmDev& G = a.gemm[kind_of(ph)];
          const int pb = G.cta_piece[cta], pe = G.cta_piece[cta + 1];
          uint64_t tw_w = 0, tw_x = 0, tw_acc = 0, t_issue = 0, t_first = 0;
          int xk0 = 0;   // resident: first K tile of the slice
          if (G.resident && pb < pe) {
            xk0 = G.pieces[pb].kt0;
            for (int p = pb + 1; p < pe; ++p) xk0 = min(xk0, G.pieces[p].kt0);
            const uint64_t t0 = a.probe ? global_timer_ns() : 0;
            if (!mbar_wait(xr_full, xp & 1u, a.err, kSiteMmaX)) {
              ok = false;
              break;
            }
            if (a.probe) tw_x += global_timer_ns() - t0;
          }
          for (int p = pb; p < pe && ok; ++p) {
            const FwdPiece pc = G.pieces[p];
            const uint32_t buf = au & 1u;
            const uint64_t ta0 = a.probe ? global_timer_ns() : 0;
            if (au >= 2 && !mbar_wait(&acc_empty[buf], ((au >> 1) - 1) & 1u, a.err, kSiteMmaAcc)) {
              ok = false;
              break;
            }
            if (a.probe) tw_acc += global_timer_ns() - ta0;
            tc_fence_after();
            const uint32_t d = tmem + buf * static_cast<uint32_t>(a.n_pad);
            for (int kt = pc.kt0; kt < pc.kt1; ++kt, ++u) {
              const int s = static_cast<int>(u % S), xs = static_cast<int>(xu % SX);
              const uint64_t t0 = a.probe ? global_timer_ns() : 0;
              if (!mbar_wait(&full_w[s], (u / S) & 1u, a.err, kSiteMmaW)) {
                ok = false;
                break;
              }
              const uint64_t t1 = a.probe ? global_timer_ns() : 0;
              if (!G.resident && !mbar_wait(&full_x[xs], (xu / SX) & 1u, a.err, kSiteMmaX)) {
                ok = false;
                break;
              }
              uint64_t t2 = 0;
              if (a.probe) {
                t2 = global_timer_ns();
                tw_w += t1 - t0;
                tw_x += t2 - t1;
                if (!t_first) t_first = t2;
              }
              tc_fence_after();
              const uint32_t wa = smem_u32(ring + s * kSlot);
              const uint32_t xa = smem_u32(aux + (G.resident ? (kt - xk0) : xs) * a.x_bytes);
#pragma unroll
              for (int kk = 0; kk < 4; ++kk) {
                const uint64_t adesc = desc_sw128(wa + kk * 32);
                umma_bf16(d, adesc, desc_sw128(xa + kk * 32), idesc, (kt > pc.kt0 || kk > 0) ? 1u : 0u);
                umma_bf16(d, adesc, desc_sw128(xa + xhalf + kk * 32), idesc, 1u);
              }
              umma_commit(&empty_w[s]);
              if (!G.resident) {
                umma_commit(&empty_x[xs]);
                ++xu;
              }
              if (a.probe) t_issue += global_timer_ns() - t2;
            }
            if (!ok) break;
            umma_commit(&acc_full[buf]);
            ++au;
          }
          if (pb < pe) {
            if (G.resident) {
              umma_commit(xr_free);   // the slice may be overwritten once these MMAs completed
              ++xp;
            }
            probe(a, l, 3 * kind_of(ph) + 1);
            probe_set(a, l, 16 + kind_of(ph), tw_w);
            probe_set(a, l, 20 + kind_of(ph), tw_x);
            probe_set(a, l, 32 + kind_of(ph), t_issue);
            probe_set(a, l, 36 + kind_of(ph), tw_acc);
            probe_set(a, l, 40 + kind_of(ph), t_first);
          }
        }
      }
    }
  } else if (warp == kWarpX) {
    // ================================================================ activation loader
    // The whole warp copies each K step's hi and lo activation tiles (n_pad
    // rows x 64 bf16 each) with cp.async from L2 into the 128-byte-swizzled
    // layout the MMA descriptors expect -- through the load/store path, so the
    // copies never queue behind the producer's weight and K/V streams in the
    // TMA unit.  Up to SX - 1 K steps are in flight; a stage is announced on
    // full_x once its copies have landed, and everything is announced before
    // any blocking wait on a step counter.
    const int np = a.n_pad, chunks = np * 16;
    const uint32_t tile_bytes = static_cast<uint32_t>(np) * 128;
    const int depth = SX - 1;
    uint32_t xu = 0, xa = 0;   // stages issued / announced (pipelined steps)
    uint32_t xp = 0;           // slices loaded (resident steps)
    bool ok = true;
    auto announce = [&](int keep) {   // announce the oldest stages until at most `keep` are in flight
      if (static_cast<int>(xu - xa) <= keep) return;
      cp_async_wait_pending(keep);
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0)
        for (; static_cast<int>(xu - xa) > keep; ++xa) mbar_arrive(&full_x[xa % SX]);
      xa = xu - keep;
    };
    for (int l = 0; l < L && ok; ++l) {
      for (int kind = 0; kind < FWD_KINDS && ok; ++kind) {
        const FwdGemmDev& G = a.gemm[kind];
        const int pb = G.cta_piece[cta], pe = G.cta_piece[cta + 1];
        if (pb == pe) continue;
        const int* cnt = nullptr;
        int target = 0, K = a.d;
        const __nv_bfloat16 *xh = a.x_hi, *xl = a.x_lo;
        if (kind == FWD_QKV) {
          if (l > 0) {
            cnt = cnt_done + FWD_DOWN;
            target = l * a.gemm[FWD_DOWN].tiles;
          }
        } else if (kind == FWD_O) {
          cnt = cnt_comb;
          target = (l + 1) * P;
          xh = a.o_hi;
          xl = a.o_lo;
          K = a.n_q * a.hd;
        } else if (kind == FWD_GU) {
          cnt = cnt_done + FWD_O;
          target = (l + 1) * a.gemm[FWD_O].tiles;
        } else {
          cnt = cnt_done + FWD_GU;
          target = (l + 1) * a.gemm[FWD_GU].tiles;
          xh = a.a_hi;
          xl = a.a_lo;
          K = a.ff;
        }
        announce(0);
        if (cnt)
          ok = __shfl_sync(0xffffffffu, lane == 0 ? (wait_counter(cnt, target, a.err, kSiteXDep + kind) ? 1 : 0) : 0,
                           0) != 0;
        if (!ok) break;
        if (lane == 0) probe(a, l, 3 * kind);
        if (G.resident) {
          // the whole K range of this CTA's pieces, once, after the MMAs reading the previous slice completed
          int k0 = G.pieces[pb].kt0, k1 = G.pieces[pb].kt1;
          for (int p = pb + 1; p < pe; ++p) {
            k0 = min(k0, G.pieces[p].kt0);
            k1 = max(k1, G.pieces[p].kt1);
          }
          if (xp > 0 && !__all_sync(0xffffffffu, mbar_wait(xr_free, (xp - 1) & 1u, a.err, kSiteXEmpty))) {
            ok = false;
            break;
          }
          for (int kt = k0; kt < k1; ++kt) {
            const uint32_t st = smem_u32(aux + (kt - k0) * a.x_bytes);
            for (int id = lane; id < chunks; id += 32) {
              const int tsel = id >= np * 8 ? 1 : 0;
              const int r = (id >> 3) - tsel * np, j = id & 7;
              const __nv_bfloat16* src = (tsel ? xl : xh) + static_cast<int64_t>(r) * K + kt * 64 + j * 8;
              cp_async16_cg(st + tsel * tile_bytes + r * 128 + ((j ^ (r & 7)) << 4), src);
            }
          }
          cp_async_commit();
          cp_async_wait_pending(0);
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) mbar_arrive(xr_full);
          ++xp;
          continue;
        }
        for (int p = pb; p < pe && ok; ++p) {
          const FwdPiece pc = G.pieces[p];
          for (int kt = pc.kt0; kt < pc.kt1; ++kt) {
            const int xs = static_cast<int>(xu % SX);
            if (xu >= static_cast<uint32_t>(SX) &&
                !__all_sync(0xffffffffu, mbar_wait(&empty_x[xs], ((xu / SX) - 1) & 1u, a.err, kSiteXEmpty))) {
              ok = false;
              break;
            }
            const uint32_t st = smem_u32(aux + xs * a.x_bytes);
            for (int id = lane; id < chunks; id += 32) {
              const int tsel = id >= np * 8 ? 1 : 0;
              const int r = (id >> 3) - tsel * np, j = id & 7;
              const __nv_bfloat16* src = (tsel ? xl : xh) + static_cast<int64_t>(r) * K + kt * 64 + j * 8;
              cp_async16_cg(st + tsel * tile_bytes + r * 128 + ((j ^ (r & 7)) << 4), src);
            }
            cp_async_commit();
            ++xu;   // counted before announcing: this stage is one of the pending ones
            announce(depth);
          }
        }
      }
    }
    announce(0);
  } else if (warp == kWarpMerger) {
    // ================================================================ merger
    uint32_t k = 0;
    bool ok = true;
    for (int l = 0; l < L; ++l) {
      if (!TWO_ROWS)
        for (int si = seg0; si < seg1; ++si) {
          const AttnSeg sg = a.wk.segs[si];
          if (sg.kind != 0) continue;
          if (ok) ok = __all_sync(0xffffffffu, mbar_wait(seg_full, k & 1u, a.err, kSiteMerger));
          if (ok) merge_warp_states<HD>(a.group, mo, mm, mlv, sg.slot, lane, a.apart_o, a.apart_ml);
          __syncwarp();
          if (lane == 0) mbar_arrive(seg_free);
          ++k;
        }
      named_bar_sync(kBarAttn, kMathThreads + 32);   // this CTA's attention slots of layer l are written
    }
  } else {
    // ================================================================ math warps
    const int mt = threadIdx.x - kWarpMath0 * 32;
    const int mw = warp - kWarpMath0;
    uint32_t u = 0, au = 0, n_priv = 0;
    bool ok = true;
    auto drain = [&](int kind, int l) {
      const FwdGemmDev& G = a.gemm[kind];
      uint64_t t_fence = 0, t_arrive = 0;
      const int np2 = a.n_pad / 2;
      const int row = (warp & 3) * 32 + lane;   // TMEM lane quadrant of this warp
      const int c_lo = (mw >> 2) * np2;
      for (int p = G.cta_piece[cta]; p < G.cta_piece[cta + 1]; ++p) {
        const FwdPiece pc = G.pieces[p];
        const uint32_t buf = au & 1u;
        if (ok) ok = __all_sync(0xffffffffu, mbar_wait(&acc_full[buf], (au >> 1) & 1u, a.err, kSiteDrain));
        tc_fence_after();
        if (ok) {
          float* dst = a.acc + (static_cast<int64_t>(pc.tile) * 128 + row) * a.n_pad;
          const uint32_t taddr = tmem + (static_cast<uint32_t>((warp & 3) * 32) << 16) + buf * a.n_pad;
          for (int c0 = c_lo; c0 < c_lo + np2; c0 += 8) {
            if (c0 >= a.n) break;
            float v[8];
            tmem_ld8(taddr + c0, v);
            red_add_v4(dst + c0, v[0], v[1], v[2], v[3]);
            red_add_v4(dst + c0 + 4, v[4], v[5], v[6], v[7]);
          }
          const uint64_t t0 = a.probe ? global_timer_ns() : 0;
          __threadfence();   // this thread's reductions are performed before the arrival below
          if (a.probe) t_fence += global_timer_ns() - t0;
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&acc_empty[buf]);
        ++au;
        // the tile's arrival count; the last piece to arrive runs the epilogue
        const uint64_t ta = a.probe ? global_timer_ns() : 0;
        named_bar_sync(kBarMath, kMathThreads);
        if (mt == 0) {
          int last = 0;
          if (ok) {
            __threadfence();
            const int npt = G.tile_np[pc.tile];
            const int old = atomicAdd(a.counters + a.tile_cnt_off[kind] + pc.tile, 1);
            last = old + 1 == (l + 1) * npt;
            __threadfence();
          }
          *s_flag = last;
        }
        named_bar_sync(kBarMath, kMathThreads);
        const bool last = *s_flag != 0;
        named_bar_sync(kBarMath, kMathThreads);   // every thread has read the flag before it is reused
        if (a.probe) t_arrive += global_timer_ns() - ta;
        if (last) {
          __threadfence();
          finalize_tile(a, kind, pc.tile, l, mt, s_rs, s_sq);
          fence_proxy_async_global();
          named_bar_sync(kBarMath, kMathThreads);
          if (mt == 0) {
            __threadfence();
            atomicAdd(cnt_done + kind, 1);
          }
        }
      }
      if (mt == 0 && G.cta_piece[cta] < G.cta_piece[cta + 1]) {
        probe(a, l, 3 * kind + 2);
        probe_set(a, l, 24 + kind, t_fence);
        probe_set(a, l, 28 + kind, t_arrive);
      }
    };
    // broadcast of a wait done by math thread 0
    auto math_wait = [&](const int* cnt, int target, int site) {
      if (mt == 0) *s_flag = (ok && wait_counter(cnt, target, a.err, site)) ? 1 : 0;
      named_bar_sync(kBarMath, kMathThreads);
      ok = *s_flag != 0;
      named_bar_sync(kBarMath, kMathThreads);
    };

    for (int l = 0; l < L; ++l) {
      // ---------------------------------------------------------------- QKV
      drain(FWD_QKV, l);
      trace_phase(a, l, 0, mt);
      u += s_cnt[0];
      // ---------------------------------------------------------------- attention
      math_wait(cnt_done + FWD_QKV, (l + 1) * a.gemm[FWD_QKV].tiles, kSiteQ);
      if (mt == 0) probe(a, l, 12);
      for (int si = seg0; si < seg1; ++si) {
        const AttnSeg sg = a.wk.segs[si];
        const bool shared = sg.kind == 1;
        const int cand = shared ? (mw < sg.n_cands ? a.wk.cands[sg.cand + mw] : -1) : (mw < sg.n_pages ? sg.cand : -1);
        WarpQ<HD> q;
        if (cand >= 0 && ok) {
          const int64_t q0 = (static_cast<int64_t>(cand) * a.n_q + static_cast<int64_t>(sg.g) * a.group) * HD;
          load_q<HD, TWO_ROWS>(q, a.q_hi + q0, a.q_lo + q0, a.group, lane);
        }
        WarpState<HD> st;
        st.reset();
        for (int p0 = 0; p0 < sg.n_pages; p0 += kStagePages) {
          const int npg = min(kStagePages, sg.n_pages - p0);
          const int ns = (npg + kPPS - 1) / kPPS;
          for (int j = 0; j < ns; ++j) {
            const uint32_t v = u + j;
            if (ok) ok = __all_sync(0xffffffffu, mbar_wait(&full_w[v % S], (v / S) & 1u, a.err, kSiteAttnFull));
          }
          if (ok && cand >= 0) {
            if (!shared) {   // page mw of this stage
              if (mw < npg) {
                const int valid = p0 + mw == sg.n_pages - 1 ? sg.last_valid : 16;
                const uint32_t kb = smem_u32(ring + ((u + mw / kPPS) % S) * kSlot + (mw % kPPS) * kPage);
                process_page<HD, TWO_ROWS>(q, kb, kb + kBlock, valid, lane, st);
              }
            } else {         // every page of this stage, for this warp's candidate
              for (int pi = 0; pi < npg; ++pi) {
                const int valid = p0 + pi == sg.n_pages - 1 ? sg.last_valid : 16;
                const uint32_t kb = smem_u32(ring + ((u + pi / kPPS) % S) * kSlot + (pi % kPPS) * kPage);
                process_page<HD, TWO_ROWS>(q, kb, kb + kBlock, valid, lane, st);
              }
            }
          }
          __syncwarp();
          if (lane == 0)
            for (int j = 0; j < ns; ++j) {   // the eighth warp done with a slot frees it
              const int s = static_cast<int>((u + j) % S);
              if ((atomicAdd(&attn_rel[s], 1) + 1) % (kMathThreads / 32) == 0) mbar_arrive(&empty_w[s]);
            }
          u += ns;
        }
        if (cand >= 0 && ok) finish_state<HD, TWO_ROWS>(st);
        if (!shared && !TWO_ROWS) {
          if (n_priv > 0) ok = __all_sync(0xffffffffu, mbar_wait(seg_free, (n_priv - 1) & 1u, a.err, kSiteSegFree)) && ok;
          stash_state<HD>(st, cand >= 0 && ok, mw, a.group, lane, mo, mm, mlv);
          __syncwarp();
          if (lane == 0) mbar_arrive(seg_full);
          ++n_priv;
        } else if (cand >= 0 && ok) {
          const int slot_id = shared ? a.wk.slots[sg.slot + mw] : sg.slot + mw;
          store_state_slot<HD, TWO_ROWS>(st, slot_id, a.group, lane, a.apart_o, a.apart_ml);
        }
      }
      named_bar_sync(kBarAttn, kMathThreads + 32);
      if (mt == 0) {
        probe(a, l, 13);
        __threadfence();
        atomicAdd(cnt_attn, 1);
      }
      trace_phase(a, l, 1, mt);
      // ---------------------------------------------------------------- combine
      math_wait(cnt_attn, (l + 1) * P, kSiteAttnDone);
      if (mt == 0) probe(a, l, 14);
      {
        const int64_t off = static_cast<int64_t>(l) * a.n * a.n_q * HD;
        const AttnMerge mg{a.q, a.kself, a.vself, a.o_hi, a.o_lo, nullptr, a.dbg_attn ? a.dbg_attn + off : nullptr};
        for (int unit = cta; unit < a.n * a.n_kv && ok; unit += P) {
          const int b = unit / a.n_kv, g = unit - b * a.n_kv;
          combine_group<HD, kRows>(mt, b, g, a.wk.slot_base[unit], a.wk.nslots[unit], a.n_q, a.n_kv, a.group,
                                   a.apart_o, a.apart_ml, mg, aux,
                                   [] { named_bar_sync(kBarMath, kMathThreads); });
          named_bar_sync(kBarMath, kMathThreads);
        }
      }
      fence_proxy_async_global();
      named_bar_sync(kBarMath, kMathThreads);
      if (mt == 0) {
        probe(a, l, 15);
        __threadfence();
        atomicAdd(cnt_comb, 1);
      }
      trace_phase(a, l, 2, mt);
      // ---------------------------------------------------------------- O, gate/up, down
      drain(FWD_O, l);
      trace_phase(a, l, 3, mt);
      drain(FWD_GU, l);
      trace_phase(a, l, 4, mt);
      drain(FWD_DOWN, l);
      trace_phase(a, l, 5, mt);
      u += s_cnt[2] + s_cnt[3] + s_cnt[4];
    }
  }
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == kWarpMma) {
    tc_fence_after();
    tmem_dealloc(tmem, a.tmem_cols);
  }
  trace_end(ts);
}

template <int HD, bool TWO>
cudaError_t set_smem_fwd() {
  return cudaFuncSetAttribute(forward_kernel<HD, TWO>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(kMaxSmem));
}

}  // namespace

bool split_gemm(int tiles, int ktiles, int n_ctas, int resident_kt, FwdGemmHost& g) {
  g.tiles = tiles;
  g.ktiles = ktiles;
  g.pieces.clear();
  g.cta_piece.assign(static_cast<size_t>(n_ctas) + 1, 0);
  g.tile_np.assign(static_cast<size_t>(tiles), 0);
  g.resident = resident_kt > 0 ? 1 : 0;
  // k-groups of r K tiles: one group (plain stream-K) unless the slice must stay within resident_kt
  int G = 1, r = ktiles;
  if (resident_kt > 0 && ktiles > resident_kt) {
    G = (ktiles + resident_kt - 1) / resident_kt;
    r = (ktiles + G - 1) / G;
    G = (ktiles + r - 1) / r;
  }
  for (int grp = 0; grp < G; ++grp) {
    const int k0 = grp * r, k1 = std::min(ktiles, k0 + r), rg = k1 - k0;
    // the group's CTAs, in proportion to its share of K; every group needs one
    const int c0 = static_cast<int>(static_cast<int64_t>(n_ctas) * k0 / ktiles);
    const int c1 = static_cast<int>(static_cast<int64_t>(n_ctas) * k1 / ktiles);
    if (c1 <= c0) return false;
    const int C = c1 - c0;
    const int64_t U = static_cast<int64_t>(tiles) * rg;
    for (int j = 0; j < C; ++j) {
      g.cta_piece[c0 + j] = static_cast<int32_t>(g.pieces.size());
      const int64_t u0 = U * j / C, u1 = U * (j + 1) / C;
      for (int64_t u = u0; u < u1;) {
        FwdPiece p;
        p.tile = static_cast<int32_t>(u / rg);
        p.kt0 = static_cast<int32_t>(k0 + u % rg);
        p.kt1 = static_cast<int32_t>(std::min<int64_t>(k1, p.kt0 + (u1 - u)));
        p.pad = 0;
        g.pieces.push_back(p);
        ++g.tile_np[p.tile];
        u += p.kt1 - p.kt0;
      }
    }
  }
  g.cta_piece[n_ctas] = static_cast<int32_t>(g.pieces.size());
  return true;
}

bool plan_forward(int hd, int group, int n_pad, FwdPlan& p) {
  if (n_pad < 16 || n_pad > 256 || n_pad % 16) return false;
  const bool two = group > 8;
  p.x_bytes = static_cast<uint32_t>(2 * n_pad * 128);   // hi and lo tiles of one 64-wide K step
  uint32_t x_ring;
  if (n_pad <= 32) {   // small batches: each CTA's activation slice (<= 64 KB) is loaded once per step
    p.resident_kt = static_cast<int>(kResidentBytes / p.x_bytes);
    p.x_stages = 8;
    x_ring = kResidentBytes;
  } else {             // larger batches: activation tiles pipelined per K step
    p.resident_kt = 0;
    p.x_stages = n_pad <= 64 ? 4 : 2;
    x_ring = p.x_stages * p.x_bytes;
  }
  const uint32_t merge = two ? 0u : static_cast<uint32_t>(kStateWarps * 8 * hd * 4 + 2 * kStateWarps * 8 * 4);
  size_t comb = 0;
  if (hd == 128)
    comb = two ? CombineShape<128, 16>::kBytes : CombineShape<128, 8>::kBytes;
  else
    comb = two ? CombineShape<64, 16>::kBytes : CombineShape<64, 8>::kBytes;
  uint32_t aux = std::max<uint32_t>(x_ring, std::max<uint32_t>(merge, static_cast<uint32_t>(comb)));
  aux = (aux + 1023) & ~1023u;
  const int64_t room = static_cast<int64_t>(kMaxSmem) - 1024 - kMiscBytes - aux;
  int slots = static_cast<int>(room / kSlot);
  if (slots > kMaxSlots) slots = kMaxSlots;
  if (slots < 4) return false;   // one attention stage of eight pages needs four slots (hd 128)
  p.ring_slots = slots;
  p.aux_off = static_cast<uint32_t>(slots) * kSlot;
  p.misc_off = p.aux_off + aux;
  p.smem_bytes = static_cast<size_t>(p.misc_off) + kMiscBytes + 1024;
  uint32_t cols = 32;
  while (cols < static_cast<uint32_t>(2 * n_pad)) cols <<= 1;
  p.tmem_cols = cols;
  return p.smem_bytes <= kMaxSmem;
}

cudaError_t forward_configure() {
  cudaError_t e;
  if ((e = set_smem_fwd<64, false>()) != cudaSuccess) return e;
  if ((e = set_smem_fwd<64, true>()) != cudaSuccess) return e;
  if ((e = set_smem_fwd<128, false>()) != cudaSuccess) return e;
  return set_smem_fwd<128, true>();
}

cudaError_t launch_forward(const FwdMaps& maps, const FwdArgs& a, int grid, cudaStream_t stream, bool cooperative,
                           unsigned long long* ts) {
  FwdPlan p;
  if (!plan_forward(a.hd, a.group, a.n_pad, p)) return cudaErrorInvalidValue;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = p.smem_bytes;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = cooperative ? 1 : 0;
  const bool two = a.group > 8;
  if (a.hd == 128)
    return two ? cudaLaunchKernelEx(&cfg, forward_kernel<128, true>, maps, a, ts)
               : cudaLaunchKernelEx(&cfg, forward_kernel<128, false>, maps, a, ts);
  return two ? cudaLaunchKernelEx(&cfg, forward_kernel<64, true>, maps, a, ts)
             : cudaLaunchKernelEx(&cfg, forward_kernel<64, false>, maps, a, ts);
}

}  // namespace kvprm
