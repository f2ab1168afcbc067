// Warp-level building blocks of the paged decode attention (App. A.3 read-out,
// head = softmax(q^T K / sqrt(d_k)) V for the verify token's query), used by
// the attention kernels (attention.cu):
//  - WarpQ / load_q: one warp's query rows as mma.m16n8k16 A fragments, hi and
//    lo bf16 parts of the fp32 query (packed into the two 8-row halves of one
//    MMA when the group has <= 8 heads, two MMAs otherwise);
//  - WarpState / process_page: the online softmax over one 16-token page held
//    in shared memory under the 128-byte swizzle (scores in log2 units);
//  - finish_state / stash_state / store_state_slot: end of a run of pages;
//  - merge_warp_states: fold eight warps' states into one partial slot;
//  - combine_group: merge a (candidate, kv head)'s partial slots with the
//    verify token's own key/value entry into the attention output.
#pragma once

#include <cuda_bf16.h>

#include "kernels.h"
#include "ptx.cuh"

namespace kvprm {
namespace ac {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr int kStateWarps = 8;   // warps whose states a private run's merge folds

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

// Online-softmax state of one warp: per thread rows gid (and gid + 8 when two
// rows) of the running maximum, the running sum and O.
template <int HD>
struct WarpState {
  float m[2], l[2];
  float o[HD / 8][4];
  __device__ __forceinline__ void reset() {
    m[0] = m[1] = -INFINITY;
    l[0] = l[1] = 0.f;
#pragma unroll
    for (int n = 0; n < HD / 8; ++n) o[n][0] = o[n][1] = o[n][2] = o[n][3] = 0.f;
  }
};

// Score one page (16 tokens, `valid` of them real) for one warp's query rows
// and fold it into the online softmax state.  The K fragments of the whole
// page are loaded first and S is accumulated in four independent chains; O is
// rescaled only when some row's maximum grew (the factor is exactly 1
// otherwise).
template <int HD, bool TWO_ROWS>
__device__ __forceinline__ void process_page(const WarpQ<HD>& q, uint32_t kbase, uint32_t vbase, int valid, int lane,
                                             WarpState<HD>& st) {
  const int tig = lane & 3;
  const float sl2 = kLog2e * rsqrtf(static_cast<float>(HD));
  // S = Q K^T for the page's 16 tokens (two n-tiles of 8 tokens)
  float s0[4] = {0.f, 0.f, 0.f, 0.f}, s1[4] = {0.f, 0.f, 0.f, 0.f};
  float t0[4] = {0.f, 0.f, 0.f, 0.f}, t1[4] = {0.f, 0.f, 0.f, 0.f};
  {
    const int mi = lane >> 3, r = lane & 7;
    const int tok = (mi >> 1) * 8 + r;
    uint32_t kb[HD / 16][4];
#pragma unroll
    for (int ks = 0; ks < HD / 16; ++ks) {
      const int hdc = ks * 16 + (mi & 1) * 8;
      const uint32_t addr = kbase + (hdc >> 6) * 2048 + tok * 128 + ((((hdc & 63) >> 3) ^ (tok & 7)) << 4);
      ldsm_x4(addr, kb[ks][0], kb[ks][1], kb[ks][2], kb[ks][3]);
    }
#pragma unroll
    for (int ks = 0; ks < HD / 16; ++ks) {
      float(&d0)[4] = (ks & 1) ? t0 : s0;
      float(&d1)[4] = (ks & 1) ? t1 : s1;
      mma_bf16_16816(d0, q.a0[ks], q.a1[ks], q.a2[ks], q.a3[ks], kb[ks][0], kb[ks][1]);
      mma_bf16_16816(d1, q.a0[ks], q.a1[ks], q.a2[ks], q.a3[ks], kb[ks][2], kb[ks][3]);
      if (TWO_ROWS) {
        mma_bf16_16816(d0, q.b0[ks], q.b1[ks], q.b2[ks], q.b3[ks], kb[ks][0], kb[ks][1]);
        mma_bf16_16816(d1, q.b0[ks], q.b1[ks], q.b2[ks], q.b3[ks], kb[ks][2], kb[ks][3]);
      }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      s0[i] += t0[i];
      s1[i] += t1[i];
    }
  }
  const int c0 = tig * 2, c1 = tig * 2 + 1, c2 = 8 + tig * 2, c3 = 9 + tig * 2;
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
    x[r][0] = c0 < valid ? x[r][0] * sl2 : -INFINITY;
    x[r][1] = c1 < valid ? x[r][1] * sl2 : -INFINITY;
    x[r][2] = c2 < valid ? x[r][2] * sl2 : -INFINITY;
    x[r][3] = c3 < valid ? x[r][3] * sl2 : -INFINITY;
    float mx = fmaxf(fmaxf(x[r][0], x[r][1]), fmaxf(x[r][2], x[r][3]));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
    const float m_new = fmaxf(st.m[r], mx);
    if (__any_sync(0xffffffffu, m_new > st.m[r])) {   // warp-uniform: rescale O by 2^(m_old - m_new)
      const float alpha = exp2f(st.m[r] - m_new);
      st.l[r] *= alpha;
      if (!TWO_ROWS) {   // one head per thread row: both MMA row halves rescale together
#pragma unroll
        for (int n = 0; n < HD / 8; ++n) {
          st.o[n][0] *= alpha;
          st.o[n][1] *= alpha;
          st.o[n][2] *= alpha;
          st.o[n][3] *= alpha;
        }
      } else {
#pragma unroll
        for (int n = 0; n < HD / 8; ++n) {
          st.o[n][2 * r] *= alpha;
          st.o[n][2 * r + 1] *= alpha;
        }
      }
      st.m[r] = m_new;
    }
    float p[4];
#pragma unroll
    for (int i2 = 0; i2 < 4; ++i2) p[i2] = exp2f(x[r][i2] - m_new);
    st.l[r] += (p[0] + p[1]) + (p[2] + p[3]);
    float hi[4], lo[4];
#pragma unroll
    for (int i2 = 0; i2 < 4; ++i2) {
      hi[i2] = __bfloat162float(__float2bfloat16_rn(p[i2]));
      lo[i2] = p[i2] - hi[i2];
    }
    if (!TWO_ROWS) {
      ph[0] = pack_bf16(hi[0], hi[1]);   // row gid: P_hi
      ph[1] = pack_bf16(lo[0], lo[1]);   // row gid + 8: P_lo
      ph[2] = pack_bf16(hi[2], hi[3]);
      ph[3] = pack_bf16(lo[2], lo[3]);
    } else {
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
    uint32_t vb[HD / 16][4];
#pragma unroll
    for (int j2 = 0; j2 < HD / 16; ++j2) {
      const int hdc = j2 * 16 + (mi >> 1) * 8;
      const uint32_t addr = vbase + (hdc >> 6) * 2048 + tok * 128 + ((((hdc & 63) >> 3) ^ (tok & 7)) << 4);
      ldsm_x4_t(addr, vb[j2][0], vb[j2][1], vb[j2][2], vb[j2][3]);
    }
#pragma unroll
    for (int j2 = 0; j2 < HD / 16; ++j2) {
      mma_bf16_16816(st.o[2 * j2], ph[0], ph[1], ph[2], ph[3], vb[j2][0], vb[j2][1]);
      mma_bf16_16816(st.o[2 * j2 + 1], ph[0], ph[1], ph[2], ph[3], vb[j2][2], vb[j2][3]);
      if (TWO_ROWS) {
        mma_bf16_16816(st.o[2 * j2], pl[0], pl[1], pl[2], pl[3], vb[j2][0], vb[j2][1]);
        mma_bf16_16816(st.o[2 * j2 + 1], pl[0], pl[1], pl[2], pl[3], vb[j2][2], vb[j2][3]);
      }
    }
  }
}

// Two pages (A, then B) of a shared run for one warp's packed query rows (group <= 8).  The
// arithmetic of two process_page calls, except that the two pages' 32 scores per row meet one
// running-maximum update (the online softmax over a 32-token block), so the second page's score
// MMAs, maximum and exponentials proceed beside the first's: a warp scoring several pages of a
// stage for one candidate is otherwise held by each page's chain of dependent steps.
template <int HD>
__device__ __forceinline__ void process_page_pair(const WarpQ<HD>& q, uint32_t kbA, uint32_t vbA, int validA,
                                                  uint32_t kbB, uint32_t vbB, int validB, int lane,
                                                  WarpState<HD>& st) {
  const int tig = lane & 3;
  const float sl2 = kLog2e * rsqrtf(static_cast<float>(HD));
  // S = Q K^T for both pages: [page][n-tile of 8 tokens][4] (four independent accumulation chains)
  float s[2][2][4];
#pragma unroll
  for (int pg = 0; pg < 2; ++pg)
#pragma unroll
    for (int nt = 0; nt < 2; ++nt)
#pragma unroll
      for (int i = 0; i < 4; ++i) s[pg][nt][i] = 0.f;
  {
    const int mi = lane >> 3, r = lane & 7;
    const int tok = (mi >> 1) * 8 + r;
#pragma unroll
    for (int pg = 0; pg < 2; ++pg) {
      const uint32_t kbase = pg ? kbB : kbA;
#pragma unroll
      for (int h = 0; h < HD / 64; ++h) {   // K fragments of four K steps at a time (register budget)
        uint32_t kb[4][4];
#pragma unroll
        for (int k4 = 0; k4 < 4; ++k4) {
          const int hdc = (4 * h + k4) * 16 + (mi & 1) * 8;
          const uint32_t addr = kbase + (hdc >> 6) * 2048 + tok * 128 + ((((hdc & 63) >> 3) ^ (tok & 7)) << 4);
          ldsm_x4(addr, kb[k4][0], kb[k4][1], kb[k4][2], kb[k4][3]);
        }
#pragma unroll
        for (int k4 = 0; k4 < 4; ++k4) {
          const int ks = 4 * h + k4;
          mma_bf16_16816(s[pg][0], q.a0[ks], q.a1[ks], q.a2[ks], q.a3[ks], kb[k4][0], kb[k4][1]);
          mma_bf16_16816(s[pg][1], q.a0[ks], q.a1[ks], q.a2[ks], q.a3[ks], kb[k4][2], kb[k4][3]);
        }
      }
    }
  }
  const int c0 = tig * 2, c1 = tig * 2 + 1, c2 = 8 + tig * 2, c3 = 9 + tig * 2;
  float x[2][4];
  float mx = -INFINITY;
#pragma unroll
  for (int pg = 0; pg < 2; ++pg) {
    const int valid = pg ? validB : validA;
    // hi (row gid) + lo (row gid + 8) parts of the same head
    x[pg][0] = c0 < valid ? (s[pg][0][0] + s[pg][0][2]) * sl2 : -INFINITY;
    x[pg][1] = c1 < valid ? (s[pg][0][1] + s[pg][0][3]) * sl2 : -INFINITY;
    x[pg][2] = c2 < valid ? (s[pg][1][0] + s[pg][1][2]) * sl2 : -INFINITY;
    x[pg][3] = c3 < valid ? (s[pg][1][1] + s[pg][1][3]) * sl2 : -INFINITY;
    mx = fmaxf(mx, fmaxf(fmaxf(x[pg][0], x[pg][1]), fmaxf(x[pg][2], x[pg][3])));
  }
  mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
  mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
  const float m_new = fmaxf(st.m[0], mx);
  if (__any_sync(0xffffffffu, m_new > st.m[0])) {   // warp-uniform: rescale O by 2^(m_old - m_new)
    const float alpha = exp2f(st.m[0] - m_new);
    st.l[0] *= alpha;
#pragma unroll
    for (int n = 0; n < HD / 8; ++n) {
      st.o[n][0] *= alpha;
      st.o[n][1] *= alpha;
      st.o[n][2] *= alpha;
      st.o[n][3] *= alpha;
    }
    st.m[0] = m_new;
  }
  uint32_t ph[2][4];   // A fragments of P per page: rows gid = P_hi, gid + 8 = P_lo
#pragma unroll
  for (int pg = 0; pg < 2; ++pg) {
    float p[4];
#pragma unroll
    for (int i2 = 0; i2 < 4; ++i2) p[i2] = exp2f(x[pg][i2] - m_new);
    st.l[0] += (p[0] + p[1]) + (p[2] + p[3]);
    float hi[4], lo[4];
#pragma unroll
    for (int i2 = 0; i2 < 4; ++i2) {
      hi[i2] = __bfloat162float(__float2bfloat16_rn(p[i2]));
      lo[i2] = p[i2] - hi[i2];
    }
    ph[pg][0] = pack_bf16(hi[0], hi[1]);
    ph[pg][1] = pack_bf16(lo[0], lo[1]);
    ph[pg][2] = pack_bf16(hi[2], hi[3]);
    ph[pg][3] = pack_bf16(lo[2], lo[3]);
  }
  // O += P V for page A, then page B (V^T fragments through ldmatrix.trans)
  const int mi = lane >> 3;
  const int tok = (mi & 1) * 8 + (lane & 7);
#pragma unroll
  for (int pg = 0; pg < 2; ++pg) {
    const uint32_t vbase = pg ? vbB : vbA;
#pragma unroll
    for (int h = 0; h < HD / 64; ++h) {   // V fragments of four 16-column groups at a time (register budget)
      uint32_t vb[4][4];
#pragma unroll
      for (int k4 = 0; k4 < 4; ++k4) {
        const int hdc = (4 * h + k4) * 16 + (mi >> 1) * 8;
        const uint32_t addr = vbase + (hdc >> 6) * 2048 + tok * 128 + ((((hdc & 63) >> 3) ^ (tok & 7)) << 4);
        ldsm_x4_t(addr, vb[k4][0], vb[k4][1], vb[k4][2], vb[k4][3]);
      }
#pragma unroll
      for (int k4 = 0; k4 < 4; ++k4) {
        const int j2 = 4 * h + k4;
        mma_bf16_16816(st.o[2 * j2], ph[pg][0], ph[pg][1], ph[pg][2], ph[pg][3], vb[k4][0], vb[k4][1]);
        mma_bf16_16816(st.o[2 * j2 + 1], ph[pg][0], ph[pg][1], ph[pg][2], ph[pg][3], vb[k4][2], vb[k4][3]);
      }
    }
  }
}

// End of a run of pages for one warp: fold the lo-part rows onto their heads
// (packed layout) and quad-reduce the row sums.
template <int HD, bool TWO_ROWS>
__device__ __forceinline__ void finish_state(WarpState<HD>& st) {
  if (!TWO_ROWS) {
#pragma unroll
    for (int n = 0; n < HD / 8; ++n) {
      st.o[n][0] += st.o[n][2];
      st.o[n][1] += st.o[n][3];
    }
  }
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    st.l[r] += __shfl_xor_sync(0xffffffffu, st.l[r], 1);
    st.l[r] += __shfl_xor_sync(0xffffffffu, st.l[r], 2);
  }
}

// Hand warp `w`'s finished state (packed layout, group <= 8) to the merge
// through shared memory: mo [8 warps][8 rows][HD], mm / ml [8 warps][8 rows].
// A warp that scored nothing marks its rows with m = -inf.
template <int HD>
__device__ __forceinline__ void stash_state(const WarpState<HD>& st, bool scored, int w, int group, int lane,
                                            float* mo, float* mm, float* ml) {
  const int gid = lane >> 2, tig = lane & 3;
  if (scored) {
    if (gid < group) {
#pragma unroll
      for (int n = 0; n < HD / 8; ++n)
        *reinterpret_cast<float2*>(mo + (w * 8 + gid) * HD + n * 8 + tig * 2) = make_float2(st.o[n][0], st.o[n][1]);
      if (tig == 0) {
        mm[w * 8 + gid] = st.m[0];
        ml[w * 8 + gid] = st.l[0];
      }
    }
  } else if (lane < 8) {
    mm[w * 8 + lane] = -INFINITY;
    ml[w * 8 + lane] = 0.f;
  }
}

// Write a warp's finished state to partial slot `slot_id`: row r of the group
// at part_o[(slot_id * group + r) * HD] and (m, l) at part_ml[(...) * 2].
template <int HD, bool TWO_ROWS>
__device__ __forceinline__ void store_state_slot(const WarpState<HD>& st, int slot_id, int group, int lane,
                                                 float* part_o, float* part_ml) {
  const int gid = lane >> 2, tig = lane & 3;
#pragma unroll
  for (int r = 0; r < (TWO_ROWS ? 2 : 1); ++r) {
    const int row = gid + 8 * r;
    if (row < group) {
      const int64_t pr = static_cast<int64_t>(slot_id) * group + row;
      float* dst = part_o + pr * HD;
#pragma unroll
      for (int n = 0; n < HD / 8; ++n)
        *reinterpret_cast<float2*>(dst + n * 8 + tig * 2) = make_float2(st.o[n][2 * r], st.o[n][2 * r + 1]);
      if (tig == 0) *reinterpret_cast<float2*>(part_ml + pr * 2) = make_float2(st.m[r], st.l[r]);
    }
  }
}

// One warp folds query row r of the eight stashed warp states of a private run:
//   M = max_w m_w, L = sum_w 2^(m_w - M) l_w, O = sum_w 2^(m_w - M) O_w
// into dst_o[0 .. HD) and dst_ml[0 .. 2) = (M, L).
template <int HD>
__device__ __forceinline__ void merge_row(int r, const float* mo, const float* mm, const float* ml, int lane,
                                          float* dst_o, float* dst_ml) {
  constexpr int kPer = HD / 32;
  float mw[kStateWarps], M = -INFINITY;
#pragma unroll
  for (int w = 0; w < kStateWarps; ++w) {
    mw[w] = mm[w * 8 + r];
    M = fmaxf(M, mw[w]);
  }
  float acc[kPer], L = 0.f;
#pragma unroll
  for (int j = 0; j < kPer; ++j) acc[j] = 0.f;
#pragma unroll
  for (int w = 0; w < kStateWarps; ++w) {
    if (mw[w] == -INFINITY) continue;   // an idle warp: its O rows are not written
    const float f = exp2f(mw[w] - M);
    L += f * ml[w * 8 + r];
#pragma unroll
    for (int j = 0; j < kPer; ++j) acc[j] += f * mo[(w * 8 + r) * HD + lane + 32 * j];
  }
#pragma unroll
  for (int j = 0; j < kPer; ++j) dst_o[lane + 32 * j] = acc[j];
  if (lane == 0) *reinterpret_cast<float2*>(dst_ml) = make_float2(M, L);
}

// One warp folds the eight stashed warp states of a private run into partial slot `slot`, row by row.
template <int HD>
__device__ __forceinline__ void merge_warp_states(int group, const float* mo, const float* mm, const float* ml,
                                                  int slot, int lane, float* part_o, float* part_ml) {
  for (int r = 0; r < group; ++r) {
    const int64_t pr = static_cast<int64_t>(slot) * group + r;
    merge_row<HD>(r, mo, mm, ml, lane, part_o + pr * HD, part_ml + pr * 2);
  }
}

// Combine of one (candidate row b, kv head g): W warps (8 or 4; threads tid < 32 W)
// fold its partial slots [first, first + ns), U at a time per warp with every
// load of a round issued before the first use, into a running (M, L, O) per
// query head of the group; the warps' states and the verify token's own entry
// (s_self = q . k_self, value v_self) are then merged through shared memory:
//   M* = max(s_self, M_w), o = (2^(s_self - M*) v_self + sum_w 2^(M_w - M*) O_w)
//                              / (2^(s_self - M*) + sum_w 2^(M_w - M*) L_w).
// In a depth-k readout (mg.depth > 1) row b is verify token t = b % depth and the
// self entries are its candidate's tokens 0 .. t (rows b - t .. b), each a term
// 2^(s_j - M*) v_j of the same sums (the DEEP variant);
// written as a bf16 (hi, lo) pair (and optional fp32 copies).  `smem` holds
// CombineShape::kBytes; sync() is a barrier over exactly the 32 W threads.  A
// caller running several groups back to back syncs between them.
template <int HD, int ROWS, int W_ = 8>
struct CombineShape {
  static constexpr int W = W_;                              // warps
  static constexpr int U = HD * ROWS <= 512 ? 2 : 1;        // slots in flight per warp
  static constexpr size_t kAcc = 0;                                         // [W][ROWS][HD]
  static constexpr size_t kM = kAcc + sizeof(float) * W * ROWS * HD;        // [W][ROWS]
  static constexpr size_t kL = kM + sizeof(float) * W * ROWS;               // [W][ROWS]
  static constexpr size_t kSelf = kL + sizeof(float) * W * ROWS;            // [ROWS][kMaxReadoutDepth]
  static constexpr size_t kBytes = kSelf + sizeof(float) * ROWS * kMaxReadoutDepth;
};

template <int HD, int ROWS, int W_ = 8, bool DEEP = false, typename Sync>
__device__ __forceinline__ void combine_group(int tid, int b, int g, int first, int ns, int n_q, int n_kv, int group,
                                              const float* __restrict__ part_o, const float* __restrict__ part_ml,
                                              const AttnMerge& mg, uint8_t* smem, Sync sync) {
  using CS = CombineShape<HD, ROWS, W_>;
  constexpr int kPer = HD / 32, W = CS::W, U = CS::U;
  constexpr int kOut = (ROWS * HD + W * 32 - 1) / (W * 32);   // outputs per thread in the final phase
  float* s_acc = reinterpret_cast<float*>(smem + CS::kAcc);
  float* s_m = reinterpret_cast<float*>(smem + CS::kM);
  float* s_l = reinterpret_cast<float*>(smem + CS::kL);
  float* s_self = reinterpret_cast<float*>(smem + CS::kSelf);
  const int warp = tid >> 5, lane = tid & 31;
  const int64_t hq0 = static_cast<int64_t>(b) * n_q + static_cast<int64_t>(g) * group;
  const int64_t hk = static_cast<int64_t>(b) * n_kv + g;
  // Every global load of the first round is issued before any is used: this
  // warp's first U slots, the q / k_self rows of head `warp` and this thread's
  // v_self values for the final phase.
  float2 ml[U];
  float v[U][ROWS][kPer];
#pragma unroll
  for (int k = 0; k < U; ++k) {
    const int sk = warp + k * W;
    const int64_t pr = (static_cast<int64_t>(first) + (sk < ns ? sk : 0)) * group;
    ml[k] = (sk < ns && lane < group) ? __ldcg(reinterpret_cast<const float2*>(part_ml + (pr + lane) * 2))
                                      : make_float2(-INFINITY, 0.f);
#pragma unroll
    for (int r = 0; r < ROWS; ++r)
#pragma unroll
      for (int j = 0; j < kPer; ++j)
        v[k][r][j] = (sk < ns && r < group) ? __ldcg(part_o + (pr + r) * HD + lane + 32 * j) : 0.f;
  }
  float qd[kPer], kd[kPer];
#pragma unroll
  for (int j = 0; j < kPer; ++j) {
    qd[j] = warp < group ? __ldcg(mg.q + (hq0 + warp) * HD + lane + 32 * j) : 0.f;
    kd[j] = warp < group ? __ldcg(mg.kself + hk * HD + lane + 32 * j) : 0.f;
  }
  float vsf[kOut];
#pragma unroll
  for (int i = 0; i < kOut; ++i) {
    const int idx = tid + i * W * 32;
    vsf[i] = idx < group * HD ? __ldcg(mg.vself + hk * HD + idx % HD) : 0.f;
  }
  // the self entries' scores of head `warp`: token t's own (k_self already loaded) and, in a
  // depth-k readout, its candidate's earlier tokens (rows b - t .. b - 1)
  // DEEP (a depth-k readout): a compiled variant of its own, so that the single-entry form keeps its code
  const int t_self = DEEP ? b % mg.depth : 0, n_self = DEEP ? t_self + 1 : 1;
  const int64_t hk0 = hk - static_cast<int64_t>(t_self) * n_kv;
  if (warp < group) {
    for (int e = 0; e < n_self; ++e) {
      float dot = 0.f;
#pragma unroll
      for (int j = 0; j < kPer; ++j)
        dot += qd[j] * (e == t_self ? kd[j] : __ldcg(mg.kself + (hk0 + e * n_kv) * HD + lane + 32 * j));
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) dot += __shfl_xor_sync(0xffffffffu, dot, off);
      if (lane == 0) s_self[warp * kMaxReadoutDepth + e] = dot * (kLog2e * rsqrtf(static_cast<float>(HD)));
    }
  }
  for (int r = warp + W; r < group; r += W) {   // heads beyond the warp count (G > W; k_self is loaded by all)
    for (int e = 0; e < n_self; ++e) {
      float dot = 0.f;
#pragma unroll
      for (int j = 0; j < kPer; ++j)
        dot += __ldcg(mg.q + (hq0 + r) * HD + lane + 32 * j) *
               (e == t_self ? kd[j] : __ldcg(mg.kself + (hk0 + e * n_kv) * HD + lane + 32 * j));
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) dot += __shfl_xor_sync(0xffffffffu, dot, off);
      if (lane == 0) s_self[r * kMaxReadoutDepth + e] = dot * (kLog2e * rsqrtf(static_cast<float>(HD)));
    }
  }
  float M[ROWS], L[ROWS], acc[ROWS][kPer];
#pragma unroll
  for (int r = 0; r < ROWS; ++r) {
    M[r] = -INFINITY;
    L[r] = 0.f;
#pragma unroll
    for (int j = 0; j < kPer; ++j) acc[r][j] = 0.f;
  }
  for (int s0 = warp;; s0 += U * W) {
#pragma unroll
    for (int k = 0; k < U; ++k)
#pragma unroll
      for (int r = 0; r < ROWS; ++r) {
        const float mr = __shfl_sync(0xffffffffu, ml[k].x, r), lr = __shfl_sync(0xffffffffu, ml[k].y, r);
        if (mr == -INFINITY) continue;   // past the last slot (warp-uniform)
        const float Mn = fmaxf(M[r], mr);
        const float sc = exp2f(M[r] - Mn), wv = exp2f(mr - Mn);
        L[r] = L[r] * sc + wv * lr;
#pragma unroll
        for (int j = 0; j < kPer; ++j) acc[r][j] = acc[r][j] * sc + wv * v[k][r][j];
        M[r] = Mn;
      }
    if (s0 + U * W >= ns) break;
    // the next round of slots (more than U * W slots only)
#pragma unroll
    for (int k = 0; k < U; ++k) {
      const int sk = s0 + U * W + k * W;
      const int64_t pr = (static_cast<int64_t>(first) + (sk < ns ? sk : 0)) * group;
      ml[k] = (sk < ns && lane < group) ? __ldcg(reinterpret_cast<const float2*>(part_ml + (pr + lane) * 2))
                                        : make_float2(-INFINITY, 0.f);
#pragma unroll
      for (int r = 0; r < ROWS; ++r)
#pragma unroll
        for (int j = 0; j < kPer; ++j)
          v[k][r][j] = (sk < ns && r < group) ? __ldcg(part_o + (pr + r) * HD + lane + 32 * j) : 0.f;
    }
  }
#pragma unroll
  for (int r = 0; r < ROWS; ++r) {
    if (r < group) {
#pragma unroll
      for (int j = 0; j < kPer; ++j) s_acc[(warp * ROWS + r) * HD + lane + 32 * j] = acc[r][j];
      if (lane == 0) {
        s_m[warp * ROWS + r] = M[r];
        s_l[warp * ROWS + r] = L[r];
      }
    }
  }
  sync();
#pragma unroll
  for (int i = 0; i < kOut; ++i) {
    const int idx = tid + i * W * 32;
    if (idx >= group * HD) break;
    const int r = idx / HD, d = idx - r * HD;
    const float* ss = s_self + r * kMaxReadoutDepth;
    float Mt = ss[0];
    for (int e = 1; e < n_self; ++e) Mt = fmaxf(Mt, ss[e]);
#pragma unroll
    for (int w = 0; w < W; ++w) Mt = fmaxf(Mt, s_m[w * ROWS + r]);
    float num = 0.f, den = 0.f;
    for (int e = 0; e < n_self; ++e) {   // the self entries (one without a depth-k readout)
      const float ws = exp2f(ss[e] - Mt);
      num += ws * (e == t_self ? vsf[i] : __ldcg(mg.vself + (hk0 + e * n_kv) * HD + d));
      den += ws;
    }
#pragma unroll
    for (int w = 0; w < W; ++w) {
      const float mw = s_m[w * ROWS + r];
      if (mw == -INFINITY) continue;
      const float f = exp2f(mw - Mt);
      num += f * s_acc[(w * ROWS + r) * HD + d];
      den += f * s_l[w * ROWS + r];
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
}

}  // namespace ac
}  // namespace kvprm
