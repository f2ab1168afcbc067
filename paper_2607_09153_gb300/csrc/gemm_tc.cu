// Projection GEMMs of the verify-token forward, batched over candidates (the
// c_ffn * d^2 term of Eq. cost_kv): Y[n][m] = sum_k W[m][k] * X[n][k].
//
// The weight matrix is the streamed operand (read once from HBM per call), so
// it is the MMA's A operand: M = 128 weight rows per CTA, N = the candidate
// batch padded to a multiple of 16 (16..256), K in 64-element tiles.  A
// producer thread streams W and X tiles with TMA (128-byte swizzle) through a
// multi-stage mbarrier ring; one thread issues tcgen05.mma (kind::f16, bf16 x
// bf16 -> fp32) into a TMEM accumulator.  The activation X arrives as a bf16
// (hi, lo) pair, X = hi + lo to ~2^-17 relative, so the contraction sees the
// fp32 activation (the weights are bf16 by definition).  The hi and lo tiles
// sit back to back in shared memory and one MMA of N = 2 n_pad covers both
// (each weight K slice is read from shared memory once -- the MMA issue rate
// is bounded by those reads at this small N); the two accumulator halves are
// added when TMEM is read.  Beyond N = 256 each half takes its own MMA.
//
// K is split across the CTAs of a thread-block cluster (one cluster per
// 128-row tile) so that every SM streams weights.  The splits are reduced
// inside the cluster through distributed shared memory in rank order
// (deterministic, no float atomics): each CTA parks its accumulator in its own
// shared memory, and CTA r sums the candidate columns [r*N/cs, (r+1)*N/cs)
// over all ranks and applies the epilogue of the step:
//   PLAIN  out[n][m] = y
//   QKV    RoPE on the q and k rows (rotate-half pairs inside a head) -> q
//          (fp32 and bf16 hi/lo), self k, self v (fp32)
//   RESID  h[n][m] += y, the tile's sum of squares of the new h per
//          candidate, and h ⊙ g (g = the next RMSNorm's gain) as the next
//          projection's bf16 hi/lo input
//   SILU   rows are 64 gate rows and the matching 64 up rows (two TMA boxes
//          per stage); a = SiLU(gate) * up as a bf16 hi/lo pair
// An RMSNorm x = g ⊙ h / sqrt(mean(h^2) + eps) between two projections is
// thereby split: the per-candidate factor r = 1/sqrt(mean(h^2) + eps) is a
// scalar of the column, so W x = r (W (h ⊙ g)); the residual epilogue writes
// h ⊙ g and the per-tile sums of squares, and the QKV and SILU epilogues scale
// their accumulators by r before RoPE / SiLU.  No normalisation kernel runs
// between the projections.
#include <type_traits>
#include "kernels.h"
#include "ptx.cuh"

namespace kvprm {

namespace {

constexpr int kBM = 128;
constexpr int kBK = 64;
constexpr uint32_t kWTileBytes = kBM * kBK * 2;   // 16 KB
// after the ring: barriers, TMEM slot and 64 block-sum floats (512 B), then 256
// per-column RMSNorm factors (1 KB)
constexpr size_t kTailBytes = 512 + 1024 + 4096;   // barriers, RMSNorm factors, preloaded residual
constexpr int kHPreCols = 8;                        // residual columns preloaded per rank (128 rows each)
constexpr size_t kGemmMaxSmem = 200 * 1024;         // dynamic shared memory the kernel is configured for

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~static_cast<uintptr_t>(1023));
}

__device__ __forceinline__ void store_hilo(__nv_bfloat16* hi, __nv_bfloat16* lo, int64_t i, float x) {
  const __nv_bfloat16 h = __float2bfloat16_rn(x);
  hi[i] = h;
  lo[i] = __float2bfloat16_rn(x - __bfloat162float(h));
}

// LARGE (n_pad >= 64, one kernel image per batch class so that the small-batch code keeps its own
// register allocation): the residual epilogue issues a 16-column group's residual loads before
// using any and sums each column's squares in one pass over the parked tile, clusters of 4 reduce
// with 16-byte DSMEM loads, and the epilogues move 4 or 8 consecutive rows of a column per thread
// with 16-byte accesses (the 4-warp CTA is otherwise bound by 2- and 4-byte stores and by one load
// latency per column).
template <bool LARGE>
__global__ void __launch_bounds__(256, 2) gemm_cluster_kernel(const __grid_constant__ CUtensorMap tmW,
                                                           const __grid_constant__ CUtensorMap tmX,
                                                           const __grid_constant__ CUtensorMap tmXlo, int has_lo,
                                                           const __grid_constant__ CUtensorMap tmB,
                                                           const __grid_constant__ CUtensorMap tmT,
                                                           const __grid_constant__ CUtensorMap tmTlo, int k_main,
                                                           int k_tiles, int cs, int stages, uint32_t tmem_cols,
                                                           int n_pad, int mt_arg, GemmEpilogue ep, int* err,
                                                           unsigned long long* ts) {
  trace_begin(ts);
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  // m-tiles of this CTA (LARGE only): a stage holds mt weight tiles, then the activation tile(s)
  const int mt = LARGE ? mt_arg : 1;
  const uint32_t x_bytes = static_cast<uint32_t>(n_pad) * kBK * 2;
  const uint32_t w_bytes = kWTileBytes * static_cast<uint32_t>(mt);
  const uint32_t stage_bytes = w_bytes + x_bytes * (has_lo ? 2u : 1u);
  const uint32_t acc_bytes = static_cast<uint32_t>(n_pad) * kBM * 4;
  const uint32_t ring_bytes = stages * stage_bytes > acc_bytes ? stages * stage_bytes : acc_bytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + ring_bytes);
  uint64_t* empty = full + stages;
  uint64_t* done = empty + stages;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);
  float* red = reinterpret_cast<float*>(tmem_slot + 4);   // 64 floats for per-column block sums
  float* rsc = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(full) + 512);   // RMSNorm factor per column
  float* hpre = rsc + 256;   // RESID: this rank's columns of h for the tile's rows, [c - cbeg][128]

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int m_tile0 = blockIdx.x / cs * mt;   // first m-tile of this CTA
  const uint32_t rank = cluster_rank();
  const int kps = (k_tiles + cs - 1) / cs;
  const int kt0 = static_cast<int>(rank) * kps;
  const int kt1 = min(k_tiles, kt0 + kps);
  const int nk = kt1 > kt0 ? kt1 - kt0 : 0;
  const bool silu = ep.mode == GemmEpilogue::SILU;
  // this rank's candidate columns in the reduction and the epilogue
  const int cols = n_pad / cs;
  const int cbeg = static_cast<int>(rank) * cols;
  const int cend = min(cbeg + cols, ep.n_valid);
  const int nc = cend > cbeg ? cend - cbeg : 0;
  const bool hpreload = ep.mode == GemmEpilogue::RESID && nc <= kHPreCols && mt == 1;
  constexpr int kEpiBatch = LARGE ? 8 : 1;

  if (threadIdx.x == 0) {
    for (int s = 0; s < stages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(done, 1);
    fence_mbar_init();
    tma_prefetch_desc(&tmW);
    tma_prefetch_desc(&tmX);
    if (has_lo) tma_prefetch_desc(&tmXlo);
    if (k_main < k_tiles) {
      tma_prefetch_desc(&tmB);
      tma_prefetch_desc(&tmT);
      if (has_lo) tma_prefetch_desc(&tmTlo);
    }
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, tmem_cols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // Let the next kernel in the stream start its own independent prologue and
  // streaming now (or, with late_trigger, once the partials are parked); it
  // waits for this grid's completion before touching what this grid writes.
  if (!ep.late_trigger) grid_dep_launch();

  if (warp == 0 && lane == 0 && nk > 0) {
    // ---------------- TMA producer
    const uint64_t pol_w = policy_evict_first();
    const uint64_t pol_x = policy_evict_last();
    // K tiles [0, k_main) come from W and x; a scorer adapter's tiles after them from B and t
    auto load_w = [&](uint8_t* st, int kt, uint64_t* bar) {
      const CUtensorMap* wm = kt < k_main ? &tmW : &tmB;
      const int kx = (kt < k_main ? kt : kt - k_main) * kBK;
      for (int t = 0; t < mt; ++t) {
        const int m_tile = m_tile0 + t;
        uint8_t* wt = st + t * kWTileBytes;
        if (!silu) {
          tma_load_2d(wt, wm, bar, kx, m_tile * kBM, pol_w);
        } else {   // 64 gate rows, then the matching 64 up rows
          tma_load_2d(wt, wm, bar, kx, m_tile * 64, pol_w);
          tma_load_2d(wt + kWTileBytes / 2, wm, bar, kx, ep.ff + m_tile * 64, pol_w);
        }
      }
    };
    auto load_x = [&](uint8_t* st, int kt, uint64_t* bar) {
      const bool main = kt < k_main;
      const int kx = (main ? kt : kt - k_main) * kBK;
      tma_load_2d(st + w_bytes, main ? &tmX : &tmT, bar, kx, 0, pol_x);
      if (has_lo) tma_load_2d(st + w_bytes + x_bytes, main ? &tmXlo : &tmTlo, bar, kx, 0, pol_x);
    };
    // Weights do not depend on the preceding kernel: start streaming the first
    // ring's worth of W before waiting for the activations it produces.
    const int pre = min(stages, nk);
    for (int i = 0; i < pre; ++i) {
      mbar_arrive_expect_tx(&full[i], stage_bytes);
      load_w(smem + i * stage_bytes, kt0 + i, &full[i]);
    }
    grid_dep_wait();
    trace_event(ts, 0);   // the preceding kernel has completed
    for (int i = 0; i < pre; ++i) load_x(smem + i * stage_bytes, kt0 + i, &full[i]);
    for (int i = pre; i < nk; ++i) {
      const int s = i % stages;
      const uint32_t use = static_cast<uint32_t>(i / stages);
      if (!mbar_wait(&empty[s], (use & 1u) ^ 1u, err)) break;
      uint8_t* st = smem + s * stage_bytes;
      mbar_arrive_expect_tx(&full[s], stage_bytes);
      load_w(st, kt0 + i, &full[s]);
      load_x(st, kt0 + i, &full[s]);
    }
  } else if (warp >= 2) {
    // ---------------- while the weights stream: the RMSNorm factor of each of this rank's columns
    // (QKV, SILU), from the residual stream's tile sums of squares the preceding kernel wrote; the
    // parking barrier below orders these writes before the epilogue reads them
    grid_dep_wait();
    if (ep.rs_sumsq)
      for (int t0 = threadIdx.x - 64; t0 < nc; t0 += blockDim.x - 64) {   // nc <= 256 columns
        const int c = cbeg + t0;
        float ssum = 0.f;
        for (int t = 0; t < ep.rs_tiles; ++t) ssum += ep.rs_sumsq[static_cast<int64_t>(t) * ep.n_valid + c];
        rsc[t0] = 1.0f / sqrtf(ssum / ep.rs_d + ep.rs_eps);
      }
    // RESID: the residual values the epilogue adds to, read now rather than after the MMAs, when
    // the next kernel's weight stream may be competing for the memory system
    if (hpreload)
      for (int idx = threadIdx.x - 64; idx < nc * kBM; idx += blockDim.x - 64) {
        const int c = cbeg + idx / kBM, gm = m_tile0 * kBM + idx % kBM;
        hpre[idx] = gm < ep.M ? ep.h[static_cast<int64_t>(c) * ep.M + gm] : 0.f;
      }
  } else if (warp == 1 && nk > 0) {
    // ---------------- MMA issuer (the whole warp; one elected lane issues)
    // With the hi and lo activation tiles stored back to back (2 n_pad rows
    // under the same swizzle), one MMA of N = 2 n_pad reads each weight K
    // slice from shared memory once: columns [0, n_pad) accumulate W hi,
    // [n_pad, 2 n_pad) accumulate W lo, summed when the accumulator is read.
    // Beyond N = 256 the two halves take one MMA each into the same columns.
    // With two m-tiles per CTA, tile t accumulates from TMEM column t tile_cols (half the
    // allocation, a power of two).
    const bool merged = has_lo && 2 * n_pad <= 256;
    const bool two = has_lo && !merged;
    const uint32_t idesc = idesc_bf16_f32(kBM, merged ? 2 * n_pad : n_pad);
    const uint32_t tile_cols = tmem_cols / static_cast<uint32_t>(mt);
    for (int i = 0; i < nk; ++i) {
      const int s = i % stages;
      const uint32_t use = static_cast<uint32_t>(i / stages);
      if (!__all_sync(0xffffffffu, mbar_wait(&full[s], use & 1u, err))) break;
      if (i == 0 && lane == 0) trace_event(ts, 1);   // first weight and activation tiles landed
      tc_fence_after();
      const uint64_t a0 = desc_sw128(smem_u32(smem + s * stage_bytes));   // K step kk: + 2 kk (32 bytes)
      const uint64_t b0 = a0 + (w_bytes >> 4);
      const uint64_t l0 = b0 + static_cast<uint64_t>(x_bytes >> 4);
      const uint32_t acc0 = i > 0 ? 1u : 0u;
      for (int t = 0; t < mt; ++t) {
        const uint32_t d = tmem + static_cast<uint32_t>(t) * tile_cols;
        const uint64_t at = a0 + static_cast<uint64_t>(t) * (kWTileBytes >> 4);
        if (two) {
#pragma unroll
          for (int kk = 0; kk < kBK / 16; ++kk) {
            umma_bf16_w(d, at + 2 * kk, b0 + 2 * kk, idesc, kk > 0 ? 1u : acc0);
            umma_bf16_w(d, at + 2 * kk, l0 + 2 * kk, idesc, 1u);
          }
        } else {
#pragma unroll
          for (int kk = 0; kk < kBK / 16; ++kk) umma_bf16_w(d, at + 2 * kk, b0 + 2 * kk, idesc, kk > 0 ? 1u : acc0);
        }
      }
      umma_commit_w(&empty[s]);
    }
    umma_commit_w(done);
  }
  __syncwarp();

  // ---------------- accumulator -> own shared memory, acc[c][m] (fp32, c < n_pad, m < 128)
  const bool have = nk > 0 ? __all_sync(0xffffffffu, mbar_wait(done, 0, err)) : true;
  if (threadIdx.x == 0) trace_event(ts, 2);   // all MMAs of this CTA completed
  tc_fence_after();
  float* acc = reinterpret_cast<float*>(smem);   // the ring is idle once `done` has fired
  // 4 warps, or 8 (the large-batch image): warps w and w + 4 share TMEM lane quadrant w,
  // i.e. the tile's rows 32 w .. 32 w + 31, and take alternate 16-column groups (or columns)
  const int nw = static_cast<int>(blockDim.x >> 5), nwh = nw >> 2, wh = warp >> 2;
  const int m = (warp & 3) * 32 + lane;
  const bool merged = has_lo && 2 * n_pad <= 256;
  const uint32_t tile_cols = tmem_cols / static_cast<uint32_t>(mt);
  // one m-tile at a time: park it, reduce it over the cluster (split K), write its epilogue; with two
  // tiles and split K the second is parked once every peer has read this CTA's first partial
  for (int tt = 0; tt < mt; ++tt) {
    const int m_tile = m_tile0 + tt;
    const uint32_t tcol = static_cast<uint32_t>(tt) * tile_cols;
    if (tt > 0 && cs > 1) cluster_wait();   // matches the arrive after the previous tile's reduction
    for (int c0 = 16 * wh; c0 < n_pad; c0 += 16 * nwh) {
      float v[16];
      if (nk > 0 && have) {
        const uint32_t t = tmem + (static_cast<uint32_t>((warp & 3) * 32) << 16) + tcol + static_cast<uint32_t>(c0);
        tmem_ld16(t, v);
        if (merged) {
          float w[16];
          tmem_ld16(t + static_cast<uint32_t>(n_pad), w);
#pragma unroll
          for (int j = 0; j < 16; ++j) v[j] += w[j];
        }
      } else {
#pragma unroll
        for (int j = 0; j < 16; ++j) v[j] = 0.f;
      }
#pragma unroll
      for (int j = 0; j < 16; ++j) acc[(c0 + j) * kBM + m] = v[j];
    }
    tc_fence_before();
    if (tt == 0 || cs > 1) {
      cluster_sync();   // every rank's partial is parked
      if (tt == 0) {
        if (threadIdx.x == 0) trace_event(ts, 3);
        if (ep.late_trigger) grid_dep_launch();
        // ---------------- reduce this rank's candidate columns over the cluster, then the epilogue
        grid_dep_wait();   // outputs may still be read by kernels that precede this one
      }
      // Step 1: acc[c][m] <- sum over ranks of acc_r[c][m] for this rank's columns
      // (only this rank reads them, so it may overwrite its own copy).  Two columns
      // per round trip when the cluster has <= 8 ranks (four with 16-byte loads in
      // the large-batch image's clusters of 4), all peer loads in flight.
      // Without split K (cs = 1) the parked accumulator is already the sum.
      if (LARGE && (cs == 4 || cs == 8)) {
        // four consecutive rows of one column per thread (a warp covers a column's 128 rows), 16 / CS
        // columns per round: 16 loads of 16 bytes in flight, the CS ranks' copies of each; warp w takes
        // columns cbeg + w, cbeg + w + nw, ...
        auto vreduce = [&](auto cs_c) {
          constexpr int CS = decltype(cs_c)::value, PER = 16 / CS;
          const int rq = static_cast<int>(threadIdx.x) & 31, cg = static_cast<int>(threadIdx.x) >> 5;
          for (int c0 = cbeg + cg; c0 < cend; c0 += nw * PER) {
            float4 v[16];
#pragma unroll
            for (int k = 0; k < 16; ++k) {   // rank k % CS of column c0 + nw (k / CS)
              const int cc = c0 + nw * (k / CS);
              v[k] = cc < cend ? ld_cluster4(acc + cc * kBM + 4 * rq, static_cast<uint32_t>(k % CS))
                               : make_float4(0.f, 0.f, 0.f, 0.f);
            }
#pragma unroll
            for (int j = 0; j < PER; ++j) {
              const int cc = c0 + nw * j;
              if (cc >= cend) continue;
              const float4* u = v + CS * j;
              auto add = [](float4 x, float4 y) { return make_float4(x.x + y.x, x.y + y.y, x.z + y.z, x.w + y.w); };
              float4 r = add(add(u[0], u[1]), add(u[2], u[3]));
              if constexpr (CS == 8) r = add(r, add(add(u[4], u[5]), add(u[6], u[7])));
              *reinterpret_cast<float4*>(acc + cc * kBM + 4 * rq) = r;
            }
          }
        };
        if (cs == 4)
          vreduce(std::integral_constant<int, 4>{});
        else
          vreduce(std::integral_constant<int, 8>{});
      } else if (cs > 1) {
        const int step = cs <= 8 ? 2 : 1;
        for (int c = cbeg + wh * step; c < cend; c += step * nwh) {
          const bool two = step == 2 && c + 1 < cend;
          float v[16];
#pragma unroll
          for (int k = 0; k < 16; ++k) {
            const int r = step == 2 ? (k & 7) : k;
            const int cc = (step == 2 && k >= 8) ? c + 1 : c;
            const bool use = r < cs && (cc == c || two);
            v[k] = use ? ld_cluster(acc + cc * kBM + m, static_cast<uint32_t>(r)) : 0.f;
          }
          if (step == 2) {
            float s0 = 0.f, s1 = 0.f;
#pragma unroll
            for (int k = 0; k < 8; ++k) {
              s0 += v[k];
              s1 += v[8 + k];
            }
            __syncwarp();
            acc[c * kBM + m] = s0;
            if (two) acc[(c + 1) * kBM + m] = s1;
          } else {
            float s0 = 0.f;
#pragma unroll
            for (int k = 0; k < 16; ++k) s0 += v[k];
            acc[c * kBM + m] = s0;
          }
        }
      }
      if (threadIdx.x == 0) trace_event(ts, 4);   // this rank's columns are reduced over the cluster
      // no peer reads this tile's partial any more once every rank has arrived here: arrive now and
      // wait only before this shared memory is reused (the next tile's parking, or the exit), so the
      // barrier's latency hides behind the epilogue
      __syncwarp();
      cluster_arrive();
    }
    __syncthreads();   // every warp's reduced columns are in acc
    if (threadIdx.x == 0) trace_event(ts, 5);
    // QKV with the per-head q/k RMSNorm: the factor of each (column, head of this tile) over the
    // head's hd rows of the RMSNorm-scaled projection, 1/sqrt(mean(y^2) + eps) times the column's
    // RMSNorm factor (v heads keep the latter alone); parked where RESID preloads its residual
    float* qkf = hpre;   // [column][head of the tile]
    if (ep.mode == GemmEpilogue::QKV && ep.qn_gain) {
      const int hpt = kBM / ep.hd;   // heads per tile: 1 (hd 128) or 2 (hd 64)
      for (int it = warp; it < nc * hpt; it += nw) {
        const int cl = it / hpt, hh = it % hpt;
        const float* col = acc + (cbeg + cl) * kBM + hh * ep.hd;
        float sq = 0.f;
        for (int r = lane; r < ep.hd; r += 32) sq += col[r] * col[r];
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, off);
        if (lane == 0) {
          const float rs = ep.rs_sumsq ? rsc[cl] : 1.f;
          const int head = m_tile * (kBM / ep.hd) + hh;
          qkf[cl * 2 + hh] = head < ep.n_q + ep.n_kv ? rs / sqrtf(rs * rs * sq / ep.hd + ep.rs_eps) : rs;
        }
      }
      __syncthreads();
    }
    // Step 2: the epilogue over (row, column) pairs, all threads in parallel
    if (ep.mode == GemmEpilogue::PLAIN) {
      const int gm = m_tile * kBM + m;
      if (gm < ep.M)
        for (int c = cbeg + wh; c < cend; c += nwh) ep.out[static_cast<int64_t>(c) * ep.M + gm] = acc[c * kBM + m];
    } else if (LARGE && ep.mode == GemmEpilogue::LOWRANK) {   // t = s (A x), hi/lo [n][r]; large image only
      const int gm = m_tile * kBM + m;
      if (gm < ep.M)
        for (int c = cbeg + wh; c < cend; c += nwh)
          store_hilo(ep.t_hi, ep.t_lo, static_cast<int64_t>(c) * ep.M + gm, ep.lr_scale * acc[c * kBM + m]);
    } else if (ep.mode == GemmEpilogue::RESID && LARGE) {
      // pass 1, 16 columns at a time with the group's residual loads in flight before the first use:
      // h += acc, the next projection's input, and hv^2 parked in place of acc (each (column, row)
      // slot is this thread's own)
      const int gm = m_tile * kBM + m;
      const float gain = (ep.gain_next && gm < ep.M) ? __bfloat162float(ep.gain_next[gm]) : 0.f;
      if ((ep.M & 3) == 0) {
        // four consecutive rows of one column per thread (a warp covers one column's 128 rows):
        // 16-byte residual loads and stores, 8-byte hi/lo stores; eight columns' loads in flight
        const int rq = static_cast<int>(threadIdx.x) & 31, cg = static_cast<int>(threadIdx.x) >> 5;
        const int gm0 = m_tile * kBM + 4 * rq;
        const bool rows_ok = gm0 < ep.M;   // M % 4 == 0: the four rows are all valid or all past M
        float g4[4] = {0.f, 0.f, 0.f, 0.f};
        if (ep.gain_next && rows_ok) {
          const uint2 gb = *reinterpret_cast<const uint2*>(ep.gain_next + gm0);
          const float2 ga = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&gb.x));
          const float2 gc = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&gb.y));
          g4[0] = ga.x;
          g4[1] = ga.y;
          g4[2] = gc.x;
          g4[3] = gc.y;
        }
        for (int c0 = cbeg + cg; c0 < cend; c0 += nw * 8) {
          float4 h_in[8];
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const int c = c0 + nw * k;
            h_in[k] = (c < cend && rows_ok) ? *reinterpret_cast<const float4*>(ep.h + static_cast<int64_t>(c) * ep.M + gm0)
                                            : make_float4(0.f, 0.f, 0.f, 0.f);
          }
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const int c = c0 + nw * k;
            if (c >= cend) break;
            float4* ap = reinterpret_cast<float4*>(acc + c * kBM + 4 * rq);
            const float4 a = *ap;
            float4 hv = make_float4(0.f, 0.f, 0.f, 0.f);
            if (rows_ok) {
              hv = make_float4(h_in[k].x + a.x, h_in[k].y + a.y, h_in[k].z + a.z, h_in[k].w + a.w);
              const int64_t o = static_cast<int64_t>(c) * ep.M + gm0;
              *reinterpret_cast<float4*>(ep.h + o) = hv;
              if (ep.h_copy) *reinterpret_cast<float4*>(ep.h_copy + o) = hv;
              if (ep.gain_next) {
                const float x[4] = {hv.x * g4[0], hv.y * g4[1], hv.z * g4[2], hv.w * g4[3]};
                uint32_t hi[2], lo[2];
#pragma unroll
                for (int e = 0; e < 2; ++e) {
                  const __nv_bfloat162 h2 = __floats2bfloat162_rn(x[2 * e], x[2 * e + 1]);
                  const float2 hf = __bfloat1622float2(h2);
                  const __nv_bfloat162 l2 = __floats2bfloat162_rn(x[2 * e] - hf.x, x[2 * e + 1] - hf.y);
                  hi[e] = *reinterpret_cast<const uint32_t*>(&h2);
                  lo[e] = *reinterpret_cast<const uint32_t*>(&l2);
                }
                *reinterpret_cast<uint2*>(ep.x_hi + o) = make_uint2(hi[0], hi[1]);
                *reinterpret_cast<uint2*>(ep.x_lo + o) = make_uint2(lo[0], lo[1]);
              }
            }
            *ap = make_float4(hv.x * hv.x, hv.y * hv.y, hv.z * hv.z, hv.w * hv.w);
          }
        }
      } else {   // warps w and w + 4 share rows: alternate 16-column groups
        for (int c0 = cbeg + 16 * wh; c0 < cend; c0 += 16 * nwh) {
          float h_in[16];
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            const int c = c0 + j;
            h_in[j] = (c < cend && gm < ep.M) ? ep.h[static_cast<int64_t>(c) * ep.M + gm] : 0.f;
          }
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            const int c = c0 + j;
            if (c >= cend) break;
            float hv = 0.f;
            if (gm < ep.M) {
              hv = h_in[j] + acc[c * kBM + m];
              ep.h[static_cast<int64_t>(c) * ep.M + gm] = hv;
              if (ep.gain_next) store_hilo(ep.x_hi, ep.x_lo, static_cast<int64_t>(c) * ep.M + gm, hv * gain);
            }
            acc[c * kBM + m] = hv * hv;
          }
        }
      }
      __syncthreads();
      // pass 2: each column's sum of squares over the tile's 128 rows, eight threads per column
      // (rows part + 8 q, the start of q rotated per column so that a warp's four columns hit
      // different banks), warp-uniform trip count for the shuffles
      for (int t0 = 0; t0 < nc * 8; t0 += blockDim.x) {
        const int t = t0 + static_cast<int>(threadIdx.x);
        const int cl = t >> 3, part = t & 7;
        float sq = 0.f;
        if (t < nc * 8) {
          const float* col = acc + (cbeg + cl) * kBM + part;
#pragma unroll
          for (int q = 0; q < 16; ++q) sq += col[8 * ((q + (cl & 3)) & 15)];
        }
        sq += __shfl_xor_sync(0xffffffffu, sq, 1);
        sq += __shfl_xor_sync(0xffffffffu, sq, 2);
        sq += __shfl_xor_sync(0xffffffffu, sq, 4);
        if (t < nc * 8 && part == 0) ep.sumsq[static_cast<int64_t>(m_tile) * ep.n_valid + cbeg + cl] = sq;
      }
    } else if (ep.mode == GemmEpilogue::RESID) {
      const int gm = m_tile * kBM + m;
      float* sq_s = red;   // [16 columns][4 warps]
      for (int c0 = cbeg; c0 < cend; c0 += 16) {
        const int c1 = min(cend, c0 + 16);
        {
          for (int c = c0; c < c1; ++c) {
            float hv = 0.f;
            if (gm < ep.M) {
              float* hp = ep.h + static_cast<int64_t>(c) * ep.M + gm;
              hv = (hpreload ? hpre[(c - cbeg) * kBM + m] : *hp) + acc[c * kBM + m];
              *hp = hv;
              if (ep.h_copy) ep.h_copy[static_cast<int64_t>(c) * ep.M + gm] = hv;
              if (ep.gain_next)
                store_hilo(ep.x_hi, ep.x_lo, static_cast<int64_t>(c) * ep.M + gm, hv * __bfloat162float(ep.gain_next[gm]));
            }
            float sq = hv * hv;
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, off);
            if (lane == 0) sq_s[(c - c0) * 4 + warp] = sq;
          }
        }
        __syncthreads();
        if (threadIdx.x < c1 - c0) {
          const float* q4 = sq_s + threadIdx.x * 4;
          ep.sumsq[static_cast<int64_t>(m_tile) * ep.n_valid + c0 + threadIdx.x] = (q4[0] + q4[1]) + (q4[2] + q4[3]);
        }
        __syncthreads();
      }
    } else if (ep.mode == GemmEpilogue::SILU && LARGE && (ep.ff & 7) == 0) {
      // eight consecutive rows of one column per thread (8 row groups x 16 column groups): 16-byte
      // loads from the parked tile and one 16-byte store for each of the hi and lo halves (2-byte
      // stores, 256 per warp and tile at B = 256, bound the scalar form); the exponential and the
      // divide take the fast intrinsics
      const int rg = static_cast<int>(threadIdx.x) & 7, cg = static_cast<int>(threadIdx.x) >> 3;
      const int j0 = m_tile * 64 + 8 * rg;   // ff % 8 == 0: a row group is all valid or all past ff
      if (j0 < ep.ff) {
#pragma unroll 2
        for (int c = cbeg + cg; c < cend; c += 4 * nw) {   // 4 nw column groups of 8 threads
          const float rs = ep.rs_sumsq ? rsc[c - cbeg] : 1.f;
          const float4* gp = reinterpret_cast<const float4*>(acc + c * kBM + 8 * rg);
          const float4* up = reinterpret_cast<const float4*>(acc + c * kBM + 64 + 8 * rg);
          const float4 g0 = gp[0], g1 = gp[1], u0 = up[0], u1 = up[1];
          const float g[8] = {g0.x, g0.y, g0.z, g0.w, g1.x, g1.y, g1.z, g1.w};
          const float u[8] = {u0.x, u0.y, u0.z, u0.w, u1.x, u1.y, u1.z, u1.w};
          uint32_t hi[4], lo[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float ga = g[2 * e] * rs, gb = g[2 * e + 1] * rs;
            const float a = __fdividef(ga, 1.0f + __expf(-ga)) * (u[2 * e] * rs);
            const float b = __fdividef(gb, 1.0f + __expf(-gb)) * (u[2 * e + 1] * rs);
            const __nv_bfloat162 h2 = __floats2bfloat162_rn(a, b);
            const float2 hf = __bfloat1622float2(h2);
            const __nv_bfloat162 l2 = __floats2bfloat162_rn(a - hf.x, b - hf.y);
            hi[e] = *reinterpret_cast<const uint32_t*>(&h2);
            lo[e] = *reinterpret_cast<const uint32_t*>(&l2);
          }
          const int64_t o = static_cast<int64_t>(c) * ep.ff + j0;
          *reinterpret_cast<uint4*>(ep.a_hi + o) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
          *reinterpret_cast<uint4*>(ep.a_lo + o) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
          if (ep.gu_save) {   // gate and up pre-activations (after the RMSNorm factor) for a backward pass
            float4* gs = reinterpret_cast<float4*>(ep.gu_save + static_cast<int64_t>(c) * 2 * ep.ff + j0);
            float4* us = reinterpret_cast<float4*>(ep.gu_save + static_cast<int64_t>(c) * 2 * ep.ff + ep.ff + j0);
            gs[0] = make_float4(g[0] * rs, g[1] * rs, g[2] * rs, g[3] * rs);
            gs[1] = make_float4(g[4] * rs, g[5] * rs, g[6] * rs, g[7] * rs);
            us[0] = make_float4(u[0] * rs, u[1] * rs, u[2] * rs, u[3] * rs);
            us[1] = make_float4(u[4] * rs, u[5] * rs, u[6] * rs, u[7] * rs);
          }
        }
      }
    } else if (ep.mode == GemmEpilogue::SILU) {
      // 2 nhalf column groups of 64 threads (rows m and m + 64 of a column share a group)
      const int r = m & 63, ng = 2 * nwh, grp = (m >> 6) + 2 * wh;
      const int j = m_tile * 64 + r;
      if (j < ep.ff)
        for (int c0 = cbeg + grp; c0 < cend; c0 += ng * kEpiBatch) {
          float g[kEpiBatch], u[kEpiBatch];   // a batch's operands, read before its first store
#pragma unroll
          for (int k = 0; k < kEpiBatch; ++k) {
            const int c = c0 + ng * k;
            const bool ok = c < cend;
            const float rs = (ok && ep.rs_sumsq) ? rsc[c - cbeg] : 1.f;
            g[k] = ok ? acc[c * kBM + r] * rs : 0.f;
            u[k] = ok ? acc[c * kBM + 64 + r] * rs : 0.f;
          }
#pragma unroll
          for (int k = 0; k < kEpiBatch; ++k) {
            const int c = c0 + ng * k;
            if (c < cend) {
              store_hilo(ep.a_hi, ep.a_lo, static_cast<int64_t>(c) * ep.ff + j, g[k] / (1.0f + expf(-g[k])) * u[k]);
              if (ep.gu_save) {   // gate and up pre-activations for a backward pass
                ep.gu_save[static_cast<int64_t>(c) * 2 * ep.ff + j] = g[k];
                ep.gu_save[static_cast<int64_t>(c) * 2 * ep.ff + ep.ff + j] = u[k];
              }
            }
          }
        }
    } else if (LARGE && (ep.hd & 7) == 0) {
      // QKV, four consecutive RoPE pairs (i .. i + 3, partners i + half ..) of one column per
      // thread (16 pair groups x 8 column groups): 16-byte loads of the parked tile and the
      // rotation, 16-byte fp32 and 8-byte hi/lo stores; two columns' operands in flight
      const int pq = 4 * (static_cast<int>(threadIdx.x) & 15), cg = static_cast<int>(threadIdx.x) >> 4;
      const int hd = ep.hd, half = hd / 2;
      const int row_a = (pq / half) * hd + (pq % half);   // half % 4 == 0: the four pairs share a head
      const int row_b = row_a + half;
      const int grow = m_tile * kBM + row_a;
      const int head = grow / hd, i = grow % hd;
      const bool rot = head < ep.n_q + ep.n_kv;
      // per-head q/k RMSNorm: the gains of these rows (q heads: q_norm, k heads: k_norm)
      const bool qkn = ep.qn_gain != nullptr && rot;
      float gna[4] = {1.f, 1.f, 1.f, 1.f}, gnb[4] = {1.f, 1.f, 1.f, 1.f};
      if (qkn) {
        const __nv_bfloat16* gsrc = head < ep.n_q ? ep.qn_gain : ep.kn_gain;
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          gna[e] = __bfloat162float(gsrc[i + e]);
          gnb[e] = __bfloat162float(gsrc[i + half + e]);
        }
      }
      const int hh_tile = row_a / hd;   // head of this tile
      auto store4 = [&](float* dst, __nv_bfloat16* dhi, __nv_bfloat16* dlo, int64_t o, const float (&x)[4]) {
        *reinterpret_cast<float4*>(dst + o) = make_float4(x[0], x[1], x[2], x[3]);
        if (dhi) {
          uint32_t hi[2], lo[2];
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            const __nv_bfloat162 h2 = __floats2bfloat162_rn(x[2 * e], x[2 * e + 1]);
            const float2 hf = __bfloat1622float2(h2);
            const __nv_bfloat162 l2 = __floats2bfloat162_rn(x[2 * e] - hf.x, x[2 * e + 1] - hf.y);
            hi[e] = *reinterpret_cast<const uint32_t*>(&h2);
            lo[e] = *reinterpret_cast<const uint32_t*>(&l2);
          }
          *reinterpret_cast<uint2*>(dhi + o) = make_uint2(hi[0], hi[1]);
          *reinterpret_cast<uint2*>(dlo + o) = make_uint2(lo[0], lo[1]);
        }
      };
      if (head < ep.n_q + 2 * ep.n_kv) {
#pragma unroll 2
        for (int c = cbeg + cg; c < cend; c += 2 * nw) {   // 2 nw column groups of 16 threads
          const float rs = ep.qn_gain ? qkf[(c - cbeg) * 2 + hh_tile] : (ep.rs_sumsq ? rsc[c - cbeg] : 1.f);
          const float4 a4 = *reinterpret_cast<const float4*>(acc + c * kBM + row_a);
          const float4 b4 = *reinterpret_cast<const float4*>(acc + c * kBM + row_b);
          float4 r0 = make_float4(1.f, 0.f, 1.f, 0.f), r1 = r0;   // (cos, sin) of pairs i, i+1 / i+2, i+3
          if (rot) {
            const float4* rp = reinterpret_cast<const float4*>(ep.rope + c * half + i);
            r0 = rp[0];
            r1 = rp[1];
          }
          const float cs_[4] = {r0.x, r0.z, r1.x, r1.z}, sn_[4] = {r0.y, r0.w, r1.y, r1.w};
          const float av[4] = {a4.x * rs * gna[0], a4.y * rs * gna[1], a4.z * rs * gna[2], a4.w * rs * gna[3]};
          const float bv[4] = {b4.x * rs * gnb[0], b4.y * rs * gnb[1], b4.z * rs * gnb[2], b4.w * rs * gnb[3]};
          float oa[4], ob[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            if (rot) {
              oa[e] = av[e] * cs_[e] - bv[e] * sn_[e];
              ob[e] = bv[e] * cs_[e] + av[e] * sn_[e];
            } else {
              oa[e] = av[e];
              ob[e] = bv[e];
            }
          }
          if (head < ep.n_q) {
            const int64_t o = (static_cast<int64_t>(c) * ep.n_q + head) * hd + i;
            store4(ep.q, ep.q_hi, ep.q_lo, o, oa);
            store4(ep.q, ep.q_hi, ep.q_lo, o + half, ob);
          } else {
            const bool is_k = head < ep.n_q + ep.n_kv;
            const int kvh = is_k ? head - ep.n_q : head - ep.n_q - ep.n_kv;
            float* dst = is_k ? ep.kself : ep.vself;
            const int64_t o = (static_cast<int64_t>(c) * ep.n_kv + kvh) * hd + i;
            store4(dst, nullptr, nullptr, o, oa);
            store4(dst, nullptr, nullptr, o + half, ob);
          }
        }
      }
    } else {   // QKV: pair p = m & 63 of this tile, 2 nhalf column groups of 64 threads
      const int p = m & 63, ng = 2 * nwh, grp = (m >> 6) + 2 * wh;
      const int hd = ep.hd, half = hd / 2;
      const int row_a = (p / half) * hd + (p % half);   // first element of the pair, within the tile
      const int row_b = row_a + half;
      const int grow = m_tile * kBM + row_a;              // row of W_qkv
      const int head = grow / hd, i = grow % hd;          // i < half
      const bool rot = head < ep.n_q + ep.n_kv;   // q and k rows take RoPE, v rows do not
      // per-head q/k RMSNorm (q heads: q_norm, k heads: k_norm gains of these two rows)
      float gna = 1.f, gnb = 1.f;
      if (ep.qn_gain && rot) {
        const __nv_bfloat16* gsrc = head < ep.n_q ? ep.qn_gain : ep.kn_gain;
        gna = __bfloat162float(gsrc[i]);
        gnb = __bfloat162float(gsrc[i + half]);
      }
      const int hh_tile = row_a / hd;
      for (int c0 = cbeg + grp; c0 < cend; c0 += ng * kEpiBatch) {
        // a batch's operands (accumulator pair and rotation), read before its first store
        float av[kEpiBatch], bv[kEpiBatch];
        float2 cs2[kEpiBatch];
#pragma unroll
        for (int k = 0; k < kEpiBatch; ++k) {
          const int c = c0 + ng * k;
          const bool ok = c < cend;
          const float rs = !ok ? 1.f : (ep.qn_gain ? qkf[(c - cbeg) * 2 + hh_tile] : (ep.rs_sumsq ? rsc[c - cbeg] : 1.f));
          av[k] = ok ? acc[c * kBM + row_a] * rs * gna : 0.f;
          bv[k] = ok ? acc[c * kBM + row_b] * rs * gnb : 0.f;
          cs2[k] = (ok && rot) ? ep.rope[c * half + i] : make_float2(1.f, 0.f);
        }
#pragma unroll
        for (int k = 0; k < kEpiBatch; ++k) {
          const int c = c0 + ng * k;
          if (c >= cend) break;
          float a = av[k], b = bv[k];
          if (rot) {
            const float a2 = a * cs2[k].x - b * cs2[k].y;
            const float b2 = b * cs2[k].x + a * cs2[k].y;
            a = a2;
            b = b2;
          }
          if (head < ep.n_q) {
            const int64_t o = (static_cast<int64_t>(c) * ep.n_q + head) * hd + i;
            ep.q[o] = a;
            ep.q[o + half] = b;
            store_hilo(ep.q_hi, ep.q_lo, o, a);
            store_hilo(ep.q_hi, ep.q_lo, o + half, b);
          } else if (head < ep.n_q + 2 * ep.n_kv) {
            const bool is_k = head < ep.n_q + ep.n_kv;
            const int kvh = is_k ? head - ep.n_q : head - ep.n_q - ep.n_kv;
            float* dst = (is_k ? ep.kself : ep.vself) + (static_cast<int64_t>(c) * ep.n_kv + kvh) * hd + i;
            dst[0] = a;
            dst[half] = b;
          }
        }
      }
    }
    if (tt + 1 < mt) __syncthreads();   // every thread is done with acc before the next tile is parked
  }
  (void)nc;
  if (threadIdx.x == 0) trace_event(ts, 6);   // this thread's epilogue written
  __syncwarp();
  cluster_wait();   // peers have finished reading this CTA's partial
  if (threadIdx.x == 0) trace_event(ts, 7);
  if (warp == 1) tmem_dealloc(tmem, tmem_cols);
  trace_end(ts);
}

}  // namespace

GemmPlan plan_gemm(int M, int K, int n_pad, int num_sms, bool has_lo, bool gate_up) {
  GemmPlan p;
  p.has_lo = has_lo;
  p.gate_up = gate_up;
  p.m_tiles = gate_up ? (M + 63) / 64 : (M + kBM - 1) / kBM;   // gate/up: M = d_ff, 64 pairs per tile
  p.k_tiles = (K + kBK - 1) / kBK;
  const uint32_t stage_bytes = kWTileBytes + static_cast<uint32_t>(n_pad) * kBK * 2 * (has_lo ? 2u : 1u);
  int stages = static_cast<int>((112u * 1024u) / stage_bytes);
  p.stages = stages < 2 ? 2 : (stages > 8 ? 8 : stages);
  // the parked accumulator (n_pad x 128 fp32) reuses the ring
  size_t ring = static_cast<size_t>(p.stages) * stage_bytes;
  const size_t acc = static_cast<size_t>(n_pad) * kBM * 4;
  if (ring < acc) ring = acc;
  p.smem_bytes = ring + 1024 /*align*/ + kTailBytes;
  // cluster size: the largest power of two <= 16 that keeps the CTA count within what fits on the
  // SMs at once (two per SM when two CTAs' shared memory fits, else one: at B = 256 a stage holds
  // 64 KB of activations) and gives every rank at least two K tiles
  const int per_sm = p.smem_bytes + 1024 <= 228u * 1024u / 2 ? 2 : 1;
  // A cluster is placed whole on one GPC.  With two CTAs per SM, a grid that needs (nearly) every
  // slot cannot be placed in one wave while the preceding kernel still holds part of the SMs
  // (programmatic dependent launch places this grid's first clusters early, half-filling SMs in a
  // pattern that strands slots): the 7B QKV projection at B = 64, 36 clusters of 8 = 288 of 304
  // slots, had its last clusters start ~10 us after the preceding kernel ended.  Such grids keep
  // within 7/8 of the slots.
  const int slots = per_sm == 2 ? per_sm * num_sms * 7 / 8 : per_sm * num_sms;
  int cs = 1;
  while (cs < 16 && p.m_tiles * cs * 2 <= slots && cs * 4 <= p.k_tiles && cs * 2 <= n_pad) cs *= 2;
  p.cluster = cs;
  p.splits = cs;
  p.kt_per_split = (p.k_tiles + cs - 1) / cs;
  // a ring deeper than the K tiles one CTA streams only holds shared memory
  // that overlapping kernels could use
  if (p.stages > p.kt_per_split) p.stages = p.kt_per_split < 2 ? 2 : p.kt_per_split;
  ring = static_cast<size_t>(p.stages) * stage_bytes;
  if (ring < acc) ring = acc;
  p.smem_bytes = ring + 1024 /*align*/ + kTailBytes;
  uint32_t cols = 32;
  const int need = (has_lo && 2 * n_pad <= 256) ? 2 * n_pad : n_pad;   // merged hi/lo accumulator halves
  while (cols < static_cast<uint32_t>(need)) cols <<= 1;
  p.tmem_cols = cols;
  // gate/up at large batches without split K: when one-tile CTAs would need two waves, a CTA takes
  // two m-tiles, so that every stage's activation tile (four times the weight tile at B = 256 with
  // the lo half) serves both, and the grid fits on the SMs at once
  if (gate_up && n_pad > 64 && cs == 1 && p.m_tiles % 2 == 0 && p.m_tiles > per_sm * num_sms) {
    const uint32_t st2 = 2 * kWTileBytes + static_cast<uint32_t>(n_pad) * kBK * 2 * (has_lo ? 2u : 1u);
    int stages2 = static_cast<int>((192u * 1024u) / st2);
    if (stages2 > 8) stages2 = 8;
    if (stages2 > p.kt_per_split) stages2 = p.kt_per_split;
    size_t ring2 = static_cast<size_t>(stages2) * st2;
    if (ring2 < acc) ring2 = acc;
    const size_t smem2 = ring2 + 1024 + kTailBytes;
    if (stages2 >= 2 && 2 * cols <= 512 && smem2 <= kGemmMaxSmem && (p.m_tiles / 2) <= num_sms) {
      p.mt = 2;
      p.stages = stages2;
      p.smem_bytes = smem2;
      p.tmem_cols = 2 * cols;
    }
  }
  // long split-K loops at large batches (the 7B down projection at B = 256: 74 K tiles per rank): two
  // m-tiles per CTA over twice the ranks, the same CTA count.  A 96 KB stage then carries 16 MMAs
  // (~1 us), enough to cover its own loading (~0.8 us), where one tile's 8 MMAs left the tensor pipe
  // waiting a third of the time; the second tile's parking and cluster reduction cost less than those
  // stalls once the K loop is long
  if (!gate_up && n_pad >= 128 && per_sm == 1 && p.mt == 1 && cs >= 2 && cs * 2 <= 8 && p.m_tiles % 2 == 0 &&
      p.kt_per_split >= 32) {
    const int cs2 = cs * 2;
    const uint32_t st2 = 2 * kWTileBytes + static_cast<uint32_t>(n_pad) * kBK * 2 * (has_lo ? 2u : 1u);
    const int kps2 = (p.k_tiles + cs2 - 1) / cs2;
    int stages2 = static_cast<int>((192u * 1024u) / st2);
    if (stages2 > 8) stages2 = 8;
    if (stages2 > kps2) stages2 = kps2;
    size_t ring2 = static_cast<size_t>(stages2) * st2;
    if (ring2 < acc) ring2 = acc;
    const size_t smem2 = ring2 + 1024 + kTailBytes;
    if (stages2 >= 2 && 2 * p.tmem_cols <= 512 && smem2 <= kGemmMaxSmem && (p.m_tiles / 2) * cs2 <= num_sms &&
        cs2 * 4 <= p.k_tiles && n_pad % cs2 == 0) {
      p.mt = 2;
      p.cluster = cs2;
      p.splits = cs2;
      p.kt_per_split = kps2;
      p.stages = stages2;
      p.smem_bytes = smem2;
      p.tmem_cols = 2 * p.tmem_cols;
    }
  }
  // the large-batch image runs eight warps instead of four (registers for two such CTAs per SM), so
  // that the parking, the cluster reduction and the epilogue after the MMAs run on twice the warps
  p.threads = n_pad >= 64 ? 256 : 128;
  return p;
}

cudaError_t gemm_configure() {
  cudaError_t e = cudaFuncSetAttribute(gemm_cluster_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(kGemmMaxSmem));
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(gemm_cluster_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(kGemmMaxSmem));
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(gemm_cluster_kernel<false>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(gemm_cluster_kernel<true>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
}

cudaError_t launch_gemm(const GemmPlan& p, const CUtensorMap* tmW, const CUtensorMap* tmX, const CUtensorMap* tmXlo,
                        const GemmEpilogue& ep, int n_pad, int* err, cudaStream_t stream, bool pdl,
                        unsigned long long* ts, const GemmLowRank* lr) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((p.m_tiles + p.mt - 1) / p.mt * p.cluster, 1, 1);
  const bool large = n_pad >= 64 || ep.mode == GemmEpilogue::LOWRANK;
  if (p.threads != 128 && (p.threads != 256 || !large)) return cudaErrorInvalidValue;
  cfg.blockDim = dim3(static_cast<unsigned>(p.threads), 1, 1);
  cfg.dynamicSmemBytes = p.smem_bytes;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = p.cluster;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 2 : 1;
  const CUtensorMap& xlo = p.has_lo ? *tmXlo : *tmX;
  // without an adapter every K tile is W's and x's (the extra maps are never read)
  const bool with_lr = lr && lr->b && lr->t_hi && (!p.has_lo || lr->t_lo);
  if (with_lr && (lr->k_main < 1 || lr->k_main >= p.k_tiles)) return cudaErrorInvalidValue;
  const CUtensorMap& mb = with_lr ? *lr->b : *tmW;
  const CUtensorMap& mt = with_lr ? *lr->t_hi : *tmX;
  const CUtensorMap& mtl = with_lr ? (p.has_lo ? *lr->t_lo : *lr->t_hi) : xlo;
  const int k_main = with_lr ? lr->k_main : p.k_tiles;
  // the adapter's A x (LOWRANK) runs on the large-batch image at every batch size, so that the
  // small-batch image keeps its register allocation
  if (large)
    return cudaLaunchKernelEx(&cfg, gemm_cluster_kernel<true>, *tmW, *tmX, xlo, p.has_lo ? 1 : 0, mb, mt, mtl, k_main,
                              p.k_tiles, p.cluster, p.stages, p.tmem_cols, n_pad, p.mt, ep, err, ts);
  if (p.mt != 1) return cudaErrorInvalidValue;   // two m-tiles per CTA exist in the large-batch image only
  return cudaLaunchKernelEx(&cfg, gemm_cluster_kernel<false>, *tmW, *tmX, xlo, p.has_lo ? 1 : 0, mb, mt, mtl, k_main,
                            p.k_tiles, p.cluster, p.stages, p.tmem_cols, n_pad, 1, ep, err, ts);
}

}  // namespace kvprm
