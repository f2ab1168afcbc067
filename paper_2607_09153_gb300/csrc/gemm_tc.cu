// Projection GEMM for the verify token, batched over candidates (the
// c_ffn * d^2 term of Eq. cost_kv): part[s][n][m] = sum_{k in split s} W[m][k] * X[n][k].
//
// The activation X arrives as a pair of bf16 tensors (hi, lo) with
// X = hi + lo to ~2^-17 relative: each K step issues two MMAs (W*hi, W*lo)
// into the same fp32 accumulator, so the contraction sees the fp32
// activation, not a bf16 rounding of it (the weights are bf16 by definition).
//
// The weight matrix is the streamed operand (read once from HBM per call), so
// it is the MMA's A operand: M = 128 weight rows per CTA, N = the candidate
// batch padded to a multiple of 16 (16..256), K in 64-element tiles.  A
// producer thread streams W and X tiles with TMA (128-byte swizzle) through a
// multi-stage mbarrier ring; one thread issues tcgen05.mma (kind::f16, bf16 x
// bf16 -> fp32) into a TMEM accumulator; four warps read TMEM back with
// tcgen05.ld and store fp32 split-K partials.  K is split across CTAs so that
// every SM streams weights; the consumer kernel reduces the splits in a fixed
// order (deterministic, no float atomics) fused with its own epilogue.
#include "kernels.h"
#include "ptx.cuh"

namespace kvprm {

namespace {

constexpr int kBM = 128;
constexpr int kBK = 64;
constexpr uint32_t kWTileBytes = kBM * kBK * 2;   // 16 KB

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~static_cast<uintptr_t>(1023));
}

__global__ void __launch_bounds__(128) gemm_wstream_kernel(const __grid_constant__ CUtensorMap tmW,
                                                           const __grid_constant__ CUtensorMap tmX,
                                                           const __grid_constant__ CUtensorMap tmXlo, int has_lo,
                                                           float* __restrict__ part, int M, int n_valid, int n_pad,
                                                           int k_tiles, int kt_per_split, int stages,
                                                           uint32_t tmem_cols, int* err) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  const uint32_t x_bytes = static_cast<uint32_t>(n_pad) * kBK * 2;
  const uint32_t stage_bytes = kWTileBytes + x_bytes * (has_lo ? 2u : 1u);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + stages * stage_bytes);
  uint64_t* empty = full + stages;
  uint64_t* done = empty + stages;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int m_tile = blockIdx.x, split = blockIdx.y;
  const int kt0 = split * kt_per_split;
  const int kt1 = min(k_tiles, kt0 + kt_per_split);
  const int nk = kt1 - kt0;

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
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, tmem_cols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0 && lane == 0) {
    // ---------------- TMA producer
    const uint64_t pol_w = policy_evict_first();
    const uint64_t pol_x = policy_evict_last();
    // Weights do not depend on the preceding kernel: start streaming the first
    // ring's worth of W before waiting for the activations it produces.
    const int pre = min(stages, nk);
    for (int i = 0; i < pre; ++i) {
      uint8_t* st = smem + i * stage_bytes;
      mbar_arrive_expect_tx(&full[i], stage_bytes);
      tma_load_2d(st, &tmW, &full[i], (kt0 + i) * kBK, m_tile * kBM, pol_w);
    }
    grid_dep_wait();
    for (int i = 0; i < pre; ++i) {
      tma_load_2d(smem + i * stage_bytes + kWTileBytes, &tmX, &full[i], (kt0 + i) * kBK, 0, pol_x);
      if (has_lo)
        tma_load_2d(smem + i * stage_bytes + kWTileBytes + x_bytes, &tmXlo, &full[i], (kt0 + i) * kBK, 0, pol_x);
    }
    for (int i = pre; i < nk; ++i) {
      const int s = i % stages;
      const uint32_t use = static_cast<uint32_t>(i / stages);
      if (!mbar_wait(&empty[s], (use & 1u) ^ 1u, err)) break;
      uint8_t* st = smem + s * stage_bytes;
      mbar_arrive_expect_tx(&full[s], stage_bytes);
      tma_load_2d(st, &tmW, &full[s], (kt0 + i) * kBK, m_tile * kBM, pol_w);
      tma_load_2d(st + kWTileBytes, &tmX, &full[s], (kt0 + i) * kBK, 0, pol_x);
      if (has_lo) tma_load_2d(st + kWTileBytes + x_bytes, &tmXlo, &full[s], (kt0 + i) * kBK, 0, pol_x);
    }
  } else if (warp == 1 && lane == 0) {
    // ---------------- MMA issuer
    const uint32_t idesc = idesc_bf16_f32(kBM, n_pad);
    bool ok = true;
    for (int i = 0; i < nk && ok; ++i) {
      const int s = i % stages;
      const uint32_t use = static_cast<uint32_t>(i / stages);
      if (!mbar_wait(&full[s], use & 1u, err)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t a_base = smem_u32(smem + s * stage_bytes);
      const uint32_t b_base = a_base + kWTileBytes;
#pragma unroll
      for (int kk = 0; kk < kBK / 16; ++kk) {
        const uint64_t a_desc = desc_sw128(a_base + kk * 32);
        umma_bf16(tmem, a_desc, desc_sw128(b_base + kk * 32), idesc, (i > 0 || kk > 0) ? 1u : 0u);
        if (has_lo) umma_bf16(tmem, a_desc, desc_sw128(b_base + x_bytes + kk * 32), idesc, 1u);
      }
      umma_commit(&empty[s]);
    }
    umma_commit(done);
  }
  __syncwarp();

  // ---------------- epilogue: TMEM -> registers -> fp32 partials
  const bool have = __all_sync(0xffffffffu, mbar_wait(done, 0, err));   // also reconverges the warp
  tc_fence_after();
  grid_dep_launch();
  grid_dep_wait();
  const int m = m_tile * kBM + warp * 32 + lane;
  if (have && nk > 0) {
    float* out = part + static_cast<size_t>(split) * n_valid * M;
    for (int c0 = 0; c0 < n_pad; c0 += 16) {
      float v[16];
      tmem_ld16(tmem + (static_cast<uint32_t>(warp * 32) << 16) + static_cast<uint32_t>(c0), v);
      if (m < M) {
#pragma unroll
        for (int j = 0; j < 16; ++j)
          if (c0 + j < n_valid) out[static_cast<size_t>(c0 + j) * M + m] = v[j];
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) tmem_dealloc(tmem, tmem_cols);
}

}  // namespace

GemmPlan plan_gemm(int M, int K, int n_pad, int num_sms, bool has_lo) {
  GemmPlan p;
  p.has_lo = has_lo;
  p.m_tiles = (M + kBM - 1) / kBM;
  p.k_tiles = (K + kBK - 1) / kBK;
  const uint32_t stage_bytes = kWTileBytes + static_cast<uint32_t>(n_pad) * kBK * 2 * (has_lo ? 2u : 1u);
  int stages = static_cast<int>((112u * 1024u) / stage_bytes);
  p.stages = stages < 2 ? 2 : (stages > 8 ? 8 : stages);
  p.smem_bytes = static_cast<size_t>(p.stages) * stage_bytes + 1024 /*align*/ + 256 /*barriers*/;
  const int target = 2 * num_sms;
  int s = target / p.m_tiles;
  if (s < 1) s = 1;
  if (s > p.k_tiles) s = p.k_tiles;
  p.kt_per_split = (p.k_tiles + s - 1) / s;
  p.splits = (p.k_tiles + p.kt_per_split - 1) / p.kt_per_split;
  uint32_t cols = 32;
  while (cols < static_cast<uint32_t>(n_pad)) cols <<= 1;
  p.tmem_cols = cols;
  return p;
}

cudaError_t gemm_configure() {
  return cudaFuncSetAttribute(gemm_wstream_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
}

cudaError_t launch_gemm(const GemmPlan& p, const CUtensorMap* tmW, const CUtensorMap* tmX, const CUtensorMap* tmXlo,
                        float* part, int M, int n_valid, int n_pad, int* err, cudaStream_t stream, bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.m_tiles, p.splits, 1);
  cfg.blockDim = dim3(128, 1, 1);
  cfg.dynamicSmemBytes = p.smem_bytes;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, gemm_wstream_kernel, *tmW, *tmX, p.has_lo ? *tmXlo : *tmX, p.has_lo ? 1 : 0, part,
                            M, n_valid, n_pad, p.k_tiles, p.kt_per_split, p.stages, p.tmem_cols, err);
}

}  // namespace kvprm
