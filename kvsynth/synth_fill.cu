// kvsynth device generator: the device twin of synth.c (same SplitMix64
// streams, same quantile table, same element indexing), used to fill weights
// and the paged K/V pool directly in HBM.  Test infrastructure: it holds none
// of the scoring method's arithmetic and is not part of the scoring library.
#include <cstdint>
#include <cuda_runtime.h>

namespace {

constexpr uint64_t kGamma = 0x9E3779B97F4A7C15ULL;
constexpr uint64_t kKvTidBase = 0x4B560000ULL;

__host__ __device__ inline uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}
__host__ __device__ inline uint64_t stream_key(uint64_t seed, uint64_t tid) { return mix64(seed ^ (tid * kGamma)); }
__device__ inline uint64_t draw(uint64_t key, uint64_t n) { return mix64(key + (n + 1) * kGamma); }

__global__ void fill_kernel(uint16_t* __restrict__ out, int64_t n, uint64_t key, const uint16_t* __restrict__ table) {
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
    out[i] = __ldg(table + (draw(key, (uint64_t)i) >> 48));
}

// One thread per element of one layer of the pool [n_pages][2][n_kv][P][hd].
__global__ void pool_kernel(uint16_t* __restrict__ pool, int64_t n_pages, const int32_t* __restrict__ pseg,
                            const int32_t* __restrict__ poff, int P, int n_kv, int hd, uint64_t kk, uint64_t kvk,
                            const uint16_t* __restrict__ table) {
  const int64_t total = n_pages * 2 * n_kv * (int64_t)P * hd;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
    int64_t row = e / hd;
    int d = (int)(e - row * hd);
    int s = (int)(row % P);
    int64_t r2 = row / P;
    int h = (int)(r2 % n_kv);
    int64_t r3 = r2 / n_kv;
    int w = (int)(r3 & 1);
    int64_t pg = r3 >> 1;
    int32_t seg = pseg[pg * P + s], off = poff[pg * P + s];
    uint16_t v = 0;
    if (seg >= 0) {
      uint64_t tok = ((uint64_t)(uint32_t)seg << 24) | (uint64_t)(uint32_t)off;
      uint64_t n = (tok * (uint64_t)n_kv + (uint64_t)h) * (uint64_t)hd + (uint64_t)d;
      v = __ldg(table + (draw(w ? kvk : kk, n) >> 48));
    }
    pool[e] = v;
  }
}

int grid_for(int64_t n) {
  int64_t g = (n + 255) / 256;
  if (g > 152 * 32) g = 152 * 32;
  if (g < 1) g = 1;
  return (int)g;
}

}  // namespace

extern "C" {

int synth_dev_fill(uint16_t* out, int64_t n, uint64_t seed, uint64_t tid, const uint16_t* table_dev, void* stream) {
  if (n <= 0) return 0;
  fill_kernel<<<grid_for(n), 256, 0, (cudaStream_t)stream>>>(out, n, stream_key(seed, tid), table_dev);
  return (int)cudaGetLastError();
}

int synth_dev_kv_pool_layer(uint16_t* pool_layer, int64_t n_pages, const int32_t* page_seg, const int32_t* page_off,
                            int page_size, int n_kv, int hd, int layer, uint64_t seed, const uint16_t* table_dev,
                            void* stream) {
  int64_t total = n_pages * 2 * n_kv * (int64_t)page_size * hd;
  if (total <= 0) return 0;
  uint64_t kk = stream_key(seed, kKvTidBase + 2ULL * (uint64_t)layer);
  uint64_t kvk = stream_key(seed, kKvTidBase + 2ULL * (uint64_t)layer + 1ULL);
  pool_kernel<<<grid_for(total), 256, 0, (cudaStream_t)stream>>>(pool_layer, n_pages, page_seg, page_off, page_size,
                                                                 n_kv, hd, kk, kvk, table_dev);
  return (int)cudaGetLastError();
}

}  // extern "C"
