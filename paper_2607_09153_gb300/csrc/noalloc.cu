// kvprm_attention_noalloc: the paged attention read-out for callers that must
// not allocate device memory -- for example a serving runtime that reserves
// all of its GPU memory up front and forbids allocations afterwards, or code
// that runs inside another framework's memory-managed region where a
// cudaMalloc would break the owner's accounting or stall on a device-wide
// synchronisation.  It needs no context: its scratch (the attention work list built
// on the host from the block table and lengths, the query split into bf16
// hi/lo parts, the split partials and an error word) lives in one file-scope device array, so every GPU that loads
// this library holds that array until the process exits.
//
// Set-up: the first call on a device (with that device current) looks up the
// array's device address with cudaGetSymbolAddress and configures the kernels;
// make that first call before any stream capture.  All calls share the array
// and it keeps the last call's contents, so calls that overlap on the GPU (on
// different streams, or from several host threads) race and corrupt each
// other's results; serialise them.
//
// Each call builds its attention schedule on the host and uploads it into the
// array with cudaMemcpyAsync from pageable host memory, so the call returns
// only once the driver has staged those bytes (the host waits for the copy
// engine).  For the same reason a call on a stream that is being captured is
// refused: a graph would keep the host address of a buffer that later calls
// overwrite, and the schedule of that one call.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstdint>
#include <cstring>
#include <mutex>

#include "../../include/kvprm.h"
#include "kernels.h"

namespace {

static __device__ __align__(256) unsigned char g_scratch[KVPRM_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;

struct DeviceState {
  bool ready = false;
  unsigned char* scratch = nullptr;
};
std::mutex g_mu;
DeviceState g_dev[kMaxDevices];
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

// Once per device, with that device current: the array's device address and
// the kernels' shared-memory limits.  Returns a KVPRM_* status.
int setup_current_device(unsigned char** scratch) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return KVPRM_ECUDA;
  std::lock_guard<std::mutex> lock(g_mu);
  DeviceState& s = g_dev[dev];
  if (!s.ready) {
    void* ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, g_scratch) != cudaSuccess || ptr == nullptr) return KVPRM_ECUDA;
    if (kvprm::attention_configure() != cudaSuccess) return KVPRM_ECUDA;
    if (!g_encode) {
      void* fn = nullptr;
      cudaDriverEntryPointQueryResult q;
      if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) !=
              cudaSuccess ||
          !fn || q != cudaDriverEntryPointSuccess)
        return KVPRM_ECUDA;
      g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    }
    s.scratch = static_cast<unsigned char*>(ptr);
    s.ready = true;
  }
  *scratch = s.scratch;
  return KVPRM_OK;
}

size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

struct Carve {
  size_t err, segs, cta, pages, cands, slots, base, nslots, qhi, qlo, ohi, olo, pml, po, total;
};

// Layout of the scratch array for one call: the error word, the attention
// schedule, the query's bf16 hi/lo parts, the
// output's hi/lo parts (the kernel always writes them) and the partial slots.
Carve carve(int n, int n_q, int n_kv, int hd, const kvprm::AttnWorkHost& w) {
  Carve c;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t at = off;
    off = align256(off + bytes);
    return at;
  };
  c.err = take(sizeof(int));
  c.segs = take(sizeof(kvprm::AttnSeg) * w.segs.size());
  c.cta = take(sizeof(int32_t) * w.cta_seg.size());
  c.pages = take(sizeof(int32_t) * w.pages.size());
  c.cands = take(sizeof(int32_t) * w.cands.size());
  c.slots = take(sizeof(int32_t) * w.slots.size());
  c.base = take(sizeof(int32_t) * w.slot_base.size());
  c.nslots = take(sizeof(int32_t) * w.nslots.size());
  const size_t qe = static_cast<size_t>(n) * n_q * hd;
  c.qhi = take(2 * qe);
  c.qlo = take(2 * qe);
  c.ohi = take(2 * qe);
  c.olo = take(2 * qe);
  const size_t group = static_cast<size_t>(n_q / n_kv);
  c.pml = take(sizeof(float) * static_cast<size_t>(w.n_slots) * group * 2);
  c.po = take(sizeof(float) * static_cast<size_t>(w.n_slots) * group * hd);
  c.total = off;
  return c;
}

}  // namespace

extern "C" int kvprm_attention_noalloc(const void* kv_layer, int64_t n_pages, const int32_t* block_table,
                                       int32_t max_blocks_per_seq, const int32_t* seq_lens, int32_t n_candidates,
                                       int32_t n_q_heads, int32_t n_kv_heads, int32_t head_dim, const float* q,
                                       const float* k_self, const float* v_self, float* out, void* stream) {
  const int n = n_candidates;
  if (n < 0 || n_q_heads < 1 || n_kv_heads < 1 || max_blocks_per_seq < 1 || n_pages < 0) return KVPRM_EINVAL;
  if (head_dim != 64 && head_dim != 128) return KVPRM_EUNSUPPORTED;
  if (n_q_heads % n_kv_heads || n_q_heads / n_kv_heads > 16) return KVPRM_EUNSUPPORTED;
  if (n == 0) return KVPRM_OK;
  if (!block_table || !seq_lens || !q || !k_self || !v_self || !out) return KVPRM_EINVAL;
  auto al16 = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; };
  if (!al16(q) || !al16(k_self) || !al16(v_self)) return KVPRM_EINVAL;
  // host-side validation of the tables, as in kvprm_attention
  int max_pages = 0;
  for (int b = 0; b < n; ++b) {
    const int L = seq_lens[b];
    if (L < 0) return KVPRM_EINVAL;
    if (static_cast<int64_t>(L) > static_cast<int64_t>(max_blocks_per_seq) * 16) return KVPRM_ECAPACITY;
    const int np = (L + 15) / 16;
    if (np > max_pages) max_pages = np;
    for (int j = 0; j < np; ++j) {
      const int32_t p = block_table[static_cast<int64_t>(b) * max_blocks_per_seq + j];
      if (p < 0 || p >= n_pages) return KVPRM_EINDEX;
    }
  }
  if (max_pages > 0 && (!kv_layer || !al16(kv_layer))) return KVPRM_EINVAL;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  {
    cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(st, &cap) != cudaSuccess) return KVPRM_ECUDA;
    if (cap != cudaStreamCaptureStatusNone) return KVPRM_EUNSUPPORTED;
  }

  unsigned char* scratch = nullptr;
  int rc = setup_current_device(&scratch);
  if (rc) return rc;

  kvprm::AttnShape as;
  as.n_q = n_q_heads;
  as.n_kv = n_kv_heads;
  as.hd = head_dim;
  as.group = n_q_heads / n_kv_heads;
  as.max_blocks = max_blocks_per_seq;
  int dev = 0, sms = 148;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return KVPRM_ECUDA;
  // the attention schedule, with shared-prefix runs if they fit the array,
  // else with private runs only
  thread_local kvprm::AttnWorkHost work;
  Carve cv;
  bool fits = false;
  for (int share = 1; share >= 0 && !fits; --share) {
    if (!kvprm::build_attn_work(block_table, seq_lens, n, max_blocks_per_seq, n_kv_heads, n_q_heads / n_kv_heads, sms,
                                SIZE_MAX, share != 0,
                                work))
      continue;
    cv = carve(n, n_q_heads, n_kv_heads, head_dim, work);
    fits = cv.total <= static_cast<size_t>(KVPRM_NOALLOC_SCRATCH_BYTES);
  }
  if (!fits) return KVPRM_ECAPACITY;

  // tensor map over this layer's pages (built on the host stack; no allocation)
  const void* pool = kv_layer;
  int64_t pages = n_pages;
  if (max_pages == 0) {   // nothing is read from the pool; any valid address serves the map
    pool = scratch;
    pages = 1;
  }
  if (2 * pages >= (static_cast<int64_t>(1) << 31)) return KVPRM_EUNSUPPORTED;
  as.layer_pages = pages;
  CUtensorMap tm;
  if (kvprm::encode_pool_map(g_encode, &tm, pool, pages, n_kv_heads, head_dim) != CUDA_SUCCESS) return KVPRM_ECUDA;

  int* err = reinterpret_cast<int*>(scratch + cv.err);
  kvprm::HiLo Q{reinterpret_cast<__nv_bfloat16*>(scratch + cv.qhi), reinterpret_cast<__nv_bfloat16*>(scratch + cv.qlo)};
  __nv_bfloat16* ohi = reinterpret_cast<__nv_bfloat16*>(scratch + cv.ohi);
  __nv_bfloat16* olo = reinterpret_cast<__nv_bfloat16*>(scratch + cv.olo);
  float* pml = reinterpret_cast<float*>(scratch + cv.pml);
  float* po = reinterpret_cast<float*>(scratch + cv.po);
  kvprm::AttnWork wk;
  wk.segs = reinterpret_cast<const kvprm::AttnSeg*>(scratch + cv.segs);
  wk.cta_seg = reinterpret_cast<const int32_t*>(scratch + cv.cta);
  wk.pages = reinterpret_cast<const int32_t*>(scratch + cv.pages);
  wk.cands = reinterpret_cast<const int32_t*>(scratch + cv.cands);
  wk.slots = reinterpret_cast<const int32_t*>(scratch + cv.slots);
  wk.slot_base = reinterpret_cast<const int32_t*>(scratch + cv.base);
  wk.nslots = reinterpret_cast<const int32_t*>(scratch + cv.nslots);
  wk.n_ctas = work.n_ctas;
  wk.tc_seg0 = work.tc_seg0;
  wk.n_tc = work.n_tc;   // 0: this entry point schedules shared pages on the persistent kernel only
  wk.tc_cta = nullptr;
  wk.n_tc_ctas = 0;
  wk.fuse_cs = 0;   // the persistent plan and a combine launch

  // the error word must start at zero; everything else is written before it is read
  if (cudaMemsetAsync(err, 0, sizeof(int), st) != cudaSuccess) return KVPRM_ECUDA;
  // pageable host sources: each copy is staged by the driver before it returns,
  // so the thread-local work list may be rebuilt by the next call
  auto up = [&](size_t off, const void* src, size_t bytes) {
    return bytes == 0 || cudaMemcpyAsync(scratch + off, src, bytes, cudaMemcpyHostToDevice, st) == cudaSuccess;
  };
  if (!up(cv.segs, work.segs.data(), sizeof(kvprm::AttnSeg) * work.segs.size()) ||
      !up(cv.cta, work.cta_seg.data(), sizeof(int32_t) * work.cta_seg.size()) ||
      !up(cv.pages, work.pages.data(), sizeof(int32_t) * work.pages.size()) ||
      !up(cv.cands, work.cands.data(), sizeof(int32_t) * work.cands.size()) ||
      !up(cv.slots, work.slots.data(), sizeof(int32_t) * work.slots.size()) ||
      !up(cv.base, work.slot_base.data(), sizeof(int32_t) * work.slot_base.size()) ||
      !up(cv.nslots, work.nslots.data(), sizeof(int32_t) * work.nslots.size()))
    return KVPRM_ECUDA;
  if (kvprm::launch_split_hilo(q, static_cast<int64_t>(n) * n_q_heads * head_dim, Q, st) != cudaSuccess)
    return KVPRM_ECUDA;
  const kvprm::AttnMerge mg{q, k_self, v_self, ohi, olo, out, nullptr};
  if (kvprm::launch_attention(as, wk, &tm, 0, Q.hi, Q.lo, po, pml, mg, err, st, false) != cudaSuccess)
    return KVPRM_ECUDA;
  if (kvprm::launch_attn_combine(as, wk, n, po, pml, mg, st, false) != cudaSuccess) return KVPRM_ECUDA;
  return KVPRM_OK;
}
