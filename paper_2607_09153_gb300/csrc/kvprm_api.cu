// C ABI of the KV-PRM scoring library (declared in include/kvprm.h): context
// creation, host-side validation, block-table upload, tensor maps, the
// per-call launch sequence of the verify-token forward (Sec. 4.1 Eq. score),
// and its replay as a CUDA graph.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <string>
#include <vector>

#include "../../include/kvprm.h"
#include "kernels.h"

using kvprm::AttnShape;
using kvprm::GemmPlan;
using kvprm::ModelDims;
typedef __nv_bfloat16 bf16;

namespace {

struct CallPlan {
  int n = 0, n_pad = 0, max_pages = 0;
  GemmPlan g_qkv, g_o, g_gu, g_down;
  // scorer adapter: the A x launches, and each projection's K tiles of W (the rest are B's)
  GemmPlan l_qkv, l_o, l_gu, l_down;
  int k_qkv = 0, k_o = 0, k_gu = 0, k_down = 0;
  int attn_ctas = 0;   // grid of the attention (see build_attn_work)
};

struct GraphKey {
  int n = -1, n_pad = -1, attn_ctas = -1, tc_ctas = -1, n_tc = -1, debug = -1, profile = -1, pdl = -1, trace = -1;
  int fuse_cs = -1;
  int layer_waits = -1;
  int lora_rank = -1;
  int depth = -1;
  const void* pool = nullptr;
  int64_t n_pages = -1;
  bool operator==(const GraphKey& o) const {
    return n == o.n && n_pad == o.n_pad && attn_ctas == o.attn_ctas && tc_ctas == o.tc_ctas && n_tc == o.n_tc &&
           fuse_cs == o.fuse_cs && layer_waits == o.layer_waits && lora_rank == o.lora_rank && depth == o.depth &&
           debug == o.debug && profile == o.profile && pdl == o.pdl && trace == o.trace && pool == o.pool &&
           n_pages == o.n_pages;
  }
};

struct ProfMark {
  int cls;
  cudaEvent_t a, b;
};

// Forward intermediates a backward pass needs (kvprm_score_grad), per layer l at l * (max_candidates
// rows) of each array: the rotated q and the self k / v as the attention consumed them, the
// attention output o and its softmax log-normaliser, the residual stream after the attention block
// and after the layer, and the gate / up pre-activations.
struct FwdSaves {
  float *q = nullptr, *k = nullptr, *v = nullptr, *o = nullptr, *lse = nullptr;
  float *hmid = nullptr, *hout = nullptr, *gu = nullptr;
};

// State of the KV Steering backward pass, built by the first kvprm_score_grad call on a context.
struct GradState {
  bool ready = false;
  // library-owned transposed weights W^T [in][out] and their tensor maps (the backward's products
  // dx = W^T dy run on the forward's GEMM with these as the streamed operand)
  std::vector<__nv_bfloat16*> wt;   // per layer: qkv, o, gate_up, down
  std::vector<CUtensorMap> tm_qkv, tm_o, tm_gu, tm_down;
  FwdSaves sv;
  float *dh = nullptr, *tmp = nullptr, *D = nullptr, *dq = nullptr, *dks = nullptr, *dvs = nullptr;
  __nv_bfloat16 *ghi = nullptr, *glo = nullptr;   // a gradient as the next product's bf16 hi/lo input
  int tm_npad = -1;
  CUtensorMap tm_d_hi{}, tm_d_lo{}, tm_gu_hi{}, tm_gu_lo{}, tm_qkv_hi{}, tm_qkv_lo{};
  // per call: work units of the attention backward, shared-page flags and page lists
  int4* units = nullptr;
  size_t units_cap = 0;
  uint8_t* shared = nullptr;
  size_t shared_cap = 0;
  int32_t* lists = nullptr;   // [shared pages][all referenced pages]
  size_t lists_cap = 0;
  int n_shared = 0, n_ref = 0;   // of the last call
  float* grad_own = nullptr;   // kvprm_steer's gradient buffer
  size_t grad_own_bytes = 0;
  // the forward with saves and the backward of a call, captured once and replayed while every launch
  // parameter and buffer they bake in is unchanged (the key)
  cudaGraphExec_t gexec = nullptr;
  std::vector<int64_t> gkey;
  std::vector<ProfMark> marks;   // unused: profiled calls run eagerly
};

}  // namespace

struct kvprm_ctx {
  kvprm_config cfg{};
  int device = 0, num_sms = 148;
  ModelDims md{};
  AttnShape as{};
  PFN_cuTensorMapEncodeTiled_v12000 encode = nullptr;
  // borrowed weights
  const bf16 *embed = nullptr, *final_norm = nullptr, *w_plus = nullptr, *w_minus = nullptr;
  std::vector<const bf16*> attn_norm, mlp_norm;
  std::vector<const bf16*> q_norm, k_norm;   // per-head q/k RMSNorm gains (cfg.qk_norm)
  std::vector<CUtensorMap> tm_qkv, tm_o, tm_gu, tm_down;
  std::vector<const void*> w_qkv_src, w_o_src, w_gu_src, w_down_src;   // the borrowed matrices
  // depth-k readout (kvprm_set_readout_depth): verify tokens per candidate; candidate b of a call is
  // rows b depth .. b depth + depth - 1 of the batch (expanded tables below)
  int depth = 1;
  std::vector<int32_t> row_bt, row_sl;
  // scorer adapter (kvprm_set_lora; rank 0: the merged weights alone): per projection (QKV, O,
  // gate/up, down) and layer the maps of A and B, and t = scale (A x) as hi/lo [npad_max][rank]
  int lora_rank = 0;
  float lora_scale = 0.f;
  std::vector<CUtensorMap> tm_la[4], tm_lb[4];
  bf16 *thi = nullptr, *tlo = nullptr;
  size_t t_cap = 0;
  int tm_t_npad = -1;
  CUtensorMap tm_thi{}, tm_tlo{};
  // workspace
  int npad_max = 16;
  float* h = nullptr;
  bf16 *xhi = nullptr, *xlo = nullptr, *ohi = nullptr, *olo = nullptr, *ahi = nullptr, *alo = nullptr;
  float* sumsq = nullptr;   // [ceil(d / 128)][Bmax] per-tile sums of squares of h
  int d_tiles = 0;
  float *q = nullptr, *kself = nullptr, *vself = nullptr;
  bf16 *qhi = nullptr, *qlo = nullptr;
  float *apart_o = nullptr, *apart_ml = nullptr;   // [slot_cap][group][hd], [slot_cap][group][2]
  size_t slot_cap = 0;
  float2* rope = nullptr;
  int32_t* tables_d = nullptr;   // [Bmax] seq_lens, [Bmax][max_blocks] block table, then the attention work
  // attention work list: host plan of the current call and fixed offsets (ints) in tables_d / staging
  kvprm::AttnWorkHost work_host;
  size_t off_segs = 0, off_cta = 0, off_pages = 0, off_cands = 0, off_slots = 0, off_base = 0, off_nslots = 0,
         off_tc_cta = 0;
  size_t tables_ints = 0;
  size_t cap_segs = 0, cap_pages = 0, cap_cands = 0;
  int share_mode = 3;   // sharing of pages referenced by several candidates (build_attn_work)
  bool fuse_combine = true;   // the combine inside the attention launch where the call qualifies
  float* rewards_d = nullptr;
  int* err_d = nullptr;
  float* dbg = nullptr;
  float *dbg_q = nullptr, *dbg_k = nullptr, *dbg_v = nullptr;
  float* dbg_h = nullptr;
  unsigned long long* tc_prof = nullptr;   // tensor-core attention wait profile (debug flag 32)
  bf16* dummy_pool = nullptr;
  int debug_flags = 0;
  int last_n = 0;
  // pinned staging
  int32_t* staging = nullptr;
  float* h_rewards = nullptr;
  int* h_err = nullptr;
  cudaEvent_t staging_ev = nullptr;
  bool staging_pending = false;
  // activation tensor maps (depend on the padded batch)
  int tm_x_npad = -1;
  CUtensorMap tm_xhi{}, tm_xlo{}, tm_ohi{}, tm_olo{}, tm_ahi{}, tm_alo{};
  // pool tensor map (depends on the caller's pool)
  const void* pool_ptr = nullptr;
  int64_t pool_pages = -1;
  int64_t pool_units = -1;
  CUtensorMap tm_pool{}, tm_pool_tc{};
  // library-owned device pool for kvprm_score_host
  void* dev_pool = nullptr;
  size_t dev_pool_bytes = 0;
  // graph replay
  cudaStream_t cap_stream = nullptr;
  // the tensor-core attention's stream when it runs beside the private pages' launch
  cudaStream_t side_stream = nullptr;
  cudaEvent_t ev_fork = nullptr, ev_join = nullptr;
  // kvprm_score_host: the cache is copied layer by layer on one copy stream, one event per layer;
  // while layer_waits is set, the forward being enqueued waits for layer l's event before layer l's
  // attention, so scoring overlaps the copy of the later layers
  cudaStream_t copy_stream = nullptr;
  std::vector<cudaEvent_t> layer_ready;
  cudaEvent_t pool_free = nullptr;
  bool layer_waits = false;
  const void* host_pool = nullptr;   // source of those copies, set for the duration of the call
  size_t host_pool_bytes = 0;

  bool use_graph = true, use_pdl = true;
  GraphKey gkey;
  cudaGraphExec_t gexec = nullptr;
  std::vector<ProfMark> graph_marks;
  // device timeline trace of the last call: [slot][2] (see trace_begin / trace_end)
  bool trace = false;
  unsigned long long* trace_d = nullptr;
  int trace_cap = 0, trace_n = 0;
  std::vector<int> trace_cls;
  // profiling
  bool profile = false;
  std::vector<ProfMark> live_marks;   // marks recorded in the current (non-graph) capture
  int64_t prof_launches[KVPRM_PROF_N] = {};
  double prof_ms[KVPRM_PROF_N] = {};
  std::string last_error;
  cudaStream_t last_stream = nullptr;
  // failure-detection hooks: a scoring call reports an injected CUDA failure instead of launching
  // (kvprm_debug_inject_error); a flag that nothing sets, for the bounded-wait probe
  int inject_fail = 0;
  int* probe_flag = nullptr;
  GradState grad;
  bool grad_cuda_cores = false;   // KVPRM_GRAD_CUDA_CORES=1: the attention backward on the CUDA cores
};

namespace {

int fail(kvprm_ctx* c, int code, const char* fmt, ...) __attribute__((format(printf, 3, 4)));
int fail(kvprm_ctx* c, int code, const char* fmt, ...) {
  if (c) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof(buf), fmt, ap);
    va_end(ap);
    c->last_error = buf;
  }
  return code;
}

int cuda_fail(kvprm_ctx* c, cudaError_t e, const char* what) {
  return fail(c, KVPRM_ECUDA, "%s: %s (%s)", what, cudaGetErrorName(e), cudaGetErrorString(e));
}

#define CK(call, what)                                     \
  do {                                                     \
    cudaError_t e_ = (call);                               \
    if (e_ != cudaSuccess) return cuda_fail(ctx, e_, what); \
  } while (0)

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

int make_map(kvprm_ctx* ctx, CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer, uint32_t box_inner,
             uint32_t box_outer, const char* what) {
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {inner * 2};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = ctx->encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                           CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                           CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(ctx, KVPRM_ECUDA, "cuTensorMapEncodeTiled(%s) failed with %d", what, (int)r);
  return KVPRM_OK;
}

// Device and pinned-host bytes the library may still allocate, process-wide (-1: no limit); lowered
// by every allocation while set (kvprm_debug_set_alloc_limit, a failure-detection test hook).
std::atomic<long long> g_alloc_budget{-1};

bool take_budget(size_t bytes) {
  long long cur = g_alloc_budget.load();
  while (cur >= 0) {
    if (static_cast<long long>(bytes) > cur) return false;
    if (g_alloc_budget.compare_exchange_weak(cur, cur - static_cast<long long>(bytes))) return true;
  }
  return true;
}

template <typename T>
int dalloc(kvprm_ctx* ctx, T** p, size_t count, const char* what) {
  if (!take_budget(count * sizeof(T))) {
    *p = nullptr;
    return fail(ctx, KVPRM_ENOMEM, "allocation of %s (%zu bytes) exceeds the allocation budget", what,
                count * sizeof(T));
  }
  cudaError_t e = cudaMalloc(reinterpret_cast<void**>(p), count * sizeof(T) > 0 ? count * sizeof(T) : 16);
  if (e != cudaSuccess) {
    *p = nullptr;
    cudaGetLastError();
    return fail(ctx, KVPRM_ENOMEM, "cudaMalloc(%s, %zu bytes): %s", what, count * sizeof(T), cudaGetErrorString(e));
  }
  e = cudaMemset(*p, 0, count * sizeof(T) > 0 ? count * sizeof(T) : 16);
  if (e != cudaSuccess) return cuda_fail(ctx, e, "cudaMemset");
  return KVPRM_OK;
}

void free_ctx(kvprm_ctx* c) {
  if (!c) return;
  cudaFree(c->h);
  cudaFree(c->xhi);
  cudaFree(c->xlo);
  cudaFree(c->ohi);
  cudaFree(c->olo);
  cudaFree(c->ahi);
  cudaFree(c->alo);
  cudaFree(c->thi);
  cudaFree(c->tlo);
  cudaFree(c->qhi);
  cudaFree(c->qlo);
  cudaFree(c->sumsq);
  cudaFree(c->trace_d);
  cudaFree(c->q);
  cudaFree(c->kself);
  cudaFree(c->vself);
  cudaFree(c->apart_o);
  cudaFree(c->apart_ml);
  cudaFree(c->rope);
  cudaFree(c->tables_d);
  cudaFree(c->rewards_d);
  cudaFree(c->err_d);
  cudaFree(c->dbg);
  cudaFree(c->dbg_q);
  cudaFree(c->dbg_k);
  cudaFree(c->dbg_v);
  cudaFree(c->dbg_h);
  cudaFree(c->tc_prof);
  cudaFree(c->dummy_pool);
  cudaFree(c->dev_pool);
  cudaFree(c->probe_flag);
  {
    GradState& g = c->grad;
    for (auto* p : g.wt) cudaFree(p);
    cudaFree(g.sv.q);
    cudaFree(g.dh);
    cudaFree(g.ghi);
    cudaFree(g.glo);
    cudaFree(g.units);
    cudaFree(g.shared);
    cudaFree(g.lists);
    cudaFree(g.grad_own);
    if (g.gexec) cudaGraphExecDestroy(g.gexec);
  }
  if (c->staging) cudaFreeHost(c->staging);
  if (c->h_rewards) cudaFreeHost(c->h_rewards);
  if (c->h_err) cudaFreeHost(c->h_err);
  if (c->staging_ev) cudaEventDestroy(c->staging_ev);
  if (c->gexec) cudaGraphExecDestroy(c->gexec);
  for (auto& m : c->graph_marks) {
    if (m.a) cudaEventDestroy(m.a);
    if (m.b) cudaEventDestroy(m.b);
  }
  for (auto& m : c->live_marks) {
    cudaEventDestroy(m.a);
    cudaEventDestroy(m.b);
  }
  if (c->cap_stream) cudaStreamDestroy(c->cap_stream);
  if (c->side_stream) cudaStreamDestroy(c->side_stream);
  if (c->ev_fork) cudaEventDestroy(c->ev_fork);
  if (c->ev_join) cudaEventDestroy(c->ev_join);
  if (c->copy_stream) cudaStreamDestroy(c->copy_stream);
  for (cudaEvent_t ev : c->layer_ready)
    if (ev) cudaEventDestroy(ev);
  if (c->pool_free) cudaEventDestroy(c->pool_free);

  delete c;
}

// ---------------------------------------------------------------- per-call checks and plan
int validate_tables(kvprm_ctx* ctx, int64_t n_pages, const int32_t* bt, const int32_t* sl, int32_t n, int* max_pages) {
  if (n < 0) return fail(ctx, KVPRM_EINVAL, "n_candidates = %d is negative", n);
  if (n > ctx->cfg.max_candidates)
    return fail(ctx, KVPRM_ECAPACITY, "n_candidates = %d exceeds max_candidates = %d", n, ctx->cfg.max_candidates);
  if (n > 0 && (!bt || !sl)) return fail(ctx, KVPRM_EINVAL, "block_table and seq_lens must not be NULL");
  const int mb = ctx->cfg.max_blocks_per_seq;
  int mp = 0;
  for (int b = 0; b < n; ++b) {
    const int L = sl[b];
    if (L < 0) return fail(ctx, KVPRM_EINVAL, "seq_lens[%d] = %d is negative", b, L);
    if (static_cast<int64_t>(L) > static_cast<int64_t>(mb) * 16)
      return fail(ctx, KVPRM_ECAPACITY, "seq_lens[%d] = %d exceeds 16 * max_blocks_per_seq = %lld", b, L,
                  static_cast<long long>(mb) * 16);
    const int np = (L + 15) / 16;
    if (np > mp) mp = np;
    for (int j = 0; j < np; ++j) {
      const int32_t p = bt[static_cast<int64_t>(b) * mb + j];
      if (p < 0 || p >= n_pages)
        return fail(ctx, KVPRM_EINDEX, "block_table[%d][%d] = %d is outside [0, %lld)", b, j, p,
                    static_cast<long long>(n_pages));
    }
  }
  *max_pages = mp;
  return KVPRM_OK;
}

// Plan the attention work of this call on the host (build_attn_work); a
// sharing plan that does not fit the context's work arrays falls back to
// private runs, which always fit.
int plan_work(kvprm_ctx* ctx, const int32_t* bt, const int32_t* sl, int32_t n, bool allow_fused) {
  kvprm::AttnWorkHost& w = ctx->work_host;
  const int mb = ctx->cfg.max_blocks_per_seq, nkv = ctx->cfg.n_kv_heads;
  auto fits = [&]() {
    return w.segs.size() <= ctx->cap_segs && w.pages.size() <= ctx->cap_pages && w.cands.size() <= ctx->cap_cands &&
           w.slots.size() <= ctx->slot_cap && static_cast<size_t>(w.n_ctas) <= static_cast<size_t>(ctx->num_sms) &&
           static_cast<size_t>(w.n_tc_ctas) <= static_cast<size_t>(ctx->num_sms);
  };
  if (ctx->fuse_combine && allow_fused &&
      kvprm::build_attn_work_fused(bt, sl, n, mb, nkv, ctx->md.n_q / nkv, ctx->num_sms, ctx->slot_cap, w) && fits())
    return KVPRM_OK;
  bool ok = kvprm::build_attn_work(bt, sl, n, mb, nkv, ctx->md.n_q / nkv, ctx->num_sms, ctx->slot_cap, ctx->share_mode, w);
  if (ok && !fits() && ctx->share_mode)
    ok = kvprm::build_attn_work(bt, sl, n, mb, nkv, ctx->md.n_q / nkv, ctx->num_sms, ctx->slot_cap, 0, w);
  if (!ok || !fits())
    return fail(ctx, KVPRM_ECAPACITY, "attention work list exceeds the context's capacity");
  return KVPRM_OK;
}

// Copy the tables and the planned work into pinned staging and then to the device.
int upload_tables(kvprm_ctx* ctx, const int32_t* bt, const int32_t* sl, int32_t n, cudaStream_t st) {
  const int Bmax = ctx->cfg.max_candidates, mb = ctx->cfg.max_blocks_per_seq;
  if (ctx->staging_pending) {
    CK(cudaEventSynchronize(ctx->staging_ev), "cudaEventSynchronize(staging)");
    ctx->staging_pending = false;
  }
  const kvprm::AttnWorkHost& w = ctx->work_host;
  int32_t* S = ctx->staging;
  constexpr size_t kSegInts = sizeof(kvprm::AttnSeg) / sizeof(int32_t);
  std::memcpy(S, sl, sizeof(int32_t) * n);
  std::memcpy(S + Bmax, bt, sizeof(int32_t) * static_cast<size_t>(n) * mb);
  struct Part {
    size_t off;
    const void* src;
    size_t ints;
  } parts[] = {
      {ctx->off_segs, w.segs.data(), w.segs.size() * kSegInts},
      {ctx->off_cta, w.cta_seg.data(), w.cta_seg.size()},
      {ctx->off_pages, w.pages.data(), w.pages.size()},
      {ctx->off_cands, w.cands.data(), w.cands.size()},
      {ctx->off_slots, w.slots.data(), w.slots.size()},
      {ctx->off_base, w.slot_base.data(), w.slot_base.size()},
      {ctx->off_nslots, w.nslots.data(), w.nslots.size()},
      {ctx->off_tc_cta, w.tc_cta.data(), w.tc_cta.size()},
  };
  for (const Part& p : parts)
    if (p.ints) std::memcpy(S + p.off, p.src, sizeof(int32_t) * p.ints);
  auto up = [&](size_t off, size_t ints) -> cudaError_t {
    if (ints == 0) return cudaSuccess;
    return cudaMemcpyAsync(ctx->tables_d + off, S + off, ints * sizeof(int32_t), cudaMemcpyHostToDevice, st);
  };
  CK(up(0, static_cast<size_t>(Bmax) + static_cast<size_t>(n) * mb), "cudaMemcpyAsync(tables)");
  for (const Part& p : parts) CK(up(p.off, p.ints), "cudaMemcpyAsync(attention work)");
  CK(cudaEventRecord(ctx->staging_ev, st), "cudaEventRecord(staging)");
  ctx->staging_pending = true;
  return KVPRM_OK;
}

// Stale-maximum margin of the tensor-core attention (debug flag 16: rescale on
// every new maximum, which exercises the rescale path).
float tc_margin(const kvprm_ctx* ctx) { return (ctx->debug_flags & 16) ? 0.f : 8.f; }

kvprm::AttnWork device_work(kvprm_ctx* ctx) {
  kvprm::AttnWork wk;
  wk.segs = reinterpret_cast<const kvprm::AttnSeg*>(ctx->tables_d + ctx->off_segs);
  wk.cta_seg = ctx->tables_d + ctx->off_cta;
  wk.pages = ctx->tables_d + ctx->off_pages;
  wk.cands = ctx->tables_d + ctx->off_cands;
  wk.slots = ctx->tables_d + ctx->off_slots;
  wk.slot_base = ctx->tables_d + ctx->off_base;
  wk.nslots = ctx->tables_d + ctx->off_nslots;
  wk.n_ctas = ctx->work_host.n_ctas;
  wk.tc_seg0 = ctx->work_host.tc_seg0;
  wk.n_tc = ctx->work_host.n_tc;
  wk.tc_cta = ctx->tables_d + ctx->off_tc_cta;
  wk.n_tc_ctas = ctx->work_host.n_tc_ctas;
  wk.fuse_cs = ctx->work_host.fuse_cs;
  return wk;
}

int ensure_pool_map(kvprm_ctx* ctx, const void* pool, int64_t n_pages, int layers) {
  const int64_t units = static_cast<int64_t>(layers) * n_pages;   // (layer, page) pairs
  if (ctx->pool_ptr == pool && ctx->pool_pages == n_pages && ctx->pool_units == units) return KVPRM_OK;
  if (2 * units >= (static_cast<int64_t>(1) << 31))
    return fail(ctx, KVPRM_EUNSUPPORTED, "pool of %lld layer pages exceeds the 2^30 tensor-map coordinate limit",
                static_cast<long long>(units));
  CUresult r = kvprm::encode_pool_map(ctx->encode, &ctx->tm_pool, pool, units, ctx->cfg.n_kv_heads,
                                      ctx->cfg.head_dim);
  if (r != CUDA_SUCCESS) return fail(ctx, KVPRM_ECUDA, "cuTensorMapEncodeTiled(kv pool) failed with %d", (int)r);
  r = kvprm::encode_pool_map_tc(ctx->encode, &ctx->tm_pool_tc, pool, units, ctx->cfg.n_kv_heads, ctx->cfg.head_dim);
  if (r != CUDA_SUCCESS) return fail(ctx, KVPRM_ECUDA, "cuTensorMapEncodeTiled(kv pool, 2 KB box) failed with %d", (int)r);
  ctx->pool_ptr = pool;
  ctx->pool_pages = n_pages;
  ctx->pool_units = units;
  return KVPRM_OK;
}

int ensure_x_maps(kvprm_ctx* ctx, int n_pad) {
  if (ctx->tm_x_npad == n_pad) return KVPRM_OK;
  int rc;
  const uint64_t d = ctx->md.d, dq = static_cast<uint64_t>(ctx->md.n_q) * ctx->md.hd, ff = ctx->md.ff;
  if ((rc = make_map(ctx, &ctx->tm_xhi, ctx->xhi, d, n_pad, 64, n_pad, "x_hi"))) return rc;
  if ((rc = make_map(ctx, &ctx->tm_xlo, ctx->xlo, d, n_pad, 64, n_pad, "x_lo"))) return rc;
  if ((rc = make_map(ctx, &ctx->tm_ohi, ctx->ohi, dq, n_pad, 64, n_pad, "o_hi"))) return rc;
  if ((rc = make_map(ctx, &ctx->tm_olo, ctx->olo, dq, n_pad, 64, n_pad, "o_lo"))) return rc;
  if ((rc = make_map(ctx, &ctx->tm_ahi, ctx->ahi, ff, n_pad, 64, n_pad, "a_hi"))) return rc;
  if ((rc = make_map(ctx, &ctx->tm_alo, ctx->alo, ff, n_pad, 64, n_pad, "a_lo"))) return rc;
  ctx->tm_x_npad = n_pad;
  return KVPRM_OK;
}

// the adapter's t = scale (A x) buffer as the K-extension operand of a batch padded to n_pad
int ensure_t_maps(kvprm_ctx* ctx, int n_pad) {
  if (ctx->lora_rank == 0 || ctx->tm_t_npad == n_pad) return KVPRM_OK;
  int rc;
  const uint64_t r = static_cast<uint64_t>(ctx->lora_rank);
  if ((rc = make_map(ctx, &ctx->tm_thi, ctx->thi, r, n_pad, 64, n_pad, "t_hi"))) return rc;
  if ((rc = make_map(ctx, &ctx->tm_tlo, ctx->tlo, r, n_pad, 64, n_pad, "t_lo"))) return rc;
  ctx->tm_t_npad = n_pad;
  return KVPRM_OK;
}

CallPlan make_plan(kvprm_ctx* ctx, int n, int max_pages) {
  CallPlan p;
  p.n = n;
  p.n_pad = (n + 15) / 16 * 16;
  p.max_pages = max_pages;
  const ModelDims& m = ctx->md;
  // with an adapter each projection's K loop runs on over B's r columns (W's last tile zero-padded)
  const int r = ctx->lora_rank;
  auto kt = [](int K) { return (K + 63) / 64; };
  auto keff = [&](int K) { return r ? 64 * kt(K) + r : K; };
  p.g_qkv = kvprm::plan_gemm(m.qkv_rows, keff(m.d), p.n_pad, ctx->num_sms, true, false);
  p.g_o = kvprm::plan_gemm(m.d, keff(m.n_q * m.hd), p.n_pad, ctx->num_sms, true, false);
  p.g_gu = kvprm::plan_gemm(m.ff, keff(m.d), p.n_pad, ctx->num_sms, true, true);
  p.g_down = kvprm::plan_gemm(m.d, keff(m.ff), p.n_pad, ctx->num_sms, true, false);
  if (r) {
    p.l_qkv = kvprm::plan_gemm(r, m.d, p.n_pad, ctx->num_sms, true, false);
    p.l_o = kvprm::plan_gemm(r, m.n_q * m.hd, p.n_pad, ctx->num_sms, true, false);
    p.l_gu = kvprm::plan_gemm(r, m.d, p.n_pad, ctx->num_sms, true, false);
    p.l_down = kvprm::plan_gemm(r, m.ff, p.n_pad, ctx->num_sms, true, false);
    p.k_qkv = kt(m.d);
    p.k_o = kt(m.n_q * m.hd);
    p.k_gu = kt(m.d);
    p.k_down = kt(m.ff);
  }
  p.attn_ctas = ctx->work_host.n_ctas;
  return p;
}

// ---------------------------------------------------------------- launch sequence
struct Enq {
  kvprm_ctx* ctx;
  cudaStream_t st;
  bool pdl;
  bool prof;
  std::vector<ProfMark>* marks;
  bool capturing = false;
  cudaError_t rec(cudaEvent_t ev) {
    return capturing ? cudaEventRecordWithFlags(ev, st, cudaEventRecordExternal) : cudaEventRecord(ev, st);
  }
  int begin(int cls, cudaEvent_t* ev_b) {
    if (!prof) return KVPRM_OK;
    ProfMark m{cls, nullptr, nullptr};
    CK(cudaEventCreate(&m.a), "cudaEventCreate");
    CK(cudaEventCreate(&m.b), "cudaEventCreate");
    CK(rec(m.a), "cudaEventRecord");
    marks->push_back(m);
    *ev_b = m.b;
    return KVPRM_OK;
  }
  // count a launch whose time is part of an enclosing mark (no events of its own)
  void count(int cls) {
    if (prof) marks->push_back(ProfMark{cls, nullptr, nullptr});
  }
  unsigned long long* trace_slot(int cls) {
    if (!ctx->trace || ctx->trace_n >= ctx->trace_cap) return nullptr;
    ctx->trace_cls.push_back(cls);
    return ctx->trace_d + kvprm::kTraceStride * static_cast<size_t>(ctx->trace_n++);
  }
  int end(cudaEvent_t ev_b) {
    if (!prof) return KVPRM_OK;
    CK(rec(ev_b), "cudaEventRecord");
    return KVPRM_OK;
  }
};

#define LAUNCH(cls, expr, what)                    \
  do {                                             \
    unsigned long long* TS = E.trace_slot(cls);    \
    (void)TS;                                      \
    cudaEvent_t evb_ = nullptr;                    \
    int rc_ = E.begin(cls, &evb_);                 \
    if (rc_) return rc_;                           \
    cudaError_t e_ = (expr);                       \
    if (e_ != cudaSuccess) return cuda_fail(ctx, e_, what); \
    rc_ = E.end(evb_);                             \
    if (rc_) return rc_;                           \
  } while (0)

// The attention step of one layer: shared pages on the tensor cores (when the
// plan has any) and the private pages, into partial slots.  When the plan gave
// the two launches disjoint SMs (share mode 3) the tensor-core launch runs on
// the side stream, forked here and joined before returning, so both read
// their pages at once; a profiled call then times the pair as one step.
int enqueue_attention(kvprm_ctx* ctx, Enq& E, const kvprm::AttnShape& as, const kvprm::AttnWork& wk, int layer,
                      const kvprm::HiLo& Q, const kvprm::AttnMerge& mg, bool pdl) {
  cudaStream_t st = E.st;
  unsigned long long* tc_prof = (ctx->debug_flags & 32) ? ctx->tc_prof : nullptr;
  if (wk.n_tc > 0 && ctx->work_host.tc_concurrent) {
    cudaEvent_t evb = nullptr;
    int rc = E.begin(KVPRM_PROF_ATTN, &evb);
    if (rc) return rc;
    CK(cudaEventRecord(ctx->ev_fork, st), "cudaEventRecord(fork)");
    CK(cudaStreamWaitEvent(ctx->side_stream, ctx->ev_fork, 0), "cudaStreamWaitEvent(fork)");
    {
      unsigned long long* TS = E.trace_slot(KVPRM_PROF_ATTN_TC);
      cudaError_t e = kvprm::launch_attention_tc(as, wk, &ctx->tm_pool_tc, layer, Q.hi, Q.lo, ctx->apart_o,
                                                 ctx->apart_ml, tc_margin(ctx), ctx->err_d, ctx->side_stream, false,
                                                 TS, tc_prof);
      if (e != cudaSuccess) return cuda_fail(ctx, e, "attention_tc");
      E.count(KVPRM_PROF_ATTN_TC);
    }
    CK(cudaEventRecord(ctx->ev_join, ctx->side_stream), "cudaEventRecord(join)");
    {
      unsigned long long* TS = E.trace_slot(KVPRM_PROF_ATTN);
      cudaError_t e = kvprm::launch_attention(as, wk, &ctx->tm_pool, layer, Q.hi, Q.lo, ctx->apart_o, ctx->apart_ml,
                                              mg, ctx->err_d, st, pdl, TS);
      if (e != cudaSuccess) return cuda_fail(ctx, e, "attention");
    }
    CK(cudaStreamWaitEvent(st, ctx->ev_join, 0), "cudaStreamWaitEvent(join)");
    return E.end(evb);
  }
  if (wk.n_tc > 0)
    LAUNCH(KVPRM_PROF_ATTN_TC,
           kvprm::launch_attention_tc(as, wk, &ctx->tm_pool_tc, layer, Q.hi, Q.lo, ctx->apart_o, ctx->apart_ml,
                                      tc_margin(ctx), ctx->err_d, st, pdl, TS, tc_prof),
           "attention_tc");
  LAUNCH(KVPRM_PROF_ATTN,
         kvprm::launch_attention(as, wk, &ctx->tm_pool, layer, Q.hi, Q.lo, ctx->apart_o, ctx->apart_ml, mg,
                                 ctx->err_d, st, pdl, TS),
         "attention");
  return KVPRM_OK;
}

int enqueue_forward(kvprm_ctx* ctx, const CallPlan& P, Enq& E, const FwdSaves* sv = nullptr) {
  const ModelDims& m = ctx->md;
  const int n = P.n, np = P.n_pad;
  const int32_t* sl = ctx->tables_d;
  cudaStream_t st = E.st;
  const bool pdl = E.pdl;
  const int NL = ctx->cfg.n_layers;
  const kvprm::HiLo X{ctx->xhi, ctx->xlo}, O{ctx->ohi, ctx->olo};
  kvprm::GemmEpilogue eq;   // QKV projection -> rotated q, self k / v
  eq.mode = kvprm::GemmEpilogue::QKV;
  eq.M = m.qkv_rows;
  eq.n_valid = n;
  eq.rope = ctx->rope;
  eq.n_q = m.n_q;
  eq.n_kv = m.n_kv;
  eq.hd = m.hd;
  eq.q = ctx->q;
  eq.q_hi = ctx->qhi;
  eq.q_lo = ctx->qlo;
  eq.kself = ctx->kself;
  eq.vself = ctx->vself;
  // the pre-attention RMSNorm's per-candidate factor, from the residual stream's tile sums of squares
  eq.rs_sumsq = ctx->sumsq;
  eq.rs_tiles = ctx->d_tiles;
  eq.rs_d = m.d;
  eq.rs_eps = m.eps;
  kvprm::GemmEpilogue er;   // O and down projections -> residual stream + tile sums of squares
  er.mode = kvprm::GemmEpilogue::RESID;
  er.M = m.d;
  er.n_valid = n;
  er.h = ctx->h;
  er.sumsq = ctx->sumsq;
  er.x_hi = X.hi;   // h ⊙ (next RMSNorm gain): the next projection's input
  er.x_lo = X.lo;
  kvprm::GemmEpilogue es;   // gate/up projection -> SiLU(gate) * up
  es.mode = kvprm::GemmEpilogue::SILU;
  es.M = m.ff;
  es.n_valid = n;
  es.ff = m.ff;
  es.a_hi = ctx->ahi;
  es.a_lo = ctx->alo;
  es.rs_sumsq = ctx->sumsq;   // the pre-MLP RMSNorm's per-candidate factor
  es.rs_tiles = ctx->d_tiles;
  es.rs_d = m.d;
  es.rs_eps = m.eps;
  kvprm::GemmEpilogue et;   // scorer adapter: t = scale (A x), the K extension of the projection after it
  et.mode = kvprm::GemmEpilogue::LOWRANK;
  et.M = ctx->lora_rank;
  et.n_valid = n;
  et.lr_scale = ctx->lora_scale;
  et.t_hi = ctx->thi;
  et.t_lo = ctx->tlo;
  const bool lora = ctx->lora_rank > 0;
  // launch A x of projection j (0 QKV, 1 O, 2 gate/up, 3 down) of layer l on the projection's input
  // maps; returns the K extension the projection itself then takes
  auto adapter = [&](int j, int l, const GemmPlan& g, const CUtensorMap* xh, const CUtensorMap* xl, int k_main,
                     kvprm::GemmLowRank* lr) -> int {
    static const char* what[4] = {"adapter_qkv", "adapter_o", "adapter_gate_up", "adapter_down"};
    LAUNCH(KVPRM_PROF_LORA, kvprm::launch_gemm(g, &ctx->tm_la[j][l], xh, xl, et, np, ctx->err_d, st, pdl, TS), what[j]);
    lr->b = &ctx->tm_lb[j][l];
    lr->t_hi = &ctx->tm_thi;
    lr->t_lo = &ctx->tm_tlo;
    lr->k_main = k_main;
    return KVPRM_OK;
  };
  ctx->trace_n = 0;
  ctx->trace_cls.clear();
  if (ctx->trace)
    CK(cudaMemsetAsync(ctx->trace_d, 0xFF, sizeof(unsigned long long) * kvprm::kTraceStride * ctx->trace_cap, st),
       "trace reset");
  LAUNCH(KVPRM_PROF_FUSED,
         kvprm::launch_rope_table(sl, n, m.hd, ctx->cfg.rope_base, ctx->depth, ctx->rope, st, false, TS), "rope");
  LAUNCH(KVPRM_PROF_FUSED,
         kvprm::launch_embed_norm(m, ctx->embed, ctx->attn_norm[0], n, ctx->h, ctx->sumsq, X, st, pdl, TS),
         "embed_norm");
  for (int l = 0; l < NL; ++l) {
    kvprm::GemmLowRank lr_qkv, lr_o, lr_gu, lr_down;
    int arc;
    if (lora && (arc = adapter(0, l, P.l_qkv, &ctx->tm_xhi, &ctx->tm_xlo, P.k_qkv, &lr_qkv))) return arc;
    kvprm::GemmEpilogue eq_l = eq;   // this layer's per-head q/k RMSNorm gains, if the scorer has them
    if (ctx->cfg.qk_norm) {
      eq_l.qn_gain = ctx->q_norm[l];
      eq_l.kn_gain = ctx->k_norm[l];
    }
    const size_t Bm = static_cast<size_t>(ctx->cfg.max_candidates);
    if (sv) {   // a backward pass follows: this layer's q, self k / v go to their saved slots
      eq_l.q = sv->q + l * Bm * m.n_q * m.hd;
      eq_l.kself = sv->k + l * Bm * m.n_kv * m.hd;
      eq_l.vself = sv->v + l * Bm * m.n_kv * m.hd;
    }
    LAUNCH(KVPRM_PROF_GEMM_QKV,
           kvprm::launch_gemm(P.g_qkv, &ctx->tm_qkv[l], &ctx->tm_xhi, &ctx->tm_xlo, eq_l, np, ctx->err_d, st, pdl, TS,
                              lora ? &lr_qkv : nullptr),
           "gemm_qkv");
    if (ctx->debug_flags & 2) {
      const size_t nq = static_cast<size_t>(n) * m.n_q * m.hd, nk = static_cast<size_t>(n) * m.n_kv * m.hd;
      CK(cudaMemcpyAsync(ctx->dbg_q + l * nq, eq_l.q, nq * 4, cudaMemcpyDeviceToDevice, st), "debug q");
      CK(cudaMemcpyAsync(ctx->dbg_k + l * nk, eq_l.kself, nk * 4, cudaMemcpyDeviceToDevice, st), "debug k");
      CK(cudaMemcpyAsync(ctx->dbg_v + l * nk, eq_l.vself, nk * 4, cudaMemcpyDeviceToDevice, st), "debug v");
    }
    float* dbg = (ctx->debug_flags & 1) ? ctx->dbg + static_cast<size_t>(l) * n * m.n_q * m.hd : nullptr;
    kvprm::AttnMerge mg{eq_l.q, eq_l.kself, eq_l.vself, O.hi, O.lo, nullptr, dbg, ctx->depth};
    if (sv) {
      mg.out_f32 = sv->o + l * Bm * m.n_q * m.hd;
      mg.lse = sv->lse + l * Bm * m.n_q;
    }
    const kvprm::AttnWork wk = device_work(ctx);
    if (ctx->layer_waits)   // this layer's pages are still being copied in (kvprm_score_host)
      CK(cudaStreamWaitEvent(st, ctx->layer_ready[l], E.capturing ? cudaEventWaitExternal : cudaEventWaitDefault),
         "cudaStreamWaitEvent(layer pages)");
    {
      const int rc = enqueue_attention(ctx, E, ctx->as, wk, l, kvprm::HiLo{ctx->qhi, ctx->qlo}, mg, pdl);
      if (rc) return rc;
    }
    if (wk.fuse_cs == 0)   // else the attention launch merged the slots itself
      LAUNCH(KVPRM_PROF_COMBINE,
             kvprm::launch_attn_combine(ctx->as, wk, n, ctx->apart_o, ctx->apart_ml, mg, st, pdl, TS,
                                        (ctx->debug_flags & 64) != 0),
             "attn_combine");
    kvprm::GemmEpilogue er_o = er;   // h += W_o o; x = h ⊙ g_mlp for the gate/up projection
    er_o.gain_next = ctx->mlp_norm[l];
    er_o.late_trigger = true;   // gate/up CTAs fit beside the O projection's
    if (sv) er_o.h_copy = sv->hmid + l * Bm * m.d;
    if (lora && (arc = adapter(1, l, P.l_o, &ctx->tm_ohi, &ctx->tm_olo, P.k_o, &lr_o))) return arc;
    LAUNCH(KVPRM_PROF_GEMM_O,
           kvprm::launch_gemm(P.g_o, &ctx->tm_o[l], &ctx->tm_ohi, &ctx->tm_olo, er_o, np, ctx->err_d, st, pdl, TS,
                              lora ? &lr_o : nullptr),
           "gemm_o");
    if (lora && (arc = adapter(2, l, P.l_gu, &ctx->tm_xhi, &ctx->tm_xlo, P.k_gu, &lr_gu))) return arc;
    kvprm::GemmEpilogue es_l = es;
    if (sv) es_l.gu_save = sv->gu + l * Bm * 2 * m.ff;
    LAUNCH(KVPRM_PROF_GEMM_GATE_UP,
           kvprm::launch_gemm(P.g_gu, &ctx->tm_gu[l], &ctx->tm_xhi, &ctx->tm_xlo, es_l, np, ctx->err_d, st, pdl, TS,
                              lora ? &lr_gu : nullptr),
           "gemm_gate_up");
    kvprm::GemmEpilogue er_d = er;   // h += W_down a; x = h ⊙ g_attn of the next layer
    er_d.gain_next = l + 1 < NL ? ctx->attn_norm[l + 1] : nullptr;
    if (sv) er_d.h_copy = sv->hout + l * Bm * m.d;
    if (lora && (arc = adapter(3, l, P.l_down, &ctx->tm_ahi, &ctx->tm_alo, P.k_down, &lr_down))) return arc;
    LAUNCH(KVPRM_PROF_GEMM_DOWN,
           kvprm::launch_gemm(P.g_down, &ctx->tm_down[l], &ctx->tm_ahi, &ctx->tm_alo, er_d, np, ctx->err_d, st, pdl,
                              TS, lora ? &lr_down : nullptr),
           "gemm_down");
    if (l + 1 == NL) {
      LAUNCH(KVPRM_PROF_FUSED,
             kvprm::launch_head(m, ctx->h, ctx->sumsq, ctx->d_tiles, n, ctx->depth, ctx->final_norm, ctx->w_plus,
                                ctx->w_minus, ctx->rewards_d, st, pdl, TS),
             "reward_head");
    }
    if (ctx->debug_flags & 4) {
      const size_t nh = static_cast<size_t>(n) * m.d;
      CK(cudaMemcpyAsync(ctx->dbg_h + l * nh, ctx->h, nh * 4, cudaMemcpyDeviceToDevice, st), "debug h");
    }
  }
  return KVPRM_OK;
}

int accumulate_marks(kvprm_ctx* ctx, std::vector<ProfMark>& marks, bool destroy) {
  for (auto& mk : marks) {
    float ms = 0.f;
    if (mk.a) CK(cudaEventElapsedTime(&ms, mk.a, mk.b), "cudaEventElapsedTime");
    ctx->prof_launches[mk.cls] += 1;
    ctx->prof_ms[mk.cls] += ms;
    if (destroy && mk.a) {
      cudaEventDestroy(mk.a);
      cudaEventDestroy(mk.b);
    }
  }
  if (destroy) marks.clear();
  return KVPRM_OK;
}

void drop_graph(kvprm_ctx* ctx) {
  if (ctx->gexec) cudaGraphExecDestroy(ctx->gexec);
  ctx->gexec = nullptr;
  for (auto& m : ctx->graph_marks) {
    if (m.a) cudaEventDestroy(m.a);
    if (m.b) cudaEventDestroy(m.b);
  }
  ctx->graph_marks.clear();
  ctx->gkey = GraphKey();
}

// Host-resident cache pages into the device pool by SM loads of pinned host memory: every thread
// moves 16 bytes per step, four steps in flight (grid-stride).  Measured on GB300 (8 GB of pinned
// memory): 64 CTAs of 4 warps hold the host link at ~211 GB/s on every copy, where copy-engine
// copies of the same buffer ran at ~211 GB/s on most copies and ~120 GB/s on others.  Small CTAs
// (128 threads, no shared memory, the maximum shared-memory carve-out) share SMs with the scoring
// kernels that run meanwhile.
__global__ void __launch_bounds__(128) pool_pull_kernel(const uint4* __restrict__ src, uint4* __restrict__ dst,
                                                        int64_t n) {
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x;
  for (; i + 3 * stride < n; i += 4 * stride) {
    const uint4 a = src[i], b = src[i + stride], c = src[i + 2 * stride], d = src[i + 3 * stride];
    dst[i] = a;
    dst[i + stride] = b;
    dst[i + 2 * stride] = c;
    dst[i + 3 * stride] = d;
  }
  for (; i < n; i += stride) dst[i] = src[i];
}

constexpr int kPoolPullCtas = 64;

// Copy `bytes` (a multiple of 16; both addresses 16-byte aligned, else cudaErrorInvalidValue) from
// device-accessible pinned host memory `src` into device memory `dst`.
cudaError_t launch_pool_pull(const void* src, void* dst, size_t bytes, cudaStream_t stream) {
  if (bytes == 0) return cudaSuccess;
  if ((reinterpret_cast<uintptr_t>(src) | reinterpret_cast<uintptr_t>(dst) | bytes) & 15u) return cudaErrorInvalidValue;
  // the SMs keep the shared-memory configuration of the scoring kernels while these CTAs sit beside
  // them (a CTA preferring a larger L1 would wait for an SM to drain first)
  static const cudaError_t carve =
      cudaFuncSetAttribute(pool_pull_kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                           static_cast<int>(cudaSharedmemCarveoutMaxShared));
  if (carve != cudaSuccess) return carve;
  pool_pull_kernel<<<kPoolPullCtas, 128, 0, stream>>>(static_cast<const uint4*>(src), static_cast<uint4*>(dst),
                                                      static_cast<int64_t>(bytes / 16));
  return cudaGetLastError();
}

// The device address of host memory [p, p + bytes) when the GPU can read all of it as pinned memory:
// its first and last byte page-locked (cudaMemoryTypeHost) and mapped at one contiguous device range,
// p and bytes 16-byte aligned; else null (pageable memory, or anything the query cannot vouch for).
const void* pinned_device_view(const void* p, size_t bytes) {
  if (!p || bytes == 0 || !aligned16(p) || (bytes & 15u)) return nullptr;
  const uint8_t* last = static_cast<const uint8_t*>(p) + bytes - 1;
  cudaPointerAttributes a0{}, a1{};
  if (cudaPointerGetAttributes(&a0, p) != cudaSuccess || cudaPointerGetAttributes(&a1, last) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  if (a0.type != cudaMemoryTypeHost || a1.type != cudaMemoryTypeHost || !a0.devicePointer || !a1.devicePointer)
    return nullptr;
  if (static_cast<const uint8_t*>(a1.devicePointer) - static_cast<const uint8_t*>(a0.devicePointer) !=
      static_cast<std::ptrdiff_t>(bytes - 1))
    return nullptr;
  return aligned16(a0.devicePointer) ? a0.devicePointer : nullptr;
}

// kvprm_score_host's cache copy: layer by layer, in layer order on ONE copy stream (the copy engine
// drains one stream's queue before the next, so layers spread over several streams arrive out of
// order), after the work already on `st` (an earlier call may still read the pool, and this call's
// tables go first, so that the small table copies do not queue behind the cache); layer l's event
// gates layer l's attention.  Pinned host memory is pulled by SM loads (launch_pool_pull) in 64 MB
// launches, so that a scoring kernel whose CTAs cannot be placed beside the copy's waits for at most
// one launch (~0.3 ms): with one launch per layer (1 GB, ~5 ms) the long 8B call took 248-264 ms,
// in 64 MB launches 177 ms, and 172 ms with the forward launched without programmatic dependent
// launch (score_device), against 163 ms for its 34 GB at the link's ~211 GB/s.  Other host memory
// goes through the copy engine.
int enqueue_pool_copy(kvprm_ctx* ctx, cudaStream_t st) {
  CK(cudaEventRecord(ctx->pool_free, st), "cudaEventRecord(pool free)");
  const size_t layer_bytes = ctx->host_pool_bytes / static_cast<size_t>(ctx->cfg.n_layers);
  cudaStream_t cs = ctx->copy_stream;
  CK(cudaStreamWaitEvent(cs, ctx->pool_free, 0), "cudaStreamWaitEvent(pool)");
  const void* src = pinned_device_view(ctx->host_pool, ctx->host_pool_bytes);
  const size_t piece = size_t(64) << 20;
  for (int l = 0; l < ctx->cfg.n_layers; ++l) {
    uint8_t* dst = static_cast<uint8_t*>(ctx->dev_pool) + l * layer_bytes;
    if (src) {
      for (size_t off = 0; off < layer_bytes; off += piece)
        CK(launch_pool_pull(static_cast<const uint8_t*>(src) + l * layer_bytes + off, dst + off,
                            std::min(piece, layer_bytes - off), cs),
           "pool_pull_kernel");
    } else {
      CK(cudaMemcpyAsync(dst, static_cast<const uint8_t*>(ctx->host_pool) + l * layer_bytes, layer_bytes,
                         cudaMemcpyHostToDevice, cs),
         "cudaMemcpyAsync(pool layer)");
    }
    CK(cudaEventRecord(ctx->layer_ready[l], cs), "cudaEventRecord(layer ready)");
  }
  return KVPRM_OK;
}

// Score into ctx->rewards_d on stream `st` (stream-ordered).  With `prepared` set, the call is
// planned and its tables uploaded (stream-ordered on `st`), and its plan returned there instead of
// enqueueing the forward (the gradient call enqueues the forward together with the backward).
int score_device(kvprm_ctx* ctx, const void* kv_pages, int64_t n_pages, const int32_t* bt, const int32_t* sl, int32_t n,
                 cudaStream_t st, const FwdSaves* sv = nullptr, CallPlan* prepared = nullptr) {
  int max_pages = 0;
  int rc = validate_tables(ctx, n_pages, bt, sl, n, &max_pages);
  if (rc) return rc;
  if (n == 0) return KVPRM_OK;
  // depth-k readout: each candidate's verify tokens are rows of the batch over the candidate's pages
  const int D = ctx->depth;
  if (D > 1) {
    if (static_cast<int64_t>(n) * D > ctx->cfg.max_candidates)
      return fail(ctx, KVPRM_ECAPACITY, "n_candidates x readout depth = %lld exceeds max_candidates = %d",
                  static_cast<long long>(n) * D, ctx->cfg.max_candidates);
    const int mb = ctx->cfg.max_blocks_per_seq;
    ctx->row_bt.resize(static_cast<size_t>(n) * D * mb);
    ctx->row_sl.resize(static_cast<size_t>(n) * D);
    for (int b = 0; b < n; ++b)
      for (int t = 0; t < D; ++t) {
        const size_t row = static_cast<size_t>(b) * D + t;
        ctx->row_sl[row] = sl[b];
        std::memcpy(ctx->row_bt.data() + row * mb, bt + static_cast<size_t>(b) * mb, sizeof(int32_t) * mb);
      }
    bt = ctx->row_bt.data();
    sl = ctx->row_sl.data();
    n *= D;
  }
  const void* pool = kv_pages;
  int64_t pages = n_pages;
  if (max_pages == 0) {   // no cached token anywhere: the pool is never read
    pool = ctx->dummy_pool;
    pages = 1;
  } else {
    if (!kv_pages) return fail(ctx, KVPRM_EINVAL, "kv_pages is NULL");
    if (!aligned16(kv_pages)) return fail(ctx, KVPRM_EINVAL, "kv_pages is not 16-byte aligned");
  }
  if ((rc = ensure_pool_map(ctx, pool, pages, ctx->cfg.n_layers))) return rc;
  ctx->as.layer_pages = pages;
  // a depth-k readout's rows share their candidate's pages: the persistent plan scores each page once
  // per candidate, and its combine adds the causal verify-token entries
  if ((rc = plan_work(ctx, bt, sl, n, D == 1))) return rc;
  const CallPlan P = make_plan(ctx, n, max_pages);
  if ((rc = ensure_x_maps(ctx, P.n_pad))) return rc;
  if ((rc = ensure_t_maps(ctx, P.n_pad))) return rc;
  if ((rc = upload_tables(ctx, bt, sl, n, st))) return rc;
  if (ctx->layer_waits && (rc = enqueue_pool_copy(ctx, st))) return rc;
  ctx->last_n = n;
  ctx->last_stream = st;
  if (ctx->inject_fail) {   // failure-detection hook: report a failed launch, enqueue nothing more
    ctx->inject_fail = 0;
    return cuda_fail(ctx, cudaErrorLaunchFailure, "injected failure of the forward's launch");
  }
  if (prepared) {
    *prepared = P;
    return KVPRM_OK;
  }

  // While the cache of a host-buffer call is being copied in by SM loads, no launch is made early:
  // a kernel that programmatic dependent launch places ahead of its predecessor's end holds SM slots
  // the copy's CTAs would use (long 8B from pinned memory: 177.5 ms per call with, 171.5 ms without).
  const bool pdl = ctx->use_pdl && !ctx->profile && !ctx->layer_waits;
  if (!ctx->use_graph || sv) {   // a forward that keeps its intermediates runs eagerly
    Enq E{ctx, st, pdl, ctx->profile, &ctx->live_marks};
    if ((rc = enqueue_forward(ctx, P, E, sv))) return rc;
    if (ctx->profile) {
      CK(cudaStreamSynchronize(st), "cudaStreamSynchronize(profile)");
      if ((rc = accumulate_marks(ctx, ctx->live_marks, true))) return rc;
    }
    return KVPRM_OK;
  }
  GraphKey key;
  key.n = n;
  key.n_pad = P.n_pad;
  key.attn_ctas = P.attn_ctas;
  key.tc_ctas = ctx->work_host.n_tc_ctas * (ctx->work_host.tc_concurrent ? -1 : 1);
  key.fuse_cs = ctx->work_host.fuse_cs;
  key.layer_waits = ctx->layer_waits ? 1 : 0;
  key.lora_rank = ctx->lora_rank;
  key.depth = ctx->depth;
  key.n_tc = ctx->work_host.n_tc > 0 ? 1 : 0;
  key.debug = ctx->debug_flags;
  key.profile = ctx->profile ? 1 : 0;
  key.pdl = pdl ? 1 : 0;
  key.trace = ctx->trace ? 1 : 0;
  key.pool = pool;
  key.n_pages = pages;
  if (!(ctx->gexec && key == ctx->gkey)) {
    drop_graph(ctx);
    CK(cudaStreamBeginCapture(ctx->cap_stream, cudaStreamCaptureModeThreadLocal), "cudaStreamBeginCapture");
    Enq E{ctx, ctx->cap_stream, pdl, ctx->profile, &ctx->graph_marks};
    E.capturing = true;
    rc = enqueue_forward(ctx, P, E);
    cudaGraph_t graph = nullptr;
    cudaError_t e = cudaStreamEndCapture(ctx->cap_stream, &graph);
    if (rc) {
      if (graph) cudaGraphDestroy(graph);
      return rc;
    }
    if (e != cudaSuccess) return cuda_fail(ctx, e, "cudaStreamEndCapture");
    e = cudaGraphInstantiate(&ctx->gexec, graph, 0);
    cudaGraphDestroy(graph);
    if (e != cudaSuccess) {
      ctx->gexec = nullptr;
      return cuda_fail(ctx, e, "cudaGraphInstantiate");
    }
    ctx->gkey = key;
  }
  CK(cudaGraphLaunch(ctx->gexec, st), "cudaGraphLaunch");
  if (ctx->profile) {
    CK(cudaStreamSynchronize(st), "cudaStreamSynchronize(profile)");
    if ((rc = accumulate_marks(ctx, ctx->graph_marks, false))) return rc;
  }
  return KVPRM_OK;
}

int finish_blocking(kvprm_ctx* ctx, int32_t n, float* rewards, cudaStream_t st) {
  if (n == 0) return KVPRM_OK;
  CK(cudaMemcpyAsync(ctx->h_rewards, ctx->rewards_d, sizeof(float) * n, cudaMemcpyDeviceToHost, st),
     "cudaMemcpyAsync(rewards)");
  CK(cudaMemcpyAsync(ctx->h_err, ctx->err_d, sizeof(int), cudaMemcpyDeviceToHost, st), "cudaMemcpyAsync(err)");
  CK(cudaStreamSynchronize(st), "cudaStreamSynchronize");
  if (*ctx->h_err) {
    const int site = *ctx->h_err;
    cudaMemsetAsync(ctx->err_d, 0, sizeof(int), st);
    return fail(ctx, KVPRM_ETIMEOUT, "a bounded device wait timed out (code %d); results are invalid", site);
  }
  std::memcpy(rewards, ctx->h_rewards, sizeof(float) * n);
  return KVPRM_OK;
}

// ---------------------------------------------------------------- KV Steering: backward pass
// First kvprm_score_grad call: transposed weight copies, forward saves and backward buffers, sized
// for max_candidates.
int ensure_grad(kvprm_ctx* ctx, cudaStream_t st) {
  GradState& g = ctx->grad;
  if (g.ready) return KVPRM_OK;
  const ModelDims& m = ctx->md;
  const int NL = ctx->cfg.n_layers;
  const size_t Bm = static_cast<size_t>(ctx->cfg.max_candidates);
  const size_t nqh = static_cast<size_t>(m.n_q) * m.hd, nkh = static_cast<size_t>(m.n_kv) * m.hd;
  int rc;
  // saves: one allocation carved per array
  const size_t per_layer = Bm * (nqh + 2 * nkh + nqh + m.n_q + 2 * static_cast<size_t>(m.d) + 2 * static_cast<size_t>(m.ff));
  float* base = nullptr;
  if ((rc = dalloc(ctx, &base, per_layer * NL, "backward saves"))) return rc;
  FwdSaves& sv = g.sv;
  float* p = base;
  auto take = [&](size_t per) {
    float* r = p;
    p += per * NL;
    return r;
  };
  sv.q = take(Bm * nqh);
  sv.k = take(Bm * nkh);
  sv.v = take(Bm * nkh);
  sv.o = take(Bm * nqh);
  sv.lse = take(Bm * m.n_q);
  sv.hmid = take(Bm * m.d);
  sv.hout = take(Bm * m.d);
  sv.gu = take(Bm * 2 * static_cast<size_t>(m.ff));
  // backward buffers
  const size_t wmax = std::max<size_t>(std::max<size_t>(m.ff, m.d), nqh);
  const size_t gmax = std::max<size_t>(std::max<size_t>(2 * static_cast<size_t>(m.ff), m.qkv_rows), m.d);
  float* bb = nullptr;
  if ((rc = dalloc(ctx, &bb, Bm * (m.d + wmax + m.n_q + nqh + 2 * nkh), "backward buffers"))) return rc;
  g.dh = bb;
  g.tmp = g.dh + Bm * m.d;
  g.D = g.tmp + Bm * wmax;
  g.dq = g.D + Bm * m.n_q;
  g.dks = g.dq + Bm * nqh;
  g.dvs = g.dks + Bm * nkh;
  if ((rc = dalloc(ctx, &g.ghi, static_cast<size_t>(ctx->npad_max) * gmax, "backward hi"))) return rc;
  if ((rc = dalloc(ctx, &g.glo, static_cast<size_t>(ctx->npad_max) * gmax, "backward lo"))) return rc;
  // transposed weights: W [out][in] -> W^T [in][out], from the borrowed weights' tensor-map bases
  g.tm_qkv.resize(NL);
  g.tm_o.resize(NL);
  g.tm_gu.resize(NL);
  g.tm_down.resize(NL);
  struct Mat {
    int out, in;
  } mats[4] = {{m.qkv_rows, m.d}, {m.d, m.n_q * m.hd}, {2 * m.ff, m.d}, {m.d, m.ff}};
  for (int l = 0; l < NL; ++l) {
    const void* src[4] = {ctx->w_qkv_src[l], ctx->w_o_src[l], ctx->w_gu_src[l], ctx->w_down_src[l]};
    CUtensorMap* maps[4] = {&g.tm_qkv[l], &g.tm_o[l], &g.tm_gu[l], &g.tm_down[l]};
    for (int j = 0; j < 4; ++j) {
      bf16* wt = nullptr;
      if ((rc = dalloc(ctx, &wt, static_cast<size_t>(mats[j].out) * mats[j].in, "transposed weights"))) return rc;
      g.wt.push_back(wt);
      CK(kvprm::launch_transpose(static_cast<const bf16*>(src[j]), wt, mats[j].out, mats[j].in, st), "transpose");
      // W^T [in][out]: M = in rows, K = out columns
      if ((rc = make_map(ctx, maps[j], wt, mats[j].out, mats[j].in, 64, 128, "transposed weights"))) return rc;
    }
  }
  g.ready = true;
  return KVPRM_OK;
}

int ensure_grad_maps(kvprm_ctx* ctx, int n_pad) {
  GradState& g = ctx->grad;
  if (g.tm_npad == n_pad) return KVPRM_OK;
  const ModelDims& m = ctx->md;
  int rc;
  if ((rc = make_map(ctx, &g.tm_d_hi, g.ghi, m.d, n_pad, 64, n_pad, "grad hi (d)"))) return rc;
  if ((rc = make_map(ctx, &g.tm_d_lo, g.glo, m.d, n_pad, 64, n_pad, "grad lo (d)"))) return rc;
  if ((rc = make_map(ctx, &g.tm_gu_hi, g.ghi, 2 * static_cast<uint64_t>(m.ff), n_pad, 64, n_pad, "grad hi (gu)")))
    return rc;
  if ((rc = make_map(ctx, &g.tm_gu_lo, g.glo, 2 * static_cast<uint64_t>(m.ff), n_pad, 64, n_pad, "grad lo (gu)")))
    return rc;
  if ((rc = make_map(ctx, &g.tm_qkv_hi, g.ghi, m.qkv_rows, n_pad, 64, n_pad, "grad hi (qkv)"))) return rc;
  if ((rc = make_map(ctx, &g.tm_qkv_lo, g.glo, m.qkv_rows, n_pad, 64, n_pad, "grad lo (qkv)"))) return rc;
  g.tm_npad = n_pad;
  return KVPRM_OK;
}

template <typename T>
int grow(kvprm_ctx* ctx, T** p, size_t* cap, size_t need, const char* what) {
  if (need <= *cap) return KVPRM_OK;
  cudaFree(*p);
  *p = nullptr;
  *cap = 0;
  int rc = dalloc(ctx, p, need, what);
  if (rc) return rc;
  *cap = need;
  return KVPRM_OK;
}

// The gradient of sum_b -log P(+)_b with respect to the pages (all layers) into grad [N_L][n_pages]
// [2][n_kv][16][hd] (fp32), and P(+) into ctx->rewards_d.  Blocking (the caller synchronises); on
// return *n_ref / ref_pages hold the pages the tables reference (device list at lists + n_shared).
int score_grad_device(kvprm_ctx* ctx, const void* kv_pages, int64_t n_pages, const int32_t* bt, const int32_t* sl,
                      int32_t n, float* grad, cudaStream_t st, int* n_ref_out) {
  if (ctx->lora_rank) return fail(ctx, KVPRM_EUNSUPPORTED, "the backward pass takes the merged weights (no adapter)");
  if (ctx->depth != 1) return fail(ctx, KVPRM_EUNSUPPORTED, "the backward pass takes one verify token (depth 1)");
  if (ctx->cfg.qk_norm) return fail(ctx, KVPRM_EUNSUPPORTED, "the backward pass does not implement the q/k norm");
  if (n > 0 && !grad) return fail(ctx, KVPRM_EINVAL, "the gradient buffer is NULL");
  if (grad && (reinterpret_cast<uintptr_t>(grad) & 15u)) return fail(ctx, KVPRM_EINVAL, "grad is not 16-byte aligned");
  int max_pages = 0;
  int rc = validate_tables(ctx, n_pages, bt, sl, n, &max_pages);
  if (rc) return rc;
  *n_ref_out = 0;
  if (n == 0) return KVPRM_OK;
  if ((rc = ensure_grad(ctx, st))) return rc;
  GradState& g = ctx->grad;
  // the call's plan and tables (the forward itself is enqueued below, with the backward)
  CallPlan P;
  if ((rc = score_device(ctx, kv_pages, n_pages, bt, sl, n, st, &g.sv, &P))) return rc;
  const ModelDims& m = ctx->md;
  const int NL = ctx->cfg.n_layers, mb = ctx->cfg.max_blocks_per_seq;
  const int np = (n + 15) / 16 * 16;
  if ((rc = ensure_grad_maps(ctx, np))) return rc;
  // host plan: work units (candidate, kv head, <= 8 pages) and the pages several candidates read
  std::vector<int4> units;
  std::vector<uint8_t> refs(static_cast<size_t>(n_pages > 0 ? n_pages : 1), 0);
  constexpr int kUnitPages = kvprm::kBackUnitPagesMax;
  for (int b = 0; b < n; ++b) {
    const int pages = (sl[b] + 15) / 16;
    for (int j = 0; j < pages; ++j) {
      uint8_t& r = refs[bt[static_cast<int64_t>(b) * mb + j]];
      if (r < 2) ++r;
    }
    for (int gg = 0; gg < m.n_kv; ++gg)
      for (int j0 = 0; j0 < pages; j0 += kUnitPages) units.push_back(make_int4(b, gg, j0, std::min(pages, j0 + kUnitPages)));
  }
  std::vector<int32_t> lists;   // shared pages, then every referenced page
  for (int64_t p = 0; p < n_pages; ++p)
    if (refs[p] >= 2) lists.push_back(static_cast<int32_t>(p));
  const int n_shared = static_cast<int>(lists.size());
  for (int64_t p = 0; p < n_pages; ++p)
    if (refs[p] >= 1) lists.push_back(static_cast<int32_t>(p));
  for (auto& r : refs) r = r >= 2 ? 1 : 0;
  if ((rc = grow(ctx, &g.units, &g.units_cap, std::max<size_t>(units.size(), 1), "backward units"))) return rc;
  if ((rc = grow(ctx, &g.shared, &g.shared_cap, refs.size(), "shared-page flags"))) return rc;
  if ((rc = grow(ctx, &g.lists, &g.lists_cap, std::max<size_t>(lists.size(), 1), "page lists"))) return rc;
  if (!units.empty())
    CK(cudaMemcpyAsync(g.units, units.data(), sizeof(int4) * units.size(), cudaMemcpyHostToDevice, st), "units");
  CK(cudaMemcpyAsync(g.shared, refs.data(), refs.size(), cudaMemcpyHostToDevice, st), "shared flags");
  if (!lists.empty())
    CK(cudaMemcpyAsync(g.lists, lists.data(), sizeof(int32_t) * lists.size(), cudaMemcpyHostToDevice, st), "lists");
  g.n_shared = n_shared;
  g.n_ref = static_cast<int>(lists.size()) - n_shared;
  *n_ref_out = g.n_ref;
  const int64_t page_elems = static_cast<int64_t>(2) * m.n_kv * 16 * m.hd;
  const size_t Bm = static_cast<size_t>(ctx->cfg.max_candidates);
  const int nqh = m.n_q * m.hd, nkh = m.n_kv * m.hd;
  const FwdSaves& sv = g.sv;
  // the forward with its saves, then the backward, on stream `s`
  auto enqueue = [&](cudaStream_t s, Enq& E) -> int {
    int r = enqueue_forward(ctx, P, E, &sv);
    if (r) return r;
    CK(kvprm::launch_zero_pages(grad, g.lists, n_shared, NL, n_pages, page_elems, s), "zero shared pages");
    // the backward products on the forward's GEMM (plain fp32 epilogue) against the transposed weights
    auto gemm = [&](const CUtensorMap* w, int M, int K, const CUtensorMap* xh, const CUtensorMap* xl, float* out) {
      const GemmPlan gp = kvprm::plan_gemm(M, K, np, ctx->num_sms, true, false);
      kvprm::GemmEpilogue ep;
      ep.mode = kvprm::GemmEpilogue::PLAIN;
      ep.M = M;
      ep.n_valid = n;
      ep.out = out;
      return kvprm::launch_gemm(gp, w, xh, xl, ep, np, ctx->err_d, s, ctx->use_pdl);
    };
    CK(kvprm::launch_head_back(ctx->h, ctx->rewards_d, ctx->final_norm, ctx->w_plus, ctx->w_minus, n, m.d, m.eps, g.dh,
                               g.ghi, g.glo, s),
       "head backward");
    for (int l = NL - 1; l >= 0; --l) {
      // feed-forward block: da = W_down^T dh; [du; dt]; dx2 = W_gate_up^T [du; dt]; dh_mid
      CK(gemm(&g.tm_down[l], m.ff, m.d, &g.tm_d_hi, &g.tm_d_lo, g.tmp), "W_down^T product");
      CK(kvprm::launch_silu_back(g.tmp, sv.gu + l * Bm * 2 * m.ff, n, m.ff, g.ghi, g.glo, s), "SiLU backward");
      CK(gemm(&g.tm_gu[l], m.d, 2 * m.ff, &g.tm_gu_hi, &g.tm_gu_lo, g.tmp), "W_gate_up^T product");
      CK(kvprm::launch_rms_back(sv.hmid + l * Bm * m.d, nullptr, ctx->mlp_norm[l], g.tmp, g.dh, n, m.d, m.eps, g.dh,
                                g.ghi, g.glo, s),
         "pre-MLP RMSNorm backward");
      // attention block: do = W_o^T dh_mid, then the read-out's backward into this layer's pages
      CK(gemm(&g.tm_o[l], nqh, m.d, &g.tm_d_hi, &g.tm_d_lo, g.tmp), "W_o^T product");
      kvprm::AttnBackArgs a;
      a.n = n;
      a.n_q = m.n_q;
      a.n_kv = m.n_kv;
      a.hd = m.hd;
      a.q = sv.q + l * Bm * nqh;
      a.kself = sv.k + l * Bm * nkh;
      a.vself = sv.v + l * Bm * nkh;
      a.o = sv.o + l * Bm * nqh;
      a.dout = g.tmp;
      a.lse = sv.lse + l * Bm * m.n_q;
      a.D = g.D;
      a.dq = g.dq;
      a.dks = g.dks;
      a.dvs = g.dvs;
      a.units = g.units;
      a.n_units = static_cast<int>(units.size());
      a.seq_lens = ctx->tables_d;
      a.block_table = ctx->tables_d + ctx->cfg.max_candidates;
      a.max_blocks = mb;
      a.pool_layer = kv_pages ? static_cast<const bf16*>(kv_pages) + l * n_pages * page_elems : nullptr;
      a.shared = g.shared;
      a.grad_layer = grad + l * n_pages * page_elems;
      a.err = ctx->err_d;
      a.tm_pool = kv_pages && !ctx->grad_cuda_cores ? &ctx->tm_pool : nullptr;   // the forward's map of this pool
      a.layer_page0 = static_cast<int64_t>(l) * n_pages;
      CK(kvprm::launch_attn_back(a, s), "attention backward");
      if (l == 0) break;   // below layer 0 lies only the verify token's embedding
      // QKV projection: [dq; dk; dv] before RoPE, dx1 = W_qkv^T [...], dh of the layer below
      CK(kvprm::launch_rope_back(g.dq, g.dks, g.dvs, ctx->rope, n, m.n_q, m.n_kv, m.hd, g.ghi, g.glo, s), "RoPE backward");
      CK(gemm(&g.tm_qkv[l], m.d, m.qkv_rows, &g.tm_qkv_hi, &g.tm_qkv_lo, g.tmp), "W_qkv^T product");
      CK(kvprm::launch_rms_back(sv.hout + (l - 1) * Bm * m.d, nullptr, ctx->attn_norm[l], g.tmp, g.dh, n, m.d, m.eps,
                                g.dh, g.ghi, g.glo, s),
         "pre-attention RMSNorm backward");
    }
    return KVPRM_OK;
  };
  if (!ctx->use_graph || ctx->profile) {   // eager (profiled calls time each launch)
    Enq E{ctx, st, ctx->use_pdl && !ctx->profile, ctx->profile, &ctx->live_marks};
    if ((rc = enqueue(st, E))) return rc;
    if (ctx->profile) {
      CK(cudaStreamSynchronize(st), "cudaStreamSynchronize(profile)");
      if ((rc = accumulate_marks(ctx, ctx->live_marks, true))) return rc;
    }
    return KVPRM_OK;
  }
  // the graph of this call: everything its launches take by value or by address
  const std::vector<int64_t> key = {
      n, P.n_pad, P.attn_ctas, ctx->work_host.n_tc_ctas, ctx->work_host.tc_concurrent ? 1 : 0,
      ctx->work_host.fuse_cs, ctx->work_host.n_tc > 0 ? 1 : 0, ctx->work_host.n_ctas, ctx->debug_flags,
      ctx->use_pdl ? 1 : 0, ctx->trace ? 1 : 0, ctx->layer_waits ? 1 : 0, ctx->as.layer_pages,
      reinterpret_cast<int64_t>(kv_pages), n_pages, reinterpret_cast<int64_t>(grad),
      static_cast<int64_t>(units.size()), n_shared, static_cast<int64_t>(lists.size()),
      reinterpret_cast<int64_t>(g.units), reinterpret_cast<int64_t>(g.lists), reinterpret_cast<int64_t>(g.shared),
      ctx->grad_cuda_cores ? 1 : 0, reinterpret_cast<int64_t>(ctx->pool_ptr)};
  if (!(g.gexec && key == g.gkey)) {
    if (g.gexec) cudaGraphExecDestroy(g.gexec);
    g.gexec = nullptr;
    g.gkey.clear();
    CK(cudaStreamBeginCapture(ctx->cap_stream, cudaStreamCaptureModeThreadLocal), "cudaStreamBeginCapture(gradient)");
    Enq E{ctx, ctx->cap_stream, ctx->use_pdl, false, &g.marks};
    E.capturing = true;
    rc = enqueue(ctx->cap_stream, E);
    cudaGraph_t graph = nullptr;
    cudaError_t e = cudaStreamEndCapture(ctx->cap_stream, &graph);
    if (rc) {
      if (graph) cudaGraphDestroy(graph);
      return rc;
    }
    if (e != cudaSuccess) return cuda_fail(ctx, e, "cudaStreamEndCapture(gradient)");
    e = cudaGraphInstantiate(&g.gexec, graph, 0);
    cudaGraphDestroy(graph);
    if (e != cudaSuccess) {
      g.gexec = nullptr;
      return cuda_fail(ctx, e, "cudaGraphInstantiate(gradient)");
    }
    g.gkey = key;
  }
  CK(cudaGraphLaunch(g.gexec, st), "cudaGraphLaunch(gradient)");
  return KVPRM_OK;
}

bool env_off(const char* name) {
  const char* v = std::getenv(name);
  return v && v[0] == '1';
}

}  // namespace

// ======================================================================== C ABI
extern "C" {

int kvprm_create(const kvprm_config* cfg, const kvprm_weights* w, kvprm_ctx** out) {
  if (!out) return KVPRM_EINVAL;
  *out = nullptr;
  if (!cfg || !w) return KVPRM_EINVAL;
  const kvprm_config& c = *cfg;
  if (c.n_layers < 1 || c.d_model < 64 || c.n_q_heads < 1 || c.n_kv_heads < 1 || c.d_ff < 64) return KVPRM_EINVAL;
  if (c.page_size != 16) return KVPRM_EUNSUPPORTED;
  if (c.head_dim != 64 && c.head_dim != 128) return KVPRM_EUNSUPPORTED;
  if (c.n_q_heads % c.n_kv_heads != 0) return KVPRM_EINVAL;
  if (c.n_q_heads / c.n_kv_heads > 16) return KVPRM_EUNSUPPORTED;
  if (c.d_model % 64 || c.d_ff % 64 || (c.n_q_heads * c.head_dim) % 64) return KVPRM_EUNSUPPORTED;
  if (c.max_candidates < 1 || c.max_candidates > 256) return KVPRM_ECAPACITY;
  if (c.max_blocks_per_seq < 1) return KVPRM_EINVAL;
  if (!(c.rms_eps >= 0.f) || !(c.rope_base > 0.f)) return KVPRM_EINVAL;
  if (c.qk_norm != 0 && c.qk_norm != 1) return KVPRM_EINVAL;
  if (c.qk_norm) {
    if (!w->q_norm || !w->k_norm) return KVPRM_EINVAL;
    for (int l = 0; l < c.n_layers; ++l)
      if (!w->q_norm[l] || !w->k_norm[l]) return KVPRM_EINVAL;
  }
  if (!w->embed_verify || !w->final_norm || !w->w_plus || !w->w_minus || !w->attn_norm || !w->w_qkv || !w->w_o ||
      !w->mlp_norm || !w->w_gate_up || !w->w_down)
    return KVPRM_EINVAL;
  for (int l = 0; l < c.n_layers; ++l)
    if (!w->attn_norm[l] || !w->w_qkv[l] || !w->w_o[l] || !w->mlp_norm[l] || !w->w_gate_up[l] || !w->w_down[l])
      return KVPRM_EINVAL;
  for (int l = 0; l < c.n_layers; ++l)
    if (!aligned16(w->w_qkv[l]) || !aligned16(w->w_o[l]) || !aligned16(w->w_gate_up[l]) || !aligned16(w->w_down[l]))
      return KVPRM_EINVAL;

  kvprm_ctx* ctx = new (std::nothrow) kvprm_ctx();
  if (!ctx) return KVPRM_ENOMEM;
  ctx->cfg = c;
  int rc = KVPRM_OK;
#define CREATE_CK(call)             \
  do {                              \
    if ((rc = (call)) != KVPRM_OK) { \
      free_ctx(ctx);                \
      return rc;                    \
    }                               \
  } while (0)
  auto cu = [&](cudaError_t e, const char* what) { return e == cudaSuccess ? KVPRM_OK : cuda_fail(ctx, e, what); };
  CREATE_CK(cu(cudaGetDevice(&ctx->device), "cudaGetDevice"));
  CREATE_CK(cu(cudaDeviceGetAttribute(&ctx->num_sms, cudaDevAttrMultiProcessorCount, ctx->device), "sm count"));
  {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    CREATE_CK(cu(cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q),
                 "cudaGetDriverEntryPointByVersion"));
    if (!fn || q != cudaDriverEntryPointSuccess) {
      free_ctx(ctx);
      return KVPRM_ECUDA;
    }
    ctx->encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  }
  CREATE_CK(cu(kvprm::gemm_configure(), "gemm_configure"));
  CREATE_CK(cu(kvprm::attention_configure(), "attention_configure"));
  CREATE_CK(cu(kvprm::grad_configure(), "grad_configure"));

  ModelDims& m = ctx->md;
  m.d = c.d_model;
  m.n_q = c.n_q_heads;
  m.n_kv = c.n_kv_heads;
  m.hd = c.head_dim;
  m.ff = c.d_ff;
  m.qkv_rows = (c.n_q_heads + 2 * c.n_kv_heads) * c.head_dim;
  m.eps = c.rms_eps;
  AttnShape& as = ctx->as;
  as.n_q = m.n_q;
  as.n_kv = m.n_kv;
  as.hd = m.hd;
  as.group = m.n_q / m.n_kv;
  as.max_blocks = c.max_blocks_per_seq;
  as.layer_pages = 0;   // set per call from the pool

  ctx->embed = static_cast<const bf16*>(w->embed_verify);
  ctx->final_norm = static_cast<const bf16*>(w->final_norm);
  ctx->w_plus = static_cast<const bf16*>(w->w_plus);
  ctx->w_minus = static_cast<const bf16*>(w->w_minus);
  const int NL = c.n_layers;
  ctx->attn_norm.resize(NL);
  ctx->mlp_norm.resize(NL);
  ctx->tm_qkv.resize(NL);
  ctx->tm_o.resize(NL);
  ctx->tm_gu.resize(NL);
  ctx->tm_down.resize(NL);
  if (c.qk_norm) {
    ctx->q_norm.resize(NL);
    ctx->k_norm.resize(NL);
    for (int l = 0; l < NL; ++l) {
      ctx->q_norm[l] = static_cast<const bf16*>(w->q_norm[l]);
      ctx->k_norm[l] = static_cast<const bf16*>(w->k_norm[l]);
    }
  }
  ctx->w_qkv_src.assign(w->w_qkv, w->w_qkv + NL);
  ctx->w_o_src.assign(w->w_o, w->w_o + NL);
  ctx->w_gu_src.assign(w->w_gate_up, w->w_gate_up + NL);
  ctx->w_down_src.assign(w->w_down, w->w_down + NL);
  for (int l = 0; l < NL; ++l) {
    ctx->attn_norm[l] = static_cast<const bf16*>(w->attn_norm[l]);
    ctx->mlp_norm[l] = static_cast<const bf16*>(w->mlp_norm[l]);
    CREATE_CK(make_map(ctx, &ctx->tm_qkv[l], w->w_qkv[l], m.d, m.qkv_rows, 64, 128, "w_qkv"));
    CREATE_CK(make_map(ctx, &ctx->tm_o[l], w->w_o[l], static_cast<uint64_t>(m.n_q) * m.hd, m.d, 64, 128, "w_o"));
    CREATE_CK(make_map(ctx, &ctx->tm_gu[l], w->w_gate_up[l], m.d, 2 * static_cast<uint64_t>(m.ff), 64, 64,
                       "w_gate_up"));
    CREATE_CK(make_map(ctx, &ctx->tm_down[l], w->w_down[l], m.ff, m.d, 64, 128, "w_down"));
  }

  const int Bmax = c.max_candidates;
  ctx->npad_max = (Bmax + 15) / 16 * 16;
  const size_t Bp = ctx->npad_max;
  CREATE_CK(dalloc(ctx, &ctx->h, static_cast<size_t>(Bmax) * m.d, "h"));
  CREATE_CK(dalloc(ctx, &ctx->xhi, Bp * m.d, "x_hi"));
  CREATE_CK(dalloc(ctx, &ctx->xlo, Bp * m.d, "x_lo"));
  CREATE_CK(dalloc(ctx, &ctx->ohi, Bp * m.n_q * m.hd, "o_hi"));
  CREATE_CK(dalloc(ctx, &ctx->olo, Bp * m.n_q * m.hd, "o_lo"));
  CREATE_CK(dalloc(ctx, &ctx->ahi, Bp * m.ff, "a_hi"));
  CREATE_CK(dalloc(ctx, &ctx->alo, Bp * m.ff, "a_lo"));
  ctx->d_tiles = (m.d + 127) / 128;
  CREATE_CK(dalloc(ctx, &ctx->sumsq, static_cast<size_t>(ctx->d_tiles) * Bmax, "tile sums of squares"));
  CREATE_CK(dalloc(ctx, &ctx->q, static_cast<size_t>(Bmax) * m.n_q * m.hd, "q"));
  CREATE_CK(dalloc(ctx, &ctx->qhi, static_cast<size_t>(Bmax) * m.n_q * m.hd, "q_hi"));
  CREATE_CK(dalloc(ctx, &ctx->qlo, static_cast<size_t>(Bmax) * m.n_q * m.hd, "q_lo"));
  CREATE_CK(dalloc(ctx, &ctx->kself, static_cast<size_t>(Bmax) * m.n_kv * m.hd, "k_self"));
  CREATE_CK(dalloc(ctx, &ctx->vself, static_cast<size_t>(Bmax) * m.n_kv * m.hd, "v_self"));
  ctx->slot_cap = kvprm::attn_slot_capacity(Bmax, m.n_kv, ctx->num_sms);
  const size_t group = static_cast<size_t>(m.n_q / m.n_kv);
  CREATE_CK(dalloc(ctx, &ctx->apart_o, ctx->slot_cap * group * m.hd, "attn partials"));
  CREATE_CK(dalloc(ctx, &ctx->apart_ml, ctx->slot_cap * group * 2, "attn stats"));
  CREATE_CK(dalloc(ctx, &ctx->rope, static_cast<size_t>(Bmax) * (m.hd / 2), "rope table"));
  {
    const size_t tbl = static_cast<size_t>(Bmax) * (1 + c.max_blocks_per_seq);
    auto al8 = [](size_t x) { return (x + 7) & ~static_cast<size_t>(7); };
    // private runs need at most Bmax * n_kv + n_ctas segments, Bmax * max_blocks
    // pages and no candidate lists; sharing plans beyond these fall back to them
    const size_t bkv = static_cast<size_t>(Bmax) * m.n_kv;
    ctx->cap_segs = 8 * bkv + 4 * static_cast<size_t>(ctx->num_sms);
    ctx->cap_pages = static_cast<size_t>(Bmax) * c.max_blocks_per_seq;
    ctx->cap_cands = static_cast<size_t>(Bmax) * c.max_blocks_per_seq;
    ctx->off_segs = al8(tbl);
    ctx->off_cta = al8(ctx->off_segs + ctx->cap_segs * (sizeof(kvprm::AttnSeg) / sizeof(int32_t)));
    ctx->off_pages = al8(ctx->off_cta + ctx->num_sms + 1);
    ctx->off_cands = al8(ctx->off_pages + ctx->cap_pages);
    ctx->off_slots = al8(ctx->off_cands + ctx->cap_cands);
    ctx->off_base = al8(ctx->off_slots + ctx->slot_cap);
    ctx->off_nslots = al8(ctx->off_base + bkv);
    ctx->off_tc_cta = al8(ctx->off_nslots + bkv);
    ctx->tables_ints = al8(ctx->off_tc_cta + ctx->num_sms + 1);
  }
  CREATE_CK(dalloc(ctx, &ctx->tables_d, ctx->tables_ints, "tables and attention work"));
  CREATE_CK(dalloc(ctx, &ctx->rewards_d, static_cast<size_t>(Bmax), "rewards"));
  CREATE_CK(dalloc(ctx, &ctx->err_d, 1, "err"));
  CREATE_CK(dalloc(ctx, &ctx->dummy_pool, static_cast<size_t>(NL) * 2 * m.n_kv * 16 * m.hd, "dummy pool"));
  CREATE_CK(dalloc(ctx, &ctx->probe_flag, 1, "wait probe flag"));
  {
    if (!take_budget(sizeof(int32_t) * ctx->tables_ints + sizeof(float) * Bmax + sizeof(int))) {
      free_ctx(ctx);
      return KVPRM_ENOMEM;
    }
    cudaError_t e =
        cudaMallocHost(reinterpret_cast<void**>(&ctx->staging), sizeof(int32_t) * ctx->tables_ints);
    if (e == cudaSuccess) e = cudaMallocHost(reinterpret_cast<void**>(&ctx->h_rewards), sizeof(float) * Bmax);
    if (e == cudaSuccess) e = cudaMallocHost(reinterpret_cast<void**>(&ctx->h_err), sizeof(int));
    if (e != cudaSuccess) {
      cudaGetLastError();
      free_ctx(ctx);
      return KVPRM_ENOMEM;
    }
  }
  CREATE_CK(cu(cudaEventCreateWithFlags(&ctx->staging_ev, cudaEventDisableTiming), "cudaEventCreate"));
  CREATE_CK(cu(cudaStreamCreateWithFlags(&ctx->cap_stream, cudaStreamNonBlocking), "cudaStreamCreate"));
  CREATE_CK(cu(cudaStreamCreateWithFlags(&ctx->side_stream, cudaStreamNonBlocking), "cudaStreamCreate"));
  CREATE_CK(cu(cudaEventCreateWithFlags(&ctx->ev_fork, cudaEventDisableTiming), "cudaEventCreate"));
  CREATE_CK(cu(cudaEventCreateWithFlags(&ctx->ev_join, cudaEventDisableTiming), "cudaEventCreate"));
  CREATE_CK(cu(cudaStreamCreateWithFlags(&ctx->copy_stream, cudaStreamNonBlocking), "cudaStreamCreate"));
  ctx->layer_ready.assign(static_cast<size_t>(c.n_layers), nullptr);
  for (cudaEvent_t& ev : ctx->layer_ready)
    CREATE_CK(cu(cudaEventCreateWithFlags(&ev, cudaEventDisableTiming), "cudaEventCreate"));
  CREATE_CK(cu(cudaEventCreateWithFlags(&ctx->pool_free, cudaEventDisableTiming), "cudaEventCreate"));
  ctx->use_graph = !env_off("KVPRM_NO_GRAPH");
  ctx->use_pdl = !env_off("KVPRM_NO_PDL");
  ctx->grad_cuda_cores = env_off("KVPRM_GRAD_CUDA_CORES");
  // shared pages: on the tensor cores at head_dim 128, else one warp per candidate
  ctx->fuse_combine = !env_off("KVPRM_NO_FUSED_COMBINE");
  ctx->share_mode = env_off("KVPRM_NO_SHARING")
                        ? 0
                        : ((c.head_dim == 128 && !env_off("KVPRM_NO_TC_SHARING")) ? (env_off("KVPRM_TC_SERIAL") ? 2 : 3)
                                                                                   : 1);
  CREATE_CK(cu(cudaDeviceSynchronize(), "cudaDeviceSynchronize(create)"));
#undef CREATE_CK
  *out = ctx;
  return KVPRM_OK;
}

int kvprm_set_readout_depth(kvprm_ctx* ctx, int32_t depth) {
  if (!ctx) return KVPRM_EINVAL;
  if (depth < 1 || depth > kvprm::kMaxReadoutDepth)
    return fail(ctx, KVPRM_EINVAL, "readout depth %d outside [1, %d]", depth, kvprm::kMaxReadoutDepth);
  if (depth != ctx->depth) drop_graph(ctx);
  ctx->depth = depth;
  return KVPRM_OK;
}

int kvprm_set_lora(kvprm_ctx* ctx, int32_t rank, float scale, const kvprm_lora* lora) {
  if (!ctx) return KVPRM_EINVAL;
  if (rank == 0) {   // back to the merged weights alone
    if (ctx->lora_rank != 0) drop_graph(ctx);
    ctx->lora_rank = 0;
    ctx->lora_scale = 0.f;
    return KVPRM_OK;
  }
  if (rank < 64 || rank > 1024 || rank % 64)
    return fail(ctx, KVPRM_EINVAL, "adapter rank %d: a multiple of 64 in [64, 1024], or 0", rank);
  if (!lora) return fail(ctx, KVPRM_EINVAL, "kvprm_lora is NULL");
  if (!std::isfinite(scale)) return fail(ctx, KVPRM_EINVAL, "adapter scale is not finite");
  const ModelDims& m = ctx->md;
  const int NL = ctx->cfg.n_layers;
  const void* const* a_of[4] = {lora->a_qkv, lora->a_o, lora->a_gate_up, lora->a_down};
  const void* const* b_of[4] = {lora->b_qkv, lora->b_o, lora->b_gate_up, lora->b_down};
  const uint64_t in_of[4] = {static_cast<uint64_t>(m.d), static_cast<uint64_t>(m.n_q) * m.hd,
                             static_cast<uint64_t>(m.d), static_cast<uint64_t>(m.ff)};
  const uint64_t out_of[4] = {static_cast<uint64_t>(m.qkv_rows), static_cast<uint64_t>(m.d),
                              2 * static_cast<uint64_t>(m.ff), static_cast<uint64_t>(m.d)};
  static const char* nm[4] = {"qkv", "o", "gate_up", "down"};
  for (int j = 0; j < 4; ++j) {
    if (!a_of[j] || !b_of[j]) return fail(ctx, KVPRM_EINVAL, "adapter factor arrays of %s are NULL", nm[j]);
    for (int l = 0; l < NL; ++l)
      if (!a_of[j][l] || !b_of[j][l] || !aligned16(a_of[j][l]) || !aligned16(b_of[j][l]))
        return fail(ctx, KVPRM_EINVAL, "adapter factor of %s, layer %d, is NULL or not 16-byte aligned", nm[j], l);
  }
  // every map first, so that a failure leaves the context as it was
  std::vector<CUtensorMap> la[4], lb[4];
  int rc;
  for (int j = 0; j < 4; ++j) {
    la[j].resize(NL);
    lb[j].resize(NL);
    for (int l = 0; l < NL; ++l) {
      // A [r][in]: 128-row tiles of the A x launch; B [out][r]: the projection's own weight tile rows
      if ((rc = make_map(ctx, &la[j][l], a_of[j][l], in_of[j], static_cast<uint64_t>(rank), 64, 128, "adapter A")))
        return rc;
      if ((rc = make_map(ctx, &lb[j][l], b_of[j][l], static_cast<uint64_t>(rank), out_of[j], 64, j == 2 ? 64 : 128,
                         "adapter B")))
        return rc;
    }
  }
  const size_t need = static_cast<size_t>(ctx->npad_max) * rank;
  if (need > ctx->t_cap) {
    bf16 *th = nullptr, *tl = nullptr;
    if ((rc = dalloc(ctx, &th, need, "adapter t_hi"))) return rc;
    if ((rc = dalloc(ctx, &tl, need, "adapter t_lo"))) {
      cudaFree(th);
      return rc;
    }
    CK(cudaDeviceSynchronize(), "cudaDeviceSynchronize(adapter buffers)");
    cudaFree(ctx->thi);
    cudaFree(ctx->tlo);
    ctx->thi = th;
    ctx->tlo = tl;
    ctx->t_cap = need;
  } else if (rank != ctx->lora_rank) {
    // padding rows of t (candidates >= n) are read as K-extension columns: keep them zero
    CK(cudaMemset(ctx->thi, 0, sizeof(bf16) * ctx->t_cap), "cudaMemset(t_hi)");
    CK(cudaMemset(ctx->tlo, 0, sizeof(bf16) * ctx->t_cap), "cudaMemset(t_lo)");
  }
  for (int j = 0; j < 4; ++j) {
    ctx->tm_la[j] = std::move(la[j]);
    ctx->tm_lb[j] = std::move(lb[j]);
  }
  ctx->lora_rank = rank;
  ctx->lora_scale = scale;
  ctx->tm_t_npad = -1;
  drop_graph(ctx);
  return KVPRM_OK;
}

void kvprm_destroy(kvprm_ctx* ctx) {
  if (!ctx) return;
  cudaDeviceSynchronize();
  free_ctx(ctx);
}

const char* kvprm_last_error(const kvprm_ctx* ctx) { return ctx ? ctx->last_error.c_str() : ""; }

int kvprm_score_async(kvprm_ctx* ctx, const void* kv_pages, int64_t n_pages, const int32_t* block_table,
                      const int32_t* seq_lens, int32_t n, float* d_rewards, void* stream) {
  if (!ctx) return KVPRM_EINVAL;
  if (n > 0 && !d_rewards) return fail(ctx, KVPRM_EINVAL, "d_rewards is NULL");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  int rc = score_device(ctx, kv_pages, n_pages, block_table, seq_lens, n, st);
  if (rc || n == 0) return rc;
  CK(cudaMemcpyAsync(d_rewards, ctx->rewards_d, sizeof(float) * n, cudaMemcpyDeviceToDevice, st),
     "cudaMemcpyAsync(d_rewards)");
  return KVPRM_OK;
}

int kvprm_score(kvprm_ctx* ctx, const void* kv_pages, int64_t n_pages, const int32_t* block_table,
                const int32_t* seq_lens, int32_t n, float* rewards, void* stream) {
  if (!ctx) return KVPRM_EINVAL;
  if (n > 0 && !rewards) return fail(ctx, KVPRM_EINVAL, "rewards is NULL");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  int rc = score_device(ctx, kv_pages, n_pages, block_table, seq_lens, n, st);
  if (rc) return rc;
  return finish_blocking(ctx, n, rewards, st);
}

int kvprm_score_host(kvprm_ctx* ctx, const void* h_kv_pages, int64_t n_pages, const int32_t* block_table,
                     const int32_t* seq_lens, int32_t n, float* rewards, void* stream) {
  if (!ctx) return KVPRM_EINVAL;
  if (n > 0 && !rewards) return fail(ctx, KVPRM_EINVAL, "rewards is NULL");
  if (n_pages < 0) return fail(ctx, KVPRM_EINVAL, "n_pages is negative");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const size_t bytes = static_cast<size_t>(ctx->cfg.n_layers) * n_pages * 2 * ctx->cfg.n_kv_heads * 16 *
                       ctx->cfg.head_dim * sizeof(bf16);
  const void* pool = nullptr;
  if (bytes > 0) {
    if (!h_kv_pages) return fail(ctx, KVPRM_EINVAL, "h_kv_pages is NULL");
    if (bytes > ctx->dev_pool_bytes) {
      CK(cudaStreamSynchronize(st), "cudaStreamSynchronize(pool grow)");
      cudaFree(ctx->dev_pool);
      ctx->dev_pool = nullptr;
      ctx->dev_pool_bytes = 0;
      drop_graph(ctx);
      ctx->pool_ptr = nullptr;
      if (!take_budget(bytes)) return fail(ctx, KVPRM_ENOMEM, "device pool of %zu bytes exceeds the allocation budget", bytes);
      cudaError_t e = cudaMalloc(&ctx->dev_pool, bytes);
      if (e != cudaSuccess) {
        cudaGetLastError();
        return fail(ctx, KVPRM_ENOMEM, "cudaMalloc(device pool, %zu bytes) failed", bytes);
      }
      ctx->dev_pool_bytes = bytes;
    }
    pool = ctx->dev_pool;
  }
  ctx->layer_waits = bytes > 0;
  ctx->host_pool = h_kv_pages;
  ctx->host_pool_bytes = bytes;
  int rc = score_device(ctx, pool, n_pages, block_table, seq_lens, n, st);
  ctx->layer_waits = false;
  ctx->host_pool = nullptr;
  ctx->host_pool_bytes = 0;
  if (rc) {
    // a call that failed after its cache copy was enqueued still returns only once nothing reads the
    // caller's host buffer any more
    if (bytes > 0 && cudaStreamSynchronize(ctx->copy_stream) != cudaSuccess) cudaGetLastError();
    return rc;
  }
  return finish_blocking(ctx, n, rewards, st);
}

int kvprm_attention(kvprm_ctx* ctx, const void* kv_layer, int64_t n_pages, const int32_t* block_table,
                    const int32_t* seq_lens, int32_t n, const void* q, const void* k_self, const void* v_self,
                    float* out, void* stream) {
  if (!ctx) return KVPRM_EINVAL;
  int max_pages = 0;
  int rc = validate_tables(ctx, n_pages, block_table, seq_lens, n, &max_pages);
  if (rc) return rc;
  if (n == 0) return KVPRM_OK;
  if (!q || !k_self || !v_self || !out) return fail(ctx, KVPRM_EINVAL, "q, k_self, v_self and out must be non-NULL");
  if (!aligned16(q) || !aligned16(k_self) || !aligned16(v_self))
    return fail(ctx, KVPRM_EINVAL, "q, k_self and v_self must be 16-byte aligned");
  const kvprm::HiLo Q{ctx->qhi, ctx->qlo};
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const void* pool = kv_layer;
  int64_t pages = n_pages;
  if (max_pages == 0) {
    pool = ctx->dummy_pool;
    pages = 1;
  } else {
    if (!kv_layer) return fail(ctx, KVPRM_EINVAL, "kv_layer is NULL");
    if (!aligned16(kv_layer)) return fail(ctx, KVPRM_EINVAL, "kv_layer is not 16-byte aligned");
  }
  if ((rc = ensure_pool_map(ctx, pool, pages, 1))) return rc;
  if ((rc = plan_work(ctx, block_table, seq_lens, n, true))) return rc;
  if ((rc = upload_tables(ctx, block_table, seq_lens, n, st))) return rc;
  AttnShape as = ctx->as;
  as.layer_pages = pages;
  Enq E{ctx, st, false, ctx->profile, &ctx->live_marks};
  LAUNCH(KVPRM_PROF_FUSED,
         kvprm::launch_split_hilo(static_cast<const float*>(q), static_cast<int64_t>(n) * ctx->md.n_q * ctx->md.hd, Q,
                                  st),
         "split_hilo");
  const kvprm::AttnMerge mg{static_cast<const float*>(q), static_cast<const float*>(k_self),
                            static_cast<const float*>(v_self), ctx->ohi, ctx->olo, out, nullptr};
  const kvprm::AttnWork wk = device_work(ctx);
  if ((rc = enqueue_attention(ctx, E, as, wk, 0, Q, mg, false))) return rc;
  if (wk.fuse_cs == 0)
    LAUNCH(KVPRM_PROF_COMBINE,
           kvprm::launch_attn_combine(as, wk, n, ctx->apart_o, ctx->apart_ml, mg, st, false, TS,
                                      (ctx->debug_flags & 64) != 0),
           "attn_combine");
  ctx->last_n = n;
  ctx->last_stream = st;
  if (ctx->profile) {
    CK(cudaStreamSynchronize(st), "cudaStreamSynchronize(profile)");
    if ((rc = accumulate_marks(ctx, ctx->live_marks, true))) return rc;
  }
  // the next full score call must rebuild its pool map (this call pointed it at one layer)
  ctx->pool_ptr = nullptr;
  drop_graph(ctx);
  return KVPRM_OK;
}

int kvprm_projection(kvprm_ctx* ctx, const void* W, int32_t M, int32_t K, const void* X, int32_t n, float* Y,
                     void* stream) {
  if (!ctx) return KVPRM_EINVAL;
  if (!W || !X || !Y) return fail(ctx, KVPRM_EINVAL, "W, X and Y must be non-NULL");
  if (M < 1 || K < 8 || K % 8) return fail(ctx, KVPRM_EINVAL, "bad projection shape M=%d K=%d", M, K);
  if (n < 1 || n > ctx->cfg.max_candidates)
    return fail(ctx, KVPRM_ECAPACITY, "n = %d outside [1, max_candidates = %d]", n, ctx->cfg.max_candidates);
  if (!aligned16(W) || !aligned16(X)) return fail(ctx, KVPRM_EINVAL, "W and X must be 16-byte aligned");
  const int n_pad = (n + 15) / 16 * 16;
  const GemmPlan g = kvprm::plan_gemm(M, K, n_pad, ctx->num_sms, false, false);
  CUtensorMap tw, tx;
  int rc;
  if ((rc = make_map(ctx, &tw, W, K, M, 64, 128, "W"))) return rc;
  if ((rc = make_map(ctx, &tx, X, K, n, 64, n_pad, "X"))) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  kvprm::GemmEpilogue ep;
  ep.mode = kvprm::GemmEpilogue::PLAIN;
  ep.M = M;
  ep.n_valid = n;
  ep.out = Y;
  Enq E{ctx, st, false, ctx->profile, &ctx->live_marks};
  LAUNCH(KVPRM_PROF_GEMM_QKV, kvprm::launch_gemm(g, &tw, &tx, nullptr, ep, n_pad, ctx->err_d, st, false), "gemm");
  ctx->last_stream = st;
  if (ctx->profile) {
    CK(cudaStreamSynchronize(st), "cudaStreamSynchronize(profile)");
    if ((rc = accumulate_marks(ctx, ctx->live_marks, true))) return rc;
  }
  return KVPRM_OK;
}

int kvprm_debug_hidden(kvprm_ctx* ctx, float* d_out) {
  if (!ctx || !d_out) return KVPRM_EINVAL;
  CK(cudaMemcpyAsync(d_out, ctx->h, sizeof(float) * ctx->last_n * ctx->md.d, cudaMemcpyDeviceToDevice,
                     ctx->last_stream),
     "cudaMemcpyAsync(hidden)");
  return KVPRM_OK;
}

int kvprm_set_debug(kvprm_ctx* ctx, int flags) {
  if (!ctx) return KVPRM_EINVAL;
  if ((flags & 1) && !ctx->dbg) {
    const size_t count = static_cast<size_t>(ctx->cfg.n_layers) * ctx->cfg.max_candidates * ctx->md.n_q * ctx->md.hd;
    int rc = dalloc(ctx, &ctx->dbg, count, "debug capture");
    if (rc) return rc;
  }
  const size_t NB = static_cast<size_t>(ctx->cfg.n_layers) * ctx->cfg.max_candidates;
  if ((flags & 2) && !ctx->dbg_q) {
    int rc = dalloc(ctx, &ctx->dbg_q, NB * ctx->md.n_q * ctx->md.hd, "debug q");
    if (!rc) rc = dalloc(ctx, &ctx->dbg_k, NB * ctx->md.n_kv * ctx->md.hd, "debug k");
    if (!rc) rc = dalloc(ctx, &ctx->dbg_v, NB * ctx->md.n_kv * ctx->md.hd, "debug v");
    if (rc) return rc;
  }
  if ((flags & 4) && !ctx->dbg_h) {
    int rc = dalloc(ctx, &ctx->dbg_h, NB * ctx->md.d, "debug h");
    if (rc) return rc;
  }
  if ((flags & 32) && !ctx->tc_prof) {
    int rc = dalloc(ctx, &ctx->tc_prof, kvprm::kTcEventLog + static_cast<size_t>(ctx->num_sms) * 16,
                    "tensor-core attention profile");
    if (rc) return rc;
  }
  ctx->debug_flags = flags;
  return KVPRM_OK;
}

int kvprm_debug_layers(kvprm_ctx* ctx, int which, void* d_out) {
  if (!ctx || !d_out) return KVPRM_EINVAL;
  const size_t L = static_cast<size_t>(ctx->cfg.n_layers) * ctx->last_n;
  const void* src = nullptr;
  size_t bytes = 0;
  if (which >= 1 && which <= 3) {
    if (!(ctx->debug_flags & 2)) return fail(ctx, KVPRM_EINVAL, "q/k/v capture (flag 2) is not enabled");
    src = which == 1 ? ctx->dbg_q : (which == 2 ? ctx->dbg_k : ctx->dbg_v);
    bytes = L * (which == 1 ? ctx->md.n_q : ctx->md.n_kv) * ctx->md.hd * 4;
  } else if (which == 4) {
    if (!(ctx->debug_flags & 4)) return fail(ctx, KVPRM_EINVAL, "hidden-state capture (flag 4) is not enabled");
    src = ctx->dbg_h;
    bytes = L * ctx->md.d * 4;
  } else if (which == 5) {
    if (!(ctx->debug_flags & 32) || !ctx->tc_prof)
      return fail(ctx, KVPRM_EINVAL, "tensor-core attention profile (flag 32) is not enabled");
    src = ctx->tc_prof;
    bytes = (kvprm::kTcEventLog + static_cast<size_t>(ctx->num_sms) * 16) * sizeof(unsigned long long);
  } else {
    return fail(ctx, KVPRM_EINVAL, "unknown capture %d", which);
  }
  CK(cudaMemcpyAsync(d_out, src, bytes, cudaMemcpyDeviceToDevice, ctx->last_stream), "cudaMemcpyAsync(debug)");
  return KVPRM_OK;
}

int kvprm_debug_attn_out(kvprm_ctx* ctx, float* d_out) {
  if (!ctx || !d_out) return KVPRM_EINVAL;
  if (!(ctx->debug_flags & 1) || !ctx->dbg) return fail(ctx, KVPRM_EINVAL, "debug capture is not enabled");
  const size_t count = static_cast<size_t>(ctx->cfg.n_layers) * ctx->last_n * ctx->md.n_q * ctx->md.hd;
  CK(cudaMemcpyAsync(d_out, ctx->dbg, count * sizeof(float), cudaMemcpyDeviceToDevice, ctx->last_stream),
     "cudaMemcpyAsync(debug)");
  return KVPRM_OK;
}

int kvprm_resolve(kvprm_ctx* ctx, int32_t b, int64_t* phys_row) {
  if (!ctx || !phys_row) return KVPRM_EINVAL;
  if (b < 0 || b >= ctx->last_n) return fail(ctx, KVPRM_EINVAL, "candidate %d not in the last call", b);
  cudaStream_t st = ctx->last_stream;
  int32_t L = 0;
  CK(cudaMemcpyAsync(&L, ctx->tables_d + b, sizeof(int32_t), cudaMemcpyDeviceToHost, st), "cudaMemcpy(len)");
  CK(cudaStreamSynchronize(st), "cudaStreamSynchronize");
  if (L == 0) return KVPRM_OK;
  int64_t* d = nullptr;
  CK(cudaMalloc(&d, sizeof(int64_t) * L), "cudaMalloc(resolve)");
  cudaError_t e = kvprm::launch_resolve(ctx->tables_d + ctx->cfg.max_candidates, ctx->tables_d,
                                        ctx->cfg.max_blocks_per_seq, b, d, st);
  if (e == cudaSuccess) e = cudaMemcpyAsync(phys_row, d, sizeof(int64_t) * L, cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  cudaFree(d);
  if (e != cudaSuccess) return cuda_fail(ctx, e, "resolve");
  return KVPRM_OK;
}

int kvprm_plan_projection(int32_t M, int32_t K, int32_t n_pad, int32_t num_sms, int32_t has_lo, int32_t gate_up,
                          kvprm_projection_plan* out) {
  if (!out || M < 1 || K < 1 || num_sms < 1 || n_pad < 16 || n_pad % 16) return KVPRM_EINVAL;
  if (n_pad > 256) return KVPRM_EUNSUPPORTED;   // a context holds at most 256 candidates
  const GemmPlan g = kvprm::plan_gemm(M, K, n_pad, num_sms, has_lo != 0, gate_up != 0);
  out->m_tiles = g.m_tiles;
  out->k_tiles = g.k_tiles;
  out->kt_per_split = g.kt_per_split;
  out->cluster = g.cluster;
  out->tiles_per_cta = g.mt;
  out->stages = g.stages;
  out->tmem_cols = static_cast<int32_t>(g.tmem_cols);
  out->smem_bytes = static_cast<int64_t>(g.smem_bytes);
  out->threads = g.threads;
  return KVPRM_OK;
}

int kvprm_plan_attention(const int32_t* block_table, int32_t max_blocks_per_seq, const int32_t* seq_lens,
                         int32_t n_candidates, int32_t n_kv_heads, int32_t group, int32_t n_ctas, int32_t share,
                         kvprm_attn_plan* plan) {
  if (!plan || n_candidates < 0 || max_blocks_per_seq < 1 || n_kv_heads < 1 || group < 1 || group > 16 ||
      n_ctas < 1)
    return KVPRM_EINVAL;
  if (n_candidates > 0 && (!block_table || !seq_lens)) return KVPRM_EINVAL;
  for (int b = 0; b < n_candidates; ++b)
    if (seq_lens[b] < 0 || static_cast<int64_t>(seq_lens[b]) > static_cast<int64_t>(max_blocks_per_seq) * 16)
      return KVPRM_EINVAL;
  kvprm::AttnWorkHost w;
  const bool fuse = share >= 0 && (share & KVPRM_PLAN_FUSE) != 0;
  share = share < 0 ? 0 : (share & ~KVPRM_PLAN_FUSE);
  if (!(fuse && kvprm::build_attn_work_fused(block_table, seq_lens, n_candidates, max_blocks_per_seq, n_kv_heads,
                                             group, n_ctas, SIZE_MAX, w)) &&
      !kvprm::build_attn_work(block_table, seq_lens, n_candidates, max_blocks_per_seq, n_kv_heads, group, n_ctas,
                              SIZE_MAX, share > 3 ? 3 : share, w))
    return KVPRM_ECAPACITY;
  plan->fuse_cs = w.fuse_cs;
  plan->n_segs = static_cast<int32_t>(w.segs.size());
  plan->n_ctas = w.n_ctas;
  plan->n_pages = static_cast<int32_t>(w.pages.size());
  plan->n_cands = static_cast<int32_t>(w.cands.size());
  plan->n_slot_refs = static_cast<int32_t>(w.slots.size());
  plan->n_slots = w.n_slots;
  plan->n_tc_ctas = w.n_tc_ctas;
  constexpr size_t kSegInts = sizeof(kvprm::AttnSeg) / sizeof(int32_t);
  static_assert(kSegInts == 8, "segment layout");
  auto fits = [](const int32_t* p, int64_t cap, size_t need) { return need == 0 || (p && cap >= static_cast<int64_t>(need)); };
  if (!fits(plan->segs, plan->segs_cap, w.segs.size()) || !fits(plan->cta_seg, plan->cta_cap, w.cta_seg.size()) ||
      !fits(plan->pages, plan->pages_cap, w.pages.size()) || !fits(plan->cands, plan->cands_cap, w.cands.size()) ||
      !fits(plan->slots, plan->slots_cap, w.slots.size()) || !fits(plan->tc_cta, plan->tc_cta_cap, w.tc_cta.size()) ||
      (!w.slot_base.empty() && (!plan->slot_base || !plan->nslots)))
    return KVPRM_ECAPACITY;
  if (!w.segs.empty()) std::memcpy(plan->segs, w.segs.data(), sizeof(kvprm::AttnSeg) * w.segs.size());
  if (!w.cta_seg.empty()) std::memcpy(plan->cta_seg, w.cta_seg.data(), sizeof(int32_t) * w.cta_seg.size());
  if (!w.pages.empty()) std::memcpy(plan->pages, w.pages.data(), sizeof(int32_t) * w.pages.size());
  if (!w.cands.empty()) std::memcpy(plan->cands, w.cands.data(), sizeof(int32_t) * w.cands.size());
  if (!w.slots.empty()) std::memcpy(plan->slots, w.slots.data(), sizeof(int32_t) * w.slots.size());
  if (!w.tc_cta.empty()) std::memcpy(plan->tc_cta, w.tc_cta.data(), sizeof(int32_t) * w.tc_cta.size());
  if (!w.slot_base.empty()) {
    std::memcpy(plan->slot_base, w.slot_base.data(), sizeof(int32_t) * w.slot_base.size());
    std::memcpy(plan->nslots, w.nslots.data(), sizeof(int32_t) * w.nslots.size());
  }
  return KVPRM_OK;
}

int kvprm_score_grad(kvprm_ctx* ctx, const void* kv_pages, int64_t n_pages, const int32_t* block_table,
                     const int32_t* seq_lens, int32_t n_candidates, float* d_grad, float* rewards, void* stream) {
  if (!ctx) return KVPRM_EINVAL;
  if (n_candidates > 0 && !rewards) return fail(ctx, KVPRM_EINVAL, "rewards is NULL");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  int n_ref = 0;
  int rc = score_grad_device(ctx, kv_pages, n_pages, block_table, seq_lens, n_candidates, d_grad, st, &n_ref);
  if (rc) return rc;
  return finish_blocking(ctx, n_candidates, rewards, st);
}

int kvprm_steer(kvprm_ctx* ctx, void* kv_pages, int64_t n_pages, const int32_t* block_table, const int32_t* seq_lens,
                int32_t n_candidates, float eta, int32_t steps, float* p_first, float* p_last, void* stream) {
  if (!ctx) return KVPRM_EINVAL;
  if (steps < 0) return fail(ctx, KVPRM_EINVAL, "steps = %d is negative", steps);
  if (!std::isfinite(eta)) return fail(ctx, KVPRM_EINVAL, "eta is not finite");
  if (n_candidates < 0) return fail(ctx, KVPRM_EINVAL, "n_candidates is negative");
  if (n_pages < 0) return fail(ctx, KVPRM_EINVAL, "n_pages is negative");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (n_candidates == 0) return KVPRM_OK;
  const ModelDims& m = ctx->md;
  const int64_t page_elems = static_cast<int64_t>(2) * m.n_kv * 16 * m.hd;
  const size_t bytes = static_cast<size_t>(ctx->cfg.n_layers) * static_cast<size_t>(n_pages) * page_elems * 4;
  GradState& g = ctx->grad;
  int rc;
  if (bytes > g.grad_own_bytes) {
    CK(cudaStreamSynchronize(st), "cudaStreamSynchronize(steering buffer)");
    size_t cap = g.grad_own_bytes / 4;
    if ((rc = grow(ctx, &g.grad_own, &cap, bytes / 4, "steering gradient"))) {
      g.grad_own_bytes = 0;
      return rc;
    }
    g.grad_own_bytes = bytes;
  }
  std::vector<float> host(static_cast<size_t>(n_candidates));
  for (int t = 0; t < steps; ++t) {
    int n_ref = 0;
    if ((rc = score_grad_device(ctx, kv_pages, n_pages, block_table, seq_lens, n_candidates, g.grad_own, st, &n_ref)))
      return rc;
    if (t == 0 && p_first && (rc = finish_blocking(ctx, n_candidates, p_first, st))) return rc;
    // every referenced page (the list after the shared ones), every layer
    CK(kvprm::launch_steer_update(static_cast<bf16*>(kv_pages), g.grad_own, g.lists + g.n_shared, n_ref,
                                  ctx->cfg.n_layers, n_pages, page_elems, eta, st),
       "steering update");
  }
  if ((rc = score_device(ctx, kv_pages, n_pages, block_table, seq_lens, n_candidates, st))) return rc;
  if ((rc = finish_blocking(ctx, n_candidates, host.data(), st))) return rc;
  if (steps == 0 && p_first) std::memcpy(p_first, host.data(), sizeof(float) * n_candidates);
  if (p_last) std::memcpy(p_last, host.data(), sizeof(float) * n_candidates);
  return KVPRM_OK;
}

int kvprm_debug_set_alloc_limit(int64_t bytes) {
  g_alloc_budget.store(bytes < 0 ? -1 : static_cast<long long>(bytes));
  return KVPRM_OK;
}

int kvprm_debug_inject_error(kvprm_ctx* ctx, int32_t where) {
  if (!ctx) return KVPRM_EINVAL;
  if (where != 0 && where != 1) return fail(ctx, KVPRM_EINVAL, "injection point %d: 0 (none) or 1", where);
  ctx->inject_fail = where;
  return KVPRM_OK;
}

int kvprm_debug_wait_probe(kvprm_ctx* ctx, int32_t limit_us, void* stream) {
  if (!ctx) return KVPRM_EINVAL;
  if (limit_us < 1 || limit_us > 2000000) return fail(ctx, KVPRM_EINVAL, "wait limit %d us outside [1, 2e6]", limit_us);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  CK(kvprm::launch_wait_probe(ctx->probe_flag, ctx->err_d, 1000ull * static_cast<unsigned long long>(limit_us), st),
     "wait probe");
  ctx->last_stream = st;
  return KVPRM_OK;
}

int kvprm_check_device(kvprm_ctx* ctx) {
  if (!ctx) return KVPRM_EINVAL;
  CK(cudaStreamSynchronize(ctx->last_stream), "cudaStreamSynchronize");
  CK(cudaMemcpy(ctx->h_err, ctx->err_d, sizeof(int), cudaMemcpyDeviceToHost), "cudaMemcpy(err)");
  if (*ctx->h_err) {
    const int site = *ctx->h_err;
    CK(cudaMemset(ctx->err_d, 0, sizeof(int)), "cudaMemset(err)");
    return fail(ctx, KVPRM_ETIMEOUT, "a bounded device wait timed out (code %d)", site);
  }
  return KVPRM_OK;
}

int kvprm_set_trace(kvprm_ctx* ctx, int enable) {
  if (!ctx) return KVPRM_EINVAL;
  if (enable && !ctx->trace_d) {
    ctx->trace_cap = 2 + 8 * ctx->cfg.n_layers + 8;
    int rc = dalloc(ctx, &ctx->trace_d, static_cast<size_t>(kvprm::kTraceStride) * ctx->trace_cap, "trace");
    if (rc) return rc;
  }
  ctx->trace = enable != 0;
  return KVPRM_OK;
}

int kvprm_get_trace(kvprm_ctx* ctx, int32_t max_records, int32_t* cls, double* start_us, double* end_us) {
  return kvprm_get_trace_events(ctx, max_records, cls, start_us, end_us, nullptr);
}

int kvprm_get_trace_events(kvprm_ctx* ctx, int32_t max_records, int32_t* cls, double* start_us, double* end_us,
                           double* events_us) {
  if (!ctx || max_records < 0 || (max_records > 0 && (!cls || !start_us || !end_us))) return -KVPRM_EINVAL;
  if (!ctx->trace_d || ctx->trace_n == 0) return 0;
  if (cudaStreamSynchronize(ctx->last_stream) != cudaSuccess) return -KVPRM_ECUDA;
  constexpr int R = kvprm::kTraceStride;
  std::vector<unsigned long long> raw(static_cast<size_t>(R) * ctx->trace_n);
  if (cudaMemcpy(raw.data(), ctx->trace_d, raw.size() * sizeof(unsigned long long), cudaMemcpyDeviceToHost) !=
      cudaSuccess)
    return -KVPRM_ECUDA;
  unsigned long long t0 = ~0ull;
  for (int i = 0; i < ctx->trace_n; ++i)
    if (raw[R * i] < t0) t0 = raw[R * i];
  auto rel = [&](unsigned long long v, bool complemented) {
    if (v == ~0ull) return -1.0;
    return 1e-3 * static_cast<double>((complemented ? ~v : v) - t0);
  };
  const int n = ctx->trace_n < max_records ? ctx->trace_n : max_records;
  for (int i = 0; i < n; ++i) {
    cls[i] = ctx->trace_cls[i];
    start_us[i] = rel(raw[R * i], false);
    end_us[i] = rel(raw[R * i + 1], true);
    if (events_us)
      for (int e = 0; e < kvprm::kTraceEvents; ++e) events_us[i * kvprm::kTraceEvents + e] = rel(raw[R * i + 2 + e], true);
  }
  return n;
}

int kvprm_set_profile(kvprm_ctx* ctx, int enable) {
  if (!ctx) return KVPRM_EINVAL;
  if (enable && !ctx->profile) {
    for (int i = 0; i < KVPRM_PROF_N; ++i) {
      ctx->prof_launches[i] = 0;
      ctx->prof_ms[i] = 0.0;
    }
  }
  ctx->profile = enable != 0;
  return KVPRM_OK;
}

int kvprm_get_profile(kvprm_ctx* ctx, int64_t* launches, double* total_ms) {
  if (!ctx || !launches || !total_ms) return KVPRM_EINVAL;
  for (int i = 0; i < KVPRM_PROF_N; ++i) {
    launches[i] = ctx->prof_launches[i];
    total_ms[i] = ctx->prof_ms[i];
  }
  return KVPRM_OK;
}

}  // extern "C"
