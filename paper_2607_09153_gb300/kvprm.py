"""ctypes binding of the scoring library's C ABI (include/kvprm.h).

Names mirror the C entry points; this module only marshals arguments (device
pointers from torch tensors, host arrays from numpy) and turns non-zero status
codes into exceptions.  Every step of the scoring path runs in the CUDA
library; there is no Python or CPU fallback: if the library cannot be built or
loaded, importing it raises.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

from . import build as _build

KVPRM_OK, KVPRM_EINVAL, KVPRM_ECAPACITY, KVPRM_EINDEX, KVPRM_ECUDA, KVPRM_ENOMEM, KVPRM_ETIMEOUT, \
    KVPRM_EUNSUPPORTED = range(8)
PROF_NAMES = ("gemm_qkv", "gemm_o", "gemm_gate_up", "gemm_down", "attention", "combine", "fused", "attention_tc",
              "adapter")


class KvprmError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"kvprm error {code}: {msg}")
        self.code = code


class KvprmConfig(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int32), ("d_model", ctypes.c_int32), ("n_q_heads", ctypes.c_int32),
                ("n_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32), ("d_ff", ctypes.c_int32),
                ("page_size", ctypes.c_int32), ("rope_base", ctypes.c_float), ("rms_eps", ctypes.c_float),
                ("qk_norm", ctypes.c_int32), ("max_candidates", ctypes.c_int32), ("max_blocks_per_seq", ctypes.c_int32)]


_VPP = ctypes.POINTER(ctypes.c_void_p)


class KvprmWeights(ctypes.Structure):
    _fields_ = [("embed_verify", ctypes.c_void_p), ("final_norm", ctypes.c_void_p), ("w_plus", ctypes.c_void_p),
                ("w_minus", ctypes.c_void_p), ("attn_norm", _VPP), ("w_qkv", _VPP), ("w_o", _VPP),
                ("mlp_norm", _VPP), ("w_gate_up", _VPP), ("w_down", _VPP), ("q_norm", _VPP), ("k_norm", _VPP)]


class KvprmProjectionPlan(ctypes.Structure):
    _fields_ = [(k, ctypes.c_int32) for k in ("m_tiles", "k_tiles", "kt_per_split", "cluster", "tiles_per_cta",
                                               "stages", "tmem_cols")] + [("smem_bytes", ctypes.c_int64),
                                                                          ("threads", ctypes.c_int32)]


class KvprmLora(ctypes.Structure):
    _fields_ = [(k, _VPP) for k in ("a_qkv", "b_qkv", "a_o", "b_o", "a_gate_up", "b_gate_up", "a_down", "b_down")]


LORA_FACTORS = ("a_qkv", "b_qkv", "a_o", "b_o", "a_gate_up", "b_gate_up", "a_down", "b_down")


class KvprmAttnPlan(ctypes.Structure):
    _fields_ = [("n_segs", ctypes.c_int32), ("n_ctas", ctypes.c_int32), ("n_pages", ctypes.c_int32),
                ("n_cands", ctypes.c_int32), ("n_slot_refs", ctypes.c_int32), ("n_slots", ctypes.c_int32),
                ("segs", ctypes.POINTER(ctypes.c_int32)), ("segs_cap", ctypes.c_int64),
                ("cta_seg", ctypes.POINTER(ctypes.c_int32)), ("cta_cap", ctypes.c_int64),
                ("pages", ctypes.POINTER(ctypes.c_int32)), ("pages_cap", ctypes.c_int64),
                ("cands", ctypes.POINTER(ctypes.c_int32)), ("cands_cap", ctypes.c_int64),
                ("slots", ctypes.POINTER(ctypes.c_int32)), ("slots_cap", ctypes.c_int64),
                ("slot_base", ctypes.POINTER(ctypes.c_int32)), ("nslots", ctypes.POINTER(ctypes.c_int32)),
                ("n_tc_ctas", ctypes.c_int32), ("tc_cta", ctypes.POINTER(ctypes.c_int32)), ("tc_cta_cap", ctypes.c_int64),
                ("fuse_cs", ctypes.c_int32)]

KVPRM_PLAN_FUSE = 16


_lib = None


def lib() -> ctypes.CDLL:
    """Load (building first if the sources changed) the in-tree libkvprm.so."""
    global _lib
    if _lib is None:
        path = _build.build()
        L = ctypes.CDLL(path)
        vp, i32, i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
        i32p, i64p, f32p = ctypes.POINTER(ctypes.c_int32), ctypes.POINTER(ctypes.c_int64), ctypes.POINTER(ctypes.c_float)
        L.kvprm_create.argtypes = [ctypes.POINTER(KvprmConfig), ctypes.POINTER(KvprmWeights), ctypes.POINTER(vp)]
        L.kvprm_destroy.argtypes = [vp]
        L.kvprm_destroy.restype = None
        L.kvprm_last_error.argtypes = [vp]
        L.kvprm_last_error.restype = ctypes.c_char_p
        L.kvprm_score.argtypes = [vp, vp, i64, i32p, i32p, i32, f32p, vp]
        L.kvprm_score_async.argtypes = [vp, vp, i64, i32p, i32p, i32, vp, vp]
        L.kvprm_score_host.argtypes = [vp, vp, i64, i32p, i32p, i32, f32p, vp]
        L.kvprm_attention.argtypes = [vp, vp, i64, i32p, i32p, i32, vp, vp, vp, vp, vp]
        L.kvprm_projection.argtypes = [vp, vp, i32, i32, vp, i32, vp, vp]
        L.kvprm_set_lora.argtypes = [vp, i32, ctypes.c_float, ctypes.POINTER(KvprmLora)]
        L.kvprm_set_readout_depth.argtypes = [vp, i32]
        L.kvprm_plan_projection.argtypes = [i32, i32, i32, i32, i32, i32, ctypes.POINTER(KvprmProjectionPlan)]
        L.kvprm_debug_hidden.argtypes = [vp, vp]
        L.kvprm_attention_noalloc.argtypes = [vp, i64, i32p, i32, i32p, i32, i32, i32, i32, vp, vp, vp, vp, vp]
        L.kvprm_set_debug.argtypes = [vp, ctypes.c_int]
        L.kvprm_debug_attn_out.argtypes = [vp, vp]
        L.kvprm_debug_layers.argtypes = [vp, ctypes.c_int, vp]
        L.kvprm_resolve.argtypes = [vp, i32, i64p]
        L.kvprm_check_device.argtypes = [vp]
        L.kvprm_debug_set_alloc_limit.argtypes = [i64]
        L.kvprm_score_grad.argtypes = [vp, vp, i64, i32p, i32p, i32, vp, f32p, vp]
        L.kvprm_steer.argtypes = [vp, vp, i64, i32p, i32p, i32, ctypes.c_float, i32, f32p, f32p, vp]
        L.kvprm_debug_inject_error.argtypes = [vp, i32]
        L.kvprm_debug_wait_probe.argtypes = [vp, i32, vp]
        L.kvprm_set_profile.argtypes = [vp, ctypes.c_int]
        L.kvprm_set_trace.argtypes = [vp, ctypes.c_int]
        L.kvprm_get_trace.argtypes = [vp, i32, i32p, ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_double)]
        L.kvprm_get_trace_events.argtypes = [vp, i32, i32p, ctypes.POINTER(ctypes.c_double),
                                             ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_double)]
        L.kvprm_get_profile.argtypes = [vp, i64p, ctypes.POINTER(ctypes.c_double)]
        L.kvprm_plan_attention.argtypes = [i32p, i32, i32p, i32, i32, i32, i32, i32, ctypes.POINTER(KvprmAttnPlan)]
        _lib = L
    return _lib


def library_path() -> str:
    return _build.LIB


def _check(ctx, rc: int) -> None:
    if rc != KVPRM_OK:
        msg = lib().kvprm_last_error(ctx).decode() if ctx else ""
        raise KvprmError(rc, msg)


def _i32(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.int32)


def _p(a: np.ndarray, t):
    return a.ctypes.data_as(ctypes.POINTER(t))


# ------------------------------------------------------------------ same-name wrappers
def kvprm_create(config: KvprmConfig, weights: KvprmWeights) -> ctypes.c_void_p:
    ctx = ctypes.c_void_p()
    rc = lib().kvprm_create(ctypes.byref(config), ctypes.byref(weights), ctypes.byref(ctx))
    if rc != KVPRM_OK:
        raise KvprmError(rc, "kvprm_create failed")
    return ctx


def kvprm_destroy(ctx) -> None:
    lib().kvprm_destroy(ctx)


def kvprm_score(ctx, kv_pages_ptr: int, n_pages: int, block_table, seq_lens, n: int, stream_ptr: int = 0) -> np.ndarray:
    bt, sl = _i32(block_table), _i32(seq_lens)
    out = np.zeros(n, np.float32)
    _check(ctx, lib().kvprm_score(ctx, kv_pages_ptr, n_pages, _p(bt, ctypes.c_int32), _p(sl, ctypes.c_int32), n,
                                  _p(out, ctypes.c_float), stream_ptr))
    return out


def kvprm_score_async(ctx, kv_pages_ptr: int, n_pages: int, block_table, seq_lens, n: int, d_rewards_ptr: int,
                      stream_ptr: int = 0) -> None:
    bt, sl = _i32(block_table), _i32(seq_lens)
    _check(ctx, lib().kvprm_score_async(ctx, kv_pages_ptr, n_pages, _p(bt, ctypes.c_int32), _p(sl, ctypes.c_int32),
                                        n, d_rewards_ptr, stream_ptr))


def kvprm_score_host(ctx, h_kv_pages_ptr: int, n_pages: int, block_table, seq_lens, n: int, stream_ptr: int = 0,
                     out: np.ndarray | None = None) -> np.ndarray:
    bt, sl = _i32(block_table), _i32(seq_lens)
    if out is None:
        out = np.zeros(n, np.float32)
    _check(ctx, lib().kvprm_score_host(ctx, h_kv_pages_ptr, n_pages, _p(bt, ctypes.c_int32), _p(sl, ctypes.c_int32),
                                       n, _p(out, ctypes.c_float), stream_ptr))
    return out


def kvprm_score_grad(ctx, kv_pages_ptr: int, n_pages: int, block_table, seq_lens, n: int, d_grad_ptr: int,
                     stream_ptr: int = 0) -> np.ndarray:
    """KV Steering gradient: d(sum_b -log P(+)_b)/d(keys, values) into the device fp32 buffer d_grad
    (the pool's layout); returns P(+) [n]."""
    bt, sl = _i32(block_table), _i32(seq_lens)
    out = np.zeros(n, np.float32)
    _check(ctx, lib().kvprm_score_grad(ctx, kv_pages_ptr, n_pages, _p(bt, ctypes.c_int32), _p(sl, ctypes.c_int32), n,
                                       d_grad_ptr, _p(out, ctypes.c_float), stream_ptr))
    return out


def kvprm_steer(ctx, kv_pages_ptr: int, n_pages: int, block_table, seq_lens, n: int, eta: float, steps: int,
                stream_ptr: int = 0) -> tuple[np.ndarray, np.ndarray]:
    """`steps` KV Steering steps on the (caller-owned, written) pages; returns P(+) before and after."""
    bt, sl = _i32(block_table), _i32(seq_lens)
    p0 = np.zeros(n, np.float32)
    p1 = np.zeros(n, np.float32)
    _check(ctx, lib().kvprm_steer(ctx, kv_pages_ptr, n_pages, _p(bt, ctypes.c_int32), _p(sl, ctypes.c_int32), n,
                                  float(eta), int(steps), _p(p0, ctypes.c_float), _p(p1, ctypes.c_float), stream_ptr))
    return p0, p1


def kvprm_attention(ctx, kv_layer_ptr: int, n_pages: int, block_table, seq_lens, n: int, q_ptr: int, k_self_ptr: int,
                    v_self_ptr: int, out_ptr: int, stream_ptr: int = 0) -> None:
    bt, sl = _i32(block_table), _i32(seq_lens)
    _check(ctx, lib().kvprm_attention(ctx, kv_layer_ptr, n_pages, _p(bt, ctypes.c_int32), _p(sl, ctypes.c_int32), n,
                                      q_ptr, k_self_ptr, v_self_ptr, out_ptr, stream_ptr))


def kvprm_projection(ctx, W_ptr: int, M: int, K: int, X_ptr: int, n: int, Y_ptr: int, stream_ptr: int = 0) -> None:
    _check(ctx, lib().kvprm_projection(ctx, W_ptr, M, K, X_ptr, n, Y_ptr, stream_ptr))


def kvprm_plan_projection(M: int, K: int, n_pad: int, num_sms: int, has_lo: bool = True,
                          gate_up: bool = False) -> dict:
    """The projection GEMM's launch plan (host only)."""
    out = KvprmProjectionPlan()
    rc = lib().kvprm_plan_projection(int(M), int(K), int(n_pad), int(num_sms), int(has_lo), int(gate_up),
                                     ctypes.byref(out))
    if rc != 0:
        raise KvprmError(rc, "kvprm_plan_projection: bad arguments")
    return {k: getattr(out, k) for k, _ in KvprmProjectionPlan._fields_}


def kvprm_set_readout_depth(ctx, depth: int) -> None:
    _check(ctx, lib().kvprm_set_readout_depth(ctx, int(depth)))


def kvprm_set_lora(ctx, rank: int, scale: float, lora: KvprmLora | None) -> None:
    _check(ctx, lib().kvprm_set_lora(ctx, int(rank), float(scale), ctypes.byref(lora) if lora is not None else None))


def kvprm_debug_hidden(ctx, d_out_ptr: int) -> None:
    _check(ctx, lib().kvprm_debug_hidden(ctx, d_out_ptr))


def kvprm_attention_noalloc(kv_layer_ptr: int, n_pages: int, block_table, seq_lens, n_q_heads: int, n_kv_heads: int,
                            head_dim: int, q_ptr: int, k_self_ptr: int, v_self_ptr: int, out_ptr: int,
                            stream_ptr: int = 0) -> None:
    """The attention read-out through the entry point that allocates nothing (no context)."""
    bt, sl = _i32(block_table), _i32(seq_lens)
    n = len(sl)
    rc = lib().kvprm_attention_noalloc(kv_layer_ptr, n_pages, _p(bt, ctypes.c_int32), bt.shape[1] if bt.ndim == 2 else 1,
                                       _p(sl, ctypes.c_int32), n, n_q_heads, n_kv_heads, head_dim, q_ptr, k_self_ptr,
                                       v_self_ptr, out_ptr, stream_ptr)
    if rc != KVPRM_OK:
        raise KvprmError(rc, "kvprm_attention_noalloc failed")


def kvprm_plan_attention(block_table, seq_lens, n_kv_heads: int, group: int, n_ctas: int, share: int = 1) -> dict:
    """The attention schedule of a call (host only): dict of numpy arrays
    segs [n_segs][8], cta_seg, pages, cands, slots, slot_base, nslots, fuse_cs.  share: 0 none,
    1 shared runs on the persistent CTAs, 2 shared pages on the tensor cores, 3 as 2 with the SMs
    split between the two launches; | KVPRM_PLAN_FUSE tries the fused-combine plan first."""
    bt, sl = _i32(block_table), _i32(seq_lens)
    n = len(sl)
    mb = bt.shape[1] if bt.ndim == 2 and bt.shape[1] > 0 else 1
    bt = bt.reshape(max(n, 1) if n else 1, -1) if n else np.zeros((1, 1), np.int32)
    plan = KvprmAttnPlan()
    rc = lib().kvprm_plan_attention(_p(bt, ctypes.c_int32), mb, _p(sl, ctypes.c_int32), n, n_kv_heads, group, n_ctas,
                                    int(share), ctypes.byref(plan))
    if rc not in (KVPRM_OK, KVPRM_ECAPACITY):
        raise KvprmError(rc, "kvprm_plan_attention failed")
    bufs = {"segs": np.zeros((max(plan.n_segs, 1), 8), np.int32), "cta_seg": np.zeros(max(plan.n_ctas + 1, 1), np.int32),
            "pages": np.zeros(max(plan.n_pages, 1), np.int32), "cands": np.zeros(max(plan.n_cands, 1), np.int32),
            "slots": np.zeros(max(plan.n_slot_refs, 1), np.int32),
            "slot_base": np.zeros(max(n * n_kv_heads, 1), np.int32), "nslots": np.zeros(max(n * n_kv_heads, 1), np.int32),
            "tc_cta": np.zeros(max(plan.n_tc_ctas + 1, 1), np.int32)}
    plan.segs, plan.segs_cap = _p(bufs["segs"], ctypes.c_int32), bufs["segs"].shape[0]
    plan.cta_seg, plan.cta_cap = _p(bufs["cta_seg"], ctypes.c_int32), bufs["cta_seg"].size
    plan.pages, plan.pages_cap = _p(bufs["pages"], ctypes.c_int32), bufs["pages"].size
    plan.cands, plan.cands_cap = _p(bufs["cands"], ctypes.c_int32), bufs["cands"].size
    plan.slots, plan.slots_cap = _p(bufs["slots"], ctypes.c_int32), bufs["slots"].size
    plan.slot_base, plan.nslots = _p(bufs["slot_base"], ctypes.c_int32), _p(bufs["nslots"], ctypes.c_int32)
    plan.tc_cta, plan.tc_cta_cap = _p(bufs["tc_cta"], ctypes.c_int32), bufs["tc_cta"].size
    rc = lib().kvprm_plan_attention(_p(bt, ctypes.c_int32), mb, _p(sl, ctypes.c_int32), n, n_kv_heads, group, n_ctas,
                                    int(share), ctypes.byref(plan))
    if rc != KVPRM_OK:
        raise KvprmError(rc, "kvprm_plan_attention failed")
    return {"segs": bufs["segs"][:plan.n_segs], "cta_seg": bufs["cta_seg"][:plan.n_ctas + 1] if plan.n_ctas else
            np.zeros(1, np.int32), "pages": bufs["pages"][:plan.n_pages], "cands": bufs["cands"][:plan.n_cands],
            "slots": bufs["slots"][:plan.n_slot_refs], "slot_base": bufs["slot_base"][:n * n_kv_heads],
            "nslots": bufs["nslots"][:n * n_kv_heads], "n_ctas": plan.n_ctas, "n_slots": plan.n_slots,
            "tc_cta": bufs["tc_cta"][:plan.n_tc_ctas + 1] if plan.n_tc_ctas else np.zeros(1, np.int32),
            "n_tc_ctas": plan.n_tc_ctas, "fuse_cs": plan.fuse_cs}


def kvprm_set_debug(ctx, flags: int) -> None:
    _check(ctx, lib().kvprm_set_debug(ctx, flags))


def kvprm_debug_attn_out(ctx, d_out_ptr: int) -> None:
    _check(ctx, lib().kvprm_debug_attn_out(ctx, d_out_ptr))


def kvprm_debug_layers(ctx, which: int, d_out_ptr: int) -> None:
    _check(ctx, lib().kvprm_debug_layers(ctx, which, d_out_ptr))


def kvprm_resolve(ctx, b: int, length: int) -> np.ndarray:
    out = np.zeros(max(length, 1), np.int64)
    _check(ctx, lib().kvprm_resolve(ctx, b, _p(out, ctypes.c_int64)))
    return out[:length]


def kvprm_check_device(ctx) -> None:
    _check(ctx, lib().kvprm_check_device(ctx))


def kvprm_debug_set_alloc_limit(n_bytes: int) -> None:
    """Failure-detection hook: the library may allocate at most n_bytes more (-1: no limit)."""
    rc = lib().kvprm_debug_set_alloc_limit(int(n_bytes))
    if rc != KVPRM_OK:
        raise KvprmError(rc, "kvprm_debug_set_alloc_limit failed")


def kvprm_debug_inject_error(ctx, where: int = 1) -> None:
    _check(ctx, lib().kvprm_debug_inject_error(ctx, int(where)))


def kvprm_debug_wait_probe(ctx, limit_us: int, stream_ptr: int = 0) -> None:
    _check(ctx, lib().kvprm_debug_wait_probe(ctx, int(limit_us), stream_ptr))


def kvprm_set_profile(ctx, enable: bool) -> None:
    _check(ctx, lib().kvprm_set_profile(ctx, int(enable)))


def kvprm_set_trace(ctx, enable: bool) -> None:
    _check(ctx, lib().kvprm_set_trace(ctx, int(enable)))


def kvprm_get_trace(ctx, max_records: int = 4096) -> list:
    """[(class name, start us, end us)] of the last call's launches, in issue order."""
    cls = np.zeros(max_records, np.int32)
    t0 = np.zeros(max_records, np.float64)
    t1 = np.zeros(max_records, np.float64)
    n = lib().kvprm_get_trace(ctx, max_records, _p(cls, ctypes.c_int32),
                              t0.ctypes.data_as(ctypes.POINTER(ctypes.c_double)),
                              t1.ctypes.data_as(ctypes.POINTER(ctypes.c_double)))
    if n < 0:
        _check(ctx, -n)
    return [(PROF_NAMES[cls[i]], float(t0[i]), float(t1[i])) for i in range(n)]


def kvprm_get_trace_events(ctx, max_records: int = 4096) -> list:
    """[(class name, start us, end us, [8 milestone us or -1])] of the last call's launches, in issue order."""
    dp = ctypes.POINTER(ctypes.c_double)
    cls = np.zeros(max_records, np.int32)
    t0 = np.zeros(max_records, np.float64)
    t1 = np.zeros(max_records, np.float64)
    ev = np.zeros((max_records, 8), np.float64)
    n = lib().kvprm_get_trace_events(ctx, max_records, _p(cls, ctypes.c_int32), t0.ctypes.data_as(dp),
                                     t1.ctypes.data_as(dp), ev.ctypes.data_as(dp))
    if n < 0:
        _check(ctx, -n)
    return [(PROF_NAMES[cls[i]], float(t0[i]), float(t1[i]), ev[i].tolist()) for i in range(n)]


def kvprm_get_profile(ctx) -> dict:
    """{class name: (launches, total ms)} since profiling was enabled."""
    k = len(PROF_NAMES)
    n = np.zeros(k, np.int64)
    ms = np.zeros(k, np.float64)
    _check(ctx, lib().kvprm_get_profile(ctx, _p(n, ctypes.c_int64), ms.ctypes.data_as(ctypes.POINTER(ctypes.c_double))))
    return {PROF_NAMES[i]: (int(n[i]), float(ms[i])) for i in range(k)}


# ------------------------------------------------------------------ torch convenience
class Scorer:
    """Owns a context for a scorer whose weights are torch bf16 CUDA tensors.

    weights = {'embed_verify', 'final_norm', 'w_plus', 'w_minus'} -> tensor, and
    'layers' -> list of {'attn_norm', 'w_qkv', 'w_o', 'mlp_norm', 'w_gate_up', 'w_down'} (plus 'q_norm' and
    'k_norm' with qk_norm=True)."""

    def __init__(self, n_layers, d_model, n_q_heads, n_kv_heads, head_dim, d_ff, weights: dict, max_candidates: int,
                 max_blocks_per_seq: int, rope_base: float = 1e4, rms_eps: float = 1e-6, qk_norm: bool = False):
        self.cfg = KvprmConfig(n_layers, d_model, n_q_heads, n_kv_heads, head_dim, d_ff, 16, rope_base, rms_eps,
                               int(qk_norm), max_candidates, max_blocks_per_seq)
        arr = ctypes.c_void_p * n_layers
        lay = weights["layers"]
        kinds = ("attn_norm", "w_qkv", "w_o", "mlp_norm", "w_gate_up", "w_down") + (("q_norm", "k_norm") if qk_norm else ())
        self._arrays = {k: arr(*[lay[l][k].data_ptr() for l in range(n_layers)]) for k in kinds}
        self._weights = weights   # keep the tensors alive
        cast = lambda a: ctypes.cast(a, _VPP)  # noqa: E731
        self.w = KvprmWeights(weights["embed_verify"].data_ptr(), weights["final_norm"].data_ptr(),
                              weights["w_plus"].data_ptr(), weights["w_minus"].data_ptr(),
                              cast(self._arrays["attn_norm"]), cast(self._arrays["w_qkv"]), cast(self._arrays["w_o"]),
                              cast(self._arrays["mlp_norm"]), cast(self._arrays["w_gate_up"]),
                              cast(self._arrays["w_down"]), cast(self._arrays["q_norm"]) if qk_norm else None,
                              cast(self._arrays["k_norm"]) if qk_norm else None)
        self.ctx = kvprm_create(self.cfg, self.w)

    def set_depth(self, depth: int) -> None:
        """Depth-k readout: k verify tokens per candidate, the reward read at the last one."""
        kvprm_set_readout_depth(self.ctx, depth)

    def set_lora(self, rank: int, alpha: float = 32.0, factors: list | None = None) -> None:
        """Scorer adapter on every projection (rank 0: merged weights alone); factors[l] holds
        {'a_qkv', 'b_qkv', 'a_o', 'b_o', 'a_gate_up', 'b_gate_up', 'a_down', 'b_down'} bf16 tensors."""
        if rank == 0:
            kvprm_set_lora(self.ctx, 0, 0.0, None)
            return
        n = self.cfg.n_layers
        arr = ctypes.c_void_p * n
        self._lora_arrays = {k: arr(*[factors[l][k].data_ptr() for l in range(n)]) for k in LORA_FACTORS}
        self._lora_factors = factors   # keep the tensors alive
        lo = KvprmLora(*[ctypes.cast(self._lora_arrays[k], _VPP) for k in LORA_FACTORS])
        kvprm_set_lora(self.ctx, rank, alpha / rank, lo)

    def close(self):
        if self.ctx:
            kvprm_destroy(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def score(self, kv_pages, block_table, seq_lens, stream=None) -> np.ndarray:
        import torch
        st = (stream or torch.cuda.current_stream()).cuda_stream
        n_pages = kv_pages.shape[1]
        return kvprm_score(self.ctx, kv_pages.data_ptr(), n_pages, block_table, seq_lens, len(seq_lens), st)

    def score_host(self, kv_pages, block_table, seq_lens, stream=None) -> np.ndarray:
        """As score, with kv_pages a contiguous CPU bf16 tensor (pinned memory is copied in by the
        library's copy kernel at the host link's full rate; pageable memory by the copy engine)."""
        import torch
        if kv_pages.device.type != "cpu" or not kv_pages.is_contiguous():
            raise ValueError("score_host takes a contiguous CPU tensor; use score for a device cache")
        st = (stream or torch.cuda.current_stream()).cuda_stream
        return kvprm_score_host(self.ctx, kv_pages.data_ptr(), kv_pages.shape[1], block_table, seq_lens, len(seq_lens),
                                st)

    def score_async(self, kv_pages, block_table, seq_lens, d_rewards, stream=None) -> None:
        import torch
        st = (stream or torch.cuda.current_stream()).cuda_stream
        kvprm_score_async(self.ctx, kv_pages.data_ptr(), kv_pages.shape[1], block_table, seq_lens, len(seq_lens),
                          d_rewards.data_ptr(), st)
