"""CPU oracle for KV-PRM verify-token scoring -- TEST INFRASTRUCTURE ONLY.

A plain fp64 C restatement of the scoring definition (Sec. 4.1 Eq. score,
App. A.3 attention read-out, App. B.2 judgment tokens), compiled with gcc and
bound here with ctypes.  Only tests/, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this package; the CUDA scoring
library neither links nor calls it, and the two share no code.

Parity status: every function is pinned (tests/test_oracle_pins.py and
tests/test_oracle_mutants.py) by closed forms, invariants, a library
cross-check and a brute-force full causal re-encode (oracle/reencode.py);
the paper prints no worked numeric example, so no value is pinned to a
number printed in the paper.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_BUILD = os.path.join(_HERE, "_build")
SRC = os.path.join(_HERE, "kvprm_oracle.c")
LIB = os.path.join(_BUILD, "libkvprm_oracle.so")

_u16p = ctypes.POINTER(ctypes.c_uint16)
_f64p = ctypes.POINTER(ctypes.c_double)


def _lib_path(mutant: int = 0) -> str:
    return LIB if mutant == 0 else os.path.join(_BUILD, f"libkvprm_oracle_mutant{mutant}.so")


def build(mutant: int = 0, verbose: bool = False) -> str:
    """Compile the oracle (or a planted-mistake variant used by the mutation tests)."""
    os.makedirs(_BUILD, exist_ok=True)
    out = _lib_path(mutant)
    if not os.path.exists(out) or os.path.getmtime(out) < os.path.getmtime(SRC):
        cmd = ["gcc", "-O2", "-std=c11", "-shared", "-fPIC", "-pthread", f"-DORACLE_MUTANT={mutant}", "-o", out, SRC,
               "-lm"]
        subprocess.run(cmd, check=True, capture_output=not verbose)
    return out


class OracleCfg(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int), ("d_model", ctypes.c_int), ("n_q_heads", ctypes.c_int),
                ("n_kv_heads", ctypes.c_int), ("head_dim", ctypes.c_int), ("d_ff", ctypes.c_int),
                ("rope_base", ctypes.c_double), ("rms_eps", ctypes.c_double), ("mirror", ctypes.c_int),
                ("nthreads", ctypes.c_int), ("lora_rank", ctypes.c_int), ("lora_scale", ctypes.c_double),
                ("depth", ctypes.c_int), ("qk_norm", ctypes.c_int)]

    @staticmethod
    def from_arch(arch, mirror: bool = True, nthreads: int | None = None, depth: int = 1) -> "OracleCfg":
        rank = int(getattr(arch, "lora_rank", 0))
        return OracleCfg(arch.n_layers, arch.d_model, arch.n_q_heads, arch.n_kv_heads, arch.head_dim, arch.d_ff,
                         float(arch.rope_base), float(arch.rms_eps), int(mirror),
                         int(nthreads or max(1, os.cpu_count() or 1)), rank,
                         float(arch.lora_alpha) / rank if rank else 0.0, int(depth),
                         int(bool(getattr(arch, "qk_norm", False))))


class DenseWeights(ctypes.Structure):
    _fields_ = [("top", _u16p * 4), ("layer", ctypes.POINTER(_u16p) * 16)]


class DenseKV(ctypes.Structure):
    _fields_ = [("n_cand", ctypes.c_int), ("per_token", ctypes.c_int64), ("K", ctypes.POINTER(_u16p)),
                ("V", ctypes.POINTER(_u16p)), ("lens", ctypes.POINTER(ctypes.c_int64))]


_libs: dict[int, ctypes.CDLL] = {}


def lib(mutant: int = 0) -> ctypes.CDLL:
    if mutant not in _libs:
        L = ctypes.CDLL(build(mutant))
        L.oracle_bf16_round.restype = ctypes.c_double
        L.oracle_bf16_round.argtypes = [ctypes.c_double]
        L.oracle_rmsnorm.argtypes = [_f64p, _u16p, ctypes.c_int, ctypes.c_double, _f64p]
        L.oracle_rope.argtypes = [_f64p, ctypes.c_int, ctypes.c_double, ctypes.c_double]
        L.oracle_attend.argtypes = [_f64p, _u16p, _u16p, ctypes.c_int64, ctypes.c_int64, _f64p, _f64p, ctypes.c_int,
                                    _f64p, _f64p]
        L.oracle_reward.restype = ctypes.c_double
        L.oracle_reward.argtypes = [_f64p, _u16p, _u16p, ctypes.c_int]
        L.oracle_score.argtypes = [ctypes.POINTER(OracleCfg), ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
                                   ctypes.c_void_p, ctypes.c_int, ctypes.POINTER(ctypes.c_int32),
                                   ctypes.POINTER(ctypes.c_int64), _f64p, _f64p, _f64p, _f64p, _f64p]
        _libs[mutant] = L
    return _libs[mutant]


def _f64(a):
    a = np.ascontiguousarray(a, dtype=np.float64)
    return a, a.ctypes.data_as(_f64p)


def _u16(a):
    a = np.ascontiguousarray(a, dtype=np.uint16)
    return a, a.ctypes.data_as(_u16p)


# ------------------------------------------------------------------ primitives
def bf16_round(x: float, mutant: int = 0) -> float:
    return lib(mutant).oracle_bf16_round(float(x))


def rmsnorm(h, g_bits, eps: float, mutant: int = 0) -> np.ndarray:
    h, hp = _f64(h)
    g, gp = _u16(g_bits)
    out = np.empty_like(h)
    lib(mutant).oracle_rmsnorm(hp, gp, h.size, eps, out.ctypes.data_as(_f64p))
    return out


def rope(x, pos: float, base: float, mutant: int = 0) -> np.ndarray:
    x = np.array(x, dtype=np.float64, copy=True)
    lib(mutant).oracle_rope(x.ctypes.data_as(_f64p), x.size, float(pos), float(base))
    return x


def attend(q, K_bits, V_bits, k_self, v_self, mutant: int = 0):
    """One query head against L cached bf16 keys/values plus the self entry.
    Returns (o [hd], weights [L+1])."""
    q, qp = _f64(q)
    hd = q.size
    K, Kp = _u16(np.asarray(K_bits).reshape(-1, hd))
    V, Vp = _u16(np.asarray(V_bits).reshape(-1, hd))
    L = K.shape[0]
    ks, ksp = _f64(k_self)
    vs, vsp = _f64(v_self)
    o = np.empty(hd)
    w = np.empty(L + 1)
    lib(mutant).oracle_attend(qp, Kp, Vp, L, hd, ksp, vsp, hd, o.ctypes.data_as(_f64p), w.ctypes.data_as(_f64p))
    return o, w


def reward(x, wp_bits, wm_bits, mutant: int = 0) -> float:
    x, xp = _f64(x)
    wp, wpp = _u16(wp_bits)
    wm, wmp = _u16(wm_bits)
    return lib(mutant).oracle_reward(xp, wpp, wmp, x.size)


# ------------------------------------------------------------------ scorer
class Result:
    def __init__(self, p_plus, attn, hidden, qkv=None, h_layers=None):
        self.p_plus, self.attn, self.hidden, self.qkv, self.h_layers = p_plus, attn, hidden, qkv, h_layers


def _score(arch, wfn, wuser, kvfn, kvuser, cand_ids, lens, mirror, want_attn, want_hidden, nthreads, mutant,
           want_layers=False, depth: int = 1):
    n = len(cand_ids)
    rows = n * depth   # per-row outputs: candidate i's verify tokens are rows i depth .. i depth + depth - 1
    ids = np.ascontiguousarray(cand_ids, np.int32)
    lens = np.ascontiguousarray(lens, np.int64)
    p = np.empty(n)
    attn = np.empty((arch.n_layers, rows, arch.n_q_heads * arch.head_dim)) if want_attn else None
    hid = np.empty((n, arch.d_model)) if want_hidden else None
    qkv = np.empty((arch.n_layers, rows, arch.qkv_rows)) if want_layers else None
    hl = np.empty((arch.n_layers, rows, arch.d_model)) if want_layers else None
    cfg = OracleCfg.from_arch(arch, mirror, nthreads, depth)
    rc = lib(mutant).oracle_score(ctypes.byref(cfg), wfn, wuser, kvfn, kvuser, n,
                                  ids.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)),
                                  lens.ctypes.data_as(ctypes.POINTER(ctypes.c_int64)), p.ctypes.data_as(_f64p),
                                  attn.ctypes.data_as(_f64p) if attn is not None else None,
                                  hid.ctypes.data_as(_f64p) if hid is not None else None,
                                  qkv.ctypes.data_as(_f64p) if qkv is not None else None,
                                  hl.ctypes.data_as(_f64p) if hl is not None else None)
    if rc != 0:
        raise RuntimeError(f"oracle_score failed with code {rc}")
    return Result(p, attn, hid, qkv, hl)


def score_synth(w, tables, cand_ids=None, mirror: bool = True, want_attn: bool = True, want_hidden: bool = False,
                nthreads: int | None = None, mutant: int = 0, want_layers: bool = False, depth: int = 1) -> Result:
    """Score candidates of a kvsynth workload; K/V come from their logical token identities.  depth > 1:
    a depth-k readout (k verify tokens, causal among themselves; per-row outputs have len(ids) * k rows)."""
    import kvsynth
    prov = kvsynth.Providers(w, tables, nthreads)
    ids = list(range(w.n_candidates)) if cand_ids is None else list(cand_ids)
    lens = [len(w.cand_seg[i]) for i in ids]
    return _score(w.arch, prov.weight_fn, prov.user, prov.kv_fn, prov.user, ids, lens, mirror, want_attn, want_hidden,
                  nthreads, mutant, want_layers, depth)


def score_dense(arch, weights: dict, kv: list, mirror: bool = True, want_attn: bool = True, want_hidden: bool = False,
                nthreads: int | None = None, mutant: int = 0, depth: int = 1) -> Result:
    """Score from explicit arrays.  weights = {'top': {kind: bits}, 'layers': [{kind: bits}]} (kinds 4..9, the
    adapter factors 10..17 when arch.lora_rank > 0, the q/k norm gains 18, 19 when arch.qk_norm);
    kv[l][b] = (K_bits [L_b][nkv][hd], V_bits [L_b][nkv][hd])."""
    keep = []
    dw = DenseWeights()
    for k in range(4):
        a, ap = _u16(weights["top"][k])
        keep.append(a)
        dw.top[k] = ap
    kinds = list(range(4, 10))
    if getattr(arch, "lora_rank", 0):   # with an adapter: its factors too
        kinds += list(range(10, 18))
    if getattr(arch, "qk_norm", False):   # with the per-head q/k norm: its gains
        kinds += [18, 19]
    for kind in kinds:
        j = kind - 4
        ptrs = (_u16p * arch.n_layers)()
        for l in range(arch.n_layers):
            a, ap = _u16(weights["layers"][l][kind])
            keep.append(a)
            ptrs[l] = ap
        keep.append(ptrs)
        dw.layer[j] = ctypes.cast(ptrs, ctypes.POINTER(_u16p))
    n = len(kv[0])
    lens = np.asarray([np.asarray(kv[0][b][0]).shape[0] for b in range(n)], np.int64)
    Kp = (_u16p * (arch.n_layers * n))()
    Vp = (_u16p * (arch.n_layers * n))()
    for l in range(arch.n_layers):
        for b in range(n):
            K, kp = _u16(kv[l][b][0])
            V, vp = _u16(kv[l][b][1])
            keep += [K, V]
            Kp[l * n + b] = kp
            Vp[l * n + b] = vp
    dk = DenseKV(n, arch.n_kv_heads * arch.head_dim, Kp, Vp, lens.ctypes.data_as(ctypes.POINTER(ctypes.c_int64)))
    keep += [Kp, Vp, lens, dw, dk]
    L = lib(mutant)
    wfn = ctypes.cast(L.oracle_dense_weight_provider, ctypes.c_void_p).value
    kvfn = ctypes.cast(L.oracle_dense_kv_provider, ctypes.c_void_p).value
    return _score(arch, wfn, ctypes.cast(ctypes.pointer(dw), ctypes.c_void_p).value, kvfn,
                  ctypes.cast(ctypes.pointer(dk), ctypes.c_void_p).value, list(range(n)), lens, mirror, want_attn,
                  want_hidden, nthreads, mutant, False, depth)
