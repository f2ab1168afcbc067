"""Seeded synthetic inputs for KV-PRM verify-token scoring.

This package is the one module both sides use: the CPU oracle (``oracle/``)
and the CUDA scoring library (``paper_2607_09153_gb300``).  It holds the
scorer architectures and workload shapes, the cache-sharing structure of each
workload (distinct caches, a beam prefix, an MCTS tree), the paging of logical
tokens into physical pages, and bit-exact host (C) and device (CUDA) fills.
It contains none of the scoring method's arithmetic.

Value recipe: bf16 bit patterns ``table[SplitMix64(key, n) >> 48]`` where the
65,536-entry table holds bf16(offset + scale * Phi^-1((i + 0.5) / 65536)):
N(0, 1) for cached keys/values, N(0, 0.02) for weights, 1 + gain_std * N(0, 1)
for RMSNorm gains (gain_std = 0 gives the standard all-ones initialisation).
"""
from __future__ import annotations

import ctypes
import os
import shutil
import subprocess
from dataclasses import dataclass, field

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_BUILD = os.path.join(_HERE, "_build")
HOST_LIB = os.path.join(_BUILD, "libkvsynth_host.so")
DEV_LIB = os.path.join(_BUILD, "libkvsynth_dev.so")

# weight kinds (same numbering the oracle's provider interface uses)
EMBED, FINAL_NORM, W_PLUS, W_MINUS, ATTN_NORM, W_QKV, W_O, MLP_NORM, W_GATE_UP, W_DOWN = range(10)
# low-rank adapter factors of each projection (y = W x + scale B (A x)): A [r][in], B [out][r]
(LORA_A_QKV, LORA_B_QKV, LORA_A_O, LORA_B_O, LORA_A_GATE_UP, LORA_B_GATE_UP, LORA_A_DOWN,
 LORA_B_DOWN) = range(10, 18)
LORA_KINDS = tuple(range(10, 18))
# per-head RMSNorm gains of q and k (Qwen3-style q/k norm), [head_dim] per layer
Q_NORM, K_NORM = 18, 19
QK_NORM_KINDS = (Q_NORM, K_NORM)
LAYER_KINDS = (ATTN_NORM, W_QKV, W_O, MLP_NORM, W_GATE_UP, W_DOWN)
GAIN_KINDS = (FINAL_NORM, ATTN_NORM, MLP_NORM, Q_NORM, K_NORM)


# --------------------------------------------------------------------------- build
def build(verbose: bool = False, device: bool | None = None) -> None:
    """Compile the host generator (gcc) and, when nvcc is present, its device twin."""
    os.makedirs(_BUILD, exist_ok=True)
    src = os.path.join(_HERE, "synth.c")
    if _stale(HOST_LIB, [src]):
        cmd = ["gcc", "-O2", "-std=c11", "-shared", "-fPIC", "-pthread", "-o", HOST_LIB, src]
        subprocess.run(cmd, check=True, capture_output=not verbose)
    nvcc = shutil.which("nvcc") or ("/usr/local/cuda/bin/nvcc" if os.path.exists("/usr/local/cuda/bin/nvcc") else None)
    if device is None:
        device = nvcc is not None
    if device:
        cu = os.path.join(_HERE, "synth_fill.cu")
        if _stale(DEV_LIB, [cu]):
            cmd = [nvcc, "-O3", "-std=c++17", "-gencode", "arch=compute_103a,code=sm_103a", "-shared",
                   "-Xcompiler", "-fPIC", "-o", DEV_LIB, cu]
            subprocess.run(cmd, check=True, capture_output=not verbose)


def _stale(out: str, srcs: list[str]) -> bool:
    if not os.path.exists(out):
        return True
    t = os.path.getmtime(out)
    return any(os.path.getmtime(s) > t for s in srcs)


_host = None
_dev = None


def host_lib() -> ctypes.CDLL:
    global _host
    if _host is None:
        build(device=False)
        lib = ctypes.CDLL(HOST_LIB)
        u16p, i32p = ctypes.POINTER(ctypes.c_uint16), ctypes.POINTER(ctypes.c_int32)
        lib.synth_fill.argtypes = [u16p, ctypes.c_int64, ctypes.c_uint64, ctypes.c_uint64, u16p, ctypes.c_int]
        lib.synth_kv_logical.argtypes = [u16p, u16p, ctypes.c_int64, i32p, i32p, ctypes.c_int, ctypes.c_int,
                                         ctypes.c_int, ctypes.c_uint64, u16p, ctypes.c_int]
        lib.synth_kv_pool_layer.argtypes = [u16p, ctypes.c_int64, i32p, i32p, ctypes.c_int, ctypes.c_int,
                                            ctypes.c_int, ctypes.c_int, ctypes.c_uint64, u16p, ctypes.c_int]
        lib.synth_weight_tid.restype = ctypes.c_uint64
        lib.synth_weight_tid.argtypes = [ctypes.c_int, ctypes.c_int]
        _host = lib
    return _host


def dev_lib() -> ctypes.CDLL:
    global _dev
    if _dev is None:
        build(device=True)
        lib = ctypes.CDLL(DEV_LIB)
        vp = ctypes.c_void_p
        lib.synth_dev_fill.argtypes = [vp, ctypes.c_int64, ctypes.c_uint64, ctypes.c_uint64, vp, vp]
        lib.synth_dev_kv_pool_layer.argtypes = [vp, ctypes.c_int64, vp, vp, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                                ctypes.c_int, ctypes.c_uint64, vp, vp]
        _dev = lib
    return _dev


def _nthreads() -> int:
    return max(1, min(64, os.cpu_count() or 1))


def _p(a: np.ndarray, t):
    return a.ctypes.data_as(ctypes.POINTER(t))


# --------------------------------------------------------------------------- tables
def f64_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float64 values to bf16 (round to nearest, ties to even); return bit patterns."""
    x = np.asarray(x, dtype=np.float64)
    m, e = np.frexp(x)                      # x = m * 2^e, 0.5 <= |m| < 1
    q = np.rint(m * 256.0)                  # 8 significant bits, ties to even
    v = np.ldexp(q / 256.0, e)              # exactly representable in bf16
    return (v.astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)


def bf16_bits_to_f64(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def quantile_table(scale: float = 1.0, offset: float = 0.0) -> np.ndarray:
    from scipy.special import ndtri
    p = (np.arange(65536, dtype=np.float64) + 0.5) / 65536.0
    return f64_to_bf16_bits(offset + scale * ndtri(p))


@dataclass
class Tables:
    kv: np.ndarray      # N(0, 1)
    w: np.ndarray       # N(0, 0.02)
    g: np.ndarray       # 1 + gain_std * N(0, 1)
    qkv: np.ndarray | None = None   # W_qkv draws when set (N(0, qkv_std)), else those of `w`

    @staticmethod
    def make(gain_std: float = 0.0, qkv_std: float | None = None) -> "Tables":
        """qkv_std: draw W_qkv at this std instead of 0.02.  Wider query/key projections give scores
        q.k / sqrt(hd) tens of units apart, the peaked attention of a trained scorer."""
        kv = quantile_table(1.0)
        w = quantile_table(0.02)
        g = quantile_table(gain_std, 1.0) if gain_std > 0 else np.full(65536, 0x3F80, dtype=np.uint16)
        qkv = quantile_table(qkv_std) if qkv_std is not None else None
        return Tables(kv, w, g, qkv)

    def for_kind(self, kind: int) -> np.ndarray:
        if kind in GAIN_KINDS:
            return self.g
        if kind == W_QKV and self.qkv is not None:
            return self.qkv
        return self.w


# --------------------------------------------------------------------------- architectures
@dataclass(frozen=True)
class Arch:
    n_layers: int
    d_model: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    d_ff: int
    rope_base: float = 1e4
    rms_eps: float = 1e-6
    page_size: int = 16
    lora_rank: int = 0          # 0: merged scorer weights; else an adapter of this rank on every projection
    lora_alpha: float = 32.0    # adapter scale alpha / rank
    qk_norm: bool = False       # per-head RMSNorm of q and k (gains [head_dim] per layer) before RoPE

    @property
    def lora_scale(self) -> float:
        return self.lora_alpha / self.lora_rank if self.lora_rank else 0.0

    def layer_kinds(self) -> tuple[int, ...]:
        return LAYER_KINDS + (LORA_KINDS if self.lora_rank else ()) + (QK_NORM_KINDS if self.qk_norm else ())

    @property
    def qkv_rows(self) -> int:
        return (self.n_q_heads + 2 * self.n_kv_heads) * self.head_dim

    def weight_shape(self, kind: int) -> tuple[int, ...]:
        d, hd, r = self.d_model, self.head_dim, self.lora_rank
        return {
            EMBED: (d,), FINAL_NORM: (d,), W_PLUS: (d,), W_MINUS: (d,), ATTN_NORM: (d,),
            W_QKV: (self.qkv_rows, d), W_O: (d, self.n_q_heads * hd), MLP_NORM: (d,),
            W_GATE_UP: (2 * self.d_ff, d), W_DOWN: (d, self.d_ff),
            LORA_A_QKV: (r, d), LORA_B_QKV: (self.qkv_rows, r), LORA_A_O: (r, self.n_q_heads * hd), LORA_B_O: (d, r),
            LORA_A_GATE_UP: (r, d), LORA_B_GATE_UP: (2 * self.d_ff, r), LORA_A_DOWN: (r, self.d_ff),
            LORA_B_DOWN: (d, r), Q_NORM: (hd,), K_NORM: (hd,),
        }[kind]

    def weight_bytes(self) -> int:
        per_layer = sum(int(np.prod(self.weight_shape(k))) for k in self.layer_kinds())
        top = sum(int(np.prod(self.weight_shape(k))) for k in (EMBED, FINAL_NORM, W_PLUS, W_MINUS))
        return 2 * (self.n_layers * per_layer + top)

    def kv_bytes_per_token(self) -> int:
        return self.n_layers * 2 * self.n_kv_heads * self.head_dim * 2


ARCH_TINY = Arch(2, 256, 4, 2, 64, 1024)
ARCH_1P5B = Arch(28, 1536, 12, 2, 128, 8960)
ARCH_7B = Arch(28, 3584, 28, 4, 128, 18944)
ARCH_8B = Arch(32, 4096, 32, 8, 128, 14336)


# --------------------------------------------------------------------------- workloads
@dataclass
class Workload:
    """Candidates' logical token identities plus their paging into a shuffled pool."""
    name: str
    arch: Arch
    seed: int
    cand_seg: list[np.ndarray]          # per candidate: segment id of each logical position
    cand_off: list[np.ndarray]          # per candidate: offset within that segment
    block_table: np.ndarray = field(default=None)   # int32 [B][max_blocks], -1 where unused
    seq_lens: np.ndarray = field(default=None)      # int32 [B]
    page_seg: np.ndarray = field(default=None)      # int32 [n_pages][P], -1 = empty slot
    page_off: np.ndarray = field(default=None)      # int32 [n_pages][P]
    gain_std: float = 0.0

    @property
    def n_candidates(self) -> int:
        return len(self.cand_seg)

    @property
    def n_pages(self) -> int:
        return int(self.page_seg.shape[0])

    @property
    def max_blocks(self) -> int:
        return int(self.block_table.shape[1])

    def logical_tokens(self) -> int:
        return int(self.seq_lens.sum())

    def unique_kv_bytes(self) -> int:
        """Bytes of the pages the block tables reference (each counted once), all layers."""
        P = self.arch.page_size
        used = set()
        for b in range(self.n_candidates):
            nb = (int(self.seq_lens[b]) + P - 1) // P
            used.update(self.block_table[b, :nb].tolist())
        return len(used) * P * self.arch.kv_bytes_per_token()

    def logical_kv_bytes(self) -> int:
        return self.logical_tokens() * self.arch.kv_bytes_per_token()


def _segments_to_tokens(segs: list[tuple[int, int]]) -> tuple[np.ndarray, np.ndarray]:
    if not segs:
        return np.zeros(0, np.int32), np.zeros(0, np.int32)
    seg = np.concatenate([np.full(n, s, np.int32) for s, n in segs])
    off = np.concatenate([np.arange(n, dtype=np.int32) for s, n in segs])
    return seg, off


def paginate(w: Workload, extra_pages: int = 3, max_blocks: int | None = None) -> Workload:
    """Assign physical pages: pages with identical token content are shared, the
    physical ids are a seeded permutation, and a few never-referenced decoy pages
    are added.  A partially shared page (a parent's tail followed by a child's
    first tokens) is its own page per distinct content (copy-on-write)."""
    P = w.arch.page_size
    rng = np.random.default_rng(w.seed + 7)
    content: dict[bytes, int] = {}
    uniq_seg, uniq_off = [], []
    logical = []
    for seg, off in zip(w.cand_seg, w.cand_off):
        L = len(seg)
        ids = []
        for j in range((L + P - 1) // P):
            s = np.full(P, -1, np.int32)
            o = np.full(P, -1, np.int32)
            n = min(P, L - j * P)
            s[:n] = seg[j * P:j * P + n]
            o[:n] = off[j * P:j * P + n]
            key = s.tobytes() + o.tobytes()
            u = content.get(key)
            if u is None:
                u = len(uniq_seg)
                content[key] = u
                uniq_seg.append(s)
                uniq_off.append(o)
            ids.append(u)
        logical.append(ids)
    n_uniq = len(uniq_seg)
    n_pages = n_uniq + extra_pages
    perm = rng.permutation(n_pages).astype(np.int32)
    page_seg = np.empty((n_pages, P), np.int32)
    page_off = np.empty((n_pages, P), np.int32)
    for u in range(n_uniq):
        page_seg[perm[u]] = uniq_seg[u]
        page_off[perm[u]] = uniq_off[u]
    decoy_seg = (1 << 20) - 1
    for k in range(extra_pages):
        page_seg[perm[n_uniq + k]] = decoy_seg
        page_off[perm[n_uniq + k]] = np.arange(P, dtype=np.int32) + k * P
    mb = max([len(x) for x in logical] + [1])
    if max_blocks is not None:
        assert max_blocks >= mb
        mb = max_blocks
    bt = np.full((len(logical), mb), -1, np.int32)
    for b, ids in enumerate(logical):
        if ids:
            bt[b, :len(ids)] = perm[np.asarray(ids)]
    w.block_table = bt
    w.seq_lens = np.asarray([len(s) for s in w.cand_seg], np.int32)
    w.page_seg, w.page_off = page_seg, page_off
    return w


def workload_from_segments(name: str, arch: Arch, seed: int, segs_per_cand: list[list[tuple[int, int]]],
                           gain_std: float = 0.0, extra_pages: int = 3, max_blocks: int | None = None) -> Workload:
    cs, co = [], []
    for segs in segs_per_cand:
        s, o = _segments_to_tokens(segs)
        cs.append(s)
        co.append(o)
    return paginate(Workload(name, arch, seed, cs, co, gain_std=gain_std), extra_pages, max_blocks)


def distinct(name: str, arch: Arch, seed: int, lens: list[int], **kw) -> Workload:
    """Each candidate owns one segment (a distinct cache)."""
    return workload_from_segments(name, arch, seed, [[(b, L)] if L > 0 else [] for b, L in enumerate(lens)], **kw)


def shared_prefix(name: str, arch: Arch, seed: int, B: int, prefix: int, suffix: int, **kw) -> Workload:
    """Beam step: every candidate = one shared prefix segment + its own suffix segment."""
    return workload_from_segments(name, arch, seed, [[(0, prefix), (1 + b, suffix)] for b in range(B)], **kw)


def mcts_tree(name: str, arch: Arch, seed: int, branching: int = 4, depth: int = 4, lo: int = 256, hi: int = 2048,
              **kw) -> Workload:
    """Leaves of a complete `branching`-ary tree of `depth` edge levels; each edge is
    a segment with a seeded uniform integer length in [lo, hi]; leaves in tree order."""
    rng = np.random.default_rng(seed)
    paths = [[]]
    next_seg = 0
    for _ in range(depth):
        new = []
        for p in paths:
            for _c in range(branching):
                n = int(rng.integers(lo, hi + 1))
                new.append(p + [(next_seg, n)])
                next_seg += 1
        paths = new
    return workload_from_segments(name, arch, seed, paths, **kw)


WORKLOAD_NAMES = ("tiny", "qwen1p5b_b16_l2048", "beam7b_b64_p4096_s512", "long8b_b8_l32768", "mcts7b_b256_d4")


def make_workload(name: str, gain_std: float = 0.0) -> Workload:
    """The five scoring workloads (seed = 1000 + index)."""
    i = WORKLOAD_NAMES.index(name)
    seed = 1000 + i
    if name == "tiny":
        return distinct(name, ARCH_TINY, seed, [128] * 4, gain_std=gain_std)
    if name == "qwen1p5b_b16_l2048":
        return distinct(name, ARCH_1P5B, seed, [2048] * 16, gain_std=gain_std)
    if name == "beam7b_b64_p4096_s512":
        return shared_prefix(name, ARCH_7B, seed, 64, 4096, 512, gain_std=gain_std)
    if name == "long8b_b8_l32768":
        return distinct(name, ARCH_8B, seed, [32768] * 8, gain_std=gain_std)
    if name == "mcts7b_b256_d4":
        return mcts_tree(name, ARCH_7B, seed, gain_std=gain_std)
    raise KeyError(name)


# --------------------------------------------------------------------------- host fills
def host_weight(arch: Arch, kind: int, layer: int, seed: int, tables: Tables) -> np.ndarray:
    shape = arch.weight_shape(kind)
    out = np.empty(int(np.prod(shape)), np.uint16)
    lib = host_lib()
    tid = lib.synth_weight_tid(kind, layer if kind >= ATTN_NORM else 0)
    table = tables.for_kind(kind)
    lib.synth_fill(_p(out, ctypes.c_uint16), out.size, seed, tid, _p(table, ctypes.c_uint16), _nthreads())
    return out.reshape(shape)


def host_weights(arch: Arch, seed: int, tables: Tables) -> dict:
    """All weights as bf16 bit arrays: {'top': {kind: arr}, 'layers': [{kind: arr}]}"""
    top = {k: host_weight(arch, k, 0, seed, tables) for k in (EMBED, FINAL_NORM, W_PLUS, W_MINUS)}
    layers = [{k: host_weight(arch, k, l, seed, tables) for k in arch.layer_kinds()} for l in range(arch.n_layers)]
    return {"top": top, "layers": layers}


def host_kv_logical(w: Workload, layer: int, cand: int, tables: Tables) -> tuple[np.ndarray, np.ndarray]:
    a = w.arch
    L = len(w.cand_seg[cand])
    K = np.empty((L, a.n_kv_heads, a.head_dim), np.uint16)
    V = np.empty_like(K)
    seg = np.ascontiguousarray(w.cand_seg[cand], np.int32)
    off = np.ascontiguousarray(w.cand_off[cand], np.int32)
    host_lib().synth_kv_logical(_p(K, ctypes.c_uint16), _p(V, ctypes.c_uint16), L, _p(seg, ctypes.c_int32),
                                _p(off, ctypes.c_int32), a.n_kv_heads, a.head_dim, layer, w.seed,
                                _p(tables.kv, ctypes.c_uint16), _nthreads())
    return K, V


def host_kv_pool(w: Workload, tables: Tables, layers: list[int] | None = None) -> np.ndarray:
    """Paged pool [N_L][n_pages][2][n_kv][P][hd] as bf16 bits (small workloads only)."""
    a = w.arch
    layers = list(range(a.n_layers)) if layers is None else layers
    pool = np.empty((len(layers), w.n_pages, 2, a.n_kv_heads, a.page_size, a.head_dim), np.uint16)
    ps = np.ascontiguousarray(w.page_seg, np.int32)
    po = np.ascontiguousarray(w.page_off, np.int32)
    for i, l in enumerate(layers):
        host_lib().synth_kv_pool_layer(_p(pool[i], ctypes.c_uint16), w.n_pages, _p(ps, ctypes.c_int32),
                                       _p(po, ctypes.c_int32), a.page_size, a.n_kv_heads, a.head_dim, l, w.seed,
                                       _p(tables.kv, ctypes.c_uint16), _nthreads())
    return pool


# --------------------------------------------------------------------------- device fills
class DeviceInputs:
    """Weights and the paged K/V pool generated directly in HBM (torch tensors)."""

    def __init__(self, w: Workload, tables: Tables, device: str = "cuda:0", stream=None, pool_slack_pages: int = 0):
        import torch
        self.w, self.arch = w, w.arch
        a = w.arch
        dev = torch.device(device)
        self.stream = stream if stream is not None else torch.cuda.current_stream(dev)
        sp = ctypes.c_void_p(self.stream.cuda_stream)
        lib = dev_lib()
        t_kv = torch.from_numpy(tables.kv.view(np.int16)).to(dev)
        t_w = torch.from_numpy(tables.w.view(np.int16)).to(dev)
        t_g = torch.from_numpy(tables.g.view(np.int16)).to(dev)
        t_q = torch.from_numpy(tables.qkv.view(np.int16)).to(dev) if tables.qkv is not None else t_w
        hl = host_lib()

        def fill(kind, layer):
            shape = a.weight_shape(kind)
            t = torch.empty(shape, dtype=torch.bfloat16, device=dev)
            tid = hl.synth_weight_tid(kind, layer if kind >= ATTN_NORM else 0)
            table = t_g if kind in GAIN_KINDS else (t_q if kind == W_QKV else t_w)
            rc = lib.synth_dev_fill(t.data_ptr(), t.numel(), w.seed, tid, table.data_ptr(), sp)
            assert rc == 0, rc
            return t

        self.top = {k: fill(k, 0) for k in (EMBED, FINAL_NORM, W_PLUS, W_MINUS)}
        self.layers = [{k: fill(k, l) for k in a.layer_kinds()} for l in range(a.n_layers)]
        P = a.page_size
        self.n_pages = w.n_pages + pool_slack_pages
        self.pool = torch.empty((a.n_layers, self.n_pages, 2, a.n_kv_heads, P, a.head_dim), dtype=torch.bfloat16,
                                device=dev)
        pseg = np.full((self.n_pages, P), -1, np.int32)
        poff = np.zeros((self.n_pages, P), np.int32)
        pseg[:w.n_pages] = w.page_seg
        poff[:w.n_pages] = w.page_off
        d_seg = torch.from_numpy(pseg).to(dev)
        d_off = torch.from_numpy(poff).to(dev)
        for l in range(a.n_layers):
            rc = lib.synth_dev_kv_pool_layer(self.pool[l].data_ptr(), self.n_pages, d_seg.data_ptr(),
                                             d_off.data_ptr(), P, a.n_kv_heads, a.head_dim, l, w.seed,
                                             t_kv.data_ptr(), sp)
            assert rc == 0, rc
        self.stream.synchronize()
        del d_seg, d_off, t_kv, t_w, t_g, t_q


# --------------------------------------------------------------------------- oracle providers
class SynthModel(ctypes.Structure):
    """Mirror of synth.c's `synth_model` (weights and per-candidate token identities)."""
    _fields_ = [
        ("seed", ctypes.c_uint64),
        ("table_w", ctypes.POINTER(ctypes.c_uint16)),
        ("table_g", ctypes.POINTER(ctypes.c_uint16)),
        ("table_kv", ctypes.POINTER(ctypes.c_uint16)),
        ("nthreads", ctypes.c_int),
        ("n_kv", ctypes.c_int),
        ("hd", ctypes.c_int),
        ("n_cand", ctypes.c_int),
        ("cand_len", ctypes.POINTER(ctypes.c_int64)),
        ("cand_seg", ctypes.POINTER(ctypes.POINTER(ctypes.c_int32))),
        ("cand_off", ctypes.POINTER(ctypes.POINTER(ctypes.c_int32))),
        ("table_qkv", ctypes.POINTER(ctypes.c_uint16)),
    ]


class Providers:
    """C function pointers + user data that feed a workload's weights and logical
    K/V (by token identity, not by page) to a consumer such as the oracle."""

    def __init__(self, w: Workload, tables: Tables, nthreads: int | None = None):
        lib = host_lib()
        a = w.arch
        self._keep = [tables.w, tables.g, tables.kv, tables.qkv]
        segs = [np.ascontiguousarray(s, np.int32) for s in w.cand_seg]
        offs = [np.ascontiguousarray(o, np.int32) for o in w.cand_off]
        self._keep += segs + offs
        i32p = ctypes.POINTER(ctypes.c_int32)
        seg_arr = (i32p * len(segs))(*[_p(s, ctypes.c_int32) for s in segs])
        off_arr = (i32p * len(offs))(*[_p(o, ctypes.c_int32) for o in offs])
        lens = np.asarray([len(s) for s in segs], np.int64)
        self._keep += [seg_arr, off_arr, lens]
        self.model = SynthModel(w.seed, _p(tables.w, ctypes.c_uint16), _p(tables.g, ctypes.c_uint16),
                                _p(tables.kv, ctypes.c_uint16), nthreads or _nthreads(), a.n_kv_heads, a.head_dim,
                                len(segs), _p(lens, ctypes.c_int64), seg_arr, off_arr,
                                _p(tables.qkv, ctypes.c_uint16) if tables.qkv is not None else None)
        self.weight_fn = ctypes.cast(lib.synth_weight_provider, ctypes.c_void_p).value
        self.kv_fn = ctypes.cast(lib.synth_kv_provider, ctypes.c_void_p).value
        self.user = ctypes.cast(ctypes.pointer(self.model), ctypes.c_void_p).value
