"""Shared helpers of the GPU parity tests: run a kvsynth workload through the
C-ABI scoring library and compare with the CPU oracle."""
from __future__ import annotations

import numpy as np
import pytest

import kvsynth as ks
import oracle

P_PLUS_ATOL = 1e-3        # absolute tolerance on P(+)
ATTN_RTOL = 2e-3          # per (layer, candidate): ||o_gpu - o_ref||_inf / ||o_ref||_inf


def require_gpu():
    import torch
    if not torch.cuda.is_available():
        pytest.fail("no CUDA device: GPU tests must run on a GB300")
    return torch


def make_scorer(dev: ks.DeviceInputs, max_candidates: int, max_blocks: int):
    from paper_2607_09153_gb300 import Scorer
    a = dev.arch
    wt = {"embed_verify": dev.top[ks.EMBED], "final_norm": dev.top[ks.FINAL_NORM], "w_plus": dev.top[ks.W_PLUS],
          "w_minus": dev.top[ks.W_MINUS],
          "layers": [{"attn_norm": L[ks.ATTN_NORM], "w_qkv": L[ks.W_QKV], "w_o": L[ks.W_O], "mlp_norm": L[ks.MLP_NORM],
                      "w_gate_up": L[ks.W_GATE_UP], "w_down": L[ks.W_DOWN],
                      **({"q_norm": L[ks.Q_NORM], "k_norm": L[ks.K_NORM]} if a.qk_norm else {})} for L in dev.layers]}
    sc = Scorer(a.n_layers, a.d_model, a.n_q_heads, a.n_kv_heads, a.head_dim, a.d_ff, wt, max_candidates, max_blocks,
                a.rope_base, a.rms_eps, qk_norm=a.qk_norm)
    if a.lora_rank:   # the scorer adapter, kept apart from the weights
        names = dict(zip(ks.LORA_KINDS, ("a_qkv", "b_qkv", "a_o", "b_o", "a_gate_up", "b_gate_up", "a_down", "b_down")))
        sc.set_lora(a.lora_rank, a.lora_alpha, [{names[k]: L[k] for k in ks.LORA_KINDS} for L in dev.layers])
    return sc


def run_gpu(w: ks.Workload, tables: ks.Tables, debug: bool = True, dev=None, scorer=None, extra_flags: int = 0,
            depth: int = 1):
    """Score every candidate on the GPU; returns (rewards [B], attn [N_L][B depth][nq*hd] or None).
    extra_flags: further kvprm_set_debug bits (16: rescale on every new attention row maximum);
    depth > 1: a depth-k readout (candidate b's verify tokens are attention rows b depth + t)."""
    torch = require_gpu()
    import paper_2607_09153_gb300 as kp
    dev = dev or ks.DeviceInputs(w, tables)
    sc = scorer or make_scorer(dev, max(1, w.n_candidates * depth), w.max_blocks)
    a = w.arch
    if depth > 1:
        sc.set_depth(depth)
    if debug or extra_flags:
        kp.kvprm_set_debug(sc.ctx, (1 if debug else 0) | extra_flags)
    r = sc.score(dev.pool, w.block_table, w.seq_lens)
    attn = None
    if debug:
        out = torch.empty((a.n_layers, w.n_candidates * depth, a.n_q_heads * a.head_dim), dtype=torch.float32,
                          device="cuda")
        kp.kvprm_debug_attn_out(sc.ctx, out.data_ptr())
        torch.cuda.synchronize()
        attn = out.cpu().numpy().astype(np.float64)
    kp.kvprm_check_device(sc.ctx)
    return r.astype(np.float64), attn, dev, sc


def attn_rel_err(gpu: np.ndarray, ref: np.ndarray) -> np.ndarray:
    """[N_L][n] relative inf-norm error per (layer, candidate)."""
    num = np.abs(gpu - ref).max(axis=-1)
    den = np.abs(ref).max(axis=-1)
    return num / np.maximum(den, 1e-30)


def compare(w, tables, cand_ids=None, gpu_rewards=None, gpu_attn=None, label="", depth: int = 1):
    """Against the oracle in exact mode: bf16 weights and cache, every activation exact."""
    ids = list(range(w.n_candidates)) if cand_ids is None else list(cand_ids)
    ref = oracle.score_synth(w, tables, ids, mirror=False, depth=depth)
    dp = np.abs(gpu_rewards[ids] - ref.p_plus)
    msg = f"{label}: max |dP| = {dp.max():.3e}"
    if gpu_attn is not None:
        rows = [i * depth + t for i in ids for t in range(depth)]   # the oracle's rows, in the same order
        e = attn_rel_err(gpu_attn[:, rows], ref.attn)
        msg += f", max attn rel err = {e.max():.3e}"
        assert e.max() <= ATTN_RTOL, msg + f" (worst layer/cand {np.unravel_index(e.argmax(), e.shape)})"
    assert dp.max() <= P_PLUS_ATOL, msg
    print(msg)
    return ref


# ---------------------------------------------------------------- peaked attention inputs
class PlantedCase:
    """One layer's paged cache with planted keys, and queries aimed at them, so that the softmax of
    the attention read-out is peaked: scores q.k / sqrt(hd) tens of units apart, one key (or a run of
    identical keys) dominating, the largest score arriving late in the sequence.

    The plant is keyed by token identity (segment, offset) and applied twice, independently: to the
    paged pool (through page_seg / page_off) and to each candidate's logical K/V (through cand_seg /
    cand_off), so the block-table walk is still checked against the logical sequence."""

    def __init__(self, w: ks.Workload, tables: ks.Tables, seed: int, needles: list, runs: list = (),
                 broad_std: float = 15.0):
        a = w.arch
        self.w, self.arch = w, a
        rng = np.random.default_rng(seed)
        nkv, hd, G = a.n_kv_heads, a.head_dim, a.n_q_heads // a.n_kv_heads
        self.pool = ks.host_kv_pool(w, tables, layers=[0])[0]          # [pages][2][nkv][16][hd]
        self.K, self.V = [], []
        for b in range(w.n_candidates):
            K, V = ks.host_kv_logical(w, 0, b, tables)
            self.K.append(K)
            self.V.append(V)
        keys = {}

        def plant(seg, off, g, key_bits):
            hit = (w.page_seg == seg) & (w.page_off == off)
            pg, slot = np.nonzero(hit)
            self.pool[pg, 0, g, slot, :] = key_bits
            for b in range(w.n_candidates):
                j = np.nonzero((w.cand_seg[b] == seg) & (w.cand_off[b] == off))[0]
                self.K[b][j, g, :] = key_bits

        # needles: (seg, off) -> one key per kv head, drawn N(0, 1) and rounded to bf16
        for seg, off in needles:
            kb = ks.f64_to_bf16_bits(rng.normal(0, 1, (nkv, hd)))
            keys[(seg, off)] = kb
            for g in range(nkv):
                plant(seg, off, g, kb[g])
        # identical-key runs: (seg, off0, count) all carry the same key per kv head
        for seg, off0, count in runs:
            kb = ks.f64_to_bf16_bits(rng.normal(0, 1, (nkv, hd)))
            keys[(seg, off0)] = kb
            for off in range(off0, off0 + count):
                for g in range(nkv):
                    plant(seg, off, g, kb[g])
        # queries: per candidate the key of its latest planted identity, scaled per head so that the
        # top score is ~10 .. ~70 units above the rest; every fourth head a broad N(0, broad_std)
        # query (scores spread over tens of units without a planted target)
        B, nq = w.n_candidates, a.n_q_heads
        self.q = np.empty((B, nq, hd), np.float32)
        alphas = np.array([1.0, 2.5, 4.5, 6.0])
        for b in range(B):
            pos = {ident: max(np.nonzero((w.cand_seg[b] == ident[0]) & (w.cand_off[b] == ident[1]))[0], default=-1)
                   for ident in keys}
            target = max(pos, key=pos.get) if pos and max(pos.values()) >= 0 else None
            for h in range(nq):
                g = h // G
                if target is None or h % 4 == 3:
                    self.q[b, h] = rng.normal(0, broad_std, hd).astype(np.float32)
                else:
                    kf = ks.bf16_bits_to_f64(keys[target][g])
                    self.q[b, h] = (alphas[h % 4] * kf + rng.normal(0, 0.05, hd)).astype(np.float32)
        self.kself = rng.normal(0, 1, (B, nkv, hd)).astype(np.float32)
        self.vself = rng.normal(0, 1, (B, nkv, hd)).astype(np.float32)

    def expected(self) -> np.ndarray:
        """The oracle's read-out o [B][nq][hd] (fp64) of every (candidate, head)."""
        a = self.arch
        G = a.n_q_heads // a.n_kv_heads
        out = np.empty((self.w.n_candidates, a.n_q_heads, a.head_dim))
        for b in range(self.w.n_candidates):
            for h in range(a.n_q_heads):
                g = h // G
                out[b, h], _ = oracle.attend(self.q[b, h].astype(np.float64), self.K[b][:, g, :], self.V[b][:, g, :],
                                             self.kself[b, g].astype(np.float64), self.vself[b, g].astype(np.float64))
        return out

    def score_spread(self) -> float:
        """Largest gap between a row's top score and its median score (in units of q.k / sqrt(hd))."""
        a = self.arch
        G = a.n_q_heads // a.n_kv_heads
        gap = 0.0
        for b in range(self.w.n_candidates):
            if len(self.K[b]) == 0:
                continue
            for h in range(a.n_q_heads):
                Kf = ks.bf16_bits_to_f64(self.K[b][:, h // G, :])
                s = Kf @ self.q[b, h].astype(np.float64) / np.sqrt(a.head_dim)
                gap = max(gap, float(s.max() - np.median(s)))
        return gap

    def device(self):
        torch = require_gpu()
        pool = torch.from_numpy(self.pool.view(np.int16)).cuda()
        q, k, v = (torch.from_numpy(np.ascontiguousarray(x)).cuda() for x in (self.q, self.kself, self.vself))
        return pool, q, k, v


def row_rel_err(got: np.ndarray, ref: np.ndarray) -> float:
    """Largest per-(candidate, head) relative inf-norm error."""
    num = np.abs(got - ref).max(axis=-1)
    den = np.maximum(np.abs(ref).max(axis=-1), 1e-30)
    return float((num / den).max())
