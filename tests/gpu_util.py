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
                      "w_gate_up": L[ks.W_GATE_UP], "w_down": L[ks.W_DOWN]} for L in dev.layers]}
    sc = Scorer(a.n_layers, a.d_model, a.n_q_heads, a.n_kv_heads, a.head_dim, a.d_ff, wt, max_candidates, max_blocks,
                a.rope_base, a.rms_eps)
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
