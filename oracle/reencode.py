"""Brute-force full causal re-encode -- TEST INFRASTRUCTURE ONLY.

The paper's premise (Sec. 1 and Sec. 4.1): scoring appends one verify token to
the end of the trajectory and reads the generator's cache instead of
re-encoding.  So the verify-against-cache result must equal what the same
decoder computes at the last position when the whole sequence
[x_0 .. x_{L-1}, v] is run through a plain causal forward (the Text-PRM style
computation of Eq. flops_forward, O(L^2)).  This module is that plain forward,
written independently of the C oracle with PyTorch CPU library routines in
float64 (``scaled_dot_product_attention`` with a causal mask and grouped
heads, ``rms_norm``, ``silu``); with ``arch.qk_norm`` each head's q and k are
RMS-normalised (``rms_norm`` over head_dim, gains of kinds 18 and 19) before RoPE.  It returns the last position's P(+) and
attention outputs and the per-layer key/value cache of positions < L, which is
what a generator would have left behind.

Rounding: cached keys/values are stored in bf16 (a bf16 model's cache).  With
``mirror=True`` the bf16 roundings of the precision contract are applied at
every position (projection inputs, q, k, v, attention output, SiLU product,
final x); with ``mirror=False`` only the cache of positions < L is rounded.
"""
from __future__ import annotations

import numpy as np
import torch
import torch.nn.functional as F


def _bits_to_f64(b) -> torch.Tensor:
    u = np.asarray(b, dtype=np.uint16).astype(np.uint32) << 16
    return torch.from_numpy(u.view(np.float32).astype(np.float64))


def _to_bf16_bits(x: np.ndarray) -> np.ndarray:
    m, e = np.frexp(np.asarray(x, dtype=np.float64))
    v = np.ldexp(np.rint(m * 256.0) / 256.0, e)
    return (v.astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)


def round_bf16(x: torch.Tensor) -> torch.Tensor:
    """Direct float64 -> bf16 rounding (nearest, ties to even), returned as float64."""
    return _bits_to_f64(_to_bf16_bits(x.numpy())).reshape(x.shape)


def _rope_tables(T: int, hd: int, base: float):
    inv = base ** (-torch.arange(0, hd, 2, dtype=torch.float64) / hd)     # [hd/2]
    ang = torch.arange(T, dtype=torch.float64)[:, None] * inv[None, :]     # [T, hd/2]
    ang = torch.cat([ang, ang], dim=-1)                                    # [T, hd]
    return ang.cos(), ang.sin()


def _rotate_half(x: torch.Tensor) -> torch.Tensor:
    h = x.shape[-1] // 2
    return torch.cat([-x[..., h:], x[..., :h]], dim=-1)


def reencode(arch, weights: dict, xs: np.ndarray, mirror: bool = True, depth: int = 1):
    """Causal forward over [xs; e_v x depth] (depth verify tokens, the depth-k readout).  xs: [L, d]
    float64 hidden inputs of the trajectory.

    Returns (p_plus of the last position, attn, cache): attn [N_L, nq*hd] at the last position for
    depth 1, else [N_L, depth, nq*hd] at the verify positions; cache[l] = (K_bits, V_bits), each
    [L, nkv, hd] uint16 (post-RoPE keys)."""
    d, nq, nkv, hd, ff = arch.d_model, arch.n_q_heads, arch.n_kv_heads, arch.head_dim, arch.d_ff
    L = xs.shape[0]
    T = L + depth
    top = weights["top"]
    e_v = _bits_to_f64(top[0])
    h = torch.cat([torch.as_tensor(xs, dtype=torch.float64).reshape(L, d), e_v[None, :].expand(depth, d)], dim=0)
    cos, sin = _rope_tables(T, hd, arch.rope_base)
    rb = round_bf16 if mirror else (lambda t: t)
    cache, attn_last = [], []
    for l in range(arch.n_layers):
        lw = weights["layers"][l]
        g_attn, g_mlp = _bits_to_f64(lw[4]), _bits_to_f64(lw[7])
        W_qkv = _bits_to_f64(lw[5]).reshape(-1, d)
        W_o = _bits_to_f64(lw[6]).reshape(d, nq * hd)
        W_gu = _bits_to_f64(lw[8]).reshape(2 * ff, d)
        W_d = _bits_to_f64(lw[9]).reshape(d, ff)

        x = rb(F.rms_norm(h, (d,), weight=g_attn, eps=arch.rms_eps))
        qkv = x @ W_qkv.T
        q = qkv[:, :nq * hd].reshape(T, nq, hd)
        k = qkv[:, nq * hd:(nq + nkv) * hd].reshape(T, nkv, hd)
        v = qkv[:, (nq + nkv) * hd:].reshape(T, nkv, hd)
        if getattr(arch, "qk_norm", False):   # per-head RMSNorm of q and k (gains kinds 18, 19) before RoPE
            q = F.rms_norm(q, (hd,), weight=_bits_to_f64(lw[18]), eps=arch.rms_eps)
            k = F.rms_norm(k, (hd,), weight=_bits_to_f64(lw[19]), eps=arch.rms_eps)
        q = q * cos[:, None, :] + _rotate_half(q) * sin[:, None, :]
        k = k * cos[:, None, :] + _rotate_half(k) * sin[:, None, :]
        if mirror:
            q, k, v = rb(q), rb(k), rb(v)
        else:
            k = torch.cat([round_bf16(k[:L]), k[L:]], dim=0)
            v = torch.cat([round_bf16(v[:L]), v[L:]], dim=0)
        cache.append((_to_bf16_bits(k[:L].numpy()), _to_bf16_bits(v[:L].numpy())))
        o = F.scaled_dot_product_attention(q.transpose(0, 1)[None], k.transpose(0, 1)[None],
                                           v.transpose(0, 1)[None], is_causal=True, enable_gqa=True)
        o = o[0].transpose(0, 1).reshape(T, nq * hd)
        attn_last.append(o[L].clone() if depth == 1 else o[L:].clone())
        h = h + rb(o) @ W_o.T
        x = rb(F.rms_norm(h, (d,), weight=g_mlp, eps=arch.rms_eps))
        gu = x @ W_gu.T
        a = rb(F.silu(gu[:, :ff]) * gu[:, ff:])
        h = h + a @ W_d.T
    x = rb(F.rms_norm(h[T - 1:T], (d,), weight=_bits_to_f64(top[1]), eps=arch.rms_eps))[0]
    z = torch.stack([x @ _bits_to_f64(top[3]), x @ _bits_to_f64(top[2])])     # [z_-, z_+]
    p_plus = torch.softmax(z, dim=0)[1].item()
    return p_plus, torch.stack(attn_last).numpy(), cache
