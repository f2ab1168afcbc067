"""Pins for the CPU oracle: checks against facts the paper and the mathematics
fix, written as plain functions so the mutation tests can run them against
oracle builds with planted mistakes.  Each raises AssertionError on failure."""
from __future__ import annotations

import math

import numpy as np
import torch
import torch.nn.functional as F

import kvsynth as ks
import oracle
from oracle.reencode import reencode

RNG = np.random.default_rng(20260101)


def _bits(x):
    return ks.f64_to_bf16_bits(np.asarray(x, dtype=np.float64))


def pin_bf16_round(m=0):
    # ties to even around 1.0 (bf16 spacing 2^-7 there) and torch's own fp32->bf16 rounding
    assert oracle.bf16_round(1.0 + 2.0 ** -8, m) == 1.0
    assert oracle.bf16_round(1.0 + 3 * 2.0 ** -8, m) == 1.0 + 2.0 ** -6
    assert oracle.bf16_round(-(1.0 + 3 * 2.0 ** -8), m) == -(1.0 + 2.0 ** -6)
    x = RNG.normal(0, 3, 2000).astype(np.float32)
    ref = torch.from_numpy(x).to(torch.bfloat16).double().numpy()
    got = np.array([oracle.bf16_round(float(v), m) for v in x])
    assert np.array_equal(got, ref)


def pin_rmsnorm(m=0):
    d, eps = 64, 1e-6
    g = _bits(RNG.normal(1, 0.2, d))
    gf = ks.bf16_bits_to_f64(g)
    for c in (0.5, -3.0, 1e-3):
        out = oracle.rmsnorm(np.full(d, c), g, eps, m)
        np.testing.assert_allclose(out, c / math.sqrt(c * c + eps) * gf, rtol=1e-14, atol=0)
    h = RNG.normal(0, 1, d)
    ref = F.rms_norm(torch.from_numpy(h), (d,), weight=torch.from_numpy(gf), eps=eps).numpy()
    np.testing.assert_allclose(oracle.rmsnorm(h, g, eps, m), ref, rtol=1e-13)


def pin_rope(m=0):
    hd, base = 64, 1e4
    x = RNG.normal(0, 1, hd)
    np.testing.assert_array_equal(oracle.rope(x, 0.0, base, m), x)
    for p in (1.0, 17.0, 4096.0, 32768.0):
        np.testing.assert_allclose(np.linalg.norm(oracle.rope(x, p, base, m)), np.linalg.norm(x), rtol=1e-13)
    # one pair (hd = 2): a plain rotation by `pos` radians
    r = oracle.rope(np.array([1.0, 0.0]), 0.7, base, m)
    np.testing.assert_allclose(r, [math.cos(0.7), math.sin(0.7)], rtol=1e-15, atol=1e-16)
    # relative position: <R(m)q, R(n)k> depends on m - n only
    q, k = RNG.normal(0, 1, hd), RNG.normal(0, 1, hd)
    a = oracle.rope(q, 100.0, base, m) @ oracle.rope(k, 90.0, base, m)
    b = oracle.rope(q, 1010.0, base, m) @ oracle.rope(k, 1000.0, base, m)
    assert abs(a - b) < 1e-10 * (1 + abs(a))


def pin_attend(m=0):
    hd = 64
    q = RNG.normal(0, 1, hd)
    ks_, vs_ = RNG.normal(0, 1, hd), RNG.normal(0, 1, hd)
    # (i) empty cache: the verify token reads its own value
    o, w = oracle.attend(q, np.zeros((0, hd), np.uint16), np.zeros((0, hd), np.uint16), ks_, vs_, m)
    np.testing.assert_array_equal(o, vs_)
    np.testing.assert_array_equal(w, [1.0])
    # (ii) identical keys (all equal to the self key): the mean of the values
    L = 9
    kb = np.tile(_bits(ks_), (L, 1))
    ksr = ks.bf16_bits_to_f64(_bits(ks_))
    V = _bits(RNG.normal(0, 1, (L, hd)))
    o, w = oracle.attend(q, kb, V, ksr, vs_, m)
    mean = (ks.bf16_bits_to_f64(V).sum(0) + vs_) / (L + 1)
    np.testing.assert_allclose(o, mean, rtol=1e-12, atol=1e-14)
    # (iii) q = 0: uniform weights
    K = _bits(RNG.normal(0, 1, (L, hd)))
    o, w = oracle.attend(np.zeros(hd), K, V, ks_, vs_, m)
    np.testing.assert_allclose(o, mean, rtol=1e-12, atol=1e-14)
    # (iv) two entries: weight of the cached one is sigmoid(s_1 - s_self)
    o, w = oracle.attend(q, K[:1], V[:1], ks_, vs_, m)
    s1 = q @ ks.bf16_bits_to_f64(K[0]) / math.sqrt(hd)
    s2 = q @ ks_ / math.sqrt(hd)
    np.testing.assert_allclose(w[0], 1.0 / (1.0 + math.exp(s2 - s1)), rtol=1e-13)
    # (v) weights sum to one; (vi) invariance to the order of cached positions
    L = 257
    K = _bits(RNG.normal(0, 1, (L, hd)))
    V = _bits(RNG.normal(0, 1, (L, hd)))
    o, w = oracle.attend(q, K, V, ks_, vs_, m)
    assert abs(w.sum() - 1.0) < 1e-12
    perm = RNG.permutation(L)
    o2, _ = oracle.attend(q, K[perm], V[perm], ks_, vs_, m)
    np.testing.assert_allclose(o2, o, rtol=1e-12, atol=1e-14)
    # library cross-check: causal SDPA row L over [K; k_self]
    Kf = torch.from_numpy(np.vstack([ks.bf16_bits_to_f64(K), ks_[None]]))
    Vf = torch.from_numpy(np.vstack([ks.bf16_bits_to_f64(V), vs_[None]]))
    ref = F.scaled_dot_product_attention(torch.from_numpy(q)[None, None], Kf[None], Vf[None])[0, 0].numpy()
    np.testing.assert_allclose(o, ref, rtol=1e-11, atol=1e-13)


def pin_reward(m=0):
    d = 128
    x = RNG.normal(0, 1, d)
    w1 = _bits(RNG.normal(0, 0.02, d))
    w2 = _bits(RNG.normal(0, 0.02, d))
    assert oracle.reward(x, w1, w1, m) == 0.5
    p = oracle.reward(x, w1, w2, m)
    zp, zm = ks.bf16_bits_to_f64(w1) @ x, ks.bf16_bits_to_f64(w2) @ x
    ref = torch.softmax(torch.tensor([zm, zp], dtype=torch.float64), 0)[1].item()
    assert abs(p - ref) < 1e-15
    assert abs(oracle.reward(x, w2, w1, m) - (1 - p)) < 1e-15


def pin_reencode(m=0, lens=(0, 1, 5, 16, 17, 40), mirror=True, arch=None):
    """Verify-against-cache == last position of a full causal forward over [x; v]."""
    arch = arch or ks.ARCH_TINY
    t = ks.Tables.make(0.2)
    W = ks.host_weights(arch, 77, t)
    for L in lens:
        xs = np.random.default_rng(1000 + L).normal(0, 1, (L, arch.d_model))
        p, attn, cache = reencode(arch, W, xs, mirror)
        r = oracle.score_dense(arch, W, [[cache[l]] for l in range(arch.n_layers)], mirror=mirror, mutant=m)
        assert abs(p - r.p_plus[0]) < 1e-12, (L, p, r.p_plus[0])
        np.testing.assert_allclose(r.attn[:, 0], attn, rtol=1e-9, atol=1e-12)


def pin_lora_merged(m=0):
    """The scorer adapter (Sec. 4.1 f_{theta + Delta theta}; App. B.1 r, alpha) equals its merged weights:
    W x + s B (A x) = (W + s B A) x.  With A a column selection (one 1 per row) and W and s B on a grid of
    2^-10 below 256 steps, W + s B A is exactly a bf16 matrix, so the unmerged scorer (rank 64, s = 1/2)
    and the merged one must agree to fp64 rounding on every projection, in both modes."""
    import dataclasses
    base = ks.ARCH_TINY
    arch = dataclasses.replace(base, lora_rank=64)
    s, r = arch.lora_scale, arch.lora_rank
    assert s == 0.5
    rng = np.random.default_rng(515)
    W = ks.host_weights(base, 78, ks.Tables.make(0.2))
    proj = [(ks.W_QKV, ks.LORA_A_QKV, ks.LORA_B_QKV), (ks.W_O, ks.LORA_A_O, ks.LORA_B_O),
            (ks.W_GATE_UP, ks.LORA_A_GATE_UP, ks.LORA_B_GATE_UP), (ks.W_DOWN, ks.LORA_A_DOWN, ks.LORA_B_DOWN)]
    unmerged = {"top": W["top"], "layers": []}
    merged = {"top": W["top"], "layers": []}
    for l in range(arch.n_layers):
        lu, lm = dict(W["layers"][l]), dict(W["layers"][l])
        for kw, ka, kb in proj:
            rows, cols = base.weight_shape(kw)
            w0 = rng.integers(-100, 101, (rows, cols)) * 2.0 ** -10
            b = rng.integers(-100, 101, (rows, r)) * 2.0 ** -10 / s
            sel = rng.choice(cols, r, replace=False)
            a = np.zeros((r, cols))
            a[np.arange(r), sel] = 1.0
            wm = w0.copy()
            wm[:, sel] += s * b
            for v in (w0, a, b, wm):   # every value is a bf16 number
                assert np.array_equal(ks.bf16_bits_to_f64(_bits(v)), v)
            lu[kw], lu[ka], lu[kb] = _bits(w0), _bits(a), _bits(b)
            lm[kw] = _bits(wm)
        unmerged["layers"].append(lu)
        merged["layers"].append(lm)
    kv_rng = np.random.default_rng(516)
    lens = (0, 7, 33)
    kv = [[tuple(_bits(kv_rng.normal(0, 1, (L, base.n_kv_heads, base.head_dim))) for _ in range(2)) for L in lens]
          for _ in range(base.n_layers)]
    for mirror in (False, True):
        ru = oracle.score_dense(arch, unmerged, kv, mirror=mirror, mutant=m)
        rm = oracle.score_dense(base, merged, kv, mirror=mirror, mutant=m)
        assert np.abs(ru.p_plus - rm.p_plus).max() < 1e-12, (mirror, ru.p_plus, rm.p_plus)
        np.testing.assert_allclose(ru.attn, rm.attn, rtol=1e-9, atol=1e-12)
    # and the adapter is not a no-op on these weights
    rb = oracle.score_dense(base, {"top": W["top"], "layers": [
        {k: v for k, v in lu.items() if k < ks.LORA_A_QKV} for lu in unmerged["layers"]]}, kv, mirror=False, mutant=m)
    assert np.abs(rb.p_plus - rm.p_plus).max() > 1e-6


def pin_depth_reencode(m=0, depth=3, lens=(0, 5, 17)):
    """Depth-k readout (Sec. 3 R_k; Sec. 5, k > 1 verify tokens) == the last k positions of a full causal
    forward over [x; v, .., v]: verify token t sits at position L + t and sees the cache and tokens 0..t."""
    arch = ks.ARCH_TINY
    t = ks.Tables.make(0.2)
    W = ks.host_weights(arch, 79, t)
    for mirror in (True, False):
        for L in lens:
            xs = np.random.default_rng(2000 + L).normal(0, 1, (L, arch.d_model))
            p, attn, cache = reencode(arch, W, xs, mirror, depth=depth)
            r = oracle.score_dense(arch, W, [[cache[l]] for l in range(arch.n_layers)], mirror=mirror, mutant=m,
                                   depth=depth)
            assert abs(p - r.p_plus[0]) < 1e-12, (L, mirror, p, r.p_plus[0])
            np.testing.assert_allclose(r.attn, attn, rtol=1e-9, atol=1e-12)


def pin_qk_norm(m=0):
    """With the per-head q/k RMSNorm (the paper's Qwen3 scorers) the verify-against-cache path still
    equals the last position of the full causal re-encode, which normalises with torch's rms_norm; the
    gains are drawn 1 + 0.2 N(0, 1), so a norm placed after RoPE or a swapped gain changes the result."""
    import dataclasses
    arch = dataclasses.replace(ks.ARCH_TINY, qk_norm=True)
    for mirror in (False, True):
        pin_reencode(m, lens=(0, 5, 17, 40), mirror=mirror, arch=arch)
    # the norm must change the result: the same weights without it score differently
    t = ks.Tables.make(0.2)
    W = ks.host_weights(arch, 77, t)
    xs = np.random.default_rng(5).normal(0, 1, (17, arch.d_model))
    p_on, _, _ = reencode(arch, W, xs, False)
    p_off, _, _ = reencode(ks.ARCH_TINY, W, xs, False)
    assert abs(p_on - p_off) > 1e-6


# ---------------------------------------------------------------- KV Steering gradient (oracle/kvgrad.py)
def _grad_case(seed=91, lens=(20, 7), arch=None):
    """Tiny scorer with random gains and a random bf16 cache of the given lengths per candidate."""
    arch = arch or ks.ARCH_TINY
    t = ks.Tables.make(0.2)
    W = ks.host_weights(arch, seed, t)
    rng = np.random.default_rng(seed)
    kv = [[(ks.f64_to_bf16_bits(rng.normal(0, 1, (L, arch.n_kv_heads, arch.head_dim))),
            ks.f64_to_bf16_bits(rng.normal(0, 1, (L, arch.n_kv_heads, arch.head_dim)))) for L in lens]
          for _ in range(arch.n_layers)]
    return arch, W, kv


def pin_grad_forward(m=0):
    """The gradient oracle's own forward gives the C oracle's P(+) (two independent restatements of
    Eq. score)."""
    from oracle import kvgrad
    arch, W, kv = _grad_case()
    p, _, _ = kvgrad.score_grad(arch, W, kv, mutant=m if m >= 21 else 0)
    r = oracle.score_dense(arch, W, kv, mirror=False, mutant=m if m < 21 else 0)
    np.testing.assert_allclose(p, r.p_plus, rtol=0, atol=1e-12)


def pin_grad_fd(m=0):
    """Central finite differences of l = -log P(+) at sampled cached keys and values of every layer
    (steps of 1e-4 in fp64: truncation error ~1e-9 relative) equal the analytic gradient."""
    from oracle import kvgrad
    arch, W, kv = _grad_case()
    kvf = [[(kvgrad.bits_to_f64(K), kvgrad.bits_to_f64(V)) for K, V in row] for row in kv]
    p, dK, dV = kvgrad.score_grad(arch, W, kvf, mutant=m if m >= 21 else 0)
    rng = np.random.default_rng(3)
    hstep = 1e-4
    worst = 0.0
    for _ in range(24):
        l = int(rng.integers(arch.n_layers))
        b = int(rng.integers(len(kvf[0])))
        which = int(rng.integers(2))
        A = kvf[l][b][which]
        j, g, e = (int(rng.integers(n)) for n in A.shape)
        vals = []
        for sign in (1, -1):
            A[j, g, e] += sign * hstep
            vals.append(-np.log(kvgrad.score_grad(arch, W, kvf)[0][b]))
            A[j, g, e] -= sign * hstep
        fd = (vals[0] - vals[1]) / (2 * hstep)
        an = (dK if which == 0 else dV)[l][b][j, g, e]
        scale = max(np.abs(dK[l][b]).max(), np.abs(dV[l][b]).max())
        worst = max(worst, abs(fd - an) / scale)
    assert worst < 1e-6, worst


def _torch_neg_log_p(arch, W, Ks, Vs):
    """-log P(+) of one candidate written with torch library routines (rms_norm, softmax, silu) on
    cache tensors Ks[l], Vs[l] [L][n_kv][hd] that may require grad."""
    import torch.nn.functional as F
    d, nq, nkv, hd, ff = arch.d_model, arch.n_q_heads, arch.n_kv_heads, arch.head_dim, arch.d_ff
    f = lambda b: torch.from_numpy(ks.bf16_bits_to_f64(b))  # noqa: E731
    L = Ks[0].shape[0]
    inv = arch.rope_base ** (-torch.arange(0, hd, 2, dtype=torch.float64) / hd)
    ang = torch.cat([L * inv, L * inv])
    cos, sin = ang.cos(), ang.sin()
    rot = lambda x: x * cos + torch.cat([-x[..., hd // 2:], x[..., :hd // 2]], -1) * sin  # noqa: E731
    h = f(W["top"][0])
    for l in range(arch.n_layers):
        lw = W["layers"][l]
        x = F.rms_norm(h, (d,), weight=f(lw[4]), eps=arch.rms_eps)
        qkv = f(lw[5]).reshape(-1, d) @ x
        q = rot(qkv[:nq * hd].reshape(nq, hd))
        k = rot(qkv[nq * hd:(nq + nkv) * hd].reshape(nkv, hd))
        v = qkv[(nq + nkv) * hd:].reshape(nkv, hd)
        Kall = torch.cat([Ks[l], k[None]], 0)                  # [L+1][nkv][hd]
        Vall = torch.cat([Vs[l], v[None]], 0)
        Kg = Kall.repeat_interleave(nq // nkv, dim=1)          # [L+1][nq][hd]
        Vg = Vall.repeat_interleave(nq // nkv, dim=1)
        w = torch.softmax((Kg * q[None]).sum(-1) / hd ** 0.5, dim=0)   # [L+1][nq]
        o = (w[..., None] * Vg).sum(0)
        h = h + f(lw[6]).reshape(d, nq * hd) @ o.reshape(-1)
        x = F.rms_norm(h, (d,), weight=f(lw[7]), eps=arch.rms_eps)
        gu = f(lw[8]).reshape(2 * ff, d) @ x
        h = h + f(lw[9]).reshape(d, ff) @ (F.silu(gu[:ff]) * gu[ff:])
    x = F.rms_norm(h, (d,), weight=f(W["top"][1]), eps=arch.rms_eps)
    z = torch.stack([x @ f(W["top"][3]), x @ f(W["top"][2])])
    return -torch.log_softmax(z, 0)[1]


def pin_grad_autograd(m=0):
    """torch autograd through that separately written forward gives the oracle's gradient."""
    from oracle import kvgrad
    arch, W, kv = _grad_case(seed=92, lens=(13, 0, 33))
    p, dK, dV = kvgrad.score_grad(arch, W, kv, mutant=m if m >= 21 else 0)
    for b in range(len(kv[0])):
        Ks = [torch.from_numpy(ks.bf16_bits_to_f64(kv[l][b][0])).requires_grad_() for l in range(arch.n_layers)]
        Vs = [torch.from_numpy(ks.bf16_bits_to_f64(kv[l][b][1])).requires_grad_() for l in range(arch.n_layers)]
        loss = _torch_neg_log_p(arch, W, Ks, Vs)
        assert abs(loss.item() + np.log(p[b])) < 1e-12
        loss.backward()
        for l in range(arch.n_layers):
            np.testing.assert_allclose(dK[l][b], Ks[l].grad.numpy(), rtol=1e-9, atol=1e-13)
            np.testing.assert_allclose(dV[l][b], Vs[l].grad.numpy(), rtol=1e-9, atol=1e-13)


ALL_PINS = [pin_bf16_round, pin_rmsnorm, pin_rope, pin_attend, pin_reward, pin_reencode, pin_lora_merged,
            pin_depth_reencode, pin_qk_norm, pin_grad_forward, pin_grad_fd, pin_grad_autograd]
