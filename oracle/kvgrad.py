"""KV Steering oracle -- TEST INFRASTRUCTURE ONLY.

Only tests/ and bench.py's CPU-baseline leg may import this module; the CUDA
scoring library neither imports nor calls it, and the two share no code.

KV Steering (Sec. 6 "Discussion on Broader Applications of KV-PRM"; App. C,
Algorithm "KV Steering at agent handoff") treats the KV-PRM score as a
differentiable function of the cache: with loss l = -log P(+)(kv), one step is
kv <- kv - eta * grad_kv l, repeated T times.  This module computes, in plain
float64 NumPy, for each candidate b:

  * the verify-token forward of Sec. 4.1 Eq. score (the same definition as the
    C oracle, kvprm_oracle.c, written again here with every intermediate kept):
      x1 = RMSNorm(h) g_attn;  [q; k; v] = W_qkv x1;  q, k = RoPE(q, k; p = L_b)
      s_j = q_h . K_j / sqrt(hd) over the cache and the token's own key
      w = softmax(s);  o_h = sum_j w_j V_j (+ w_self v)
      h_mid = h + W_o o;  x2 = RMSNorm(h_mid) g_mlp;  [u; t] = W_gate_up x2
      h' = h_mid + W_down (SiLU(u) * t);  finally x = RMSNorm(h) g_final,
      P(+) = sigmoid(w_plus . x - w_minus . x)
  * the loss l_b = -log P(+)_b and its gradient with respect to every cached
    key K_j and value V_j of every layer, by the chain rule taken in reverse
    order of those steps (no automatic differentiation):
      dl/dz_+ = -(1 - P), dl/dz_- = 1 - P
      RMSNorm  y = h r g, r = (mean h^2 + eps)^-1/2:
               dh = r (g * dy) - h r^3 (sum_i g_i dy_i h_i) / d
      SiLU-gated MLP:  da = W_down^T dh;  du = da t SiLU'(u);  dt = da SiLU(u)
      softmax read-out, per head:  D = do . o;  ds_j = w_j (do . V_j - D)
               dV_j += w_j do;  dK_j += ds_j q / sqrt(hd);
               dq = sum_j ds_j K_j / sqrt(hd) (cache and self entry)
      RoPE backward = rotation by the negative angle.
  * Candidates that share a page (a beam prefix, MCTS ancestors) each
    contribute their own gradient to it; a batch's gradient is that of the
    summed loss sum_b l_b, so a shared page receives the sum over its
    candidates (reading of the algorithm for a batch of trajectories).

Steering keeps the cache in bf16 (the paper's precision, App. B.1): a step is
kv <- RNE_bf16(kv - eta * grad), the gradient taken at the current bf16 cache.

Scope: merged scorer weights, one verify token, no q/k norm (the forms the
GPU gradient implements).  Parity status: pinned by central finite
differences of this module's own forward, by torch autograd through a
separately written torch forward (tests/oracle_pins.py), and the forward's
P(+) by the C oracle.
"""
from __future__ import annotations

import numpy as np

# weight kinds (the providers' numbering)
EMBED, FINAL_NORM, W_PLUS, W_MINUS, ATTN_NORM, W_QKV, W_O, MLP_NORM, W_GATE_UP, W_DOWN = range(10)


def bits_to_f64(b) -> np.ndarray:
    """bf16 bit patterns -> float64 values."""
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def round_bf16(x: np.ndarray) -> np.ndarray:
    """Nearest bf16 value of each float64 (ties to even), as float64."""
    x = np.asarray(x, dtype=np.float64)
    m, e = np.frexp(x)
    return np.ldexp(np.rint(m * 256.0) / 256.0, e)


def _rmsnorm(h, g, eps):
    r = 1.0 / np.sqrt(np.mean(h * h) + eps)
    return h * r * g, r


def _rmsnorm_back(h, g, r, dy):
    """Gradient of y = h r g (r = (mean h^2 + eps)^-1/2) with respect to h."""
    return r * (g * dy) - h * (r ** 3) * np.dot(g * dy, h) / h.size


def _rope_angles(pos, hd, base):
    i = np.arange(hd // 2, dtype=np.float64)
    ang = pos * base ** (-2.0 * i / hd)
    return np.cos(ang), np.sin(ang)


def _rope(x, c, s):
    """Rotate-half pairs (i, i + hd/2) of x [..., hd] by angle (c, s)."""
    h = x.shape[-1] // 2
    a, b = x[..., :h], x[..., h:]
    return np.concatenate([a * c - b * s, b * c + a * s], axis=-1)


def _rope_back(dy, c, s):
    h = dy.shape[-1] // 2
    da, db = dy[..., :h], dy[..., h:]
    return np.concatenate([da * c + db * s, db * c - da * s], axis=-1)


def _silu(u):
    return u / (1.0 + np.exp(-u))


def _silu_prime(u):
    sg = 1.0 / (1.0 + np.exp(-u))
    return sg * (1.0 + u * (1.0 - sg))


def _as_f64(a):
    a = np.asarray(a)
    return bits_to_f64(a) if a.dtype == np.uint16 else a.astype(np.float64)


def score_grad(arch, weights: dict, kv: list, mutant: int = 0):
    """P(+), l = -log P(+) and dl/dK, dl/dV for every candidate.

    weights = {'top': {kind: bf16 bits}, 'layers': [{kind: bf16 bits}]}; kv[l][b] = (K, V), each
    [L_b][n_kv][hd] as bf16 bits or float64 values.  Returns (p_plus [n], dK, dV) with dK[l][b] and
    dV[l][b] float64 [L_b][n_kv][hd] (candidate b's logical positions; the caller adds the
    contributions of candidates that share a page).
    mutant > 0 plants one mistake in the reverse pass (used only by the tests of the pins):
    21 drops the -D term of the softmax backward, 22 rotates the RoPE backward the wrong way,
    23 drops the second term of the RMSNorm backward."""
    d, nq, nkv, hd, ff = arch.d_model, arch.n_q_heads, arch.n_kv_heads, arch.head_dim, arch.d_ff
    G = nq // nkv
    NL = arch.n_layers
    eps = arch.rms_eps
    n = len(kv[0])
    top = {k: bits_to_f64(v) for k, v in weights["top"].items()}
    lays = [{k: bits_to_f64(v) for k, v in L.items() if k in (ATTN_NORM, W_QKV, W_O, MLP_NORM, W_GATE_UP, W_DOWN)}
            for L in weights["layers"]]
    for l in range(NL):
        lays[l][W_QKV] = lays[l][W_QKV].reshape((nq + 2 * nkv) * hd, d)
        lays[l][W_O] = lays[l][W_O].reshape(d, nq * hd)
        lays[l][W_GATE_UP] = lays[l][W_GATE_UP].reshape(2 * ff, d)
        lays[l][W_DOWN] = lays[l][W_DOWN].reshape(d, ff)
    scale = 1.0 / np.sqrt(hd)
    p_plus = np.empty(n)
    dK = [[None] * n for _ in range(NL)]
    dV = [[None] * n for _ in range(NL)]
    for b in range(n):
        Ks = [_as_f64(kv[l][b][0]).reshape(-1, nkv, hd) for l in range(NL)]
        Vs = [_as_f64(kv[l][b][1]).reshape(-1, nkv, hd) for l in range(NL)]
        L = Ks[0].shape[0]
        c, s = _rope_angles(float(L), hd, arch.rope_base)
        # ---------------- forward, every intermediate kept
        h = top[EMBED].copy()
        save = []
        for l in range(NL):
            P = lays[l]
            x1, r1 = _rmsnorm(h, P[ATTN_NORM], eps)
            qkv = P[W_QKV] @ x1
            q = _rope(qkv[:nq * hd].reshape(nq, hd), c, s)
            ks = _rope(qkv[nq * hd:(nq + nkv) * hd].reshape(nkv, hd), c, s)
            vs = qkv[(nq + nkv) * hd:].reshape(nkv, hd)
            o = np.empty((nq, hd))
            w_all = np.empty((nq, L + 1))
            for hh in range(nq):
                g = hh // G
                sc = np.concatenate([Ks[l][:, g, :] @ q[hh], [ks[g] @ q[hh]]]) * scale
                w = np.exp(sc - sc.max())
                w /= w.sum()
                w_all[hh] = w
                o[hh] = w[:L] @ Vs[l][:, g, :] + w[L] * vs[g]
            h_mid = h + P[W_O] @ o.reshape(-1)
            x2, r2 = _rmsnorm(h_mid, P[MLP_NORM], eps)
            gu = P[W_GATE_UP] @ x2
            u, t = gu[:ff], gu[ff:]
            h_out = h_mid + P[W_DOWN] @ (_silu(u) * t)
            save.append((h, r1, q, ks, vs, o, w_all, h_mid, r2, u, t))
            h = h_out
        xf, rf = _rmsnorm(h, top[FINAL_NORM], eps)
        z_p, z_m = top[W_PLUS] @ xf, top[W_MINUS] @ xf
        pp = 1.0 / (1.0 + np.exp(z_m - z_p))
        p_plus[b] = pp
        # ---------------- reverse pass of l = -log P(+)
        dxf = (1.0 - pp) * (top[W_MINUS] - top[W_PLUS])
        dh = _rmsnorm_back(h, top[FINAL_NORM], rf, dxf)
        if mutant == 23:
            dh = rf * (top[FINAL_NORM] * dxf)
        for l in reversed(range(NL)):
            P = lays[l]
            h_in, r1, q, ks, vs, o, w_all, h_mid, r2, u, t = save[l]
            # feed-forward block
            da = P[W_DOWN].T @ dh
            du = da * t * _silu_prime(u)
            dt = da * _silu(u)
            dx2 = P[W_GATE_UP].T @ np.concatenate([du, dt])
            dh_mid = dh + _rmsnorm_back(h_mid, P[MLP_NORM], r2, dx2)
            # attention block
            do = (P[W_O].T @ dh_mid).reshape(nq, hd)
            dq = np.zeros((nq, hd))
            dks = np.zeros((nkv, hd))
            dvs = np.zeros((nkv, hd))
            gK = np.zeros((L, nkv, hd))
            gV = np.zeros((L, nkv, hd))
            for hh in range(nq):
                g = hh // G
                w = w_all[hh]
                D = 0.0 if mutant == 21 else do[hh] @ o[hh]
                dp = np.concatenate([Vs[l][:, g, :] @ do[hh], [vs[g] @ do[hh]]])
                ds = w * (dp - D)
                gV[:, g, :] += np.outer(w[:L], do[hh])
                gK[:, g, :] += np.outer(ds[:L], q[hh]) * scale
                dvs[g] += w[L] * do[hh]
                dks[g] += ds[L] * q[hh] * scale
                dq[hh] = (ds[:L] @ Ks[l][:, g, :] + ds[L] * ks[g]) * scale
            dK[l][b], dV[l][b] = gK, gV
            sn = -s if mutant == 22 else s
            dqkv = np.concatenate([_rope_back(dq, c, sn).reshape(-1), _rope_back(dks, c, sn).reshape(-1),
                                   dvs.reshape(-1)])
            dx1 = P[W_QKV].T @ dqkv
            dh = dh_mid + _rmsnorm_back(h_in, P[ATTN_NORM], r1, dx1)
    return p_plus, dK, dV


def loss(arch, weights: dict, kv: list) -> np.ndarray:
    """l_b = -log P(+)_b of every candidate (the forward of score_grad)."""
    p, _, _ = score_grad(arch, weights, kv)
    return -np.log(p)


def pool_grad(w, dK, dV, n_layers: int) -> dict:
    """Sum the candidates' logical gradients into their physical pages: {(layer, page): [2][n_kv][16][hd]}
    for every page a block table references (a page several candidates read gets their sum)."""
    P = 16
    out = {}
    for b in range(w.n_candidates):
        L = int(w.seq_lens[b])
        for j in range(L):
            page = int(w.block_table[b, j // P])
            for l in range(n_layers):
                key = (l, page)
                if key not in out:
                    out[key] = np.zeros((2,) + dK[l][b].shape[1:2] + (P,) + dK[l][b].shape[2:])
                out[key][0, :, j % P, :] += dK[l][b][j]
                out[key][1, :, j % P, :] += dV[l][b][j]
    return out


def steer(arch, weights: dict, kv: list, eta: float, steps: int, shared=None):
    """Algorithm "KV Steering at agent handoff" with the cache kept in bf16: T times
    kv <- RNE_bf16(kv - eta * grad_kv sum_b l_b).  kv[l][b] = (K, V) float64 (bf16 values); `shared`
    maps each candidate's logical positions to physical pages (w, a kvsynth workload) so that a page
    several candidates read takes one update with their summed gradient; without it every candidate's
    cache is its own.  Returns (kv after the steps, P(+) before each step and after the last)."""
    NL = arch.n_layers
    kv = [[(_as_f64(kv[l][b][0]).copy(), _as_f64(kv[l][b][1]).copy()) for b in range(len(kv[0]))]
          for l in range(NL)]
    history = []
    for _ in range(steps):
        p, dK, dV = score_grad(arch, weights, kv)
        history.append(p)
        if shared is not None:   # sum over the candidates that read each physical position
            w = shared
            P = 16
            acc = {}
            for b in range(w.n_candidates):
                for j in range(int(w.seq_lens[b])):
                    key = (int(w.block_table[b, j // P]), j % P)
                    for l in range(NL):
                        a = acc.setdefault((l,) + key, [0.0, 0.0])
                        a[0] = a[0] + dK[l][b][j]
                        a[1] = a[1] + dV[l][b][j]
            for b in range(w.n_candidates):
                for j in range(int(w.seq_lens[b])):
                    key = (int(w.block_table[b, j // P]), j % P)
                    for l in range(NL):
                        gk, gv = acc[(l,) + key]
                        dK[l][b][j] = gk
                        dV[l][b][j] = gv
        for l in range(NL):
            for b in range(len(kv[0])):
                K, V = kv[l][b]
                kv[l][b] = (round_bf16(K - eta * dK[l][b]), round_bf16(V - eta * dV[l][b]))
    p, _, _ = score_grad(arch, weights, kv)
    history.append(p)
    return kv, history
