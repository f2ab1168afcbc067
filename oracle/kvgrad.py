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


def _layer(arch, L):
    """One layer's matrices as float64 (converted when needed, so that a full-size model need not be
    held in float64 at once)."""
    d, nq, nkv, hd, ff = arch.d_model, arch.n_q_heads, arch.n_kv_heads, arch.head_dim, arch.d_ff
    return {ATTN_NORM: bits_to_f64(L[ATTN_NORM]), MLP_NORM: bits_to_f64(L[MLP_NORM]),
            W_QKV: bits_to_f64(L[W_QKV]).reshape((nq + 2 * nkv) * hd, d),
            W_O: bits_to_f64(L[W_O]).reshape(d, nq * hd),
            W_GATE_UP: bits_to_f64(L[W_GATE_UP]).reshape(2 * ff, d),
            W_DOWN: bits_to_f64(L[W_DOWN]).reshape(d, ff)}


def score_grad(arch, weights: dict, kv: list, mutant: int = 0):
    """P(+), l = -log P(+) and dl/dK, dl/dV for every candidate.

    weights = {'top': {kind: bf16 bits}, 'layers': [{kind: bf16 bits}]}; kv[l][b] = (K, V), each
    [L_b][n_kv][hd] as bf16 bits or float64 values.  Returns (p_plus [n], dK, dV) with dK[l][b] and
    dV[l][b] float64 [L_b][n_kv][hd] (candidate b's logical positions; the caller adds the
    contributions of candidates that share a page).  The candidates' rows go through each projection
    together (one matrix product per step); the attention read-out runs per candidate and head.
    mutant > 0 plants one mistake in the reverse pass (used only by the tests of the pins):
    21 drops the -D term of the softmax backward, 22 rotates the RoPE backward the wrong way,
    23 drops the second term of the RMSNorm backward."""
    d, nq, nkv, hd, ff = arch.d_model, arch.n_q_heads, arch.n_kv_heads, arch.head_dim, arch.d_ff
    G = nq // nkv
    NL = arch.n_layers
    eps = arch.rms_eps
    n = len(kv[0])
    top = {k: bits_to_f64(v) for k, v in weights["top"].items()}
    scale = 1.0 / np.sqrt(hd)
    Ks = [[_as_f64(kv[l][b][0]).reshape(-1, nkv, hd) for b in range(n)] for l in range(NL)]
    Vs = [[_as_f64(kv[l][b][1]).reshape(-1, nkv, hd) for b in range(n)] for l in range(NL)]
    lens = [Ks[0][b].shape[0] for b in range(n)]
    cs = [_rope_angles(float(L), hd, arch.rope_base) for L in lens]
    c = np.stack([x[0] for x in cs])[:, None, :]   # [n][1][hd/2]
    s = np.stack([x[1] for x in cs])[:, None, :]

    def rms(h, g):   # rows of h
        r = 1.0 / np.sqrt(np.mean(h * h, axis=1) + eps)
        return h * r[:, None] * g, r

    def rms_back(h, g, r, dy):
        return r[:, None] * (g * dy) - h * (r ** 3)[:, None] * np.sum(g * dy * h, axis=1)[:, None] / d

    # ---------------- forward, every intermediate kept
    h = np.tile(top[EMBED], (n, 1))
    save = []
    for l in range(NL):
        P = _layer(arch, weights["layers"][l])
        x1, r1 = rms(h, P[ATTN_NORM])
        qkv = x1 @ P[W_QKV].T
        q = _rope(qkv[:, :nq * hd].reshape(n, nq, hd), c, s)
        ks = _rope(qkv[:, nq * hd:(nq + nkv) * hd].reshape(n, nkv, hd), c, s)
        vs = qkv[:, (nq + nkv) * hd:].reshape(n, nkv, hd)
        o = np.empty((n, nq, hd))
        w_all = []
        for b in range(n):
            wb = np.empty((nq, lens[b] + 1))
            for hh in range(nq):
                g = hh // G
                sc = np.concatenate([Ks[l][b][:, g, :] @ q[b, hh], [ks[b, g] @ q[b, hh]]]) * scale
                w = np.exp(sc - sc.max())
                w /= w.sum()
                wb[hh] = w
                o[b, hh] = w[:lens[b]] @ Vs[l][b][:, g, :] + w[lens[b]] * vs[b, g]
            w_all.append(wb)
        h_mid = h + o.reshape(n, -1) @ P[W_O].T
        x2, r2 = rms(h_mid, P[MLP_NORM])
        gu = x2 @ P[W_GATE_UP].T
        u, t = gu[:, :ff], gu[:, ff:]
        h_out = h_mid + (_silu(u) * t) @ P[W_DOWN].T
        save.append((h, r1, q, ks, vs, o, w_all, h_mid, r2, u, t))
        h = h_out
    xf, rf = rms(h, top[FINAL_NORM])
    z_p, z_m = xf @ top[W_PLUS], xf @ top[W_MINUS]
    p_plus = 1.0 / (1.0 + np.exp(z_m - z_p))
    # ---------------- reverse pass of sum_b -log P(+)_b
    dxf = (1.0 - p_plus)[:, None] * (top[W_MINUS] - top[W_PLUS])[None, :]
    dh = rms_back(h, top[FINAL_NORM], rf, dxf)
    if mutant == 23:
        dh = rf[:, None] * (top[FINAL_NORM] * dxf)
    dK = [[None] * n for _ in range(NL)]
    dV = [[None] * n for _ in range(NL)]
    for l in reversed(range(NL)):
        P = _layer(arch, weights["layers"][l])
        h_in, r1, q, ks, vs, o, w_all, h_mid, r2, u, t = save[l]
        # feed-forward block
        da = dh @ P[W_DOWN]
        du = da * t * _silu_prime(u)
        dt = da * _silu(u)
        dx2 = np.concatenate([du, dt], axis=1) @ P[W_GATE_UP]
        dh_mid = dh + rms_back(h_mid, P[MLP_NORM], r2, dx2)
        # attention block
        do = (dh_mid @ P[W_O]).reshape(n, nq, hd)
        dq = np.zeros((n, nq, hd))
        dks = np.zeros((n, nkv, hd))
        dvs = np.zeros((n, nkv, hd))
        for b in range(n):
            L = lens[b]
            gK = np.zeros((L, nkv, hd))
            gV = np.zeros((L, nkv, hd))
            for hh in range(nq):
                g = hh // G
                w = w_all[b][hh]
                D = 0.0 if mutant == 21 else do[b, hh] @ o[b, hh]
                dp = np.concatenate([Vs[l][b][:, g, :] @ do[b, hh], [vs[b, g] @ do[b, hh]]])
                ds = w * (dp - D)
                gV[:, g, :] += np.outer(w[:L], do[b, hh])
                gK[:, g, :] += np.outer(ds[:L], q[b, hh]) * scale
                dvs[b, g] += w[L] * do[b, hh]
                dks[b, g] += ds[L] * q[b, hh] * scale
                dq[b, hh] = (ds[:L] @ Ks[l][b][:, g, :] + ds[L] * ks[b, g]) * scale
            dK[l][b], dV[l][b] = gK, gV
        sn = -s if mutant == 22 else s
        dqkv = np.concatenate([_rope_back(dq, c, sn).reshape(n, -1), _rope_back(dks, c, sn).reshape(n, -1),
                               dvs.reshape(n, -1)], axis=1)
        dx1 = dqkv @ P[W_QKV]
        dh = dh_mid + rms_back(h_in, P[ATTN_NORM], r1, dx1)
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
