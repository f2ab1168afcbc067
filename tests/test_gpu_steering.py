"""GPU parity of KV Steering (Sec. 6; App. C, Algorithm "KV Steering at agent handoff"): the
gradient of sum_b -log P(+)_b with respect to every cached key and value (kvprm_score_grad) against
the fp64 oracle (oracle/kvgrad.py), on the tiny configuration, the 1.5B-shaped configuration at full
size, ragged and shared-page caches (a page several candidates read holds their summed gradient) and
both head widths; then steering steps (kvprm_steer) against the oracle's bf16 steps.

Tolerance: per layer, max |g_gpu - g_ref| / max |g_ref| over the referenced pages <= 2e-3 -- the
attention read-out's tolerance, since the backward runs the same fp32 arithmetic (fp32 softmax
weights and accumulations, bf16 hi/lo pairs into the tensor-core products); P(+) within 1e-3."""
import numpy as np
import pytest

import kvsynth as ks
from oracle import kvgrad
from tests.gpu_util import P_PLUS_ATOL, make_scorer, require_gpu

pytestmark = pytest.mark.gpu

GRAD_RTOL = 2e-3


def _oracle(w, t, ids=None):
    """Oracle gradient of the candidates `ids` (all by default) summed into physical pages."""
    a = w.arch
    ids = list(range(w.n_candidates)) if ids is None else list(ids)
    W = ks.host_weights(a, w.seed, t)
    kv = [[ks.host_kv_logical(w, l, b, t) for b in ids] for l in range(a.n_layers)]
    p, dK, dV = kvgrad.score_grad(a, W, kv)
    pages = {}
    for i, b in enumerate(ids):
        for j in range(int(w.seq_lens[b])):
            page = int(w.block_table[b, j // 16])
            for l in range(a.n_layers):
                e = pages.setdefault((l, page), np.zeros((2, a.n_kv_heads, 16, a.head_dim)))
                e[0, :, j % 16, :] += dK[l][i][j]
                e[1, :, j % 16, :] += dV[l][i][j]
    return p, pages, W, kv


def _gpu_grad(w, t, dev=None):
    torch = require_gpu()
    import paper_2607_09153_gb300 as kp
    dev = dev or ks.DeviceInputs(w, t)
    sc = make_scorer(dev, w.n_candidates, w.max_blocks)
    grad = torch.full(dev.pool.shape, float("nan"), dtype=torch.float32, device="cuda")
    p = kp.kvprm_score_grad(sc.ctx, dev.pool.data_ptr(), dev.n_pages, w.block_table, w.seq_lens, w.n_candidates,
                            grad.data_ptr(), torch.cuda.current_stream().cuda_stream)
    kp.kvprm_check_device(sc.ctx)
    return p, grad, dev, sc


def _compare(label, w, p_gpu, grad, p_ref, pages, ids=None):
    ids = list(range(w.n_candidates)) if ids is None else list(ids)
    dp = float(np.abs(p_gpu[ids] - p_ref).max())
    a = w.arch
    worst = 0.0
    for l in range(a.n_layers):
        keys = sorted(k for k in pages if k[0] == l)
        ref = np.stack([pages[k] for k in keys])
        got = grad[l][[k[1] for k in keys]].cpu().numpy().astype(np.float64)
        assert np.isfinite(got).all(), f"{label}: layer {l} has unwritten or non-finite gradient entries"
        err = np.abs(got - ref).max() / max(np.abs(ref).max(), 1e-30)
        worst = max(worst, err)
    print(f"{label}: max |dP| = {dp:.3e}, max per-layer gradient rel err = {worst:.3e}")
    assert dp <= P_PLUS_ATOL
    assert worst <= GRAD_RTOL, f"{label}: {worst:.3e}"


def _check_steered(label, w, host, kv_ref, eta, pages):
    """Steered bf16 pages against the oracle's step.  Each value may differ from the oracle's by one
    bf16 ulp of rounding plus eta times the gradient's own tolerance (GRAD_RTOL times the layer's
    largest gradient entry): the GPU steps along its own gradient, which agrees with the oracle's to
    that tolerance.  Away from cancellation that bound is under one ulp; the count of values that
    differ at all stays under 1 %."""
    a = w.arch
    gmax = [max(np.abs(v).max() for k, v in pages.items() if k[0] == l) for l in range(a.n_layers)]
    n_diff = n_all = 0
    worst = 0.0
    for b in range(w.n_candidates):
        for j in range(int(w.seq_lens[b])):
            page, slot = int(w.block_table[b, j // 16]), j % 16
            for l in range(a.n_layers):
                for which in (0, 1):
                    got_bits = host[l, page, which, :, slot, :]
                    ref_bits = ks.f64_to_bf16_bits(kv_ref[l][b][which][j])
                    got, ref = kvgrad.bits_to_f64(got_bits), kvgrad.bits_to_f64(ref_bits)
                    ulp = np.abs(kvgrad.bits_to_f64(ref_bits + 1) - ref)
                    bound = ulp + eta * GRAD_RTOL * gmax[l]
                    err = np.abs(got - ref)
                    assert (err <= bound).all(), (label, b, j, l, which, float((err / bound).max()))
                    worst = max(worst, float((err / bound).max()))
                    n_diff += int((got_bits != ref_bits).sum())
                    n_all += got_bits.size
    print(f"{label}: {n_diff} of {n_all} values differ from the oracle's step; worst error / bound {worst:.3f}")
    assert n_diff <= 0.01 * n_all


@pytest.mark.parametrize("gain_std", [0.0, 0.2])
def test_grad_tiny(gain_std):
    t = ks.Tables.make(gain_std)
    w = ks.make_workload("tiny", gain_std=gain_std)
    p, grad, dev, sc = _gpu_grad(w, t)
    p_ref, pages, _, _ = _oracle(w, t)
    _compare(f"tiny g{gain_std}", w, p, grad, p_ref, pages)
    sc.close()


@pytest.mark.parametrize("make", [
    # ragged lengths with partial last pages, an empty cache, head_dim 64
    lambda: ks.distinct("g_rag", ks.ARCH_TINY, 501, [0, 1, 15, 17, 100, 257], gain_std=0.2),
    # a tree: pages read by 2, 4 and 8 leaves (accumulated gradients), head_dim 64
    lambda: ks.mcts_tree("g_tree", ks.ARCH_TINY, 502, branching=2, depth=3, lo=5, hi=40, gain_std=0.2),
    # head_dim 128, G = 7, a prefix shared by 8 candidates (its forward on the tensor cores)
    lambda: ks.shared_prefix("g_tc", ks.Arch(2, 256, 14, 2, 128, 512), 503, 8, 96, 21, gain_std=0.2),
    # G = 16 (the widest grouping)
    lambda: ks.distinct("g_g16", ks.Arch(2, 512, 16, 1, 64, 512), 504, [0, 50, 129], gain_std=0.2),
])
def test_grad_shapes(make):
    t = ks.Tables.make(0.2)
    w = make()
    p, grad, dev, sc = _gpu_grad(w, t)
    p_ref, pages, _, _ = _oracle(w, t)
    _compare(w.name, w, p, grad, p_ref, pages)
    sc.close()


def test_grad_peaked():
    """Peaked attention (W_qkv drawn wide): softmax weights far from uniform in every layer."""
    t = ks.Tables.make(0.2, qkv_std=0.5)
    w = ks.distinct("g_peak", ks.ARCH_TINY, 505, [30, 128, 200], gain_std=0.2)
    p, grad, dev, sc = _gpu_grad(w, t)
    p_ref, pages, _, _ = _oracle(w, t)
    _compare("peaked", w, p, grad, p_ref, pages)
    sc.close()


def test_grad_full_size_1p5b():
    """The 1.5B-shaped configuration at full size (28 layers, 16 x 2048): the whole batch's gradient
    on the GPU, sampled candidates (distinct caches: each page's gradient is its candidate's) against
    the oracle."""
    t = ks.Tables.make()
    w = ks.make_workload("qwen1p5b_b16_l2048")
    p, grad, dev, sc = _gpu_grad(w, t)
    ids = [0, 7, 15]
    p_ref, pages, _, _ = _oracle(w, t, ids)
    _compare("qwen1p5b_b16_l2048 sampled", w, p, grad, p_ref, pages, ids)
    sc.close()


def test_steer_steps():
    """kvprm_steer: one and then two more bf16 steps on a copy of the pages, against the oracle's
    steps; every candidate's P(+) rises on the first step."""
    torch = require_gpu()
    import paper_2607_09153_gb300 as kp
    t = ks.Tables.make(0.2)
    w = ks.distinct("steer", ks.ARCH_TINY, 506, [40, 77, 128, 5], gain_std=0.2)
    dev = ks.DeviceInputs(w, t)
    sc = make_scorer(dev, w.n_candidates, w.max_blocks)
    p_ref, pages, W, kv = _oracle(w, t)
    gmax = max(np.abs(v).max() for v in pages.values())
    eta = 0.05 / gmax
    pool = dev.pool.clone()
    st = torch.cuda.current_stream().cuda_stream
    p0, p1 = kp.kvprm_steer(sc.ctx, pool.data_ptr(), dev.n_pages, w.block_table, w.seq_lens, w.n_candidates, eta, 1, st)
    assert np.abs(p0 - p_ref).max() <= P_PLUS_ATOL
    assert (p1 > p0).all(), (p0, p1)
    kv_ref, hist = kvgrad.steer(w.arch, W, kv, eta, 1)
    assert np.abs(p1 - hist[-1]).max() <= P_PLUS_ATOL
    print(f"steer: P(+) {np.round(p0, 5)} -> {np.round(p1, 5)}")
    host = pool.cpu().view(torch.int16).numpy().view(np.uint16)
    _check_steered("steer", w, host, kv_ref, eta, pages)
    # the untouched decoy pages are as they were
    refs = set(int(x) for b in range(w.n_candidates) for x in w.block_table[b, :(int(w.seq_lens[b]) + 15) // 16])
    decoys = [p for p in range(dev.n_pages) if p not in refs]
    assert torch.equal(pool[:, decoys], dev.pool[:, decoys])
    # two more steps keep raising P(+)
    q0, q2 = kp.kvprm_steer(sc.ctx, pool.data_ptr(), dev.n_pages, w.block_table, w.seq_lens, w.n_candidates, eta, 2, st)
    assert np.allclose(q0, p1, atol=1e-6) and (q2 > q0).all()
    sc.close()


def test_grad_scope_errors():
    torch = require_gpu()
    import dataclasses
    import paper_2607_09153_gb300 as kp
    t = ks.Tables.make(0.2)
    w = ks.distinct("g_err", ks.ARCH_TINY, 507, [20, 40], gain_std=0.2)
    dev = ks.DeviceInputs(w, t)
    sc = make_scorer(dev, 4, w.max_blocks)
    grad = torch.zeros(dev.pool.shape, dtype=torch.float32, device="cuda")
    st = torch.cuda.current_stream().cuda_stream
    with pytest.raises(kp.KvprmError) as e:
        kp.kvprm_score_grad(sc.ctx, dev.pool.data_ptr(), dev.n_pages, w.block_table, w.seq_lens, 2, 0, st)
    assert e.value.code == kp.KVPRM_EINVAL
    sc.set_depth(2)
    with pytest.raises(kp.KvprmError) as e:
        kp.kvprm_score_grad(sc.ctx, dev.pool.data_ptr(), dev.n_pages, w.block_table, w.seq_lens, 2, grad.data_ptr(), st)
    assert e.value.code == kp.KVPRM_EUNSUPPORTED
    sc.set_depth(1)
    r = kp.kvprm_score_grad(sc.ctx, dev.pool.data_ptr(), dev.n_pages, w.block_table, w.seq_lens, 2, grad.data_ptr(), st)
    assert np.isfinite(r).all()
    sc.close()
    wl = ks.distinct("g_err", dataclasses.replace(ks.ARCH_TINY, lora_rank=64), 507, [20, 40], gain_std=0.2)
    devl = ks.DeviceInputs(wl, t)
    scl = make_scorer(devl, 4, wl.max_blocks)
    with pytest.raises(kp.KvprmError) as e:
        kp.kvprm_score_grad(scl.ctx, devl.pool.data_ptr(), devl.n_pages, wl.block_table, wl.seq_lens, 2,
                            grad.data_ptr(), st)
    assert e.value.code == kp.KVPRM_EUNSUPPORTED
    scl.close()


def test_steer_shared_prefix():
    """kvprm_steer on a beam-shaped cache whose prefix 8 candidates read (the forward scores it on the
    tensor cores; its gradient is accumulated from every candidate): one step against the oracle's
    step with the summed gradient applied once to each shared page."""
    torch = require_gpu()
    import paper_2607_09153_gb300 as kp
    t = ks.Tables.make(0.2)
    w = ks.shared_prefix("steer_sp", ks.Arch(2, 256, 14, 2, 128, 512), 508, 8, 96, 21, gain_std=0.2)
    dev = ks.DeviceInputs(w, t)
    sc = make_scorer(dev, w.n_candidates, w.max_blocks)
    p_ref, pages, W, kv = _oracle(w, t)
    eta = 0.05 / max(np.abs(v).max() for v in pages.values())
    pool = dev.pool.clone()
    st = torch.cuda.current_stream().cuda_stream
    p0, p1 = kp.kvprm_steer(sc.ctx, pool.data_ptr(), dev.n_pages, w.block_table, w.seq_lens, w.n_candidates, eta, 1, st)
    assert np.abs(p0 - p_ref).max() <= P_PLUS_ATOL
    kv_ref, hist = kvgrad.steer(w.arch, W, kv, eta, 1, shared=w)
    assert np.abs(p1 - hist[-1]).max() <= P_PLUS_ATOL
    print(f"steer shared prefix: P(+) {np.round(p0, 4)} -> {np.round(p1, 4)}")
    host = pool.cpu().view(torch.int16).numpy().view(np.uint16)
    _check_steered("steer shared prefix", w, host, kv_ref, eta, pages)
    sc.close()


def test_grad_mcts_tree_hd128():
    """A small MCTS tree on the 7B grouping: pages read by 9 (tensor-core forward), 3 and 1 candidates,
    ragged edges with partial pages copied per child."""
    t = ks.Tables.make(0.2)
    w = ks.mcts_tree("g_tree128", ks.Arch(2, 256, 14, 2, 128, 512), 509, branching=3, depth=3, lo=20, hi=70,
                     gain_std=0.2)
    p, grad, dev, sc = _gpu_grad(w, t)
    p_ref, pages, _, _ = _oracle(w, t)
    _compare(w.name, w, p, grad, p_ref, pages)
    sc.close()


def test_grad_graph_matches_eager(monkeypatch):
    """The gradient call's captured graph (the default) against the same call with eager launches
    (KVPRM_NO_GRAPH=1): the same kernels, so the same values up to the order of float atomics on
    pages several candidates read; and a second replay of the graph agrees with the first."""
    torch = require_gpu()
    import paper_2607_09153_gb300 as kp
    t = ks.Tables.make(0.2)
    w = ks.mcts_tree("g_graph", ks.ARCH_TINY, 510, branching=2, depth=3, lo=5, hi=60, gain_std=0.2)
    dev = ks.DeviceInputs(w, t)
    st = torch.cuda.current_stream().cuda_stream
    out = []
    for eager in (False, True):
        if eager:
            monkeypatch.setenv("KVPRM_NO_GRAPH", "1")
        sc = make_scorer(dev, w.n_candidates, w.max_blocks)
        grads = []
        for _ in range(2):
            grad = torch.full(dev.pool.shape, float("nan"), dtype=torch.float32, device="cuda")
            p = kp.kvprm_score_grad(sc.ctx, dev.pool.data_ptr(), dev.n_pages, w.block_table, w.seq_lens,
                                    w.n_candidates, grad.data_ptr(), st)
            grads.append((p, grad))
        kp.kvprm_check_device(sc.ctx)
        out.append(grads)
        sc.close()
    refs = set(int(x) for b in range(w.n_candidates) for x in w.block_table[b, :(int(w.seq_lens[b]) + 15) // 16])
    idx = sorted(refs)
    (pg0, g0), (pg1, g1) = out[0]
    (pe, ge), _ = out[1]
    scale = float(ge[:, idx].abs().max())
    for p, g in ((pg0, g0), (pg1, g1)):
        assert np.abs(p - pe).max() <= 1e-6
        assert float((g[:, idx] - ge[:, idx]).abs().max()) <= 1e-5 * scale
