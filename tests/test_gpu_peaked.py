"""GPU parity where the softmax of the attention read-out is peaked (App. A.3: a trained scorer's
query singles out a few cached positions): scores q.k / sqrt(hd) tens of units apart, one planted
key dominating late in the sequence, runs of identical keys sharing the top score, and broad
queries whose scores spread over tens of units.  Every attention plan is covered: the fused-combine
plan, the persistent kernel with the combine launch, shared runs of <= 4 candidates on the
persistent kernel, the tensor-core tiles of shared pages with the production rescale margin, an
MCTS tree mixing the last two, both forms of the combine launch, and (end to end) the depth-k
combine.  Tolerances are the ones every parity test uses: 2e-3 relative per (candidate, head) or
(layer, candidate), 1e-3 on P(+)."""
import numpy as np
import pytest

import kvsynth as ks
import oracle
from tests.gpu_util import ATTN_RTOL, PlantedCase, compare, make_scorer, require_gpu, row_rel_err, run_gpu

pytestmark = pytest.mark.gpu

ARCH_G6 = ks.Arch(1, 256, 12, 2, 128, 256)    # 1.5B heads, one layer (projections unused here)
ARCH_G7 = ks.Arch(1, 256, 14, 2, 128, 256)    # 7B-like grouping: shared groups of >= 6 on the tensor cores
ARCH_H64 = ks.Arch(1, 256, 4, 2, 64, 256)     # head_dim 64: shared pages on the persistent kernel only


def _last(w, b):
    return int(w.cand_seg[b][-1]), int(w.cand_off[b][-1])


def _run(case: PlantedCase, label: str, min_spread: float = 30.0, flags: int = 0):
    torch = require_gpu()
    import paper_2607_09153_gb300 as kp
    w, a = case.w, case.arch
    spread = case.score_spread()
    assert spread >= min_spread, f"{label}: top-to-median score gap {spread:.1f} is not peaked"
    dev = ks.DeviceInputs(ks.distinct("host", a, 1, [16]), ks.Tables.make())   # weights for a context only
    sc = make_scorer(dev, w.n_candidates, w.max_blocks)
    if flags:
        kp.kvprm_set_debug(sc.ctx, flags)
    pool, q, k, v = case.device()
    B = w.n_candidates
    out = torch.full((B, a.n_q_heads, a.head_dim), float("nan"), dtype=torch.float32, device="cuda")
    kp.kvprm_attention(sc.ctx, pool.data_ptr(), w.n_pages, w.block_table, w.seq_lens, B, q.data_ptr(),
                       k.data_ptr(), v.data_ptr(), out.data_ptr(), torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    kp.kvprm_check_device(sc.ctx)
    got = out.cpu().numpy().astype(np.float64)
    ref = case.expected()
    err = row_rel_err(got, ref)
    print(f"{label}: score gap {spread:.1f}, max rel err {err:.3e}")
    assert np.isfinite(got).all()
    assert err <= ATTN_RTOL, f"{label}: {err:.3e}"
    sc.close()
    return got, ref


def test_peaked_fused_combine():
    # equal lengths, nothing shared: the fused-combine plan (clusters merging through DSMEM)
    w = ks.distinct("pk_fused", ARCH_G6, 201, [1024] * 4)
    needles = [_last(w, b) for b in range(4)] + [(1, 700)]
    _run(PlantedCase(w, ks.Tables.make(), 1, needles, runs=[(2, 1000, 24)]), "fused combine")


@pytest.mark.parametrize("flat", [False, True])
def test_peaked_persistent_and_combine(flat):
    # ragged lengths: the persistent kernel (private runs, merger warp) and the combine launch (its
    # general form, or the flat form with debug flag 64); candidate 4's top score is a run of 64
    # identical keys near its end, candidate 6 has no cache
    lens = [1, 17, 250, 2049, 4096, 33, 0]
    w = ks.distinct("pk_persist", ARCH_G6, 202, lens)
    needles = [_last(w, b) for b in (0, 1, 2, 3, 5)] + [(3, 5)]
    _run(PlantedCase(w, ks.Tables.make(), 2, needles, runs=[(4, 4000, 64)]), f"persistent + combine flat={flat}",
         flags=64 if flat else 0)


def test_peaked_shared_runs():
    # three candidates share a prefix: a shared run of 3 on the persistent kernel (replica warps)
    w = ks.shared_prefix("pk_shared", ARCH_G6, 203, 3, 1024, 100)
    needles = [(0, 1010), (1, 99)]   # a late prefix key for candidates 1, 2; candidate 0's own suffix
    _run(PlantedCase(w, ks.Tables.make(), 3, needles, runs=[(0, 900, 16)]), "shared runs of 3")


def test_peaked_shared_runs_hd64():
    # head_dim 64: every shared group on the persistent kernel, groups of 2 .. 8
    w = ks.mcts_tree("pk_tree64", ARCH_H64, 204, branching=2, depth=3, lo=40, hi=300)
    needles = [_last(w, b) for b in range(0, w.n_candidates, 2)] + [(0, 30)]
    _run(PlantedCase(w, ks.Tables.make(), 4, needles), "tree, head_dim 64")


@pytest.mark.parametrize("B,prefix,suffix", [(24, 2064, 37), (8, 4096, 16)])
def test_peaked_tensor_cores(B, prefix, suffix):
    # a shared prefix of >= 6 candidates: tensor-core tiles with the production rescale margin; the
    # dominant key sits at the prefix's end (after every other chunk) or in a candidate's suffix
    w = ks.shared_prefix("pk_tc", ARCH_G7, 205 + B, B, prefix, suffix)
    needles = [(0, prefix - 3)] + [(1 + b, suffix - 1) for b in range(0, B, 3)]
    _run(PlantedCase(w, ks.Tables.make(), 5 + B, needles, runs=[(0, prefix - 300, 64)]),
         f"tensor cores B={B} prefix={prefix}")


@pytest.mark.parametrize("flat", [False, True])
def test_peaked_tree_mixed(flat):
    # MCTS tree: depth-1 groups of 9 on the tensor cores, depth-2 groups of 3 on the persistent kernel
    w = ks.mcts_tree("pk_tree", ARCH_G7, 206, branching=3, depth=3, lo=100, hi=400)
    needles = [_last(w, b) for b in range(w.n_candidates)] + [(0, 50)]
    _run(PlantedCase(w, ks.Tables.make(), 6, needles, runs=[(0, 10, 32)]),
         f"tree, tensor cores + shared runs, flat={flat}", flags=64 if flat else 0)


# ---------------------------------------------------------------- end to end, peaked query/key projections
def _layer0_gap(w, tables, ref):
    """Top-to-median score gap of layer 0 over the oracle's own rotated q and the cache."""
    a = w.arch
    G = a.n_q_heads // a.n_kv_heads
    gap = 0.0
    for i in range(min(4, w.n_candidates)):
        K, _ = ks.host_kv_logical(w, 0, i, tables)
        if len(K) == 0:
            continue
        q = ref.qkv[0, i, :a.n_q_heads * a.head_dim].reshape(a.n_q_heads, a.head_dim)
        for h in range(a.n_q_heads):
            s = ks.bf16_bits_to_f64(K[:, h // G, :]) @ q[h] / np.sqrt(a.head_dim)
            gap = max(gap, float(s.max() - np.median(s)))
    return gap


@pytest.mark.parametrize("name,arch,qkv_std,make,depth", [
    ("tiny", ks.ARCH_TINY, 0.5, lambda a: ks.distinct("pe_tiny", a, 211, [128] * 4, gain_std=0.2), 1),
    ("tiny ragged", ks.ARCH_TINY, 0.5, lambda a: ks.distinct("pe_rag", a, 212, [0, 5, 100, 333], gain_std=0.2), 1),
    ("1.5B layers fused", ks.Arch(2, 1536, 12, 2, 128, 8960), 0.2,
     lambda a: ks.distinct("pe_15", a, 213, [2048] * 8, gain_std=0.2), 1),
    ("7B layers shared prefix", ks.Arch(2, 3584, 28, 4, 128, 18944), 0.1,
     lambda a: ks.shared_prefix("pe_7b", a, 214, 12, 1024, 64, gain_std=0.2), 1),
    ("tiny depth 3", ks.ARCH_TINY, 0.5, lambda a: ks.distinct("pe_d3", a, 215, [0, 17, 100, 250], gain_std=0.2), 3),
])
def test_peaked_end_to_end(name, arch, qkv_std, make, depth):
    """The whole scorer with W_qkv drawn wide, so that every layer's attention is peaked; P(+) and
    every layer's attention output against the oracle (exact mode)."""
    t = ks.Tables.make(0.2, qkv_std=qkv_std)
    w = make(arch)
    r, attn, dev, sc = run_gpu(w, t, depth=depth)
    ref = compare(w, t, gpu_rewards=r, gpu_attn=attn, label=f"peaked {name}", depth=depth)
    lay = oracle.score_synth(w, t, list(range(min(4, w.n_candidates))), mirror=False, want_layers=True)
    gap = _layer0_gap(w, t, lay)
    print(f"peaked {name}: layer-0 top-to-median score gap {gap:.1f}")
    assert gap >= 15.0
    del ref
    sc.close()
