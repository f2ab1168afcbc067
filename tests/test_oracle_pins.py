"""The CPU oracle against closed forms, invariants, library routines and a
brute-force causal re-encode (see tests/oracle_pins.py)."""
import numpy as np
import pytest

import kvsynth as ks
import oracle
from tests import oracle_pins as P


def test_bf16_round():
    P.pin_bf16_round()


def test_rmsnorm():
    P.pin_rmsnorm()


def test_rope():
    P.pin_rope()


def test_attend():
    P.pin_attend()


def test_reward():
    P.pin_reward()


@pytest.mark.parametrize("depth", [2, 4])
def test_depth_readout_reencode(depth):
    P.pin_depth_reencode(depth=depth)


def test_qk_norm_reencode():
    P.pin_qk_norm()


def test_grad_forward_matches_c_oracle():
    P.pin_grad_forward()


def test_grad_finite_differences():
    P.pin_grad_fd()


def test_grad_autograd():
    P.pin_grad_autograd()


def test_steer_step_lowers_each_loss():
    """One step of KV Steering (App. C) with the cache kept in bf16 lowers -log P(+) of every candidate
    with a distinct cache, and a shared page takes the summed gradient of the candidates reading it."""
    from oracle import kvgrad
    arch, W, kv = P._grad_case(seed=93, lens=(40, 25, 64))
    _, dK, dV = kvgrad.score_grad(arch, W, kv)
    gmax = max(max(np.abs(dK[l][b]).max(), np.abs(dV[l][b]).max()) for l in range(2) for b in range(3))
    eta = 0.05 / gmax
    kv2, hist = kvgrad.steer(arch, W, kv, eta, 1)
    assert (hist[1] > hist[0]).all(), hist
    # every updated value is a bf16 value
    for l in range(arch.n_layers):
        for b in range(3):
            for A in kv2[l][b]:
                assert np.array_equal(kvgrad.round_bf16(A), A)
    # a shared prefix: the steered pages are identical for every candidate reading them
    w = ks.shared_prefix("steer_pin", arch, 94, 3, 32, 9)
    t = ks.Tables.make(0.2)
    Wt = ks.host_weights(arch, w.seed, t)
    kvw = [[ks.host_kv_logical(w, l, b, t) for b in range(3)] for l in range(arch.n_layers)]
    kv3, hist3 = kvgrad.steer(arch, Wt, kvw, 0.5, 1, shared=w)
    for l in range(arch.n_layers):
        for b in (1, 2):
            assert np.array_equal(kv3[l][b][0][:32], kv3[l][0][0][:32])


def test_lora_equals_merged():
    P.pin_lora_merged()


def test_lora_synth_provider():
    """The seeded generator supplies the adapter factors: with rank 64 the scores move away from the
    merged scorer's, and a zero-scale adapter (alpha = 0) gives the merged scorer's scores exactly."""
    import dataclasses
    t = ks.Tables.make(0.2)
    w = ks.distinct("lora", ks.ARCH_TINY, 11, [0, 20, 70], gain_std=0.2)
    r0 = oracle.score_synth(w, t, mirror=False)
    w.arch = dataclasses.replace(ks.ARCH_TINY, lora_rank=64)
    r1 = oracle.score_synth(w, t, mirror=False)
    assert np.abs(r1.p_plus - r0.p_plus).max() > 1e-4
    w.arch = dataclasses.replace(ks.ARCH_TINY, lora_rank=64, lora_alpha=0.0)
    r2 = oracle.score_synth(w, t, mirror=False)
    assert np.array_equal(r2.p_plus, r0.p_plus)


@pytest.mark.parametrize("mirror", [True, False])
def test_reencode_tiny(mirror):
    P.pin_reencode(mirror=mirror)


def test_reencode_wide_groups():
    # G = 6 query heads per kv head (the 1.5B layout), shrunk
    arch = ks.Arch(2, 192, 6, 1, 32, 256)
    P.pin_reencode(lens=(0, 3, 33), arch=arch)


def test_logical_vs_paged_cache():
    """The logical K/V the oracle reads equal the pool pages the block table names."""
    t = ks.Tables.make()
    w = ks.mcts_tree("t", ks.ARCH_TINY, 5, branching=2, depth=3, lo=5, hi=40)
    pool = ks.host_kv_pool(w, t, layers=[1])[0]          # [n_pages][2][nkv][P][hd]
    P_ = w.arch.page_size
    for b in range(w.n_candidates):
        K, V = ks.host_kv_logical(w, 1, b, t)
        L = int(w.seq_lens[b])
        pos = np.arange(L)
        pages = w.block_table[b, pos // P_]
        np.testing.assert_array_equal(pool[pages, 0, :, pos % P_, :], K)
        np.testing.assert_array_equal(pool[pages, 1, :, pos % P_, :], V)


def test_sharing_structure():
    w = ks.make_workload("beam7b_b64_p4096_s512")
    # 256 shared prefix pages + 32 own pages per candidate (page aligned)
    assert len(set(w.block_table[:, :256].ravel().tolist())) == 256
    assert (w.block_table[:, :256] == w.block_table[0, :256]).all()
    own = w.block_table[:, 256:288]
    assert len(set(own.ravel().tolist())) == 64 * 32
    t = ks.make_workload("mcts7b_b256_d4")
    assert t.n_candidates == 256 and 4 * 256 <= t.seq_lens.min() and t.seq_lens.max() <= 4 * 2048


def test_oracle_threads_agree():
    t = ks.Tables.make(0.2)
    w = ks.distinct("t", ks.ARCH_TINY, 3, [0, 7, 33])
    a = oracle.score_synth(w, t, nthreads=1)
    b = oracle.score_synth(w, t, nthreads=4)
    np.testing.assert_array_equal(a.p_plus, b.p_plus)
    np.testing.assert_array_equal(a.attn, b.attn)


def test_golden_regression():
    """Oracle outputs on the seeded tiny workloads match the committed fixture
    (written by tests/golden/make_golden.py, which calls only the oracle)."""
    import json
    import os
    from tests.golden.make_golden import compute
    with open(os.path.join(os.path.dirname(__file__), "golden", "oracle_tiny.json")) as f:
        ref = json.load(f)
    got = compute()
    for k in ref:
        np.testing.assert_allclose(got[k]["p_plus"], ref[k]["p_plus"], rtol=0, atol=1e-12)
        np.testing.assert_allclose(got[k]["attn_absmax"], ref[k]["attn_absmax"], rtol=1e-10)
