"""GPU parity: the C-ABI CUDA scoring path against the CPU oracle (exact mode:
bf16 weights and cache, exact activations) on seeded inputs -- P(+) within 1e-3
absolute; every layer's attention output within 2e-3 relative inf-norm, full
chain, not teacher-forced -- plus edge cases, indexing and error handling."""
import numpy as np
import pytest

import kvsynth as ks
import oracle
from tests.gpu_util import ATTN_RTOL, compare, make_scorer, require_gpu, run_gpu

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("gain_std", [0.0, 0.2])
def test_tiny_workload(gain_std):
    t = ks.Tables.make(gain_std)
    w = ks.make_workload("tiny", gain_std=gain_std)
    r, attn, _, _ = run_gpu(w, t)
    compare(w, t, gpu_rewards=r, gpu_attn=attn, label=f"tiny g{gain_std}")


def test_ragged_and_page_edges():
    t = ks.Tables.make(0.2)
    w = ks.distinct("ragged", ks.ARCH_TINY, 21, [0, 1, 15, 16, 17, 31, 33, 100, 257, 1000], gain_std=0.2)
    r, attn, _, _ = run_gpu(w, t)
    compare(w, t, gpu_rewards=r, gpu_attn=attn, label="ragged")


def test_all_empty_caches():
    t = ks.Tables.make(0.2)
    w = ks.distinct("empty", ks.ARCH_TINY, 22, [0, 0, 0], gain_std=0.2)
    r, attn, _, _ = run_gpu(w, t)
    compare(w, t, gpu_rewards=r, gpu_attn=attn, label="empty")


def test_shared_pages_tree():
    t = ks.Tables.make(0.2)
    w = ks.mcts_tree("tree", ks.ARCH_TINY, 23, branching=3, depth=3, lo=5, hi=70, gain_std=0.2)
    r, attn, _, _ = run_gpu(w, t)
    compare(w, t, gpu_rewards=r, gpu_attn=attn, label="tree")


# head_dim 128 with G = 7: pages shared by several candidates are scored on the
# tensor cores (tiles of <= 18 candidates x 7 heads) instead of per warp
ARCH_G7 = ks.Arch(2, 256, 14, 2, 128, 512)


@pytest.mark.parametrize("B,prefix,suffix", [(40, 528, 37), (3, 64, 1), (18, 16, 5), (20, 530, 40)])
def test_tc_shared_prefix(B, prefix, suffix):
    t = ks.Tables.make(0.2)
    w = ks.shared_prefix("tc_prefix", ARCH_G7, 31 + B, B, prefix, suffix, gain_std=0.2)
    r, attn, _, _ = run_gpu(w, t)
    compare(w, t, gpu_rewards=r, gpu_attn=attn, label=f"tensor-core prefix B={B} prefix={prefix}")


@pytest.mark.parametrize("rescale_always", [False, True])
def test_tc_long_prefix(rescale_always):
    # 36 candidates (two tiles) share 11,200 tokens: every tensor-core part spans >= 5
    # chunks, so K/V stages are reused and S buffers alternate; flag 16 forces the
    # running-maximum rescale of O in TMEM on every new maximum
    t = ks.Tables.make(0.2)
    w = ks.shared_prefix("tc_long", ARCH_G7, 37, 36, 11200, 23, gain_std=0.2)
    r, attn, _, _ = run_gpu(w, t, extra_flags=16 if rescale_always else 0)
    compare(w, t, gpu_rewards=r, gpu_attn=attn, label=f"tensor-core long prefix rescale_always={rescale_always}")


def test_tc_tree():
    t = ks.Tables.make(0.2)
    w = ks.mcts_tree("tc_tree", ARCH_G7, 41, branching=3, depth=3, lo=5, hi=90, gain_std=0.2)
    r, attn, _, _ = run_gpu(w, t)
    compare(w, t, gpu_rewards=r, gpu_attn=attn, label="tensor-core tree")


@pytest.mark.parametrize("B", [1, 17, 40])
def test_batch_padding(B):
    t = ks.Tables.make(0.2)
    lens = [(37 * b) % 300 for b in range(B)]
    w = ks.distinct("batch", ks.ARCH_TINY, 24 + B, lens, gain_std=0.2)
    r, attn, _, _ = run_gpu(w, t)
    compare(w, t, gpu_rewards=r, gpu_attn=attn, label=f"B={B}")


@pytest.mark.parametrize("arch,lens", [
    (ks.Arch(2, 1536, 12, 2, 128, 8960), [2048] * 16),                   # 1.5B layer shapes, G = 6
    (ks.Arch(2, 3584, 28, 4, 128, 18944), [1, 300, 4096, 777, 64, 2000]),  # 7B layer shapes, G = 7
    (ks.Arch(2, 4096, 32, 8, 128, 14336), [5000, 4096, 1]),               # 8B layer shapes, G = 4
    (ks.Arch(2, 512, 16, 1, 64, 512), [0, 50, 129]),                      # G = 16 (two MMA row groups)
])
def test_layer_shapes(arch, lens):
    t = ks.Tables.make(0.2)
    w = ks.distinct("shapes", arch, 31, lens, gain_std=0.2)
    r, attn, _, _ = run_gpu(w, t)
    compare(w, t, gpu_rewards=r, gpu_attn=attn, label=f"arch {arch.d_model}/{arch.n_q_heads}/{arch.n_kv_heads}")


def test_two_tile_gate_up():
    """7B layer shapes at 200 candidates (padded to 208): the gate/up projection's one-tile CTAs
    would not fit on the SMs at once, so each CTA takes two m-tiles (two accumulators of N = 208
    side by side in TMEM, one activation stage for both); sampled candidates against the oracle."""
    t = ks.Tables.make(0.2)
    lens = [(53 * b) % 257 for b in range(200)]
    w = ks.distinct("two_tile", ks.Arch(2, 3584, 28, 4, 128, 18944), 57, lens, gain_std=0.2)
    r, attn, dev, sc = run_gpu(w, t)
    assert np.isfinite(r).all()
    ids = [0, 1, 100, 127, 128, 199]
    compare(w, t, cand_ids=ids, gpu_rewards=r, gpu_attn=attn, label="two-tile gate/up")
    sc.close()


@pytest.mark.parametrize("lens", [[16 * 9] * 4,            # 8 (candidate, kv head) pairs: clusters of 8
                                  [16 * 33 - 5] * 20,       # 40 pairs: clusters of 2
                                  [40] * 76,                # 152 pairs: one CTA each
                                  [100, 110, 120, 125]])    # about equal lengths, ragged last pages
@pytest.mark.parametrize("fused", [True, False])
def test_fused_combine(lens, fused, monkeypatch):
    # the combine merged by each cluster's rank 0 inside the attention launch, and the same calls
    # with the persistent plan and a combine launch
    if not fused:
        monkeypatch.setenv("KVPRM_NO_FUSED_COMBINE", "1")
    t = ks.Tables.make(0.2)
    w = ks.distinct("fused", ks.ARCH_TINY, 41 + len(lens), lens, gain_std=0.2)
    r, attn, _, _ = run_gpu(w, t)
    compare(w, t, gpu_rewards=r, gpu_attn=attn, label=f"fused={fused} lens={lens[:2]}x{len(lens)}")


def test_narrow_combine():
    # more (candidate, kv head) pairs than one wave of the general combine (240 candidates x 4 kv
    # heads = 960 > 6 x 152; a context holds at most 256 candidates), and than the SMs: the flat combine
    t = ks.Tables.make(0.2)
    lens = [int(x) for x in np.random.default_rng(47).integers(0, 60, size=240)]
    w = ks.distinct("narrow", ks.Arch(2, 256, 8, 4, 64, 512), 47, lens, gain_std=0.2)
    r, attn, _, _ = run_gpu(w, t)
    compare(w, t, gpu_rewards=r, gpu_attn=attn, label="narrow combine, 240 candidates x 4 kv heads")


def test_narrow_combine_depth_readout():
    # the same number of pairs from a depth-2 readout (120 candidates x 2 rows x 4 kv heads): the
    # general combine with four warps per pair and the causal verify-token entries
    t = ks.Tables.make(0.2)
    lens = [int(x) for x in np.random.default_rng(48).integers(0, 60, size=120)]
    w = ks.distinct("narrow_d2", ks.Arch(2, 256, 8, 4, 64, 512), 48, lens, gain_std=0.2)
    r, attn, _, _ = run_gpu(w, t, depth=2)
    compare(w, t, gpu_rewards=r, gpu_attn=attn, label="narrow combine, depth 2", depth=2)


# debug flag 64: the flat combine at every batch size
@pytest.mark.parametrize("make", [
    # empty and ragged caches, one to many partial slots per (candidate, kv head), head_dim 64
    lambda: ks.distinct("flat", ks.ARCH_TINY, 61, [0, 1, 15, 17, 300, 2500], gain_std=0.2),
    # head_dim 128, G = 7, shared pages (tensor-core and persistent partials) and private suffixes
    lambda: ks.shared_prefix("flat_tc", ARCH_G7, 62, 20, 530, 40, gain_std=0.2),
    lambda: ks.mcts_tree("flat_tree", ARCH_G7, 63, branching=3, depth=3, lo=5, hi=90, gain_std=0.2),
    # G = 16 (16 warps per CTA)
    lambda: ks.distinct("flat_g16", ks.Arch(2, 512, 16, 1, 64, 512), 64, [0, 50, 129, 3000], gain_std=0.2),
])
def test_flat_combine(make):
    t = ks.Tables.make(0.2)
    w = make()
    r, attn, _, _ = run_gpu(w, t, extra_flags=64)
    compare(w, t, gpu_rewards=r, gpu_attn=attn, label=f"flat combine {w.name}")


def test_attention_teacher_forced():
    """kvprm_attention on given fp32 q / self k / self v against the oracle's read-out."""
    torch = require_gpu()
    import paper_2607_09153_gb300 as kp
    arch = ks.Arch(1, 512, 12, 2, 128, 512)
    t = ks.Tables.make()
    w = ks.distinct("attn", arch, 41, [0, 1, 16, 17, 250, 2049, 4096])
    dev = ks.DeviceInputs(w, t)
    sc = make_scorer(dev, w.n_candidates, w.max_blocks)
    rng = np.random.default_rng(5)
    B, nq, nkv, hd = w.n_candidates, arch.n_q_heads, arch.n_kv_heads, arch.head_dim
    qf = rng.normal(0, 0.8, (B, nq, hd)).astype(np.float32)
    kf = rng.normal(0, 1, (B, nkv, hd)).astype(np.float32)
    vf = rng.normal(0, 1, (B, nkv, hd)).astype(np.float32)
    q, k, v = (torch.from_numpy(a).cuda() for a in (qf, kf, vf))
    out = torch.empty((B, nq, hd), dtype=torch.float32, device="cuda")
    kp.kvprm_attention(sc.ctx, dev.pool[0].data_ptr(), dev.n_pages, w.block_table, w.seq_lens, B, q.data_ptr(),
                       k.data_ptr(), v.data_ptr(), out.data_ptr(), torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    got = out.cpu().numpy().astype(np.float64)
    worst = 0.0
    for b in range(B):
        K, V = ks.host_kv_logical(w, 0, b, t)
        for h in range(nq):
            g = h // (nq // nkv)
            o, _ = oracle.attend(qf[b, h].astype(np.float64), K[:, g, :], V[:, g, :], kf[b, g].astype(np.float64),
                                 vf[b, g].astype(np.float64))
            e = np.abs(got[b, h] - o).max() / np.abs(o).max()
            worst = max(worst, e)
    print(f"teacher-forced attention: max rel err {worst:.3e}")
    assert worst <= ATTN_RTOL


def test_resolve_bit_exact():
    import paper_2607_09153_gb300 as kp
    t = ks.Tables.make()
    w = ks.mcts_tree("resolve", ks.ARCH_TINY, 42, branching=2, depth=3, lo=3, hi=50)
    _, _, dev, sc = run_gpu(w, t, debug=False)
    for b in range(w.n_candidates):
        L = int(w.seq_lens[b])
        got = kp.kvprm_resolve(sc.ctx, b, L)
        pos = np.arange(L)
        ref = w.block_table[b, pos // 16].astype(np.int64) * 16 + pos % 16
        np.testing.assert_array_equal(got, ref)
        # and the rows it names hold the candidate's logical tokens
        seg = w.page_seg.reshape(-1)[got]
        off = w.page_off.reshape(-1)[got]
        np.testing.assert_array_equal(seg, w.cand_seg[b])
        np.testing.assert_array_equal(off, w.cand_off[b])


def test_deterministic_and_host_path():
    import paper_2607_09153_gb300 as kp
    torch = require_gpu()
    t = ks.Tables.make(0.2)
    w = ks.distinct("det", ks.ARCH_TINY, 43, [5, 600, 1234, 64], gain_std=0.2)
    r1, _, dev, sc = run_gpu(w, t, debug=False)
    r2 = sc.score(dev.pool, w.block_table, w.seq_lens)
    assert np.array_equal(r1.astype(np.float32), r2)
    sp = torch.cuda.current_stream().cuda_stream
    # the host cache pinned, pageable, and pinned at an address 8 bytes off a 16-byte boundary: the
    # same rewards, bit for bit, and the pinned buffer again after the others
    host_pool = dev.pool.cpu().pin_memory()
    r3 = kp.kvprm_score_host(sc.ctx, host_pool.data_ptr(), dev.n_pages, w.block_table, w.seq_lens, w.n_candidates, sp)
    assert np.array_equal(r3, r2)
    pageable = dev.pool.cpu()
    assert not pageable.is_pinned()
    r4 = kp.kvprm_score_host(sc.ctx, pageable.data_ptr(), dev.n_pages, w.block_table, w.seq_lens, w.n_candidates, sp)
    assert np.array_equal(r4, r2)
    raw = torch.empty(host_pool.numel() * 2 + 16, dtype=torch.uint8).pin_memory()
    off = (8 - raw.data_ptr()) % 16
    raw[off:off + host_pool.numel() * 2].copy_(host_pool.view(-1).view(torch.uint8))
    r5 = kp.kvprm_score_host(sc.ctx, raw.data_ptr() + off, dev.n_pages, w.block_table, w.seq_lens, w.n_candidates, sp)
    assert np.array_equal(r5, r2)
    r6 = kp.kvprm_score_host(sc.ctx, host_pool.data_ptr(), dev.n_pages, w.block_table, w.seq_lens, w.n_candidates, sp)
    assert np.array_equal(r6, r2)
    d = torch.empty(w.n_candidates, dtype=torch.float32, device="cuda")
    sc.score_async(dev.pool, w.block_table, w.seq_lens, d)
    torch.cuda.synchronize()
    assert np.array_equal(d.cpu().numpy(), r2)


def test_host_side_errors():
    import paper_2607_09153_gb300 as kp
    t = ks.Tables.make()
    w = ks.distinct("err", ks.ARCH_TINY, 44, [20, 40])
    _, _, dev, sc = run_gpu(w, t, debug=False)
    bt = w.block_table.copy()
    bt[1, 1] = dev.n_pages            # out of range page id
    with pytest.raises(kp.KvprmError) as e:
        sc.score(dev.pool, bt, w.seq_lens)
    assert e.value.code == 3
    bt = w.block_table.copy()
    bt[0, 2] = -7                     # beyond ceil(20/16) = 2 blocks: ignored
    sc.score(dev.pool, bt, w.seq_lens)
    with pytest.raises(kp.KvprmError) as e:    # longer than max_blocks * 16
        sc.score(dev.pool, w.block_table, np.array([20, 16 * w.max_blocks + 1], np.int32))
    assert e.value.code == 2
    with pytest.raises(kp.KvprmError) as e:    # more candidates than the context holds
        kp.kvprm_score(sc.ctx, dev.pool.data_ptr(), dev.n_pages, np.zeros((3, w.max_blocks), np.int32),
                       np.zeros(3, np.int32), 3)
    assert e.value.code == 2
    with pytest.raises(kp.KvprmError) as e:
        sc.score(dev.pool, w.block_table, np.array([20, -1], np.int32))
    assert e.value.code == 1
    assert kp.kvprm_score(sc.ctx, 0, 0, np.zeros((0, 1), np.int32), np.zeros(0, np.int32), 0).size == 0


# ---------------------------------------------------------------- scorer adapter (kvprm_set_lora)
def _lora_arch(arch, rank):
    import dataclasses
    return dataclasses.replace(arch, lora_rank=rank)


@pytest.mark.parametrize("arch,rank,lens,sample", [
    (ks.ARCH_TINY, 64, [0, 50, 129, 200], None),                                    # r = 64: half an A tile
    (ks.ARCH_TINY, 1024, [7, 90], None),                                             # the largest rank
    (ks.Arch(2, 1536, 12, 2, 128, 8960), 256, [2048] * 16, None),                   # 1.5B layers, small image
    (ks.Arch(2, 3584, 28, 4, 128, 18944), 256, [(37 * b) % 300 for b in range(64)],  # 7B layers, B = 64
     [0, 1, 31, 63]),
    (ks.Arch(2, 3584, 28, 4, 128, 18944), 128, [(53 * b) % 257 for b in range(200)],  # two m-tiles per gate/up CTA
     [0, 100, 199]),
])
def test_lora(arch, rank, lens, sample):
    """Every projection y = W x + (alpha / r) B (A x) with the factors kept apart (Sec. 4.1, App. B.1):
    t = s A x on its own launch, then W x + B t as one K loop; against the oracle's fp64 adapter."""
    t = ks.Tables.make(0.2)
    w = ks.distinct("lora", _lora_arch(arch, rank), 61 + rank, lens, gain_std=0.2)
    r, attn, dev, sc = run_gpu(w, t)
    compare(w, t, cand_ids=sample, gpu_rewards=r, gpu_attn=attn, label=f"adapter r={rank} d={arch.d_model}")
    sc.close()


def test_lora_switch_and_errors():
    """Rank 0 restores the merged scorer bit for bit; bad arguments leave the context as it was."""
    import paper_2607_09153_gb300 as kp
    t = ks.Tables.make(0.2)
    w = ks.distinct("lora_sw", _lora_arch(ks.ARCH_TINY, 64), 71, [3, 40, 100], gain_std=0.2)
    dev = ks.DeviceInputs(w, t)
    sc = make_scorer(dev, 8, w.max_blocks)
    with_lora = sc.score(dev.pool, w.block_table, w.seq_lens)
    sc.set_lora(0)
    merged = sc.score(dev.pool, w.block_table, w.seq_lens)
    w0 = ks.distinct("lora_sw", ks.ARCH_TINY, 71, [3, 40, 100], gain_std=0.2)   # same seed: same weights and cache
    dev0 = ks.DeviceInputs(w0, t)
    fresh = make_scorer(dev0, 8, w0.max_blocks)
    base = fresh.score(dev0.pool, w0.block_table, w0.seq_lens)
    assert np.array_equal(merged, base)
    assert np.abs(with_lora - merged).max() > 1e-5
    for bad in (32, 100, 2048, -64):
        with pytest.raises(kp.KvprmError):
            kp.kvprm_set_lora(sc.ctx, bad, 0.5, None)
    with pytest.raises(kp.KvprmError):
        kp.kvprm_set_lora(sc.ctx, 64, 0.5, None)
    assert np.array_equal(sc.score(dev.pool, w.block_table, w.seq_lens), merged)
    fresh.close()
    sc.close()


# ---------------------------------------------------------------- depth-k readout (kvprm_set_readout_depth)
@pytest.mark.parametrize("arch,depth,make", [
    (ks.ARCH_TINY, 3, lambda a: ks.distinct("depth", a, 81, [0, 17, 100, 250], gain_std=0.2)),
    (ks.Arch(2, 1536, 12, 2, 128, 8960), 4, lambda a: ks.distinct("depth", a, 82, [2048] * 4, gain_std=0.2)),
    # 8 rows per candidate on the tensor-core path for a 64-row shared prefix group (G = 7)
    (ks.Arch(2, 3584, 28, 4, 128, 18944), 2, lambda a: ks.shared_prefix("depth", a, 83, 8, 256, 40, gain_std=0.2)),
])
def test_depth_readout(arch, depth, make):
    """k verify tokens per candidate, causal among themselves, reward at the last (Sec. 3 R_k, Sec. 5):
    every token's attention output per layer and P(+) against the oracle's depth-k readout."""
    t = ks.Tables.make(0.2)
    w = make(arch)
    r, attn, dev, sc = run_gpu(w, t, depth=depth)
    compare(w, t, gpu_rewards=r, gpu_attn=attn, label=f"depth {depth} d={arch.d_model}", depth=depth)
    # depth 1 on the same context gives the single-token scores
    sc.set_depth(1)
    r1 = sc.score(dev.pool, w.block_table, w.seq_lens)
    ref1 = oracle.score_synth(w, t, mirror=False)
    assert np.abs(r1 - ref1.p_plus).max() <= 1e-3
    sc.close()


def test_depth_errors():
    import paper_2607_09153_gb300 as kp
    t = ks.Tables.make(0.2)
    w = ks.distinct("depth_err", ks.ARCH_TINY, 84, [5, 9, 30], gain_std=0.2)
    dev = ks.DeviceInputs(w, t)
    sc = make_scorer(dev, 4, w.max_blocks)   # room for 4 rows
    for bad in (0, 9, -1):
        with pytest.raises(kp.KvprmError):
            sc.set_depth(bad)
    sc.set_depth(2)   # 3 candidates x 2 rows > 4
    with pytest.raises(kp.KvprmError):
        sc.score(dev.pool, w.block_table, w.seq_lens)
    sc.set_depth(1)
    r = sc.score(dev.pool, w.block_table, w.seq_lens)
    assert np.isfinite(r).all()
    sc.close()


def test_lora_with_depth_readout():
    """Both extensions at once: a rank-64 adapter on every projection and 3 verify tokens per candidate."""
    t = ks.Tables.make(0.2)
    w = ks.distinct("lora_depth", _lora_arch(ks.ARCH_TINY, 64), 91, [0, 33, 140], gain_std=0.2)
    r, attn, dev, sc = run_gpu(w, t, depth=3)
    compare(w, t, gpu_rewards=r, gpu_attn=attn, label="adapter r=64 with depth 3", depth=3)
    sc.close()


# ---------------------------------------------------------------- per-head q/k RMSNorm (kvprm_config.qk_norm)
def _qk(arch):
    import dataclasses
    return dataclasses.replace(arch, qk_norm=True)


@pytest.mark.parametrize("make", [
    lambda: ks.distinct("qkn_tiny", _qk(ks.ARCH_TINY), 401, [0, 5, 128, 333], gain_std=0.2),     # hd 64, two heads a tile
    lambda: ks.distinct("qkn_15", _qk(ks.Arch(2, 1536, 12, 2, 128, 8960)), 402, [2048] * 16, gain_std=0.2),
    lambda: ks.shared_prefix("qkn_7b", _qk(ks.Arch(2, 3584, 28, 4, 128, 18944)), 403, 64, 256, 20, gain_std=0.2),
])
def test_qk_norm(make):
    """The paper's Qwen3 scorers normalise each q and k head before RoPE (Sec. 5 "Setup"): the QKV
    epilogue's per-head RMSNorm (small- and large-batch kernel images) against the oracle's."""
    t = ks.Tables.make(0.2)
    w = make()
    r, attn, dev, sc = run_gpu(w, t)
    ids = None if w.n_candidates <= 16 else [0, 1, 31, 63]
    compare(w, t, cand_ids=ids, gpu_rewards=r, gpu_attn=attn, label=f"qk_norm {w.name}")
    sc.close()
