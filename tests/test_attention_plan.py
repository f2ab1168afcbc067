"""Host logic of the paged-attention schedule (kvprm_plan_attention; no GPU).

The read-out of App. A.3 is split into segments of pages scored per kv head;
whatever the split, every cached token of every candidate must be scored
exactly once per kv head, every partial slot must belong to exactly one
(candidate, kv head), and the CTAs must get equal shares of the work.  These
checks recompute all of that from the block tables, independently of the
planner."""
import collections

import numpy as np
import pytest

import kvsynth as ks
import paper_2607_09153_gb300.kvprm as kp

PRIVATE_COST, SHARED_COST_PER_CAND = 4, 2   # the planner's per-page cost model
TC_CHUNK_COST, TC_CTA_COST = 26, 180        # its tensor-core launch: per 64-token chunk, per CTA


def check_plan(bt, sl, n_kv, group, n_ctas, share):
    share = int(share)
    flags = share & kp.KVPRM_PLAN_FUSE
    bt = np.asarray(bt, np.int32)
    sl = np.asarray(sl, np.int32)
    n = len(sl)
    p = kp.kvprm_plan_attention(bt, sl, n_kv, group, n_ctas, share)
    share &= ~flags
    segs, cta = p["segs"], p["cta_seg"]
    # expected multiset of (b, g, page, valid tokens)
    want = collections.Counter()
    for b in range(n):
        npg = (int(sl[b]) + 15) // 16
        for g in range(n_kv):
            for j in range(npg):
                want[(b, g, int(bt[b, j]), 16 if j < npg - 1 else int(sl[b]) - 16 * (npg - 1))] += 1
    got = collections.Counter()
    used = collections.defaultdict(list)   # (b, g) -> slots
    assert p["n_ctas"] <= n_ctas
    if p["n_ctas"]:
        assert cta[0] == 0 and np.all(np.diff(cta) >= 0)
        assert cta[-1] == len(segs) if share < 2 else cta[-1] <= len(segs)
    cost = np.zeros(max(p["n_ctas"], 1))
    for k in range(p["n_ctas"]):
        for s in segs[cta[k]:cta[k + 1]]:
            kind, g, c, nc, off, npg, last, slot = (int(x) for x in s)
            assert 0 <= g < n_kv and npg >= 1 and 1 <= last <= 16
            pages = p["pages"][off:off + npg]
            if kind == 0:
                cands = [c]
                k_slots = 1 if group <= 8 else min(8, npg)
                slots = [[slot + i for i in range(k_slots)]]
                cost[k] += PRIVATE_COST * npg
            else:
                # kind 1: shared runs on the persistent CTAs (share 1, or share >= 2 for pages
                # shared by fewer candidates than a tensor-core tile is worth)
                assert kind == 1 and share >= 1 and 1 <= nc <= 8 and last == 16
                cands = [int(x) for x in p["cands"][c:c + nc]]
                # (8 // nc) replica warps per candidate, slot w of the segment for warp w (candidate w % nc)
                reps = 8 // nc
                slots = [[int(p["slots"][slot + w]) for w in range(reps * nc) if w % nc == k2] for k2 in range(nc)]
                cost[k] += SHARED_COST_PER_CAND * nc * npg
            for b, sls in zip(cands, slots):
                used[(b, g)] += sls
                for i, pg in enumerate(pages):
                    got[(b, g, int(pg), last if i == npg - 1 else 16)] += 1
    # tensor-core segments (share >= 2) follow the persistent CTAs' segments
    tc0 = int(cta[-1]) if p["n_ctas"] else 0
    for s in segs[tc0:]:
        kind, g, c, nc, off, npg, last, slot = (int(x) for x in s)
        assert kind == 2 and share >= 2 and 0 <= g < n_kv and npg >= 1 and last == 16
        assert 1 <= nc <= 128 // group, "a tile holds at most 128 query rows"
        for b, sl_ in zip(p["cands"][c:c + nc], p["slots"][slot:slot + nc]):
            used[(int(b), g)].append(int(sl_))
            for pg in p["pages"][off:off + npg]:
                got[(int(b), g, int(pg), 16)] += 1
    assert got == want, "every cached token scored exactly once per kv head"
    for b in range(n):
        for g in range(n_kv):
            base, cnt = int(p["slot_base"][b * n_kv + g]), int(p["nslots"][b * n_kv + g])
            assert sorted(used[(b, g)]) == list(range(base, base + cnt)), (b, g)
    assert int(p["nslots"].sum()) == p["n_slots"]
    if p["n_ctas"] > 1:
        total = cost.sum()
        unit = PRIVATE_COST if share == 0 else max(PRIVATE_COST, SHARED_COST_PER_CAND * 8)
        assert np.abs(cost - total / p["n_ctas"]).max() <= unit, "equal CTA shares up to one page"
    return p


@pytest.mark.parametrize("name", ["tiny", "qwen1p5b_b16_l2048", "beam7b_b64_p4096_s512", "long8b_b8_l32768",
                                  "mcts7b_b256_d4"])
@pytest.mark.parametrize("share", [0, 1, 2, 3])
def test_workload_plans(name, share):
    w = ks.make_workload(name)
    a = w.arch
    p = check_plan(w.block_table, w.seq_lens, a.n_kv_heads, a.n_q_heads // a.n_kv_heads, 152, share)
    if not share:
        assert (p["segs"][:, 0] == 0).all()
    if share == 3 and p["n_tc_ctas"] and p["n_ctas"]:
        assert p["n_ctas"] + p["n_tc_ctas"] <= 152, "side by side, the two launches share the SMs"
    if share >= 2 and name in ("beam7b_b64_p4096_s512", "mcts7b_b256_d4"):
        tc = p["segs"][p["segs"][:, 0] == 2]
        # at most one tensor-core CTA per SM, equal chunk counts up to one, every kind-2 segment owned once;
        # within a (tile, kv head) every piece but the last is whole 4-page chunks
        tcc, nt = p["tc_cta"], p["n_tc_ctas"]
        assert 1 <= nt <= 152 and tcc[0] == len(p["segs"]) - len(tc) and tcc[-1] == len(p["segs"])
        per_cta = [sum((int(x[5]) + 3) // 4 for x in p["segs"][tcc[k]:tcc[k + 1]]) for k in range(nt)]
        assert max(per_cta) - min(per_cta) <= 1
        parts = collections.defaultdict(list)
        for s in tc:
            parts[(int(s[2]), int(s[1]))].append((int(s[4]), int(s[5])))
        for lst in parts.values():
            lst.sort()
            assert all(npg % 4 == 0 for _, npg in lst[:-1])
            assert all(o0 + n0 == o1 for (o0, n0), (o1, _) in zip(lst, lst[1:])), "parts tile the run's pages"


def test_shared_prefix_is_read_once_per_chunk():
    # 20 candidates share a 10-page prefix, then own 3 pages each
    n, pre, own = 20, 10, 3
    bt = np.zeros((n, pre + own), np.int32)
    for b in range(n):
        bt[b, :pre] = np.arange(pre)
        bt[b, pre:] = pre + own * b + np.arange(own)
    sl = np.full(n, 16 * (pre + own) - 5, np.int32)
    p = check_plan(bt, sl, 2, 4, 16, True)
    shared = p["segs"][p["segs"][:, 0] == 1]
    # the prefix pages go to shared segments of <= 8 candidates: ceil(20 / 8) = 3 chunks per head
    per_head = collections.Counter()
    for s in shared:
        per_head[int(s[1])] += int(s[5])
    assert per_head == {0: 3 * pre, 1: 3 * pre}


def test_shared_prefix_tensor_core_tiles():
    # 40 candidates share a 33-page prefix (G = 7: tiles of <= 18 candidates -> 3 tiles of 13-14)
    n, pre, own = 40, 33, 2
    bt = np.zeros((n, pre + own), np.int32)
    for b in range(n):
        bt[b, :pre] = np.arange(pre)
        bt[b, pre:] = pre + own * b + np.arange(own)
    sl = np.full(n, 16 * (pre + own) - 3, np.int32)
    p = check_plan(bt, sl, 2, 7, 24, 2)
    tc = p["segs"][p["segs"][:, 0] == 2]
    assert sorted(set(tc[:, 3].tolist())) == [13, 14], "candidates spread evenly over the fewest tiles"
    per_tile_head = collections.Counter()
    for s in tc:
        per_tile_head[(int(s[2]), int(s[1]))] += int(s[5])
    assert len(per_tile_head) == 3 * 2 and set(per_tile_head.values()) == {pre}, "each tile reads the prefix once"


@pytest.mark.parametrize("share", [1, 2, 3])
def test_tiles_with_the_same_candidates_share_one_run(share):
    # an MCTS-like tree: pages 0..9 shared by all 32 candidates (G = 7: two tensor-core tiles of
    # 16), pages 10..21 by candidates 0..15 and pages 22..29 by candidates 16..31, then 2 own pages
    # each.  Each tile of the 32-candidate group has the same candidates as one of the smaller
    # groups: one run over both groups' pages (10 + 12 or 10 + 8).  On the persistent kernel (runs
    # of <= 8 candidates) the same holds run by run.
    n = 32
    bt = np.zeros((n, 24), np.int32)
    sl = np.zeros(n, np.int32)
    for b in range(n):
        mid = (10 + np.arange(12)) if b < 16 else (22 + np.arange(8))
        row = np.concatenate([np.arange(10), mid, 100 + 2 * b + np.arange(2)])
        bt[b, :len(row)] = row
        sl[b] = 16 * len(row) - 5
    p = check_plan(bt, sl, 2, 7, 40, share)
    kind = 2 if share >= 2 else 1
    runs = collections.defaultdict(int)   # (candidate offset, kv head) -> pages
    for seg in p["segs"][p["segs"][:, 0] == kind]:
        runs[(int(seg[2]), int(seg[1]))] += int(seg[5])
    if kind == 2:
        assert sorted(runs.values()) == [18, 18, 22, 22], runs
    else:
        assert sorted(runs.values()) == [18] * 4 + [22] * 4, runs


@pytest.mark.parametrize("n_share, kind", [(4, 1), (5, 1), (6, 2), (9, 2)])
def test_small_shared_groups_stay_on_the_persistent_kernel(n_share, kind):
    # pages shared by fewer than 6 candidates are scored as kind-1 runs even in the tensor-core modes
    n, pre, own = 12, 9, 2
    bt = np.zeros((n, pre + own), np.int32)
    for b in range(n):
        bt[b, :pre] = np.arange(pre) if b < n_share else 100 + pre * b + np.arange(pre)
        bt[b, pre:] = 1000 + own * b + np.arange(own)
    sl = np.full(n, 16 * (pre + own), np.int32)
    for share in (2, 3):
        p = check_plan(bt, sl, 2, 7, 24, share)
        shared = p["segs"][p["segs"][:, 0] != 0]
        assert len(shared) and set(shared[:, 0].tolist()) == {kind}


def test_concurrent_split_shares_the_sms():
    # a shared prefix (tensor cores) and private suffixes (persistent kernel) side by side
    n, pre, own = 40, 64, 24
    bt = np.zeros((n, pre + own), np.int32)
    for b in range(n):
        bt[b, :pre] = np.arange(pre)
        bt[b, pre:] = pre + own * b + np.arange(own)
    sl = np.full(n, 16 * (pre + own), np.int32)
    p3 = check_plan(bt, sl, 2, 7, 64, 3)
    assert p3["n_tc_ctas"] >= 1 and p3["n_ctas"] >= 1 and p3["n_tc_ctas"] + p3["n_ctas"] <= 64
    # the split minimises the later launch's end under the cost model: a tensor-core CTA costs 26 per
    # 64-token chunk plus 180, a private page 4 (both per kv head)
    chunks = 2 * ((pre + 3) // 4) * len(set(p3["segs"][p3["segs"][:, 0] == 2][:, 2].tolist()))
    units = 2 * n * own * PRIVATE_COST

    def later_end(x):
        return max(-(-chunks // x) * TC_CHUNK_COST + TC_CTA_COST, -(-units // (64 - x)))

    x = p3["n_tc_ctas"]
    assert all(later_end(x) <= later_end(y) for y in range(1, 64))
    p2 = check_plan(bt, sl, 2, 7, 64, 2)   # serial: each launch planned over all SMs
    assert p2["n_ctas"] == 64 and p2["n_tc_ctas"] == 64


@pytest.mark.parametrize("name, cs", [("tiny", 8), ("qwen1p5b_b16_l2048", 4), ("long8b_b8_l32768", 0),
                                      ("beam7b_b64_p4096_s512", 0), ("mcts7b_b256_d4", 0)])
def test_fused_combine_plan(name, cs):
    # equal lengths, no sharing, group <= 8 and few pages per CTA: pair p on cluster p, one slot per rank
    w = ks.make_workload(name)
    a = w.arch
    n_kv, group = a.n_kv_heads, a.n_q_heads // a.n_kv_heads
    p = check_plan(w.block_table, w.seq_lens, n_kv, group, 152, 3 | kp.KVPRM_PLAN_FUSE)
    assert p["fuse_cs"] == cs
    if not cs:
        return
    n = len(w.seq_lens)
    assert p["n_ctas"] == n * n_kv * cs <= 152 and len(p["segs"]) == p["n_ctas"]
    for k in range(p["n_ctas"]):
        (seg,) = p["segs"][p["cta_seg"][k]:p["cta_seg"][k + 1]]
        pr, r = divmod(k, cs)
        b, g = divmod(pr, n_kv)
        assert seg[0] == 0 and seg[2] == b and seg[1] == g and seg[7] == pr * cs + r
        npg = (int(w.seq_lens[b]) + 15) // 16
        assert seg[5] == (r + 1) * npg // cs - r * npg // cs and seg[5] <= 64
    assert (p["slot_base"] == np.arange(n * n_kv) * cs).all() and (p["nslots"] == cs).all()


@pytest.mark.parametrize("case", ["ragged", "shared", "repeat", "empty", "wide_group"])
def test_fused_combine_plan_declines(case):
    n, npg = 6, 8
    bt = np.arange(n * npg, dtype=np.int32).reshape(n, npg)
    sl = np.full(n, 16 * npg, np.int32)
    group = 4
    if case == "ragged":
        sl[0] = 16 * 4   # 4 pages against 8
    elif case == "shared":
        bt[1, 0] = bt[0, 0]
    elif case == "repeat":
        bt[2, 3] = bt[2, 2]
    elif case == "empty":
        sl[3] = 0
    else:
        group = 12
    p = check_plan(bt, sl, 2, group, 152, 1 | kp.KVPRM_PLAN_FUSE)
    assert p["fuse_cs"] == 0


def test_repeated_page_in_one_candidate_stays_private():
    bt = np.array([[3, 3, 4], [3, 3, 5]], np.int32)   # page 3 listed twice by both candidates
    sl = np.array([48, 48], np.int32)
    p = check_plan(bt, sl, 1, 2, 4, True)
    assert (p["segs"][:, 0] == 0).all()


def test_partial_last_page_is_never_shared():
    bt = np.array([[0, 1], [0, 1]], np.int32)
    sl = np.array([20, 20], np.int32)   # page 1 is partial (4 tokens) for both
    p = check_plan(bt, sl, 1, 1, 4, True)
    for s in p["segs"]:
        if s[0] == 1:
            assert 1 not in set(p["pages"][s[4]:s[4] + s[5]].tolist())


@pytest.mark.parametrize("lens", [[0], [0, 0, 0], [1], [16], [17], [0, 1, 15, 16, 17, 31, 33, 100, 257, 1000]])
@pytest.mark.parametrize("n_ctas", [1, 3, 152])
@pytest.mark.parametrize("share", [1, 2, 3])
def test_edges(lens, n_ctas, share):
    n = len(lens)
    mb = max(1, max((L + 15) // 16 for L in lens))
    bt = np.arange(n * mb, dtype=np.int32).reshape(n, mb)
    p = check_plan(bt, lens, 2, 3, n_ctas, share)
    for b, L in enumerate(lens):
        if L == 0:
            assert (p["nslots"][b * 2:(b + 1) * 2] == 0).all(), "an empty cache has no partial: self entry only"


def test_two_row_groups_count_one_slot_per_busy_warp():
    bt = np.arange(3 * 40, dtype=np.int32).reshape(3, 40)
    sl = np.array([5, 100, 640], np.int32)
    check_plan(bt, sl, 1, 16, 7, True)


def test_deterministic():
    w = ks.make_workload("mcts7b_b256_d4")
    a = w.arch
    p1 = kp.kvprm_plan_attention(w.block_table, w.seq_lens, a.n_kv_heads, a.n_q_heads // a.n_kv_heads, 152)
    p2 = kp.kvprm_plan_attention(w.block_table, w.seq_lens, a.n_kv_heads, a.n_q_heads // a.n_kv_heads, 152)
    for k in ("segs", "cta_seg", "pages", "cands", "slots", "slot_base", "nslots"):
        assert np.array_equal(p1[k], p2[k]), k


def test_bad_arguments():
    with pytest.raises(kp.KvprmError):
        kp.kvprm_plan_attention(np.zeros((1, 1), np.int32), [17], 1, 1, 4)   # 17 tokens > 16 * 1 block
    with pytest.raises(kp.KvprmError):
        kp.kvprm_plan_attention(np.zeros((1, 1), np.int32), [1], 1, 17, 4)   # G > 16


@pytest.mark.parametrize("k", [2, 4, 8])
def test_depth_rows_stream_each_page_once(k):
    """A depth-k readout expands each candidate into k rows over the same pages (kvprm_set_readout_depth):
    the schedule must score every token for every row, yet stream each (page, kv head) once, the k rows
    forming one sharing group (shared runs below 6 rows, the tensor-core path from 6)."""
    w = ks.make_workload("qwen1p5b_b16_l2048")
    bt = np.repeat(np.asarray(w.block_table, np.int32), k, axis=0)
    sl = np.repeat(np.asarray(w.seq_lens, np.int32), k)
    p = check_plan(bt, sl, 2, 6, 152, 3)
    streams = collections.Counter()
    for s in p["segs"]:
        kind, g, c, nc, off, npg, last, slot = (int(x) for x in s)
        assert kind != 0, "a row of a depth-k candidate was planned as private pages"
        for pg in p["pages"][off:off + npg]:
            streams[(int(pg), g)] += 1
    assert set(streams.values()) == {1}


@pytest.mark.parametrize("share", [1, 3])
def test_sparse_page_ids_plan_alike(share):
    """Page ids far larger than the number of references (and a negative one, which only the host-only
    planner entry accepts unchecked) take the planner's hash-map path instead of its dense arrays:
    the schedule is the same up to the renaming of the pages."""
    w = ks.mcts_tree("sparse", ks.Arch(1, 256, 14, 2, 128, 256), 29, branching=3, depth=3, lo=5, hi=90)
    bt, sl = np.asarray(w.block_table, np.int32), np.asarray(w.seq_lens, np.int32)
    dense = check_plan(bt, sl, 2, 7, 64, share)
    for rename in (lambda x: x * 4099 + 11, lambda x: x - 1):
        bt2 = rename(bt.astype(np.int64)).astype(np.int32)
        p = kp.kvprm_plan_attention(bt2, sl, 2, 7, 64, share)
        for k in ("segs", "cta_seg", "cands", "slots", "slot_base", "nslots"):
            np.testing.assert_array_equal(p[k], dense[k], err_msg=k)
        np.testing.assert_array_equal(p["pages"], rename(np.asarray(dense["pages"], np.int64)).astype(np.int32))
