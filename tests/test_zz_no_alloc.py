"""kvprm_attention_noalloc, the attention entry point for callers that cannot allocate device
memory (its scratch is a static device array): its output against the CPU oracle's read-out and
against the context-based kvprm_attention, on two calls in a row, for distinct caches and for a
beam-shaped shared prefix (shared runs laid out in the array), with peaked softmax.

This file is collected last so that a run stopping at the first failure has already run every
other test; it also passes alone in a fresh process."""
import numpy as np
import pytest

import kvsynth as ks
from tests.gpu_util import ATTN_RTOL, PlantedCase, make_scorer, require_gpu, row_rel_err

pytestmark = pytest.mark.gpu

ARCH = ks.Arch(1, 512, 12, 2, 128, 512)


def _cases():
    w1 = ks.distinct("noalloc", ARCH, 51, [0, 1, 17, 300, 2049, 4096, 33])
    w2 = ks.shared_prefix("noalloc_beam", ARCH, 52, 5, 1040, 70)   # 5 candidates share 65 pages
    return [("distinct", PlantedCase(w1, ks.Tables.make(), 51, [(b, int(L) - 1) for b, L in enumerate(w1.seq_lens)
                                                                 if L > 0])),
            ("shared prefix", PlantedCase(w2, ks.Tables.make(), 52, [(0, 1030), (2, 69)], runs=[(0, 500, 32)]))]


@pytest.mark.parametrize("which", [0, 1])
def test_noalloc_matches_oracle_twice(which):
    torch = require_gpu()
    import paper_2607_09153_gb300 as kp
    label, case = _cases()[which]
    w, a = case.w, case.arch
    B, nq, nkv, hd = w.n_candidates, a.n_q_heads, a.n_kv_heads, a.head_dim
    pool, q, k, v = case.device()
    stream = torch.cuda.current_stream().cuda_stream
    ref = case.expected()
    # the context entry point on the same inputs
    dev = ks.DeviceInputs(ks.distinct("host", a, 1, [16]), ks.Tables.make())
    sc = make_scorer(dev, B, w.max_blocks)
    ctx_out = torch.empty((B, nq, hd), dtype=torch.float32, device="cuda")
    kp.kvprm_attention(sc.ctx, pool.data_ptr(), w.n_pages, w.block_table, w.seq_lens, B, q.data_ptr(), k.data_ptr(),
                       v.data_ptr(), ctx_out.data_ptr(), stream)
    torch.cuda.synchronize()
    c = ctx_out.cpu().numpy().astype(np.float64)
    for call in range(2):
        out = torch.full((B, nq, hd), float("nan"), dtype=torch.float32, device="cuda")
        kp.kvprm_attention_noalloc(pool.data_ptr(), w.n_pages, w.block_table, w.seq_lens, nq, nkv, hd, q.data_ptr(),
                                   k.data_ptr(), v.data_ptr(), out.data_ptr(), stream)
        torch.cuda.synchronize()
        got = out.cpu().numpy().astype(np.float64)
        assert np.isfinite(got).all(), f"{label} call {call}: unwritten outputs"
        err = row_rel_err(got, ref)
        err_ctx = row_rel_err(got, c)
        print(f"no-alloc {label} call {call}: max rel err vs oracle {err:.3e}, vs kvprm_attention {err_ctx:.3e}")
        assert err <= ATTN_RTOL and err_ctx <= ATTN_RTOL
    sc.close()


def test_noalloc_rejects_oversize():
    torch = require_gpu()
    import paper_2607_09153_gb300 as kp
    # 256 candidates x 128 query heads x 128 dims: the query's hi/lo parts and the
    # combine's hi/lo output alone take 4 x 8 MiB, beyond the 32 MiB scratch array
    B, nq, nkv, hd = 256, 128, 8, 128
    q = torch.zeros((B, nq, hd), dtype=torch.float32, device="cuda")
    k = torch.zeros((B, nkv, hd), dtype=torch.float32, device="cuda")
    with pytest.raises(kp.KvprmError) as e:
        kp.kvprm_attention_noalloc(0, 0, np.zeros((B, 1), np.int32), np.zeros(B, np.int32), nq, nkv, hd,
                                   q.data_ptr(), k.data_ptr(), k.data_ptr(), q.data_ptr(), 0)
    assert e.value.code == 2


def test_noalloc_refuses_capturing_stream():
    """A call on a stream being captured returns KVPRM_EUNSUPPORTED and enqueues nothing."""
    torch = require_gpu()
    import paper_2607_09153_gb300 as kp
    B, nq, nkv, hd = 2, 12, 2, 128
    q = torch.zeros((B, nq, hd), dtype=torch.float32, device="cuda")
    k = torch.zeros((B, nkv, hd), dtype=torch.float32, device="cuda")
    out = torch.zeros((B, nq, hd), dtype=torch.float32, device="cuda")
    x = torch.zeros(16, device="cuda")
    s = torch.cuda.Stream()
    g = torch.cuda.CUDAGraph()
    codes = []
    with torch.cuda.graph(g, stream=s, capture_error_mode="thread_local"):
        try:
            kp.kvprm_attention_noalloc(0, 0, np.zeros((B, 1), np.int32), np.zeros(B, np.int32), nq, nkv, hd,
                                       q.data_ptr(), k.data_ptr(), k.data_ptr(), out.data_ptr(), s.cuda_stream)
        except kp.KvprmError as e:
            codes.append(e.code)
        x.add_(1.0)   # the graph needs one node
    torch.cuda.synchronize()
    assert codes == [kp.KVPRM_EUNSUPPORTED]
