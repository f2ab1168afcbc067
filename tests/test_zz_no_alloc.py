"""kvprm_attention_noalloc, the attention entry point for callers that cannot
allocate device memory (its scratch is a static device array), against the
context-based kvprm_attention on the same inputs, on two calls in a row.

This file is collected last so that a run stopping at the first failure has
already run every other test; it also passes alone in a fresh process."""
import numpy as np
import pytest

import kvsynth as ks
from tests.gpu_util import ATTN_RTOL, make_scorer, require_gpu

pytestmark = pytest.mark.gpu


def _rel(a, b):
    return float(np.abs(a - b).max() / np.abs(b).max())


def test_noalloc_matches_context_entry_point_twice():
    torch = require_gpu()
    import paper_2607_09153_gb300 as kp
    arch = ks.Arch(1, 512, 12, 2, 128, 512)
    t = ks.Tables.make()
    w = ks.distinct("noalloc", arch, 51, [0, 1, 17, 300, 2049, 4096, 33])
    dev = ks.DeviceInputs(w, t)
    sc = make_scorer(dev, w.n_candidates, w.max_blocks)
    B, nq, nkv, hd = w.n_candidates, arch.n_q_heads, arch.n_kv_heads, arch.head_dim
    rng = np.random.default_rng(7)
    q, k, v = (torch.from_numpy(rng.normal(0, s, shape).astype(np.float32)).cuda()
               for s, shape in ((0.8, (B, nq, hd)), (1.0, (B, nkv, hd)), (1.0, (B, nkv, hd))))
    stream = torch.cuda.current_stream().cuda_stream
    ref = torch.empty((B, nq, hd), dtype=torch.float32, device="cuda")
    kp.kvprm_attention(sc.ctx, dev.pool[0].data_ptr(), dev.n_pages, w.block_table, w.seq_lens, B, q.data_ptr(),
                       k.data_ptr(), v.data_ptr(), ref.data_ptr(), stream)
    torch.cuda.synchronize()
    r = ref.cpu().numpy()
    for call in range(2):
        out = torch.full((B, nq, hd), float("nan"), dtype=torch.float32, device="cuda")
        kp.kvprm_attention_noalloc(dev.pool[0].data_ptr(), dev.n_pages, w.block_table, w.seq_lens, nq, nkv, hd,
                                   q.data_ptr(), k.data_ptr(), v.data_ptr(), out.data_ptr(), stream)
        torch.cuda.synchronize()
        got = out.cpu().numpy()
        assert np.isfinite(got).all(), f"call {call}: unwritten outputs"
        err = _rel(got, r)
        print(f"no-alloc call {call}: max rel diff vs kvprm_attention {err:.3e}")
        assert err <= ATTN_RTOL
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
