"""Failure detection on the host side of the GPU path, in forms that fault and hang nothing: an
allocation budget that makes the library's allocations fail as if the device were full, an
injected CUDA failure reported by a scoring call, and a bounded device wait that runs out because
the flag it waits for is never set.  After each failure the context scores correctly again."""
import numpy as np
import pytest

import kvsynth as ks
from tests.gpu_util import compare, make_scorer, require_gpu

pytestmark = pytest.mark.gpu


@pytest.fixture
def tiny():
    require_gpu()
    t = ks.Tables.make(0.2)
    w = ks.distinct("fail", ks.ARCH_TINY, 301, [0, 40, 128, 77], gain_std=0.2)
    dev = ks.DeviceInputs(w, t)
    yield w, t, dev


def _scores_ok(sc, w, t, dev):
    r = sc.score(dev.pool, w.block_table, w.seq_lens)
    compare(w, t, gpu_rewards=r.astype(np.float64), label="after the failure")
    return r


def test_allocation_budget(tiny):
    import paper_2607_09153_gb300 as kp
    torch = require_gpu()
    w, t, dev = tiny
    try:
        kp.kvprm_debug_set_alloc_limit(1 << 16)   # far below a context's workspace
        with pytest.raises(kp.KvprmError) as e:
            make_scorer(dev, w.n_candidates, w.max_blocks)
        assert e.value.code == kp.KVPRM_ENOMEM
        kp.kvprm_debug_set_alloc_limit(-1)
        sc = make_scorer(dev, w.n_candidates, w.max_blocks)
        r0 = _scores_ok(sc, w, t, dev)
        # the host-cache call must grow its device pool: refused under a zero budget, context intact
        kp.kvprm_debug_set_alloc_limit(0)
        host_pool = dev.pool.cpu().pin_memory()
        st = torch.cuda.current_stream().cuda_stream
        with pytest.raises(kp.KvprmError) as e:
            kp.kvprm_score_host(sc.ctx, host_pool.data_ptr(), dev.n_pages, w.block_table, w.seq_lens,
                                w.n_candidates, st)
        assert e.value.code == kp.KVPRM_ENOMEM
        assert "budget" in str(e.value)
        assert np.array_equal(sc.score(dev.pool, w.block_table, w.seq_lens), r0)
        kp.kvprm_debug_set_alloc_limit(-1)
        r1 = kp.kvprm_score_host(sc.ctx, host_pool.data_ptr(), dev.n_pages, w.block_table, w.seq_lens,
                                 w.n_candidates, st)
        assert np.array_equal(r1, r0)
        sc.close()
    finally:
        kp.kvprm_debug_set_alloc_limit(-1)


def test_injected_cuda_error(tiny):
    import paper_2607_09153_gb300 as kp
    w, t, dev = tiny
    sc = make_scorer(dev, w.n_candidates, w.max_blocks)
    r0 = _scores_ok(sc, w, t, dev)
    kp.kvprm_debug_inject_error(sc.ctx, 1)
    with pytest.raises(kp.KvprmError) as e:
        sc.score(dev.pool, w.block_table, w.seq_lens)
    assert e.value.code == kp.KVPRM_ECUDA and "injected" in str(e.value)
    kp.kvprm_check_device(sc.ctx)   # nothing ran, nothing timed out
    assert np.array_equal(sc.score(dev.pool, w.block_table, w.seq_lens), r0)
    sc.close()


def test_bounded_wait_gives_up(tiny):
    import paper_2607_09153_gb300 as kp
    torch = require_gpu()
    w, t, dev = tiny
    sc = make_scorer(dev, w.n_candidates, w.max_blocks)
    r0 = _scores_ok(sc, w, t, dev)
    st = torch.cuda.current_stream().cuda_stream
    kp.kvprm_debug_wait_probe(sc.ctx, 2000, st)   # 2 ms on a flag that nothing sets
    with pytest.raises(kp.KvprmError) as e:
        kp.kvprm_check_device(sc.ctx)
    assert e.value.code == kp.KVPRM_ETIMEOUT and "code 9" in str(e.value)
    kp.kvprm_check_device(sc.ctx)   # the error word was cleared
    # a blocking call that follows a timed-out wait reports it, then the context scores again
    kp.kvprm_debug_wait_probe(sc.ctx, 1000, st)
    with pytest.raises(kp.KvprmError) as e:
        sc.score(dev.pool, w.block_table, w.seq_lens)
    assert e.value.code == kp.KVPRM_ETIMEOUT
    assert np.array_equal(sc.score(dev.pool, w.block_table, w.seq_lens), r0)
    with pytest.raises(kp.KvprmError):
        kp.kvprm_debug_wait_probe(sc.ctx, 0, st)
    sc.close()
