"""Full-size parity: each benchmark workload at its full size, scored on the GPU
for the whole batch through the same graph-replayed launch sequence bench.py
times; the oracle (exact mode) scores sampled candidates one by one and every
sampled candidate's P(+) and per-layer attention outputs are compared."""
import numpy as np
import pytest

import kvsynth as ks
from tests.gpu_util import compare, run_gpu

pytestmark = pytest.mark.gpu


def _sample(w):
    L = w.seq_lens
    ids = {0, w.n_candidates - 1, int(np.argmin(L)), int(np.argmax(L))}
    return sorted(ids)


@pytest.mark.parametrize("name", ["qwen1p5b_b16_l2048", "beam7b_b64_p4096_s512", "long8b_b8_l32768",
                                  "mcts7b_b256_d4"])
def test_full_size_sampled(name):
    t = ks.Tables.make()
    w = ks.make_workload(name)
    r, attn, dev, sc = run_gpu(w, t)
    assert np.isfinite(r).all() and (r > 0).all() and (r < 1).all()
    ids = _sample(w)
    compare(w, t, cand_ids=ids, gpu_rewards=r, gpu_attn=attn, label=f"{name} sampled {ids}")
    sc.close()
    del dev
