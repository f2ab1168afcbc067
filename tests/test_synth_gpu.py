"""The device generator fills exactly the bits the host generator does."""
import numpy as np
import pytest

import kvsynth as ks

pytestmark = pytest.mark.gpu


def test_device_fill_matches_host():
    import torch
    if not torch.cuda.is_available():
        pytest.fail("no CUDA device")
    t = ks.Tables.make(0.2)
    w = ks.mcts_tree("fill", ks.ARCH_TINY, 9, branching=2, depth=2, lo=3, hi=40, gain_std=0.2)
    dev = ks.DeviceInputs(w, t)
    host_pool = ks.host_kv_pool(w, t)
    assert np.array_equal(dev.pool.cpu().view(torch.int16).numpy().view(np.uint16), host_pool)
    for l in range(w.arch.n_layers):
        for kind, tensor in dev.layers[l].items():
            ref = ks.host_weight(w.arch, kind, l, w.seed, t)
            assert np.array_equal(tensor.cpu().view(torch.int16).numpy().view(np.uint16), ref), (l, kind)
    for kind, tensor in dev.top.items():
        ref = ks.host_weight(w.arch, kind, 0, w.seed, t)
        assert np.array_equal(tensor.cpu().view(torch.int16).numpy().view(np.uint16), ref), kind
