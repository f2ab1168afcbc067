"""GPU parity on seeded random sharing structures: forests of cached segments whose leaves are the
candidates, so that one call mixes private pages, shared runs of 2 to 8 candidates on the
persistent kernel (whole stages, ragged last stages and the paired-page path), groups of 6 or more
candidates on the tensor cores, partial pages copied per child, and empty caches; several head
groupings (G = 1, 2, 6, 7, 16) and head dims, a depth-2 readout and a scorer adapter.  Every
candidate's P(+) and every layer's attention output are compared with the oracle at the tolerances
every parity test uses (1e-3 on P(+), 2e-3 relative on the attention output)."""
import numpy as np
import pytest

import kvsynth as ks
from tests.gpu_util import compare, run_gpu

pytestmark = pytest.mark.gpu


def random_forest(seed: int, n_roots: int, depth: int, branching: int, lo: int, hi: int, n_empty: int = 0,
                  max_leaves: int = 96) -> list:
    """Leaves of `n_roots` random trees (each node has 1..branching children, a branch stops early
    with probability 1/4), edges of uniform integer length in [lo, hi]; plus `n_empty` empty caches."""
    rng = np.random.default_rng(seed)
    paths = []
    seg = 0

    def grow(prefix, d):
        nonlocal seg
        if len(paths) >= max_leaves:
            return
        if d == depth or (d > 0 and rng.random() < 0.25):
            paths.append(prefix)
            return
        for _ in range(int(rng.integers(1, branching + 1))):
            n = int(rng.integers(lo, hi + 1))
            grow(prefix + [(seg, n)], d + 1)
            seg += 1

    for _ in range(n_roots):
        grow([], 0)
    paths += [[] for _ in range(n_empty)]
    order = rng.permutation(len(paths))   # candidates in no particular tree order
    return [paths[i] for i in order]


CASES = [
    # (label, arch, seed, roots, depth, branching, lo, hi, empty, readout depth)
    ("G7 hd128 forest", ks.Arch(1, 256, 14, 2, 128, 256), 301, 2, 3, 6, 40, 400, 2, 1),
    ("G6 hd128 two layers", ks.Arch(2, 256, 12, 2, 128, 256), 302, 3, 3, 4, 16, 300, 1, 1),
    ("G2 hd64 tiny-shaped", ks.Arch(2, 256, 4, 2, 64, 1024), 303, 2, 4, 4, 1, 200, 3, 1),
    ("G16 hd64 two MMA row groups", ks.Arch(1, 512, 16, 1, 64, 512), 304, 2, 3, 5, 8, 250, 1, 1),
    ("G1 hd64", ks.Arch(1, 256, 4, 4, 64, 256), 305, 3, 3, 3, 20, 300, 0, 1),
    ("G7 hd128 wide fan-out", ks.Arch(1, 256, 14, 2, 128, 256), 306, 1, 2, 10, 100, 700, 0, 1),
    ("G7 hd128 depth-2 readout", ks.Arch(1, 256, 14, 2, 128, 256), 307, 2, 3, 5, 30, 300, 1, 2),
]


@pytest.mark.parametrize("case", CASES, ids=[c[0] for c in CASES])
def test_random_forest(case):
    label, arch, seed, roots, depth, branching, lo, hi, empty, k = case
    paths = random_forest(seed, roots, depth, branching, lo, hi, empty)
    if k > 1:
        paths = paths[:256 // k]
    w = ks.workload_from_segments(label.replace(" ", "_"), arch, seed, paths, gain_std=0.2)
    assert w.n_candidates * k <= 256
    t = ks.Tables.make(0.2)
    r, attn, _, _ = run_gpu(w, t, depth=k)
    assert np.isfinite(r).all()
    compare(w, t, gpu_rewards=r, gpu_attn=attn, label=f"{label}: {w.n_candidates} candidates, "
            f"{w.n_pages} pages", depth=k)


def test_random_forest_adapter():
    """The same kind of forest through a scorer with an adapter of rank 64 on every projection."""
    import dataclasses
    arch = dataclasses.replace(ks.Arch(2, 256, 12, 2, 128, 512), lora_rank=64)
    paths = random_forest(308, 2, 3, 4, 16, 250, 1)
    w = ks.workload_from_segments("random_adapter", arch, 308, paths, gain_std=0.2)
    t = ks.Tables.make(0.2)
    r, attn, _, _ = run_gpu(w, t)
    compare(w, t, gpu_rewards=r, gpu_attn=attn, label=f"adapter forest: {w.n_candidates} candidates")
