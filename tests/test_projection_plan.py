"""The projection GEMM's launch plan (kvprm_plan_projection, host only) over the workloads' shapes,
batch paddings and adapter ranks: the invariants the kernel relies on (shared memory within the
configured limit, split-K ranks dividing the batch columns, the K tiles covered, tensor memory for
every tile's accumulator, two-tile plans in one wave)."""
import pytest

import kvsynth as ks
import paper_2607_09153_gb300 as kp

SMS = 152
MAX_SMEM = 200 * 1024


def _shapes(a, rank=0):
    kx = lambda K: 64 * ((K + 63) // 64) + rank if rank else K  # noqa: E731  (adapter K extension)
    return [("qkv", a.qkv_rows, kx(a.d_model), False), ("o", a.d_model, kx(a.n_q_heads * a.head_dim), False),
            ("gate_up", a.d_ff, kx(a.d_model), True), ("down", a.d_model, kx(a.d_ff), False)]


@pytest.mark.parametrize("arch", [ks.ARCH_TINY, ks.ARCH_1P5B, ks.ARCH_7B, ks.ARCH_8B])
@pytest.mark.parametrize("n_pad", [16, 32, 48, 64, 96, 128, 192, 208, 256])
@pytest.mark.parametrize("rank", [0, 64, 256])
def test_projection_plan_invariants(arch, n_pad, rank):
    for name, M, K, gu in _shapes(arch, rank):
        p = kp.kvprm_plan_projection(M, K, n_pad, SMS, True, gu)
        tag = f"{name} M={M} K={K} n_pad={n_pad}"
        assert p["smem_bytes"] <= MAX_SMEM, tag
        assert p["cluster"] in (1, 2, 4, 8, 16) and n_pad % p["cluster"] == 0, tag
        assert p["tiles_per_cta"] in (1, 2), tag
        assert 2 <= p["stages"] <= 8, tag
        k_tiles = (K + 63) // 64
        assert p["k_tiles"] == k_tiles, tag
        assert p["kt_per_split"] == (k_tiles + p["cluster"] - 1) // p["cluster"], tag
        assert p["m_tiles"] == ((M + 63) // 64 if gu else (M + 127) // 128), tag
        need = 2 * n_pad if 2 * n_pad <= 256 else n_pad   # hi and lo halves side by side, else summed
        cols = p["tmem_cols"]
        assert cols <= 512 and cols & (cols - 1) == 0 and cols // p["tiles_per_cta"] >= need, tag
        assert p["threads"] == (256 if n_pad >= 64 else 128), tag   # eight warps on the large-batch image
        if p["tiles_per_cta"] == 2:   # two m-tiles per CTA: the grid fits the SMs at once
            grid = (p["m_tiles"] + 1) // 2 * p["cluster"]
            assert grid <= SMS and p["m_tiles"] % 2 == 0, tag


def test_projection_plan_large_batch_choices():
    """The plans the 7B scorer at 256 candidates runs: gate/up and down take two m-tiles per CTA."""
    a = ks.ARCH_7B
    gu = kp.kvprm_plan_projection(a.d_ff, a.d_model, 256, SMS, True, True)
    down = kp.kvprm_plan_projection(a.d_model, a.d_ff, 256, SMS, True, False)
    qkv = kp.kvprm_plan_projection(a.qkv_rows, a.d_model, 256, SMS, True, False)
    assert (gu["tiles_per_cta"], gu["cluster"]) == (2, 1)
    assert (down["tiles_per_cta"], down["cluster"]) == (2, 8)
    assert (qkv["tiles_per_cta"], qkv["cluster"]) == (1, 4)
    assert gu["threads"] == down["threads"] == qkv["threads"] == 256


def test_projection_plan_errors():
    for args in [(0, 64, 16, SMS), (64, 0, 16, SMS), (64, 64, 24, SMS), (64, 64, 16, 0)]:
        with pytest.raises(kp.KvprmError):
            kp.kvprm_plan_projection(*args)


def test_projection_plan_beyond_context_batch():
    # a context holds at most 256 candidates: larger padded batches are not plannable
    for n_pad in (272, 512, 1024):
        with pytest.raises(kp.KvprmError) as e:
            kp.kvprm_plan_projection(4608, 3584, n_pad, SMS)
        assert e.value.code == kp.KVPRM_EUNSUPPORTED
    assert kp.kvprm_plan_projection(4608, 3584, 256, SMS)["tmem_cols"] <= 512


@pytest.mark.parametrize("arch", [ks.ARCH_TINY, ks.ARCH_1P5B, ks.ARCH_7B, ks.ARCH_8B])
@pytest.mark.parametrize("n_pad", [16, 32, 64, 96, 128, 256])
def test_projection_plan_cluster_placement(arch, n_pad):
    """Whole clusters are placed on one GPC: where two CTAs share an SM, a split-K grid keeps within
    7/8 of the CTA slots, so that it is placed in one wave beside the preceding kernel's CTAs (the
    7B QKV projection at B = 64 takes clusters of 4, 144 CTAs, not 36 clusters of 8 = 288 of 304)."""
    for name, M, K, gu in _shapes(arch):
        p = kp.kvprm_plan_projection(M, K, n_pad, SMS, True, gu)
        if p["cluster"] == 1:
            continue
        two_per_sm = p["smem_bytes"] + 1024 <= 228 * 1024 // 2
        ctas = (p["m_tiles"] + p["tiles_per_cta"] - 1) // p["tiles_per_cta"] * p["cluster"]
        assert ctas <= (2 * SMS * 7 // 8 if two_per_sm else SMS), f"{name} n_pad={n_pad}: {ctas} CTAs"
    qkv = kp.kvprm_plan_projection(ks.ARCH_7B.qkv_rows, ks.ARCH_7B.d_model, 64, SMS)
    assert (qkv["cluster"], qkv["m_tiles"]) == (4, 36)
