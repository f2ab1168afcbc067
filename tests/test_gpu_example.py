"""The usage example of README.md, run as written (random bf16 weights and cache from torch): one
blocking call scores four candidates; candidates whose block tables list the same pages, in any
order, receive the same P(+) (the read-out is a softmax over the cached positions, so their order
does not matter)."""
import numpy as np
import pytest

from tests.gpu_util import require_gpu

pytestmark = pytest.mark.gpu


def readme_example():
    import torch
    from paper_2607_09153_gb300 import Scorer

    L, d, nq, nkv, hd, ff = 2, 256, 4, 2, 64, 1024       # layers, d_model, heads, head_dim, MLP width
    torch.manual_seed(0)
    bf = dict(dtype=torch.bfloat16, device="cuda")
    w = lambda *shape: (0.02 * torch.randn(*shape, device="cuda")).to(torch.bfloat16)  # noqa: E731
    weights = {"embed_verify": w(d), "final_norm": torch.ones(d, **bf), "w_plus": w(d), "w_minus": w(d),
               "layers": [{"attn_norm": torch.ones(d, **bf), "w_qkv": w((nq + 2 * nkv) * hd, d), "w_o": w(d, nq * hd),
                           "mlp_norm": torch.ones(d, **bf), "w_gate_up": w(2 * ff, d), "w_down": w(d, ff)}
                          for _ in range(L)]}
    scorer = Scorer(L, d, nq, nkv, hd, ff, weights, max_candidates=4, max_blocks_per_seq=8)
    kv = torch.randn(L, 32, 2, nkv, 16, hd, **bf)      # per layer 32 pages of 16 tokens: [K, V][head][token][dim]
    block_table = np.arange(32, dtype=np.int32).reshape(4, 8)   # candidate b reads pages 8 b .. 8 b + 7
    seq_lens = np.array([128, 128, 100, 5], dtype=np.int32)      # cached tokens per candidate
    p_plus = scorer.score(kv, block_table, seq_lens)             # numpy float32 [4]
    return scorer, kv, block_table, seq_lens, p_plus


def test_readme_example():
    require_gpu()
    scorer, kv, bt, lens, p = readme_example()
    assert p.shape == (4,) and np.all((p > 0) & (p < 1)), p
    # candidates 1 and 2 read candidate 0's pages, candidate 2 in reverse order
    bt2 = bt.copy()
    bt2[1] = bt[0]
    bt2[2] = bt[0][::-1]
    lens2 = np.full(4, 128, np.int32)
    p2 = scorer.score(kv, bt2, lens2)
    assert abs(p2[0] - p[0]) < 1e-6 and abs(p2[1] - p2[0]) < 1e-6 and abs(p2[2] - p2[0]) < 1e-5, (p, p2)
    # the same cache held in host memory (pinned, then pageable): the same rewards, bit for bit
    assert np.array_equal(scorer.score_host(kv.cpu().pin_memory(), bt, lens), p)
    assert np.array_equal(scorer.score_host(kv.cpu(), bt, lens), p)
    with pytest.raises(ValueError):
        scorer.score_host(kv, bt, lens)
    scorer.close()
