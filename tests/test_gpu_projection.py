"""The tcgen05 projection GEMM alone (kvprm_projection) against an fp64 matmul
of the same bf16 inputs, over shapes that exercise one vs many K tiles per
CTA, ring wrap-around, and batch padding."""
import numpy as np
import pytest

import kvsynth as ks
from tests.gpu_util import make_scorer, require_gpu

pytestmark = pytest.mark.gpu

SHAPES = [  # (M, K, n)
    (256, 1024, 4),        # one K tile per CTA
    (2048, 1536, 16),      # 2 K tiles per CTA
    (1536, 8960, 16),      # 6 K tiles per CTA (= ring depth)
    (17920, 1536, 16),     # 12 K tiles per CTA (ring wraps)
    (38912, 1024, 16),     # 16 K tiles per CTA, one split
    (4608, 3584, 64),
    (3584, 18944, 64),
    (37888, 3584, 256),
    (512, 256, 33),
]


@pytest.fixture(scope="module")
def ctx():
    require_gpu()
    arch = ks.Arch(1, 3584, 28, 4, 128, 18944)    # sizes the context's split-K partial buffer
    t = ks.Tables.make()
    w = ks.distinct("proj", arch, 1, [16])
    dev = ks.DeviceInputs(w, t)
    sc = make_scorer(dev, 256, 4)
    yield sc
    sc.close()


@pytest.mark.parametrize("M,K,n", SHAPES)
def test_projection(ctx, M, K, n):
    torch = require_gpu()
    import paper_2607_09153_gb300 as kp
    rng = np.random.default_rng(M + K + n)
    Wb = ks.f64_to_bf16_bits(rng.normal(0, 0.02, (M, K)))
    Xb = ks.f64_to_bf16_bits(rng.normal(0, 1, (n, K)))
    W = torch.from_numpy(Wb.view(np.int16)).cuda()
    X = torch.from_numpy(Xb.view(np.int16)).cuda()
    Y = torch.full((n, M), float("nan"), dtype=torch.float32, device="cuda")
    kp.kvprm_projection(ctx.ctx, W.data_ptr(), M, K, X.data_ptr(), n, Y.data_ptr(),
                        torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    got = Y.cpu().numpy().astype(np.float64)
    ref = ks.bf16_bits_to_f64(Xb) @ ks.bf16_bits_to_f64(Wb).T
    err = np.abs(got - ref).max() / np.abs(ref).max()
    print(f"projection M={M} K={K} n={n}: rel err {err:.3e}")
    assert np.isfinite(got).all()
    assert err < 1e-5
