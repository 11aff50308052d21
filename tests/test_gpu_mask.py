"""aces_tree_mask against the oracle's parent-pointer walk: every bit of the
packed mask and every depth must match."""
import numpy as np
import pytest

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def A():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_02514_gb300 as A
    A.load()
    return A


@pytest.mark.parametrize("F,L", [([1, 1, 0], 2), ([4] * 16, 17), ([6, 5, 5, 5, 5, 4, 4, 4, 4, 4, 3, 3, 3, 3, 3, 3], 1),
                                 ([0, 0, 0, 0], 3), ([31, 0, 2], 7)])
def test_tree_mask_matches_oracle(A, orc, F, L):
    mask, depth = A.tree_mask(F, L)
    torch.cuda.synchronize()
    want, wdepth = orc.tree_mask(F, len(F), L)
    n = want.shape[0]
    words = mask.cpu().numpy().view(np.uint32)
    bits = ((words[:, :, None] >> np.arange(32, dtype=np.uint32)) & 1).astype(bool).reshape(n, -1)
    assert not bits[:, n:].any()
    np.testing.assert_array_equal(bits[:, :n], want)
    np.testing.assert_array_equal(depth.cpu().numpy(), wdepth)
