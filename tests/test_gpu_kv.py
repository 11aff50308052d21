"""aces_compact_kv (COMPACT_KV / ROLLBACK_KV of Alg. 1) against the oracle's
plain slice copies: the whole KV array and the new lengths must match bit
for bit, for hits (with and without overlapping source and destination),
full accepts, misses and out-of-range trees."""
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


def _case(seed, planes, B, H, S, D, K, L, dtype):
    rng = np.random.default_rng(seed)
    if dtype == "bf16":
        kv = rng.integers(0, 1 << 16, size=(planes, B, H, S, D), dtype=np.uint16)
    else:
        kv = rng.standard_normal((planes, B, H, S, D)).astype(np.float32)
    t = rng.integers(0, S // 2, size=B).astype(np.int32)
    al = rng.integers(0, K + 1, size=B).astype(np.int32)
    n_slots = 3 * K
    slot = rng.integers(-2, n_slots, size=B).astype(np.int32)
    slot[al == K] = -2
    t[0], al[0], slot[0] = 3, K - 1, 0          # distance 1: overlapping move
    t[1], al[1], slot[1] = S - K - 1, 0, 2      # tree passes the end
    al[2], slot[2] = 1, -1                      # a miss
    al[3], slot[3] = K, -2                      # the whole chain accepted
    return kv, t, al, slot


@pytest.mark.parametrize("dtype,D", [("bf16", 64), ("bf16", 128), ("f32", 36)])
def test_compact_kv_matches_oracle(A, orc, dtype, D):
    planes, B, H, S, K, L = 6, 48, 4, 160, 8, 5
    kv, t, al, slot = _case(61, planes, B, H, S, D, K, L, dtype)
    want, want_len = orc.compact_kv(kv, t, al, slot, K, L)
    if dtype == "bf16":
        g = torch.from_numpy(kv.view(np.int16)).cuda().view(torch.bfloat16)
    else:
        g = torch.from_numpy(kv).cuda()
    n = A.compact_kv(g, *(torch.from_numpy(x).cuda() for x in (t, al, slot)), K, L)
    torch.cuda.synchronize()
    got = g.view(torch.int16).cpu().numpy().view(np.uint16) if dtype == "bf16" else g.cpu().numpy()
    np.testing.assert_array_equal(n.cpu().numpy(), want_len)
    np.testing.assert_array_equal(got, want)
    assert (want_len == -1).any() and (slot >= 0).any() and (slot == -1).any() and (slot == -2).any()
