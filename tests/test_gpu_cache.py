"""Branch cache (Sec. III-C) at large fan-outs, against the float64 oracle.

Fan-outs above 8 take the one-pass path: the union of the per-thread top-8
lists, sorted in shared memory, holds the F_d largest whenever no thread
dropped an id above the F_d-th entry.  Otherwise the kernel repeats its pass
eight maxima at a time.  Both must give the oracle's branches bit for bit.
"""
import dataclasses

import numpy as np
import pytest

import gen
from tests import parity

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def A():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_02514_gb300 as A
    A.load()
    return A


def _check(A, orc, q, xt, F):
    c = A.cache_build(torch.from_numpy(q).cuda(), torch.from_numpy(xt).cuda(), F)
    torch.cuda.synchronize()
    gbt, gbp = c["branch_tok"].cpu().numpy(), c["branch_prob"].cpu().numpy()
    obt, obp = orc.cache_build(q, xt, F)
    parity.compare_cache(gbt, gbp, obt, obp)
    return gbt


@pytest.mark.parametrize("F", [[64] * 16, [9, 17, 33, 64, 128, 256, 8, 4, 2, 1, 0, 65, 100, 12, 40, 24]],
                         ids=["F64", "mixed"])
def test_large_fanouts_on_the_benchmark_rows(A, orc, F):
    w = dataclasses.replace(gen.WORKLOADS["b256_k16_v256000_bf16"], B=3)
    inp = gen.generate(w)
    gbt = _check(A, orc, inp["q"], inp["xt"], F)
    assert (gbt >= 0).mean() > 0.99  # the draft support holds hundreds of ids


def test_one_thread_holding_more_than_eight_falls_back_to_repeated_passes(A, orc):
    # 40 large q values in the chunks of one thread (ids 4 * (256 m) + e):
    # its list keeps 8 of them, so the union cannot prove the top 32
    V, K = 32768, 2
    rng = np.random.default_rng(71)
    q = rng.random((1, K, V)).astype(np.float32) * 1e-6
    ids = np.array([4 * 256 * m + e for m in range(10) for e in range(4)])
    q[0, :, ids] = rng.uniform(0.5, 1.0, size=(len(ids), K)).astype(np.float32)
    q /= q.sum(-1, keepdims=True)
    xt = np.array([[5, 7]], np.int32)
    _check(A, orc, q.astype(np.float32), xt, [32, 40])


def test_fanout_at_the_limit_on_dense_rows(A, orc):
    V, K = 32000, 2
    rng = np.random.default_rng(72)
    q = rng.random((2, K, V))
    q = (q / q.sum(-1, keepdims=True)).astype(np.float32)
    xt = rng.integers(0, V, size=(2, K)).astype(np.int32)
    _check(A, orc, q, xt, [1024, 1000])
