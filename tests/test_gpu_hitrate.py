"""Cache hit rate of the GPU pipeline (verify + cache build + lookup) for the
three tree shapes of the paper's ablation (Sec. V, Table 2): a single chain
(no branches), a uniform split of the branch budget and the geometric decay
of Sec. IV-C from aces_branch_alloc.

The oracle gives each sequence's exact hit probability given its drafted
chain (orc_hit_prob; pinned against a simulation of the protocol), so the
GPU's empirical hit rate over many uniform draws must match the mean of
those probabilities within 5 standard deviations.  The expected ordering
single < uniform < geometric is checked on the oracle's values.
"""
import numpy as np
import pytest

import gen

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

B, K, V, B_ALLOC = 4096, 8, 4000, 16
DRAWS = 4


@pytest.fixture(scope="module")
def A():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_02514_gb300 as A
    A.load()
    return A


@pytest.fixture(scope="module")
def setup(A, orc):
    w = gen.make_workload(B, K, V, "f32", rho=0.97, T=0.6, top_p=0.9, k=0, seed=93)
    inp = gen.generate(w, workers=8)
    ov = orc.verify(inp["z"], inp["q"], inp["xt"], inp["u"], w.T, w.top_p, 0)
    alpha = float(np.minimum(1.0, ov["ratio"]).mean())
    shapes = {"single": [0] * K, "uniform": [B_ALLOC // K] * K,
              "geometric": A.branch_alloc(B_ALLOC, K, alpha, 1.0)}
    rng = np.random.default_rng(94)
    draws = [((rng.integers(1, 1 << 24, size=(B, K + 1))) / float(1 << 24)).astype(np.float32)
             for _ in range(DRAWS)]
    return w, inp, shapes, draws


def _empirical(A, w, inp, F, draws):
    z = torch.from_numpy(inp["z"]).cuda()
    q = torch.from_numpy(inp["q"]).cuda()
    xt = torch.from_numpy(inp["xt"]).cuda()
    cache = A.cache_build(q, xt, F)
    hits = 0
    for u in draws:
        out = A.verify(z, q, xt, torch.from_numpy(u).cuda(), w.T, w.top_p, 0)
        slot = A.cache_lookup(cache["branch_tok"], F, out["accept_len"], out["out_token"])
        hits += int(((slot >= 0) | (slot == -2)).sum().item())
    return hits / (len(draws) * w.B)


def test_hit_rates_of_the_three_shapes(A, orc, setup):
    w, inp, shapes, draws = setup
    pred = {}
    for name, F in shapes.items():
        assert sum(F) == (0 if name == "single" else B_ALLOC)
        bt, _ = orc.cache_build(inp["q"], inp["xt"], F)
        hp, pp = orc.hit_prob(inp["z"], inp["q"], inp["xt"], w.T, w.top_p, bt, F)
        emp = _empirical(A, w, inp, F, draws)
        sd = np.sqrt(np.sum(hp * (1.0 - hp)) / DRAWS) / w.B
        assert abs(emp - hp.mean()) < 5 * sd + 1e-4, (name, emp, hp.mean(), sd)
        pred[name] = hp.mean()
    assert pred["single"] < pred["uniform"] < pred["geometric"], pred
