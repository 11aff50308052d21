"""Parity with draft distributions of dense support.

The generator's draft sampler cuts q below 1e-4 of its largest weight, so q
has support on a few percent of the vocabulary.  These tests build q from
the generator's draft logits in two other ways and compare the CUDA path
with the float64 oracle on the result:
  * the reading of the survey table: q = the same temperature and top-p
    warp the target goes through (the oracle's warp, Sec. II-A), cast to
    float32;
  * q = softmax(zd / T) with no cut (top_p = 1): every id has q > 0.
The draft tokens are redrawn from each q by inverse CDF.  Shapes: the
32000-id float32 workload and the 256000-id bfloat16 workload, a few
sequences each.
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


def _with_q(orc, w, q_top_p, seed):
    inp = dict(gen.generate_sequences(w, range(w.B), draft_logits=True))
    p = orc.warp(inp.pop("zd"), w.T, q_top_p)[0][:, : w.K]
    q = (p / p.sum(-1, keepdims=True)).astype(np.float32)
    rng = np.random.default_rng(seed)
    xt = np.empty((w.B, w.K), np.int32)
    for b in range(w.B):
        for i in range(w.K):
            c = np.cumsum(q[b, i], dtype=np.float64)
            j = min(int(np.searchsorted(c, rng.random() * c[-1], side="right")), w.V - 1)
            while q[b, i, j] <= 0.0:
                j -= 1
            xt[b, i] = j
    inp["q"], inp["xt"] = q, xt
    return inp


def _dev(inp):
    z = inp["z"]
    zt = torch.from_numpy(z.view(np.int16)).cuda().view(torch.bfloat16) if z.dtype == np.uint16 \
        else torch.from_numpy(z).cuda()
    return zt, torch.from_numpy(inp["q"]).cuda(), torch.from_numpy(inp["xt"]).cuda(), torch.from_numpy(inp["u"]).cuda()


@pytest.mark.parametrize("name,B", [("b16_k8_v32000_f32", 6), ("b256_k16_v256000_bf16", 4)], ids=["v32000", "v256000"])
@pytest.mark.parametrize("kind", ["nucleus", "dense"])
def test_dense_draft_distribution(A, orc, name, B, kind):
    w = dataclasses.replace(gen.WORKLOADS[name], B=B)
    inp = _with_q(orc, w, w.top_p if kind == "nucleus" else 1.0, seed=61)
    if kind == "dense":
        assert (inp["q"] > 0).mean() > 0.99
    z, q, xt, u = _dev(inp)
    g = A.verify(z, q, xt, u, w.T, w.top_p, w.k)
    c = A.cache_build(q, xt, w.F)
    torch.cuda.synchronize()
    g = {key: v.cpu().numpy() for key, v in g.items()}
    o = orc.verify(inp["z"], inp["q"], inp["xt"], inp["u"], w.T, w.top_p, w.k)
    res = parity.compare_verify(inp, g, o, w.top_p, inp["z"].dtype == np.uint16, w.k)
    assert res["checked_seqs"] >= B - 1, res
    gbt, gbp = c["branch_tok"].cpu().numpy(), c["branch_prob"].cpu().numpy()
    obt, obp = orc.cache_build(inp["q"], inp["xt"], w.F)
    parity.compare_cache(gbt, gbp, obt, obp)
    if kind == "dense":  # every branch slot is filled
        assert (gbt >= 0).all()
    slot = A.cache_lookup(c["branch_tok"], w.F, torch.from_numpy(g["accept_len"]).cuda(),
                          torch.from_numpy(g["out_token"]).cuda()).cpu().numpy()
    np.testing.assert_array_equal(slot, orc.cache_lookup(gbt, w.F, g["accept_len"], g["out_token"]))
