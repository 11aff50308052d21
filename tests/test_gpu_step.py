"""aces_cloud_step: verification and cache build of one batch in one call.

The cache build runs on the library's own stream, forked from the caller's
stream and joined back to it.  Its results must be bit-identical to
aces_verify followed by aces_cache_build, and the fork and join must order
it after the caller's earlier work and before the caller's later work: the
inputs are written on a fresh stream right before the call and the outputs
copied on that stream right after it.
"""
import numpy as np
import pytest

import gen

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def A():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_02514_gb300 as A
    A.load()
    return A


@pytest.mark.parametrize("name", ["b16_k8_v32000_f32", "b64_k8_v152064_bf16", "b1_k4_v32000_f32"])
def test_cloud_step_equals_the_separate_calls(A, name):
    w = gen.WORKLOADS[name]
    inp = gen.generate(w)
    z = torch.from_numpy(inp["z"].view(np.int16)).cuda().view(torch.bfloat16) if w.dtype == "bf16" \
        else torch.from_numpy(inp["z"]).cuda()
    q, xt, u = (torch.from_numpy(inp[key]).cuda() for key in ("q", "xt", "u"))
    ref = dict(A.verify(z, q, xt, u, w.T, w.top_p, w.k))
    ref.update(A.cache_build(q, xt, w.F))
    torch.cuda.synchronize()

    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        # inputs written on the caller's stream just before the call
        z2, q2, xt2, u2 = (t.clone() for t in (torch.zeros_like(z), torch.zeros_like(q),
                                                torch.zeros_like(xt), torch.zeros_like(u)))
        for dst, src in ((z2, z), (q2, q), (xt2, xt), (u2, u)):
            dst.copy_(src, non_blocking=True)
        got = A.cloud_step(z2, q2, xt2, u2, w.T, w.top_p, w.k, w.F)
        # outputs read on the caller's stream just after it
        got = {key: v.clone() for key, v in got.items()}
    torch.cuda.synchronize()
    assert set(got) == set(ref)
    for key in ref:
        assert torch.equal(got[key], ref[key]), key
