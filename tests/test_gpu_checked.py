"""The checked build on small and ragged cases.

libacespec_checked.so is the library compiled with -DACES_CHECKED: every
data-dependent shared- and global-memory index of every kernel (row kernels,
resolve, cache, resample, KV compaction) is checked against its array's
bound, and the first index out of range is recorded (site, index, bound)
instead of used.  Nothing traps.  These tests build it (about a minute),
route the package's calls to it, run the small and ragged parity cases, the
path cases and the other entry points, compare with the float64 oracle, and
require the record to stay empty.
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
    from paper_2609_02514_gb300 import build
    build.build(checked=True)
    A.use_checked(True)
    A.checked_violation()  # start from an empty record
    yield A
    A.use_checked(False)


def _dev(inp):
    z = inp["z"]
    zt = torch.from_numpy(z.view(np.int16)).cuda().view(torch.bfloat16) if z.dtype == np.uint16 \
        else torch.from_numpy(z).cuda()
    return zt, torch.from_numpy(inp["q"]).cuda(), torch.from_numpy(inp["xt"]).cuda(), torch.from_numpy(inp["u"]).cuda()


def _verify_all(A, orc, w, inp, exact=False):
    z, q, xt, u = _dev(inp)
    g = A.verify(z, q, xt, u, w.T, w.top_p, w.k, exact=exact)
    F = tuple(min(3, w.V - 1) for _ in range(w.K))
    c = A.cache_build(q, xt, F)
    slot = A.cache_lookup(c["branch_tok"], F, g["accept_len"], g["out_token"])
    rs = A.resample_sparse(g["accept_len"], g["topk_ids"], g["topk_probs"], g["tail_mass"], g["row_status"], q, u)
    torch.cuda.synchronize()
    assert A.checked_violation() is None
    gn = {key: v.cpu().numpy() for key, v in g.items()}
    o = orc.verify(inp["z"], inp["q"], inp["xt"], inp["u"], w.T, w.top_p, w.k)
    parity.compare_verify(inp, gn, o, w.top_p, inp["z"].dtype == np.uint16, w.k)
    obt, obp = orc.cache_build(inp["q"], inp["xt"], F)
    parity.compare_cache(c["branch_tok"].cpu().numpy(), c["branch_prob"].cpu().numpy(), obt, obp)
    np.testing.assert_array_equal(slot.cpu().numpy(),
                                  orc.cache_lookup(c["branch_tok"].cpu().numpy(), F, gn["accept_len"], gn["out_token"]))
    assert rs["token"].shape == (w.B,)


CASES = [
    dict(B=1, K=4, V=32000, dtype="f32", T=1.0, top_p=1.0, k=16),       # the first workload's shape
    dict(B=3, K=2, V=10007, dtype="f32", T=0.7, top_p=0.9, k=37),       # unaligned rows: general path
    dict(B=2, K=3, V=4099, dtype="bf16", T=1.3, top_p=0.95, k=5),       # unaligned bf16 rows
    dict(B=4, K=5, V=8200, dtype="bf16", T=0.6, top_p=0.8, k=64),       # aligned, ragged last tile
    dict(B=2, K=16, V=20000, dtype="f32", T=1.0, top_p=1.0, k=256),     # top_p = 1, largest payload
    dict(B=5, K=1, V=65544, dtype="bf16", T=2.0, top_p=0.99, k=16),     # flat rows: exact fallback
    dict(B=3, K=4, V=128256, dtype="bf16", T=1.0, top_p=0.9, k=32, sigma=3.0, rho=0.5),  # value mode
]


@pytest.mark.parametrize("cfg", CASES, ids=lambda c: f"{c['dtype']}_V{c['V']}_p{c['top_p']}")
def test_no_index_out_of_range(A, orc, cfg):
    cfg = dict(cfg)
    w = gen.make_workload(cfg.pop("B"), cfg.pop("K"), cfg.pop("V"), seed=13, **cfg)
    inp = gen.generate(w)
    _verify_all(A, orc, w, inp)
    _verify_all(A, orc, w, inp, exact=True)


def test_no_index_out_of_range_on_degenerate_rows(A, orc):
    w = gen.make_workload(8, 3, 4096, "f32", T=1.0, top_p=0.9, k=8, seed=21)
    inp = dict(gen.generate(w))
    z, q, xt, u = (inp[key].copy() for key in ("z", "q", "xt", "u"))
    z[0, 1, 17] = np.nan
    z[1, 0, :] = -np.inf
    z[2, 2, 5] = np.inf
    z[3, 0, ::2] = -np.inf
    xt[4, 0] = 4096 + 3
    q[5, 0, xt[5, 0]] = 0.0
    z[7, :, :] = 0.5
    inp.update(z=z, q=q, xt=xt, u=u)
    zt, qt, xtt, ut = _dev(inp)
    A.verify(zt, qt, xtt, ut, w.T, w.top_p, w.k)
    torch.cuda.synchronize()
    assert A.checked_violation() is None


def test_no_index_out_of_range_in_the_edge_kernels(A):
    # KV compaction and the tree mask on a small tree (hits, misses, full accept)
    B, K, H, D, planes, t0 = 4, 3, 2, 64, 2, 8
    F = [2, 2, 1]
    bl = K + 1
    S = t0 + K + sum(F) * bl
    kv = torch.randn(planes, B, H, S, D, device="cuda").to(torch.bfloat16)
    pref = torch.full((B,), t0, dtype=torch.int32, device="cuda")
    al = torch.tensor([0, 1, 3, 2], dtype=torch.int32, device="cuda")
    slot = torch.tensor([1, -1, -2, 4], dtype=torch.int32, device="cuda")
    A.compact_kv(kv, pref, al, slot, K, bl)
    A.tree_mask(F, bl)
    torch.cuda.synchronize()
    assert A.checked_violation() is None
