"""Losslessness of the GPU verification (Sec. II-A, the modified rejection
sampling of Chen et al. that AceSpec's cloud step runs).

With draft tokens drawn from q, the token emitted at each position (the
accepted draft token, or the residual / bonus draw at the first rejection)
follows the warped target distribution p exactly, whatever q is.  These are
the oracle's own statistical pins run on the CUDA path: many sequences share
one set of 16-id target and draft rows, and chi-square tests (p-value > 1e-3,
fixed seeds) compare the emitted tokens with p, computed here from the
library softmax and a brute-force nucleus.  The sequences go through the
library in launches of CHUNK sequences.
"""
import numpy as np
import pytest
from scipy import stats

import gen
from tests import parity
from tests.test_oracle_pins import _batch, _norm, _order, _pq, _softmax

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

CHUNK = 200_000


@pytest.fixture(scope="module")
def A():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_02514_gb300 as A
    A.load()
    return A


def _to_dev(z, bf16):
    if bf16:
        return torch.from_numpy(z.view(np.int16)).cuda().view(torch.bfloat16)
    return torch.from_numpy(z).cuda()


def _verify_many(A, z_rows, q_rows, n, seed, T, top_p, k=0, bf16=False):
    """accept_len, out_token and draft tokens of n sequences sharing the rows
    (z_rows already bf16 bit patterns when bf16)."""
    acc, tok, xts = [], [], []
    zr = gen.bf16_to_f32(z_rows) if bf16 else z_rows
    for c in range(n // CHUNK):
        z, q, xt, u = _batch(zr, q_rows, CHUNK, seed + c)
        if bf16:
            z = np.ascontiguousarray(np.broadcast_to(z_rows, z.shape))
        g = A.verify(_to_dev(z, bf16), torch.from_numpy(q).cuda(), torch.from_numpy(xt).cuda(),
                     torch.from_numpy(u).cuda(), T, top_p, k)
        torch.cuda.synchronize()
        acc.append(g["accept_len"].cpu().numpy())
        tok.append(g["out_token"].cpu().numpy())
        xts.append(xt)
    return np.concatenate(acc), np.concatenate(tok), np.concatenate(xts)


def _nucleus_p(z, T, top_p):
    pi = _softmax(z, T)
    o = _order(z)
    nkeep = z.size if top_p >= 1 else int(np.argmax(np.cumsum(pi[o]) >= top_p)) + 1
    p = np.zeros_like(pi)
    p[o[:nkeep]] = pi[o[:nkeep]] / pi[o[:nkeep]].sum()
    return p


@pytest.mark.parametrize("top_p,bf16", [(1.0, False), (0.7, False), (0.7, True)],
                         ids=["f32_full", "f32_nucleus", "bf16_nucleus"])
def test_gpu_first_emitted_token_is_distributed_as_target(A, top_p, bf16):
    zt, qd, _ = _pq(31)
    T, n = 0.9, 1_000_000
    zrows = np.stack([zt, zt])
    if bf16:
        zrows = gen.f32_to_bf16(zrows)
        zt = gen.bf16_to_f32(zrows)[0].astype(np.float32)
    acc, tok, xt = _verify_many(A, zrows, qd[None], n, 32, T, top_p, 16, bf16)
    emitted = np.where(acc >= 1, xt[:, 0], tok)
    p = _nucleus_p(zt, T, top_p)
    counts = np.bincount(emitted, minlength=zt.size)
    assert counts[p == 0].sum() == 0
    sup = p > 0
    assert stats.chisquare(counts[sup], p[sup] * n).pvalue > 1e-3


def test_gpu_accept_law_is_geometric(A):
    # i.i.d. positions with acceptance alpha = sum_x min(p, q):
    # P(pi = i) = alpha^i (1 - alpha), P(pi = K) = alpha^K (Sec. III-A)
    zt, qd, p = _pq(21)
    K, n = 6, 400_000
    acc, _, _ = _verify_many(A, np.stack([zt] * (K + 1)), np.stack([qd] * K), n, 22, 1.0, 1.0)
    alpha = np.minimum(p, qd.astype(np.float64)).sum()
    counts = np.bincount(acc, minlength=K + 1)
    probs = np.array([alpha ** i * (1 - alpha) for i in range(K)] + [alpha ** K])
    assert stats.chisquare(counts, probs * n).pvalue > 1e-3


def test_gpu_second_and_bonus_tokens_are_distributed_as_target(A):
    rng = np.random.default_rng(41)
    V, n = 16, 1_000_000
    z0, z1, z2 = (rng.normal(0, 1.2, V).astype(np.float32) for _ in range(3))
    q0, q1 = (_norm(np.exp(rng.normal(0, 1.2, V))).astype(np.float32) for _ in range(2))
    acc, tok, xt = _verify_many(A, np.stack([z0, z1, z2]), np.stack([q0, q1]), n, 42, 1.0, 1.0)
    sel = acc >= 1
    second = np.where(acc[sel] >= 2, xt[sel, 1], tok[sel])
    assert stats.chisquare(np.bincount(second, minlength=V), _softmax(z1, 1.0) * sel.sum()).pvalue > 1e-3
    allacc = acc == 2
    counts2 = np.bincount(tok[allacc], minlength=V)
    assert stats.chisquare(counts2, _softmax(z2, 1.0) * allacc.sum()).pvalue > 1e-3


def test_gpu_draws_equal_the_oracle_on_a_subset(A, orc):
    # the same sequences through both sides: bit-exact accept_len and
    # out_token except where the flag rules allow a rounding difference
    zt, qd, _ = _pq(31)
    z, q, xt, u = _batch(np.stack([zt, zt]), qd[None], 4000, 77)
    g = A.verify(torch.from_numpy(z).cuda(), torch.from_numpy(q).cuda(), torch.from_numpy(xt).cuda(),
                 torch.from_numpy(u).cuda(), 0.9, 0.7, 16)
    torch.cuda.synchronize()
    g = {key: v.cpu().numpy() for key, v in g.items()}
    o = orc.verify(z, q, xt, u, 0.9, 0.7, 16)
    inp = {"z": z, "q": q, "xt": xt, "u": u}
    res = parity.compare_verify(inp, g, o, 0.7, False, 16)
    assert res["checked_seqs"] >= 3900
