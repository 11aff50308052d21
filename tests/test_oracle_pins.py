"""Pins of the float64 oracle against facts fixed outside it.

Each test checks the oracle against a closed form from the paper, a library
routine, an invariant or brute force on tiny inputs, chosen so that a dropped
term, a wrong sign, a wrong index or a transposed operand in the oracle fails
at least one of them.  None of these tests touch the GPU.
"""
import itertools

import numpy as np
import pytest
from scipy import special, stats


def _softmax(z, T):
    return special.softmax(np.asarray(z, np.float64) / T)


def _order(z):
    z = np.asarray(z, np.float64)
    return np.lexsort((np.arange(z.size), -z))


def _batch(z_rows, q_rows, n, seed):
    """n sequences that all share the given target rows [K+1,V] and draft rows
    [K,V]; draft tokens drawn from q, uniforms in (0,1)."""
    rng = np.random.default_rng(seed)
    z_rows = np.asarray(z_rows, np.float32)
    q_rows = np.asarray(q_rows, np.float32)
    R, V = z_rows.shape
    K = R - 1
    z = np.ascontiguousarray(np.broadcast_to(z_rows, (n, R, V)))
    q = np.ascontiguousarray(np.broadcast_to(q_rows, (n, K, V)))
    xt = np.empty((n, K), np.int32)
    for i in range(K):
        c = np.cumsum(q_rows[i].astype(np.float64))
        xt[:, i] = np.minimum(np.searchsorted(c, rng.random(n) * c[-1], side="right"), V - 1)
    u = ((rng.integers(1, 1 << 24, size=(n, R))) / float(1 << 24)).astype(np.float32)
    return z, q, xt, u


def _norm(x):
    x = np.asarray(x, np.float64)
    return x / x.sum()


# --------------------------------------------------------------------------
# step 1-2: temperature softmax and nucleus


@pytest.mark.parametrize("T", [0.3, 1.0, 1.7])
def test_top_p_one_is_library_softmax(orc, T):
    rng = np.random.default_rng(1)
    z = rng.normal(0, 3, 50).astype(np.float32)
    out = orc.sparsify(z[None], T, 1.0, 50)
    ref = _softmax(z, T)
    o = _order(z)
    np.testing.assert_array_equal(out["topk_ids"][0], o)
    np.testing.assert_allclose(out["topk_probs"][0], ref[o], rtol=1e-12, atol=0)
    assert abs(out["tail"][0]) < 1e-12


@pytest.mark.parametrize("seed", range(6))
def test_nucleus_is_minimal_max_mass_subset_bruteforce(orc, seed):
    rng = np.random.default_rng(100 + seed)
    V = 9
    z = rng.normal(0, 2, V).astype(np.float32)
    T = float(rng.uniform(0.5, 1.5))
    pi = _softmax(z, T)
    for top_p in (0.3, 0.55, 0.8, 0.95, 0.999):
        best = None
        for c in range(1, V + 1):
            masses = [(sum(pi[list(s)]), s) for s in itertools.combinations(range(V), c)]
            ok = [m for m in masses if m[0] >= top_p]
            if ok:
                best = max(ok)
                break
        mass, subset = best
        out = orc.sparsify(z[None], T, top_p, V)
        n = int(out["n_nuc"][0])
        assert n == len(subset)
        ids = out["topk_ids"][0][:n]
        assert set(ids.tolist()) == set(subset)
        np.testing.assert_allclose(out["topk_probs"][0][:n], pi[ids] / mass, rtol=1e-12)
        assert (out["topk_ids"][0][n:] == -1).all()
        assert (out["topk_probs"][0][n:] == 0).all()


def test_equal_logits_break_ties_by_lower_id(orc):
    z = np.array([1.0, 3.0, 3.0, 0.5, 3.0, 1.0], np.float32)
    out = orc.sparsify(z[None], 1.0, 1.0, 6)
    np.testing.assert_array_equal(out["topk_ids"][0], [1, 2, 4, 0, 5, 3])
    # top_p reached inside the tie: exactly the lowest ids of the tied group are kept
    pi = _softmax(z, 1.0)
    top_p = float(pi[1] + pi[2] - 1e-9)
    out = orc.sparsify(z[None], 1.0, top_p, 6)
    assert out["n_nuc"][0] == 2
    np.testing.assert_array_equal(out["topk_ids"][0][:3], [1, 2, -1])


def test_topk_payload_matches_full_sort(orc):
    rng = np.random.default_rng(7)
    V, k = 4096, 64
    z = rng.normal(0, 3, V).astype(np.float32)
    z[rng.choice(V, 300)] = z[5]   # plenty of exact ties
    out = orc.sparsify(z[None], 0.9, 1.0, k)
    o = _order(z)[:k]
    pi = _softmax(z, 0.9)
    np.testing.assert_array_equal(out["topk_ids"][0], o)
    np.testing.assert_allclose(out["topk_probs"][0], pi[o], rtol=1e-12)
    np.testing.assert_allclose(out["tail"][0], 1.0 - pi[o].sum(), atol=1e-12)


def test_minus_inf_logits_have_zero_mass_and_nan_rows_are_flagged(orc):
    z = np.array([[0.0, -np.inf, 2.0, -np.inf, 1.0],
                  [0.0, np.nan, 1.0, 2.0, 3.0],
                  [-np.inf] * 5,
                  [0.0, np.inf, 1.0, 2.0, 3.0]], np.float32)
    out = orc.sparsify(z, 1.0, 1.0, 5)
    np.testing.assert_array_equal(out["topk_ids"][0], [2, 4, 0, -1, -1])
    np.testing.assert_allclose(out["topk_probs"][0][:3], _softmax([2.0, 1.0, 0.0], 1.0), rtol=1e-12)
    assert list(out["row_status"]) == [0, orc.ROW_NONFINITE, orc.ROW_NONFINITE, orc.ROW_NONFINITE]
    assert (out["topk_ids"][1:] == -1).all()


# --------------------------------------------------------------------------
# steps 3-5: accept test, first rejection, residual, losslessness


def _pq(seed, V=16, T=1.0):
    rng = np.random.default_rng(seed)
    zt = rng.normal(0, 1.5, V).astype(np.float32)
    qd = _norm(np.exp(rng.normal(0, 1.5, V))).astype(np.float32)
    return zt, qd, _softmax(zt, T)


def test_accept_rate_equals_sum_min_p_q(orc):
    zt, qd, p = _pq(11)
    n = 1_000_000
    z, q, xt, u = _batch(np.stack([zt, zt]), qd[None], n, 12)
    out = orc.verify(z, q, xt, u, 1.0, 1.0, 0)
    rate = (out["accept_len"] == 1).mean()
    alpha = np.minimum(p, q[0, 0].astype(np.float64)).sum()
    sd = np.sqrt(alpha * (1 - alpha) / n)
    assert abs(rate - alpha) < 5 * sd, (rate, alpha)


def test_expected_accepted_length_closed_form(orc):
    # Sec. III-A: with i.i.d. acceptance alpha per position, the expected
    # number of accepted tokens per round is (1 - alpha^gamma) / (1 - alpha);
    # it counts emitted tokens capped at gamma, i.e. E[min(pi + 1, gamma)].
    zt, qd, p = _pq(21)
    K, n = 6, 300_000
    z, q, xt, u = _batch(np.stack([zt] * (K + 1)), np.stack([qd] * K), n, 22)
    out = orc.verify(z, q, xt, u, 1.0, 1.0, 0)
    L = np.minimum(out["accept_len"] + 1, K)
    alpha = np.minimum(p, qd.astype(np.float64)).sum()
    expect = (1 - alpha ** K) / (1 - alpha)
    assert abs(L.mean() - expect) < 5 * L.std() / np.sqrt(n), (L.mean(), expect)
    # the whole law of pi is geometric: P(pi = i) = alpha^i (1 - alpha), P(pi = K) = alpha^K
    counts = np.bincount(out["accept_len"], minlength=K + 1)
    probs = np.array([alpha ** i * (1 - alpha) for i in range(K)] + [alpha ** K])
    assert stats.chisquare(counts, probs * n).pvalue > 1e-3


@pytest.mark.parametrize("top_p", [1.0, 0.7])
def test_first_emitted_token_is_distributed_as_target(orc, top_p):
    # Lossless verification (Sec. II-A, Chen et al.): the emitted token
    # follows the (warped) target distribution exactly.
    zt, qd, _ = _pq(31)
    T = 0.9
    n = 1_000_000
    z, q, xt, u = _batch(np.stack([zt, zt]), qd[None], n, 32)
    out = orc.verify(z, q, xt, u, T, top_p, 16)
    tok = np.where(out["accept_len"] >= 1, xt[:, 0], out["out_token"])
    # target distribution from the library softmax and a brute-force nucleus
    pi = _softmax(zt, T)
    o = _order(zt)
    c = np.cumsum(pi[o])
    nkeep = zt.size if top_p >= 1 else int(np.argmax(c >= top_p)) + 1
    p = np.zeros_like(pi)
    p[o[:nkeep]] = pi[o[:nkeep]] / pi[o[:nkeep]].sum()
    counts = np.bincount(tok, minlength=zt.size)
    assert counts[p == 0].sum() == 0
    sup = p > 0
    assert stats.chisquare(counts[sup], p[sup] * n).pvalue > 1e-3


def test_second_emitted_token_is_distributed_as_target(orc):
    rng = np.random.default_rng(41)
    V, n = 16, 1_000_000
    z0 = rng.normal(0, 1.2, V).astype(np.float32)
    z1 = rng.normal(0, 1.2, V).astype(np.float32)
    z2 = rng.normal(0, 1.2, V).astype(np.float32)
    q0 = _norm(np.exp(rng.normal(0, 1.2, V))).astype(np.float32)
    q1 = _norm(np.exp(rng.normal(0, 1.2, V))).astype(np.float32)
    z, q, xt, u = _batch(np.stack([z0, z1, z2]), np.stack([q0, q1]), n, 42)
    out = orc.verify(z, q, xt, u, 1.0, 1.0, 0)
    sel = out["accept_len"] >= 1
    tok = np.where(out["accept_len"][sel] >= 2, xt[sel, 1], out["out_token"][sel])
    p1 = _softmax(z1, 1.0)
    counts = np.bincount(tok, minlength=V)
    assert stats.chisquare(counts, p1 * sel.sum()).pvalue > 1e-3
    # bonus token (both accepted) follows the last target row
    allacc = out["accept_len"] == 2
    counts2 = np.bincount(out["out_token"][allacc], minlength=V)
    assert stats.chisquare(counts2, _softmax(z2, 1.0) * allacc.sum()).pvalue > 1e-3


def test_residual_follows_normalised_positive_part(orc):
    # At a rejection the corrected token is drawn from norm(max(0, p - q)).
    zt, qd, p = _pq(51)
    n = 400_000
    z, q, xt, u = _batch(np.stack([zt, zt]), qd[None], n, 52)
    out = orc.verify(z, q, xt, u, 1.0, 1.0, 0)
    rej = out["accept_len"] == 0
    r = np.maximum(p - qd.astype(np.float64), 0.0)
    r /= r.sum()
    counts = np.bincount(out["out_token"][rej], minlength=zt.size)
    assert counts[r == 0].sum() == 0
    assert stats.chisquare(counts[r > 0], r[r > 0] * rej.sum()).pvalue > 1e-3
    # the rejected draft token is never re-emitted (its residual is zero)
    assert not np.any(out["out_token"][rej] == xt[rej, 0])
    np.testing.assert_allclose(out["res_sum"][rej], np.maximum(p - qd, 0).sum(), rtol=1e-6)


def test_inverse_cdf_uses_vocab_order_and_strict_inequality(orc):
    # bonus draw on a uniform two-token row: u < 1/2 picks id 0, u >= 1/2 id 1
    z = np.zeros((3, 1, 2), np.float32)
    q = np.full((3, 0, 2), 0.5, np.float32)
    xt = np.zeros((3, 0), np.int32)
    u = np.array([[0.25], [0.5], [0.75]], np.float32)
    out = orc.verify(z, q, xt, u, 1.0, 1.0, 0)
    assert list(out["accept_len"]) == [0, 0, 0]
    assert list(out["out_token"]) == [0, 1, 1]


def test_bad_draft_probability_forces_reject(orc):
    z = np.array([[[0.0, 1.0, 2.0], [0.0, 0.0, 0.0]]], np.float32)
    q = np.array([[[0.5, 0.5, 0.0]]], np.float32)
    xt = np.array([[2]], np.int32)                  # drafted an id with q = 0
    u = np.array([[0.01, 0.5]], np.float32)
    out = orc.verify(z, q, xt, u, 1.0, 1.0, 3)
    assert out["accept_len"][0] == 0
    assert out["row_status"][0, 0] & orc.ROW_BAD_Q
    assert out["out_token"][0] == 2                 # residual mass sits where q = 0


def test_residual_reads_draft_only_where_target_is_positive(orc):
    # nucleus of z = [5, 0, 0] at top_p = 0.5 is {0}, so p = (1, 0, 0).  The
    # draft token 1 has p = 0 and is rejected; r = max(0, p - q) = (0.5, 0, 0)
    # for any valid q, so token 0 is emitted.  A negative q at id 2 (p = 0)
    # is never read; a negative q at id 0 makes the residual row invalid.
    z = np.array([[[5.0, 0.0, 0.0], [0.0, 0.0, 0.0]]] * 2, np.float32)
    q = np.array([[[0.5, 0.7, -0.2]], [[-0.1, 0.7, 0.4]]], np.float32)
    xt = np.array([[1], [1]], np.int32)
    u = np.array([[0.01, 0.999], [0.01, 0.999]], np.float32)
    out = orc.verify(z, q, xt, u, 1.0, 0.5, 0)
    assert list(out["accept_len"]) == [0, 0]
    assert out["row_status"][0, 0] == 0 and out["out_token"][0] == 0
    assert out["res_sum"][0] == pytest.approx(0.5, abs=1e-15)
    assert out["row_status"][1, 0] & orc.ROW_BAD_Q and out["out_token"][1] == -1


# --------------------------------------------------------------------------
# step 7-8: branch cache


def test_cache_build_matches_full_sort_excluding_draft_token(orc):
    rng = np.random.default_rng(61)
    B, K, V = 3, 4, 500
    q = rng.random((B, K, V)).astype(np.float32)
    q[q < 0.3] = 0.0
    q[0, 1, 10:20] = q[0, 1, 5]                    # ties resolved by lower id
    q = (q / q.sum(-1, keepdims=True)).astype(np.float32)
    xt = rng.integers(0, V, (B, K)).astype(np.int32)
    xt[0, 1] = 5
    F = np.array([3, 7, 0, 5], np.int32)
    bt, bp = orc.cache_build(q, xt, F)
    off = np.concatenate([[0], np.cumsum(F)[:-1]])
    for b in range(B):
        for d in range(K):
            qq = q[b, d].astype(np.float64)
            ids = [x for x in np.lexsort((np.arange(V), -qq)) if x != xt[b, d] and qq[x] > 0][: F[d]]
            got = bt[b, off[d]: off[d] + F[d]]
            np.testing.assert_array_equal(got[: len(ids)], ids)
            assert (got[len(ids):] == -1).all()
            np.testing.assert_allclose(bp[b, off[d]: off[d] + len(ids)],
                                       qq[ids] / (1 - qq[xt[b, d]]), rtol=1e-12)


def test_cache_with_every_alternative_sums_to_one(orc):
    rng = np.random.default_rng(62)
    V = 64
    q = _norm(rng.random(V) + 0.01)
    q32 = q.astype(np.float32)[None, None]
    xt = np.array([[17]], np.int32)
    bt, bp = orc.cache_build(q32, xt, np.array([V - 1], np.int32))
    assert sorted(bt[0].tolist()) == [x for x in range(V) if x != 17]
    assert abs(bp.sum() - 1.0) < 1e-6


def test_cache_lookup_exhaustive(orc):
    F = np.array([2, 0, 3], np.int32)
    K = 3
    bt = np.array([[7, 9, 4, 5, 6]], np.int32)   # depth0: 7,9  depth1: -  depth2: 4,5,6
    table = {(0, 7): 0, (0, 9): 1, (2, 4): 2, (2, 5): 3, (2, 6): 4}
    for pi in range(K + 1):
        for tok in range(-1, 11):
            slot = orc.cache_lookup(bt, F, np.array([pi], np.int32), np.array([tok], np.int32))[0]
            expect = -2 if pi == K else table.get((pi, tok), -1)
            assert slot == expect, (pi, tok, slot)


# --------------------------------------------------------------------------
# Sec. IV-C: geometric branch allocation


@pytest.mark.parametrize("B_alloc,gamma,alpha,beta", [(64, 16, 0.9, 1.0), (40, 8, 0.6, 0.5),
                                                       (17, 5, 0.99, 2.0), (100, 16, 0.3, 1.0)])
def test_branch_allocation_geometric_sum_and_decay(orc, B_alloc, gamma, alpha, beta):
    real, ints = orc.branch_alloc(B_alloc, gamma, alpha, beta)
    eta = alpha ** (1 / (beta + 1))
    assert abs(sum(real) - B_alloc) < 1e-9 * B_alloc            # geometric series closes the budget
    assert all(real[i + 1] / real[i] == pytest.approx(eta) for i in range(gamma - 1))
    assert sum(ints) == B_alloc
    assert all(ints[i] >= ints[i + 1] for i in range(gamma - 1))
    assert all(abs(a - b) < 1 for a, b in zip(ints, real))


def test_branch_allocation_uniform_limit(orc):
    real, ints = orc.branch_alloc(48, 8, 1.0, 1.0)
    assert ints == [6] * 8


def test_branch_allocation_golden(orc):
    import os
    path = os.path.join(os.path.dirname(__file__), "golden", "branch_alloc.txt")
    for line in open(path):
        if not line.strip() or line.startswith("#"):
            continue
        a, b, c, d, rest = line.split(None, 4)
        _, ints = orc.branch_alloc(int(a), int(b), float(c), float(d))
        assert ints == [int(x) for x in rest.split()]


# --------------------------------------------------------------------------
# step 9: edge-side resample from the sparse payload (Alg. 1 RESAMPLE)


def _sparse_case(ids0, probs0, tail0, q0, u_draw):
    """One sequence, K = 1, rejected at position 0: payload of row 0 given."""
    k = len(ids0)
    ids = np.full((1, 2, k), -1, np.int32)
    probs = np.zeros((1, 2, k), np.float32)
    tail = np.ones((1, 2), np.float32)
    ids[0, 0] = ids0
    probs[0, 0] = probs0
    tail[0, 0] = tail0
    q = np.asarray([[q0]], np.float32)
    u = np.array([[0.5, u_draw]], np.float32)
    return dict(accept_len=np.array([0], np.int32), ids=ids, probs=probs, tail=tail,
                row_status=np.zeros((1, 2), np.int32), q=q, u=u)


@pytest.mark.parametrize("u_draw,token", [(0.5, 0), (0.9, 1)])
def test_sparse_resample_tail_below_draft_mass(orc, u_draw, token):
    # payload {0: 0.5, 1: 0.3}, tail 0.2; q uniform over 4 ids.  Outside the
    # payload q holds 0.5 > 0.2, so the spread tail never exceeds q there:
    # r^ = (0.25, 0.05, 0, 0).  u * 0.3 < 0.25 picks id 0, else id 1.
    c = _sparse_case([0, 1], [0.5, 0.3], 0.2, [0.25, 0.25, 0.25, 0.25], u_draw)
    o = orc.resample_sparse(c["accept_len"], c["ids"], c["probs"], c["tail"], c["row_status"], c["q"], c["u"])
    assert o["token"][0] == token and o["status"][0] == 0
    np.testing.assert_allclose(o["dist"][0], [0.25 / 0.3, 0.05 / 0.3, 0.0, 0.0], atol=1e-6)


@pytest.mark.parametrize("u_draw,token", [(0.3, 1), (0.6, 2), (0.9, 3)])
def test_sparse_resample_tail_spread_like_the_draft(orc, u_draw, token):
    # q = (0.7, 0.2, 0.05, 0.05): outside the payload q holds 0.1 and the
    # tail 0.2, so p^ = 2 q there and r^ = q = 0.05 on ids 2 and 3;
    # on the payload r^ = (max(0, 0.5 - 0.7), 0.3 - 0.2) = (0, 0.1).
    c = _sparse_case([0, 1], [0.5, 0.3], 0.2, [0.7, 0.2, 0.05, 0.05], u_draw)
    o = orc.resample_sparse(c["accept_len"], c["ids"], c["probs"], c["tail"], c["row_status"], c["q"], c["u"])
    assert o["token"][0] == token
    np.testing.assert_allclose(o["dist"][0], [0.0, 0.5, 0.25, 0.25], atol=1e-6)
    assert o["res_sum"][0] == pytest.approx(0.2, abs=1e-7)


def test_sparse_resample_bonus_row_uses_the_payload(orc):
    # pi = K: no draft row; the draw follows the payload probabilities
    c = _sparse_case([3, 1, 2], [0.6, 0.3, 0.1], 0.0, [0.25] * 4, 0.95)
    c["accept_len"][0] = 1
    c["ids"][0, 1] = [3, 1, 2]
    c["probs"][0, 1] = [0.6, 0.3, 0.1]
    c["tail"][0, 1] = 0.0
    o = orc.resample_sparse(c["accept_len"], c["ids"], c["probs"], c["tail"], c["row_status"], c["q"], c["u"])
    np.testing.assert_allclose(o["dist"][0], [0.0, 0.3, 0.1, 0.6], atol=1e-7)
    assert o["token"][0] == 3          # 0.95 > 0.3 + 0.1 in id order


def test_sparse_resample_invalid_rows(orc):
    c = _sparse_case([0, 1], [0.5, 0.3], 0.2, [-0.1, 0.5, 0.3, 0.3], 0.5)
    o = orc.resample_sparse(c["accept_len"], c["ids"], c["probs"], c["tail"], c["row_status"], c["q"], c["u"])
    assert o["token"][0] == -1 and o["status"][0] == orc.ROW_BAD_Q      # q < 0 on the payload
    c = _sparse_case([0, 1], [0.5, 0.3], 0.2, [0.25] * 4, 0.5)
    c["row_status"][0, 0] = orc.ROW_NONFINITE
    o = orc.resample_sparse(c["accept_len"], c["ids"], c["probs"], c["tail"], c["row_status"], c["q"], c["u"])
    assert o["token"][0] == -1 and o["status"][0] == orc.ROW_NONFINITE


def _verify_then_resample(orc, seed, k, top_p=0.9, T=1.0, V=2000, n=300):
    rng = np.random.default_rng(seed)
    zd = rng.normal(0.0, 2.0, (n, 2, V))
    z = (0.8 * zd + 0.6 * rng.normal(0.0, 2.0, (n, 2, V))).astype(np.float32)
    qw = np.exp((zd[:, :1] - zd[:, :1].max(-1, keepdims=True)) / T)
    q = (qw / qw.sum(-1, keepdims=True)).astype(np.float32)
    xt = np.array([[np.searchsorted(np.cumsum(q[b, 0], dtype=np.float64), rng.random() * 0.999)] for b in range(n)],
                  np.int32).clip(0, V - 1)
    u = ((rng.integers(1, 1 << 24, size=(n, 2))) / float(1 << 24)).astype(np.float32)
    ov = orc.verify(z, q, xt, u, T, top_p, k)
    os_ = orc.resample_sparse(ov["accept_len"], ov["topk_ids"], ov["topk_probs"].astype(np.float32),
                              ov["tail"].astype(np.float32), ov["row_status"], q, u)
    p, _ = orc.warp(z, T, top_p)
    return z, q, u, ov, os_, p


def test_sparse_resample_is_the_exact_draw_when_the_nucleus_fits(orc):
    # k >= every nucleus size: tail = 0 and p^ = p, so the edge's draw is the
    # cloud's exact residual draw, token for token
    z, q, u, ov, os_, p = _verify_then_resample(orc, 71, k=256, top_p=0.8, T=0.5)
    assert ov["n_nuc"].max() <= 256
    n = len(u)
    pi = ov["accept_len"]
    same = 0
    for b in range(n):
        s = ov["res_sum"][b]
        t = ov["res_target"][b]
        if any(np.isfinite(c) and abs(t - c) < 1e-6 * s for c in (ov["res_cj"][b], ov["res_cjm1"][b])):
            continue
        assert os_["token"][b] == ov["out_token"][b], b
        same += 1
        # the distribution drawn from is norm(max(0, p_pi - q_pi)) (or p_K)
        r = p[b, pi[b]] - (q[b, 0] if pi[b] < 1 else 0.0)
        r = np.maximum(r, 0.0)
        if r.sum() == 0.0:
            r = p[b, pi[b]]
        np.testing.assert_allclose(os_["dist"][b], r / r.sum(), atol=1e-6)
    assert same >= n - 3


def test_sparse_resample_distance_shrinks_with_payload_size(orc):
    # total-variation distance between the edge's distribution and the exact
    # residual, averaged over sequences: 0 once k covers every nucleus, and
    # never larger for a larger payload on these rows
    tvs = []
    for k in (4, 16, 64, 256):
        z, q, u, ov, os_, p = _verify_then_resample(orc, 72, k=k, top_p=0.8, T=0.5, n=120)
        pi = ov["accept_len"]
        d = []
        for b in range(len(u)):
            r = np.maximum(p[b, pi[b]] - (q[b, 0] if pi[b] < 1 else 0.0), 0.0)
            if r.sum() == 0.0:
                r = p[b, pi[b]]
            d.append(0.5 * np.abs(os_["dist"][b] - r / r.sum()).sum())
        tvs.append(float(np.mean(d)))
    assert tvs[0] > 0.01
    assert all(a >= b - 1e-9 for a, b in zip(tvs, tvs[1:])), tvs
    assert tvs[-1] < 1e-6, tvs


def test_sparse_resample_tv_golden_table():
    # the committed table of the edge's distance to the exact residual is
    # reproduced by the oracle (two rows of the smallest workload)
    import os
    import sys
    here = os.path.dirname(os.path.abspath(__file__))
    sys.path.insert(0, os.path.join(here, "golden"))
    import make_sparse_tv as mk
    want = {}
    for line in open(os.path.join(here, "golden", "sparse_resample_tv.txt")):
        if line.startswith("#") or not line.strip():
            continue
        f = line.split()
        want[(f[0], int(f[1]))] = line.strip()
    for k in (4, 64):
        assert mk.fmt("b16_k8_v32000_f32", k, mk.row("b16_k8_v32000_f32", k)) == want[("b16_k8_v32000_f32", k)]


# --------------------------------------------------------------------------
# cache hit probability (Sec. III-C; Eq. for P_hit in Sec. IV-C)


def _hit_batch(orc, n, F, seed, V=16, K=3):
    rng = np.random.default_rng(seed)
    z_rows = rng.normal(0.0, 1.5, (K + 1, V))
    q_rows = _softmax(z_rows[:K] + rng.normal(0.0, 1.0, (K, V)), 1.0).reshape(K, V)
    z, q, xt, u = _batch(z_rows, q_rows, n, seed + 1)
    return z, q, xt, u


def test_hit_probability_matches_simulation_of_the_protocol(orc):
    # the oracle's own verify + cache + lookup, repeated over uniforms, hits
    # as often as the closed form predicts (5 sigma)
    F = [3, 2, 1]
    z, q, xt, u = _hit_batch(orc, 40000, F, 81)
    ov = orc.verify(z, q, xt, u, 1.0, 1.0, 0)
    bt, _ = orc.cache_build(q, xt, F)
    slot = orc.cache_lookup(bt, F, ov["accept_len"], ov["out_token"])
    hits = (slot >= 0) | (slot == -2)
    hp, pp = orc.hit_prob(z, q, xt, 1.0, 1.0, bt, F)
    sd = np.sqrt(np.sum(hp * (1 - hp))) / len(hp)
    assert abs(hits.mean() - hp.mean()) < 5 * sd, (hits.mean(), hp.mean(), sd)
    assert 0.2 < hp.mean() < 0.99


def test_hit_probability_closed_forms(orc):
    z, q, xt, u = _hit_batch(orc, 200, [0, 0, 0], 82)
    ov = orc.verify(z, q, xt, u, 1.0, 1.0, 0)
    a = np.minimum(1.0, ov["ratio"])
    # no branches: only a fully accepted chain is recovered
    bt0, _ = orc.cache_build(q, xt, [0, 0, 0])
    hp, pp = orc.hit_prob(z, q, xt, 1.0, 1.0, bt0, [0, 0, 0])
    np.testing.assert_allclose(hp, np.prod(a, axis=1), rtol=1e-12)
    np.testing.assert_allclose(pp, np.prod(a, axis=1), rtol=1e-12)
    # every alternative cached (q has full support here): always recovered
    Fall = [15, 15, 15]
    bt1, _ = orc.cache_build(q, xt, Fall)
    hp, pp = orc.hit_prob(z, q, xt, 1.0, 1.0, bt1, Fall)
    np.testing.assert_allclose(hp, 1.0, atol=1e-12)
    np.testing.assert_allclose(pp, 1.0, atol=1e-12)


def test_hit_rate_golden_table():
    # the committed hit-rate table is reproduced by the oracle (one regime)
    import os
    import sys
    here = os.path.dirname(os.path.abspath(__file__))
    sys.path.insert(0, os.path.join(here, "golden"))
    import make_hit_rates as mk
    lines = [ln.strip() for ln in open(os.path.join(here, "golden", "hit_rates.txt")) if not ln.startswith("#")]
    got = mk.rows(*mk.REGIMES[0])
    assert got == lines[:len(got)]


# --------------------------------------------------------------------------
# COMPACT_KV / ROLLBACK_KV (Alg. 1)


def test_compact_kv_hand_example(orc):
    # one plane, one head, D = 1, positions labelled by their index: prefix
    # of 3, main chain of K = 2 (positions 3-4), branches of 2 (slot 0 at
    # 5-6, slot 1 at 7-8, slot 2 at 9-10)
    kv = np.arange(12, dtype=np.float32).reshape(1, 1, 1, 12, 1).repeat(4, axis=1)
    al = np.array([0, 1, 2, 1], np.int32)
    slot = np.array([1, 2, -2, -1], np.int32)
    out, n = orc.compact_kv(kv, [3, 3, 3, 3], al, slot, 2, 2)
    assert list(n) == [5, 6, 5, 4]
    assert out[0, 0, 0, :, 0].tolist() == [0, 1, 2, 7, 8, 5, 6, 7, 8, 9, 10, 11]    # slot 1 behind t+0
    assert out[0, 1, 0, :, 0].tolist() == [0, 1, 2, 3, 9, 10, 6, 7, 8, 9, 10, 11]   # slot 2 behind t+1
    assert (out[0, 2:] == kv[0, 2:]).all()                                          # accept / miss: no move


def test_compact_kv_overlapping_move_and_bounds(orc):
    # branch rows overlap their destination (distance 1 < length 3)
    kv = np.arange(10, dtype=np.float32).reshape(1, 1, 1, 10, 1)
    out, n = orc.compact_kv(kv, [2], [1], [0], 2, 3)   # src 4..6 -> dst 3..5
    assert n[0] == 6
    assert out[0, 0, 0, :, 0].tolist() == [0, 1, 2, 4, 5, 6, 6, 7, 8, 9]
    out, n = orc.compact_kv(kv, [6], [0], [0], 2, 3)   # src 8..10 passes the end
    assert n[0] == -1 and (out == kv).all()


# --------------------------------------------------------------------------
# tree attention mask (Sec. III-C)


def test_tree_mask_hand_example(orc):
    # K = 3 main tokens m0 m1 m2; one branch at depth 0 (b0 b0'), one at
    # depth 1 (b1 b1'); branch_len 2 -> 7 tree tokens
    mask, depth = orc.tree_mask([1, 1, 0], 3, 2)
    want = np.array([
        # m0 m1 m2 b0 b0' b1 b1'
        [1, 0, 0, 0, 0, 0, 0],   # m0
        [1, 1, 0, 0, 0, 0, 0],   # m1
        [1, 1, 1, 0, 0, 0, 0],   # m2
        [0, 0, 0, 1, 0, 0, 0],   # b0: replaces m0, sees no main token
        [0, 0, 0, 1, 1, 0, 0],   # b0'
        [1, 0, 0, 0, 0, 1, 0],   # b1: replaces m1, sees m0
        [1, 0, 0, 0, 0, 1, 1],   # b1'
    ], bool)
    assert (mask == want).all()
    assert depth.tolist() == [0, 1, 2, 0, 1, 1, 2]


def test_tree_mask_invariants(orc):
    F, K, L = [3, 2, 2, 1, 0, 1], 6, 4
    mask, depth = orc.tree_mask(F, K, L)
    n = K + sum(F) * L
    assert mask.shape == (n, n)
    assert (np.triu(mask, 1) == 0).all()                  # ancestors come first in the packed order
    assert (np.diag(mask)).all()
    assert (mask.sum(1) == depth + 1).all()
    # a branch token at depth d, offset o sees d main tokens and o + 1 branch tokens
    s = 0
    for d in range(K):
        for _ in range(F[d]):
            for o in range(L):
                q = K + s * L + o
                assert mask[q, :K].sum() == d and mask[q, K:].sum() == o + 1 and depth[q] == d + o
            s += 1
