"""Host-side budgeting and branch allocation (Sec. IV-B, IV-C) in the library,
checked against the oracle's allocator and against closed forms.  No GPU."""
import itertools

import pytest

import paper_2609_02514_gb300 as A


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2609_02514_gb300 import build
    build.build()
    A.load()


@pytest.mark.parametrize("B_alloc,gamma,alpha,beta", list(itertools.product(
    [0, 1, 7, 40, 64, 200, 1000], [1, 4, 8, 16], [0.3, 0.6, 0.9, 0.99, 1.0], [0.5, 1.0, 3.0])))
def test_branch_alloc_matches_the_oracle(orc, B_alloc, gamma, alpha, beta):
    _, want = orc.branch_alloc(B_alloc, gamma, alpha, beta)
    got = A.branch_alloc(B_alloc, gamma, alpha, beta)
    assert got == want
    assert sum(got) == B_alloc


def test_branch_alloc_decays_and_rejects_bad_arguments():
    F = A.branch_alloc(64, 16, 0.9, 1.0)
    assert F == sorted(F, reverse=True) and F[0] > F[-1]
    for bad in ((-1, 4, 0.9, 1.0), (8, 0, 0.9, 1.0), (8, 17, 0.9, 1.0), (8, 4, 0.0, 1.0), (8, 4, 1.2, 1.0),
                (8, 4, 0.9, 0.0), (8, 4, float("nan"), 1.0)):
        with pytest.raises(A.AcespecError):
            A.branch_alloc(*bad)


def test_tree_budget_inverts_a_linear_latency_profile():
    # T(B) = 5 ms + 0.25 ms * B: RTT + T_verify = 30 ms fits B = 100
    lat = [0.005 + 0.00025 * b for b in range(1, 401)]
    assert A.tree_budget(lat, 0.025, 0.005, 1000) == 100
    assert A.tree_budget(lat, 0.025, 0.005, 64) == 64          # B_max caps it
    assert A.tree_budget(lat, 0.0, 0.0, 1000) == 0             # nothing fits
    assert A.tree_budget(lat, 10.0, 0.0, 1000) == 400          # the whole table fits
    for bad in (([0.2, 0.1], 0.1, 0.1, 8), ([], 0.1, 0.1, 8), ([0.1], -1.0, 0.1, 8), ([0.1], 0.1, 0.1, -1)):
        with pytest.raises((A.AcespecError, ValueError)):
            A.tree_budget(*bad)
