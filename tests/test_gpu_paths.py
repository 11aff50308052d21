"""Parity on inputs built to drive each branch of the fast row kernel.

The workspace's first int32 words count, per call, the rows handed to the
exact general kernel, bounded-wait timeouts, rows certified only by the full
sketch histogram (the top group maxima kept per thread were not enough),
rows whose candidates were ordered by bitonic sort (more than 512), rows the
general kernel finished by radix selection, rows split over several CTAs,
and rows the general kernel finished by its bfloat16 value histogram.  Each
test asserts the branch it targets was taken, then compares every output
with the float64 oracle under the rules of tests/parity.py.
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


def _run(A, orc, w, z):
    """Verify the generator's q, x~, u with the logits z on both sides."""
    inp = gen.generate(w)
    inp["z"] = z
    if z.dtype == np.uint16:
        zt = torch.from_numpy(z.view(np.int16)).cuda().view(torch.bfloat16)
    else:
        zt = torch.from_numpy(z).cuda()
    q, xt, u = (torch.from_numpy(inp[key]).cuda() for key in ("q", "xt", "u"))
    ws = torch.zeros(A.workspace_bytes(w.B, w.K, w.V, w.k), dtype=torch.uint8, device="cuda")
    g = A.verify(zt, q, xt, u, w.T, w.top_p, w.k, workspace=ws)
    torch.cuda.synchronize()
    g = {key: v.cpu().numpy() for key, v in g.items()}
    counters = ws[:28].view(torch.int32).cpu().numpy().tolist()
    o = orc.verify(z, inp["q"], inp["xt"], inp["u"], w.T, w.top_p, w.k)
    res = parity.compare_verify(inp, g, o, w.top_p, z.dtype == np.uint16, w.k)
    return counters, res


def _plateau(B, K, V, n_hot, group, seed):
    """-30 everywhere except n_hot ids, one per sketch group, near 0."""
    rng = np.random.default_rng(seed)
    z = np.full((B, K + 1, V), -30.0, np.float32)
    j = np.arange(n_hot)
    ids = j * group + (j % group)
    for b in range(B):
        for i in range(K + 1):
            z[b, i, ids] = rng.uniform(0.0, 1.5, n_hot).astype(np.float32)
    return z


def test_second_tier_certification_and_bitonic_order(A, orc):
    # 1500 near-equal ids in 1500 different sketch groups (16 float32 logits
    # each): the 512 per-thread top maxima carry too little mass, the full
    # sketch certifies, and the nucleus (~1200 ids) is ordered by bitonic sort
    w = gen.make_workload(2, 2, 32000, "f32", T=1.0, top_p=0.8, k=64, seed=31)
    counters, res = _run(A, orc, w, _plateau(2, 2, 32000, 1500, 16, 31))
    fallback, timeouts, second_tier, bitonic, radix, split, valhist = counters
    assert fallback == 0 and timeouts == 0
    # a row split over CTAs bins every part's top maxima, which here covers
    # every hot group: the first tier then suffices
    assert second_tier == 6 - split and bitonic == 6, counters
    assert res["checked_seqs"] == 2


def test_more_candidates_than_capacity_falls_back(A, orc):
    # 3000 near-equal ids: the nucleus alone exceeds the 2048 candidates the
    # fast kernel holds, so every row goes to the exact general kernel
    w = gen.make_workload(2, 1, 64000, "f32", T=1.0, top_p=0.8, k=32, seed=32)
    counters, res = _run(A, orc, w, _plateau(2, 1, 64000, 3000, 16, 32))
    assert counters[0] == 4, counters
    assert res["checked_seqs"] == 2


def test_first_tier_suffices_on_the_benchmark_rows(A, orc):
    # the first 4 sequences of the 256000-id benchmark workload (68 rows):
    # nearly every row is certified by the per-thread top maxima, and all
    # are ranked directly on the fast path
    w = dataclasses.replace(gen.WORKLOADS["b256_k16_v256000_bf16"], B=4)
    z = gen.generate(w)["z"]
    counters, res = _run(A, orc, w, z)
    fallback, timeouts, second_tier, bitonic = counters[:4]
    assert fallback == 0 and timeouts == 0 and bitonic == 0, counters
    assert second_tier <= 3, counters
    assert res["checked_seqs"] >= 3


@pytest.mark.parametrize("dtype,V", [("bf16", 600000), ("f32", 300000), ("f32", 600000)],
                         ids=["bf16_gc8", "f32_gc8", "f32_general"])
def test_large_vocabularies(A, orc, dtype, V):
    # bf16 at 600000 ids and f32 at 300000 use 8 chunks per sketch group;
    # f32 at 600000 exceeds the sketch and runs on the general kernel
    w = gen.make_workload(1, 1, V, dtype, T=0.8, top_p=0.9, k=48, seed=34)
    z = gen.generate(w)["z"]
    counters, res = _run(A, orc, w, z)
    assert counters[1] == 0
    assert res["checked_seqs"] == 1


def _bf16(z):
    return gen.f32_to_bf16(np.ascontiguousarray(z, dtype=np.float32))


def test_value_histogram_takes_large_nucleus_bf16_rows(A, orc):
    # rows of the 128256-id recipe (nuclei of thousands of ids): the sketch
    # cannot order them, and the general kernel finishes every one by counting
    # ids per bf16 value (the crossing lies among the 4096 values below the max)
    w = gen.make_workload(2, 2, 128256, "bf16", sigma=3.0, rho=0.5, T=1.0, top_p=0.9, k=32, seed=41)
    z = gen.generate(w)["z"]
    counters, res = _run(A, orc, w, z)
    fallback, radix, valhist = counters[0], counters[4], counters[6]
    assert fallback >= 1 and valhist == fallback and radix == 0, counters
    assert res["checked_seqs"] >= 1


def test_value_histogram_declines_a_crossing_below_its_window(A, orc):
    # flat rows (T=2, top_p=0.99): the crossing lies among negative logits,
    # whose keys are below the window (below every tiny positive value); the
    # binned path takes the rows
    w = gen.make_workload(3, 2, 65536, "bf16", T=2.0, top_p=0.99, k=64, seed=41)
    z = gen.generate(w)["z"]
    counters, res = _run(A, orc, w, z)  # (compares every unflagged output)
    fallback, valhist = counters[0], counters[6]
    assert fallback >= 1 and valhist == 0, counters


@pytest.mark.parametrize("n_vals,V,expect_valhist", [(40, 32000, True), (24, 65536, False)],
                         ids=["ties_within_capacity", "ties_beyond_capacity"])
def test_value_histogram_ties(A, orc, n_vals, V, expect_valhist):
    # logits from a few distinct bf16 values: the crossing value is shared by
    # ~V/n_vals ids, taken in id order.  Up to 1024 of them the value
    # histogram orders them itself; beyond that the binned path takes the row.
    w = gen.make_workload(2, 2, V, "bf16", T=1.0, top_p=0.7, k=32, seed=42)
    rng = np.random.default_rng(42)
    vals = np.linspace(-2.0, 2.0, n_vals).astype(np.float32)
    z = _bf16(vals[rng.integers(0, n_vals, size=(2, 3, V))])
    counters, res = _run(A, orc, w, z)
    fallback, valhist = counters[0], counters[6]
    assert fallback == 6, counters
    assert (valhist == 6) if expect_valhist else (valhist == 0), counters
    assert res["checked_seqs"] >= 1


def test_value_histogram_top_p_one_rows(A, orc):
    # top_p = 1 on bf16 rows: 3000 ids spread over the sketch groups with
    # values in [1, 1.05] (seven bf16 values, all within one sketch bin), the
    # rest at -30.  The k-th id lies among ~3000 candidates, more than the
    # fast kernel holds, so it hands every row over with its max and exp-sum;
    # the value histogram counts the finite ids itself (the whole row is the
    # nucleus) and takes the payload, ties in id order, from the top value.
    V, n_hot = 64000, 3000
    w = gen.make_workload(2, 1, V, "bf16", T=1.0, top_p=1.0, k=64, seed=44)
    rng = np.random.default_rng(44)
    z = np.full((2, 2, V), -30.0, np.float32)
    j = np.arange(n_hot)
    ids = j * 16 + (j % 16)
    for b in range(2):
        for i in range(2):
            z[b, i, ids] = rng.uniform(1.0, 1.05, n_hot).astype(np.float32)
    counters, res = _run(A, orc, w, _bf16(z))
    assert counters[0] == 4 and counters[6] == 4 and counters[4] == 0, counters
    assert res["checked_seqs"] >= 1


def test_signed_zeros_on_the_general_path(A, orc):
    # -0 and +0 are one value (one order key): the nucleus and the payload take
    # them in id order whatever their signs.  Ten positive ids, then a run of
    # 512 zeros of random sign (16 whole sketch groups, so the one-max-per-group
    # bound cannot certify the row), the rest at -20.  Zero lies ~16000 bf16
    # keys below a max near 1, beyond the value histogram's window, so the
    # binned path takes the rows.
    V = 32000
    w = gen.make_workload(2, 1, V, "bf16", T=1.0, top_p=0.999, k=64, seed=43)
    rng = np.random.default_rng(43)
    z = np.full((2, 2, V), -20.0, np.float32)
    z[:, :, 100:110] = rng.uniform(0.5, 1.0, size=(2, 2, 10)).astype(np.float32)
    z[:, :, 1024:1536] = np.where(rng.random((2, 2, 512)) < 0.5, np.float32(0.0), np.float32(-0.0))
    counters, res = _run(A, orc, w, _bf16(z))
    assert counters[0] == 4 and counters[6] == 0, counters
    assert res["checked_seqs"] >= 1
