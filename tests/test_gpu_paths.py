"""Parity on inputs built to drive each branch of the row kernels.

The workspace's first ten int32 words count, per call: rows handed to the
exact general kernel, bounded-wait timeouts (reserved), bfloat16 rows the
single-pass kernel finished from its value counts, rows whose candidates were
ordered by bitonic sort (more than 512), rows the general kernel finished by
radix selection, rows whose nucleus cut was left to the resolve step, rows
the general kernel finished by its bfloat16 value histogram, accept tests
that ranked the draft token among the ids of the crossing value, rows that
published their depth, rows that took their depth from finished rows, and
rows whose values were counted in a second pass.  Each test
asserts the branch it targets was taken, then compares every output with the
float64 oracle under the rules of tests/parity.py.  Tests of the general
kernel's own branches call the exact entry point (every row on that kernel).
"""
import dataclasses
import math

import numpy as np
import pytest

import gen
from tests import parity

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

(FALLBACK, TIMEOUTS, VALUE_MODE, BITONIC, RADIX, LAZY, GEN_VALHIST, TIE_RANK, PUBLISHED, HINTED, RECOUNT, SHORT,
 SKETCH_LED) = range(13)


@pytest.fixture(scope="module")
def A():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_02514_gb300 as A
    A.load()
    return A


def _run(A, orc, w, z, exact=False, inp=None):
    """Verify the generator's q, x~, u (or inp's) with the logits z on both sides."""
    inp = dict(gen.generate(w)) if inp is None else inp
    inp["z"] = z
    if z.dtype == np.uint16:
        zt = torch.from_numpy(z.view(np.int16)).cuda().view(torch.bfloat16)
    else:
        zt = torch.from_numpy(z).cuda()
    q, xt, u = (torch.from_numpy(inp[key]).cuda() for key in ("q", "xt", "u"))
    ws = torch.zeros(A.workspace_bytes(w.B, w.K, w.V, w.k), dtype=torch.uint8, device="cuda")
    g = A.verify(zt, q, xt, u, w.T, w.top_p, w.k, workspace=ws, exact=exact)
    torch.cuda.synchronize()
    g = {key: v.cpu().numpy() for key, v in g.items()}
    counters = ws[A.COUNTERS_OFFSET:A.COUNTERS_OFFSET + 64].view(torch.int32).cpu().numpy().tolist()
    o = orc.verify(z, inp["q"], inp["xt"], inp["u"], w.T, w.top_p, w.k)
    res = parity.compare_verify(inp, g, o, w.top_p, z.dtype == np.uint16, w.k)
    return counters, res


def _bf16(z):
    return gen.f32_to_bf16(np.ascontiguousarray(z, dtype=np.float32))


def _sampled_ids(V, dtype):
    """Ids the single-pass kernel reads in its first iteration: tiles of 32
    16-byte chunks, tile t of the row order at (t * p) mod ntile, p the
    smallest integer >= ntile / 64 coprime with ntile, t < 64."""
    epc = 8 if dtype == "bf16" else 4
    ntile = -(-(V // epc) // 32)
    p = max(1, ntile // 64)
    while math.gcd(p, ntile) != 1:
        p += 1
    ids = []
    for t in range(min(64, ntile)):
        tile = t * p % ntile
        ids.append(np.arange(tile * 32 * epc, min((tile + 1) * 32 * epc, V)))
    return np.concatenate(ids)


# ---------------------------------------------------------------------------
# the single-pass kernel


def test_value_counts_on_the_benchmark_rows(A, orc):
    # the first 4 sequences of the 256000-id benchmark workload (68 rows, the
    # first rows of a call: D = 10 T): counted per bf16 value, the payload
    # re-read from the sketch's groups; no row needs the general kernel
    w = dataclasses.replace(gen.WORKLOADS["b256_k16_v256000_bf16"], B=4)
    z = gen.generate(w)["z"]
    counters, res = _run(A, orc, w, z)
    assert counters[TIMEOUTS] == 0 and counters[FALLBACK] == 0 and counters[VALUE_MODE] == 68, counters
    assert res["checked_seqs"] >= 3


def test_large_nuclei_leave_the_cut_to_the_resolve_step(A, orc):
    # rows of the 128256-id recipe (nuclei of thousands of ids, k = 32): the
    # crossing value's ids are not among the payload's, so the cut is left to
    # the resolve step, which finds it for the drawn rows
    w = gen.make_workload(3, 4, 128256, "bf16", sigma=3.0, rho=0.5, T=1.0, top_p=0.9, k=32, seed=41)
    z = gen.generate(w)["z"]
    counters, res = _run(A, orc, w, z)
    assert counters[FALLBACK] == 0 and counters[VALUE_MODE] == 15 and counters[LAZY] == 15, counters
    assert res["checked_seqs"] >= 2


def test_exact_cut_when_the_nucleus_fits_the_payload(A, orc):
    # 50 dominant ids at 15 outside the sampled tiles, 60000 ids in [6, 8]:
    # the sample sees only the bulk; the running max reaches 15 later.  The
    # nucleus (about 35 of the 50 tied ids) is shorter than k, so the payload
    # re-read holds every id of the crossing value and the cut is exact
    V = 65536
    w = gen.make_workload(2, 1, V, "bf16", T=1.0, top_p=0.5, k=64, seed=45)
    rng = np.random.default_rng(45)
    samp = _sampled_ids(V, "bf16")
    rest = np.setdiff1d(np.arange(V), samp)
    z = np.full((2, 2, V), -30.0, np.float32)
    for b in range(2):
        for i in range(2):
            z[b, i, rng.choice(V, 60000, replace=False)] = rng.uniform(6.0, 8.0, 60000)
            z[b, i, rng.choice(rest, 50, replace=False)] = 15.0
    counters, res = _run(A, orc, w, _bf16(z))
    assert counters[FALLBACK] == 0 and counters[VALUE_MODE] == 4 and counters[LAZY] == 0, counters
    assert res["checked_seqs"] >= 1


def test_draft_token_on_the_crossing_value(A, orc):
    # the draft token of every draft row is moved to an id holding that row's
    # crossing value (the n_nuc-th id in order), with q > 0 there: the accept
    # test ranks it among the ids of that value, which were not read
    w = gen.make_workload(2, 3, 128256, "bf16", sigma=3.0, rho=0.5, T=1.0, top_p=0.9, k=32, seed=46)
    inp = dict(gen.generate(w))
    z = inp["z"]
    zf = gen.bf16_to_f32(z).astype(np.float64)
    o = orc.verify(z, inp["q"], inp["xt"], inp["u"], w.T, w.top_p, w.k)
    xt = inp["xt"].copy()
    q = inp["q"].copy()
    for b in range(w.B):
        for i in range(w.K):
            row = zf[b, i]
            order = np.lexsort((np.arange(w.V), -row))
            v = row[order[o["n_nuc"][b, i] - 1]]
            same = np.flatnonzero(row == v)
            x = int(same[len(same) // 2])  # one in the middle: in or out of the nucleus
            xt[b, i] = x
            if q[b, i, x] <= 0.0:
                q[b, i, x] = 1e-3
    inp["xt"], inp["q"] = xt, q
    counters, res = _run(A, orc, w, z, inp=inp)
    assert counters[TIE_RANK] >= 1 and counters[FALLBACK] == 0, counters
    assert res["checked_seqs"] >= 1


def _tied_top(V, n_top, seed):
    """Rows of n_top ids at 10 spread over the row, the rest at -30."""
    rng = np.random.default_rng(seed)
    z = np.full((2, 2, V), -30.0, np.float32)
    for b in range(2):
        for i in range(2):
            z[b, i, rng.choice(V, n_top, replace=False)] = 10.0
    return _bf16(z)


def test_payload_ties_ordered_by_bitonic_sort(A, orc):
    # 700 ids tied at the top value, top_p = 0.5001 (the crossing, 351 ids
    # in, is not within 1e-6 of it), k = 64: the crossing value is the
    # payload's last value, so all 700 of its ids are re-read (more than the
    # 512 ranked directly: bitonic sort) and the cut is exact
    V = 65536
    w = gen.make_workload(2, 1, V, "bf16", T=1.0, top_p=0.5001, k=64, seed=51)
    counters, res = _run(A, orc, w, _tied_top(V, 700, 51))
    assert counters[FALLBACK] == 0 and counters[BITONIC] == 4 and counters[LAZY] == 0, counters
    assert res["checked_seqs"] == 2


def test_payload_ties_beyond_the_candidate_area_fall_back(A, orc):
    # 1500 ids tied at the payload's last value: more than the 1024 that the
    # re-read keeps, so the exact general kernel takes the rows
    V = 65536
    w = gen.make_workload(2, 1, V, "bf16", T=1.0, top_p=0.5001, k=64, seed=52)
    counters, res = _run(A, orc, w, _tied_top(V, 1500, 52))
    assert counters[FALLBACK] == 4, counters
    assert res["checked_seqs"] == 2


def test_bitonic_order_for_many_candidates(A, orc):
    # 1500 near-equal float32 ids spread over the row, the rest far below:
    # the list holds them all and the nucleus (~1200 ids) is ordered by
    # bitonic sort
    V = 32000
    w = gen.make_workload(2, 2, V, "f32", T=1.0, top_p=0.8, k=64, seed=31)
    rng = np.random.default_rng(31)
    z = np.full((2, 3, V), -30.0, np.float32)
    ids = np.arange(1500) * 21
    z[:, :, ids] = rng.uniform(0.0, 0.5, size=(2, 3, 1500)).astype(np.float32)
    counters, res = _run(A, orc, w, z)
    assert counters[FALLBACK] == 0 and counters[BITONIC] == 6, counters
    assert res["checked_seqs"] == 2


def test_more_candidates_than_the_list_falls_back(A, orc):
    # 5000 near-equal float32 ids, each in its own chunk: the capture
    # exceeds the 3584 records of a one-wave launch (1536 in larger ones),
    # so every row goes to the exact general kernel
    V = 128000
    w = gen.make_workload(2, 1, V, "f32", T=1.0, top_p=0.8, k=32, seed=32)
    rng = np.random.default_rng(32)
    z = np.full((2, 2, V), -30.0, np.float32)
    ids = np.arange(5000) * 21
    z[:, :, ids] = rng.uniform(0.0, 0.5, size=(2, 2, 5000)).astype(np.float32)
    counters, res = _run(A, orc, w, z)
    assert counters[FALLBACK] == 4, counters
    assert res["checked_seqs"] == 2


def test_a_misleading_sample_is_still_counted(A, orc):
    # the sampled tiles hold 300 ids near 10 and nothing else; the rest of
    # the row holds 20000 ids at 5, which carry most of the mass.  The counts
    # reach 10 T below the running max, so the crossing is found on chip
    V = 65536
    w = gen.make_workload(2, 1, V, "bf16", T=1.0, top_p=0.9, k=16, seed=47)
    rng = np.random.default_rng(47)
    samp = _sampled_ids(V, "bf16")
    rest = np.setdiff1d(np.arange(V), samp)
    z = np.full((2, 2, V), -30.0, np.float32)
    for b in range(2):
        for i in range(2):
            z[b, i, rng.choice(samp, 300, replace=False)] = rng.uniform(9.8, 10.0, 300)
            z[b, i, rng.choice(rest, 20000, replace=False)] = 5.0
    counters, res = _run(A, orc, w, _bf16(z))
    assert counters[FALLBACK] == 0 and counters[VALUE_MODE] == 4, counters
    assert res["checked_seqs"] >= 1


def test_crossing_below_the_counted_values_is_counted_again(A, orc):
    # one id at 16 and 60000 ids at 5 (T = 1) carry about equal mass, so the
    # top_p = 0.9 crossing lies 11 T below the max, beyond D = 10 T: a second
    # pass counts the row from its max down and finds it (k = 1: the payload
    # is the top id, the crossing value's ids are left to the resolve step)
    V = 65536
    w = gen.make_workload(2, 1, V, "bf16", T=1.0, top_p=0.9, k=1, seed=53)
    rng = np.random.default_rng(53)
    z = np.full((2, 2, V), -30.0, np.float32)
    for b in range(2):
        for i in range(2):
            z[b, i, rng.choice(V, 60000, replace=False)] = 5.0
            z[b, i, rng.integers(V)] = 16.0
    counters, res = _run(A, orc, w, _bf16(z))
    assert counters[FALLBACK] == 0 and counters[RECOUNT] == 4 and counters[LAZY] == 4, counters
    assert res["checked_seqs"] >= 1


def test_a_max_above_the_value_window_is_counted_again(A, orc):
    # flat rows in [2, 3] with one id at 1000 outside the sample: it lies
    # beyond the 1024 counted values (at most 767 below the sample's max);
    # the second pass anchors the window at the row max
    V = 65536
    w = gen.make_workload(2, 1, V, "bf16", T=1.0, top_p=0.9, k=16, seed=48)
    rng = np.random.default_rng(48)
    samp = set(_sampled_ids(V, "bf16").tolist())
    far = next(x for x in range(V - 1, 0, -1) if x not in samp)
    z = rng.uniform(2.0, 3.0, size=(2, 2, V)).astype(np.float32)
    z[:, :, far] = 1000.0
    counters, res = _run(A, orc, w, _bf16(z))
    assert counters[FALLBACK] == 0 and counters[RECOUNT] == 4, counters
    assert res["checked_seqs"] >= 1


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_later_rows_take_their_depth_from_finished_rows(A, orc, dtype):
    # 1088 rows, more than run at once: rows that start after 32 have
    # finished take D from those rows' depths (bf16: the counts' lower end;
    # float32: the capture threshold, running max - D).  Shapes of the
    # 128256-id and of the 32000-id float32 workloads.
    if dtype == "bf16":
        w = gen.make_workload(96, 16, 128256, "bf16", sigma=3.0, rho=0.5, T=1.0, top_p=0.9, k=32, seed=54)
    else:
        w = gen.make_workload(64, 16, 32000, "f32", sigma=3.0, rho=0.8, T=0.8, top_p=0.9, k=32, seed=54)
    inp = gen.generate(w)
    counters, res = _run(A, orc, w, inp["z"], inp=dict(inp))
    # (float32 rows whose capture overflows the 1536 recorded chunks go to
    # the exact general kernel)
    assert counters[HINTED] >= 200 and counters[FALLBACK] <= (8 if dtype == "bf16" else 200), counters
    assert res["checked_seqs"] >= 32


def test_short_rows_lead_later_rows_to_the_sketch(A, orc):
    # 1088 rows shaped like the 256000-id workload (T = 0.6, top_p = 0.8,
    # k = 128: nuclei of tens of ids).  Once 32 rows have finished, all of
    # them short, later rows stream without counting and read back only the
    # sketch groups that can hold the nucleus.
    w = gen.make_workload(64, 16, 256000, "bf16", sigma=3.0, rho=0.9, T=0.6, top_p=0.8, k=128, seed=57)
    inp = gen.generate(w)
    counters, res = _run(A, orc, w, inp["z"], inp=dict(inp))
    assert counters[FALLBACK] == 0 and counters[SHORT] >= 200 and counters[SKETCH_LED] >= 200, counters
    assert res["checked_seqs"] >= 32


def _verify_ws(A, w, inp, ws):
    zt = torch.from_numpy(inp["z"].view(np.int16)).cuda().view(torch.bfloat16)
    q, xt, u = (torch.from_numpy(inp[key]).cuda() for key in ("q", "xt", "u"))
    g = A.verify(zt, q, xt, u, w.T, w.top_p, w.k, workspace=ws)
    torch.cuda.synchronize()
    counters = ws[A.COUNTERS_OFFSET:A.COUNTERS_OFFSET + 64].view(torch.int32).cpu().numpy().tolist()
    return {key: v.cpu().numpy() for key, v in g.items()}, counters


def test_hints_carried_to_the_next_call_change_no_result(A, orc):
    # 680 rows shaped like the 256000-id workload, twice on one workspace:
    # the first call's first wave has no hints; the second call takes the
    # first call's from the workspace, so all its rows are hinted and nearly
    # all take the sketch-led pass.  Hints choose a pass only: the same bits, the
    # oracle's results.  A workspace whose hint area holds another call's
    # hints or noise gives the same bits too.
    w = gen.make_workload(40, 16, 256000, "bf16", sigma=3.0, rho=0.9, T=0.6, top_p=0.8, k=128, seed=61)
    inp = dict(gen.generate(w))
    rows = w.B * (w.K + 1)
    ws = torch.zeros(A.workspace_bytes(w.B, w.K, w.V, w.k), dtype=torch.uint8, device="cuda")
    g1, c1 = _verify_ws(A, w, inp, ws)
    g2, c2 = _verify_ws(A, w, inp, ws)
    # (a few rows start while this call's own first rows say that fewer than
    # 98% were short, and count instead)
    assert c1[HINTED] < rows and c2[HINTED] == rows and c2[SKETCH_LED] >= rows - rows // 32, (c1, c2)
    assert c2[SKETCH_LED] > c1[SKETCH_LED], (c1, c2)
    for key in g1:
        assert np.array_equal(g1[key], g2[key]), key
    o = orc.verify(inp["z"], inp["q"], inp["xt"], inp["u"], w.T, w.top_p, w.k)
    res = parity.compare_verify(inp, g2, o, w.top_p, True, w.k)
    assert res["checked_seqs"] >= 32
    # another call's hints (another top_p) and then noise in the hint area
    w2 = gen.make_workload(40, 16, 256000, "bf16", sigma=3.0, rho=0.9, T=0.6, top_p=0.5, k=128, seed=61)
    _verify_ws(A, w2, inp, ws)
    g3, c3 = _verify_ws(A, w, inp, ws)
    assert c3[HINTED] < rows, c3
    ws[:256] = torch.randint(0, 256, (256,), dtype=torch.uint8, device="cuda")
    g4, _ = _verify_ws(A, w, inp, ws)
    for key in g1:
        assert np.array_equal(g1[key], g3[key]) and np.array_equal(g1[key], g4[key]), key


def test_sketch_led_row_with_a_long_nucleus_counts_again(A, orc):
    # The first 800 rows have four dominant ids (short nuclei), the last
    # 288 flat logits (nuclei of most of the row).  Rows that start after
    # the short ones finished take the sketch-led pass; for the flat ones
    # the groups it marks do not hold the crossing, and the row is counted
    # in a second pass instead.
    B, K, V = 64, 16, 32768
    w = gen.make_workload(B, K, V, "bf16", T=1.0, top_p=0.9, k=16, seed=58)
    rng = np.random.default_rng(58)
    rows = B * (K + 1)
    z = rng.uniform(0.0, 1.0, size=(rows, V)).astype(np.float32)
    for r in range(800):
        z[r, rng.choice(V, 4, replace=False)] = 12.0 + rng.uniform(0.0, 0.5, 4)
    counters, res = _run(A, orc, w, _bf16(z.reshape(B, K + 1, V)))
    assert counters[FALLBACK] == 0 and counters[SKETCH_LED] >= 100 and counters[RECOUNT] >= 1, counters
    assert res["checked_seqs"] >= 32


@pytest.mark.parametrize("dtype,V", [("bf16", 600000), ("bf16", 1 << 20), ("f32", 300000), ("f32", 1 << 20)],
                         ids=["bf16_600k", "bf16_1m", "f32_300k", "f32_1m"])
def test_large_vocabularies(A, orc, dtype, V):
    w = gen.make_workload(4, 1, V, dtype, T=0.8, top_p=0.9, k=48, seed=34)
    z = gen.generate(w)["z"]
    counters, res = _run(A, orc, w, z)
    assert counters[TIMEOUTS] == 0
    assert res["checked_seqs"] >= 1


# ---------------------------------------------------------------------------
# the exact general kernel (every row handed over: aces_verify_exact)


def test_general_value_histogram_takes_large_nucleus_bf16_rows(A, orc):
    w = gen.make_workload(2, 2, 128256, "bf16", sigma=3.0, rho=0.5, T=1.0, top_p=0.9, k=32, seed=41)
    z = gen.generate(w)["z"]
    counters, res = _run(A, orc, w, z, exact=True)
    assert counters[FALLBACK] == 6 and counters[GEN_VALHIST] == 6 and counters[RADIX] == 0, counters
    assert res["checked_seqs"] >= 1


def test_general_value_histogram_declines_a_crossing_below_its_window(A, orc):
    # flat rows (T=2, top_p=0.99): the crossing lies among negative logits,
    # whose keys are below the window (below every tiny positive value); the
    # binned path takes the rows
    w = gen.make_workload(3, 2, 65536, "bf16", T=2.0, top_p=0.99, k=64, seed=41)
    z = gen.generate(w)["z"]
    counters, res = _run(A, orc, w, z, exact=True)
    assert counters[FALLBACK] == 9 and counters[GEN_VALHIST] == 0, counters


@pytest.mark.parametrize("n_vals,V,expect_valhist", [(40, 32000, True), (24, 65536, False)],
                         ids=["ties_within_capacity", "ties_beyond_capacity"])
def test_general_value_histogram_ties(A, orc, n_vals, V, expect_valhist):
    # logits from a few distinct bf16 values: the crossing value is shared by
    # ~V/n_vals ids, taken in id order.  Up to 1024 of them the value
    # histogram orders them itself; beyond that the binned path takes the row.
    w = gen.make_workload(2, 2, V, "bf16", T=1.0, top_p=0.7, k=32, seed=42)
    rng = np.random.default_rng(42)
    vals = np.linspace(-2.0, 2.0, n_vals).astype(np.float32)
    z = _bf16(vals[rng.integers(0, n_vals, size=(2, 3, V))])
    counters, res = _run(A, orc, w, z, exact=True)
    assert counters[FALLBACK] == 6, counters
    assert (counters[GEN_VALHIST] == 6) if expect_valhist else (counters[GEN_VALHIST] == 0), counters
    assert res["checked_seqs"] >= 1


def test_ties_on_the_single_pass_kernel(A, orc):
    # the same few-valued rows on aces_verify: whatever the kernel decides,
    # ids of the crossing value are taken in id order
    w = gen.make_workload(2, 2, 32000, "bf16", T=1.0, top_p=0.7, k=32, seed=42)
    rng = np.random.default_rng(42)
    vals = np.linspace(-2.0, 2.0, 40).astype(np.float32)
    z = _bf16(vals[rng.integers(0, 40, size=(2, 3, 32000))])
    counters, res = _run(A, orc, w, z)
    assert res["checked_seqs"] >= 1


def test_general_value_histogram_top_p_one_rows(A, orc):
    # top_p = 1 on bf16 rows: 3000 ids with values in [1, 1.05] (seven bf16
    # values), the rest at -30.  The value histogram counts the finite ids
    # itself (the whole row is the nucleus) and takes the payload, ties in id
    # order, from the top value.
    V, n_hot = 64000, 3000
    w = gen.make_workload(2, 1, V, "bf16", T=1.0, top_p=1.0, k=64, seed=44)
    rng = np.random.default_rng(44)
    z = np.full((2, 2, V), -30.0, np.float32)
    j = np.arange(n_hot)
    ids = j * 16 + (j % 16)
    for b in range(2):
        for i in range(2):
            z[b, i, ids] = rng.uniform(1.0, 1.05, n_hot).astype(np.float32)
    counters, res = _run(A, orc, w, _bf16(z), exact=True)
    assert counters[FALLBACK] == 4 and counters[GEN_VALHIST] == 4 and counters[RADIX] == 0, counters
    assert res["checked_seqs"] >= 1
    # and on aces_verify
    counters, res = _run(A, orc, w, _bf16(z))
    assert res["checked_seqs"] >= 1


def test_signed_zeros_on_the_general_path(A, orc):
    # -0 and +0 are one value (one order key): the nucleus and the payload take
    # them in id order whatever their signs.  Ten positive ids, then a run of
    # 512 zeros of random sign, the rest at -20.  Zero lies ~16000 bf16 keys
    # below a max near 1, beyond the value histogram's window, so the binned
    # path takes the rows.
    V = 32000
    w = gen.make_workload(2, 1, V, "bf16", T=1.0, top_p=0.999, k=64, seed=43)
    rng = np.random.default_rng(43)
    z = np.full((2, 2, V), -20.0, np.float32)
    z[:, :, 100:110] = rng.uniform(0.5, 1.0, size=(2, 2, 10)).astype(np.float32)
    z[:, :, 1024:1536] = np.where(rng.random((2, 2, 512)) < 0.5, np.float32(0.0), np.float32(-0.0))
    counters, res = _run(A, orc, w, _bf16(z), exact=True)
    assert counters[FALLBACK] == 4 and counters[GEN_VALHIST] == 0, counters
    assert res["checked_seqs"] >= 1
    # and on aces_verify (the list holds the zeros)
    counters, res = _run(A, orc, w, _bf16(z))
    assert res["checked_seqs"] >= 1


def test_general_radix_path(A, orc):
    # float32 rows of 5000 tied ids at 0 (the rest at -30), top_p = 0.5001
    # (the crossing, 2501 ids in, is 1e-4 from it: not flagged): the crossing
    # bin holds more ids than the binned path collects (2048), so the radix
    # selection finishes the rows; ties go by id
    V = 32768
    w = gen.make_workload(2, 1, V, "f32", T=1.0, top_p=0.5001, k=16, seed=49)
    rng = np.random.default_rng(49)
    z = np.full((2, 2, V), -30.0, np.float32)
    for b in range(2):
        for i in range(2):
            z[b, i, rng.choice(V, 5000, replace=False)] = 0.0
    counters, res = _run(A, orc, w, z, exact=True)
    assert counters[FALLBACK] == 4 and counters[RADIX] >= 1, counters
    assert res["checked_seqs"] >= 1
