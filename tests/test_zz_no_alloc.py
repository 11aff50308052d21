"""aces_verify_noalloc: verification for callers that cannot allocate.

Some callers have no device allocator on their serving path (cudaMalloc
synchronizes the whole device; some embedding runtimes own all device
memory), so they cannot pass aces_verify a workspace.  aces_verify_noalloc
runs the same kernels on a fixed scratch array inside the library.  These
tests call it through the C ABI and check that two calls in a row give the
same results as aces_verify on the same inputs, with the tolerances the
parity tests use (exact for ids, lengths, tokens and status; probabilities
1e-5 absolute for float32 logits, 2e-3 relative for bfloat16).

This file is collected last so that a run stopping at the first failure has
already run every other test; it also passes on its own in a fresh process.
"""
import ctypes

import numpy as np
import pytest

import gen

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

SCRATCH_BYTES = 1 << 20   # ACES_NOALLOC_SCRATCH_BYTES in include/acespec.h


@pytest.fixture(scope="module")
def lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_02514_gb300 as A
    lib = A.load()
    P, I, F = ctypes.c_void_p, ctypes.c_int, ctypes.c_float
    lib.aces_verify_noalloc.argtypes = [P, I, P, P, P, I, I, I, F, F, P, P, I, P, P, P, P, P]
    lib.aces_verify_noalloc.restype = I
    return lib


def _inputs(w):
    d = gen.generate(w)
    if w.dtype == "bf16":
        z = torch.from_numpy(d["z"].view(np.int16)).cuda().view(torch.bfloat16)
    else:
        z = torch.from_numpy(d["z"]).cuda()
    return z, torch.from_numpy(d["q"]).cuda(), torch.from_numpy(d["xt"]).cuda(), torch.from_numpy(d["u"]).cuda()


def _outputs(B, K, k):
    i32 = dict(dtype=torch.int32, device="cuda")
    return dict(accept_len=torch.full((B,), -7, **i32), out_token=torch.full((B,), -7, **i32),
                row_status=torch.full((B, K + 1), -7, **i32), topk_ids=torch.full((B, K + 1, k), -7, **i32),
                topk_probs=torch.full((B, K + 1, k), -7.0, device="cuda"),
                tail_mass=torch.full((B, K + 1), -7.0, device="cuda"))


def _p(t):
    return ctypes.c_void_p(t.data_ptr())


def _noalloc(lib, z, q, xt, u, w, k, o):
    B, R, V = z.shape
    dt = 1 if z.dtype == torch.bfloat16 else 0
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    return lib.aces_verify_noalloc(_p(z), dt, _p(q), _p(xt), _p(u), B, R - 1, V, w.T, w.top_p,
                                   _p(o["accept_len"]), _p(o["out_token"]), k, _p(o["topk_ids"]),
                                   _p(o["topk_probs"]), _p(o["tail_mass"]), _p(o["row_status"]), stream)


def _compare(got, ref, bf16):
    for key in ("accept_len", "out_token", "row_status", "topk_ids"):
        np.testing.assert_array_equal(got[key].cpu().numpy(), ref[key].cpu().numpy(), err_msg=key)
    for key in ("topk_probs", "tail_mass"):
        g = got[key].cpu().numpy().astype(np.float64)
        r = ref[key].cpu().numpy().astype(np.float64)
        if bf16:
            assert np.all(np.abs(g - r) <= 2e-3 * np.abs(r) + 1e-12), key
        else:
            assert np.all(np.abs(g - r) <= 1e-5), key


def test_two_calls_in_a_row_match_aces_verify(lib):
    import paper_2609_02514_gb300 as A
    cases = [gen.make_workload(12, 8, 32000, "bf16", T=0.8, top_p=0.9, k=32, seed=41),
             gen.make_workload(5, 16, 20000, "f32", T=1.0, top_p=1.0, k=64, seed=42)]
    for w in cases:          # two calls in a row, on different shapes and inputs
        z, q, xt, u = _inputs(w)
        ref = A.verify(z, q, xt, u, w.T, w.top_p, w.k)
        got = _outputs(w.B, w.K, w.k)
        assert _noalloc(lib, z, q, xt, u, w, w.k, got) == 0
        torch.cuda.synchronize()
        _compare(got, ref, w.dtype == "bf16")


def test_same_inputs_twice_give_identical_outputs(lib):
    w = gen.make_workload(8, 4, 40000, "bf16", T=0.7, top_p=0.95, k=16, seed=43)
    z, q, xt, u = _inputs(w)
    first = _outputs(w.B, w.K, w.k)
    second = _outputs(w.B, w.K, w.k)
    assert _noalloc(lib, z, q, xt, u, w, w.k, first) == 0
    assert _noalloc(lib, z, q, xt, u, w, w.k, second) == 0
    torch.cuda.synchronize()
    for key in first:
        np.testing.assert_array_equal(first[key].cpu().numpy(), second[key].cpu().numpy(), err_msg=key)


def test_largest_batch_runs_without_nucleus_lists(lib):
    # B = 876 at K = 16 is the largest batch the scratch holds; its residual
    # draws scan whole rows, aces_verify's use the stored nucleus lists.
    import paper_2609_02514_gb300 as A
    w = gen.make_workload(876, 16, 1000, "f32", T=1.0, top_p=0.6, k=8, seed=44)
    assert A.workspace_bytes(w.B, w.K, w.V, w.k) > SCRATCH_BYTES
    z, q, xt, u = _inputs(w)
    ref = A.verify(z, q, xt, u, w.T, w.top_p, w.k)
    got = _outputs(w.B, w.K, w.k)
    assert _noalloc(lib, z, q, xt, u, w, w.k, got) == 0
    torch.cuda.synchronize()
    _compare(got, ref, False)


def test_batch_beyond_the_scratch_is_rejected(lib):
    B, K, V, k = 877, 16, 1000, 8          # needs more than ACES_NOALLOC_SCRATCH_BYTES
    z = torch.zeros(B, K + 1, V, device="cuda")
    q = torch.full((B, K, V), 1.0 / V, device="cuda")
    xt = torch.zeros(B, K, dtype=torch.int32, device="cuda")
    u = torch.full((B, K + 1), 0.5, device="cuda")
    o = _outputs(B, K, k)
    w = gen.make_workload(B, K, V, "f32", T=1.0, top_p=0.9, k=k)
    assert _noalloc(lib, z, q, xt, u, w, k, o) == 2       # ACES_ERR_UNSUPPORTED
    torch.cuda.synchronize()
    assert (o["accept_len"] == -7).all()                   # nothing was launched


def test_matches_the_oracle(lib, orc):
    # one case compared with the float64 oracle directly (the other tests
    # compare with aces_verify, itself compared with the oracle elsewhere)
    from tests import parity
    w = gen.make_workload(6, 8, 32000, "bf16", T=0.8, top_p=0.9, k=32, seed=45)
    d = gen.generate(w)
    z, q, xt, u = _inputs(w)
    got = _outputs(w.B, w.K, w.k)
    assert _noalloc(lib, z, q, xt, u, w, w.k, got) == 0
    torch.cuda.synchronize()
    g = {key: v.cpu().numpy() for key, v in got.items()}
    o = orc.verify(d["z"], d["q"], d["xt"], d["u"], w.T, w.top_p, w.k)
    res = parity.compare_verify(d, g, o, w.top_p, True, w.k)
    assert res["checked_seqs"] >= w.B - 1, res
