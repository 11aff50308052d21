"""Parity of aces_resample_sparse (the edge's draw from the sparse payload,
Alg. 1 RESAMPLE) with the float64 oracle.

Both sides get the same inputs: the oracle's own verification of a seeded
workload (its accept lengths, row status and payload, the payload cast to
float32) plus the draft rows and uniforms.  Tokens and status must match
exactly, except for sequences whose draw lies within 1e-6 of the total of a
prefix-sum boundary (tests/parity.py's residual rule).
"""
import dataclasses

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


def _oracle_payload(orc, inp, w, k):
    ov = orc.verify(inp["z"], inp["q"], inp["xt"], inp["u"], w.T, w.top_p, k)
    return dict(accept_len=ov["accept_len"].astype(np.int32), ids=ov["topk_ids"].astype(np.int32),
                probs=ov["topk_probs"].astype(np.float32), tail=ov["tail"].astype(np.float32),
                row_status=ov["row_status"].astype(np.int32)), ov


def _both(A, orc, pay, q, u):
    o = orc.resample_sparse(pay["accept_len"], pay["ids"], pay["probs"], pay["tail"], pay["row_status"], q, u)
    d = {key: torch.from_numpy(np.ascontiguousarray(v)).cuda() for key, v in pay.items()}
    g = A.resample_sparse(d["accept_len"], d["ids"], d["probs"], d["tail"], d["row_status"],
                          torch.from_numpy(q).cuda(), torch.from_numpy(u).cuda())
    torch.cuda.synchronize()
    return {key: v.cpu().numpy() for key, v in g.items()}, o


def _compare(g, o):
    B = len(o["token"])
    np.testing.assert_array_equal(g["status"], o["status"])
    checked = 0
    for b in range(B):
        s, t = o["res_sum"][b], o["res_target"][b]
        if np.isfinite(s) and any(np.isfinite(c) and abs(t - c) < 1e-6 * s
                                  for c in (o["res_cj"][b], o["res_cjm1"][b])):
            continue
        assert g["token"][b] == o["token"][b], f"seq {b}: gpu {g['token'][b]} oracle {o['token'][b]}"
        checked += 1
    return checked


@pytest.mark.parametrize("name,k", [("b16_k8_v32000_f32", 4), ("b16_k8_v32000_f32", 32),
                                    ("b16_k8_v32000_f32", 256), ("b1_k4_v32000_f32", 16)])
def test_resample_matches_oracle(A, orc, name, k):
    w = gen.WORKLOADS[name]
    inp = gen.generate(w)
    pay, ov = _oracle_payload(orc, inp, w, k)
    g, o = _both(A, orc, pay, inp["q"], inp["u"])
    assert _compare(g, o) >= w.B - 1
    if k == 4:
        assert (pay["tail"][np.arange(w.B), pay["accept_len"]] > 0).any()   # the spread path ran


def test_resample_bf16_workload_sampled(A, orc):
    # sequences of the 152064-id Zipf-head workload, small payload: the tail
    # is spread over the whole vocabulary
    w = dataclasses.replace(gen.WORKLOADS["b64_k8_v152064_bf16"], B=12)
    inp = gen.generate(w)
    pay, ov = _oracle_payload(orc, inp, w, 8)
    g, o = _both(A, orc, pay, inp["q"], inp["u"])
    assert _compare(g, o) >= w.B - 1


def test_resample_equals_exact_draw_when_nucleus_fits(A):
    # GPU verify then GPU resample with k covering every nucleus: the edge's
    # token is the cloud's exact residual token
    w = dataclasses.replace(gen.WORKLOADS["b256_k16_v256000_bf16"], B=32)
    inp = gen.generate(w)
    z = torch.from_numpy(inp["z"].view(np.int16)).cuda().view(torch.bfloat16)
    q, xt, u = (torch.from_numpy(inp[key]).cuda() for key in ("q", "xt", "u"))
    out = A.verify(z, q, xt, u, w.T, w.top_p, 256)
    g = A.resample_sparse(out["accept_len"], out["topk_ids"], out["topk_probs"], out["tail_mass"],
                          out["row_status"], q, u)
    torch.cuda.synchronize()
    tail_pi = out["tail_mass"][torch.arange(w.B, device="cuda"), out["accept_len"].long()]
    fits = (tail_pi == 0).cpu().numpy()
    assert fits.sum() >= w.B - 2
    same = (g["token"] == out["out_token"]).cpu().numpy()
    assert same[fits].mean() >= 0.95, same[fits].mean()


def test_resample_degenerate_rows(A, orc):
    w = gen.make_workload(6, 2, 3000, "f32", T=1.0, top_p=0.9, k=6, seed=51)
    inp = gen.generate(w)
    pay, ov = _oracle_payload(orc, inp, w, 6)
    q = inp["q"].copy()
    al = pay["accept_len"].copy()
    al[0] = 2                                        # bonus row: payload alone
    pay["row_status"][1, al[1]] |= 1                 # row pi NONFINITE
    pay["ids"][2, al[2]] = -1                        # empty payload
    if al[3] < 2:
        q[3, al[3], pay["ids"][3, al[3], 0]] = -0.5  # negative q on the payload
    if al[4] < 2:
        pay["tail"][4, al[4]] = 0.5                  # tail spread: reads all of q ...
        q[4, al[4], (pay["ids"][4, al[4], 0] + 1) % w.V] = np.nan   # ... and meets a NaN
    pay["accept_len"] = al
    g, o = _both(A, orc, pay, q, inp["u"])
    _compare(g, o)
    assert g["status"][1] == 1 and g["token"][1] == -1
    assert g["token"][2] == -1
    if al[3] < 2:
        assert g["status"][3] == 2 and g["token"][3] == -1
    if al[4] < 2:
        assert g["status"][4] == 2 and g["token"][4] == -1
