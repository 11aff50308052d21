"""Writes tests/golden/sparse_resample_tv.txt: how far the edge's draw from the
sparse payload (Alg. 1 RESAMPLE) is from the exact residual draw, as a
function of the payload size k.

For the first 8 sequences of three seeded workloads and each k, the oracle
verifies the sequences, draws from the payload of row pi (orc_resample_sparse)
and compares the distribution it drew from with the exact one,
norm(max(0, p_pi - q_pi)) (p_K for the bonus row).  Each line: workload k
mean_tv max_tv tail_frac token_agree, where tail_frac is the fraction of
sequences whose row pi has a tail above 1e-6 (nucleus larger than k) and
token_agree the fraction whose sparse token equals the exact token.
Calls only the oracle package and the input generator.
"""
import dataclasses
import os
import sys

import numpy as np

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__)))))
import gen  # noqa: E402
from oracle import oracle as O  # noqa: E402

WORKLOADS = ["b16_k8_v32000_f32", "b64_k8_v152064_bf16", "b256_k16_v256000_bf16"]
KS = [1, 4, 16, 64, 128, 256]
NSEQ = 8


def row(name, k, nseq=NSEQ):
    w = dataclasses.replace(gen.WORKLOADS[name], B=nseq)
    inp = gen.generate(w)
    ov = O.verify(inp["z"], inp["q"], inp["xt"], inp["u"], w.T, w.top_p, k)
    os_ = O.resample_sparse(ov["accept_len"], ov["topk_ids"], ov["topk_probs"].astype(np.float32),
                            ov["tail"].astype(np.float32), ov["row_status"], inp["q"], inp["u"])
    p, _ = O.warp(inp["z"], w.T, w.top_p)
    tv, tail_pos, agree = [], 0, 0
    for b in range(nseq):
        pi = int(ov["accept_len"][b])
        r = p[b, pi] - (inp["q"][b, pi].astype(np.float64) if pi < w.K else 0.0)
        r = np.maximum(r, 0.0)
        if r.sum() == 0.0:
            r = p[b, pi]
        tv.append(0.5 * np.abs(os_["dist"][b] - r / r.sum()).sum())
        tail_pos += int(ov["tail"][b, pi] > 1e-6)
        agree += int(os_["token"][b] == ov["out_token"][b])
    return float(np.mean(tv)), float(np.max(tv)), tail_pos / nseq, agree / nseq


def fmt(name, k, vals):
    return f"{name} {k} {vals[0]:.6e} {vals[1]:.6e} {vals[2]:.4f} {vals[3]:.4f}"


if __name__ == "__main__":
    out = os.path.join(os.path.dirname(os.path.abspath(__file__)), "sparse_resample_tv.txt")
    with open(out, "w") as f:
        f.write("# workload k mean_tv max_tv tail_frac token_agree  (first 8 sequences; oracle only)\n")
        for name in WORKLOADS:
            for k in KS:
                f.write(fmt(name, k, row(name, k)) + "\n")
