"""Writes tests/golden/hit_rates.txt: expected cache hit rate of the three tree
shapes of the paper's ablation (single chain, uniform, geometric decay of
Sec. IV-C) on seeded synthetic rows, from the oracle alone.

For each regime (target-draft correlation rho, temperature T) the oracle
verifies 512 sequences of K = 8 drafts over V = 4000 ids, estimates the
acceptance rate alpha, allocates B_alloc branches per shape, builds the
branches and averages the per-sequence hit probability (orc_hit_prob) and
the product form of Sec. IV-C.  Each line: rho T alpha B_alloc shape F
hit_rate product_form.  Calls only the oracle package and the input
generator.
"""
import os
import sys

import numpy as np

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__)))))
import gen  # noqa: E402
from oracle import oracle as O  # noqa: E402

K, V, NSEQ = 8, 4000, 512
REGIMES = [(0.97, 0.6), (0.95, 0.5), (0.9, 1.0)]
BUDGETS = [16, 32]


def rows(rho, T, nseq=NSEQ):
    w = gen.make_workload(nseq, K, V, "f32", rho=rho, T=T, top_p=0.9, k=0, seed=95)
    inp = gen.generate(w)
    ov = O.verify(inp["z"], inp["q"], inp["xt"], inp["u"], w.T, w.top_p, 0)
    alpha = float(np.minimum(1.0, ov["ratio"]).mean())
    out = []
    for b_alloc in BUDGETS:
        shapes = [("single", [0] * K), ("uniform", [b_alloc // K] * K),
                  ("geometric", O.branch_alloc(b_alloc, K, alpha, 1.0)[1])]
        for name, F in shapes:
            bt, _ = O.cache_build(inp["q"], inp["xt"], F)
            hp, pp = O.hit_prob(inp["z"], inp["q"], inp["xt"], w.T, w.top_p, bt, F)
            out.append(f"{rho} {T} {alpha:.4f} {b_alloc} {name} {','.join(str(f) for f in F)} "
                       f"{hp.mean():.4f} {pp.mean():.4f}")
    return out


if __name__ == "__main__":
    path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "hit_rates.txt")
    with open(path, "w") as f:
        f.write("# rho T alpha B_alloc shape F hit_rate product_form  (K=8, V=4000, 512 sequences; oracle only)\n")
        for rho, T in REGIMES:
            for line in rows(rho, T):
                f.write(line + "\n")
