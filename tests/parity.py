"""Comparison of the CUDA path's outputs with the float64 oracle.

Tolerances and flag rules:
  * accepted lengths, emitted tokens, payload ids, branch ids, slots and row
    status bits must be bit-exact;
  * a sequence is flagged (its accept_len / out_token are only checked for
    validity) when, at some row i <= pi (oracle), |u_i - p/q| < 1e-5, when
    the residual draw is within 1e-6 * sum(r) of a prefix-sum boundary
    (|u_K sum r - C_j| or |u_K sum r - C_{j-1}|), or when a row i <= pi has
    a flagged nucleus;
  * a row's nucleus is flagged when its cumulative mass before or at the
    crossing id is within 1e-6 of top_p (membership and payload ids then
    are only checked for validity);
  * probabilities: 1e-5 absolute for float32 logits, 2e-3 relative for
    bfloat16 logits (tail mass: 1e-5 absolute, or 2e-3 relative / 1e-6
    absolute for bfloat16).
"""
from __future__ import annotations

import numpy as np

ACCEPT_FLAG = 1e-5
MASS_FLAG = 1e-6
RESID_FLAG = 1e-6


def nucleus_flags(orc_out, top_p):
    cp, ca = orc_out["cum_prev"], orc_out["cum_at"]
    if top_p >= 1.0:
        return np.zeros(cp.shape, bool)
    with np.errstate(invalid="ignore"):
        return (np.abs(cp - top_p) < MASS_FLAG) | (np.abs(ca - top_p) < MASS_FLAG)


def sequence_flags(inp, orc_out, top_p):
    u = inp["u"].astype(np.float64)
    B, R = u.shape
    K = R - 1
    pi = orc_out["accept_len"]
    nflag = nucleus_flags(orc_out, top_p)
    flags = np.zeros(B, bool)
    for b in range(B):
        for i in range(min(pi[b], K - 1) + 1 if K > 0 else 0):
            if abs(u[b, i] - orc_out["ratio"][b, i]) < ACCEPT_FLAG:
                flags[b] = True
        if nflag[b, : pi[b] + 1].any():
            flags[b] = True
        s = orc_out["res_sum"][b]
        if np.isfinite(s):
            t = orc_out["res_target"][b]
            for c in (orc_out["res_cj"][b], orc_out["res_cjm1"][b]):
                if np.isfinite(c) and abs(t - c) < RESID_FLAG * s:
                    flags[b] = True
    return flags


def _prob_close(got, ref, bf16):
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    if bf16:
        return np.abs(got - ref) <= 2e-3 * np.abs(ref) + 1e-12
    return np.abs(got - ref) <= 1e-5


def compare_payload(gpu, orc_out, top_p, bf16, rows_mask=None):
    """Returns a dict of counts; raises AssertionError on a mismatch."""
    gid = gpu["topk_ids"].reshape(-1, gpu["topk_ids"].shape[-1])
    gp = gpu["topk_probs"].reshape(gid.shape)
    gt = gpu["tail_mass"].reshape(-1)
    oid = orc_out["topk_ids"].reshape(gid.shape)
    op = orc_out["topk_probs"].reshape(gid.shape)
    ot = orc_out["tail"].reshape(-1)
    st = orc_out["row_status"].reshape(-1)
    nflag = nucleus_flags(orc_out, top_p).reshape(-1)
    n_flag = 0
    worst = 0.0
    for r in range(gid.shape[0]):
        if rows_mask is not None and not rows_mask[r]:
            continue
        if st[r] & 1:
            assert (gid[r] == -1).all() and (gp[r] == 0).all(), f"row {r}: NONFINITE payload"
            continue
        if nflag[r]:
            n_flag += 1
            valid = gid[r][gid[r] >= 0]
            assert len(set(valid.tolist())) == len(valid), f"row {r}: duplicate ids"
            continue
        if not np.array_equal(gid[r], oid[r]):
            bad = np.nonzero(gid[r] != oid[r])[0][:5]
            raise AssertionError(f"row {r}: payload ids differ at {bad}: gpu {gid[r][bad]} oracle {oid[r][bad]}")
        ok = _prob_close(gp[r], op[r], bf16)
        assert ok.all(), f"row {r}: payload probs differ: {gp[r][~ok][:4]} vs {op[r][~ok][:4]}"
        worst = max(worst, float(np.max(np.abs(gp[r] - op[r]))))
        tol = max(2e-3 * abs(ot[r]), 1e-6) if bf16 else 1e-5
        assert abs(gt[r] - ot[r]) <= tol, f"row {r}: tail {gt[r]} vs {ot[r]}"
    return dict(flagged_rows=n_flag, max_prob_err=worst)


def compare_verify(inp, gpu, orc_out, top_p, bf16, k):
    """Bit-exact accept_len / out_token / row_status on unflagged sequences,
    payload per compare_payload."""
    B = inp["u"].shape[0]
    K = inp["u"].shape[1] - 1
    V = inp["q"].shape[-1] if inp["q"].ndim == 3 else None
    flags = sequence_flags(inp, orc_out, top_p)
    al, tok = gpu["accept_len"], gpu["out_token"]
    assert ((al >= 0) & (al <= K)).all()
    n_checked = 0
    for b in range(B):
        if flags[b]:
            continue
        n_checked += 1
        assert al[b] == orc_out["accept_len"][b], \
            f"seq {b}: accept_len {al[b]} vs oracle {orc_out['accept_len'][b]}"
        assert tok[b] == orc_out["out_token"][b], \
            f"seq {b}: out_token {tok[b]} vs oracle {orc_out['out_token'][b]} (pi={al[b]})"
    # row status: exact except rows after a flagged sequence's divergence
    gst = gpu["row_status"].reshape(B, K + 1)
    ost = orc_out["row_status"].reshape(B, K + 1)
    for b in range(B):
        if flags[b]:
            continue
        # the BAD_Q bit of the residual row is only known to the side that drew it
        assert np.array_equal(gst[b], ost[b]), f"seq {b}: row_status {gst[b]} vs {ost[b]}"
    res = dict(flagged_seqs=int(flags.sum()), checked_seqs=n_checked)
    if k > 0:
        res.update(compare_payload(gpu, orc_out, top_p, bf16))
    if V is not None:
        res["V"] = V
    return res


def compare_cache(gpu_bt, gpu_bp, orc_bt, orc_bp):
    np.testing.assert_array_equal(gpu_bt, orc_bt)
    assert np.all(np.abs(gpu_bp.astype(np.float64) - orc_bp) <= 1e-5), \
        float(np.max(np.abs(gpu_bp - orc_bp)))
