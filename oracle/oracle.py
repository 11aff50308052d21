"""ctypes front end of the float64 CPU oracle (acespec_oracle.c).

TEST INFRASTRUCTURE ONLY: imported by the test suite, the smoke check and the
benchmark's CPU-baseline leg.  The product path never imports this module.

All functions take numpy arrays as produced by the ``gen`` package (bfloat16
logits as uint16 bits, widened here exactly to float32) and return numpy
arrays.  Probabilities come back as float64.
"""
from __future__ import annotations

import ctypes
import os
import shutil
import subprocess
import threading
from math import floor

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "acespec_oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

ROW_NONFINITE = 1
ROW_BAD_Q = 2


def build(force: bool = False) -> str:
    """Compile the oracle with the host C compiler (OpenMP when available)."""
    if not force and os.path.exists(_LIB_PATH) and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC):
        return _LIB_PATH
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        raise RuntimeError("no C compiler found to build the oracle")
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    base = [cc, "-O2", "-std=c11", "-shared", "-fPIC", "-o", tmp, _SRC, "-lm"]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True, capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = ctypes.CDLL(_LIB_PATH)
            P = ctypes.c_void_p
            I = ctypes.c_int
            D = ctypes.c_double
            lib.orc_sparsify.argtypes = [P, I, I, D, D, I, P, P, P, P, P, P, P]
            lib.orc_verify.argtypes = [P, P, P, P, I, I, I, D, D, I, P, P, P, P, P, P, P, P, P, P, P, P, P, P]
            lib.orc_cache_build.argtypes = [P, P, P, I, I, I, P, P]
            lib.orc_cache_lookup.argtypes = [P, P, I, I, P, P, P]
            lib.orc_warp.argtypes = [P, I, I, D, D, P, P]
            lib.orc_hit_prob.argtypes = [P, P, P, I, I, I, D, D, P, P, P, P]
            lib.orc_resample_sparse.argtypes = [P, P, P, P, P, P, P, I, I, I, I, P, P, P, P, P, P, P]
            lib.orc_num_threads.argtypes = []
            lib.orc_set_threads.argtypes = [I]
            for f in (lib.orc_sparsify, lib.orc_verify, lib.orc_cache_build, lib.orc_cache_lookup,
                      lib.orc_num_threads, lib.orc_set_threads):
                f.restype = I
            _lib = lib
    return _lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _logits_f32(z: np.ndarray) -> np.ndarray:
    if z.dtype == np.uint16:   # bfloat16 bits -> float32, exact
        return (z.astype(np.uint32) << 16).view(np.float32)
    return np.ascontiguousarray(z, dtype=np.float32)


def num_threads() -> int:
    return int(_load().orc_num_threads())


def set_threads(n: int) -> int:
    """Threads of the oracle's parallel loops from now on; returns the previous count."""
    return int(_load().orc_set_threads(int(n)))


def sparsify(z, T: float, top_p: float, k: int):
    """Steps 1, 2 and 6 on every row of z [..., V]."""
    lib = _load()
    zf = _logits_f32(z)
    V = zf.shape[-1]
    rows = zf.size // V
    zf = zf.reshape(rows, V)
    ids = np.empty((rows, k), np.int32)
    probs = np.empty((rows, k), np.float64)
    tail = np.empty(rows, np.float64)
    st = np.empty(rows, np.int32)
    cp = np.empty(rows, np.float64)
    ca = np.empty(rows, np.float64)
    nn = np.empty(rows, np.int32)
    if lib.orc_sparsify(_ptr(zf), rows, V, float(T), float(top_p), int(k), _ptr(ids), _ptr(probs),
                        _ptr(tail), _ptr(st), _ptr(cp), _ptr(ca), _ptr(nn)):
        raise MemoryError("oracle allocation failed")
    return dict(topk_ids=ids, topk_probs=probs, tail=tail, row_status=st, cum_prev=cp, cum_at=ca,
                n_nuc=nn)


def verify(z, q, xt, u, T: float, top_p: float, k: int):
    """Steps 1-6 for B sequences: z [B,K+1,V], q [B,K,V], xt [B,K], u [B,K+1]."""
    lib = _load()
    zf = _logits_f32(z)
    B, R, V = zf.shape
    K = R - 1
    q = np.ascontiguousarray(q, dtype=np.float32)
    xt = np.ascontiguousarray(xt, dtype=np.int32)
    u = np.ascontiguousarray(u, dtype=np.float32)
    assert q.shape == (B, K, V) and xt.shape == (B, K) and u.shape == (B, R)
    kk = max(int(k), 0)
    out = dict(
        accept_len=np.empty(B, np.int32), out_token=np.empty(B, np.int32),
        topk_ids=np.empty((B, R, max(kk, 1)), np.int32), topk_probs=np.empty((B, R, max(kk, 1)), np.float64),
        tail=np.empty((B, R), np.float64), row_status=np.empty((B, R), np.int32),
        ratio=np.empty((B, max(K, 1)), np.float64), cum_prev=np.empty((B, R), np.float64),
        cum_at=np.empty((B, R), np.float64), n_nuc=np.empty((B, R), np.int32),
        res_target=np.empty(B, np.float64), res_cj=np.empty(B, np.float64),
        res_cjm1=np.empty(B, np.float64), res_sum=np.empty(B, np.float64))
    o = out
    if lib.orc_verify(_ptr(zf), _ptr(q), _ptr(xt), _ptr(u), B, K, V, float(T), float(top_p), kk,
                      _ptr(o["accept_len"]), _ptr(o["out_token"]), _ptr(o["topk_ids"]),
                      _ptr(o["topk_probs"]), _ptr(o["tail"]), _ptr(o["row_status"]), _ptr(o["ratio"]),
                      _ptr(o["cum_prev"]), _ptr(o["cum_at"]), _ptr(o["n_nuc"]), _ptr(o["res_target"]),
                      _ptr(o["res_cj"]), _ptr(o["res_cjm1"]), _ptr(o["res_sum"])):
        raise MemoryError("oracle allocation failed")
    if kk == 0:
        for key in ("topk_ids", "topk_probs", "tail"):
            out.pop(key)
    return out


def cache_build(q, xt, F):
    """Step 7: q [B,K,V], xt [B,K], F [K] -> branch_tok, branch_prob [B, sum F]."""
    lib = _load()
    q = np.ascontiguousarray(q, dtype=np.float32)
    xt = np.ascontiguousarray(xt, dtype=np.int32)
    F = np.ascontiguousarray(F, dtype=np.int32)
    B, K, V = q.shape
    tot = int(F.sum())
    bt = np.empty((B, max(tot, 1)), np.int32)
    bp = np.empty((B, max(tot, 1)), np.float64)
    if lib.orc_cache_build(_ptr(q), _ptr(xt), _ptr(F), B, K, V, _ptr(bt), _ptr(bp)):
        raise MemoryError("oracle allocation failed")
    return bt[:, :tot], bp[:, :tot]


def cache_lookup(branch_tok, F, accept_len, token):
    """Step 8: slot per sequence (-1 miss, -2 full accept)."""
    lib = _load()
    F = np.ascontiguousarray(F, dtype=np.int32)
    K = F.shape[0]
    tot = int(F.sum())
    B = accept_len.shape[0]
    bt = np.ascontiguousarray(branch_tok, dtype=np.int32).reshape(B, tot) if tot else np.zeros((B, 1), np.int32)
    al = np.ascontiguousarray(accept_len, dtype=np.int32)
    tk = np.ascontiguousarray(token, dtype=np.int32)
    slot = np.empty(B, np.int32)
    lib.orc_cache_lookup(_ptr(bt), _ptr(F), B, K, _ptr(al), _ptr(tk), _ptr(slot))
    return slot


def branch_alloc(B_alloc: int, gamma: int, alpha: float, beta: float):
    """Geometric-decay branch allocation of Sec. IV-C.

    eta = alpha^(1/(beta+1)); F*_k = B_alloc (1-eta)/(1-eta^gamma) eta^k
    (the closed form after solving the Lagrangian condition under the budget
    sum F_k = B_alloc).  Integers: floor, then the remaining units go to the
    largest fractional parts, ties to the shallower depth.
    Returns (real-valued F*, integer F).
    """
    eta = alpha ** (1.0 / (beta + 1.0))
    if eta == 1.0:
        real = [B_alloc / gamma] * gamma
    else:
        real = [B_alloc * (1.0 - eta) / (1.0 - eta ** gamma) * eta ** kk for kk in range(gamma)]
    ints = [int(floor(r)) for r in real]
    left = B_alloc - sum(ints)
    rema = sorted(range(gamma), key=lambda kk: (-(real[kk] - ints[kk]), kk))
    for kk in rema[:left]:
        ints[kk] += 1
    return real, ints


def warp(z, T: float, top_p: float):
    """Steps 1-2: the nucleus-renormalised target p of every row of z [..., V]."""
    lib = _load()
    zf = _logits_f32(z)
    V = zf.shape[-1]
    rows = zf.size // V
    p = np.empty((rows, V), np.float64)
    st = np.empty(rows, np.int32)
    if lib.orc_warp(_ptr(zf), rows, V, float(T), float(top_p), _ptr(p), _ptr(st)):
        raise MemoryError("oracle allocation failed")
    return p.reshape(zf.shape), st.reshape(zf.shape[:-1])


def resample_sparse(accept_len, ids, probs, tail, row_status, q, u):
    """Step 9: the edge's draw from the payload of row pi (Alg. 1 RESAMPLE).

    accept_len [B], ids/probs [B, K+1, k] (probs as float32), tail [B, K+1],
    row_status [B, K+1], q [B, K, V], u [B, K+1].  Returns token, status,
    the flag diagnostics and dist [B, V] (the normalised distribution drawn from).
    """
    lib = _load()
    ids = np.ascontiguousarray(ids, np.int32)
    B, R, k = ids.shape
    K = R - 1
    q = np.ascontiguousarray(q, np.float32)
    V = q.shape[-1]
    al = np.ascontiguousarray(accept_len, np.int32)
    pr = np.ascontiguousarray(probs, np.float32)
    tl = np.ascontiguousarray(tail, np.float32)
    rs = np.ascontiguousarray(row_status, np.int32)
    uu = np.ascontiguousarray(u, np.float32)
    out = dict(token=np.empty(B, np.int32), status=np.empty(B, np.int32),
               res_target=np.empty(B, np.float64), res_cj=np.empty(B, np.float64),
               res_cjm1=np.empty(B, np.float64), res_sum=np.empty(B, np.float64),
               dist=np.empty((B, V), np.float64))
    o = out
    if lib.orc_resample_sparse(_ptr(al), _ptr(ids), _ptr(pr), _ptr(tl), _ptr(rs), _ptr(q), _ptr(uu), B, K, V, k,
                               _ptr(o["token"]), _ptr(o["status"]), _ptr(o["res_target"]), _ptr(o["res_cj"]),
                               _ptr(o["res_cjm1"]), _ptr(o["res_sum"]), _ptr(o["dist"])):
        raise MemoryError("oracle allocation failed")
    return out


def hit_prob(z, q, xt, T: float, top_p: float, branch_tok, F):
    """Per-sequence probability that the cache recovers the sequence (lookup
    slot >= 0 or -2) given z, q, x~ and the branches, and the product form
    prod_k (a_k + (1 - a_k) R_k) of Sec. IV-C with the same per-row terms."""
    lib = _load()
    zf = _logits_f32(z)
    B, R, V = zf.shape
    K = R - 1
    q = np.ascontiguousarray(q, np.float32)
    xt = np.ascontiguousarray(xt, np.int32)
    bt = np.ascontiguousarray(branch_tok, np.int32)
    Fa = np.ascontiguousarray(F, np.int32)
    hp = np.empty(B, np.float64)
    pp = np.empty(B, np.float64)
    if lib.orc_hit_prob(_ptr(zf), _ptr(q), _ptr(xt), B, K, V, float(T), float(top_p), _ptr(bt), _ptr(Fa),
                        _ptr(hp), _ptr(pp)):
        raise MemoryError("oracle allocation failed")
    return hp, pp


def compact_kv(kv, prefix_len, accept_len, slot, K: int, branch_len: int):
    """COMPACT_KV / ROLLBACK_KV of Alg. 1 on a KV array [planes, B, H, S, D].

    The tree of every sequence is packed after its prefix of prefix_len[b]
    positions: the main chain (K positions), then the branches in slot order,
    branch_len positions each.  After the lookup:
      slot >= 0  (hit):   the branch's rows move right behind the accepted
                          tokens, positions t + pi ...; new length
                          t + pi + branch_len;
      slot == -2 (all accepted): nothing moves; new length t + K;
      slot == -1 (miss):  the rejected drafts are dropped; new length t + pi.
    A sequence whose tree would pass the end of the array gets new length -1
    and nothing moves.  Returns (new kv, new lengths).  Plain slice copies.
    """
    kv = np.array(kv, copy=True)
    S = kv.shape[3]
    B = kv.shape[1]
    new_len = np.empty(B, np.int32)
    for b in range(B):
        t, pi, s = int(prefix_len[b]), int(accept_len[b]), int(slot[b])
        total = 0
        if t < 0 or pi < 0 or pi > K:
            new_len[b] = -1
            continue
        if s >= 0:
            src = t + K + s * branch_len
            if src + branch_len > S:
                new_len[b] = -1
                continue
            block = kv[:, b, :, src:src + branch_len, :].copy()
            kv[:, b, :, t + pi:t + pi + branch_len, :] = block
            total = t + pi + branch_len
        elif s == -2:
            total = t + K
        else:
            total = t + pi
        new_len[b] = total if total <= S else -1
    return kv, new_len


def tree_mask(F, K: int, branch_len: int):
    """Tree attention mask of the packed branch forward (Sec. III-C, Fig. for
    the tree mask), by walking parent pointers.

    Packed order: the main chain (K tokens), then the branches in slot order
    (depth 0's F_0 branches first), branch_len tokens each: the alternative
    token at depth d and its drafted continuation.  A token's parent is the
    token before it on its path: main token m -> m - 1; the first token of a
    branch at depth d -> main token d - 1 (none at depth 0); a later branch
    token -> the one before it in its branch.  mask[q, k] is True when k is q
    or one of its ancestors (every tree token also sees the whole shared
    prefix, which the mask leaves out); depth[q] = number of ancestors.
    """
    F = [int(f) for f in F]
    n_branch = sum(F)
    n = K + n_branch * branch_len
    parent = [-1] * n
    for m in range(1, K):
        parent[m] = m - 1
    s = 0
    for d in range(K):
        for _ in range(F[d]):
            base = K + s * branch_len
            parent[base] = d - 1
            for o in range(1, branch_len):
                parent[base + o] = base + o - 1
            s += 1
    mask = np.zeros((n, n), bool)
    depth = np.zeros(n, np.int32)
    for q in range(n):
        k = q
        while k >= 0:
            mask[q, k] = True
            k = parent[k]
        depth[q] = int(mask[q].sum()) - 1
    return mask, depth
