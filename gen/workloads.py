"""Synthetic workloads shaped like the paper's model pairs (Sec. V-A).

Each workload is one draft/target pair of vocabulary size V, B sequences and a
draft length K (gamma in the paper).  Every sequence b is generated from its
own counter-based Philox stream keyed by (seed, b), so any subset of
sequences of a full-size workload can be regenerated exactly on its own.

Recipe (per sequence, positions i = 0..K):
  * draft logits  zd[i, :] ~ N(0, sigma^2)
  * target logits z[i, :]  = rho * zd + sqrt(1 - rho^2) * N(0, sigma^2),
    or, when rho is None, z = zd + N(0, noise^2)
  * optional Zipf head: 100 ids (one fixed random set per workload) get
    +2 * ln(101 / rank), rank = 1..100, added to both zd and z
  * logits are rounded to float32 (and then to bfloat16, round-to-nearest-
    even, for bf16 workloads)
  * draft distribution q[i, :] for i < K: tempered weights
    exp((zd - max zd) / T) restricted to ids whose weight is >= draft_min_p
    (1e-4 by default) of the largest (a min-p style support cut of the draft
    sampler; 0 keeps every id), normalised, stored as float32.  This stands
    in for the edge model's output Q.
  * draft token x~[i] is drawn from the float32 q[i] by inverse CDF.
  * uniforms u[i] for i <= K are float32 in (0, 1): u[:, i<K] drive the
    accept tests and u[:, K] the single residual / bonus draw.
The real datasets (GSM8K, HumanEval, Alpaca) and model weights are not
available; these rows stand in for their per-position distributions.
"""
from __future__ import annotations

import dataclasses
import os
from typing import Optional, Sequence

import numpy as np

DRAFT_MIN_P = 1e-4          # support cut of the synthetic draft sampler
ZIPF_HEAD = 100


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    B: int
    K: int
    V: int
    dtype: str              # "f32" or "bf16" for the target logits
    sigma: float
    rho: Optional[float]
    noise: float
    zipf: bool
    T: float
    top_p: float
    k: int
    F: tuple
    seed: int
    draft_min_p: float = 1e-4  # support cut of the draft sampler (0: every id keeps q > 0)

    @property
    def rows(self) -> int:
        return self.B * (self.K + 1)


# F for the 128256-vocabulary workload comes from the geometric-decay
# allocation (Sec. IV-C) with B_alloc = 64, gamma = 16, alpha = 0.9, beta = 1
# (eta = 0.9487), rounded to integers by largest remainder.
_F_GEOM_64_16 = (6, 5, 5, 5, 5, 4, 4, 4, 4, 4, 3, 3, 3, 3, 3, 3)

WORKLOADS = {
    w.name: w for w in [
        Workload("b1_k4_v32000_f32", 1, 4, 32000, "f32", 3.0, None, 1.0, False,
                 1.0, 1.0, 16, (2,) * 4, 1001),
        Workload("b16_k8_v32000_f32", 16, 8, 32000, "f32", 3.0, 0.8, 0.0, False,
                 0.8, 0.9, 32, (4,) * 8, 1002),
        Workload("b64_k8_v152064_bf16", 64, 8, 152064, "bf16", 4.0, 0.7, 0.0, True,
                 0.7, 0.95, 64, (4,) * 8, 1003),
        Workload("b128_k16_v128256_bf16", 128, 16, 128256, "bf16", 3.0, 0.5, 0.0, False,
                 1.0, 0.9, 32, _F_GEOM_64_16, 1004),
        Workload("b256_k16_v256000_bf16", 256, 16, 256000, "bf16", 3.0, 0.9, 0.0, False,
                 0.6, 0.8, 128, (4,) * 16, 1005),
    ]
}


def f32_to_bf16(x: np.ndarray) -> np.ndarray:
    """Round float32 to bfloat16 (round-to-nearest-even); returns uint16 bits."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    nan = (b & 0x7FFFFFFF) > 0x7F800000
    r = ((b >> 16) & 1) + np.uint32(0x7FFF)
    out = ((b + r) >> 16).astype(np.uint16)
    out[nan] = ((b[nan] >> 16) | 0x40).astype(np.uint16)
    return out


def bf16_to_f32(h: np.ndarray) -> np.ndarray:
    """Widen bfloat16 bits (uint16) to float32 exactly."""
    return (np.ascontiguousarray(h, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def _zipf_head(w: Workload):
    rng = np.random.Generator(np.random.Philox(np.random.SeedSequence([w.seed, 2 ** 31])))
    ids = rng.choice(w.V, ZIPF_HEAD, replace=False)
    bias = 2.0 * np.log((ZIPF_HEAD + 1.0) / np.arange(1, ZIPF_HEAD + 1))
    return ids, bias


def _one_sequence(w: Workload, b: int, head, draft_logits: bool = False):
    """Returns (z float32 [K+1,V], q float32 [K,V], xt int32 [K], u float32 [K+1]),
    plus the draft logits zd float32 [K+1,V] when draft_logits is set."""
    rng = np.random.Generator(np.random.Philox(np.random.SeedSequence([w.seed, b])))
    K, V = w.K, w.V
    big = V >= 100000
    dt = np.float32 if big else np.float64
    zd = rng.standard_normal((K + 1, V), dtype=dt)
    zd *= dt(w.sigma)
    n = rng.standard_normal((K + 1, V), dtype=dt)
    if w.rho is None:
        z = zd + n * dt(w.noise)
    else:
        z = dt(w.rho) * zd + dt(np.sqrt(1.0 - w.rho * w.rho) * w.sigma) * n
    if head is not None:
        ids, bias = head
        zd[:, ids] += bias.astype(dt)
        z[:, ids] += bias.astype(dt)
    z32 = z.astype(np.float32)
    q = np.empty((K, V), np.float32)
    xt = np.empty(K, np.int32)
    for i in range(K):
        d = zd[i].astype(np.float64)
        wgt = np.exp((d - d.max()) / w.T)
        if w.draft_min_p > 0.0:
            wgt[wgt < w.draft_min_p] = 0.0
        q[i] = (wgt / wgt.sum()).astype(np.float32)
        c = np.cumsum(q[i], dtype=np.float64)
        t = rng.random() * c[-1]
        j = int(np.searchsorted(c, t, side="right"))
        j = min(j, V - 1)
        while q[i, j] <= 0.0:       # never pick an id outside the draft support
            j -= 1
        xt[i] = j
    u = (rng.integers(1, 1 << 24, size=K + 1).astype(np.float64) / float(1 << 24)).astype(np.float32)
    if draft_logits:
        return z32, q, xt, u, zd.astype(np.float32)
    return z32, q, xt, u


def make_workload(B: int, K: int, V: int, dtype: str = "bf16", sigma: float = 3.0,
                  rho: Optional[float] = 0.8, noise: float = 1.0, zipf: bool = False, T: float = 1.0,
                  top_p: float = 0.9, k: int = 16, F: Sequence[int] = (), seed: int = 7,
                  name: str = "custom") -> Workload:
    """An ad-hoc workload with the same recipe (for ragged and edge-case tests)."""
    F = tuple(F) if F else (2,) * K
    return Workload(name, B, K, V, dtype, sigma, rho, noise, zipf, T, top_p, k, F, seed)


def _resolve(w) -> Workload:
    return WORKLOADS[w] if isinstance(w, str) else w


def _fill(args):
    w, seqs, shm_names, shapes = args
    from multiprocessing import shared_memory
    head = _zipf_head(w) if w.zipf else None
    shms = [shared_memory.SharedMemory(name=s) for s in shm_names]
    try:
        zbuf = np.ndarray(shapes[0][0], dtype=shapes[0][1], buffer=shms[0].buf)
        qbuf = np.ndarray(shapes[1][0], dtype=shapes[1][1], buffer=shms[1].buf)
        xbuf = np.ndarray(shapes[2][0], dtype=shapes[2][1], buffer=shms[2].buf)
        ubuf = np.ndarray(shapes[3][0], dtype=shapes[3][1], buffer=shms[3].buf)
        for pos, b in seqs:
            z, q, xt, u = _one_sequence(w, b, head)
            zbuf[pos] = f32_to_bf16(z) if w.dtype == "bf16" else z
            qbuf[pos] = q
            xbuf[pos] = xt
            ubuf[pos] = u
        del zbuf, qbuf, xbuf, ubuf
    finally:
        for s in shms:
            s.close()
    return len(seqs)


def generate_sequences(name, seqs: Sequence[int], workers: int = 0, B: Optional[int] = None,
                       draft_logits: bool = False):
    """Generate the listed sequences of workload `name` (a name or a Workload).

    Returns a dict with z ([n,K+1,V] float32, or uint16 bfloat16 bits), q
    ([n,K,V] float32), xt ([n,K] int32), u ([n,K+1] float32) and the workload;
    with draft_logits also zd ([n,K+1,V] float32, the draft logits q was
    made from; one process).  `workers` > 1 uses a spawn-started process
    pool (safe after CUDA init).
    """
    w = _resolve(name)
    seqs = [int(s) for s in seqs]
    n = len(seqs)
    zdt = np.uint16 if w.dtype == "bf16" else np.float32
    shapes = [((n, w.K + 1, w.V), zdt), ((n, w.K, w.V), np.float32),
              ((n, w.K), np.int32), ((n, w.K + 1), np.float32)]
    if workers <= 1 or n < 4 or draft_logits:
        head = _zipf_head(w) if w.zipf else None
        z = np.empty(*shapes[0]); q = np.empty(*shapes[1])
        xt = np.empty(*shapes[2]); u = np.empty(*shapes[3])
        zd = np.empty((n, w.K + 1, w.V), np.float32) if draft_logits else None
        for pos, b in enumerate(seqs):
            r = _one_sequence(w, b, head, draft_logits)
            zz, qq, xx, uu = r[:4]
            z[pos] = f32_to_bf16(zz) if w.dtype == "bf16" else zz
            q[pos] = qq; xt[pos] = xx; u[pos] = uu
            if draft_logits:
                zd[pos] = r[4]
        out = dict(z=z, q=q, xt=xt, u=u, w=w, seqs=np.array(seqs))
        if draft_logits:
            out["zd"] = zd
        return out
    import multiprocessing as mp
    from multiprocessing import shared_memory
    shms = [shared_memory.SharedMemory(create=True, size=max(1, int(np.prod(s)) * np.dtype(d).itemsize))
            for s, d in shapes]
    try:
        items = list(enumerate(seqs))
        chunks = [items[i::workers] for i in range(workers)]
        ctx = mp.get_context("spawn")
        with ctx.Pool(workers) as pool:
            pool.map(_fill, [(w, c, [s.name for s in shms], shapes) for c in chunks if c])
        out = [np.ndarray(s, dtype=d, buffer=m.buf).copy() for (s, d), m in zip(shapes, shms)]
    finally:
        for m in shms:
            m.close()
            m.unlink()
    return dict(z=out[0], q=out[1], xt=out[2], u=out[3], w=w, seqs=np.array(seqs))


def generate(name, workers: int = 0, B: Optional[int] = None):
    """Generate the first B (default: all) sequences of workload `name`."""
    w = _resolve(name)
    nb = w.B if B is None else B
    if workers == 0:
        workers = min(16, os.cpu_count() or 1) if w.V * w.K * nb > 50_000_000 else 1
    return generate_sequences(w, range(nb), workers=workers)
