#!/usr/bin/env python
"""Benchmark of the AceSpec hot path on GB300.

One step = one pass of the whole path over one batch: aces_verify (temperature
softmax, nucleus, accept tests, first rejection, residual/bonus draw, fused
sparse top-k payload) + aces_cache_build (per-depth branch cache) +
aces_cache_lookup, on the B=256, K=16, V=256000 bfloat16 workload
(T=0.6, top_p=0.8, k=128, F=[4]*16).  Inputs (6.4 GB) are larger than L2, so
no flush is needed between steps.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl acespec|reference]

Prints one JSON line on rank 0.  With N > 1 (torchrun) every rank processes
its own B sequences (weak scaling, no collective on the data path) and the
timing is the max over ranks.  `--impl reference` times the float64 CPU
oracle on a bounded sample of the same workload instead.
"""
from __future__ import annotations

import argparse
import ctypes
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "verified rows/s and achieved HBM GB/s (fraction of GB300 peak) for verify+sparsify"
WORKLOAD = "b256_k16_v256000_bf16"
SWEEP_B = (32, 64, 128, 256)
# kernels of one step: k_rows_cap, k_rows_general, k_resolve_seg,
# k_resolve_pick (aces_verify), k_cache_build, k_cache_lookup
KERNELS_PER_STEP = 6
VERIFY_KERNELS = ["k_rows_cap", "k_rows_general", "k_resolve_seg", "k_resolve_pick"]
# path counters at the start of the workspace (int32 words)
PATHS = ["rows_on_general_kernel", "timeouts", "rows_value_histogram", "rows_bitonic_order",
         "general_rows_radix", "rows_cut_left_to_resolve", "general_rows_value_histogram",
         "accept_tests_ranked_among_ties", "rows_published_depth", "rows_depth_from_finished_rows",
         "rows_counted_twice", "short_rows_published", "rows_sketch_led"]


# ---------------------------------------------------------------------------
# clocks during the timed region: NVML polled at ~1 ms plus nvidia-smi (read only)
class ClockSampler:
    REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown",
               0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown"}

    def __init__(self, pci_bus_id: str | None):
        self.samples = []
        self.smi_lines = []
        self._stop = threading.Event()
        self._nvml = None
        self._h = None
        self.max_mhz = None
        try:
            nv = ctypes.CDLL("libnvidia-ml.so.1")
            if nv.nvmlInit_v2() == 0:
                h = ctypes.c_void_p()
                ok = -1
                if pci_bus_id:
                    ok = nv.nvmlDeviceGetHandleByPciBusId_v2(pci_bus_id.encode(), ctypes.byref(h))
                if ok != 0:
                    ok = nv.nvmlDeviceGetHandleByIndex_v2(0, ctypes.byref(h))
                if ok == 0:
                    self._nvml, self._h = nv, h
                    mx = ctypes.c_uint()
                    if nv.nvmlDeviceGetMaxClockInfo(h, 1, ctypes.byref(mx)) == 0:
                        self.max_mhz = mx.value
        except OSError:
            pass
        self._smi = None

    def _poll(self):
        nv, h = self._nvml, self._h
        clk = ctypes.c_uint()
        rs = ctypes.c_ulonglong()
        pw = ctypes.c_uint()
        while not self._stop.is_set():
            if nv.nvmlDeviceGetClockInfo(h, 1, ctypes.byref(clk)) == 0:
                r = rs.value if nv.nvmlDeviceGetCurrentClocksEventReasons(h, ctypes.byref(rs)) == 0 else 0
                p = pw.value / 1000.0 if nv.nvmlDeviceGetPowerUsage(h, ctypes.byref(pw)) == 0 else None
                self.samples.append((clk.value, r, p))
            time.sleep(0.001)

    def __enter__(self):
        try:
            q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
                 "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
                 "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
            self._smi = subprocess.Popen(["nvidia-smi", f"--query-gpu={q}", "--format=csv,noheader",
                                          "-lms", "50"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL,
                                         text=True)
        except OSError:
            self._smi = None
        if self._nvml is not None:
            self._t = threading.Thread(target=self._poll, daemon=True)
            self._t.start()
        return self

    def __exit__(self, *exc):
        self._stop.set()
        if self._nvml is not None:
            self._t.join()
        if self._smi is not None:
            self._smi.terminate()
            try:
                out, _ = self._smi.communicate(timeout=5)
                self.smi_lines = [ln for ln in out.splitlines() if ln.strip()]
            except subprocess.TimeoutExpired:
                self._smi.kill()
        return False

    def summary(self):
        mhz = [s[0] for s in self.samples]
        reasons = set()
        for _, r, _ in self.samples:
            for bit, name in self.REASONS.items():
                if r & bit:
                    reasons.add(name)
        smi_mhz = []
        for ln in self.smi_lines:
            f = [x.strip() for x in ln.split(",")]
            try:
                smi_mhz.append(float(f[1].split()[0]))
                if self.max_mhz is None:
                    self.max_mhz = float(f[2].split()[0])
                for name, col in (("hw_slowdown", 5), ("hw_thermal_slowdown", 6), ("sw_thermal_slowdown", 7),
                                  ("sw_power_cap", 8)):
                    if f[col].lower() == "active":
                        reasons.add(name)
            except (IndexError, ValueError):
                pass
        allm = mhz or smi_mhz
        pw = [s[2] for s in self.samples if s[2] is not None]
        return {"sm_mhz": statistics.median(allm) if allm else None, "sm_max_mhz": self.max_mhz,
                "reasons": sorted(reasons), "samples": len(mhz), "smi_samples": len(smi_mhz),
                "power_w_max": max(pw) if pw else None}


# ---------------------------------------------------------------------------
def measured_peak():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        d = json.load(open(p))
        return float(d["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return 6800.0, "fallback"


# device code behind each profiled kernel (its file and the shared device header)
KERNEL_SOURCES = {
    "aces_verify": ("common.cuh", "rows_cap.cu", "rows_general.cu", "resolve.cu"),
    "k_cache_build": ("common.cuh", "cache.cu"),
}


def _code_only(text: str) -> str:
    """The source without its comments and blank space (a change of comments
    alone leaves the kernel, and so the captured counters, as they were)."""
    import re
    text = re.sub(r"/\*.*?\*/", " ", text, flags=re.S)
    text = re.sub(r"//[^\n]*", " ", text)
    return " ".join(text.split())


def kernel_source_hash(kernel: str) -> str:
    h = hashlib.sha256()
    for f in KERNEL_SOURCES[kernel]:
        h.update(_code_only(open(os.path.join(ROOT, "paper_2609_02514_gb300", "csrc", f)).read()).encode())
    return h.hexdigest()[:16]


def profiled_traffic(kernel: str, units: float):
    """DRAM bytes per launch from the committed ncu summary, scaled to the
    timed launch's units; None when the kernels changed since the capture."""
    p = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        d = json.load(open(p))
    except (OSError, ValueError):
        return None
    e = d.get("kernels", {}).get(kernel)
    if not e or kernel not in KERNEL_SOURCES or e.get("source_hash") != kernel_source_hash(kernel):
        return None
    return e["dram_bytes"] * units / e["units"]


def verify_bytes(B, K, V, k, zsize, n_resid_q):
    """Algorithmic bytes of one aces_verify call with a payload of k.

    Reads: every logit once, q at the K draft tokens, the draft tokens and
    the uniforms, and q at the residual row's nucleus ids (n_resid_q floats
    over the batch; the residual max(0, p - q) is 0 wherever p = 0).
    Writes: payload, tail and status per row, token and length per sequence.
    """
    rd = B * (K + 1) * V * zsize + n_resid_q * 4 + B * K * 12 + B * (K + 1) * 4
    wr = B * (K + 1) * (8 * k + 4) + B * 8 + B * (K + 1) * 4
    return rd + wr


def resid_q_count(out, K, k):
    """q floats the residual step needs: the nucleus of each rejecting
    sequence's row pi, counted from its payload (a lower bound of the nucleus
    size when that exceeds k)."""
    if k == 0:
        return 0
    al = out["accept_len"].cpu().numpy()
    ids = out["topk_ids"].cpu().numpy()
    rej = np.nonzero(al < K)[0]
    return int((ids[rej, al[rej]] >= 0).sum())


def resample_bytes(B, K, V, k, n_spread):
    """Algorithmic bytes of one aces_resample_sparse call: per sequence the
    payload of row pi (ids, probs, tail, status), q at its ids, the length
    and the uniform, the token and status; the whole q row pi for the
    n_spread sequences whose payload has a positive tail."""
    return B * (k * 12 + 4 + 4 + 4 + 4 + 8) + n_spread * V * 4


def cache_bytes(B, K, V, S):
    return B * K * V * 4 + B * K * 4 + B * S * 8


# ---------------------------------------------------------------------------
def shard(rank: int, B: int) -> range:
    """Sequences of this rank: every rank gets its own B sequences (weak scaling)."""
    return range(rank * B, (rank + 1) * B)


def max_over_ranks(x: float, dist=None, device=None) -> float:
    """The largest x over all ranks (the job's time is its slowest rank's)."""
    if dist is None:
        return x
    import torch
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def init_dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def reference_arm(args, ws, rank):
    """Times the float64 CPU oracle as it stands on a bounded sample."""
    if rank != 0:
        return
    import gen
    from oracle import oracle as O
    O.build()
    w = gen.WORKLOADS[args.workload]
    cores = O.num_threads()
    nseq = max(1, min(cores, w.B, args.ref_seqs))
    inp = gen.generate_sequences(w, range(nseq), workers=min(16, os.cpu_count() or 1))
    rows = nseq * (w.K + 1)

    def step():
        O.verify(inp["z"], inp["q"], inp["xt"], inp["u"], w.T, w.top_p, w.k)
        O.cache_build(inp["q"], inp["xt"], w.F)

    for _ in range(args.warmup):
        step()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        step()
    dt = time.perf_counter() - t0
    val = rows * args.steps / dt
    sample = f"{nseq} of {w.B} sequences ({rows} target rows + {nseq * w.K} draft rows) per step"
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": val, "unit": "rows/s", "n_gpus": ws,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt / args.steps * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": config_of(w),
        "cpu_baseline": {"value": val, "unit": "rows/s", "cores": cores, "kind": "oracle", "sample": sample},
        "e2e": {"value": val, "unit": "rows/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }), flush=True)


def config_of(w):
    zb = w.B * (w.K + 1) * w.V * (2 if w.dtype == "bf16" else 4)
    qb = w.B * w.K * w.V * 4
    return {"workload": w.name if w.B == gen_B(w) else f"{w.name} (first {w.B} sequences)", "B": w.B, "K": w.K,
            "V": w.V, "logits": w.dtype, "T": w.T, "top_p": w.top_p, "k": w.k, "F": list(w.F),
            "l2": f"inputs (z {zb / 1e9:.2f} GB + q {qb / 1e9:.2f} GB) exceed the 129 MB L2; no flush",
            "parallelism": "one process per GPU, sequences sharded, no collective",
            "step": "aces_cloud_step (verification, with the cache build on the library's side stream) "
                    "+ aces_cache_lookup"}


def gen_B(w):
    import gen
    return gen.WORKLOADS[w.name].B


def cpu_baseline(w, inp):
    from oracle import oracle as O
    O.build()
    cores = O.num_threads()
    nseq = min(w.B, max(1, cores))
    sub = {k: inp[k][:nseq] for k in ("z", "q", "xt", "u")}
    t0 = time.perf_counter()
    O.verify(sub["z"], sub["q"], sub["xt"], sub["u"], w.T, w.top_p, w.k)
    O.cache_build(sub["q"], sub["xt"], w.F)
    dt = time.perf_counter() - t0
    rows = nseq * (w.K + 1)
    return {"value": rows / dt, "unit": "rows/s", "cores": cores, "kind": "oracle",
            "sample": f"{nseq} of {w.B} sequences: verify+sparsify ({rows} rows) and cache build "
                      f"({nseq * w.K} rows), OpenMP over sequences, {dt:.1f} s"}


def oracle_rates(w, inp, seqs_all, seqs_one):
    """The oracle as it stands on the machine's host cores: verify+sparsify rows/s
    with every core (OpenMP over sequences) and with one thread, each on a
    bounded sample of the workload's sequences."""
    from oracle import oracle as O
    O.build()
    cores = O.num_threads()

    def rate(nseq):
        sub = {k: inp[k][:nseq] for k in ("z", "q", "xt", "u")}
        t0 = time.perf_counter()
        O.verify(sub["z"], sub["q"], sub["xt"], sub["u"], w.T, w.top_p, w.k)
        dt = time.perf_counter() - t0
        return nseq * (w.K + 1) / dt, dt

    n_all = max(1, min(w.B, seqs_all, cores))
    v_all, t_all = rate(n_all)
    prev = O.set_threads(1)
    try:
        n_one = max(1, min(w.B, seqs_one))
        v_one, t_one = rate(n_one)
    finally:
        O.set_threads(prev)
    return {"value": v_all, "unit": "rows/s", "cores": cores, "kind": "oracle",
            "sample": f"{n_all} of {w.B} sequences ({n_all * (w.K + 1)} rows), verify+sparsify, {t_all:.2f} s",
            "one_thread": {"value": v_one, "unit": "rows/s", "cores": 1,
                           "sample": f"{n_one} sequence(s) ({n_one * (w.K + 1)} rows), {t_one:.2f} s"}}


def per_config(A, torch, dev, stream, peak, peak_kind, have=None, cpu=True):
    """aces_verify (k > 0) and aces_cache_build on every paper-shaped
    workload at full size: CUDA-event times, algorithmic bytes, the fraction
    of the measured HBM peak, the rows on each kernel path, and the oracle
    timed beside it.  `have` maps a workload name to its already resident
    inputs (host arrays, device tensors)."""
    import gen
    entries = []
    for name, w in gen.WORKLOADS.items():
        if have and name in have:
            inp, d = have[name]
        else:
            inp = gen.generate_sequences(w, range(w.B), workers=min(16, os.cpu_count() or 1))
            z = torch.from_numpy(inp["z"].view(np.int16)).view(torch.bfloat16) if w.dtype == "bf16" \
                else torch.from_numpy(inp["z"])
            d = {"z": z.to(dev), "q": torch.from_numpy(inp["q"]).to(dev),
                 "xt": torch.from_numpy(inp["xt"]).to(dev), "u": torch.from_numpy(inp["u"]).to(dev)}
        B, K, V, k = w.B, w.K, w.V, w.k
        zsize = 2 if w.dtype == "bf16" else 4
        wsb = torch.zeros(A.workspace_bytes(B, K, V, k), dtype=torch.uint8, device=dev)
        out = A.verify(d["z"], d["q"], d["xt"], d["u"], w.T, w.top_p, k, workspace=wsb)
        cache = A.cache_build(d["q"], d["xt"], w.F)
        for _ in range(3):
            A.verify(d["z"], d["q"], d["xt"], d["u"], w.T, w.top_p, k, out=out, workspace=wsb)
        torch.cuda.synchronize()
        n = 20
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n)]
        for e0, e1 in ev:
            e0.record(stream)
            A.verify(d["z"], d["q"], d["xt"], d["u"], w.T, w.top_p, k, out=out, workspace=wsb)
            e1.record(stream)
        torch.cuda.synchronize()
        vms = statistics.median(e0.elapsed_time(e1) for e0, e1 in ev)
        paths = dict(zip(PATHS, wsb[A.COUNTERS_OFFSET:A.COUNTERS_OFFSET + 64].view(torch.int32).cpu().numpy().tolist()))
        paths.pop("timeouts")
        vb = verify_bytes(B, K, V, k, zsize, resid_q_count(out, K, k))
        for _ in range(3):
            A.cache_build(d["q"], d["xt"], w.F, out=cache)
        for e0, e1 in ev:
            e0.record(stream)
            A.cache_build(d["q"], d["xt"], w.F, out=cache)
            e1.record(stream)
        torch.cuda.synchronize()
        cms = statistics.median(e0.elapsed_time(e1) for e0, e1 in ev)
        cb = cache_bytes(B, K, V, int(sum(w.F)))
        rows = B * (K + 1)
        gbs = vb / (vms * 1e-3) / 1e9
        e = {"workload": name, "B": B, "K": K, "V": V, "logits": w.dtype, "T": w.T, "top_p": w.top_p, "k": k,
             "F": list(w.F),
             "verify_sparsify": {"ms": vms, "rows_per_s": rows / (vms * 1e-3), "alg_bytes": vb, "gbs": gbs,
                                 "kernels": VERIFY_KERNELS, "paths": paths,
                                 "l2": "logits %.1f MB %s the 129 MB L2; back-to-back calls" % (
                                     rows * V * zsize / 1e6, "exceed" if rows * V * zsize > 129e6 else "fit in")},
             "roofline_verify_sparsify": {"bound": "hbm", "kernel": "aces_verify", "achieved": gbs, "peak": peak,
                                          "unit": "GB/s", "frac": gbs / peak, "peak_kind": peak_kind},
             "cache_build": {"ms": cms, "alg_bytes": cb, "gbs": cb / (cms * 1e-3) / 1e9,
                             "frac": cb / (cms * 1e-3) / 1e9 / peak, "kernels": ["k_cache_build"]}}
        if cpu:
            e["cpu_baseline"] = oracle_rates(w, inp, 16, 1)
        entries.append(e)
        del d, out, cache, wsb
        torch.cuda.empty_cache()
    return entries


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="acespec", choices=["acespec", "reference"])
    ap.add_argument("--workload", default=WORKLOAD)
    ap.add_argument("--ref-seqs", type=int, default=16)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-sweep", action="store_true")
    ap.add_argument("--no-extras", action="store_true",
                    help="skip the resample and KV-compaction timings (small profiling runs)")
    ap.add_argument("--e2e-steps", type=int, default=0)
    ap.add_argument("--B", type=int, default=0, help="use only the first B sequences (small profiling runs)")
    ap.add_argument("--no-per-config", action="store_true", help="skip the five paper-shaped workloads' entries")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)
    ws, rank, local = init_dist()

    if args.impl == "reference":
        reference_arm(args, ws, rank)
        return

    import torch

    import gen
    import paper_2609_02514_gb300 as A

    w = gen.WORKLOADS[args.workload]
    if args.B:
        import dataclasses
        w = dataclasses.replace(w, B=min(args.B, w.B))
    # host inputs first (spawn pool), this rank's shard of sequences
    inp = gen.generate_sequences(w, shard(rank, w.B), workers=min(16, os.cpu_count() or 1))

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    pg = None
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
        pg = dist
    A.load()
    B, K, V, k = w.B, w.K, w.V, w.k
    S = int(sum(w.F))
    zsize = 2 if w.dtype == "bf16" else 4

    # pinned host copies (e2e) and device-resident inputs
    zh = torch.from_numpy(inp["z"].view(np.int16)).view(torch.bfloat16) if w.dtype == "bf16" \
        else torch.from_numpy(inp["z"])
    host = {"z": zh.pin_memory(), "q": torch.from_numpy(inp["q"]).pin_memory(),
            "xt": torch.from_numpy(inp["xt"]).pin_memory(), "u": torch.from_numpy(inp["u"]).pin_memory()}
    d = {key: t.to(dev) for key, t in host.items()}
    out = A.verify(d["z"], d["q"], d["xt"], d["u"], w.T, w.top_p, k)
    cache = A.cache_build(d["q"], d["xt"], w.F)
    slot = A.cache_lookup(cache["branch_tok"], w.F, out["accept_len"], out["out_token"])
    wsb = torch.zeros(A.workspace_bytes(B, K, V, k), dtype=torch.uint8, device=dev)
    torch.cuda.synchronize()
    stream = torch.cuda.current_stream(dev)

    both = dict(out)
    both.update(cache)

    def step():
        # verification and cache build in one call (the cache build overlaps
        # the verification on the library's side stream), then the lookup
        A.cloud_step(d["z"], d["q"], d["xt"], d["u"], w.T, w.top_p, k, w.F, out=both, workspace=wsb)
        A.cache_lookup(both["branch_tok"], w.F, both["accept_len"], both["out_token"], out=slot)

    def parts_step(ev):
        # the same work as three sequential calls, timed part by part
        ev[0].record(stream)
        A.verify(d["z"], d["q"], d["xt"], d["u"], w.T, w.top_p, k, out=out, workspace=wsb)
        ev[1].record(stream)
        A.cache_build(d["q"], d["xt"], w.F, out=cache)
        ev[2].record(stream)
        A.cache_lookup(cache["branch_tok"], w.F, out["accept_len"], out["out_token"], out=slot)
        ev[3].record(stream)

    def barrier():
        if pg is not None:
            pg.barrier()
        torch.cuda.synchronize()

    for _ in range(args.warmup):
        step()
    pci = None
    try:
        pci = torch.cuda.get_device_properties(dev).pci_bus_id  # may not exist on every torch
    except AttributeError:
        pass
    barrier()
    with ClockSampler(pci) as clocks:
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        t0.record(stream)
        for i in range(args.steps):
            step()
        t1.record(stream)
        barrier()
    ms_total = max_over_ranks(t0.elapsed_time(t1), pg, dev)
    ms_step = ms_total / args.steps
    # per-part times (sequential calls), outside the timed region
    n_parts = min(args.steps, 20)
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(n_parts)]
    for _ in range(2):
        parts_step(evs[0])
    for i in range(n_parts):
        parts_step(evs[i])
    torch.cuda.synchronize()
    part_ms = {
        "verify_sparsify": statistics.mean(e[0].elapsed_time(e[1]) for e in evs),
        "cache_build": statistics.mean(e[1].elapsed_time(e[2]) for e in evs),
        "cache_lookup": statistics.mean(e[2].elapsed_time(e[3]) for e in evs),
    }
    rows = B * (K + 1)
    value = ws * rows / (ms_step * 1e-3)

    al = out["accept_len"].cpu().numpy()
    n_rej = int((al < K).sum())
    n_resid_q = resid_q_count(out, K, k)
    paths = dict(zip(PATHS, wsb[A.COUNTERS_OFFSET:A.COUNTERS_OFFSET + 64].view(torch.int32).cpu().numpy().tolist()))
    paths.pop("timeouts")
    peak, peak_kind = measured_peak()
    vb = verify_bytes(B, K, V, k, zsize, n_resid_q)
    cb = cache_bytes(B, K, V, S)
    parts = {
        "verify_sparsify": {"ms": part_ms["verify_sparsify"], "rows_per_s": rows / (part_ms["verify_sparsify"] * 1e-3),
                            "alg_bytes": vb, "gbs": vb / (part_ms["verify_sparsify"] * 1e-3) / 1e9,
                            "kernels": VERIFY_KERNELS,
                            "paths": paths, "rejecting_sequences": n_rej},
        "cache_build": {"ms": part_ms["cache_build"], "alg_bytes": cb,
                        "gbs": cb / (part_ms["cache_build"] * 1e-3) / 1e9, "kernels": ["k_cache_build"]},
        "cache_lookup": {"ms": part_ms["cache_lookup"], "kernels": ["k_cache_lookup"]},
    }
    if not args.no_extras:
        # edge-side draw from the sparse payload (Alg. 1 RESAMPLE), timed apart from the step
        rs_out = A.resample_sparse(out["accept_len"], out["topk_ids"], out["topk_probs"], out["tail_mass"],
                                   out["row_status"], d["q"], d["u"])
        for _ in range(3):
            A.resample_sparse(out["accept_len"], out["topk_ids"], out["topk_probs"], out["tail_mass"],
                              out["row_status"], d["q"], d["u"], out=rs_out)
        r0 = torch.cuda.Event(enable_timing=True)
        r1 = torch.cuda.Event(enable_timing=True)
        r0.record(stream)
        for _ in range(args.steps):
            A.resample_sparse(out["accept_len"], out["topk_ids"], out["topk_probs"], out["tail_mass"],
                              out["row_status"], d["q"], d["u"], out=rs_out)
        r1.record(stream)
        torch.cuda.synchronize()
        rs_ms = r0.elapsed_time(r1) / args.steps
        tail_pi = out["tail_mass"][torch.arange(B, device=dev), out["accept_len"].long()].cpu().numpy()
        n_spread = int((tail_pi > 0).sum())
        rb = resample_bytes(B, K, V, k, n_spread)
        parts["resample_sparse"] = {"ms": rs_ms, "alg_bytes": rb, "gbs": rb / (rs_ms * 1e-3) / 1e9,
                                    "sequences_reading_whole_q_row": n_spread, "kernels": ["k_resample_sparse"],
                                    "note": "edge-side draw from row pi's payload; not part of the step"}
        # COMPACT_KV after the lookup (Alg. 1), timed apart from the step: a draft
        # model's KV cache (28 layers x {K, V}, 8 heads, head dim 128, bf16) for
        # the first 64 sequences, prefix of 512 positions, branches of K + 1
        kb = min(B, 64)
        planes, kh, kd, t0, bl = 56, 8, 128, 512, K + 1
        S_kv = t0 + K + S * bl
        kv = torch.empty(planes, kb, kh, S_kv, kd, dtype=torch.bfloat16, device=dev)
        pref = torch.full((kb,), t0, dtype=torch.int32, device=dev)
        new_len = torch.empty(kb, dtype=torch.int32, device=dev)
        kv_args = (kv, pref, out["accept_len"][:kb], slot[:kb], K, bl)
        for _ in range(3):
            A.compact_kv(*kv_args, new_len=new_len)
        # the moved rows (tens of MB) fit in L2: flush it (write 256 MB) before each timed call
        flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
        kv_ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                 for _ in range(args.steps)]
        for e0, e1 in kv_ev:
            flush.fill_(1)
            e0.record(stream)
            A.compact_kv(*kv_args, new_len=new_len)
            e1.record(stream)
        torch.cuda.synchronize()
        kv_ms = statistics.mean(e0.elapsed_time(e1) for e0, e1 in kv_ev)
        del flush
        n_hit = int((slot[:kb] >= 0).sum().item())
        kvb = 2 * n_hit * planes * kh * bl * kd * 2
        parts["compact_kv"] = {"ms": kv_ms, "alg_bytes": kvb, "gbs": kvb / (kv_ms * 1e-3) / 1e9, "hits": n_hit,
                               "sequences": kb, "kernels": ["k_compact_kv"],
                               "note": "KV [56, 64, 8, %d, 128] bf16; moved rows read + written; L2 flushed before each "
                                       "call; not part of the step" % S_kv}
        del kv
    if not args.no_extras:
        # the cache build at a fan-out of 64 per depth (one pass over q when
        # the union of the per-thread lists proves the top 64), and on draft
        # distributions of dense support (no min-p cut; the first 64 sequences)
        def time_cache(qq, xx, FF, n=10):
            o = A.cache_build(qq, xx, FF)
            for _ in range(3):
                A.cache_build(qq, xx, FF, out=o)
            c0 = torch.cuda.Event(enable_timing=True)
            c1 = torch.cuda.Event(enable_timing=True)
            c0.record(stream)
            for _ in range(n):
                A.cache_build(qq, xx, FF, out=o)
            c1.record(stream)
            torch.cuda.synchronize()
            return c0.elapsed_time(c1) / n
        F64 = [64] * K
        ms64 = time_cache(d["q"], d["xt"], F64)
        cb64 = cache_bytes(B, K, V, 64 * K)
        parts["cache_build_F64"] = {"ms": ms64, "alg_bytes": cb64, "gbs": cb64 / (ms64 * 1e-3) / 1e9,
                                    "vs_F_of_the_step": ms64 / part_ms["cache_build"], "kernels": ["k_cache_build"],
                                    "note": "F = [64] * K on the step's q; not part of the step"}
        import dataclasses
        bd = min(B, 64)
        wd = dataclasses.replace(w, B=bd, draft_min_p=0.0)
        dq = gen.generate_sequences(wd, shard(rank, bd), workers=min(16, os.cpu_count() or 1))
        qd = torch.from_numpy(dq["q"]).to(dev)
        xd = torch.from_numpy(dq["xt"]).to(dev)
        msd = time_cache(qd, xd, list(w.F))
        msd64 = time_cache(qd, xd, F64)
        msm = time_cache(d["q"][:bd], d["xt"][:bd], list(w.F))
        cbd = cache_bytes(bd, K, V, S)
        parts["cache_build_dense_q"] = {
            "sequences": bd, "ms": msd, "gbs": cbd / (msd * 1e-3) / 1e9, "ms_F64": msd64,
            "ms_same_sequences_min_p_q": msm, "support": float((qd > 0).float().mean().item()),
            "kernels": ["k_cache_build"],
            "note": "q = tempered softmax of the draft logits with no support cut; not part of the step"}
        del qd, xd, dq
    for p in parts.values():
        if "gbs" in p:
            p["frac_of_peak"] = p["gbs"] / peak
    dom = max(("verify_sparsify", "cache_build"), key=lambda n: part_ms[n])
    dom_kernel = "aces_verify" if dom == "verify_sparsify" else "k_cache_build"
    roof = {"bound": "hbm", "kernel": dom_kernel, "achieved": parts[dom]["gbs"], "peak": peak, "unit": "GB/s",
            "frac": parts[dom]["gbs"] / peak, "peak_kind": peak_kind,
            "traffic": profiled_traffic(dom_kernel, B)}
    roof_v = {"bound": "hbm", "kernel": "aces_verify", "achieved": parts["verify_sparsify"]["gbs"], "peak": peak,
              "unit": "GB/s", "frac": parts["verify_sparsify"]["gbs"] / peak, "peak_kind": peak_kind,
              "traffic": profiled_traffic("aces_verify", B)}

    # B sweep at V = 256000 (verify + sparsify only, device-resident inputs)
    sweep = []
    if not args.no_sweep and rank == 0:
        for bs in SWEEP_B:
            if bs > B:
                continue
            sub = {key: d[key][:bs] for key in ("z", "q", "xt", "u")}
            o2 = A.verify(sub["z"], sub["q"], sub["xt"], sub["u"], w.T, w.top_p, k)
            ws2 = torch.zeros(A.workspace_bytes(bs, K, V, k), dtype=torch.uint8, device=dev)
            for _ in range(3):
                A.verify(sub["z"], sub["q"], sub["xt"], sub["u"], w.T, w.top_p, k, out=o2, workspace=ws2)
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            n = 10
            e0.record(stream)
            for _ in range(n):
                A.verify(sub["z"], sub["q"], sub["xt"], sub["u"], w.T, w.top_p, k, out=o2, workspace=ws2)
            e1.record(stream)
            torch.cuda.synchronize()
            ms = e0.elapsed_time(e1) / n
            by = verify_bytes(bs, K, V, k, zsize, resid_q_count(o2, K, k))
            sweep.append({"B": bs, "ms": ms, "rows_per_s": bs * (K + 1) / (ms * 1e-3), "gbs": by / (ms * 1e-3) / 1e9,
                          "frac_of_peak": by / (ms * 1e-3) / 1e9 / peak})

    # end to end through the public API: pinned host inputs in, results out
    e2e_steps = args.e2e_steps or min(args.steps, 30)
    res_keys = ["accept_len", "out_token", "row_status", "topk_ids", "topk_probs", "tail_mass"]
    host_out = {key: torch.empty_like(out[key], device="cpu").pin_memory() for key in res_keys}
    host_cache = {key: torch.empty_like(cache[key], device="cpu").pin_memory() for key in cache}
    host_slot = torch.empty_like(slot, device="cpu").pin_memory()
    h2d = sum(t.numel() * t.element_size() for t in host.values())
    d2h = sum(t.numel() * t.element_size() for t in host_out.values()) + \
        sum(t.numel() * t.element_size() for t in host_cache.values()) + host_slot.numel() * 4

    def e2e_step():
        for key in host:
            d[key].copy_(host[key], non_blocking=True)
        step()
        for key in res_keys:
            host_out[key].copy_(out[key], non_blocking=True)
        for key in cache:
            host_cache[key].copy_(cache[key], non_blocking=True)
        host_slot.copy_(slot, non_blocking=True)
        stream.synchronize()

    for _ in range(2):
        e2e_step()
    barrier()
    t = time.perf_counter()
    for _ in range(e2e_steps):
        e2e_step()
    barrier()
    e2e_s = max_over_ranks((time.perf_counter() - t) / e2e_steps, pg, dev)
    e2e = {"value": ws * rows / e2e_s, "unit": "rows/s", "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
           "ms_per_step": e2e_s * 1e3}

    cpu = None
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(w, inp)

    # the five paper-shaped workloads, one entry each (N = 1 only)
    pc = None
    if rank == 0 and ws == 1 and not args.no_per_config:
        del host, host_out, host_cache
        have = {w.name: (inp, d)} if w.B == gen_B(w) else None
        pc = per_config(A, torch, dev, stream, peak, peak_kind, have=have, cpu=not args.no_cpu_baseline)

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "rows/s", "n_gpus": ws, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32", "data": "synthetic", "config": config_of(w),
            "roofline": roof, "roofline_verify_sparsify": roof_v, "cpu_baseline": cpu, "e2e": e2e,
            "gpu_launches": KERNELS_PER_STEP * args.steps, "clocks": clocks.summary(), "parts": parts, "sweep": sweep,
            "per_config": pc,
        }
        print(json.dumps(line), flush=True)
    if pg is not None:
        pg.barrier()
        pg.destroy_process_group()


if __name__ == "__main__":
    main()
