"""AceSpec verify / sparsify / state-cache path on one GB300 GPU.

Thin Python binding of libacespec.so (declared in include/acespec.h).  The
functions below only marshal arguments: output tensors are allocated with
PyTorch on the inputs' device, pointers and the current CUDA stream are
handed to the C ABI, and every step of the computation runs in the
library's CUDA kernels.  There is no CPU fallback: calling any function
without the built library, or with host tensors, raises.

    verify(z, q, xt, u, T, top_p, k)      Sec. III-B, lossless verification
                                          fused with the sparse payload
    sparsify(z, T, top_p, k)              Sec. III-B / V-C downlink payload
    cache_build(q, xt, F)                 Sec. III-C branch cache
    cache_lookup(branch_tok, F, pi, tok)  Algorithm 1 state recovery
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

__all__ = ["load", "use_checked", "checked_violation", "lib_path", "workspace_bytes", "verify", "sparsify", "cache_build", "cache_lookup",
           "ROW_NONFINITE", "ROW_BAD_Q", "COUNTERS_OFFSET", "AcespecError"]

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB_PATH = os.path.join(_HERE, "libacespec.so")
_LIB_CHECKED = os.path.join(_HERE, "libacespec_checked.so")
_lock = threading.Lock()
_lib = None          # the library every function below calls
_libs = {}           # loaded libraries by path

# byte offset of the 16 path counters in a workspace (int32; after the hints
# a call leaves for the next one)
COUNTERS_OFFSET = 256

ROW_NONFINITE = 1
ROW_BAD_Q = 2
ACES_F32 = 0
ACES_BF16 = 1
_STATUS = {0: "ok", 1: "invalid argument", 2: "unsupported argument", 3: "CUDA launch error"}


class AcespecError(RuntimeError):
    def __init__(self, fn, code):
        super().__init__(f"{fn} failed: {_STATUS.get(code, code)} (status {code})")
        self.code = code


def lib_path() -> str:
    return _LIB_PATH


def load():
    """Load libacespec.so (built by __graft_entry__.build() or build.py)."""
    global _lib
    with _lock:
        if _lib is None:
            _lib = _open(_LIB_PATH)
        return _lib


def use_checked(on: bool = True):
    """Route every call of this module to the checked test build,
    libacespec_checked.so (built with build.build(checked=True)), or back to
    the product library.  Returns the library now in use."""
    global _lib
    with _lock:
        _lib = _open(_LIB_CHECKED if on else _LIB_PATH)
        return _lib


def checked_violation():
    """(site, index, bound) of the first out-of-range index the checked
    build met since the last call, or None; clears the record."""
    lib = load()
    if not hasattr(lib, "aces_checked_violation"):
        raise RuntimeError("the product library has no index checks: call use_checked() first")
    out = (ctypes.c_ulonglong * 3)()
    _check("aces_checked_violation", lib.aces_checked_violation(out))
    return None if out[0] == 0 else (int(out[0]), int(out[1]), int(out[2]))


def _open(path):
    if path in _libs:
        return _libs[path]
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing: build it with `python -m paper_2609_02514_gb300.build`")
    lib = ctypes.CDLL(path)
    P, I, F, S = ctypes.c_void_p, ctypes.c_int, ctypes.c_float, ctypes.c_size_t
    lib.aces_workspace_bytes.argtypes = [I, I, I, I]
    lib.aces_workspace_bytes.restype = S
    lib.aces_verify.argtypes = [P, I, P, P, P, I, I, I, F, F, P, P, I, P, P, P, P, P, S, P]
    lib.aces_verify_exact.argtypes = lib.aces_verify.argtypes
    lib.aces_sparsify.argtypes = [P, I, I, I, F, F, I, P, P, P, P, P, S, P]
    lib.aces_cache_build.argtypes = [P, P, P, I, I, I, P, P, P]
    lib.aces_cloud_step.argtypes = [P, I, P, P, P, I, I, I, F, F, P, P, I, P, P, P, P, P, P, P, P, S, P]
    lib.aces_cache_lookup.argtypes = [P, P, I, I, P, P, P, P]
    lib.aces_resample_sparse.argtypes = [P, P, P, P, P, P, P, I, I, I, I, P, P, P]
    lib.aces_compact_kv.argtypes = [P, I, I, I, I, I, I, P, P, P, I, I, P, P]
    lib.aces_tree_tokens.argtypes = [P, I, I]
    lib.aces_tree_tokens.restype = I
    lib.aces_tree_mask.argtypes = [P, I, I, P, P, P]
    lib.aces_tree_budget.argtypes = [P, I, ctypes.c_double, ctypes.c_double, I, P]
    lib.aces_branch_alloc.argtypes = [I, I, ctypes.c_double, ctypes.c_double, P]
    lib.aces_status_string.argtypes = [I]
    lib.aces_status_string.restype = ctypes.c_char_p
    for f in (lib.aces_verify, lib.aces_verify_exact, lib.aces_sparsify, lib.aces_cache_build,
              lib.aces_cache_lookup, lib.aces_resample_sparse, lib.aces_tree_budget, lib.aces_branch_alloc,
              lib.aces_compact_kv, lib.aces_tree_mask):
        f.restype = I
    if hasattr(lib, "aces_checked_violation"):
        lib.aces_checked_violation.argtypes = [P]
        lib.aces_checked_violation.restype = I
    _libs[path] = lib
    return lib


def _check(fn, code):
    if code != 0:
        raise AcespecError(fn, code)


def _cuda(t: torch.Tensor, name: str) -> torch.Tensor:
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return t


def _p(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(dev):
    return ctypes.c_void_p(torch.cuda.current_stream(dev).cuda_stream)


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.float32:
        return ACES_F32
    if t.dtype == torch.bfloat16:
        return ACES_BF16
    raise ValueError(f"target logits must be float32 or bfloat16, got {t.dtype}")


def workspace_bytes(B: int, K: int, V: int, k: int) -> int:
    return int(load().aces_workspace_bytes(int(B), int(K), int(V), int(k)))


def verify(target_logits, draft_probs, draft_tokens, uniforms, T: float, top_p: float, k: int = 0,
           out: dict | None = None, workspace: torch.Tensor | None = None, exact: bool = False):
    """Lossless verification of B drafted chains (+ sparse payload when k > 0).

    target_logits [B, K+1, V] float32/bfloat16, draft_probs [B, K, V] float32,
    draft_tokens [B, K] int32, uniforms [B, K+1] float32.
    Returns a dict of device tensors: accept_len [B], out_token [B],
    row_status [B, K+1] and, when k > 0, topk_ids / topk_probs [B, K+1, k],
    tail_mass [B, K+1].  `out` may supply preallocated outputs (same keys).
    exact=True calls aces_verify_exact (every row on the exact general
    kernel; same results, slower).
    """
    lib = load()
    z = _cuda(target_logits, "target_logits")
    q = _cuda(draft_probs, "draft_probs")
    xt = _cuda(draft_tokens, "draft_tokens")
    u = _cuda(uniforms, "uniforms")
    if z.dim() != 3:
        raise ValueError("target_logits must be [B, K+1, V]")
    B, R, V = z.shape
    K = R - 1
    if q.dtype != torch.float32 or tuple(q.shape) != (B, K, V):
        raise ValueError("draft_probs must be float32 [B, K, V]")
    if xt.dtype != torch.int32 or tuple(xt.shape) != (B, K):
        raise ValueError("draft_tokens must be int32 [B, K]")
    if u.dtype != torch.float32 or tuple(u.shape) != (B, R):
        raise ValueError("uniforms must be float32 [B, K+1]")
    dev = z.device
    o = {} if out is None else dict(out)
    i32 = dict(dtype=torch.int32, device=dev)
    f32 = dict(dtype=torch.float32, device=dev)
    o.setdefault("accept_len", torch.empty(B, **i32))
    o.setdefault("out_token", torch.empty(B, **i32))
    o.setdefault("row_status", torch.empty(B, R, **i32))
    if k > 0:
        o.setdefault("topk_ids", torch.empty(B, R, k, **i32))
        o.setdefault("topk_probs", torch.empty(B, R, k, **f32))
        o.setdefault("tail_mass", torch.empty(B, R, **f32))
    need = workspace_bytes(B, K, V, k)
    ws = workspace if workspace is not None else torch.empty(max(need, 16), dtype=torch.uint8, device=dev)
    fn = lib.aces_verify_exact if exact else lib.aces_verify
    code = fn(_p(z), _dtype_code(z), _p(q), _p(xt), _p(u), B, K, V, float(T), float(top_p),
              _p(o["accept_len"]), _p(o["out_token"]), int(k), _p(o.get("topk_ids")),
              _p(o.get("topk_probs")), _p(o.get("tail_mass")), _p(o["row_status"]),
              _p(ws), ws.numel(), _stream(dev))
    _check("aces_verify_exact" if exact else "aces_verify", code)
    return o


def sparsify(target_logits, T: float, top_p: float, k: int, out: dict | None = None,
             workspace: torch.Tensor | None = None):
    """Sparse top-k payload of every row of target_logits [rows, V] (or [..., V])."""
    lib = load()
    z = _cuda(target_logits, "target_logits")
    V = z.shape[-1]
    rows = z.numel() // V
    dev = z.device
    lead = tuple(z.shape[:-1])
    o = {} if out is None else dict(out)
    o.setdefault("topk_ids", torch.empty(*lead, k, dtype=torch.int32, device=dev))
    o.setdefault("topk_probs", torch.empty(*lead, k, dtype=torch.float32, device=dev))
    o.setdefault("tail_mass", torch.empty(*lead, dtype=torch.float32, device=dev))
    o.setdefault("row_status", torch.empty(*lead, dtype=torch.int32, device=dev))
    need = workspace_bytes(rows, 0, V, k)
    ws = workspace if workspace is not None else torch.empty(max(need, 16), dtype=torch.uint8, device=dev)
    code = lib.aces_sparsify(_p(z), _dtype_code(z), rows, V, float(T), float(top_p), int(k),
                             _p(o["topk_ids"]), _p(o["topk_probs"]), _p(o["tail_mass"]),
                             _p(o["row_status"]), _p(ws), ws.numel(), _stream(dev))
    _check("aces_sparsify", code)
    return o


def _f_host(F):
    arr = (ctypes.c_int32 * len(F))(*[int(f) for f in F])
    return arr


def cache_build(draft_probs, draft_tokens, F, out: dict | None = None):
    """Branch cache: q [B,K,V] float32, x~ [B,K] int32, F (K ints) ->
    branch_tok [B, sum F] int32, branch_prob [B, sum F] float32."""
    lib = load()
    q = _cuda(draft_probs, "draft_probs")
    xt = _cuda(draft_tokens, "draft_tokens")
    B, K, V = q.shape
    if len(F) != K:
        raise ValueError("F must have K entries")
    tot = int(sum(int(f) for f in F))
    dev = q.device
    o = {} if out is None else dict(out)
    o.setdefault("branch_tok", torch.empty(B, tot, dtype=torch.int32, device=dev))
    o.setdefault("branch_prob", torch.empty(B, tot, dtype=torch.float32, device=dev))
    code = lib.aces_cache_build(_p(q), _p(xt), _f_host(F), B, K, V, _p(o["branch_tok"]),
                                _p(o["branch_prob"]), _stream(dev))
    _check("aces_cache_build", code)
    return o


def cloud_step(target_logits, draft_probs, draft_tokens, uniforms, T: float, top_p: float, k: int, F,
               out: dict | None = None, workspace: torch.Tensor | None = None):
    """verify() and cache_build() of the same batch in one call (the cache
    build runs concurrently on the library's own stream).  Returns the keys of
    both: accept_len, out_token, row_status, the payload when k > 0,
    branch_tok and branch_prob."""
    lib = load()
    z = _cuda(target_logits, "target_logits")
    q = _cuda(draft_probs, "draft_probs")
    xt = _cuda(draft_tokens, "draft_tokens")
    u = _cuda(uniforms, "uniforms")
    if z.dim() != 3:
        raise ValueError("target_logits must be [B, K+1, V]")
    B, R, V = z.shape
    K = R - 1
    if q.dtype != torch.float32 or tuple(q.shape) != (B, K, V):
        raise ValueError("draft_probs must be float32 [B, K, V]")
    if xt.dtype != torch.int32 or tuple(xt.shape) != (B, K):
        raise ValueError("draft_tokens must be int32 [B, K]")
    if u.dtype != torch.float32 or tuple(u.shape) != (B, R):
        raise ValueError("uniforms must be float32 [B, K+1]")
    if len(F) != K:
        raise ValueError("F must have K entries")
    tot = int(sum(int(f) for f in F))
    dev = z.device
    o = {} if out is None else dict(out)
    i32 = dict(dtype=torch.int32, device=dev)
    f32 = dict(dtype=torch.float32, device=dev)
    o.setdefault("accept_len", torch.empty(B, **i32))
    o.setdefault("out_token", torch.empty(B, **i32))
    o.setdefault("row_status", torch.empty(B, R, **i32))
    if k > 0:
        o.setdefault("topk_ids", torch.empty(B, R, k, **i32))
        o.setdefault("topk_probs", torch.empty(B, R, k, **f32))
        o.setdefault("tail_mass", torch.empty(B, R, **f32))
    o.setdefault("branch_tok", torch.empty(B, tot, **i32))
    o.setdefault("branch_prob", torch.empty(B, tot, **f32))
    need = workspace_bytes(B, K, V, k)
    ws = workspace if workspace is not None else torch.empty(max(need, 16), dtype=torch.uint8, device=dev)
    code = lib.aces_cloud_step(_p(z), _dtype_code(z), _p(q), _p(xt), _p(u), B, K, V, float(T), float(top_p),
                               _p(o["accept_len"]), _p(o["out_token"]), int(k), _p(o.get("topk_ids")),
                               _p(o.get("topk_probs")), _p(o.get("tail_mass")), _p(o["row_status"]), _f_host(F),
                               _p(o["branch_tok"]), _p(o["branch_prob"]), _p(ws), ws.numel(), _stream(dev))
    _check("aces_cloud_step", code)
    return o


def cache_lookup(branch_tok, F, accept_len, token, out: torch.Tensor | None = None):
    """slot [B] int32: off_pi + j on a hit, -1 on a miss, -2 when pi == K."""
    lib = load()
    bt = _cuda(branch_tok, "branch_tok")
    al = _cuda(accept_len, "accept_len")
    tk = _cuda(token, "token")
    B = al.shape[0]
    K = len(F)
    slot = out if out is not None else torch.empty(B, dtype=torch.int32, device=al.device)
    code = lib.aces_cache_lookup(_p(bt), _f_host(F), B, K, _p(al), _p(tk), _p(slot), _stream(al.device))
    _check("aces_cache_lookup", code)
    return slot


def resample_sparse(accept_len, topk_ids, topk_probs, tail_mass, row_status, draft_probs, uniforms,
                    out: dict | None = None):
    """Edge-side draw from the sparse payload of row pi (Alg. 1 RESAMPLE).

    accept_len [B], topk_ids / topk_probs [B,K+1,k], tail_mass / row_status
    [B,K+1] (as written by verify), draft_probs [B,K,V] float32, uniforms
    [B,K+1] float32 -> token [B] int32, status [B] int32.
    """
    lib = load()
    al = _cuda(accept_len, "accept_len")
    ids = _cuda(topk_ids, "topk_ids")
    pr = _cuda(topk_probs, "topk_probs")
    tl = _cuda(tail_mass, "tail_mass")
    st = _cuda(row_status, "row_status")
    q = _cuda(draft_probs, "draft_probs")
    u = _cuda(uniforms, "uniforms")
    B, K, V = q.shape
    k = ids.shape[-1]
    dev = q.device
    o = {} if out is None else dict(out)
    o.setdefault("token", torch.empty(B, dtype=torch.int32, device=dev))
    o.setdefault("status", torch.empty(B, dtype=torch.int32, device=dev))
    code = lib.aces_resample_sparse(_p(al), _p(ids), _p(pr), _p(tl), _p(st), _p(q), _p(u), B, K, V, k,
                                    _p(o["token"]), _p(o["status"]), _stream(dev))
    _check("aces_resample_sparse", code)
    return o


def tree_budget(draft_latency_s, rtt_s: float, verify_s: float, B_max: int) -> int:
    """Network-aware budget B* (Sec. IV-B) from the drafting times of tree sizes 1..n."""
    lib = load()
    n = len(draft_latency_s)
    arr = (ctypes.c_double * n)(*[float(t) for t in draft_latency_s])
    out = ctypes.c_int(0)
    _check("aces_tree_budget", lib.aces_tree_budget(arr, n, float(rtt_s), float(verify_s), int(B_max),
                                                    ctypes.byref(out)))
    return int(out.value)


def branch_alloc(B_alloc: int, gamma: int, alpha: float, beta: float) -> list:
    """Integer branch counts F_0..F_{gamma-1} of the geometric-decay allocation (Sec. IV-C)."""
    lib = load()
    F = (ctypes.c_int32 * int(gamma))()
    _check("aces_branch_alloc", lib.aces_branch_alloc(int(B_alloc), int(gamma), float(alpha), float(beta), F))
    return [int(f) for f in F]


def compact_kv(kv, prefix_len, accept_len, slot, K: int, branch_len: int, new_len: torch.Tensor | None = None):
    """COMPACT_KV / ROLLBACK_KV (Alg. 1) in place on kv [planes, B, H, S, D];
    returns new_len [B] int32."""
    lib = load()
    kv = _cuda(kv, "kv")
    t = _cuda(prefix_len, "prefix_len")
    al = _cuda(accept_len, "accept_len")
    sl = _cuda(slot, "slot")
    planes, B, H, S, D = kv.shape
    out = new_len if new_len is not None else torch.empty(B, dtype=torch.int32, device=kv.device)
    code = lib.aces_compact_kv(_p(kv), kv.element_size(), planes, B, H, S, D, _p(t), _p(al), _p(sl), int(K),
                               int(branch_len), _p(out), _stream(kv.device))
    _check("aces_compact_kv", code)
    return out


def tree_mask(F, branch_len: int, device=None):
    """Tree attention mask (Sec. III-C): mask [n, ceil(n/32)] int32 words (bit
    j of word w: key 32 w + j allowed) and depth [n] int32 on the device."""
    lib = load()
    K = len(F)
    n = int(lib.aces_tree_tokens(_f_host(F), K, int(branch_len)))
    if n < 0:
        raise ValueError("invalid tree shape")
    dev = torch.device("cuda") if device is None else torch.device(device)
    mask = torch.empty(n, (n + 31) // 32, dtype=torch.int32, device=dev)
    depth = torch.empty(n, dtype=torch.int32, device=dev)
    _check("aces_tree_mask", lib.aces_tree_mask(_f_host(F), K, int(branch_len), _p(mask), _p(depth),
                                                _stream(dev)))
    return mask, depth
