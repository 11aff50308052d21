"""Host-side checks of the C ABI: the library builds, loads without a GPU,
exports every function include/acespec.h declares, sizes its workspace, and
rejects invalid arguments before touching the device."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "acespec.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2609_02514_gb300 import build
    import paper_2609_02514_gb300 as A
    build.build()
    return A.load()


def declared_functions(checked=False):
    """Functions the header declares; those of the checked build's block
    (#ifdef ACES_CHECKED) only when checked is set."""
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    if not checked:
        text = re.sub(r"#ifdef ACES_CHECKED.*?#endif", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(aces_[a-z_]+)\s*\(", text)))


def test_header_declares_the_four_entry_points():
    names = declared_functions()
    for n in ("aces_verify", "aces_sparsify", "aces_cache_build", "aces_cache_lookup",
              "aces_workspace_bytes", "aces_status_string"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name
    # the checked build's extra function is not in the product library
    extra = set(declared_functions(checked=True)) - set(declared_functions())
    assert extra == {"aces_checked_violation"}


def test_workspace_sizes(lib):
    ws = lib.aces_workspace_bytes
    assert ws(256, 16, 256000, 128) >= 256 * 17 * 32
    assert ws(1, 4, 32000, 16) > 0
    assert ws(5, 0, 100, 4) > 0            # sparsify sizing
    for bad in ((0, 4, 100, 4), (1, 17, 100, 4), (1, 4, 1, 1), (1, 4, (1 << 20) + 1, 4), (1, 4, 100, 257)):
        assert ws(*bad) == 0, bad


def test_status_strings(lib):
    assert lib.aces_status_string(0) == b"ok"
    assert lib.aces_status_string(1) == b"invalid argument"


FAKE = ctypes.c_void_p(0x10000)   # never dereferenced: validation fails first


def _verify(lib, **kw):
    a = dict(z=FAKE, dt=1, q=FAKE, xt=FAKE, u=FAKE, B=2, K=4, V=1000, T=1.0, top_p=0.9, al=FAKE, tok=FAKE,
             k=8, ids=FAKE, probs=FAKE, tail=FAKE, st=FAKE, ws=FAKE, wsb=1 << 20, s=None)
    a.update(kw)
    return lib.aces_verify(a["z"], a["dt"], a["q"], a["xt"], a["u"], a["B"], a["K"], a["V"], a["T"],
                           a["top_p"], a["al"], a["tok"], a["k"], a["ids"], a["probs"], a["tail"], a["st"],
                           a["ws"], a["wsb"], a["s"])


@pytest.mark.parametrize("kw,code", [
    (dict(B=0), 1), (dict(K=0), 1), (dict(K=17), 1), (dict(V=1), 1), (dict(V=(1 << 20) + 1), 1),
    (dict(T=0.0), 2), (dict(T=-1.0), 1), (dict(T=float("inf")), 1), (dict(T=float("nan")), 1),
    (dict(top_p=0.0), 1), (dict(top_p=1.0001), 1), (dict(top_p=float("nan")), 1),
    (dict(k=-1), 1), (dict(k=257), 1), (dict(V=10, k=11), 1), (dict(dt=7), 2),
    (dict(z=None), 1), (dict(q=None), 1), (dict(xt=None), 1), (dict(u=None), 1), (dict(al=None), 1),
    (dict(tok=None), 1), (dict(st=None), 1), (dict(ids=None), 1), (dict(ws=None), 1),
    (dict(wsb=16), 1), (dict(ws=ctypes.c_void_p(0x10008)), 1),
])
def test_verify_rejects_invalid_arguments(lib, kw, code):
    assert _verify(lib, **kw) == code


def _step(lib, **kw):
    F = (ctypes.c_int32 * 4)(2, 2, 2, 2)
    a = dict(z=FAKE, dt=1, q=FAKE, xt=FAKE, u=FAKE, B=2, K=4, V=1000, T=1.0, top_p=0.9, al=FAKE, tok=FAKE,
             k=8, ids=FAKE, probs=FAKE, tail=FAKE, st=FAKE, F=F, bt=FAKE, bp=FAKE, ws=FAKE, wsb=1 << 20, s=None)
    a.update(kw)
    return lib.aces_cloud_step(a["z"], a["dt"], a["q"], a["xt"], a["u"], a["B"], a["K"], a["V"], a["T"],
                               a["top_p"], a["al"], a["tok"], a["k"], a["ids"], a["probs"], a["tail"], a["st"],
                               a["F"], a["bt"], a["bp"], a["ws"], a["wsb"], a["s"])


@pytest.mark.parametrize("kw,code", [
    # the checks of aces_verify ...
    (dict(B=0), 1), (dict(K=17), 1), (dict(T=0.0), 2), (dict(top_p=0.0), 1), (dict(k=257), 1),
    (dict(dt=7), 2), (dict(z=None), 1), (dict(u=None), 1), (dict(ws=None), 1), (dict(wsb=16), 1),
    # ... and those of aces_cache_build, all before any launch
    (dict(F=None), 1), (dict(F=(ctypes.c_int32 * 4)(2, -1, 2, 2)), 1),
    (dict(V=5000, F=(ctypes.c_int32 * 4)(2, 2000, 2, 2)), 2), (dict(bt=None), 1), (dict(bp=None), 1),
])
def test_cloud_step_rejects_invalid_arguments(lib, kw, code):
    assert _step(lib, **kw) == code


def test_cache_calls_reject_invalid_arguments(lib):
    F = (ctypes.c_int32 * 4)(2, 2, 2, 2)
    Fbad = (ctypes.c_int32 * 4)(2, -1, 2, 2)
    Fbig = (ctypes.c_int32 * 4)(2, 2000, 2, 2)
    cb = lib.aces_cache_build
    assert cb(FAKE, FAKE, Fbad, 2, 4, 5000, FAKE, FAKE, None) == 1
    assert cb(FAKE, FAKE, Fbig, 2, 4, 5000, FAKE, FAKE, None) == 2
    assert cb(FAKE, FAKE, F, 2, 4, 2, FAKE, FAKE, None) == 1       # F_d > V - 1
    assert cb(FAKE, FAKE, None, 2, 4, 5000, FAKE, FAKE, None) == 1
    assert cb(None, FAKE, F, 2, 4, 5000, FAKE, FAKE, None) == 1
    assert cb(FAKE, FAKE, F, 2, 0, 5000, FAKE, FAKE, None) == 1
    cl = lib.aces_cache_lookup
    assert cl(FAKE, F, 2, 4, FAKE, FAKE, None, None) == 1
    assert cl(FAKE, Fbad, 2, 4, FAKE, FAKE, FAKE, None) == 1
    sp = lib.aces_sparsify
    assert sp(FAKE, 0, 4, 1000, 1.0, 0.9, 0, FAKE, FAKE, FAKE, FAKE, FAKE, 1 << 20, None) == 1   # k = 0
    assert sp(FAKE, 0, 0, 1000, 1.0, 0.9, 4, FAKE, FAKE, FAKE, FAKE, FAKE, 1 << 20, None) == 1


def test_binding_refuses_host_tensors():
    torch = pytest.importorskip("torch")
    import paper_2609_02514_gb300 as A
    z = torch.zeros(1, 3, 16)
    with pytest.raises(ValueError):
        A.verify(z, torch.zeros(1, 2, 16), torch.zeros(1, 2, dtype=torch.int32), torch.zeros(1, 3), 1.0, 0.9, 4)


def _resample(lib, **kw):
    a = dict(al=FAKE, ids=FAKE, probs=FAKE, tail=FAKE, st=FAKE, q=FAKE, u=FAKE, B=2, K=4, V=1000, k=8,
             tok=FAKE, stat=FAKE, s=None)
    a.update(kw)
    return lib.aces_resample_sparse(a["al"], a["ids"], a["probs"], a["tail"], a["st"], a["q"], a["u"], a["B"],
                                    a["K"], a["V"], a["k"], a["tok"], a["stat"], a["s"])


@pytest.mark.parametrize("kw", [
    dict(B=0), dict(K=0), dict(K=17), dict(V=1), dict(V=(1 << 20) + 1), dict(k=0), dict(k=257),
    dict(V=10, k=11), dict(al=None), dict(ids=None), dict(probs=None), dict(tail=None), dict(st=None),
    dict(q=None), dict(u=None), dict(tok=None), dict(stat=None),
])
def test_resample_sparse_rejects_invalid_arguments(lib, kw):
    assert _resample(lib, **kw) == 1


def _compact(lib, **kw):
    a = dict(kv=ctypes.c_void_p(0x10000), eb=2, planes=4, B=2, H=2, S=64, D=64, t=FAKE, al=FAKE, sl=FAKE, K=4,
             L=5, nl=FAKE, s=None)
    a.update(kw)
    return lib.aces_compact_kv(a["kv"], a["eb"], a["planes"], a["B"], a["H"], a["S"], a["D"], a["t"], a["al"],
                               a["sl"], a["K"], a["L"], a["nl"], a["s"])


@pytest.mark.parametrize("kw", [
    dict(kv=None), dict(t=None), dict(al=None), dict(sl=None), dict(nl=None), dict(eb=3), dict(planes=0),
    dict(B=0), dict(H=0), dict(S=0), dict(D=0), dict(K=0), dict(K=17), dict(L=0), dict(D=4),
    dict(kv=ctypes.c_void_p(0x10008)),
])
def test_compact_kv_rejects_invalid_arguments(lib, kw):
    assert _compact(lib, **kw) == 1


def test_tree_tokens_and_mask_validation(lib):
    F = (ctypes.c_int32 * 3)(1, 1, 0)
    assert lib.aces_tree_tokens(F, 3, 2) == 7
    assert lib.aces_tree_tokens(F, 3, 0) == -1
    assert lib.aces_tree_tokens(None, 3, 2) == -1
    Fbad = (ctypes.c_int32 * 3)(1, -1, 0)
    assert lib.aces_tree_tokens(Fbad, 3, 2) == -1
    assert lib.aces_tree_mask(F, 3, 2, None, FAKE, None) == 1
    assert lib.aces_tree_mask(F, 3, 0, FAKE, FAKE, None) == 1
