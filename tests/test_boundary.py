"""The C-ABI boundary without a GPU: the library builds, loads and exports every
function declared in include/adapld.h, and argument errors are reported with
the documented codes before anything is enqueued (every call here fails
validation, so no CUDA work is attempted)."""
import ctypes
import os
import re

import pytest

from paper_2606_05742_gb300 import build, native

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "adapld.h")


@pytest.fixture(scope="module")
def lib():
    build.build()
    return native.load()


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"^[A-Za-z_][\w\s\*]*?\b(adapld_\w+)\s*\(", src, flags=re.M)))


def test_header_declares_expected_entry_points():
    decl = declared_functions()
    for name in ("adapld_lexical_match", "adapld_semantic_topk", "adapld_build_draft_tree",
                 "adapld_step"):
        assert name in decl
    assert sorted(native.EXPORTED) == decl


def test_library_exports_every_declared_symbol(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name


def test_checked_build_exports_every_declared_symbol():
    """The checked debug build (every kernel index tested) has the same ABI."""
    chk = native.load_library(build.build(checked=True))
    for name in declared_functions():
        assert hasattr(chk, name), name
    assert chk.adapld_status_string(-9) == native.load().adapld_status_string(-9)


def test_status_strings(lib):
    for code in (0, -1, -2, -3, -4, -5, -6, -7, -8, -9, -10, -11, -12, -13, -14, -15, -16, -17,
                 -20):
        s = native.status_string(code)
        assert s and s != "unknown status"
    assert native.status_string(-999) == "unknown status"


def test_tree_nodes_and_workspace(lib):
    p = native.make_params(5, 32, 4, 16, 1)
    assert native.tree_nodes(p) == 1 + 16 + 4 * 2
    assert native.workspace_bytes(8, 131072, 8192, p) > 0
    assert native.workspace_bytes(0, 10, 8, p) == 0          # bad B
    assert native.workspace_bytes(1, 10, 12, p) == 0         # d % 8 != 0
    assert native.workspace_bytes(1, 10, 16392, p) == 0      # d too large
    assert native.workspace_bytes(1, 1 << 31, 8, p) == 0     # B*ld too large
    assert native.workspace_bytes(1, 0, 8, p) == 0           # bad ld


FAKE = 1 << 20  # a 16-byte aligned non-null address; never dereferenced here


def _step(lib, **kw):
    a = dict(tokens=FAKE, ld=64, lengths=FAKE, reps=FAKE, d=16, query=FAKE, next_topk=None, Kn=0,
             B=2, p=native.make_params(3, 8, 2, 8), ws=FAKE, ws_bytes=1 << 30)
    a.update(kw)
    so = native.StepOut(FAKE, FAKE, FAKE, FAKE, FAKE, None,
                        native.TreeOut(FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, None))
    if "out" in kw:
        so = kw["out"]
    return lib.adapld_step(a["tokens"], a["ld"], a["lengths"], a["reps"], a["d"], a["query"],
                           a["next_topk"], a["Kn"], a["B"], ctypes.byref(a["p"]),
                           ctypes.byref(so), a["ws"], a["ws_bytes"], None)


@pytest.mark.parametrize("kw,code", [
    (dict(tokens=None), -1),
    (dict(reps=None), -1),
    (dict(B=0), -2),
    (dict(B=65536, ld=1), -2),
    (dict(p=native.make_params(0, 8, 2, 8)), -3),
    (dict(p=native.make_params(9, 8, 2, 8)), -3),
    (dict(p=native.make_params(3, 0, 2, 8)), -4),
    (dict(p=native.make_params(3, 33, 2, 8)), -4),
    (dict(p=native.make_params(3, 8, -1, 8)), -5),
    (dict(p=native.make_params(3, 8, 65, 8)), -5),
    (dict(p=native.make_params(3, 8, 2, 0)), -6),
    (dict(p=native.make_params(3, 8, 2, 257)), -6),
    (dict(d=12), -7),
    (dict(d=0), -7),
    (dict(reps=FAKE + 4), -8),
    (dict(query=FAKE + 8), -8),
    (dict(ws=None), -9),
    (dict(ws_bytes=16), -9),
    (dict(ld=0), -10),
    (dict(ld=1 << 31), -11),
    (dict(p=native.make_params(3, 8, 64, 256, 16)), -11),
    (dict(p=native.make_params(3, 8, 2, 8, 0)), -12),
    (dict(p=native.make_params(3, 8, 2, 8, 17)), -12),
    (dict(next_topk=FAKE, Kn=0), -13),
    (dict(next_topk=FAKE, Kn=65), -13),
    (dict(p=native.make_params(3, 8, 2, 8, 1, float("nan"))), -14),
])
def test_step_argument_errors(lib, kw, code):
    assert _step(lib, **kw) == code


def test_step_null_outputs(lib):
    so = native.StepOut(FAKE, FAKE, None, FAKE, FAKE, None,
                        native.TreeOut(FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, None))
    assert _step(lib, out=so) == -1
    so = native.StepOut(FAKE, FAKE, FAKE, FAKE, FAKE, None,
                        native.TreeOut(FAKE, FAKE, FAKE, FAKE, None, FAKE, None))
    assert _step(lib, out=so) == -1


def test_entry_point_argument_errors(lib):
    L = lib
    assert L.adapld_lexical_match(FAKE, 64, FAKE, 0, 3, 8, FAKE, FAKE, FAKE, FAKE, FAKE,
                                  1 << 30, None) == -2
    assert L.adapld_lexical_match(FAKE, 64, FAKE, 2, 9, 8, FAKE, FAKE, FAKE, FAKE, FAKE,
                                  1 << 30, None) == -3
    assert L.adapld_lexical_match(FAKE, 64, FAKE, 2, 3, 8, None, FAKE, FAKE, FAKE, FAKE,
                                  1 << 30, None) == -1
    assert L.adapld_lexical_match(FAKE, 64, FAKE, 2, 3, 8, FAKE, FAKE, FAKE, FAKE, FAKE,
                                  8, None) == -9
    assert L.adapld_semantic_topk(FAKE, 64, 16, FAKE, FAKE, None, 2, 40, 0.1, FAKE, FAKE, FAKE,
                                  FAKE, 1 << 30, None) == -4
    assert L.adapld_semantic_topk(FAKE + 2, 64, 16, FAKE, FAKE, None, 2, 8, 0.1, FAKE, FAKE,
                                  FAKE, FAKE, 1 << 30, None) == -8
    assert L.adapld_semantic_topk(FAKE, 64, 20, FAKE, FAKE, None, 2, 8, 0.1, FAKE, FAKE, FAKE,
                                  FAKE, 1 << 30, None) == -7
    to = native.TreeOut(FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, None)
    p = native.make_params(3, 8, 2, 8)
    assert L.adapld_build_draft_tree(FAKE, 64, FAKE, FAKE, 16, FAKE, 2, FAKE, FAKE, FAKE, FAKE,
                                     None, 0, None, ctypes.byref(p), None, None, FAKE, 1 << 30,
                                     None) == -1
    bad = native.make_params(3, 8, 2, 8, 1)
    bad.k = 0
    assert L.adapld_build_draft_tree(FAKE, 64, FAKE, FAKE, 16, FAKE, 2, FAKE, FAKE, FAKE, FAKE,
                                     None, 0, None, ctypes.byref(bad), ctypes.byref(to), None,
                                     FAKE, 1 << 30, None) == -4
    for e in (native.Embeddings(None, 10, 16), native.Embeddings(FAKE + 2, 10, 16),
              native.Embeddings(FAKE, 0, 16), native.Embeddings(FAKE, 10, 12)):
        assert L.adapld_build_draft_tree(FAKE, 64, FAKE, FAKE, 16, FAKE, 2, FAKE, FAKE, FAKE,
                                         FAKE, None, 0, ctypes.byref(e), ctypes.byref(p),
                                         ctypes.byref(to), None, FAKE, 1 << 30, None) == -16
        assert L.adapld_embedding_topk(FAKE, 64, FAKE, ctypes.byref(e), None, 2, 8, 0.1, FAKE,
                                       FAKE, FAKE, None, FAKE, 1 << 30, None) == -16
    good = native.Embeddings(FAKE, 10, 16)
    assert L.adapld_embedding_topk(FAKE, 64, FAKE, None, None, 2, 8, 0.1, FAKE, FAKE, FAKE,
                                   None, FAKE, 1 << 30, None) == -1
    assert L.adapld_embedding_topk(FAKE, 64, FAKE, ctypes.byref(good), None, 2, 0, 0.1, FAKE,
                                   FAKE, FAKE, None, FAKE, 1 << 30, None) == -4
    v = ctypes.c_int32(0)
    assert L.adapld_read_device_status(None, ctypes.byref(v), None) == -1


def _accept(lib, **kw):
    a = dict(logits=FAKE, V=64, draft_tokens=FAKE, parents=FAKE, n_nodes=FAKE, B=2, N=8,
             n_accept=FAKE, new_tokens=FAKE, n_new=FAKE, tokens=None, ld=0, lengths=None,
             node_reps=None, reps=None, d=0, query=None, status=None, ws=FAKE,
             ws_bytes=1 << 30)
    a.update(kw)
    return lib.adapld_accept_greedy(*a.values(), None)


@pytest.mark.parametrize("kw,code", [
    (dict(logits=None), -1),
    (dict(n_new=None), -1),
    (dict(tokens=FAKE), -1),                       # tokens without lengths
    (dict(lengths=FAKE), -1),
    (dict(tokens=FAKE, lengths=FAKE, ld=16, node_reps=FAKE, d=16), -1),  # no reps/query
    (dict(B=0), -2),
    (dict(B=65536), -2),
    (dict(N=0), -11),
    (dict(N=1025), -11),
    (dict(V=0), -17),
    (dict(V=60), -17),
    (dict(logits=FAKE + 2), -17),
    (dict(tokens=FAKE, lengths=FAKE, ld=0), -10),
    (dict(tokens=FAKE, lengths=FAKE, ld=16, node_reps=FAKE, reps=FAKE, query=FAKE, d=12), -7),
    (dict(tokens=FAKE, lengths=FAKE, ld=16, node_reps=FAKE + 8, reps=FAKE, query=FAKE, d=16),
     -8),
    (dict(ws=None), -9),
    (dict(ws_bytes=64), -9),
    (dict(ws=FAKE + 4), -8),
])
def test_accept_argument_errors(lib, kw, code):
    assert _accept(lib, **kw) == code


def test_step_from_host_argument_errors(lib):
    p = native.make_params(3, 8, 2, 8)
    so = native.StepOut(FAKE, FAKE, FAKE, FAKE, FAKE, None,
                        native.TreeOut(FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, None))
    args = [FAKE, 64, FAKE, FAKE, 16, FAKE, 2, ctypes.byref(p), FAKE, FAKE, FAKE, FAKE,
            ctypes.byref(so), ctypes.byref(so), FAKE, 1 << 30, None]
    for i in (0, 2, 3, 5, 8, 9, 10, 11, 12, 13):     # each required pointer
        bad = list(args)
        bad[i] = None
        assert lib.adapld_step_from_host(*bad) == -1, i
    bad = list(args)
    bad[6] = 0
    assert lib.adapld_step_from_host(*bad) == -2
    bad = list(args)
    bad[4] = 12
    assert lib.adapld_step_from_host(*bad) == -7
    # the step's own checks on the device buffers also run before the first
    # copy: without a GPU an enqueued copy would fail with ADAPLD_ERR_CUDA
    # (-20), so each of these codes shows that nothing was enqueued
    bad = list(args)
    bad[14] = None                                   # no workspace
    assert lib.adapld_step_from_host(*bad) == -9
    bad = list(args)
    bad[15] = 64                                     # workspace too small
    assert lib.adapld_step_from_host(*bad) == -9
    bad = list(args)
    bad[14] = FAKE + 4                               # misaligned workspace
    assert lib.adapld_step_from_host(*bad) == -8
    bad = list(args)
    bad[10] = FAKE + 2                               # misaligned device reps
    assert lib.adapld_step_from_host(*bad) == -8
    bad = list(args)
    bad[11] = FAKE + 8                               # misaligned device query
    assert lib.adapld_step_from_host(*bad) == -8
    so_missing = native.StepOut(FAKE, FAKE, None, FAKE, FAKE, None,
                                native.TreeOut(FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, None))
    bad = list(args)
    bad[12] = ctypes.byref(so_missing)               # a required device output
    assert lib.adapld_step_from_host(*bad) == -1
    bad = list(args)
    p_bad = native.make_params(3, 40, 2, 8)          # k out of range
    bad[7] = ctypes.byref(p_bad)
    assert lib.adapld_step_from_host(*bad) == -4


def test_binding_fails_loudly_without_library(monkeypatch, tmp_path):
    monkeypatch.setattr(native, "LIB_PATH", str(tmp_path / "missing.so"))
    monkeypatch.setattr(native, "_lib", None)
    with pytest.raises(RuntimeError, match="no CPU fallback"):
        native.load()
