"""The workspace-free semantic fallback, adapld_semantic_topk_static().

It serves callers that can pass device pointers for their inputs and outputs
but cannot obtain any other device memory (for instance a library embedded in a
server whose GPU memory belongs to another allocator).  Its scratch is a
device array inside the library, so these tests check, through the C ABI, that
two calls in a row give the same candidates and scores as the regular entry
point with a caller workspace and as the oracle, that batches of different
sizes in a row (up to the array's limit) stay correct, that a batch above the
limit is refused, and that an expired device wait is visible through
adapld_semantic_topk_static_status().  This file is collected last on
purpose; it must pass alone in a fresh process as well as after the other GPU
tests.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle
from paper_2606_05742_gb300 import build, native, synth
from tests import parity
from tests.parity import SCORE_ATOL

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    build.build()
    return native.load()


def _device(w):
    tok = torch.from_numpy(w.tokens).cuda()
    ln = torch.from_numpy(w.lengths).cuda()
    reps = torch.from_numpy(w.reps.view(np.int16)).cuda().view(torch.bfloat16)
    q = torch.from_numpy(w.query.view(np.int16)).cuda().view(torch.bfloat16)
    return tok, ln, reps, q


def _outputs(B, k):
    return (torch.full((B, k), -7, dtype=torch.int32, device="cuda"),
            torch.full((B, k), 7.0, dtype=torch.float32, device="cuda"),
            torch.full((B,), -7, dtype=torch.int32, device="cuda"))


def _static_call(lib, w, reps, q, ln, k, tau, active=None):
    c, s, n = _outputs(w.B, k)
    rc = lib.adapld_semantic_topk_static(
        reps.data_ptr(), w.ld, w.d, q.data_ptr(), ln.data_ptr(),
        None if active is None else active.data_ptr(), w.B, k, tau, c.data_ptr(),
        s.data_ptr(), n.data_ptr(), torch.cuda.current_stream().cuda_stream)
    assert rc == 0, native.status_string(rc)
    st = ctypes.c_int32(-1)
    rc = lib.adapld_semantic_topk_static_status(ctypes.byref(st),
                                                torch.cuda.current_stream().cuda_stream)
    assert rc == 0, native.status_string(rc)
    return c.cpu().numpy(), s.cpu().numpy(), n.cpu().numpy(), st.value


def _workspace_call(w, reps, q, ln, k, tau, active=None):
    p = native.make_params(w.n_max, k, w.W, w.D)
    ws = native.allocate_workspace(w.B, w.ld, w.d, p)
    c, s, n = _outputs(w.B, k)
    native.semantic_topk(reps, q, ln, k, tau, c, s, n, ws, active=active)
    torch.cuda.synchronize()
    assert native.read_device_status(ws) == 0
    return c.cpu().numpy(), s.cpu().numpy(), n.cpu().numpy()


def _check_against_references(w, got, ref, sel, tau, oracle_seqs):
    gc, gs, gn = got
    rc, rs, rn = ref
    assert (rn[sel] == gn[sel]).all(), "counts"
    assert (rc[sel] == gc[sel]).all(), "candidates"
    if sel.any():
        assert np.abs(rs[sel] - gs[sel]).max() <= SCORE_ATOL, "scores"
    # unselected rows are left as the caller wrote them
    assert (gc[~sel] == -7).all() and (gn[~sel] == -7).all()
    rep = parity.Report()
    for b in oracle_seqs:
        length = int(w.lengths[b])
        if not sel[b] or length < 1 or length > w.ld:
            continue
        s_all = oracle.scores_all(w.reps[b], w.query[b], length)
        eps = parity.eps_rows(w.reps[b][: length - 1], w.query[b], w.d)
        parity.check_semantic_list(gc[b], gs[b], int(gn[b]), s_all, eps, w.k, tau, rep,
                                   f"seq {b}")
        oc, _ = oracle.semantic(w.reps[b], w.query[b], length, w.k, tau)
        if [int(x) for x in gc[b, : gn[b]]] != oc:
            rep.tie_resolved += 1
    assert rep.tie_resolved == 0, rep


@pytest.mark.parametrize("tau,use_active", [(0.1, True), (float("-inf"), False)])
def test_static_scratch_matches_workspace_entry_point(lib, tau, use_active):
    w = synth.make_workload(3, B=12, L=3001, d=512, nohit=0.5, seed=31,
                            lengths=[3001, 2000, 17, 1, 2999, 3001, 640, 2, 3001, 1500, 900, 3000])
    tok, ln, reps, q = _device(w)
    B, k = w.B, w.k
    active = (torch.arange(B, device="cuda") % 3 != 1).to(torch.uint8) if use_active else None
    ref = _workspace_call(w, reps, q, ln, k, tau, active)
    sel = np.ones(B, bool) if active is None else active.cpu().numpy().astype(bool)
    for call in range(2):
        gc, gs, gn, st = _static_call(lib, w, reps, q, ln, k, tau, active)
        assert st == 0, f"call {call}: device status {st}"
        _check_against_references(w, (gc, gs, gn), ref, sel, tau, range(B))
    assert (ref[2][sel] > 0).any()


def test_static_scratch_batch_sizes_in_a_row(lib):
    """The largest batch the array holds, then a small one, then the largest
    again: the plan and the slots move with B inside the shared array, so
    each call must still match the workspace entry point and the oracle."""
    big = synth.make_workload(4, B=native.STATIC_MAX_B, L=40, d=16, nohit=1.0, seed=77, V=50)
    small = synth.make_workload(2, B=5, L=1200, d=136, nohit=1.0, seed=78)
    for w, tau in ((big, float("-inf")), (small, 0.1), (big, 0.1)):
        tok, ln, reps, q = _device(w)
        ref = _workspace_call(w, reps, q, ln, w.k, tau)
        gc, gs, gn, st = _static_call(lib, w, reps, q, ln, w.k, tau)
        assert st == 0
        sel = np.ones(w.B, bool)
        seqs = range(w.B) if w.B <= 16 else range(0, w.B, 37)
        _check_against_references(w, (gc, gs, gn), ref, sel, tau, seqs)


def test_static_scratch_reports_an_expired_wait(lib, monkeypatch):
    """With the test switch the semantic kernel's producer issues no copy, so
    its bounded waits run out: the call still returns ADAPLD_OK (the failure
    is on the device), and adapld_semantic_topk_static_status() shows
    ADAPLD_DEV_TIMEOUT.  The next normal call clears the word and is correct."""
    w = synth.make_workload(2, B=4, L=3000, d=256, nohit=1.0, seed=51)
    tok, ln, reps, q = _device(w)
    monkeypatch.setenv("ADAPLD_TEST_SEMANTIC_STALL", "1")
    _, _, _, st = _static_call(lib, w, reps, q, ln, w.k, 0.1)
    assert st & native.DEV_TIMEOUT
    monkeypatch.delenv("ADAPLD_TEST_SEMANTIC_STALL")
    ref = _workspace_call(w, reps, q, ln, w.k, 0.1)
    gc, gs, gn, st = _static_call(lib, w, reps, q, ln, w.k, 0.1)
    assert st == 0
    _check_against_references(w, (gc, gs, gn), ref, np.ones(w.B, bool), 0.1, range(w.B))
    assert native.semantic_topk_static_status() == 0


def test_static_scratch_rejects_too_large_batch(lib):
    B, ld, d = native.STATIC_MAX_B + 1, 4, 8
    buf = torch.zeros(B * ld * d + 64, dtype=torch.bfloat16, device="cuda")
    ints = torch.zeros(B * 32 + 64, dtype=torch.int32, device="cuda")
    flts = torch.zeros(B * 32, dtype=torch.float32, device="cuda")
    rc = lib.adapld_semantic_topk_static(buf.data_ptr(), ld, d, buf.data_ptr(), ints.data_ptr(),
                                         None, B, 8, 0.1, ints.data_ptr(), flts.data_ptr(),
                                         ints.data_ptr(), None)
    assert rc == native.ERR_STATIC_LIMIT
    assert "1024" in native.status_string(rc)
