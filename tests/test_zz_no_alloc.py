"""The workspace-free semantic fallback, adapld_semantic_topk_static().

It serves callers that can pass device pointers for their inputs and outputs
but cannot obtain any other device memory (for instance a library embedded in a
server whose GPU memory belongs to another allocator).  Its scratch is a
device array inside the library, so this test checks, through the C ABI, that
two calls in a row give the same candidates and scores as the regular entry
point with a caller workspace, and that a batch above the array's limit is
refused.  This file is collected last on purpose; it must pass alone in a fresh
process as well as after the other GPU tests.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2606_05742_gb300 import build, native, synth
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


@pytest.mark.parametrize("tau,use_active", [(0.1, True), (float("-inf"), False)])
def test_static_scratch_matches_workspace_entry_point(lib, tau, use_active):
    w = synth.make_workload(3, B=12, L=3001, d=512, nohit=0.5, seed=31,
                            lengths=[3001, 2000, 17, 1, 2999, 3001, 640, 2, 3001, 1500, 900, 3000])
    tok, ln, reps, q = _device(w)
    B, k = w.B, w.k
    active = (torch.arange(B, device="cuda") % 3 != 1).to(torch.uint8) if use_active else None
    p = native.make_params(w.n_max, k, w.W, w.D)
    ws = native.allocate_workspace(B, w.ld, w.d, p)

    def outputs():
        return (torch.full((B, k), -7, dtype=torch.int32, device="cuda"),
                torch.full((B, k), 7.0, dtype=torch.float32, device="cuda"),
                torch.full((B,), -7, dtype=torch.int32, device="cuda"))

    ref_c, ref_s, ref_n = outputs()
    native.semantic_topk(reps, q, ln, k, tau, ref_c, ref_s, ref_n, ws, active=active)
    torch.cuda.synchronize()
    sel = np.ones(B, bool) if active is None else active.cpu().numpy().astype(bool)
    for call in range(2):
        c, s, n = outputs()
        rc = lib.adapld_semantic_topk_static(
            reps.data_ptr(), w.ld, w.d, q.data_ptr(), ln.data_ptr(),
            None if active is None else active.data_ptr(), B, k, tau, c.data_ptr(),
            s.data_ptr(), n.data_ptr(), torch.cuda.current_stream().cuda_stream)
        assert rc == 0, native.status_string(rc)
        torch.cuda.synchronize()
        rn, gn = ref_n.cpu().numpy(), n.cpu().numpy()
        rcand, gcand = ref_c.cpu().numpy(), c.cpu().numpy()
        rs, gs = ref_s.cpu().numpy(), s.cpu().numpy()
        assert (rn[sel] == gn[sel]).all(), f"call {call}: counts"
        assert (rcand[sel] == gcand[sel]).all(), f"call {call}: candidates"
        assert np.abs(rs[sel] - gs[sel]).max() <= SCORE_ATOL, f"call {call}: scores"
        # unselected rows are left as the caller wrote them
        assert (gcand[~sel] == -7).all() and (gn[~sel] == -7).all()
    assert (ref_n.cpu().numpy()[sel] > 0).any()


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
