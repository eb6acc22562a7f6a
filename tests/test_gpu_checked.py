"""The checked debug build (libadapld_checked.so, -DADAPLD_CHECKED): every
computed index in the kernels is tested before the access it guards, and a
failure raises ADAPLD_DEV_INTERNAL instead of touching memory.  It stands in
for a memory checker on this GPU.  Small parity workloads of every kind run
through it: no check may fire (device status 0) and every output must equal
the normal build's bit for bit (the checks change no arithmetic); the normal
build's outputs are the ones the parity tests compare with the oracle."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_05742_gb300 import build, native, synth

pytestmark = pytest.mark.gpu
NEG_INF = float("-inf")


@pytest.fixture(scope="module")
def libs():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    build.build()
    normal = native.load()
    checked = native.load_library(build.build(checked=True))
    return normal, checked


def _step(w, P, emb=None, next_topk=None):
    tok = torch.from_numpy(np.ascontiguousarray(w.tokens)).cuda()
    ln = torch.from_numpy(np.ascontiguousarray(w.lengths)).cuda()
    reps = torch.from_numpy(np.ascontiguousarray(w.reps).view(np.int16)).cuda().view(
        torch.bfloat16)
    q = torch.from_numpy(np.ascontiguousarray(w.query).view(np.int16)).cuda().view(torch.bfloat16)
    E = torch.from_numpy(emb.view(np.int16)).cuda().view(torch.bfloat16) if emb is not None else None
    nt = torch.from_numpy(next_topk).cuda() if next_topk is not None else None
    p = native.make_params(P["n_max"], P["k"], P["W"], P["D"], P["succ_len"], P["tau"],
                           P["flags"])
    eng = native.Engine(w.B, w.ld, w.d, p)
    eng.run(tok, ln, reps, q, next_topk=nt, emb=E)
    torch.cuda.synchronize()
    return eng.out.to_host(), native.read_device_status(eng.ws)


def _both(libs, monkeypatch, w, P, **kw):
    normal, checked = libs
    monkeypatch.setattr(native, "_lib", normal)
    ref, st = _step(w, P, **kw)
    assert st == 0
    monkeypatch.setattr(native, "_lib", checked)
    got, st = _step(w, P, **kw)
    monkeypatch.setattr(native, "_lib", normal)
    assert st == 0, f"a checked index failed (device status {st})"
    for key in ref:
        assert np.array_equal(ref[key], got[key], equal_nan=True), key


def _P(w, **over):
    P = dict(n_max=w.n_max, k=w.k, W=w.W, D=w.D, succ_len=w.succ_len, tau=w.tau, flags=0)
    P.update(over)
    return P


CASES = [  # (cfg, B, L, d, seed, overrides)
    (1, 3, 2048, 256, 1, {}), (2, 8, 1500, 128, 0, {}), (3, 6, 2500, 640, 0, {}),
    (4, 40, 300, 8, 3, {}), (5, 4, 4000, 256, 0, {"tau": NEG_INF}),
    (5, 4, 20000, 64, 2, {"W": 8, "k": 32, "flags": oracle.SUCC_ON_STRICT}),
    (5, 3, 70001, 32, 4, {"n_max": 8, "tau": NEG_INF}),
    (2, 5, 300, 64, 5, {"W": 64, "k": 32, "D": 200, "succ_len": 4}),
    (4, 300, 40, 16, 6, {}),
]


@pytest.mark.parametrize("cfg,B,L,d,seed,over", CASES)
def test_checked_build_single_cache(libs, monkeypatch, cfg, B, L, d, seed, over):
    w = synth.make_workload(cfg, B=B, L=L, d=d, seed=seed, nohit=0.5,
                            lengths=[L] + [max(1, L - 37 * i) for i in range(1, B)])
    _both(libs, monkeypatch, w, _P(w, **over))


@pytest.mark.parametrize("cfg,B,L,d,de,V,seed", [(2, 8, 1500, 128, 64, 4096, 0),
                                                 (4, 20, 500, 64, 8, 2048, 3),
                                                 (5, 3, 20000, 64, 256, 4096, 5),
                                                 (4, 150, 300, 32, 64, 2500, 12)])
def test_checked_build_embeddings(libs, monkeypatch, cfg, B, L, d, de, V, seed):
    w = synth.make_workload(cfg, B=B, L=L, d=d, V=V, seed=seed, nohit=0.6)
    E = synth.make_embeddings(w, V, de, seed)
    for flags in (0, oracle.SUCC_ON_STRICT):
        _both(libs, monkeypatch, w, _P(w, flags=flags), emb=E)


def test_checked_build_next_token_table(libs, monkeypatch):
    w = synth.make_workload(3, B=5, L=900, d=64, seed=9, nohit=0.4, V=500)
    tk = synth.make_next_topk(w.tokens, w.lengths, 500, 6, seed=9)
    _both(libs, monkeypatch, w, _P(w), next_topk=tk)
