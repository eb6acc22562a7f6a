"""GPU parity: the CUDA path (through the C ABI) against the CPU oracle on the
same seeded inputs.  Integer outputs bit-exact, scores within 1e-2, cosine
decisions tie-tolerant within the fp32 error bound (see tests/parity.py)."""
import ctypes
import os
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import pytest
import torch

import oracle
from paper_2606_05742_gb300 import build, native, synth
from tests import parity
from tests.conftest import load_golden

pytestmark = pytest.mark.gpu
NEG_INF = float("-inf")


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    build.build()
    native.load()


def to_dev(w):
    """numpy workload -> torch CUDA tensors (tokens, lengths, reps, query)."""
    tok = torch.from_numpy(np.ascontiguousarray(w.tokens)).cuda()
    ln = torch.from_numpy(np.ascontiguousarray(w.lengths)).cuda()
    reps = torch.from_numpy(np.ascontiguousarray(w.reps).view(np.int16)).cuda().view(torch.bfloat16)
    q = torch.from_numpy(np.ascontiguousarray(w.query).view(np.int16)).cuda().view(torch.bfloat16)
    return tok, ln, reps, q


def P_of(w, tau=None, flags=0, **over):
    P = dict(n_max=w.n_max, k=w.k, W=w.W, D=w.D, succ_len=w.succ_len,
             tau=w.tau if tau is None else tau, flags=flags)
    P.update(over)
    return P


def params(P):
    return native.make_params(P["n_max"], P["k"], P["W"], P["D"], P["succ_len"], P["tau"],
                              P["flags"])


def run_step(w, P, next_topk=None, emb=None):
    tok, ln, reps, q = to_dev(w)
    eng = native.Engine(w.B, w.ld, w.d, params(P))
    nt = torch.from_numpy(next_topk).cuda() if next_topk is not None else None
    E = torch.from_numpy(emb.view(np.int16)).cuda().view(torch.bfloat16) if emb is not None else None
    eng.run(tok, ln, reps, q, next_topk=nt, emb=E)
    torch.cuda.synchronize()
    assert native.read_device_status(eng.ws) == 0
    return eng.out.to_host()


def succ_extensions(g, b):
    n = int(g["n_nodes"][b])
    par = g["parents"][b, :n]
    heads = [i for i in range(1, n) if par[i] == 0]
    if g["hit_kind"][b] == oracle.LEX:
        heads = [i for i in heads if i != 1]
    return sum(1 for h in heads if (par == h).any())


def check_all(w, g, P, next_topk=None, full_eps=True, seqs=None, emb=None, ties=0):
    """Every sequence (or `seqs`) against the oracle.  `ties` is the number of
    sequences whose GPU result may differ from the oracle's only inside an
    fp32 near-tie (see tests/parity.py); None leaves it unchecked (inputs
    built to be tie-heavy)."""
    rep = parity.Report()
    seqs = range(w.B) if seqs is None else seqs
    for b in seqs:
        parity.compare_sequence(b, w.tokens[b], int(w.lengths[b]), w.ld, w.reps[b], w.query[b],
                                g, P, rep, None if next_topk is None else next_topk[b],
                                full_eps, emb)
    hk = g["hit_kind"]
    exp_stats = [int((hk == 1).sum()), int((hk == 2).sum()), int(w.B - (hk == 1).sum() - (hk == 2).sum()),
                 sum(succ_extensions(g, b) for b in range(w.B))]
    assert g["stats"].tolist() == exp_stats
    if ties is not None:
        assert rep.tie_resolved == ties, rep
    return rep


def compare_device_workload(w, g, P, emb=None):
    """Every sequence of a workload generated on the device against the
    oracle (per-row error bounds), on a host thread pool: the oracle is C and
    releases the GIL, and numpy's bound computation mostly does too.  Each
    sequence's rows are copied to the host by its own worker."""
    tokens = w.tokens.cpu().numpy()
    lengths = w.lengths.cpu().numpy()

    def one(b):
        rep = parity.Report()
        R = w.reps[b].view(torch.int16).cpu().numpy().view(np.uint16)
        q = w.query[b].view(torch.int16).cpu().numpy().view(np.uint16)
        parity.compare_sequence(b, tokens[b], int(lengths[b]), w.ld, R, q, g, P, rep,
                                full_eps=True, emb=emb)
        return rep

    workers = max(1, min(w.B, os.cpu_count() or 4, 16))
    with ThreadPoolExecutor(max_workers=workers) as ex:
        rep = parity.Report.merge(ex.map(one, range(w.B)))
    assert rep.exact + rep.tie_resolved == w.B
    return rep


def bf16_rows(rows, d):
    out = np.zeros((len(rows), d), np.float32)
    for i, r in enumerate(rows):
        out[i, : len(r)] = r
    return synth.f32_to_bf16_bits(out)


def single(tokens, R, q, n_max, k, W, D, succ_len=1, tau=0.1):
    L, d = R.shape
    return synth.Workload(0, 1, L, d, n_max, k, W, D, succ_len, tau,
                          np.asarray(tokens, np.int32)[None], np.array([L], np.int32), R[None],
                          q[None], np.array([], int))


# ---------------------------------------------------------------- golden cases
def test_worked_example_lexical():
    g0 = load_golden("worked_example_lexical.txt")
    M = [int(x) for x in g0["tokens"]]
    L, d = len(M), 8
    row = synth.f32_to_bf16_bits(np.random.default_rng(0).standard_normal(d).astype(np.float32))
    R = np.tile(row, (L, 1))
    w = single(M, R, R[L - 1], 2, 8, 2, 8)
    g = run_step(w, P_of(w))
    n = int(g["n_nodes"][0])
    assert g["hit_kind"][0] == 1 and g["match_n"][0] == 2
    assert g["cand"][0, : g["n_cand"][0]].tolist() == [int(x) for x in g0["cand"]]
    assert g["draft_tokens"][0, :n].tolist() == [int(x) for x in g0["tree_tokens"]]
    assert g["parents"][0, :n].tolist() == [int(x) for x in g0["tree_parents"]]
    assert g["positions"][0, :n].tolist() == [int(x) for x in g0["tree_positions"]]
    for i in range(n):
        assert np.flatnonzero(g["mask"][0, i]).tolist() == [int(x) for x in g0[f"mask_row{i}"]]
    check_all(w, g, P_of(w))


def test_worked_example_semantic():
    g0 = load_golden("worked_example_semantic.txt")
    M = [int(x) for x in g0["tokens"]]
    L = len(M)
    R = bf16_rows([[float(x) for x in g0[f"row{i}"]] for i in range(L)], 8)
    q = bf16_rows([[float(x) for x in g0["query"]]], 8)[0]
    w = single(M, R, q, 3, 3, 2, 4)
    g = run_step(w, P_of(w))
    n = int(g["n_nodes"][0])
    assert g["hit_kind"][0] == 2
    assert g["cand"][0, :3].tolist() == [int(x) for x in g0["cand"]]
    np.testing.assert_allclose(g["score"][0, :3], [float(x) for x in g0["score"]], atol=1e-6)
    assert g["draft_tokens"][0, :n].tolist() == [int(x) for x in g0["tree_tokens"]]
    assert g["parents"][0, :n].tolist() == [int(x) for x in g0["tree_parents"]]
    assert g["positions"][0, :n].tolist() == [int(x) for x in g0["tree_positions"]]
    assert g["stats"].tolist() == [0, 1, 0, 2]
    check_all(w, g, P_of(w))


# ------------------------------------------------------ seeded small workloads
SMALL = [  # (cfg, B, L, d, seed)
    (1, 1, 700, 64, 0), (1, 3, 2048, 256, 1), (2, 8, 1500, 128, 0), (2, 6, 3000, 520, 2),
    (3, 6, 2500, 640, 0), (4, 24, 600, 96, 0), (4, 40, 300, 8, 3), (5, 4, 4000, 256, 0),
]


@pytest.mark.parametrize("cfg,B,L,d,seed", SMALL)
def test_small_workloads(cfg, B, L, d, seed):
    rng = np.random.default_rng(seed)
    lengths = rng.integers(max(2, L // 3), L + 1, size=B).astype(np.int32)
    lengths[0] = L
    w = synth.make_workload(cfg, B=B, L=L, d=d, ld=L + 5, lengths=lengths, seed=seed)
    for tau in (0.1, NEG_INF):
        P = P_of(w, tau=tau)
        check_all(w, run_step(w, P), P)


@pytest.mark.parametrize("d", [8, 136, 2048, 2056, 4096, 4104, 5120, 6144, 6152, 8192, 8200,
                               12288, 12296, 16384])
def test_every_dimension_variant(d):
    L = 96 if d > 4096 else 300
    w = synth.make_workload(3, B=4, L=L, d=d, nohit=0.75, seed=d)
    for tau in (0.1, NEG_INF):
        P = P_of(w, tau=tau)
        check_all(w, run_step(w, P), P)


def test_rows_spread_over_all_ctas():
    """Far more rows than CTAs: every CTA range straddles sequence boundaries."""
    w = synth.make_workload(2, B=5, L=30011, d=64, nohit=1.0, seed=5,
                            lengths=[30011, 17, 29000, 1, 12345])
    for tau in (0.1, NEG_INF):
        P = P_of(w, tau=tau, k=32)
        check_all(w, run_step(w, P), P)


def test_many_short_sequences():
    """Thousands of short sequences: plans and tickets over B far above the
    CTA count and a block's width, in both retrieval modes."""
    V = 2000
    w = synth.make_workload(4, B=3000, L=40, d=16, V=V, nohit=0.5, seed=7)
    P = P_of(w)
    check_all(w, run_step(w, P), P)
    E = synth.make_embeddings(w, V, 16, 7)
    check_all(w, run_step(w, P, emb=E), P, emb=E)


def test_fewer_rows_than_ctas():
    w = synth.make_workload(2, B=3, L=9, d=16, nohit=1.0, seed=6, lengths=[9, 4, 2])
    for tau in (0.1, NEG_INF):
        P = P_of(w, tau=tau)
        check_all(w, run_step(w, P), P)


def test_exact_ties_break_to_recent():
    """Identical rows give identical fp32 scores: order must be by position."""
    L, d = 400, 64
    M = np.arange(L, dtype=np.int32) % 97
    M[-1] = 1000                              # no lexical hit
    rng = np.random.default_rng(3)
    R = synth.f32_to_bf16_bits(rng.standard_normal((L, d)).astype(np.float32))
    R[5:: 7] = R[0]
    q = R[0].copy()
    w = single(M, R, q, 3, 32, 3, 6)
    P = P_of(w, tau=NEG_INF)
    g = run_step(w, P)
    tied = sorted([j for j in range(L - 1) if (R[j] == R[0]).all()], reverse=True)[:32]
    assert g["cand"][0].tolist() == tied
    check_all(w, g, P)


@pytest.mark.parametrize("lengths", [[0, 1, 2, 3, 50, 51], [1, 1, 1, 1, 1, 1], [2, 2, 3, 3, 4, 4]])
@pytest.mark.parametrize("n_max,k,W", [(8, 1, 0), (1, 3, 3), (4, 32, 64)])
def test_edge_lengths(lengths, n_max, k, W):
    w = synth.make_workload(4, B=6, L=50, d=16, ld=50, seed=9, nohit=0.5,
                            lengths=[min(x, 50) for x in lengths])
    w.lengths = np.asarray(lengths, np.int32)   # 51 > ld: invalid on purpose
    P = P_of(w, n_max=n_max, k=k, W=W, tau=NEG_INF)
    check_all(w, run_step(w, P), P)


@pytest.mark.parametrize("flags", [oracle.NO_LEX_RERANK, oracle.SUCC_ON_STRICT, oracle.NO_SEMANTIC,
                                   oracle.NO_BRANCH, oracle.NO_SUCC,
                                   oracle.NO_LEX_RERANK | oracle.NO_BRANCH | oracle.NO_SEMANTIC])
def test_ablation_flags(flags):
    w = synth.make_workload(2, B=12, L=2000, d=128, nohit=0.5, seed=11)
    P = P_of(w, flags=flags)
    check_all(w, run_step(w, P), P)


@pytest.mark.parametrize("succ_len", [2, 5])
def test_longer_successors(succ_len):
    w = synth.make_workload(2, B=8, L=1200, d=64, nohit=0.75, seed=12)
    P = P_of(w, succ_len=succ_len, flags=oracle.SUCC_ON_STRICT)
    check_all(w, run_step(w, P), P)


@pytest.mark.parametrize("flags", [0, oracle.SUCC_ON_STRICT])
def test_maximum_tree(flags):
    """The largest tree the boundary takes: 1 + D + W(1 + succ_len) = 1024
    nodes (D = 255, W = 64, succ_len = 11, k = 32, n_max = 8), 64 branches from
    a 64-wide next-token table, so every branch scans for successors and
    2048 successor rows per sequence are scored."""
    V = 4000
    w = synth.make_workload(2, B=4, L=2000, d=64, V=V, nohit=0.5, seed=91)
    tk = synth.make_next_topk(w.tokens, w.lengths, V, 64, seed=91)
    P = P_of(w, n_max=8, k=32, W=64, D=255, succ_len=11, flags=flags, tau=NEG_INF)
    g = run_step(w, P, next_topk=tk)
    assert g["draft_tokens"].shape[1] == 1024
    assert int(g["n_nodes"].max()) > 300
    check_all(w, g, P, next_topk=tk)


def test_maximum_batch():
    """B = 65535, the largest batch (every kernel's grid y at its limit), of
    short ragged histories; the oracle checks the first and last sequences
    and a seeded sample, the statistics cover every sequence."""
    B = 65535
    rng = np.random.default_rng(65535)
    lengths = rng.integers(1, 13, size=B).astype(np.int32)
    w = synth.make_workload(4, B=B, L=12, d=8, V=50, nohit=0.3, seed=5, lengths=lengths)
    P = P_of(w, tau=NEG_INF)
    g = run_step(w, P)
    sample = sorted({0, 1, B - 2, B - 1, *rng.choice(B, 1500, replace=False).tolist()})
    check_all(w, g, P, seqs=sample)


def test_next_token_table():
    w = synth.make_workload(2, B=6, L=400, d=64, nohit=0.5, seed=13)
    tk = synth.make_next_topk(w.tokens, w.lengths, 32000, 6)
    P = P_of(w)
    check_all(w, run_step(w, P, next_topk=tk), P, next_topk=tk)


def test_standalone_entry_points():
    """lexical -> semantic (selected sequences) -> tree, as three calls."""
    w = synth.make_workload(2, B=10, L=900, d=128, nohit=0.5, seed=14)
    P = P_of(w)
    tok, ln, reps, q = to_dev(w)
    p = params(P)
    out = native.Outputs.allocate(w.B, p)
    ws = native.allocate_workspace(w.B, w.ld, w.d, p)
    native.lexical_match(tok, ln, w.n_max, w.k, out.hit_kind, out.match_n, out.cand, out.n_cand, ws)
    torch.cuda.synchronize()
    hk = out.hit_kind.cpu().numpy()
    for b in range(w.B):
        n, c = oracle.lexical(w.tokens[b], w.n_max, w.k)
        assert hk[b] == (1 if n else 0)
        assert out.cand[b, : out.n_cand[b]].tolist() == c
    active = (out.hit_kind != 1).to(torch.uint8)
    native.semantic_topk(reps, q, ln, w.k, w.tau, out.cand, out.score, out.n_cand, ws,
                         active=active)
    torch.cuda.synchronize()
    nc = out.n_cand.cpu().numpy()
    out.hit_kind.copy_(torch.where(out.hit_kind == 1, out.hit_kind,
                                   torch.where(out.n_cand > 0, 2, 0).to(torch.int32)))
    out.status.zero_()
    out.stats.zero_()
    native.build_draft_tree(tok, ln, reps, q, out.hit_kind, out.cand, out.score, out.n_cand, p,
                            out, ws)
    torch.cuda.synchronize()
    g = out.to_host()
    g["match_n"] = np.array([oracle.lexical(w.tokens[b], w.n_max, w.k)[0] for b in range(w.B)])
    assert (nc[hk == 1] >= 1).all()
    check_all(w, g, P)
    # the fallback alone over every sequence, pure top-k
    cand = torch.empty((w.B, w.k), dtype=torch.int32, device="cuda")
    score = torch.empty((w.B, w.k), dtype=torch.float32, device="cuda")
    n_c = torch.empty(w.B, dtype=torch.int32, device="cuda")
    native.semantic_topk(reps, q, ln, w.k, NEG_INF, cand, score, n_c, ws)
    torch.cuda.synchronize()
    rep = parity.Report()
    for b in range(w.B):
        L = int(w.lengths[b])
        s_all = oracle.scores_all(w.reps[b], w.query[b], L)
        eps = parity.eps_rows(w.reps[b][: L - 1], w.query[b], w.d)
        parity.check_semantic_list(cand[b].cpu().numpy(), score[b].cpu().numpy(), int(n_c[b]),
                                   s_all, eps, w.k, NEG_INF, rep)


def test_repeated_calls_reuse_workspace():
    w = synth.make_workload(4, B=16, L=700, d=64, seed=15)
    P = P_of(w)
    tok, ln, reps, q = to_dev(w)
    eng = native.Engine(w.B, w.ld, w.d, params(P))
    eng.ws.fill_(0xA5)                      # garbage workspace: every call must reset it
    first = None
    for _ in range(3):
        eng.run(tok, ln, reps, q)
        torch.cuda.synchronize()
        g = eng.out.to_host()
        if first is None:
            first = g
        for key in first:
            assert np.array_equal(first[key], g[key], equal_nan=True), key
    check_all(w, first, P)


# ------------------------------------------------ randomised configurations
@pytest.mark.parametrize("case", range(64))
def test_random_configurations(case):
    """Random parameter combinations (n_max, k, W, D, succ_len, tau, ablation
    flags, ragged lengths, d, the next-token table, the embedding table)
    against the oracle, so rarely combined paths (the fused tree stage with
    a table and flags, several slices with few rows, ...) meet it too."""
    rng = np.random.default_rng(5000 + case)
    cfg = int(rng.integers(1, 6))
    B = int(rng.integers(1, 24))
    L = int(rng.choice([2, 7, 300, 1500, 5000, 9000]))
    d = int(rng.choice([8, 64, 136, 512, 1024]))
    V = int(rng.choice([300, 4000, 20000]))
    lengths = [int(x) for x in rng.integers(1, L + 1, size=B)]
    lengths[0] = L
    w = synth.make_workload(cfg, B=B, L=L, d=d, V=V, nohit=float(rng.choice([0.0, 0.5, 1.0])),
                            seed=case, lengths=lengths)
    flags = 0
    for f in (oracle.NO_LEX_RERANK, oracle.SUCC_ON_STRICT, oracle.NO_SEMANTIC, oracle.NO_BRANCH,
              oracle.NO_SUCC):
        if rng.random() < 0.2:
            flags |= f
    P = P_of(w, tau=float(rng.choice([NEG_INF, 0.0, 0.1, 0.5])), flags=flags,
             n_max=int(rng.integers(1, 9)), k=int(rng.integers(1, 33)),
             W=int(rng.integers(0, 9)), D=int(rng.integers(1, 41)),
             succ_len=int(rng.integers(1, 5)))
    tk = synth.make_next_topk(w.tokens, w.lengths, V, int(rng.integers(1, 9)),
                              seed=case) if rng.random() < 0.3 else None
    E = synth.make_embeddings(w, V, int(rng.choice([8, 64, 200])), case) \
        if rng.random() < 0.4 else None
    check_all(w, run_step(w, P, next_topk=tk, emb=E), P, next_topk=tk, emb=E)


# ----------------------------------------------------- full-size workloads
@pytest.mark.parametrize("cfg", [1, 2, 3, 4, 5])
def test_full_size_config(cfg):
    """The five workload shapes at full size, launched as the benchmark does;
    every sequence is checked against the oracle element by element (per-row
    error bounds), and none may need the near-tie allowance."""
    w = synth.make_workload(cfg, device="cuda")
    P = P_of(w)
    eng = native.Engine(w.B, w.ld, w.d, params(P))
    eng.run(w.tokens, w.lengths, w.reps, w.query)
    torch.cuda.synchronize()
    assert native.read_device_status(eng.ws) == 0
    g = eng.out.to_host()
    rep = compare_device_workload(w, g, P)
    print(f"config {cfg}: {rep}")
    assert rep.tie_resolved == 0, rep
    hk = g["hit_kind"]
    assert g["stats"].tolist()[:3] == [int((hk == 1).sum()), int((hk == 2).sum()),
                                       int((hk == 0).sum())]
    # planted near-duplicates are found for every forced miss
    for b in [int(x) for x in w.forced]:
        assert g["hit_kind"][b] == 2
        got = set(g["cand"][b, : g["n_cand"][b]].tolist())
        assert set(w.planted[b][: w.k]) <= got or len(got) == w.k


TUNINGS = {64: ["1,4,2", "2,8,3", "3,16,4"], 4096: ["1,2,5", "2,4,2", "3,8,2"],
           5120: ["1,2,3", "2,4,2"], 8192: ["1,1,8", "2,2,2", "1,4,3"],
           12288: ["1,1,2", "2,2,2"], 16384: ["1,1,4", "2,2,2"]}


@pytest.mark.parametrize("d", sorted(TUNINGS))
def test_semantic_launch_shapes(d, monkeypatch):
    """Every rows-per-stage variant and CTAs-per-SM choice of the semantic
    kernel gives a valid ranking (the shape only changes the schedule)."""
    L = 200 if d > 4096 else 700
    w = synth.make_workload(5, B=3, L=L, d=d, nohit=1.0, seed=d + 7)
    for tun in TUNINGS[d]:
        monkeypatch.setenv("ADAPLD_SEMANTIC_TUNING", tun)
        for tau in (0.1, NEG_INF):
            P = P_of(w, tau=tau)
            check_all(w, run_step(w, P), P)


def test_long_history_many_chunks():
    """More than 32 lexical chunks and successor slices per sequence (merges
    that need several groups of 32 parts)."""
    w = synth.make_workload(5, B=2, L=300000, d=8, nohit=0.5, seed=41, V=64)
    for tau in (0.1, NEG_INF):
        P = P_of(w, tau=tau)
        check_all(w, run_step(w, P), P)


@pytest.mark.parametrize("xmax", ["1", "2", "3", "8", "16"])
def test_lexical_cluster_shapes(xmax, monkeypatch):
    """Every cluster width of the lexical kernel (CTAs per sequence, hence
    chunks per CTA from 1 to 9) gives the oracle's outcome: histories of
    several 8192-position chunks, rows that start off a 16-byte boundary
    (odd ld), ragged lengths, a small vocabulary (many hits) and n_max = 8."""
    monkeypatch.setenv("ADAPLD_LEXICAL_CLUSTER", xmax)
    w = synth.make_workload(5, B=5, L=70001, d=8, V=64, nohit=0.2, seed=43,
                            lengths=[70001, 8193, 16385, 2, 40000])
    for n_max in (1, 8):
        P = P_of(w, tau=NEG_INF, n_max=n_max)
        check_all(w, run_step(w, P), P)


@pytest.mark.parametrize("B,L,W,k", [(3, 900, 2, 8), (4, 9000, 3, 8), (3, 20000, 4, 32),
                                     (5, 40000, 8, 32), (20, 70000, 1, 4), (3, 100000, 2, 16),
                                     (2, 131073, 64, 32)])
def test_tree_cluster_shapes(B, L, W, k):
    """The single-kernel tree stage over clusters of 1 to 16 CTAs per
    sequence (history slices from 1 to 16, scored rows from a few to 2048,
    several rows per warp), against the oracle, with and without the
    text-rule successors of lexical hits (their rerank runs across the
    cluster before the branch set)."""
    w = synth.make_workload(5, B=B, L=L, d=64, V=300, nohit=0.5, seed=L + W,
                            lengths=[L] + [max(2, L - 977 * i) for i in range(1, B)])
    for flags in (0, oracle.SUCC_ON_STRICT):
        P = P_of(w, tau=NEG_INF, W=W, k=k, flags=flags)
        check_all(w, run_step(w, P), P)


def test_semantic_wait_timeout_is_reported_and_recoverable(monkeypatch):
    """Failure path without a fault: with the test switch the semantic
    kernel's producer issues no copy, so every bounded wait expires; the call
    must report ADAPLD_DEV_TIMEOUT through the workspace status word, and the
    next normal call on the same context must succeed with correct results."""
    w = synth.make_workload(2, B=4, L=3000, d=256, nohit=1.0, seed=51)
    P = P_of(w)
    tok, ln, reps, q = to_dev(w)
    eng = native.Engine(w.B, w.ld, w.d, params(P))
    monkeypatch.setenv("ADAPLD_TEST_SEMANTIC_STALL", "1")
    eng.run(tok, ln, reps, q)
    torch.cuda.synchronize()
    assert native.read_device_status(eng.ws) & native.DEV_TIMEOUT
    monkeypatch.delenv("ADAPLD_TEST_SEMANTIC_STALL")
    g = run_step(w, P)
    check_all(w, g, P)


def test_concurrent_calls_from_threads():
    """Two host threads, each with its own stream, workspace and outputs,
    issue steps concurrently (the library keeps no shared state): each gets
    the single-threaded result."""
    import threading
    V = 4000
    ws_ = [synth.make_workload(2, B=5, L=2000, d=64, V=V, nohit=0.6, seed=94 + i)
           for i in range(2)]
    refs = [run_step(w, P_of(w)) for w in ws_]
    results, errors = [None, None], []

    def worker(i):
        try:
            w = ws_[i]
            s = torch.cuda.Stream()
            with torch.cuda.stream(s):
                tok, ln, reps, q = to_dev(w)
                eng = native.Engine(w.B, w.ld, w.d, params(P_of(w)))
                call = eng.bind(tok, ln, reps, q, stream=s)
                for _ in range(20):
                    call()
                s.synchronize()
                results[i] = eng.out.to_host()
        except Exception as e:  # reported below
            errors.append(e)

    th = [threading.Thread(target=worker, args=(i,)) for i in range(2)]
    for t in th:
        t.start()
    for t in th:
        t.join()
    assert not errors, errors
    for ref, got in zip(refs, results):
        for key in ref:
            assert np.array_equal(ref[key], got[key], equal_nan=True), key


@pytest.mark.parametrize("mode", ["plain", "embeddings"])
def test_bound_step_matches_run(mode):
    """Engine.bind marshals the arguments once; its calls give the step's
    outputs, also after the buffers' contents change in place."""
    V = 4000
    w = synth.make_workload(2, B=6, L=1500, d=64, V=V, nohit=0.5, seed=92)
    E = synth.make_embeddings(w, V, 64, 92) if mode == "embeddings" else None
    P = P_of(w)
    ref = run_step(w, P, emb=E)
    tok, ln, reps, q = to_dev(w)
    Ed = torch.from_numpy(E.view(np.int16)).cuda().view(torch.bfloat16) if E is not None else None
    eng = native.Engine(w.B, w.ld, w.d, params(P))
    call = eng.bind(tok, ln, reps, q, emb=Ed)
    call()
    torch.cuda.synchronize()
    got = eng.out.to_host()
    for key in ref:
        assert np.array_equal(ref[key], got[key], equal_nan=True), key
    # a shorter history in place: the next call sees it
    ln[0] = 700
    w.lengths[0] = 700
    ref2 = run_step(w, P, emb=E)
    call()
    torch.cuda.synchronize()
    got2 = eng.out.to_host()
    for key in ref2:
        assert np.array_equal(ref2[key], got2[key], equal_nan=True), key


@pytest.mark.parametrize("mode", ["plain", "embeddings"])
def test_step_replays_from_a_cuda_graph(mode):
    """A step (and the verification after it) captured once in a CUDA graph
    and replayed gives the eager outputs: the calls enqueue device work only
    (no host synchronisation, no allocation), so a serving loop can capture
    them with its decode step."""
    V = 4000
    w = synth.make_workload(2, B=6, L=1500, d=64, V=V, nohit=0.5, seed=91)
    E = synth.make_embeddings(w, V, 64, 91) if mode == "embeddings" else None
    P = P_of(w)
    ref = run_step(w, P, emb=E)
    tok, ln, reps, q = to_dev(w)
    Ed = torch.from_numpy(E.view(np.int16)).cuda().view(torch.bfloat16) if E is not None else None
    eng = native.Engine(w.B, w.ld, w.d, params(P))
    N = eng.out.draft_tokens.shape[1]
    lg = torch.randn((w.B, N, 512), device="cuda").to(torch.bfloat16)
    n_acc = torch.zeros(w.B, dtype=torch.int32, device="cuda")
    new = torch.zeros((w.B, N), dtype=torch.int32, device="cuda")
    n_new = torch.zeros(w.B, dtype=torch.int32, device="cuda")
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):            # warm-up outside the capture
        eng.run(tok, ln, reps, q, emb=Ed)
        native.accept_greedy(lg, eng.out.draft_tokens, eng.out.parents, eng.out.n_nodes, n_acc,
                             new, n_new, eng.ws)
    torch.cuda.synchronize()
    want_acc = n_acc.clone()
    for t in eng.out.tensors():
        t.zero_()
    n_acc.zero_()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        eng.run(tok, ln, reps, q, emb=Ed)
        native.accept_greedy(lg, eng.out.draft_tokens, eng.out.parents, eng.out.n_nodes, n_acc,
                             new, n_new, eng.ws)
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    assert native.read_device_status(eng.ws) == 0
    got = eng.out.to_host()
    for key in ref:
        assert np.array_equal(ref[key], got[key], equal_nan=True), key
    assert torch.equal(n_acc, want_acc)


def test_step_from_host_matches_device_path():
    """adapld_step_from_host: host inputs in, host outputs out, in one call,
    equal to the device-resident step; twice on the same buffers."""
    w = synth.make_workload(2, B=7, L=900, d=64, nohit=0.5, seed=93)
    P = P_of(w)
    ref = run_step(w, P)
    p = params(P)
    eng = native.Engine(w.B, w.ld, w.d, p)
    tok_h = torch.from_numpy(np.ascontiguousarray(w.tokens)).pin_memory()
    len_h = torch.from_numpy(np.ascontiguousarray(w.lengths)).pin_memory()
    reps_h = torch.from_numpy(np.ascontiguousarray(w.reps).view(np.int16)).view(
        torch.bfloat16).pin_memory()
    q_h = torch.from_numpy(np.ascontiguousarray(w.query).view(np.int16)).view(
        torch.bfloat16).pin_memory()
    dev = (torch.empty(tok_h.shape, dtype=torch.int32, device="cuda"),
           torch.empty(len_h.shape, dtype=torch.int32, device="cuda"),
           torch.empty(reps_h.shape, dtype=torch.bfloat16, device="cuda"),
           torch.empty(q_h.shape, dtype=torch.bfloat16, device="cuda"))
    host_out = native.Outputs.allocate(w.B, p, device="cpu", pin_memory=True)
    call, h2d, d2h = eng.bind_from_host(tok_h, len_h, reps_h, q_h, dev, host_out)
    assert h2d == w.tokens.nbytes + w.lengths.nbytes + w.reps.nbytes + w.query.nbytes
    assert d2h == host_out.nbytes()
    for _ in range(2):
        for t in host_out.tensors():
            t.zero_()
        call()
        torch.cuda.synchronize()
        got = {n: t.numpy() for n, t in zip(
            ["hit_kind", "match_n", "cand", "score", "n_cand", "status", "anchor", "draft_tokens",
             "parents", "positions", "mask", "n_nodes", "stats"], host_out.tensors())}
        for key in ref:
            assert np.array_equal(ref[key], got[key], equal_nan=True), key


def test_step_from_host_rejects_before_copying():
    """adapld_step_from_host checks every argument of the step (workspace
    size, alignment of the device buffers, device outputs) before its first
    copy: a rejected call leaves the device buffers untouched and enqueues
    nothing."""
    w = synth.make_workload(2, B=3, L=300, d=64, nohit=0.5, seed=95)
    p = params(P_of(w))
    eng = native.Engine(w.B, w.ld, w.d, p)
    tok_h = torch.from_numpy(np.ascontiguousarray(w.tokens)).pin_memory()
    len_h = torch.from_numpy(np.ascontiguousarray(w.lengths)).pin_memory()
    reps_h = torch.from_numpy(np.ascontiguousarray(w.reps).view(np.int16)).view(
        torch.bfloat16).pin_memory()
    q_h = torch.from_numpy(np.ascontiguousarray(w.query).view(np.int16)).view(
        torch.bfloat16).pin_memory()
    # device inputs one element longer than needed, so a misaligned view fits
    raw = [torch.full((t.numel() + 8,), 7, dtype=t.dtype, device="cuda")
           for t in (tok_h, len_h, reps_h, q_h)]
    dev = [r[: t.numel()] for r, t in zip(raw, (tok_h, len_h, reps_h, q_h))]
    host_out = native.Outputs.allocate(w.B, p, device="cpu", pin_memory=True)
    so_d, so_h = eng.out.c_struct(), host_out.c_struct()
    lib = native.load()
    stream = torch.cuda.current_stream()
    ws_bytes = eng.ws.numel()

    def call(reps_d=None, ws_bytes=ws_bytes, ws_ptr=None):
        return lib.adapld_step_from_host(
            tok_h.data_ptr(), w.ld, len_h.data_ptr(), reps_h.data_ptr(), w.d, q_h.data_ptr(), w.B,
            ctypes.byref(p), dev[0].data_ptr(), dev[1].data_ptr(),
            reps_d if reps_d is not None else dev[2].data_ptr(), dev[3].data_ptr(),
            ctypes.byref(so_d), ctypes.byref(so_h),
            ws_ptr if ws_ptr is not None else eng.ws.data_ptr(), ws_bytes, stream.cuda_stream)

    torch.cuda.synchronize()
    assert call(ws_bytes=ws_bytes - 256) == native.ERR_WORKSPACE
    assert call(reps_d=raw[2].data_ptr() + 2) == native.ERR_ALIGN
    assert call(ws_ptr=eng.ws.data_ptr() + 4) == native.ERR_ALIGN
    torch.cuda.synchronize()
    for r in raw:                                    # no copy reached the device
        assert (r == 7).all()
    assert call() == 0                               # the same buffers, valid call
    torch.cuda.synchronize()
    assert (dev[0].cpu() == tok_h.flatten()).all()


def test_end_to_end_from_host_matches_device_path():
    """The public end-to-end call (pinned host inputs, copies on side streams,
    outputs copied back) returns what the device-resident call returns."""
    w = synth.make_workload(4, B=12, L=900, d=128, seed=61)
    P = P_of(w)
    g = run_step(w, P)
    eng = native.Engine(w.B, w.ld, w.d, params(P))
    tok_h = torch.from_numpy(w.tokens).pin_memory()
    len_h = torch.from_numpy(w.lengths).pin_memory()
    reps_h = torch.from_numpy(w.reps.view(np.int16)).view(torch.bfloat16).pin_memory()
    q_h = torch.from_numpy(w.query.view(np.int16)).view(torch.bfloat16).pin_memory()
    dev = (torch.empty(tok_h.shape, dtype=tok_h.dtype, device="cuda"),
           torch.empty(len_h.shape, dtype=len_h.dtype, device="cuda"),
           torch.empty(reps_h.shape, dtype=reps_h.dtype, device="cuda"),
           torch.empty(q_h.shape, dtype=q_h.dtype, device="cuda"))
    host_out = [torch.empty(x.shape, dtype=x.dtype).pin_memory() for x in eng.out.tensors()]
    for _ in range(2):
        h2d, d2h = eng.run_from_host(tok_h, len_h, reps_h, q_h, dev, host_out)
        torch.cuda.synchronize()
        names = ["hit_kind", "match_n", "cand", "score", "n_cand", "status", "anchor",
                 "draft_tokens", "parents", "positions", "mask", "n_nodes", "stats"]
        for name, t in zip(names, host_out):
            assert np.array_equal(t.numpy(), g[name], equal_nan=True), name
    assert h2d == w.tokens.nbytes + w.lengths.nbytes + w.reps.nbytes + w.query.nbytes


# --------------------------------------------- token-embedding (two-representation) mode
EMB_CASES = [  # (cfg, B, L, d, de, V, seed)
    (2, 8, 1500, 128, 64, 4096, 0), (5, 4, 3000, 256, 4096, 8192, 1),
    (3, 6, 2000, 640, 136, 3000, 2), (4, 20, 500, 64, 8, 2048, 3),
    (5, 3, 1200, 64, 8192, 2048, 4),
    (5, 3, 20000, 64, 256, 4096, 5),    # several chunks and slices per history
    (2, 16, 900, 64, 512, 3000, 6),     # 9-16 fallback queries: two query tiles
    (3, 12, 1500, 64, 1040, 4000, 7),   # a table width that ends in a partial slice
    # batches above 16 sequences (the per-sequence lists whatever the switch)
    (4, 24, 700, 64, 144, 2048, 9),
    (2, 40, 900, 64, 256, 3000, 8),
    (4, 220, 400, 32, 64, 2500, 11),    # more than 128 fallback sequences
]


@pytest.mark.parametrize("union", ["1", "0"])
@pytest.mark.parametrize("cfg,B,L,d,de,V,seed", EMB_CASES)
def test_embedding_mode(cfg, B, L, d, de, V, seed, union, monkeypatch):
    """Eq. 4 over token embeddings, Eq. 6 rerank of the semantic candidates,
    and the successor backoff of Sec. 3.5, against the oracle; through the
    union pass (batches of up to 16: every table row of the batch read once,
    tensor cores) and through the per-sequence lists (ADAPLD_EMB_UNION=0,
    and every batch above 16)."""
    monkeypatch.setenv("ADAPLD_EMB_UNION", union)
    w = synth.make_workload(cfg, B=B, L=L, d=d, V=V, nohit=0.6, seed=seed)
    E = synth.make_embeddings(w, V, de, seed)
    backoff = 0
    for tau in (0.1, NEG_INF):
        P = P_of(w, tau=tau)
        g = run_step(w, P, emb=E)
        check_all(w, g, P, emb=E)
        o = oracle.step(w.tokens, w.lengths, w.reps, w.query, w.n_max, w.k, w.W, w.D,
                        w.succ_len, tau, 0, emb=E)
        assert (o.hit == g["hit_kind"]).all()
        for b in range(w.B):
            if o.hit[b] == oracle.SEM:
                L_b = int(w.lengths[b])
                backoff += sum(1 for i in range(1, int(o.n_nodes[b]))
                               if o.parents[b, i] == 0 and
                               not (w.tokens[b, : L_b - 1] == o.tokens[b, i]).any())
    print("branches needing the backoff:", backoff)


@pytest.mark.parametrize("flags,table", [
    (oracle.SUCC_ON_STRICT, False), (oracle.SUCC_ON_STRICT, True),
    (oracle.NO_SEMANTIC | oracle.SUCC_ON_STRICT, True), (oracle.NO_LEX_RERANK, False),
    (oracle.NO_SUCC, False)])
def test_embedding_mode_ablations(flags, table):
    """Variants of the two-representation step: successors on lexical hits
    (with the next-token table their branch tokens may never have occurred,
    so their backoff needs the distinct-token lists of lexical-hit
    sequences, which the tree stage builds itself when the fallback is off),
    no rerank, no successors."""
    V = 3000
    w = synth.make_workload(2, B=10, L=1200, d=64, V=V, nohit=0.5, seed=85)
    E = synth.make_embeddings(w, V, 64, 85)
    tk = synth.make_next_topk(w.tokens, w.lengths, V, 5) if table else None
    P = P_of(w, flags=flags)
    check_all(w, run_step(w, P, next_topk=tk, emb=E), P, next_topk=tk, emb=E)


def test_embedding_mode_with_next_token_table():
    w = synth.make_workload(2, B=6, L=700, d=64, V=4096, nohit=0.5, seed=71)
    E = synth.make_embeddings(w, 4096, 64, 71)
    tk = synth.make_next_topk(w.tokens, w.lengths, 4096, 5)
    P = P_of(w)
    check_all(w, run_step(w, P, next_topk=tk, emb=E), P, next_topk=tk, emb=E)


def test_embedding_topk_standalone():
    w = synth.make_workload(3, B=7, L=2500, d=16, V=5000, nohit=1.0, seed=72)
    de = 256
    E = synth.make_embeddings(w, 5000, de, 72)
    tok, ln, _, _ = to_dev(w)
    Ed = torch.from_numpy(E.view(np.int16)).cuda().view(torch.bfloat16)
    p = native.make_params(w.n_max, w.k, w.W, w.D)
    ws = native.allocate_workspace(w.B, w.ld, w.d, p)
    cand = torch.full((w.B, w.k), -7, dtype=torch.int32, device="cuda")
    score = torch.zeros((w.B, w.k), dtype=torch.float32, device="cuda")
    n = torch.full((w.B,), -7, dtype=torch.int32, device="cuda")
    status = torch.zeros(w.B, dtype=torch.int32, device="cuda")
    active = (torch.arange(w.B, device="cuda") != 3).to(torch.uint8)
    for tau in (0.1, NEG_INF):
        native.embedding_topk(tok, ln, Ed, w.k, tau, cand, score, n, ws, active=active,
                              status=status)
        torch.cuda.synchronize()
        assert native.read_device_status(ws) == 0
        rep = parity.Report()
        for b in range(w.B):
            if b == 3:
                assert int(n[b]) == -7
                continue
            L_b = int(w.lengths[b])
            s_all, eps = parity.emb_scores(w.tokens[b], L_b, E)
            parity.check_semantic_list(cand[b].cpu().numpy(), score[b].cpu().numpy(), int(n[b]),
                                       s_all, eps, w.k, tau, rep, f"seq {b}")
        assert int(status.sum()) == 0


def _emb_topk(w, E, tau, active=None):
    tok, ln, _, _ = to_dev(w)
    Ed = torch.from_numpy(E.view(np.int16)).cuda().view(torch.bfloat16)
    ws = native.allocate_workspace(w.B, w.ld, w.d, params(P_of(w)))
    cand = torch.full((w.B, w.k), -7, dtype=torch.int32, device="cuda")
    score = torch.zeros((w.B, w.k), dtype=torch.float32, device="cuda")
    n = torch.full((w.B,), -7, dtype=torch.int32, device="cuda")
    native.embedding_topk(tok, ln, Ed, w.k, tau, cand, score, n, ws, active=active)
    torch.cuda.synchronize()
    assert native.read_device_status(ws) == 0
    return cand.cpu().numpy(), score.cpu().numpy(), n.cpu().numpy()


def test_embedding_equal_rows_interleave_by_recency():
    """Tokens with bitwise equal table rows score exactly alike, so their
    positions interleave by recency in the Eq. 4 ranking; a frequent token
    whose row equals the anchor's fills the whole list with its most recent
    positions.  The GPU scores each distinct token once and expands the
    tokens back to positions: the lists must equal the oracle's."""
    V, de = 600, 64
    w = synth.make_workload(2, B=3, L=900, d=32, V=V, nohit=1.0, seed=81)
    E = synth.make_embeddings(w, V, de, 81)
    a0 = int(w.tokens[0, w.lengths[0] - 1])
    a1 = int(w.tokens[1, w.lengths[1] - 1])
    for t in (7, 11):
        assert t not in (a0, a1)
    E[7] = E[a0]
    E[11] = E[a0]
    w.tokens[0, [100, 250, 400, 600, 880]] = 7
    w.tokens[0, [150, 300, 620, 890]] = 11
    E[3] = E[a1]                        # token 3 is frequent under the Zipf draw
    assert (w.tokens[1, : w.lengths[1] - 1] == 3).sum() > w.k
    for tau in (0.1, NEG_INF):
        cand, score, n = _emb_topk(w, E, tau)
        for b in range(w.B):
            L_b = int(w.lengths[b])
            oc, _ = oracle.semantic_emb(w.tokens[b], L_b, E, w.k, tau)
            assert cand[b, : n[b]].tolist() == oc, (b, tau)
        want0 = sorted([j for j in range(w.lengths[0] - 1) if w.tokens[0, j] in (7, 11)],
                       reverse=True)[: w.k]
        assert cand[0, : w.k].tolist() == want0
        assert (w.tokens[1, cand[1, : w.k]] == 3).all()
        P = P_of(w, tau=tau)
        check_all(w, run_step(w, P, emb=E), P, emb=E)


def test_embedding_standalone_calls_match_the_step():
    """lexical -> embedding fallback -> tree with the table (the tree call
    builds the distinct-token lists for the backoff itself) gives the step's
    trees."""
    V = 3000
    w = synth.make_workload(3, B=6, L=2500, d=64, V=V, nohit=0.7, seed=82)
    E = synth.make_embeddings(w, V, 64, 82)
    Ed = torch.from_numpy(E.view(np.int16)).cuda().view(torch.bfloat16)
    P = P_of(w)
    p = params(P)
    g_step = run_step(w, P, emb=E)
    tok, ln, reps, q = to_dev(w)
    out = native.Outputs.allocate(w.B, p)
    ws = native.allocate_workspace(w.B, w.ld, w.d, p)
    native.lexical_match(tok, ln, w.n_max, w.k, out.hit_kind, out.match_n, out.cand, out.n_cand, ws)
    active = (out.hit_kind != 1).to(torch.uint8)
    native.embedding_topk(tok, ln, Ed, w.k, w.tau, out.cand, out.score, out.n_cand, ws,
                          active=active)
    out.hit_kind.copy_(torch.where(out.hit_kind == 1, out.hit_kind,
                                   torch.where(out.n_cand > 0, 2, 0).to(torch.int32)))
    out.status.zero_()
    out.stats.zero_()
    native.build_draft_tree(tok, ln, reps, q, out.hit_kind, out.cand, out.score, out.n_cand, p,
                            out, ws, emb=Ed)
    torch.cuda.synchronize()
    assert native.read_device_status(ws) == 0
    g = out.to_host()
    for key in ("hit_kind", "anchor", "draft_tokens", "parents", "positions", "mask", "n_nodes"):
        assert np.array_equal(g[key], g_step[key]), key


@pytest.mark.parametrize("lengths", [[0, 1, 2, 3, 50, 51], [2, 2, 3, 3, 4, 4]])
def test_embedding_mode_edge_lengths(lengths):
    """Empty, one- and two-token histories and a length past ld in
    two-representation mode (the distinct-token lists of such histories are
    empty or a single token)."""
    V = 300
    w = synth.make_workload(4, B=6, L=50, d=16, ld=50, V=V, seed=83, nohit=0.5,
                            lengths=[min(x, 50) for x in lengths])
    w.lengths = np.asarray(lengths, np.int32)   # 51 > ld: invalid on purpose
    E = synth.make_embeddings(w, V, 16, 83)
    for tau in (0.1, NEG_INF):
        P = P_of(w, tau=tau)
        check_all(w, run_step(w, P, emb=E), P, emb=E)


@pytest.mark.parametrize("kind", ["one_token", "all_distinct"])
def test_embedding_mode_extreme_histories(kind):
    """A history of one repeated token (one list entry, every position tied)
    and a history of all-distinct tokens (the list is the whole history)."""
    V = 9000
    w = synth.make_workload(2, B=2, L=5000, d=32, V=V, seed=84, nohit=1.0)
    L = int(w.lengths[0])
    if kind == "one_token":
        w.tokens[0, : L - 1] = 17
        w.tokens[0, L - 1] = 18
    else:
        w.tokens[0, :L] = np.random.default_rng(84).permutation(V)[:L]
    E = synth.make_embeddings(w, V, 32, 84)
    for tau in (0.1, NEG_INF):
        P = P_of(w, tau=tau)
        check_all(w, run_step(w, P, emb=E), P, emb=E)


def test_embedding_mode_vocabulary_beyond_the_union_bitmap():
    """A batch whose table has more rows than the union pass's bitmap covers
    (short histories, a large vocabulary) keeps the per-sequence lists; the
    results match the oracle all the same, as does a batch just inside."""
    for L, V in ((20, 50000), (200, 4000)):
        w = synth.make_workload(2, B=3, L=L, d=32, V=V, nohit=1.0, seed=86)
        E = synth.make_embeddings(w, V, 32, 86)
        for tau in (0.1, NEG_INF):
            P = P_of(w, tau=tau)
            check_all(w, run_step(w, P, emb=E), P, emb=E)


def test_embedding_mode_token_out_of_table():
    """A token id outside the table reads row 0 and is flagged, no fault."""
    w = synth.make_workload(2, B=3, L=400, d=32, V=1000, nohit=1.0, seed=73)
    E = synth.make_embeddings(w, 1000, 32, 73)
    w.tokens[1, 10] = 5000
    w.tokens[2, 399] = -3           # the anchor itself
    P = P_of(w)
    tok, ln, reps, q = to_dev(w)
    eng = native.Engine(w.B, w.ld, w.d, params(P))
    eng.run(tok, ln, reps, q, emb=torch.from_numpy(E.view(np.int16)).cuda().view(torch.bfloat16))
    torch.cuda.synchronize()
    assert native.read_device_status(eng.ws) == 0
    st = eng.out.status.cpu().numpy()
    assert st[1] & native.SEQ_BAD_TOKEN and st[2] & native.SEQ_BAD_TOKEN
    assert not st[0] & native.SEQ_BAD_TOKEN


@pytest.mark.parametrize("cfg", [2, 3, 4, 5])
def test_full_size_embedding(cfg):
    """A full-size workload with a vocabulary x d embedding table (config 5:
    128256 x 8192, 2.1 GB), launched as the benchmark's embedding mode does;
    every sequence against the oracle.  Config 5 (8 sequences) takes the
    union pass, configs 2-4 (32-256 sequences) the per-sequence lists."""
    w = synth.make_workload(cfg, device="cuda")
    V, de = synth.CONFIGS[cfg]["V"], w.d
    Ed = synth.make_embeddings(w, V, de, 0)
    P = P_of(w)
    eng = native.Engine(w.B, w.ld, w.d, params(P))
    eng.run(w.tokens, w.lengths, w.reps, w.query, emb=Ed)
    torch.cuda.synchronize()
    assert native.read_device_status(eng.ws) == 0
    g = eng.out.to_host()
    E = Ed.view(torch.int16).cpu().numpy().view(np.uint16)
    rep = compare_device_workload(w, g, P, emb=E)
    print(f"config {cfg} with embeddings: {rep}")
    assert rep.tie_resolved == 0, rep
    for b in [int(x) for x in w.forced]:
        assert g["hit_kind"][b] == 2


def test_kernel_launch_counter():
    """adapld_kernel_launches() counts the kernels the library enqueues: the
    same step adds the same count each time (its kernels: lexical, semantic,
    tree stage at least), and a call refused by the argument checks adds
    none."""
    w = synth.make_workload(5, B=3, L=20000, d=64, nohit=0.5, seed=91)
    P = P_of(w)
    tok, ln, reps, q = to_dev(w)
    eng = native.Engine(w.B, w.ld, w.d, params(P))
    eng.run(tok, ln, reps, q)
    torch.cuda.synchronize()
    n0 = native.kernel_launches()
    eng.run(tok, ln, reps, q)
    n1 = native.kernel_launches()
    eng.run(tok, ln, reps, q)
    n2 = native.kernel_launches()
    torch.cuda.synchronize()
    assert n1 - n0 == n2 - n1 >= 3
    with pytest.raises(native.AdapldError):
        native.step(tok, ln, reps, q, params(P), eng.out, eng.ws[:64])  # workspace too small
    assert native.kernel_launches() == n2
