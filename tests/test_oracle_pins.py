"""Pins of the CPU oracle against things other than itself: hand-built worked
examples, brute force on tiny inputs, textbook/library routines, closed forms,
exact rational arithmetic, structural invariants and the paper's printed
trigger rates.  No GPU is needed."""
import math
from fractions import Fraction

import numpy as np
import pytest

import oracle
from paper_2606_05742_gb300 import synth
from tests.conftest import load_golden

NEG_INF = float("-inf")


# ----------------------------------------------------------------- helpers
def ints(v):
    return [int(x) for x in v]


def rows_to_bf16(rows, d):
    """Small exact rows -> bf16 bit patterns, zero-padded to d."""
    out = np.zeros((len(rows), d), np.float32)
    for i, r in enumerate(rows):
        out[i, : len(r)] = r
    return synth.f32_to_bf16_bits(out)


def lexical_bruteforce(M, n_max, k):
    """Independent formulation: sliding windows over the history without the
    anchor, longest suffix first (Eq. 3 generalised)."""
    M = np.asarray(M)
    L = len(M)
    for n in range(min(n_max, L - 1), 0, -1):
        win = np.lib.stride_tricks.sliding_window_view(M[: L - 1], n)
        hits = np.flatnonzero((win == M[L - n:]).all(axis=1)) + n - 1
        if len(hits):
            return n, sorted(hits.tolist(), reverse=True)[:k]
    return 0, []


def closure_mask(parents):
    """Ancestor-or-self relation as the reflexive-transitive closure of the
    parent relation, by repeated boolean matrix products."""
    n = len(parents)
    A = np.eye(n, dtype=bool)
    P = np.zeros((n, n), bool)
    for i, p in enumerate(parents):
        if p >= 0:
            P[i, p] = True
    R = A.copy()
    for _ in range(n):
        R = R | (R.astype(np.int64) @ P.astype(np.int64) > 0)
    return R


def np_cos(R, q):
    Rf = synth.bf16_bits_to_f32(R).astype(np.float64)
    qf = synth.bf16_bits_to_f32(q).astype(np.float64)
    num = Rf @ qf
    den = np.linalg.norm(Rf, axis=1) * np.linalg.norm(qf)
    out = np.zeros_like(num)
    nz = den > 0
    out[nz] = num[nz] / den[nz]
    return out


# ------------------------------------------------------- worked examples
def test_worked_example_lexical():
    g = load_golden("worked_example_lexical.txt")
    M = np.array(ints(g["tokens"]), np.int32)
    L = len(M)
    n_max, k, W, D, sl, d = (int(g[x][0]) for x in ("n_max", "k", "W", "D", "succ_len", "d"))
    rng = np.random.default_rng(0)
    row = rng.standard_normal(d).astype(np.float32)
    R = synth.f32_to_bf16_bits(np.tile(row, (L, 1)))
    q = R[L - 1].copy()
    res = oracle.step(M[None], [L], R[None], q[None], n_max, k, W, D, sl, 0.1)
    assert res.hit[0] == int(g["hit"][0]) == oracle.LEX
    assert res.match_n[0] == int(g["match_n"][0])
    assert res.cand[0, : res.n_cand[0]].tolist() == ints(g["cand"])
    assert res.anchor[0] == int(g["anchor"][0])
    n = res.n_nodes[0]
    assert res.tokens[0, :n].tolist() == ints(g["tree_tokens"])
    assert res.parents[0, :n].tolist() == ints(g["tree_parents"])
    assert res.positions[0, :n].tolist() == ints(g["tree_positions"])
    for i in range(n):
        assert np.flatnonzero(res.mask[0, i]).tolist() == ints(g[f"mask_row{i}"])
    assert (res.tokens[0, n:] == -1).all() and (res.mask[0, n:] == 0).all()


def test_worked_example_semantic():
    g = load_golden("worked_example_semantic.txt")
    M = np.array(ints(g["tokens"]), np.int32)
    L = len(M)
    n_max, k, W, D, sl, d = (int(g[x][0]) for x in ("n_max", "k", "W", "D", "succ_len", "d"))
    R = rows_to_bf16([[float(x) for x in g[f"row{i}"]] for i in range(L)], d)
    q = rows_to_bf16([[float(x) for x in g["query"]]], d)[0]
    res = oracle.step(M[None], [L], R[None], q[None], n_max, k, W, D, sl, float(g["tau"][0]))
    assert res.hit[0] == int(g["hit"][0]) == oracle.SEM
    assert res.match_n[0] == 0
    assert res.cand[0, : res.n_cand[0]].tolist() == ints(g["cand"])
    np.testing.assert_allclose(res.score[0, : res.n_cand[0]], [float(x) for x in g["score"]],
                               rtol=0, atol=1e-15)
    assert res.anchor[0] == int(g["anchor"][0])
    n = res.n_nodes[0]
    assert res.tokens[0, :n].tolist() == ints(g["tree_tokens"])
    assert res.parents[0, :n].tolist() == ints(g["tree_parents"])
    assert res.positions[0, :n].tolist() == ints(g["tree_positions"])
    for i in range(n):
        assert np.flatnonzero(res.mask[0, i]).tolist() == ints(g[f"mask_row{i}"])
    assert res.stats.tolist() == [0, 1, 0, 2]


# ---------------------------------------------------------------- lexical
@pytest.mark.parametrize("seed", range(40))
def test_lexical_matches_bruteforce(seed):
    rng = np.random.default_rng(seed)
    L = int(rng.integers(1, 24))
    V = int(rng.integers(2, 5))
    M = rng.integers(0, V, size=L).astype(np.int32)
    for n_max in (1, 2, 3, 5, 8):
        for k in (1, 3, 32):
            assert oracle.lexical(M, n_max, k) == lexical_bruteforce(M, n_max, k)


@pytest.mark.parametrize("seed", range(20))
def test_lexical_nmax1_is_eq3(seed):
    """n_max = 1 is exactly Eq. 3: every earlier position holding the anchor."""
    rng = np.random.default_rng(100 + seed)
    M = rng.integers(0, 6, size=int(rng.integers(2, 200))).astype(np.int32)
    hits = np.flatnonzero(M[:-1] == M[-1])[::-1]
    n, c = oracle.lexical(M, 1, 1000)
    assert c == hits.tolist()
    assert n == (1 if len(hits) else 0)


@pytest.mark.parametrize("seed", range(20))
def test_lexical_most_recent_is_str_rfind(seed):
    """The most recent candidate of the longest suffix agrees with the
    library's substring search (str.rfind over a character encoding)."""
    rng = np.random.default_rng(200 + seed)
    M = rng.integers(0, 3, size=int(rng.integers(2, 40))).astype(np.int32)
    s = "".join(chr(97 + t) for t in M)
    L = len(M)
    n_max = 4
    n, c = oracle.lexical(M, n_max, 8)
    exp_n, exp_j = 0, None
    for m in range(min(n_max, L - 1), 0, -1):
        i = s.rfind(s[L - m:], 0, L - 1)
        if i >= 0:
            exp_n, exp_j = m, i + m - 1
            break
    assert n == exp_n
    if exp_j is not None:
        assert c[0] == exp_j


def test_lexical_edge_cases():
    assert oracle.lexical([7], 3, 4) == (0, [])
    assert oracle.lexical([7, 7], 3, 4) == (1, [0])
    assert oracle.lexical([1, 2], 3, 4) == (0, [])
    # a longer match wins over more recent shorter ones
    assert oracle.lexical([1, 2, 3, 9, 3, 2, 3], 3, 4) == (2, [2])
    # k caps the list, most recent kept
    assert oracle.lexical([4, 4, 4, 4, 4], 1, 2) == (1, [3, 2])


def test_forced_no_hit_sequences_miss():
    w = synth.make_workload(2, B=12, L=600, d=8, nohit=0.5)
    assert len(w.forced) == 6
    for b in range(w.B):
        n, c = oracle.lexical(w.tokens[b], w.n_max, w.k)
        if b in w.forced:
            assert n == 0 and c == []


def test_forced_miss_over_a_full_vocabulary():
    """A history that holds every id of a small vocabulary can only miss
    with id V; the embedding table then grows a row for it."""
    V = 300
    w = synth.make_workload(5, B=3, L=9000, d=8, V=V, nohit=1.0, seed=2064)
    for b in range(w.B):
        ln = int(w.lengths[b])
        assert oracle.lexical(w.tokens[b, :ln], w.n_max, w.k)[0] == 0
    assert int(w.tokens.max()) == V
    E = synth.make_embeddings(w, V, 8, 1)
    assert E.shape == (V + 1, 8)


# --------------------------------------------------------------- semantic
def test_cosine_closed_forms():
    rng = np.random.default_rng(1)
    x = synth.f32_to_bf16_bits(rng.standard_normal(64).astype(np.float32))
    neg = x ^ np.uint16(0x8000)
    twice = synth.f32_to_bf16_bits(2 * synth.bf16_bits_to_f32(x))
    zero = np.zeros(64, np.uint16)
    assert abs(oracle.cosine(x, x) - 1) < 1e-15
    assert abs(oracle.cosine(x, neg) + 1) < 1e-15
    assert abs(oracle.cosine(x, twice) - 1) < 1e-15
    assert oracle.cosine(x, zero) == 0.0 and oracle.cosine(zero, zero) == 0.0
    e0 = rows_to_bf16([[1, 0]], 8)[0]
    e1 = rows_to_bf16([[0, 3]], 8)[0]
    assert oracle.cosine(e0, e1) == 0.0


@pytest.mark.parametrize("seed", range(10))
def test_cosine_exact_rational(seed):
    """fp64 cosine agrees with exact rational arithmetic to a few ulps."""
    rng = np.random.default_rng(300 + seed)
    a = rng.integers(-50, 51, size=16).astype(np.float32)
    b = rng.integers(-50, 51, size=16).astype(np.float32)
    xa, xb = synth.f32_to_bf16_bits(a), synth.f32_to_bf16_bits(b)
    fa = [Fraction(float(v)) for v in synth.bf16_bits_to_f32(xa)]
    fb = [Fraction(float(v)) for v in synth.bf16_bits_to_f32(xb)]
    xy = sum(p * r for p, r in zip(fa, fb))
    nn = sum(p * p for p in fa) * sum(r * r for r in fb)
    exact = float(xy) / math.sqrt(float(nn))
    assert abs(oracle.cosine(xa, xb) - exact) <= 4e-16 * max(1.0, abs(exact))


@pytest.mark.parametrize("seed", range(8))
def test_semantic_full_sort(seed):
    """tau = -inf, k = len-1 turns the fallback into a full descending sort:
    compare with numpy's fp64 matrix product and lexsort."""
    rng = np.random.default_rng(400 + seed)
    L, d = int(rng.integers(2, 60)), 8 * int(rng.integers(1, 5))
    R = synth.f32_to_bf16_bits(rng.standard_normal((L, d)).astype(np.float32))
    if seed % 2:  # force exact score ties: duplicate rows
        R[1::3] = R[0]
    q = R[L - 1]
    s = np_cos(R[: L - 1], q)
    j = np.arange(L - 1)
    order = np.lexsort((-j, -s))
    c, sc = oracle.semantic(R, q, L, L - 1, NEG_INF)
    assert c == order.tolist()
    np.testing.assert_allclose(sc, s[order], rtol=0, atol=1e-14)


@pytest.mark.parametrize("tau", [0.1, 0.0, -0.2, 0.5])
def test_semantic_threshold_and_cap(tau):
    rng = np.random.default_rng(5)
    L, d, k = 300, 16, 7
    R = synth.f32_to_bf16_bits(rng.standard_normal((L, d)).astype(np.float32))
    q = R[L - 1]
    s = np_cos(R[: L - 1], q)
    j = np.arange(L - 1)
    keep = np.flatnonzero(s >= tau)
    order = keep[np.lexsort((-j[keep], -s[keep]))][:k]
    c, _ = oracle.semantic(R, q, L, k, tau)
    assert c == order.tolist()


def test_semantic_planted_rows_rank_first():
    w = synth.make_workload(2, B=2, L=700, d=1024, nohit=1.0)
    for b in range(w.B):
        c, s = oracle.semantic(w.reps[b], w.query[b], 700, w.k, 0.1)
        assert sorted(c) == sorted(w.planted[b])
        for v in s:
            assert abs(v - 1 / 1.09) < 0.03
        # noise rows stay far below the threshold (std 1/sqrt(d))
        all_s = oracle.scores_all(w.reps[b], w.query[b], 700)
        noise = np.delete(all_s, w.planted[b])
        assert np.abs(noise).max() < 0.2


def test_semantic_degenerate():
    R = rows_to_bf16([[1, 0]], 8)
    assert oracle.semantic(R, R[0], 1, 4, NEG_INF) == ([], [])
    R = rows_to_bf16([[0, 0], [1, 0]], 8)
    c, s = oracle.semantic(R, R[1], 2, 4, NEG_INF)
    assert c == [0] and s == [0.0]           # zero row scores 0
    assert oracle.semantic(R, R[1], 2, 4, 0.1) == ([], [])


# ------------------------------------------------------------------ rerank
@pytest.mark.parametrize("seed", range(6))
def test_rerank_is_argmax(seed):
    rng = np.random.default_rng(500 + seed)
    L, d = 40, 16
    R = synth.f32_to_bf16_bits(rng.standard_normal((L, d)).astype(np.float32))
    q = synth.f32_to_bf16_bits(rng.standard_normal(d).astype(np.float32))
    cands = sorted(rng.choice(L - 1, size=6, replace=False).tolist(), reverse=True)
    c, s = oracle.rerank(R, q, cands)
    sc = np_cos(R[cands], q)
    order = np.lexsort((-np.array(cands), -sc))
    assert c == [cands[i] for i in order]
    assert c[0] == cands[int(np.argmax(sc))]


# -------------------------------------------------------------------- tree
def _random_case(rng):
    L = int(rng.integers(2, 14))
    V = int(rng.integers(2, 5))
    d = 8
    M = rng.integers(0, V, size=L).astype(np.int32)
    # rows from a small integer set: exact cosines, frequent exact ties
    R = rows_to_bf16(rng.integers(-2, 3, size=(L, 3)).tolist(), d)
    q = R[L - 1]
    return M, L, R, q, d


@pytest.mark.parametrize("seed", range(60))
@pytest.mark.parametrize("flags", [0, oracle.SUCC_ON_STRICT, oracle.NO_LEX_RERANK,
                                   oracle.NO_BRANCH, oracle.NO_SUCC, oracle.NO_SEMANTIC])
def test_tree_invariants(seed, flags):
    rng = np.random.default_rng(600 + seed)
    M, L, R, q, d = _random_case(rng)
    n_max, k, W, D, sl = 3, 4, int(rng.integers(1, 4)), int(rng.integers(1, 6)), int(rng.integers(1, 3))
    tau = NEG_INF if seed % 3 == 0 else 0.1
    res = oracle.step(M[None], [L], R[None], q[None], n_max, k, W, D, sl, tau, flags)
    nmax = oracle.tree_nodes(D, W, sl)
    n = int(res.n_nodes[0])
    hit = int(res.hit[0])
    tok, par, pos = res.tokens[0], res.parents[0], res.positions[0]
    assert 1 <= n <= nmax
    assert tok[0] == M[L - 1] and par[0] == -1 and pos[0] == L - 1
    assert all(0 <= par[i] < i for i in range(1, n))
    mask = res.mask[0, :n, :n].astype(bool)
    assert (mask == closure_mask(par[:n].tolist())).all()
    depth = mask.sum(axis=1) - 1
    assert (pos[:n] == L - 1 + depth).all()
    assert (tok[n:] == -1).all() and (par[n:] == -1).all() and (pos[n:] == -1).all()
    assert not res.mask[0, n:].any() and not res.mask[0, :, n:].any()
    # retrieval outcome vs Eq. 3 / Eq. 5
    ln, lc = lexical_bruteforce(M, n_max, k)
    cands = res.cand[0, : res.n_cand[0]].tolist()
    if ln:
        assert hit == oracle.LEX and sorted(cands, reverse=True) == lc
    elif flags & oracle.NO_SEMANTIC:
        assert hit == oracle.NONE
    else:
        exp = [j for j in range(L - 1) if oracle.cosine(R[j], q) >= tau]
        assert hit == (oracle.SEM if exp else oracle.NONE)
    if hit == oracle.NONE:
        assert n == 1 and res.anchor[0] == -1
        return
    js = cands[0]
    assert res.anchor[0] == js
    children = [i for i in range(1, n) if par[i] == 0]
    main = []
    if hit == oracle.LEX:
        l = min(D, L - 1 - js)
        main = M[js + 1: js + 1 + l].tolist()
        chain = [1 + i for i in range(l)]
        assert tok[chain].tolist() == main
        assert [par[c] for c in chain] == [0] + chain[:-1]
    # branch rule (Eq. 10-11) with the memory-read surrogate
    exp_br = []
    if not flags & oracle.NO_BRANCH:
        exp_br = list(dict.fromkeys(int(M[c + 1]) for c in cands))[:W]
        if hit == oracle.LEX:
            exp_br = [t for t in exp_br if t != main[0]]
    br_nodes = [c for c in children if not (hit == oracle.LEX and c == 1)]
    assert [int(tok[c]) for c in br_nodes] == exp_br
    # successors (Eq. 13-15), Algorithm 1 by default
    want = (not flags & (oracle.NO_SUCC | oracle.NO_BRANCH)) and (
        hit == oracle.SEM or bool(flags & oracle.SUCC_ON_STRICT))
    Rf = synth.bf16_bits_to_f32(R).astype(np.float64)
    for c in br_nodes:
        kids = [i for i in range(n) if par[i] == c]
        b = int(tok[c])
        occ = [t for t in range(L - 2, -1, -1) if M[t] == b][:k]
        if not want or not occ:
            assert kids == []
            continue
        ref = Rf[js + 1]
        sc = [float(Rf[t] @ ref / (np.linalg.norm(Rf[t]) * np.linalg.norm(ref)))
              if np.linalg.norm(Rf[t]) * np.linalg.norm(ref) > 0 else 0.0 for t in occ]
        best = max(range(len(occ)), key=lambda i: (sc[i], occ[i]))
        tb = occ[best]
        exp_s = M[tb + 1: min(tb + sl, L - 1) + 1].tolist()
        got, cur = [], c
        while True:
            kids = [i for i in range(n) if par[i] == cur]
            if not kids:
                break
            assert len(kids) == 1
            cur = kids[0]
            got.append(int(tok[cur]))
        assert got == exp_s


def test_pld_special_case():
    """With the rerank and branches off, the draft is the span after the most
    recent occurrence of the longest suffix: prompt-lookup decoding, which
    the library's substring search reproduces."""
    rng = np.random.default_rng(9)
    for _ in range(30):
        L = int(rng.integers(3, 50))
        M = rng.integers(0, 3, size=L).astype(np.int32)
        d = 8
        R = synth.f32_to_bf16_bits(rng.standard_normal((L, d)).astype(np.float32))
        D = 5
        res = oracle.step(M[None], [L], R[None], R[L - 1][None], 3, 4, 2, D, 1, 0.1,
                          oracle.NO_LEX_RERANK | oracle.NO_BRANCH | oracle.NO_SEMANTIC)
        s = "".join(chr(97 + t) for t in M)
        exp = [int(M[-1])]
        for m in range(min(3, L - 1), 0, -1):
            i = s.rfind(s[L - m:], 0, L - 1)
            if i >= 0:
                j = i + m - 1
                exp += M[j + 1: j + 1 + min(D, L - 1 - j)].tolist()
                break
        n = res.n_nodes[0]
        assert res.tokens[0, :n].tolist() == exp


def test_next_topk_branches():
    """Paper-faithful branch source: the first W ids of the cached top-K row at
    j*, minus the main path's first token on a strict hit (Eq. 10-11)."""
    M = np.array([5, 7, 9, 5, 7, 3, 5, 7], np.int32)
    L, d = 8, 8
    R = synth.f32_to_bf16_bits(np.ones((L, d), np.float32))
    tk = np.full((1, L, 4), -1, np.int32)
    tk[0, 4] = [3, 11, 12, 13]    # main[0] = 3 is in the top-W
    res = oracle.step(M[None], [L], R[None], R[L - 1][None], 2, 8, 3, 8, 1, 0.1, 0, tk)
    n = res.n_nodes[0]
    assert res.tokens[0, :n].tolist() == [7, 3, 5, 7, 11, 12]
    tk[0, 4] = [20, 21, 22, 3]    # main[0] outside the top-W: W branches remain
    res = oracle.step(M[None], [L], R[None], R[L - 1][None], 2, 8, 3, 8, 1, 0.1, 0, tk)
    n = res.n_nodes[0]
    assert res.tokens[0, :n].tolist() == [7, 3, 5, 7, 20, 21, 22]


def test_invalid_and_short_lengths():
    M = np.array([[3, 4, 3, 4]], np.int32)
    R = np.zeros((1, 4, 8), np.uint16)
    q = np.zeros((1, 8), np.uint16)
    for ln, exp_nodes in ((0, 0), (5, 0), (1, 1)):
        res = oracle.step(M, [ln], R, q, 3, 4, 2, 4, 1, 0.1)
        assert res.n_nodes[0] == exp_nodes and res.hit[0] == oracle.NONE
        assert res.anchor[0] == -1


def test_trigger_rates_pin_algorithm1():
    """Table 9's trigger frequencies (avg / triggered latency) equal Table
    10's retrieval outcome rates: successor drafting runs on semantic hits
    only (Algorithm 1), not on every branch as the prose could suggest."""
    g = load_golden("table9_table10_trigger_rates.txt")
    lex, sem, none, rec = (float(x) / 100 for x in g["hit_rates"])
    rate = {k: float(g[k][1]) / float(g[k][0]) for k in
            ("semantic_fallback", "rerank", "branch", "successor")}
    assert abs(rate["successor"] - sem) < 0.01
    assert abs(rate["successor"] - (lex + sem)) > 0.5
    assert abs(rate["semantic_fallback"] - (sem + none)) < 0.01
    assert abs(rate["rerank"] - (lex + sem)) < 0.01
    assert abs(rate["branch"] - (lex + sem)) < 0.02
    assert abs(sem / (sem + none) - rec) < 1e-3          # Eq. 18, R_rec
    # and the oracle follows that rule by default
    w = synth.make_workload(2, B=10, L=400, d=16, nohit=0.5)
    res = oracle.step(w.tokens, w.lengths, w.reps, w.query, w.n_max, w.k, w.W, w.D, 1, 0.1)
    for b in range(w.B):
        if res.hit[b] != oracle.SEM:
            assert _extended_branches(res, b) == 0
    assert res.stats[1] > 0 and res.stats[3] > 0
    assert res.stats[3] == sum(_extended_branches(res, b) for b in range(w.B))
    res2 = oracle.step(w.tokens, w.lengths, w.reps, w.query, w.n_max, w.k, w.W, w.D, 1, 0.1,
                       oracle.SUCC_ON_STRICT)
    assert res2.stats[3] > res.stats[3]


def _extended_branches(res, b):
    """Branch nodes (children of the root other than the main chain's head)
    that carry a successor child."""
    n = int(res.n_nodes[b])
    par = res.parents[b, :n]
    heads = [i for i in range(1, n) if par[i] == 0]
    if res.hit[b] == oracle.LEX:
        heads = [i for i in heads if i != 1]
    return sum(1 for h in heads if (par == h).any())


def test_semantic_threshold_is_inclusive():
    """Eq. 4 keeps cos >= tau: rows whose exact cosine equals tau stay in."""
    R = rows_to_bf16([[0, 1], [3, 4], [1, 1], [1, 0]], 8)   # cos 0, 0.6, 0.707 vs (1,0)
    q = R[3]
    c, s = oracle.semantic(R, q, 4, 8, 0.6)
    assert c == [2, 1] and s[1] == 0.6
    c, s = oracle.semantic(R, q, 4, 8, 0.0)
    assert c == [2, 1, 0] and s[2] == 0.0


# ------------------------------------------------- token-embedding fallback
def test_worked_example_embedding():
    g = load_golden("worked_example_embedding.txt")
    M = np.array(ints(g["tokens"]), np.int32)
    L = len(M)
    n_max, k, W, D, sl, d = (int(g[x][0]) for x in ("n_max", "k", "W", "D", "succ_len", "d"))
    E = rows_to_bf16([[float(x) for x in g[f"emb{v}"]] for v in range(6)], d)
    R = rows_to_bf16([[float(x) for x in g[f"row{i}"]] for i in range(L)], d)
    q = rows_to_bf16([[float(x) for x in g["query"]]], d)[0]
    res = oracle.step(M[None], [L], R[None], q[None], n_max, k, W, D, sl, float(g["tau"][0]),
                      emb=E)
    assert res.hit[0] == int(g["hit"][0]) == oracle.SEM
    assert res.cand[0, : res.n_cand[0]].tolist() == ints(g["cand"])
    np.testing.assert_allclose(res.score[0, : res.n_cand[0]], [float(x) for x in g["score"]],
                               atol=1e-15)
    assert res.anchor[0] == int(g["anchor"][0])
    n = res.n_nodes[0]
    assert res.tokens[0, :n].tolist() == ints(g["tree_tokens"])
    assert res.parents[0, :n].tolist() == ints(g["tree_parents"])
    assert res.positions[0, :n].tolist() == ints(g["tree_positions"])
    single = oracle.step(M[None], [L], R[None], q[None], n_max, k, W, D, sl, 0.1)
    assert single.cand[0, :2].tolist() == [2, 3]


@pytest.mark.parametrize("seed", range(6))
def test_embedding_fallback_reduces_to_single_cache(seed):
    """All-distinct tokens with E = R (token v's embedding is row v) and the
    query equal to the anchor's row make Eq. 4 over embeddings coincide with
    the single-cache fallback, which is pinned above."""
    rng = np.random.default_rng(700 + seed)
    L, d, k = int(rng.integers(3, 80)), 16, 5
    R = synth.f32_to_bf16_bits(rng.standard_normal((L, d)).astype(np.float32))
    M = np.arange(L, dtype=np.int32)
    q = R[L - 1]
    for tau in (0.1, NEG_INF):
        assert oracle.semantic_emb(M, L, R, k, tau) == oracle.semantic(R, q, L, k, tau)
    # the steps agree up to successor drafting, which only the embedding mode
    # can back off for a branch token with no earlier occurrence
    a = oracle.step(M[None], [L], R[None], q[None], 3, k, 2, 4, 1, NEG_INF, oracle.NO_SUCC,
                    emb=R)
    b = oracle.step(M[None], [L], R[None], q[None], 3, k, 2, 4, 1, NEG_INF, oracle.NO_SUCC)
    for name in ("hit", "cand", "score", "anchor", "tokens", "parents", "mask", "n_nodes"):
        assert np.array_equal(getattr(a, name), getattr(b, name)), name


@pytest.mark.parametrize("seed", range(20))
def test_embedding_fallback_bruteforce(seed):
    rng = np.random.default_rng(800 + seed)
    V, L, de, k = int(rng.integers(3, 9)), int(rng.integers(2, 40)), 8, 4
    M = rng.integers(0, V, size=L).astype(np.int32)
    E = rows_to_bf16(rng.integers(-2, 3, size=(V, 3)).tolist(), de)
    Ef = synth.bf16_bits_to_f32(E).astype(np.float64)
    ea = Ef[M[-1]]
    s = np.array([Ef[v] @ ea / (np.linalg.norm(Ef[v]) * np.linalg.norm(ea))
                  if np.linalg.norm(Ef[v]) * np.linalg.norm(ea) > 0 else 0.0 for v in M[:-1]])
    j = np.arange(L - 1)
    for tau in (0.1, NEG_INF):
        keep = np.flatnonzero(s >= tau)
        order = keep[np.lexsort((-j[keep], -s[keep]))][:k]
        c, sc = oracle.semantic_emb(M, L, E, k, tau)
        assert c == order.tolist()
        np.testing.assert_allclose(sc, s[order], atol=1e-12)


@pytest.mark.parametrize("seed", range(20))
def test_successor_backoff_bruteforce(seed):
    """A branch token that never occurs earlier backs off to the embedding
    fallback with the branch token as the query anchor (Sec. 3.5)."""
    rng = np.random.default_rng(900 + seed)
    V, L, d, k = 8, int(rng.integers(4, 30)), 8, 3
    M = rng.integers(0, V - 2, size=L).astype(np.int32)   # tokens V-2, V-1 never occur
    E = rows_to_bf16(rng.integers(-2, 3, size=(V, 3)).tolist(), d)
    R = rows_to_bf16(rng.integers(-2, 3, size=(L, 3)).tolist(), d)
    js = int(rng.integers(0, L - 1))
    Ef = synth.bf16_bits_to_f32(E).astype(np.float64)
    Rf = synth.bf16_bits_to_f32(R).astype(np.float64)

    def cos(x, y):
        n = np.linalg.norm(x) * np.linalg.norm(y)
        return float(x @ y / n) if n > 0 else 0.0

    for b in (V - 1, int(M[0])):
        occ = [t for t in range(L - 2, -1, -1) if M[t] == b][:k]
        if not occ:
            es = [(cos(Ef[M[t]], Ef[b]), t) for t in range(L - 1)]
            es = [x for x in es if x[0] >= 0.1]
            occ = [t for _, t in sorted(es, key=lambda x: (-x[0], -x[1]))[:k]]
        exp_s = [cos(Rf[t], Rf[js + 1]) for t in occ]
        t, sc = oracle.successor_candidates_emb(M, L, R, d, E, 0.1, js, b, k)
        assert t == occ
        np.testing.assert_allclose(sc, exp_s, atol=1e-12)
    # without a table a token that never occurs has no successor candidates
    assert oracle.successor_candidates(M, L, R, d, js, V - 1, k) == ([], [])


@pytest.mark.parametrize("seed", range(20))
def test_anchor_backoff_is_the_fallback(seed):
    """A semantic hit's anchor never occurred earlier (else the lexical match
    holds at n = 1); when it is a branch token its backoff of Sec. 3.5 -- Eq. 4
    with the anchor as the query -- returns the fallback's own candidate list,
    which the GPU step takes over instead of scoring the rows again."""
    rng = np.random.default_rng(950 + seed)
    V, L, d, k = 9, int(rng.integers(3, 40)), 8, int(rng.integers(1, 6))
    M = rng.integers(0, V - 1, size=L).astype(np.int32)
    M[-1] = V - 1                                   # the anchor: no earlier occurrence
    E = rows_to_bf16(rng.integers(-2, 3, size=(V, 3)).tolist(), d)
    R = rows_to_bf16(rng.integers(-2, 3, size=(L, 3)).tolist(), d)
    js = int(rng.integers(0, L - 1))
    assert oracle.lexical(M, 3, k)[0] == 0          # no lexical hit
    for tau in (0.1, NEG_INF):
        c, _ = oracle.semantic_emb(M, L, E, k, tau)
        t, _ = oracle.successor_candidates_emb(M, L, R, d, E, tau, js, int(M[-1]), k)
        assert t == c


# ---------------------------------------------------- greedy verification
def _logits_rows(g, case, N, V):
    L = np.zeros((N, V), np.float32)
    for i in range(N):
        key = f"{case}_node{i}"
        if key in g:
            vals = g[key]
            for t, v in zip(vals[0::2], vals[1::2]):
                L[i, int(t)] = float(v)
    return synth.f32_to_bf16_bits(L)


@pytest.mark.parametrize("case", ["A", "B", "C"])
def test_worked_example_verify(case):
    g = load_golden("worked_example_verify.txt")
    tok = np.array(ints(g["tree_tokens"]), np.int32)
    par = np.array(ints(g["tree_parents"]), np.int32)
    V = int(g["vocab"][0])
    lg = _logits_rows(g, case, len(tok), V)
    acc, new, path = oracle.verify_greedy(lg, tok, par, len(tok))
    assert acc == int(g[f"{case}_accept"][0])
    assert new == ints(g[f"{case}_new"])
    assert path == ints(g[f"{case}_path"])


def _verify_bruteforce(lg, tok, par, n):
    target = [int(np.argmax(synth.bf16_bits_to_f32(lg[i]))) for i in range(n)]
    ok = [True] + [False] * (n - 1)
    for i in range(1, n):
        ok[i] = ok[par[i]] and tok[i] == target[par[i]]
    deepest = max((i for i in range(n) if ok[i]), key=lambda i: _depth(par, i))
    chain = []
    cur = deepest
    while cur != 0:
        chain.append(cur)
        cur = par[cur]
    chain = chain[::-1]
    return len(chain), [int(tok[c]) for c in chain] + [target[deepest]], [0] + chain


def _depth(par, i):
    d = 0
    while par[i] >= 0:
        i = par[i]
        d += 1
    return d


@pytest.mark.parametrize("seed", range(40))
def test_verify_bruteforce_on_built_trees(seed):
    """Trees built by the oracle itself; logits with small integer values so
    maxima tie often; numpy's argmax takes the first maximum."""
    rng = np.random.default_rng(1000 + seed)
    M, L, R, q, d = _random_case(rng)
    flags = [0, oracle.SUCC_ON_STRICT][seed % 2]
    res = oracle.step(M[None], [L], R[None], q[None], 3, 4, 3, 5, 2, NEG_INF, flags)
    n = int(res.n_nodes[0])
    tok, par = res.tokens[0, :n], res.parents[0, :n]
    V = 6
    # bias each node's logits towards a child's token half of the time
    lg = rng.integers(-2, 3, size=(n, V)).astype(np.float32)
    for i in range(n):
        kids = [c for c in range(n) if par[c] == i]
        if kids and rng.random() < 0.6:
            t = int(tok[kids[int(rng.integers(len(kids)))]])
            if t < V:
                lg[i, t] = 5.0
    M2 = np.where(tok >= V, V - 1, tok).astype(np.int32)   # keep tokens inside the vocabulary
    lgb = synth.f32_to_bf16_bits(lg)
    assert oracle.verify_greedy(lgb, M2, par, n) == _verify_bruteforce(lgb, M2, par, n)


def test_verify_chain_is_longest_matching_prefix():
    """A chain tree (prompt-lookup draft): the accepted tokens are the longest
    prefix of the draft agreeing with the target's choices."""
    rng = np.random.default_rng(5)
    for _ in range(30):
        n = int(rng.integers(1, 9))
        tok = rng.integers(0, 4, size=n).astype(np.int32)
        par = np.arange(-1, n - 1, dtype=np.int32)
        target = rng.integers(0, 4, size=n)
        lg = np.full((n, 4), -1.0, np.float32)
        lg[np.arange(n), target] = 1.0
        acc, new, path = oracle.verify_greedy(synth.f32_to_bf16_bits(lg), tok, par, n)
        m = 0
        while m + 1 < n and tok[m + 1] == target[m]:
            m += 1
        assert acc == m and new == tok[1:m + 1].tolist() + [int(target[m])]


def test_accept_appends_tokens_and_rows():
    rng = np.random.default_rng(6)
    B, N, V, d, ld = 3, 5, 12, 8, 10
    tok = np.tile(np.array([7, 3, 5, 7, 9], np.int32), (B, 1))
    par = np.tile(np.array([-1, 0, 1, 2, 0], np.int32), (B, 1))
    n_nodes = np.array([5, 5, 0], np.int32)
    lg = np.zeros((B, N, V), np.float32)
    lg[0, 0, 3] = lg[0, 1, 5] = lg[0, 2, 4] = 1.0      # accept 3, 5; bonus 4
    lg[1, 0, 9] = lg[1, 4, 2] = 1.0                    # accept 9; bonus 2
    lgb = synth.f32_to_bf16_bits(lg)
    tokens = np.arange(B * ld, dtype=np.int32).reshape(B, ld)
    lengths = np.array([5, 9, 4], np.int32)
    node_reps = synth.f32_to_bf16_bits(rng.standard_normal((B, N, d)).astype(np.float32))
    reps = np.zeros((B, ld, d), np.uint16)
    query = np.zeros((B, d), np.uint16)
    t0, r0 = tokens.copy(), reps.copy()
    r = oracle.accept_greedy(lgb, tok, par, n_nodes, tokens, lengths, node_reps, reps, query)
    assert r.n_accept.tolist() == [2, 1, 0] and r.n_new.tolist() == [3, 2, 0]
    assert r.new_tokens[0, :3].tolist() == [3, 5, 4] and r.new_tokens[1, :2].tolist() == [9, 2]
    assert r.full.tolist() == [0, 1, 0]                 # 9 + 2 > 10: no room
    assert lengths.tolist() == [8, 9, 4]
    assert tokens[0, 5:8].tolist() == [3, 5, 4] and (tokens[1] == t0[1]).all()
    assert (reps[0, 5] == node_reps[0, 0]).all() and (reps[0, 6] == node_reps[0, 1]).all()
    assert (reps[0, 7] == node_reps[0, 2]).all() and (query[0] == node_reps[0, 2]).all()
    assert (reps[1] == r0[1]).all() and (reps[2] == r0[2]).all()


def test_accept_exact_fit():
    """An append that fills the capacity exactly (len + n_new == ld) happens."""
    tok = np.array([[7, 3, 5, 7, 9]], np.int32)
    par = np.array([[-1, 0, 1, 2, 0]], np.int32)
    lg = np.zeros((1, 5, 12), np.float32)
    lg[0, 0, 3] = lg[0, 1, 5] = lg[0, 2, 4] = 1.0      # 3 new tokens
    tokens = np.zeros((1, 10), np.int32)
    lengths = np.array([7], np.int32)
    r = oracle.accept_greedy(synth.f32_to_bf16_bits(lg), tok, par, np.array([5], np.int32),
                             tokens, lengths)
    assert r.full.tolist() == [0] and lengths.tolist() == [10]
    assert tokens[0, 7:].tolist() == [3, 5, 4]
