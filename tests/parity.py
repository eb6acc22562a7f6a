"""GPU-vs-oracle comparison helpers used by the ``gpu`` tests.

Integer results (retrieval outcome, lexical match length and candidate set,
tree structure, tokens, parents, positions, mask) must match bit-exactly.
Floating-point scores must match within 1e-2 absolute.  Where a cosine decides
an integer (which candidates enter the top-k, their order, the argmax of
Eq. 7 and Eq. 14), the GPU computes in fp32 and the oracle in fp64, so two
candidates whose fp64 scores differ by less than the rigorous fp32 error bound
eps may legitimately swap: the GPU's choice is then accepted if it is valid
under the oracle's scores within eps, and the rest of the step is re-derived
by the oracle from the GPU's own candidate list (conditional parity), which
must then match exactly.

eps for cos(x, y) with bf16 inputs, fp32 products (exact) and fp32
accumulation of d terms in any order, then two square roots, a product and a
division (each correctly rounded): |err| <= gamma_d (A + |c|) + 5u|c| with
u = 2^-24, gamma_d ~ d u and A = sum|x_i y_i| / (|x||y|) <= 1.  The bound
below doubles the unit roundoff for margin.
"""
from __future__ import annotations

import numpy as np

import oracle
from paper_2606_05742_gb300 import synth

SCORE_ATOL = 1e-2          # absolute score tolerance (bf16 inputs, fp32 accumulation)
U2 = 2.0 ** -23


def eps_rows(R: np.ndarray, ref: np.ndarray, d: int, chunk: int = 2048) -> np.ndarray:
    """Per-row error bound of the fp32 cosine of each row of R against ref."""
    rf = synth.bf16_bits_to_f32(ref).astype(np.float64)
    nr = np.linalg.norm(rf)
    out = np.empty(R.shape[0])
    for i in range(0, R.shape[0], chunk):
        x = synth.bf16_bits_to_f32(R[i:i + chunk]).astype(np.float64)
        nx = np.linalg.norm(x, axis=1)
        den = nx * nr
        A = np.where(den > 0, np.abs(x) @ np.abs(rf) / np.where(den > 0, den, 1), 0.0)
        c = np.where(den > 0, x @ rf / np.where(den > 0, den, 1), 0.0)
        out[i:i + chunk] = (d + 8) * U2 * (A + np.abs(c)) + 1e-6
    return out


def eps_uniform(d: int) -> float:
    """The same bound with A <= 1 and |c| <= 1 (no per-row data needed)."""
    return (d + 8) * U2 * 2.0 + 1e-6


class Report:
    def __init__(self):
        self.exact = 0
        self.tie_resolved = 0
        self.max_score_err = 0.0

    def __repr__(self):
        return (f"exact={self.exact} tie_resolved={self.tie_resolved} "
                f"max_score_err={self.max_score_err:.3g}")

    @staticmethod
    def merge(reports) -> "Report":
        out = Report()
        for r in reports:
            out.exact += r.exact
            out.tie_resolved += r.tie_resolved
            out.max_score_err = max(out.max_score_err, r.max_score_err)
        return out


def check_semantic_list(gc, gs, gn, s_all, eps, k, tau, rep: Report, where=""):
    """Validates a GPU semantic top-k list against every fp64 score."""
    C = [int(x) for x in gc[:gn]]
    S = np.asarray(gs[:gn], dtype=np.float64)
    n_rows = len(s_all)
    assert len(set(C)) == len(C), f"{where}: duplicate candidates {C}"
    assert all(0 <= j < n_rows for j in C), f"{where}: candidate out of range {C}"
    assert (np.asarray(gc[gn:]) == -1).all(), f"{where}: cand padding"
    if gn:
        err = np.abs(S - s_all[C]).max()
        rep.max_score_err = max(rep.max_score_err, float(err))
        assert err <= SCORE_ATOL, f"{where}: score error {err}"
    # membership at the threshold
    for j in C:
        assert s_all[j] >= tau - eps[j], f"{where}: row {j} below tau"
    n_lo = min(k, int((s_all >= tau + eps).sum()))
    n_hi = min(k, int((s_all >= tau - eps).sum()))
    assert n_lo <= gn <= n_hi, f"{where}: count {gn} not in [{n_lo}, {n_hi}]"
    # order: no adjacent pair inverted by more than the bound
    for a, b in zip(C, C[1:]):
        assert s_all[b] <= s_all[a] + eps[a] + eps[b], f"{where}: order {a} {b}"
    # completeness: nothing left out clearly beats what is in
    inside = np.zeros(n_rows, bool)
    inside[C] = True
    out_idx = np.flatnonzero(~inside & (s_all >= tau - eps))
    if gn == k and gn:
        last = C[-1]
        bad = out_idx[s_all[out_idx] > s_all[last] + eps[out_idx] + eps[last]]
        assert len(bad) == 0, f"{where}: rows {bad[:5]} beat the last candidate"
    elif len(out_idx):
        bad = out_idx[s_all[out_idx] >= tau + eps[out_idx]]
        assert len(bad) == 0, f"{where}: rows {bad[:5]} above tau missing"


def check_candidate_set(C, s_all, eps, k, tau, where=""):
    """A candidate set (any order) is a valid top-k-above-tau set under the
    fp64 scores within the bound (membership, count, completeness)."""
    n_rows = len(s_all)
    assert len(set(C)) == len(C), f"{where}: duplicate candidates {C}"
    assert all(0 <= j < n_rows for j in C), f"{where}: candidate out of range {C}"
    for j in C:
        assert s_all[j] >= tau - eps[j], f"{where}: row {j} below tau"
    n_lo = min(k, int((s_all >= tau + eps).sum()))
    n_hi = min(k, int((s_all >= tau - eps).sum()))
    assert n_lo <= len(C) <= n_hi, f"{where}: count {len(C)} not in [{n_lo}, {n_hi}]"
    inside = np.zeros(n_rows, bool)
    inside[C] = True
    out_idx = np.flatnonzero(~inside & (s_all >= tau - eps))
    if len(C) == k and C:
        worst = min(C, key=lambda j: (s_all[j], j))
        bad = out_idx[s_all[out_idx] > s_all[worst] + eps[out_idx] + eps[worst]]
        assert len(bad) == 0, f"{where}: rows {bad[:5]} beat the worst candidate"
    elif len(out_idx):
        bad = out_idx[s_all[out_idx] >= tau + eps[out_idx]]
        assert len(bad) == 0, f"{where}: rows {bad[:5]} above tau missing"


def emb_scores(M, length, E):
    """cos(E[M[j]], E[M[len-1]]) for j in [0, len-2] (fp64) and the bounds."""
    rows = np.ascontiguousarray(E[np.asarray(M[: length - 1])])
    ea = E[int(M[length - 1])]
    return oracle.scores_all(rows, ea, length), eps_rows(rows, ea, E.shape[1]) if length > 1 \
        else np.zeros(0)


def _successor_ok(M, length, R, d, js, btok, chain, k, succ_len, emb=None, tau=0.1):
    """The GPU's successor chain for branch token btok is the continuation of
    some candidate whose Eq. 13 score is within the bound of the best (the
    candidates being the lexical occurrences, or the embedding backoff)."""
    if emb is not None:
        ts, ss = oracle.successor_candidates_emb(M, length, R, d, emb, tau, js, btok, 2 * k)
        lex = [t for t in range(length - 2, -1, -1) if M[t] == btok]
        if lex:
            ts, ss = ts[:k], ss[:k]
    else:
        ts, ss = oracle.successor_candidates(M, length, R, d, js, btok, k)
    if not ts:
        return chain == []
    ss = np.asarray(ss)
    e = eps_rows(R[np.asarray(ts)], R[js + 1], d)
    best = int(np.argmax(ss))
    for i, t in enumerate(ts):
        if ss[i] >= ss[best] - e[i] - e[best]:
            exp = [int(x) for x in M[t + 1: min(t + succ_len, length - 1) + 1]]
            if exp == chain:
                return True
    return False


def _chain_nodes(par, n, head):
    """Nodes below ``head`` (each the single child of the previous)."""
    nodes, cur = [], head
    while True:
        kids = [i for i in range(n) if par[i] == cur]
        if not kids:
            return nodes
        cur = kids[0]
        nodes.append(cur)


def compare_sequence(b, M, length, ld, R, q, g, P, rep: Report, topk_table=None, full_eps=True,
                     emb=None):
    """Checks sequence b of a GPU step (host dict g) against the oracle.
    P: dict(n_max, k, W, D, succ_len, tau, flags); topk_table: this
    sequence's [ld][Kn] next-token table or None."""
    k, W, D, sl, tau, flags = P["k"], P["W"], P["D"], P["succ_len"], P["tau"], P["flags"]
    d = q.shape[0]
    where = f"seq {b}"
    N = oracle.tree_nodes(D, W, sl)
    hit = int(g["hit_kind"][b])
    if length < 1 or length > ld:
        assert hit == oracle.NONE and int(g["n_nodes"][b]) == 0, where
        assert int(g["status"][b]) & 1, where
        assert (g["draft_tokens"][b] == -1).all() and not g["mask"][b].any(), where
        return
    assert int(g["status"][b]) == 0, where
    M = np.asarray(M[:length])
    gn = int(g["n_cand"][b])
    gc = g["cand"][b]
    gs = g["score"][b]
    ln, lc = oracle.lexical(M, P["n_max"], k)
    assert int(g["match_n"][b]) == ln, f"{where}: match_n {g['match_n'][b]} != {ln}"
    tied = False
    if ln:
        assert hit == oracle.LEX, where
        C = [int(x) for x in gc[:gn]]
        assert sorted(C, reverse=True) == lc, f"{where}: lexical set {C} != {lc}"
        if flags & oracle.NO_LEX_RERANK:
            assert C == lc, where
            assert np.isnan(gs[:gn]).all(), where
        else:
            oc, os_ = oracle.rerank(R, q, lc)
            s_map = dict(zip(oc, os_))
            e = eps_rows(R[np.asarray(C)], q, d)
            for i, j in enumerate(C):
                err = abs(float(gs[i]) - s_map[j])
                rep.max_score_err = max(rep.max_score_err, err)
                assert err <= SCORE_ATOL, f"{where}: rerank score {err}"
            for i in range(len(C) - 1):
                assert s_map[C[i + 1]] <= s_map[C[i]] + e[i] + e[i + 1], f"{where}: rerank order"
            tied = C != oc
    elif flags & oracle.NO_SEMANTIC:
        assert hit == oracle.NONE and gn == 0, where
    elif emb is not None:
        # Eq. 4 over token embeddings selects the set, Eq. 6 orders it
        s_emb, e_emb = emb_scores(M, length, emb)
        C = [int(x) for x in gc[:gn]]
        assert (np.asarray(gc[gn:]) == -1).all(), f"{where}: cand padding"
        check_candidate_set(C, s_emb, e_emb, k, tau, where)
        assert hit == (oracle.SEM if gn else oracle.NONE), where
        if gn:
            s_map = dict(zip(*oracle.rerank(R, q, C)))
            e = eps_rows(R[np.asarray(C)], q, d)
            for i, j in enumerate(C):
                err = abs(float(gs[i]) - s_map[j])
                rep.max_score_err = max(rep.max_score_err, err)
                assert err <= SCORE_ATOL, f"{where}: rerank score {err}"
            for i in range(len(C) - 1):
                assert s_map[C[i + 1]] <= s_map[C[i]] + e[i] + e[i + 1], f"{where}: rerank order"
        oc, _ = oracle.semantic_emb(M, length, emb, k, tau)
        tied = sorted(C) != sorted(oc) or C != oracle.rerank(R, q, oc)[0]
    else:
        s_all = oracle.scores_all(R, q, length)
        eps = eps_rows(R[: length - 1], q, d) if full_eps else np.full(length - 1, eps_uniform(d))
        check_semantic_list(gc, gs, gn, s_all, eps, k, tau, rep, where)
        assert hit == (oracle.SEM if gn else oracle.NONE), where
        oc, _ = oracle.semantic(R, q, length, k, tau)
        tied = [int(x) for x in gc[:gn]] != oc
    # conditional tree: the oracle's construction from the GPU's ranked list
    cands = [int(x) for x in gc[:gn]]
    topk_row = topk_table[cands[0]] if (topk_table is not None and cands) else None
    T = oracle.tree_from(M, length, R, d, hit, cands, k, W, D, sl, flags, topk_row, emb=emb,
                         tau=tau)
    n = int(g["n_nodes"][b])
    assert int(g["anchor"][b]) == T.anchor, where
    gt, gp, gpos, gm = g["draft_tokens"][b], g["parents"][b], g["positions"][b], g["mask"][b]
    same = (n == T.n_nodes and (gt == T.tokens).all() and (gp == T.parents).all()
            and (gpos == T.positions).all() and (gm == T.mask).all())
    if not same:
        # only successor choices may differ, and only within the bound
        assert n == T.n_nodes and (gp == T.parents).all(), f"{where}: tree structure"
        assert (gpos == T.positions).all() and (gm == T.mask).all(), f"{where}: tree layout"
        heads = [c for c in range(1, n) if gp[c] == 0 and not (hit == oracle.LEX and c == 1)]
        succ_nodes = {c: _chain_nodes(gp, n, c) for c in heads}
        in_chain = {i for v in succ_nodes.values() for i in v}
        for i in range(n):
            if i not in in_chain:
                assert int(gt[i]) == int(T.tokens[i]), f"{where}: node {i}"
        for c, nodes in succ_nodes.items():
            chain = [int(gt[i]) for i in nodes]
            if chain != [int(T.tokens[i]) for i in nodes]:
                assert _successor_ok(M, length, R, d, T.anchor, int(gt[c]), chain, k, sl,
                                     emb, tau), f"{where}: successor below node {c}"
                tied = True
    if tied:
        rep.tie_resolved += 1
    else:
        rep.exact += 1
    assert g["draft_tokens"][b].shape[0] == N


def host_outputs(out) -> dict:
    return out.to_host()
