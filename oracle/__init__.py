"""ctypes binding of the AdaPLD CPU oracle (``adapld_oracle.c``).

Test infrastructure only: the tests, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline leg are the only callers.  The oracle is a plain fp64
restatement of the paper's definitions (Sec. 3.3-3.5, Eq. 3-15, Algorithm 1)
and shares no code with the CUDA library.

Arrays are numpy: tokens int32, representations as uint16 bf16 bit patterns.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "adapld_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")

# Retrieval outcomes (Eq. 5 / Algorithm 1) and ablation switches, restated
# here from the paper independently of the CUDA library's header.
NONE, LEX, SEM = 0, 1, 2
NO_LEX_RERANK = 1
SUCC_ON_STRICT = 2
NO_SEMANTIC = 4
NO_BRANCH = 8
NO_SUCC = 16


def build(force: bool = False) -> str:
    """Compile the oracle with the host C compiler (plain C99, -O2)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(
            ["gcc", "-std=c99", "-O2", "-ffp-contract=off", "-fPIC", "-shared",
             _SRC, "-o", tmp, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


_lib = None


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        P = ctypes.c_void_p
        i32, i64, f64, u32 = ctypes.c_int32, ctypes.c_int64, ctypes.c_double, ctypes.c_uint32
        lib.oracle_cosine.argtypes = [P, P, i32]
        lib.oracle_cosine.restype = f64
        lib.oracle_lexical.argtypes = [P, i32, i32, i32, P, P, P]
        lib.oracle_lexical.restype = ctypes.c_int
        lib.oracle_semantic.argtypes = [P, i32, P, i32, i32, f64, P, P]
        lib.oracle_semantic.restype = i32
        lib.oracle_scores_all.argtypes = [P, i32, P, i32, P]
        lib.oracle_scores_all.restype = None
        lib.oracle_rerank.argtypes = [P, i32, P, P, P, i32]
        lib.oracle_rerank.restype = None
        lib.oracle_successor_candidates.argtypes = [P, i32, P, i32, i32, i32, i32, P, P]
        lib.oracle_successor_candidates.restype = i32
        lib.oracle_tree_from.argtypes = [P, i32, P, i32, i32, P, i32, P, i32, i32, i32, i32,
                                         i32, u32, i32, P, P, P, P, P, P]
        lib.oracle_tree_from.restype = i32
        lib.oracle_step.argtypes = [P, i64, P, P, i32, P, P, i32, i32, i32, i32, i32, i32,
                                    i32, f64, u32, i32, P, P, P, P, P, P, P, P, P, P, P, P]
        lib.oracle_step.restype = None
        lib.oracle_step_emb.argtypes = [P, i64, P, P, i32, P, P, i32, P, i32, i32, i32, i32,
                                        i32, i32, i32, f64, u32, i32, P, P, P, P, P, P, P, P,
                                        P, P, P, P]
        lib.oracle_step_emb.restype = None
        lib.oracle_semantic_emb.argtypes = [P, i32, P, i32, i32, f64, P, P]
        lib.oracle_semantic_emb.restype = i32
        lib.oracle_successor_candidates_emb.argtypes = [P, i32, P, i32, P, i32, f64, i32, i32,
                                                        i32, P, P]
        lib.oracle_successor_candidates_emb.restype = i32
        lib.oracle_tree_from_emb.argtypes = [P, i32, P, i32, P, i32, f64, i32, P, i32, P, i32,
                                             i32, i32, i32, i32, u32, i32, P, P, P, P, P, P]
        lib.oracle_tree_from_emb.restype = i32
        lib.oracle_verify_greedy.argtypes = [P, i32, P, P, i32, P, P, P]
        lib.oracle_verify_greedy.restype = i32
        lib.oracle_accept_greedy.argtypes = [P, i32, P, P, P, i32, i32, P, P, P, P, i64, P, P, P,
                                             i32, P, P]
        lib.oracle_accept_greedy.restype = None
        _lib = lib
    return _lib


def _p(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def tree_nodes(draft_len: int, branch_width: int, succ_len: int) -> int:
    """Node capacity of one draft tree: root + main chain + branch paths."""
    return 1 + draft_len + branch_width * (1 + succ_len)


def cosine(x, y) -> float:
    """cos(x, y) of two bf16 vectors (uint16 bit patterns), in fp64."""
    x = _c(x, np.uint16)
    y = _c(y, np.uint16)
    assert x.shape == y.shape and x.ndim == 1
    return _load().oracle_cosine(_p(x), _p(y), x.shape[0])


def lexical(M, n_max: int, k: int):
    """Eq. 3, longest suffix first: returns (match_n, [candidates desc j])."""
    M = _c(M, np.int32)
    cand = np.full(max(k, 1), -1, np.int32)
    mn = np.zeros(1, np.int32)
    nc = np.zeros(1, np.int32)
    _load().oracle_lexical(_p(M), M.shape[0], n_max, k, _p(mn), _p(cand), _p(nc))
    return int(mn[0]), cand[: int(nc[0])].tolist()


def semantic(R, q, length: int, k: int, tau: float):
    """Eq. 4 capped at k: returns ([positions], [scores]) best first."""
    R = _c(R, np.uint16)
    q = _c(q, np.uint16)
    d = q.shape[0]
    cand = np.full(max(k, 1), -1, np.int32)
    score = np.zeros(max(k, 1), np.float64)
    n = _load().oracle_semantic(_p(R), d, _p(q), length, k, float(tau), _p(cand), _p(score))
    return cand[:n].tolist(), score[:n].tolist()


def semantic_emb(M, length: int, E, k: int, tau: float):
    """Eq. 4 over token embeddings, cos(E[M[j]], E[M[len-1]]), capped at k:
    returns ([positions], [scores]) best first."""
    M = _c(M, np.int32)
    E = _c(E, np.uint16)
    cand = np.full(max(k, 1), -1, np.int32)
    score = np.zeros(max(k, 1), np.float64)
    n = _load().oracle_semantic_emb(_p(M), length, _p(E), E.shape[1], k, float(tau), _p(cand),
                                    _p(score))
    return cand[:n].tolist(), score[:n].tolist()


def successor_candidates_emb(M, length: int, R, d: int, E, tau: float, j_star: int, b: int,
                             k: int):
    """Sec. 3.5 lexical-first backoff for branch token b (embedding fallback
    when b never occurs), each candidate scored by Eq. 13."""
    M = _c(M, np.int32)
    R = _c(R, np.uint16)
    E = _c(E, np.uint16)
    t = np.zeros(max(k, 1), np.int32)
    s = np.zeros(max(k, 1), np.float64)
    n = _load().oracle_successor_candidates_emb(_p(M), length, _p(R), d, _p(E), E.shape[1],
                                                float(tau), j_star, b, k, _p(t), _p(s))
    return t[:n].tolist(), s[:n].tolist()


def scores_all(R, q, length: int) -> np.ndarray:
    """Every Eq. 4 score cos(R[j], q), j in [0, length-2], in fp64."""
    R = _c(R, np.uint16)
    q = _c(q, np.uint16)
    out = np.zeros(max(length - 1, 0), np.float64)
    if length > 1:
        _load().oracle_scores_all(_p(R), q.shape[0], _p(q), length, _p(out))
    return out


def rerank(R, q, cands):
    """Eq. 6-7: returns (candidates re-sorted best first, their scores)."""
    R = _c(R, np.uint16)
    q = _c(q, np.uint16)
    c = _c(cands, np.int32).copy()
    s = np.zeros(max(len(c), 1), np.float64)
    _load().oracle_rerank(_p(R), q.shape[0], _p(q), _p(c), _p(s), len(c))
    return c.tolist(), s[: len(c)].tolist()


def successor_candidates(M, length: int, R, d: int, j_star: int, b: int, k: int):
    """Eq. 13: k most recent t with M[t] = b, t <= len-2, and cos(R[t], R[j*+1])."""
    M = _c(M, np.int32)
    R = _c(R, np.uint16)
    t = np.zeros(max(k, 1), np.int32)
    s = np.zeros(max(k, 1), np.float64)
    n = _load().oracle_successor_candidates(_p(M), length, _p(R), d, j_star, b, k, _p(t), _p(s))
    return t[:n].tolist(), s[:n].tolist()


@dataclass
class Tree:
    anchor: int
    tokens: np.ndarray
    parents: np.ndarray
    positions: np.ndarray
    mask: np.ndarray
    n_nodes: int
    succ_ext: int


def tree_from(M, length: int, R, d: int, hit: int, cands, k: int, W: int, D: int,
              succ_len: int = 1, flags: int = 0, topk_row=None, emb=None,
              tau: float = 0.1) -> Tree:
    """Draft tree (Sec. 3.5, Algorithm 1) from a retrieval outcome and its
    ranked candidate list (cands[0] is the anchor j*); with an embedding
    table `emb`, successor drafting backs off to the embedding fallback."""
    M = _c(M, np.int32)
    R = _c(R, np.uint16)
    c = _c(cands, np.int32) if len(cands) else np.zeros(1, np.int32)
    nmax = tree_nodes(D, W, succ_len)
    tok = np.zeros(nmax, np.int32)
    par = np.zeros(nmax, np.int32)
    pos = np.zeros(nmax, np.int32)
    mask = np.zeros((nmax, nmax), np.uint8)
    anchor = np.zeros(1, np.int32)
    nn = np.zeros(1, np.int32)
    if topk_row is not None:
        tr = _c(topk_row, np.int32)
        trp, kn = _p(tr), tr.shape[0]
    else:
        trp, kn = None, 0
    if emb is not None:
        E = _c(emb, np.uint16)
        Ep, de = _p(E), E.shape[1]
    else:
        Ep, de = None, 0
    ext = _load().oracle_tree_from_emb(_p(M), length, _p(R), d, Ep, de, float(tau), hit, _p(c),
                                       len(cands), trp, kn, k, W, D, succ_len, flags, nmax,
                                       _p(anchor), _p(tok), _p(par), _p(pos), _p(mask), _p(nn))
    return Tree(int(anchor[0]), tok, par, pos, mask, int(nn[0]), int(ext))


@dataclass
class StepResult:
    hit: np.ndarray
    match_n: np.ndarray
    anchor: np.ndarray
    cand: np.ndarray
    score: np.ndarray
    n_cand: np.ndarray
    tokens: np.ndarray
    parents: np.ndarray
    positions: np.ndarray
    mask: np.ndarray
    n_nodes: np.ndarray
    stats: np.ndarray


def step(tokens, lengths, reps, query, n_max: int, k: int, W: int, D: int,
         succ_len: int = 1, tau: float = 0.1, flags: int = 0, next_topk=None,
         emb=None) -> StepResult:
    """One draft-construction step for a batch (layouts as in the library):
    tokens [B][ld] int32, lengths [B], reps [B][ld][d] bf16 bits,
    query [B][d] bf16 bits, next_topk [B][ld][Kn] int32 or None, emb [V][de]
    bf16 bits (token embeddings) or None."""
    tokens = _c(tokens, np.int32)
    lengths = _c(lengths, np.int32)
    reps = _c(reps, np.uint16)
    query = _c(query, np.uint16)
    B, ld = tokens.shape
    d = query.shape[1]
    assert reps.shape == (B, ld, d)
    nmax = tree_nodes(D, W, succ_len)
    hit = np.zeros(B, np.int32)
    mn = np.zeros(B, np.int32)
    anchor = np.zeros(B, np.int32)
    cand = np.zeros((B, k), np.int32)
    score = np.zeros((B, k), np.float64)
    nc = np.zeros(B, np.int32)
    tok = np.zeros((B, nmax), np.int32)
    par = np.zeros((B, nmax), np.int32)
    pos = np.zeros((B, nmax), np.int32)
    mask = np.zeros((B, nmax, nmax), np.uint8)
    nn = np.zeros(B, np.int32)
    stats = np.zeros(4, np.int64)
    if next_topk is not None:
        nt = _c(next_topk, np.int32)
        ntp, kn = _p(nt), nt.shape[2]
    else:
        ntp, kn = None, 0
    if emb is not None:
        E = _c(emb, np.uint16)
        Ep, de = _p(E), E.shape[1]
    else:
        Ep, de = None, 0
    _load().oracle_step_emb(_p(tokens), ld, _p(lengths), _p(reps), d, _p(query), Ep, de, ntp,
                            kn, B, n_max, k, W, D, succ_len, float(tau), flags, nmax,
                            _p(hit), _p(mn), _p(anchor), _p(cand), _p(score), _p(nc), _p(tok),
                            _p(par), _p(pos), _p(mask), _p(nn), _p(stats))
    return StepResult(hit, mn, anchor, cand, score, nc, tok, par, pos, mask, nn, stats)


def verify_greedy(logits, tokens, parents, n_nodes: int):
    """Greedy tree verification (Sec. 3.6, Eq. 16 at temperature 0): returns
    (accepted draft count, new tokens incl. the bonus, path of nodes)."""
    lg = _c(logits, np.uint16)
    tk = _c(tokens, np.int32)
    pr = _c(parents, np.int32)
    N, V = lg.shape
    nt = np.full(max(N, 1), -1, np.int32)
    path = np.zeros(max(N, 1), np.int32)
    nn = np.zeros(1, np.int32)
    acc = _load().oracle_verify_greedy(_p(lg), V, _p(tk), _p(pr), n_nodes, _p(nt), _p(path),
                                       _p(nn))
    n = int(nn[0])
    return int(acc), nt[:n].tolist(), path[:n].tolist()


@dataclass
class AcceptResult:
    n_accept: np.ndarray
    new_tokens: np.ndarray
    n_new: np.ndarray
    full: np.ndarray


def accept_greedy(logits, draft_tokens, parents, n_nodes, tokens=None, lengths=None,
                  node_reps=None, reps=None, query=None) -> AcceptResult:
    """Verification and append for a batch; tokens/lengths/reps/query (numpy,
    modified in place) are optional (all or none for the append)."""
    lg = _c(logits, np.uint16)
    B, N, V = lg.shape
    tk = _c(draft_tokens, np.int32)
    pr = _c(parents, np.int32)
    nn = _c(n_nodes, np.int32)
    n_acc = np.zeros(B, np.int32)
    new = np.zeros((B, N), np.int32)
    n_new = np.zeros(B, np.int32)
    full = np.zeros(B, np.int32)
    if tokens is not None:
        assert tokens.dtype == np.int32 and tokens.flags.c_contiguous
        ld = tokens.shape[1]
        args = [_p(tokens), ld, _p(lengths)]
    else:
        args = [None, 0, None]
    if node_reps is not None:
        nr = _c(node_reps, np.uint16)
        d = nr.shape[2]
        args += [_p(nr), _p(reps), d, _p(query)]
    else:
        args += [None, None, 0, None]
    _load().oracle_accept_greedy(_p(lg), V, _p(tk), _p(pr), _p(nn), B, N, _p(n_acc), _p(new),
                                 _p(n_new), *args, _p(full))
    return AcceptResult(n_acc, new, n_new, full)
