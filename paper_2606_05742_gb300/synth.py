"""Seeded synthetic workloads shaped like the paper's draft-construction inputs.

This module only draws inputs; it holds none of the method's arithmetic and is
the one piece shared by the CUDA path's tests/benchmark and the CPU oracle.

The paper measures on Spec-Bench, CodeEditorBench, AIME 2024, MATH-500 and
MMLU-Pro with Vicuna / Qwen3 hidden states (Sec. 4.1, Tables 5-6).  None of
that is available here, so these generators stand in for it:

* token history: Zipf(s = 1.1) ids over the vocabulary, with a fraction of the
  positions copied from earlier 8-64 token spans (input-grounded reuse,
  Sec. 3.1 and Table 11), so lexical hits occur naturally;
* forced lexical misses: a seeded subset of sequences whose last token is
  replaced by the smallest id absent from the rest of the history (this also
  removes every longer suffix match), bracketing the paper's measured
  semantic / no-hit rates (Table 10);
* representation cache: i.i.d. N(0, 1) bf16 rows with planted near-duplicates
  of a hidden base vector v (v + 0.3 N(0, I)) and a query drawn the same way,
  so the semantic fallback has a well-separated answer (cos ~ 1/1.09 against
  noise of std 1/sqrt(d)); the row of the last position is set to the query,
  since row len-1 and the query are the same prefix state.

Sequence b of config c with seed s draws from ``numpy.random.default_rng([s,
c, b])`` (tokens) and ``[s, c, b, 1]`` (CPU representations), or from a torch
CUDA generator seeded from the same tuple (device representations), so a
sequence is the same whether generated alone or inside its batch.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import Optional

import numpy as np

# The five workload shapes: (B, L, vocab, copy rate, d, forced no-hit fraction,
# planted rows (None = config-1 style noisy copy of one row), n_max, k, W, D).
CONFIGS = {
    1: dict(B=1, L=2048, V=32000, copy=0.30, d=4096, nohit=0.0, planted=None,
            n_max=3, k=8, W=2, D=8),
    2: dict(B=32, L=8192, V=32000, copy=0.20, d=4096, nohit=0.40, planted=4,
            n_max=4, k=8, W=3, D=10),
    3: dict(B=64, L=32768, V=128256, copy=0.10, d=5120, nohit=0.60, planted=4,
            n_max=4, k=16, W=4, D=12),
    4: dict(B=256, L=4096, V=32000, copy=0.25, d=4096, nohit=0.30, planted=4,
            n_max=3, k=8, W=2, D=8),
    5: dict(B=8, L=131072, V=128256, copy=0.05, d=8192, nohit=0.80, planted=16,
            n_max=5, k=32, W=4, D=16),
}
TAU = 0.1          # semantic threshold used throughout the paper's experiments
SUCC_LEN = 1       # one successor token per branch
ZIPF_S = 1.1
MEAN_SPAN = 36.0   # mean of U{8..64}
NOISE = 0.3        # planted-row / query perturbation


def describe(cfg_id: int) -> str:
    c = CONFIGS[cfg_id]
    return (f"B={c['B']} L={c['L']} d={c['d']} vocab={c['V']} copy={c['copy']} "
            f"nohit={c['nohit']} n_max={c['n_max']} k={c['k']} W={c['W']} D={c['D']}")


def copy_event_prob(copy_rate: float) -> float:
    """Per-position probability of starting a copied span so that the expected
    copied fraction equals ``copy_rate`` (mean span 36)."""
    return copy_rate / (MEAN_SPAN - (MEAN_SPAN - 1.0) * copy_rate)


_ZIPF_CDF = {}


def _zipf_cdf(V: int) -> np.ndarray:
    if V not in _ZIPF_CDF:
        w = np.arange(1, V + 1, dtype=np.float64) ** (-ZIPF_S)
        c = np.cumsum(w)
        _ZIPF_CDF[V] = c / c[-1]
    return _ZIPF_CDF[V]


def gen_tokens(rng: np.random.Generator, L: int, V: int, copy_rate: float) -> np.ndarray:
    """Zipf ids with copied spans (see module docstring)."""
    cdf = _zipf_cdf(V)
    toks = np.minimum(np.searchsorted(cdf, rng.random(L), side="right"), V - 1).astype(np.int32)
    u = rng.random(L)
    span = rng.integers(8, 65, size=L)
    start_u = rng.random(L)
    pi = copy_event_prob(copy_rate)
    events = np.flatnonzero(u < pi)
    events = events[events >= 64]
    p_next = 0
    for e in events:
        if e < p_next:
            continue
        s_len = int(span[e])
        s = int(start_u[e] * (e - s_len + 1))
        end = min(e + s_len, L)
        toks[e:end] = toks[s:s + (end - e)]
        p_next = e + s_len
    return toks


def force_no_hit(toks: np.ndarray, length: int, V: int) -> None:
    """Replace the last token by the smallest id absent from the history."""
    seen = np.zeros(V + 1, dtype=bool)
    seen[toks[: length - 1]] = True
    toks[length - 1] = int(np.argmin(seen))


def forced_set(cfg_id: int, B: int, frac: float, seed: int) -> np.ndarray:
    n = int(math.floor(frac * B + 0.5))
    rng = np.random.default_rng([seed, cfg_id, 1_000_003])
    return np.sort(rng.permutation(B)[:n])


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round-to-nearest-even fp32 -> bf16, returned as uint16 bit patterns."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    r = ((u >> 16) & 1) + np.uint32(0x7FFF)
    return ((u + r) >> 16).astype(np.uint16)


def bf16_bits_to_f32(h: np.ndarray) -> np.ndarray:
    return (np.asarray(h, dtype=np.uint32) << 16).view(np.float32)


@dataclass
class Workload:
    cfg_id: int
    B: int
    ld: int
    d: int
    n_max: int
    k: int
    W: int
    D: int
    succ_len: int
    tau: float
    tokens: object            # [B][ld] int32 (numpy or torch)
    lengths: object           # [B] int32
    reps: object              # [B][ld][d] bf16 (numpy uint16 bits or torch bf16)
    query: object             # [B][d]
    forced: np.ndarray        # indices of forced lexical misses
    planted: list = field(default_factory=list)  # per sequence planted rows
    device: str = "cpu"


def make_tokens(cfg_id: int, *, B: Optional[int] = None, L: Optional[int] = None,
                ld: Optional[int] = None, lengths=None, seed: int = 0,
                nohit: Optional[float] = None, V: Optional[int] = None):
    """The token histories of ``make_workload`` with the same arguments (the
    same seeds), without the representation cache: (tokens [B][ld] int32,
    lengths [B] int32, forced misses)."""
    c = CONFIGS[cfg_id]
    B = c["B"] if B is None else B
    L = c["L"] if L is None else L
    V = c["V"] if V is None else V
    ld = L if ld is None else ld
    frac = c["nohit"] if nohit is None else nohit
    if lengths is None:
        lengths = np.full(B, L, dtype=np.int32)
    lengths = np.asarray(lengths, dtype=np.int32)
    assert lengths.shape == (B,) and int(lengths.max()) <= ld
    tokens = np.zeros((B, ld), dtype=np.int32)
    forced = forced_set(cfg_id, B, frac, seed)
    fset = set(forced.tolist())
    for b in range(B):
        rng = np.random.default_rng([seed, cfg_id, b])
        tokens[b] = gen_tokens(rng, ld, V, c["copy"])
        ln = int(lengths[b])
        if b in fset and ln >= 1:
            force_no_hit(tokens[b], ln, V)
    return tokens, lengths, forced


def make_workload(cfg_id: int, *, device: str = "cpu", B: Optional[int] = None,
                  L: Optional[int] = None, d: Optional[int] = None, ld: Optional[int] = None,
                  lengths=None, seed: int = 0, nohit: Optional[float] = None,
                  planted: Optional[int] = -1, V: Optional[int] = None) -> Workload:
    """Build config ``cfg_id`` (optionally resized) on ``device``.

    ``device="cpu"`` returns numpy arrays (representations as uint16 bf16
    bits); ``"cuda"`` returns torch tensors with the representation cache drawn
    on the GPU in row chunks.  ``lengths`` gives ragged sequences (each <= ld).
    """
    c = dict(CONFIGS[cfg_id])
    B = c["B"] if B is None else B
    L = c["L"] if L is None else L
    d = c["d"] if d is None else d
    ld = L if ld is None else ld
    n_plant = c["planted"] if planted == -1 else planted
    tokens, lengths, forced = make_tokens(cfg_id, B=B, L=L, ld=ld, lengths=lengths, seed=seed,
                                          nohit=nohit, V=V)

    planted_rows = []
    if device == "cpu":
        reps = np.zeros((B, ld, d), dtype=np.uint16)
        query = np.zeros((B, d), dtype=np.uint16)
        for b in range(B):
            rng = np.random.default_rng([seed, cfg_id, b, 1])
            R = rng.standard_normal((ld, d), dtype=np.float32)
            ln = int(lengths[b])
            q, rows = _plant(rng, R, ln, d, n_plant)
            planted_rows.append(rows)
            if ln >= 1:
                R[ln - 1] = q
            reps[b] = f32_to_bf16_bits(R)
            query[b] = f32_to_bf16_bits(q)
        tok_out, len_out = tokens, lengths
    else:
        import torch
        dev = torch.device(device)
        reps = torch.empty((B, ld, d), dtype=torch.bfloat16, device=dev)
        query = torch.empty((B, d), dtype=torch.bfloat16, device=dev)
        chunk = max(1, (1 << 26) // d)
        for b in range(B):
            g = torch.Generator(device=dev)
            g.manual_seed(_torch_seed(seed, cfg_id, b))
            for r0 in range(0, ld, chunk):
                r1 = min(ld, r0 + chunk)
                reps[b, r0:r1] = torch.randn((r1 - r0, d), generator=g, device=dev,
                                             dtype=torch.float32).to(torch.bfloat16)
            rng = np.random.default_rng([seed, cfg_id, b, 1])
            ln = int(lengths[b])
            q, rows = _plant_torch(rng, g, reps[b], ln, d, n_plant)
            planted_rows.append(rows)
            query[b] = q.to(torch.bfloat16)
            if ln >= 1:
                reps[b, ln - 1] = query[b]
        tok_out = torch.from_numpy(tokens).to(dev)
        len_out = torch.from_numpy(lengths).to(dev)
    return Workload(cfg_id, B, ld, d, c["n_max"], c["k"], c["W"], c["D"], SUCC_LEN, TAU,
                    tok_out, len_out, reps, query, forced, planted_rows, device)


def _torch_seed(seed: int, cfg_id: int, b: int) -> int:
    return int(np.random.default_rng([seed, cfg_id, b, 2]).integers(0, 2**62))


def _plant(rng, R, ln, d, n_plant):
    """Planted near-duplicates (numpy, fp32 before rounding to bf16)."""
    if ln < 2:
        return rng.standard_normal(d, dtype=np.float32), []
    if n_plant is None:           # config-1 style: the query is a noisy copy of one row
        r = int(rng.integers(0, ln - 1))
        q = R[r] + np.float32(NOISE) * rng.standard_normal(d, dtype=np.float32)
        return q.astype(np.float32), [r]
    v = rng.standard_normal(d, dtype=np.float32)
    m = min(n_plant, ln - 1)
    rows = np.sort(rng.choice(ln - 1, size=m, replace=False)).tolist()
    for r in rows:
        R[r] = v + np.float32(NOISE) * rng.standard_normal(d, dtype=np.float32)
    q = v + np.float32(NOISE) * rng.standard_normal(d, dtype=np.float32)
    return q.astype(np.float32), rows


def _plant_torch(rng, g, Rb, ln, d, n_plant):
    """Planted near-duplicates on the device (positions from numpy, values from
    the torch generator)."""
    import torch
    dev = Rb.device

    def randn():
        return torch.randn(d, generator=g, device=dev, dtype=torch.float32)

    if ln < 2:
        return randn(), []
    if n_plant is None:
        r = int(rng.integers(0, ln - 1))
        q = Rb[r].float() + NOISE * randn()
        return q, [r]
    v = randn()
    m = min(n_plant, ln - 1)
    rows = np.sort(rng.choice(ln - 1, size=m, replace=False)).tolist()
    for r in rows:
        Rb[r] = (v + NOISE * randn()).to(torch.bfloat16)
    return v + NOISE * randn(), rows


def make_next_topk(tokens: np.ndarray, lengths: np.ndarray, V: int, Kn: int,
                   seed: int = 0) -> np.ndarray:
    """A synthetic cached next-token top-K table [B][ld][Kn] (distinct ids per
    row): with probability 1/2 the observed continuation comes first, the rest
    are Zipf draws.  Stands in for the target model's TopK(p(.|M_<=j))."""
    B, ld = tokens.shape
    rng = np.random.default_rng([seed, 77, B, ld])
    cdf = _zipf_cdf(V)
    out = np.full((B, ld, Kn), -1, dtype=np.int32)
    for b in range(B):
        for j in range(ld):
            row = []
            if j + 1 < lengths[b] and rng.random() < 0.5:
                row.append(int(tokens[b, j + 1]))
            while len(row) < Kn:
                t = int(min(np.searchsorted(cdf, rng.random(), side="right"), V - 1))
                if t not in row:
                    row.append(t)
            out[b, j] = row
    return out


def make_embeddings(w: Workload, V: int, de: int, seed: int = 0, synonyms: int = 3):
    """A token-embedding table E[V][de] (bf16) for the two-representation
    mode: i.i.d. N(0,1) rows, and for every forced lexical miss, `synonyms`
    tokens of its history (always including the token just before the
    anchor) get rows E[a] + 0.3 N(0, I) around the anchor's row, so the
    embedding fallback (Eq. 4) finds them and a candidate right before the
    anchor makes the anchor itself a branch token with no earlier
    occurrence (the successor backoff of Sec. 3.5).  numpy uint16 bits on
    the CPU, a torch bf16 tensor when the workload lives on a GPU.  A forced
    miss in a history that already holds all V ids takes id V
    (`force_no_hit`), so the table gets max(V, largest id + 1) rows."""
    tokens = w.tokens if isinstance(w.tokens, np.ndarray) else w.tokens.cpu().numpy()
    lengths = w.lengths if isinstance(w.lengths, np.ndarray) else w.lengths.cpu().numpy()
    rng = np.random.default_rng([seed, 31337, V, de])
    V = max(V, int(tokens.max()) + 1) if tokens.size else V
    plants = []
    for b in w.forced:
        ln = int(lengths[b])
        if ln < 3 or ln > tokens.shape[1]:   # too short, or an invalid length
            continue
        a = int(tokens[b, ln - 1])
        hist = tokens[b, : ln - 1]
        pick = {int(hist[-1])}
        cand = np.unique(hist[hist != a])
        extra = rng.permutation(cand)[: max(0, synonyms - 1)]
        pick.update(int(x) for x in extra)
        pick.discard(a)
        plants.append((a, sorted(pick)))
    if w.device == "cpu":
        E = rng.standard_normal((V, de), dtype=np.float32)
        for a, vs in plants:
            for v in vs:
                E[v] = E[a] + np.float32(NOISE) * rng.standard_normal(de, dtype=np.float32)
        return f32_to_bf16_bits(E)
    import torch
    dev = torch.device(w.device)
    g = torch.Generator(device=dev)
    g.manual_seed(int(rng.integers(0, 2**62)))
    E = torch.empty((V, de), dtype=torch.bfloat16, device=dev)
    chunk = max(1, (1 << 26) // de)
    for r0 in range(0, V, chunk):
        r1 = min(V, r0 + chunk)
        E[r0:r1] = torch.randn((r1 - r0, de), generator=g, device=dev,
                               dtype=torch.float32).to(torch.bfloat16)
    for a, vs in plants:
        ea = E[a].float()
        for v in vs:
            E[v] = (ea + NOISE * torch.randn(de, generator=g, device=dev,
                                             dtype=torch.float32)).to(torch.bfloat16)
    return E
