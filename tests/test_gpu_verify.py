"""Greedy verification and the memory append on the GPU (adapld_accept_greedy)
against the oracle, bit for bit: the target's choice per node (first index
of the maximum bf16 logit), the accepted path, the new tokens and the
appended tokens, hidden-state rows and query (Sec. 3.6, Eq. 16 at
temperature 0; Algorithm 1)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_05742_gb300 import build, native, synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    build.build()
    native.load()


def cuda_i32(x):
    return torch.from_numpy(np.ascontiguousarray(x, dtype=np.int32)).cuda()


def cuda_bf16(bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).cuda().view(torch.bfloat16)


def host_bits(t):
    return t.view(torch.int16).cpu().numpy().view(np.uint16)


def run_both(logits, draft, parents, n_nodes, memory=None, node_reps=None, ws=None):
    """adapld_accept_greedy and oracle.accept_greedy on the same inputs.
    memory = (tokens [B][ld], lengths [B], reps [B][ld][d] bits, query [B][d]
    bits) or None; the oracle appends into copies."""
    B, N, V = logits.shape
    o_mem = None
    if memory is not None:
        o_mem = [np.array(m, copy=True) for m in memory]
    o = oracle.accept_greedy(logits, draft, parents, n_nodes,
                             *(o_mem[:2] if o_mem else (None, None)),
                             node_reps if memory is not None else None,
                             *(o_mem[2:] if o_mem and node_reps is not None else (None, None)))
    n_acc = torch.full((B,), -9, dtype=torch.int32, device="cuda")
    new = torch.full((B, N), -9, dtype=torch.int32, device="cuda")
    n_new = torch.full((B,), -9, dtype=torch.int32, device="cuda")
    st = torch.full((B,), -9, dtype=torch.int32, device="cuda")
    if ws is None:
        ws = native.allocate_workspace(B, 1, 8, native.make_params(1, 1, 0, 1))
    kw = {}
    if memory is not None:
        kw = dict(tokens=cuda_i32(memory[0]), lengths=cuda_i32(memory[1]))
        if node_reps is not None:
            kw.update(node_reps=cuda_bf16(node_reps), reps=cuda_bf16(memory[2]),
                      query=cuda_bf16(memory[3]))
    native.accept_greedy(cuda_bf16(logits), cuda_i32(draft), cuda_i32(parents), cuda_i32(n_nodes),
                         n_acc, new, n_new, ws, status=st, **kw)
    torch.cuda.synchronize()
    gpu = dict(n_accept=n_acc.cpu().numpy(), new=new.cpu().numpy(), n_new=n_new.cpu().numpy(),
               status=st.cpu().numpy())
    if memory is not None:
        gpu["tokens"] = kw["tokens"].cpu().numpy()
        gpu["lengths"] = kw["lengths"].cpu().numpy()
        if node_reps is not None:
            gpu["reps"] = host_bits(kw["reps"])
            gpu["query"] = host_bits(kw["query"])
    return gpu, o, o_mem


def assert_same(gpu, o, o_mem):
    assert (gpu["n_accept"] == o.n_accept).all()
    assert (gpu["n_new"] == o.n_new).all()
    assert (gpu["new"] == o.new_tokens).all()
    assert ((gpu["status"] & native.SEQ_FULL) != 0).tolist() == (o.full != 0).tolist()
    if o_mem is not None:
        assert (gpu["tokens"] == o_mem[0]).all()
        assert (gpu["lengths"] == o_mem[1]).all()
        if "reps" in gpu:
            assert (gpu["reps"] == o_mem[2]).all()
            assert (gpu["query"] == o_mem[3]).all()


def planted_logits(draft, parents, n_nodes, V, rng, p_accept=0.7, spread=3):
    """bf16 logits [B][N][V]: small random integers (many exact ties, so the
    first-index rule decides) plus, with probability p_accept, a clear maximum
    at one child's token, so that paths of several tokens get accepted."""
    B, N = draft.shape
    lg = rng.integers(-spread, spread, size=(B, N, V)).astype(np.float32)
    for b in range(B):
        n = int(n_nodes[b])
        for i in range(n):
            kids = [c for c in range(1, n) if parents[b, c] == i]
            if kids and rng.random() < p_accept:
                t = int(draft[b, kids[int(rng.integers(len(kids)))]])
                if 0 <= t < V:
                    lg[b, i, t] = 8.0
    return synth.f32_to_bf16_bits(lg)


def step_trees(cfg, seed, V, **kw):
    """Trees from a real GPU step on a small workload of config `cfg`."""
    w = synth.make_workload(cfg, seed=seed, V=V, **kw)
    p = native.make_params(w.n_max, w.k, w.W, w.D, w.succ_len, w.tau, 0)
    eng = native.Engine(w.B, w.ld, w.d, p)
    tok = cuda_i32(w.tokens)
    ln = cuda_i32(w.lengths)
    eng.run(tok, ln, cuda_bf16(w.reps), cuda_bf16(w.query))
    torch.cuda.synchronize()
    g = eng.out.to_host()
    return w, g, eng


@pytest.mark.parametrize("seed,with_reps", [(0, True), (1, True), (2, False), (3, True)])
def test_trees_from_a_step(seed, with_reps):
    rng = np.random.default_rng(1100 + seed)
    V = 512
    lengths = [600, 600, 600, 0, 640, 600, 300, 1, 600, 639]
    w, g, eng = step_trees(2, seed, V, B=10, L=600, d=64, ld=640, nohit=0.5, lengths=lengths)
    lg = planted_logits(g["draft_tokens"], g["parents"], g["n_nodes"], V, rng)
    node_reps = None
    if with_reps:
        node_reps = synth.f32_to_bf16_bits(
            rng.standard_normal(g["draft_tokens"].shape + (w.d,)).astype(np.float32))
    mem = (w.tokens, w.lengths, w.reps, w.query)
    gpu, o, o_mem = run_both(lg, g["draft_tokens"], g["parents"], g["n_nodes"], mem,
                             node_reps, ws=eng.ws)
    assert_same(gpu, o, o_mem)
    assert o.n_accept.max() >= 2          # the planted choices were accepted somewhere
    assert o.full[4] == 1                 # length == ld: no room for the new tokens
    assert (gpu["status"][4] & native.SEQ_FULL) != 0


def test_verification_only_and_repeated_calls():
    """Without the append, twice on one workspace (the per-call counters
    start again from zero)."""
    rng = np.random.default_rng(7)
    V = 1024
    w, g, eng = step_trees(4, 5, V, B=12, L=3000, d=32, nohit=0.5)
    for rep in range(2):
        lg = planted_logits(g["draft_tokens"], g["parents"], g["n_nodes"], V, rng)
        gpu, o, _ = run_both(lg, g["draft_tokens"], g["parents"], g["n_nodes"], ws=eng.ws)
        assert_same(gpu, o, None)
        assert (gpu["status"] == 0).all()


def chain_tree(N, n, toks):
    draft = np.full((1, N), -1, np.int32)
    par = np.full((1, N), -1, np.int32)
    draft[0, :n] = toks[:n]
    par[0, 1:n] = np.arange(n - 1)
    return draft, par


def test_hand_built_trees():
    """Whole chain accepted; root-only tree (the bonus token alone); an empty
    tree; all logits equal (choice 0); two children with the same token (the
    first in node order wins); a child stored before its parent."""
    V, N = 64, 8
    B = 6
    draft = np.full((B, N), -1, np.int32)
    par = np.full((B, N), -1, np.int32)
    nn = np.zeros(B, np.int32)
    lg = np.zeros((B, N, V), np.float32)
    # 0: chain 0-1-2-3-4 of tokens 5,6,7,8 all chosen, bonus 9
    draft[0, :5] = [0, 5, 6, 7, 8]
    par[0, 1:5] = [0, 1, 2, 3]
    nn[0] = 5
    for i, t in enumerate([5, 6, 7, 8, 9]):
        lg[0, i, t] = 1.0
    # 1: root only: bonus = argmax at the root
    draft[1, 0] = 3
    nn[1] = 1
    lg[1, 0, 40] = 2.0
    # 2: empty tree
    nn[2] = 0
    # 3: all-equal logits: the choice is token 0, which child 1 carries
    draft[3, :3] = [1, 0, 0]
    par[3, 1:3] = [0, 0]
    nn[3] = 3
    # 4: siblings 1 and 2 both carry token 11; only node 2 has a child (12)
    draft[4, :4] = [0, 11, 11, 12]
    par[4, 1:4] = [0, 0, 2]
    nn[4] = 4
    lg[4, 0, 11] = 3.0
    lg[4, 1, 12] = 3.0
    lg[4, 2, 12] = 3.0
    # 5: node 1 is the child of node 2
    draft[5, :3] = [0, 21, 20]
    par[5, 1:3] = [2, 0]
    nn[5] = 3
    lg[5, 0, 20] = 1.0
    lg[5, 2, 21] = 1.0
    lg[5, 1, 33] = 1.0
    bits = synth.f32_to_bf16_bits(lg)
    gpu, o, _ = run_both(bits, draft, par, nn)
    assert_same(gpu, o, None)
    assert gpu["n_accept"].tolist() == [4, 0, 0, 1, 1, 2]
    assert gpu["new"][0, :5].tolist() == [5, 6, 7, 8, 9]
    assert gpu["new"][1, :2].tolist() == [40, -1] and gpu["n_new"][1] == 1
    assert gpu["n_new"][2] == 0 and (gpu["new"][2] == -1).all()
    assert gpu["new"][3, :2].tolist() == [0, 0]
    assert gpu["new"][4, :3].tolist() == [11, 12, -1]  # through node 1, the first in order
    assert gpu["new"][5, :3].tolist() == [20, 21, 33]


def test_choice_across_row_splits():
    """Rows long enough to be split over several CTAs (V = 40960): equal
    maxima in different splits go to the first index; -0 and +0 tie; the
    maximum at the last index; a row of equal values."""
    V, N = 40960, 4
    lg = np.full((1, N, V), -2.0, np.float32)
    lg[0, 0, 30000] = 5.0
    lg[0, 0, 100] = 5.0
    lg[0, 1, :] = -1.0
    lg[0, 2, 17000] = 0.0
    lg[0, 2, 50] = -0.0
    lg[0, 3, V - 1] = 7.0
    draft = np.array([[0, 100, 0, 50]], np.int32)
    par = np.array([[-1, 0, 1, 2]], np.int32)
    nn = np.array([4], np.int32)
    gpu, o, _ = run_both(synth.f32_to_bf16_bits(lg), draft, par, nn)
    assert_same(gpu, o, None)
    assert gpu["n_accept"][0] == 3
    assert gpu["new"][0].tolist() == [100, 0, 50, V - 1]


def test_maximum_trees_from_a_step():
    """Trees of the largest size (1024 nodes: D = 255, W = 64, succ_len = 11,
    branches from a 64-wide next-token table, successors on every hit) from
    a GPU step, verified and appended (tokens, hidden-state rows, query)."""
    rng = np.random.default_rng(1024)
    V = 4000
    w = synth.make_workload(2, B=3, L=2000, ld=2600, d=64, V=V, nohit=0.5, seed=91)
    tk = synth.make_next_topk(w.tokens, w.lengths, V, 64, seed=91)
    p = native.make_params(8, 32, 64, 255, 11, float("-inf"), oracle.SUCC_ON_STRICT)
    eng = native.Engine(w.B, w.ld, w.d, p)
    eng.run(cuda_i32(w.tokens), cuda_i32(w.lengths), cuda_bf16(w.reps), cuda_bf16(w.query),
            next_topk=cuda_i32(tk))
    torch.cuda.synchronize()
    g = eng.out.to_host()
    assert g["draft_tokens"].shape[1] == 1024 and int(g["n_nodes"].max()) > 300
    lg = planted_logits(g["draft_tokens"], g["parents"], g["n_nodes"], V, rng, p_accept=0.9)
    node_reps = synth.f32_to_bf16_bits(
        rng.standard_normal(g["draft_tokens"].shape + (w.d,)).astype(np.float32))
    mem = (w.tokens, w.lengths, w.reps, w.query)
    gpu, o, o_mem = run_both(lg, g["draft_tokens"], g["parents"], g["n_nodes"], mem,
                             node_reps, ws=eng.ws)
    assert_same(gpu, o, o_mem)
    assert o.n_accept.max() >= 8


@pytest.mark.parametrize("N,depth", [(300, 200), (600, 450)])
def test_deep_chains(N, depth):
    """Chains of N nodes (N x S <= 1024 caps the row splits: at N = 600 one
    CTA walks every 32 KB group of its row) accepted to a planted depth."""
    V = 40960
    rng = np.random.default_rng(N)
    B = 2
    draft = np.full((B, N), -1, np.int32)
    par = np.full((B, N), -1, np.int32)
    draft[:, 1:] = rng.integers(0, V, size=(B, N - 1))
    par[:, 1:] = np.arange(N - 1)
    nn = np.array([N, N - 7], np.int32)
    lg = rng.integers(-4, 4, size=(B, N, V)).astype(np.float32)
    for b in range(B):
        for i in range(min(depth, int(nn[b]) - 1)):
            lg[b, i, draft[b, i + 1]] = 9.0
    gpu, o, _ = run_both(synth.f32_to_bf16_bits(lg), draft, par, nn)
    assert_same(gpu, o, None)
    assert gpu["n_accept"].tolist() == [depth, depth]


def test_append_boundaries():
    """len + n_new == ld appends (exact fit); one more is FULL with nothing
    appended; a length outside [0, ld] is reported and nothing is appended."""
    V, N, ld, d = 32, 4, 10, 16
    draft, par = chain_tree(N, 3, [0, 4, 5])
    draft = np.repeat(draft, 4, 0)
    par = np.repeat(par, 4, 0)
    nn = np.full(4, 3, np.int32)
    lg = np.zeros((4, N, V), np.float32)
    lg[:, 0, 4] = 1.0
    lg[:, 1, 5] = 1.0
    lg[:, 2, 6] = 1.0                  # everything accepted: n_new = 3
    bits = synth.f32_to_bf16_bits(lg)
    rng = np.random.default_rng(3)
    tokens = rng.integers(0, V, size=(4, ld)).astype(np.int32)
    lengths = np.array([7, 8, 11, 0], np.int32)
    reps = synth.f32_to_bf16_bits(rng.standard_normal((4, ld, d)).astype(np.float32))
    query = synth.f32_to_bf16_bits(rng.standard_normal((4, d)).astype(np.float32))
    node_reps = synth.f32_to_bf16_bits(rng.standard_normal((4, N, d)).astype(np.float32))
    # the oracle does not model a length outside [0, ld]: compare rows 0, 1, 3
    keep = [0, 1, 3]
    mem = (tokens[keep], lengths[keep], reps[keep], query[keep])
    gpu, o, o_mem = run_both(bits[keep], draft[keep], par[keep], nn[keep], mem, node_reps[keep])
    assert_same(gpu, o, o_mem)
    assert gpu["lengths"].tolist() == [10, 8, 3]
    assert gpu["status"].tolist() == [0, native.SEQ_FULL, 0]
    # the bad length, on the GPU alone
    mem = (tokens, lengths, reps, query)
    B = 4
    n_acc = torch.empty(B, dtype=torch.int32, device="cuda")
    new = torch.empty((B, N), dtype=torch.int32, device="cuda")
    n_new = torch.empty(B, dtype=torch.int32, device="cuda")
    st = torch.empty(B, dtype=torch.int32, device="cuda")
    tk, ln = cuda_i32(tokens), cuda_i32(lengths)
    ws = native.allocate_workspace(B, 1, 8, native.make_params(1, 1, 0, 1))
    native.accept_greedy(cuda_bf16(bits), cuda_i32(draft), cuda_i32(par), cuda_i32(nn), n_acc,
                         new, n_new, ws, tokens=tk, lengths=ln, node_reps=cuda_bf16(node_reps),
                         reps=cuda_bf16(reps), query=cuda_bf16(query), status=st)
    torch.cuda.synchronize()
    assert st.cpu().tolist()[2] == native.SEQ_BAD_LENGTH
    assert ln.cpu().tolist()[2] == 11 and (tk.cpu().numpy()[2] == tokens[2]).all()
    assert n_new.cpu().tolist()[2] == 3


def test_full_size_config5():
    """Trees of a full step of the long-context workload (8 x 131072 tokens,
    d = 8192) and target logits over the full 128256-token vocabulary."""
    w = synth.make_workload(5, device="cuda")
    p = native.make_params(w.n_max, w.k, w.W, w.D, w.succ_len, w.tau, 0)
    eng = native.Engine(w.B, w.ld, w.d, p)
    eng.run(w.tokens, w.lengths, w.reps, w.query)
    torch.cuda.synchronize()
    g = eng.out.to_host()
    V = synth.CONFIGS[5]["V"]
    B, N = g["draft_tokens"].shape
    gen = torch.Generator(device="cuda")
    gen.manual_seed(5)
    lg = torch.randn((B, N, V), generator=gen, device="cuda").to(torch.bfloat16)
    rng = np.random.default_rng(5)
    for b in range(B):
        n = int(g["n_nodes"][b])
        for i in range(n):
            kids = [c for c in range(1, n) if g["parents"][b, c] == i]
            if kids and rng.random() < 0.7:
                lg[b, i, int(g["draft_tokens"][b, kids[0]])] = 10.0
    n_acc = torch.empty(B, dtype=torch.int32, device="cuda")
    new = torch.empty((B, N), dtype=torch.int32, device="cuda")
    n_new = torch.empty(B, dtype=torch.int32, device="cuda")
    trees = [cuda_i32(g[k]) for k in ("draft_tokens", "parents", "n_nodes")]
    native.accept_greedy(lg, *trees, n_acc, new, n_new, eng.ws)
    torch.cuda.synchronize()
    o = oracle.accept_greedy(host_bits(lg), g["draft_tokens"], g["parents"], g["n_nodes"])
    assert (n_acc.cpu().numpy() == o.n_accept).all()
    assert (n_new.cpu().numpy() == o.n_new).all()
    assert (new.cpu().numpy() == o.new_tokens).all()
    assert o.n_accept.max() >= 1


@pytest.mark.parametrize("case", range(48))
def test_random_trees(case):
    """Random trees (every parent before its child, random fan-out), tie-heavy
    logits with planted choices, random lengths and capacities, the append
    with and without hidden states, against the oracle."""
    rng = np.random.default_rng(700 + case)
    B = int(rng.integers(1, 12))
    N = int(rng.integers(1, 80))
    V = int(rng.choice([8, 64, 1000, 20000]))
    ld = int(rng.integers(4, 200))
    d = int(rng.choice([8, 32, 136]))
    draft = np.full((B, N), -1, np.int32)
    par = np.full((B, N), -1, np.int32)
    nn = rng.integers(0, N + 1, size=B).astype(np.int32)
    for b in range(B):
        for i in range(1, int(nn[b])):
            par[b, i] = int(rng.integers(0, i))
        draft[b, : nn[b]] = rng.integers(0, V, size=int(nn[b]))
    lg = planted_logits(draft, par, nn, V, rng, p_accept=float(rng.uniform(0.3, 0.95)),
                        spread=int(rng.integers(1, 4)))
    mode = case % 3  # 0: verification only, 1: append tokens, 2: append tokens and rows
    mem, node_reps = None, None
    if mode:
        tokens = rng.integers(0, V, size=(B, ld)).astype(np.int32)
        lengths = rng.integers(0, ld + 1, size=B).astype(np.int32)
        reps = synth.f32_to_bf16_bits(rng.standard_normal((B, ld, d)).astype(np.float32))
        query = synth.f32_to_bf16_bits(rng.standard_normal((B, d)).astype(np.float32))
        mem = (tokens, lengths, reps, query)
        if mode == 2:
            node_reps = synth.f32_to_bf16_bits(
                rng.standard_normal((B, N, d)).astype(np.float32))
    gpu, o, o_mem = run_both(lg, draft, par, nn, mem, node_reps)
    assert_same(gpu, o, o_mem)


@pytest.mark.parametrize("case,N,V", [(0, 1024, 16384), (1, 1024, 16392), (2, 300, 128256),
                                      (3, 700, 40000)])
def test_random_large_trees(case, N, V):
    """Large random trees (up to the 1024-node maximum, parents within 8 of
    their child, so paths run deep) over vocabularies at, just past and far
    past one 16384-entry row split, tie-heavy logits with planted choices."""
    rng = np.random.default_rng(9100 + case)
    B = 2
    draft = np.full((B, N), -1, np.int32)
    par = np.full((B, N), -1, np.int32)
    nn = np.array([N, int(rng.integers(1, N))], np.int32)
    for b in range(B):
        for i in range(1, int(nn[b])):
            par[b, i] = int(rng.integers(max(0, i - 8), i))
        draft[b, : nn[b]] = rng.integers(0, V, size=int(nn[b]))
    lg = rng.integers(-3, 3, size=(B, N, V)).astype(np.float32)
    for b in range(B):
        kids = {}
        for c in range(1, int(nn[b])):
            kids.setdefault(int(par[b, c]), []).append(c)
        for i, ks in kids.items():
            if rng.random() < 0.9:  # plant a child with children of its own when there is one
                inner = [c for c in ks if c in kids] or ks
                lg[b, i, draft[b, inner[int(rng.integers(len(inner)))]]] = 7.0
    gpu, o, o_mem = run_both(synth.f32_to_bf16_bits(lg), draft, par, nn)
    assert_same(gpu, o, o_mem)
    assert o.n_accept.max() >= 4
