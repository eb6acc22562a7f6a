"""Benchmark of one AdaPLD draft-construction step (lexical anchoring ->
semantic fallback -> rerank + draft tree) over B sequences on GB300.

Default workload: the largest-context shape (B=8, L=131072, d=8192, 80%
forced lexical misses, n_max=5, k=32, W=4, D=16, tau=0.1), synthetic and
seeded, resident in HBM (17.2 GB, far above the 129 MB L2, so no flush is
needed between steps).  Prints one JSON line.

  python bench.py [--gpus N --steps K --warmup W] [--impl native|reference]

Under torchrun each rank runs its own batch (weak scaling, no collective on
the data path); rank 0 prints the line with the max-over-ranks time.
``--impl reference`` times the CPU oracle instead (rank 0 only), on a bounded
sample of the same workload.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "draft-construction steps/sec (B seqs, device-timed) and achieved HBM GB/s vs peak"
UNIT = "steps/s"


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["native", "reference"], default="native")
    ap.add_argument("--config", type=int, default=5)
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--embeddings", action="store_true",
                    help="two-representation mode: token-embedding fallback (vocab x d table)")
    ap.add_argument("--batch", type=int, default=None,
                    help="override B (profiling of small cases; not the headline workload)")
    ap.add_argument("--no-verify", dest="verify", action="store_false",
                    help="skip timing greedy verification of the step's trees against "
                         "synthetic target logits [B][nodes][V]")
    ap.add_argument("--verify", dest="verify", action="store_true", help=argparse.SUPPRESS)
    ap.add_argument("--flags", default="",
                    help="ablation variants (Table 4), comma-separated: no_lex_rerank, "
                         "succ_on_strict, no_semantic, no_branch, no_succ")
    ap.add_argument("--e2e-steps", type=int, default=5)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    return ap.parse_args()


def semantic_traffic(algorithmic_bytes: int):
    """DRAM traffic of one semantic-kernel launch, from the committed ncu
    capture (traffic/algorithmic ratio, scaled to this launch's bytes, which
    grow in proportion), or None once the kernel source differs from the
    captured one."""
    import hashlib
    prof = os.path.join(ROOT, "profiles", "semantic_kernel_config5_B2.md")
    csrc = os.path.join(ROOT, "paper_2606_05742_gb300", "csrc")
    if not os.path.exists(prof):
        return None
    text = open(prof).read()
    for name in ("semantic.cu", "common.cuh"):
        h = hashlib.sha256(open(os.path.join(csrc, name), "rb").read()).hexdigest()
        if f"{name} sha256 {h}" not in text:
            return None
    ratio = [ln.split(":", 1)[1] for ln in text.splitlines() if ln.startswith("traffic_ratio:")]
    return int(float(ratio[0]) * algorithmic_bytes) if ratio else None


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            pk = json.load(f)
        return float(pk["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


# ------------------------------------------------------- multi-process
def max_over_ranks(value: float, device=None) -> float:
    """The maximum of a per-rank value over the process group (the value
    itself without one).  Used for the slowest rank's elapsed time."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return value
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(world: int, steps: int, max_ms: float) -> float:
    """Whole-job steps/s: every rank runs `steps` steps of its own batch of B
    sequences (weak scaling), so the job completes world*steps in the slowest
    rank's time."""
    return world * steps / (max_ms / 1000.0)


def rank_seed(seed: int, rank: int) -> int:
    """Each rank draws its own batch."""
    return seed + rank


# --------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons during the timed
    region (read-only queries)."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.idx = gpu_index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                 "-lms", "100", "-i", str(self.idx)],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except (OSError, ValueError):
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                smax.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm)}


# --------------------------------------------------------- oracle timing
class OracleRun:
    """The CPU oracle timed on the benchmark's own workload: every sequence of
    the batch at full length, the same bytes the GPU step reads (host copies
    of the device inputs), one sequence per task on a pool of host threads
    (the C oracle runs outside the GIL).  One step = the oracle's whole
    draft-construction step over the batch."""

    def __init__(self, tokens, lengths, reps, query, n_max, k, W, D, succ_len, tau, flags=0):
        self.args = (tokens, lengths, reps, query)
        self.params = (n_max, k, W, D, succ_len, tau, flags)
        self.B = tokens.shape[0]
        self.hit = None

    def step(self, threads: int) -> float:
        """Runs one step on `threads` host threads; returns its wall time (s)."""
        import concurrent.futures as cf

        import oracle
        tokens, lengths, reps, query = self.args
        n_max, k, W, D, succ_len, tau, flags = self.params
        hit = np.zeros(self.B, np.int32)

        def one(b):
            r = oracle.step(tokens[b:b + 1], lengths[b:b + 1], reps[b:b + 1], query[b:b + 1],
                            n_max, k, W, D, succ_len, tau, flags)
            hit[b] = r.hit[0]

        s = time.perf_counter()
        if threads == 1:
            for b in range(self.B):
                one(b)
        else:
            with cf.ThreadPoolExecutor(max_workers=threads) as ex:
                list(ex.map(one, range(self.B)))
        wall = time.perf_counter() - s
        self.hit = hit
        return wall

    def outcomes(self) -> dict:
        h = self.hit
        return {"lexical": int((h == 1).sum()), "semantic": int((h == 2).sum()),
                "none": int((h == 0).sum())}

    def desc(self, threads: int, cfg_id: int) -> str:
        plural = "s" if threads > 1 else ""
        return (f"oracle (plain C, fp64) on {threads} host thread{plural}, one sequence per "
                f"task: whole steps over the full config-{cfg_id} batch ({self.B} sequences, "
                "full length, the GPU step's own inputs copied to the host)")


def host_threads(batch: int) -> int:
    return max(1, min(batch, os.cpu_count() or 1))


def host_copy(w):
    """numpy copies of a device workload's inputs (bf16 as uint16 bits)."""
    import torch
    tok = w.tokens.cpu().numpy()
    ln = w.lengths.cpu().numpy()
    reps = w.reps.view(torch.int16).cpu().numpy().view(np.uint16)
    q = w.query.view(torch.int16).cpu().numpy().view(np.uint16)
    return tok, ln, reps, q


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    from paper_2606_05742_gb300 import synth
    import torch
    flags = parse_flags(args.flags)
    if args.embeddings:
        print(json.dumps({"impl": "reference", "unavailable": "the reference arm times the "
                          "single-cache step only"}), flush=True)
        return
    if torch.cuda.is_available():  # the native arm's bytes, drawn on the GPU, copied here
        w = synth.make_workload(args.config, device="cuda", seed=args.seed, B=args.batch)
        tok, ln, reps, q = host_copy(w)
        del w
        torch.cuda.empty_cache()
    else:
        w = synth.make_workload(args.config, seed=args.seed, B=args.batch)
        tok, ln, reps, q = w.tokens, w.lengths, w.reps, w.query
    c = synth.CONFIGS[args.config]
    run = OracleRun(tok, ln, reps, q, c["n_max"], c["k"], c["W"], c["D"], 1, synth.TAU, flags)
    threads = host_threads(run.B)
    for _ in range(args.warmup):
        run.step(threads)
    walls = []
    for _ in range(args.steps):  # whole steps, bounded by wall time
        walls.append(run.step(threads))
        if sum(walls) > 120:
            break
    total = sum(walls)
    value = len(walls) / total
    conf = workload_config(args.config, args.batch, flags, None)
    conf["outcomes"] = run.outcomes()
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT,
        "n_gpus": args.gpus, "steps": len(walls), "warmup": args.warmup,
        "ms_per_step": 1000.0 * total / len(walls), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": conf, "parallelism": "host threads (rank 0 only)", "accumulate": "fp64",
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle",
                         "sample": run.desc(threads, args.config)},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def workload_config(cfg_id, batch=None, flags=0, emb_shape=None):
    """The workload as both arms describe it (the same object for the same
    arguments)."""
    from paper_2606_05742_gb300 import synth
    c = synth.CONFIGS[cfg_id]
    B = c["B"] if batch is None else batch
    conf = {"workload": f"config{cfg_id}: {synth.describe(cfg_id)} tau={synth.TAU}",
            "B": B, "L": c["L"], "d": c["d"], "global_batch": B,
            "l2": "inputs larger than L2 (no flush needed)"}
    if emb_shape is not None:
        conf["workload"] += (f" + token-embedding fallback ({emb_shape[0]} x {emb_shape[1]} "
                             "table; two-representation mode)")
    if flags:
        conf["workload"] += f" ablation flags {flags}"
        conf["flags"] = flags
    if batch is not None:
        conf["workload"] += f" (resized: B={B})"
    return conf


# ---------------------------------------------------------- native arm
FLAG_NAMES = {"no_lex_rerank": 1, "succ_on_strict": 2, "no_semantic": 4, "no_branch": 8,
              "no_succ": 16}


def parse_flags(text):
    flags = 0
    for name in filter(None, (x.strip().lower() for x in text.split(","))):
        if name not in FLAG_NAMES:
            raise SystemExit(f"unknown flag {name!r}; known: {', '.join(FLAG_NAMES)}")
        flags |= FLAG_NAMES[name]
    return flags


def algorithmic_bytes(w, g, lengths, tokens, flags=0, emb_dim=None):
    """Bytes the step must move at minimum (no re-reads), per kernel.  With a
    token-embedding table of dimension emb_dim (two-representation mode) the
    fallback needs one table row per distinct token of the fallback
    histories and anchors taken together (the score depends only on the
    token, and a row serves every sequence holding it) plus one pass over
    each history's ids, and a successor backoff one row per distinct token
    of its sequence."""
    d, k = w.d, w.k
    hk = g["hit_kind"]
    semantic = not flags & FLAG_NAMES["no_semantic"]
    active = (hk != 1) & semantic
    lex_bytes = int(4 * lengths.sum())

    def distinct(b):
        L = int(lengths[b])
        return int(np.unique(tokens[b, : L - 1]).size) if L >= 2 else 0

    if emb_dim is None:
        sem_rows = int(sum(lengths[b] - 1 for b in range(w.B) if active[b] and lengths[b] >= 2))
        n_active = int(active.sum())
        sem_bytes = (sem_rows * d * 2 + n_active * d * 2 + 4 * w.B) if semantic else 0
    else:
        fb = [b for b in range(w.B) if active[b] and lengths[b] >= 2]
        union = (np.unique(np.concatenate([tokens[b, : int(lengths[b])] for b in fb])).size
                 if fb else 0)
        sem_bytes = int(union) * emb_dim * 2 + sum(4 * int(lengths[b]) for b in fb)
        sem_bytes += 4 * w.B if semantic else 0
    # tree kernel: rerank rows + query for lexical hits, successor scan + rows
    succ_on = w.W > 0 and not flags & (FLAG_NAMES["no_succ"] | FLAG_NAMES["no_branch"])
    gathered = 0
    succ_scan = 0
    backoff = 0
    for b in range(w.B):
        L = int(lengths[b])
        if hk[b] == 1 and not flags & FLAG_NAMES["no_lex_rerank"]:
            gathered += int(g["n_cand"][b]) + 1
        if emb_dim is not None and hk[b] == 2:     # Eq. 6 rerank of the fallback's list
            gathered += int(g["n_cand"][b]) + 1
        if succ_on and (hk[b] == 2 or (hk[b] == 1 and flags & FLAG_NAMES["succ_on_strict"])):
            n = int(g["n_nodes"][b])
            par = g["parents"][b, :n]
            # branch heads hang off the root; on a lexical hit node 1 is main[0]
            heads = [i for i in range(1, n) if par[i] == 0 and not (hk[b] == 1 and i == 1)]
            succ_scan += 4 * (L - 1)
            gathered += 1
            for h in heads:
                t = int(g["draft_tokens"][b, h])
                occ = int((tokens[b, : L - 1] == t).sum())
                if occ == 0 and emb_dim is not None:   # backoff: the branch token's row
                    backoff += (distinct(b) + 1) * emb_dim * 2 + 4 * L
                    gathered += min(k, L - 1)
                else:
                    gathered += min(k, occ)
    N = g["draft_tokens"].shape[1]
    out_bytes = w.B * (N * 12 + N * N + k * 8 + 32)
    tree_bytes = gathered * d * 2 + succ_scan + backoff + out_bytes
    return {"lexical": lex_bytes, "semantic": sem_bytes, "tree": tree_bytes,
            "step": lex_bytes + sem_bytes + tree_bytes}


def run_native(args):
    import torch
    import torch.distributed as dist

    from paper_2606_05742_gb300 import native, synth

    flags = parse_flags(args.flags)
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)

    def barrier():
        if world > 1:
            dist.barrier()

    cfg = args.config
    w = synth.make_workload(cfg, device=str(dev), seed=rank_seed(args.seed, rank), B=args.batch)
    p = native.make_params(w.n_max, w.k, w.W, w.D, w.succ_len, w.tau, flags)
    eng = native.Engine(w.B, w.ld, w.d, p, device=dev)
    stream = torch.cuda.current_stream(dev)
    emb = None
    if args.embeddings:
        emb = synth.make_embeddings(w, synth.CONFIGS[cfg]["V"], w.d, rank_seed(args.seed, rank))

    for _ in range(max(3, args.warmup)):
        eng.run(w.tokens, w.lengths, w.reps, w.query, emb=emb)
    torch.cuda.synchronize(dev)
    if native.read_device_status(eng.ws) != 0:
        raise RuntimeError("device status raised during warm-up")
    g = eng.out.to_host()
    lengths = w.lengths.cpu().numpy()
    tokens = w.tokens.cpu().numpy()
    nbytes = algorithmic_bytes(w, g, lengths, tokens, flags,
                               emb_dim=None if emb is None else int(emb.shape[1]))

    # Timed region A (the headline): K steps back to back, CUDA events only at
    # the two ends, so consecutive kernels keep their programmatic-launch
    # overlap.  Timed region B: K more steps with events around each kernel,
    # for the per-kernel durations (the roofline) and the stage breakdown.
    K = args.steps
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(6)] for _ in range(K)]
    for row in ev:                       # torch creates CUDA events lazily, on first record
        for e in row:
            e.record(stream)
    clocks = ClockSampler(torch.cuda.current_device()) if rank == 0 else None
    start = torch.cuda.Event(enable_timing=True)
    end = torch.cuda.Event(enable_timing=True)
    barrier()
    torch.cuda.synchronize(dev)
    if clocks:
        clocks.start()
        time.sleep(0.3)
    call = eng.bind(w.tokens, w.lengths, w.reps, w.query, emb=emb, stream=stream)
    launches0 = native.kernel_launches()
    start.record(stream)
    for i in range(K):
        call()
    end.record(stream)
    launches = native.kernel_launches() - launches0  # counted by the library
    torch.cuda.synchronize(dev)
    barrier()
    total_ms = start.elapsed_time(end)
    startb = torch.cuda.Event(enable_timing=True)
    endb = torch.cuda.Event(enable_timing=True)
    startb.record(stream)
    for i in range(K):
        native.step(w.tokens, w.lengths, w.reps, w.query, p, eng.out, eng.ws,
                    events=native.StepEvents(*[e.cuda_event for e in ev[i]]), emb=emb)
    endb.record(stream)
    torch.cuda.synchronize(dev)
    barrier()
    clk = clocks.stop() if clocks else None
    total_b_ms = startb.elapsed_time(endb)
    if native.read_device_status(eng.ws) != 0:
        raise RuntimeError("device status raised during the timed region")
    semantic_on = not flags & FLAG_NAMES["no_semantic"]
    stage = {name: [r[2 * i].elapsed_time(r[2 * i + 1]) for r in ev]
             for i, name in enumerate(("lexical", "semantic", "tree"))
             if name != "semantic" or semantic_on}
    # the dominant kernel: the semantic top-k, or without it the tree stage
    dom_name, dom_kernel = (("semantic", "semantic_kernel" if emb is None else
                             "rep_insert/count/scatter + semantic_kernel (gather) + expand")
                            if semantic_on
                            else ("tree", "succ_scan_kernel + tree_kernel"))
    sem_ms = stage[dom_name]
    total_ms = max_over_ranks(total_ms, dev)
    ms_per_step = total_ms / K
    value = job_throughput(world, K, total_ms)

    # greedy verification (Sec. 3.6) of this step's trees against synthetic
    # target logits; not part of the step (the target model sits in between)
    verify = None
    if args.verify:
        V = synth.CONFIGS[cfg]["V"]
        Bn, N = eng.out.draft_tokens.shape
        gen = torch.Generator(device=dev)
        gen.manual_seed(rank_seed(args.seed, rank))
        logits = torch.randn((Bn, N, V), generator=gen, device=dev).to(torch.bfloat16)
        n_acc = torch.empty(Bn, dtype=torch.int32, device=dev)
        new_t = torch.empty((Bn, N), dtype=torch.int32, device=dev)
        n_new = torch.empty(Bn, dtype=torch.int32, device=dev)
        trees = (eng.out.draft_tokens, eng.out.parents, eng.out.n_nodes)
        for _ in range(3):
            native.accept_greedy(logits, *trees, n_acc, new_t, n_new, eng.ws)
        # events around each call: the device time of one call (counter
        # reset + kernel), whatever the host takes to issue the next one
        vev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(K)]
        for e0, e1 in vev:
            e0.record(stream)
            e1.record(stream)
        torch.cuda.synchronize(dev)
        for e0, e1 in vev:
            e0.record(stream)
            native.accept_greedy(logits, *trees, n_acc, new_t, n_new, eng.ws)
            e1.record(stream)
        torch.cuda.synchronize(dev)
        vms = statistics.median(e0.elapsed_time(e1) for e0, e1 in vev)
        nodes = int(eng.out.n_nodes.sum().item())
        vbytes = nodes * V * 2
        verify = {"ms": vms, "logits_bytes": vbytes, "gbs": vbytes / (vms / 1000.0) / 1e9,
                  "vocab": V, "nodes": nodes, "timing": "median over calls of per-call events"}
        del logits

    # end-to-end through the public API from pinned host buffers
    e2e = None
    host_in = None  # numpy views of the pinned host inputs (also the oracle's inputs)
    if not args.no_e2e and emb is None:
        tok_h = w.tokens.cpu().pin_memory()
        len_h = w.lengths.cpu().pin_memory()
        # the host inputs are written by the CPU, as a host producer would
        # write them (a pinned buffer last written by the GPU read back over
        # the host link at a fraction of the rate in probes)
        reps_h = w.reps.cpu().pin_memory()
        q_h = w.query.cpu().pin_memory()
        host_in = (tok_h.numpy(), len_h.numpy(),
                   reps_h.view(torch.int16).numpy().view(np.uint16),
                   q_h.view(torch.int16).numpy().view(np.uint16))
        dev_in = (torch.empty_like(w.tokens), torch.empty_like(w.lengths),
                  torch.empty_like(w.reps), torch.empty_like(w.query))
        host_out = native.Outputs.allocate(w.B, p, device="cpu", pin_memory=True)
        # one C call per step: host inputs -> device, the step, outputs -> host
        e2e_call, h2d, d2h = eng.bind_from_host(tok_h, len_h, reps_h, q_h, dev_in, host_out,
                                                stream=stream)
        e2e_call()
        torch.cuda.synchronize(dev)
        KE = args.e2e_steps
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        barrier()
        torch.cuda.synchronize(dev)
        e0.record(stream)
        for _ in range(KE):
            e2e_call()
        e1.record(stream)
        torch.cuda.synchronize(dev)
        barrier()
        te = max_over_ranks(e0.elapsed_time(e1), dev)
        e2e = {"value": job_throughput(world, KE, te), "unit": UNIT,
               "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h)}
        del dev_in

    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return

    peak, peak_kind = peaks()
    sem_avg_ms = sum(sem_ms) / len(sem_ms)
    achieved = nbytes[dom_name] / (sem_avg_ms / 1000.0) / 1e9
    step_gbs = nbytes["step"] / (ms_per_step / 1000.0) / 1e9
    cpu = None
    if not args.no_cpu_baseline and emb is None:
        # whole oracle steps over the same batch: one step on every host
        # thread it can use, then one on a single thread (about 10-30 s of
        # host CPU work at configs 3 and 5)
        if host_in is None:
            host_in = host_copy(w)
        run = OracleRun(*host_in, w.n_max, w.k, w.W, w.D, w.succ_len, w.tau, flags)
        threads = host_threads(w.B)
        walls = [run.step(threads) for _ in range(2)]
        wall1 = run.step(1)
        cpu = {"value": len(walls) / sum(walls), "unit": UNIT, "cores": threads,
               "kind": "oracle", "sample": run.desc(threads, cfg) + f"; {len(walls)} steps",
               "value_1_thread": 1.0 / wall1, "sample_1_thread": run.desc(1, cfg) + "; 1 step",
               "outcomes_match": run.outcomes() == {
                   "lexical": int((g["hit_kind"] == 1).sum()),
                   "semantic": int((g["hit_kind"] == 2).sum()),
                   "none": int((g["hit_kind"] == 0).sum())}}
    host_in = None
    hk = g["hit_kind"]
    conf = workload_config(cfg, args.batch, flags,
                           None if emb is None else (int(emb.shape[0]), int(emb.shape[1])))
    conf["outcomes"] = {"lexical": int((hk == 1).sum()), "semantic": int((hk == 2).sum()),
                        "none": int((hk == 0).sum())}
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K,
        "warmup": max(3, args.warmup), "ms_per_step": ms_per_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": conf,
        "parallelism": f"replicas x{world} (batch per GPU)", "accumulate": "fp32",
        "sequence_steps_per_s": value * w.B,
        "roofline": {"bound": "hbm", "kernel": dom_kernel,
                     "achieved": achieved, "peak": peak, "peak_kind": peak_kind,
                     "unit": "GB/s", "frac": achieved / peak,
                     "traffic": (semantic_traffic(nbytes["semantic"])
                                 if emb is None and semantic_on else None),
                     "algorithmic_bytes": nbytes[dom_name], "avg_launch_ms": sem_avg_ms},
        "step_hbm": {"achieved": step_gbs, "frac": step_gbs / peak,
                     "algorithmic_bytes": nbytes["step"]},
        "stage_ms": {name: sum(v) / len(v) for name, v in stage.items()},
        "ms_per_step_with_stage_events": total_b_ms / K,
        "cpu_baseline": cpu,
        "e2e": e2e,
        "verify": verify,
        "gpu_launches": launches,
        "clocks": clk,
    }
    print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def main():
    args = parse()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_native(args)


if __name__ == "__main__":
    main()
