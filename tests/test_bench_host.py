"""Host-side helpers of bench.py (no GPU): ablation flag parsing and the
algorithmic byte count under each variant."""
import os

import numpy as np
import pytest

import bench
from paper_2606_05742_gb300 import native


def test_flag_names_match_the_library():
    assert bench.FLAG_NAMES == {"no_lex_rerank": native.NO_LEX_RERANK,
                                "succ_on_strict": native.SUCC_ON_STRICT,
                                "no_semantic": native.NO_SEMANTIC,
                                "no_branch": native.NO_BRANCH, "no_succ": native.NO_SUCC}
    assert bench.parse_flags("") == 0
    assert bench.parse_flags("no_succ, NO_BRANCH") == native.NO_SUCC | native.NO_BRANCH
    with pytest.raises(SystemExit):
        bench.parse_flags("no_such_flag")


class _W:
    B, d, k, W = 3, 16, 4, 2


def test_algorithmic_bytes_by_variant():
    L = 10
    tokens = np.tile(np.arange(L, dtype=np.int32) % 5, (3, 1))
    lengths = np.full(3, L, np.int32)
    # sequence 0 lexical (3 candidates), 1 semantic, 2 nothing
    g = {"hit_kind": np.array([1, 2, 0]), "n_cand": np.array([3, 2, 0]),
         "n_nodes": np.array([4, 3, 1]),
         "parents": np.array([[-1, 0, 1, 0], [-1, 0, 0, -1], [-1, -1, -1, -1]]),
         "draft_tokens": np.array([[4, 0, 1, 2], [4, 1, 3, -1], [4, -1, -1, -1]])}
    base = bench.algorithmic_bytes(_W, g, lengths, tokens)
    assert base["lexical"] == 4 * 30
    assert base["semantic"] == 2 * (9 * 16 * 2 + 16 * 2) + 4 * 3   # two sequences scan
    no_sem = bench.algorithmic_bytes(_W, g, lengths, tokens, native.NO_SEMANTIC)
    assert no_sem["semantic"] == 0
    # rerank rows of the lexical hit: 3 candidates + the query
    no_rr = bench.algorithmic_bytes(_W, g, lengths, tokens, native.NO_LEX_RERANK)
    assert base["tree"] - no_rr["tree"] == 4 * 16 * 2
    # successors of the semantic hit: scan 4*(L-1), the reference row, and
    # min(k, occurrences) rows per branch head (tokens 1 and 3: 2 each in 0..8)
    no_succ = bench.algorithmic_bytes(_W, g, lengths, tokens, native.NO_SUCC)
    assert base["tree"] - no_succ["tree"] == 4 * 9 + (1 + 2 + 2) * 16 * 2
    # text-rule successors add the lexical hit's branch head (node 3, token 2)
    strict = bench.algorithmic_bytes(_W, g, lengths, tokens, native.SUCC_ON_STRICT)
    assert strict["tree"] - base["tree"] == 4 * 9 + (1 + 2) * 16 * 2


def test_reference_arm_prints_one_line(capsys):
    """`bench.py --impl reference` times whole oracle steps over the full
    workload on host threads and prints the contract's JSON line, with the
    same config object the native arm prints (small workload: config 1)."""
    import json
    import argparse
    args = argparse.Namespace(config=1, seed=0, steps=2, warmup=1, gpus=1, batch=None,
                              flags="", embeddings=False)
    bench.run_reference(args)
    out = [ln for ln in capsys.readouterr().out.splitlines() if ln.startswith("{")]
    assert len(out) == 1
    line = json.loads(out[0])
    assert line["impl"] == "reference" and line["value"] > 0 and line["steps"] == 2
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["cores"] >= 1
    assert line["e2e"] == {"value": line["value"], "unit": line["unit"],
                           "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
    conf = bench.workload_config(1)
    conf["outcomes"] = line["config"]["outcomes"]
    assert line["config"] == conf
    assert sum(conf["outcomes"].values()) == conf["B"]


def test_algorithmic_bytes_embedding_mode():
    """With a token-embedding table the fallback counts one row per distinct
    token of the fallback histories and anchors together (each row read
    once) and one pass over each history's ids."""
    L = 10
    tokens = np.tile(np.arange(L, dtype=np.int32) % 5, (3, 1))   # 5 distinct in 0..8
    lengths = np.full(3, L, np.int32)
    g = {"hit_kind": np.array([1, 2, 0]), "n_cand": np.array([3, 2, 0]),
         "n_nodes": np.array([4, 3, 1]),
         "parents": np.array([[-1, 0, 1, 0], [-1, 0, 0, -1], [-1, -1, -1, -1]]),
         "draft_tokens": np.array([[4, 0, 1, 2], [4, 1, 7, -1], [4, -1, -1, -1]])}
    de = 8
    x = bench.algorithmic_bytes(_W, g, lengths, tokens, emb_dim=de)
    assert x["semantic"] == 5 * de * 2 + 2 * 4 * L + 4 * 3
    base = bench.algorithmic_bytes(_W, g, lengths, tokens)
    # the semantic hit adds its Eq. 6 rerank rows (2 + query); its branch
    # token 7 never occurs: the backoff gathers the 5 distinct rows + anchor
    # and scores min(k, L-1) positions instead of none
    extra = (2 + 1) * 16 * 2 + (5 + 1) * de * 2 + 4 * L + 4 * 16 * 2
    assert x["tree"] - base["tree"] == extra


def test_oracle_run_times_whole_steps_of_the_batch():
    """The CPU baseline runs the oracle's whole step over every sequence of
    the batch (one per task): the outcomes it reports are the oracle's own,
    whatever the thread count."""
    import oracle
    from paper_2606_05742_gb300 import synth
    w = synth.make_workload(2, B=5, L=600, d=16, nohit=0.4, seed=3)
    run = bench.OracleRun(w.tokens, w.lengths, w.reps, w.query, w.n_max, w.k, w.W, w.D,
                          w.succ_len, w.tau)
    assert run.step(3) > 0
    ref = oracle.step(w.tokens, w.lengths, w.reps, w.query, w.n_max, w.k, w.W, w.D,
                      w.succ_len, w.tau)
    assert (run.hit == ref.hit).all()
    o = run.outcomes()
    assert o["none"] + o["lexical"] + o["semantic"] == 5 and o["lexical"] >= 1
    run.step(1)
    assert (run.hit == ref.hit).all()


def test_workload_config_is_shared_by_both_arms():
    a = bench.workload_config(5)
    assert a == bench.workload_config(5, None, 0, None)
    assert a["B"] == 8 and a["L"] == 131072 and a["d"] == 8192
    r = bench.workload_config(2, batch=4, flags=native.NO_SUCC)
    assert r["B"] == r["global_batch"] == 4 and r["flags"] == native.NO_SUCC


def test_profile_summaries_describe_the_current_sources():
    """Every ncu summary under profiles/ records the sha256 of the sources it
    was captured against; each must match the source as it stands, or the
    summary must say how the current file (named by its current hash)
    differs.  The semantic kernel's summary, which the benchmark scales into
    roofline.traffic, must match exactly."""
    import glob
    import hashlib
    import re

    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    csrc = os.path.join(root, "paper_2606_05742_gb300", "csrc")
    current = {os.path.basename(f): hashlib.sha256(open(f, "rb").read()).hexdigest()
               for f in glob.glob(os.path.join(csrc, "*.cu*"))}
    summaries = sorted(glob.glob(os.path.join(root, "profiles", "*.md")))
    assert summaries
    for path in summaries:
        text = open(path).read()
        recorded = re.findall(r"([a-z_]+\.cuh?) sha256 ([0-9a-f]{64})", text)
        assert recorded, f"{os.path.basename(path)} records no source hashes"
        for name, h in recorded:
            assert name in current, (path, name)
            assert h == current[name] or current[name] in text, (
                f"{os.path.basename(path)}: {name} changed since the capture")
    assert bench.semantic_traffic(10**9) is not None
