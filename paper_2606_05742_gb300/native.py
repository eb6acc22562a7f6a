"""ctypes binding of ``libadapld.so`` (C ABI in ``include/adapld.h``).

Argument marshalling only: every step of the draft-construction path runs in
the library's CUDA kernels.  Tensors are torch CUDA tensors (device memory and
streams are PyTorch's); the functions pass their data pointers and the current
stream to the C ABI and raise :class:`AdapldError` on a non-zero status.  There
is no CPU fallback: if the library is missing the first call raises.
"""
from __future__ import annotations

import ctypes
import math
import os
from dataclasses import dataclass
from typing import Optional

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libadapld.so")

# ---- constants mirrored from include/adapld.h ----------------------------------
HIT_NONE, HIT_LEX, HIT_SEM = 0, 1, 2
NO_LEX_RERANK = 1
SUCC_ON_STRICT = 2
NO_SEMANTIC = 4
NO_BRANCH = 8
NO_SUCC = 16
SEQ_BAD_LENGTH = 1
SEQ_BAD_CANDIDATE = 2
SEQ_BAD_TOKEN = 4
SEQ_FULL = 8
DEV_TIMEOUT = 1
DEV_INTERNAL = 2

EXPORTED = [
    "adapld_tree_nodes", "adapld_workspace_bytes", "adapld_status_string",
    "adapld_lexical_match", "adapld_semantic_topk", "adapld_build_draft_tree",
    "adapld_step", "adapld_step_ex", "adapld_read_device_status",
    "adapld_semantic_topk_static", "adapld_embedding_topk", "adapld_accept_greedy",
    "adapld_step_from_host", "adapld_semantic_topk_static_status", "adapld_kernel_launches",
]
STATIC_MAX_B = 1024
ERR_NULL = -1
ERR_ALIGN = -8
ERR_WORKSPACE = -9
ERR_STATIC_LIMIT = -15


class AdapldError(RuntimeError):
    def __init__(self, code: int, where: str):
        super().__init__(f"{where}: {status_string(code)} (status {code})")
        self.code = code


class Params(ctypes.Structure):
    _fields_ = [("n_max", ctypes.c_int32), ("k", ctypes.c_int32),
                ("branch_width", ctypes.c_int32), ("draft_len", ctypes.c_int32),
                ("succ_len", ctypes.c_int32), ("tau", ctypes.c_float),
                ("flags", ctypes.c_uint32)]


def make_params(n_max: int, k: int, branch_width: int, draft_len: int, succ_len: int = 1,
                tau: float = 0.1, flags: int = 0) -> Params:
    return Params(n_max, k, branch_width, draft_len, succ_len, tau, flags)


class TreeOut(ctypes.Structure):
    _fields_ = [("anchor", ctypes.c_void_p), ("draft_tokens", ctypes.c_void_p),
                ("parents", ctypes.c_void_p), ("positions", ctypes.c_void_p),
                ("mask", ctypes.c_void_p), ("n_nodes", ctypes.c_void_p),
                ("stats", ctypes.c_void_p)]


class StepOut(ctypes.Structure):
    _fields_ = [("hit_kind", ctypes.c_void_p), ("match_n", ctypes.c_void_p),
                ("cand", ctypes.c_void_p), ("score", ctypes.c_void_p),
                ("n_cand", ctypes.c_void_p), ("status", ctypes.c_void_p),
                ("tree", TreeOut)]


class Embeddings(ctypes.Structure):
    """Token-embedding table [vocab][dim] bf16 (two-representation mode)."""
    _fields_ = [("table", ctypes.c_void_p), ("vocab", ctypes.c_int32), ("dim", ctypes.c_int32)]

    @staticmethod
    def of(table) -> "Embeddings":
        V, dim = table.shape
        return Embeddings(table.data_ptr(), V, dim)


class StepEvents(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in
                ("lexical_begin", "lexical_end", "semantic_begin", "semantic_end",
                 "tree_begin", "tree_end")]


_lib = None


def _configure(lib: ctypes.CDLL) -> ctypes.CDLL:
    P, i32, i64, sz, f32 = (ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t,
                            ctypes.c_float)
    lib.adapld_tree_nodes.argtypes = [P]
    lib.adapld_tree_nodes.restype = i32
    lib.adapld_workspace_bytes.argtypes = [i32, i64, i32, P]
    lib.adapld_workspace_bytes.restype = sz
    lib.adapld_status_string.argtypes = [ctypes.c_int]
    lib.adapld_status_string.restype = ctypes.c_char_p
    lib.adapld_lexical_match.argtypes = [P, i64, P, i32, i32, i32, P, P, P, P, P, sz, P]
    lib.adapld_semantic_topk.argtypes = [P, i64, i32, P, P, P, i32, i32, f32, P, P, P, P, sz, P]
    lib.adapld_build_draft_tree.argtypes = [P, i64, P, P, i32, P, i32, P, P, P, P, P, i32, P,
                                            P, P, P, P, sz, P]
    lib.adapld_step.argtypes = [P, i64, P, P, i32, P, P, i32, i32, P, P, P, sz, P]
    lib.adapld_step_ex.argtypes = [P, i64, P, P, i32, P, P, i32, i32, P, P, P, sz, P, P, P]
    lib.adapld_embedding_topk.argtypes = [P, i64, P, P, P, i32, i32, f32, P, P, P, P, P, sz, P]
    lib.adapld_read_device_status.argtypes = [P, P, P]
    lib.adapld_semantic_topk_static.argtypes = [P, i64, i32, P, P, P, i32, i32, f32, P, P, P, P]
    lib.adapld_semantic_topk_static_status.argtypes = [P, P]
    lib.adapld_accept_greedy.argtypes = [P, i32, P, P, P, i32, i32, P, P, P, P, i64, P, P, P,
                                         i32, P, P, P, sz, P]
    lib.adapld_step_from_host.argtypes = [P, i64, P, P, i32, P, i32, P, P, P, P, P, P, P, P, sz,
                                          P]
    lib.adapld_kernel_launches.argtypes = []
    lib.adapld_kernel_launches.restype = ctypes.c_ulonglong
    for f in ("adapld_lexical_match", "adapld_semantic_topk", "adapld_build_draft_tree",
              "adapld_step", "adapld_step_ex", "adapld_read_device_status",
              "adapld_semantic_topk_static", "adapld_embedding_topk",
              "adapld_accept_greedy", "adapld_step_from_host",
              "adapld_semantic_topk_static_status"):
        getattr(lib, f).restype = ctypes.c_int
    return lib


def load() -> ctypes.CDLL:
    """Loads the CUDA library; raises if it has not been built."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(
                f"{LIB_PATH} is missing: build it first (python -c 'import __graft_entry__ as g; "
                "g.build()'); there is no CPU fallback")
        _lib = _configure(ctypes.CDLL(LIB_PATH))
    return _lib


def load_library(path: str) -> ctypes.CDLL:
    """Another build of the library (e.g. the checked debug build), configured
    like the default one; not cached."""
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing; there is no CPU fallback")
    return _configure(ctypes.CDLL(path))


def status_string(code: int) -> str:
    return load().adapld_status_string(code).decode()


def _check(rc: int, where: str) -> None:
    if rc != 0:
        raise AdapldError(rc, where)


def _ptr(t) -> Optional[int]:
    return None if t is None else t.data_ptr()


def _stream(stream) -> int:
    import torch
    s = torch.cuda.current_stream() if stream is None else stream
    return s.cuda_stream


def tree_nodes(p: Params) -> int:
    return load().adapld_tree_nodes(ctypes.byref(p))


def workspace_bytes(B: int, ld: int, d: int, p: Optional[Params] = None) -> int:
    return load().adapld_workspace_bytes(B, ld, d, ctypes.byref(p) if p is not None else None)


def lexical_match(tokens, lengths, n_max: int, k: int, hit_kind, match_n, cand, n_cand, ws,
                  stream=None) -> None:
    B, ld = tokens.shape
    rc = load().adapld_lexical_match(_ptr(tokens), ld, _ptr(lengths), B, n_max, k, _ptr(hit_kind),
                                     _ptr(match_n), _ptr(cand), _ptr(n_cand), _ptr(ws),
                                     ws.numel() * ws.element_size(), _stream(stream))
    _check(rc, "adapld_lexical_match")


def semantic_topk(reps, query, lengths, k: int, tau: float, cand, score, n_cand, ws,
                  active=None, stream=None) -> None:
    B, ld, d = reps.shape
    rc = load().adapld_semantic_topk(_ptr(reps), ld, d, _ptr(query), _ptr(lengths),
                                     _ptr(active), B, k, tau, _ptr(cand), _ptr(score),
                                     _ptr(n_cand), _ptr(ws), ws.numel() * ws.element_size(),
                                     _stream(stream))
    _check(rc, "adapld_semantic_topk")


def semantic_topk_static(reps, query, lengths, k: int, tau: float, cand, score, n_cand,
                         active=None, stream=None) -> None:
    """adapld_semantic_topk_static: the semantic fallback for callers that
    cannot supply a workspace (scratch in the library's own device array;
    B <= 1024; calls must not overlap on the GPU)."""
    B, ld, d = reps.shape
    rc = load().adapld_semantic_topk_static(_ptr(reps), ld, d, _ptr(query), _ptr(lengths),
                                            _ptr(active), B, k, tau, _ptr(cand), _ptr(score),
                                            _ptr(n_cand), _stream(stream))
    _check(rc, "adapld_semantic_topk_static")


def kernel_launches() -> int:
    """Kernels the library has enqueued in this process (adapld_kernel_launches)."""
    return int(load().adapld_kernel_launches())


def semantic_topk_static_status(stream=None) -> int:
    """ADAPLD_DEV_* bits of the last adapld_semantic_topk_static call on the
    current device (synchronises the stream)."""
    st = ctypes.c_int32(-1)
    _check(load().adapld_semantic_topk_static_status(ctypes.byref(st), _stream(stream)),
           "adapld_semantic_topk_static_status")
    return st.value


def _tree_out(anchor, draft_tokens, parents, positions, mask, n_nodes, stats=None) -> TreeOut:
    return TreeOut(_ptr(anchor), _ptr(draft_tokens), _ptr(parents), _ptr(positions),
                   _ptr(mask), _ptr(n_nodes), _ptr(stats))


def build_draft_tree(tokens, lengths, reps, query, hit_kind, cand, score, n_cand, p: Params,
                     out: "Outputs", ws, next_topk=None, emb=None, stream=None) -> None:
    B, ld, d = reps.shape
    to = _tree_out(out.anchor, out.draft_tokens, out.parents, out.positions, out.mask,
                   out.n_nodes, out.stats)
    kn = next_topk.shape[2] if next_topk is not None else 0
    e = Embeddings.of(emb) if emb is not None else None
    rc = load().adapld_build_draft_tree(
        _ptr(tokens), ld, _ptr(lengths), _ptr(reps), d, _ptr(query), B, _ptr(hit_kind),
        _ptr(cand), _ptr(score), _ptr(n_cand), _ptr(next_topk), kn,
        ctypes.byref(e) if e is not None else None, ctypes.byref(p),
        ctypes.byref(to), _ptr(out.status), _ptr(ws), ws.numel() * ws.element_size(),
        _stream(stream))
    _check(rc, "adapld_build_draft_tree")


def embedding_topk(tokens, lengths, emb, k: int, tau: float, cand, score, n_cand, ws,
                   active=None, status=None, stream=None) -> None:
    """Eq. 4 over token embeddings (adapld_embedding_topk)."""
    B, ld = tokens.shape
    e = Embeddings.of(emb)
    rc = load().adapld_embedding_topk(_ptr(tokens), ld, _ptr(lengths), ctypes.byref(e),
                                      _ptr(active), B, k, tau, _ptr(cand), _ptr(score),
                                      _ptr(n_cand), _ptr(status), _ptr(ws),
                                      ws.numel() * ws.element_size(), _stream(stream))
    _check(rc, "adapld_embedding_topk")


@dataclass
class Outputs:
    """Device output buffers of one step (layouts as in adapld_step_out)."""
    hit_kind: object
    match_n: object
    cand: object
    score: object
    n_cand: object
    status: object
    anchor: object
    draft_tokens: object
    parents: object
    positions: object
    mask: object
    n_nodes: object
    stats: object

    @staticmethod
    def allocate(B: int, p: Params, device="cuda", pin_memory=False) -> "Outputs":
        """Buffers on `device` ("cpu" with pin_memory=True: page-locked host
        buffers for adapld_step_from_host)."""
        import torch
        N = 1 + p.draft_len + p.branch_width * (1 + p.succ_len)
        i32 = dict(dtype=torch.int32, device=device, pin_memory=pin_memory)
        return Outputs(
            torch.empty(B, **i32), torch.empty(B, **i32), torch.empty((B, p.k), **i32),
            torch.empty((B, p.k), dtype=torch.float32, device=device, pin_memory=pin_memory),
            torch.empty(B, **i32), torch.empty(B, **i32), torch.empty(B, **i32),
            torch.empty((B, N), **i32), torch.empty((B, N), **i32), torch.empty((B, N), **i32),
            torch.empty((B, N, N), dtype=torch.uint8, device=device, pin_memory=pin_memory),
            torch.empty(B, **i32), torch.empty(4, **i32))

    def c_struct(self) -> StepOut:
        return StepOut(_ptr(self.hit_kind), _ptr(self.match_n), _ptr(self.cand),
                       _ptr(self.score), _ptr(self.n_cand), _ptr(self.status),
                       _tree_out(self.anchor, self.draft_tokens, self.parents, self.positions,
                                 self.mask, self.n_nodes, self.stats))

    def tensors(self):
        return [self.hit_kind, self.match_n, self.cand, self.score, self.n_cand, self.status,
                self.anchor, self.draft_tokens, self.parents, self.positions, self.mask,
                self.n_nodes, self.stats]

    def nbytes(self) -> int:
        return sum(t.numel() * t.element_size() for t in self.tensors())

    def to_host(self) -> dict:
        names = ["hit_kind", "match_n", "cand", "score", "n_cand", "status", "anchor",
                 "draft_tokens", "parents", "positions", "mask", "n_nodes", "stats"]
        return {n: t.cpu().numpy() for n, t in zip(names, self.tensors())}


def allocate_workspace(B: int, ld: int, d: int, p: Params, device="cuda"):
    import torch
    nbytes = workspace_bytes(B, ld, d, p)
    if nbytes == 0:
        raise AdapldError(-7, "adapld_workspace_bytes")
    return torch.empty(nbytes, dtype=torch.uint8, device=device)


def step(tokens, lengths, reps, query, p: Params, out: Outputs, ws, next_topk=None,
         events: Optional[StepEvents] = None, stream=None, emb=None) -> None:
    """One draft-construction step (adapld_step, or adapld_step_ex with
    events and/or a token-embedding table `emb` [vocab][dim] bf16)."""
    B, ld, d = reps.shape
    so = out.c_struct()
    kn = next_topk.shape[2] if next_topk is not None else 0
    lib = load()
    args = (_ptr(tokens), ld, _ptr(lengths), _ptr(reps), d, _ptr(query), _ptr(next_topk), kn, B,
            ctypes.byref(p), ctypes.byref(so), _ptr(ws), ws.numel() * ws.element_size())
    if events is None and emb is None:
        rc = lib.adapld_step(*args, _stream(stream))
    else:
        e = Embeddings.of(emb) if emb is not None else None
        rc = lib.adapld_step_ex(*args, ctypes.byref(e) if e is not None else None,
                                ctypes.byref(events) if events is not None else None,
                                _stream(stream))
    _check(rc, "adapld_step")


def accept_greedy(logits, draft_tokens, parents, n_nodes, n_accept, new_tokens, n_new, ws,
                  tokens=None, lengths=None, node_reps=None, reps=None, query=None,
                  status=None, stream=None) -> None:
    """Greedy tree verification and the memory append (adapld_accept_greedy).
    logits [B][N][V] bf16; optional append into tokens/lengths (and, with
    node_reps [B][N][d], reps/query)."""
    B, N, V = logits.shape
    ld = tokens.shape[1] if tokens is not None else 0
    d = node_reps.shape[2] if node_reps is not None else 0
    rc = load().adapld_accept_greedy(
        _ptr(logits), V, _ptr(draft_tokens), _ptr(parents), _ptr(n_nodes), B, N, _ptr(n_accept),
        _ptr(new_tokens), _ptr(n_new), _ptr(tokens), ld, _ptr(lengths), _ptr(node_reps),
        _ptr(reps), d, _ptr(query), _ptr(status), _ptr(ws), ws.numel() * ws.element_size(),
        _stream(stream))
    _check(rc, "adapld_accept_greedy")


def read_device_status(ws, stream=None) -> int:
    v = ctypes.c_int32(0)
    _check(load().adapld_read_device_status(_ptr(ws), ctypes.byref(v), _stream(stream)),
           "adapld_read_device_status")
    return int(v.value)


class BoundCall:
    """A library call with its arguments marshalled once (see Engine.bind)."""

    def __init__(self, fn, args, keep, name):
        self._fn, self._args, self._keep, self._name = fn, args, keep, name

    def __call__(self) -> None:
        rc = self._fn(*self._args)
        if rc:
            _check(rc, self._name)


class Engine:
    """Owns the device buffers for repeated steps over B sequences of capacity
    ld and dimension d, and offers the end-to-end call from host tensors."""

    def __init__(self, B: int, ld: int, d: int, p: Params, device="cuda"):
        import torch
        self.B, self.ld, self.d, self.p = B, ld, d, p
        self.device = torch.device(device)
        self.out = Outputs.allocate(B, p, device)
        self.ws = allocate_workspace(B, ld, d, p, device)

    def run(self, tokens, lengths, reps, query, next_topk=None, events=None, stream=None,
            emb=None):
        step(tokens, lengths, reps, query, self.p, self.out, self.ws, next_topk, events, stream,
             emb)
        return self.out

    def bind_from_host(self, tokens_h, lengths_h, reps_h, query_h, dev_inputs, host_out,
                       stream=None):
        """The end-to-end step through adapld_step_from_host, arguments
        marshalled once: each call copies the host inputs (page-locked) into
        `dev_inputs` (tokens, lengths, reps, query on the device), runs the
        step into self.out and copies every output into `host_out` (an
        Outputs of page-locked host tensors).  Returns (call, h2d bytes, d2h
        bytes)."""
        B, ld, d = reps_h.shape
        tok_d, len_d, reps_d, q_d = dev_inputs
        so_d = self.out.c_struct()
        so_h = host_out.c_struct()
        lib = load()
        args = (_ptr(tokens_h), ld, _ptr(lengths_h), _ptr(reps_h), d, _ptr(query_h), B,
                ctypes.byref(self.p), _ptr(tok_d), _ptr(len_d), _ptr(reps_d), _ptr(q_d),
                ctypes.byref(so_d), ctypes.byref(so_h), _ptr(self.ws),
                self.ws.numel() * self.ws.element_size(), _stream(stream))
        h2d = sum(t.numel() * t.element_size() for t in (tokens_h, lengths_h, reps_h, query_h))
        return (BoundCall(lib.adapld_step_from_host, args, [so_d, so_h, self.p],
                          "adapld_step_from_host"), h2d, host_out.nbytes())

    def bind(self, tokens, lengths, reps, query, next_topk=None, stream=None, emb=None):
        """The step on fixed buffers with its arguments marshalled once: the
        returned callable enqueues one step per call (a decode loop updates
        the buffers' contents in place between calls)."""
        B, ld, d = reps.shape
        so = self.out.c_struct()
        kn = next_topk.shape[2] if next_topk is not None else 0
        lib = load()
        args = [_ptr(tokens), ld, _ptr(lengths), _ptr(reps), d, _ptr(query), _ptr(next_topk),
                kn, B, ctypes.byref(self.p), ctypes.byref(so), _ptr(self.ws),
                self.ws.numel() * self.ws.element_size()]
        keep = [so, self.p]
        if emb is None:
            fn = lib.adapld_step
        else:
            e = Embeddings.of(emb)
            keep.append(e)
            fn = lib.adapld_step_ex
            args += [ctypes.byref(e), None]
        args.append(_stream(stream))
        return BoundCall(fn, tuple(args), keep, "adapld_step")

    def run_from_host(self, tokens_h, lengths_h, reps_h, query_h, dev_inputs, host_out,
                      stream=None, copy_streams: int = 4):
        """End-to-end step from pinned host inputs: copies them into the
        device buffers ``dev_inputs`` (tokens, lengths, reps, query), runs the
        step and copies every output back into the pinned ``host_out`` list
        (same order as :meth:`Outputs.tensors`).  The representation cache is
        copied in ``copy_streams`` row blocks on side streams so that several
        copy engines share the host link.  Returns bytes moved (host->device,
        device->host)."""
        import torch
        main = torch.cuda.current_stream(self.device) if stream is None else stream
        tok_d, len_d, reps_d, q_d = dev_inputs
        if getattr(self, "_copy_streams", None) is None or len(self._copy_streams) != copy_streams:
            self._copy_streams = [torch.cuda.Stream(device=self.device)
                                  for _ in range(copy_streams)]
        h2d = 0
        start = torch.cuda.Event()
        start.record(main)
        rows_h = reps_h.view(-1, reps_h.shape[-1])
        rows_d = reps_d.view(-1, reps_d.shape[-1])
        n = rows_h.shape[0]
        bounds = [n * i // copy_streams for i in range(copy_streams + 1)]
        for s, lo, hi in zip(self._copy_streams, bounds[:-1], bounds[1:]):
            s.wait_event(start)
            with torch.cuda.stream(s):
                rows_d[lo:hi].copy_(rows_h[lo:hi], non_blocking=True)
            done = torch.cuda.Event()
            done.record(s)
            main.wait_event(done)
        h2d += reps_h.numel() * reps_h.element_size()
        with torch.cuda.stream(main):
            for src, dst in ((tokens_h, tok_d), (lengths_h, len_d), (query_h, q_d)):
                dst.copy_(src, non_blocking=True)
                h2d += src.numel() * src.element_size()
            self.run(tok_d, len_d, reps_d, q_d, stream=main)
            d2h = 0
            for src, dst in zip(self.out.tensors(), host_out):
                dst.copy_(src, non_blocking=True)
                d2h += src.numel() * src.element_size()
        return h2d, d2h
