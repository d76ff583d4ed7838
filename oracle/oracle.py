"""CPU oracle for the GBA aggregate-and-apply step (arXiv 2205.11048).

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline leg are the only users.  The product library never
imports this module and shares no code with ``gba_oracle.c``.

``OracleGBA`` is the parameter server of Alg. 2 reduced to one process: a FIFO
gradient buffer that pops the shortest prefix of messages whose local batches
reach the global batch (Sec. 4.1: apply once N_a gradients are buffered), then
runs one global step of ``gba_oracle.c`` on them.  State is kept only for a
tracked set of rows per table and of dense elements; rows are independent of
one another, so any subset evolves exactly as it would in the full model.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from dataclasses import dataclass, field

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "gba_oracle.c")
_LIB = os.path.join(_HERE, "libgba_oracle.so")

ADAGRAD = 0
ADAM = 1
INT32_MAX = 2**31 - 1


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (no fused multiply-add, plain -O2)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(
            ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-shared",
             "-fPIC", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


class _Opt(ctypes.Structure):
    _fields_ = [("kind", ctypes.c_int32), ("lr", ctypes.c_float), ("init_acc", ctypes.c_float),
                ("beta1", ctypes.c_float), ("beta2", ctypes.c_float), ("eps", ctypes.c_float)]


class _Table(ctypes.Structure):
    _fields_ = [("V", ctypes.c_int64), ("d", ctypes.c_int32), ("id_mode", ctypes.c_int32),
                ("opt", _Opt), ("n_track", ctypes.c_int64),
                ("track", ctypes.POINTER(ctypes.c_int64)),
                ("w", ctypes.POINTER(ctypes.c_float)), ("s0", ctypes.POINTER(ctypes.c_float)),
                ("s1", ctypes.POINTER(ctypes.c_float)), ("ver", ctypes.POINTER(ctypes.c_int64))]


class _Dense(ctypes.Structure):
    _fields_ = [("D", ctypes.c_int64), ("opt", _Opt), ("n_track", ctypes.c_int64),
                ("track", ctypes.POINTER(ctypes.c_int64)),
                ("w", ctypes.POINTER(ctypes.c_float)), ("s0", ctypes.POINTER(ctypes.c_float)),
                ("s1", ctypes.POINTER(ctypes.c_float))]


class _Rule(ctypes.Structure):
    _fields_ = [("iota", ctypes.c_int32), ("row_staleness", ctypes.c_int32),
                ("sparse_denominator", ctypes.c_int32), ("decay", ctypes.c_int32),
                ("lambda_", ctypes.c_float), ("drop_latest", ctypes.c_int32)]


class Stats(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int64) for n in (
        "msgs_kept", "msgs_dropped", "dense_stale_sum", "dense_stale_max", "pairs",
        "pairs_dropped", "row_stale_sum", "row_stale_max", "occurrences", "rows_touched",
        "rows_applied")]

    def as_dict(self):
        return {n: int(getattr(self, n)) for n, _ in self._fields_}


_lib = None


def load(path: str):
    """Load an oracle library (the default build, or a copy compiled elsewhere)."""
    L = ctypes.CDLL(path)
    _declare(L)
    return L


def lib():
    global _lib
    if _lib is None:
        _lib = load(build())
    return _lib


def _declare(L):
    """Set the ctypes signatures of the oracle's exported functions."""
    L.gbao_splitmix64.restype = ctypes.c_uint64
    L.gbao_splitmix64.argtypes = [ctypes.c_uint64]
    L.gbao_init_weight.restype = ctypes.c_float
    L.gbao_init_weight.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_uint64]
    L.gbao_table_tag.restype = ctypes.c_uint64
    L.gbao_table_tag.argtypes = [ctypes.c_int32]
    L.gbao_dense_tag.restype = ctypes.c_uint64
    L.gbao_dense_tag.argtypes = []
    L.gbao_init_table.argtypes = [ctypes.POINTER(_Table), ctypes.c_int32, ctypes.c_uint64]
    L.gbao_init_dense.argtypes = [ctypes.POINTER(_Dense), ctypes.c_uint64]
    L.gbao_select_prefix.restype = ctypes.c_int32
    L.gbao_select_prefix.argtypes = [ctypes.POINTER(ctypes.c_int32), ctypes.c_int32,
                                        ctypes.c_int64]
    L.gbao_step.restype = ctypes.c_int
    L.gbao_step.argtypes = [
        ctypes.c_int64, ctypes.POINTER(_Rule), ctypes.c_int32, ctypes.POINTER(ctypes.c_int64),
        ctypes.c_int32, ctypes.POINTER(_Table), ctypes.POINTER(ctypes.c_void_p),
        ctypes.POINTER(ctypes.c_int64), ctypes.POINTER(ctypes.c_void_p),
        ctypes.POINTER(_Dense), ctypes.POINTER(ctypes.c_void_p),
        ctypes.POINTER(ctypes.c_int32), ctypes.POINTER(ctypes.c_void_p),
        ctypes.POINTER(ctypes.c_void_p), ctypes.POINTER(Stats)]


def splitmix64(x: int) -> int:
    return int(lib().gbao_splitmix64(ctypes.c_uint64(x & (2**64 - 1))))


def init_weight(seed: int, tag: int, e: int) -> float:
    return float(lib().gbao_init_weight(seed & (2**64 - 1), tag, e))


def table_tag(t: int) -> int:
    return int(lib().gbao_table_tag(t))


def dense_tag() -> int:
    return int(lib().gbao_dense_tag())


def select_prefix(B, G: int) -> int:
    arr = np.ascontiguousarray(np.asarray(B, dtype=np.int32))
    return int(lib().gbao_select_prefix(
        arr.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)), len(arr), int(G)))


def _fptr(a):
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_float)) if a is not None else None


def _iptr(a):
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_int64))


@dataclass
class OptSpec:
    kind: int = ADAGRAD
    lr: float = 0.01
    init_acc: float = 0.1
    beta1: float = 0.9
    beta2: float = 0.999
    eps: float = 1e-8

    def c(self) -> _Opt:
        return _Opt(self.kind, self.lr, self.init_acc, self.beta1, self.beta2, self.eps)


@dataclass
class TableSpec:
    rows: int
    dim: int
    opt: OptSpec = field(default_factory=OptSpec)
    id_mode: int = 0   # 0: row = id, 1: row = uint64(id) mod rows, 2: each id its own row


@dataclass
class Message:
    """One worker push: token, local batch, per-table ids/rows, dense gradient."""
    token: int
    local_batch: int
    ids: list          # per table: int64 [n]
    rows: list         # per table: float32 [n, d]
    dense: np.ndarray  # float32 [D]


class _TableState:
    def __init__(self, spec: TableSpec, t: int, track, seed: int, L):
        self.spec = spec
        self.track = np.ascontiguousarray(np.asarray(track, dtype=np.int64))
        assert np.all(np.diff(self.track) > 0), "tracked rows must be strictly increasing"
        n, d = len(self.track), spec.dim
        self.w = np.zeros(n * d, np.float32)
        self.s0 = np.zeros(n * d, np.float32)
        self.s1 = np.zeros(n * d, np.float32) if spec.opt.kind == ADAM else None
        self.ver = np.zeros(n, np.int64)
        self.c = _Table(spec.rows, spec.dim, spec.id_mode, spec.opt.c(), n, _iptr(self.track),
                        _fptr(self.w), _fptr(self.s0), _fptr(self.s1), _iptr(self.ver))
        L.gbao_init_table(ctypes.byref(self.c), t, seed & (2**64 - 1))

    def row_index(self, rows):
        return np.searchsorted(self.track, rows)


class _DenseState:
    def __init__(self, D: int, opt: OptSpec, track, seed: int, L):
        self.track = np.ascontiguousarray(
            np.arange(D, dtype=np.int64) if track is None else np.asarray(track, np.int64))
        n = len(self.track)
        self.w = np.zeros(n, np.float32)
        self.s0 = np.zeros(n, np.float32)
        self.s1 = np.zeros(n, np.float32) if opt.kind == ADAM else None
        self.c = _Dense(D, opt.c(), n, _iptr(self.track), _fptr(self.w), _fptr(self.s0),
                        _fptr(self.s1))
        L.gbao_init_dense(ctypes.byref(self.c), seed & (2**64 - 1))


class OracleGBA:
    """The aggregate-and-apply state machine of Alg. 2 on the CPU."""

    def __init__(self, tables, dense_size: int, dense_opt: OptSpec, global_batch: int,
                 iota: int = INT32_MAX, row_staleness: int = 0, sparse_denominator: int = 0,
                 seed: int = 0, track_rows=None, track_dense=None, library=None, decay: int = 0,
                 lam: float = 1.0, drop_latest: int = 0):
        self.L = library if library is not None else lib()
        self.specs = list(tables)
        self.D = int(dense_size)
        self.G = int(global_batch)
        self.rule = _Rule(int(iota), int(row_staleness), int(sparse_denominator), int(decay),
                          float(lam), int(drop_latest))
        self.k = 0
        self.fifo: list[Message] = []
        self.tables = []
        for t, spec in enumerate(self.specs):
            tr = np.arange(spec.rows, dtype=np.int64) if track_rows is None or \
                track_rows[t] is None else track_rows[t]
            self.tables.append(_TableState(spec, t, tr, seed, self.L))
        self.dense = _DenseState(self.D, dense_opt, track_dense, seed, self.L)
        self.last_keep = None
        self.last_count = None
        self.last_kept = None
        self.last_stats = None
        self._c_tables = (_Table * max(1, len(self.tables)))(*[ts.c for ts in self.tables])

    def push(self, msg: Message) -> None:
        self.fifo.append(msg)

    def pull_version(self) -> int:
        return self.k

    def try_apply(self) -> int:
        B = np.ascontiguousarray(np.array([m.local_batch for m in self.fifo], dtype=np.int32))
        M = int(self.L.gbao_select_prefix(
            B.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)), len(B), self.G))
        if M == 0:
            return 0
        batch, self.fifo = self.fifo[:M], self.fifo[M:]
        self.apply_messages(batch)
        return 1

    def apply_messages(self, batch) -> None:
        """Run one global step on exactly these popped messages."""
        M, T = len(batch), len(self.tables)
        tokens = np.array([m.token for m in batch], dtype=np.int64)
        keep = []  # hold references while C reads them
        ids_p = (ctypes.c_void_p * max(1, T * M))()
        rows_p = (ctypes.c_void_p * max(1, T * M))()
        n_arr = np.zeros(max(1, T * M), dtype=np.int64)
        for t in range(T):
            d = self.specs[t].dim
            for m, msg in enumerate(batch):
                ids = np.ascontiguousarray(np.asarray(msg.ids[t], dtype=np.int64))
                rows = np.ascontiguousarray(np.asarray(msg.rows[t], dtype=np.float32))
                assert rows.size == ids.size * d
                keep += [ids, rows]
                ids_p[t * M + m] = ids.ctypes.data
                rows_p[t * M + m] = rows.ctypes.data
                n_arr[t * M + m] = ids.size
        dense_p = (ctypes.c_void_p * max(1, M))()
        for m, msg in enumerate(batch):
            g = np.ascontiguousarray(np.asarray(msg.dense, dtype=np.float32))
            assert g.size == self.D
            keep.append(g)
            dense_p[m] = g.ctypes.data
        keep_out = np.zeros(max(1, M), dtype=np.int32)
        counts = [np.zeros(len(ts.track), np.int64) for ts in self.tables]
        kept = [np.zeros(len(ts.track), np.int64) for ts in self.tables]
        cnt_p = (ctypes.c_void_p * max(1, T))(*[c.ctypes.data for c in counts])
        kept_p = (ctypes.c_void_p * max(1, T))(*[c.ctypes.data for c in kept])
        st = Stats()
        rc = self.L.gbao_step(self.k, ctypes.byref(self.rule), M, _iptr(tokens), T,
                             self._c_tables, ids_p, _iptr(n_arr), rows_p,
                             ctypes.byref(self.dense.c), dense_p,
                             keep_out.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)), cnt_p,
                             kept_p, ctypes.byref(st))
        if rc != 0:
            raise ValueError("id out of range (id_mode 0) or the reserved id INT64_MIN (id_mode 2)")
        self.k += 1
        self.last_keep = keep_out[:M].copy()
        self.last_count = counts
        self.last_kept = kept
        self.last_stats = st.as_dict()
