"""ctypes binding of libgba (include/gba.h): the same entry points, argument
marshalling only.  Every step of the aggregate-and-apply path runs in the
library's CUDA kernels; there is no Python or CPU fallback, and loading fails
loudly when the library has not been built.

``GBA`` is a small convenience wrapper that passes torch tensors' device
pointers; torch is only used for device memory and streams.
"""
from __future__ import annotations

import ctypes
import os
import re

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libgba.so")
HEADER = os.path.join(os.path.dirname(_HERE), "include", "gba.h")

GBA_OK = 0
GBA_E_ARG = -1
GBA_E_ID_RANGE = -2
GBA_E_OOM = -3
GBA_E_CUDA = -4
GBA_E_DEVICE_TIMEOUT = -5
GBA_E_STATE = -6
GBA_E_FULL = -7
STATUS_NAMES = {0: "GBA_OK", -1: "GBA_E_ARG", -2: "GBA_E_ID_RANGE", -3: "GBA_E_OOM",
                -4: "GBA_E_CUDA", -5: "GBA_E_DEVICE_TIMEOUT", -6: "GBA_E_STATE",
                -7: "GBA_E_FULL"}
ADAGRAD, ADAM = 0, 1
DIRECT, MODULO, HASH = 0, 1, 2
INT32_MAX = 2**31 - 1
KERNEL_NAMES = ["weights", "sort_hist", "sort_pass", "seg_scan", "row_long", "row_apply",
                "dense", "init", "other"]


class GBAError(RuntimeError):
    def __init__(self, status, msg=""):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {msg}")
        self.status = status


class gba_opt_desc(ctypes.Structure):
    _fields_ = [("kind", ctypes.c_int32), ("lr", ctypes.c_float),
                ("adagrad_init_acc", ctypes.c_float), ("beta1", ctypes.c_float),
                ("beta2", ctypes.c_float), ("eps", ctypes.c_float)]


class gba_table_desc(ctypes.Structure):
    _fields_ = [("rows", ctypes.c_int64), ("dim", ctypes.c_int32), ("id_mode", ctypes.c_int32),
                ("max_ids_per_msg", ctypes.c_int64), ("opt", gba_opt_desc)]


class gba_staleness_desc(ctypes.Structure):
    _fields_ = [("iota", ctypes.c_int32), ("row_staleness", ctypes.c_int32),
                ("sparse_denominator", ctypes.c_int32), ("decay", ctypes.c_int32),
                ("lambda_", ctypes.c_float), ("drop_latest", ctypes.c_int32)]


class gba_sparse_grad(ctypes.Structure):
    _fields_ = [("ids", ctypes.c_void_p), ("n", ctypes.c_int64), ("rows", ctypes.c_void_p)]


class gba_stats_t(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int64) for n in (
        "steps", "msgs_kept", "msgs_dropped", "dense_stale_sum", "dense_stale_max", "pairs",
        "pairs_dropped", "row_stale_sum", "row_stale_max", "occurrences", "rows_touched",
        "rows_applied", "occurrences_kept")]

    def as_dict(self):
        return {n: int(getattr(self, n)) for n, _ in self._fields_}


class gba_kernel_times_t(ctypes.Structure):
    _fields_ = [("launches", ctypes.c_int64 * len(KERNEL_NAMES)),
                ("ms", ctypes.c_double * len(KERNEL_NAMES))]


_P = ctypes.c_void_p
_SIGNATURES = {
    "gba_create": (ctypes.c_int, [ctypes.POINTER(gba_table_desc), ctypes.c_int32, ctypes.c_int64,
                                  ctypes.POINTER(gba_opt_desc), ctypes.c_int64, ctypes.c_int32,
                                  ctypes.POINTER(gba_staleness_desc), ctypes.c_uint64, _P,
                                  ctypes.POINTER(_P)]),
    "gba_push": (ctypes.c_int, [_P, ctypes.c_int64, ctypes.POINTER(gba_sparse_grad), _P,
                                ctypes.c_int32]),
    "gba_push_ref": (ctypes.c_int, [_P, ctypes.c_int64, ctypes.POINTER(gba_sparse_grad), _P,
                                    ctypes.c_int32]),
    "gba_try_apply": (ctypes.c_int32, [_P]),
    "gba_pull_version": (ctypes.c_int64, [_P]),
    "gba_sync": (ctypes.c_int, [_P]),
    "gba_get_table": (ctypes.c_int, [_P, ctypes.c_int32, ctypes.POINTER(_P), ctypes.POINTER(_P),
                                     ctypes.POINTER(_P), ctypes.POINTER(_P)]),
    "gba_get_dense": (ctypes.c_int, [_P, ctypes.POINTER(_P), ctypes.POINTER(_P),
                                     ctypes.POINTER(_P)]),
    "gba_stats": (ctypes.c_int, [_P, ctypes.POINTER(gba_stats_t)]),
    "gba_last_error": (ctypes.c_char_p, [_P]),
    "gba_destroy": (None, [_P]),
    "gba_set_timing": (ctypes.c_int, [_P, ctypes.c_int32]),
    "gba_kernel_times": (ctypes.c_int, [_P, ctypes.POINTER(gba_kernel_times_t)]),
    "gba_set_debug": (ctypes.c_int, [_P, ctypes.c_int32]),
    "gba_set_overlap": (ctypes.c_int, [_P, ctypes.c_int32]),
    "gba_join": (ctypes.c_int, [_P]),
    "gba_set_eager_dense": (ctypes.c_int, [_P, ctypes.c_int32]),
    "gba_table_capacity": (ctypes.c_int, [_P, ctypes.c_int32, ctypes.POINTER(ctypes.c_int64)]),
    "gba_lookup_rows": (ctypes.c_int, [_P, ctypes.c_int32, _P, ctypes.c_int64, _P]),
    "gba_pull": (ctypes.c_int, [_P, ctypes.c_int32, _P, ctypes.c_int64, _P]),
    "gba_token_list_create": (ctypes.c_int, [ctypes.c_int64, ctypes.c_int32, ctypes.POINTER(_P)]),
    "gba_fetch_token": (ctypes.c_int, [_P, ctypes.POINTER(ctypes.c_int64)]),
    "gba_token_list_state": (ctypes.c_int, [_P, ctypes.POINTER(ctypes.c_int64),
                                            ctypes.POINTER(ctypes.c_int64)]),
    "gba_token_list_destroy": (None, [_P]),
    "gba_debug_segments": (ctypes.c_int, [_P, ctypes.c_int64, _P, _P, _P, _P,
                                          ctypes.POINTER(ctypes.c_int64)]),
    "gba_debug_sorted": (ctypes.c_int, [_P, ctypes.c_int64, _P, _P,
                                        ctypes.POINTER(ctypes.c_int64)]),
    "gba_debug_keep": (ctypes.c_int, [_P, ctypes.c_int32, _P, ctypes.POINTER(ctypes.c_int32)]),
    "gba_debug_set_wait_limit": (ctypes.c_int, [_P, ctypes.c_int64]),
    "gba_debug_withhold_dense_copies": (ctypes.c_int, [_P, ctypes.c_int32]),
    "gba_selftest_wait_timeout": (ctypes.c_int, [ctypes.c_int64, _P]),
    "gba_version_string": (ctypes.c_char_p, []),
    "gba_device_binary_version": (ctypes.c_int32, []),
    "gba_sort_ids_static": (ctypes.c_int, [_P, ctypes.c_int64, ctypes.c_int64, ctypes.c_int32,
                                           _P, _P, _P]),
}

_lib = None


def header_functions(path: str = HEADER):
    """Names of the functions include/gba.h declares."""
    text = open(path).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(gba_[a-z_0-9]+)\s*\(", text)))


def load(path: str = LIB_PATH):
    """Load libgba.so and declare its signatures (raises if it is missing)."""
    global _lib
    if _lib is not None and path == LIB_PATH:
        return _lib
    if not os.path.exists(path):
        raise ImportError(f"libgba.so not built: {path} (run __graft_entry__.build())")
    L = ctypes.CDLL(path)
    for name, (res, args) in _SIGNATURES.items():
        fn = getattr(L, name)
        fn.restype = res
        fn.argtypes = args
    if path == LIB_PATH:
        _lib = L
    return L


def check(status, h=None, what=""):
    if status < 0:
        msg = what
        if h:
            msg += " " + (load().gba_last_error(h) or b"").decode()
        raise GBAError(status, msg)
    return status


# ---- thin functional wrappers with the ABI's names ------------------------------------

def gba_create(tables, dense_size, dense_opt, global_batch, max_buffered_msgs, staleness,
               init_seed, cuda_stream=None):
    L = load()
    arr = (gba_table_desc * max(1, len(tables)))(*tables)
    h = _P()
    st = check(L.gba_create(arr, len(tables), dense_size,
                            ctypes.byref(dense_opt) if dense_opt is not None else None,
                            global_batch, max_buffered_msgs,
                            ctypes.byref(staleness) if staleness is not None else None,
                            init_seed & (2**64 - 1), cuda_stream, ctypes.byref(h)),
               what="gba_create")
    return h, st


def gba_push(h, token, per_table, dense_grad, local_batch):
    arr = (gba_sparse_grad * max(1, len(per_table)))(*per_table)
    return load().gba_push(h, token, arr, dense_grad, local_batch)


def gba_push_ref(h, token, per_table, dense_grad, local_batch):
    arr = (gba_sparse_grad * max(1, len(per_table)))(*per_table)
    return load().gba_push_ref(h, token, arr, dense_grad, local_batch)


def gba_try_apply(h):
    return load().gba_try_apply(h)


def gba_pull_version(h):
    return load().gba_pull_version(h)


def gba_sync(h):
    return load().gba_sync(h)


def gba_destroy(h):
    load().gba_destroy(h)


# ---- convenience wrapper over torch tensors --------------------------------------------

def opt_desc(kind=ADAGRAD, lr=0.01, init_acc=0.1, beta1=0.9, beta2=0.999, eps=1e-8):
    return gba_opt_desc(kind, lr, init_acc, beta1, beta2, eps)


def gba_for_workload(cfg, max_buf=None, seed=None, overlap=False, **rule):
    """A handle sized for a workload description (a `workload.WorkloadCfg`:
    tables, dense size, optimizers, global batch, tolerance iota), with room
    for max_buf buffered messages (default two global batches)."""
    def od(o):
        return opt_desc(o.kind, o.lr, o.init_acc, o.beta1, o.beta2, o.eps)
    tables = [(tb.rows, tb.dim, tb.id_mode, cfg.max_ids_per_msg(t), od(tb.opt))
              for t, tb in enumerate(cfg.tables)]
    rule = rule or dict(iota=cfg.iota)
    g = GBA(tables, cfg.D, od(cfg.dense_opt), cfg.G, max_buf or 2 * cfg.M,
            seed=cfg.seed if seed is None else seed, **rule)
    if overlap:
        g.set_overlap(True)
    return g


class GBA:
    """One parameter-server state on the current CUDA device."""

    def __init__(self, tables, dense_size, dense_opt, global_batch, max_buffered_msgs,
                 iota=INT32_MAX, row_staleness=0, sparse_denominator=0, seed=0, stream=None,
                 decay=0, lam=1.0, drop_latest=0):
        """tables: list of (rows, dim, id_mode, max_ids_per_msg, gba_opt_desc)."""
        import torch
        self.torch = torch
        self.L = load()
        self.dims = [int(t[1]) for t in tables]
        self.rows = [int(t[0]) for t in tables]
        self.opts = [t[4] for t in tables]
        self.D = int(dense_size)
        self.dense_opt = dense_opt
        descs = [gba_table_desc(int(r), int(d), int(m), int(mx), o) for (r, d, m, mx, o) in tables]
        st = gba_staleness_desc(int(iota), int(row_staleness), int(sparse_denominator),
                                int(decay), float(lam), int(drop_latest))
        if stream is None:
            stream = torch.cuda.current_stream()
        self.stream = stream
        self.h, _ = gba_create(descs, self.D, dense_opt, int(global_batch),
                               int(max_buffered_msgs), st, int(seed),
                               ctypes.c_void_p(stream.cuda_stream))
        self._keep = []  # tensors referenced by pushed-by-reference messages

    def close(self):
        if self.h:
            self.L.gba_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def _grads(self, ids, rows):
        out = []
        for t in range(len(self.dims)):
            i, r = ids[t], rows[t]
            n = int(i.numel())
            out.append(gba_sparse_grad(i.data_ptr() if n else None, n,
                                       r.data_ptr() if n else None))
        return out

    def push(self, token, ids, rows, dense, local_batch):
        """Copying push; tensors may live on the device or in (pinned) host memory."""
        return check(gba_push(self.h, int(token), self._grads(ids, rows),
                              dense.data_ptr() if self.D else None, int(local_batch)),
                     self.h, "gba_push")

    def push_ref(self, token, ids, rows, dense, local_batch):
        """Push by reference (device tensors that stay valid until applied)."""
        return check(gba_push_ref(self.h, int(token), self._grads(ids, rows),
                                  dense.data_ptr() if self.D else None, int(local_batch)),
                     self.h, "gba_push_ref")

    def try_apply(self):
        return check(gba_try_apply(self.h), self.h, "gba_try_apply")

    def version(self):
        return int(gba_pull_version(self.h))

    def sync(self):
        return check(gba_sync(self.h), self.h, "gba_sync")

    def table(self, t):
        """Copies (on the device) of table t: w [rows, dim], slot0, slot1, ver."""
        w, s0, s1, v = _P(), _P(), _P(), _P()
        check(self.L.gba_get_table(self.h, t, ctypes.byref(w), ctypes.byref(s0),
                                   ctypes.byref(s1), ctypes.byref(v)), self.h)
        rows = self.capacity(t)
        n = rows * self.dims[t]
        torch = self.torch
        self.sync()
        out = []
        for p, cnt, dt in ((w, n, torch.float32), (s0, n, torch.float32), (s1, n, torch.float32),
                           (v, rows, torch.int32)):
            out.append(None if not p.value else _copy_device(p.value, cnt, dt))
        out[0] = out[0].view(rows, self.dims[t])
        out[1] = out[1].view(rows, self.dims[t])
        if out[2] is not None:
            out[2] = out[2].view(rows, self.dims[t])
        return out

    def table_rows(self, t, rows):
        """w, slot0, slot1, ver of selected rows of table t (device tensors)."""
        w, s0, s1, v = _P(), _P(), _P(), _P()
        check(self.L.gba_get_table(self.h, t, ctypes.byref(w), ctypes.byref(s0),
                                   ctypes.byref(s1), ctypes.byref(v)), self.h)
        self.sync()
        torch = self.torch
        d = self.dims[t]
        cap = self.capacity(t)
        idx = torch.as_tensor(rows, dtype=torch.int64, device="cuda")
        res = []
        for p in (w, s0, s1):
            if not p.value:
                res.append(None)
                continue
            res.append(_gather_rows(p.value, cap, d, idx))
        res.append(_gather_rows(v.value, cap, 1, idx, torch.int32).view(-1))
        return res

    def dense(self):
        w, s0, s1 = _P(), _P(), _P()
        check(self.L.gba_get_dense(self.h, ctypes.byref(w), ctypes.byref(s0), ctypes.byref(s1)),
              self.h)
        self.sync()
        torch = self.torch
        return [None if not p.value else _copy_device(p.value, self.D, torch.float32)
                for p in (w, s0, s1)]

    def stats(self):
        s = gba_stats_t()
        check(self.L.gba_stats(self.h, ctypes.byref(s)), self.h)
        return s.as_dict()

    def pull(self, t, ids):
        """Current rows of table t for the device int64 tensor ids (pull responding)."""
        torch = self.torch
        ids = ids.contiguous()
        out = torch.empty(ids.numel(), self.dims[t], dtype=torch.float32, device=ids.device)
        check(self.L.gba_pull(self.h, int(t), ids.data_ptr() if ids.numel() else None,
                              ids.numel(), out.data_ptr() if ids.numel() else None),
              self.h, "gba_pull")
        return out

    def capacity(self, t):
        """Rows the arrays of table t hold now (slots of a HASH table)."""
        r = ctypes.c_int64()
        check(self.L.gba_table_capacity(self.h, int(t), ctypes.byref(r)), self.h)
        return int(r.value)

    def lookup(self, t, ids):
        """Slots of the device int64 tensor ids in HASH table t (-1: absent)."""
        torch = self.torch
        ids = ids.contiguous()
        out = torch.empty(ids.numel(), dtype=torch.int64, device=ids.device)
        if ids.numel():
            check(self.L.gba_lookup_rows(self.h, int(t), ids.data_ptr(), ids.numel(),
                                         out.data_ptr()), self.h, "gba_lookup_rows")
        return out

    def set_eager_dense(self, on=True):
        check(self.L.gba_set_eager_dense(self.h, int(on)), self.h, "gba_set_eager_dense")

    def join(self):
        """Order the handle's stream after every step enqueued so far."""
        check(self.L.gba_join(self.h), self.h, "gba_join")

    def set_overlap(self, on=True):
        check(self.L.gba_set_overlap(self.h, int(on)), self.h)

    def set_debug(self, on=True):
        check(self.L.gba_set_debug(self.h, int(on)), self.h)

    def set_timing(self, on=True):
        check(self.L.gba_set_timing(self.h, int(on)), self.h)

    def kernel_times(self):
        kt = gba_kernel_times_t()
        check(self.L.gba_kernel_times(self.h, ctypes.byref(kt)), self.h)
        return {KERNEL_NAMES[i]: (int(kt.launches[i]), float(kt.ms[i])) for i in range(len(KERNEL_NAMES))}

    def set_wait_limit(self, ns):
        check(self.L.gba_debug_set_wait_limit(self.h, int(ns)), self.h)

    def withhold_dense_copies(self, on=True):
        check(self.L.gba_debug_withhold_dense_copies(self.h, 1 if on else 0), self.h)

    def segments(self, cap=None):
        """Dedup output of the last step: (table, row, count, kept) numpy arrays."""
        import numpy as np
        n = ctypes.c_int64()
        if cap is None:
            self.L.gba_debug_segments(self.h, 0, None, None, None, None, ctypes.byref(n))
            cap = int(n.value)
        t = np.zeros(cap, np.int32)
        r = np.zeros(cap, np.int64)
        c = np.zeros(cap, np.int64)
        k = np.zeros(cap, np.int64)
        check(self.L.gba_debug_segments(self.h, cap, t.ctypes.data, r.ctypes.data, c.ctypes.data,
                                        k.ctypes.data, ctypes.byref(n)), self.h)
        u = int(n.value)
        return t[:u], r[:u], c[:u], k[:u]

    def sorted_keys(self):
        import numpy as np
        n = ctypes.c_int64()
        self.L.gba_debug_sorted(self.h, 0, None, None, ctypes.byref(n))
        cap = int(n.value)
        keys = np.zeros(cap, np.uint32)
        occ = np.zeros(cap, np.uint32)
        check(self.L.gba_debug_sorted(self.h, cap, keys.ctypes.data, occ.ctypes.data,
                                      ctypes.byref(n)), self.h)
        return keys, occ

    def keep(self, cap=4096):
        import numpy as np
        out = np.zeros(cap, np.int32)
        M = ctypes.c_int32()
        check(self.L.gba_debug_keep(self.h, cap, out.ctypes.data, ctypes.byref(M)), self.h)
        return out[:M.value]


class _DevArray:
    """Minimal __cuda_array_interface__ over library-owned device memory."""

    def __init__(self, ptr, nbytes):
        self.__cuda_array_interface__ = {"shape": (nbytes,), "typestr": "|u1",
                                         "data": (ptr, False), "version": 3}


def _copy_device(ptr, n, dtype):
    import torch
    elem = torch.empty((), dtype=dtype).element_size()
    raw = torch.as_tensor(_DevArray(ptr, n * elem), device="cuda")
    return raw.view(dtype).clone()


def _gather_rows(ptr, rows, d, idx, dtype=None):
    import torch
    dtype = dtype or torch.float32
    elem = torch.empty((), dtype=dtype).element_size()
    raw = torch.as_tensor(_DevArray(ptr, rows * d * elem), device="cuda").view(dtype)
    return raw.view(rows, d).index_select(0, idx).clone()


class TokenList:
    """The token list of Sec. 4.1 / Alg. 2 (see gba_token_list_create)."""

    def __init__(self, repeats, workers):
        self.L = load()
        self.h = _P()
        check(self.L.gba_token_list_create(int(repeats), int(workers), ctypes.byref(self.h)),
              what="gba_token_list_create")

    def fetch(self):
        t = ctypes.c_int64()
        check(self.L.gba_fetch_token(self.h, ctypes.byref(t)), what="gba_fetch_token")
        return int(t.value)

    def state(self):
        q, f = ctypes.c_int64(), ctypes.c_int64()
        check(self.L.gba_token_list_state(self.h, ctypes.byref(q), ctypes.byref(f)))
        return int(q.value), int(f.value)

    def close(self):
        if self.h:
            self.L.gba_token_list_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
