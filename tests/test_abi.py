"""The C-ABI library loads and exports every symbol include/gba.h declares, and
rejects bad arguments before touching a GPU (no compute calls here)."""
import ctypes
import subprocess

import pytest

from paper_2205_11048_gb300 import binding as B


@pytest.fixture(scope="module")
def L():
    import __graft_entry__
    __graft_entry__.build()
    return B.load()


def test_exports_every_declared_symbol(L):
    declared = B.header_functions()
    assert len(declared) >= 15
    out = subprocess.run(["nm", "-D", "--defined-only", B.LIB_PATH], capture_output=True,
                         text=True, check=True).stdout
    exported = {ln.split()[-1] for ln in out.splitlines() if " T " in ln}
    missing = [f for f in declared if f not in exported]
    assert not missing, missing
    for f in declared:
        assert hasattr(L, f)
    # every declared function has a binding signature
    assert set(declared) <= set(B._SIGNATURES)


def test_library_is_built_for_sm103a_only():
    """Every translation unit and the link are compiled for sm_103a and nothing else."""
    from paper_2205_11048_gb300 import build as BLD
    assert BLD.ARCH == ["-gencode", "arch=compute_103a,code=sm_103a"]


def test_no_device_code_without_a_gpu(L):
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present (the GPU test checks the version)")
    assert L.gba_device_binary_version() == B.GBA_E_CUDA


def _table(rows=100, dim=16, mode=0, mx=10, kind=0, init=0.1):
    return B.gba_table_desc(rows, dim, mode, mx, B.opt_desc(kind, 0.01, init))


def _create(L, tables, D=8, G=4, max_buf=4, st=None, dense_opt=None):
    h = ctypes.c_void_p()
    arr = (B.gba_table_desc * max(1, len(tables)))(*tables)
    dopt = dense_opt if dense_opt is not None else B.opt_desc()
    return L.gba_create(arr, len(tables), D, ctypes.byref(dopt) if D else None, G, max_buf,
                        ctypes.byref(st) if st else None, 0, None, ctypes.byref(h)), h


@pytest.mark.parametrize("bad", [
    dict(tables=[_table(rows=0)]), dict(tables=[_table(dim=0)]), dict(tables=[_table(dim=257)]),
    dict(tables=[_table(mode=3)]), dict(tables=[_table(mx=-1)]),
    dict(tables=[_table(mode=2, rows=2**30 + 1)]),
    dict(tables=[_table(kind=5)]), dict(tables=[_table(init=0.0)]),
    dict(tables=[_table(rows=2**31), _table(rows=2**31)]),
    dict(tables=[_table()], G=0), dict(tables=[_table()], max_buf=0),
    dict(tables=[_table()], D=-1),
    dict(tables=[_table()], st=B.gba_staleness_desc(-1, 0, 0)),
    dict(tables=[_table()], st=B.gba_staleness_desc(1, 2, 0)),
    dict(tables=[_table()], st=B.gba_staleness_desc(1, 0, 3)),
    dict(tables=[_table()], st=B.gba_staleness_desc(1, 0, 0, 2, 1.0, 0)),
    dict(tables=[_table()], st=B.gba_staleness_desc(1, 0, 0, 1, 0.0, 0)),
    dict(tables=[_table()], st=B.gba_staleness_desc(1, 0, 0, 1, 1.5, 0)),
    dict(tables=[_table()], st=B.gba_staleness_desc(1024, 0, 0, 1, 0.5, 0)),
    dict(tables=[_table()], st=B.gba_staleness_desc(1, 0, 0, 0, 1.0, -1)),
    dict(tables=[_table()], dense_opt=B.opt_desc(1, 0.01, 0.1, 1.0, 0.999, 1e-8)),
])
def test_create_rejects_bad_arguments(L, bad):
    st, h = _create(L, **bad)
    assert st == B.GBA_E_ARG
    assert not h.value


def test_null_handle_calls_are_safe(L):
    assert L.gba_try_apply(None) == B.GBA_E_ARG
    assert L.gba_pull_version(None) == -1
    assert L.gba_sync(None) == B.GBA_E_ARG
    assert L.gba_push(None, 0, None, None, 1) == B.GBA_E_ARG
    assert L.gba_stats(None, None) == B.GBA_E_ARG
    L.gba_destroy(None)
    assert L.gba_last_error(None) == b""
    assert L.gba_selftest_wait_timeout(-1, None) == B.GBA_E_ARG
    # every other entry point that takes a handle refuses a NULL one
    for call in (lambda: L.gba_push_ref(None, 0, None, None, 1),
                 lambda: L.gba_join(None), lambda: L.gba_set_overlap(None, 1),
                 lambda: L.gba_set_eager_dense(None, 1), lambda: L.gba_set_timing(None, 1),
                 lambda: L.gba_set_debug(None, 1), lambda: L.gba_kernel_times(None, None),
                 lambda: L.gba_get_table(None, 0, None, None, None, None),
                 lambda: L.gba_get_dense(None, None, None, None),
                 lambda: L.gba_table_capacity(None, 0, None),
                 lambda: L.gba_lookup_rows(None, 0, None, 0, None),
                 lambda: L.gba_pull(None, 0, None, 0, None),
                 lambda: L.gba_debug_segments(None, 0, None, None, None, None, None),
                 lambda: L.gba_debug_sorted(None, 0, None, None, None),
                 lambda: L.gba_debug_keep(None, 0, None, None),
                 lambda: L.gba_debug_set_wait_limit(None, 0),
                 lambda: L.gba_debug_withhold_dense_copies(None, 1)):
        assert call() == B.GBA_E_ARG


def test_create_without_gpu_fails_cleanly(L):
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    st, h = _create(L, [_table()])
    assert st in (B.GBA_E_CUDA, B.GBA_E_OOM)
    assert not h.value
