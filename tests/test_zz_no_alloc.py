"""The allocation-free sort entry point, through the C ABI (needs a GPU).

gba_sort_ids_static serves callers that must not allocate device memory when
they need a sort: a runtime that reserved all device memory up front, or an
allocator's own hook, which cannot call back into cudaMalloc.  It must give
exactly what the library's regular path gives for the same ids: the stable
radix sort that gba_try_apply performs, read back with gba_debug_sorted.  Two
calls in a row share the fixed scratch array, so the second call also checks
that stale contents of the first do not leak into its result.

This file is collected last so that a run stopping at the first failure has
run every other test first."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2205_11048_gb300 import binding as B

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def L():
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(0)
    return B.load()


def regular_path_sort(ids, rows, id_mode):
    """Sorted rows and input order from the regular step (gba_try_apply)."""
    n = ids.numel()
    tables = [(rows, 4, id_mode, n, B.opt_desc())]
    g = B.GBA(tables, 0, None, 1, 2, seed=0)
    grads = torch.zeros(n, 4, device="cuda")
    g.push_ref(0, [ids], [grads], torch.zeros(0, device="cuda"), 1)
    assert g.try_apply() == 1
    keys, occ = g.sorted_keys()
    g.close()
    return keys, occ


def static_sort_rc(L, ids, rows, id_mode):
    n = ids.numel()
    out_rows = torch.empty(max(n, 1), dtype=torch.int32, device="cuda")
    out_order = torch.empty(max(n, 1), dtype=torch.int32, device="cuda")
    stream = torch.cuda.current_stream()
    rc = L.gba_sort_ids_static(ids.data_ptr(), n, rows, id_mode, out_rows.data_ptr(),
                               out_order.data_ptr(), ctypes.c_void_p(stream.cuda_stream))
    return rc, (out_rows[:n].cpu().numpy().view(np.uint32),
                out_order[:n].cpu().numpy().view(np.uint32))


def static_sort(L, ids, rows, id_mode):
    rc, out = static_sort_rc(L, ids, rows, id_mode)
    assert rc == B.GBA_OK, B.STATUS_NAMES.get(rc, rc)
    return out


def check_against_regular(L, ids, rows, mode):
    got_rows, got_order = static_sort(L, ids, rows, mode)
    want_rows, want_order = regular_path_sort(ids, rows, mode)
    assert np.array_equal(got_rows, want_rows)
    assert np.array_equal(got_order, want_order)
    assert np.all(np.diff(got_rows.astype(np.int64)) >= 0)


def test_two_calls_match_the_regular_path(L):
    gen = torch.Generator(device="cuda").manual_seed(11)
    # call 1: DIRECT ids with a hot set, several sort tiles and a ragged tail
    rows1 = 1_000_003
    hot = torch.randint(0, 50, (40_000,), generator=gen, device="cuda")
    cold = torch.randint(0, rows1, (260_001,), generator=gen, device="cuda")
    ids1 = torch.cat([cold[:100_000], hot, cold[100_000:]]).to(torch.int64)
    # call 2: hashed 64-bit ids (MODULO), fewer of them and fewer key bits
    rows2 = 40_009
    ids2 = torch.randint(-2**62, 2**62, (77_777,), generator=gen, device="cuda",
                         dtype=torch.int64)
    for ids, rows, mode in ((ids1, rows1, B.DIRECT), (ids2, rows2, B.MODULO)):
        check_against_regular(L, ids, rows, mode)


def test_id_out_of_range_then_a_good_call(L):
    """A DIRECT id outside [0, rows) is reported; the next call starts from
    cleared error words and sorts correctly."""
    gen = torch.Generator(device="cuda").manual_seed(3)
    ids = torch.randint(0, 5000, (10_000,), generator=gen, device="cuda", dtype=torch.int64)
    bad = ids.clone()
    bad[7_777] = 5000
    rc, _ = static_sort_rc(L, bad, 5000, B.DIRECT)
    assert rc == B.GBA_E_ID_RANGE
    bad[7_777] = -1
    rc, _ = static_sort_rc(L, bad, 5000, B.DIRECT)
    assert rc == B.GBA_E_ID_RANGE
    check_against_regular(L, ids, 5000, B.DIRECT)


@pytest.mark.parametrize("n", [1, 2047, 2049])
@pytest.mark.parametrize("rows", [1, (1 << 24) + 1])
def test_small_and_ragged_inputs(L, n, rows):
    """One id, one id short of a sort tile, one past it; a single row (one
    pass, all keys equal) and 25-bit keys (four passes)."""
    gen = torch.Generator(device="cuda").manual_seed(n + rows)
    ids = torch.randint(0, rows, (n,), generator=gen, device="cuda", dtype=torch.int64)
    check_against_regular(L, ids, rows, B.DIRECT)


def test_limits_are_refused(L):
    big = B.load().gba_sort_ids_static(None, (1 << 20) + 1, 10, 0, None, None, None)
    assert big == B.GBA_E_ARG
    assert L.gba_sort_ids_static(None, 0, 10, 0, None, None, None) == B.GBA_OK
    assert L.gba_sort_ids_static(None, 5, 0, 0, None, None, None) == B.GBA_E_ARG
