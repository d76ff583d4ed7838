"""The token list (Sec. 4.1; Alg. 2 token generation and pull responding
threads) through the C ABI; it needs no GPU.

The paper fixes: token values start at zero and each value repeats M times,
so the i-th token handed out is floor(i / M) (the sentence of Sec. 4.1; the
formula printed after it, floor(i / K) with K = ceil(Q / M), repeats values K
times and is taken as garbled); the queue is refilled under a lock whenever it
holds fewer tokens than there are workers."""
import threading

import pytest

from paper_2205_11048_gb300 import binding as B


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


@pytest.mark.parametrize("M,workers", [(1, 1), (4, 4), (32, 40), (128, 100), (3, 7)])
def test_ith_token_is_i_div_m(M, workers):
    tl = B.TokenList(M, workers)
    got = [tl.fetch() for _ in range(5 * M + 3)]
    assert got == [i // M for i in range(5 * M + 3)]
    # ascending, each value exactly M times
    for v in range(5):
        assert got.count(v) == M
    # after every fetch the refill has topped the queue up to one token per worker
    assert tl.state() == (workers, 5 * M + 3)
    tl.close()


def test_bad_arguments():
    L = B.load()
    h = B._P()
    assert L.gba_token_list_create(0, 4, B.ctypes.byref(h)) == B.GBA_E_ARG
    assert L.gba_token_list_create(4, 0, B.ctypes.byref(h)) == B.GBA_E_ARG
    assert L.gba_token_list_create(4, 4, None) == B.GBA_E_ARG
    assert L.gba_fetch_token(None, None) == B.GBA_E_ARG
    L.gba_token_list_destroy(None)


def test_concurrent_fetches_hand_out_each_index_once():
    """Pull responding threads fetch concurrently: together they receive exactly
    the tokens floor(i / M) for i = 0 .. n-1, each thread in ascending order."""
    M, workers, threads, each = 16, 24, 8, 500
    tl = B.TokenList(M, workers)
    out = [[] for _ in range(threads)]

    def run(j):
        for _ in range(each):
            out[j].append(tl.fetch())

    ts = [threading.Thread(target=run, args=(j,)) for j in range(threads)]
    for t in ts:
        t.start()
    for t in ts:
        t.join()
    allv = sorted(v for o in out for v in o)
    assert allv == [i // M for i in range(threads * each)]
    for o in out:
        assert o == sorted(o)
    tl.close()
