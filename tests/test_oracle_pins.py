"""The CPU oracle against what the paper and mathematics fix (no GPU)."""
import numpy as np
import pytest

from oracle import oracle as O
from tests import _pins


@pytest.fixture(scope="module")
def L():
    return O.lib()


@pytest.mark.parametrize("pin", _pins.ALL_PINS, ids=lambda p: p.__name__)
def test_pin(pin, L):
    pin(L)


def test_splitmix64_published_outputs():
    g = _pins.load_golden()["splitmix64_seed0"]
    gamma = 0x9E3779B97F4A7C15
    for i, want in enumerate(g["outputs"]):
        # output i of the generator started at state 0 is the hash of state i * gamma
        assert O.splitmix64((i * gamma) % 2**64) == int(want, 16)


def test_init_weights_exact_and_in_range():
    vals = np.array([O.init_weight(1234, O.table_tag(t), e) for t in range(3) for e in range(4000)])
    assert np.all(vals >= -1 / 16) and np.all(vals < 1 / 16)
    # exact multiples of 2^-27 (24-bit integers scaled by a power of two)
    q = vals * 2**27
    assert np.all(q == np.round(q))
    # roughly uniform: mean near 0, variance near (1/8)^2 / 12
    assert abs(vals.mean()) < 2e-3
    assert abs(vals.var() - (1 / 8) ** 2 / 12) < 2e-4
    # distinct arrays get distinct streams
    assert O.init_weight(1, O.table_tag(0), 5) != O.init_weight(1, O.table_tag(1), 5)
    assert O.init_weight(1, O.dense_tag(), 5) != O.init_weight(1, O.table_tag(0), 5)


def test_select_prefix():
    assert O.select_prefix([], 4) == 0
    assert O.select_prefix([1, 1, 1], 4) == 0
    assert O.select_prefix([1, 1, 2, 9], 4) == 3
    assert O.select_prefix([5, 1], 4) == 1
    assert O.select_prefix([256] * 4, 1024) == 4


def test_id_out_of_range_is_an_error():
    tb = O.TableSpec(4, 1)
    orc = O.OracleGBA([tb], 1, O.OptSpec(), 1)
    orc.push(O.Message(0, 1, [np.array([4], np.int64)], [np.ones((1, 1), np.float32)],
                       np.ones(1, np.float32)))
    with pytest.raises(ValueError):
        orc.try_apply()


def test_modulo_ids_and_tracking_subset():
    """MODULO ids map by uint64 residue (negative ids included), and a tracked
    subset of rows evolves exactly as the same rows of the full table."""
    rng = np.random.default_rng(5)
    V, d, D, M = 13, 2, 3, 3
    msgs = []
    for s in range(3):
        batch = []
        for m in range(M):
            ids = rng.integers(-2**62, 2**62, size=7).astype(np.int64)
            batch.append(O.Message(s, 1, [ids], [(rng.standard_normal((7, d)) * .1).astype(np.float32)],
                                   (rng.standard_normal(D)).astype(np.float32)))
        msgs.append(batch)
    spec = O.TableSpec(V, d, O.OptSpec(O.ADAM, 0.01), id_mode=1)
    full = O.OracleGBA([spec], D, O.OptSpec(), M, iota=0, seed=3)
    sub_rows = np.array([1, 4, 12], np.int64)
    sub = O.OracleGBA([spec], D, O.OptSpec(), M, iota=0, seed=3, track_rows=[sub_rows],
                      track_dense=np.array([2], np.int64))
    for batch in msgs:
        for m in batch:
            full.push(m)
            sub.push(m)
        full.try_apply()
        sub.try_apply()
    fw = full.tables[0].w.reshape(V, d)[sub_rows]
    assert np.array_equal(fw, sub.tables[0].w.reshape(-1, d))
    assert np.array_equal(full.tables[0].ver[sub_rows], sub.tables[0].ver)
    assert full.dense.w[2] == sub.dense.w[0]
    # the residue is taken on the unsigned 64-bit value
    ids = np.concatenate([m.ids[0] for m in msgs[0]])
    rows = (ids.view(np.uint64) % np.uint64(V)).astype(np.int64)
    touched = np.unique(rows)
    full2 = O.OracleGBA([spec], D, O.OptSpec(), M, iota=0, seed=3)
    for m in msgs[0]:
        full2.push(m)
    full2.try_apply()
    assert np.nonzero(full2.last_count[0])[0].tolist() == touched.tolist()
