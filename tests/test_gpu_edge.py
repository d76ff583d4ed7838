"""Edge cases of the CUDA path against the CPU oracle, and its error handling
(needs a GPU).  No case here faults or hangs the device: bad ids are caught by
the kernels' own range checks, waits are bounded."""
import ctypes

import numpy as np
import pytest
import torch

from oracle import oracle as O
from paper_2205_11048_gb300 import binding as B
from paper_2205_11048_gb300 import workload as W
from tests import _harness as H

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(0)


def msg(token, ids_per_table, dims, D, B_=1, scale=0.01, gen=None, dtype_ids=torch.int64):
    gen = gen or torch.Generator(device="cuda").manual_seed(token * 7 + len(ids_per_table))
    ids = [torch.as_tensor(i, dtype=dtype_ids, device="cuda") for i in ids_per_table]
    rows = [torch.randn(i.numel(), d, generator=gen, device="cuda") * scale
            for i, d in zip(ids, dims)]
    dense = torch.randn(D, generator=gen, device="cuda") * scale
    return dict(token=token, local_batch=B_, ids=ids, rows=rows, dense=dense)


def cfg_of(tables, D, G, dense_kind=W.ADAM, iota=1):
    """tables: list of (rows, dim, id_mode, opt kind)."""
    tcs = tuple(W.TableCfg(r, d, 1, 0, 1.1, mode, W.OptCfg(kind, 0.01 if kind == 0 else 0.001))
                for (r, d, mode, kind) in tables)
    return W.WorkloadCfg("edge", M=G, B=1, tables=tcs, D=D,
                         dense_opt=W.OptCfg(dense_kind, 0.01 if dense_kind == 0 else 0.001),
                         stale=W.StaleCfg("fresh"), iota=iota, seed=3)


def run_custom(cfg, steps, rule=None, max_buf=64, max_ids=None, by_ref=False, tol=H.TOL_ONE_STEP):
    """steps: list of lists of message dicts; every step must trigger exactly once."""
    tables = [(tb.rows, tb.dim, tb.id_mode, max_ids or 4096, H.opt_desc(tb.opt))
              for tb in cfg.tables]
    rule = rule or dict(iota=cfg.iota)
    g = B.GBA(tables, cfg.D, H.opt_desc(cfg.dense_opt), cfg.G, max_buf, seed=cfg.seed, **rule)
    g.set_debug(True)
    orc = H.make_oracle(cfg, rule=rule)
    stats = {}
    for batch in steps:
        for m in batch:
            (g.push_ref if by_ref else g.push)(m["token"], m["ids"], m["rows"], m["dense"],
                                               m["local_batch"])
            orc.push(H.to_oracle(m))
        a, b = g.try_apply(), orc.try_apply()
        assert a == b == 1
        H.accumulate_stats(stats, orc.last_stats, orc)
        if cfg.tables:
            H.compare_segments(g, orc, True)
        H.compare_state(g, orc, tol)
    g.sync()
    H.compare_stats(g, stats)
    return g, orc


def test_hand_example_matches_golden_exactly():
    """The hand-worked golden example, through the CUDA path: exact values."""
    from tests import _pins
    gj = _pins.load_golden()["adagrad"]
    F = _pins.F
    lr, acc0 = F(gj["table"]["lr"]), F(gj["table"]["init_acc"])
    tables = [(4, 2, 0, 8, B.opt_desc(0, lr, acc0))]
    g = B.GBA(tables, 2, B.opt_desc(0, lr, acc0), 2, 8, iota=gj["iota"], seed=12345)
    w0 = g.table(0)[0].cpu().numpy().astype(np.float64)
    dw0 = g.dense()[0].cpu().numpy().astype(np.float64)
    for step in gj["steps"]:
        for m in step["messages"]:
            ids = torch.tensor(m["ids"], dtype=torch.int64, device="cuda")
            rows = torch.tensor(m["rows"], dtype=torch.float32, device="cuda")
            g.push(m["token"], [ids], [rows], torch.tensor(m["dense"], dtype=torch.float32,
                                                           device="cuda"), m["B"])
        assert g.try_apply() == 1
        e = step["expect"]
        assert g.keep().tolist() == e["keep"]
        w, s0, _, ver = g.table(0)
        for r in range(4):
            assert (w[r].cpu().numpy().astype(np.float64) - w0[r]).tolist() == \
                [F(v) for v in e["dw"][str(r)]]
            assert s0[r].cpu().numpy().astype(np.float64).tolist() == \
                [F(v) for v in e["acc"][str(r)]]
        assert ver.cpu().tolist() == e["ver"]
        dw, ds0, _ = g.dense()
        assert (dw.cpu().numpy().astype(np.float64) - dw0).tolist() == \
            [F(v) for v in e["dense_dw"]]
        assert ds0.cpu().numpy().astype(np.float64).tolist() == [F(v) for v in e["dense_acc"]]
    g.close()


@pytest.mark.parametrize("variant", [0, 1, 2])
def test_rule_option_goldens_exactly(variant):
    """The hand-worked steps of the optional readings (kept-message and M
    denominators, message staleness for rows), through the CUDA path."""
    from tests import _pins
    gj = _pins.load_golden()["rule_options"]
    var = gj["variants"][variant]
    F = _pins.F
    lr, acc0 = F(gj["table"]["lr"]), F(gj["table"]["init_acc"])
    tables = [(4, 2, 0, 8, B.opt_desc(0, lr, acc0))]
    g = B.GBA(tables, 2, B.opt_desc(0, lr, acc0), 2, 8, seed=4321, **var["rule"])
    w0 = g.table(0)[0].cpu().numpy().astype(np.float64)
    dw0 = g.dense()[0].cpu().numpy().astype(np.float64)
    for step in (gj["step0"], var["step1"]):
        for m in step["messages"]:
            ids = torch.tensor(m["ids"], dtype=torch.int64, device="cuda")
            rows = torch.tensor(m["rows"], dtype=torch.float32, device="cuda")
            g.push(m["token"], [ids], [rows], torch.tensor(m["dense"], dtype=torch.float32,
                                                           device="cuda"), m["B"])
        assert g.try_apply() == 1
        e = step["expect"]
        assert g.keep().tolist() == e["keep"]
        w, s0, _, ver = g.table(0)
        for r in range(4):
            assert (w[r].cpu().numpy().astype(np.float64) - w0[r]).tolist() == \
                [F(v) for v in e["dw"][str(r)]]
            assert s0[r].cpu().numpy().astype(np.float64).tolist() == \
                [F(v) for v in e["acc"][str(r)]]
        assert ver.cpu().tolist() == e["ver"]
        dw, ds0, _ = g.dense()
        assert (dw.cpu().numpy().astype(np.float64) - dw0).tolist() == \
            [F(v) for v in e["dense_dw"]]
        assert ds0.cpu().numpy().astype(np.float64).tolist() == [F(v) for v in e["dense_acc"]]
    g.close()


@pytest.mark.parametrize("name", ["geometric", "hop_bw"])
def test_decay_variant_goldens_exactly(name):
    """The hand-worked steps of geometric decay (lambda^s) and Hop-BW's ignored
    latest gradients, through the CUDA path: exact values."""
    from tests import _pins
    gj = _pins.load_golden()["decay_variants"]
    var = gj[name]
    F = _pins.F
    lr, acc0 = F(gj["table"]["lr"]), F(gj["table"]["init_acc"])
    tables = [(4, 2, 0, 8, B.opt_desc(0, lr, acc0))]
    g = B.GBA(tables, 2, B.opt_desc(0, lr, acc0), var["global_batch"], 8, seed=4321,
              **var["rule"])
    w0 = g.table(0)[0].cpu().numpy().astype(np.float64)
    dw0 = g.dense()[0].cpu().numpy().astype(np.float64)
    for step in var["steps"]:
        for m in step["messages"]:
            ids = torch.tensor(m["ids"], dtype=torch.int64, device="cuda")
            rows = torch.tensor(m["rows"], dtype=torch.float32, device="cuda")
            g.push(m["token"], [ids], [rows], torch.tensor(m["dense"], dtype=torch.float32,
                                                           device="cuda"), m["B"])
        assert g.try_apply() == 1
        e = step["expect"]
        assert g.keep().tolist() == e["keep"]
        w, s0, _, ver = g.table(0)
        for r in range(4):
            assert (w[r].cpu().numpy().astype(np.float64) - w0[r]).tolist() == \
                [F(v) for v in e["dw"][str(r)]]
            assert s0[r].cpu().numpy().astype(np.float64).tolist() == \
                [F(v) for v in e["acc"][str(r)]]
        assert ver.cpu().tolist() == e["ver"]
        dw, ds0, _ = g.dense()
        assert (dw.cpu().numpy().astype(np.float64) - dw0).tolist() == \
            [F(v) for v in e["dense_dw"]]
        assert ds0.cpu().numpy().astype(np.float64).tolist() == [F(v) for v in e["dense_acc"]]
    g.close()


@pytest.mark.parametrize("rule", [dict(iota=6, decay=1, lam=0.7),
                                  dict(iota=3, decay=1, lam=0.5, row_staleness=1),
                                  dict(iota=O.INT32_MAX, drop_latest=1),
                                  dict(iota=2, decay=1, lam=0.9, drop_latest=2,
                                       sparse_denominator=1)])
@pytest.mark.parametrize("kind", [0, 1])
def test_decay_variants_against_the_oracle(rule, kind):
    """Geometric decay and Hop-BW on a random stream with stale tokens, hot
    rows (long rows) and two row widths, Adagrad and Adam."""
    rng = np.random.default_rng(17 + kind)
    cfg = cfg_of([(500, 16, 0, kind), (300, 6, 0, kind)], D=1031, G=6, dense_kind=kind)
    steps = []
    for k in range(5):
        batch = []
        for m in range(6):
            n0 = int(rng.integers(0, 400))
            ids0 = np.concatenate([rng.zipf(1.4, n0) % 500, np.full(int(rng.integers(0, 90)), 7)])
            ids1 = rng.integers(0, 300, int(rng.integers(0, 50)))
            tok = max(0, k - int(rng.integers(0, 5)))
            batch.append(msg(tok, [ids0, ids1], [16, 6], 1031))
        steps.append(batch)
    run_custom(cfg, steps, rule=rule)


@pytest.mark.parametrize("dim", [1, 3, 4, 8, 19, 24, 64, 128, 200, 256])
@pytest.mark.parametrize("kind", [0, 1])
def test_row_widths_and_optimizers(dim, kind):
    rng = np.random.default_rng(dim * 10 + kind)
    cfg = cfg_of([(997, dim, 0, kind)], D=33, G=3, iota=1)
    steps = []
    for k in range(3):
        batch = []
        for m in range(3):
            n = int(rng.integers(0, 300))
            ids = rng.zipf(1.3, n) % 997
            tok = max(0, k - int(rng.integers(0, 3)))
            batch.append(msg(tok, [ids], [dim], 33))
        steps.append(batch)
    run_custom(cfg, steps)


def test_empty_messages_and_empty_steps():
    cfg = cfg_of([(50, 4, 0, 0), (30, 8, 0, 1)], D=5, G=3)
    steps = [
        [msg(0, [[], []], [4, 8], 5), msg(0, [[1, 2], []], [4, 8], 5), msg(0, [[], [7]], [4, 8], 5)],
        [msg(1, [[], []], [4, 8], 5)] * 3,            # no ids at all in the step
        [msg(2, [[3] * 500, []], [4, 8], 5), msg(2, [[], []], [4, 8], 5),
         msg(2, [[3], [29]], [4, 8], 5)],
    ]
    run_custom(cfg, steps)


def test_everything_dropped():
    """All messages beyond iota: dense still steps (Adam moments move), no row moves."""
    cfg = cfg_of([(40, 4, 0, 1)], D=9, G=2, iota=0)
    steps = [[msg(0, [[1, 2]], [4], 9), msg(0, [[2, 3]], [4], 9)],
             [msg(1, [[5]], [4], 9), msg(1, [[6]], [4], 9)],
             [msg(0, [[1, 7]], [4], 9), msg(0, [[2]], [4], 9)]]   # staleness 2 > 0
    g, orc = run_custom(cfg, steps)
    assert orc.last_keep.tolist() == [0, 0]


def test_single_message_steps_and_token_ahead():
    cfg = cfg_of([(20, 4, 0, 0)], D=4, G=1, iota=0)
    steps = [[msg(0, [[1]], [4], 4)], [msg(5, [[1, 1, 2]], [4], 4)], [msg(2, [[2]], [4], 4)]]
    run_custom(cfg, steps)


@pytest.mark.parametrize("rule", [dict(iota=1, row_staleness=1),
                                  dict(iota=1, sparse_denominator=1),
                                  dict(iota=1, sparse_denominator=2),
                                  dict(iota=O.INT32_MAX)])
def test_rule_options(rule):
    rng = np.random.default_rng(4)
    cfg = cfg_of([(300, 8, 0, 0)], D=17, G=4)
    steps = []
    for k in range(5):
        steps.append([msg(max(0, k - int(rng.integers(0, 4))), [rng.integers(0, 300, 50)], [8], 17)
                      for _ in range(4)])
    run_custom(cfg, steps, rule=rule)


def test_modulo_negative_ids():
    rng = np.random.default_rng(8)
    cfg = cfg_of([(1009, 16, 1, 0)], D=8, G=2)
    steps = [[msg(0, [rng.integers(-2**62, 2**62, 400)], [16], 8) for _ in range(2)]
             for _ in range(2)]
    run_custom(cfg, steps)


def test_varying_local_batches_overshoot():
    """Apply when the buffered local batches reach G; the shortest prefix is popped."""
    cfg = cfg_of([(64, 4, 0, 0)], D=4, G=10)
    a = [msg(0, [[1]], [4], 4, B_=3), msg(0, [[2]], [4], 4, B_=3), msg(0, [[1]], [4], 4, B_=5)]
    tables = [(64, 4, 0, 16, B.opt_desc())]
    g = B.GBA(tables, 4, B.opt_desc(1, 0.001), 10, 8, iota=1, seed=3)
    orc = H.make_oracle(cfg)
    for m in a[:2]:
        g.push(m["token"], m["ids"], m["rows"], m["dense"], m["local_batch"])
        orc.push(H.to_oracle(m))
    assert g.try_apply() == 0 and orc.try_apply() == 0
    extra = msg(0, [[9]], [4], 4, B_=7)
    for m in (a[2], extra):
        g.push(m["token"], m["ids"], m["rows"], m["dense"], m["local_batch"])
        orc.push(H.to_oracle(m))
    assert g.try_apply() == 1 and orc.try_apply() == 1
    H.compare_state(g, orc, H.TOL_ONE_STEP)
    assert g.try_apply() == 0 and orc.try_apply() == 0   # 7 < 10 buffered
    g.close()


def test_hot_row_spanning_many_warps():
    """One row with 200K occurrences in a step: its kept occurrences fill
    hundreds of chunks, summed by different warps and merged in chunk order by
    the warp that finishes the last one."""
    gen = torch.Generator(device="cuda").manual_seed(1)
    cfg = cfg_of([(5000, 16, 0, 1)], D=4, G=4, iota=2)
    steps = []
    for k in range(2):
        batch = []
        for m in range(4):
            hot = torch.full((50_000,), 17, dtype=torch.int64, device="cuda")
            cold = torch.randint(0, 5000, (3000,), generator=gen, device="cuda")
            ids = torch.cat([hot[:25_000], cold, hot[25_000:]])
            batch.append(msg(max(0, k - m % 3), [ids.cpu().numpy()], [16], 4))
        steps.append(batch)
    run_custom(cfg, steps, max_ids=60_000)


@pytest.mark.parametrize("dim", [64, 12, 14])  # 14: the register path (not a multiple of 4)
@pytest.mark.parametrize("rule", [None, dict(iota=2, decay=1, lam=0.5)])
def test_kept_count_boundaries_of_the_row_kernels(dim, rule):
    """Rows whose kept occurrences sit on each side of the row kernels' limits
    -- 4 (short rows), 32 (one lane group per row) and multiples of the
    128-occurrence chunks -- against the oracle: all messages kept, stale
    messages dropped, and geometric weights."""
    counts = [1, 2, 4, 5, 6, 31, 32, 33, 64, 127, 128, 129, 130, 255, 256, 257, 300]
    V, M, D = len(counts) + 3, 8, 37
    iota = (rule or {}).get("iota", 1)
    cfg = cfg_of([(V, dim, 0, 0)], D=D, G=M, iota=iota)
    rng = np.random.default_rng(dim)

    def batch(k, stale):
        per = [[] for _ in range(M)]
        for r, c in enumerate(counts):
            for _ in range(c):
                per[int(rng.integers(0, M))].append(r)
        toks = [max(0, k - 3) if m in stale else k for m in range(M)]
        return [msg(toks[m], [np.array(per[m], np.int64)], [dim], D,
                    gen=torch.Generator(device="cuda").manual_seed(100 * k + m)) for m in range(M)]

    steps = [batch(0, []), batch(1, []), batch(2, [1, 5]), batch(3, [0]), batch(4, [])]
    run_custom(cfg, steps, rule=rule)


@pytest.mark.parametrize("D", [2048 * 152 * 2 + 6, 2048 * 152 * 3 * 2 + 2048 + 6])
def test_dense_tiles_over_many_ctas(D):
    """Dense sizes that give some CTAs more tiles than others, a short last
    tile and a ragged tail of 2 elements, every element against the oracle."""
    cfg = cfg_of([], D=D, G=3)
    run_custom(cfg, [[msg(0, [], [], D), msg(0, [], [], D), msg(0, [], [], D)],
                     [msg(1, [], [], D), msg(0, [], [], D), msg(1, [], [], D)]], by_ref=True)


def test_dense_only_and_tables_only():
    cfg = cfg_of([], D=1031, G=2)
    run_custom(cfg, [[msg(0, [], [], 1031), msg(0, [], [], 1031)]] * 2)
    cfg = cfg_of([(100, 4, 0, 0)], D=0, G=2)
    run_custom(cfg, [[msg(0, [[1, 2]], [4], 0), msg(0, [[2]], [4], 0)]] * 2)


@pytest.mark.parametrize("D", [1, 2, 3, 4, 5, 1023, 1024, 1025, 4097, 100_003])
def test_dense_sizes(D):
    cfg = cfg_of([(10, 4, 0, 0)], D=D, G=3)
    run_custom(cfg, [[msg(0, [[1]], [4], D), msg(0, [[]], [4], D), msg(0, [[2]], [4], D)],
                     [msg(1, [[1]], [4], D), msg(0, [[3]], [4], D), msg(1, [[]], [4], D)]],
               by_ref=True)


def test_ragged_sort_sizes():
    """Step sizes around the sort and segment-scan tiles (2048 positions) and
    the classification tiles (2048 row records)."""
    rng = np.random.default_rng(2)
    for n in (1, 63, 64, 65, 2047, 2048, 2049, 4095, 4096, 4097, 12289):
        cfg = cfg_of([(70_000, 8, 0, 0)], D=4, G=1)
        run_custom(cfg, [[msg(0, [rng.integers(0, 70_000, n)], [8], 4)]], max_ids=n)


# ---------------------------------------------------------------------------
# errors

def test_id_out_of_range_fails_the_step_without_touching_state():
    tables = [(10, 4, 0, 8, B.opt_desc())]
    g = B.GBA(tables, 4, B.opt_desc(), 1, 4, seed=1)
    w_before = _raw_table_w(g, 0)
    d_before = _raw_dense(g)
    m = msg(0, [[3, 10]], [4], 4)   # id 10 is outside [0, 10)
    g.push(m["token"], m["ids"], m["rows"], m["dense"], 1)
    rc = g.L.gba_try_apply(g.h)
    if rc == 1:
        rc = g.L.gba_sync(g.h)
    assert rc == B.GBA_E_ID_RANGE
    assert g.L.gba_try_apply(g.h) == B.GBA_E_STATE
    torch.cuda.synchronize()
    assert torch.equal(_raw_table_w(g, 0), w_before)
    assert torch.equal(_raw_dense(g), d_before)
    g.close()


def _raw_table_w(g, t):
    w, s0, s1, v = ctypes.c_void_p(), ctypes.c_void_p(), ctypes.c_void_p(), ctypes.c_void_p()
    g.L.gba_get_table(g.h, t, ctypes.byref(w), ctypes.byref(s0), ctypes.byref(s1),
                      ctypes.byref(v))
    torch.cuda.synchronize()
    n = g.rows[t] * g.dims[t]
    return B._copy_device(w.value, n, torch.float32)


def _raw_dense(g):
    w, s0, s1 = ctypes.c_void_p(), ctypes.c_void_p(), ctypes.c_void_p()
    g.L.gba_get_dense(g.h, ctypes.byref(w), ctypes.byref(s0), ctypes.byref(s1))
    torch.cuda.synchronize()
    return B._copy_device(w.value, g.D, torch.float32)


def test_push_validation_and_full_buffer():
    tables = [(10, 4, 0, 3, B.opt_desc())]
    g = B.GBA(tables, 4, B.opt_desc(), 100, 2, seed=1)
    m = msg(0, [[1, 2]], [4], 4)
    L, h = g.L, g.h
    good = [B.gba_sparse_grad(m["ids"][0].data_ptr(), 2, m["rows"][0].data_ptr())]
    too_many = [B.gba_sparse_grad(m["ids"][0].data_ptr(), 4, m["rows"][0].data_ptr())]
    assert B.gba_push(h, -1, good, m["dense"].data_ptr(), 1) == B.GBA_E_ARG
    assert B.gba_push(h, 0, good, m["dense"].data_ptr(), 0) == B.GBA_E_ARG
    assert B.gba_push(h, 0, too_many, m["dense"].data_ptr(), 1) == B.GBA_E_ARG
    assert B.gba_push(h, 0, good, None, 1) == B.GBA_E_ARG
    assert B.gba_push_ref(h, 0, good, m["dense"].data_ptr() + 4, 1) == B.GBA_E_ARG  # misaligned
    assert B.gba_push(h, 0, good, m["dense"].data_ptr(), 1) == B.GBA_OK
    assert B.gba_push(h, 0, good, m["dense"].data_ptr(), 1) == B.GBA_OK
    assert B.gba_push(h, 0, good, m["dense"].data_ptr(), 1) == B.GBA_E_FULL
    assert L.gba_try_apply(h) == 0
    g.close()


def test_bounded_wait_gives_up():
    """A device wait on a flag nothing sets returns GBA_E_DEVICE_TIMEOUT and
    the context stays usable."""
    L = B.load()
    assert L.gba_selftest_wait_timeout(2_000_000, None) == B.GBA_E_DEVICE_TIMEOUT
    x = torch.ones(4, device="cuda")
    assert float((x * 2).sum()) == 8.0


def test_tiny_wait_limit_in_sort_is_reported_or_harmless():
    """With a zero wait limit the onesweep look-back gives up whenever a
    predecessor tile is not ready yet; the step then fails with
    GBA_E_DEVICE_TIMEOUT (or succeeds if no tile had to wait).  No dense
    parameters here, so only the sort's waits are exercised."""
    rng = np.random.default_rng(0)
    cfg = cfg_of([(200_000, 8, 0, 0)], D=0, G=1)
    tables = [(200_000, 8, 0, 300_000, B.opt_desc())]
    g = B.GBA(tables, 0, None, 1, 4, seed=1)
    g.set_wait_limit(0)
    m = msg(0, [rng.integers(0, 200_000, 300_000)], [8], 0)
    g.push(m["token"], m["ids"], m["rows"], m["dense"], 1)
    rc = g.L.gba_try_apply(g.h)
    if rc == 1:
        rc = g.L.gba_sync(g.h)
    assert rc in (B.GBA_OK, B.GBA_E_DEVICE_TIMEOUT)
    g.close()
    # the device is still usable: a fresh handle runs a step
    g2 = B.GBA(tables, 0, None, 1, 4, seed=1)
    g2.push(m["token"], m["ids"], m["rows"], m["dense"], 1)
    assert g2.try_apply() == 1
    g2.sync()
    g2.close()


def test_tiny_wait_limit_in_dense_is_reported_or_harmless():
    """A dense-only step with a zero wait limit: the dense kernel's mbarrier
    waits give up whenever a stage is not ready at the first try, the producer
    stops issuing copies and waits (with its own bound) for the ones in
    flight, and the step reports GBA_E_DEVICE_TIMEOUT -- or completes if no
    wait had to give up.  Either way the context stays usable and a fresh
    handle applies a step afterwards."""
    D, M = 3_000_001, 6
    dense_opt = B.opt_desc(W.ADAM, 0.001)
    gen = torch.Generator(device="cuda").manual_seed(9)
    grads = [torch.randn(D, generator=gen, device="cuda") * 0.01 for _ in range(M)]
    g = B.GBA([], D, dense_opt, M, 2 * M, seed=2)
    g.set_wait_limit(0)
    for i in range(M):
        g.push_ref(0, [], [], grads[i], 1)
    rc = g.L.gba_try_apply(g.h)
    if rc == 1:
        rc = g.L.gba_sync(g.h)
    assert rc in (B.GBA_OK, B.GBA_E_DEVICE_TIMEOUT)
    g.close()
    g2 = B.GBA([], D, dense_opt, M, 2 * M, seed=2)
    for i in range(M):
        g2.push_ref(0, [], [], grads[i], 1)
    assert g2.try_apply() == 1
    g2.sync()
    w, _, _ = g2.dense()
    assert torch.isfinite(w).all()
    g2.close()


def test_dense_waits_run_out_when_copies_are_withheld():
    """K5's bounded waits, forced: the producer issues no copies, so every
    consumer waits on a stage nothing fills; after the 1 ms limit each wait
    gives up, the step reports GBA_E_DEVICE_TIMEOUT, the handle stays failed,
    and the context is still usable (a fresh handle applies a step that
    matches the oracle's dense update)."""
    D, M = 1_000_003, 4
    dense_opt = B.opt_desc(W.ADAGRAD, 0.01)
    gen = torch.Generator(device="cuda").manual_seed(13)
    grads = [torch.randn(D, generator=gen, device="cuda") * 0.01 for _ in range(M)]
    g = B.GBA([], D, dense_opt, M, 2 * M, seed=3)
    g.set_wait_limit(1_000_000)
    g.withhold_dense_copies(True)
    for i in range(M):
        g.push_ref(0, [], [], grads[i], 1)
    rc = g.L.gba_try_apply(g.h)
    if rc == 1:
        rc = g.L.gba_sync(g.h)
    assert rc == B.GBA_E_DEVICE_TIMEOUT
    assert g.L.gba_try_apply(g.h) != 1  # the handle stays failed
    g.close()
    torch.cuda.synchronize()
    g2 = B.GBA([], D, dense_opt, M, 2 * M, seed=3)
    for i in range(M):
        g2.push_ref(0, [], [], grads[i], 1)
    assert g2.try_apply() == 1
    g2.sync()
    w, _, _ = g2.dense()
    orc = O.OracleGBA([], D, O.OptSpec(O.ADAGRAD, 0.01), M, seed=3,
                      track_dense=np.arange(0, D, 997, dtype=np.int64))
    for i in range(M):
        orc.push(O.Message(0, 1, [], [], grads[i].cpu().numpy()))
    assert orc.try_apply() == 1
    got = w.cpu().numpy()[np.arange(0, D, 997)]
    np.testing.assert_allclose(got, orc.dense.w, rtol=1e-5, atol=1e-7)
    g2.close()


def test_device_code_is_sm103a():
    """The kernels run from sm_103a device code on this GPU."""
    assert B.load().gba_device_binary_version() == 103


@pytest.mark.parametrize("dim,mode", [(16, 0), (3, 0), (64, 1), (19, 1)])
def test_pull_returns_the_current_rows(dim, mode):
    """Pull responding (Alg. 2): after a few steps, gba_pull gives exactly the
    oracle's rows for any ids (duplicates, MODULO residues of negative ids)."""
    rng = np.random.default_rng(dim + 100 * mode)
    V = 997
    cfg = cfg_of([(V, dim, mode, 0)], D=7, G=3, iota=1)
    steps = []
    for k in range(3):
        batch = []
        for m in range(3):
            n = int(rng.integers(1, 200))
            ids = rng.zipf(1.3, n) % V if mode == 0 else rng.integers(-2**62, 2**62, n)
            batch.append(msg(max(0, k - int(rng.integers(0, 2))), [ids], [dim], 7))
        steps.append(batch)
    g, orc = run_custom(cfg, steps)
    if mode == 0:
        ids = rng.integers(0, V, 1000)
    else:
        ids = np.concatenate([rng.integers(-2**62, 2**62, 500),
                              np.concatenate([s_[0]["ids"][0].cpu().numpy() for s_ in steps])])
    ids_t = torch.as_tensor(ids, dtype=torch.int64, device="cuda")
    got = g.pull(0, ids_t).cpu().numpy()
    rows = H.rows_of(cfg, 0, ids.astype(np.int64))
    want = orc.tables[0].w.reshape(V, dim)[rows]
    assert np.array_equal(got, want)
    assert g.pull(0, ids_t[:0]).shape == (0, dim)
    g.sync()
    g.close()


def test_pull_orders_after_overlapping_steps():
    """With steps overlapping, a pull still sees every step enqueued before it."""
    cfg = W.reduced(2)
    g = H.make_gpu(cfg, overlap=True, debug=False)
    orc = H.make_oracle(cfg)
    for k in range(3):
        for m in W.generate_step(cfg, k, "cuda"):
            H.push_gpu(g, m)
            orc.push(H.to_oracle(m))
        assert g.try_apply() == 1 and orc.try_apply() == 1
    ids = torch.arange(0, cfg.tables[0].rows, 7, dtype=torch.int64, device="cuda")
    got = g.pull(0, ids).cpu().numpy()
    want = orc.tables[0].w.reshape(cfg.tables[0].rows, -1)[ids.cpu().numpy()]
    assert np.array_equal(got, want)
    g.close()


def test_pull_of_an_out_of_range_id_is_latched():
    tables = [(100, 8, 0, 16, B.opt_desc())]
    g = B.GBA(tables, 0, None, 1, 4, seed=1)
    ids = torch.tensor([3, 100, 5], dtype=torch.int64, device="cuda")
    out = g.pull(0, ids)
    assert int(g.L.gba_sync(g.h)) == B.GBA_E_ID_RANGE
    o = out.cpu().numpy()
    assert np.all(o[1] == 0)
    w = _raw_table_w(g, 0).view(100, 8).cpu().numpy()
    assert np.array_equal(o[[0, 2]], w[[3, 5]])
    g.close()


@pytest.mark.parametrize("by_ref", [False, True])
@pytest.mark.parametrize("rule", [dict(iota=2), dict(iota=5, decay=1, lam=0.8)])
def test_eager_dense_equals_buffered(by_ref, rule):
    """Eager push-time aggregation of the dense gradients gives the buffered
    mode's state bit for bit, and matches the oracle, with varying local
    batches (steps of different sizes, overshoot) and stale tokens."""
    rng = np.random.default_rng(5 + by_ref)
    cfg = cfg_of([(400, 8, 0, 0)], D=20_011, G=6, dense_kind=1)
    stream = []
    k_expected = 0
    for k in range(6):
        acc = 0
        while acc < cfg.G:  # one step's messages: local batches summing to >= G
            b = int(rng.integers(1, 4))
            m = msg(max(0, k - int(rng.integers(0, 4))), [rng.integers(0, 400, 40)], [8], 20_011,
                    B_=b)
            stream.append(m)
            acc += b
    outs = []
    for eager in (False, True):
        tables = [(400, 8, 0, 4096, H.opt_desc(cfg.tables[0].opt))]
        g = B.GBA(tables, cfg.D, H.opt_desc(cfg.dense_opt), cfg.G, 64, seed=cfg.seed, **rule)
        if eager:
            g.set_eager_dense(True)
        orc = H.make_oracle(cfg, rule=rule)
        n_steps = 0
        for m in stream:
            (g.push_ref if by_ref else g.push)(m["token"], m["ids"], m["rows"], m["dense"],
                                               m["local_batch"])
            orc.push(H.to_oracle(m))
            a, c = g.try_apply(), orc.try_apply()
            assert a == c
            n_steps += a
        g.sync()
        H.compare_state(g, orc, H.TOL_ONE_STEP)
        outs.append([t.cpu() for t in g.dense()[:3] if t is not None] + [g.table(0)[0].cpu()])
        assert n_steps >= 6
        g.close()
    for a, b in zip(*outs):
        assert torch.equal(a, b)


def test_eager_dense_refusals_and_capacity():
    tables = [(100, 4, 0, 16, B.opt_desc())]
    g = B.GBA(tables, 1000, B.opt_desc(1, 0.001), 4, 64, seed=1, iota=3, drop_latest=1)
    with pytest.raises(B.GBAError) as e:
        g.set_eager_dense(True)
    assert e.value.status == B.GBA_E_ARG
    g.close()
    g = B.GBA(tables, 1000, B.opt_desc(1, 0.001), 4, 64, seed=1, iota=3)
    m = msg(0, [[1, 2]], [4], 1000, B_=4)
    g.push(m["token"], m["ids"], m["rows"], m["dense"], 4)
    with pytest.raises(B.GBAError) as e:  # messages are buffered
        g.set_eager_dense(True)
    assert e.value.status == B.GBA_E_STATE
    assert g.try_apply() == 1
    g.set_eager_dense(True)
    # each message fills a whole step: eight pending steps fit, a ninth does not
    for i in range(8):
        g.push(m["token"], m["ids"], m["rows"], m["dense"], 4)
    rc = g.L.gba_push(g.h, 0, (B.gba_sparse_grad * 1)(*g._grads(m["ids"], m["rows"])),
                      m["dense"].data_ptr(), 4)
    assert rc == B.GBA_E_FULL
    for i in range(8):
        assert g.try_apply() == 1
    assert g.try_apply() == 0
    g.sync()
    g.close()


def test_hash_table_grows_and_matches_the_oracle():
    """An expandable hash table of 64-bit ids (every distinct id its own row)
    next to a DIRECT table: it starts at 1024 slots and doubles several times
    as new ids arrive; dedup output, state, tags and pulls (of stored and of
    never-seen ids) match the oracle, which keys rows by id."""
    rng = np.random.default_rng(23)
    ranks = 30_000
    salt = 0x5DEECE66D
    tcs = (W.TableCfg(1000, 16, 1, 0, 1.1, W.HASH, W.OptCfg(W.ADAGRAD, 0.01)),
           W.TableCfg(300, 8, 1, 0, 1.1, W.DIRECT, W.OptCfg(W.ADAM, 0.001)))
    cfg = W.WorkloadCfg("hash", M=4, B=1, tables=tcs, D=77, dense_opt=W.OptCfg(W.ADAM, 0.001),
                        stale=W.StaleCfg("fresh"), iota=2, seed=8)
    steps = []
    for k in range(8):
        batch = []
        for m in range(4):
            r = torch.as_tensor(rng.zipf(1.2, 2000) % ranks, dtype=torch.int64)
            ids0 = W.hash64(r ^ salt)
            ids1 = rng.integers(0, 300, 50)
            batch.append(msg(max(0, k - int(rng.integers(0, 4))), [ids0.numpy(), ids1], [16, 8], 77))
        steps.append(batch)
    all_ids = np.unique(np.concatenate([m["ids"][0].cpu().numpy() for b in steps for m in b]))
    unseen = W.hash64(torch.arange(ranks, ranks + 40, dtype=torch.int64) ^ salt).numpy()
    track0 = np.unique(np.concatenate([all_ids, unseen]))
    tables = [(1000, 16, W.HASH, 8192, H.opt_desc(tcs[0].opt)),
              (300, 8, W.DIRECT, 8192, H.opt_desc(tcs[1].opt))]
    g = B.GBA(tables, 77, H.opt_desc(cfg.dense_opt), 4, 16, seed=cfg.seed, iota=2)
    g.set_debug(True)
    assert g.capacity(0) == 1024
    orc = H.make_oracle(cfg, track_rows=[track0, None])
    for batch in steps:
        for m in batch:
            g.push(m["token"], m["ids"], m["rows"], m["dense"], 1)
            orc.push(H.to_oracle(m))
        assert g.try_apply() == 1 and orc.try_apply() == 1
        # dedup output: the hash table reports ids; compare as sets ordered by id
        t_g, r_g, c_g, k_g = g.segments()
        sel = t_g == 0
        order = np.argsort(r_g[sel])
        touched = np.nonzero(orc.last_count[0])[0]
        assert np.array_equal(r_g[sel][order], track0[touched])
        assert np.array_equal(c_g[sel][order], orc.last_count[0][touched])
        assert np.array_equal(k_g[sel][order], orc.last_kept[0][touched])
        # state of every tracked id the table holds; ids it does not hold were never pushed
        slots = g.lookup(0, torch.as_tensor(track0, device="cuda")).cpu().numpy()
        have = slots >= 0
        assert np.all(np.isin(track0[have], all_ids))
        w, s0, _, ver = g.table_rows(0, slots[have])
        ts = orc.tables[0]
        assert np.array_equal(ver.cpu().numpy().astype(np.int64), ts.ver[have])
        assert H.rel_err(w.cpu().numpy(), ts.w.reshape(-1, 16)[have]) <= H.TOL_ONE_STEP
        assert H.rel_err(s0.cpu().numpy(), ts.s0.reshape(-1, 16)[have]) <= H.TOL_ONE_STEP
        assert np.all(ts.ver[~have] == 0)
    assert g.capacity(0) >= 2 * 1024  # the table grew
    # pulls: stored ids give their rows, never-seen ids their initial values
    got = g.pull(0, torch.as_tensor(track0, device="cuda")).cpu().numpy()
    assert H.rel_err(got, orc.tables[0].w.reshape(-1, 16)) <= H.TOL_ONE_STEP
    unseen_idx = np.searchsorted(track0, unseen)
    assert np.array_equal(got[unseen_idx], orc.tables[0].w.reshape(-1, 16)[unseen_idx])
    g.sync()
    g.close()


def test_hash_table_reserved_id_fails_the_step():
    tables = [(1000, 4, W.HASH, 16, B.opt_desc())]
    g = B.GBA(tables, 0, None, 1, 4, seed=1)
    ids = torch.tensor([5, -2**63, 7], dtype=torch.int64, device="cuda")
    g.push(0, [ids], [torch.zeros(3, 4, device="cuda")], torch.zeros(0, device="cuda"), 1)
    assert g.L.gba_try_apply(g.h) == 1
    assert g.L.gba_sync(g.h) == B.GBA_E_ID_RANGE
    g.close()
