"""Host-side pieces of the benchmark and the binding, on the CPU: the
algorithmic bytes per step (the survey's definition written out), and the
handle arguments built from a workload description."""
import numpy as np

import bench
from paper_2205_11048_gb300 import binding as B
from paper_2205_11048_gb300 import workload as W


def test_algorithmic_bytes_of_the_1e7x32_workload():
    cfg = W.config(2)  # one 1e7 x 32 Adagrad table, 1M dense parameters with Adam
    steps = 4
    n, n_kept, u, m_kept = 851968, 759560, 338193, 28
    delta = dict(occurrences=n * steps, occurrences_kept=n_kept * steps,
                 rows_applied=u * steps, msgs_kept=m_kept * steps, rows_touched=365444 * steps)
    b, per = bench.alg_bytes(cfg, delta, steps)
    d, D = 32, 1_000_000
    assert b["sort"] == 8 * n                                   # the ids
    assert b["rows"] == 4 * d * n_kept + 2 * 2 * 4 * d * u + 8 * u  # kept rows, w + acc, tag
    assert b["dense"] == 4 * D * m_kept + 2 * 3 * 4 * D           # kept grads, w + m + v
    assert b["total"] == b["sort"] + b["rows"] + b["dense"]
    assert per["u_applied"] == u and per["occ_kept"] == n_kept


def test_handle_arguments_from_a_workload(monkeypatch):
    seen = []

    class Fake:
        def __init__(self, *a, **k):
            seen.append((a, k))
            self.overlap = False

        def set_overlap(self, on):
            self.overlap = on

    monkeypatch.setattr(B, "GBA", Fake)
    for n in range(1, 6):
        cfg = W.config(n)
        g = B.gba_for_workload(cfg, overlap=True)
        (tables, D, dense_opt, G, max_buf), kw = seen[-1]
        assert [t[:4] for t in tables] == [(tb.rows, tb.dim, tb.id_mode, cfg.max_ids_per_msg(i))
                                           for i, tb in enumerate(cfg.tables)]
        assert [t[4].kind for t in tables] == [tb.opt.kind for tb in cfg.tables]
        assert (D, G, max_buf) == (cfg.D, cfg.G, 2 * cfg.M)
        # the descriptor holds C floats
        assert dense_opt.kind == cfg.dense_opt.kind and dense_opt.lr == float(np.float32(cfg.dense_opt.lr))
        assert kw == dict(seed=cfg.seed, iota=cfg.iota) and g.overlap
    B.gba_for_workload(W.config(1), row_staleness=1)
    assert seen[-1][1] == dict(seed=W.config(1).seed, row_staleness=1)


def test_dense_bytes_of_the_two_dense_modes():
    """Buffered: the apply reads every kept gradient (4D each) and the state.
    Eager: a kept push reads its gradient and updates the step's compensated
    pair (4D + 8D + 8D; the first kept push only writes the pair, 4D + 8D), and
    the apply reads the pair (8D) and the state."""
    cfg = W.config(4)  # 64M dense parameters with Adam
    D, m = cfg.D, 15.0
    state = 2 * 3 * 4 * D
    buf = bench.dense_traffic(cfg, {"m_kept": m}, "buffered")
    assert buf["bytes_per_step"] == buf["bytes_per_apply"] == 4 * D * m + state
    assert buf["bytes_per_kept_push"] == 0.0 and buf["buffer_bytes_per_message"] == 4 * D
    eag = bench.dense_traffic(cfg, {"m_kept": m}, "eager")
    pushes = 12 * D + 20 * D * (m - 1)
    assert abs(eag["bytes_per_kept_push"] * m - pushes) < 1e-3 * pushes
    assert eag["bytes_per_apply"] == 8 * D + state
    assert abs(eag["bytes_per_step"] - (pushes + 8 * D + state)) < 1e-3 * pushes
    assert eag["buffer_bytes_per_pending_step"] == 8 * D
    # no kept message: nothing is pushed into the pair
    assert bench.dense_traffic(cfg, {"m_kept": 0.0}, "eager")["bytes_per_kept_push"] == 0.0


def test_workload_variants_for_the_bench():
    """Shaped profiling cases keep the message structure and shrink the state;
    hash-id tables start at a power of two at least twice the rows; a hash
    table too large for one GPU is refused before any allocation."""
    base = W.config(5)
    s = bench.workload_cfg(5, "as-configured", 4_000_000, 2_000_000)
    assert s.tables[0].rows == 4_000_000 and s.D == 2_000_000
    assert (s.M, s.B, s.tables[0].dim, s.tables[0].fields) == (base.M, base.B, base.tables[0].dim,
                                                               base.tables[0].fields)
    assert s.name != base.name and "shaped" in s.name
    h = bench.workload_cfg(2, "hash")
    cap = h.tables[0].rows
    assert h.tables[0].id_mode == W.HASH and cap & (cap - 1) == 0
    assert cap >= 2 * W.config(2).tables[0].rows and cap // 2 < 2 * W.config(2).tables[0].rows
    import pytest
    with pytest.raises(SystemExit):
        bench.workload_cfg(5, "hash")


def test_config_dict_states_the_l2_rule():
    """Each global batch's ids and gradients against the 129 MB L2: larger for
    the headline workload, smaller (and said so) for the tiny one."""
    big = bench.config_dict(W.config(5), 1)
    assert big["l2"].startswith("inputs larger than L2") and big["workload"] == W.config(5).name
    small = bench.config_dict(W.config(1), 1)
    assert small["l2"].startswith("inputs smaller than L2")
    assert big["parallelism"] == "replicas x1" and bench.config_dict(W.config(5), 4)["parallelism"] == "replicas x4"


def test_traffic_is_tied_to_the_kernel_code(tmp_path, monkeypatch):
    """The committed DRAM traffic of a kernel class is reported only while the
    class's code (comments aside) is the code it was measured on."""
    src = "int a; // note\n/* block\n comment */ int b;\n"
    assert bench._code_only(src) == bench._code_only(src.replace("note", "other remark"))
    assert bench._code_only(src) != bench._code_only(src.replace("int b", "int c"))
    (tmp_path / "profiles").mkdir()
    (tmp_path / "k.cu").write_text(src)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    monkeypatch.setitem(bench.KERNEL_SOURCES, "dense", ["k.cu"])
    sha = bench.source_sha(["k.cu"])
    (tmp_path / "profiles" / "traffic.json").write_text(
        '{"w": {"dense": {"dram_bytes_per_step": 123.0, "source_sha": "%s"}}}' % sha)
    assert bench.measured_traffic("dense", "w") == 123.0
    assert bench.measured_traffic("dense", "other") is None
    (tmp_path / "k.cu").write_text(src.replace("int b", "int c"))
    assert bench.measured_traffic("dense", "w") is None
