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
