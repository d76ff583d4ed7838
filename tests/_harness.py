"""Runs one message stream through the CUDA library and the CPU oracle and
compares them.  Test infrastructure: used by the GPU tests and the smoke check."""
from __future__ import annotations

import numpy as np
import torch

from oracle import oracle as O
from paper_2205_11048_gb300 import binding as B
from paper_2205_11048_gb300 import workload as W

# Tolerances of the parity contract: one apply step, and after 100 steps.
TOL_ONE_STEP = 1e-5
TOL_MANY_STEPS = 1e-4


def opt_spec(o: W.OptCfg) -> O.OptSpec:
    return O.OptSpec(o.kind, o.lr, o.init_acc, o.beta1, o.beta2, o.eps)


def opt_desc(o: W.OptCfg):
    return B.opt_desc(o.kind, o.lr, o.init_acc, o.beta1, o.beta2, o.eps)


def make_gpu(cfg: W.WorkloadCfg, max_buf=None, seed=None, debug=True, rule=None, overlap=False):
    g = B.gba_for_workload(cfg, max_buf=max_buf, seed=seed, overlap=overlap, **(rule or {}))
    if debug:
        g.set_debug(True)
    return g


def make_oracle(cfg: W.WorkloadCfg, track_rows=None, track_dense=None, seed=None, rule=None):
    specs = [O.TableSpec(tb.rows, tb.dim, opt_spec(tb.opt), tb.id_mode) for tb in cfg.tables]
    rule = rule or dict(iota=cfg.iota)
    return O.OracleGBA(specs, cfg.D, opt_spec(cfg.dense_opt), cfg.G,
                       seed=cfg.seed if seed is None else seed, track_rows=track_rows,
                       track_dense=track_dense, **rule)


def to_oracle(msg) -> O.Message:
    return O.Message(int(msg["token"]), int(msg["local_batch"]),
                     [i.detach().cpu().numpy() for i in msg["ids"]],
                     [r.detach().cpu().numpy() for r in msg["rows"]],
                     msg["dense"].detach().cpu().numpy())


def push_gpu(g: B.GBA, msg, by_ref=False):
    f = g.push_ref if by_ref else g.push
    f(msg["token"], msg["ids"], msg["rows"], msg["dense"], msg["local_batch"])


def rel_err(a: np.ndarray, b: np.ndarray) -> float:
    """max_i |a-b| / max(|b|, 1e-3 * max_j |b_j|) over one tensor."""
    a = np.asarray(a, np.float64).ravel()
    b = np.asarray(b, np.float64).ravel()
    if b.size == 0:
        return 0.0
    floor = 1e-3 * float(np.max(np.abs(b)))
    den = np.maximum(np.abs(b), floor if floor > 0 else 1e-30)
    return float(np.max(np.abs(a - b) / den))


def rows_of(cfg, t, ids_np):
    """The oracle's row of each id: the id itself (DIRECT, and HASH tables,
    where every distinct id is a row), or its unsigned residue (MODULO)."""
    tb = cfg.tables[t]
    if tb.id_mode in (W.DIRECT, W.HASH):
        return ids_np.astype(np.int64)
    return (ids_np.view(np.uint64) % np.uint64(tb.rows)).astype(np.int64)


def compare_segments(g: B.GBA, orc: O.OracleGBA, full_tracking: bool):
    """Dedup output of the last step: bit-exact against the oracle's."""
    t_g, r_g, c_g, k_g = g.segments()
    for t, ts in enumerate(orc.tables):
        sel = t_g == t
        rows_g, cnt_g, kept_g = r_g[sel], c_g[sel], k_g[sel]
        assert np.all(np.diff(rows_g) > 0), "unique rows must be strictly increasing"
        cnt_o = orc.last_count[t]
        touched_o = np.nonzero(cnt_o)[0]
        if full_tracking:
            assert np.array_equal(rows_g, ts.track[touched_o]), f"unique rows differ (table {t})"
            assert np.array_equal(cnt_g, cnt_o[touched_o]), f"message counts differ (table {t})"
            assert np.array_equal(kept_g, orc.last_kept[t][touched_o]), f"kept counts differ ({t})"
        else:
            pos = np.searchsorted(ts.track, rows_g)
            pos = np.minimum(pos, len(ts.track) - 1)
            hit = ts.track[pos] == rows_g
            assert np.array_equal(rows_g[hit], ts.track[touched_o]), f"sampled rows differ ({t})"
            assert np.array_equal(cnt_g[hit], cnt_o[touched_o])
            assert np.array_equal(kept_g[hit], orc.last_kept[t][touched_o])
    keep_g = g.keep()
    assert np.array_equal(keep_g, orc.last_keep), "message weights differ"


def compare_state(g: B.GBA, orc: O.OracleGBA, tol: float, full_dense=True):
    """Tables and dense state: floats within tol (R14 metric), tags bit-exact,
    never-updated rows bit-identical."""
    worst = {}
    for t, ts in enumerate(orc.tables):
        d = ts.spec.dim
        w, s0, s1, ver = g.table_rows(t, ts.track)
        w, s0 = w.cpu().numpy(), s0.cpu().numpy()
        ver = ver.cpu().numpy()
        assert np.array_equal(ver.astype(np.int64), ts.ver), f"tags differ (table {t})"
        ow = ts.w.reshape(-1, d)
        os0 = ts.s0.reshape(-1, d)
        untouched = ts.ver == 0
        assert np.array_equal(w[untouched], ow[untouched]), "untouched rows must be bit-identical"
        worst[f"t{t}.w"] = rel_err(w, ow)
        worst[f"t{t}.s0"] = rel_err(s0, os0)
        if ts.s1 is not None:
            worst[f"t{t}.s1"] = rel_err(s1.cpu().numpy(), ts.s1.reshape(-1, d))
    if orc.D > 0:
        dw, ds0, ds1 = g.dense()
        idx = torch.as_tensor(orc.dense.track, device="cuda")
        worst["dense.w"] = rel_err(dw[idx].cpu().numpy(), orc.dense.w)
        worst["dense.s0"] = rel_err(ds0[idx].cpu().numpy(), orc.dense.s0)
        if orc.dense.s1 is not None:
            worst["dense.s1"] = rel_err(ds1[idx].cpu().numpy(), orc.dense.s1)
    bad = {k: v for k, v in worst.items() if not v <= tol}
    assert not bad, f"tolerance {tol} exceeded: {bad}"
    return worst


def compare_stats(g: B.GBA, orc_stats_sum: dict):
    s = g.stats()
    for key in ("msgs_kept", "msgs_dropped", "dense_stale_sum", "pairs", "pairs_dropped",
                "row_stale_sum", "occurrences", "rows_touched", "rows_applied",
                "occurrences_kept"):
        assert s[key] == orc_stats_sum[key], (key, s[key], orc_stats_sum[key])
    for key in ("dense_stale_max", "row_stale_max"):
        assert s[key] == orc_stats_sum[key], (key, s[key], orc_stats_sum[key])


def accumulate_stats(acc: dict, step: dict, orc=None):
    if orc is not None:
        acc["occurrences_kept"] = acc.get("occurrences_kept", 0) + int(
            sum(int(k.sum()) for k in orc.last_kept))
    for k, v in step.items():
        if k.endswith("_max"):
            acc[k] = max(acc.get(k, 0), v)
        else:
            acc[k] = acc.get(k, 0) + v
    return acc


def run_parity(cfg: W.WorkloadCfg, steps: int, tol: float, by_ref=False, check_every=1,
               track_rows=None, track_dense=None, max_buf=None, rule=None, device="cuda",
               messages=None, overlap=False):
    """Feed the same stream to both sides for `steps` global steps and compare."""
    full = track_rows is None
    g = make_gpu(cfg, max_buf=max_buf, rule=rule, overlap=overlap)
    orc = make_oracle(cfg, track_rows, track_dense, rule=rule)
    stats = {}
    worst = {}
    keep_alive = []
    for k in range(steps):
        msgs = messages(k) if messages else W.generate_step(cfg, k, device)
        for m in msgs:
            push_gpu(g, m, by_ref)
            orc.push(to_oracle(m))
        if by_ref:
            keep_alive.append(msgs)
        assert g.try_apply() == 1
        assert orc.try_apply() == 1
        accumulate_stats(stats, orc.last_stats, orc)
        compare_segments(g, orc, full) if orc.tables else None
        if (k + 1) % check_every == 0 or k == steps - 1:
            worst = compare_state(g, orc, tol)
        if len(keep_alive) > 2:
            g.sync()
            keep_alive.pop(0)
    g.sync()
    if full:
        compare_stats(g, stats)
    assert g.version() == steps == orc.pull_version()
    g.close()
    return worst


def rows_of_gpu(tb, ids: torch.Tensor) -> torch.Tensor:
    """Row of each id (int64 tensor on the device): DIRECT ids as they are,
    MODULO ids by the residue of their unsigned 64-bit value."""
    if tb.id_mode == W.DIRECT:
        return ids
    V = tb.rows
    r = torch.remainder(ids, V)
    wrap = (1 << 64) % V            # 2^64 mod V, added for negative ids
    return torch.where(ids < 0, torch.remainder(r + wrap, V), r)


def run_fullsize(cfg: W.WorkloadCfg, steps: int, tol: float, n_hot=150, n_rand=1500,
                 n_dense=20000, seed=0, overlap=True):
    """Full-size workload in the benchmark's launch configuration (messages
    pushed by reference), checked against the oracle on a sample of rows (hot
    and random rows touched by the first step) and of dense parameters."""
    g = make_gpu(cfg, debug=False, overlap=overlap)
    gen = torch.Generator().manual_seed(seed)
    first = W.generate_step(cfg, 0, "cuda")
    track = []
    for t, tb in enumerate(cfg.tables):
        rows = torch.cat([rows_of_gpu(tb, m["ids"][t]) for m in first])
        u, cnt = torch.unique(rows, return_counts=True)
        hot = u[torch.argsort(cnt, descending=True)[:n_hot]]
        pick = torch.randperm(u.numel(), generator=gen)[:n_rand].to(u.device)
        rnd = u[pick]
        cold = torch.randint(0, tb.rows, (50,), generator=gen).to(u.device)
        track.append(torch.unique(torch.cat([hot, rnd, cold])))
    dense_idx = torch.unique(torch.cat([
        torch.randint(0, cfg.D, (n_dense,), generator=gen),
        torch.tensor([0, 1, 2, 3, cfg.D - 1, cfg.D - 2]).clamp(0, cfg.D - 1)]))
    orc = make_oracle(cfg, track_rows=[t.cpu().numpy() for t in track],
                      track_dense=dense_idx.numpy())
    dense_host = [np.zeros(cfg.D, np.float32) for _ in range(cfg.M)]
    dense_dev_idx = dense_idx.to("cuda")
    for k in range(steps):
        msgs = first if k == 0 else W.generate_step(cfg, k, "cuda")
        for i, m in enumerate(msgs):
            push_gpu(g, m, by_ref=True)
            ids_f, rows_f = [], []
            for t, tb in enumerate(cfg.tables):
                sel = torch.isin(rows_of_gpu(tb, m["ids"][t]), track[t])
                ids_f.append(m["ids"][t][sel].cpu().numpy())
                rows_f.append(m["rows"][t][sel].cpu().numpy())
            dh = dense_host[i]
            dh[dense_idx.numpy()] = m["dense"][dense_dev_idx].cpu().numpy()
            orc.push(O.Message(int(m["token"]), int(m["local_batch"]), ids_f, rows_f, dh.copy()))
        assert g.try_apply() == 1
        assert orc.try_apply() == 1
        g.sync()
        keep_g = g.keep()
        assert np.array_equal(keep_g, orc.last_keep), "message weights differ"
        msgs = None
    worst = compare_state(g, orc, tol)
    g.close()
    return worst
