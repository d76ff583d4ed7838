"""Pins of the CPU oracle: checks against what the paper and mathematics fix.

Each pin takes an oracle library handle so the same checks can be run against
copies of the oracle with a planted mistake (test_oracle_mutations.py).
"""
from __future__ import annotations

import json
import os
from fractions import Fraction

import numpy as np

from oracle import oracle as O

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def load_golden(name="hand_example.json"):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def F(s) -> float:
    return float(Fraction(str(s)))


def _msg(j, n_tables=1):
    ids = np.array(j["ids"], dtype=np.int64)
    rows = np.array(j["rows"], dtype=np.float32).reshape(len(ids), -1)
    return O.Message(j["token"], j["B"], [ids], [rows], np.array(j["dense"], np.float32))


# ---------------------------------------------------------------------------
def pin_hand_adagrad(L):
    """Two hand-worked steps (Eq. (1) drops, per-ID tags, both denominators)."""
    g = load_golden()["adagrad"]
    tb = O.TableSpec(g["table"]["rows"], g["table"]["dim"],
                     O.OptSpec(O.ADAGRAD, F(g["table"]["lr"]), F(g["table"]["init_acc"])))
    dopt = O.OptSpec(O.ADAGRAD, F(g["dense"]["lr"]), F(g["dense"]["init_acc"]))
    orc = O.OracleGBA([tb], g["dense"]["D"], dopt, g["global_batch"], iota=g["iota"],
                      seed=12345, library=L)
    w0 = orc.tables[0].w.astype(np.float64).reshape(tb.rows, tb.dim).copy()
    dw0 = orc.dense.w.astype(np.float64).copy()
    for step in g["steps"]:
        assert orc.pull_version() == step["k"]
        for m in step["messages"]:
            orc.push(_msg(m))
        assert orc.try_apply() == 1
        e = step["expect"]
        assert orc.last_keep.tolist() == e["keep"], ("keep", orc.last_keep)
        cnt = orc.last_count[0]
        kept = orc.last_kept[0]
        touched = np.nonzero(cnt)[0].tolist()
        assert touched == e["touched"], ("touched", touched)
        assert cnt[touched].tolist() == e["count"], ("count", cnt)
        assert kept[touched].tolist() == e["kept"], ("kept", kept)
        w = orc.tables[0].w.astype(np.float64).reshape(tb.rows, tb.dim)
        acc = orc.tables[0].s0.reshape(tb.rows, tb.dim)
        for r in range(tb.rows):
            want_dw = [F(v) for v in e["dw"][str(r)]]
            assert (w[r] - w0[r]).tolist() == want_dw, ("dw", r, (w[r] - w0[r]).tolist())
            assert acc[r].astype(np.float64).tolist() == [F(v) for v in e["acc"][str(r)]], \
                ("acc", r)
        assert orc.tables[0].ver.tolist() == e["ver"], ("ver", orc.tables[0].ver)
        dw = (orc.dense.w.astype(np.float64) - dw0).tolist()
        assert dw == [F(v) for v in e["dense_dw"]], ("dense dw", dw)
        assert orc.dense.s0.astype(np.float64).tolist() == [F(v) for v in e["dense_acc"]]
        for key, val in e["stats"].items():
            assert orc.last_stats[key] == val, ("stats", key, orc.last_stats[key], val)


def _check_hand_step(orc, tb, e, w0, dw0):
    assert orc.last_keep.tolist() == e["keep"], ("keep", orc.last_keep)
    cnt = orc.last_count[0]
    kept = orc.last_kept[0]
    touched = np.nonzero(cnt)[0].tolist()
    assert touched == e["touched"], ("touched", touched)
    assert cnt[touched].tolist() == e["count"], ("count", cnt)
    assert kept[touched].tolist() == e["kept"], ("kept", kept)
    w = orc.tables[0].w.astype(np.float64).reshape(tb.rows, tb.dim)
    acc = orc.tables[0].s0.reshape(tb.rows, tb.dim)
    for r in range(tb.rows):
        assert (w[r] - w0[r]).tolist() == [F(v) for v in e["dw"][str(r)]], \
            ("dw", r, (w[r] - w0[r]).tolist())
        assert acc[r].astype(np.float64).tolist() == [F(v) for v in e["acc"][str(r)]], ("acc", r)
    assert orc.tables[0].ver.tolist() == e["ver"], ("ver", orc.tables[0].ver)
    dw = (orc.dense.w.astype(np.float64) - dw0).tolist()
    assert dw == [F(v) for v in e["dense_dw"]], ("dense dw", dw)
    assert orc.dense.s0.astype(np.float64).tolist() == [F(v) for v in e["dense_acc"]]
    for key, val in e["stats"].items():
        assert orc.last_stats[key] == val, ("stats", key, orc.last_stats[key], val)


def pin_hand_rule_options(L):
    """Hand-worked steps of the optional readings: a row's sum divided by its
    kept messages, or by M; rows decayed by the message staleness k - token."""
    g = load_golden()["rule_options"]
    for var in g["variants"]:
        tb = O.TableSpec(g["table"]["rows"], g["table"]["dim"],
                         O.OptSpec(O.ADAGRAD, F(g["table"]["lr"]), F(g["table"]["init_acc"])))
        dopt = O.OptSpec(O.ADAGRAD, F(g["dense"]["lr"]), F(g["dense"]["init_acc"]))
        orc = O.OracleGBA([tb], g["dense"]["D"], dopt, g["global_batch"], seed=4321, library=L,
                          **var["rule"])
        w0 = orc.tables[0].w.astype(np.float64).reshape(tb.rows, tb.dim).copy()
        dw0 = orc.dense.w.astype(np.float64).copy()
        for step in (g["step0"], var["step1"]):
            assert orc.pull_version() == step["k"]
            for m in step["messages"]:
                orc.push(_msg(m))
            assert orc.try_apply() == 1
            _check_hand_step(orc, tb, step["expect"], w0, dw0)


def pin_hand_decay_variants(L):
    """Hand-worked steps of geometric decay (lambda^s) and of Hop-BW's ignored
    latest gradients, exact in float32."""
    g = load_golden()["decay_variants"]
    for name in ("geometric", "hop_bw"):
        var = g[name]
        tb = O.TableSpec(g["table"]["rows"], g["table"]["dim"],
                         O.OptSpec(O.ADAGRAD, F(g["table"]["lr"]), F(g["table"]["init_acc"])))
        dopt = O.OptSpec(O.ADAGRAD, F(g["dense"]["lr"]), F(g["dense"]["init_acc"]))
        orc = O.OracleGBA([tb], g["dense"]["D"], dopt, var["global_batch"], seed=4321, library=L,
                          **var["rule"])
        w0 = orc.tables[0].w.astype(np.float64).reshape(tb.rows, tb.dim).copy()
        dw0 = orc.dense.w.astype(np.float64).copy()
        for step in var["steps"]:
            assert orc.pull_version() == step["k"]
            for m in step["messages"]:
                orc.push(_msg(m))
            assert orc.try_apply() == 1
            _check_hand_step(orc, tb, step["expect"], w0, dw0)


def pin_decay_special_cases(L, seed=31):
    """lambda = 1 is Eq. (1) and drop_latest = 0 ignores nothing: both give the
    default rule's state bit for bit; drop_latest = M keeps no gradient, so
    only the dense optimizer moves (with a zero gradient)."""
    rng = np.random.default_rng(seed)
    V, d, D, M = 11, 3, 7, 4
    batches = [random_messages(rng, M, V, d, D, 0, 6, tokens=[max(0, s - int(t)) for t in
                                                           rng.integers(0, 4, M)])
               for s in range(4)]
    def run(**rule):
        tb = O.TableSpec(V, d, O.OptSpec(O.ADAM, 0.003))
        orc = O.OracleGBA([tb], D, O.OptSpec(O.ADAM, 0.001), M, iota=2, seed=9, library=L, **rule)
        for b in batches:
            for m in b:
                orc.push(m)
            assert orc.try_apply() == 1
        return orc
    base = run()
    for rule in (dict(decay=1, lam=1.0), dict(drop_latest=0)):
        o = run(**rule)
        assert np.array_equal(o.tables[0].w, base.tables[0].w), rule
        assert np.array_equal(o.tables[0].ver, base.tables[0].ver), rule
        assert np.array_equal(o.dense.w, base.dense.w), rule
    none = run(drop_latest=M)
    assert np.all(none.tables[0].ver == 0)
    # with a zero gradient Adam's first step moves nothing: m = v = 0
    tb = O.TableSpec(V, d, O.OptSpec(O.ADAM, 0.003))
    fresh = O.OracleGBA([tb], D, O.OptSpec(O.ADAM, 0.001), M, iota=2, seed=9, library=L)
    assert np.array_equal(none.dense.w, fresh.dense.w) and np.all(none.dense.s1 == 0)
    # geometric weights fall with staleness: lambda^s for the kept dense gradients
    o = run(decay=1, lam=0.5)
    assert not np.array_equal(o.dense.w, base.dense.w)


def pin_hand_adam(L):
    """One textbook Adam step with dyadic hyper-parameters."""
    g = load_golden()["adam"]
    t = g["table"]
    opt = O.OptSpec(O.ADAM, F(t["lr"]), 0.0, F(t["beta1"]), F(t["beta2"]), F(t["eps"]))
    dd = g["dense"]
    dopt = O.OptSpec(O.ADAM, F(dd["lr"]), 0.0, F(dd["beta1"]), F(dd["beta2"]), F(dd["eps"]))
    tb = O.TableSpec(t["rows"], t["dim"], opt)
    orc = O.OracleGBA([tb], dd["D"], dopt, g["global_batch"], iota=g["iota"], seed=7,
                      library=L)
    w0 = orc.tables[0].w.astype(np.float64).reshape(tb.rows, tb.dim).copy()
    dw0 = orc.dense.w.astype(np.float64).copy()
    orc.push(_msg(g["message"]))
    assert orc.try_apply() == 1
    e = g["expect"]
    w = orc.tables[0].w.astype(np.float64).reshape(tb.rows, tb.dim)
    m = orc.tables[0].s0.reshape(tb.rows, tb.dim)
    v = orc.tables[0].s1.reshape(tb.rows, tb.dim)
    for r in range(tb.rows):
        assert (w[r] - w0[r]).tolist() == [F(x) for x in e["dw"][str(r)]], ("adam dw", r)
        assert m[r].astype(np.float64).tolist() == [F(x) for x in e["m"][str(r)]], ("m", r)
        assert v[r].astype(np.float64).tolist() == [F(x) for x in e["v"][str(r)]], ("v", r)
    assert (orc.dense.w.astype(np.float64) - dw0).tolist() == [F(x) for x in e["dense_dw"]]
    assert orc.dense.s0.astype(np.float64).tolist() == [F(x) for x in e["dense_m"]]
    assert orc.dense.s1.astype(np.float64).tolist() == [F(x) for x in e["dense_v"]]
    assert orc.tables[0].ver.tolist() == e["ver"]


# ---------------------------------------------------------------------------
def random_messages(rng, M, V, d, D, n_lo=0, n_hi=6, tokens=None, B=1, id_hi=None):
    msgs = []
    for m in range(M):
        n = int(rng.integers(n_lo, n_hi + 1))
        ids = rng.integers(0, V if id_hi is None else id_hi, size=n).astype(np.int64)
        rows = (rng.standard_normal((n, d)) * 0.01).astype(np.float32)
        dense = (rng.standard_normal(D) * 0.01).astype(np.float32)
        tok = 0 if tokens is None else int(tokens[m])
        msgs.append(O.Message(tok, B, [ids], [rows], dense))
    return msgs


def pin_sync_closed_form(L, seed=3):
    """Zero staleness (all tokens = k): the step equals synchronous training on
    the concatenated global batch.  The reference here is linear algebra: the
    per-row gradient is D^-1 A^T G with A the occurrence-to-row incidence, G the
    stacked gradient rows and D the number of messages containing each row;
    the dense gradient is the mean of the M dense gradients.  The optimizer is
    applied in float64 and compared with a relative tolerance."""
    rng = np.random.default_rng(seed)
    V, d, D, M = 23, 3, 17, 5
    tb = O.TableSpec(V, d, O.OptSpec(O.ADAGRAD, 0.05, 0.1))
    orc = O.OracleGBA([tb], D, O.OptSpec(O.ADAGRAD, 0.02, 0.1), M, iota=0, seed=99,
                      library=L)
    for step in range(3):
        w0 = orc.tables[0].w.astype(np.float64).reshape(V, d).copy()
        a0 = orc.tables[0].s0.astype(np.float64).reshape(V, d).copy()
        dw0 = orc.dense.w.astype(np.float64).copy()
        da0 = orc.dense.s0.astype(np.float64).copy()
        msgs = random_messages(rng, M, V, d, D, 1, 9, tokens=[orc.k] * M)
        A = np.zeros((0, V))
        G = np.zeros((0, d))
        P = np.zeros((M, V))
        for m, msg in enumerate(msgs):
            inc = np.zeros((len(msg.ids[0]), V))
            inc[np.arange(len(msg.ids[0])), msg.ids[0]] = 1.0
            A = np.vstack([A, inc])
            G = np.vstack([G, msg.rows[0].astype(np.float64)])
            P[m, msg.ids[0]] = 1.0
        c = P.sum(axis=0)
        S = A.T @ G
        touched = c > 0
        ghat = np.zeros((V, d))
        ghat[touched] = S[touched] / c[touched, None]
        a1 = a0 + ghat**2
        with np.errstate(divide="ignore", invalid="ignore"):  # untouched rows are not used
            w1 = np.where(touched[:, None], w0 - 0.05 * ghat / np.sqrt(a1), w0)
        a1 = np.where(touched[:, None], a1, a0)
        gbar = np.mean(np.stack([m.dense.astype(np.float64) for m in msgs]), axis=0)
        da1 = da0 + gbar**2
        dw1 = dw0 - 0.02 * gbar / np.sqrt(da1)
        for msg in msgs:
            orc.push(msg)
        assert orc.try_apply() == 1
        assert orc.last_keep.tolist() == [1] * M
        w = orc.tables[0].w.astype(np.float64).reshape(V, d)
        a = orc.tables[0].s0.astype(np.float64).reshape(V, d)
        np.testing.assert_allclose(w, w1, rtol=2e-6, atol=1e-9)
        np.testing.assert_allclose(a, a1, rtol=2e-6, atol=1e-12)
        np.testing.assert_allclose(orc.dense.w, dw1, rtol=2e-6, atol=1e-9)
        np.testing.assert_allclose(orc.dense.s0, da1, rtol=2e-6, atol=1e-12)
        assert orc.last_count[0].tolist() == c.astype(np.int64).tolist()


def pin_decay_boundary(L):
    """Eq. (1): staleness exactly iota keeps, iota + 1 drops, for the dense
    decision (k - token) and the row decision (tag - token) separately; a row
    not updated since the token is kept even when its message is dense-dropped;
    iota = INT32_MAX keeps everything (BSP)."""
    for iota in (0, 1, 3, O.INT32_MAX):
        V, d, D = 6, 2, 3
        tb = O.TableSpec(V, d, O.OptSpec(O.ADAGRAD, 0.01, 0.1))
        orc = O.OracleGBA([tb], D, O.OptSpec(O.ADAGRAD, 0.01, 0.1), 1, iota=iota, seed=5,
                          library=L)
        z = np.zeros(D, np.float32)
        # Each warm-up step is fresh and updates row 1, so afterwards tag(row 1) = k.
        depth = 6 if iota == O.INT32_MAX else iota + 2
        for _ in range(depth):
            orc.push(O.Message(orc.k, 1, [np.array([1], np.int64)],
                               [np.ones((1, d), np.float32)], z))
            assert orc.try_apply() == 1
        assert int(orc.tables[0].ver[1]) == orc.k
        # (lag, dense kept, row 1 kept, row 4 kept); row 4 has tag 0 (never updated)
        cases = [(0, 1, 1, 1), (orc.k, 1, 1, 1)] if iota == O.INT32_MAX else \
            [(iota, 1, 1, 1), (iota + 1, 0, 0, 1)]
        for lag, want_dense, want_row1, want_row4 in cases:
            k = orc.k
            token = k - lag
            assert token >= 0
            orc.tables[0].ver[4] = 0
            orc.push(O.Message(token, 1, [np.array([1, 4], np.int64)],
                               [np.ones((2, d), np.float32)], z))
            assert orc.try_apply() == 1
            assert orc.last_keep.tolist() == [want_dense], (iota, lag, orc.last_keep)
            assert int(orc.last_kept[0][1]) == want_row1, (iota, lag, "row1")
            assert int(orc.last_kept[0][4]) == want_row4, (iota, lag, "row4")
            assert int(orc.tables[0].ver[4]) == k + 1
            assert int(orc.tables[0].ver[1]) == (k + 1 if want_row1 else k)
    # negative staleness (token ahead of k) clamps to 0 and keeps
    tb = O.TableSpec(4, 1, O.OptSpec(O.ADAGRAD, 0.01, 0.1))
    orc = O.OracleGBA([tb], 1, O.OptSpec(O.ADAGRAD, 0.01, 0.1), 1, iota=0, seed=1, library=L)
    orc.push(O.Message(7, 1, [np.array([2], np.int64)], [np.ones((1, 1), np.float32)],
                       np.ones(1, np.float32)))
    assert orc.try_apply() == 1 and orc.last_keep.tolist() == [1]
    assert orc.last_stats["dense_stale_sum"] == 0


def pin_fifo_prefix(L):
    """Alg. 2: apply once at least the global batch is buffered, popping the
    oldest messages; the rest stay buffered."""
    tb = O.TableSpec(4, 1)
    orc = O.OracleGBA([tb], 1, O.OptSpec(), 4, iota=O.INT32_MAX, seed=0, library=L)
    one = np.ones(1, np.float32)
    for b in (1, 2):
        orc.push(O.Message(0, b, [np.array([0], np.int64)], [np.ones((1, 1), np.float32)], one))
    assert orc.try_apply() == 0 and orc.pull_version() == 0
    orc.push(O.Message(0, 2, [np.array([1], np.int64)], [np.ones((1, 1), np.float32)], one))
    orc.push(O.Message(0, 5, [np.array([2], np.int64)], [np.ones((1, 1), np.float32)], one))
    assert orc.try_apply() == 1
    assert len(orc.fifo) == 1 and orc.fifo[0].local_batch == 5
    assert orc.last_count[0].tolist() == [2, 1, 0, 0]
    assert orc.try_apply() == 1 and len(orc.fifo) == 0
    assert orc.try_apply() == 0


def pin_order_invariance(L, seed=11):
    """Permuting the messages of a global batch leaves every integer output
    identical and floats within one float32 ulp (double accumulation)."""
    rng = np.random.default_rng(seed)
    V, d, D, M = 9, 4, 11, 4
    base = random_messages(rng, M, V, d, D, 0, 7, tokens=[0, 1, 2, 0])
    results = []
    for perm in ([0, 1, 2, 3], [3, 1, 0, 2], [2, 3, 1, 0]):
        tb = O.TableSpec(V, d, O.OptSpec(O.ADAM, 0.001))
        orc = O.OracleGBA([tb], D, O.OptSpec(O.ADAM, 0.001), M, iota=1, seed=4, library=L)
        # two warm-up steps so tags differ across rows
        for s in range(2):
            for msg in random_messages(np.random.default_rng(100 + s), M, V, d, D, 1, 5,
                                       tokens=[s] * M):
                orc.push(msg)
            orc.try_apply()
        for i in perm:
            orc.push(base[i])
        orc.try_apply()
        results.append((orc.tables[0].w.copy(), orc.tables[0].s0.copy(),
                        orc.tables[0].ver.copy(), orc.last_count[0].copy(),
                        orc.last_kept[0].copy(), orc.dense.w.copy(),
                        sorted(orc.last_keep.tolist()), orc.last_stats))
    ref = results[0]
    for r in results[1:]:
        assert np.array_equal(r[2], ref[2]) and np.array_equal(r[3], ref[3])
        assert np.array_equal(r[4], ref[4]) and r[6] == ref[6] and r[7] == ref[7]
        for a, b in ((r[0], ref[0]), (r[1], ref[1]), (r[5], ref[5])):
            ulp = np.spacing(np.abs(b).astype(np.float32))
            assert np.all(np.abs(a - b) <= ulp)


# ---------------------------------------------------------------------------
def brute_force_run(specs, D, dense_opt, G, iota, steps, seed, keys=None):
    """A literal restatement for tiny inputs: enumerate every (message,
    occurrence) pair, keep a dictionary per row, and round to float32 after
    every operation in the stated order.  keys[t] lists table t's row keys
    (default: 0..rows-1); a key x starts from the initial values of element
    x*d + j (modulo 2^64), so keys may be arbitrary 64-bit ids."""
    f32 = np.float32
    t_specs = specs
    if keys is None:
        keys = [range(sp.rows) for sp in t_specs]
    init_w = {}
    for t, sp in enumerate(t_specs):
        for x in keys[t]:
            for j in range(sp.dim):
                e = (int(x) * sp.dim + j) % 2**64
                init_w[(t, int(x), j)] = f32(O.init_weight(seed, O.table_tag(t), e))
    W = dict(init_w)
    S0 = {key: (f32(t_specs[key[0]].opt.init_acc) if t_specs[key[0]].opt.kind == O.ADAGRAD
                else f32(0)) for key in W}
    S1 = {key: f32(0) for key in W}
    ver = {(t, int(x)): 0 for t in range(len(t_specs)) for x in keys[t]}
    DW = [f32(O.init_weight(seed, O.dense_tag(), e)) for e in range(D)]
    DS0 = [f32(dense_opt.init_acc) if dense_opt.kind == O.ADAGRAD else f32(0)] * D
    DS1 = [f32(0)] * D

    def bc(beta, t):
        p = 1.0
        for _ in range(t):
            p = p * float(f32(beta))
        return f32(1.0 - p)

    def upd(opt, w, s0, s1, g, t):
        lr, b1, b2, eps = f32(opt.lr), f32(opt.beta1), f32(opt.beta2), f32(opt.eps)
        if opt.kind == O.ADAGRAD:
            a = f32(s0 + f32(g * g))
            return f32(w - f32(f32(lr * g) / f32(np.sqrt(a)))), a, s1
        m = f32(f32(b1 * s0) + f32(f32(f32(1) - b1) * g))
        v = f32(f32(b2 * s1) + f32(f32(f32(1) - b2) * f32(g * g)))
        mh = f32(m / bc(opt.beta1, t))
        vh = f32(v / bc(opt.beta2, t))
        return f32(w - f32(f32(lr * mh) / f32(f32(np.sqrt(vh)) + eps))), m, v

    k = 0
    for batch in steps:
        M = len(batch)
        f = [1 if max(0, k - m.token) <= iota else 0 for m in batch]
        for e in range(D):
            s = 0.0
            for m in range(M):
                if f[m]:
                    s += float(batch[m].dense[e])
            g = f32(f32(s) / f32(M))
            DW[e], DS0[e], DS1[e] = upd(dense_opt, DW[e], DS0[e], DS1[e], g, k + 1)
        for t, sp in enumerate(t_specs):
            pairs = {}   # row -> list of (m, keep, grad row)
            for m, msg in enumerate(batch):
                for o, i in enumerate(msg.ids[t]):
                    x = int(i)
                    keep = max(0, ver[(t, x)] - msg.token) <= iota
                    pairs.setdefault(x, []).append((m, keep, msg.rows[t][o]))
            for x, occ in sorted(pairs.items()):
                if not any(kp for _, kp, _ in occ):
                    continue
                c = len({m for m, _, _ in occ})
                for j in range(sp.dim):
                    s = 0.0
                    for _, kp, row in occ:
                        if kp:
                            s += float(row[j])
                    g = f32(f32(s) / f32(c))
                    key = (t, x, j)
                    W[key], S0[key], S1[key] = upd(sp.opt, W[key], S0[key], S1[key], g, k + 1)
                ver[(t, x)] = k + 1
        k += 1
    return W, S0, S1, ver, DW, DS0, DS1


def pin_brute_force(L, seed=21):
    """Bit-for-bit agreement with the brute-force restatement on tiny inputs."""
    rng = np.random.default_rng(seed)
    for kind in (O.ADAGRAD, O.ADAM):
        V, d, D, M = 8, 3, 4, 4
        specs = [O.TableSpec(V, d, O.OptSpec(kind, 0.03)), O.TableSpec(5, 2, O.OptSpec(kind, 0.02))]
        dopt = O.OptSpec(kind, 0.01)
        orc = O.OracleGBA(specs, D, dopt, M, iota=1, seed=77, library=L)
        steps = []
        for s in range(3):
            toks = [max(0, s - int(rng.integers(0, 3))) for _ in range(M)]
            batch = []
            for m in range(M):
                ids, rows = [], []
                for sp in specs:
                    n = int(rng.integers(0, 5))
                    ids.append(rng.integers(0, sp.rows, n).astype(np.int64))
                    rows.append((rng.standard_normal((n, sp.dim)) * 0.5).astype(np.float32))
                batch.append(O.Message(toks[m], 1, ids, rows,
                                       (rng.standard_normal(D) * 0.5).astype(np.float32)))
            steps.append(batch)
            for msg in batch:
                orc.push(msg)
            assert orc.try_apply() == 1
        W, S0, S1, ver, DW, DS0, DS1 = brute_force_run(specs, D, dopt, M, 1, steps, 77)
        for t, sp in enumerate(specs):
            w = orc.tables[t].w.reshape(sp.rows, sp.dim)
            s0 = orc.tables[t].s0.reshape(sp.rows, sp.dim)
            for x in range(sp.rows):
                assert orc.tables[t].ver[x] == ver[(t, x)]
                for j in range(sp.dim):
                    assert w[x, j] == W[(t, x, j)], ("w", kind, t, x, j)
                    assert s0[x, j] == S0[(t, x, j)], ("s0", kind, t, x, j)
                    if kind == O.ADAM:
                        assert orc.tables[t].s1.reshape(sp.rows, sp.dim)[x, j] == S1[(t, x, j)]
        assert orc.dense.w.tolist() == [float(v) for v in DW]
        assert orc.dense.s0.tolist() == [float(v) for v in DS0]


def pin_hash_ids(L, seed=41):
    """Tables of arbitrary 64-bit ids (id mode 2): with ids in [0, V) they
    evolve bit for bit as DIRECT tables; with ids anywhere in the int64 range
    (negative, beyond 2^32, repeated within a message) they agree bit for bit
    with the brute-force restatement keyed by id; the reserved id INT64_MIN
    is an error."""
    rng = np.random.default_rng(seed)
    V, d, D, M = 6, 3, 2, 4
    for kind in (O.ADAGRAD, O.ADAM):
        # small ids: the same as row = id
        direct = O.OracleGBA([O.TableSpec(V, d, O.OptSpec(kind, 0.03))], D,
                             O.OptSpec(kind, 0.01), M, iota=1, seed=5, library=L)
        hashed = O.OracleGBA([O.TableSpec(V, d, O.OptSpec(kind, 0.03), id_mode=2)], D,
                             O.OptSpec(kind, 0.01), M, iota=1, seed=5, library=L,
                             track_rows=[np.arange(V, dtype=np.int64)])
        for s in range(3):
            for m in range(M):
                n = int(rng.integers(0, 5))
                msg = O.Message(max(0, s - int(rng.integers(0, 3))), 1,
                                [rng.integers(0, V, n).astype(np.int64)],
                                [(rng.standard_normal((n, d)) * .5).astype(np.float32)],
                                (rng.standard_normal(D) * .5).astype(np.float32))
                direct.push(msg)
                hashed.push(msg)
            assert direct.try_apply() == 1 and hashed.try_apply() == 1
        assert direct.tables[0].w.tobytes() == hashed.tables[0].w.tobytes()
        assert direct.tables[0].s0.tobytes() == hashed.tables[0].s0.tobytes()
        assert direct.tables[0].ver.tolist() == hashed.tables[0].ver.tolist()

        # arbitrary ids against the brute force keyed by id
        pool = np.array([-2**63 + 1, -7, 0, 3, 2**33 + 5, 2**62 + 11], np.int64)
        spec = O.TableSpec(len(pool), d, O.OptSpec(kind, 0.03), id_mode=2)
        dopt = O.OptSpec(kind, 0.01)
        orc = O.OracleGBA([spec], D, dopt, M, iota=1, seed=9, library=L,
                          track_rows=[np.sort(pool)])
        steps = []
        for s in range(3):
            batch = []
            for m in range(M):
                n = int(rng.integers(0, 5))
                ids = pool[rng.integers(0, len(pool), n)]
                batch.append(O.Message(max(0, s - int(rng.integers(0, 3))), 1, [ids],
                                       [(rng.standard_normal((n, d)) * .5).astype(np.float32)],
                                       (rng.standard_normal(D) * .5).astype(np.float32)))
            steps.append(batch)
            for msg in batch:
                orc.push(msg)
            assert orc.try_apply() == 1
        W, S0, S1, ver, DW, _, _ = brute_force_run([spec], D, dopt, M, 1, steps, 9,
                                                    keys=[sorted(int(x) for x in pool)])
        w = orc.tables[0].w.reshape(-1, d)
        s0 = orc.tables[0].s0.reshape(-1, d)
        for r, x in enumerate(sorted(int(x) for x in pool)):
            assert orc.tables[0].ver[r] == ver[(0, x)], ("ver", kind, x)
            for j in range(d):
                assert w[r, j] == W[(0, x, j)], ("w", kind, x, j)
                assert s0[r, j] == S0[(0, x, j)], ("s0", kind, x, j)
        assert orc.dense.w.tolist() == [float(v) for v in DW]

    # the reserved id
    orc = O.OracleGBA([O.TableSpec(4, 1, id_mode=2)], 1, O.OptSpec(), 1, library=L,
                      track_rows=[np.arange(4, dtype=np.int64)])
    orc.push(O.Message(0, 1, [np.array([-2**63], np.int64)], [np.ones((1, 1), np.float32)],
                       np.ones(1, np.float32)))
    try:
        orc.try_apply()
    except ValueError:
        pass
    else:
        raise AssertionError("the reserved id was accepted")


def pin_modulo_ids(L, seed=51):
    """MODULO tables (hashing trick): a table fed arbitrary int64 ids, negative
    ones included, evolves bit for bit as a DIRECT table fed the residues of
    the ids read as unsigned 64-bit integers, computed here with Python's
    exact integer arithmetic."""
    rng = np.random.default_rng(seed)
    V, d, D, M = 7, 2, 3, 3
    for kind in (O.ADAGRAD, O.ADAM):
        mod = O.OracleGBA([O.TableSpec(V, d, O.OptSpec(kind, 0.03), id_mode=1)], D,
                          O.OptSpec(kind, 0.01), M, iota=1, seed=4, library=L)
        direct = O.OracleGBA([O.TableSpec(V, d, O.OptSpec(kind, 0.03))], D,
                             O.OptSpec(kind, 0.01), M, iota=1, seed=4, library=L)
        for s in range(3):
            for m in range(M):
                n = int(rng.integers(0, 6))
                ids = rng.integers(-2**63, 2**63 - 1, n, dtype=np.int64)
                res = np.array([(int(x) % 2**64) % V for x in ids], np.int64)
                rows = (rng.standard_normal((n, d)) * .5).astype(np.float32)
                dense = (rng.standard_normal(D) * .5).astype(np.float32)
                tok = max(0, s - int(rng.integers(0, 3)))
                mod.push(O.Message(tok, 1, [ids], [rows], dense))
                direct.push(O.Message(tok, 1, [res], [rows], dense))
            assert mod.try_apply() == 1 and direct.try_apply() == 1
        assert mod.tables[0].w.tobytes() == direct.tables[0].w.tobytes()
        assert mod.tables[0].s0.tobytes() == direct.tables[0].s0.tobytes()
        assert mod.tables[0].ver.tolist() == direct.tables[0].ver.tolist()


ALL_PINS = [pin_hand_adagrad, pin_hand_rule_options, pin_hand_decay_variants,
            pin_decay_special_cases, pin_hand_adam, pin_sync_closed_form, pin_decay_boundary,
            pin_fifo_prefix, pin_order_invariance, pin_brute_force, pin_hash_ids, pin_modulo_ids]


def pin_init_published(L):
    """The counter-based initial weights: SplitMix64's published outputs and the
    stated mapping of the top 24 bits to [-1/16, 1/16)."""
    g = load_golden()["splitmix64_seed0"]
    gamma = 0x9E3779B97F4A7C15
    for i, want in enumerate(g["outputs"]):
        assert int(L.gbao_splitmix64((i * gamma) % 2**64)) == int(want, 16)
    # e = 0, tag 0, seed = gamma: hash is output 1 of the published stream
    h = int(g["outputs"][1], 16)
    want = ((h >> 40) - 2**23) * 2.0**-27
    assert float(L.gbao_init_weight(gamma, 0, 0)) == want
