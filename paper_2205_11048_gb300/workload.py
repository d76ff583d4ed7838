"""Seeded synthetic message streams shaped like the paper's workloads.

This module generates inputs only: worker messages with a token, a local
batch, per-table feature ids and their gradient rows, and a dense gradient.
It holds none of the aggregation arithmetic; both the CUDA path and the CPU
oracle consume exactly the tensors it returns.

The paper trains on Criteo-1TB, Alimama and a private dataset (Sec. 5.1,
Table 1), none of which is available here.  The streams below stand in for
them: feature ids follow a bounded Zipf law per field (the skew of Fig. 4 and
Insight 2), each field maps ranks to rows through its own salted bijection so
hot rows differ per field, gradients are N(0, 0.01^2), and per-message
staleness follows the distributions named for each workload (Table 3 reports
GBA's average dense staleness 0.12-0.21 with maxima 9-11).

Everything is produced with torch on the requested device from a
``torch.Generator`` seeded per (workload seed, step), so a stream is
reproducible on a given device.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field, replace

import torch

ADAGRAD = 0
ADAM = 1
DIRECT = 0
MODULO = 1
HASH = 2


@dataclass(frozen=True)
class OptCfg:
    kind: int = ADAGRAD
    lr: float = 0.01
    init_acc: float = 0.1
    beta1: float = 0.9
    beta2: float = 0.999
    eps: float = 1e-8


@dataclass(frozen=True)
class TableCfg:
    rows: int
    dim: int
    fields: int               # feature fields that look up this table
    ids_per_field: float = 0  # 0: one id per sample and field; >0: Poisson mean
    zipf: float = 1.05        # exponent of the bounded Zipf law over ranks 1..rows
    id_mode: int = DIRECT     # DIRECT: id is the row; MODULO / HASH: 64-bit hashed id
    opt: OptCfg = field(default_factory=OptCfg)


@dataclass(frozen=True)
class StaleCfg:
    kind: str = "fresh"        # fresh | geometric | pareto
    mean: float = 0.0          # geometric mean on {0, 1, ...}
    straggler_frac: float = 0.0
    straggler_lo: int = 5
    straggler_hi: int = 20
    alpha: float = 1.5         # Pareto shape, x_m = 1
    cap: int = 50


@dataclass(frozen=True)
class WorkloadCfg:
    name: str
    M: int                    # messages per global batch
    B: int                    # local batch of every message
    tables: tuple
    D: int                    # dense parameters
    dense_opt: OptCfg
    stale: StaleCfg
    iota: int = 4
    seed: int = 0
    steps: int = 20

    @property
    def G(self) -> int:
        return self.M * self.B

    def ids_per_msg(self, t: int) -> float:
        tb = self.tables[t]
        per = tb.ids_per_field if tb.ids_per_field > 0 else 1
        return self.B * tb.fields * per

    def max_ids_per_msg(self, t: int) -> int:
        """An upper bound on one message's ids for table t (6 sigma over Poisson)."""
        mean = self.ids_per_msg(t)
        if self.tables[t].ids_per_field > 0:
            return int(mean + 6 * math.sqrt(mean) + 64)
        return int(mean)


ADAM_DENSE = OptCfg(kind=ADAM, lr=0.001)


def config(n: int) -> WorkloadCfg:
    """The five workloads, at full size (n = 1..5)."""
    if n == 1:
        return WorkloadCfg("c1-tiny", M=4, B=256,
                           tables=(TableCfg(100_000, 16, 26, 0, 1.1),),
                           D=200_000, dense_opt=OptCfg(ADAGRAD, 0.01),
                           stale=StaleCfg("fresh"), iota=4, seed=0, steps=20)
    if n == 2:
        return WorkloadCfg("c2-onehot-1e7x32", M=32, B=1024,
                           tables=(TableCfg(10_000_000, 32, 26, 0, 1.05),),
                           D=1_000_000, dense_opt=ADAM_DENSE,
                           stale=StaleCfg("geometric", mean=1.0, straggler_frac=0.1),
                           iota=4, seed=1, steps=20)
    if n == 3:
        return WorkloadCfg("c3-multihot-4x1.25e7x16", M=64, B=1024,
                           tables=tuple(TableCfg(12_500_000, 16, 25, 20.0, 1.2)
                                        for _ in range(4)),
                           D=2_000_000, dense_opt=ADAM_DENSE,
                           stale=StaleCfg("geometric", mean=2.0), iota=4, seed=2, steps=20)
    if n == 4:
        return WorkloadCfg("c4-dense-heavy-64M", M=16, B=1024,
                           tables=(TableCfg(1_000_000, 64, 40, 0, 1.05),),
                           D=64_000_000, dense_opt=ADAM_DENSE,
                           stale=StaleCfg("pareto", alpha=1.5, cap=50), iota=4, seed=3,
                           steps=20)
    if n == 5:
        return WorkloadCfg("c5-large-2e8x64-hashed", M=128, B=1024,
                           tables=(TableCfg(200_000_000, 64, 40, 0, 1.05, MODULO),),
                           D=8_000_000, dense_opt=ADAM_DENSE,
                           stale=StaleCfg("geometric", mean=3.0, straggler_frac=0.2),
                           iota=4, seed=4, steps=20)
    raise ValueError(n)


def reduced(n: int) -> WorkloadCfg:
    """The same five workloads scaled down so the oracle runs them in seconds
    while keeping their structure (tables, fields, skew, staleness, optimizers)."""
    c = config(n)
    if n == 1:
        return c
    if n == 2:
        return replace(c, name="c2-reduced", M=8, B=96,
                       tables=(replace(c.tables[0], rows=200_003),), D=50_001)
    if n == 3:
        return replace(c, name="c3-reduced", M=6, B=16,
                       tables=tuple(replace(tb, rows=30_011 + 7 * i)
                                    for i, tb in enumerate(c.tables)), D=20_003)
    if n == 4:
        return replace(c, name="c4-reduced", M=5, B=64,
                       tables=(replace(c.tables[0], rows=50_000),), D=300_007)
    if n == 5:
        return replace(c, name="c5-reduced", M=12, B=48,
                       tables=(replace(c.tables[0], rows=1_000_003),), D=40_000)
    raise ValueError(n)


# --------------------------------------------------------------------------
# Samplers
# --------------------------------------------------------------------------

def _helper1(x: torch.Tensor) -> torch.Tensor:
    """log1p(x) / x, continuous at 0."""
    small = x.abs() < 1e-8
    safe = torch.where(small, torch.ones_like(x), x)
    return torch.where(small, 1.0 - x * (0.5 - x * (1.0 / 3.0)), torch.log1p(safe) / safe)


def _helper2(x: torch.Tensor) -> torch.Tensor:
    """expm1(x) / x, continuous at 0."""
    small = x.abs() < 1e-8
    safe = torch.where(small, torch.ones_like(x), x)
    return torch.where(small, 1.0 + x * 0.5 * (1.0 + x * (1.0 / 3.0)), torch.expm1(safe) / safe)


def zipf_ranks(n: int, N: int, s: float, gen: torch.Generator, device) -> torch.Tensor:
    """n draws of a bounded Zipf law P(r) ~ r^-s on r = 1..N.

    Rejection-inversion of Hormann and Derflinger (1996): invert the integral
    H of the hat x^-s, round to the nearest integer, and accept unless the
    point falls in the part of the hat above the histogram bar."""
    one_minus_s = 1.0 - s

    def H(x):
        lx = torch.log(x)
        return _helper2(one_minus_s * lx) * lx

    def Hinv(y):
        t = torch.clamp(y * one_minus_s, min=-1.0)
        return torch.exp(_helper1(t) * y)

    def h(x):
        return torch.exp(-s * torch.log(x))

    f64 = dict(dtype=torch.float64, device=device)
    Hx1 = float(H(torch.tensor(1.5, **f64))) - 1.0
    HN = float(H(torch.tensor(N + 0.5, **f64)))
    sq = 2.0 - float(Hinv(H(torch.tensor(2.5, **f64)) - h(torch.tensor(2.0, **f64))))
    out = torch.empty(n, dtype=torch.int64, device=device)
    todo = torch.arange(n, device=device)
    while todo.numel() > 0:
        u = HN + torch.rand(todo.numel(), generator=gen, **f64) * (Hx1 - HN)
        x = Hinv(u)
        k = torch.clamp(torch.round(x), 1, N)
        ok = ((k - x) <= sq) | (u >= H(k + 0.5) - h(k))
        out[todo[ok]] = k[ok].to(torch.int64)
        todo = todo[~ok]
    return out


_MASK64 = (1 << 64) - 1


def _s64(v: int) -> int:
    v &= _MASK64
    return v - (1 << 64) if v >> 63 else v


def _lsr(z: torch.Tensor, s: int) -> torch.Tensor:
    return (z >> s) & ((1 << (64 - s)) - 1)


def hash64(x: torch.Tensor) -> torch.Tensor:
    """SplitMix64 output for state x (int64 two's complement, wrapping)."""
    z = x + _s64(0x9E3779B97F4A7C15)
    z = (z ^ _lsr(z, 30)) * _s64(0xBF58476D1CE4E5B9)
    z = (z ^ _lsr(z, 27)) * _s64(0x94D049BB133111EB)
    return z ^ _lsr(z, 31)


def _field_params(cfg: WorkloadCfg, t: int):
    """Per-field bijection rank -> row (a*(r-1) + b mod V, gcd(a, V) = 1) and hash salts."""
    tb = cfg.tables[t]
    g = torch.Generator().manual_seed(cfg.seed * 7919 + 104729 * (t + 1))
    params = []
    for _ in range(tb.fields):
        while True:
            a = int(torch.randint(1, max(2, tb.rows), (1,), generator=g))
            if math.gcd(a, tb.rows) == 1:
                break
        b = int(torch.randint(0, max(1, tb.rows), (1,), generator=g))
        salt = int(torch.randint(0, 2**62, (1,), generator=g))
        params.append((a, b, salt))
    return params


def _step_gen(cfg: WorkloadCfg, step: int, device, tag: int) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed((cfg.seed * 1_000_003 + step * 7_919 + tag * 104_729) & (2**62 - 1))
    return g


def draw_staleness(cfg: WorkloadCfg, n: int, gen: torch.Generator) -> list:
    """Per-message staleness in global steps (host ints)."""
    st = cfg.stale
    if st.kind == "fresh":
        return [0] * n
    if st.kind == "geometric":
        p = 1.0 / (1.0 + st.mean)
        s = torch.empty(n, dtype=torch.float64).geometric_(p, generator=gen) - 1
        if st.straggler_frac > 0:
            strag = torch.rand(n, generator=gen, dtype=torch.float64) < st.straggler_frac
            lag = torch.randint(st.straggler_lo, st.straggler_hi + 1, (n,), generator=gen)
            s = torch.where(strag, lag.to(torch.float64), s)
        return [int(v) for v in s]
    if st.kind == "pareto":
        u = 1.0 - torch.rand(n, generator=gen, dtype=torch.float64)  # (0, 1]
        x = u.pow(-1.0 / st.alpha)                                    # Pareto(x_m = 1)
        s = torch.clamp(torch.floor(x) - 1, 0, st.cap)
        return [int(v) for v in s]
    raise ValueError(st.kind)


def tokens_for_step(cfg: WorkloadCfg, k_apply: int, salt: int = 0) -> list:
    """Tokens of the M messages that global step k_apply will consume:
    token = max(0, k_apply - staleness)."""
    g = torch.Generator().manual_seed((cfg.seed * 31 + k_apply * 1_000_033 + salt) & (2**62 - 1))
    return [max(0, k_apply - s) for s in draw_staleness(cfg, cfg.M, g)]


def message_ids(cfg: WorkloadCfg, t: int, gen: torch.Generator, device) -> torch.Tensor:
    """Feature ids of one message for table t, field-major."""
    tb = cfg.tables[t]
    params = _field_params(cfg, t)
    out = []
    for (a, b, salt) in params:
        if tb.ids_per_field > 0:
            lam = torch.full((cfg.B,), float(tb.ids_per_field), dtype=torch.float32,
                             device=device)
            n = int(torch.poisson(lam, generator=gen).sum())
        else:
            n = cfg.B
        r = zipf_ranks(n, tb.rows, tb.zipf, gen, device)
        if tb.id_mode == DIRECT:
            out.append((a * (r - 1) + b) % tb.rows)
        else:
            out.append(hash64(r ^ salt))
    if not out:
        return torch.empty(0, dtype=torch.int64, device=device)
    return torch.cat(out)


def generate_step(cfg: WorkloadCfg, k_apply: int, device="cpu", tokens=None) -> list:
    """The M messages consumed by global step k_apply, in arrival order.

    Returns a list of dicts: token, local_batch, ids (per table int64 [n]),
    rows (per table float32 [n, d]), dense (float32 [D])."""
    device = torch.device(device)
    gen = _step_gen(cfg, k_apply, device, 1)
    if tokens is None:
        tokens = tokens_for_step(cfg, k_apply)
    msgs = []
    for m in range(cfg.M):
        ids, rows = [], []
        for t, tb in enumerate(cfg.tables):
            i = message_ids(cfg, t, gen, device)
            g = torch.randn(i.numel(), tb.dim, generator=gen, device=device,
                            dtype=torch.float32) * 0.01
            ids.append(i)
            rows.append(g)
        dense = torch.randn(cfg.D, generator=gen, device=device, dtype=torch.float32) * 0.01
        msgs.append(dict(token=int(tokens[m]), local_batch=cfg.B, ids=ids, rows=rows,
                         dense=dense))
    perm = torch.randperm(cfg.M, generator=torch.Generator().manual_seed(
        cfg.seed * 13 + k_apply)).tolist()
    return [msgs[i] for i in perm]
