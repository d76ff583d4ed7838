"""Benchmark of the GBA aggregate-and-apply step on GB300.

One "step" is one global step of the hot path: message weights (Eq. (1)),
the radix sort + dedup of the global batch's ids, the per-row decayed
segment-sum and row update, and the dense reduce + optimizer.

Default workload: the largest single-GPU one -- 128 workers of local batch
1024 (global batch 131,072), one 2e8 x 64 embedding table of hashed 64-bit ids
(MODULO rows) with its Adagrad accumulator, 40 one-hot Zipf(1.05) fields, 8M
dense parameters with Adam, geometric staleness (mean 3) with 20% stragglers.
Inputs are synthetic (seeded Zipf ids, N(0, 0.01^2) gradients) and resident in
HBM before the timed region; messages are pushed by reference, two distinct
global batches in turn (each larger than the 129 MB L2), with fresh tokens
every step.  The timed region ends with the library's streams joined into the
timing stream, so it covers all of the steps' work.

Prints one JSON line (rank 0).  --impl reference times the CPU oracle instead,
on the same workload description.
"""
from __future__ import annotations

import argparse
import ctypes
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "global-batch aggregate+apply steps/s; applied grad rows/s; HBM GB/s vs ~8 TB/s peak"
R_BATCHES = 2
L2_BYTES = 129e6  # GB300 L2


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            j = json.load(f)
        return float(j["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


def workload_cfg(n, id_mode="as-configured", rows=None, dense=None):
    """Workload n; id_mode "hash" turns every table into an expandable hash
    table of 64-bit ids (initial capacity: the next power of two at or above
    twice its rows).  rows / dense shrink the tables' rows and the dense size
    while keeping the message, id and staleness structure: a case of the same
    shape small enough for a multi-pass profiler capture."""
    from paper_2205_11048_gb300 import workload as W
    cfg = W.config(n)
    if rows is not None or dense is not None:
        r = rows if rows is not None else cfg.tables[0].rows
        D = dense if dense is not None else cfg.D
        cfg = W.replace(cfg, name=f"{cfg.name}-shaped-{r}x{cfg.tables[0].dim}-D{D}", D=D,
                        tables=tuple(W.replace(t, rows=r) for t in cfg.tables))
    if id_mode == "hash":
        def cap(r):
            c = 1024
            while c < 2 * r:
                c *= 2
            return c
        cfg = W.replace(cfg, name=cfg.name + "-hash-ids",
                        tables=tuple(W.replace(t, id_mode=W.HASH, rows=cap(t.rows))
                                     for t in cfg.tables))
        state = sum(t.rows * (4 * t.dim * (2 if t.opt.kind == 0 else 3) + 12) for t in cfg.tables)
        if state > 150e9:
            raise SystemExit(f"--id-mode hash: {state / 1e9:.0f} GB of table state at the initial "
                             "capacity; use --shape-rows for a smaller case")
    return cfg


def alg_bytes(cfg, st_delta, steps):
    """Algorithmic bytes per step by kernel (the bytes the method must move):
    ids 8 B per occurrence (sort), kept gradient rows 4d B, per applied row its
    state read + written (2 * S_opt * 4d B) and tag (8 B), dense: kept messages'
    gradients 4D B each plus the dense state read + written (2 * S_opt * 4D).
    The tables of every workload here share one width and optimizer; the
    counters are summed over tables."""
    assert all(t.dim == cfg.tables[0].dim and t.opt.kind == cfg.tables[0].opt.kind
               for t in cfg.tables), "tables of different widths or optimizers"
    tb = cfg.tables[0]
    d = tb.dim
    s_opt_rows = 2 if tb.opt.kind == 0 else 3
    s_opt_dense = 2 if cfg.dense_opt.kind == 0 else 3
    occ = st_delta["occurrences"] / steps
    occ_kept = st_delta["occurrences_kept"] / steps
    u_app = st_delta["rows_applied"] / steps
    m_kept = st_delta["msgs_kept"] / steps
    b = {
        "sort": 8.0 * occ,
        "rows": 4.0 * d * occ_kept + 2 * s_opt_rows * 4.0 * d * u_app + 8.0 * u_app,
        "dense": 4.0 * cfg.D * m_kept + 2 * s_opt_dense * 4.0 * cfg.D,
    }
    b["total"] = b["sort"] + b["rows"] + b["dense"]
    return b, dict(occ=occ, occ_kept=occ_kept, u_applied=u_app, m_kept=m_kept,
                   u_touched=st_delta["rows_touched"] / steps)


class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index):
        self.p = None
        try:
            self.p = subprocess.Popen(
                ["nvidia-smi", "-i", str(device_index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, ValueError):
            self.p = None

    def stop(self):
        if self.p is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.p.terminate()
        try:
            out, _ = self.p.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.p.kill()
            out, _ = self.p.communicate()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in out.strip().splitlines():
            parts = [x.strip() for x in ln.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[4:8]):
                if v.lower() == "active":
                    reasons.add(nm)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": sorted(reasons),
                "samples": len(sm)}


def _code_only(text):
    """C/CUDA source without its comments and blank lines (string literals in
    these files hold no comment markers)."""
    import re
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    text = re.sub(r"//[^\n]*", "", text)
    return "\n".join(ln.rstrip() for ln in text.splitlines() if ln.strip())


def source_sha(files):
    """Hash of the code (comments excluded) of a kernel class's sources."""
    h = hashlib.sha256()
    for f in files:
        with open(os.path.join(ROOT, f), encoding="utf-8") as fh:
            h.update(_code_only(fh.read()).encode())
    return h.hexdigest()[:16]


KERNEL_SOURCES = {
    "rows": ["paper_2205_11048_gb300/csrc/gba_rows.cu", "paper_2205_11048_gb300/csrc/gba_internal.cuh"],
    "dense": ["paper_2205_11048_gb300/csrc/gba_dense.cu", "paper_2205_11048_gb300/csrc/gba_internal.cuh"],
    "sort": ["paper_2205_11048_gb300/csrc/gba_sort.cu", "paper_2205_11048_gb300/csrc/gba_internal.cuh"],
}


def measured_traffic(kernel, workload):
    """DRAM bytes per global step of a kernel class (all its launches in one
    step) from the committed ncu launch list, if the class's sources are
    unchanged since the capture."""
    p = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(p):
        return None
    with open(p) as f:
        j = json.load(f)
    e = j.get(workload, {}).get(kernel)
    if not e or e.get("source_sha") != source_sha(KERNEL_SOURCES[kernel]):
        return None
    return e.get("dram_bytes_per_step")


def max_over_ranks(x: float, pg, device="cpu") -> float:
    """The largest value of x over all ranks (x itself without a process group)."""
    if pg is None:
        return float(x)
    import torch
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    pg.all_reduce(t, op=pg.ReduceOp.MAX)
    return float(t.item())


def job_throughput(steps_per_rank: int, world: int, max_elapsed_ms: float) -> float:
    """Whole-job steps/s: every rank's steps over the slowest rank's time."""
    return steps_per_rank * world / (max_elapsed_ms / 1e3)


def dist_setup():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def dense_traffic(cfg, per, mode):
    """Algorithmic dense bytes of one step, split into what the pushes move
    and what the apply moves.  Buffered (messages pushed by reference): the
    apply reads every kept message's gradient (4D each) and reads and writes
    the state.  Eager: a kept push reads its gradient and updates the step's
    compensated accumulator pair (4D + 8D + 8D; the first kept push of a step
    only writes it, 4D + 8D), the apply reads the pair (8D) and the state."""
    D = cfg.D
    s_opt = 2 if cfg.dense_opt.kind == 0 else 3
    state = 2 * s_opt * 4 * D
    m_kept = per["m_kept"]
    if mode == "eager":
        push = (12 * D + 20 * D * max(0.0, m_kept - 1)) / max(m_kept, 1e-9) if m_kept else 0.0
        return {"mode": "eager", "bytes_per_kept_push": push,
                "bytes_per_apply": 8 * D + state, "bytes_per_step": push * m_kept + 8 * D + state,
                "buffer_bytes_per_pending_step": 8 * D}
    return {"mode": "buffered", "bytes_per_kept_push": 0.0,
            "bytes_per_apply": 4 * D * m_kept + state, "bytes_per_step": 4 * D * m_kept + state,
            "buffer_bytes_per_message": 4 * D}


def config_dict(cfg, ws):
    """The workload description both arms print (the same dict in each)."""
    in_bytes = cfg.M * (sum(cfg.ids_per_msg(t) * (8 + 4 * tb.dim)
                            for t, tb in enumerate(cfg.tables)) + 4 * cfg.D)
    return {"workload": cfg.name, "M": cfg.M, "B": cfg.B, "G": cfg.G,
            "tables": [[t.rows, t.dim] for t in cfg.tables], "dense": cfg.D,
            "iota": cfg.iota, "batches_in_turn": R_BATCHES,
            "l2": (f"inputs larger than L2: each global batch holds {in_bytes / 1e6:.0f} MB of "
                   f"ids and gradients, {R_BATCHES} distinct batches in turn"
                   if in_bytes > L2_BYTES else
                   f"inputs smaller than L2 (no flush): each global batch holds "
                   f"{in_bytes / 1e6:.1f} MB of ids and gradients, {R_BATCHES} distinct "
                   f"batches in turn"),
            "parallelism": f"replicas x{ws}"}


def touched_rows(cfg, batches_cpu):
    """Per table, the sorted rows that the batches' ids map to."""
    import numpy as np
    from tests import _harness as H
    out = []
    for t in range(len(cfg.tables)):
        rows = [H.rows_of(cfg, t, m["ids"][t].numpy()) for b in batches_cpu for m in b]
        out.append(np.unique(np.concatenate(rows)) if rows else np.zeros(0, np.int64))
    return out


def sample_ratio(cfg):
    """r such that 1/r of one global step is about a quarter second of the
    oracle on one core (it takes about 0.66 us per id occurrence and 1.2 ns per
    dense element and message on the Grace host)."""
    n = cfg.M * sum(cfg.ids_per_msg(t) for t in range(len(cfg.tables)))
    est = 0.66e-6 * n + 1.2e-9 * cfg.M * cfg.D
    return max(1, int(round(est / 0.25)))


def oracle_rate(cfg, batches_cpu, warmup, steps, r=None):
    """The CPU oracle, as it stands, one thread, on bounded samples of global
    steps of the workload: each step pushes the batches in turn (tokens drawn
    per step as on the GPU) restricted to 1/r of the work -- the id
    occurrences of the rows x with x mod r = 0 and the dense elements
    [0, ceil(D / r)).  Rows are independent of one another and of the dense
    part, so the oracle computes for them exactly what a full step computes.
    Steps/s of the full step = 1 / (r x seconds per sampled step).  State
    initialisation and the sampling of the messages are outside the timed
    part.  Returns (steps/s, description of the sample)."""
    import numpy as np

    from oracle import oracle as O
    from paper_2205_11048_gb300 import workload as W
    from tests import _harness as H
    r = sample_ratio(cfg) if r is None else int(r)
    track = [t[t % r == 0] for t in touched_rows(cfg, batches_cpu)]
    d_s = -(-cfg.D // r)
    orc_msgs = []
    for b in batches_cpu:
        mb = []
        for m in b:
            om = H.to_oracle(m)
            keep = [H.rows_of(cfg, t, om.ids[t]) % r == 0 for t in range(len(cfg.tables))]
            mb.append(O.Message(om.token, om.local_batch, [x[k] for x, k in zip(om.ids, keep)],
                                [x[k] for x, k in zip(om.rows, keep)], om.dense))
        orc_msgs.append(mb)
    t0 = time.perf_counter()
    orc = H.make_oracle(cfg, track_rows=track, track_dense=np.arange(d_s, dtype=np.int64))
    setup_s = time.perf_counter() - t0

    def step(k):
        for m, tok in zip(orc_msgs[k % len(orc_msgs)], W.tokens_for_step(cfg, k)):
            m.token = tok
            orc.push(m)
        assert orc.try_apply() == 1

    k = 0
    for _ in range(warmup):
        step(k)
        k += 1
    t0 = time.perf_counter()
    for _ in range(steps):
        step(k)
        k += 1
    el = time.perf_counter() - t0
    n_rows = sum(len(t) for t in track)
    sample = (f"{steps} sampled steps of {cfg.name} after {warmup} warm-up steps, one thread, "
              f"{len(batches_cpu)} distinct batches in turn; each sampled step is 1/{r} of a "
              f"global step (the id occurrences of rows x with x mod {r} = 0: {n_rows} rows "
              f"touched, and dense elements [0, {d_s})); steps/s = 1 / ({r} x seconds per "
              f"sampled step); state initialised in {setup_s:.1f} s outside the timing; "
              f"{el:.1f} s timed")
    return steps / (el * r), sample


def run_reference(args):
    """The CPU oracle on this host's cores, same workload, warm-up and steps."""
    ws, rank, _ = dist_setup()
    if rank != 0:
        return
    from paper_2205_11048_gb300 import workload as W
    cfg = workload_cfg(args.config, args.id_mode, args.shape_rows, args.shape_dense)
    batches = [W.generate_step(cfg, r, "cpu") for r in range(R_BATCHES)]
    sps, sample = oracle_rate(cfg, batches, args.warmup, args.steps)
    line = {"impl": "reference", "metric": METRIC, "value": sps, "unit": "steps/s",
            "n_gpus": ws, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1e3 / sps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32", "data": "synthetic (seeded Zipf ids, "
            "N(0,0.01^2) grads; generated on the host)", "config": config_dict(cfg, ws),
            "cpu_baseline": {"value": sps, "unit": "steps/s", "cores": 1, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": sps, "unit": "steps/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def push_args(B, cfg, batch):
    """ctypes arguments of gba_push / gba_push_ref for every message of a batch."""
    out = []
    for m in batch:
        grads = (B.gba_sparse_grad * max(1, len(cfg.tables)))(*[
            B.gba_sparse_grad(m["ids"][t].data_ptr(), m["ids"][t].numel(),
                              m["rows"][t].data_ptr()) for t in range(len(cfg.tables))])
        out.append((grads, ctypes.c_void_p(m["dense"].data_ptr()), m["local_batch"]))
    return out


def run_gba(args):
    import torch

    from paper_2205_11048_gb300 import binding as B
    from paper_2205_11048_gb300 import workload as W

    ws, rank, local = dist_setup()
    torch.cuda.set_device(local)
    pg = None
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
        pg = dist
    import __graft_entry__
    if rank == 0 or ws == 1:
        __graft_entry__.build()
    if pg:
        pg.barrier()
        __graft_entry__.build()
    L = B.load()

    cfg = workload_cfg(args.config, args.id_mode, args.shape_rows, args.shape_dense)
    M = cfg.M
    # R distinct global batches, resident on this GPU
    batches = [W.generate_step(W.replace(cfg, seed=cfg.seed + 1000 * rank), r, "cuda")
               for r in range(R_BATCHES)]
    torch.cuda.synchronize()
    stream = torch.cuda.current_stream()
    # consecutive steps overlap (step k+1's sort during step k's row update)
    g = B.gba_for_workload(cfg, max_buf=2 * M, overlap=True)
    if args.dense_mode == "eager":
        g.set_eager_dense(True)  # dense gradients summed at push time
    pre = [push_args(B, cfg, b) for b in batches]
    # tokens of every step this run applies, drawn before any timing
    n_total = args.warmup + 2 * args.steps + (args.e2e_steps + 2 if args.e2e_steps > 0 else 0)
    tokens = [W.tokens_for_step(cfg, k) for k in range(n_total)]

    def step(k, push=L.gba_push_ref, args_=pre):
        tk = tokens[k]
        for i, (grads, dense, b) in enumerate(args_[k % len(args_)]):
            rc = push(g.h, tk[i], grads, dense, b)
            if rc != 0:
                raise B.GBAError(rc, "push")
        rc = L.gba_try_apply(g.h)
        if rc != 1:
            raise B.GBAError(rc, "try_apply")

    sampler = ClockSampler(local)
    k = 0
    for _ in range(args.warmup):
        step(k)
        k += 1
    g.join()
    g.sync()
    st0 = g.stats()
    g.set_timing(False)  # clears the launch counters; no events inside the timed region
    if pg:
        pg.barrier()
    torch.cuda.synchronize()
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for _ in range(args.steps):
        step(k)
        k += 1
    g.join()  # the timing stream waits for every step's segment-sum, row and dense work
    ev1.record(stream)
    torch.cuda.synchronize()
    el_ms = ev0.elapsed_time(ev1)
    if pg:
        pg.barrier()
    launches = sum(n for name, (n, _) in g.kernel_times().items() if name != "init")
    st1 = g.stats()
    delta = {key: st1[key] - st0[key] for key in st1}
    el_ms = max_over_ranks(el_ms, pg, "cuda")
    ms_per_step = el_ms / args.steps
    value = job_throughput(args.steps, ws, el_ms)

    # Per-kernel device times: a second pass of the same number of steps with
    # every launch bracketed by events on its own stream (outside the timed
    # region above; kernels of consecutive steps still run concurrently).
    g.set_timing(True)
    for _ in range(args.steps):
        step(k)
        k += 1
    g.join()
    kt = g.kernel_times()
    g.set_timing(False)
    clocks = sampler.stop()

    # roofline of the dominant kernel class: the one that must move the most
    # algorithmic bytes
    bytes_, per = alg_bytes(cfg, delta, args.steps)
    dense_split = dense_traffic(cfg, per, args.dense_mode)
    if args.dense_mode == "eager":  # the dense class then includes the push-time sums
        bytes_["total"] += dense_split["bytes_per_step"] - bytes_["dense"]
        bytes_["dense"] = dense_split["bytes_per_step"]
    classes = {"rows": kt["seg_scan"][1] + kt["row_long"][1] + kt["row_apply"][1],
               "dense": kt["dense"][1], "sort": kt["sort_hist"][1] + kt["sort_pass"][1]}
    n_launch = {"rows": kt["seg_scan"][0] + kt["row_long"][0] + kt["row_apply"][0],
                "dense": kt["dense"][0], "sort": kt["sort_hist"][0] + kt["sort_pass"][0]}
    dom = max(("rows", "dense", "sort"), key=lambda c: bytes_[c])
    launches_per_step = max(1, n_launch[dom] // args.steps)
    dur_ms = classes[dom] / args.steps  # one step's launches of that class
    peak, peak_kind = peaks()
    achieved = bytes_[dom] / (dur_ms / 1e3) / 1e9
    traffic = measured_traffic(dom, cfg.name)

    # End to end through the C ABI with host buffers: every step copies its M
    # messages from pinned host memory (gba_push) and reads the step's counters
    # back (gba_stats), on the same handle with steps no longer overlapping.
    e2e = None
    if args.e2e_steps > 0:
        g.set_overlap(False)
        hb = [dict(local_batch=m["local_batch"],
                   ids=[x.cpu().pin_memory() for x in m["ids"]],
                   rows=[x.cpu().pin_memory() for x in m["rows"]],
                   dense=m["dense"].cpu().pin_memory()) for m in batches[0]]
        h2d = sum(sum(x.numel() * 8 for x in m["ids"]) + sum(x.numel() * 4 for x in m["rows"])
                  + m["dense"].numel() * 4 for m in hb)
        pre_host = [push_args(B, cfg, hb)]
        stats_out = B.gba_stats_t()

        def e2e_step(kk):
            step(kk, push=L.gba_push, args_=pre_host)
            rc = L.gba_stats(g.h, ctypes.byref(stats_out))  # reads the step's counters
            if rc != 0:
                raise B.GBAError(rc, "stats")

        for _ in range(2):
            e2e_step(k)
            k += 1
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        for _ in range(args.e2e_steps):
            e2e_step(k)
            k += 1
        torch.cuda.synchronize()
        el = time.perf_counter() - t0
        el = max_over_ranks(el, pg, "cuda")
        e2e = {"value": ws * args.e2e_steps / el, "unit": "steps/s", "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": ctypes.sizeof(B.gba_stats_t), "steps": args.e2e_steps}
        del hb, pre_host

    cpu = None
    if rank == 0 and ws == 1 and args.cpu_steps > 0:
        cpu_batches = [[{"token": m["token"], "local_batch": m["local_batch"],
                         "ids": [x.cpu() for x in m["ids"]], "rows": [x.cpu() for x in m["rows"]],
                         "dense": m["dense"].cpu()} for m in b] for b in batches]
        # the same warm-up as the reference arm, so both report one number
        sps, sample = oracle_rate(cfg, cpu_batches, args.warmup, args.cpu_steps)
        cpu = {"value": sps, "unit": "steps/s", "cores": 1, "kind": "oracle", "sample": sample}
        del cpu_batches

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "steps/s", "n_gpus": ws,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_per_step,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
            "data": "synthetic (seeded Zipf ids, N(0,0.01^2) grads; replicas per GPU)",
            "config": config_dict(cfg, ws),
            "rows_per_s": per["occ"] * value,
            "unique_rows_per_s": per["u_touched"] * value,
            "alg_bytes_per_step": bytes_["total"],
            "alg_gbs": bytes_["total"] * value / ws / 1e9,
            "hbm_frac_of_8tbs": bytes_["total"] * value / ws / 8e12,
            "hbm_frac_of_measured": bytes_["total"] * value / ws / 1e9 / peak,
            "roofline": {"bound": "hbm", "kernel": dom, "achieved": achieved, "peak": peak,
                         "peak_kind": peak_kind, "unit": "GB/s", "frac": achieved / peak,
                         "traffic": traffic, "alg_bytes_per_launch": bytes_[dom] / launches_per_step,
                         "launches_per_step": launches_per_step,
                         "ms_per_step_in_kernel": dur_ms,
                         "timing": "CUDA events around each launch on its stream, in a second "
                                   "pass of the same steps after the timed region"},
            "kernels_ms_per_step": {n: kt[n][1] / args.steps for n in kt if n != "init"},
            "dense_mode": dense_split,
            "per_step": per,
            "clocks": clocks,
            "gpu_launches": launches,
            "e2e": e2e,
            "cpu_baseline": cpu,
        }
        print(json.dumps(line), flush=True)
    g.close()
    if pg:
        pg.barrier()
        pg.destroy_process_group()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=300)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="gba", choices=["gba", "reference"])
    ap.add_argument("--config", type=int, default=5,
                    help="workload 1-5 (default 5: the largest one that fits one GPU)")
    ap.add_argument("--e2e-steps", type=int, default=10)
    ap.add_argument("--dense-mode", default="buffered", choices=["buffered", "eager"],
                    help="eager: dense gradients summed into their step's accumulator at push")
    ap.add_argument("--id-mode", default="as-configured", choices=["as-configured", "hash"],
                    help="hash: every table an expandable hash table of 64-bit ids")
    ap.add_argument("--shape-rows", type=int, default=None,
                    help="rows of every table (profiling case of the same shape)")
    ap.add_argument("--shape-dense", type=int, default=None,
                    help="dense parameters (profiling case of the same shape)")
    ap.add_argument("--cpu-steps", type=int, default=48,
                    help="sampled oracle steps timed for the cpu_baseline leg (after --warmup "
                         "untimed ones); each is about a quarter second of one core")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.impl == "reference":
        run_reference(args)
    else:
        run_gba(args)


if __name__ == "__main__":
    main()
