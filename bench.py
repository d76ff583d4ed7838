"""Benchmark of the GBA aggregate-and-apply step on GB300.

One "step" is one global step of the hot path: message weights (Eq. (1)),
the radix sort + dedup of the global batch's ids, the per-row decayed
segment-sum and row update, and the dense reduce + optimizer.

Default workload: the 32-worker one-hot workload (1e7 x 32 embedding table,
Adagrad; 1M dense parameters, Adam; 32 messages of local batch 1024, 26 ids per
sample; geometric staleness with 10% stragglers).  Inputs are synthetic
(seeded Zipf ids, N(0, 0.01^2) gradients) and resident in HBM before the timed
region; messages are pushed by reference, R distinct global batches in turn,
with fresh tokens every step.

Prints one JSON line (rank 0).  --impl reference times the CPU oracle instead.
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
R_BATCHES = 4


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            j = json.load(f)
        return float(j["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


def workload_cfg(n):
    from paper_2205_11048_gb300 import workload as W
    return W.config(n)


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


def source_sha(files):
    h = hashlib.sha256()
    for f in files:
        with open(os.path.join(ROOT, f), "rb") as fh:
            h.update(fh.read())
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


def run_reference(args):
    """The CPU oracle, as it stands, on this host's cores, same workload."""
    ws, rank, _ = dist_setup()
    if rank != 0:
        return
    import numpy as np
    import torch

    from oracle import oracle as O
    from paper_2205_11048_gb300 import workload as W
    from tests import _harness as H
    cfg = workload_cfg(args.config)
    batches = [W.generate_step(cfg, r, "cpu") for r in range(R_BATCHES)]
    orc_msgs = [[H.to_oracle(m) for m in b] for b in batches]
    t0 = time.perf_counter()
    orc = H.make_oracle(cfg)
    setup_s = time.perf_counter() - t0
    budget = args.ref_budget_s

    def step(k):
        toks = W.tokens_for_step(cfg, k)
        for m, tok in zip(orc_msgs[k % R_BATCHES], toks):
            m.token = tok
            orc.push(m)
        assert orc.try_apply() == 1

    k = 0
    for _ in range(max(0, min(args.warmup, 3))):
        step(k)
        k += 1
    t0 = time.perf_counter()
    n = 0
    while n < args.steps and (time.perf_counter() - t0) < budget:
        step(k)
        k += 1
        n += 1
    el = time.perf_counter() - t0
    sps = n / el
    sample = (f"{n} full global steps of {cfg.name} (all {cfg.tables[0].rows} rows and "
              f"{cfg.D} dense parameters tracked), single thread, {R_BATCHES} distinct "
              f"batches in turn; state init {setup_s:.1f} s excluded")
    line = {"impl": "reference", "metric": METRIC, "value": sps, "unit": "steps/s", "n_gpus": ws,
            "steps": n, "warmup": min(args.warmup, 3), "ms_per_step": 1e3 * el / max(n, 1),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
            "data": "synthetic", "config": {"workload": cfg.name, "M": cfg.M, "B": cfg.B},
            "cpu_baseline": {"value": sps, "unit": "steps/s", "cores": 1, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": sps, "unit": "steps/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def cpu_baseline(cfg, batches_cpu, budget_s):
    """Oracle steps/s on this host, one thread, on the same batches."""
    from paper_2205_11048_gb300 import workload as W
    from tests import _harness as H
    orc_msgs = [[H.to_oracle(m) for m in b] for b in batches_cpu]
    orc = H.make_oracle(cfg)
    t0 = time.perf_counter()
    n = 0
    k = 0
    while time.perf_counter() - t0 < budget_s:
        toks = W.tokens_for_step(cfg, k)
        for m, tok in zip(orc_msgs[k % len(orc_msgs)], toks):
            m.token = tok
            orc.push(m)
        orc.try_apply()
        n += 1
        k += 1
    el = time.perf_counter() - t0
    return {"value": n / el, "unit": "steps/s", "cores": 1, "kind": "oracle",
            "sample": f"{n} full global steps of {cfg.name} on the CPU oracle, one thread, "
                      f"{el:.1f} s"}


def run_gba(args):
    import numpy as np
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

    cfg = workload_cfg(args.config)
    M = cfg.M
    # R distinct global batches, resident on this GPU
    batches = [W.generate_step(W.replace(cfg, seed=cfg.seed + 1000 * rank), r, "cuda")
               for r in range(R_BATCHES)]
    torch.cuda.synchronize()
    stream = torch.cuda.current_stream()
    # consecutive steps overlap (step k+1's sort during step k's row update)
    g = B.gba_for_workload(cfg, max_buf=2 * M, overlap=True)
    # pre-built ctypes arguments for the by-reference pushes
    pre = []
    for b in batches:
        row = []
        for m in b:
            grads = (B.gba_sparse_grad * len(cfg.tables))(*[
                B.gba_sparse_grad(m["ids"][t].data_ptr(), m["ids"][t].numel(),
                                  m["rows"][t].data_ptr()) for t in range(len(cfg.tables))])
            row.append((grads, ctypes.c_void_p(m["dense"].data_ptr()), m["local_batch"]))
        pre.append(row)
    tokens = {}

    def toks(k):
        if k not in tokens:
            tokens[k] = W.tokens_for_step(cfg, k)
        return tokens[k]

    def step(k):
        tk = toks(k)
        for i, (grads, dense, b) in enumerate(pre[k % R_BATCHES]):
            rc = L.gba_push_ref(g.h, tk[i], grads, dense, b)
            if rc != 0:
                raise B.GBAError(rc, "push_ref")
        rc = L.gba_try_apply(g.h)
        if rc != 1:
            raise B.GBAError(rc, "try_apply")

    n_total = args.warmup + args.steps
    for k in range(n_total):
        toks(k)
    k = 0
    for _ in range(args.warmup):
        step(k)
        k += 1
    g.sync()
    st0 = g.stats()
    g.set_timing(True)
    sampler = ClockSampler(local)
    time.sleep(0.3)
    if pg:
        pg.barrier()
    torch.cuda.synchronize()
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for _ in range(args.steps):
        step(k)
        k += 1
    ev1.record(stream)
    torch.cuda.synchronize()
    el_ms = ev0.elapsed_time(ev1)
    if pg:
        pg.barrier()
    clocks = sampler.stop()
    kt = g.kernel_times()
    g.sync()
    st1 = g.stats()
    delta = {key: st1[key] - st0[key] for key in st1}
    el_ms = max_over_ranks(el_ms, pg, "cuda")
    ms_per_step = el_ms / args.steps
    value = job_throughput(args.steps, ws, el_ms)
    launches = sum(kt[n][0] for n in kt if n != "init")

    # roofline of the dominant kernel class: the one that must move the most
    # algorithmic bytes (its time is measured live, concurrent steps included)
    bytes_, per = alg_bytes(cfg, delta, args.steps)
    # the row path is three kernels per table (segment reduction, rows that
    # cross windows, row update): its bytes are divided by their summed time
    classes = {"rows": kt["seg_reduce"][1] + kt["seg_cross"][1] + kt["row_update"][1],
               "dense": kt["dense"][1], "sort": kt["sort_hist"][1] + kt["sort_pass"][1]}
    dom = max(("rows", "dense", "sort"), key=lambda c: bytes_[c])
    n_launch = {"rows": kt["seg_reduce"][0] + kt["seg_cross"][0] + kt["row_update"][0],
                "dense": kt["dense"][0], "sort": kt["sort_hist"][0] + kt["sort_pass"][0]}
    launches_per_step = max(1, n_launch[dom] // args.steps)
    dur_ms = classes[dom] / args.steps  # one step's launches of that class
    peak, peak_kind = peaks()
    achieved = bytes_[dom] / (dur_ms / 1e3) / 1e9
    traffic = measured_traffic(dom, cfg.name)

    # end to end through the C ABI with host buffers: pinned host -> device
    # copies inside gba_push, one step, and a device -> host read of the counters
    e2e = None
    if args.e2e_steps > 0:
        host = []
        for b in batches[:2]:
            hb = []
            for m in b:
                hb.append(dict(token=0, local_batch=m["local_batch"],
                               ids=[x.cpu().pin_memory() for x in m["ids"]],
                               rows=[x.cpu().pin_memory() for x in m["rows"]],
                               dense=m["dense"].cpu().pin_memory()))
            host.append(hb)
        h2d = sum(sum(x.numel() * 8 for x in m["ids"]) + sum(x.numel() * 4 for x in m["rows"])
                  + m["dense"].numel() * 4 for m in host[0])
        g2 = B.gba_for_workload(cfg, max_buf=2 * M)
        pre2 = []
        for hb in host:
            row = []
            for m in hb:
                grads = (B.gba_sparse_grad * len(cfg.tables))(*[
                    B.gba_sparse_grad(m["ids"][t].data_ptr(), m["ids"][t].numel(),
                                      m["rows"][t].data_ptr()) for t in range(len(cfg.tables))])
                row.append((grads, ctypes.c_void_p(m["dense"].data_ptr()), m["local_batch"]))
            pre2.append(row)
        stats_out = B.gba_stats_t()

        def e2e_step(kk):
            tk = toks(kk % n_total)
            for i, (grads, dense, b) in enumerate(pre2[kk % 2]):
                rc = L.gba_push(g2.h, tk[i], grads, dense, b)
                if rc != 0:
                    raise B.GBAError(rc, "push")
            rc = L.gba_try_apply(g2.h)
            if rc != 1:
                raise B.GBAError(rc, "try_apply")
            rc = L.gba_stats(g2.h, ctypes.byref(stats_out))  # reads the step's counters
            if rc != 0:
                raise B.GBAError(rc, "stats")

        for kk in range(3):
            e2e_step(kk)
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        for kk in range(args.e2e_steps):
            e2e_step(3 + kk)
        torch.cuda.synchronize()
        el = time.perf_counter() - t0
        e2e = {"value": ws * args.e2e_steps / el, "unit": "steps/s", "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": ctypes.sizeof(B.gba_stats_t), "steps": args.e2e_steps}
        g2.close()

    cpu = None
    if rank == 0 and ws == 1 and args.cpu_budget_s > 0:
        cpu_batches = [[{"token": m["token"], "local_batch": m["local_batch"],
                         "ids": [x.cpu() for x in m["ids"]], "rows": [x.cpu() for x in m["rows"]],
                         "dense": m["dense"].cpu()} for m in b] for b in batches]
        cpu = cpu_baseline(cfg, cpu_batches, args.cpu_budget_s)

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "steps/s", "n_gpus": ws,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_per_step,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
            "data": "synthetic (seeded Zipf ids, N(0,0.01^2) grads; replicas per GPU)",
            "config": {"workload": cfg.name, "M": cfg.M, "B": cfg.B, "G": cfg.G,
                       "tables": [[t.rows, t.dim] for t in cfg.tables], "dense": cfg.D,
                       "iota": cfg.iota, "batches_in_turn": R_BATCHES,
                       "l2": "inputs larger than L2 (distinct global batches of "
                             f"{bytes_['total'] / 1e6:.0f} MB of algorithmic traffic each)",
                       "parallelism": f"replicas x{ws}"},
            "rows_per_s": per["occ"] * value,
            "unique_rows_per_s": per["u_touched"] * value,
            "alg_bytes_per_step": bytes_["total"],
            "alg_gbs": bytes_["total"] * value / ws / 1e9,
            "hbm_frac_of_8tbs": bytes_["total"] * value / ws / 8e12,
            "roofline": {"bound": "hbm", "kernel": dom, "achieved": achieved, "peak": peak,
                         "peak_kind": peak_kind, "unit": "GB/s", "frac": achieved / peak,
                         "traffic": traffic, "alg_bytes_per_launch": bytes_[dom] / launches_per_step,
                         "launches_per_step": launches_per_step,
                         "ms_per_step_in_kernel": dur_ms},
            "kernels_ms_per_step": {n: kt[n][1] / args.steps for n in kt if n != "init"},
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
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", default="gba", choices=["gba", "reference"])
    ap.add_argument("--config", type=int, default=2)
    ap.add_argument("--e2e-steps", type=int, default=20)
    ap.add_argument("--cpu-budget-s", type=float, default=15.0)
    ap.add_argument("--ref-budget-s", type=float, default=60.0)
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.impl == "reference":
        run_reference(args)
    else:
        run_gba(args)


if __name__ == "__main__":
    main()
