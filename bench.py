"""Benchmark: routing decisions/s of the replica simulation on GB300.

Workload (one step): the 70B 1P/2D-shaped grid -- W = 3 workers, 64 replicas
x 20 000 requests (concurrency sweep C in {16..256}, selfish and load-balanced
replicas side by side on 7 shared traces), 64k-block LRU caches per worker.
A step runs the whole path: block hashing of every trace, the replica
simulations, and the per-window PoA estimate of every replica.

  value   decisions/s (requests x workers scored) with the traces resident in
          HBM, CUDA events around K steps on the library's stream.
  e2e     the same metric through the C ABI with pinned HOST trace buffers
          (host->device copies and the result read-back inside the timed region).
  --impl reference   the CPU oracle (single thread) on a bounded sample of the
          same workload, the reference arm of this comparison.

Multi-GPU (torchrun): replicas are independent, so each rank runs its own
64-replica grid on its own traces (weak scaling); ranks only meet at the
timing barriers.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

WORKLOAD = "p2d"
WORKLOAD_DESC = ("70B 1P/2D-shaped: W=3 workers, 64 replicas x 20000 requests, C in "
                 "{16,32,64,128,256}, selfish (omega=1, tau=0) and load-balanced replicas on 7 "
                 "shared traces, prompts lognormal median 1024 max 8192 tokens, 64 Zipf(1.1) "
                 "prefix groups of 512-2048 tokens, outputs lognormal median 256, block 16, "
                 "65536-block LRU cache per worker")
METRIC = "routing decisions/s (requests x workers scored)"


def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def _max_over_ranks(values, device):
    """Element-wise maximum of `values` over all ranks (the step time of the
    slowest rank); the identity when torch.distributed is not initialised."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return [float(v) for v in values]
    t = torch.tensor([float(v) for v in values], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(v) for v in t.tolist()]


def _plan(rank: int, n_req=None):
    from paper_2606_17081_gb300 import workloads as wk
    p = wk.plan(WORKLOAD, n_req=n_req)
    if rank:
        p.trace_seeds = [s + 1000 * rank for s in p.trace_seeds]
        for r in p.replicas:
            r.seed += 1000 * rank
    return p


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled during the timed region."""
    Q = ("index,pci.bus_id,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, bus_id: str | None):
        self.bus = (bus_id or "").lower()
        self.rows = []
        self.p = None

    def start(self):
        try:
            self.p = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.Q}",
                                       "--format=csv,noheader,nounits", "-lms", "200"],
                                      stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except Exception:
            self.p = None

    def _read(self):
        for line in self.p.stdout:
            f = [x.strip() for x in line.split(",")]
            if len(f) >= 10:
                self.rows.append(f)

    def stop(self) -> dict:
        if self.p is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.p.terminate()
        try:
            self.p.wait(timeout=5)
        except Exception:
            self.p.kill()
        self.t.join(timeout=2)
        rows = self.rows
        if self.bus:
            mine = [r for r in rows if self.bus.endswith(r[1].lower()[-12:]) or
                    r[1].lower().endswith(self.bus[-12:])]
            rows = mine or rows
        sm = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        mx = [float(r[3]) for r in rows if r[3].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[k] for r in rows for k in range(4) if r[6 + k].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons,
                "samples": len(rows)}


def _table_bytes(K: int) -> int:
    """Device bytes of one worker's cache: keys + stamps (>= 4K slots in
    buckets of 8) and the stamp log (>= 4K entries)."""
    slots = 8
    while slots < 4 * K:
        slots <<= 1
    ring = 1
    while ring < 4 * K:
        ring <<= 1
    return slots * 12 + ring * 4


# DRAM bytes (read + write) of one full-size k_sim launch of this workload,
# from a one-pass ncu capture (dram__bytes_read.sum + dram__bytes_write.sum),
# with the SHA-256 of the simulation kernel's sources it was taken with.
SIM_TRAFFIC = {"bytes": 31999974144 + 6064310016,
               "sources_sha256": "0fc67a527a3b92e59a5a8de6dff6c21835b2d735ef8812b66f6dcbeb12c818d8",
               "summary": "profiles/k_sim_p2d.md"}


def _sim_traffic(full_size: bool):
    """The captured DRAM traffic per k_sim launch, or None when the kernel
    changed since the capture (or the workload is not the full-size one)."""
    import hashlib
    h = hashlib.sha256()
    for f in ("sim_kernel.cu", "rs_device.cuh", "rs_internal.h"):
        with open(os.path.join(ROOT, "paper_2606_17081_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    if not full_size or h.hexdigest() != SIM_TRAFFIC["sources_sha256"]:
        return None
    return float(SIM_TRAFFIC["bytes"])


def _alg_bytes(results, W: int) -> float:
    """Algorithmic bytes of the simulation kernel for one launch (per-unit
    figures: 32 B per first-miss probe of a bucketed table, 8 B per block hash
    read, 32 B key sector + 16 B LRU stamp/log per inserted block, 64 B per
    eviction, 16 B per touched block, per-request record bytes)."""
    b = 0.0
    for r in results:
        touched = r.hashed_blocks - r.inserted_blocks
        b += (32.0 * r.probe_blocks + 8.0 * r.hashed_blocks + 48.0 * r.inserted_blocks +
              64.0 * r.evicted_blocks + 16.0 * touched + (48.0 + 4.0 * W) * r.n_routed)
    return b


def _aux_knee(rs, ctx, p, descs, params, reps: int = 5) -> dict:
    """Outside the timed steps: the saturation-knee detector over the grid's
    concurrency sweeps, on the records of one more simulation of the grid
    (synchronous call: host argument copies, two kernels, result reads)."""
    from paper_2606_17081_gb300 import workloads as wk
    n = sum(r.n_req for r in p.replicas)
    rec, keep = rs.device_records(n, p.W)
    rs.simulate_replicas(ctx.h, descs, rs.RS_MEM_DEVICE, params, rec)
    rows = np.concatenate([[0], np.cumsum([r.n_req for r in p.replicas])]).astype(np.int64)
    load = np.array([r.C for r in p.replicas], np.float64)
    sw = wk.sweeps(p.replicas)
    out = rs.sweep_knee(ctx.h, rec, rows, load, sw)
    t0 = time.perf_counter()
    for _ in range(reps):
        out = rs.sweep_knee(ctx.h, rec, rows, load, sw)
    ms = (time.perf_counter() - t0) * 1e3 / reps
    del keep
    return {"sweep_knee": {"ms_per_call": ms, "rows": int(n), "replicas": len(params),
                           "sweeps": len(sw) - 1, "pct": 99, "theta": 0.0,
                           "first_knee_C": [float(x) for x in out["knee_load"]]}}


def _aux_variants(rs, p, descs, reps: int = 2) -> dict:
    """Outside the timed steps: the simulation kernel's device time on the same
    p2d replicas under each variant of the method (frequency eviction, Game 2
    tiers, power of two choices), and on the load-spike plan (Experiment 3).
    Each variant runs once to warm up, then `reps` times; decisions/s counts
    requests x W as the main line does."""
    from dataclasses import replace as dc_replace
    from paper_2606_17081_gb300 import workloads as wk
    out = {}

    def timed(ctx, descs_v, params_v, decisions):
        rs.simulate_replicas(ctx.h, descs_v, rs.RS_MEM_DEVICE, params_v)
        ms = []
        for _ in range(reps):
            rs.simulate_replicas(ctx.h, descs_v, rs.RS_MEM_DEVICE, params_v)
            ms.append(rs.route_last_timing(ctx.h).sim_ms)
        sim = statistics.mean(ms)
        return {"sim_ms": sim, "decisions_per_s": decisions / (sim / 1e3)}

    decisions = sum(r.n_req for r in p.replicas) * p.W
    ctx = rs.Context(W=p.W, K=p.K)
    freq = [rs.replica_params(dc_replace(r, eviction=rs.RS_EVICT_FREQ, freq_max=64, decay_s=1.0))
            for r in p.replicas]
    out["frequency_eviction"] = {**timed(ctx, descs, freq, decisions), "freq_max": 64,
                                 "decay_s": 1.0}
    p2c = [rs.replica_params(dc_replace(r, policy=rs.RS_POLICY_P2C)) for r in p.replicas]
    out["power_of_two_choices"] = timed(ctx, descs, p2c, decisions)
    ctx.close()
    ctx = rs.Context(W=p.W, K=p.K, tiered=1, tier_k2=p.K, tier_k3=2 * p.K, tier_node=1)
    base = [rs.replica_params(r) for r in p.replicas]
    out["game2_tiers"] = {**timed(ctx, descs, base, decisions), "tier_blocks": [p.K, p.K, 2 * p.K]}
    ctx.close()
    sp = wk.plan("spike")
    trs = sp.traces()
    dev = [rs.device_trace(t) for t in trs]
    ctx = rs.Context(W=sp.W, K=sp.K, theta1=sp.theta1, theta2=sp.theta2)
    out["load_spike_plan"] = {**timed(ctx, [b.desc() for b in dev],
                                      [rs.replica_params(r) for r in sp.replicas],
                                      sum(r.n_req for r in sp.replicas) * sp.W),
                              "replicas": len(sp.replicas)}
    ctx.close()
    return out


def _aux_probe(rs, d, n: int, reps: int = 5) -> dict:
    """Outside the timed steps: the batch probe (route_probe: S2's cached
    prefix for many requests against one cache snapshot) on a router instance
    of 64 workers with 65536-block caches.  The first 2000 requests (at most
    half) of a p2d trace are routed (route_batch), then the others are probed.  The
    call hashes the batch, then probes; its kernel time is the call's device
    time (CUDA events) less a block-hash call on the same batch.  probes =
    sum over (request, worker) of min(m_ij + 1, nb_i) table lookups."""
    import torch
    W, K, nr = 64, 65536, min(2000, n // 2)
    if n - nr <= 0:
        return {}
    ctx = rs.Context(W=W, K=K, n_instances=1)
    wo = torch.zeros(nr, dtype=torch.int32, device="cuda")
    rs.route_batch(ctx.h, 0, d.tokens, d.offsets, nr, d.out_len, wo)
    m = n - nr
    offs = d.offsets[nr:]
    po = torch.zeros(m * W, dtype=torch.int32, device="cuda")
    hs = torch.zeros(int(offs[-1].item()) // 16 + 1, dtype=torch.int64, device="cuda")
    rs.route_probe(ctx.h, 0, d.tokens, offs, m, po)
    tp, th = [], []
    for _ in range(reps):
        e0, e1, e2 = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
        e0.record()
        rs.route_probe(ctx.h, 0, d.tokens, offs, m, po)
        e1.record()
        rs.route_hash_blocks(ctx.h, d.tokens, offs, m, hs)
        e2.record()
        torch.cuda.synchronize()
        tp.append(e0.elapsed_time(e1))
        th.append(e1.elapsed_time(e2))
    ctx.close()
    pre = po.cpu().numpy().reshape(m, W).astype(np.int64)
    nb = (np.diff(offs.cpu().numpy()) // 16)[:, None]
    probes = int(np.minimum(pre + 1, nb).sum())
    kern = min(tp) - min(th)
    return {"workers": W, "cache_blocks": K, "routed": nr, "probed": m, "pairs": m * W,
            "probes": probes, "mean_prefix": float(pre.mean()), "call_ms": min(tp),
            "hash_ms": min(th), "kernel_ms": kern, "probes_per_s": probes / (kern / 1e3),
            "bucket_bytes_per_s": 64 * probes / (kern / 1e3)}


def run_gpu(args):
    import torch
    import torch.distributed as dist
    from paper_2606_17081_gb300 import routesim as rs

    ws, rank, local = _dist()
    torch.cuda.set_device(local)
    if ws > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    p = _plan(rank, args.n_req)
    traces = p.traces()
    ctx = rs.Context(W=p.W, K=p.K)
    dev = [rs.device_trace(t) for t in traces]
    host = [rs.host_trace(t, pinned=True) for t in traces]
    params = [rs.replica_params(r) for r in p.replicas]
    descs_d = [b.desc() for b in dev]
    descs_h = [b.desc() for b in host]
    decisions = sum(r.n_req for r in p.replicas) * p.W
    torch.cuda.synchronize()

    def barrier():
        if ws > 1:
            dist.barrier()

    def step(descs, mem):
        return rs.simulate_replicas(ctx.h, descs, mem, params)

    for _ in range(args.warmup):
        res = step(descs_d, rs.RS_MEM_DEVICE)
    bus = None
    try:
        bus = torch.cuda.get_device_properties(local).pci_bus_id
    except Exception:
        pass
    clk = ClockSampler(bus if isinstance(bus, str) else None)
    clk.start()
    time.sleep(0.4)
    # ---- device-resident timing
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    sim_ms, hash_ms, poa_ms, launches = [], [], [], 0
    barrier()
    torch.cuda.synchronize()
    ev0.record()
    for _ in range(args.steps):
        res = step(descs_d, rs.RS_MEM_DEVICE)
        t = rs.route_last_timing(ctx.h)
        sim_ms.append(t.sim_ms)
        hash_ms.append(t.hash_ms)
        poa_ms.append(t.poa_ms)
        launches += t.launches
    ev1.record()
    torch.cuda.synchronize()
    barrier()
    ms = ev0.elapsed_time(ev1)
    clocks = clk.stop()
    hashed_tokens = rs.route_last_timing(ctx.h).hashed_tokens
    # ---- end to end through the C ABI with host buffers
    for _ in range(max(1, args.warmup // 2)):
        step(descs_h, rs.RS_MEM_HOST)
    barrier()
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        step(descs_h, rs.RS_MEM_HOST)
    torch.cuda.synchronize()
    barrier()
    e2e_s = time.perf_counter() - t0
    ms, e2e_s = _max_over_ranks([ms, e2e_s], "cuda")
    aux = None
    if rank == 0:
        aux = _aux_knee(rs, ctx, p, descs_d, params)
        if not args.no_aux:
            aux["variants"] = _aux_variants(rs, p, descs_d)
            aux["probe_batch"] = _aux_probe(rs, dev[0], traces[0].n_req)
    if rank != 0:
        if ws > 1:
            dist.destroy_process_group()
        return
    status = [r.status for r in res]
    assert all(s == 0 for s in status), status
    per_step_s = ms / 1e3 / args.steps
    value = decisions * ws / per_step_s
    peak, peak_kind = _peaks()
    sim_avg = statistics.mean(sim_ms)
    alg = _alg_bytes(res, p.W)
    achieved = alg / (sim_avg / 1e3) / 1e9
    hash_avg = statistics.mean(hash_ms)
    nblocks = sum(int(t.offsets[-1]) // 16 for t in traces)
    hash_bytes = 4.0 * hashed_tokens + 8.0 * nblocks
    hash_gbs = hash_bytes / (hash_avg / 1e3) / 1e9
    h2d = sum(b.tokens.numel() * 4 + b.offsets.numel() * 8 + b.release.numel() * 8 +
              b.out_len.numel() * 4 for b in host)
    import ctypes
    d2h = len(params) * ctypes.sizeof(rs.rs_replica_result) + 8 * len(traces)
    poa = [r.poa_total for r in res]
    cpu = None if args.no_cpu_baseline else cpu_baseline(p, traces, budget_s=args.cpu_budget)
    line = {
        "metric": METRIC, "value": value, "unit": "decisions/s", "n_gpus": ws,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded traces shaped like the paper's chat workload)",
        "config": {"workload": WORKLOAD_DESC, "replicas_per_gpu": len(params),
                   "requests_per_replica": p.replicas[0].n_req, "W": p.W,
                   "cache_blocks": p.K, "parallelism": f"replicas sharded over {ws} GPU(s)",
                   "l2": "inputs larger than L2 every step (%.0f MB of tokens read, %.0f MB of "
                         "cache tables cleared and rebuilt per step; L2 129 MB)" % (
                             sum(t.tokens.nbytes for t in traces) / 1e6,
                             _table_bytes(p.K) * p.W * len(params) / 1e6)},
        "replicas_per_s": len(params) * ws / per_step_s,
        "requests_per_s": decisions * ws / p.W / per_step_s,
        "kernels_ms_per_step": {"block_hash": hash_avg, "simulate": sim_avg,
                                "poa": statistics.mean(poa_ms)},
        "roofline": {"kernel": "k_sim (replica simulation, one CTA per replica)",
                     "bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "peak_kind": peak_kind,
                     "alg_bytes_per_launch": alg, "traffic": _sim_traffic(args.n_req is None),
                     "traffic_source": SIM_TRAFFIC["summary"],
                     "note": "latency-bound event loop: 64 replicas on 152 SMs"},
        "hash_roofline": {"kernel": "k_block_hash", "bound": "hbm", "achieved": hash_gbs,
                          "peak": peak, "unit": "GB/s", "frac": hash_gbs / peak,
                          "alg_bytes_per_launch_set": hash_bytes},
        "poa_total_mean": float(np.mean(poa)),
        "e2e": {"value": decisions * ws / (e2e_s / args.steps), "unit": "decisions/s",
                "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h)},
        "clocks": clocks,
        "gpu_launches": int(launches),
        "cpu_baseline": cpu,
        "aux": aux,
    }
    print(json.dumps(line))
    if ws > 1:
        dist.destroy_process_group()


def cpu_baseline(p, traces, budget_s: float = 15.0) -> dict:
    """The oracle, single-threaded, on whole replicas of the workload until the
    budget is spent; decisions/s on one core."""
    import oracle as O
    cfg = O.OracleConfig(W=p.W, K=p.K, theta1=p.theta1, theta2=p.theta2)
    done = dec = 0
    t0 = time.perf_counter()
    # selfish / load-balanced pairs over C first, then the rest of the 64 in order
    first = [0, 5, 1, 6, 2, 7, 3, 8, 4, 9]
    order = first + [k for k in range(len(p.replicas)) if k not in first]
    for k in order:
        r = p.replicas[k]
        o = O.simulate(cfg, traces[r.trace], r.C, policy=r.policy, controller=r.controller,
                       omega=r.omega, tau=r.tau, seed=r.seed, n_req=r.n_req)
        O.poa(cfg, o)
        done += 1
        dec += r.n_req * p.W
        if time.perf_counter() - t0 > budget_s:
            break
    el = time.perf_counter() - t0
    return {"value": dec / el, "unit": "decisions/s", "cores": 1, "kind": "oracle",
            "sample": f"{done} whole replicas of the {len(p.replicas)} (20000 requests each; "
                      f"pairs 0/5, 1/6, ... first, then in order) incl. PoA, single thread, "
                      f"{el:.1f} s"}


def run_reference(args):
    """Reference arm: the CPU oracle on a bounded sample of the same workload."""
    ws, rank, local = _dist()
    if rank != 0:
        return
    p = _plan(0)
    from paper_2606_17081_gb300 import workloads as wk
    traces = [wk.make_trace(p.spec, p.trace_seeds[0])]
    import oracle as O
    cfg = O.OracleConfig(W=p.W, K=p.K)
    reps = [p.replicas[0], p.replicas[5]]      # one selfish, one load-balanced replica

    def step():
        for r in reps:
            o = O.simulate(cfg, traces[0], r.C, policy=r.policy, omega=r.omega, tau=r.tau,
                           seed=r.seed, n_req=r.n_req)
            O.poa(cfg, o)

    for _ in range(args.warmup):
        step()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        step()
    el = time.perf_counter() - t0
    dec = sum(r.n_req for r in reps) * p.W * args.steps
    v = dec / el
    sample = ("2 whole replicas per step (C=16 selfish and load-balanced, 20000 requests "
              "each) incl. PoA, oracle single thread")
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": v, "unit": "decisions/s",
        "n_gpus": ws, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": el * 1e3 / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": WORKLOAD_DESC},
        "cpu_baseline": {"value": v, "unit": "decisions/s", "cores": 1, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": v, "unit": "decisions/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0}}))


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="native", choices=["native", "reference"])
    ap.add_argument("--cpu-budget", type=float, default=15.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-aux", action="store_true",
                    help="skip the timings reported under aux.variants and aux.probe_batch")
    ap.add_argument("--n-req", type=int, default=None,
                    help="truncate every replica's trace (profiling of a small case)")
    args = ap.parse_args()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
