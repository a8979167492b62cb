"""Benchmark: routing decisions/s of the replica simulation on GB300.

Headline workload (one step): the parameter grid -- W = 6 workers, 4096 cells
(overlap weight omega x concurrency C x temperature tau x 8 seeds), each
simulated under the selfish cache-affinity policy and the load-balanced one on
its trace, i.e. 8192 simulations x 10 000 requests, 32 768-block LRU caches
per worker.  A step runs the whole path: block hashing of every trace, the
replica simulations, decision statistics and the per-window PoA estimate of
every simulation.

  value   decisions/s (requests x workers scored) with the traces resident in
          HBM, CUDA events around K steps on the library's stream.
  e2e     the same metric through the C ABI with pinned HOST trace buffers
          (host->device copies and the result read-back inside the timed region).
  aux.per_config   one timed call of every other workload (tiny, the 1P/2D and
          1P/5D grids, and the W = 64 workload at its own shape, whose traces
          are hashed chunk by chunk into resident block hashes).
  --impl reference   the CPU oracle (single thread) on a bounded sample of the
          same workload, the reference arm of this comparison.

Multi-GPU (torchrun): the replicas of the one plan are independent, so rank r
runs a contiguous range of them (strong scaling: N ranks do the N = 1 work in
pieces, with no data-path collective); ranks only meet at the timing barriers.
"""
from __future__ import annotations

import argparse
import ctypes
import json
import os
import platform
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

HEADLINE = "grid"
METRIC = "routing decisions/s (requests x workers scored)"
WORKLOAD_DESC = {
    "tiny": "W=3, 1 replica x 512 requests (Poisson 50/s), prompts 64-512 tokens from 16 "
            "shared 256-token prefixes, block 16, 2048-block LRU cache per worker, argmin, C=16",
    "p2d": "70B 1P/2D-shaped: W=3, 64 replicas x 20000 requests, C in {16..256}, selfish "
           "(omega=1, tau=0) and load-balanced replicas on 7 shared traces, prompts lognormal "
           "median 1024 max 8192 tokens, 64 Zipf(1.1) prefix groups of 512-2048 tokens, outputs "
           "lognormal median 256, 65536-block LRU cache per worker",
    "p5d": "70B 1P/5D-shaped: W=6, 256 replicas x 50000 requests, C in {32..512} x tau in "
           "{0, 0.5, 1} with Philox sampling, adaptive saturation controller on, 18 traces, "
           "65536-block LRU cache per worker",
    "grid": "parameter grid: W=6, 4096 cells (omega {0,.25,.5,1,2,4} x C {16..512} x tau "
            "{0,.5,1} x 8 trace seeds) x 2 policies (selfish, load-balanced) = 8192 simulations "
            "x 10000 requests, 32768-block LRU cache per worker, per-simulation PoA",
    "large": "W=64, 16 replicas (8 selfish, 8 coordinated) x 1000000 requests, prompts lognormal "
             "median 2048 max 32768 tokens, 1024 Zipf(1.0) prefix groups, 2^20-block LRU cache "
             "per worker, C=4096; traces hashed chunk by chunk into resident block hashes",
}


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


def rank_range(n: int, ws: int, rank: int):
    """Contiguous share [lo, hi) of n replicas for rank `rank` of ws."""
    return n * rank // ws, n * (rank + 1) // ws


def _subset(full, spec):
    """Replica indices of a profiling subset: "N" = the plan's first N
    replicas, "per-trace" = the first replica of every trace."""
    if spec == "per-trace":
        seen, idx = set(), []
        for k, r in enumerate(full.replicas):
            if r.trace not in seen:
                seen.add(r.trace)
                idx.append(k)
        return idx
    return list(range(min(int(spec), len(full.replicas))))


def _plan(name: str, rank: int = 0, ws: int = 1, n_req=None, subset=None):
    """The workload's replicas that rank `rank` of ws runs (its contiguous
    range of the one plan, traces remapped to the ones it uses); `subset`
    (a profiling option) first narrows the plan to those replicas."""
    from paper_2606_17081_gb300 import workloads as wk
    full = wk.plan(name, n_req=n_req)
    if subset is not None:
        full = wk.plan(name, n_req=n_req, replicas=_subset(full, subset))
        if ws > 1:
            raise ValueError("--replicas is a single-GPU profiling option")
        return full, 0, len(full.replicas)
    lo, hi = rank_range(len(full.replicas), ws, rank)
    if (lo, hi) == (0, len(full.replicas)):
        return full, lo, hi
    return wk.plan(name, n_req=n_req, replicas=list(range(lo, hi))), lo, hi


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


# DRAM bytes (read + write) of one full-size k_sim launch of the headline
# workload (dram__bytes_read.sum + dram__bytes_write.sum), with the SHA-256 of
# the simulation kernel's sources it was taken with; None until such a
# capture exists for these sources.  The full grid holds about 103 GB of
# cache tables, so the capture ran on 304 of its 8192 simulations (one
# resident wave, two per SM, 10 000 requests each: 234.69 GB) and is scaled by
# 8192 / 304; every simulation's tables and requests are of the same kind.
SIM_TRAFFIC = {"bytes": 234692720384 * 8192 / 304,
               "sources_sha256": "188fdf42bea8a811467ab449087524e9d353034642b819cda337c020b3f84b3f",
               "summary": "profiles/k_sim_grid.md",
               "scaled_from": "304 simulations x 10 000 requests, times 8192 / 304"}


def _sim_traffic(full_size: bool):
    """The captured DRAM traffic per k_sim launch, or None when the kernel
    changed since the capture (or the workload is not the full-size one)."""
    import hashlib
    if SIM_TRAFFIC["bytes"] is None:
        return None
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


def _roofline(results, W, sim_ms, peak, peak_kind):
    alg = _alg_bytes(results, W)
    ach = alg / (sim_ms / 1e3) / 1e9
    return {"kernel": "k_sim (replica simulation, one CTA per replica)", "bound": "hbm",
            "achieved": ach, "peak": peak, "unit": "GB/s", "frac": ach / peak,
            "peak_kind": peak_kind, "alg_bytes_per_launch": alg}


def _aux_knee(rs, ctx, p, descs, params, reps: int = 5) -> dict:
    """Outside the timed steps: the saturation-knee detector over the plan's
    concurrency sweeps, on the records of one more simulation of it
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
    kl = [float(x) for x in out["knee_load"]]
    return {"sweep_knee": {"workload": "p2d", "ms_per_call": ms, "rows": int(n),
                           "replicas": len(params), "sweeps": len(sw) - 1, "pct": 99,
                           "theta": 0.0, "first_knee_C": kl}}


def _timed_sim(rs, ctx, descs, params, reps: int = 1, warm: int = 1):
    """Device times of simulate_replicas (after `warm` untimed calls): the
    mean over `reps` calls of each phase, the last call's results and the
    kernel launches of one call."""
    for _ in range(warm):
        rs.simulate_replicas(ctx.h, descs, rs.RS_MEM_DEVICE, params)
    ts = []
    for _ in range(reps):
        res = rs.simulate_replicas(ctx.h, descs, rs.RS_MEM_DEVICE, params)
        t = rs.route_last_timing(ctx.h)
        ts.append((t.hash_ms, t.sim_ms, t.poa_ms, t.launches, t.hashed_tokens))
    m = [statistics.mean(x[k] for x in ts) for k in range(3)]
    return res, {"hash_ms": m[0], "sim_ms": m[1], "poa_ms": m[2], "launches": ts[-1][3],
                 "hashed_tokens": ts[-1][4]}


def _config_entry(p, res, t, peak, peak_kind, extra=None) -> dict:
    decisions = sum(r.n_req for r in p.replicas) * p.W
    step = t["hash_ms"] + t["sim_ms"] + t["poa_ms"]
    e = {"workload": WORKLOAD_DESC[p.name], "W": p.W, "replicas": len(p.replicas),
         "requests_per_replica": p.replicas[0].n_req, "cache_blocks": p.K,
         "decisions_per_s": decisions / (step / 1e3), "replicas_per_s": len(p.replicas) / (step / 1e3),
         "kernels_ms": {"block_hash": t["hash_ms"], "simulate": t["sim_ms"], "poa": t["poa_ms"]},
         "roofline": _roofline(res, p.W, t["sim_ms"], peak, peak_kind),
         "status": sorted({int(r.status) for r in res}),
         "poa_total_mean": float(np.mean([r.poa_total for r in res]))}
    if t.get("hashed_tokens"):
        blocks = sum(int(r.hashed_blocks) for r in res)
        e["hash_ms_note"] = "hash kernel launches only (events around them)"
    if extra:
        e.update(extra)
    return e


def _per_config(rs, peak, peak_kind, skip=(), large_n_req=None) -> dict:
    """One timed call (after one untimed) of each workload but the headline;
    the W = 64 workload streams its traces' tokens through the block-hash
    kernel into resident hashes first, then runs one untimed call on its
    first 2000 requests (allocations) and one timed call at full size."""
    import torch
    from paper_2606_17081_gb300 import streaming as stm
    out = {}
    for name in ("tiny", "p2d", "p5d"):
        if name in skip:
            continue
        p, _, _ = _plan(name)
        ctx = rs.Context(W=p.W, K=p.K, theta1=p.theta1, theta2=p.theta2)
        dev = [rs.device_trace(t) for t in p.traces()]
        descs = [b.desc() for b in dev]
        params = [rs.replica_params(r) for r in p.replicas]
        res, t = _timed_sim(rs, ctx, descs, params, reps=2 if name != "p5d" else 1)
        out[name] = _config_entry(p, res, t, peak, peak_kind)
        ctx.close()
        del dev
        torch.cuda.empty_cache()
    if "large" not in skip:
        p, _, _ = _plan("large", n_req=large_n_req)
        ctx = rs.Context(W=p.W, K=p.K, theta1=p.theta1, theta2=p.theta2)
        tm = []
        bufs = []
        for m in p.metas():
            d = {}
            bufs.append(stm.hash_streamed(ctx, m, timing=d))
            tm.append(d)
        descs = [b.desc() for b in bufs]
        from dataclasses import replace as dc_replace
        small = [rs.replica_params(dc_replace(r, n_req=min(r.n_req, 2000))) for r in p.replicas]
        rs.simulate_replicas(ctx.h, descs, rs.RS_MEM_DEVICE, small)
        params = [rs.replica_params(r) for r in p.replicas]
        res, t = _timed_sim(rs, ctx, descs, params, reps=1, warm=0)
        hash_ms = sum(d["hash_ms"] for d in tm)
        toks = sum(d["tokens"] for d in tm)
        blocks = sum(d["blocks"] for d in tm)
        t["hash_ms"] = hash_ms     # the streamed S1 (hash kernel launches only)
        hb = 4.0 * toks + 8.0 * blocks
        out["large"] = _config_entry(p, res, t, peak, peak_kind, extra={
            "streamed_hashing": {"tokens": toks, "blocks": blocks, "chunks": sum(d["chunks"] for d in tm),
                                 "token_generation_ms": sum(d["fill_ms"] for d in tm),
                                 "hash_ms": hash_ms, "hash_gbs": hb / (hash_ms / 1e3) / 1e9,
                                 "hash_frac": hb / (hash_ms / 1e3) / 1e9 / peak,
                                 "note": "tokens produced on the device by the seeded generator "
                                         "(not timed in decisions/s), hashed chunk by chunk"}})
        ctx.close()
        del bufs
        torch.cuda.empty_cache()
    return out


def _aux_variants(rs, reps: int = 2) -> dict:
    """Outside the timed steps: the simulation kernel's device time on the p2d
    replicas under each variant of the method (frequency eviction, Game 2
    tiers, power of two choices), and on the load-spike plan (Experiment 3).
    Each variant runs once to warm up, then `reps` times; decisions/s counts
    requests x W as the main line does."""
    from dataclasses import replace as dc_replace
    import torch
    from paper_2606_17081_gb300 import workloads as wk
    out = {}
    p, _, _ = _plan("p2d")
    dev = [rs.device_trace(t) for t in p.traces()]
    descs = [b.desc() for b in dev]

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
    base = [rs.replica_params(r) for r in p.replicas]
    out["knee"] = _aux_knee(rs, ctx, p, descs, base)["sweep_knee"]
    ctx.close()
    ctx = rs.Context(W=p.W, K=p.K, tiered=1, tier_k2=p.K, tier_k3=2 * p.K, tier_node=1)
    out["game2_tiers"] = {**timed(ctx, descs, base, decisions), "tier_blocks": [p.K, p.K, 2 * p.K]}
    ctx.close()
    sp = wk.plan("spike")
    sdev = [rs.device_trace(t) for t in sp.traces()]
    ctx = rs.Context(W=sp.W, K=sp.K, theta1=sp.theta1, theta2=sp.theta2)
    out["load_spike_plan"] = {**timed(ctx, [b.desc() for b in sdev],
                                      [rs.replica_params(r) for r in sp.replicas],
                                      sum(r.n_req for r in sp.replicas) * sp.W),
                              "replicas": len(sp.replicas)}
    ctx.close()
    del dev, sdev
    torch.cuda.empty_cache()
    return out


def _aux_probe(rs, n_route: int = 4096, n_probe: int = 60000, reps: int = 5,
               cache_blocks=None) -> dict:
    """Outside the timed steps: the batch probe (route_probe: S2's cached
    prefix for many requests against one cache snapshot) where its tables do
    not fit in L2: a router instance of 64 workers with 2^20-block caches (the
    W = 64 workload's), filled by routing that workload's first n_route
    requests, then the next n_probe requests probed.  The call hashes the
    batch, then probes; the probe kernel's time is the call's device time
    (CUDA events) less a block-hash call on the same batch.  lookups = sum
    over (request, worker) of min(m_ij + 1, nb_i); algorithmic bytes = 32 B
    per lookup (one bucket sector) + 8 B per block hash (read once, then
    reused by the request's W pairs) + 4 B per m_ij written."""
    import torch
    from paper_2606_17081_gb300 import workloads as wk
    p = wk.plan("large", n_req=n_route + n_probe)
    tr = p.traces()[0]
    W, K = p.W, (cache_blocks or p.K)
    ctx = rs.Context(W=W, K=K, n_instances=1)
    d = rs.device_trace(tr)
    wo = torch.zeros(n_route, dtype=torch.int32, device="cuda")
    rs.route_batch(ctx.h, 0, d.tokens, d.offsets, n_route, d.out_len, wo)
    m = tr.n_req - n_route
    offs = d.offsets[n_route:]
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
    lookups = int(np.minimum(pre + 1, nb).sum())
    kern = min(tp) - min(th)
    alg = 32.0 * lookups + 8.0 * float(nb.sum()) + 4.0 * m * W
    peak, kind = _peaks()
    return {"workers": W, "cache_blocks": K, "table_bytes": _table_bytes(K) * W,
            "routed": n_route, "probed": m, "pairs": m * W, "lookups": lookups,
            "mean_prefix": float(pre.mean()), "call_ms": min(tp), "hash_ms": min(th),
            "kernel_ms": kern, "lookups_per_s": lookups / (kern / 1e3),
            "alg_bytes": alg, "alg_gbs": alg / (kern / 1e3) / 1e9,
            "frac": alg / (kern / 1e3) / 1e9 / peak, "peak_kind": kind}


def run_gpu(args):
    import torch
    import torch.distributed as dist
    from paper_2606_17081_gb300 import routesim as rs

    ws, rank, local = _dist()
    torch.cuda.set_device(local)
    if ws > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    name = args.workload
    if args.probe_only:
        if rank == 0:
            print(json.dumps({"probe_batch_hbm": _aux_probe(rs, cache_blocks=args.probe_cache_blocks)}))
        return
    p, lo, hi = _plan(name, rank, ws, args.n_req, args.replicas)
    full = args.n_req is None and args.replicas is None
    traces = p.traces()
    ctx = rs.Context(W=p.W, K=p.K, theta1=p.theta1, theta2=p.theta2)
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
    e2e_steps = max(1, min(args.steps, args.e2e_steps))
    step(descs_h, rs.RS_MEM_HOST)
    barrier()
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(e2e_steps):
        step(descs_h, rs.RS_MEM_HOST)
    torch.cuda.synchronize()
    barrier()
    e2e_s = time.perf_counter() - t0
    status = [int(r.status) for r in res]
    assert all(s == 0 for s in status), status
    ms, e2e_s = _max_over_ranks([ms, e2e_s], "cuda")
    total_decisions = _sum_over_ranks(decisions, "cuda")
    total_replicas = _sum_over_ranks(len(params), "cuda")
    if rank != 0:
        if ws > 1:
            dist.destroy_process_group()
        return
    peak, peak_kind = _peaks()
    ctx_keep = ctx
    aux = {}
    if not args.no_aux:
        aux["per_config"] = _per_config(rs, peak, peak_kind, skip=(name,))
        aux["variants"] = _aux_variants(rs)
        aux["probe_batch_hbm"] = _aux_probe(rs)
    per_step_s = ms / 1e3 / args.steps
    value = total_decisions / per_step_s
    sim_avg = statistics.mean(sim_ms)
    roof = _roofline(res, p.W, sim_avg, peak, peak_kind)
    roof["traffic"] = _sim_traffic(full and ws == 1)
    roof["traffic_source"] = SIM_TRAFFIC["summary"]
    roof["traffic_scaled_from"] = SIM_TRAFFIC["scaled_from"]
    roof["note"] = (f"latency-bound event loop: {len(params)} simulations, "
                    f"{'two' if len(params) > 152 else 'one'} resident per SM")
    hash_avg = statistics.mean(hash_ms)
    nblocks = sum(int(np.sum(np.diff(t.offsets) // 16)) for t in traces)
    hash_bytes = 4.0 * hashed_tokens + 8.0 * nblocks
    hash_gbs = hash_bytes / (hash_avg / 1e3) / 1e9
    h2d = sum(b.tokens.numel() * 4 + b.offsets.numel() * 8 + b.release.numel() * 8 +
              b.out_len.numel() * 4 for b in host)
    d2h = len(params) * ctypes.sizeof(rs.rs_replica_result) + 8 * len(traces)
    poa = [r.poa_total for r in res]
    cpu = None if args.no_cpu_baseline else cpu_baseline(p, traces, budget_s=args.cpu_budget)
    line = {
        "metric": METRIC, "value": value, "unit": "decisions/s", "n_gpus": ws,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms / args.steps,
        "higher_is_better": True, "scaling": "strong", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded traces shaped like the paper's chat workload)",
        "config": {"workload": WORKLOAD_DESC[name], "name": name,
                   "simulations": total_replicas,
                   "requests_per_replica": p.replicas[0].n_req, "W": p.W,
                   "cache_blocks": p.K,
                   "parallelism": f"replicas of one plan partitioned over {ws} GPU(s)",
                   "l2": "inputs larger than L2 every step (%.0f MB of tokens read, %.0f MB of "
                         "cache tables cleared and rebuilt per step; L2 129 MB)" % (
                             sum(t.tokens.nbytes for t in traces) / 1e6,
                             _table_bytes(p.K) * p.W * len(params) / 1e6)},
        "replicas_per_s": total_replicas / per_step_s,
        "requests_per_s": total_decisions / p.W / per_step_s,
        "kernels_ms_per_step": {"block_hash": hash_avg, "simulate": sim_avg,
                                "poa": statistics.mean(poa_ms)},
        "roofline": roof,
        "hash_roofline": {"kernel": "k_block_hash (launches only)", "bound": "hbm",
                          "achieved": hash_gbs, "peak": peak, "unit": "GB/s",
                          "frac": hash_gbs / peak, "alg_bytes_per_launch_set": hash_bytes},
        "poa_total_mean": float(np.mean(poa)),
        "e2e": {"value": total_decisions / (e2e_s / e2e_steps), "unit": "decisions/s",
                "steps": e2e_steps, "h2d_bytes_per_step": int(h2d),
                "d2h_bytes_per_step": int(d2h)},
        "clocks": clocks,
        "gpu_launches": int(launches),
        "cpu_baseline": cpu,
        "aux": aux,
    }
    print(json.dumps(line))
    del ctx_keep
    if ws > 1:
        dist.destroy_process_group()


def _sum_over_ranks(v, device):
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return v
    t = torch.tensor([float(v)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return type(v)(t.item())


def _oracle_replicas(args):
    """Worker of the all-cores baseline: whole replicas of the plan, one after
    another, until the budget is spent; returns (replicas, decisions, s)."""
    name, idx, budget, W, K, th1, th2 = args
    sys.path.insert(0, ROOT)
    import oracle as O
    from paper_2606_17081_gb300 import workloads as wk
    p = wk.plan(name)
    cfg = O.OracleConfig(W=W, K=K, theta1=th1, theta2=th2)
    cache = {}
    done = dec = 0
    t0 = time.perf_counter()
    for k in idx:
        r = p.replicas[k]
        if r.trace not in cache:
            cache[r.trace] = wk.make_trace(p.spec, p.trace_seeds[r.trace])
        o = O.simulate(cfg, cache[r.trace], r.C, policy=r.policy, controller=r.controller,
                       omega=r.omega, tau=r.tau, seed=r.seed, n_req=r.n_req)
        O.poa(cfg, o)
        done += 1
        dec += r.n_req * W
        if time.perf_counter() - t0 > budget:
            break
    return done, dec, time.perf_counter() - t0


def _cpu_model() -> str:
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.startswith("Model name:"):
                return line.split(":", 1)[1].strip()
    except Exception:
        pass
    return platform.processor() or platform.machine()


def cpu_baseline(p, traces, budget_s: float = 15.0) -> dict:
    """The oracle on whole replicas of the workload until the budget is spent:
    on one core, and on every host core at once (one process per core, each
    on its own replicas, spawned so that no CUDA state is inherited)."""
    import multiprocessing as mp
    import oracle as O
    cfg = O.OracleConfig(W=p.W, K=p.K, theta1=p.theta1, theta2=p.theta2)
    done = dec = 0
    t0 = time.perf_counter()
    order = list(range(len(p.replicas)))
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
    ncpu = os.cpu_count() or 1
    allc = None
    try:
        ctxm = mp.get_context("spawn")
        jobs = [(p.name, order[c::ncpu], budget_s, p.W, p.K, p.theta1, p.theta2)
                for c in range(ncpu)]
        t1 = time.perf_counter()
        with ctxm.Pool(ncpu) as pool:
            parts = pool.map(_oracle_replicas, jobs)
        wall = time.perf_counter() - t1
        rd = sum(x[0] for x in parts)
        dd = sum(x[1] for x in parts)
        slow = max(x[2] for x in parts)
        allc = {"value": dd / slow, "unit": "decisions/s", "cores": ncpu, "replicas": rd,
                "wall_s": wall, "sample": f"{rd} whole replicas over {ncpu} processes "
                                          f"(replica k on process k mod {ncpu}), incl. PoA; "
                                          f"decisions over the slowest process's time"}
    except Exception as e:   # the one-core figure stands alone
        allc = {"unavailable": str(e)[:200]}
    return {"value": dec / el, "unit": "decisions/s", "cores": 1, "kind": "oracle",
            "host_cores": ncpu, "cpu_model": _cpu_model(),
            "sample": f"{done} whole replicas of the {len(p.replicas)} ({p.replicas[0].n_req} "
                      f"requests each, in plan order) incl. PoA, single thread, {el:.1f} s",
            "all_cores": allc}


def run_reference(args):
    """Reference arm: the CPU oracle on a bounded sample of the same workload."""
    ws, rank, local = _dist()
    if rank != 0:
        return
    from paper_2606_17081_gb300 import workloads as wk
    name = getattr(args, "workload", HEADLINE)
    p = wk.plan(name)
    import oracle as O
    cfg = O.OracleConfig(W=p.W, K=p.K, theta1=p.theta1, theta2=p.theta2)
    reps = p.replicas[:2]        # the first cell's selfish and load-balanced simulations
    traces = {r.trace: wk.make_trace(p.spec, p.trace_seeds[r.trace]) for r in reps}

    def step():
        for r in reps:
            o = O.simulate(cfg, traces[r.trace], r.C, policy=r.policy, controller=r.controller,
                           omega=r.omega, tau=r.tau, seed=r.seed, n_req=r.n_req)
            O.poa(cfg, o)

    for _ in range(args.warmup):
        step()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        step()
    el = time.perf_counter() - t0
    dec = sum(r.n_req for r in reps) * p.W * args.steps
    v = dec / el
    sample = (f"2 whole simulations per step (the first cell, selfish and load-balanced, "
              f"{reps[0].n_req} requests each) incl. PoA, oracle single thread")
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": v, "unit": "decisions/s",
        "n_gpus": ws, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": el * 1e3 / args.steps, "higher_is_better": True, "scaling": "strong",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": WORKLOAD_DESC[name], "name": name},
        "cpu_baseline": {"value": v, "unit": "decisions/s", "cores": 1, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": v, "unit": "decisions/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0}}))


def arg_parser() -> argparse.ArgumentParser:
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="native", choices=["native", "reference"])
    ap.add_argument("--workload", default=HEADLINE, choices=sorted(WORKLOAD_DESC))
    ap.add_argument("--e2e-steps", type=int, default=5,
                    help="steps of the end-to-end (host buffers) measurement")
    ap.add_argument("--cpu-budget", type=float, default=15.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-aux", action="store_true",
                    help="skip the timings reported under aux (other workloads, variants, "
                         "batch probe)")
    ap.add_argument("--n-req", type=int, default=None,
                    help="truncate every replica's trace (profiling of a small case)")
    ap.add_argument("--replicas", default=None,
                    help="profiling of a small case: the plan's first N replicas, or "
                         "'per-trace' (the first replica of every trace)")
    ap.add_argument("--probe-only", action="store_true",
                    help="run only the batch-probe measurement (aux.probe_batch_hbm)")
    ap.add_argument("--probe-cache-blocks", type=int, default=None,
                    help="cache blocks per worker of the batch-probe instance "
                         "(default: the W = 64 workload's 2^20)")
    return ap


def main():
    args = arg_parser().parse_args()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
