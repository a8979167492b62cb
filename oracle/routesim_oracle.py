"""ctypes wrapper of the C oracle (liboracle.so) -- test infrastructure.

Argument marshalling only: every step of the computation is in
`routesim_oracle.c`.  The shared object is compiled from that single file with
gcc (`build_oracle`), in place, on whichever machine runs the tests.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
from dataclasses import dataclass, field

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "routesim_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")

OK, ERR_INVALID, ERR_OOM, ERR_CAPACITY, ERR_COLLISION = 0, -1, -2, -3, -7
POLICY_DYNAMO, POLICY_LOADBAL = 0, 1
# static counterfactual policies of the routing-baselines discussion (§9)
POLICY_ROUNDROBIN, POLICY_RANDOM, POLICY_P2C = 2, 3, 4
# cache eviction: exact LRU, or the KV Block Manager's frequency rule (§2.2)
EVICT_LRU, EVICT_FREQ = 0, 1


def build_oracle(force: bool = False) -> str:
    """Compile liboracle.so next to its source (single-threaded C, no FMA contraction)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < max(
            os.path.getmtime(_SRC), os.path.getmtime(os.path.join(_HERE, "routesim_oracle.h"))):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math",
                               "-fPIC", "-shared", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


class _Config(C.Structure):
    _fields_ = [("W", C.c_int32), ("block", C.c_int32), ("K", C.c_int64),
                ("hash_seed", C.c_uint64), ("lat_a", C.c_double), ("lat_b", C.c_double),
                ("lat_d", C.c_double), ("cap", C.c_int32), ("w_c", C.c_double),
                ("itl", C.c_double), ("dt", C.c_double), ("alpha", C.c_double),
                ("theta1", C.c_double), ("theta2", C.c_double), ("eps_frac", C.c_double),
                ("hyst_k", C.c_int32), ("regime_tau", C.c_float * 3),
                ("regime_omega", C.c_float * 3), ("poa_window", C.c_double),
                ("tiered", C.c_int32), ("tier_node", C.c_int32), ("tier_k2", C.c_int64),
                ("tier_k3", C.c_int64), ("tier_alpha", C.c_double * 3), ("tier_gamma", C.c_double),
                ("tier_d_near", C.c_double), ("tier_d_far", C.c_double)]


class _Replica(C.Structure):
    _fields_ = [("C", C.c_int32), ("policy", C.c_int32), ("controller", C.c_int32),
                ("omega", C.c_float), ("tau", C.c_float), ("seed", C.c_uint64),
                ("n_req", C.c_int64), ("c_t1", C.c_double), ("c_t2", C.c_double),
                ("c_mid", C.c_int32), ("c_end", C.c_int32), ("eviction", C.c_int32),
                ("freq_max", C.c_int32), ("decay_s", C.c_double)]


class _Summary(C.Structure):
    _fields_ = [("status", C.c_int32), ("n_routed", C.c_int64), ("sum_ttft", C.c_double),
                ("sum_e2e", C.c_double), ("makespan", C.c_double), ("near_ties", C.c_int64),
                ("exact_ties", C.c_int64), ("sampled", C.c_int64), ("near_boundary", C.c_int64),
                ("hit_blocks", C.c_int64), ("inserted_blocks", C.c_int64),
                ("evicted_blocks", C.c_int64), ("ticks", C.c_int64),
                ("regime_switches", C.c_int64), ("final_regime", C.c_int32),
                ("max_regime", C.c_int32), ("ticks_in_regime", C.c_int64 * 3),
                ("final_ewma", C.c_double), ("first_switch_t", C.c_double),
                ("first_evict_t", C.c_double), ("rho_first_evict", C.c_double),
                ("rho_end", C.c_double), ("kv_g1", C.c_int64), ("kv_g2", C.c_int64),
                ("kv_g3", C.c_int64), ("kv_remote", C.c_int64), ("kv_recompute", C.c_int64),
                ("kv_cost", C.c_double)]


class _Records(C.Structure):
    _fields_ = [("worker", C.c_void_p), ("arrival", C.c_void_p), ("start", C.c_void_p),
                ("first_token", C.c_void_p), ("completion", C.c_void_p), ("ttft", C.c_void_p),
                ("nbt", C.c_void_p), ("n_frozen", C.c_void_p), ("prefix", C.c_void_p),
                ("cost", C.c_void_p), ("kv_cost", C.c_void_p)]


@dataclass
class OracleConfig:
    """Model constants.  Defaults: §6.4 cost-matrix constants, §6.2 controller
    (70B thresholds), Table 2 regime parameters."""
    W: int = 3
    K: int = 2048
    block: int = 16
    hash_seed: int = 0
    lat_a: float = 0.005
    lat_b: float = 0.020
    lat_d: float = 0.010
    cap: int = 64
    w_c: float = 0.015
    itl: float = 0.012
    dt: float = 5.0
    alpha: float = 0.3
    theta1: float = 0.3
    theta2: float = 2.0
    eps_frac: float = 0.1
    hyst_k: int = 3
    regime_tau: tuple = (0.0, 0.7, 0.8)
    regime_omega: tuple = (1.0, 1.0, 0.1)
    poa_window: float = 5.0
    # Game 2 tiers (§4.2, Eq. kv-cost); the paper gives no values
    tiered: int = 0
    tier_node: int = 1
    tier_k2: int = 0
    tier_k3: int = 0
    tier_alpha: tuple = (1.0, 4.0, 20.0)
    tier_gamma: float = 100.0
    tier_d_near: float = 2.0
    tier_d_far: float = 10.0

    @property
    def K_stack(self) -> int:
        """Blocks a worker holds across its tiers."""
        return self.K + (self.tier_k2 + self.tier_k3 if self.tiered else 0)

    def c(self) -> _Config:
        return _Config(self.W, self.block, self.K, self.hash_seed, self.lat_a, self.lat_b,
                       self.lat_d, self.cap, self.w_c, self.itl, self.dt, self.alpha,
                       self.theta1, self.theta2, self.eps_frac, self.hyst_k,
                       (C.c_float * 3)(*self.regime_tau), (C.c_float * 3)(*self.regime_omega),
                       self.poa_window, self.tiered, self.tier_node, self.tier_k2, self.tier_k3,
                       (C.c_double * 3)(*self.tier_alpha), self.tier_gamma, self.tier_d_near,
                       self.tier_d_far)


_lib = None


def lib():
    global _lib
    if _lib is None:
        _lib = C.CDLL(build_oracle())
        L = _lib
        L.orc_mix64.restype = C.c_uint64
        L.orc_mix64.argtypes = [C.c_uint64]
        L.orc_expf.restype = C.c_float
        L.orc_expf.argtypes = [C.c_float]
        L.orc_select.restype = C.c_int32
        L.orc_select.argtypes = [C.c_void_p, C.c_int32, C.c_float, C.c_uint32]
        L.orc_simulate.restype = C.c_int32
        L.orc_poa.restype = C.c_int64
        L.orc_static_numer.restype = C.c_int64
        L.orc_assign.restype = C.c_double
        L.orc_assign.argtypes = [C.c_void_p, C.c_int64, C.c_int32, C.c_int64, C.c_int32,
                                 C.c_void_p]
        L.orc_game_exhaustive.restype = C.c_int32
        L.orc_router_new.restype = C.c_void_p
        L.orc_router_new.argtypes = [C.POINTER(_Config), C.c_float, C.c_float, C.c_uint64,
                                     C.c_int32]
        L.orc_router_free.argtypes = [C.c_void_p]
        L.orc_router_route.restype = C.c_int32
        L.orc_router_release.restype = C.c_int32
        L.orc_router_probe.restype = C.c_int32
        L.orc_router_active.restype = C.c_int32
        L.orc_router_cache.restype = C.c_int32
    return _lib


def _p(a):
    return None if a is None else C.c_void_p(a.ctypes.data)


def _c(a, dt):
    return np.ascontiguousarray(a, dtype=dt)


# --------------------------------------------------------------------------- primitives

def mix64(z: int) -> int:
    return int(lib().orc_mix64(C.c_uint64(z & 0xFFFFFFFFFFFFFFFF)))


def philox4x32_10(ctr, key):
    c = (C.c_uint32 * 4)(*ctr)
    k = (C.c_uint32 * 2)(*key)
    o = (C.c_uint32 * 4)()
    lib().orc_philox4x32_10(c, k, o)
    return tuple(int(v) for v in o)


def expf(x) -> np.ndarray:
    x = _c(np.atleast_1d(x), np.float32)
    y = np.empty_like(x)
    lib().orc_expf_n(_p(x), _p(y), C.c_int64(x.size))
    return y


def select(cost, tau: float, u24: int = 0) -> int:
    c = _c(cost, np.float32)
    return int(lib().orc_select(_p(c), c.size, C.c_float(tau), C.c_uint32(u24)))


def hash_blocks(tokens, offsets, block: int = 16, seed: int = 0) -> np.ndarray:
    t = _c(tokens, np.int32)
    o = _c(offsets, np.int64)
    n = o.size - 1
    out = np.zeros(max(int(o[-1]) // block, 1), np.uint64)
    lib().orc_hash_blocks(_p(t), _p(o), C.c_int64(n), C.c_int32(block), C.c_uint64(seed),
                          _p(out))
    return out[: int(o[-1]) // block]


# --------------------------------------------------------------------------- simulation

def simulate(cfg: OracleConfig, trace, C_: int, policy: int = POLICY_DYNAMO,
             controller: int = 0, omega: float = 1.0, tau: float = 0.0, seed: int = 0,
             n_req=None, want_cache: bool = False, max_ticks: int = 0,
             schedule=None, eviction: int = EVICT_LRU, freq_max: int = 64,
             decay_s: float = 1.0) -> dict:
    """Run one replica.  `trace` has tokens/offsets/release/out_len arrays.
    schedule: None or (c_t1, c_t2, c_mid, c_end), the load-spike concurrency
    of Experiment 3 (C before c_t1, c_mid until c_t2, c_end after).
    eviction: EVICT_LRU, or EVICT_FREQ with its frequency cap and decay step."""
    n = trace.n_req if n_req is None else int(n_req)
    W = cfg.W
    t = _c(trace.tokens, np.int32)
    o = _c(trace.offsets, np.int64)
    rel = _c(trace.release, np.float64)
    ol = _c(trace.out_len, np.int32)
    nn = max(n, 1)
    r = {
        "worker": np.full(nn, -1, np.int32), "arrival": np.zeros(nn), "start": np.zeros(nn),
        "first_token": np.zeros(nn), "completion": np.zeros(nn), "ttft": np.zeros(nn),
        "nbt": np.zeros(nn, np.int32), "n_frozen": np.zeros(nn * W, np.uint16),
        "prefix": np.zeros(nn * W, np.uint16), "cost": np.zeros(nn * W, np.float32),
        "kv_cost": np.zeros(nn),
    }
    rec = _Records(*[_p(r[k]).value for k in ("worker", "arrival", "start", "first_token",
                                                "completion", "ttft", "nbt", "n_frozen",
                                                "prefix", "cost", "kv_cost")])
    st = schedule if schedule is not None else (0.0, 0.0, 0, 0)
    rep = _Replica(C_, policy, controller, omega, tau, seed, n, float(st[0]), float(st[1]),
                   int(st[2]), int(st[3]), int(eviction), int(freq_max), float(decay_s))
    s = _Summary()
    keys = np.zeros(W * cfg.K_stack, np.uint64) if want_cache else None
    sizes = np.zeros(W, np.int64) if want_cache else None
    te = np.zeros(max(max_ticks, 1)) if max_ticks else None
    tr = np.zeros(max(max_ticks, 1), np.int32) if max_ticks else None
    cc = cfg.c()
    st = lib().orc_simulate(C.byref(cc), _p(t), _p(o), _p(rel), _p(ol), C.byref(rep),
                            C.byref(rec), C.byref(s), _p(keys), _p(sizes), _p(te), _p(tr),
                            C.c_int64(max_ticks))
    out = {k: v[:n] if v.size == nn else v[: n * W] for k, v in r.items()}
    for k in ("n_frozen", "prefix", "cost"):
        out[k] = out[k].reshape(n, W)
    out["status"] = int(st)
    out["summary"] = {f: (list(getattr(s, f)) if f == "ticks_in_regime" else getattr(s, f))
                      for f, _ in _Summary._fields_}
    if want_cache:
        ks = cfg.K_stack
        out["cache"] = [keys[j * ks: j * ks + int(sizes[j])].copy() for j in range(W)]
    if max_ticks:
        k = min(int(s.ticks), max_ticks)
        out["tick_ewma"] = te[:k].copy()
        out["tick_regime"] = tr[:k].copy()
    return out


def poa(cfg: OracleConfig, rec: dict, method: int = 0):
    """Eq. (12) over completion-time windows; returns (numer, opt, count, total)."""
    n = rec["worker"].size
    W = cfg.W
    wk = _c(rec["worker"], np.int32)
    ct = _c(rec["completion"], np.float64)
    tt = _c(rec["ttft"], np.float64)
    nbt = _c(rec["nbt"], np.int32)
    nf = _c(np.asarray(rec["n_frozen"]).reshape(-1), np.uint16)
    pf = _c(np.asarray(rec["prefix"]).reshape(-1), np.uint16)
    routed = ct[wk >= 0]
    cap = int(np.floor(routed.max() / cfg.poa_window)) + 2 if routed.size else 1
    numer = np.zeros(cap)
    opt = np.zeros(cap)
    cnt = np.zeros(cap, np.int64)
    total = C.c_double(0.0)
    cc = cfg.c()
    nw = lib().orc_poa(C.byref(cc), C.c_int64(n), _p(wk), _p(ct), _p(tt), _p(nbt), _p(nf),
                       _p(pf), C.c_int32(method), _p(numer), _p(opt), _p(cnt), C.c_int64(cap),
                       C.byref(total))
    if nw < 0:
        raise RuntimeError(f"orc_poa failed: {nw}")
    return numer[:nw], opt[:nw], cnt[:nw], float(total.value)


def static_numer(cfg: OracleConfig, rec: dict):
    """Per Eq. (12) window, the frozen §6.4 cost of the realized assignment
    (the static counterfactual of §9): sum over the window of c_{i, worker(i)}."""
    n = rec["worker"].size
    wk = _c(rec["worker"], np.int32)
    ct = _c(rec["completion"], np.float64)
    nbt = _c(rec["nbt"], np.int32)
    nf = _c(np.asarray(rec["n_frozen"]).reshape(-1), np.uint16)
    pf = _c(np.asarray(rec["prefix"]).reshape(-1), np.uint16)
    routed = ct[wk >= 0]
    cap = int(np.floor(routed.max() / cfg.poa_window)) + 2 if routed.size else 1
    out = np.zeros(cap)
    cc = cfg.c()
    nw = lib().orc_static_numer(C.byref(cc), C.c_int64(n), _p(wk), _p(ct), _p(nbt), _p(nf),
                                _p(pf), _p(out), C.c_int64(cap))
    if nw < 0:
        raise RuntimeError(f"orc_static_numer failed: {nw}")
    return out[:nw]


def poa_static(cfg: OracleConfig, rec: dict) -> float:
    """Sum of the realized assignment's frozen costs over the sum of window OPTs."""
    _, opt, _, _ = poa(cfg, rec)
    st = static_numer(cfg, rec)
    to = float(np.sum(opt))
    return float(np.sum(st)) / to if to > 0 else 0.0


def assign(cost, capw: int, method: int = 1):
    c = _c(cost, np.float64)
    n, W = c.shape
    a = np.zeros(max(n, 1), np.int32)
    v = lib().orc_assign(_p(c), C.c_int64(n), C.c_int32(W), C.c_int64(capw), C.c_int32(method),
                         _p(a))
    return float(v), a[:n]


def game_exhaustive(o, omega: float, lat_a=0.005, lat_b=0.020, lat_d=0.010, cap=64) -> dict:
    o = _c(o, np.float64)
    n, W = o.shape
    opt, worst, best, greedy = (C.c_double() for _ in range(4))
    nne, steps = C.c_int64(), C.c_int64()
    spread = C.c_int32()
    st = lib().orc_game_exhaustive(C.c_int32(n), C.c_int32(W), _p(o), C.c_double(omega),
                                   C.c_double(lat_a), C.c_double(lat_b), C.c_double(lat_d),
                                   C.c_int32(cap), C.byref(opt), C.byref(worst), C.byref(best),
                                   C.byref(greedy), C.byref(nne), C.byref(steps),
                                   C.byref(spread))
    if st != 0:
        raise ValueError("invalid game instance")
    return {"opt": opt.value, "worst_ne": worst.value, "best_ne": best.value,
            "greedy": greedy.value, "n_ne": nne.value, "br_steps": steps.value,
            "max_ne_spread": spread.value}


class Router:
    """Live router (route_batch / route_release semantics), oracle side."""

    def __init__(self, cfg: OracleConfig, omega: float, tau: float, seed: int, n_instances: int = 1):
        self.cfg = cfg
        self._cc = cfg.c()
        self.h = lib().orc_router_new(C.byref(self._cc), omega, tau, seed, n_instances)
        if not self.h:
            raise ValueError("invalid router parameters")

    def __del__(self):
        if getattr(self, "h", None):
            lib().orc_router_free(C.c_void_p(self.h))
            self.h = None

    def route(self, instance, tokens, offsets, out_len):
        t = _c(tokens, np.int32)
        o = _c(offsets, np.int64)
        ol = _c(out_len, np.int32)
        n = o.size - 1
        W = self.cfg.W
        wk = np.zeros(max(n, 1), np.int32)
        cost = np.zeros(max(n, 1) * W, np.float32)
        pre = np.zeros(max(n, 1) * W, np.int32)
        st = lib().orc_router_route(C.c_void_p(self.h), C.c_int32(instance), _p(t), _p(o),
                                    C.c_int64(n), _p(ol), _p(wk), _p(cost), _p(pre))
        return st, wk[:n], cost[: n * W].reshape(n, W), pre[: n * W].reshape(n, W)

    def probe(self, instance, tokens, offsets):
        """m_ij of every request on every worker against the current caches
        (nothing updated): (status, int32 [n, W])."""
        t = _c(tokens, np.int32)
        o = _c(offsets, np.int64)
        n = o.size - 1
        W = self.cfg.W
        pre = np.zeros(max(n, 1) * W, np.int32)
        st = lib().orc_router_probe(C.c_void_p(self.h), C.c_int32(instance), _p(t), _p(o),
                                    C.c_int64(n), _p(pre))
        return st, pre[: n * W].reshape(n, W)

    def release(self, instance, worker, blocks):
        w = _c(worker, np.int32)
        b = _c(blocks, np.int32)
        return lib().orc_router_release(C.c_void_p(self.h), C.c_int32(instance), _p(w), _p(b),
                                        C.c_int64(w.size))

    def active(self, instance):
        a = np.zeros(self.cfg.W, np.int64)
        lib().orc_router_active(C.c_void_p(self.h), C.c_int32(instance), _p(a))
        return a

    def cache(self, instance, worker):
        keys = np.zeros(self.cfg.K, np.uint64)
        sz = C.c_int64()
        lib().orc_router_cache(C.c_void_p(self.h), C.c_int32(instance), C.c_int32(worker),
                               _p(keys), C.byref(sz))
        return keys[: sz.value].copy()


def p99(values) -> float:
    v = _c(values, np.float64)
    f = lib().orc_p99
    f.restype = C.c_double
    return float(f(_p(v), C.c_int64(v.size)))


def sweep_knee(worker, ttft, row_start, load, sweep_start, pct: int = 99,
               theta: float = 0.0) -> dict:
    """Saturation knee of load sweeps (§5.1, PoA-growth proposition, item 3;
    Experiment 2): per replica the nearest-rank pct-th percentile of its routed
    TTFTs; per sweep the divided differences d1, d2 and the first interior
    point with d2 > theta (knee_index -1 if none, -2 if loads do not increase)."""
    wk = _c(worker, np.int32)
    tt = _c(ttft, np.float64)
    rows = _c(row_start, np.int64)
    ld = _c(load, np.float64)
    sw = _c(sweep_start, np.int32)
    n_rep = rows.size - 1
    n_sw = sw.size - 1
    out = {"stat": np.zeros(max(n_rep, 1)), "d1": np.zeros(max(n_rep, 1)),
           "d2": np.zeros(max(n_rep, 1)), "knee_load": np.zeros(max(n_sw, 1)),
           "knee_index": np.zeros(max(n_sw, 1), np.int32)}
    st = lib().orc_sweep_knee(C.c_int32(n_rep), _p(rows), _p(wk), _p(tt), _p(ld),
                              C.c_int32(n_sw), _p(sw), C.c_int32(pct), C.c_double(theta),
                              _p(out["stat"]), _p(out["d1"]), _p(out["d2"]),
                              _p(out["knee_load"]), _p(out["knee_index"]))
    if st != OK:
        raise ValueError(f"orc_sweep_knee rejected the input ({st})")
    for k in ("stat", "d1", "d2"):
        out[k] = out[k][:n_rep]
    for k in ("knee_load", "knee_index"):
        out[k] = out[k][:n_sw]
    return out


def controller_run(cfg: OracleConfig, L):
    """Feed per-sample P99 values (NaN = empty window); returns (ewma, regime)."""
    x = _c(L, np.float64)
    e = np.zeros(max(x.size, 1))
    r = np.zeros(max(x.size, 1), np.int32)
    cc = cfg.c()
    lib().orc_controller_run(C.byref(cc), C.c_int64(x.size), _p(x), _p(e), _p(r))
    return e[: x.size], r[: x.size]
