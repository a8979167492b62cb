"""Python binding of libroutesim.so (include/routesim.h) -- marshalling only.

Functions carry the C entry points' names and arguments; pointers may be
given as integers, torch tensors or numpy arrays.  Every step of the
computation runs in the CUDA library: if it is not built this module raises,
it never falls back to anything else.  PyTorch is used only for device
memory and streams.
"""
from __future__ import annotations

import ctypes as C
import os
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libroutesim.so")

RS_OK, RS_ERR_INVALID, RS_ERR_OOM, RS_ERR_CAPACITY = 0, -1, -2, -3
RS_ERR_CUDA, RS_ERR_TIMEOUT, RS_ERR_STATE, RS_ERR_COLLISION = -4, -5, -6, -7
RS_POLICY_DYNAMO, RS_POLICY_LOADBAL = 0, 1
RS_POLICY_ROUNDROBIN, RS_POLICY_RANDOM, RS_POLICY_P2C = 2, 3, 4
RS_MEM_DEVICE, RS_MEM_HOST = 0, 1
RS_EVICT_LRU, RS_EVICT_FREQ = 0, 1
RS_SIM_NO_POA = 1


class rs_config(C.Structure):
    _fields_ = [("W", C.c_int32), ("block_size", C.c_int32), ("cache_blocks", C.c_int64),
                ("hash_seed", C.c_uint64), ("omega", C.c_float), ("tau", C.c_float),
                ("seed", C.c_uint64), ("lat_a", C.c_double), ("lat_b", C.c_double),
                ("lat_d", C.c_double), ("cap", C.c_int32), ("hyst_k", C.c_int32),
                ("w_c", C.c_double), ("itl", C.c_double), ("dt", C.c_double),
                ("alpha", C.c_double), ("theta1", C.c_double), ("theta2", C.c_double),
                ("eps_frac", C.c_double), ("regime_tau", C.c_float * 3),
                ("regime_omega", C.c_float * 3), ("poa_window", C.c_double),
                ("tiered", C.c_int32), ("tier_node", C.c_int32), ("tier_k2", C.c_int64),
                ("tier_k3", C.c_int64), ("tier_alpha", C.c_double * 3), ("tier_gamma", C.c_double),
                ("tier_d_near", C.c_double), ("tier_d_far", C.c_double)]


class rs_trace(C.Structure):
    _fields_ = [("tokens", C.c_void_p), ("offsets", C.c_void_p), ("release", C.c_void_p),
                ("out_len", C.c_void_p), ("n_req", C.c_int64), ("hashes", C.c_void_p)]


class rs_replica_params(C.Structure):
    _fields_ = [("trace", C.c_int32), ("C", C.c_int32), ("policy", C.c_int32),
                ("controller", C.c_int32), ("omega", C.c_float), ("tau", C.c_float),
                ("seed", C.c_uint64), ("n_req", C.c_int64), ("c_t1", C.c_double),
                ("c_t2", C.c_double), ("c_mid", C.c_int32), ("c_end", C.c_int32),
                ("eviction", C.c_int32), ("freq_max", C.c_int32), ("decay_s", C.c_double)]


class rs_replica_result(C.Structure):
    _fields_ = [("status", C.c_int32), ("final_regime", C.c_int32), ("n_routed", C.c_int64),
                ("sum_ttft", C.c_double), ("sum_e2e", C.c_double), ("makespan", C.c_double),
                ("poa_total", C.c_double), ("n_windows", C.c_int64), ("near_ties", C.c_int64),
                ("exact_ties", C.c_int64), ("sampled", C.c_int64), ("near_boundary", C.c_int64),
                ("hit_blocks", C.c_int64), ("inserted_blocks", C.c_int64),
                ("evicted_blocks", C.c_int64), ("ticks", C.c_int64),
                ("regime_switches", C.c_int64), ("max_regime", C.c_int32),
                ("reserved0", C.c_int32), ("ticks_in_regime", C.c_int64 * 3),
                ("final_ewma", C.c_double), ("probes", C.c_int64),
                ("probe_blocks", C.c_int64), ("hashed_blocks", C.c_int64),
                ("slow_path", C.c_int64), ("rebuilds", C.c_int64),
                ("first_switch_t", C.c_double), ("poa_static", C.c_double),
                ("first_evict_t", C.c_double), ("rho_first_evict", C.c_double),
                ("rho_end", C.c_double), ("kv_g1", C.c_int64), ("kv_g2", C.c_int64),
                ("kv_g3", C.c_int64), ("kv_remote", C.c_int64), ("kv_recompute", C.c_int64),
                ("kv_cost", C.c_double)]

    def as_dict(self) -> dict:
        return {f: (list(getattr(self, f)) if f == "ticks_in_regime" else getattr(self, f))
                for f, _ in self._fields_ if f != "reserved0"}


class rs_records(C.Structure):
    _fields_ = [("worker", C.c_void_p), ("arrival", C.c_void_p), ("start", C.c_void_p),
                ("first_token", C.c_void_p), ("completion", C.c_void_p), ("ttft", C.c_void_p),
                ("nbt", C.c_void_p), ("n_frozen", C.c_void_p), ("prefix", C.c_void_p),
                ("cost", C.c_void_p), ("kv_cost", C.c_void_p)]


class rs_timing(C.Structure):
    _fields_ = [("hash_ms", C.c_float), ("sim_ms", C.c_float), ("poa_ms", C.c_float),
                ("total_ms", C.c_float), ("launches", C.c_int64), ("hashed_tokens", C.c_int64)]


EXPORTS = ["rs_config_default", "route_init", "route_destroy", "route_last_error",
           "route_hash_blocks", "route_dup_flags", "route_batch", "route_probe", "route_release", "route_active",
           "simulate_replicas", "poa_estimate", "route_cache_dump", "route_last_timing",
           "poa_estimate_noalloc", "sweep_knee"]

_lib = None


class RoutesimError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"routesim status {status}: {message}")
        self.status = status


def lib():
    """The loaded CUDA library; raises if it has not been built."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with "
                               "`python -c 'import __graft_entry__ as g; g.build()'`")
        L = C.CDLL(LIB_PATH)
        vp, i32, i64 = C.c_void_p, C.c_int32, C.c_int64
        sig = {
            "rs_config_default": (None, [C.POINTER(rs_config)]),
            "route_init": (i32, [C.POINTER(vp), C.POINTER(rs_config), i32, vp]),
            "route_destroy": (None, [vp]),
            "route_last_error": (C.c_char_p, [vp]),
            "route_hash_blocks": (i32, [vp, vp, vp, i64, vp]),
            "route_dup_flags": (i32, [vp, vp, vp, i64, i64, vp]),
            "route_batch": (i32, [vp, i32, vp, vp, i32, vp, vp, vp, vp]),
            "route_probe": (i32, [vp, i32, vp, vp, i64, vp]),
            "route_release": (i32, [vp, i32, vp, vp, i32]),
            "route_active": (i32, [vp, i32, vp]),
            "simulate_replicas": (i32, [vp, C.POINTER(rs_trace), i32, i32,
                                        C.POINTER(rs_replica_params), i32,
                                        C.POINTER(rs_replica_result), C.POINTER(rs_records), i32]),
            "poa_estimate": (i32, [vp, C.POINTER(rs_records), i64, vp, vp, vp,
                                   C.POINTER(C.c_int64), C.POINTER(C.c_double)]),
            "route_cache_dump": (i32, [vp, i32, i32, i32, vp, i64, C.POINTER(C.c_int64)]),
            "route_last_timing": (i32, [vp, C.POINTER(rs_timing)]),
            "poa_estimate_noalloc": (i32, [C.POINTER(rs_config), C.POINTER(rs_records), i64, vp,
                                           vp, vp, i64, vp, vp, vp]),
            "sweep_knee": (i32, [vp, C.POINTER(rs_records), vp, i32, vp, vp, i32, i32,
                                 C.c_double, vp, vp, vp, vp, vp]),
        }
        for name, (res, args) in sig.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def _ptr(x):
    if x is None:
        return None
    if isinstance(x, int):
        return C.c_void_p(x)
    if hasattr(x, "data_ptr"):
        return C.c_void_p(x.data_ptr())
    if isinstance(x, np.ndarray):
        return C.c_void_p(x.ctypes.data)
    raise TypeError(f"cannot pass {type(x)} as a pointer")


def _check(st: int, ctx) -> None:
    if st != RS_OK:
        raise RoutesimError(st, route_last_error(ctx))


# ----------------------------------------------------------------- entry points

def rs_config_default() -> rs_config:
    c = rs_config()
    lib().rs_config_default(C.byref(c))
    return c


def route_last_error(ctx) -> str:
    m = lib().route_last_error(ctx)
    return m.decode() if m else ""


def route_init(cfg: rs_config, n_instances: int = 0, stream: int = 0):
    h = C.c_void_p()
    st = lib().route_init(C.byref(h), C.byref(cfg), n_instances, C.c_void_p(stream or None))
    _check(st, None)
    return h


def route_destroy(ctx) -> None:
    lib().route_destroy(ctx)


def route_hash_blocks(ctx, tokens, offsets, n_req: int, hashes) -> None:
    _check(lib().route_hash_blocks(ctx, _ptr(tokens), _ptr(offsets), n_req, _ptr(hashes)), ctx)


def route_dup_flags(ctx, hashes, offsets, n_req: int, max_blocks: int, flags) -> None:
    _check(lib().route_dup_flags(ctx, _ptr(hashes), _ptr(offsets), n_req, max_blocks,
                                 _ptr(flags)), ctx)


def route_probe(ctx, instance: int, tokens, offsets, n_req: int, prefix_out) -> None:
    _check(lib().route_probe(ctx, instance, _ptr(tokens), _ptr(offsets), n_req,
                             _ptr(prefix_out)), ctx)


def route_batch(ctx, instance: int, tokens, offsets, n_req: int, out_len, worker_out,
                cost_out=None, prefix_out=None) -> None:
    _check(lib().route_batch(ctx, instance, _ptr(tokens), _ptr(offsets), n_req, _ptr(out_len),
                             _ptr(worker_out), _ptr(cost_out), _ptr(prefix_out)), ctx)


def route_release(ctx, instance: int, worker, blocks, n: int) -> None:
    _check(lib().route_release(ctx, instance, _ptr(worker), _ptr(blocks), n), ctx)


def route_active(ctx, instance: int, W: int) -> np.ndarray:
    out = np.zeros(W, np.int64)
    _check(lib().route_active(ctx, instance, _ptr(out)), ctx)
    return out


def simulate_replicas(ctx, traces, trace_mem: int, params, records: rs_records | None = None,
                      flags: int = 0):
    """traces: sequence of rs_trace; params: sequence of rs_replica_params.
    Returns the ctypes array of rs_replica_result (raises on a non-OK status,
    with the per-replica results attached as `.results`)."""
    tr = (rs_trace * max(len(traces), 1))(*traces)
    pr = (rs_replica_params * max(len(params), 1))(*params)
    res = (rs_replica_result * max(len(params), 1))()
    st = lib().simulate_replicas(ctx, tr, len(traces), trace_mem, pr, len(params), res,
                                 C.byref(records) if records is not None else None, flags)
    if st != RS_OK:
        e = RoutesimError(st, route_last_error(ctx))
        e.results = res
        raise e
    return res


def poa_estimate(ctx, records: rs_records, n: int, max_windows: int):
    numer = np.zeros(max(max_windows, 1))
    opt = np.zeros(max(max_windows, 1))
    cnt = np.zeros(max(max_windows, 1), np.int64)
    nw = C.c_int64(max_windows)
    tot = C.c_double()
    _check(lib().poa_estimate(ctx, C.byref(records), n, _ptr(numer), _ptr(opt), _ptr(cnt),
                              C.byref(nw), C.byref(tot)), ctx)
    k = min(nw.value, max_windows)
    return numer[:k], opt[:k], cnt[:k], float(tot.value), int(nw.value)


def route_cache_dump(ctx, source: int, index: int, worker: int, capacity: int) -> np.ndarray:
    keys = np.zeros(max(capacity, 1), np.uint64)
    size = C.c_int64()
    _check(lib().route_cache_dump(ctx, source, index, worker, _ptr(keys), capacity,
                                  C.byref(size)), ctx)
    return keys[: min(size.value, capacity)].copy()


def route_last_timing(ctx) -> rs_timing:
    t = rs_timing()
    lib().route_last_timing(ctx, C.byref(t))
    return t


def sweep_knee(ctx, records: rs_records, row_start, load, sweep_start, pct: int = 99,
               theta: float = 0.0) -> dict:
    """Saturation knee of load sweeps over device records: per-replica
    percentile of routed TTFTs, divided differences, first interior level with
    a second difference above theta."""
    rows = np.ascontiguousarray(row_start, np.int64)
    ld = np.ascontiguousarray(load, np.float64)
    sw = np.ascontiguousarray(sweep_start, np.int32)
    nr, ns = rows.size - 1, sw.size - 1
    out = {"stat": np.zeros(max(nr, 1)), "d1": np.zeros(max(nr, 1)), "d2": np.zeros(max(nr, 1)),
           "knee_load": np.zeros(max(ns, 1)), "knee_index": np.zeros(max(ns, 1), np.int32)}
    _check(lib().sweep_knee(ctx, C.byref(records), _ptr(rows), nr, _ptr(ld), _ptr(sw), ns, pct,
                            theta, _ptr(out["stat"]), _ptr(out["d1"]), _ptr(out["d2"]),
                            _ptr(out["knee_load"]), _ptr(out["knee_index"])), ctx)
    for k in ("stat", "d1", "d2"):
        out[k] = out[k][:nr]
    for k in ("knee_load", "knee_index"):
        out[k] = out[k][:ns]
    return out


def poa_estimate_noalloc(cfg: rs_config, records: rs_records, n: int, numer_dev, opt_dev,
                         count_dev, max_windows: int, poa_total_dev, n_windows_dev,
                         stream: int = 0) -> None:
    """Same result as poa_estimate, computed in the library's fixed static
    device array (nothing allocated, for callers that cannot allocate device
    memory); outputs stay in device memory."""
    st = lib().poa_estimate_noalloc(C.byref(cfg), C.byref(records), n, _ptr(numer_dev),
                                    _ptr(opt_dev), _ptr(count_dev), max_windows,
                                    _ptr(poa_total_dev), _ptr(n_windows_dev),
                                    C.c_void_p(stream or None))
    if st != RS_OK:
        raise RoutesimError(st, "poa_estimate_noalloc rejected the call")


# ----------------------------------------------------------------- marshalling helpers

@dataclass
class TraceBuffers:
    """A trace's arrays in one memory space, kept alive with its descriptor.
    tokens None: the trace is given by its block hashes (`hashes`)."""
    tokens: object
    offsets: object
    release: object
    out_len: object
    n_req: int
    hashes: object = None

    def desc(self) -> rs_trace:
        tok = _ptr(self.tokens)
        return rs_trace(tok.value if tok is not None else None, _ptr(self.offsets).value,
                        _ptr(self.release).value, _ptr(self.out_len).value, self.n_req,
                        _ptr(self.hashes).value if self.tokens is None else None)


def device_trace(trace, device="cuda") -> TraceBuffers:
    import torch
    return TraceBuffers(torch.from_numpy(trace.tokens).to(device),
                        torch.from_numpy(trace.offsets).to(device),
                        torch.from_numpy(trace.release).to(device),
                        torch.from_numpy(trace.out_len).to(device), trace.n_req)


def host_trace(trace, pinned: bool = True) -> TraceBuffers:
    import torch
    conv = (lambda a: torch.from_numpy(a).pin_memory()) if pinned else torch.from_numpy
    return TraceBuffers(conv(trace.tokens), conv(trace.offsets), conv(trace.release),
                        conv(trace.out_len), trace.n_req)


def replica_params(r) -> rs_replica_params:
    return rs_replica_params(r.trace, r.C, r.policy, r.controller, r.omega, r.tau, r.seed, r.n_req,
                             float(getattr(r, "c_t1", 0.0)), float(getattr(r, "c_t2", 0.0)),
                             int(getattr(r, "c_mid", 0)), int(getattr(r, "c_end", 0)),
                             int(getattr(r, "eviction", RS_EVICT_LRU)),
                             int(getattr(r, "freq_max", 64)), float(getattr(r, "decay_s", 1.0)))


def device_records(rows: int, W: int, device="cuda", with_cost: bool = False,
                   with_kv: bool = False):
    """Caller-owned record tensors and the rs_records struct pointing at them."""
    import torch
    t = {
        "worker": torch.full((rows,), -1, dtype=torch.int32, device=device),
        "arrival": torch.zeros(rows, dtype=torch.float64, device=device),
        "start": torch.zeros(rows, dtype=torch.float64, device=device),
        "first_token": torch.zeros(rows, dtype=torch.float64, device=device),
        "completion": torch.zeros(rows, dtype=torch.float64, device=device),
        "ttft": torch.zeros(rows, dtype=torch.float64, device=device),
        "nbt": torch.zeros(rows, dtype=torch.int32, device=device),
        "n_frozen": torch.zeros(rows * W, dtype=torch.int16, device=device),
        "prefix": torch.zeros(rows * W, dtype=torch.int16, device=device),
    }
    if with_cost:
        t["cost"] = torch.zeros(rows * W, dtype=torch.float32, device=device)
    if with_kv:
        t["kv_cost"] = torch.zeros(rows, dtype=torch.float64, device=device)
    rec = rs_records(*[t[k].data_ptr() if k in t else None for k, _ in rs_records._fields_])
    return rec, t


class Context:
    """Owns one rs_ctx (route_init / route_destroy)."""

    def __init__(self, W: int, K: int, n_instances: int = 0, stream: int = 0, **fields):
        cfg = rs_config_default()
        cfg.W = W
        cfg.cache_blocks = K
        for k, v in fields.items():
            if k in ("regime_tau", "regime_omega"):
                setattr(cfg, k, (C.c_float * 3)(*v))
            elif k == "tier_alpha":
                setattr(cfg, k, (C.c_double * 3)(*v))
            else:
                setattr(cfg, k, v)
        self.cfg = cfg
        self.W = W
        self.K = K
        self.h = route_init(cfg, n_instances, stream)

    def close(self):
        if getattr(self, "h", None) is not None:
            route_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
