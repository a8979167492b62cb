"""Seeded synthetic request traces and replica grids (inputs only).

This module draws the inputs that both the CUDA path and the CPU oracle consume:
token ids, prompt/output lengths, prefix-group structure and release times.  It
holds none of the method's arithmetic (no hashing, no routing, no latency model):
everything here is a random draw or a table of workload shapes.

Workload shapes follow the paper's serving experiments, scaled up (§7.4: chat
prompts drawn from a few shared templates, closed-loop concurrency C held by a
semaphore; §7.7: the concurrency sweeps, the 4x4 (tau, omega) sweep, the
adaptive-controller runs).  The paper's own prompt templates are not
reproduced; prompts are uniform token ids with shared-prefix groups.

Token layout: one int32 array, requests stored back to back (CSR `offsets`,
int64, n+1 entries), the array padded with zeros to a multiple of 4 entries so
that 16-byte vector loads never leave it.

Two ways of drawing the tokens:
  "stream"   one numpy draw for the whole trace (every workload but the largest);
  "counter"  for traces too large to draw or hold on the host (the W = 64
             workload: about 2.7 G tokens per trace).  The random suffix token
             at position x of the trace's token array is the (x+1)-th output
             of SplitMix64 (Steele, Lea & Flood, OOPSLA 2014) from a per-trace
             key, reduced to the vocabulary by Lemire's multiply-shift
             ((z >> 32) * vocab) >> 32; prefix tokens come from the group's
             prefix, as in "stream".  Any range of positions can then be
             produced on its own: on the host with numpy (`TraceMeta.tokens`)
             or on the device with torch integer ops (`TraceMeta.fill_device`),
             bit for bit the same.
"""
from __future__ import annotations

from dataclasses import dataclass, field, replace
from typing import Optional

import numpy as np

VOCAB = 32000
BLOCK = 16

POLICY_DYNAMO = 0    # router cost of Eq. (1): omega * prefill blocks + active blocks
POLICY_LOADBAL = 1   # coordinated: the same cost with omega = 0, tau = 0
# static counterfactual policies (the routing-baselines discussion, §9)
POLICY_ROUNDROBIN = 2   # request i -> worker i mod W
POLICY_RANDOM = 3       # uniform worker from a Philox draw
POLICY_P2C = 4          # two distinct uniform workers, the lower Eq. (1) cost


@dataclass(frozen=True)
class TraceSpec:
    n_req: int
    vocab: int = VOCAB
    len_kind: str = "lognormal"       # "lognormal" | "uniform"
    len_median: float = 1024.0
    len_sigma: float = 0.75
    len_min: int = 16
    len_max: int = 8192
    n_groups: int = 64
    prefix_min: int = 512
    prefix_max: int = 2048
    zipf_s: Optional[float] = 1.1     # None: uniform group popularity
    out_kind: str = "lognormal"       # "lognormal" | "uniform"
    out_median: float = 256.0
    out_sigma: float = 0.5
    out_min: int = 1
    out_max: int = 4096
    rate: Optional[float] = None      # Poisson arrival rate (req/s); None = closed loop
    tokens: str = "stream"            # "stream" | "counter" (see the module docstring)
    n_meta: Optional[int] = None      # "counter": requests whose lengths etc. are drawn (>= n_req),
                                      # so that a shorter n_req gives a prefix of the full trace


@dataclass
class Trace:
    tokens: np.ndarray    # int32 [round_up(offsets[-1], 4)]
    offsets: np.ndarray   # int64 [n+1]
    release: np.ndarray   # float64 [n], seconds
    out_len: np.ndarray   # int32 [n]
    group: np.ndarray     # int32 [n], prefix group (diagnostic)

    @property
    def n_req(self) -> int:
        return int(self.offsets.shape[0] - 1)

    @property
    def n_tokens(self) -> int:
        return int(self.offsets[-1])

    def head(self, n: int) -> "Trace":
        """The first n requests as a trace of their own (same token bytes)."""
        n = min(n, self.n_req)
        end = int(self.offsets[n])
        pad = (-end) % 4
        toks = self.tokens[:end]
        if pad:
            toks = np.concatenate([toks, np.zeros(pad, np.int32)])
        return Trace(np.ascontiguousarray(toks), self.offsets[: n + 1].copy(),
                     self.release[:n].copy(), self.out_len[:n].copy(), self.group[:n].copy())


def _lengths(rng, kind, median, sigma, lo, hi, n):
    if kind == "uniform":
        return rng.integers(lo, hi + 1, size=n).astype(np.int64)
    x = np.exp(rng.normal(np.log(median), sigma, size=n))
    return np.clip(np.rint(x), lo, hi).astype(np.int64)


def make_trace(spec: TraceSpec, seed: int) -> Trace:
    """Draw one trace.  Same (spec, seed) -> same bytes on any machine with numpy."""
    if spec.tokens == "counter":
        return trace_meta(spec, seed).trace(spec.n_req)
    rng = np.random.default_rng([int(seed), 0x5EED7ACE])
    n = int(spec.n_req)
    G = int(spec.n_groups)
    plen = rng.integers(spec.prefix_min, spec.prefix_max + 1, size=G).astype(np.int64)
    prefixes = [rng.integers(0, spec.vocab, size=int(p), dtype=np.int32) for p in plen]
    if spec.zipf_s is None:
        group = rng.integers(0, G, size=n).astype(np.int32)
    else:
        w = 1.0 / np.power(np.arange(1, G + 1, dtype=np.float64), spec.zipf_s)
        group = rng.choice(G, size=n, p=w / w.sum()).astype(np.int32)
    L = _lengths(rng, spec.len_kind, spec.len_median, spec.len_sigma, spec.len_min, spec.len_max, n)
    O = _lengths(rng, spec.out_kind, spec.out_median, spec.out_sigma, spec.out_min, spec.out_max, n)
    if spec.rate is None:
        release = np.zeros(n, np.float64)
    else:
        release = np.cumsum(rng.exponential(1.0 / spec.rate, size=n))
    offsets = np.zeros(n + 1, np.int64)
    np.cumsum(L, out=offsets[1:])
    total = int(offsets[-1])
    tokens = np.zeros(total + ((-total) % 4), np.int32)
    tokens[:total] = rng.integers(0, spec.vocab, size=total, dtype=np.int32)
    for i in range(n):
        g = int(group[i])
        k = int(min(plen[g], L[i]))
        o = int(offsets[i])
        tokens[o:o + k] = prefixes[g][:k]
    return Trace(tokens, offsets, release.astype(np.float64), O.astype(np.int32), group)


# SplitMix64 (Steele, Lea & Flood, OOPSLA 2014): state_n = key + n * GAMMA, and
# output_n is the state passed through its finalizer (two xor-shift-multiply
# rounds and a last xor-shift).
SM_GAMMA = 0x9E3779B97F4A7C15
SM_M1 = 0xBF58476D1CE4E5B9
SM_M2 = 0x94D049BB133111EB


def sm_output_np(x: np.ndarray, key: int) -> np.ndarray:
    """SplitMix64 outputs number x + 1 (x >= 0, int64 array) from `key`."""
    z = (np.asarray(x).astype(np.uint64) + np.uint64(1)) * np.uint64(SM_GAMMA) + np.uint64(key)
    z = (z ^ (z >> np.uint64(30))) * np.uint64(SM_M1)
    z = (z ^ (z >> np.uint64(27))) * np.uint64(SM_M2)
    return z ^ (z >> np.uint64(31))


def _sm_tokens_np(x: np.ndarray, key: int, vocab: int) -> np.ndarray:
    """Suffix tokens at trace positions x (int64): Lemire reduction of the
    high 32 bits of SplitMix64 output x + 1."""
    z = sm_output_np(x, key)
    return (((z >> np.uint64(32)) * np.uint64(vocab)) >> np.uint64(32)).astype(np.int32)


def _s64(c: int) -> int:
    """A 64-bit constant as the signed value with the same bits."""
    return c - (1 << 64) if c >= (1 << 63) else c


def _sm_tokens_torch(x, key: int, vocab: int):
    """The same on int64 torch tensors: products wrap modulo 2^64 and shifts
    are made logical by masking the sign-extended bits."""
    def lsr(z, k):
        return (z >> k) & ((1 << (64 - k)) - 1)
    z = (x + 1) * _s64(SM_GAMMA) + _s64(key)
    z = (z ^ lsr(z, 30)) * _s64(SM_M1)
    z = (z ^ lsr(z, 27)) * _s64(SM_M2)
    z = z ^ lsr(z, 31)
    import torch
    return ((lsr(z, 32) * vocab) >> 32).to(torch.int32)


@dataclass
class TraceMeta:
    """A "counter" trace without its tokens: per-request lengths, groups and
    times for n_meta requests, the groups' prefix tokens (`pool`, CSR by
    `pool_off`) and the suffix stream's key.  Tokens of any position range
    come from `tokens` (host) or `fill_device` (device), identically."""
    offsets: np.ndarray   # int64 [n+1]
    release: np.ndarray   # float64 [n]
    out_len: np.ndarray   # int32 [n]
    group: np.ndarray     # int32 [n]
    kpref: np.ndarray     # int64 [n]: leading tokens taken from the group's prefix
    pool: np.ndarray      # int32: the groups' prefixes back to back
    pool_off: np.ndarray  # int64 [G+1]
    key: int
    vocab: int

    @property
    def n_req(self) -> int:
        return int(self.offsets.shape[0] - 1)

    def tokens(self, x0: int, x1: int) -> np.ndarray:
        """int32 tokens at trace positions x0 .. x1-1 (positions past the last
        request hold suffix-stream values)."""
        out = _sm_tokens_np(np.arange(x0, x1, dtype=np.int64), self.key, self.vocab)
        # the leading kpref[i] tokens of every request in range come from its prefix
        i0 = max(int(np.searchsorted(self.offsets, x0, side="right")) - 1, 0)
        i1 = min(int(np.searchsorted(self.offsets, x1, side="left")), self.n_req)
        for i in range(i0, i1):
            a = int(self.offsets[i])
            b = a + int(self.kpref[i])
            lo, hi = max(a, x0), min(b, x1)
            if lo < hi:
                src = int(self.pool_off[int(self.group[i])]) + (lo - a)
                out[lo - x0:hi - x0] = self.pool[src:src + (hi - lo)]
        return out

    def trace(self, n: int) -> Trace:
        """The first n requests with their tokens (host memory)."""
        n = min(int(n), self.n_req)
        end = int(self.offsets[n])
        toks = np.zeros(end + ((-end) % 4), np.int32)
        step = 1 << 24
        for x0 in range(0, end, step):
            x1 = min(end, x0 + step)
            toks[x0:x1] = self.tokens(x0, x1)
        return Trace(toks, self.offsets[: n + 1].copy(), self.release[:n].copy(),
                     self.out_len[:n].copy(), self.group[:n].copy())

    def device(self, device="cuda") -> dict:
        """The tables `fill_device` reads, as device tensors."""
        import torch
        return {k: torch.from_numpy(getattr(self, k)).to(device)
                for k in ("offsets", "group", "kpref", "pool", "pool_off")}

    def fill_device(self, dev: dict, x0: int, x1: int, out, step: int = 1 << 25) -> None:
        """Writes the tokens of positions x0 .. x1-1 into the int32 device
        tensor `out` (at least x1 - x0 entries) with torch integer ops, in
        steps of `step` positions."""
        import torch
        offs, grp, kp = dev["offsets"], dev["group"], dev["kpref"]
        pool, poff = dev["pool"], dev["pool_off"]
        n = self.n_req
        for a in range(x0, x1, step):
            b = min(x1, a + step)
            x = torch.arange(a, b, dtype=torch.int64, device=offs.device)
            req = (torch.searchsorted(offs, x, right=True) - 1).clamp_(max=n - 1)
            p = x - offs[req]
            k = kp[req]
            idx = poff[grp[req].long()] + torch.minimum(p, k - 1).clamp_(min=0)
            pre = pool[idx.clamp_(max=pool.numel() - 1)]
            suf = _sm_tokens_torch(x, self.key, self.vocab)
            out[a - x0:b - x0] = torch.where(p < k, pre, suf)


def trace_meta(spec: TraceSpec, seed: int) -> TraceMeta:
    """Lengths, groups, times and prefix tokens of a "counter" trace, drawn for
    spec.n_meta (default n_req) requests; the suffix tokens are never drawn
    here.  Same (spec, seed) -> same values on any machine with numpy."""
    rng = np.random.default_rng([int(seed), 0x5EED7ACE])
    n = int(spec.n_meta if spec.n_meta is not None else spec.n_req)
    G = int(spec.n_groups)
    plen = rng.integers(spec.prefix_min, spec.prefix_max + 1, size=G).astype(np.int64)
    pool = rng.integers(0, spec.vocab, size=int(plen.sum()), dtype=np.int32)
    pool_off = np.zeros(G + 1, np.int64)
    np.cumsum(plen, out=pool_off[1:])
    if spec.zipf_s is None:
        group = rng.integers(0, G, size=n).astype(np.int32)
    else:
        w = 1.0 / np.power(np.arange(1, G + 1, dtype=np.float64), spec.zipf_s)
        group = rng.choice(G, size=n, p=w / w.sum()).astype(np.int32)
    L = _lengths(rng, spec.len_kind, spec.len_median, spec.len_sigma, spec.len_min, spec.len_max, n)
    O = _lengths(rng, spec.out_kind, spec.out_median, spec.out_sigma, spec.out_min, spec.out_max, n)
    if spec.rate is None:
        release = np.zeros(n, np.float64)
    else:
        release = np.cumsum(rng.exponential(1.0 / spec.rate, size=n))
    key = int(rng.integers(0, 1 << 63, dtype=np.int64)) * 2 + int(rng.integers(0, 2))
    offsets = np.zeros(n + 1, np.int64)
    np.cumsum(L, out=offsets[1:])
    kpref = np.minimum(plen[group], L).astype(np.int64)
    return TraceMeta(offsets, release.astype(np.float64), O.astype(np.int32), group, kpref, pool,
                     pool_off, key, int(spec.vocab))


@dataclass
class Replica:
    trace: int            # index into Plan.trace_seeds
    C: int                # closed-loop concurrency
    policy: int           # POLICY_DYNAMO | POLICY_LOADBAL
    controller: int       # 1: adaptive controller of §6 on
    omega: float
    tau: float
    seed: int             # Philox key for temperature sampling
    n_req: int            # requests of the trace this replica routes
    # load-spike schedule (Experiment 3): C before c_t1, c_mid on [c_t1, c_t2),
    # c_end after; c_mid = 0 keeps C throughout
    c_t1: float = 0.0
    c_t2: float = 0.0
    c_mid: int = 0
    c_end: int = 0
    # cache eviction: 0 exact LRU, 1 the KV Block Manager's frequency rule
    # with its frequency cap and decay step (s)
    eviction: int = 0
    freq_max: int = 64
    decay_s: float = 1.0


@dataclass
class Plan:
    name: str
    W: int
    K: int                                  # cache blocks per worker
    spec: TraceSpec
    trace_seeds: list
    replicas: list = field(default_factory=list)
    theta1: float = 0.3                     # s, 70B thresholds of §6.2
    theta2: float = 2.0

    def traces(self):
        return [make_trace(self.spec, s) for s in self.trace_seeds]

    def metas(self):
        """The traces without tokens ("counter" specs only), each cut to
        spec.n_req requests."""
        out = []
        for s in self.trace_seeds:
            m = trace_meta(self.spec, s)
            n = self.spec.n_req
            out.append(TraceMeta(m.offsets[: n + 1].copy(), m.release[:n].copy(),
                                 m.out_len[:n].copy(), m.group[:n].copy(), m.kpref[:n].copy(),
                                 m.pool, m.pool_off, m.key, m.vocab))
        return out


TINY_SPEC = TraceSpec(n_req=512, len_kind="uniform", len_min=64, len_max=512,
                      n_groups=16, prefix_min=256, prefix_max=256, zipf_s=None,
                      out_kind="uniform", out_min=16, out_max=256, rate=50.0)
P2D_SPEC = TraceSpec(n_req=20000)
P5D_SPEC = TraceSpec(n_req=50000)
GRID_SPEC = TraceSpec(n_req=10000)
LARGE_SPEC = TraceSpec(n_req=1_000_000, len_median=2048.0, len_max=32768, n_groups=1024,
                       zipf_s=1.0, tokens="counter", n_meta=1_000_000)


def plan(name: str, n_req: Optional[int] = None, replicas: Optional[list] = None) -> Plan:
    """The replica grid of one workload.

    n_req truncates every trace (tests run the oracle on a prefix); `replicas`
    keeps only the listed replica indices (in that order).
    """
    if name == "tiny":
        spec = TINY_SPEC
        p = Plan(name, W=3, K=2048, spec=spec, trace_seeds=[0])
        p.replicas = [Replica(0, 16, POLICY_DYNAMO, 0, 1.0, 0.0, 0, spec.n_req)]
    elif name == "p2d":
        # 70B 1P/2D-shaped: W=3, C sweep, selfish vs load-balanced on the same trace.
        spec = P2D_SPEC
        Cs = [16, 32, 64, 128, 256]
        reps = []
        for r in range(64):
            pol = POLICY_DYNAMO if (r // 5) % 2 == 0 else POLICY_LOADBAL
            om = 1.0 if pol == POLICY_DYNAMO else 0.0
            reps.append(Replica(r // 10, Cs[r % 5], pol, 0, om, 0.0, r // 10, spec.n_req))
        p = Plan(name, W=3, K=65536, spec=spec, trace_seeds=list(range(7)), replicas=reps)
    elif name == "p5d":
        # 70B 1P/5D-shaped: W=6, C x T cells, adaptive controller on.
        spec = P5D_SPEC
        Cs = [32, 64, 128, 256, 512]
        Ts = [0.0, 0.5, 1.0]
        reps = []
        for r in range(256):
            cell = r % 15
            reps.append(Replica(r // 15, Cs[cell % 5], POLICY_DYNAMO, 1, 1.0, Ts[cell // 5],
                                r // 15, spec.n_req))
        p = Plan(name, W=6, K=65536, spec=spec, trace_seeds=list(range(18)), replicas=reps)
    elif name == "grid":
        # omega x C x T x seed; every cell also runs the coordinated policy on its trace.
        spec = GRID_SPEC
        Ws = [0.0, 0.25, 0.5, 1.0, 2.0, 4.0]
        Cs = [16, 32, 64, 128, 256, 512]
        Ts = [0.0, 0.5, 1.0]
        reps = []
        for r in range(4096):
            cell = r % 108
            rs = r // 108
            ts = rs % 8
            C = Cs[(cell // 6) % 6]
            reps.append(Replica(ts, C, POLICY_DYNAMO, 0, Ws[cell % 6], Ts[cell // 36], rs, spec.n_req))
            reps.append(Replica(ts, C, POLICY_LOADBAL, 0, 0.0, 0.0, rs, spec.n_req))
        p = Plan(name, W=6, K=32768, spec=spec, trace_seeds=list(range(8)), replicas=reps)
    elif name == "spike":
        # Experiment 3's three-phase load spike, C = 32 -> 128 -> 32 for
        # 120 / 180 / 120 s, on the 70B 1P/2D topology (2 decode workers):
        # static routing (tau = 0, omega = 1 throughout) against the adaptive
        # controller, three seeds each; the requests outlast the 420 s.
        spec = P2D_SPEC
        reps = []
        for sd in range(3):
            for ctl in (0, 1):
                reps.append(Replica(sd, 32, POLICY_DYNAMO, ctl, 1.0, 0.0, sd, 9000,
                                    c_t1=120.0, c_t2=300.0, c_mid=128, c_end=32))
        p = Plan(name, W=2, K=65536, spec=spec, trace_seeds=list(range(3)), replicas=reps)
    elif name == "sat":
        # Experiment 2's saturation sweep: nine concurrency levels on the 70B
        # 1P/2D topology, static routing and the adaptive controller, three
        # seeds; each (seed, controller) pair is one sweep of increasing C.
        spec = P2D_SPEC
        Cs = [1, 4, 8, 16, 32, 64, 128, 256, 512]
        reps = []
        for sd in range(3):
            for ctl in (0, 1):
                for C in Cs:
                    reps.append(Replica(sd, C, POLICY_DYNAMO, ctl, 1.0, 0.0, sd, 6000))
        p = Plan(name, W=3, K=65536, spec=spec, trace_seeds=list(range(3)), replicas=reps)
    elif name == "large":
        spec = LARGE_SPEC
        reps = []
        for r in range(16):
            pol = POLICY_DYNAMO if r < 8 else POLICY_LOADBAL
            reps.append(Replica(r % 8, 4096, pol, 0, 1.0 if pol == POLICY_DYNAMO else 0.0, 0.0,
                                r % 8, spec.n_req))
        p = Plan(name, W=64, K=1 << 20, spec=spec, trace_seeds=list(range(8)), replicas=reps)
    else:
        raise ValueError(f"unknown workload {name!r}")
    if n_req is not None:
        p.spec = replace(p.spec, n_req=min(n_req, p.spec.n_req))
        for r in p.replicas:
            r.n_req = min(r.n_req, p.spec.n_req)
    if replicas is not None:
        keep = [p.replicas[i] for i in replicas]
        used = sorted({r.trace for r in keep})
        remap = {t: k for k, t in enumerate(used)}
        p.trace_seeds = [p.trace_seeds[t] for t in used]
        for r in keep:
            r.trace = remap[r.trace]
        p.replicas = keep
    return p


def sweeps(replicas) -> list:
    """Boundaries of the load sweeps of a replica list: maximal runs of
    consecutive replicas that differ only in C, with C increasing.  Returns
    sweep_start (len = sweeps + 1) for the knee detector."""
    def same(a, b):
        return (a.trace, a.policy, a.controller, a.omega, a.tau, a.seed, a.n_req, a.c_t1,
                a.c_t2, a.c_mid, a.c_end) == (b.trace, b.policy, b.controller, b.omega, b.tau,
                                              b.seed, b.n_req, b.c_t1, b.c_t2, b.c_mid, b.c_end)
    start = [0]
    for k in range(1, len(replicas)):
        a, b = replicas[k - 1], replicas[k]
        if not (same(a, b) and b.C > a.C):
            start.append(k)
    if replicas:
        start.append(len(replicas))
    return start
