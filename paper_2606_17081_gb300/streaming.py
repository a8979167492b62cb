"""Block hashing (S1) of traces too large to hold as tokens.

A prompt enters the router only through the block hashes of §2.2, and Eq. (1)'s
cached-prefix term is computed from them.  For a trace of billions of tokens
(the W = 64 workload: about 2.7 G tokens, 10.8 GB, per trace) the tokens are
therefore produced chunk by chunk into one device buffer and hashed there with
route_hash_blocks; only the 8-byte hashes of the whole trace stay in HBM, and
simulate_replicas takes the trace by its hashes (rs_trace.tokens = NULL).

Chunks hold whole requests and start on a 16-token boundary b: hashing
requests i0 .. i1-1 from a buffer that starts at token b, with offsets rebased
by b and the output advanced by b / 16, writes exactly their entries of the
trace's hash layout (request i's k-th hash at floor(offsets[i] / 16) + k).
This module only orders the calls; the hashing runs in the library's kernel
and the tokens come from the caller's producer (the seeded generator of
`workloads`).
"""
from __future__ import annotations

import numpy as np

from . import routesim as rs


def hash_streamed(ctx, meta, n_req=None, chunk_tokens: int = 1 << 26, device="cuda",
                  timing: dict | None = None) -> rs.TraceBuffers:
    """The first n_req requests of `meta` (a workloads.TraceMeta) as a device
    trace given by its block hashes.  `timing` (optional dict) receives the
    device time of the token production and of the hash calls (ms) and the
    token count."""
    import torch
    n = meta.n_req if n_req is None else min(int(n_req), meta.n_req)
    offs = meta.offsets[: n + 1]
    total = int(offs[-1])
    longest = int(np.diff(offs).max()) if n else 0
    chunk = max(int(chunk_tokens), longest + 32)
    dev_tab = meta.device(device)
    offs_dev = torch.from_numpy(np.ascontiguousarray(offs)).to(device)
    hashes = torch.zeros(total // 16 + 1, dtype=torch.int64, device=device)
    buf = torch.zeros(chunk + 64, dtype=torch.int32, device=device)
    ev = [] if timing is not None else None
    i0 = 0
    while i0 < n:
        base = (int(offs[i0]) // 16) * 16
        # the most whole requests whose tokens fit the buffer from base on
        i1 = int(np.searchsorted(offs, base + chunk, side="right")) - 1
        i1 = min(max(i1, i0 + 1), n)
        end = int(offs[i1])
        cnt = (end - base + 3) // 4 * 4
        if ev is not None:
            e = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
            e[0].record()
        meta.fill_device(dev_tab, base, base + cnt, buf)
        rel = offs_dev[i0:i1 + 1] - base
        if ev is not None:
            e[1].record()
        rs.route_hash_blocks(ctx.h, buf, rel, i1 - i0, hashes.data_ptr() + 8 * (base // 16))
        if ev is not None:
            e[2].record()
            ev.append(e)
        # (one stream: the next fill waits for this hash; rel's memory is
        # reused in stream order)
        i0 = i1
    if timing is not None:
        torch.cuda.synchronize()
        timing["fill_ms"] = sum(e[0].elapsed_time(e[1]) for e in ev)
        timing["hash_ms"] = sum(e[1].elapsed_time(e[2]) for e in ev)
        timing["tokens"] = total
        timing["blocks"] = int(np.sum(np.diff(offs) // 16))
        timing["chunks"] = len(ev)
    del buf
    return rs.TraceBuffers(None, offs_dev,
                           torch.from_numpy(np.ascontiguousarray(meta.release[:n])).to(device),
                           torch.from_numpy(np.ascontiguousarray(meta.out_len[:n])).to(device),
                           n, hashes)
