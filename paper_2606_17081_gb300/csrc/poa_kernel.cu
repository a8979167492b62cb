// PoA estimate of Eq. (12) (K4).
//
// k_poa_prep (one CTA per replica): window of every request = floor of its
// completion time over the window length; frozen costs
// c_ij = a n_ij + b + d/(C - n_ij)^2 - w_c o_ij of the §6.4 matrix; a stable
// bucket sort of the requests by window (request order kept inside a window).
//
// k_poa_solve (a few CTAs per replica, one warp per window): OPT of the window =
// minimum-cost assignment of its requests to W workers of capacity
// max(C_j, ceil(n/W)) each (the replicated-column square matrix of §6.4).
// Every request first takes its cheapest worker; that is optimal unless a
// worker exceeds its capacity.  Otherwise the excess requests are taken out
// (what stays is optimal for its own subset: every row sits at its minimum)
// and put back one at a time along a shortest augmenting path (successive
// shortest paths), found by Bellman-Ford on the W worker nodes with edge
// weights min over the requests at j of (c_qk - c_qj).  The edge weights are
// kept across augmentations: a request that moves in lowers its worker's
// weights in O(W); only a worker that lost the request behind one of its
// minima is rescanned.
//
// k_poa_total (one warp per replica): the whole-run PoA, sum of observed
// latency over sum of OPT across the replica's windows; and the static
// counterfactual of §9, the realized assignment's frozen cost over OPT.
#include "rs_device.cuh"

namespace rs {

__device__ __forceinline__ double frozen_cost(const ModelConsts& mc, int nf, int m, int nbt) {
  const double t1 = __dmul_rn(mc.lat_a, (double)nf);
  const double t2 = __dadd_rn(t1, mc.lat_b);
  const double den = (double)(mc.cap - nf);
  const double f = __dadd_rn(t2, __ddiv_rn(mc.lat_d, __dmul_rn(den, den)));
  const double o = nbt > 0 ? __ddiv_rn((double)m, (double)nbt) : 0.0;
  return __dsub_rn(f, __dmul_rn(mc.w_c, o));
}

struct PoaPrepShared {
  long long maxw;
  int overflow;
  int wn[NT_POA / 32];
  int wk[NT_POA / 32][32];
  int wc[NT_POA / 32][32];
  long long scan_w[NT_POA / 32];
  long long carry;
};

__global__ void __launch_bounds__(NT_POA) k_poa_prep(const PoaProblem* __restrict__ probs,
                                                     PoaBuffers b, ModelConsts mc) {
  __shared__ PoaPrepShared P;
  const PoaProblem pr = probs[blockIdx.x];
  const int W = mc.W;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (b.wprob)   // the owner of every window slot of this problem
    for (int64_t w = threadIdx.x; w < pr.win_cap; w += NT_POA) b.wprob[pr.win_base + w] = blockIdx.x;
  if (threadIdx.x == 0) {
    P.maxw = -1;
    P.overflow = W > POA_WMAX_WIDE;
    P.carry = 0;
  }
  if (lane == 0) P.wn[warp] = 0;
  __syncthreads();
  if (P.overflow) {
    if (threadIdx.x == 0) b.nwin[blockIdx.x] = -2;
    return;
  }
  long long mx = -1;
  for (int64_t q = threadIdx.x; q < pr.n; q += NT_POA) {
    const int64_t r = pr.rec_base + q;
    const int wk = b.rec.worker[r];
    int key = -1;
    if (wk >= 0) {
      const long long w = (long long)floor(__ddiv_rn(b.rec.completion[r], mc.poa_window));
      if (w >= pr.win_cap || w < 0) P.overflow = 1;
      else key = (int)w;
      mx = w > mx ? w : mx;
    }
    b.wkey[pr.scratch_base + q] = key;
  }
  for (int o = 16; o > 0; o >>= 1) {
    const long long v = __shfl_xor_sync(FULL_MASK, mx, o);
    mx = v > mx ? v : mx;
  }
  if (lane == 0 && mx >= 0) atomicMax(&P.maxw, mx);
  __syncthreads();
  if (P.overflow) {
    if (threadIdx.x == 0) b.nwin[blockIdx.x] = -1;
    return;
  }
  const int64_t nw = P.maxw + 1;
  int64_t* cnt = b.wcnt + pr.win_base;
  int64_t* wst = b.wstart + pr.win_base + blockIdx.x;   // nw + 1 entries
  int64_t* fill = b.wfill + pr.win_base;
  for (int64_t w = threadIdx.x; w < nw; w += NT_POA) cnt[w] = 0;
  __syncthreads();
  for (int64_t q = threadIdx.x; q < pr.n; q += NT_POA) {
    const int key = b.wkey[pr.scratch_base + q];
    if (key >= 0) atomicAdd(reinterpret_cast<unsigned long long*>(cnt + key), 1ull);
  }
  __syncthreads();
  // exclusive scan of the window counts
  for (int64_t w0 = 0; w0 < nw; w0 += NT_POA) {
    const int64_t w = w0 + threadIdx.x;
    long long v = w < nw ? (long long)cnt[w] : 0;
    long long x = v;
    for (int o = 1; o < 32; o <<= 1) {
      const long long y = __shfl_up_sync(FULL_MASK, x, o);
      if (lane >= o) x += y;
    }
    if (lane == 31) P.scan_w[warp] = x;
    __syncthreads();
    long long off = P.carry;
    for (int i = 0; i < warp; i++) off += P.scan_w[i];
    if (w < nw) {
      wst[w] = off + x - v;
      fill[w] = off + x - v;
    }
    __syncthreads();
    if (threadIdx.x == NT_POA - 1) {
      long long tot = 0;
      for (int i = 0; i < NT_POA / 32; i++) tot += P.scan_w[i];
      P.carry += tot;
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) wst[nw] = P.carry;
  __syncthreads();
  // stable scatter: rank inside the chunk = earlier warps' equal keys + earlier lanes
  for (int64_t q0 = 0; q0 < pr.n; q0 += NT_POA) {
    const int64_t q = q0 + threadIdx.x;
    const int key = q < pr.n ? b.wkey[pr.scratch_base + q] : -1;
    const unsigned peers = __match_any_sync(FULL_MASK, key);
    const int intra = __popc(peers & ((1u << lane) - 1u));
    const bool leader = (__ffs(peers) - 1) == lane;
    if (leader) {
      const int idx = atomicAdd(&P.wn[warp], 1);
      P.wk[warp][idx] = key;
      P.wc[warp][idx] = __popc(peers);
    }
    __syncthreads();
    if (key >= 0) {
      int cross = 0;
      for (int v = 0; v < warp; v++)
        for (int e = 0; e < P.wn[v]; e++)
          if (P.wk[v][e] == key) cross += P.wc[v][e];
      const int64_t d = pr.scratch_base + fill[key] + cross + intra;
      b.order[d] = (int32_t)q;
      // the frozen cost row, stored at the request's sorted position
      const int64_t r = pr.rec_base + q;
      const int nbt = b.rec.nbt[r];
      double* cr = b.cost + d * W;
      for (int j = 0; j < W; j++)
        cr[j] = frozen_cost(mc, b.rec.n_frozen[r * W + j], b.rec.prefix[r * W + j], nbt);
    }
    __syncthreads();
    if (leader && key >= 0)
      atomicAdd(reinterpret_cast<unsigned long long*>(fill + key), (unsigned long long)__popc(peers));
    if (lane == 0) P.wn[warp] = 0;
    __syncthreads();
  }
  if (threadIdx.x == 0) b.nwin[blockIdx.x] = nw;
}

struct PoaWarpShared {
  int counts[POA_WMAX];
  double dist[POA_WMAX];                           // shortest-path distances of one augmentation
  int pred[POA_WMAX];
  double wmin[POA_WMAX][POA_WMAX];
  int wrow[POA_WMAX][POA_WMAX];
  int mv_row[POA_WMAX + 1], mv_to[POA_WMAX + 1];   // requests moved by the last augmentation
  int dirty[POA_WMAX];                             // workers whose edge weights need a rescan
  int nmv;
  double num, opt;
  int err;
};

// Order-preserving map of a double onto uint64: x < y (IEEE, neither NaN,
// not both zero) iff dorder(x) < dorder(y); comparisons on the serial paths
// then run on the integer units instead of the FP64 pipe.
__device__ __forceinline__ uint64_t dorder(double x) {
  const uint64_t u = (uint64_t)__double_as_longlong(x);
  return (u >> 63) ? ~u : (u | 0x8000000000000000ull);
}
__device__ __forceinline__ double dunorder(uint64_t k) {
  const uint64_t u = (k >> 63) ? (k & 0x7FFFFFFFFFFFFFFFull) : ~k;
  return __longlong_as_double((long long)u);
}
constexpr uint64_t DKEY_NONE = ~0ull;   // above dorder of every double but NaN

// Edge weights out of worker j: for every k, the cheapest move of a request now
// at j to k, min over those requests of c_qk - c_qj (ties: lowest row).
template <int WT>
__device__ __forceinline__ void poa_edges_from(PoaWarpShared& S, const PoaBuffers& b,
                                               int64_t base, int64_t m, int W, int j, int lane) {
  // per lane: the cheapest move to each k among its rows, as order keys
  // (registers: the loops run over the compile-time bound WT >= W with k < W
  // guards);
  // four rows per lane in flight, each lane's rows in increasing order so
  // that ties keep the lowest row
  uint64_t lk[WT];
  int lr[WT];
#pragma unroll
  for (int k = 0; k < WT; k++) { lk[k] = DKEY_NONE; lr[k] = -1; }
  for (int64_t r0 = lane; r0 < m; r0 += 128) {
    int at[4];
#pragma unroll
    for (int u = 0; u < 4; u++) at[u] = r0 + 32 * u < m ? b.asg[base + r0 + 32 * u] : -1;
#pragma unroll
    for (int u = 0; u < 4; u++) {
      if (at[u] != j) continue;
      const int64_t r = r0 + 32 * u;
      const double* cr = b.cost + (base + r) * W;
      const double cj = cr[j];
#pragma unroll
      for (int k = 0; k < WT; k++) {
        if (k < W && k != j) {
          const uint64_t key = dorder(__dsub_rn(cr[k], cj));
          if (key < lk[k]) { lk[k] = key; lr[k] = (int)r; }
        }
      }
    }
  }
#pragma unroll
  for (int k = 0; k < WT; k++) {
    if (k < W) {
      uint64_t key = lk[k];
      int rr = lr[k];
      for (int o = 16; o > 0; o >>= 1) {
        const uint64_t k2 = __shfl_xor_sync(FULL_MASK, key, o);
        const int r2 = __shfl_xor_sync(FULL_MASK, rr, o);
        if (r2 >= 0 && (rr < 0 || k2 < key || (k2 == key && r2 < rr))) { key = k2; rr = r2; }
      }
      if (lane == 0) {
        S.wmin[j][k] = rr >= 0 ? dunorder(key) : __longlong_as_double(0x7FF0000000000000ll);
        S.wrow[j][k] = rr;
      }
    }
  }
}

struct PoaSolveShared {
  PoaWarpShared w[NT_POA / 32];
};

__device__ __forceinline__ double warp_sum(double v) {
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(FULL_MASK, v, o);
  return v;
}

// The next window a solver warp takes: with b.wnext the warps of the whole
// grid take window slots from the counter in order (a replica's windows
// spread over the GPU, so a few heavy replicas do not hold the end of the
// launch); without it the warps of problem blockIdx.x's CTAs stride over its
// windows (next, stride).  Returns false when no window is left.
__device__ __forceinline__ bool poa_next(const PoaProblem* __restrict__ probs, const PoaBuffers& b,
                                         int lane, int64_t& next, int64_t stride, int* pi,
                                         int64_t* w) {
  for (;;) {
    if (b.wnext) {
      unsigned long long item = 0;
      if (lane == 0) item = atomicAdd(b.wnext, 1ull);
      item = __shfl_sync(FULL_MASK, item, 0);
      if ((int64_t)item >= b.nslots) return false;
      const int p = b.wprob[item];
      const int64_t ww = (int64_t)item - probs[p].win_base;
      const int64_t nw = b.nwin[p];
      if (nw < 0 || ww >= nw) continue;   // a spare slot, or a problem that overflowed
      *pi = p;
      *w = ww;
      return true;
    }
    const int64_t nw = b.nwin[blockIdx.x];
    const int64_t ww = next;
    next += stride;
    if (nw < 0 || ww >= nw) return false;
    *pi = (int)blockIdx.x;
    *w = ww;
    return true;
  }
}

// WT: a compile-time bound on W (the exact W for the common 3 and 6, else
// POA_WMAX), so that the unrolled per-worker loops hold no dead iterations:
// the solver's warps run different phases at once and its code must stay
// small for the instruction cache.
template <int WT>
__global__ void __launch_bounds__(NT_POA) k_poa_solve(const PoaProblem* __restrict__ probs,
                                                      PoaBuffers b, ModelConsts mc) {
  __shared__ PoaSolveShared P;
  const int W = mc.W;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  PoaWarpShared& S = P.w[warp];
  int64_t next = (int64_t)blockIdx.y * (NT_POA / 32) + warp;
  const int64_t stride = (int64_t)gridDim.y * (NT_POA / 32);
  int pi;
  int64_t w;
  // (a problem whose windows overflowed: k_poa_total reports it)
  while (poa_next(probs, b, lane, next, stride, &pi, &w)) {
    const PoaProblem pr = probs[pi];
    const int64_t* wst = b.wstart + pr.win_base + pi;
    const int64_t s0 = wst[w];
    const int64_t m = wst[w + 1] - s0;
    const int64_t base = pr.scratch_base + s0;   // window rows in order[], asg[]
    if (m == 0) {
      if (lane == 0) {
        b.wnum[pr.win_base + w] = 0.0;
        b.wopt[pr.win_base + w] = 0.0;
        b.wstat[pr.win_base + w] = 0.0;
        b.wcnt[pr.win_base + w] = 0;
      }
      continue;
    }
    int64_t capw = (m + W - 1) / W;
    if (capw < mc.cap) capw = mc.cap;
    if (lane < W) S.counts[lane] = 0;
    if (lane == 0) S.err = 0;
    __syncwarp();
    double num = 0.0, nst = 0.0;
    for (int64_t r = lane; r < m; r += 32) {
      const int q = b.order[base + r];
      const double* cr = b.cost + (base + r) * W;
      nst += cr[b.rec.worker[pr.rec_base + q]];   // the realized assignment's frozen cost
      int best = 0;
      double bc = cr[0];
      for (int j = 1; j < W; j++)
        if (cr[j] < bc) { bc = cr[j]; best = j; }
      b.asg[base + r] = best;
      atomicAdd(&S.counts[best], 1);
      num += b.rec.ttft[pr.rec_base + q];
    }
    num = warp_sum(num);
    nst = warp_sum(nst);
    __syncwarp();
    int over = 0;
    for (int j = 0; j < W; j++) over |= S.counts[j] > capw;
    if (over) {
      // take out the excess, latest rows first
      if (lane == 0) {
        int64_t nrem = 0;
        for (int64_t r = m - 1; r >= 0; r--) {
          const int j = b.asg[base + r];
          if (S.counts[j] > capw) {
            S.counts[j]--;
            b.asg[base + r] = -1;
            b.wkey[base + nrem++] = (int32_t)r;   // wkey reused as the removal list
          }
        }
        S.num = (double)nrem;
      }
      __syncwarp();
      const int64_t nrem = (int64_t)S.num;
      for (int j = 0; j < W; j++) poa_edges_from<WT>(S, b, base, m, W, j, lane);
      __syncwarp();
      for (int64_t e = 0; e < nrem; e++) {
        const int64_t r0 = b.wkey[base + e];
        const double* c0 = b.cost + (base + r0) * W;
        // Bellman-Ford from the request's costs, in Jacobi rounds: lane k < W
        // owns target k and every round reads the previous round's distances
        // (shortest paths have at most W - 1 edges).  Exact cycles are >= 0;
        // relaxing only on gains above 1e-12 keeps rounding-level negative
        // cycles from looping the predecessors.
        double dk = __longlong_as_double(0x7FF0000000000000ll);
        int pk = -1;
        if (lane < W) dk = c0[lane];
        for (int it = 0; it < W; it++) {
          // the best way into k this round (lowest j on ties), then one
          // FP64 test against the gain threshold
          uint64_t bk = DKEY_NONE;
          int bj = -1;
#pragma unroll
          for (int j = 0; j < WT; j++) {
            const double dj = __shfl_sync(FULL_MASK, dk, j);
            if (j < W && lane < W && j != lane && S.wrow[j][lane] >= 0) {
              const uint64_t key = dorder(__dadd_rn(dj, S.wmin[j][lane]));
              if (key < bk) { bk = key; bj = j; }
            }
          }
          int ch = 0;
          if (bj >= 0) {
            const double v = dunorder(bk);
            if (v < dk - 1e-12) { dk = v; pk = bj; ch = 1; }
          }
          if (!__any_sync(FULL_MASK, ch)) break;
        }
        // target: the nearest worker with room (ties: lowest index)
        uint64_t key = ~0ull;
        if (lane < W && S.counts[lane] < capw) key = dorder(dk);
        int tl = lane;
        for (int o = 16; o > 0; o >>= 1) {
          const uint64_t k2 = __shfl_xor_sync(FULL_MASK, key, o);
          const int t2 = __shfl_xor_sync(FULL_MASK, tl, o);
          if (k2 < key || (k2 == key && t2 < tl)) { key = k2; tl = t2; }
        }
        if (lane < W) { S.dist[lane] = dk; S.pred[lane] = pk; }
        __syncwarp();
        if (lane == 0) {
          const int tgt = key == ~0ull ? -1 : tl;
          int nmv = 0;
          for (int j = 0; j < W; j++) S.dirty[j] = 0;
          if (tgt < 0) {
            S.err = 1;
          } else {
            // walk the path back from its end: each edge j -> k moves the
            // request behind S.wrow[j][k] from j to k
            int k = tgt, steps = 0;
            while (S.pred[k] >= 0 && steps <= W) {
              const int j = S.pred[k];
              const int r = S.wrow[j][k];
              S.mv_row[nmv] = r;
              S.mv_to[nmv++] = k;
              // j loses r: its weights need a rescan where r was the minimum
              for (int k2 = 0; k2 < W; k2++) S.dirty[j] |= S.wrow[j][k2] == r;
              k = j;
              steps++;
            }
            if (steps > W) {
              S.err = 1;
              nmv = 0;
            } else {
              for (int t = 0; t < nmv; t++) b.asg[base + S.mv_row[t]] = S.mv_to[t];
              b.asg[base + r0] = k;
              S.mv_row[nmv] = (int)r0;
              S.mv_to[nmv++] = k;
              S.counts[tgt]++;
            }
          }
          S.nmv = nmv;
        }
        __syncwarp();
        if (S.err) break;
        // requests that moved in lower their new worker's weights (lane k2
        // keeps column k2; moves in path order)
        const int nmv = S.nmv;
        for (int t = 0; t < nmv; t++) {
          const int r = S.mv_row[t], to = S.mv_to[t];
          const int k2 = lane;
          if (k2 < W && k2 != to) {
            const double* cr = b.cost + (base + r) * W;
            const double v = __dsub_rn(cr[k2], cr[to]);
            const int wr = S.wrow[to][k2];
            if (wr < 0 || v < S.wmin[to][k2] || (v == S.wmin[to][k2] && r < wr)) {
              S.wmin[to][k2] = v;
              S.wrow[to][k2] = r;
            }
          }
        }
        __syncwarp();
        for (int j = 0; j < W; j++)
          if (S.dirty[j]) poa_edges_from<WT>(S, b, base, m, W, j, lane);
        __syncwarp();
      }
    }
    double opt = 0.0;
    for (int64_t r = lane; r < m; r += 32) {
      const int a = b.asg[base + r];
      opt += a >= 0 ? b.cost[(base + r) * W + a] : __longlong_as_double(0x7FF8000000000000ll);
    }
    opt = warp_sum(opt);
    if (lane == 0) {
      b.wnum[pr.win_base + w] = num;
      b.wstat[pr.win_base + w] = nst;
      b.wopt[pr.win_base + w] = S.err ? __longlong_as_double(0x7FF8000000000000ll) : opt;
      b.wcnt[pr.win_base + w] = m;
    }
    __syncwarp();
  }
}

// The same OPT for W > POA_WMAX workers, one warp per CTA with its window's
// W x W edge weights in shared memory.  Lane l owns the target workers
// k = l, l + 32: it keeps column k of the weights (one pass over the rows
// updates every source at once) and relaxes dist[k] in Bellman-Ford, all
// targets of a round in parallel (rounds until nothing changes, at most W), so
// that no step costs O(W^2) on one lane.
struct PoaWide {
  double* wmin;   // [W][W]
  double* dist;   // [W]
  int* wrow;      // [W][W]
  int* pred;      // [W]
  int* counts;    // [W]
  int* dirty;     // [W]
  int* mv_row;    // [W + 1]
  int* mv_to;     // [W + 1]
};

__host__ __device__ inline size_t poa_wide_smem(int W) {
  const size_t w = (size_t)W;
  return w * w * 12 + w * 12 + w * 8 + 2 * (w + 1) * 4;
}

// Recompute the weights out of every source j with dirty[j] (all of them when
// all is set): min over the requests at j of c_qk - c_qj, ties to the lowest
// row.  Rows go 128 at a time: four assignment loads per lane, the rows at a
// rescanned worker compacted in order into `sel`, then taken four at a time
// with their cost slices loaded together (lane l keeps columns l, l + 32).
__device__ __forceinline__ void wide_rescan(const PoaWide& S, const PoaBuffers& b, int64_t base,
                                            int64_t m, int W, int lane, bool all, int* sel) {
  const double inf = __longlong_as_double(0x7FF0000000000000ll);
  for (int k = lane; k < W; k += 32)
    for (int j = 0; j < W; j++)
      if (all || S.dirty[j]) { S.wmin[j * W + k] = inf; S.wrow[j * W + k] = -1; }
  for (int64_t r0 = 0; r0 < m; r0 += 128) {
    int at[4];
#pragma unroll
    for (int u = 0; u < 4; u++) {
      const int64_t r = r0 + 32 * u + lane;
      at[u] = r < m ? b.asg[base + r] : -1;
    }
    int ns = 0;
#pragma unroll
    for (int u = 0; u < 4; u++) {
      const bool hit = at[u] >= 0 && (all || S.dirty[at[u]]);
      const unsigned msk = __ballot_sync(FULL_MASK, hit);
      if (hit) sel[ns + __popc(msk & ((1u << lane) - 1u))] = (int)(32 * u + lane);
      ns += __popc(msk);
    }
    __syncwarp();
    for (int t0 = 0; t0 < ns; t0 += 4) {
      double c0[4], c1[4], cj[4];
      int rr[4], jj[4];
#pragma unroll
      for (int u = 0; u < 4; u++) {
        rr[u] = -1;
        if (t0 + u < ns) {
          const int64_t r = r0 + sel[t0 + u];
          rr[u] = (int)r;
          jj[u] = b.asg[base + r];
          const double* cr = b.cost + (base + r) * W;
          c0[u] = lane < W ? cr[lane] : 0.0;
          c1[u] = lane + 32 < W ? cr[lane + 32] : 0.0;
          cj[u] = cr[jj[u]];
        }
      }
#pragma unroll
      for (int u = 0; u < 4; u++) {
        if (rr[u] < 0) continue;
        const int j = jj[u];
        if (lane < W && lane != j) {
          const double v = __dsub_rn(c0[u], cj[u]);
          if (v < S.wmin[j * W + lane]) { S.wmin[j * W + lane] = v; S.wrow[j * W + lane] = rr[u]; }
        }
        if (lane + 32 < W && lane + 32 != j) {
          const double v = __dsub_rn(c1[u], cj[u]);
          if (v < S.wmin[j * W + lane + 32]) {
            S.wmin[j * W + lane + 32] = v;
            S.wrow[j * W + lane + 32] = rr[u];
          }
        }
      }
    }
    __syncwarp();
  }
}

__global__ void __launch_bounds__(32, 1) k_poa_solve_wide(const PoaProblem* __restrict__ probs,
                                                       PoaBuffers b, ModelConsts mc) {
  extern __shared__ __align__(16) unsigned char wsm[];
  const int W = mc.W;
  PoaWide S;
  {
    unsigned char* q = wsm;
    S.wmin = reinterpret_cast<double*>(q); q += (size_t)W * W * 8;
    S.dist = reinterpret_cast<double*>(q); q += (size_t)W * 8;
    S.wrow = reinterpret_cast<int*>(q); q += (size_t)W * W * 4;
    S.pred = reinterpret_cast<int*>(q); q += (size_t)W * 4;
    S.counts = reinterpret_cast<int*>(q); q += (size_t)W * 4;
    S.dirty = reinterpret_cast<int*>(q); q += (size_t)W * 4;
    S.mv_row = reinterpret_cast<int*>(q); q += (size_t)(W + 1) * 4;
    S.mv_to = reinterpret_cast<int*>(q);
  }
  __shared__ int s_err, s_nmv;
  __shared__ long long s_nrem;
  __shared__ int s_sel[128];          // rows of a rescan chunk
  __shared__ int s_pj[POA_WMAX_WIDE + 1], s_pr[POA_WMAX_WIDE + 1];   // the last path's edges
  const int lane = threadIdx.x;
  int64_t next = blockIdx.y;
  const int64_t stride = gridDim.y;
  int pi;
  int64_t w;
  while (poa_next(probs, b, lane, next, stride, &pi, &w)) {
    const PoaProblem pr = probs[pi];
    const int64_t* wst = b.wstart + pr.win_base + pi;
    const int64_t s0 = wst[w];
    const int64_t m = wst[w + 1] - s0;
    const int64_t base = pr.scratch_base + s0;
    if (m == 0) {
      if (lane == 0) {
        b.wnum[pr.win_base + w] = 0.0;
        b.wopt[pr.win_base + w] = 0.0;
        b.wstat[pr.win_base + w] = 0.0;
        b.wcnt[pr.win_base + w] = 0;
      }
      continue;
    }
    int64_t capw = (m + W - 1) / W;
    if (capw < mc.cap) capw = mc.cap;
    for (int j = lane; j < W; j += 32) S.counts[j] = 0;
    if (lane == 0) s_err = 0;
    __syncwarp();
    double num = 0.0, nst = 0.0;
    for (int64_t r = lane; r < m; r += 32) {
      const int q = b.order[base + r];
      const double* cr = b.cost + (base + r) * W;
      nst += cr[b.rec.worker[pr.rec_base + q]];
      int best = 0;
      double bc = cr[0];
      for (int j = 1; j < W; j++)
        if (cr[j] < bc) { bc = cr[j]; best = j; }
      b.asg[base + r] = best;
      atomicAdd(&S.counts[best], 1);
      num += b.rec.ttft[pr.rec_base + q];
    }
    num = warp_sum(num);
    nst = warp_sum(nst);
    __syncwarp();
    int over = 0;
    for (int j = lane; j < W; j += 32) over |= S.counts[j] > capw;
    if (__any_sync(FULL_MASK, over)) {
      if (lane == 0) {   // take out the excess, latest rows first
        long long nrem = 0;
        for (int64_t r = m - 1; r >= 0; r--) {
          const int j = b.asg[base + r];
          if (S.counts[j] > capw) {
            S.counts[j]--;
            b.asg[base + r] = -1;
            b.wkey[base + nrem++] = (int32_t)r;
          }
        }
        s_nrem = nrem;
      }
      __syncwarp();
      const int64_t nrem = s_nrem;
      wide_rescan(S, b, base, m, W, lane, true, s_sel);
      __syncwarp();
      for (int64_t e = 0; e < nrem; e++) {
        const int64_t r0 = b.wkey[base + e];
        const double* c0 = b.cost + (base + r0) * W;
        for (int k = lane; k < W; k += 32) { S.dist[k] = c0[k]; S.pred[k] = -1; }
        __syncwarp();
        // Jacobi rounds: every target reads the previous round's distances;
        // the best way into a target (lowest j on ties) is found on order
        // keys, then tested once against the gain threshold.  Only gains
        // above 1e-12 count (exact cycles are >= 0; rounding-level negative
        // ones must not loop the predecessors).  A round relaxes only the
        // edges out of sources whose distance changed in the round before:
        // an edge out of an unchanged source was tested against a distance
        // that has only fallen since, so it cannot pass now.
        uint64_t act = W >= 64 ? ~0ull : ((1ull << W) - 1ull);
        for (int it = 0; it < W && act; it++) {
          int ch[2] = {0, 0};
          double nd[2];
          int np[2];
          uint64_t bk[2] = {DKEY_NONE, DKEY_NONE};
          int bj[2] = {-1, -1};
          // sources four at a time, both targets together: the loads and
          // additions of a group are independent (one warp per CTA has no
          // other warps to hide their latency); sources in increasing order,
          // so ties keep the lowest j
          for (uint64_t a = act; a;) {
            int js[4];
#pragma unroll
            for (int u = 0; u < 4; u++) {
              js[u] = a ? __ffsll((long long)a) - 1 : -1;
              a &= a ? a - 1 : 0ull;
            }
            double dj[4];
#pragma unroll
            for (int u = 0; u < 4; u++) dj[u] = js[u] >= 0 ? S.dist[js[u]] : 0.0;
#pragma unroll
            for (int h = 0; h < 2; h++) {
              const int k = lane + 32 * h;
              if (k >= W) continue;
              uint64_t key[4];
#pragma unroll
              for (int u = 0; u < 4; u++) {
                const int j = js[u];
                key[u] = DKEY_NONE;
                if (j >= 0 && j != k && S.wrow[j * W + k] >= 0)
                  key[u] = dorder(__dadd_rn(dj[u], S.wmin[j * W + k]));
              }
#pragma unroll
              for (int u = 0; u < 4; u++)
                if (key[u] < bk[h]) { bk[h] = key[u]; bj[h] = js[u]; }
            }
          }
#pragma unroll
          for (int h = 0; h < 2; h++) {
            const int k = lane + 32 * h;
            nd[h] = 0.0;
            np[h] = -1;
            if (k >= W) continue;
            nd[h] = S.dist[k];
            np[h] = S.pred[k];
            if (bj[h] >= 0) {
              const double v = dunorder(bk[h]);
              if (v < nd[h] - 1e-12) { nd[h] = v; np[h] = bj[h]; ch[h] = 1; }
            }
          }
          __syncwarp();
#pragma unroll
          for (int h = 0; h < 2; h++) {
            const int k = lane + 32 * h;
            if (k < W) { S.dist[k] = nd[h]; S.pred[k] = np[h]; }
          }
          act = (uint64_t)__ballot_sync(FULL_MASK, ch[0]) |
                ((uint64_t)__ballot_sync(FULL_MASK, ch[1]) << 32);
          __syncwarp();
        }
        // target: the nearest worker with room (ties: lowest index)
        uint64_t tkey = DKEY_NONE;
        int tl = -1;
#pragma unroll
        for (int h = 0; h < 2; h++) {
          const int k = lane + 32 * h;
          if (k < W && S.counts[k] < capw) {
            const uint64_t key = dorder(S.dist[k]);
            if (tl < 0 || key < tkey) { tkey = key; tl = k; }
          }
        }
        for (int o = 16; o > 0; o >>= 1) {
          const uint64_t k2 = __shfl_xor_sync(FULL_MASK, tkey, o);
          const int t2 = __shfl_xor_sync(FULL_MASK, tl, o);
          if (t2 >= 0 && (tl < 0 || k2 < tkey || (k2 == tkey && t2 < tl))) { tkey = k2; tl = t2; }
        }
        if (lane == 0) {
          const int tgt = tl;
          int nmv = 0;
          if (tgt < 0) {
            s_err = 1;
          } else {
            // walk the path back from its end: edge j -> k moves the request
            // behind wrow[j][k] from j to k
            int k = tgt, steps = 0;
            while (S.pred[k] >= 0 && steps <= W) {
              const int j = S.pred[k];
              const int r = S.wrow[j * W + k];
              s_pj[nmv] = j;
              s_pr[nmv] = r;
              S.mv_row[nmv] = r;
              S.mv_to[nmv++] = k;
              k = j;
              steps++;
            }
            if (steps > W) {
              s_err = 1;
              nmv = 0;
            } else {
              for (int t = 0; t < nmv; t++) b.asg[base + S.mv_row[t]] = S.mv_to[t];
              b.asg[base + r0] = k;
              S.mv_row[nmv] = (int)r0;
              S.mv_to[nmv++] = k;
              S.counts[tgt]++;
            }
          }
          s_nmv = nmv;
        }
        __syncwarp();
        // a source that lost its request needs a rescan where that request
        // was the minimum of one of its weights
        for (int j = lane; j < W; j += 32) S.dirty[j] = 0;
        __syncwarp();
        if (!s_err) {
          const int npath = s_nmv - 1;
          for (int t = 0; t < npath; t++) {
            const int j = s_pj[t], r = s_pr[t];
            bool hit = false;
            for (int k2 = lane; k2 < W; k2 += 32) hit |= S.wrow[j * W + k2] == r;
            if (__any_sync(FULL_MASK, hit) && lane == 0) S.dirty[j] = 1;
          }
        }
        __syncwarp();
        __syncwarp();
        if (s_err) break;
        // requests that moved in lower their new worker's weights; a dirty
        // worker is rescanned whole instead
        const int nmv = s_nmv;
        for (int t = 0; t < nmv; t++) {
          const int r = S.mv_row[t], to = S.mv_to[t];
          if (S.dirty[to]) continue;
          const double* cr = b.cost + (base + r) * W;
          const double ct = cr[to];
          for (int k2 = lane; k2 < W; k2 += 32) {
            if (k2 == to) continue;
            const double v = __dsub_rn(cr[k2], ct);
            const int wr = S.wrow[to * W + k2];
            if (wr < 0 || v < S.wmin[to * W + k2] || (v == S.wmin[to * W + k2] && r < wr)) {
              S.wmin[to * W + k2] = v;
              S.wrow[to * W + k2] = r;
            }
          }
        }
        int anyd = 0;
        for (int j = lane; j < W; j += 32) anyd |= S.dirty[j];
        if (__any_sync(FULL_MASK, anyd)) wide_rescan(S, b, base, m, W, lane, false, s_sel);
        __syncwarp();
      }
    }
    double opt = 0.0;
    for (int64_t r = lane; r < m; r += 32) {
      const int a = b.asg[base + r];
      opt += a >= 0 ? b.cost[(base + r) * W + a] : __longlong_as_double(0x7FF8000000000000ll);
    }
    opt = warp_sum(opt);
    if (lane == 0) {
      b.wnum[pr.win_base + w] = num;
      b.wstat[pr.win_base + w] = nst;
      b.wopt[pr.win_base + w] = s_err ? __longlong_as_double(0x7FF8000000000000ll) : opt;
      b.wcnt[pr.win_base + w] = m;
    }
    __syncwarp();
  }
}

// Whole-run PoA of every replica: one warp per replica, windows summed in
// order by lane 0 (the same order as a sequential sum).
__global__ void __launch_bounds__(NT_POA) k_poa_total(int nprob, PoaBuffers b,
                                                      const PoaProblem* __restrict__ probs) {
  const int lane = threadIdx.x & 31;
  const int p = (int)(((int64_t)blockIdx.x * NT_POA + threadIdx.x) >> 5);
  if (p >= nprob || lane != 0) return;
  const PoaProblem pr = probs[p];
  const int64_t nw = b.nwin[p];
  double tot = __longlong_as_double(0x7FF8000000000000ll), tst = tot;
  if (nw >= 0) {
    double tn = 0.0, to = 0.0, ts = 0.0;
    for (int64_t w = 0; w < nw; w++) {
      tn += b.wnum[pr.win_base + w];
      to += b.wopt[pr.win_base + w];
      ts += b.wstat[pr.win_base + w];
    }
    tot = to > 0.0 ? tn / to : 0.0;
    tst = to > 0.0 ? ts / to : 0.0;
  }
  b.total[p] = tot;
  if (b.total_static) b.total_static[p] = tst;
  if (b.res) {
    b.res[p].poa_total = tot;
    b.res[p].poa_static = tst;
    b.res[p].n_windows = nw;
  }
}

// Last window of each problem: the largest floor(completion / window) over
// its routed rows (-1 when none is routed).  The host sizes the
// window-indexed scratch from it before k_poa_prep, so that every window the
// records span has a slot.  A completion that is negative or not finite is
// skipped here (k_poa_prep reports it as an overflow); indices are clamped
// at 2^62.
__global__ void __launch_bounds__(NT_POA) k_poa_span(const PoaProblem* __restrict__ probs,
                                                     rs_records rec, double window,
                                                     long long* __restrict__ maxw) {
  __shared__ long long red[NT_POA / 32];
  const PoaProblem pr = probs[blockIdx.x];
  long long mx = -1;
  for (int64_t q = threadIdx.x; q < pr.n; q += NT_POA) {
    const int64_t r = pr.rec_base + q;
    if (rec.worker[r] < 0) continue;
    const double w = floor(__ddiv_rn(rec.completion[r], window));
    if (!(w >= 0.0)) continue;
    const long long k = w < 4.611686018427387904e18 ? (long long)w : (1ll << 62);
    mx = k > mx ? k : mx;
  }
  for (int o = 16; o > 0; o >>= 1) {
    const long long v = __shfl_xor_sync(FULL_MASK, mx, o);
    mx = v > mx ? v : mx;
  }
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = mx;
  __syncthreads();
  if (threadIdx.x == 0) {
    long long m = red[0];
    for (int w = 1; w < NT_POA / 32; w++) m = red[w] > m ? red[w] : m;
    maxw[blockIdx.x] = m;
  }
}

cudaError_t launch_poa_span(const PoaProblem* d_prob, int nprob, const rs_records& rec,
                            double window, long long* maxw, cudaStream_t st) {
  if (nprob <= 0) return cudaSuccess;
  k_poa_span<<<nprob, NT_POA, 0, st>>>(d_prob, rec, window, maxw);
  return cudaGetLastError();
}

cudaError_t launch_poa(const PoaProblem* d_prob, int nprob, const PoaBuffers& b,
                       const ModelConsts& mc, cudaStream_t st) {
  if (nprob <= 0) return cudaSuccess;
  k_poa_prep<<<nprob, NT_POA, 0, st>>>(d_prob, b, mc);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  // a few CTAs per replica so that a handful of replicas still fill the GPU
  int dev = 0, sms = 152;
  if (cudaGetDevice(&dev) == cudaSuccess)
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  int split = (4 * sms + nprob - 1) / nprob;
  split = split < 1 ? 1 : (split > 16 ? 16 : split);
  const size_t wsmem = poa_wide_smem(mc.W);
  if (mc.W > POA_WMAX &&
      (e = cudaFuncSetAttribute(k_poa_solve_wide, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)wsmem)) != cudaSuccess)
    return e;
  if (b.wnext) {
    // one wave of CTAs whose warps take the windows from the counter
    if ((e = cudaMemsetAsync(b.wnext, 0, sizeof(unsigned long long), st)) != cudaSuccess) return e;
    int per_sm = 0;
    if (mc.W <= POA_WMAX) {
      void (*kern)(const PoaProblem*, PoaBuffers, ModelConsts) =
          mc.W == 3 ? k_poa_solve<3> : (mc.W == 6 ? k_poa_solve<6> : k_poa_solve<POA_WMAX>);
      if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, NT_POA, 0)) !=
          cudaSuccess)
        return e;
      int64_t g = (b.nslots + NT_POA / 32 - 1) / (NT_POA / 32);
      const int64_t cap = (int64_t)sms * (per_sm > 0 ? per_sm : 1);
      g = g < cap ? g : cap;
      kern<<<(unsigned)(g > 0 ? g : 1), NT_POA, 0, st>>>(d_prob, b, mc);
    } else {
      if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_poa_solve_wide, 32,
                                                             wsmem)) != cudaSuccess)
        return e;
      int64_t g = b.nslots;
      const int64_t cap = (int64_t)sms * (per_sm > 0 ? per_sm : 1);
      g = g < cap ? g : cap;
      k_poa_solve_wide<<<(unsigned)(g > 0 ? g : 1), 32, wsmem, st>>>(d_prob, b, mc);
    }
  } else if (mc.W <= POA_WMAX) {
    void (*kern)(const PoaProblem*, PoaBuffers, ModelConsts) =
        mc.W == 3 ? k_poa_solve<3> : (mc.W == 6 ? k_poa_solve<6> : k_poa_solve<POA_WMAX>);
    kern<<<dim3(nprob, split), NT_POA, 0, st>>>(d_prob, b, mc);
  } else {
    // one warp per CTA: 8x the CTAs for the same windows in flight
    const int wsplit = split * (NT_POA / 32) > 128 ? 128 : split * (NT_POA / 32);
    k_poa_solve_wide<<<dim3(nprob, wsplit), 32, wsmem, st>>>(d_prob, b, mc);
  }
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  k_poa_total<<<(nprob + NT_POA / 32 - 1) / (NT_POA / 32), NT_POA, 0, st>>>(nprob, b, d_prob);
  return cudaGetLastError();
}

}  // namespace rs
