// Live routing (route_batch / route_release) on one router instance.
//
// One CTA routes a batch of requests of one instance in array order: for each
// request, the cached prefix of every worker, the Eq. (1) cost with the
// instance's active blocks, the Eq. (2) choice, and the chosen worker's cache
// and load update -- the same steps as a simulated arrival, without the
// event loop (completions are reported by the caller through route_release).
#include "rs_device.cuh"

namespace rs {

struct RouterShared {
  UpdateShared us;
  uint32_t scan_pos;
  int warp_tot[NT_SIM / 32];
  unsigned long long probes;
  int64_t off0, off1;
  int status, nopen, jstar, rebuild;
  uint64_t ordinal;
};

__global__ void __launch_bounds__(NT_SIM) k_route_batch(
    RouterState s, int32_t instance, const int64_t* __restrict__ offsets,
    const uint64_t* __restrict__ hashes, int32_t n_req, const int32_t* __restrict__ out_len,
    int32_t* __restrict__ worker_out, float* __restrict__ cost_out, int32_t* __restrict__ prefix_out,
    int nbmax, TableGeom g, ModelConsts mc, float omega, float tau, uint64_t seed) {
  extern __shared__ __align__(16) unsigned char smem[];
  __shared__ RouterShared R;
  const int W = mc.W;
  const size_t nb_cap = (size_t)(nbmax > 0 ? nbmax : 1);
  size_t dup = 1;
  while (dup < 2 * nb_cap) dup <<= 1;
  unsigned char* p = smem;
  auto take = [&](size_t bytes) {
    unsigned char* r = p;
    p += (bytes + 15) & ~(size_t)15;
    return r;
  };
  uint64_t* hbuf = reinterpret_cast<uint64_t*>(take(8 * nb_cap));
  UpdateScratch sc;
  sc.dupset = reinterpret_cast<uint64_t*>(take(8 * dup));
  sc.dupmask = (uint32_t)(dup - 1);
  int64_t* A = reinterpret_cast<int64_t*>(take(8 * (size_t)W));
  CacheMeta* meta = reinterpret_cast<CacheMeta*>(take(sizeof(CacheMeta) * (size_t)W));
  sc.slot = reinterpret_cast<uint32_t*>(take(4 * nb_cap));
  sc.pst = reinterpret_cast<uint32_t*>(take(4 * nb_cap));
  sc.fslot = reinterpret_cast<uint32_t*>(take(4 * nb_cap));
  sc.vslot = reinterpret_cast<uint32_t*>(take(8 * nb_cap));
  sc.vt = reinterpret_cast<uint32_t*>(take(8 * nb_cap));
  sc.owner = reinterpret_cast<int32_t*>(take(8 * nb_cap));
  sc.victim = reinterpret_cast<int32_t*>(take(8 * nb_cap));
  int32_t* wm = reinterpret_cast<int32_t*>(take(4 * (size_t)W));
  int32_t* wopen = reinterpret_cast<int32_t*>(take(4 * (size_t)W));
  float* wcost = reinterpret_cast<float*>(take(4 * (size_t)W));
  sc.kind = take(nb_cap);
  sc.evk = take(nb_cap);
  sc.touched = take(2 * nb_cap);

  for (uint32_t q = threadIdx.x; q <= sc.dupmask; q += NT_SIM) sc.dupset[q] = 0ull;
  for (int j = threadIdx.x; j < W; j += NT_SIM) {
    A[j] = s.active[j];
    meta[j] = s.meta[j];
  }
  if (threadIdx.x == 0) {
    R.status = *s.status;
    R.ordinal = *s.ordinal;
    R.probes = 0;
  }
  __syncthreads();
  auto table = [&](int j) {
    TableView t;
    t.keys = s.keys + (size_t)j * g.slots;
    t.stamp = s.stamp + (size_t)j * g.slots;
    t.log = s.log + (size_t)j * g.R;
    t.fexp = nullptr;
    t.bmask = g.bmask;
    t.rmask = g.rmask;
    return t;
  };
  const int CH = max(32, ((4 * NT_SIM) / W) & ~31);
  for (int32_t i = 0; i < n_req && R.status == RS_OK; i++) {
    const int64_t o0 = offsets[i], o1 = offsets[i + 1];
    const int64_t Lp = o1 - o0;
    const int64_t nb64 = Lp >> 4;
    if (nb64 > (int64_t)g.K || nb64 > (int64_t)nbmax) {
      __syncthreads();
      if (threadIdx.x == 0) R.status = RS_ERR_CAPACITY;
      __syncthreads();
      break;
    }
    const int nb = (int)nb64;
    const int nbt = (int)((Lp + 15) >> 4);
    for (int k = threadIdx.x; k < nb; k += NT_SIM) hbuf[k] = __ldg(hashes + (o0 >> 4) + k);
    for (int j = threadIdx.x; j < W; j += NT_SIM) {
      wm[j] = nb;
      wopen[j] = j;
    }
    if (threadIdx.x == 0) R.nopen = W;
    __syncthreads();
    // cached prefix on every worker
    int err = 0;
    for (int c0 = 0;;) {
      const int nopen = R.nopen;
      const int len = min(CH, nb - c0);
      const int total = len > 0 ? nopen * len : 0;
      for (int it = threadIdx.x; it < total; it += NT_SIM) {
        const int jj = wopen[it / len];
        const int k = c0 + it % len;
        if (k < wm[jj] && table_find(table(jj), hbuf[k], &err) == SLOT_NONE) atomicMin(&wm[jj], k);
      }
      __syncthreads();
      c0 += CH;
      if (threadIdx.x == 0) {
        int no = 0;
        if (c0 < nb)
          for (int j = 0; j < W; j++)
            if (wm[j] >= c0) wopen[no++] = j;
        R.nopen = no;
      }
      __syncthreads();
      if (R.nopen == 0) break;
    }
    if (err) R.status = RS_ERR_TIMEOUT;
    for (int j = threadIdx.x; j < W; j += NT_SIM) {
      const float cj = router_cost(omega, (int64_t)nbt - wm[j], A[j]);
      wcost[j] = cj;
      if (cost_out) cost_out[(size_t)i * W + j] = cj;
      if (prefix_out) prefix_out[(size_t)i * W + j] = wm[j];
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      const uint32_t u24 = tau > 0.0f ? draw_u24(seed, R.ordinal, (uint32_t)instance, TAG_ROUTE) : 0u;
      R.jstar = select_worker(wcost, W, tau, u24, nullptr);
      CacheMeta* mt = &meta[R.jstar];
      const uint64_t span = (uint64_t)mt->T - mt->head + (uint64_t)nb;
      R.rebuild = span > g.R || mt->tombs > g.slots / 8 || (uint64_t)mt->T + nb > STAMP_LIMIT;
      update_reset(&R.us);
      R.us.err = 0;
    }
    __syncthreads();
    const int js = R.jstar;
    const TableView tv = table(js);
    if (R.rebuild) cache_rebuild<NT_SIM>(tv, &meta[js], g.K, s.tmp, R.warp_tot, &R.us);
    cache_lookup_all<NT_SIM>(tv, hbuf, nb, sc, &R.us, &R.probes);
    __syncthreads();
    if (R.us.dup) {
      if (threadIdx.x == 0) R.status = RS_ERR_COLLISION;
      __syncthreads();
      break;
    }
    cache_apply<NT_SIM>(tv, &meta[js], g.K, hbuf, nb, sc, &R.us, R.warp_tot, &R.scan_pos);
    if (threadIdx.x == 0) {
      if (R.us.err) R.status = R.us.err;
      A[js] += (Lp + out_len[i] + 15) >> 4;
      worker_out[i] = js;
      R.ordinal++;
    }
    __syncthreads();
  }
  __syncthreads();
  for (int j = threadIdx.x; j < W; j += NT_SIM) {
    s.active[j] = A[j];
    s.meta[j] = meta[j];
  }
  if (threadIdx.x == 0) {
    *s.status = R.status;
    *s.ordinal = R.ordinal;
  }
}

size_t router_smem(int W, int nbmax) {
  const size_t nb = (size_t)(nbmax > 0 ? nbmax : 1);
  size_t dup = 1;
  while (dup < 2 * nb) dup <<= 1;
  auto r16 = [](size_t x) { return (x + 15) & ~(size_t)15; };
  return r16(8 * nb) + r16(8 * dup) + r16(8 * (size_t)W) + r16(sizeof(CacheMeta) * (size_t)W) +
         3 * r16(4 * nb) + 4 * r16(8 * nb) + 3 * r16(4 * (size_t)W) + 2 * r16(nb) + r16(2 * nb);
}

cudaError_t launch_route_batch(const RouterState& s, int32_t instance, const int64_t* offsets,
                               const uint64_t* hashes, int32_t n_req, const int32_t* out_len,
                               int32_t* worker_out, float* cost_out, int32_t* prefix_out,
                               int nbmax, const TableGeom& g, const ModelConsts& mc, float omega,
                               float tau, uint64_t seed, cudaStream_t st) {
  if (n_req <= 0) return cudaSuccess;
  const size_t smem = router_smem(mc.W, nbmax);
  cudaError_t e = cudaFuncSetAttribute(k_route_batch, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  k_route_batch<<<1, NT_SIM, smem, st>>>(s, instance, offsets, hashes, n_req, out_len, worker_out,
                                         cost_out, prefix_out, nbmax, g, mc, omega, tau, seed);
  return cudaGetLastError();
}

// Completions: subtract, then clamp at zero (equal to clamping after every
// subtraction, since a release only subtracts).  Invalid workers are skipped
// and flagged in *bad.
__global__ void k_route_release(int64_t* active, const int32_t* __restrict__ worker,
                                const int32_t* __restrict__ blocks, int32_t n, int32_t W,
                                int32_t* bad) {
  for (int32_t i = threadIdx.x; i < n; i += blockDim.x) {
    const int w = worker[i];
    if (w < 0 || w >= W) {
      atomicExch(bad, 1);
      continue;
    }
    atomicAdd(reinterpret_cast<unsigned long long*>(active + w),
              (unsigned long long)(-(long long)blocks[i]));
  }
  __syncthreads();
  for (int j = threadIdx.x; j < W; j += blockDim.x)
    if (active[j] < 0) active[j] = 0;
}

cudaError_t launch_route_release(const RouterState& s, const int32_t* worker, const int32_t* blocks,
                                 int32_t n, int32_t W, cudaStream_t st) {
  if (n <= 0) return cudaSuccess;
  k_route_release<<<1, 256, 0, st>>>(s.active, worker, blocks, n, W, s.status + 1);
  return cudaGetLastError();
}

__global__ void k_clear_tables(uint64_t* keys, uint32_t* stamp, size_t nslots, CacheMeta* meta,
                               size_t nmeta) {
  const size_t stride = (size_t)gridDim.x * blockDim.x;
  for (size_t s = (size_t)blockIdx.x * blockDim.x + threadIdx.x; s < nslots; s += stride) {
    keys[s] = KEY_EMPTY;
    stamp[s] = STAMP_NONE;
  }
  for (size_t s = (size_t)blockIdx.x * blockDim.x + threadIdx.x; s < nmeta; s += stride)
    meta[s] = CacheMeta{};
}

cudaError_t launch_clear_tables(uint64_t* keys, uint32_t* stamp, size_t nslots, CacheMeta* meta,
                                size_t nmeta, cudaStream_t st) {
  k_clear_tables<<<152 * 4, 256, 0, st>>>(keys, stamp, nslots, meta, nmeta);
  return cudaGetLastError();
}

// Batch probe (route_probe): the first-miss prefix m_ij of S2 for every
// (request, worker) pair against one snapshot of the tables (only read).
//
// A pair walks its request's blocks in order until the first one absent from
// the worker's table; a walk of m_ij + 1 dependent lookups per thread would
// leave a warp waiting for its longest walk with most lanes idle (most pairs
// miss at block 0, a few follow a shared prefix for many blocks).  So a warp
// takes 64 consecutive pairs (request-major, two per lane) and runs them
// together in steps: at each step the a pairs still open share the warp's 64
// lookup slots, each pair the next `share` blocks of its walk, share =
// min(64 / a, 2^step) (one block per pair at the first step, doubling as the
// open pairs thin out, so no pair looks up more than about twice the blocks
// its answer needs); both slots of a lane are issued before either is used.
// A pair's window ends its walk at its first absent block (or the prompt's
// end), else the walk moves on by `share`.  Lookups: one 64-byte bucket (two
// 32-byte sectors) and one 8-byte hash each.
constexpr int PROBE_NT = 256;

// Position of the n-th (0-based) set bit of x; x has more than n set bits.
__device__ __forceinline__ int nth_set_bit64(uint64_t x, int n) {
  int pos = 0;
#pragma unroll
  for (int w = 32; w >= 1; w >>= 1) {
    const int c = __popcll(x & ((1ull << w) - 1ull));
    if (n >= c) {
      n -= c;
      x >>= w;
      pos += w;
    }
  }
  return pos;
}

struct ProbePair {
  int64_t hbase;   // index of the request's first block hash
  int32_t start;   // next block of the walk
  int32_t nb;      // full blocks of the request
  int32_t j;       // worker
  int32_t pad;
};

__global__ void __launch_bounds__(PROBE_NT) k_probe_batch(RouterState s,
                                                          const int64_t* __restrict__ offsets,
                                                          const uint64_t* __restrict__ hashes,
                                                          int64_t n_req, int W, TableGeom g,
                                                          int32_t* __restrict__ prefix_out) {
  __shared__ ProbePair sp[PROBE_NT / 32][64];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  ProbePair* P = sp[warp];
  const int64_t total = n_req * W;
  const int64_t ngroups = (total + 63) >> 6;
  const int64_t gw = ((int64_t)blockIdx.x * PROBE_NT + threadIdx.x) >> 5;
  const int64_t nw = ((int64_t)gridDim.x * PROBE_NT) >> 5;
  for (int64_t grp = gw; grp < ngroups; grp += nw) {
    const int64_t e0 = grp << 6;
    // this lane's two pairs: slots lane and lane + 32
    int32_t m[2] = {0, 0};
    bool open[2] = {false, false};
#pragma unroll
    for (int h = 0; h < 2; h++) {
      const int q = lane + 32 * h;
      const int64_t e = e0 + q;
      ProbePair pp{0, 0, 0, 0, 0};
      if (e < total) {
        const int64_t i = e / W;
        const int64_t o0 = __ldg(offsets + i);
        const int64_t nbl = (__ldg(offsets + i + 1) - o0) >> 4;
        pp.hbase = o0 >> 4;
        pp.nb = (int32_t)(nbl < 0x7FFFFFFF ? nbl : 0x7FFFFFFF);
        pp.j = (int32_t)(e - i * W);
        open[h] = pp.nb > 0;
      }
      P[q] = pp;
    }
    uint64_t act = (uint64_t)__ballot_sync(FULL_MASK, open[0]) |
                   ((uint64_t)__ballot_sync(FULL_MASK, open[1]) << 32);
    for (int step = 0; act != 0ull; step++) {
      __syncwarp();
      const int a = __popcll(act);
      int share = 64 / a;
      if (step < 6 && share > (1 << step)) share = 1 << step;
      // lookups of slots lane and lane + 32: pair (its rank r among the open
      // ones) and block start + off
      bool miss[2] = {false, false};
      bool live[2] = {false, false};
      uint64_t hk[2] = {0ull, 0ull};
      TableView tv[2];
#pragma unroll
      for (int h = 0; h < 2; h++) {
        const int q = lane + 32 * h;
        const int r = q / share;
        if (r < a) {
          const int pi = nth_set_bit64(act, r);
          const ProbePair pp = P[pi];
          const int64_t k = (int64_t)pp.start + (q - r * share);
          live[h] = true;
          if (k >= pp.nb) {
            miss[h] = true;   // past the prompt: the walk ends at nb
          } else {
            hk[h] = __ldg(hashes + pp.hbase + k);
            const size_t wj = (size_t)pp.j;
            tv[h].keys = s.keys + wj * g.slots;
            tv[h].stamp = s.stamp + wj * g.slots;
            tv[h].log = s.log + wj * g.R;
            tv[h].fexp = nullptr;
            tv[h].bmask = g.bmask;
            tv[h].rmask = g.rmask;
          }
        }
      }
      int err = 0;
#pragma unroll
      for (int h = 0; h < 2; h++)
        if (live[h] && !miss[h]) miss[h] = table_find(tv[h], hk[h], &err) == SLOT_NONE;
      const uint64_t mm = (uint64_t)__ballot_sync(FULL_MASK, miss[0]) |
                          ((uint64_t)__ballot_sync(FULL_MASK, miss[1]) << 32);
      // each pair's owner closes its walk at the window's first miss, or moves on
      const uint64_t wmask = share >= 64 ? ~0ull : ((1ull << share) - 1ull);
#pragma unroll
      for (int h = 0; h < 2; h++) {
        const int q = lane + 32 * h;
        if (!open[h]) continue;
        const int r = __popcll(act & ((1ull << q) - 1ull));
        const uint64_t bits = (mm >> (r * share)) & wmask;
        const int32_t st = P[q].start;
        if (bits) {
          m[h] = st + __ffsll((long long)bits) - 1;
          open[h] = false;
        } else if (st + share >= P[q].nb) {
          m[h] = P[q].nb;
          open[h] = false;
        }
      }
      __syncwarp();   // every lane has read the starts of this step
#pragma unroll
      for (int h = 0; h < 2; h++)
        if (open[h]) P[lane + 32 * h].start += share;
      act = (uint64_t)__ballot_sync(FULL_MASK, open[0]) |
            ((uint64_t)__ballot_sync(FULL_MASK, open[1]) << 32);
    }
#pragma unroll
    for (int h = 0; h < 2; h++) {
      const int64_t e = e0 + lane + 32 * h;
      if (e < total) prefix_out[e] = m[h];
    }
    __syncwarp();
  }
}

cudaError_t launch_probe_batch(const RouterState& s, const int64_t* offsets, const uint64_t* hashes,
                               int64_t n_req, int W, const TableGeom& g, int32_t* prefix_out,
                               cudaStream_t st) {
  if (n_req <= 0) return cudaSuccess;
  int dev = 0, sms = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  const int64_t groups = (n_req * W + 63) / 64;   // 64 pairs per warp
  int64_t nblk = (groups + PROBE_NT / 32 - 1) / (PROBE_NT / 32);
  if (nblk > (int64_t)sms * 8) nblk = (int64_t)sms * 8;
  k_probe_batch<<<(unsigned)nblk, PROBE_NT, 0, st>>>(s, offsets, hashes, n_req, W, g, prefix_out);
  return cudaGetLastError();
}

}  // namespace rs
