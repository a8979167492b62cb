// Closed-loop routing simulation (K3): one CTA per replica, persistent.
//
// Per replica the CTA runs the whole event loop of the paper's serving
// setting: a client holding C requests in flight (§7.4), completions and
// controller samples in time order, then for every arriving request the
// routing step of Algorithm 1 -- cached-prefix probe of every worker, the
// Eq. (1) cost, the Eq. (2) choice (with the Table 2 parameters of the
// current Eq. (11) regime when the controller is on), the chosen worker's
// LRU cache update and load update -- and its Eq. (9) latency.
//
// Thread 0 owns the scalar event state (completion heap, FIFO queues,
// controller) in shared memory; every data-parallel step (hash staging,
// probes, the cache update, controller percentile) uses the whole CTA.
// Floating point follows the paper's formulas operation by operation
// (explicit _rn intrinsics, no contraction).
#include "rs_device.cuh"

namespace rs {

__host__ __device__ inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

struct SimLayout {
  size_t f_a, f_o, h_t, hbuf, dupset;
  size_t f_req, f_worker, f_blk, f_O, f_next, h_f, freestk, owner, victim;
  size_t slot, pst, vslot, vt;
  size_t wmeta, winserv, wA, wqh, wqt, wm, wcost, wopen;
  size_t kind, evk, touched;
  size_t total;
  uint32_t dupmask;
};

__host__ __device__ inline SimLayout make_sim_layout(int W, int nbmax, int cmax) {
  SimLayout L;
  size_t o = 0;
  const size_t nb = (size_t)(nbmax > 0 ? nbmax : 1);
  const size_t nv = 2 * nb;
  const size_t C = (size_t)(cmax > 0 ? cmax : 1);
  size_t dup = 1;
  while (dup < 2 * nb) dup <<= 1;
  L.dupmask = (uint32_t)(dup - 1);
#define TAKE(field, bytes, al) \
  o = align_up(o, al);         \
  L.field = o;                 \
  o += (bytes);
  TAKE(f_a, 8 * C, 16)
  TAKE(f_o, 8 * C, 8)
  TAKE(h_t, 8 * C, 8)
  TAKE(hbuf, 8 * nb, 16)
  TAKE(dupset, 8 * dup, 16)
  TAKE(wA, 8 * (size_t)W, 8)
  TAKE(f_req, 4 * C, 4)
  TAKE(f_worker, 4 * C, 4)
  TAKE(f_blk, 4 * C, 4)
  TAKE(f_O, 4 * C, 4)
  TAKE(f_next, 4 * C, 4)
  TAKE(h_f, 4 * C, 4)
  TAKE(freestk, 4 * C, 4)
  TAKE(owner, 4 * nv, 4)
  TAKE(victim, 4 * nv, 4)
  TAKE(slot, 4 * nb, 4)
  TAKE(pst, 4 * nb, 4)
  TAKE(vslot, 4 * nv, 4)
  TAKE(vt, 4 * nv, 4)
  TAKE(wmeta, sizeof(CacheMeta) * (size_t)W, 16)
  TAKE(winserv, 4 * (size_t)W, 4)
  TAKE(wqh, 4 * (size_t)W, 4)
  TAKE(wqt, 4 * (size_t)W, 4)
  TAKE(wm, 4 * (size_t)W, 4)
  TAKE(wcost, 4 * (size_t)W, 4)
  TAKE(wopen, 4 * (size_t)W, 4)
  TAKE(kind, nb, 1)
  TAKE(evk, nb, 1)
  TAKE(touched, nv, 1)
#undef TAKE
  L.total = align_up(o, 16);
  return L;
}

size_t sim_smem_bytes(int W, int nbmax, int cmax) { return make_sim_layout(W, nbmax, cmax).total; }

struct SimScalars {
  double prev_arrival, a_cur, rel, rel_next, makespan, sum_ttft, sum_e2e, min_ft, lastL, ewma;
  int64_t next_tick, np, off0, off1, noff0, noff1;
  int64_t near_ties, exact_ties, sampled, near_bd, hit_blocks, inserted, evicted, slow, rebuilds;
  int64_t ticks, switches, tir[3], n_routed, probe_blocks, hashed_blocks;
  unsigned long long probes;
  uint64_t sel_prefix;
  int32_t in_flight, nheap, nfree, phase, evres, status, O, nO, jstar, regime, up_cnt, down_cnt;
  int32_t have_L, have_ewma, max_regime, pend_cur, nopen, sel_kk, rebuild, nw;
  float tau_cur, omega_cur;
  UpdateShared us;
  uint32_t scan_pos;
  int warp_tot[NT_SIM / 32];
  int hist[256];
  double red[NT_SIM / 32];
};

// Everything a device helper needs, resolved once per CTA.
struct SimCtx {
  SimScalars* S;
  const SimDesc* d;
  const SimBuffers* b;
  const SimLaunch* L;
  int sid;
  double *f_a, *f_o, *h_t;
  uint64_t* hbuf;
  int32_t *f_req, *f_worker, *f_blk, *f_O, *f_next, *h_f, *freestk;
  CacheMeta* wmeta;
  int32_t *winserv, *wqh, *wqt, *wm, *wopen;
  int64_t* wA;
  float* wcost;
  UpdateScratch sc;
  double *pend_ft[2], *pend_tt[2], *pend_win;

  __device__ TableView table(int j) const {
    TableView t;
    const size_t wi = (size_t)sid * L->mc.W + j;
    t.keys = b->keys + wi * L->g.slots;
    t.stamp = b->stamp + wi * L->g.slots;
    t.log = b->log + wi * L->g.R;
    t.bmask = L->g.bmask;
    t.rmask = L->g.rmask;
    return t;
  }
};

// ------------------------------------------------------------ event machinery (thread 0)

__device__ __forceinline__ bool ev_less(const SimCtx& c, double ta, int fa, double tb, int fb) {
  return ta < tb || (ta == tb && c.f_req[fa] < c.f_req[fb]);
}

__device__ void heap_push(SimCtx& c, double t, int f) {
  int i = c.S->nheap++;
  c.h_t[i] = t;
  c.h_f[i] = f;
  while (i > 0) {
    const int p = (i - 1) >> 1;
    if (!ev_less(c, c.h_t[i], c.h_f[i], c.h_t[p], c.h_f[p])) break;
    const double tt = c.h_t[i]; c.h_t[i] = c.h_t[p]; c.h_t[p] = tt;
    const int ff = c.h_f[i]; c.h_f[i] = c.h_f[p]; c.h_f[p] = ff;
    i = p;
  }
}

__device__ void heap_pop(SimCtx& c, double* t, int* f) {
  *t = c.h_t[0];
  *f = c.h_f[0];
  const int n = --c.S->nheap;
  c.h_t[0] = c.h_t[n];
  c.h_f[0] = c.h_f[n];
  int i = 0;
  for (;;) {
    const int l = 2 * i + 1, r = l + 1;
    int s = i;
    if (l < n && ev_less(c, c.h_t[l], c.h_f[l], c.h_t[s], c.h_f[s])) s = l;
    if (r < n && ev_less(c, c.h_t[r], c.h_f[r], c.h_t[s], c.h_f[s])) s = r;
    if (s == i) break;
    const double tt = c.h_t[i]; c.h_t[i] = c.h_t[s]; c.h_t[s] = tt;
    const int ff = c.h_f[i]; c.h_f[i] = c.h_f[s]; c.h_f[s] = ff;
    i = s;
  }
}

// Eq. (9) with beta = 2: f(n) = a n + b + d / (cap - n)^2
__device__ __forceinline__ double latency_f(const ModelConsts& mc, int n) {
  const double t1 = __dmul_rn(mc.lat_a, (double)n);
  const double t2 = __dadd_rn(t1, mc.lat_b);
  const double den = (double)(mc.cap - n);
  const double t3 = __ddiv_rn(mc.lat_d, __dmul_rn(den, den));
  return __dadd_rn(t2, t3);
}

__device__ void start_service(SimCtx& c, int f, int j, double t) {
  SimScalars& S = *c.S;
  const ModelConsts& mc = c.L->mc;
  const int n = ++c.winserv[j];
  const double fv = latency_f(mc, n);
  const double svc = __dsub_rn(fv, __dmul_rn(mc.w_c, c.f_o[f]));
  const double ft = __dadd_rn(t, svc);
  const double a = c.f_a[f];
  const double tt = __dsub_rn(ft, a);
  const double ct = __dadd_rn(ft, __dmul_rn((double)c.f_O[f], mc.itl));
  const int64_t row = c.d->rec_base + c.f_req[f];
  c.b->rec.start[row] = t;
  c.b->rec.first_token[row] = ft;
  c.b->rec.ttft[row] = tt;
  c.b->rec.completion[row] = ct;
  heap_push(c, ct, f);
  if (c.d->controller) {
    const int cur = S.pend_cur;
    c.pend_ft[cur][S.np] = ft;
    c.pend_tt[cur][S.np] = tt;
    S.np++;
    if (ft < S.min_ft) S.min_ft = ft;
  }
  S.sum_ttft = __dadd_rn(S.sum_ttft, tt);
  S.sum_e2e = __dadd_rn(S.sum_e2e, __dsub_rn(ct, a));
}

__device__ void complete(SimCtx& c, int f, double t) {
  SimScalars& S = *c.S;
  const int j = c.f_worker[f];
  c.winserv[j]--;
  c.wA[j] -= c.f_blk[f];
  S.in_flight--;
  if (t > S.makespan) S.makespan = t;
  c.freestk[S.nfree++] = f;
  const int f2 = c.wqh[j];
  if (f2 >= 0) {
    c.wqh[j] = c.f_next[f2];
    if (c.wqh[j] < 0) c.wqt[j] = -1;
    start_service(c, f2, j, t);
  }
}

// EWMA of Eq. (10) and the hysteretic regime of Eq. (11); one sample.
__device__ void ctl_sample(SimCtx& c, bool has_window, double Lw) {
  SimScalars& S = *c.S;
  const ModelConsts& mc = c.L->mc;
  double L = 0.0;
  if (has_window) {
    L = Lw;
    S.have_L = 1;
    S.lastL = L;
  } else if (S.have_L) {
    L = S.lastL;
  }
  if (S.have_L) {
    if (!S.have_ewma) {
      S.ewma = L;
      S.have_ewma = 1;
    } else {
      S.ewma = __dadd_rn(__dmul_rn(mc.alpha, L), __dmul_rn(__dsub_rn(1.0, mc.alpha), S.ewma));
    }
    bool up = false, down = false;
    if (S.regime == 0) up = S.ewma >= mc.theta1;
    if (S.regime == 1) {
      up = S.ewma >= mc.theta2;
      down = S.ewma < __dsub_rn(mc.theta1, __dmul_rn(mc.eps_frac, mc.theta1));
    }
    if (S.regime == 2) down = S.ewma < __dsub_rn(mc.theta2, __dmul_rn(mc.eps_frac, mc.theta2));
    S.up_cnt = up ? S.up_cnt + 1 : 0;
    S.down_cnt = down ? S.down_cnt + 1 : 0;
    if (S.up_cnt >= mc.hyst_k) {
      S.regime++;
      S.up_cnt = S.down_cnt = 0;
      S.switches++;
    } else if (S.down_cnt >= mc.hyst_k) {
      S.regime--;
      S.up_cnt = S.down_cnt = 0;
      S.switches++;
    }
    if (S.regime > S.max_regime) S.max_regime = S.regime;
  }
  S.tir[S.regime]++;
  S.ticks++;
  S.next_tick++;
  if (S.ticks >= TICK_LIMIT) S.status = RS_ERR_CAPACITY;
}

__device__ __forceinline__ double tick_time(const SimCtx& c) {
  return c.d->controller ? __dmul_rn((double)c.S->next_tick, c.L->mc.dt) : __longlong_as_double(0x7FF0000000000000ll);
}

// Advances events for the current request (thread 0).  Returns 1 when a
// controller sample with a non-empty window is due (the CTA computes it),
// 0 when the arrival time is known and every event up to it is processed.
__device__ int events_advance(SimCtx& c) {
  SimScalars& S = *c.S;
  const double INF = __longlong_as_double(0x7FF0000000000000ll);
  if (S.phase == 0) {
    double T = S.prev_arrival;
    if (S.in_flight >= c.d->C) {
      for (;;) {
        if (S.status != RS_OK) return 0;
        if (S.nheap == 0) {   // cannot happen: every request in flight is in service or queued
          S.status = RS_ERR_TIMEOUT;
          S.a_cur = T;
          S.phase = 1;
          return 0;
        }
        const double tc = c.h_t[0];
        const double tt = tick_time(c);
        if (tt < tc) {
          if (S.min_ft >= tt) { ctl_sample(c, false, 0.0); continue; }
          return 1;
        }
        double t;
        int f;
        heap_pop(c, &t, &f);
        complete(c, f, t);
        if (t > T) T = t;
        break;
      }
    }
    S.a_cur = S.rel > T ? S.rel : T;
    S.phase = 1;
  }
  const double a = S.a_cur;
  for (;;) {
    if (S.status != RS_OK) return 0;
    const double tc = S.nheap > 0 ? c.h_t[0] : INF;
    const double tt = tick_time(c);
    if (tc <= tt) {
      if (tc > a) break;
      double t;
      int f;
      heap_pop(c, &t, &f);
      complete(c, f, t);
    } else {
      if (tt > a) break;
      if (S.min_ft >= tt) { ctl_sample(c, false, 0.0); continue; }
      return 1;
    }
  }
  return 0;
}

// ------------------------------------------------------------ controller sample (CTA)

// The window holds the TTFTs of requests whose first token came before the
// sample time and after the previous sample; its nearest-rank P99 (exact
// radix selection over the float64 bit patterns, TTFT > 0) feeds Eq. (10).
__device__ void tick_cta(SimCtx& c) {
  SimScalars& S = *c.S;
  const double tt = __dmul_rn((double)S.next_tick, c.L->mc.dt);
  const int cur = S.pend_cur;
  const int64_t np = S.np;
  const double* sft = c.pend_ft[cur];
  const double* stt = c.pend_tt[cur];
  double* dft = c.pend_ft[cur ^ 1];
  double* dtt = c.pend_tt[cur ^ 1];
  int64_t nkeep = 0, nwin = 0;
  double mft = __longlong_as_double(0x7FF0000000000000ll);
  for (int64_t p0 = 0; p0 < np; p0 += NT_SIM) {
    const int64_t p = p0 + threadIdx.x;
    bool keep = false, inwin = false;
    double f = 0.0, v = 0.0;
    if (p < np) {
      f = sft[p];
      v = stt[p];
      inwin = f < tt;
      keep = !inwin;
    }
    int t1, t2;
    const int r1 = cta_rank<NT_SIM>(keep, S.warp_tot, &t1);
    const int r2 = cta_rank<NT_SIM>(inwin, S.warp_tot, &t2);
    if (keep) {
      dft[nkeep + r1] = f;
      dtt[nkeep + r1] = v;
      mft = fmin(mft, f);
    }
    if (inwin) c.pend_win[nwin + r2] = v;
    nkeep += t1;
    nwin += t2;
  }
  // CTA minimum of the kept first-token times
  for (int o = 16; o > 0; o >>= 1) mft = fmin(mft, __shfl_xor_sync(FULL_MASK, mft, o));
  if ((threadIdx.x & 31) == 0) S.red[threadIdx.x >> 5] = mft;
  if (threadIdx.x == 0) {
    S.sel_prefix = 0;
    S.sel_kk = (int)((99 * nwin + 99) / 100);
  }
  __syncthreads();
  double L = 0.0;
  if (nwin > 0) {
    for (int shift = 56; shift >= 0; shift -= 8) {
      for (int q = threadIdx.x; q < 256; q += NT_SIM) S.hist[q] = 0;
      __syncthreads();
      const uint64_t pre = S.sel_prefix;
      const uint64_t mhi = shift == 56 ? 0ull : (~0ull << (shift + 8));
      for (int64_t p = threadIdx.x; p < nwin; p += NT_SIM) {
        const uint64_t bits = (uint64_t)__double_as_longlong(c.pend_win[p]);
        if ((bits & mhi) == (pre & mhi)) atomicAdd(&S.hist[(bits >> shift) & 255], 1);
      }
      __syncthreads();
      if (threadIdx.x == 0) {
        int cum = 0;
        for (int dg = 0; dg < 256; dg++) {
          if (cum + S.hist[dg] >= S.sel_kk) {
            S.sel_prefix = pre | ((uint64_t)dg << shift);
            S.sel_kk -= cum;
            break;
          }
          cum += S.hist[dg];
        }
      }
      __syncthreads();
    }
    L = __longlong_as_double((long long)S.sel_prefix);
  }
  if (threadIdx.x == 0) {
    double m = S.red[0];
    for (int w = 1; w < NT_SIM / 32; w++) m = fmin(m, S.red[w]);
    S.np = nkeep;
    S.pend_cur = cur ^ 1;
    S.min_ft = m;
    ctl_sample(c, nwin > 0, L);
  }
  __syncthreads();
}

// ------------------------------------------------------------ routing step (CTA)

// m_j: leading blocks of the prompt found in worker j's cache, for every j.
// Rounds of CH blocks per still-undecided worker; a worker is decided once a
// miss is found below the round's end.
__device__ void probe_prefixes(SimCtx& c, int nb) {
  SimScalars& S = *c.S;
  const int W = c.L->mc.W;
  const int CH = max(32, ((4 * NT_SIM) / W) & ~31);
  int c0 = 0;
  int err = 0;
  unsigned long long cnt = 0;
  for (;;) {
    const int nopen = S.nopen;
    const int len = min(CH, nb - c0);
    const int total = len > 0 ? nopen * len : 0;
    for (int it = threadIdx.x; it < total; it += NT_SIM) {
      const int jj = c.wopen[it / len];
      const int k = c0 + it % len;
      if (k < c.wm[jj]) {
        cnt++;
        if (table_find(c.table(jj), c.hbuf[k], &err) == SLOT_NONE) atomicMin(&c.wm[jj], k);
      }
    }
    __syncthreads();
    c0 += CH;
    if (threadIdx.x == 0) {
      int no = 0;
      if (c0 < nb)
        for (int j = 0; j < W; j++)
          if (c.wm[j] >= c0) c.wopen[no++] = j;
      S.nopen = no;
    }
    __syncthreads();
    if (S.nopen == 0) break;
  }
  if (cnt) atomicAdd(&S.probes, cnt);
  if (err) S.status = RS_ERR_TIMEOUT;
}

// Cache update of the chosen worker (CTA).
__device__ void update_chosen(SimCtx& c, int j, int nb) {
  SimScalars& S = *c.S;
  const TableGeom& g = c.L->g;
  const TableView tv = c.table(j);
  CacheMeta* meta = &c.wmeta[j];
  if (threadIdx.x == 0) {
    const uint64_t span = (uint64_t)meta->T - meta->head + (uint64_t)nb;
    S.rebuild = span > g.R || meta->tombs > g.slots / 8 || (uint64_t)meta->T + nb > STAMP_LIMIT;
    update_reset(&S.us);
    S.us.err = 0;
  }
  __syncthreads();
  if (S.rebuild) {
    cache_rebuild<NT_SIM>(tv, meta, g.K, c.b->tmp + (size_t)c.sid * g.K, S.warp_tot, &S.us);
    if (threadIdx.x == 0) S.rebuilds++;
  }
  cache_lookup_all<NT_SIM>(tv, c.hbuf, nb, c.sc, &S.us, &S.probes);
  __syncthreads();
  if (S.us.dup) {
    if (threadIdx.x == 0) S.status = RS_ERR_COLLISION;
    __syncthreads();
    return;
  }
  cache_apply<NT_SIM>(tv, meta, g.K, c.hbuf, nb, c.sc, &S.us, S.warp_tot, &S.scan_pos);
  if (threadIdx.x == 0) {
    if (S.us.err) S.status = S.us.err;
    S.inserted += S.us.n_ins;
    S.evicted += S.us.n_victims;
    S.slow += S.us.slow;
  }
  __syncthreads();
}

__global__ void __launch_bounds__(NT_SIM) k_sim(const SimDesc* __restrict__ descs, SimBuffers b,
                                                SimLaunch L) {
  extern __shared__ __align__(16) unsigned char smem[];
  __shared__ SimScalars S;
  const int sid = blockIdx.x;
  const SimDesc d = descs[sid];
  const int W = L.mc.W;
  const ModelConsts& mc = L.mc;
  const SimLayout lay = make_sim_layout(W, L.nbmax, L.cmax);
  SimCtx c;
  c.S = &S;
  c.d = &d;
  c.b = &b;
  c.L = &L;
  c.sid = sid;
  c.f_a = reinterpret_cast<double*>(smem + lay.f_a);
  c.f_o = reinterpret_cast<double*>(smem + lay.f_o);
  c.h_t = reinterpret_cast<double*>(smem + lay.h_t);
  c.hbuf = reinterpret_cast<uint64_t*>(smem + lay.hbuf);
  c.f_req = reinterpret_cast<int32_t*>(smem + lay.f_req);
  c.f_worker = reinterpret_cast<int32_t*>(smem + lay.f_worker);
  c.f_blk = reinterpret_cast<int32_t*>(smem + lay.f_blk);
  c.f_O = reinterpret_cast<int32_t*>(smem + lay.f_O);
  c.f_next = reinterpret_cast<int32_t*>(smem + lay.f_next);
  c.h_f = reinterpret_cast<int32_t*>(smem + lay.h_f);
  c.freestk = reinterpret_cast<int32_t*>(smem + lay.freestk);
  c.wmeta = reinterpret_cast<CacheMeta*>(smem + lay.wmeta);
  c.winserv = reinterpret_cast<int32_t*>(smem + lay.winserv);
  c.wqh = reinterpret_cast<int32_t*>(smem + lay.wqh);
  c.wqt = reinterpret_cast<int32_t*>(smem + lay.wqt);
  c.wm = reinterpret_cast<int32_t*>(smem + lay.wm);
  c.wopen = reinterpret_cast<int32_t*>(smem + lay.wopen);
  c.wA = reinterpret_cast<int64_t*>(smem + lay.wA);
  c.wcost = reinterpret_cast<float*>(smem + lay.wcost);
  c.sc.slot = reinterpret_cast<uint32_t*>(smem + lay.slot);
  c.sc.pst = reinterpret_cast<uint32_t*>(smem + lay.pst);
  c.sc.kind = smem + lay.kind;
  c.sc.evk = smem + lay.evk;
  c.sc.vslot = reinterpret_cast<uint32_t*>(smem + lay.vslot);
  c.sc.vt = reinterpret_cast<uint32_t*>(smem + lay.vt);
  c.sc.owner = reinterpret_cast<int32_t*>(smem + lay.owner);
  c.sc.touched = smem + lay.touched;
  c.sc.victim = reinterpret_cast<int32_t*>(smem + lay.victim);
  c.sc.dupset = reinterpret_cast<uint64_t*>(smem + lay.dupset);
  c.sc.dupmask = lay.dupmask;
  double* pend = b.pend + (size_t)sid * 5 * b.pend_cap;
  c.pend_ft[0] = pend;
  c.pend_tt[0] = pend + b.pend_cap;
  c.pend_ft[1] = pend + 2 * b.pend_cap;
  c.pend_tt[1] = pend + 3 * b.pend_cap;
  c.pend_win = pend + 4 * b.pend_cap;

  // ---- initial state: empty caches, idle workers
  {
    const size_t nsl = (size_t)W * L.g.slots;
    uint64_t* keys = b.keys + (size_t)sid * nsl;
    uint32_t* st = b.stamp + (size_t)sid * nsl;
    for (size_t s = threadIdx.x; s < nsl / 2; s += NT_SIM)
      reinterpret_cast<ulonglong2*>(keys)[s] = make_ulonglong2(KEY_EMPTY, KEY_EMPTY);
    for (size_t s = threadIdx.x; s < nsl / 4; s += NT_SIM)
      reinterpret_cast<uint4*>(st)[s] = make_uint4(STAMP_NONE, STAMP_NONE, STAMP_NONE, STAMP_NONE);
    for (uint32_t s = threadIdx.x; s <= lay.dupmask; s += NT_SIM) c.sc.dupset[s] = 0ull;
    for (int p = threadIdx.x; p < d.C; p += NT_SIM) c.freestk[p] = d.C - 1 - p;
    for (int j = threadIdx.x; j < W; j += NT_SIM) {
      c.wmeta[j] = CacheMeta{0u, 0u, 0u, 0u};
      c.winserv[j] = 0;
      c.wA[j] = 0;
      c.wqh[j] = -1;
      c.wqt[j] = -1;
    }
    if (threadIdx.x == 0) {
      SimScalars z;
      memset(&z, 0, sizeof z);
      S = z;
      S.min_ft = __longlong_as_double(0x7FF0000000000000ll);
      S.next_tick = 1;
      S.nfree = d.C;
      if (d.n_req > 0) {
        S.noff0 = d.offsets[0];
        S.noff1 = d.offsets[1];
        S.rel_next = d.release[0];
        S.nO = d.out_len[0];
      }
    }
    __syncthreads();
  }

  const int64_t n = d.n_req;
  for (int64_t i = 0; i < n; i++) {
    if (threadIdx.x == 0) {
      S.off0 = S.noff0;
      S.off1 = S.noff1;
      S.rel = S.rel_next;
      S.O = S.nO;
      S.phase = 0;
    }
    __syncthreads();
    // ---- completions and controller samples up to the arrival
    for (;;) {
      if (threadIdx.x == 0) S.evres = events_advance(c);
      __syncthreads();
      if (S.evres == 0) break;
      tick_cta(c);
    }
    if (S.status != RS_OK) break;
    // ---- prefetch the next request's scalars
    if (threadIdx.x == 32 && i + 1 < n) {
      S.noff0 = d.offsets[i + 1];
      S.noff1 = d.offsets[i + 2];
      S.rel_next = d.release[i + 1];
      S.nO = d.out_len[i + 1];
    }
    const int64_t Lp = S.off1 - S.off0;
    const int64_t nb64 = Lp >> 4;
    if (nb64 > (int64_t)L.g.K) {
      if (threadIdx.x == 0) S.status = RS_ERR_CAPACITY;
      break;
    }
    const int nb = (int)nb64;
    const int nbt = (int)((Lp + 15) >> 4);
    const int64_t blk = (Lp + S.O + 15) >> 4;
    const double a = S.a_cur;
    const int64_t row = d.rec_base + i;
    // ---- stage the prompt's block hashes; regime parameters (Algorithm 1)
    const uint64_t* hsrc = d.hashes + (S.off0 >> 4);
    for (int k = threadIdx.x; k < nb; k += NT_SIM) c.hbuf[k] = __ldg(hsrc + k);
    for (int j = threadIdx.x; j < W; j += NT_SIM) {
      c.wm[j] = nb;
      c.wopen[j] = j;
    }
    if (threadIdx.x == 0) {
      S.nopen = W;
      float tau = d.tau, om = d.omega;
      if (d.policy == RS_POLICY_LOADBAL) {
        tau = 0.0f;
        om = 0.0f;
      } else if (d.controller && S.regime > 0) {
        tau = mc.regime_tau[S.regime];
        om = mc.regime_omega[S.regime];
      }
      S.tau_cur = tau;
      S.omega_cur = om;
    }
    __syncthreads();
    // ---- cached prefix on every worker
    probe_prefixes(c, nb);
    // ---- Eq. (1) costs and the frozen loads of Eq. (12)
    for (int j = threadIdx.x; j < W; j += NT_SIM) {
      const float cj = router_cost(S.omega_cur, (int64_t)nbt - c.wm[j], c.wA[j]);
      c.wcost[j] = cj;
      const int nf = min(c.winserv[j] + 1, mc.cap - 1);
      b.rec.n_frozen[row * W + j] = (uint16_t)nf;
      b.rec.prefix[row * W + j] = (uint16_t)c.wm[j];
      if (mc.write_cost) b.rec.cost[row * W + j] = cj;
    }
    __syncthreads();
    // ---- Eq. (2) choice
    if (threadIdx.x == 0) {
      for (int j = 0; j < W; j++) S.probe_blocks += min(c.wm[j] + 1, nb);
      S.hashed_blocks += nb;
      const float tau = S.tau_cur;
      const uint32_t u24 = tau > 0.0f ? draw_u24(d.seed, (uint64_t)i, 0u, TAG_SIM) : 0u;
      int nbd = 0;
      S.jstar = select_worker(c.wcost, W, tau, u24, &nbd);
      if (W >= 2) {
        const int bmin = argmin_lowest(c.wcost, W);
        float c2 = __int_as_float(0x7F800000);
        for (int j = 0; j < W; j++)
          if (j != bmin && c.wcost[j] < c2) c2 = c.wcost[j];
        const double diff = (double)c2 - (double)c.wcost[bmin];
        if (diff <= 1e-6 * fabs((double)c2)) S.near_ties++;
        if (c2 == c.wcost[bmin]) S.exact_ties++;
      }
      if (tau > 0.0f) {
        S.sampled++;
        S.near_bd += nbd;
      }
    }
    __syncthreads();
    const int js = S.jstar;
    // ---- the chosen worker's LRU cache
    update_chosen(c, js, nb);
    if (S.status != RS_OK) break;
    // ---- load, records, service start or FIFO queue
    if (threadIdx.x == 0) {
      const int f = c.freestk[--S.nfree];
      c.f_req[f] = (int32_t)i;
      c.f_worker[f] = js;
      c.f_blk[f] = (int32_t)blk;
      c.f_O[f] = S.O;
      c.f_a[f] = a;
      c.f_o[f] = nbt > 0 ? __ddiv_rn((double)c.wm[js], (double)nbt) : 0.0;
      c.f_next[f] = -1;
      c.wA[js] += blk;
      S.in_flight++;
      S.hit_blocks += c.wm[js];
      b.rec.worker[row] = js;
      b.rec.arrival[row] = a;
      b.rec.nbt[row] = nbt;
      if (c.winserv[js] < mc.cap - 1) {
        start_service(c, f, js, a);
      } else {
        if (c.wqt[js] >= 0) c.f_next[c.wqt[js]] = f; else c.wqh[js] = f;
        c.wqt[js] = f;
      }
      S.prev_arrival = a;
      S.n_routed++;
    }
    __syncthreads();
  }
  // ---- drain: remaining completions start the queued requests
  if (threadIdx.x == 0 && S.status == RS_OK) {
    while (S.nheap > 0) {
      double t;
      int f;
      heap_pop(c, &t, &f);
      complete(c, f, t);
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    rs_replica_result r;
    memset(&r, 0, sizeof r);
    r.status = S.status;
    r.final_regime = S.regime;
    r.n_routed = S.n_routed;
    r.sum_ttft = S.sum_ttft;
    r.sum_e2e = S.sum_e2e;
    r.makespan = S.makespan;
    r.poa_total = 0.0;
    r.n_windows = 0;
    r.near_ties = S.near_ties;
    r.exact_ties = S.exact_ties;
    r.sampled = S.sampled;
    r.near_boundary = S.near_bd;
    r.hit_blocks = S.hit_blocks;
    r.inserted_blocks = S.inserted;
    r.evicted_blocks = S.evicted;
    r.ticks = S.ticks;
    r.regime_switches = S.switches;
    r.max_regime = S.max_regime;
    r.ticks_in_regime[0] = S.tir[0];
    r.ticks_in_regime[1] = S.tir[1];
    r.ticks_in_regime[2] = S.tir[2];
    r.final_ewma = S.have_ewma ? S.ewma : -1.0;
    r.probes = (int64_t)S.probes;
    r.probe_blocks = S.probe_blocks;
    r.hashed_blocks = S.hashed_blocks;
    r.slow_path = S.slow;
    r.rebuilds = S.rebuilds;
    b.res[sid] = r;
  }
  for (int j = threadIdx.x; j < W; j += NT_SIM) b.meta_out[(size_t)sid * W + j] = c.wmeta[j];
}

cudaError_t launch_sim(const SimDesc* d_desc, const SimBuffers& b, const SimLaunch& L,
                       cudaStream_t st) {
  if (L.nsim <= 0) return cudaSuccess;
  const size_t smem = sim_smem_bytes(L.mc.W, L.nbmax, L.cmax);
  cudaError_t e = cudaFuncSetAttribute(k_sim, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  k_sim<<<L.nsim, NT_SIM, smem, st>>>(d_desc, b, L);
  return cudaGetLastError();
}

}  // namespace rs
