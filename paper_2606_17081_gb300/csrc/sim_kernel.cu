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
// Per request i (256 threads, 8 warps):
//   probe      warps 0-6: cached prefix m_ij on every worker; warp 7, at the
//              same time: request i's completions and controller samples up
//              to its arrival;
//   choose     every warp alike: Eq. (1) costs and the Eq. (2) choice (no
//              barrier after it);
//   update     warps 0-6 (named barrier 1): the chosen worker's cache;
//   control    warp 7, at the same time (once the update group has read its
//              inputs, named barrier 3): the decision's records and
//              statistics, request i's load, service start and latency, then
//              request i+1's scalars and block hashes into the other buffer.
// The control work is serial and runs on float64, whose dependent-operation
// latency on this GPU is long; the cache update is memory-bound.  Neither needs
// the other's results, so they overlap.  Times are ordered through an integer
// key of their bit patterns (same order as the float64 comparison, no FP64
// compare on the serial path).  Floating point follows the paper's formulas
// operation by operation (explicit _rn intrinsics, no contraction).
#include "rs_device.cuh"

namespace rs {

constexpr int NT_UPD = NT_SIM - 32;      // threads of the cache-update group (warps 0-6)
constexpr int CTL = NT_SIM - 32;         // the control thread (lane 0 of warp 7)
constexpr int FTAB_MAX = 1024;           // f(n) tabulated for n < FTAB_MAX
constexpr int PROBE_CAP = SIM_PROBE_CAP;   // W * nb up to which the probe captures every slot

__host__ __device__ inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

struct SimLayout {
  size_t ftab, f_oitl, f_a, f_o, h_k, hbuf0, hbuf1, dupset, wA;
  size_t f_req, f_worker, f_blk, f_next, h_f, freestk, owner, victim;
  size_t slot, pst, fslot, pslot, pfree, vslot, vt;
  size_t wmeta, wfreq, wtier, ptier, winserv, wqh, wqt, wm, wcost, wopen, wabs;
  size_t kind, evk, touched;
  size_t total;
  size_t slot_bytes;   // per-replica global bytes of the slot arrays (0: in shared memory)
  uint32_t dupmask;
};

// slots_global: the per-request slot arrays (times, links, the event heap;
// 56 bytes per request in flight) live in global memory, for concurrencies
// whose slots do not fit in shared memory; their offsets are then relative to
// the replica's global slot area.
__host__ __device__ inline SimLayout make_sim_layout(int W, int nbmax, int cmax, int nft,
                                                     bool slots_global = false,
                                                     bool tiered = false) {
  SimLayout L;
  size_t o = 0, og = 0;
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
#define TAKES(field, bytes, al)  /* a slot array */ \
  if (slots_global) {                               \
    og = align_up(og, al);                          \
    L.field = og;                                   \
    og += (bytes);                                  \
  } else {                                          \
    TAKE(field, bytes, al)                          \
  }
  TAKE(ftab, 8 * (size_t)(nft > 0 ? nft : 1), 16)
  TAKES(f_oitl, 8 * C, 8)
  TAKES(f_a, 8 * C, 8)
  TAKES(f_o, 8 * C, 8)
  TAKES(h_k, 8 * C, 8)
  TAKE(hbuf0, 8 * nb, 16)
  TAKE(hbuf1, 8 * nb, 16)
  TAKE(dupset, 8 * dup, 16)
  TAKE(wA, 8 * (size_t)W, 8)
  TAKES(f_req, 4 * C, 4)
  TAKES(f_worker, 4 * C, 4)
  TAKES(f_blk, 4 * C, 4)
  TAKES(f_next, 4 * C, 4)
  TAKES(h_f, 4 * C, 4)
  TAKES(freestk, 4 * C, 4)
  TAKE(owner, 4 * nv, 4)
  TAKE(victim, 4 * nv, 4)
  TAKE(slot, 4 * nb, 4)
  TAKE(pst, 4 * nb, 4)
  TAKE(fslot, 4 * nb, 4)
  TAKE(pslot, 4 * (size_t)PROBE_CAP, 16)
  TAKE(pfree, 4 * (size_t)PROBE_CAP, 16)
  TAKE(vslot, 4 * nv, 4)
  TAKE(vt, 4 * nv, 4)
  TAKE(wmeta, sizeof(CacheMeta) * (size_t)W, 16)
  TAKE(wfreq, sizeof(FreqMeta) * (size_t)W, 8)
  TAKE(wtier, tiered ? sizeof(TierMeta) * (size_t)W : 0, 8)
  TAKE(ptier, tiered ? (size_t)PROBE_CAP : 0, 4)
  TAKE(winserv, 4 * (size_t)W, 4)
  TAKE(wqh, 4 * (size_t)W, 4)
  TAKE(wqt, 4 * (size_t)W, 4)
  TAKE(wm, 4 * (size_t)W, 4)
  TAKE(wcost, 4 * (size_t)W * (NT_SIM / 32), 4)   // one cost row per warp
  TAKE(wopen, (size_t)(NT_SIM / 32) * WMAX, 4)
  TAKE(wabs, 4 * (size_t)W, 4)
  TAKE(kind, nb, 1)
  TAKE(evk, nb, 1)
  TAKE(touched, nv, 1)
#undef TAKES
#undef TAKE
  L.total = align_up(o, 16);
  L.slot_bytes = slots_global ? align_up(og, 256) : 0;
  return L;
}

__host__ __device__ inline int ftab_size(int cap) { return cap < FTAB_MAX ? cap : FTAB_MAX; }

size_t sim_smem_bytes(int W, int nbmax, int cmax, int cap, bool slots_global, bool tiered) {
  return make_sim_layout(W, nbmax, cmax, ftab_size(cap), slots_global, tiered).total;
}

size_t sim_slot_bytes(int cmax) {
  return make_sim_layout(1, 1, cmax, 1, true).slot_bytes;
}

// One request as the loop sees it (two live at once: i and i+1).
struct ReqState {
  int64_t off0;
  double oitl;     // O * itl
  int64_t blk;     // ceil((L + O) / 16): active blocks while unfinished
  double a;        // arrival
  double rel;      // client release time
  double twait;    // while waiting for a free client slot: the time reached
  int nb, nbt, O, phase, full;   // phase 0 new, 2 waiting for a slot, 1 arrival known
  int dup;                       // two blocks of the prompt share a chained hash
  float tau, omega;
};

// Request i's scalars as read from the trace (control thread).
struct RawReq {
  int64_t o0, o1;
  double rel;
  int O, dup;
};

struct SimScalars {
  ReqState q[2];
  RawReq nraw;                 // the request after the next one to arrive, as read
  double prev_arrival, min_ft, tick_t, lastL, ewma, sum_ttft, sum_e2e, makespan, first_switch_t;
  int64_t first_evict_i, first_live;   // first evicting update: request, resident blocks after it
  int64_t next_tick, np;
  int64_t near_ties, exact_ties, sampled, near_bd, hit_blocks, inserted, evicted, slow, rebuilds;
  int64_t ticks, switches, tir[3], n_routed, probe_blocks, hashed_blocks;
  unsigned long long probes;
  uint64_t sel_prefix;
  int32_t in_flight, nheap, nfree, evres, status, jstar, regime, up_cnt, down_cnt;
  int32_t have_L, have_ewma, max_regime, pend_cur, sel_kk;
  uint32_t dclock;             // decay step of the request being updated (frequency eviction)
  int64_t kv[5];               // Game 2: own G1 / G2 / G3, remote, recompute blocks
  double kv_cost;              // summed Eq. kv-cost
  int kvacc[10];               // one request's Game 2 categories (update group)
  int64_t tier_out;            // blocks the last update pushed out of G1
  UpdateShared us;
  uint32_t scan_pos;
  int warp_tot[NT_SIM / 32];
  int hist[256];
  double red[NT_SIM / 32];
  FreqShared fs;               // the frequency update's scalars
};

// Everything a device helper needs, resolved once per CTA.
struct SimCtx {
  SimScalars* S;
  const SimDesc* d;
  const SimBuffers* b;
  const SimLaunch* L;
  int sid;
  double *f_a, *f_o, *ftab, *f_oitl;
  uint64_t* h_k;
  uint64_t *hbuf0, *hbuf1;
  int32_t *f_req, *f_worker, *f_blk, *f_next, *h_f, *freestk;
  CacheMeta* wmeta;
  FreqMeta* wfreq;
  TierMeta* wtier;    // Game 2 band boundaries per worker (tiered)
  uint8_t* ptier;     // [W][nb] tier of each (worker, block) pair, 0 = absent (tiered)
  int32_t *winserv, *wqh, *wqt, *wm, *wabs;
  uint8_t* wopen;     // [NT_SIM / 32][WMAX] each probing warp's open workers
  uint32_t *pslot, *pfree;
  int64_t* wA;
  float* wcost;
  UpdateScratch sc;
  double *pend_ft0, *pend_tt0, *pend_ft1, *pend_tt1, *pend_win;

  __device__ __forceinline__ uint64_t* hbuf(int p) const { return p ? hbuf1 : hbuf0; }
  __device__ __forceinline__ double* pend_ft(int p) const { return p ? pend_ft1 : pend_ft0; }
  __device__ __forceinline__ double* pend_tt(int p) const { return p ? pend_tt1 : pend_tt0; }

  __device__ __forceinline__ TableView table(int j) const {
    TableView t;
    const size_t wi = (size_t)sid * L->mc.W + j;
    t.keys = b->keys + wi * L->g.slots;
    t.stamp = b->stamp + wi * L->g.slots;
    t.log = b->log + wi * L->g.R;
    t.fexp = b->fexp ? b->fexp + wi * L->g.slots : nullptr;
    t.bmask = L->g.bmask;
    t.rmask = L->g.rmask;
    return t;
  }
};

// Monotone integer key of a float64 (same order as the float64 comparison
// for every non-NaN value) and its inverse.
__device__ __forceinline__ uint64_t tkey(double x) {
  const uint64_t b = (uint64_t)__double_as_longlong(x);
  return (b >> 63) ? ~b : (b | 0x8000000000000000ull);
}
__device__ __forceinline__ double tval(uint64_t k) {
  const uint64_t b = (k >> 63) ? (k & 0x7FFFFFFFFFFFFFFFull) : ~k;
  return __longlong_as_double((long long)b);
}
constexpr uint64_t KEY_INF = 0xFFF0000000000000ull;   // tkey(+infinity)

// ------------------------------------------------------------ event machinery (control thread)

__device__ __forceinline__ bool ev_less(const SimCtx& c, uint64_t ka, int fa, uint64_t kb, int fb) {
  return ka < kb || (ka == kb && c.f_req[fa] < c.f_req[fb]);
}

// The completions heap: 4-ary (children of i at 4i+1 .. 4i+4), half the
// levels of a binary heap on the control thread's dependent chain; ev_less is
// a strict total order (time, then request), so the pops are the same events
// in the same order whatever the heap's shape.
constexpr int HEAP_D = 4;

__device__ __forceinline__ void heap_push(SimCtx& c, uint64_t k, int f) {
  int i = c.S->nheap++;
  while (i > 0) {
    const int p = (i - 1) / HEAP_D;
    if (!ev_less(c, k, f, c.h_k[p], c.h_f[p])) break;
    c.h_k[i] = c.h_k[p];
    c.h_f[i] = c.h_f[p];
    i = p;
  }
  c.h_k[i] = k;
  c.h_f[i] = f;
}

__device__ __forceinline__ void heap_pop(SimCtx& c, uint64_t* k, int* f) {
  *k = c.h_k[0];
  *f = c.h_f[0];
  const int n = --c.S->nheap;
  const uint64_t lk = c.h_k[n];
  const int lf = c.h_f[n];
  int i = 0;
  for (;;) {
    const int c0 = HEAP_D * i + 1;
    if (c0 >= n) break;
    const int c1 = min(c0 + HEAP_D, n);
    // the children's keys first (independent loads), then their minimum
    uint64_t kk[HEAP_D];
#pragma unroll
    for (int q = 0; q < HEAP_D; q++) kk[q] = c0 + q < c1 ? c.h_k[c0 + q] : KEY_INF;
    int s = c0;
    uint64_t ks = kk[0];
    int fs = c.h_f[c0];
#pragma unroll
    for (int q = 1; q < HEAP_D; q++) {
      if (c0 + q >= c1) break;
      const int fq = c.h_f[c0 + q];
      if (ev_less(c, kk[q], fq, ks, fs)) {
        s = c0 + q;
        ks = kk[q];
        fs = fq;
      }
    }
    if (!ev_less(c, ks, fs, lk, lf)) break;
    c.h_k[i] = ks;
    c.h_f[i] = fs;
    i = s;
  }
  c.h_k[i] = lk;
  c.h_f[i] = lf;
}

// Eq. (9) with beta = 2: f(n) = a n + b + d / (cap - n)^2
__device__ __forceinline__ double latency_f(const ModelConsts& mc, int n) {
  const double t1 = __dmul_rn(mc.lat_a, (double)n);
  const double t2 = __dadd_rn(t1, mc.lat_b);
  const double den = (double)(mc.cap - n);
  const double t3 = __ddiv_rn(mc.lat_d, __dmul_rn(den, den));
  return __dadd_rn(t2, t3);
}

// Service of slot f starts on worker j at time t: TTFT = wait + f(n) - w_c o.
__device__ __forceinline__ void start_service(SimCtx& c, int f, int j, double t) {
  SimScalars& S = *c.S;
  const ModelConsts& mc = c.L->mc;
  const int n = ++c.winserv[j];
  const double fv = n < FTAB_MAX ? c.ftab[n] : latency_f(mc, n);
  const double svc = __dsub_rn(fv, c.f_o[f]);          // f_o holds w_c * o
  const double ft = __dadd_rn(t, svc);
  const double tt = __dsub_rn(ft, c.f_a[f]);
  const double ct = __dadd_rn(ft, c.f_oitl[f]);         // O * itl
  const int64_t row = c.d->rec_base + c.f_req[f];
  c.b->rec.start[row] = t;
  c.b->rec.first_token[row] = ft;
  c.b->rec.ttft[row] = tt;
  c.b->rec.completion[row] = ct;
  heap_push(c, tkey(ct), f);
  if (c.d->controller) {
    const int cur = S.pend_cur;
    c.pend_ft(cur)[S.np] = ft;
    c.pend_tt(cur)[S.np] = tt;
    S.np++;
    if (tkey(ft) < tkey(S.min_ft)) S.min_ft = ft;
  }
}

__device__ __forceinline__ void complete(SimCtx& c, int f, double t) {
  SimScalars& S = *c.S;
  const int j = c.f_worker[f];
  c.winserv[j]--;
  c.wA[j] -= c.f_blk[f];
  S.in_flight--;
  c.freestk[S.nfree++] = f;
  const int f2 = c.wqh[j];
  if (f2 >= 0) {
    c.wqh[j] = c.f_next[f2];
    if (c.wqh[j] < 0) c.wqt[j] = -1;
    start_service(c, f2, j, t);
  }
}

// EWMA of Eq. (10) and the hysteretic regime of Eq. (11); one sample.
__device__ __forceinline__ void ctl_sample(SimCtx& c, bool has_window, double Lw) {
  SimScalars& S = *c.S;
  const ModelConsts& mc = c.L->mc;
  const int64_t sw0 = S.switches;
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
  if (sw0 == 0 && S.switches > 0) S.first_switch_t = S.tick_t;   // this sample's time
  S.tir[S.regime]++;
  S.ticks++;
  S.next_tick++;
  S.tick_t = __dmul_rn((double)S.next_tick, mc.dt);
  if (S.ticks >= TICK_LIMIT) S.status = RS_ERR_CAPACITY;
}

__device__ __forceinline__ uint64_t tick_key(const SimCtx& c) {
  return c.d->controller ? tkey(c.S->tick_t) : KEY_INF;
}

// Advances events for request q (control thread).  Returns 1 when a
// controller sample with a non-empty window is due (the CTA computes it), 0
// when the arrival time is known and every event up to it is processed.
__device__ __forceinline__ int events_advance(SimCtx& c, ReqState& q) {
  SimScalars& S = *c.S;
  if (q.phase == 0) {
    q.twait = S.prev_arrival;
    q.phase = 2;
  }
  if (q.phase == 2) {
    // closed-loop client (§7.4): wait until fewer than C(t) requests are in
    // flight; completions, controller samples and steps of the load-spike
    // schedule in time order (ties in that order)
    const SimDesc& d = *c.d;
    for (;;) {
      const uint64_t kw = tkey(q.twait);
      const bool mid = d.c_mid > 0 && kw >= tkey(d.c_t1);
      const bool end = d.c_mid > 0 && kw >= tkey(d.c_t2);
      const int conc = end ? d.c_end : (mid ? d.c_mid : d.C);
      if (S.in_flight < conc) break;
      if (S.status != RS_OK) return 0;
      const uint64_t kc = S.nheap > 0 ? c.h_k[0] : KEY_INF;
      const uint64_t kt = tick_key(c);
      const uint64_t ks = d.c_mid <= 0 || end ? KEY_INF : tkey(mid ? d.c_t2 : d.c_t1);
      if (kc == KEY_INF && ks == KEY_INF) {   // cannot happen: a request in flight is in service
        S.status = RS_ERR_TIMEOUT;
        return 0;
      }
      if (kc <= kt && kc <= ks) {
        uint64_t k;
        int f;
        heap_pop(c, &k, &f);
        const double t = tval(k);
        complete(c, f, t);
        if (k > kw) q.twait = t;
      } else if (kt <= ks) {
        if (tkey(S.min_ft) >= kt) { ctl_sample(c, false, 0.0); continue; }
        return 1;
      } else {
        q.twait = mid ? d.c_t2 : d.c_t1;   // the schedule steps
      }
    }
    q.a = tkey(q.rel) > tkey(q.twait) ? q.rel : q.twait;
    q.phase = 1;
  }
  const uint64_t ka = tkey(q.a);
  for (;;) {
    if (S.status != RS_OK) return 0;
    const uint64_t kc = S.nheap > 0 ? c.h_k[0] : KEY_INF;
    const uint64_t kt = tick_key(c);
    if (kc <= kt) {
      if (kc > ka) break;
      uint64_t k;
      int f;
      heap_pop(c, &k, &f);
      complete(c, f, tval(k));
    } else {
      if (kt > ka) break;
      if (tkey(S.min_ft) >= kt) { ctl_sample(c, false, 0.0); continue; }
      return 1;
    }
  }
  return 0;
}

// ------------------------------------------------------------ controller sample (CTA)

// The window holds the TTFTs of requests whose first token came before the
// sample time and after the previous sample; its nearest-rank P99 (exact
// radix selection over the float64 bit patterns, TTFT > 0) feeds Eq. (10).
__device__ __forceinline__ void tick_cta(SimCtx& c) {
  SimScalars& S = *c.S;
  const double tt = S.tick_t;
  const int cur = S.pend_cur;
  const int64_t np = S.np;
  const double* sft = c.pend_ft(cur);
  const double* stt = c.pend_tt(cur);
  double* dft = c.pend_ft(cur ^ 1);
  double* dtt = c.pend_tt(cur ^ 1);
  int64_t nkeep = 0, nwin = 0;
  uint64_t mft = KEY_INF;
  const uint64_t ktt = tkey(tt);
  for (int64_t p0 = 0; p0 < np; p0 += NT_SIM) {
    const int64_t p = p0 + threadIdx.x;
    bool keep = false, inwin = false;
    double f = 0.0, v = 0.0;
    if (p < np) {
      f = sft[p];
      v = stt[p];
      inwin = tkey(f) < ktt;
      keep = !inwin;
    }
    int t1, t2;
    const int r1 = cta_rank<NT_SIM>(keep, S.warp_tot, &t1);
    const int r2 = cta_rank<NT_SIM>(inwin, S.warp_tot, &t2);
    if (keep) {
      dft[nkeep + r1] = f;
      dtt[nkeep + r1] = v;
      const uint64_t kf = tkey(f);
      mft = kf < mft ? kf : mft;
    }
    if (inwin) c.pend_win[nwin + r2] = v;
    nkeep += t1;
    nwin += t2;
  }
  for (int o = 16; o > 0; o >>= 1) {
    const uint64_t v = __shfl_xor_sync(FULL_MASK, mft, o);
    mft = v < mft ? v : mft;
  }
  if ((threadIdx.x & 31) == 0) S.red[threadIdx.x >> 5] = tval(mft);
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
  if (threadIdx.x == CTL) {
    uint64_t m = tkey(S.red[0]);
    for (int w = 1; w < NT_SIM / 32; w++) {
      const uint64_t k = tkey(S.red[w]);
      m = k < m ? k : m;
    }
    S.np = nkeep;
    S.pend_cur = cur ^ 1;
    S.min_ft = tval(m);
    ctl_sample(c, nwin > 0, L);
  }
  __syncthreads();
}

// ------------------------------------------------------------ routing step

// A warp's lookups sit at consecutive lanes; those of one worker cover
// consecutive blocks, the lane holding the window's position kw on the
// worker's span of `span` blocks.  The lanes of that span in this warp, as a
// mask: from lane - kw to lane - kw + span - 1, clipped to the warp.
__device__ __forceinline__ unsigned span_mask(int lane, int kw, int span) {
  const int lo = lane - kw > 0 ? lane - kw : 0;
  const int hi = lane - kw + span;   // one past the span's last lane
  const unsigned below_hi = hi >= 32 ? FULL_MASK : (hi > 0 ? (1u << hi) - 1u : 0u);
  return below_hi & ~((1u << lo) - 1u);
}

// Resolves ILP loaded home buckets: sl[r] the slot holding hh[r] or
// SLOT_NONE, fr[r] the first free slot of its probe path.  A bucket full of
// other keys (rare at the tables' load) continues along the probe sequence
// after all of them are scanned, so the common case runs straight through.
template <int ILP>
__device__ __forceinline__ void resolve_buckets(const SimCtx& c, const uint64_t (&v)[ILP][BUCKET],
                                                const uint32_t (&bk)[ILP],
                                                const uint64_t (&hh)[ILP], const int (&jj)[ILP],
                                                uint32_t (&sl)[ILP], uint32_t (&fr)[ILP],
                                                int* err) {
  bool cont[ILP], any = false;
#pragma unroll
  for (int r = 0; r < ILP; r++) {
    sl[r] = SLOT_NONE;
    fr[r] = SLOT_NONE;
    cont[r] = bucket_scan_masks(v[r], bk[r], hh[r], &sl[r], &fr[r]) < 0 && jj[r] >= 0;
    any |= cont[r];
  }
  if (any) {
#pragma unroll
    for (int r = 0; r < ILP; r++)
      if (cont[r]) {
        const TableView t = c.table(jj[r]);
        sl[r] = table_find_free_from(t, hh[r], (bk[r] + 1) & t.bmask, err, &fr[r]);
      }
  }
}

// m_j: leading blocks of the prompt found in worker j's cache, for every j
// (threads of the group), when W nb is too large to look every pair up at
// once.  Rounds over the workers still undecided: a round looks up the next
// `len` blocks of each open worker, with len = ILP NT / (open workers) so
// that a round is ILP lookups per thread (4 with one replica per SM under LRU,
// 1 within the two-per-SM register budget or under frequency eviction, whose
// heap leaves no registers for more), all issued before any is resolved;
// a worker is decided once a miss falls in its window.  Most workers miss at
// their first block, so the few left open after the first round get long
// windows.  Each warp lists the open workers for itself after the round's
// barrier: a miss of the next round lowers m_j only to a block at or past
// that round's start, so a worker's open state does not depend on when a
// warp reads it, and no second barrier is needed.
template <int NT, int ILP>
__device__ __forceinline__ void probe_prefixes(SimCtx& c, const uint64_t* hbuf, int nb) {
  SimScalars& S = *c.S;
  const int W = c.L->mc.W;
  const int lane = (int)(threadIdx.x & 31);
  uint8_t* wl = c.wopen + (threadIdx.x >> 5) * WMAX;   // this warp's open workers
  for (int j = lane; j < W; j += 32) wl[j] = (uint8_t)j;
  __syncwarp();
  int nopen = W;
  int c0 = 0;
  int err = 0;
  unsigned cnt = 0;
  for (;;) {
    int len = (ILP * NT) / nopen;
    if (len < 1) len = 1;
    if (len > nb - c0) len = nb - c0;   // (>= 1: the workers listed are open, so c0 < nb)
    const int total = nopen * len;      // <= ILP NT
    // open worker of lookup `it` = floor(it / len): (it + 0.5) / len lies at
    // least 0.5 / len from an integer and it < ILP NT, so the float product
    // truncates to it exactly
    const float inv_len = 1.0f / (float)len;
    int jj[ILP], kk[ILP], kw[ILP];
    uint64_t hh[ILP], v[ILP][BUCKET];
    uint32_t bk[ILP];
    // every lookup's home bucket requested before any is resolved; a thread
    // past the round's lookups repeats the round's last one (in bounds, unused)
#pragma unroll
    for (int r = 0; r < ILP; r++) {
      const int it0 = r * NT + (int)threadIdx.x;
      const int it = it0 < total ? it0 : total - 1;
      const int o = (int)(((float)it + 0.5f) * inv_len);
      const int j = wl[o];
      kw[r] = it - o * len;
      kk[r] = c0 + kw[r];
      jj[r] = it0 < total && kk[r] < c.wm[j] ? j : -1;   // (no miss known below k yet)
      hh[r] = hbuf[kk[r]];
      const TableView t = c.table(j);
      bk[r] = home_bucket(hh[r], t.bmask);
      ld_bucket(t.keys, bk[r], v[r]);
    }
    uint32_t sl[ILP], fr[ILP];
    resolve_buckets<ILP>(c, v, bk, hh, jj, sl, fr, &err);
#pragma unroll
    for (int r = 0; r < ILP; r++) {
      if (r > 0 && r * NT >= total) break;   // (uniform)
      cnt += jj[r] >= 0;
      // the first miss of the worker's window in this warp: its lanes rise
      // by one block each, so it is the window's lowest missing lane, and
      // the window's lowest lane here (kw = 0, or lane 0) records it
      const unsigned mb =
          __ballot_sync(FULL_MASK, jj[r] >= 0 && sl[r] == SLOT_NONE) & span_mask(lane, kw[r], len);
      if (jj[r] >= 0 && mb && (kw[r] == 0 || lane == 0))
        atomicMin(&c.wm[jj[r]], kk[r] + (__ffs(mb) - 1) - lane);
    }
    grp_bar<NT>();   // every miss of the round is in wm
    c0 += len;
    nopen = 0;
    for (int j0 = 0; j0 < W; j0 += 32) {
      const int j = j0 + lane;
      const bool op = c0 < nb && j < W && c.wm[j] >= c0;
      const unsigned bal = __ballot_sync(FULL_MASK, op);
      if (op) wl[nopen + __popc(bal & ((1u << lane) - 1u))] = (uint8_t)j;
      nopen += __popc(bal);
    }
    __syncwarp();
    if (nopen == 0) break;
  }
  cnt = __reduce_add_sync(FULL_MASK, cnt);
  if (lane == 0 && cnt) atomicAdd(&S.probes, (unsigned long long)cnt);
  if (err) S.status = RS_ERR_TIMEOUT;
}

// The same m_j with every (worker, block) pair looked up at once (W nb <=
// PROBE_CAP): each thread issues the first-bucket loads of ILP pairs
// before resolving them, and the slot found (or the first free slot of the
// probe path) is kept for the chosen worker's update.
// TIER: m_j counts the leading blocks in G1 (a found slot's stamp at or
// past the worker's b1); every pair's tier goes to ptier; the absent count
// is of blocks in no tier.
template <int NT, int ILP, bool TIER = false>
__device__ __forceinline__ void probe_full(SimCtx& c, const uint64_t* hbuf, int nb) {
  SimScalars& S = *c.S;
  const int W = c.L->mc.W;
  const int total = W * nb;
  const int lane = (int)(threadIdx.x & 31);
  // worker of pair `it` = floor(it / nb): (it + 0.5) / nb lies at least
  // 0.5 / nb from an integer, and with W nb <= PROBE_CAP the float product's
  // error stays far below that, so it truncates to the quotient exactly
  const float inv_nb = nb > 0 ? 1.0f / (float)nb : 0.0f;
  int err = 0;
  for (int base = 0; base < total; base += NT * ILP) {   // uniform
    int jj[ILP], kk[ILP];
    uint64_t hh[ILP], v[ILP][BUCKET];
    uint64_t stw[ILP][TIER ? 4 : 1];   // tiers: the home bucket's 8 stamps, beside its keys
    uint32_t bk[ILP];
    // every pair's home bucket requested before any is resolved; a thread
    // past the pairs repeats the last one (in bounds, unused)
#pragma unroll
    for (int r = 0; r < ILP; r++) {
      const int it0 = base + r * NT + (int)threadIdx.x;
      const int it = it0 < total ? it0 : total - 1;
      const int j = (int)(((float)it + 0.5f) * inv_nb);
      jj[r] = it0 < total ? j : -1;
      kk[r] = it - j * nb;
      hh[r] = hbuf[kk[r]];
      const TableView t = c.table(j);
      bk[r] = home_bucket(hh[r], t.bmask);
      ld_bucket(t.keys, bk[r], v[r]);
      if (TIER)   // one 32-byte sector: stamps are 4-byte, buckets of 8 start 32-byte aligned
        ld_keys4(reinterpret_cast<const uint64_t*>(t.stamp + (size_t)BUCKET * bk[r]), stw[r][0],
                 stw[r][TIER ? 1 : 0], stw[r][TIER ? 2 : 0], stw[r][TIER ? 3 : 0]);
    }
    uint32_t sl[ILP], fr[ILP];
    resolve_buckets<ILP>(c, v, bk, hh, jj, sl, fr, &err);
#pragma unroll
    for (int r = 0; r < ILP; r++) {
      const int it = base + r * NT + (int)threadIdx.x;
      bool miss = false, absent = false;
      if (jj[r] >= 0) {
        c.pslot[it] = sl[r];
        c.pfree[it] = fr[r];
        if (TIER) {
          int tier = 0;
          if (sl[r] != SLOT_NONE) {
            uint32_t st;
            if (sl[r] / BUCKET == bk[r]) {   // in the home bucket: its stamp came with the keys
              const uint32_t q = sl[r] % BUCKET;
              const uint64_t w2 = q < 2 ? stw[r][0]
                                        : (q < 4 ? stw[r][TIER ? 1 : 0]
                                                 : (q < 6 ? stw[r][TIER ? 2 : 0]
                                                          : stw[r][TIER ? 3 : 0]));
              st = (uint32_t)(q & 1u ? w2 >> 32 : w2);
            } else {
              st = __ldcg(c.table(jj[r]).stamp + sl[r]);
            }
            const TierMeta tm = c.wtier[jj[r]];
            tier = st >= tm.b1 ? 1 : (st >= tm.b2 ? 2 : 3);
          }
          c.ptier[it] = (uint8_t)tier;
          absent = sl[r] == SLOT_NONE;
          miss = tier != 1;
        } else {
          miss = sl[r] == SLOT_NONE;
        }
      }
      // per worker's lanes in this warp (blocks rise by one per lane): the
      // first miss and the absent count, recorded by the worker's lowest
      // lane here (block 0, or lane 0)
      const unsigned span = span_mask(lane, kk[r], nb);
      const unsigned mb = __ballot_sync(FULL_MASK, miss) & span;
      const unsigned nab = TIER ? __popc(__ballot_sync(FULL_MASK, absent) & span) : __popc(mb);
      // (tiers: a block below G1 ends the prefix though it is present)
      if (jj[r] >= 0 && (kk[r] == 0 || lane == 0) && (nab || (TIER && mb))) {
        if (mb) atomicMin(&c.wm[jj[r]], kk[r] + (__ffs(mb) - 1) - lane);
        if (nab) atomicAdd(&c.wabs[jj[r]], (int)nab);   // absent blocks, for the victim count
      }
    }
  }
  if (threadIdx.x == 0) S.probes += (unsigned long long)total;
  if (err) S.status = RS_ERR_TIMEOUT;
  // (the CTA barrier after the probe orders these results with their readers)
}

// Game 2 charge of request i (Eq. kv-cost, §4.2) on its worker sigma, from the
// probe's tiers (update group, before the update): per block alpha_t for
// sigma's own tier t; else the cheapest d(sigma, j) + alpha_t over other
// workers' copies (same node before other node, then the lower tier); else
// gamma.  The categories are counted, and the cost summed in a fixed order.
template <int NT>
__device__ __forceinline__ void tier_charge(SimCtx& c, int sigma, int nb, int64_t row) {
  SimScalars& S = *c.S;
  const ModelConsts& mc = c.L->mc;
  const int W = mc.W;
  const int node = sigma / mc.tier_node;
  int cnt[10];
#pragma unroll
  for (int q = 0; q < 10; q++) cnt[q] = 0;
  for (int k = threadIdx.x; k < nb; k += NT) {
    const int t = c.ptier[sigma * nb + k];
    if (t > 0) {
      cnt[t - 1]++;
      continue;
    }
    unsigned has = 0;   // bit 3 r + (q - 1): a copy at tier q, r = 0 same node, 1 other
    for (int j = 0; j < W; j++) {
      const int tj = c.ptier[j * nb + k];
      if (j == sigma || tj == 0) continue;
      has |= 1u << (3 * (j / mc.tier_node == node ? 0 : 1) + tj - 1);
    }
    int cat = 9;
    double best = __longlong_as_double(0x7FF0000000000000ll);
    for (int b = 0; b < 6; b++) {
      if (!(has >> b & 1u)) continue;
      const double v = __dadd_rn(b < 3 ? mc.tier_dn : mc.tier_df, mc.tier_alpha[b % 3]);
      if (v < best) {
        best = v;
        cat = 3 + b;
      }
    }
    cnt[cat]++;
  }
#pragma unroll
  for (int q = 0; q < 10; q++) {
    const int v = (int)__reduce_add_sync(FULL_MASK, (unsigned)cnt[q]);
    if ((threadIdx.x & 31) == 0 && v) atomicAdd(&S.kvacc[q], v);
  }
  grp_bar<NT>();
  if (threadIdx.x == 0) {
    const double* al = mc.tier_alpha;
    double cost = __dmul_rn(al[0], (double)S.kvacc[0]);
    cost = __dadd_rn(cost, __dmul_rn(al[1], (double)S.kvacc[1]));
    cost = __dadd_rn(cost, __dmul_rn(al[2], (double)S.kvacc[2]));
    for (int q = 0; q < 3; q++)
      cost = __dadd_rn(cost, __dmul_rn(__dadd_rn(mc.tier_dn, al[q]), (double)S.kvacc[3 + q]));
    for (int q = 0; q < 3; q++)
      cost = __dadd_rn(cost, __dmul_rn(__dadd_rn(mc.tier_df, al[q]), (double)S.kvacc[6 + q]));
    cost = __dadd_rn(cost, __dmul_rn(mc.tier_gamma, (double)S.kvacc[9]));
    S.kv[0] += S.kvacc[0];
    S.kv[1] += S.kvacc[1];
    S.kv[2] += S.kvacc[2];
    S.kv[3] += S.kvacc[3] + S.kvacc[4] + S.kvacc[5] + S.kvacc[6] + S.kvacc[7] + S.kvacc[8];
    S.kv[4] += S.kvacc[9];
    S.kv_cost = __dadd_rn(S.kv_cost, cost);
    if (c.b->rec.kv_cost) c.b->rec.kv_cost[row] = cost;
#pragma unroll
    for (int q = 0; q < 10; q++) S.kvacc[q] = 0;   // for the next request
  }
}

// Moves a band boundary of the recency stack past `excess` live log entries
// (they drop to the band below): the new boundary follows the excess-th live
// entry at or after *b.  CTA-wide.
template <int NT>
__device__ __forceinline__ void tier_shift(const TableView& t, const CacheMeta* meta, uint32_t* b,
                                           uint32_t excess, int* warp_tot, uint32_t* out) {
  if (excess == 0) return;
  const uint32_t T = meta->T;
  uint32_t have = 0;
  for (uint32_t p0 = *b; p0 < T; p0 += NT) {   // uniform
    const uint32_t p = p0 + threadIdx.x;
    bool live = false;
    if (p < T) live = __ldcg(t.stamp + t.log[p & t.rmask]) == p;
    int tot;
    const int r = cta_rank<NT>(live, warp_tot, &tot);
    if (live && have + (uint32_t)r == excess - 1) *out = p + 1;
    have += (uint32_t)tot;
    if (have >= excess) break;
  }
  grp_bar<NT>();
  if (threadIdx.x == 0) *b = have >= excess ? *out : T;
  grp_bar<NT>();
}

// After the chosen worker's LRU update of its whole stack: the G1 and G2
// bands move down by the live entries that no longer fit.  size0, b0: the
// stack size and boundaries before the update; us/sc: the update's record
// (kinds, present blocks' old stamps, victims).  Sets S.tier_out = blocks that
// left G1 (moved below b1, or evicted from it).
template <int NT>
__device__ __forceinline__ void tier_advance(SimCtx& c, const TableView& tv, const CacheMeta* meta,
                                             TierMeta* tm, uint32_t size0, TierMeta b0, int nb) {
  SimScalars& S = *c.S;
  const UpdateScratch& sc = c.sc;
  int d1 = 0, d2 = 0, v1 = 0;
  for (int k = threadIdx.x; k < nb; k += NT)
    if (sc.kind[k] == 0) {
      d1 += sc.pst[k] >= b0.b1;
      d2 += sc.pst[k] >= b0.b2;
    }
  const int E = S.us.n_victims;
  for (int v = threadIdx.x; v < E; v += NT) {
    const uint32_t p = sc.vt[sc.victim[v]];
    v1 += p >= b0.b1;
    d2 += p >= b0.b2;
  }
  d1 += v1;
  d1 = (int)__reduce_add_sync(FULL_MASK, (unsigned)d1);
  d2 = (int)__reduce_add_sync(FULL_MASK, (unsigned)d2);
  v1 = (int)__reduce_add_sync(FULL_MASK, (unsigned)v1);
  if ((threadIdx.x & 31) == 0) {
    atomicAdd(&S.kvacc[0], d1);   // kvacc is free between charges
    atomicAdd(&S.kvacc[1], d2);
    atomicAdd(&S.kvacc[2], v1);
  }
  grp_bar<NT>();
  const uint32_t size = meta->size;
  const int64_t k1 = c.L->k1, k12 = c.L->k12;
  const int64_t live1 = min((int64_t)size0, k1) - S.kvacc[0] + nb;
  const int64_t live2 = min((int64_t)size0, k12) - S.kvacc[1] + nb;
  const int64_t x1 = live1 - min((int64_t)size, k1);
  const int64_t x2 = live2 - min((int64_t)size, k12);
  const int vout = S.kvacc[2];
  grp_bar<NT>();
  if (threadIdx.x == 0) {
    S.kvacc[0] = S.kvacc[1] = S.kvacc[2] = 0;
    S.tier_out = (x1 > 0 ? x1 : 0) + vout;
    if ((int64_t)size <= k1) tm->b1 = meta->head;
    if ((int64_t)size <= k12) tm->b2 = meta->head;
  }
  if ((int64_t)size > k1 && x1 > 0) tier_shift<NT>(tv, meta, &tm->b1, (uint32_t)x1, S.warp_tot, &S.scan_pos);
  if ((int64_t)size > k12 && x2 > 0) tier_shift<NT>(tv, meta, &tm->b2, (uint32_t)x2, S.warp_tot, &S.scan_pos);
  grp_bar<NT>();
}

// Cache update of the chosen worker (update group, warps 0-6) for request i.
// MODE: SIM_FREQ when the launch holds replicas that evict by frequency,
// SIM_TIER for Game 2 tiers (the LRU-only kernel carries neither).
// nabs: the worker's absent blocks (from the probe); rebuild: rebuild the
// table first; dup: the prompt repeats a block hash (the update stops).
template <int MODE>
__device__ __forceinline__ void update_chosen(SimCtx& c, const uint64_t* hbuf, int j, int nb,
                                              bool full, int64_t i, int nabs, bool rebuild,
                                              bool dup) {
  constexpr bool FREQ = MODE == SIM_FREQ, TIER = MODE == SIM_TIER;
  SimScalars& S = *c.S;
  const TableGeom& g = c.L->g;
  const TableView tv = c.table(j);
  CacheMeta* meta = &c.wmeta[j];
  if (dup) {
    if (threadIdx.x == 0) S.status = RS_ERR_COLLISION;
    return;
  }
  uint64_t* gtmp = c.b->tmp + (size_t)c.sid * g.K;
  if (rebuild) {
    cache_rebuild<NT_UPD>(tv, meta, g.K, gtmp, S.warp_tot, &S.us,
                          FREQ && c.b->tmpe ? c.b->tmpe + (size_t)c.sid * g.K : nullptr,
                          FREQ ? &c.wfreq[j] : nullptr);
    if (threadIdx.x == 0) {
      S.rebuilds++;
      if (TIER) {   // stamps renumbered 0 .. size-1 in recency order
        const int64_t sz = meta->size;
        c.wtier[j].b1 = (uint32_t)(sz - min(sz, c.L->k1));
        c.wtier[j].b2 = (uint32_t)(sz - min(sz, c.L->k12));
      }
    }
    if (TIER) grp_bar<NT_UPD>();
  }
  const uint32_t size0 = meta->size;   // before this update (tiers)
  const TierMeta b0 = TIER ? c.wtier[j] : TierMeta{0u, 0u};
  const bool captured = full && !rebuild;
  if (FREQ && c.d->eviction == RS_EVICT_FREQ) {
    // the KV Block Manager's frequency rule
    const uint32_t D = S.dclock;
    FreqMeta* fm = &c.wfreq[j];
    if (captured) {
      cache_prepare_captured_freq<NT_UPD>(tv, meta, fm, g.K, c.pslot + (size_t)j * nb,
                                          c.pfree + (size_t)j * nb, nb, nabs, D, c.sc, &S.us,
                                          &S.fs, S.warp_tot, &S.scan_pos);
    } else {
      cache_lookup_all<NT_UPD, false>(tv, hbuf, nb, c.sc, &S.us, &S.probes);
      freq_present<NT_UPD>(tv, meta, fm, nb, D, c.sc, &S.us, &S.fs, &S.scan_pos);
    }
    cache_apply_freq<NT_UPD>(tv, meta, fm, g.K, hbuf, nb, D, (uint32_t)c.d->freq_max, c.sc, &S.us,
                             &S.fs, S.warp_tot, &S.scan_pos, gtmp);
  } else {
    if (captured)
      cache_prepare_captured<NT_UPD>(tv, meta, g.K, c.pslot + (size_t)j * nb,
                                     c.pfree + (size_t)j * nb, nb, nabs, c.sc, &S.us,
                                     S.warp_tot, &S.scan_pos);
    else
      cache_lookup_all<NT_UPD, false>(tv, hbuf, nb, c.sc, &S.us, &S.probes);
    cache_apply<NT_UPD>(tv, meta, g.K, hbuf, nb, c.sc, &S.us, S.warp_tot, &S.scan_pos, captured);
    if (TIER) {
      grp_bar<NT_UPD>();   // the meta update of cache_apply
      tier_advance<NT_UPD>(c, tv, meta, &c.wtier[j], size0, b0, nb);
    }
  }
  if (threadIdx.x == 0) {
    if (S.us.err) S.status = S.us.err;
    S.inserted += S.us.n_ins;
    S.evicted += S.us.n_victims;
    if ((TIER ? S.tier_out : (int64_t)S.us.n_victims) > 0 && S.first_evict_i < 0) {
      // the first update that evicted; resident blocks = inserted - evicted
      S.first_evict_i = i;
      S.first_live = S.inserted - S.evicted;
    }
    S.slow += S.us.slow;
    update_reset(&S.us);   // for the next request
    S.us.err = 0;
  }
}

// w_c * o_ij of Eq. (9) for a cached prefix of m of the prompt's nbt blocks:
// from the table of every (m, nbt) when there is one, else computed.
__device__ __forceinline__ double wco_of(const SimCtx& c, int m, int nbt) {
  if (c.b->wco_tab) return c.b->wco_tab[(size_t)m * c.b->wco_dim + nbt];
  const double o = nbt > 0 ? __ddiv_rn((double)m, (double)nbt) : 0.0;
  return __dmul_rn(c.L->mc.w_c, o);
}

// Request i's load, records and service start (control thread); wco: w_c *
// o_ij of the chosen worker.
__device__ __forceinline__ void book_request(SimCtx& c, const ReqState& q, int64_t i, double wco) {
  SimScalars& S = *c.S;
  const ModelConsts& mc = c.L->mc;
  const int js = S.jstar;
  const int f = c.freestk[--S.nfree];
  c.f_req[f] = (int32_t)i;
  c.f_worker[f] = js;
  c.f_blk[f] = (int32_t)q.blk;
  c.f_a[f] = q.a;
  c.f_o[f] = wco;
  c.f_oitl[f] = q.oitl;
  c.wA[js] += q.blk;
  S.in_flight++;
  const int64_t row = c.d->rec_base + i;
  c.b->rec.worker[row] = js;
  c.b->rec.arrival[row] = q.a;
  c.b->rec.nbt[row] = q.nbt;
  if (c.winserv[js] < mc.cap - 1) {
    start_service(c, f, js, q.a);
  } else {
    c.f_next[f] = -1;
    if (c.wqt[js] >= 0) c.f_next[c.wqt[js]] = f; else c.wqh[js] = f;
    c.wqt[js] = f;
  }
  S.prev_arrival = q.a;
  S.n_routed++;
}

// Lowest-index argmin across a warp: each lane holds the minimum of its own
// elements (cost c, index j; no element: +inf and INT_MAX); every lane ends
// with the (cost, index) that is least in (cost, then index) order.
__device__ __forceinline__ void argmin_warp(float& c, int& j) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float oc = __shfl_xor_sync(FULL_MASK, c, o);
    const int oj = __shfl_xor_sync(FULL_MASK, j, o);
    if (oc < c || (oc == c && oj < j)) {
      c = oc;
      j = oj;
    }
  }
}

__device__ __forceinline__ RawReq read_request(const SimCtx& c, int64_t i) {
  RawReq r;
  r.o0 = c.d->offsets[i];
  r.o1 = c.d->offsets[i + 1];
  r.rel = c.d->release[i];
  r.O = c.d->out_len[i];
  r.dup = c.d->dupflag[i] == 1;
  return r;
}

__device__ __forceinline__ void load_request(const SimCtx& c, ReqState& q, const RawReq& r) {
  const int64_t L = r.o1 - r.o0;
  q.off0 = r.o0;
  q.rel = r.rel;
  q.O = r.O;
  q.dup = r.dup;
  q.oitl = __dmul_rn((double)r.O, c.L->mc.itl);
  q.nb = (L >> 4) > 0x7FFFFFFF ? 0x7FFFFFFF : (int)(L >> 4);
  q.nbt = (int)((L + 15) >> 4);
  q.blk = (L + r.O + 15) >> 4;
  q.phase = 0;
  q.full = (int64_t)c.L->mc.W * (L >> 4) <= PROBE_CAP;
}

// Algorithm 1: the router parameters of the current regime (control thread).
// Called once request q's arrival is known and its events are done; with
// frequency eviction it also sets the decay step of that arrival.
template <bool FREQ>
__device__ __forceinline__ void regime_params(const SimCtx& c, ReqState& q) {
  if (FREQ && c.d->eviction == RS_EVICT_FREQ) {   // decay step of the arrival
    const double t = floor(__ddiv_rn(q.a, c.d->decay_s));
    c.S->dclock = t < 2147483648.0 ? (uint32_t)t : 2147483648u;
  }
  float tau = c.d->tau, om = c.d->omega;
  if (c.d->policy == RS_POLICY_LOADBAL) {
    tau = 0.0f;
    om = 0.0f;
  } else if (c.d->controller && c.S->regime > 0) {
    tau = c.L->mc.regime_tau[c.S->regime];
    om = c.L->mc.regime_omega[c.S->regime];
  }
  q.tau = tau;
  q.omega = om;
}

// Probe state of a request (lanes of the control warp).
__device__ __forceinline__ void probe_setup(SimCtx& c, const ReqState& q, int lane) {
  const int W = c.L->mc.W;
  for (int j = lane; j < W; j += 32) {
    c.wm[j] = q.nb;
    c.wabs[j] = 0;
  }
}

// Block hashes of a request into a staging buffer (lanes of one warp).
__device__ __forceinline__ void stage_hashes(const SimCtx& c, const ReqState& q, uint64_t* dst,
                                             int lane) {
  if (q.nb > (int)c.L->g.K) return;
  const uint64_t* src = c.d->hashes + (q.off0 >> 4);
  for (int k = lane; k < q.nb; k += 32) dst[k] = __ldg(src + k);
}

// MINB = CTAs the launch keeps resident per SM: 2 (128 registers) when there
// are more replicas than SMs, 1 (no register cap to speak of, no spills) when
// every replica has an SM to itself.
// SG: the per-request slot arrays are in global memory (a compile-time
// choice, so that in the common case the compiler knows they are shared).
template <int MINB, bool SG, int MODE>
__global__ void __launch_bounds__(NT_SIM, MINB) k_sim(const SimDesc* __restrict__ descs, SimBuffers b,
                                                SimLaunch L) {
  constexpr bool FREQ = MODE == SIM_FREQ, TIER = MODE == SIM_TIER;
  constexpr int PROBE_FULL_ILP = 2;   // lookups a thread of the full probe keeps in flight
  extern __shared__ __align__(16) unsigned char smem[];
  __shared__ SimScalars S;
  const int sid = blockIdx.x;
  const SimDesc d = descs[sid];
  const int W = L.mc.W;
  const ModelConsts& mc = L.mc;
  const int nft = ftab_size(mc.cap);
  const SimLayout lay = make_sim_layout(W, L.nbmax, L.cmax, nft, SG, TIER);
  // the slot arrays: shared memory, or this replica's global slot area
  unsigned char* slotbase;
  if constexpr (SG)
    slotbase = b.slotmem + (size_t)sid * make_sim_layout(1, 1, L.cmax, 1, true).slot_bytes;
  else
    slotbase = smem;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  SimCtx c;
  c.S = &S;
  c.d = &d;
  c.b = &b;
  c.L = &L;
  c.sid = sid;
  c.ftab = reinterpret_cast<double*>(smem + lay.ftab);
  c.f_oitl = reinterpret_cast<double*>(slotbase + lay.f_oitl);
  c.f_a = reinterpret_cast<double*>(slotbase + lay.f_a);
  c.f_o = reinterpret_cast<double*>(slotbase + lay.f_o);
  c.h_k = reinterpret_cast<uint64_t*>(slotbase + lay.h_k);
  c.hbuf0 = reinterpret_cast<uint64_t*>(smem + lay.hbuf0);
  c.hbuf1 = reinterpret_cast<uint64_t*>(smem + lay.hbuf1);
  c.f_req = reinterpret_cast<int32_t*>(slotbase + lay.f_req);
  c.f_worker = reinterpret_cast<int32_t*>(slotbase + lay.f_worker);
  c.f_blk = reinterpret_cast<int32_t*>(slotbase + lay.f_blk);
  c.f_next = reinterpret_cast<int32_t*>(slotbase + lay.f_next);
  c.h_f = reinterpret_cast<int32_t*>(slotbase + lay.h_f);
  c.freestk = reinterpret_cast<int32_t*>(slotbase + lay.freestk);
  c.wmeta = reinterpret_cast<CacheMeta*>(smem + lay.wmeta);
  c.wfreq = reinterpret_cast<FreqMeta*>(smem + lay.wfreq);
  c.wtier = reinterpret_cast<TierMeta*>(smem + lay.wtier);
  c.ptier = reinterpret_cast<uint8_t*>(smem + lay.ptier);
  c.winserv = reinterpret_cast<int32_t*>(smem + lay.winserv);
  c.wqh = reinterpret_cast<int32_t*>(smem + lay.wqh);
  c.wqt = reinterpret_cast<int32_t*>(smem + lay.wqt);
  c.wm = reinterpret_cast<int32_t*>(smem + lay.wm);
  c.wopen = reinterpret_cast<uint8_t*>(smem + lay.wopen);
  c.wabs = reinterpret_cast<int32_t*>(smem + lay.wabs);
  c.wA = reinterpret_cast<int64_t*>(smem + lay.wA);
  c.wcost = reinterpret_cast<float*>(smem + lay.wcost);
  c.sc.slot = reinterpret_cast<uint32_t*>(smem + lay.slot);
  c.sc.pst = reinterpret_cast<uint32_t*>(smem + lay.pst);
  c.sc.fslot = reinterpret_cast<uint32_t*>(smem + lay.fslot);
  c.pslot = reinterpret_cast<uint32_t*>(smem + lay.pslot);
  c.pfree = reinterpret_cast<uint32_t*>(smem + lay.pfree);
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
  c.pend_ft0 = pend;
  c.pend_tt0 = pend + b.pend_cap;
  c.pend_ft1 = pend + 2 * b.pend_cap;
  c.pend_tt1 = pend + 3 * b.pend_cap;
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
    for (int q = 1 + threadIdx.x; q < nft; q += NT_SIM) c.ftab[q] = latency_f(mc, q);
    // request slots: as many as the schedule ever holds in flight
    const int cslots = max(d.C, max(d.c_mid, d.c_end));
    for (int p = threadIdx.x; p < cslots; p += NT_SIM) c.freestk[p] = cslots - 1 - p;
    for (int j = threadIdx.x; j < W; j += NT_SIM) {
      c.wmeta[j] = CacheMeta{};
      c.wfreq[j] = FreqMeta{0u, 0u};
      if (TIER) c.wtier[j] = TierMeta{0u, 0u};
      c.winserv[j] = 0;
      c.wA[j] = 0;
      c.wqh[j] = -1;
      c.wqt[j] = -1;
    }
    if (threadIdx.x == 0) {
      memset(&S, 0, sizeof(SimScalars));
      S.min_ft = __longlong_as_double(0x7FF0000000000000ll);
      S.next_tick = 1;
      S.tick_t = mc.dt;
      S.nfree = max(d.C, max(d.c_mid, d.c_end));
      S.first_switch_t = -1.0;
      S.first_evict_i = -1;
      freq_reset(&S.fs);
    }
    __syncthreads();
  }

  const int64_t n = d.n_req;
  // ---- prologue: request 0's arrival and hashes
  if (n > 0) {
    if (threadIdx.x == CTL) {
      load_request(c, S.q[0], read_request(c, 0));
      if (n > 1) S.nraw = read_request(c, 1);
      S.evres = 0;
      update_reset(&S.us);
      S.us.err = 0;
    }
    __syncthreads();
    if (warp == NT_SIM / 32 - 1) {
      stage_hashes(c, S.q[0], c.hbuf0, lane);
      probe_setup(c, S.q[0], lane);
    }
  }
  for (int64_t i = 0; i < n; i++) {
    const int p = (int)(i & 1);
    __syncthreads();
    if (S.status != RS_OK) break;
    const int nb = S.q[p].nb;
    if (nb > (int)L.g.K) {
      if (threadIdx.x == 0) S.status = RS_ERR_CAPACITY;
      break;
    }
    const int nbt = S.q[p].nbt;
    const bool full = S.q[p].full;
    const uint64_t* hb = c.hbuf(p);
    const int64_t row = d.rec_base + i;
    if (warp < NT_SIM / 32 - 1) {
      // ---- cached prefix on every worker (warps 0-6)
      if (full) {
        probe_full<NT_UPD, PROBE_FULL_ILP, TIER>(c, hb, nb);
      } else if (TIER) {   // the tiers need every pair's slot (the host checks W nb)
        if (threadIdx.x == 0) S.status = RS_ERR_CAPACITY;
      } else {
        probe_prefixes<NT_UPD, MINB == 1 && MODE == SIM_LRU ? 4 : 1>(c, hb, nb);
      }
    } else if (lane == 0) {
      // ---- control thread, at the same time: completions and controller
      // samples up to request i's arrival (the probe needs none of them)
      S.evres = events_advance(c, S.q[p]);
      if (S.evres == 0) regime_params<FREQ>(c, S.q[p]);
    }
    __syncthreads();
    // ---- controller samples whose window needs the CTA (P99 of Eq. (10))
    while (S.evres != 0) {
      tick_cta(c);
      if (threadIdx.x == CTL) {
        S.evres = events_advance(c, S.q[p]);
        if (S.evres == 0) regime_params<FREQ>(c, S.q[p]);
      }
      __syncthreads();
    }
    if (S.status != RS_OK) break;
    // ---- Eq. (1) costs and the Eq. (2) choice, computed alike by every warp
    // (same inputs, same operations, so the same worker) so that the update
    // starts without a CTA barrier; the control warp records the decision
    const float om = S.q[p].omega, tau = S.q[p].tau;
    const bool eq2 = d.policy == RS_POLICY_DYNAMO || d.policy == RS_POLICY_LOADBAL;
    float* wc = c.wcost + (size_t)warp * W;   // this warp's cost row
    float bc = __int_as_float(0x7F800000);
    int bj = 0x7FFFFFFF;
    for (int j = lane; j < W; j += 32) {
      const float cj = router_cost(om, (int64_t)nbt - c.wm[j], c.wA[j]);
      wc[j] = cj;
      if (cj < bc || bj == 0x7FFFFFFF) {
        bc = cj;
        bj = j;
      }
    }
    argmin_warp(bc, bj);   // the lowest-index argmin (the choice at tau = 0)
    int js = bj;
    if (!eq2) {
      __syncwarp();
      int x = 0;
      if (lane == 0) x = static_policy_worker(d.policy, wc, W, d.seed, (uint64_t)i, 0u, TAG_SIM);
      js = __shfl_sync(FULL_MASK, x, 0);
    } else if (tau > 0.0f) {
      __syncwarp();
      uint32_t u24 = 0;
      if (lane == 0) u24 = draw_u24(d.seed, (uint64_t)i, 0u, TAG_SIM);
      u24 = __shfl_sync(FULL_MASK, u24, 0);
      // (the control warp also records where the draw fell)
      js = select_worker_warp(wc, W, tau, u24, bj,
                              warp == NT_SIM / 32 - 1 ? b.dstat + row * 6 + 2 : nullptr, lane);
    }
    if (warp < NT_SIM / 32 - 1) {
      // ---- the chosen worker's LRU cache (warps 0-6).  Its inputs are read
      // before the arrival that lets the control warp reset the probe state
      // and change the loads.
      const int nabs = c.wabs[js];   // absent blocks (victim count)
      // the chosen worker's table: rebuild first when its log span, its
      // tombstones or its stamps would overflow
      const CacheMeta* mt = &c.wmeta[js];
      const uint64_t span = (uint64_t)mt->T - mt->head + (uint64_t)nb;
      const bool rebuild =
          span > L.g.R || mt->tombs > L.g.slots / 8 || (uint64_t)mt->T + nb > STAMP_LIMIT;
      // two blocks of the prompt with one chained hash (a 64-bit collision,
      // flagged per request before the launch) would break the batched update
      const bool dup = S.q[p].dup != 0;
      asm volatile("bar.arrive 3, %0;" ::"n"(NT_SIM) : "memory");
      if (TIER) tier_charge<NT_UPD>(c, js, nb, row);
      update_chosen<MODE>(c, hb, js, nb, full, i, nabs, rebuild, dup);
    } else {
      asm volatile("bar.sync 3, %0;" ::"n"(NT_SIM) : "memory");   // the update group has read
      // records of the decision: frozen loads of Eq. (12), prefixes, costs;
      // the work done by the probe and the two lowest Eq. (1) costs, for the
      // near-tie statistic (counted after the run)
      int pb = 0;
      float c2 = __int_as_float(0x7F800000);
      for (int j = lane; j < W; j += 32) {
        const int m = c.wm[j];
        b.rec.n_frozen[row * W + j] = (uint16_t)min(c.winserv[j] + 1, mc.cap - 1);
        b.rec.prefix[row * W + j] = (uint16_t)m;
        if (mc.write_cost) b.rec.cost[row * W + j] = wc[j];
        pb += min(m + 1, nb);
        if (j != bj && wc[j] < c2) c2 = wc[j];
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const float x = __shfl_xor_sync(FULL_MASK, c2, o);
        if (x < c2) c2 = x;
      }
      pb = (int)__reduce_add_sync(FULL_MASK, (unsigned)pb);
      if (lane == 0) {
        float* ds = b.dstat + row * 6;
        ds[0] = bc;
        ds[1] = c2;
        if (eq2 && tau > 0.0f) S.sampled++;   // (ds[2..5] written with the draw)
        else ds[3] = -1.0f;                    // no Eq. (2) draw
        S.jstar = js;
        S.hit_blocks += c.wm[js];
        S.probe_blocks += pb;
        S.hashed_blocks += nb;
      }
      __syncwarp();
      // ---- control warp: request i's load and latency; request i+1's
      // scalars, probe state and block hashes
      ReqState& nq = S.q[p ^ 1];
      const bool more = i + 1 < n;
      // the chosen worker's w_c * o (a table load): issued first, used last
      const double wco = lane == 0 ? wco_of(c, c.wm[js], nbt) : 0.0;
      if (more) {
        // request i+1's hashes: asynchronous copies into the other staging
        // buffer, waited for before the next barrier
        const int64_t nbn = (S.nraw.o1 - S.nraw.o0) >> 4;
        if (nbn <= (int64_t)L.g.K) {
          const uint64_t* src = d.hashes + (S.nraw.o0 >> 4);
          uint64_t* dst = c.hbuf(p ^ 1);
          for (int k = lane; k < (int)nbn; k += 32) cp_async8(dst + k, src + k);
        }
        if (lane == 0) load_request(c, nq, S.nraw);
      }
      __syncwarp();
      if (more) probe_setup(c, nq, lane);
      if (lane == 0) {
        // the loads of the request after next go out first; their latency
        // overlaps the bookkeeping and the events
        RawReq raw2;
        const bool more2 = i + 2 < n;
        if (more2) raw2 = read_request(c, i + 2);
        book_request(c, S.q[p], i, wco);
        if (more2) S.nraw = raw2;
      }
      cp_async_wait_all();
      __syncwarp();   // every lane's copies of request i+1's hashes have landed
      if (MINB == 1 && more && nq.full && nq.nb <= (int)L.g.K) {
        // request i+1's home buckets on every worker, brought into L2 ahead
        // of its probe (the update running beside may still change the
        // chosen worker's; L2 holds the current data either way).  Only
        // with one replica per SM: with two, the other replica's warps fill
        // the probe's waits, and the prefetch instructions cost more than
        // they save (11% on the parameter grid)
        const uint64_t* hn = c.hbuf(p ^ 1);
        const int nbn = nq.nb;
        for (int e = lane; e < W * nbn; e += 32) {
          const int j = e / nbn;
          const TableView t = c.table(j);
          const uint32_t bk = home_bucket(hn[e - j * nbn], t.bmask);
          prefetch_l2(t.keys + (size_t)BUCKET * bk);
          prefetch_l2(t.keys + (size_t)BUCKET * bk + 4);
          if (TIER) prefetch_l2(t.stamp + (size_t)BUCKET * bk);
        }
      }
    }
  }
  __syncthreads();
  // ---- drain: remaining completions start the queued requests
  if (threadIdx.x == CTL && S.status == RS_OK) {
    while (S.nheap > 0) {
      uint64_t k;
      int f;
      heap_pop(c, &k, &f);
      complete(c, f, tval(k));
    }
  }
  __syncthreads();
  {
    double st = 0.0, se = 0.0, mk = 0.0;
    if (S.status == RS_OK)
      for (int64_t q = threadIdx.x; q < S.n_routed; q += NT_SIM) {
        const int64_t row = d.rec_base + q;
        const double ct = b.rec.completion[row];
        st = __dadd_rn(st, b.rec.ttft[row]);
        se = __dadd_rn(se, __dsub_rn(ct, b.rec.arrival[row]));
        mk = fmax(mk, ct);
      }
    for (int o = 16; o > 0; o >>= 1) {
      st = __dadd_rn(st, __shfl_xor_sync(FULL_MASK, st, o));
      se = __dadd_rn(se, __shfl_xor_sync(FULL_MASK, se, o));
      mk = fmax(mk, __shfl_xor_sync(FULL_MASK, mk, o));
    }
    __shared__ double red3[3][NT_SIM / 32];
    if (lane == 0) {
      red3[0][warp] = st;
      red3[1][warp] = se;
      red3[2][warp] = mk;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      double a0 = 0.0, a1 = 0.0, a2 = 0.0;
      for (int w = 0; w < NT_SIM / 32; w++) {
        a0 = __dadd_rn(a0, red3[0][w]);
        a1 = __dadd_rn(a1, red3[1][w]);
        a2 = fmax(a2, red3[2][w]);
      }
      S.sum_ttft = a0;
      S.sum_e2e = a1;
      S.makespan = a2;
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    rs_replica_result r;
    memset(&r, 0, sizeof r);
    r.status = S.status;
    r.final_regime = S.regime;
    r.n_routed = S.n_routed;
    r.sum_ttft = S.sum_ttft;
    r.sum_e2e = S.sum_e2e;
    r.makespan = S.makespan;
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
    r.first_switch_t = S.first_switch_t;
    // KV-cache pressure: resident blocks of every tier over W K_G1
    // (resident = inserted - evicted)
    const double cap = __dmul_rn((double)W, (double)L.k1);
    r.first_evict_t = -1.0;
    r.rho_first_evict = -1.0;
    if (S.first_evict_i >= 0) {
      r.first_evict_t = b.rec.arrival[d.rec_base + S.first_evict_i];
      r.rho_first_evict = __ddiv_rn((double)S.first_live, cap);
    }
    r.rho_end = __ddiv_rn((double)(S.inserted - S.evicted), cap);
    r.kv_g1 = S.kv[0];
    r.kv_g2 = S.kv[1];
    r.kv_g3 = S.kv[2];
    r.kv_remote = S.kv[3];
    r.kv_recompute = S.kv[4];
    r.kv_cost = S.kv_cost;
    b.res[sid] = r;
  }
  for (int j = threadIdx.x; j < W; j += NT_SIM) b.meta_out[(size_t)sid * W + j] = c.wmeta[j];
}

// w_c * (m / nbt) for every cached-prefix length m <= nbmax and prompt
// length nbt <= nbmax + 1 blocks, rounded as the latency of Eq. (9) uses it.
__global__ void k_wco_table(double* tab, int nbmax, double w_c) {
  const int dim = nbmax + 2;
  const int64_t total = (int64_t)(nbmax + 1) * dim;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < total;
       e += (int64_t)gridDim.x * blockDim.x) {
    const int m = (int)(e / dim), nbt = (int)(e % dim);
    const double o = nbt > 0 ? __ddiv_rn((double)m, (double)nbt) : 0.0;
    tab[e] = __dmul_rn(w_c, o);
  }
}

cudaError_t launch_wco_table(double* tab, int nbmax, double w_c, cudaStream_t st) {
  k_wco_table<<<152 * 4, 256, 0, st>>>(tab, nbmax, w_c);
  return cudaGetLastError();
}

// Decision statistics of every replica from the per-request records of the
// simulation: top-two Eq. (1) costs within 1e-6 relative (and equal), and
// Eq. (2) draws within 1e-6 S of a cumulative-weight boundary.
__global__ void __launch_bounds__(256) k_decision_stats(const SimDesc* __restrict__ descs,
                                                        SimBuffers b, SimLaunch L) {
  const SimDesc d = descs[blockIdx.x];
  const int64_t n = b.res[blockIdx.x].n_routed;
  long long near = 0, exact = 0, bd = 0;
  for (int64_t q = threadIdx.x; q < n; q += blockDim.x) {
    const float* ds = b.dstat + (d.rec_base + q) * 6;
    if (L.mc.W >= 2) {
      const float c1 = ds[0], c2 = ds[1];
      const double diff = (double)c2 - (double)c1;
      if (diff <= 1e-6 * fabs((double)c2)) near++;
      if (c2 == c1) exact++;
    }
    if (ds[3] >= 0.0f) {
      const double tg = (double)ds[2], S = (double)ds[3], eps = 1e-6 * S;
      const float lo = ds[4], hi = ds[5];
      if ((lo == lo && fabs(tg - (double)lo) <= eps) || (hi == hi && fabs(tg - (double)hi) <= eps))
        bd++;
    }
  }
  for (int o = 16; o > 0; o >>= 1) {
    near += __shfl_xor_sync(FULL_MASK, near, o);
    exact += __shfl_xor_sync(FULL_MASK, exact, o);
    bd += __shfl_xor_sync(FULL_MASK, bd, o);
  }
  __shared__ long long red[3][8];
  if ((threadIdx.x & 31) == 0) {
    red[0][threadIdx.x >> 5] = near;
    red[1][threadIdx.x >> 5] = exact;
    red[2][threadIdx.x >> 5] = bd;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    long long a = 0, e = 0, z = 0;
    for (int w = 0; w < (int)(blockDim.x >> 5); w++) {
      a += red[0][w];
      e += red[1][w];
      z += red[2][w];
    }
    b.res[blockIdx.x].near_ties = a;
    b.res[blockIdx.x].exact_ties = e;
    b.res[blockIdx.x].near_boundary = z;
  }
}

cudaError_t launch_decision_stats(const SimDesc* d_desc, const SimBuffers& b, const SimLaunch& L,
                                  cudaStream_t st) {
  if (L.nsim <= 0) return cudaSuccess;
  k_decision_stats<<<L.nsim, 256, 0, st>>>(d_desc, b, L);
  return cudaGetLastError();
}

cudaError_t launch_sim(const SimDesc* d_desc, const SimBuffers& b, const SimLaunch& L,
                       cudaStream_t st) {
  if (L.nsim <= 0) return cudaSuccess;
  const size_t smem = sim_smem_bytes(L.mc.W, L.nbmax, L.cmax, L.mc.cap, L.slots_global != 0,
                                    L.tiered != 0);
  int dev = 0, sms = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  // one replica per SM: the kernel may use every register
  const bool one = L.nsim <= sms;
  // Game 2 tiers, or frequency eviction state present: the kernel with that
  // variant; else the LRU-only kernel
  void (*kern)(const SimDesc*, SimBuffers, SimLaunch);
  if (L.tiered)
    kern = one ? (L.slots_global ? k_sim<1, true, SIM_TIER> : k_sim<1, false, SIM_TIER>)
               : (L.slots_global ? k_sim<2, true, SIM_TIER> : k_sim<2, false, SIM_TIER>);
  else if (b.fexp)
    kern = one ? (L.slots_global ? k_sim<1, true, SIM_FREQ> : k_sim<1, false, SIM_FREQ>)
               : (L.slots_global ? k_sim<2, true, SIM_FREQ> : k_sim<2, false, SIM_FREQ>);
  else
    kern = one ? (L.slots_global ? k_sim<1, true, SIM_LRU> : k_sim<1, false, SIM_LRU>)
               : (L.slots_global ? k_sim<2, true, SIM_LRU> : k_sim<2, false, SIM_LRU>);
  e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  kern<<<L.nsim, NT_SIM, smem, st>>>(d_desc, b, L);
  return cudaGetLastError();
}

}  // namespace rs
