/*
 * CPU oracle for the KV-cache-aware routing simulation -- TEST INFRASTRUCTURE.
 * Only tests, the smoke check and the benchmark's CPU-baseline leg use it.
 *
 * Written to be read against the paper, not to be fast: one replica at a time,
 * one request at a time, textbook data structures (chained hash map + doubly
 * linked LRU list, binary heap, Hungarian algorithm, successive shortest
 * paths).  Compile with -ffp-contract=off so that every floating-point
 * operation is rounded on its own, in the order written.
 *
 * Readings fixed where the paper is silent (each also listed in the design
 * notes of the repository):
 *  - KV blocks hold `block` tokens; only full blocks are hashed and cached.
 *  - Block hash: content g_k = the block's 64-bit little-endian token pairs
 *    folded by one multiply-xorshift each from 0x9E3779B97F4A7C15 ^ block,
 *    then the SplitMix64 finalizer; prefix H_k = H_{k-1} P + g_k mod 2^64 with
 *    H_{-1} = seed, P = 0x94D049BB133111EB; stored h_k = mix(H_k ^ k); values 0
 *    and 1 are reserved and mapped to 2 and 3.
 *  - b^prefill of Eq. (1) = ceil(L/block) - m_ij, with m_ij the number of
 *    leading blocks found in worker j's cache (first-miss prefix); the overlap
 *    o_ij of Eq. (7) is m_ij / ceil(L/block).
 *  - b^active of Eq. (1) = sum over requests routed to j and not finished
 *    (queued or in service) of ceil((L + O)/block).
 *  - Eviction: exact LRU; the chosen worker touches every full block of the
 *    prompt in order (hits move to most-recent, misses are inserted, evicting
 *    the least-recent entry when full).
 *  - Frequency eviction (the KV Block Manager of §2.2, the alternative): every
 *    block carries a frequency, 1 when inserted, doubled on a hit (at most
 *    freq_max) and lowered by 1 per decay step (never below 1); decay step
 *    floor(a_i / decay_s) at request i's arrival.  Frequency 1 is cold, 2 and
 *    more (eligible for promotion) hot.  The victim is the least recently used
 *    cold block, or the least recently used block when every block is hot.
 *  - Ties of the argmin go to the lowest worker index.  Temperature sampling
 *    uses Philox4x32-10 and a 24-bit uniform.
 *  - Service: a worker serves at most cap-1 = 63 requests at once (the pole of
 *    Eq. (9) at n = cap is never reached); extra requests wait FIFO.  TTFT =
 *    wait + f(n) - w_c * o with n the in-service count including the request.
 */
#include "routesim_oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>

/* ------------------------------------------------------------------------ */
/* Block hashing                                                             */
/* ------------------------------------------------------------------------ */

/* SplitMix64 output finalizer (Steele, Lea, Flood, OOPSLA 2014). */
uint64_t orc_mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}

/* Content of one block: its little-endian 64-bit token pairs folded in
 * order, one multiply-xorshift each (x = (x ^ w) M, then x ^= x >> 32; M
 * odd, so each step is a bijection of x and of w), then the SplitMix64
 * finalizer. */
static uint64_t block_content(const int32_t* t, int32_t block) {
  uint64_t x = 0x9E3779B97F4A7C15ULL ^ (uint64_t)block;
  for (int32_t q = 0; q < block / 2; q++) {
    uint64_t w = (uint64_t)(uint32_t)t[2 * q] | ((uint64_t)(uint32_t)t[2 * q + 1] << 32);
    x = (x ^ w) * 0xBF58476D1CE4E5B9ULL;
    x ^= x >> 32;
  }
  return orc_mix64(x);
}

/* Prefix hash of blocks 0..k (Horner): H_{-1} = seed, H_k = H_{k-1} P + g_k
 * (mod 2^64, P odd); the stored hash is mix(H_k ^ k), with the values 0 and 1
 * (the table's empty and tombstone keys) mapped to 2 and 3. */
#define PREFIX_P 0x94D049BB133111EBULL

static void hash_request(const int32_t* t, int64_t nb, int32_t block, uint64_t seed,
                         uint64_t* out) {
  uint64_t H = seed;
  for (int64_t k = 0; k < nb; k++) {
    H = H * PREFIX_P + block_content(t + k * block, block);
    uint64_t h = orc_mix64(H ^ (uint64_t)k);
    if (h < 2) h += 2;
    out[k] = h;
  }
}

void orc_hash_blocks(const int32_t* tokens, const int64_t* offsets, int64_t n_req,
                     int32_t block, uint64_t seed, uint64_t* out) {
  for (int64_t i = 0; i < n_req; i++) {
    int64_t L = offsets[i + 1] - offsets[i];
    hash_request(tokens + offsets[i], L / block, block, seed, out + offsets[i] / block);
  }
}

/* ------------------------------------------------------------------------ */
/* Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC 2011)                       */
/* ------------------------------------------------------------------------ */

void orc_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]) {
  uint32_t c0 = ctr[0], c1 = ctr[1], c2 = ctr[2], c3 = ctr[3];
  uint32_t k0 = key[0], k1 = key[1];
  for (int r = 0; r < 10; r++) {
    if (r > 0) {
      k0 += 0x9E3779B9u;
      k1 += 0xBB67AE85u;
    }
    uint64_t p0 = (uint64_t)0xD2511F53u * (uint64_t)c0;
    uint64_t p1 = (uint64_t)0xCD9E8D57u * (uint64_t)c2;
    uint32_t n0 = (uint32_t)(p1 >> 32) ^ c1 ^ k0;
    uint32_t n1 = (uint32_t)p1;
    uint32_t n2 = (uint32_t)(p0 >> 32) ^ c3 ^ k1;
    uint32_t n3 = (uint32_t)p0;
    c0 = n0; c1 = n1; c2 = n2; c3 = n3;
  }
  out[0] = c0; out[1] = c1; out[2] = c2; out[3] = c3;
}

#define TICK_LIMIT (1ll << 24)   /* controller samples per replica */
#define TAG_SIM 0x53494D31u    /* sampling stream of the simulation */
#define TAG_ROUTE 0x52545231u  /* sampling stream of the live router */

static uint32_t draw_u24(uint64_t seed, uint64_t ordinal, uint32_t stream, uint32_t tag) {
  uint32_t ctr[4] = {(uint32_t)ordinal, (uint32_t)(ordinal >> 32), stream, tag};
  uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
  uint32_t out[4];
  orc_philox4x32_10(ctr, key, out);
  return out[0] >> 8;
}

/* ------------------------------------------------------------------------ */
/* exp for the softmax of Eq. (2)                                            */
/* ------------------------------------------------------------------------ */

/* Cody-Waite: x = k ln2 + r with ln2 split in a high part (8 trailing zero
 * bits) and a low part, |r| <= ln2/2; exp(r) by its degree-7 Taylor polynomial
 * in Horner form with fused multiply-adds; scale by 2^k through the exponent
 * field.  Inputs below -87 return 0 (the result would be subnormal). */
float orc_expf(float x) {
  if (!(x >= -87.0f)) return 0.0f;
  if (x > 88.0f) return INFINITY;
  float t = x * 0x1.715476p+0f;
  float kf = nearbyintf(t);
  float r = fmaf(-kf, 0x1.62e4p-1f, x);
  r = fmaf(-kf, 0x1.7f7d1cp-20f, r);
  float p = 0x1.a01a02p-13f;
  p = fmaf(p, r, 0x1.6c16c2p-10f);
  p = fmaf(p, r, 0x1.111112p-7f);
  p = fmaf(p, r, 0x1.555556p-5f);
  p = fmaf(p, r, 0x1.555556p-3f);
  p = fmaf(p, r, 0.5f);
  p = fmaf(p, r, 1.0f);
  p = fmaf(p, r, 1.0f);
  int32_t k = (int32_t)kf;
  uint32_t bits = (uint32_t)(k + 127) << 23;
  float s;
  memcpy(&s, &bits, sizeof s);
  return p * s;
}

void orc_expf_n(const float* x, float* y, int64_t n) {
  for (int64_t i = 0; i < n; i++) y[i] = orc_expf(x[i]);
}

/* ------------------------------------------------------------------------ */
/* Worker selection, Eq. (2)                                                 */
/* ------------------------------------------------------------------------ */

static int32_t argmin_lowest(const float* c, int32_t W) {
  int32_t best = 0;
  for (int32_t j = 1; j < W; j++)
    if (c[j] < c[best]) best = j;
  return best;
}

int32_t orc_select(const float* c, int32_t W, float tau, uint32_t u24) {
  int32_t best = argmin_lowest(c, W);
  if (tau == 0.0f) return best;
  float cmin = c[best];
  float S = 0.0f;
  for (int32_t j = 0; j < W; j++) {
    float x = (c[j] - cmin) / tau;
    S = S + orc_expf(-x);
  }
  float u = (float)u24 * 0x1p-24f;
  float target = u * S;
  float cum = 0.0f;
  int32_t last = best;
  for (int32_t j = 0; j < W; j++) {
    float x = (c[j] - cmin) / tau;
    float e = orc_expf(-x);
    cum = cum + e;
    if (e > 0.0f) last = j;
    if (target < cum) return j;
  }
  return last;
}

/* near-boundary: the scaled draw lies within 1e-6 S of a cumulative boundary */
static int near_boundary(const float* c, int32_t W, float tau, uint32_t u24) {
  int32_t best = argmin_lowest(c, W);
  float cmin = c[best];
  float S = 0.0f;
  for (int32_t j = 0; j < W; j++) S = S + orc_expf(-((c[j] - cmin) / tau));
  float target = ((float)u24 * 0x1p-24f) * S;
  float cum = 0.0f;
  for (int32_t j = 0; j < W; j++) {
    cum = cum + orc_expf(-((c[j] - cmin) / tau));
    if (fabs((double)target - (double)cum) <= 1e-6 * (double)S) return 1;
  }
  return 0;
}

/* ------------------------------------------------------------------------ */
/* Exact LRU cache: chained hash map over a node pool + doubly linked list   */
/* ------------------------------------------------------------------------ */

typedef struct {
  int64_t K, size, head /* least recent */, tail /* most recent */, nfree;
  uint64_t* key;
  int64_t *prev, *next, *chain, *freel, *bucket;
  int64_t* freq;        /* frequency of each node (frequency eviction) */
  uint64_t mask;
} lru_t;

static int lru_init(lru_t* c, int64_t K) {
  memset(c, 0, sizeof *c);
  c->K = K;
  uint64_t nb = 1;
  while (nb < (uint64_t)(2 * K)) nb <<= 1;
  c->mask = nb - 1;
  c->key = (uint64_t*)malloc(sizeof(uint64_t) * K);
  c->prev = (int64_t*)malloc(sizeof(int64_t) * K);
  c->next = (int64_t*)malloc(sizeof(int64_t) * K);
  c->chain = (int64_t*)malloc(sizeof(int64_t) * K);
  c->freel = (int64_t*)malloc(sizeof(int64_t) * K);
  c->bucket = (int64_t*)malloc(sizeof(int64_t) * nb);
  c->freq = (int64_t*)malloc(sizeof(int64_t) * K);
  if (!c->key || !c->prev || !c->next || !c->chain || !c->freel || !c->bucket || !c->freq)
    return -1;
  for (uint64_t b = 0; b < nb; b++) c->bucket[b] = -1;
  for (int64_t n = 0; n < K; n++) c->freel[n] = K - 1 - n;
  c->nfree = K;
  c->head = c->tail = -1;
  return 0;
}

static void lru_free(lru_t* c) {
  free(c->key); free(c->prev); free(c->next); free(c->chain); free(c->freel); free(c->bucket);
  free(c->freq);
}

static int64_t lru_find(const lru_t* c, uint64_t key) {
  for (int64_t n = c->bucket[key & c->mask]; n >= 0; n = c->chain[n])
    if (c->key[n] == key) return n;
  return -1;
}

static void list_unlink(lru_t* c, int64_t n) {
  if (c->prev[n] >= 0) c->next[c->prev[n]] = c->next[n]; else c->head = c->next[n];
  if (c->next[n] >= 0) c->prev[c->next[n]] = c->prev[n]; else c->tail = c->prev[n];
}

static void list_push_recent(lru_t* c, int64_t n) {
  c->prev[n] = c->tail;
  c->next[n] = -1;
  if (c->tail >= 0) c->next[c->tail] = n; else c->head = n;
  c->tail = n;
}

static void lru_touch(lru_t* c, int64_t n) {
  list_unlink(c, n);
  list_push_recent(c, n);
}

/* frequency eviction: `steps` decay steps lower every frequency by 1 each,
 * never below 1 */
static void freq_decay(lru_t* c, int64_t steps) {
  for (int64_t n = c->head; n >= 0; n = c->next[n])
    c->freq[n] = c->freq[n] - steps > 1 ? c->freq[n] - steps : 1;
}

/* frequency eviction's victim: the least recently used block of frequency 1
 * (cold); when every block is hot, the least recently used block */
static int64_t freq_victim(const lru_t* c) {
  for (int64_t n = c->head; n >= 0; n = c->next[n])
    if (c->freq[n] < 2) return n;
  return c->head;
}

/* insert an absent key as most recent (frequency 1); when the cache is full
 * the LRU entry (mode LRU) or the frequency rule's victim (mode FREQ) goes
 * first.  Returns 1 if an entry was evicted. */
static int lru_insert(lru_t* c, uint64_t key, int32_t mode, uint64_t* victim_key) {
  int evicted = 0;
  if (c->size == c->K) {
    int64_t v = mode == ORC_EVICT_FREQ ? freq_victim(c) : c->head;
    if (victim_key) *victim_key = c->key[v];
    list_unlink(c, v);
    int64_t* link = &c->bucket[c->key[v] & c->mask];
    while (*link != v) link = &c->chain[*link];
    *link = c->chain[v];
    c->freel[c->nfree++] = v;
    c->size--;
    evicted = 1;
  }
  int64_t n = c->freel[--c->nfree];
  c->key[n] = key;
  c->freq[n] = 1;
  c->chain[n] = c->bucket[key & c->mask];
  c->bucket[key & c->mask] = n;
  list_push_recent(c, n);
  c->size++;
  return evicted;
}

/* removes node n (a present key) */
static void lru_remove(lru_t* c, int64_t n) {
  list_unlink(c, n);
  int64_t* link = &c->bucket[c->key[n] & c->mask];
  while (*link != n) link = &c->chain[*link];
  *link = c->chain[n];
  c->freel[c->nfree++] = n;
  c->size--;
}

/* keys from least to most recent */
static int64_t lru_dump(const lru_t* c, uint64_t* out) {
  int64_t i = 0;
  for (int64_t n = c->head; n >= 0; n = c->next[n]) out[i++] = c->key[n];
  return i;
}

static int cmp_u64(const void* a, const void* b) {
  uint64_t x = *(const uint64_t*)a, y = *(const uint64_t*)b;
  return x < y ? -1 : x > y;
}

static int has_duplicate(const uint64_t* h, int64_t nb, uint64_t* scratch) {
  memcpy(scratch, h, sizeof(uint64_t) * nb);
  qsort(scratch, nb, sizeof(uint64_t), cmp_u64);
  for (int64_t k = 1; k < nb; k++)
    if (scratch[k] == scratch[k - 1]) return 1;
  return 0;
}

/* m_ij: leading blocks found in the cache (first-miss prefix length) */
static int64_t cached_prefix(const lru_t* c, const uint64_t* h, int64_t nb) {
  int64_t m = 0;
  while (m < nb && lru_find(c, h[m]) >= 0) m++;
  return m;
}

/* the chosen worker touches the prompt's blocks in order; under frequency
 * eviction a hit doubles the block's frequency, up to freq_max */
static void cache_update(lru_t* c, const uint64_t* h, int64_t nb, int64_t* inserted,
                         int64_t* evicted, int32_t mode, int64_t freq_max) {
  for (int64_t k = 0; k < nb; k++) {
    int64_t n = lru_find(c, h[k]);
    if (n >= 0) {
      lru_touch(c, n);
      if (mode == ORC_EVICT_FREQ) c->freq[n] = 2 * c->freq[n] < freq_max ? 2 * c->freq[n] : freq_max;
    } else {
      *evicted += lru_insert(c, h[k], mode, NULL);
      *inserted += 1;
    }
  }
}

/* ------------------------------------------------------------------------ */
/* Game 2 tiers (§4.2): exclusive G1, G2, G3 caches per worker               */
/* ------------------------------------------------------------------------ */

/* key enters tier t (0 = G1) as most recent; a full tier passes its least
 * recent block down to the next tier, the last tier drops it.  Counts the
 * blocks that left G1 and the blocks dropped. */
static void tier_push(lru_t* const* tier, int32_t ntier, int32_t t, uint64_t key,
                      int64_t* left_g1, int64_t* dropped) {
  uint64_t k = key;
  for (; t < ntier; t++) {
    uint64_t v;
    if (!lru_insert(tier[t], k, ORC_EVICT_LRU, &v)) return;
    if (t == 0) (*left_g1)++;
    k = v;
  }
  (*dropped)++;
}

/* the chosen worker accesses the prompt's blocks in order: a block in G1 is
 * touched; a block in a lower tier moves to G1; an absent block is inserted
 * into G1 */
static void tier_update(lru_t* const* tier, int32_t ntier, const uint64_t* h, int64_t nb,
                        int64_t* inserted, int64_t* left_g1, int64_t* dropped) {
  for (int64_t k = 0; k < nb; k++) {
    int64_t n = lru_find(tier[0], h[k]);
    if (n >= 0) {
      lru_touch(tier[0], n);
      continue;
    }
    int found = 0;
    for (int32_t t = 1; t < ntier && !found; t++) {
      n = lru_find(tier[t], h[k]);
      if (n >= 0) {
        lru_remove(tier[t], n);
        found = 1;
      }
    }
    if (!found) *inserted += 1;
    tier_push(tier, ntier, 0, h[k], left_g1, dropped);
  }
}

/* tier (1, 2, 3) of key on a worker, 0 if absent; tid maps list index to tier */
static int32_t tier_of(lru_t* const* tier, const int32_t* tid, int32_t ntier, uint64_t key) {
  for (int32_t t = 0; t < ntier; t++)
    if (lru_find(tier[t], key) >= 0) return tid[t];
  return 0;
}

/* ------------------------------------------------------------------------ */
/* Latency model, Eq. (9) with beta = 2, constants of §6.4                   */
/* ------------------------------------------------------------------------ */

static double latency_f(const orc_config* cfg, int64_t n) {
  double t1 = cfg->lat_a * (double)n;
  double t2 = t1 + cfg->lat_b;
  double den = (double)(cfg->cap - n);
  double den2 = den * den;
  double t3 = cfg->lat_d / den2;
  return t2 + t3;
}

/* frozen cost c_ij of the §6.4 matrix */
static double frozen_cost(const orc_config* cfg, int64_t nfz, int64_t m, int64_t nbt) {
  double f = latency_f(cfg, nfz);
  double o = nbt > 0 ? (double)m / (double)nbt : 0.0;
  double t4 = cfg->w_c * o;
  return f - t4;
}

/* ------------------------------------------------------------------------ */
/* Completion heap ordered by (time, request index)                          */
/* ------------------------------------------------------------------------ */

typedef struct { double t; int64_t q; } cev;

static int cev_less(cev a, cev b) { return a.t < b.t || (a.t == b.t && a.q < b.q); }

static void heap_push(cev* h, int64_t* n, cev e) {
  int64_t i = (*n)++;
  h[i] = e;
  while (i > 0) {
    int64_t p = (i - 1) / 2;
    if (!cev_less(h[i], h[p])) break;
    cev t = h[i]; h[i] = h[p]; h[p] = t;
    i = p;
  }
}

static cev heap_pop(cev* h, int64_t* n) {
  cev top = h[0];
  h[0] = h[--(*n)];
  int64_t i = 0;
  for (;;) {
    int64_t l = 2 * i + 1, r = l + 1, s = i;
    if (l < *n && cev_less(h[l], h[s])) s = l;
    if (r < *n && cev_less(h[r], h[s])) s = r;
    if (s == i) break;
    cev t = h[i]; h[i] = h[s]; h[s] = t;
    i = s;
  }
  return top;
}

static int cmp_double(const void* a, const void* b) {
  double x = *(const double*)a, y = *(const double*)b;
  return x < y ? -1 : x > y;
}

/* ------------------------------------------------------------------------ */
/* The replica simulation                                                    */
/* ------------------------------------------------------------------------ */

typedef struct {
  int32_t regime, up_cnt, down_cnt, have_L, have_ewma;
  double lastL, ewma;
  int64_t switches;
} ctl_t;

typedef struct {
  const orc_config* cfg;
  const orc_replica* rep;
  const int32_t* tokens;
  const int64_t* offsets;
  const double* release;
  const int32_t* out_len;
  int32_t W;
  /* per request */
  int32_t* worker; double *arrival, *start, *first, *compl_t, *ttft, *o;
  int32_t* nbt; int64_t* blk; int64_t* qnext;
  uint16_t *n_frozen, *prefix; float* cost;
  /* per worker */
  lru_t* cache; int64_t *inservice, *A, *qhead, *qtail;
  lru_t *g2, *g3;      /* Game 2 tiers below G1 (tiered), else NULL */
  double* kv_cost;     /* per request, or NULL */
  /* events */
  cev* heap; int64_t nheap; int64_t in_flight;
  /* controller */
  ctl_t ctl;
  int64_t next_tick;
  int64_t* pending; int64_t npending;
  int32_t err;
  double* window;
  double* tick_ewma; int32_t* tick_regime; int64_t max_ticks;
  orc_summary* sum;
} sim_t;

static void start_service(sim_t* s, int64_t q, int32_t j, double t) {
  const orc_config* cfg = s->cfg;
  s->inservice[j]++;
  double f = latency_f(cfg, s->inservice[j]);
  double t4 = cfg->w_c * s->o[q];
  double svc = f - t4;
  double ft = t + svc;
  double tt = ft - s->arrival[q];
  double ct = ft + (double)s->out_len[q] * cfg->itl;
  s->start[q] = t;
  s->first[q] = ft;
  s->ttft[q] = tt;
  s->compl_t[q] = ct;
  cev e = {ct, q};
  heap_push(s->heap, &s->nheap, e);
  if (s->rep->controller) s->pending[s->npending++] = q;
  s->sum->sum_ttft += tt;
  s->sum->sum_e2e += ct - s->arrival[q];
}

static void complete(sim_t* s, int64_t q, double t) {
  int32_t j = s->worker[q];
  s->inservice[j]--;
  s->A[j] -= s->blk[q];
  s->in_flight--;
  if (t > s->sum->makespan) s->sum->makespan = t;
  if (s->qhead[j] >= 0) {
    int64_t q2 = s->qhead[j];
    s->qhead[j] = s->qnext[q2];
    if (s->qhead[j] < 0) s->qtail[j] = -1;
    start_service(s, q2, j, t);
  }
}

/* nearest-rank 99th percentile of v[0..n) (sorts v in place) */
static double p99_nearest_rank(double* v, int64_t n) {
  qsort(v, n, sizeof(double), cmp_double);
  return v[(99 * n + 99) / 100 - 1];
}

double orc_p99(const double* v, int64_t n) {
  if (n <= 0) return NAN;
  double* w = (double*)malloc(sizeof(double) * n);
  memcpy(w, v, sizeof(double) * n);
  double r = p99_nearest_rank(w, n);
  free(w);
  return r;
}

/* Saturation test of the PoA-growth proposition (§5.1, item 3) over load
 * sweeps, as Experiment 2 measures it: per replica, the nearest-rank pct-th
 * percentile of its routed TTFTs (sorted ascending, element ceil(pct n / 100)
 * - 1, NaN without routed requests); per sweep of replicas in increasing load,
 * the difference quotient between neighbours and the three-point second
 * divided difference at interior points; the knee is the first interior point
 * whose second difference exceeds theta.  Sweep s holds replicas
 * sweep_start[s] .. sweep_start[s+1] - 1.  Outputs for replicas outside every
 * sweep, at sweep ends, and in sweeps whose loads do not increase strictly
 * stay NaN; such a sweep reports knee index -2 and load NaN, a sweep without a
 * knee -1 and -1. */
int32_t orc_sweep_knee(int32_t n_rep, const int64_t* row_start, const int32_t* worker,
                       const double* ttft, const double* load, int32_t n_sweeps,
                       const int32_t* sweep_start, int32_t pct, double theta, double* stat,
                       double* d1, double* d2, double* knee_load, int32_t* knee_index) {
  if (pct < 1 || pct > 100 || n_rep < 0 || n_sweeps < 0) return ORC_ERR_INVALID;
  for (int32_t r = 0; r < n_rep; r++) {
    const int64_t a = row_start[r], b = row_start[r + 1];
    int64_t n = 0;
    for (int64_t i = a; i < b; i++) n += worker[i] >= 0;
    d1[r] = NAN;
    d2[r] = NAN;
    if (n == 0) {
      stat[r] = NAN;
      continue;
    }
    double* v = (double*)malloc(sizeof(double) * (size_t)n);
    if (!v) return ORC_ERR_OOM;
    int64_t m = 0;
    for (int64_t i = a; i < b; i++)
      if (worker[i] >= 0) v[m++] = ttft[i];
    qsort(v, (size_t)n, sizeof(double), cmp_double);
    stat[r] = v[((int64_t)pct * n + 99) / 100 - 1];
    free(v);
  }
  for (int32_t s = 0; s < n_sweeps; s++) {
    const int32_t a = sweep_start[s], b = sweep_start[s + 1];
    int inc = 1;
    for (int32_t r = a + 1; r < b; r++)
      if (!(load[r] > load[r - 1])) inc = 0;
    if (!inc) {
      knee_load[s] = NAN;
      knee_index[s] = -2;
      continue;
    }
    for (int32_t r = a; r + 1 < b; r++)
      d1[r] = (stat[r + 1] - stat[r]) / (load[r + 1] - load[r]);
    knee_load[s] = -1.0;
    knee_index[s] = -1;
    for (int32_t r = a + 1; r + 1 < b; r++) {
      d2[r] = 2.0 * (d1[r] - d1[r - 1]) / (load[r + 1] - load[r - 1]);
      if (knee_index[s] < 0 && d2[r] > theta) {
        knee_index[s] = r;
        knee_load[s] = load[r];
      }
    }
  }
  return ORC_OK;
}

/* Controller state update for one sample: EWMA of Eq. (10), then the
 * three-regime classifier of Eq. (11) with k-sample hysteresis (§6.2).
 * has_window = 0 means the window held no TTFT: the previous P99 is reused. */
static void ctl_sample(ctl_t* c, const orc_config* cfg, int has_window, double Lw) {
  double L = 0.0;
  if (has_window) {
    L = Lw;
    c->have_L = 1;
    c->lastL = L;
  } else if (c->have_L) {
    L = c->lastL;
  } else {
    return;   /* nothing observed yet */
  }
  if (!c->have_ewma) {
    c->ewma = L;
    c->have_ewma = 1;
  } else {
    double t1 = cfg->alpha * L;
    double t2 = (1.0 - cfg->alpha) * c->ewma;
    c->ewma = t1 + t2;
  }
  int up_ok = 0, down_ok = 0;
  if (c->regime == 0) up_ok = c->ewma >= cfg->theta1;
  if (c->regime == 1) {
    up_ok = c->ewma >= cfg->theta2;
    down_ok = c->ewma < cfg->theta1 - cfg->eps_frac * cfg->theta1;
  }
  if (c->regime == 2) down_ok = c->ewma < cfg->theta2 - cfg->eps_frac * cfg->theta2;
  c->up_cnt = up_ok ? c->up_cnt + 1 : 0;
  c->down_cnt = down_ok ? c->down_cnt + 1 : 0;
  if (c->up_cnt >= cfg->hyst_k) {
    c->regime++;
    c->up_cnt = c->down_cnt = 0;
    c->switches++;
  } else if (c->down_cnt >= cfg->hyst_k) {
    c->regime--;
    c->up_cnt = c->down_cnt = 0;
    c->switches++;
  }
}

int32_t orc_controller_run(const orc_config* cfg, int64_t n, const double* L, double* ewma,
                           int32_t* regime) {
  ctl_t c;
  memset(&c, 0, sizeof c);
  for (int64_t i = 0; i < n; i++) {
    ctl_sample(&c, cfg, !isnan(L[i]), L[i]);
    ewma[i] = c.have_ewma ? c.ewma : -1.0;
    regime[i] = c.regime;
  }
  return ORC_OK;
}

/* one controller sample at t = k * Delta: the window holds the TTFTs of
 * requests whose first token came in [(k-1) Delta, k Delta) */
static void controller_tick(sim_t* s) {
  const orc_config* cfg = s->cfg;
  double tt = (double)s->next_tick * cfg->dt;
  int64_t nw = 0, keep = 0;
  for (int64_t p = 0; p < s->npending; p++) {
    int64_t q = s->pending[p];
    if (s->first[q] < tt) s->window[nw++] = s->ttft[q];
    else s->pending[keep++] = q;
  }
  s->npending = keep;
  double L = nw > 0 ? p99_nearest_rank(s->window, nw) : 0.0;
  int64_t sw0 = s->ctl.switches;
  ctl_sample(&s->ctl, cfg, nw > 0, L);
  if (sw0 == 0 && s->ctl.switches > 0) s->sum->first_switch_t = tt;
  if (s->ctl.regime > s->sum->max_regime) s->sum->max_regime = s->ctl.regime;
  if (s->tick_ewma && s->sum->ticks < s->max_ticks) {
    s->tick_ewma[s->sum->ticks] = s->ctl.have_ewma ? s->ctl.ewma : -1.0;
    s->tick_regime[s->sum->ticks] = s->ctl.regime;
  }
  s->sum->ticks_in_regime[s->ctl.regime]++;
  s->sum->ticks++;
  s->next_tick++;
  if (s->sum->ticks >= TICK_LIMIT) s->err = ORC_ERR_CAPACITY;
}

static double next_tick_time(const sim_t* s) {
  return s->rep->controller ? (double)s->next_tick * s->cfg->dt : INFINITY;
}

/* Concurrency of the load-spike schedule at time t (Experiment 3). */
static int64_t conc_at(const orc_replica* r, double t) {
  if (r->c_mid <= 0) return r->C;
  if (t < r->c_t1) return r->C;
  if (t < r->c_t2) return r->c_mid;
  return r->c_end;
}

/* The next time after t at which the schedule's concurrency changes. */
static double next_step_time(const orc_replica* r, double t) {
  if (r->c_mid <= 0) return INFINITY;
  if (t < r->c_t1) return r->c_t1;
  if (t < r->c_t2) return r->c_t2;
  return INFINITY;
}

/* worker j's tiers from G1 down */
static void worker_tiers(sim_t* s, int32_t j, int32_t ntier, const int32_t* tid, lru_t** out) {
  for (int32_t t = 0; t < ntier; t++)
    out[t] = tid[t] == 1 ? &s->cache[j] : tid[t] == 2 ? &s->g2[j] : &s->g3[j];
}

/* blocks resident on all workers, every tier */
static int64_t resident(const sim_t* s) {
  int64_t live = 0;
  for (int32_t j = 0; j < s->W; j++) {
    live += s->cache[j].size;
    if (s->g2) live += s->g2[j].size + s->g3[j].size;
  }
  return live;
}

/* Eq. kv-cost (§4.2) of request i's blocks on worker sigma, as the caches
 * stand when it is routed: per block alpha_t for sigma's own tier t; else
 * the cheapest d(sigma, j) + alpha_t over copies on other workers (ties:
 * same node before other node, then G1 before G2 before G3); else gamma.
 * The request's cost sums the categories in a fixed order. */
static void kv_charge(sim_t* s, int32_t sigma, const uint64_t* h, int64_t nb, int32_t ntier,
                      const int32_t* tid, int64_t i) {
  const orc_config* cfg = s->cfg;
  const int32_t W = s->W;
  int64_t cnt[10] = {0};   /* own G1..G3, near G1..G3, far G1..G3, recompute */
  lru_t* own[3];
  worker_tiers(s, sigma, ntier, tid, own);
  for (int64_t k = 0; k < nb; k++) {
    const int32_t t = tier_of(own, tid, ntier, h[k]);
    if (t > 0) {
      cnt[t - 1]++;
      continue;
    }
    int has[2][3] = {{0, 0, 0}, {0, 0, 0}};
    for (int32_t j = 0; j < W; j++) {
      if (j == sigma) continue;
      lru_t* tl[3];
      worker_tiers(s, j, ntier, tid, tl);
      const int32_t tj = tier_of(tl, tid, ntier, h[k]);
      if (tj > 0) has[j / cfg->tier_node == sigma / cfg->tier_node ? 0 : 1][tj - 1] = 1;
    }
    int cat = 9;
    double best = INFINITY;
    for (int r = 0; r < 2; r++)
      for (int q = 0; q < 3; q++) {
        if (!has[r][q]) continue;
        const double v = (r == 0 ? cfg->tier_d_near : cfg->tier_d_far) + cfg->tier_alpha[q];
        if (v < best) {
          best = v;
          cat = 3 + 3 * r + q;
        }
      }
    cnt[cat]++;
  }
  const double* al = cfg->tier_alpha;
  const double dn = cfg->tier_d_near, df = cfg->tier_d_far;
  double c = al[0] * (double)cnt[0];
  c = c + al[1] * (double)cnt[1];
  c = c + al[2] * (double)cnt[2];
  for (int q = 0; q < 3; q++) c = c + (dn + al[q]) * (double)cnt[3 + q];
  for (int q = 0; q < 3; q++) c = c + (df + al[q]) * (double)cnt[6 + q];
  c = c + cfg->tier_gamma * (double)cnt[9];
  orc_summary* sum = s->sum;
  sum->kv_g1 += cnt[0];
  sum->kv_g2 += cnt[1];
  sum->kv_g3 += cnt[2];
  sum->kv_remote += cnt[3] + cnt[4] + cnt[5] + cnt[6] + cnt[7] + cnt[8];
  sum->kv_recompute += cnt[9];
  sum->kv_cost = sum->kv_cost + c;
  if (s->kv_cost) s->kv_cost[i] = c;
}

int32_t orc_simulate(const orc_config* cfg, const int32_t* tokens, const int64_t* offsets,
                     const double* release, const int32_t* out_len, const orc_replica* rep,
                     orc_records* rec, orc_summary* sum, uint64_t* cache_keys,
                     int64_t* cache_sizes, double* tick_ewma, int32_t* tick_regime,
                     int64_t max_ticks) {
  memset(sum, 0, sizeof *sum);
  sum->first_switch_t = -1.0;
  sum->first_evict_t = -1.0;
  sum->rho_first_evict = -1.0;
  const int32_t W = cfg->W;
  const int64_t n = rep->n_req;
  if (W < 1 || cfg->block < 2 || (cfg->block & 1) || cfg->K < 1 || cfg->cap < 2 || rep->C < 1 ||
      n < 0 || !(rep->tau >= 0.0f) || !(rep->omega >= 0.0f) ||
      rep->policy < ORC_POLICY_DYNAMO || rep->policy > ORC_POLICY_P2C ||
      (rep->c_mid > 0 && (rep->c_end < 1 || !(rep->c_t1 >= 0.0) || !(rep->c_t2 >= rep->c_t1))) ||
      rep->c_mid < 0 || rep->eviction < ORC_EVICT_LRU || rep->eviction > ORC_EVICT_FREQ ||
      (rep->eviction == ORC_EVICT_FREQ &&
       (rep->freq_max < 1 || rep->freq_max > (1 << 20) || !(rep->decay_s > 0.0) ||
        !(rep->decay_s < INFINITY))) ||
      (cfg->tiered &&
       (rep->eviction != ORC_EVICT_LRU || cfg->tier_k2 < 0 || cfg->tier_k3 < 0 ||
        cfg->tier_node < 1 || !(cfg->tier_alpha[0] < cfg->tier_alpha[1]) ||
        !(cfg->tier_alpha[1] < cfg->tier_alpha[2]) || !(cfg->tier_alpha[2] < cfg->tier_gamma) ||
        !(cfg->tier_gamma < INFINITY) || !(cfg->tier_alpha[0] >= 0.0) ||
        !(cfg->tier_d_near >= 0.0) || !(cfg->tier_d_far >= 0.0) ||
        !(cfg->tier_d_near < INFINITY) || !(cfg->tier_d_far < INFINITY)))) {
    sum->status = ORC_ERR_INVALID;
    return ORC_ERR_INVALID;
  }
  sim_t s;
  memset(&s, 0, sizeof s);
  s.cfg = cfg; s.rep = rep; s.tokens = tokens; s.offsets = offsets; s.release = release;
  s.out_len = out_len; s.W = W; s.sum = sum;
  s.tick_ewma = tick_ewma; s.tick_regime = tick_regime; s.max_ticks = max_ticks;
  int64_t nn = n > 0 ? n : 1;
  s.worker = rec && rec->worker ? rec->worker : (int32_t*)malloc(sizeof(int32_t) * nn);
  s.arrival = rec && rec->arrival ? rec->arrival : (double*)malloc(sizeof(double) * nn);
  s.start = rec && rec->start ? rec->start : (double*)malloc(sizeof(double) * nn);
  s.first = rec && rec->first_token ? rec->first_token : (double*)malloc(sizeof(double) * nn);
  s.compl_t = rec && rec->completion ? rec->completion : (double*)malloc(sizeof(double) * nn);
  s.ttft = rec && rec->ttft ? rec->ttft : (double*)malloc(sizeof(double) * nn);
  s.nbt = rec && rec->nbt ? rec->nbt : (int32_t*)malloc(sizeof(int32_t) * nn);
  s.n_frozen = rec ? rec->n_frozen : NULL;
  s.prefix = rec ? rec->prefix : NULL;
  s.cost = rec ? rec->cost : NULL;
  s.o = (double*)malloc(sizeof(double) * nn);
  s.blk = (int64_t*)malloc(sizeof(int64_t) * nn);
  s.qnext = (int64_t*)malloc(sizeof(int64_t) * nn);
  s.pending = (int64_t*)malloc(sizeof(int64_t) * nn);
  s.window = (double*)malloc(sizeof(double) * nn);
  s.heap = (cev*)malloc(sizeof(cev) * nn);
  s.cache = (lru_t*)calloc(W, sizeof(lru_t));
  if (cfg->tiered) {
    s.g2 = (lru_t*)calloc(W, sizeof(lru_t));
    s.g3 = (lru_t*)calloc(W, sizeof(lru_t));
  }
  s.kv_cost = rec ? rec->kv_cost : NULL;
  s.inservice = (int64_t*)calloc(W, sizeof(int64_t));
  s.A = (int64_t*)calloc(W, sizeof(int64_t));
  s.qhead = (int64_t*)malloc(sizeof(int64_t) * W);
  s.qtail = (int64_t*)malloc(sizeof(int64_t) * W);
  int64_t nbmax = 1;
  for (int64_t i = 0; i < n; i++) {
    int64_t nb = (offsets[i + 1] - offsets[i]) / cfg->block;
    if (nb > nbmax) nbmax = nb;
  }
  uint64_t* h = (uint64_t*)malloc(sizeof(uint64_t) * nbmax);
  uint64_t* hs = (uint64_t*)malloc(sizeof(uint64_t) * nbmax);
  float* c = (float*)malloc(sizeof(float) * W);
  int64_t* m = (int64_t*)malloc(sizeof(int64_t) * W);
  int32_t status = ORC_OK;
  if (!s.worker || !s.arrival || !s.start || !s.first || !s.compl_t || !s.ttft || !s.nbt ||
      !s.o || !s.blk || !s.qnext || !s.pending || !s.window || !s.heap || !s.cache ||
      !s.inservice || !s.A || !s.qhead || !s.qtail || !h || !hs || !c || !m) {
    status = ORC_ERR_OOM;
    goto done;
  }
  if (cfg->tiered && (!s.g2 || !s.g3)) { status = ORC_ERR_OOM; goto done; }
  for (int32_t j = 0; j < W; j++) {
    if (lru_init(&s.cache[j], cfg->K)) { status = ORC_ERR_OOM; goto done; }
    if (cfg->tiered && ((cfg->tier_k2 > 0 && lru_init(&s.g2[j], cfg->tier_k2)) ||
                        (cfg->tier_k3 > 0 && lru_init(&s.g3[j], cfg->tier_k3)))) {
      status = ORC_ERR_OOM;
      goto done;
    }
    s.qhead[j] = s.qtail[j] = -1;
  }
  /* the tiers of every worker as a list from G1 down, with their tier numbers */
  int32_t ntier = 1, tid[3] = {1, 2, 3};
  if (cfg->tiered) {
    if (cfg->tier_k2 > 0) tid[ntier++] = 2;
    if (cfg->tier_k3 > 0) tid[ntier++] = 3;
  }
  s.next_tick = 1;
  const int32_t B = cfg->block;
  const int64_t slots = cfg->cap - 1;
  double prev_arrival = 0.0;
  int64_t dclock = 0;   /* decay steps applied so far (frequency eviction) */

  for (int64_t i = 0; i < n; i++) {
    /* closed-loop client (§7.4): request i waits until fewer than C(t)
     * requests are in flight; completions, controller samples and steps of
     * the load-spike schedule are taken in time order (ties in that order) */
    double T = prev_arrival;
    while (s.in_flight >= conc_at(rep, T)) {
      double tc = s.nheap > 0 ? s.heap[0].t : INFINITY;
      double tt = next_tick_time(&s);
      double ts = next_step_time(rep, T);
      if (tc == INFINITY && ts == INFINITY) { status = ORC_ERR_TIMEOUT; goto done; }
      if (tc <= tt && tc <= ts) {
        cev e = heap_pop(s.heap, &s.nheap);
        complete(&s, e.q, e.t);
        if (e.t > T) T = e.t;
      } else if (tt <= ts) {
        controller_tick(&s);
        if (s.err) { status = s.err; goto done; }
      } else {
        T = ts;   /* the schedule steps to its next concurrency */
      }
    }
    double a = release[i] > T ? release[i] : T;
    /* every completion and controller sample up to the arrival, in time order */
    for (;;) {
      double tc = s.nheap > 0 ? s.heap[0].t : INFINITY;
      double tt = next_tick_time(&s);
      if (tc <= tt) {
        if (tc > a) break;
        cev e = heap_pop(s.heap, &s.nheap);
        complete(&s, e.q, e.t);
      } else {
        if (tt > a) break;
        controller_tick(&s);
        if (s.err) { status = s.err; goto done; }
      }
    }

    /* route request i at time a (Algorithm 1) */
    int64_t L = offsets[i + 1] - offsets[i];
    int64_t nb = L / B;
    int64_t nbt = (L + B - 1) / B;
    s.blk[i] = (L + out_len[i] + B - 1) / B;
    /* a prompt must fit the worker's cache (all tiers when tiered) */
    if (nb > cfg->K + (cfg->tiered ? cfg->tier_k2 + cfg->tier_k3 : 0)) {
      status = ORC_ERR_CAPACITY;
      goto done;
    }
    hash_request(tokens + offsets[i], nb, B, cfg->hash_seed, h);
    if (has_duplicate(h, nb, hs)) { status = ORC_ERR_COLLISION; goto done; }
    float tau = rep->tau, omega = rep->omega;
    if (rep->policy == ORC_POLICY_LOADBAL) {
      tau = 0.0f;
      omega = 0.0f;
    } else if (rep->controller && s.ctl.regime > 0) {
      tau = cfg->regime_tau[s.ctl.regime];
      omega = cfg->regime_omega[s.ctl.regime];
    }
    for (int32_t j = 0; j < W; j++) {
      m[j] = cached_prefix(&s.cache[j], h, nb);
      int64_t bp = nbt - m[j];
      c[j] = omega * (float)bp + (float)s.A[j];   /* Eq. (1) */
      int64_t nf = s.inservice[j] + 1;
      if (nf > slots) nf = slots;
      if (s.n_frozen) s.n_frozen[i * W + j] = (uint16_t)nf;
      if (s.prefix) s.prefix[i * W + j] = (uint16_t)m[j];
      if (s.cost) s.cost[i * W + j] = c[j];
    }
    uint32_t u24 = 0u;
    int32_t jstar;
    if (rep->policy == ORC_POLICY_ROUNDROBIN) {
      /* request i goes to worker i mod W */
      jstar = (int32_t)(i % W);
    } else if (rep->policy == ORC_POLICY_RANDOM || rep->policy == ORC_POLICY_P2C) {
      /* uniform workers from one Philox block of this request */
      uint32_t ctr[4] = {(uint32_t)i, (uint32_t)((uint64_t)i >> 32), 0u, TAG_SIM};
      uint32_t key[2] = {(uint32_t)rep->seed, (uint32_t)(rep->seed >> 32)};
      uint32_t x[4];
      orc_philox4x32_10(ctr, key, x);
      int32_t j1 = (int32_t)(((uint64_t)(x[0] >> 8) * (uint64_t)W) >> 24);
      jstar = j1;
      if (rep->policy == ORC_POLICY_P2C && W >= 2) {
        /* a second worker, uniform over the other W - 1 */
        int32_t j2 = (int32_t)(((uint64_t)(x[1] >> 8) * (uint64_t)(W - 1)) >> 24);
        if (j2 >= j1) j2++;
        int32_t lo = j1 < j2 ? j1 : j2, hi = j1 < j2 ? j2 : j1;
        jstar = c[hi] < c[lo] ? hi : lo;   /* lower Eq. (1) cost, ties to the lower index */
      }
    } else {
      if (tau > 0.0f) u24 = draw_u24(rep->seed, (uint64_t)i, 0u, TAG_SIM);
      jstar = orc_select(c, W, tau, u24);
    }
    if (W >= 2) {
      int32_t b = argmin_lowest(c, W);
      float c2 = INFINITY;
      for (int32_t j = 0; j < W; j++)
        if (j != b && c[j] < c2) c2 = c[j];
      double diff = (double)c2 - (double)c[b];
      if (diff <= 1e-6 * fabs((double)c2)) sum->near_ties++;
      if (c2 == c[b]) sum->exact_ties++;
    }
    if (tau > 0.0f && (rep->policy == ORC_POLICY_DYNAMO || rep->policy == ORC_POLICY_LOADBAL)) {
      sum->sampled++;
      sum->near_boundary += near_boundary(c, W, tau, u24);
    }
    if (rep->eviction == ORC_EVICT_FREQ) {
      /* the decay steps since the last request, applied to every block */
      double q = floor(a / rep->decay_s);
      int64_t D = q < 2147483648.0 ? (int64_t)q : 2147483648ll;
      if (D > dclock) {
        for (int32_t j = 0; j < W; j++) freq_decay(&s.cache[j], D - dclock);
        dclock = D;
      }
    }
    if (cfg->tiered) kv_charge(&s, jstar, h, nb, ntier, tid, i);
    int64_t out_g1 = 0;   /* blocks that left the chosen worker's G1 */
    if (cfg->tiered) {
      lru_t* tl[3];
      worker_tiers(&s, jstar, ntier, tid, tl);
      tier_update(tl, ntier, h, nb, &sum->inserted_blocks, &out_g1, &sum->evicted_blocks);
    } else {
      const int64_t ev0 = sum->evicted_blocks;
      cache_update(&s.cache[jstar], h, nb, &sum->inserted_blocks, &sum->evicted_blocks,
                   rep->eviction, rep->freq_max);
      out_g1 = sum->evicted_blocks - ev0;
    }
    if (out_g1 > 0 && sum->first_evict_t < 0.0) {
      sum->first_evict_t = a;
      sum->rho_first_evict = (double)resident(&s) / ((double)W * (double)cfg->K);
    }
    sum->hit_blocks += m[jstar];
    s.A[jstar] += s.blk[i];
    s.in_flight++;
    s.worker[i] = jstar;
    s.arrival[i] = a;
    s.nbt[i] = (int32_t)nbt;
    s.o[i] = nbt > 0 ? (double)m[jstar] / (double)nbt : 0.0;
    s.qnext[i] = -1;
    if (s.inservice[jstar] < slots) {
      start_service(&s, i, jstar, a);
    } else {
      if (s.qtail[jstar] >= 0) s.qnext[s.qtail[jstar]] = i; else s.qhead[jstar] = i;
      s.qtail[jstar] = i;
    }
    prev_arrival = a;
    sum->n_routed++;
  }
  /* drain: remaining completions (queued requests start as slots free) */
  while (s.nheap > 0) {
    cev e = heap_pop(s.heap, &s.nheap);
    complete(&s, e.q, e.t);
  }
  sum->final_regime = s.ctl.regime;
  sum->final_ewma = s.ctl.have_ewma ? s.ctl.ewma : -1.0;
  sum->rho_end = (double)resident(&s) / ((double)W * (double)cfg->K);
  sum->regime_switches = s.ctl.switches;
  if (cache_sizes || cache_keys) {
    /* least to most recent; tiered: G3, then G2, then G1 (one recency stack
     * of K + tier_k2 + tier_k3 blocks per worker) */
    const int64_t per = cfg->tiered ? cfg->K + cfg->tier_k2 + cfg->tier_k3 : cfg->K;
    for (int32_t j = 0; j < W; j++) {
      int64_t sz = 0;
      uint64_t* out = cache_keys ? cache_keys + (int64_t)j * per : NULL;
      if (cfg->tiered) {
        if (cfg->tier_k3 > 0) sz += out ? lru_dump(&s.g3[j], out + sz) : s.g3[j].size;
        if (cfg->tier_k2 > 0) sz += out ? lru_dump(&s.g2[j], out + sz) : s.g2[j].size;
      }
      sz += out ? lru_dump(&s.cache[j], out + sz) : s.cache[j].size;
      if (cache_sizes) cache_sizes[j] = sz;
    }
  }
done:
  sum->status = status;
  if (s.cache)
    for (int32_t j = 0; j < W; j++) lru_free(&s.cache[j]);
  if (s.g2)
    for (int32_t j = 0; j < W; j++) lru_free(&s.g2[j]);
  if (s.g3)
    for (int32_t j = 0; j < W; j++) lru_free(&s.g3[j]);
  free(s.g2);
  free(s.g3);
  if (!(rec && rec->worker)) free(s.worker);
  if (!(rec && rec->arrival)) free(s.arrival);
  if (!(rec && rec->start)) free(s.start);
  if (!(rec && rec->first_token)) free(s.first);
  if (!(rec && rec->completion)) free(s.compl_t);
  if (!(rec && rec->ttft)) free(s.ttft);
  if (!(rec && rec->nbt)) free(s.nbt);
  free(s.o); free(s.blk); free(s.qnext); free(s.pending); free(s.window); free(s.heap);
  free(s.cache); free(s.inservice); free(s.A); free(s.qhead); free(s.qtail);
  free(h); free(hs); free(c); free(m);
  return status;
}

/* ------------------------------------------------------------------------ */
/* Minimum-cost assignment (OPT of Eq. (12))                                 */
/* ------------------------------------------------------------------------ */

/* Hungarian algorithm (potentials form) on the n x (W*capw) matrix whose
 * columns replicate each worker capw times (§6.4). */
static double assign_hungarian(const double* cost, int64_t n, int32_t W, int64_t capw,
                               int32_t* assign) {
  int64_t mcols = (int64_t)W * capw;
  double* u = (double*)calloc(n + 1, sizeof(double));
  double* v = (double*)calloc(mcols + 1, sizeof(double));
  double* minv = (double*)malloc(sizeof(double) * (mcols + 1));
  int64_t* p = (int64_t*)calloc(mcols + 1, sizeof(int64_t));
  int64_t* way = (int64_t*)calloc(mcols + 1, sizeof(int64_t));
  char* used = (char*)malloc(mcols + 1);
  for (int64_t i = 1; i <= n; i++) {
    p[0] = i;
    int64_t j0 = 0;
    for (int64_t j = 0; j <= mcols; j++) { minv[j] = INFINITY; used[j] = 0; }
    do {
      used[j0] = 1;
      int64_t i0 = p[j0], j1 = 0;
      double delta = INFINITY;
      for (int64_t j = 1; j <= mcols; j++) {
        if (used[j]) continue;
        double cur = cost[(i0 - 1) * W + (j - 1) / capw] - u[i0] - v[j];
        if (cur < minv[j]) { minv[j] = cur; way[j] = j0; }
        if (minv[j] < delta) { delta = minv[j]; j1 = j; }
      }
      for (int64_t j = 0; j <= mcols; j++) {
        if (used[j]) { u[p[j]] += delta; v[j] -= delta; }
        else minv[j] -= delta;
      }
      j0 = j1;
    } while (p[j0] != 0);
    do {
      int64_t j1 = way[j0];
      p[j0] = p[j1];
      j0 = j1;
    } while (j0);
  }
  for (int64_t j = 1; j <= mcols; j++)
    if (p[j] != 0) assign[p[j] - 1] = (int32_t)((j - 1) / capw);
  free(u); free(v); free(minv); free(p); free(way); free(used);
  double total = 0.0;
  for (int64_t i = 0; i < n; i++) total += cost[i * W + assign[i]];
  return total;
}

/* Successive shortest paths with Johnson potentials and Dijkstra on
 * source -> rows (1) -> workers (cost) -> sink (capw). */
typedef struct { int64_t to, rev; int64_t capa; double cost; } edge_t;
typedef struct { double d; int64_t v; } hitem;

static void hpush(hitem* h, int64_t* n, hitem e) {
  int64_t i = (*n)++;
  h[i] = e;
  while (i > 0) {
    int64_t p = (i - 1) / 2;
    if (h[p].d <= h[i].d) break;
    hitem t = h[i]; h[i] = h[p]; h[p] = t;
    i = p;
  }
}

static hitem hpop(hitem* h, int64_t* n) {
  hitem top = h[0];
  h[0] = h[--(*n)];
  int64_t i = 0;
  for (;;) {
    int64_t l = 2 * i + 1, r = l + 1, s = i;
    if (l < *n && h[l].d < h[s].d) s = l;
    if (r < *n && h[r].d < h[s].d) s = r;
    if (s == i) break;
    hitem t = h[i]; h[i] = h[s]; h[s] = t;
    i = s;
  }
  return top;
}

static double assign_mcf(const double* cost, int64_t n, int32_t W, int64_t capw,
                         int32_t* assign) {
  int64_t V = n + W + 2, S = 0, T = n + W + 1;
  int64_t E = 2 * (n + n * (int64_t)W + W);
  edge_t* e = (edge_t*)malloc(sizeof(edge_t) * E);
  int64_t* head = (int64_t*)malloc(sizeof(int64_t) * (V + 1));
  int64_t* deg = (int64_t*)calloc(V, sizeof(int64_t));
  /* CSR adjacency: count, then fill */
  for (int64_t i = 0; i < n; i++) { deg[S]++; deg[1 + i]++; }
  for (int64_t i = 0; i < n; i++)
    for (int32_t j = 0; j < W; j++) { deg[1 + i]++; deg[1 + n + j]++; }
  for (int32_t j = 0; j < W; j++) { deg[1 + n + j]++; deg[T]++; }
  head[0] = 0;
  for (int64_t v = 0; v < V; v++) head[v + 1] = head[v] + deg[v];
  int64_t* fill = (int64_t*)malloc(sizeof(int64_t) * V);
  for (int64_t v = 0; v < V; v++) fill[v] = head[v];
#define ADD_EDGE(a, b, cp, cs)                                            \
  do {                                                                    \
    int64_t ea = fill[a]++, eb = fill[b]++;                               \
    e[ea].to = b; e[ea].rev = eb; e[ea].capa = cp; e[ea].cost = cs;       \
    e[eb].to = a; e[eb].rev = ea; e[eb].capa = 0; e[eb].cost = -(cs);     \
  } while (0)
  for (int64_t i = 0; i < n; i++) ADD_EDGE(S, 1 + i, 1, 0.0);
  for (int64_t i = 0; i < n; i++)
    for (int32_t j = 0; j < W; j++) ADD_EDGE(1 + i, 1 + n + j, 1, cost[i * W + j]);
  for (int32_t j = 0; j < W; j++) ADD_EDGE(1 + n + j, T, capw, 0.0);
#undef ADD_EDGE
  double* pot = (double*)calloc(V, sizeof(double));
  double* dist = (double*)malloc(sizeof(double) * V);
  int64_t* pe = (int64_t*)malloc(sizeof(int64_t) * V);
  hitem* hp = (hitem*)malloc(sizeof(hitem) * (E + V + 1));
  for (int64_t it = 0; it < n; it++) {
    for (int64_t v = 0; v < V; v++) { dist[v] = INFINITY; pe[v] = -1; }
    dist[S] = 0.0;
    int64_t nh = 0;
    hitem st = {0.0, S};
    hpush(hp, &nh, st);
    while (nh > 0) {
      hitem x = hpop(hp, &nh);
      if (x.d > dist[x.v]) continue;
      for (int64_t k = head[x.v]; k < head[x.v + 1]; k++) {
        if (e[k].capa <= 0) continue;
        double rc = e[k].cost + pot[x.v] - pot[e[k].to];
        if (rc < 0.0) rc = 0.0;   /* exact reduced costs are >= 0; rounding can dip below */
        double nd = dist[x.v] + rc;
        if (nd < dist[e[k].to]) {
          dist[e[k].to] = nd;
          pe[e[k].to] = k;
          hitem y = {nd, e[k].to};
          hpush(hp, &nh, y);
        }
      }
    }
    if (pe[T] < 0) break;   /* cannot happen while capacity remains */
    for (int64_t v = 0; v < V; v++)
      if (dist[v] < INFINITY) pot[v] += dist[v];
    for (int64_t v = T; v != S;) {
      int64_t k = pe[v];
      e[k].capa -= 1;
      e[e[k].rev].capa += 1;
      v = e[e[k].rev].to;
    }
  }
  int ok = 1;
  for (int64_t i = 0; i < n; i++) {
    assign[i] = -1;
    for (int64_t k = head[1 + i]; k < head[2 + i]; k++)
      if (e[k].to >= 1 + n && e[k].to <= n + W && e[k].capa == 0) {
        assign[i] = (int32_t)(e[k].to - 1 - n);
      }
    if (assign[i] < 0) ok = 0;
  }
  free(e); free(head); free(deg); free(fill); free(pot); free(dist); free(pe); free(hp);
  if (!ok) return NAN;
  double total = 0.0;
  for (int64_t i = 0; i < n; i++) total += cost[i * W + assign[i]];
  return total;
}

/* brute force over all W^n assignments that respect capw (tests only) */
static double assign_brute(const double* cost, int64_t n, int32_t W, int64_t capw,
                           int32_t* assign) {
  int32_t* cur = (int32_t*)calloc(n > 0 ? n : 1, sizeof(int32_t));
  int64_t* load = (int64_t*)calloc(W, sizeof(int64_t));
  double best = INFINITY;
  for (;;) {
    for (int32_t j = 0; j < W; j++) load[j] = 0;
    int ok = 1;
    for (int64_t i = 0; i < n; i++)
      if (++load[cur[i]] > capw) ok = 0;
    if (ok) {
      double t = 0.0;
      for (int64_t i = 0; i < n; i++) t += cost[i * W + cur[i]];
      if (t < best) {
        best = t;
        memcpy(assign, cur, sizeof(int32_t) * n);
      }
    }
    int64_t d = 0;
    while (d < n && ++cur[d] == W) cur[d++] = 0;
    if (d == n) break;
  }
  free(cur); free(load);
  return n > 0 ? best : 0.0;
}

double orc_assign(const double* cost, int64_t n, int32_t W, int64_t capw, int32_t method,
                  int32_t* assign) {
  if (n <= 0) return 0.0;
  if ((int64_t)W * capw < n) return NAN;
  if (method == 1) return assign_hungarian(cost, n, W, capw, assign);
  if (method == 3) return assign_brute(cost, n, W, capw, assign);
  return assign_mcf(cost, n, W, capw, assign);
}

/* Eq. (12): per window, sum of observed TTFT over OPT of the frozen-latency
 * matrix; windows are tumbling intervals of completion time. */
int64_t orc_poa(const orc_config* cfg, int64_t n, const int32_t* worker, const double* completion,
                const double* ttft, const int32_t* nbt, const uint16_t* n_frozen,
                const uint16_t* prefix, int32_t method, double* numer, double* opt,
                int64_t* count, int64_t n_win_cap, double* poa_total) {
  const int32_t W = cfg->W;
  int64_t nw = 0;
  for (int64_t q = 0; q < n; q++) {
    if (worker[q] < 0) continue;
    int64_t w = (int64_t)floor(completion[q] / cfg->poa_window);
    if (w + 1 > nw) nw = w + 1;
  }
  if (nw > n_win_cap) return ORC_ERR_INVALID;
  int64_t* start = (int64_t*)calloc(nw + 1, sizeof(int64_t));
  int64_t* rows = (int64_t*)malloc(sizeof(int64_t) * (n > 0 ? n : 1));
  for (int64_t q = 0; q < n; q++)
    if (worker[q] >= 0) start[(int64_t)floor(completion[q] / cfg->poa_window) + 1]++;
  for (int64_t w = 0; w < nw; w++) start[w + 1] += start[w];
  int64_t* fill = (int64_t*)malloc(sizeof(int64_t) * (nw + 1));
  memcpy(fill, start, sizeof(int64_t) * (nw + 1));
  for (int64_t q = 0; q < n; q++)   /* request order inside each window */
    if (worker[q] >= 0) rows[fill[(int64_t)floor(completion[q] / cfg->poa_window)]++] = q;
  double* cm = (double*)malloc(sizeof(double) * (n > 0 ? n : 1) * W);
  int32_t* as = (int32_t*)malloc(sizeof(int32_t) * (n > 0 ? n : 1));
  double tn = 0.0, to = 0.0;
  for (int64_t w = 0; w < nw; w++) {
    int64_t m = start[w + 1] - start[w];
    count[w] = m;
    numer[w] = 0.0;
    opt[w] = 0.0;
    if (m == 0) continue;
    for (int64_t r = 0; r < m; r++) {
      int64_t q = rows[start[w] + r];
      numer[w] += ttft[q];
      for (int32_t j = 0; j < W; j++)
        cm[r * W + j] = frozen_cost(cfg, n_frozen[q * W + j], prefix[q * W + j], nbt[q]);
    }
    int64_t capw = (m + W - 1) / W;
    if (capw < cfg->cap) capw = cfg->cap;
    int32_t meth = method;
    if (meth == 0) meth = m <= 96 ? 1 : 2;
    opt[w] = orc_assign(cm, m, W, capw, meth, as);
    tn += numer[w];
    to += opt[w];
  }
  *poa_total = to > 0.0 ? tn / to : 0.0;
  free(start); free(rows); free(fill); free(cm); free(as);
  return nw;
}

/* The static counterfactual of the routing-baselines discussion (§9): per
 * window of Eq. (12), the frozen cost of the assignment that was made,
 * sum over the window's requests of c_{i, worker(i)} with the §6.4 cost
 * matrix.  Divided by the window's OPT (orc_poa) it compares the assignment
 * itself, without queueing, with the optimum.  Returns the windows spanned. */
int64_t orc_static_numer(const orc_config* cfg, int64_t n, const int32_t* worker,
                         const double* completion, const int32_t* nbt, const uint16_t* n_frozen,
                         const uint16_t* prefix, double* numer_static, int64_t n_win_cap) {
  const int32_t W = cfg->W;
  int64_t nw = 0;
  for (int64_t q = 0; q < n; q++) {
    if (worker[q] < 0) continue;
    int64_t w = (int64_t)floor(completion[q] / cfg->poa_window);
    if (w + 1 > nw) nw = w + 1;
  }
  if (nw > n_win_cap) return ORC_ERR_INVALID;
  for (int64_t w = 0; w < nw; w++) numer_static[w] = 0.0;
  for (int64_t q = 0; q < n; q++) {   /* request order inside each window */
    if (worker[q] < 0) continue;
    int64_t w = (int64_t)floor(completion[q] / cfg->poa_window);
    int32_t j = worker[q];
    numer_static[w] += frozen_cost(cfg, n_frozen[q * W + j], prefix[q * W + j], nbt[q]);
  }
  return nw;
}

/* ------------------------------------------------------------------------ */
/* Exhaustive one-shot routing game (Def. 3, Def. 5, Def. 7)                 */
/* ------------------------------------------------------------------------ */

static double game_f(int64_t load, double a, double b, double d, int32_t cap) {
  double t1 = a * (double)load;
  double t2 = t1 + b;
  if (d == 0.0) return t2;
  double den = (double)(cap - load);
  return t2 + d / (den * den);
}

int32_t orc_game_exhaustive(int32_t n, int32_t W, const double* o, double omega,
                            double lat_a, double lat_b, double lat_d, int32_t cap,
                            double* opt, double* worst_ne, double* best_ne, double* greedy,
                            int64_t* n_ne, int64_t* br_steps, int32_t* max_ne_spread) {
  if (n < 1 || n > 12 || W < 1 || W > 8 || cap <= n) return ORC_ERR_INVALID;
  int32_t sig[16], load[8];
  for (int32_t i = 0; i < n; i++) sig[i] = 0;
  double vopt = INFINITY, vworst = -INFINITY, vbest = INFINITY;
  int64_t nne = 0;
  int32_t spread = 0;
  for (;;) {
    for (int32_t j = 0; j < W; j++) load[j] = 0;
    for (int32_t i = 0; i < n; i++) load[sig[i]]++;
    double sc = 0.0;
    int ne = 1;
    for (int32_t i = 0; i < n; i++) {
      double cur = game_f(load[sig[i]], lat_a, lat_b, lat_d, cap) - omega * o[i * W + sig[i]];
      sc += cur;
      for (int32_t k = 0; k < W && ne; k++) {
        if (k == sig[i]) continue;
        double alt = game_f(load[k] + 1, lat_a, lat_b, lat_d, cap) - omega * o[i * W + k];
        if (alt < cur - 1e-12) ne = 0;
      }
    }
    if (sc < vopt) vopt = sc;
    if (ne) {
      nne++;
      if (sc > vworst) vworst = sc;
      if (sc < vbest) vbest = sc;
      int32_t lo = load[0], hi = load[0];
      for (int32_t j = 1; j < W; j++) {
        if (load[j] < lo) lo = load[j];
        if (load[j] > hi) hi = load[j];
      }
      if (hi - lo > spread) spread = hi - lo;
    }
    int32_t d = 0;
    while (d < n && ++sig[d] == W) sig[d++] = 0;
    if (d == n) break;
  }
  /* sequential best response in index order (the router's greedy pass) */
  for (int32_t j = 0; j < W; j++) load[j] = 0;
  double vg = 0.0;
  for (int32_t i = 0; i < n; i++) {
    int32_t bk = 0;
    double bc = INFINITY;
    for (int32_t k = 0; k < W; k++) {
      double ck = game_f(load[k] + 1, lat_a, lat_b, lat_d, cap) - omega * o[i * W + k];
      if (ck < bc) { bc = ck; bk = k; }
    }
    sig[i] = bk;
    load[bk]++;
  }
  for (int32_t i = 0; i < n; i++)
    vg += game_f(load[sig[i]], lat_a, lat_b, lat_d, cap) - omega * o[i * W + sig[i]];
  /* best-response dynamics from the greedy profile */
  int64_t steps = 0;
  for (;;) {
    int moved = 0;
    for (int32_t i = 0; i < n && !moved; i++) {
      double cur = game_f(load[sig[i]], lat_a, lat_b, lat_d, cap) - omega * o[i * W + sig[i]];
      int32_t bk = -1;
      double bc = cur - 1e-12;
      for (int32_t k = 0; k < W; k++) {
        if (k == sig[i]) continue;
        double alt = game_f(load[k] + 1, lat_a, lat_b, lat_d, cap) - omega * o[i * W + k];
        if (alt < bc) { bc = alt; bk = k; }
      }
      if (bk >= 0) {
        load[sig[i]]--;
        load[bk]++;
        sig[i] = bk;
        moved = 1;
      }
    }
    if (!moved) break;
    if (++steps > 10000) { steps = -1; break; }
  }
  if (opt) *opt = vopt;
  if (worst_ne) *worst_ne = vworst;
  if (best_ne) *best_ne = vbest;
  if (greedy) *greedy = vg;
  if (n_ne) *n_ne = nne;
  if (br_steps) *br_steps = steps;
  if (max_ne_spread) *max_ne_spread = spread;
  return ORC_OK;
}

/* ------------------------------------------------------------------------ */
/* Live router (route_batch / route_release semantics)                       */
/* ------------------------------------------------------------------------ */

struct orc_router {
  orc_config cfg;
  float omega, tau;
  uint64_t seed;
  int32_t ni;
  lru_t* cache;      /* [ni * W] */
  int64_t* A;        /* [ni * W] */
  uint64_t* ordinal; /* [ni] */
};

orc_router* orc_router_new(const orc_config* cfg, float omega, float tau, uint64_t seed,
                           int32_t n_instances) {
  if (cfg->W < 1 || n_instances < 1 || !(tau >= 0.0f) || !(omega >= 0.0f)) return NULL;
  orc_router* r = (orc_router*)calloc(1, sizeof(orc_router));
  r->cfg = *cfg;
  r->omega = omega;
  r->tau = tau;
  r->seed = seed;
  r->ni = n_instances;
  int64_t nw = (int64_t)n_instances * cfg->W;
  r->cache = (lru_t*)calloc(nw, sizeof(lru_t));
  r->A = (int64_t*)calloc(nw, sizeof(int64_t));
  r->ordinal = (uint64_t*)calloc(n_instances, sizeof(uint64_t));
  for (int64_t k = 0; k < nw; k++) lru_init(&r->cache[k], cfg->K);
  return r;
}

void orc_router_free(orc_router* r) {
  if (!r) return;
  for (int64_t k = 0; k < (int64_t)r->ni * r->cfg.W; k++) lru_free(&r->cache[k]);
  free(r->cache); free(r->A); free(r->ordinal); free(r);
}

int32_t orc_router_route(orc_router* r, int32_t inst, const int32_t* tokens,
                         const int64_t* offsets, int64_t n_req, const int32_t* out_len,
                         int32_t* worker, float* cost, int32_t* prefix) {
  if (!r || inst < 0 || inst >= r->ni) return ORC_ERR_INVALID;
  const int32_t W = r->cfg.W, B = r->cfg.block;
  lru_t* cache = r->cache + (int64_t)inst * W;
  int64_t* A = r->A + (int64_t)inst * W;
  int64_t nbmax = 1;
  for (int64_t i = 0; i < n_req; i++) {
    int64_t nb = (offsets[i + 1] - offsets[i]) / B;
    if (nb > nbmax) nbmax = nb;
  }
  uint64_t* h = (uint64_t*)malloc(sizeof(uint64_t) * nbmax);
  uint64_t* hs = (uint64_t*)malloc(sizeof(uint64_t) * nbmax);
  float* c = (float*)malloc(sizeof(float) * W);
  int64_t* m = (int64_t*)malloc(sizeof(int64_t) * W);
  int32_t status = ORC_OK;
  int64_t ins = 0, ev = 0;
  for (int64_t i = 0; i < n_req; i++) {
    int64_t L = offsets[i + 1] - offsets[i];
    int64_t nb = L / B, nbt = (L + B - 1) / B;
    if (nb > r->cfg.K) { status = ORC_ERR_CAPACITY; break; }
    hash_request(tokens + offsets[i], nb, B, r->cfg.hash_seed, h);
    if (has_duplicate(h, nb, hs)) { status = ORC_ERR_COLLISION; break; }
    for (int32_t j = 0; j < W; j++) {
      m[j] = cached_prefix(&cache[j], h, nb);
      c[j] = r->omega * (float)(nbt - m[j]) + (float)A[j];
      if (cost) cost[i * W + j] = c[j];
      if (prefix) prefix[i * W + j] = (int32_t)m[j];
    }
    uint32_t u24 = r->tau > 0.0f ? draw_u24(r->seed, r->ordinal[inst], (uint32_t)inst, TAG_ROUTE)
                                 : 0u;
    int32_t js = orc_select(c, W, r->tau, u24);
    cache_update(&cache[js], h, nb, &ins, &ev, ORC_EVICT_LRU, 1);
    A[js] += (L + out_len[i] + B - 1) / B;
    worker[i] = js;
    r->ordinal[inst]++;
  }
  free(h); free(hs); free(c); free(m);
  return status;
}

/* Every request's cached prefix m_ij on every worker of an instance, against
 * the caches as they stand: the leading full blocks found (S2, the b^prefill
 * of Eq. (1)), with no cache or load touched, so that every request sees the
 * same snapshot. */
int32_t orc_router_probe(orc_router* r, int32_t inst, const int32_t* tokens,
                         const int64_t* offsets, int64_t n_req, int32_t* prefix) {
  if (!r || inst < 0 || inst >= r->ni || n_req < 0) return ORC_ERR_INVALID;
  const int32_t W = r->cfg.W, B = r->cfg.block;
  const lru_t* cache = r->cache + (int64_t)inst * W;
  int64_t nbmax = 1;
  for (int64_t i = 0; i < n_req; i++) {
    int64_t nb = (offsets[i + 1] - offsets[i]) / B;
    if (nb > nbmax) nbmax = nb;
  }
  uint64_t* h = (uint64_t*)malloc(sizeof(uint64_t) * nbmax);
  for (int64_t i = 0; i < n_req; i++) {
    const int64_t nb = (offsets[i + 1] - offsets[i]) / B;
    hash_request(tokens + offsets[i], nb, B, r->cfg.hash_seed, h);
    for (int32_t j = 0; j < W; j++) prefix[i * W + j] = (int32_t)cached_prefix(&cache[j], h, nb);
  }
  free(h);
  return ORC_OK;
}

int32_t orc_router_release(orc_router* r, int32_t inst, const int32_t* worker,
                           const int32_t* blocks, int64_t n) {
  if (!r || inst < 0 || inst >= r->ni) return ORC_ERR_INVALID;
  int64_t* A = r->A + (int64_t)inst * r->cfg.W;
  int32_t status = ORC_OK;
  for (int64_t i = 0; i < n; i++) {
    if (worker[i] < 0 || worker[i] >= r->cfg.W) {   /* skipped, reported */
      status = ORC_ERR_INVALID;
      continue;
    }
    A[worker[i]] -= blocks[i];
    if (A[worker[i]] < 0) A[worker[i]] = 0;
  }
  return status;
}

int32_t orc_router_active(orc_router* r, int32_t inst, int64_t* active) {
  if (!r || inst < 0 || inst >= r->ni) return ORC_ERR_INVALID;
  memcpy(active, r->A + (int64_t)inst * r->cfg.W, sizeof(int64_t) * r->cfg.W);
  return ORC_OK;
}

int32_t orc_router_cache(orc_router* r, int32_t inst, int32_t worker, uint64_t* keys,
                         int64_t* size) {
  if (!r || inst < 0 || inst >= r->ni || worker < 0 || worker >= r->cfg.W) return ORC_ERR_INVALID;
  *size = lru_dump(&r->cache[(int64_t)inst * r->cfg.W + worker], keys);
  return ORC_OK;
}
