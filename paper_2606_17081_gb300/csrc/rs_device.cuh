// Device building blocks of the routing library (sm_103a).
//
// Block hashing, Philox, the softmax exp, worker selection (Eq. (1), Eq. (2)),
// and the per-worker KV block cache: an open-addressing table of 64-bit block
// hashes (buckets of four 8-byte keys = one 32-byte sector) whose slots carry
// an LRU stamp, plus a ring "log" of slots in stamp order.  Exact LRU order is
// stamp order: touching or inserting a block gives it the next stamp and
// appends its slot to the log; a log entry is live iff its slot still holds
// that stamp, so the least-recent entries are the first live entries of the
// log.  A request's whole block list is applied in one CTA-wide step.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "rs_internal.h"

namespace rs {

constexpr uint64_t KEY_EMPTY = 0ull;
constexpr uint64_t KEY_TOMB = 1ull;
constexpr uint32_t STAMP_NONE = 0xFFFFFFFFu;
constexpr uint32_t SLOT_NONE = 0xFFFFFFFFu;
constexpr uint32_t STAMP_LIMIT = 0x7FFF0000u;   // compaction renumbers before this
constexpr int64_t TICK_LIMIT = 1ll << 24;       // controller samples per replica
constexpr unsigned FULL_MASK = 0xFFFFFFFFu;

// ---------------------------------------------------------------- hashing

__device__ __forceinline__ uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// content hash g of one 16-token block given as 16 words
// Content hash of one 16-token block: its 64-bit little-endian token pairs
// folded in order by one multiply-xorshift each, then the SplitMix64
// finalizer.
__device__ __forceinline__ uint64_t block_content16(const uint32_t (&w)[16]) {
  uint64_t x = 0x9E3779B97F4A7C15ull ^ 16ull;
#pragma unroll
  for (int q = 0; q < 8; q++) {
    x = (x ^ ((uint64_t)w[2 * q] | ((uint64_t)w[2 * q + 1] << 32))) * 0xBF58476D1CE4E5B9ull;
    x ^= x >> 32;
  }
  return mix64(x);
}

// Prefix hash of blocks 0..k: H_k = H_{k-1} P + g_k (mod 2^64), H_{-1} = the
// hash seed; the stored hash is mix(H_k ^ k), 0 and 1 (the table's empty and
// tombstone keys) mapped to 2 and 3.
constexpr uint64_t PREFIX_P = 0x94D049BB133111EBull;

__device__ __forceinline__ uint64_t prefix_output(uint64_t H, uint64_t k) {
  const uint64_t h = mix64(H ^ k);
  return h < 2 ? h + 2 : h;
}

// ---------------------------------------------------------------- async copies

// 8-byte global -> shared copy that completes in the background (both
// addresses 8-byte aligned); cp_async_wait_all waits for this thread's copies.
__device__ __forceinline__ void cp_async8(void* smem_dst, const void* gmem_src) {
  const unsigned d = (unsigned)__cvta_generic_to_shared(smem_dst);
  asm volatile("cp.async.ca.shared.global [%0], [%1], 8;\n" ::"r"(d), "l"(gmem_src) : "memory");
}

__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.wait_all;\n" ::: "memory");
}

// ---------------------------------------------------------------- Philox4x32-10

__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint2 k) {
#pragma unroll
  for (int r = 0; r < 10; r++) {
    if (r) {
      k.x += 0x9E3779B9u;
      k.y += 0xBB67AE85u;
    }
    const uint32_t hi0 = __umulhi(0xD2511F53u, c.x), lo0 = 0xD2511F53u * c.x;
    const uint32_t hi1 = __umulhi(0xCD9E8D57u, c.z), lo1 = 0xCD9E8D57u * c.z;
    c = make_uint4(hi1 ^ c.y ^ k.x, lo1, hi0 ^ c.w ^ k.y, lo0);
  }
  return c;
}

constexpr uint32_t TAG_SIM = 0x53494D31u;
constexpr uint32_t TAG_ROUTE = 0x52545231u;

__device__ __forceinline__ uint32_t draw_u24(uint64_t seed, uint64_t ordinal, uint32_t stream,
                                             uint32_t tag) {
  uint4 c = make_uint4((uint32_t)ordinal, (uint32_t)(ordinal >> 32), stream, tag);
  uint2 k = make_uint2((uint32_t)seed, (uint32_t)(seed >> 32));
  return philox4x32_10(c, k).x >> 8;
}

// The worker a static policy sends request `ordinal` to (round robin, uniform
// random, power of two choices; §9's routing baselines).  c: Eq. (1) costs
// (P2C only).  Random draws take words x0 and x1 of the request's Philox
// block, counter (ordinal, stream, tag) as draw_u24.
__device__ __forceinline__ int static_policy_worker(int policy, const float* c, int W,
                                                    uint64_t seed, uint64_t ordinal,
                                                    uint32_t stream, uint32_t tag) {
  if (policy == RS_POLICY_ROUNDROBIN) return (int)(ordinal % (uint64_t)W);
  const uint4 x = philox4x32_10(make_uint4((uint32_t)ordinal, (uint32_t)(ordinal >> 32), stream, tag),
                                make_uint2((uint32_t)seed, (uint32_t)(seed >> 32)));
  const int j1 = (int)(((uint64_t)(x.x >> 8) * (uint64_t)W) >> 24);
  if (policy == RS_POLICY_RANDOM || W < 2) return j1;
  int j2 = (int)(((uint64_t)(x.y >> 8) * (uint64_t)(W - 1)) >> 24);   // uniform over the others
  if (j2 >= j1) j2++;
  const int lo = j1 < j2 ? j1 : j2, hi = j1 < j2 ? j2 : j1;
  return c[hi] < c[lo] ? hi : lo;   // lower cost, ties to the lower index
}

// ---------------------------------------------------------------- exp of Eq. (2)

// Cody-Waite reduction by ln2 (split in an 8-trailing-zero high part and a
// low part) and the degree-7 Taylor polynomial of exp(r) in Horner form with
// fused multiply-adds; 2^k through the exponent field.  x < -87 gives 0.
__device__ __forceinline__ float exp_sm(float x) {
  if (!(x >= -87.0f)) return 0.0f;
  if (x > 88.0f) return __int_as_float(0x7F800000);
  const float t = __fmul_rn(x, 0x1.715476p+0f);
  const float kf = rintf(t);
  float r = __fmaf_rn(-kf, 0x1.62e4p-1f, x);
  r = __fmaf_rn(-kf, 0x1.7f7d1cp-20f, r);
  float p = 0x1.a01a02p-13f;
  p = __fmaf_rn(p, r, 0x1.6c16c2p-10f);
  p = __fmaf_rn(p, r, 0x1.111112p-7f);
  p = __fmaf_rn(p, r, 0x1.555556p-5f);
  p = __fmaf_rn(p, r, 0x1.555556p-3f);
  p = __fmaf_rn(p, r, 0.5f);
  p = __fmaf_rn(p, r, 1.0f);
  p = __fmaf_rn(p, r, 1.0f);
  const int k = (int)kf;
  return __fmul_rn(p, __int_as_float((k + 127) << 23));
}

// ---------------------------------------------------------------- selection

// Eq. (1) in fp32, rounded per operation: omega * b^prefill + b^active.
// Both counts are below 2^31 (and exact in fp32 below 2^24), so they are
// converted from 32-bit integers (the 64-bit conversion is a slower path).
__device__ __forceinline__ float router_cost(float omega, int64_t bprefill, int64_t active) {
  return __fadd_rn(__fmul_rn(omega, __int2float_rn((int)bprefill)), __int2float_rn((int)active));
}

// Lowest-index argmin over c[0..W) (one thread).
__device__ __forceinline__ int argmin_lowest(const float* c, int W) {
  int b = 0;
  for (int j = 1; j < W; j++)
    if (c[j] < c[b]) b = j;
  return b;
}

// Eq. (2): tau == 0 -> argmin; tau > 0 -> the first j whose cumulative weight
// (sequential fp32 sum in worker order) exceeds u * S.  One thread.
// ds (nullable) receives the draw's position for the near-boundary
// statistic: {u S, S, largest cumulative weight <= u S (or NaN), smallest
// cumulative weight > u S (or NaN)}.
__device__ __forceinline__ int select_worker(const float* c, int W, float tau, uint32_t u24,
                                             float* ds) {
  const int b = argmin_lowest(c, W);
  if (tau == 0.0f) return b;
  const float cmin = c[b];
  float S = 0.0f;
  for (int j = 0; j < W; j++) S = __fadd_rn(S, exp_sm(-__fdiv_rn(__fsub_rn(c[j], cmin), tau)));
  const float target = __fmul_rn(__fmul_rn((float)u24, 0x1p-24f), S);
  const float qnan = __int_as_float(0x7FC00000);
  float cum = 0.0f, lo = qnan, hi = qnan;
  int pick = -1, last = b;
  for (int j = 0; j < W; j++) {
    const float e = exp_sm(-__fdiv_rn(__fsub_rn(c[j], cmin), tau));
    cum = __fadd_rn(cum, e);
    if (e > 0.0f) last = j;
    if (pick < 0 && target < cum) {
      pick = j;
      hi = cum;
    }
    if (!(target < cum)) lo = cum;
  }
  if (ds) {
    ds[0] = target;
    ds[1] = S;
    ds[2] = lo;
    ds[3] = hi;
  }
  return pick >= 0 ? pick : last;
}

// select_worker computed by a whole warp (W <= 64; every lane returns the
// same worker): lane l computes the weights of workers l and l + 32, each
// once, and every lane then accumulates them in worker order from shuffles,
// so the sums, the draw and the statistics are those of select_worker bit
// for bit.  b: the lowest-index argmin of c.  ds (nullable) is written by
// lane 0.
__device__ __forceinline__ int select_worker_warp(const float* c, int W, float tau, uint32_t u24,
                                                  int b, float* ds, int lane) {
  if (tau == 0.0f) return b;
  const float cmin = c[b];
  float e[2];
#pragma unroll
  for (int h = 0; h < 2; h++) {
    const int j = lane + 32 * h;
    e[h] = j < W ? exp_sm(-__fdiv_rn(__fsub_rn(c[j], cmin), tau)) : 0.0f;
  }
  float S = 0.0f;
  for (int j = 0; j < W; j++) S = __fadd_rn(S, __shfl_sync(FULL_MASK, e[j >> 5], j & 31));
  const float target = __fmul_rn(__fmul_rn((float)u24, 0x1p-24f), S);
  const float qnan = __int_as_float(0x7FC00000);
  float cum = 0.0f, lo = qnan, hi = qnan;
  int pick = -1, last = b;
  for (int j = 0; j < W; j++) {
    const float ej = __shfl_sync(FULL_MASK, e[j >> 5], j & 31);
    cum = __fadd_rn(cum, ej);
    if (ej > 0.0f) last = j;
    if (pick < 0 && target < cum) {
      pick = j;
      hi = cum;
    }
    if (!(target < cum)) lo = cum;
  }
  if (ds && lane == 0) {
    ds[0] = target;
    ds[1] = S;
    ds[2] = lo;
    ds[3] = hi;
  }
  return pick >= 0 ? pick : last;
}

// ---------------------------------------------------------------- CTA helpers

// Barrier of a thread group made of the CTA's first NT threads: the whole
// 256-thread CTA uses __syncthreads, a smaller leading group the named
// barrier 1 (so the remaining warps can work on something else meanwhile).
template <int NT>
__device__ __forceinline__ void grp_bar() {
  if constexpr (NT == 256) {
    __syncthreads();
  } else {
    asm volatile("bar.sync 1, %0;" ::"n"(NT) : "memory");
  }
}

// Exclusive rank of `flag` among the CTA's threads (thread order) and the
// total; two barriers.  warp_tot: shared int[NT/32].
template <int NT>
__device__ __forceinline__ int cta_rank(bool flag, int* warp_tot, int* total) {
  const unsigned m = __ballot_sync(FULL_MASK, flag);
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  if (lane == 0) warp_tot[w] = __popc(m);
  grp_bar<NT>();
  int off = 0, tot = 0;
#pragma unroll
  for (int i = 0; i < NT / 32; i++) {
    const int v = warp_tot[i];
    off += i < w ? v : 0;
    tot += v;
  }
  grp_bar<NT>();
  *total = tot;
  return off + __popc(m & ((1u << lane) - 1u));
}

// Exclusive prefix sum of v over the group (thread order) and the total.
template <int NT>
__device__ __forceinline__ int grp_excl_scan(int v, int* warp_tot, int* total) {
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(FULL_MASK, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_tot[w] = x;
  grp_bar<NT>();
  int off = 0, tot = 0;
#pragma unroll
  for (int i = 0; i < NT / 32; i++) {
    const int t = warp_tot[i];
    off += i < w ? t : 0;
    tot += t;
  }
  grp_bar<NT>();
  *total = tot;
  return off + x - v;
}

// ---------------------------------------------------------------- cache table

constexpr int BUCKET = 8;   // keys per bucket: 64 bytes, two 32-byte sectors

struct TableView {
  uint64_t* keys;     // [BUCKET * nbuckets]
  uint32_t* stamp;    // [BUCKET * nbuckets]
  uint32_t* log;      // [rmask + 1]
  uint32_t* fexp;     // [BUCKET * nbuckets] frequency eviction state, or NULL
  uint32_t bmask;     // nbuckets - 1
  uint32_t rmask;     // log ring size - 1
};

__device__ __forceinline__ uint32_t home_bucket(uint64_t h, uint32_t bmask) {
  return (uint32_t)(h ^ (h >> 32)) & bmask;
}

// Brings the line holding p into L2 (no register result, no wait).
__device__ __forceinline__ void prefetch_l2(const void* p) {
  asm volatile("prefetch.global.L2 [%0];" ::"l"(p));
}

// Four keys (one 32-byte sector) in one 256-bit load through L2; p 32-byte
// aligned (buckets are 64-byte aligned: the key arrays start on 256-byte
// boundaries and every table holds a multiple of 8 slots).
__device__ __forceinline__ void ld_keys4(const uint64_t* p, uint64_t& a, uint64_t& b, uint64_t& c,
                                         uint64_t& d) {
  unsigned long long x0, x1, x2, x3;
  asm("ld.global.cg.v4.u64 {%0, %1, %2, %3}, [%4];"
               : "=l"(x0), "=l"(x1), "=l"(x2), "=l"(x3)
               : "l"(p));
  a = x0;
  b = x1;
  c = x2;
  d = x3;
}

// The BUCKET keys of bucket b: two independent 256-bit loads, one request
// per 32-byte sector.
__device__ __forceinline__ void ld_bucket(const uint64_t* keys, uint32_t b, uint64_t (&v)[BUCKET]) {
  const uint64_t* p = keys + (size_t)BUCKET * b;
  static_assert(BUCKET == 8, "two 32-byte sectors per bucket");
  ld_keys4(p, v[0], v[1], v[2], v[3]);
  ld_keys4(p + 4, v[4], v[5], v[6], v[7]);
}

// Slot holding h, or SLOT_NONE; *free_slot = the first EMPTY or TOMB slot of
// h's probe sequence (where an insert of h would go), with FREE_TOMB set when
// that slot held a tombstone, or SLOT_NONE.  Buckets are scanned from h's
// home bucket; a bucket with an EMPTY key ends the search (keys are never
// moved, and slots only go from EMPTY to a key, key to TOMB, TOMB to a key).
// *err is set if the scan wraps around the table.
constexpr uint32_t FREE_TOMB = 0x80000000u;

// Resolves one loaded bucket: returns 1 (found, *slot set), 0 (absent: the
// bucket holds an EMPTY key) or -1 (continue with the next bucket).  *fr, if
// still SLOT_NONE, becomes the bucket's first EMPTY or TOMB slot before the
// match (before the end when h is absent).
__device__ __forceinline__ int bucket_scan(const uint64_t (&v)[BUCKET], uint32_t b, uint64_t h,
                                           uint32_t* slot, uint32_t* fr) {
  bool empty = false;
#pragma unroll
  for (int q = 0; q < BUCKET; q++) {
    if (v[q] == h) {
      *slot = (uint32_t)BUCKET * b + q;
      return 1;
    }
    if (v[q] < 2 && *fr == SLOT_NONE)
      *fr = ((uint32_t)BUCKET * b + q) | (v[q] == KEY_TOMB ? FREE_TOMB : 0u);
    empty |= v[q] == KEY_EMPTY;
  }
  return empty ? 0 : -1;
}

// bucket_scan without branches: the eight keys give three bit masks, so the
// lanes of a warp never diverge on where h sits (the simulation's probes,
// which keep several buckets in flight per thread; a one-lookup-at-a-time
// walk is better served by the early exit above).
__device__ __forceinline__ int bucket_scan_masks(const uint64_t (&v)[BUCKET], uint32_t b,
                                                 uint64_t h, uint32_t* slot, uint32_t* fr) {
  unsigned hit = 0, fre = 0, tomb = 0;
#pragma unroll
  for (int q = 0; q < BUCKET; q++) {
    hit |= (unsigned)(v[q] == h) << q;
    fre |= (unsigned)(v[q] < 2) << q;   // EMPTY or TOMB
    tomb |= (unsigned)(v[q] == KEY_TOMB) << q;
  }
  const unsigned before = hit ? (hit & (0u - hit)) - 1u : (1u << BUCKET) - 1u;   // before the match
  const unsigned f = fre & before;
  if (f && *fr == SLOT_NONE) {
    const int q = __ffs(f) - 1;
    *fr = ((uint32_t)BUCKET * b + q) | ((tomb >> q) & 1u ? FREE_TOMB : 0u);
  }
  if (hit) {
    *slot = (uint32_t)BUCKET * b + (__ffs(hit) - 1);
    return 1;
  }
  return (fre & ~tomb) ? 0 : -1;
}

__device__ __forceinline__ uint32_t table_find_free_from(const TableView& t, uint64_t h,
                                                         uint32_t b, int* err,
                                                         uint32_t* free_slot) {
  for (uint32_t it = 0; it <= t.bmask; it++) {
    uint64_t v[BUCKET];
    ld_bucket(t.keys, b, v);
    uint32_t sl = SLOT_NONE;
    const int r = bucket_scan(v, b, h, &sl, free_slot);
    if (r >= 0) return sl;
    b = (b + 1) & t.bmask;
  }
  *err = 1;
  return SLOT_NONE;
}

__device__ __forceinline__ uint32_t table_find_free(const TableView& t, uint64_t h, int* err,
                                                    uint32_t* free_slot) {
  *free_slot = SLOT_NONE;
  return table_find_free_from(t, h, home_bucket(h, t.bmask), err, free_slot);
}

__device__ __forceinline__ uint32_t table_find(const TableView& t, uint64_t h, int* err) {
  uint32_t fr;
  return table_find_free(t, h, err, &fr);
}

// Claims the first EMPTY or TOMB slot of h's probe sequence (h known absent;
// other threads of the CTA may insert concurrently).  *was_tomb reports a
// reclaimed tombstone.
__device__ __forceinline__ uint32_t table_insert(const TableView& t, uint64_t h, int* was_tomb,
                                                 int* err) {
  uint32_t b = home_bucket(h, t.bmask);
  for (uint32_t it = 0; it <= t.bmask; it++) {
    uint64_t v[BUCKET];
    ld_bucket(t.keys, b, v);
#pragma unroll
    for (int q = 0; q < BUCKET; q++) {
      unsigned long long cur = v[q];
      unsigned long long* p =
          reinterpret_cast<unsigned long long*>(t.keys + (size_t)BUCKET * b + q);
      while (cur == KEY_EMPTY || cur == KEY_TOMB) {
        const unsigned long long prev = atomicCAS(p, cur, (unsigned long long)h);
        if (prev == cur) {
          *was_tomb = cur == KEY_TOMB;
          return (uint32_t)BUCKET * b + q;
        }
        cur = prev;
      }
    }
    b = (b + 1) & t.bmask;
  }
  *err = 1;
  return SLOT_NONE;
}

// Scratch of one CTA-wide cache update (shared memory).
struct UpdateScratch {
  uint32_t* slot;     // [nbmax] slot per request block
  uint32_t* pst;      // [nbmax] stamp of present blocks
  uint32_t* fslot;    // [nbmax] insert position seen by the lookup (FREE_TOMB flag) or SLOT_NONE
  uint8_t* kind;      // [nbmax] 1 = insert, 0 = touch
  uint8_t* evk;       // [nbmax] present block evicted before its turn
  uint32_t* vslot;    // [2*nbmax] first live log entries: slot
  uint32_t* vt;       // [2*nbmax]                          stamp
  int32_t* owner;     // [2*nbmax] request block owning that entry, or -1
  uint8_t* touched;   // [2*nbmax]
  int32_t* victim;    // [2*nbmax] indices into vslot/vt of the evicted entries
  uint64_t* dupset;   // [2*nbmax_pow2] duplicate detector
  uint32_t dupmask;
};

struct UpdateShared {   // small shared scalars of the update
  int n_absent, n_ins, reclaimed, n_victims, n_tomb, slow, err, dup;
  uint32_t pmin, gathered;
};

struct FreqShared {   // small shared scalars of the frequency update
  // where the victim search started, least e and first position of the hot
  // entries it passed, hot entries listed for the exact path
  uint32_t fstart, femin, fhot, gb;
};

// Rebuilds the table and log of one worker from its live entries in LRU
// order (stamps renumbered 0..size-1).  tmp: global scratch of >= size keys.
template <int NT>
__device__ __forceinline__ void cache_rebuild(const TableView& t, CacheMeta* meta, uint32_t K, uint64_t* tmp,
                              int* warp_tot, UpdateShared* us, uint32_t* tmpe = nullptr,
                              FreqMeta* fm = nullptr) {
  const bool fx = t.fexp != nullptr && tmpe != nullptr;   // frequencies move with their keys
  const uint32_t head = meta->head, T = meta->T;
  constexpr int PER = 8;   // log entries per thread per step: independent loads in flight
  uint32_t base = 0;
  for (uint32_t p0 = head; p0 < T; p0 += NT * PER) {
    const uint32_t pb = p0 + threadIdx.x * PER;
    uint32_t x[PER];
    bool live[PER];
    int cnt = 0;
#pragma unroll
    for (int e = 0; e < PER; e++) x[e] = pb + e < T ? t.log[(pb + e) & t.rmask] : 0u;
#pragma unroll
    for (int e = 0; e < PER; e++) {
      live[e] = pb + e < T && __ldcg(t.stamp + x[e]) == pb + e;
      cnt += live[e];
    }
    int tot;
    int off = grp_excl_scan<NT>(cnt, warp_tot, &tot);
#pragma unroll
    for (int e = 0; e < PER; e++)
      if (live[e]) {
        if (base + off < K) {
          tmp[base + off] = __ldcg(t.keys + x[e]);
          if (fx) tmpe[base + off] = __ldcg(t.fexp + x[e]);
        }
        off++;
      }
    base += tot;
  }
  grp_bar<NT>();
  if (base > K) {   // more live log entries than the cache holds: inconsistent state
    if (threadIdx.x == 0) us->err = RS_ERR_TIMEOUT;
    grp_bar<NT>();
    return;
  }
  const size_t nslots = (size_t)BUCKET * ((size_t)t.bmask + 1);
  for (size_t s = threadIdx.x; s < nslots; s += NT) {
    t.keys[s] = KEY_EMPTY;
    t.stamp[s] = STAMP_NONE;
  }
  grp_bar<NT>();
  for (uint32_t r = threadIdx.x; r < base; r += NT) {
    int wt = 0, e = 0;
    const uint32_t sl = table_insert(t, __ldcg(tmp + r), &wt, &e);
    if (e) us->err = RS_ERR_TIMEOUT;
    else {
      t.stamp[sl] = r;
      t.log[r & t.rmask] = sl;
      if (fx) t.fexp[sl] = __ldcg(tmpe + r);
    }
  }
  grp_bar<NT>();
  if (threadIdx.x == 0) {
    if (base != meta->size) us->err = RS_ERR_TIMEOUT;
    meta->head = 0;
    meta->T = base;
    meta->tombs = 0;
    if (fm) *fm = FreqMeta{0u, 0u};
  }
  grp_bar<NT>();
}

// Duplicate detector of one request's block hashes: an open-addressing set in
// shared memory; returns the slot this thread claimed (to clear it later), or
// -1, and sets *dup when h was already there.
__device__ __forceinline__ int32_t dup_claim(UpdateScratch& sc, uint64_t h, int* dup) {
  uint32_t d = (uint32_t)(h ^ (h >> 29)) & sc.dupmask;
  for (uint32_t it = 0; it <= sc.dupmask; it++) {
    const unsigned long long prev = atomicCAS(
        reinterpret_cast<unsigned long long*>(sc.dupset + d), 0ull, (unsigned long long)h);
    if (prev == 0ull) return (int32_t)d;
    if (prev == h) {
      *dup = 1;
      return -1;
    }
    d = (d + 1) & sc.dupmask;
  }
  return -1;
}

// Resets the shared scalars of one cache update.
__device__ __forceinline__ void update_reset(UpdateShared* us) {
  us->n_absent = 0;
  us->n_ins = 0;
  us->reclaimed = 0;
  us->n_victims = 0;
  us->n_tomb = 0;
  us->slow = 0;
  us->dup = 0;
  us->pmin = STAMP_NONE;
  us->gathered = 0;
}

// The frequency update's own scalars, reset once before the first update
// and at the end of each.
__device__ __forceinline__ void freq_reset(FreqShared* fs) {
  fs->femin = 0xFFFFFFFFu;
  fs->fhot = 0xFFFFFFFFu;
}

// Looks up every block of a request in one worker's cache (CTA-wide);
// fills slot[] and pst[]; counts absent blocks; detects duplicate hashes
// within the request (a shared-memory open-addressing set; each thread clears
// the slot it claimed).  us must be reset before the call.
template <int NT, bool DETECT_DUP = true>
__device__ __forceinline__ void cache_lookup_all(const TableView& t, const uint64_t* hbuf, int nb,
                                 UpdateScratch& sc, UpdateShared* us,
                                 unsigned long long* probes) {
  int nabs = 0, err = 0, dup = 0;
  uint32_t pmin = STAMP_NONE;
  for (int k = threadIdx.x; k < nb; k += NT) {
    const uint64_t h = hbuf[k];
    uint32_t fr;
    const uint32_t sl = table_find_free(t, h, &err, &fr);
    sc.slot[k] = sl;
    sc.fslot[k] = fr;
    uint32_t st = STAMP_NONE;
    if (sl != SLOT_NONE) {
      st = __ldcg(t.stamp + sl);
      pmin = min(pmin, st);
    } else {
      nabs++;
    }
    sc.pst[k] = st;
    sc.evk[k] = 0;
    if (DETECT_DUP) sc.owner[k] = dup_claim(sc, h, &dup);
  }
  nabs = __reduce_add_sync(FULL_MASK, (unsigned)nabs);
  pmin = __reduce_min_sync(FULL_MASK, pmin);
  if ((threadIdx.x & 31) == 0) {
    if (nabs) atomicAdd(&us->n_absent, nabs);
    if (pmin != STAMP_NONE) atomicMin(&us->pmin, pmin);
  }
  if (err) us->err = RS_ERR_TIMEOUT;
  if (dup) us->dup = 1;
  if (threadIdx.x == 0) atomicAdd(probes, (unsigned long long)nb);
  grp_bar<NT>();
  if (DETECT_DUP)
    for (int k = threadIdx.x; k < nb; k += NT)
      if (sc.owner[k] >= 0) sc.dupset[sc.owner[k]] = 0ull;
}

// Claims table slot x for one insert of this update in the shared-memory set
// (keys x + 1; the set is empty between uses).  Returns the set position
// claimed, or -1 when another block of the request claimed x first.
__device__ __forceinline__ int32_t slot_claim(UpdateScratch& sc, uint32_t x) {
  const unsigned long long key = (unsigned long long)x + 1ull;
  uint32_t d = (x * 0x9E3779B1u) & sc.dupmask;
  for (uint32_t it = 0; it <= sc.dupmask; it++) {
    const unsigned long long prev = atomicCAS(
        reinterpret_cast<unsigned long long*>(sc.dupset + d), 0ull, key);
    if (prev == 0ull) return (int32_t)d;
    if (prev == key) return -1;
    d = (d + 1) & sc.dupmask;
  }
  return -1;
}

// The chosen worker's lookup from slots captured by the probe (no table
// reads): stamps of present blocks, absent count, insert positions.
template <int NT>
__device__ __forceinline__ void cache_lookup_captured(const TableView& t, const uint32_t* pslot,
                                                      const uint32_t* pfree, int nb,
                                                      UpdateScratch& sc, UpdateShared* us) {
  int nabs = 0;
  uint32_t pmin = STAMP_NONE;
  for (int k = threadIdx.x; k < nb; k += NT) {
    const uint32_t sl = pslot[k];
    sc.slot[k] = sl;
    sc.fslot[k] = pfree[k];
    sc.evk[k] = 0;
    uint32_t st = STAMP_NONE;
    if (sl != SLOT_NONE) {
      st = __ldcg(t.stamp + sl);
      pmin = min(pmin, st);
    } else {
      nabs++;
    }
    sc.pst[k] = st;
  }
  nabs = __reduce_add_sync(FULL_MASK, (unsigned)nabs);
  pmin = __reduce_min_sync(FULL_MASK, pmin);
  if ((threadIdx.x & 31) == 0) {
    if (nabs) atomicAdd(&us->n_absent, nabs);
    if (pmin != STAMP_NONE) atomicMin(&us->pmin, pmin);
  }
  grp_bar<NT>();
}

// Gathers live log entries starting at meta->head until `want` are held
// (or the log ends).  Continues from us->gathered entries already held.
// Beside each entry's stamp, the first entries' buckets are read too (same
// round trip): an entry whose bucket holds an EMPTY key is marked
// VSLOT_EMPTY_OK, and evicting it may leave an EMPTY instead of a tombstone.
constexpr uint32_t VSLOT_EMPTY_OK = 0x80000000u;

template <int NT>
__device__ __forceinline__ void gather_live(const TableView& t, const CacheMeta* meta, uint32_t* pos,
                            uint32_t want, UpdateScratch& sc, UpdateShared* us, int* warp_tot) {
  const uint32_t T = meta->T;
  uint32_t have = us->gathered;
  uint32_t p0 = *pos;
  while (have < want && p0 < T) {
    const uint32_t p = p0 + threadIdx.x;
    bool live = false, empty_ok = false;
    uint32_t x = 0;
    if (p < T) {
      x = t.log[p & t.rmask];
      // buckets of the entries likely to become victims (dead entries
      // interleave, hence the margin)
      const bool look = threadIdx.x < 2 * (want - have) + 32;
      uint64_t v[BUCKET];
      if (look) ld_bucket(t.keys, x / BUCKET, v);
      live = __ldcg(t.stamp + x) == p;
      if (look) {
#pragma unroll
        for (int q = 0; q < BUCKET; q++) empty_ok |= v[q] == KEY_EMPTY;
      }
    }
    int tot;
    const int r = cta_rank<NT>(live, warp_tot, &tot);
    if (live && have + r < want) {
      sc.vslot[have + r] = x | (empty_ok ? VSLOT_EMPTY_OK : 0u);
      sc.vt[have + r] = p;
    }
    have = min(want, have + (uint32_t)tot);
    p0 += NT;
  }
  grp_bar<NT>();
  if (threadIdx.x == 0) {
    us->gathered = have;
    *pos = p0;
  }
  grp_bar<NT>();
}

// The chosen worker's update inputs from the probe's captured slots, in one
// round of loads: the stamps of the present blocks and, for the nabs - free
// victims this request needs, the first log entries after the head with
// their stamps and buckets (as gather_live's first pass).  us must be reset.
template <int NT>
__device__ __forceinline__ void cache_prepare_captured(const TableView& t, const CacheMeta* meta,
                                                       uint32_t K, const uint32_t* pslot,
                                                       const uint32_t* pfree, int nb, int nabs,
                                                       UpdateScratch& sc, UpdateShared* us,
                                                       int* warp_tot, uint32_t* scan_pos) {
  const uint32_t size = meta->size, T = meta->T, head = meta->head;
  const uint32_t free_slots = K - size;
  const uint32_t E0 = (uint32_t)nabs > free_slots ? (uint32_t)nabs - free_slots : 0u;
  // the log entries go out first ...
  const uint32_t p = head + threadIdx.x;
  const bool gp = E0 > 0 && p < T;
  uint32_t x = 0;
  if (gp) x = t.log[p & t.rmask];
  // ... then the present blocks' stamps, which do not depend on them
  uint32_t pmin = STAMP_NONE;
  for (int k = threadIdx.x; k < nb; k += NT) {
    const uint32_t sl = pslot[k];
    sc.slot[k] = sl;
    sc.fslot[k] = pfree[k];
    sc.evk[k] = 0;
    uint32_t st = STAMP_NONE;
    if (sl != SLOT_NONE) {
      st = __ldcg(t.stamp + sl);
      pmin = min(pmin, st);
    }
    sc.pst[k] = st;
  }
  // stamps and buckets of the log entries
  bool live = false, empty_ok = false;
  if (gp) {
    const bool look = threadIdx.x < 2 * E0 + 32;
    uint64_t v[BUCKET];
    if (look) ld_bucket(t.keys, x / BUCKET, v);
    live = __ldcg(t.stamp + x) == p;
    if (look) {
#pragma unroll
      for (int q = 0; q < BUCKET; q++) empty_ok |= v[q] == KEY_EMPTY;
    }
  }
  pmin = __reduce_min_sync(FULL_MASK, pmin);
  if ((threadIdx.x & 31) == 0 && pmin != STAMP_NONE) atomicMin(&us->pmin, pmin);
  int tot;
  const int r = cta_rank<NT>(live, warp_tot, &tot);
  if (live && (uint32_t)r < E0) {
    sc.vslot[r] = x | (empty_ok ? VSLOT_EMPTY_OK : 0u);
    sc.vt[r] = p;
  }
  if (threadIdx.x == 0) {
    us->n_absent = nabs;
    us->gathered = min(E0, (uint32_t)tot);
    *scan_pos = head + NT;
  }
  grp_bar<NT>();
}

// Applies one request's block list to the chosen worker's cache: exact LRU
// semantics of touching blocks 0..nb-1 in order (hits -> most recent, misses
// inserted, the least-recent entry evicted whenever the cache is full).
// Returns through us: n_victims, n_ins; updates meta.  CTA-wide.
// With `pregathered`, cache_prepare_captured has already gathered the first
// entries (us->gathered, *scan_pos).
template <int NT>
__device__ __forceinline__ void cache_apply(const TableView& t, CacheMeta* meta, uint32_t K, const uint64_t* hbuf,
                            int nb, UpdateScratch& sc, UpdateShared* us, int* warp_tot,
                            uint32_t* scan_pos, bool pregathered = false) {
  const uint32_t size = meta->size;
  const int nabs = us->n_absent;
  const uint32_t free_slots = K - size;
  const uint32_t E0 = (uint32_t)nabs > free_slots ? (uint32_t)nabs - free_slots : 0u;
  if (!pregathered) {
    if (threadIdx.x == 0) {
      us->gathered = 0;
      *scan_pos = meta->head;
    }
    grp_bar<NT>();
  }
  if (E0 > 0 && us->gathered < E0) gather_live<NT>(t, meta, scan_pos, E0, sc, us, warp_tot);
  if (E0 > 0 && us->gathered < E0) {   // fewer live entries than the size says
    if (threadIdx.x == 0) us->err = RS_ERR_TIMEOUT;
    grp_bar<NT>();
    return;
  }
  const bool fast = E0 == 0 || us->pmin > sc.vt[E0 - 1];
  if (fast) {
    for (int k = threadIdx.x; k < nb; k += NT) sc.kind[k] = sc.slot[k] == SLOT_NONE;
    for (uint32_t v = threadIdx.x; v < E0; v += NT) sc.victim[v] = (int32_t)v;
    if (threadIdx.x == 0) us->n_victims = (int)E0;
    grp_bar<NT>();
  } else {
    // exact sequential emulation over the first live entries (gathered again
    // from the head: the first pass dropped live entries past the E0-th)
    const uint32_t want = min(size, 2u * (uint32_t)nb);
    grp_bar<NT>();
    if (threadIdx.x == 0) {
      us->gathered = 0;
      *scan_pos = meta->head;
    }
    grp_bar<NT>();
    gather_live<NT>(t, meta, scan_pos, want, sc, us, warp_tot);
    const uint32_t G = us->gathered;
    for (uint32_t p = threadIdx.x; p < G; p += NT) {
      sc.owner[p] = -1;
      sc.touched[p] = 0;
    }
    grp_bar<NT>();
    const uint32_t last = G ? sc.vt[G - 1] : 0u;
    for (int k = threadIdx.x; k < nb; k += NT) {
      const uint32_t st = sc.pst[k];
      if (st != STAMP_NONE && G && st <= last) {
        uint32_t lo = 0, hi = G;   // vt is increasing: lower bound of st
        while (lo < hi) {
          const uint32_t mid = (lo + hi) >> 1;
          if (sc.vt[mid] < st) lo = mid + 1; else hi = mid;
        }
        sc.owner[lo] = k;
      }
    }
    grp_bar<NT>();
    if (threadIdx.x == 0) {
      uint32_t ptr = 0, sz = size;
      int E = 0;
      // position of each present block inside the gathered list (or none)
      for (int k = 0; k < nb; k++) {
        const bool present = sc.slot[k] != SLOT_NONE && !sc.evk[k];
        if (present) {
          sc.kind[k] = 0;
          const uint32_t st = sc.pst[k];
          if (G && st <= last) {
            uint32_t lo = 0, hi = G;
            while (lo < hi) {
              const uint32_t mid = (lo + hi) >> 1;
              if (sc.vt[mid] < st) lo = mid + 1; else hi = mid;
            }
            sc.touched[lo] = 1;
          }
        } else {
          sc.kind[k] = 1;
          if (sz == K) {
            while (ptr < G && sc.touched[ptr]) ptr++;
            if (ptr >= G) { us->err = RS_ERR_TIMEOUT; break; }
            sc.victim[E++] = (int32_t)ptr;
            if (sc.owner[ptr] >= 0) sc.evk[sc.owner[ptr]] = 1;
            ptr++;
          } else {
            sz++;
          }
        }
      }
      us->n_victims = E;
      us->slow = 1;
    }
    grp_bar<NT>();
  }
  const int E = us->n_victims;
  // evictions first, then inserts, then stamps and log.  A lookup scans whole
  // buckets and stops at the first bucket holding an EMPTY key; a bucket that
  // holds one has held one since the last rebuild (slots only become EMPTY
  // here, and only in such buckets), so no key has overflowed past it and the
  // evicted key may become EMPTY.  Elsewhere it becomes a tombstone.
  int ntomb = 0;
  for (int v = threadIdx.x; v < E; v += NT) {
    const uint32_t xv = sc.vslot[sc.victim[v]];
    const uint32_t x = xv & ~VSLOT_EMPTY_OK;
    const bool tomb = (xv & VSLOT_EMPTY_OK) == 0u;
    t.keys[x] = tomb ? KEY_TOMB : KEY_EMPTY;
    t.stamp[x] = STAMP_NONE;
    ntomb += tomb;
  }
  ntomb = __reduce_add_sync(FULL_MASK, (unsigned)ntomb);
  if ((threadIdx.x & 31) == 0 && ntomb) atomicAdd(&us->n_tomb, ntomb);
  const uint32_t T = meta->T;
  int nins = 0, recl = 0, err = 0;
  // inserts at the positions the lookup saw free: this CTA alone writes the
  // table, so a shared-memory claim per slot settles blocks that saw the same
  // position and the key is stored plainly; the others insert after the
  // barrier, along their probe path.  No barrier from the evictions is
  // needed: a position seen free is not a victim (victims hold keys), and the
  // stamps and the probing inserts come after the barrier below.
  for (int k = threadIdx.x; k < nb; k += NT) {
    if (!sc.kind[k]) continue;
    const uint32_t fr = sc.fslot[k];
    uint32_t sl = SLOT_NONE;
    int32_t cl = -1;
    if (fr != SLOT_NONE) {
      const uint32_t x = fr & ~FREE_TOMB;
      cl = slot_claim(sc, x);
      if (cl >= 0) {
        t.keys[x] = hbuf[k];
        sl = x;
        recl += (fr & FREE_TOMB) != 0;
      }
    }
    sc.slot[k] = sl;
    sc.pst[k] = (uint32_t)cl;   // pst is not needed past the decision: the claim to release
    nins++;
  }
  grp_bar<NT>();
  for (int k = threadIdx.x; k < nb; k += NT) {
    uint32_t sl = sc.slot[k];
    if (sc.kind[k]) {
      const int32_t cl = (int32_t)sc.pst[k];
      if (cl >= 0) sc.dupset[cl] = 0ull;
      if (sl == SLOT_NONE) {
        int wt = 0;
        sl = table_insert(t, hbuf[k], &wt, &err);
        recl += wt;
        sc.slot[k] = sl;
      }
    }
    if (sl != SLOT_NONE) {
      t.stamp[sl] = T + (uint32_t)k;
      t.log[(T + (uint32_t)k) & t.rmask] = sl;
    }
  }
  nins = __reduce_add_sync(FULL_MASK, (unsigned)nins);
  recl = __reduce_add_sync(FULL_MASK, (unsigned)recl);
  if ((threadIdx.x & 31) == 0) {
    if (nins) atomicAdd(&us->n_ins, nins);
    if (recl) atomicAdd(&us->reclaimed, recl);
  }
  if (err) us->err = RS_ERR_TIMEOUT;
  grp_bar<NT>();
  // (the caller's next barrier orders this with any later reader of meta)
  if (threadIdx.x == 0) {
    meta->tombs = meta->tombs + (uint32_t)us->n_tomb - (uint32_t)us->reclaimed;
    meta->size = meta->size + (uint32_t)us->n_ins - (uint32_t)E;
    if (E > 0) meta->head = sc.vt[sc.victim[E - 1]] + 1;
    meta->T = T + (uint32_t)nb;
  }
}

// ---------------------------------------------------------------- frequency eviction
//
// The KV Block Manager's rule (§2.2) in its two-class form: frequency 1 on
// insertion, doubled on a hit (at most fmax), lowered by 1 per decay step and
// never below 1; a block at frequency 1 is cold, at 2 or more hot (eligible
// for promotion).  The victim is the least recently used cold block, else the
// least recently used block.  A slot keeps the frequency lazily as e, the
// decay step from which it is back at 1: at step D the frequency is
// max(1, e - D + 1) and the block is cold iff e <= D.  Insertion sets e = D.
// The log stays in recency order, so the victims are the first live cold
// entries after the head; FreqMeta::fscan/fmin let a search skip a prefix of
// hot entries it has already passed.

// e after a hit at decay step D
__device__ __forceinline__ uint32_t freq_hit(uint32_t e, uint32_t D, uint32_t fmax) {
  const uint32_t f = e > D ? e - D + 1u : 1u;
  const uint32_t f2 = 2u * f < fmax ? 2u * f : fmax;
  return D + f2 - 1u;
}

// Where a victim search starts: fscan while the hot entries passed there
// are still hot, else the head.
__device__ __forceinline__ uint32_t freq_start(const CacheMeta* meta, const FreqMeta* fm,
                                               uint32_t D) {
  return D < fm->fmin ? fm->fscan : meta->head;
}

// The first `want` live cold log entries from *pos on (as gather_live; slot
// with VSLOT_EMPTY_OK, position).  The live hot entries passed on the way
// lower fs->femin (their least e) and fs->fhot (their first position); hot
// entries of the last chunk past the last victim count too, which only makes
// the next search start earlier.
template <int NT>
__device__ __forceinline__ void gather_cold(const TableView& t, const CacheMeta* meta, uint32_t* pos,
                                            uint32_t want, uint32_t D, UpdateScratch& sc,
                                            UpdateShared* us, FreqShared* fs, int* warp_tot) {
  const uint32_t T = meta->T;
  uint32_t have = us->gathered;
  uint32_t p0 = *pos;
  uint32_t he = 0xFFFFFFFFu, hp = 0xFFFFFFFFu;
  while (have < want && p0 < T) {
    const uint32_t p = p0 + threadIdx.x;
    bool cold = false, empty_ok = false;
    uint32_t x = 0;
    if (p < T) {
      x = t.log[p & t.rmask];
      const bool look = threadIdx.x < 2 * (want - have) + 32;
      uint64_t v[BUCKET];
      if (look) ld_bucket(t.keys, x / BUCKET, v);
      const bool live = __ldcg(t.stamp + x) == p;
      const uint32_t e = __ldcg(t.fexp + x);
      cold = live && e <= D;
      if (live && e > D) {
        he = min(he, e);
        hp = min(hp, p);
      }
      if (look) {
#pragma unroll
        for (int q = 0; q < BUCKET; q++) empty_ok |= v[q] == KEY_EMPTY;
      }
    }
    int tot;
    const int r = cta_rank<NT>(cold, warp_tot, &tot);
    if (cold && have + r < want) {
      sc.vslot[have + r] = x | (empty_ok ? VSLOT_EMPTY_OK : 0u);
      sc.vt[have + r] = p;
    }
    have = min(want, have + (uint32_t)tot);
    p0 += NT;
  }
  he = __reduce_min_sync(FULL_MASK, he);
  hp = __reduce_min_sync(FULL_MASK, hp);
  if ((threadIdx.x & 31) == 0) {
    if (he != 0xFFFFFFFFu) atomicMin(&fs->femin, he);
    if (hp != 0xFFFFFFFFu) atomicMin(&fs->fhot, hp);
  }
  grp_bar<NT>();
  if (threadIdx.x == 0) {
    us->gathered = have;
    *pos = p0;
  }
  grp_bar<NT>();
}

// The first `want` live hot entries from the head, packed (position << 32 |
// slot) into global scratch `out`, in order; fs->gb = how many.
template <int NT>
__device__ __forceinline__ void gather_hot(const TableView& t, const CacheMeta* meta, uint32_t want,
                                           uint32_t D, uint64_t* out, FreqShared* fs,
                                           int* warp_tot) {
  const uint32_t T = meta->T;
  uint32_t have = 0;
  for (uint32_t p0 = meta->head; have < want && p0 < T; p0 += NT) {
    const uint32_t p = p0 + threadIdx.x;
    bool hot = false;
    uint32_t x = 0;
    if (p < T) {
      x = t.log[p & t.rmask];
      hot = __ldcg(t.stamp + x) == p && __ldcg(t.fexp + x) > D;
    }
    int tot;
    const int r = cta_rank<NT>(hot, warp_tot, &tot);
    if (hot && have + r < want) out[have + r] = ((uint64_t)p << 32) | x;
    have = min(want, have + (uint32_t)tot);
  }
  grp_bar<NT>();
  if (threadIdx.x == 0) fs->gb = have;
  grp_bar<NT>();
}

// As cache_prepare_captured, for frequency eviction: present blocks keep
// their stamp in pst and their e in fslot (an absent block's fslot is its
// insert position); us->pmin = the least stamp of a present cold block; the
// first chunk of cold entries from the search start.  us must be reset.
template <int NT>
__device__ __forceinline__ void cache_prepare_captured_freq(const TableView& t, const CacheMeta* meta,
                                                            const FreqMeta* fm,
                                                            uint32_t K, const uint32_t* pslot,
                                                            const uint32_t* pfree, int nb, int nabs,
                                                            uint32_t D, UpdateScratch& sc,
                                                            UpdateShared* us, FreqShared* fs,
                                                            int* warp_tot, uint32_t* scan_pos) {
  const uint32_t size = meta->size, T = meta->T;
  const uint32_t start = freq_start(meta, fm, D);
  const uint32_t free_slots = K - size;
  const uint32_t E0 = (uint32_t)nabs > free_slots ? (uint32_t)nabs - free_slots : 0u;
  const uint32_t p = start + threadIdx.x;
  const bool gp = E0 > 0 && p < T;
  uint32_t x = 0;
  if (gp) x = t.log[p & t.rmask];
  uint32_t pmin = STAMP_NONE;
  for (int k = threadIdx.x; k < nb; k += NT) {
    const uint32_t sl = pslot[k];
    sc.slot[k] = sl;
    sc.evk[k] = 0;
    uint32_t st = STAMP_NONE, f = pfree[k];
    if (sl != SLOT_NONE) {
      st = __ldcg(t.stamp + sl);
      f = __ldcg(t.fexp + sl);
      if (f <= D) pmin = min(pmin, st);
    }
    sc.pst[k] = st;
    sc.fslot[k] = f;
  }
  bool cold = false, empty_ok = false;
  uint32_t he = 0xFFFFFFFFu, hp = 0xFFFFFFFFu;
  if (gp) {
    const bool look = threadIdx.x < 2 * E0 + 32;
    uint64_t v[BUCKET];
    if (look) ld_bucket(t.keys, x / BUCKET, v);
    const bool live = __ldcg(t.stamp + x) == p;
    const uint32_t e = __ldcg(t.fexp + x);
    cold = live && e <= D;
    if (live && e > D) {
      he = e;
      hp = p;
    }
    if (look) {
#pragma unroll
      for (int q = 0; q < BUCKET; q++) empty_ok |= v[q] == KEY_EMPTY;
    }
  }
  pmin = __reduce_min_sync(FULL_MASK, pmin);
  he = __reduce_min_sync(FULL_MASK, he);
  hp = __reduce_min_sync(FULL_MASK, hp);
  if ((threadIdx.x & 31) == 0) {
    if (pmin != STAMP_NONE) atomicMin(&us->pmin, pmin);
    if (he != 0xFFFFFFFFu) atomicMin(&fs->femin, he);
    if (hp != 0xFFFFFFFFu) atomicMin(&fs->fhot, hp);
  }
  int tot;
  const int r = cta_rank<NT>(cold, warp_tot, &tot);
  if (cold && (uint32_t)r < E0) {
    sc.vslot[r] = x | (empty_ok ? VSLOT_EMPTY_OK : 0u);
    sc.vt[r] = p;
  }
  if (threadIdx.x == 0) {
    us->n_absent = nabs;
    us->gathered = min(E0, (uint32_t)tot);
    fs->fstart = start;
    *scan_pos = start + NT;
  }
  grp_bar<NT>();
}

// After cache_lookup_all: present blocks' e into fslot, us->pmin = the least
// stamp of a present cold block, the search start.
template <int NT>
__device__ __forceinline__ void freq_present(const TableView& t, const CacheMeta* meta,
                                             const FreqMeta* fm, int nb, uint32_t D,
                                             UpdateScratch& sc, UpdateShared* us,
                                             FreqShared* fs, uint32_t* scan_pos) {
  if (threadIdx.x == 0) {
    us->pmin = STAMP_NONE;
    us->gathered = 0;
    fs->fstart = freq_start(meta, fm, D);
    *scan_pos = fs->fstart;
  }
  grp_bar<NT>();
  uint32_t pmin = STAMP_NONE;
  for (int k = threadIdx.x; k < nb; k += NT) {
    const uint32_t sl = sc.slot[k];
    if (sl == SLOT_NONE) continue;
    const uint32_t e = __ldcg(t.fexp + sl);
    sc.fslot[k] = e;
    if (e <= D) pmin = min(pmin, sc.pst[k]);
  }
  pmin = __reduce_min_sync(FULL_MASK, pmin);
  if ((threadIdx.x & 31) == 0 && pmin != STAMP_NONE) atomicMin(&us->pmin, pmin);
  grp_bar<NT>();
}

// Victim codes of the frequency update: >= 0 an index into vslot/vt; -1 a
// block this request inserted and evicts again (nothing to clear); <= -2 the
// slot -code - 2, cleared to a tombstone.
constexpr int32_t VICTIM_OWN_INSERT = -1;

// Binary search of stamp st among n packed (position << 32 | slot) entries
// in increasing position order; the index or -1.
__device__ __forceinline__ int32_t packed_find(const uint64_t* a, uint32_t n, uint32_t st) {
  uint32_t lo = 0, hi = n;
  while (lo < hi) {
    const uint32_t mid = (lo + hi) >> 1;
    if ((uint32_t)(__ldcg(a + mid) >> 32) < st) lo = mid + 1; else hi = mid;
  }
  return lo < n && (uint32_t)(__ldcg(a + lo) >> 32) == st ? (int32_t)lo : -1;
}

// Applies one request's block list to the chosen worker's cache under
// frequency eviction, with the semantics of touching blocks 0..nb-1 in order
// (a hit doubles the frequency and makes the block most recent, a miss
// inserts at frequency 1 after evicting the rule's victim when the cache is
// full).  Fast path: the first E0 live cold entries are the victims when no
// present cold block is older than the last of them.  Otherwise one thread
// replays the sequence over the first 2 nb cold entries (shared scratch), the
// first 2 nb hot ones (global scratch `gtmp`, only when the cold ones run
// out) and the request's own blocks.  CTA-wide; updates meta.
template <int NT>
__device__ __forceinline__ void cache_apply_freq(const TableView& t, CacheMeta* meta, FreqMeta* fm,
                                                 uint32_t K,
                                                 const uint64_t* hbuf, int nb, uint32_t D,
                                                 uint32_t fmax, UpdateScratch& sc,
                                                 UpdateShared* us, FreqShared* fs, int* warp_tot,
                                                 uint32_t* scan_pos, uint64_t* gtmp) {
  const uint32_t size = meta->size;
  const int nabs = us->n_absent;
  const uint32_t free_slots = K - size;
  const uint32_t E0 = (uint32_t)nabs > free_slots ? (uint32_t)nabs - free_slots : 0u;
  if (E0 > 0 && us->gathered < E0) gather_cold<NT>(t, meta, scan_pos, E0, D, sc, us, fs, warp_tot);
  const bool fast = E0 == 0 || (us->gathered >= E0 && us->pmin > sc.vt[E0 - 1]);
  if (fast) {
    for (int k = threadIdx.x; k < nb; k += NT) sc.kind[k] = sc.slot[k] == SLOT_NONE;
    for (uint32_t v = threadIdx.x; v < E0; v += NT) sc.victim[v] = (int32_t)v;
    if (threadIdx.x == 0) us->n_victims = (int)E0;
    grp_bar<NT>();
  } else {
    // list A: the first 2 nb live cold entries from the search start
    const uint32_t want = min(size, 2u * (uint32_t)nb);
    grp_bar<NT>();
    if (threadIdx.x == 0) {
      us->gathered = 0;
      *scan_pos = fs->fstart;
    }
    grp_bar<NT>();
    gather_cold<NT>(t, meta, scan_pos, want, D, sc, us, fs, warp_tot);
    const uint32_t G = us->gathered;
    // list B, when the cold entries ran out: the first 2 nb live hot entries
    if (G < want) {
      gather_hot<NT>(t, meta, want, D, gtmp, fs, warp_tot);
    } else if (threadIdx.x == 0) {
      fs->gb = 0;
    }
    for (uint32_t q = threadIdx.x; q < G; q += NT) {
      sc.owner[q] = -1;
      sc.touched[q] = 0;
    }
    grp_bar<NT>();
    const uint32_t last = G ? sc.vt[G - 1] : 0u;
    for (int k = threadIdx.x; k < nb; k += NT) {
      const uint32_t st = sc.pst[k];
      if (st != STAMP_NONE && G && st <= last && sc.fslot[k] <= D) {
        uint32_t lo = 0, hi = G;
        while (lo < hi) {
          const uint32_t mid = (lo + hi) >> 1;
          if (sc.vt[mid] < st) lo = mid + 1; else hi = mid;
        }
        if (lo < G && sc.vt[lo] == st) sc.owner[lo] = k;
      }
    }
    grp_bar<NT>();
    if (threadIdx.x == 0) {
      const uint32_t GB = fs->gb;
      const bool hits_cold = fmax < 2u;   // a hit at cap 1 leaves the block cold
      uint32_t pa = 0, pb = 0, sz = size;
      int qc = 0, qh = 0, E = 0;
      for (int k = 0; k < nb; k++) {
        const bool present = sc.slot[k] != SLOT_NONE && !sc.evk[k];
        if (present) {
          sc.kind[k] = 0;
          const uint32_t st = sc.pst[k];
          if (sc.fslot[k] <= D) {   // a cold entry: in list A if old enough
            if (G && st <= last) {
              uint32_t lo = 0, hi = G;
              while (lo < hi) {
                const uint32_t mid = (lo + hi) >> 1;
                if (sc.vt[mid] < st) lo = mid + 1; else hi = mid;
              }
              if (lo < G && sc.vt[lo] == st) sc.touched[lo] = 1;
            }
          } else if (GB) {          // a hot entry: in list B if old enough
            const int32_t ib = packed_find(gtmp, GB, st);
            if (ib >= 0) gtmp[ib] |= 0x80000000ull;   // touched
          }
          continue;
        }
        sc.kind[k] = 1;
        if (sz < K) {
          sz++;
          continue;
        }
        // the victim: old cold, own cold, old hot, own hot -- each oldest first
        while (pa < G && sc.touched[pa]) pa++;
        if (pa < G) {
          sc.victim[E++] = (int32_t)pa;
          const int32_t ow = sc.owner[pa];
          if (ow >= 0) {   // a block of this request, evicted before its turn
            sc.evk[ow] = 1;
            sc.fslot[ow] = SLOT_NONE;
          }
          pa++;
          continue;
        }
        while (qc < k && !(sc.kind[qc] == 1 || (hits_cold && sc.kind[qc] == 0))) qc++;
        if (qc < k) {
          if (sc.kind[qc] == 1) {
            sc.kind[qc] = 2;   // inserted and evicted again
            sc.victim[E++] = VICTIM_OWN_INSERT;
          } else {
            sc.kind[qc] = 3;   // hit, then evicted
            sc.victim[E++] = -(int32_t)sc.slot[qc] - 2;
          }
          qc++;
          continue;
        }
        while (pb < GB && (__ldcg(gtmp + pb) & 0x80000000ull)) pb++;
        if (pb < GB) {
          const uint64_t ent = __ldcg(gtmp + pb);
          const uint32_t x = (uint32_t)ent;
          sc.victim[E++] = -(int32_t)x - 2;
          // a present hot block evicted before its turn
          for (int k2 = k + 1; k2 < nb; k2++)
            if (sc.slot[k2] == x && !sc.evk[k2]) {
              sc.evk[k2] = 1;
              sc.fslot[k2] = SLOT_NONE;
            }
          pb++;
          continue;
        }
        while (qh < k && sc.kind[qh] != 0) qh++;
        if (qh < k) {
          sc.kind[qh] = 3;
          sc.victim[E++] = -(int32_t)sc.slot[qh] - 2;
          qh++;
          continue;
        }
        us->err = RS_ERR_TIMEOUT;   // nothing to evict: inconsistent state
        break;
      }
      us->n_victims = E;
      us->slow = 1;
    }
    grp_bar<NT>();
  }
  const int E = us->n_victims;
  int ntomb = 0;
  for (int v = threadIdx.x; v < E; v += NT) {
    const int32_t iv = sc.victim[v];
    if (iv == VICTIM_OWN_INSERT) continue;
    uint32_t x;
    bool tomb = true;
    if (iv >= 0) {
      const uint32_t xv = sc.vslot[iv];
      x = xv & ~VSLOT_EMPTY_OK;
      tomb = (xv & VSLOT_EMPTY_OK) == 0u;
    } else {
      x = (uint32_t)(-(iv + 2));
    }
    t.keys[x] = tomb ? KEY_TOMB : KEY_EMPTY;
    t.stamp[x] = STAMP_NONE;
    ntomb += tomb;
  }
  ntomb = __reduce_add_sync(FULL_MASK, (unsigned)ntomb);
  if ((threadIdx.x & 31) == 0 && ntomb) atomicAdd(&us->n_tomb, ntomb);
  const uint32_t T = meta->T;
  int nins = 0, recl = 0, err = 0;
  for (int k = threadIdx.x; k < nb; k += NT) {
    const int kd = sc.kind[k];
    if (kd == 2) nins++;
    if (kd != 1) continue;
    const uint32_t fr = sc.fslot[k];
    uint32_t sl = SLOT_NONE;
    int32_t cl = -1;
    if (fr != SLOT_NONE) {
      const uint32_t x = fr & ~FREE_TOMB;
      cl = slot_claim(sc, x);
      if (cl >= 0) {
        t.keys[x] = hbuf[k];
        sl = x;
        recl += (fr & FREE_TOMB) != 0;
      }
    }
    sc.slot[k] = sl;
    sc.pst[k] = (uint32_t)cl;
    nins++;
  }
  grp_bar<NT>();
  for (int k = threadIdx.x; k < nb; k += NT) {
    const int kd = sc.kind[k];
    const uint32_t pos = T + (uint32_t)k;
    if (kd >= 2) {   // evicted within this request: its log position stays dead
      t.log[pos & t.rmask] = 0u;
      continue;
    }
    uint32_t sl = sc.slot[k];
    uint32_t e = D;
    if (kd == 1) {
      const int32_t cl = (int32_t)sc.pst[k];
      if (cl >= 0) sc.dupset[cl] = 0ull;
      if (sl == SLOT_NONE) {
        int wt = 0;
        sl = table_insert(t, hbuf[k], &wt, &err);
        recl += wt;
        sc.slot[k] = sl;
      }
    } else {
      e = freq_hit(sc.fslot[k], D, fmax);
    }
    if (sl != SLOT_NONE) {
      t.stamp[sl] = pos;
      t.fexp[sl] = e;
      t.log[pos & t.rmask] = sl;
    }
  }
  nins = __reduce_add_sync(FULL_MASK, (unsigned)nins);
  recl = __reduce_add_sync(FULL_MASK, (unsigned)recl);
  if ((threadIdx.x & 31) == 0) {
    if (nins) atomicAdd(&us->n_ins, nins);
    if (recl) atomicAdd(&us->reclaimed, recl);
  }
  if (err) us->err = RS_ERR_TIMEOUT;
  grp_bar<NT>();
  if (threadIdx.x == 0) {
    meta->tombs = meta->tombs + (uint32_t)us->n_tomb - (uint32_t)us->reclaimed;
    meta->size = meta->size + (uint32_t)us->n_ins - (uint32_t)E;
    if (us->slow) {
      fm->fscan = meta->head;   // the next search starts at the head
      fm->fmin = 0;
    } else if (E > 0) {
      const uint32_t next = sc.vt[E - 1] + 1;
      if (fs->fstart == meta->head) {
        meta->head = min(fs->fhot, next);
        fm->fmin = fs->femin;
      } else {
        fm->fmin = min(fm->fmin, fs->femin);
      }
      fm->fscan = next;
    }
    meta->T = T + (uint32_t)nb;
    freq_reset(fs);
  }
}

}  // namespace rs
