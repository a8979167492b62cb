/*
 * routesim.h -- C ABI of the GB300 (sm_103a) KV-cache-aware routing library.
 *
 * The library computes, on one GPU, the request-routing mechanism that the
 * paper "The Price of Anarchy in Disaggregated Inference" analyses as a
 * congestion game with cache externalities, and its empirical PoA estimator:
 *
 *   - KV block hashing of prompts (full blocks of `block_size` tokens);
 *   - per worker, the cached-prefix length m_ij of each prompt;
 *   - the router cost of Eq. (1), c_j = omega * b_j^prefill + b_j^active (§2.2);
 *   - worker choice by argmin (tau = 0) or softmax sampling, Eq. (2);
 *   - the chosen worker's load and LRU block cache update;
 *   - per-request latency from Eq. (9) with the constants of §6.4;
 *   - the adaptive controller of §6.2-§6.4 (Eq. (10), Eq. (11), Table 2,
 *     Algorithm 1);
 *   - the PoA estimate of Eq. (12) per tumbling window.
 *
 * Conventions (every entry point):
 *   - Plain pointers and sizes only.  "_dev" pointers are CUDA device memory
 *     of the current device, "_host" pointers are host memory.
 *   - The caller owns every buffer it passes; the library owns the context,
 *     its cache tables and its scratch memory.
 *   - Work is ordered on the CUDA stream given to route_init (NULL = legacy
 *     default stream).  Calls that return results in host memory synchronise
 *     that stream before returning; the others only enqueue work.
 *   - Errors are returned as rs_status codes, never by aborting; the context
 *     keeps a message for the last error (route_last_error).  A status other
 *     than RS_OK leaves output buffers unspecified.
 *   - A context may be used by one host thread at a time.
 *
 * Readings of the paper that fix behaviour where it is silent:
 *   - only full blocks are hashed and cached; b^prefill = ceil(L/B) - m_ij and
 *     the overlap o_ij = m_ij / ceil(L/B), where m_ij counts the leading blocks
 *     found in worker j's cache;
 *   - b^active sums ceil((L + O)/B) over the worker's unfinished requests;
 *   - exact LRU eviction; the chosen worker touches the prompt's blocks in order;
 *   - argmin ties go to the lowest worker index; sampling uses Philox4x32-10
 *     with a 24-bit uniform;
 *   - a worker serves at most cap-1 requests at once (the pole of Eq. (9) at
 *     n = cap is never reached); further requests wait in FIFO order.
 */
#ifndef ROUTESIM_H
#define ROUTESIM_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  RS_OK = 0,
  RS_ERR_INVALID = -1,    /* bad argument (pointer, size, alignment, range) */
  RS_ERR_OOM = -2,        /* device or host allocation failed */
  RS_ERR_CAPACITY = -3,   /* a prompt has more full blocks than a worker cache
                             holds, or a fixed-size table would overflow */
  RS_ERR_CUDA = -4,       /* a CUDA runtime call failed (message has details) */
  RS_ERR_TIMEOUT = -5,    /* a bounded device loop gave up (inconsistent state) */
  RS_ERR_STATE = -6,      /* call not valid in the context's current state */
  RS_ERR_COLLISION = -7   /* two blocks of one prompt share a chained hash */
} rs_status;

enum { RS_POLICY_DYNAMO = 0,   /* Eq. (1) cost with the replica's omega, tau */
       RS_POLICY_LOADBAL = 1,  /* coordinated: Eq. (1) with omega = 0, tau = 0 */
       /* Static counterfactual policies of the routing-baselines discussion
        * (§9): they ignore the cache state except through P2C's cost. */
       RS_POLICY_ROUNDROBIN = 2,   /* request i -> worker i mod W */
       RS_POLICY_RANDOM = 3,       /* uniform: floor(u W), u = (Philox x0 >> 8) 2^-24 */
       RS_POLICY_P2C = 4           /* power of two choices: two distinct uniform workers
                                      (x0, x1 of one Philox draw), the lower Eq. (1)
                                      cost wins, ties to the lower index */ };

/* Eviction of the simulated per-worker caches: exact LRU, or the KV Block
 * Manager's frequency rule (§2.2; see rs_replica_params.eviction). */
enum { RS_EVICT_LRU = 0, RS_EVICT_FREQ = 1 };

enum { RS_MEM_DEVICE = 0, RS_MEM_HOST = 1 };

/* Model and controller constants.  rs_config_default() fills the paper's:
 * block 16, a = 0.005, b = 0.020, d = 0.010, beta = 2, C_j = 64, w_c = 0.015
 * (§6.4); Delta = 5 s, alpha = 0.3, theta1 = 0.3 s, theta2 = 2 s (70B, §6.2);
 * hysteresis k = 3 samples, epsilon = 0.1 theta; Table 2 regime parameters
 * (Transition tau 0.7 / omega 1.0, Saturated tau 0.8 / omega 0.1); PoA
 * window 5 s; itl 0.012 s per output token. */
typedef struct {
  int32_t W;               /* workers (1..64) */
  int32_t block_size;      /* tokens per KV block; must be 16 */
  int64_t cache_blocks;    /* LRU capacity per worker, blocks (1 .. 2^24) */
  uint64_t hash_seed;      /* h_{-1} of the block-hash chain */
  float omega, tau;        /* route_batch router parameters (>= 0) */
  uint64_t seed;           /* route_batch Philox key */
  double lat_a, lat_b, lat_d;   /* Eq. (9) constants (beta fixed at 2) */
  int32_t cap;             /* C_j, pole of Eq. (9) (2..65535); cap-1 service slots */
  int32_t hyst_k;          /* controller hysteresis samples (>= 1) */
  double w_c;              /* cache weight of the §6.4 cost matrix */
  double itl;              /* seconds per output token */
  double dt;               /* controller polling interval Delta, s (> 0) */
  double alpha;            /* EWMA weight of Eq. (10), in (0, 1] */
  double theta1, theta2;   /* Eq. (11) thresholds, s */
  double eps_frac;         /* hysteresis margin epsilon = eps_frac * theta */
  float regime_tau[3];     /* Table 2; entry 0 unused (replica's own tau) */
  float regime_omega[3];   /* Table 2; entry 0 unused (replica's own omega) */
  double poa_window;       /* window of Eq. (12), s (> 0) */
  /* Game 2 tiers (§4.2, Eq. kv-cost), simulation only.  tiered = 1 gives
   * every simulated worker the exclusive tiers G1 (cache_blocks), G2
   * (tier_k2) and G3 (tier_k3 blocks, each >= 0): an access brings a block
   * to G1, and a full tier hands its least recently used block to the next
   * (the last drops it), i.e. one recency stack of cache_blocks + tier_k2 +
   * tier_k3 blocks cut into three bands.  Routing (Eq. (1)'s cached prefix)
   * sees G1.  Every routed request is charged per full block on its worker i
   * tier_alpha[t] for its own tier t, else the cheapest d(i, j) +
   * tier_alpha[t] over copies on other workers j (d = tier_d_near when i and
   * j share a node of tier_node workers, else tier_d_far; ties: same node,
   * then the lower tier), else tier_gamma (recomputation); requires
   * 0 <= alpha_G1 < alpha_G2 < alpha_G3 < gamma < inf, finite d >= 0,
   * tier_node >= 1, W * (longest prompt's full blocks) <= 2048, and LRU
   * replicas.  Defaults (the paper gives no values): off, alpha 1 / 4 / 20,
   * gamma 100, d 2 / 10, one worker per node.  route_batch ignores tiers. */
  int32_t tiered, tier_node;
  int64_t tier_k2, tier_k3;
  double tier_alpha[3];
  double tier_gamma, tier_d_near, tier_d_far;
} rs_config;

/* Fills *cfg with the paper's constants (see above), W = 3, cache 65536. */
void rs_config_default(rs_config* cfg);

typedef struct rs_ctx rs_ctx;

/* Creates a context on the current CUDA device.  n_instances live routers
 * (route_batch state: W caches of cache_blocks each, and W load counters) are
 * allocated and cleared; n_instances may be 0 for simulation-only use.
 * cuda_stream: a cudaStream_t (or NULL).  On success *out owns the context. */
rs_status route_init(rs_ctx** out, const rs_config* cfg, int32_t n_instances, void* cuda_stream);

/* Frees the context and all library-owned device memory (synchronises). */
void route_destroy(rs_ctx* ctx);

/* Message of the last failing call on ctx ("" if none); valid until the next
 * call on ctx.  route_last_error(NULL) reports route_init failures. */
const char* route_last_error(const rs_ctx* ctx);

/* KV block hashing (§2.2 "token blocks"; the hash is this library's choice):
 * the block content g_k folds the block's 8 little-endian 64-bit token pairs
 * w in order, x = (x ^ w) * 0xBF58476D1CE4E5B9, x ^= x >> 32, from
 * x = 0x9E3779B97F4A7C15 ^ 16, then takes the SplitMix64 finalizer of x; the
 * prefix is H_k = H_{k-1} * 0x94D049BB133111EB + g_k (mod 2^64) with
 * H_{-1} = cfg.hash_seed, so equal prompt prefixes give equal hashes and a
 * change in block j changes every H_k, k >= j; the stored hash is
 * h_k = mix(H_k ^ k), with 0 and 1 mapped to 2 and 3.
 * tokens_dev: int32, 16-byte aligned, readable for round_up(offsets[n_req], 4)
 * entries.  offsets_dev: int64 [n_req + 1], non-decreasing, offsets[0] >= 0.
 * hashes_dev: uint64, request i's k-th hash at floor(offsets[i]/16) + k for
 * k < floor(L_i/16); floor(offsets[n_req]/16) entries suffice.  Asynchronous. */
rs_status route_hash_blocks(rs_ctx* ctx, const int32_t* tokens_dev, const int64_t* offsets_dev,
                            int64_t n_req, uint64_t* hashes_dev);

/* Repeated block hashes within a prompt.  A cache keyed by block hash (§2.2)
 * cannot tell apart two blocks of one prompt whose chained hashes are equal
 * (a 64-bit collision); simulate_replicas stops a replica at such a request
 * with RS_ERR_COLLISION, using these flags.  For each request i:
 *   flags_dev[i] = 1  two of its floor(L_i/16) block hashes are equal,
 *                  0  all are distinct (or it has fewer than two blocks),
 *                  2  it has more than max_blocks blocks (not checked).
 * hashes_dev/offsets_dev: the layout route_hash_blocks writes (request i's
 * k-th hash at floor(offsets[i]/16) + k; every hash >= 2, as that entry
 * produces).  flags_dev: uint8 [n_req], caller-owned.  max_blocks in
 * [1, 8192] (one shared-memory set of 2^ceil(log2(2 max_blocks)) hashes per
 * warp), else RS_ERR_INVALID.  Asynchronous on the context stream. */
rs_status route_dup_flags(rs_ctx* ctx, const uint64_t* hashes_dev, const int64_t* offsets_dev,
                          int64_t n_req, int64_t max_blocks, uint8_t* flags_dev);

/* Live routing (Algorithm 1 without the controller): routes n_req requests of
 * one router instance in array order, exactly as n_req calls of size one.
 * For each request: Eq. (1) cost with cfg.omega, the instance's active blocks
 * and its caches; Eq. (2) choice with cfg.tau (Philox counter = the
 * instance's running request ordinal); the chosen worker's cache is updated
 * and its active blocks grow by ceil((L + O)/16).
 * tokens_dev/offsets_dev as in route_hash_blocks; out_len_dev int32 [n_req];
 * worker_out_dev int32 [n_req]; cost_out_dev float [n_req*W] and
 * prefix_out_dev int32 [n_req*W] (m_ij) may be NULL.  Asynchronous; errors
 * found on the device (capacity, collision) are reported by the next
 * synchronising call on ctx. */
rs_status route_batch(rs_ctx* ctx, int32_t instance, const int32_t* tokens_dev,
                      const int64_t* offsets_dev, int32_t n_req, const int32_t* out_len_dev,
                      int32_t* worker_out_dev, float* cost_out_dev, int32_t* prefix_out_dev);

/* Cached prefixes of a batch against one router instance, read-only (§2.2, the
 * b^prefill input of Eq. (1), for many requests at once): prefix_out_dev[i*W
 * + j] = m_ij, the leading full blocks of request i found in worker j's
 * cache.  Every request sees the same snapshot -- no cache, load or ordinal
 * changes -- so a row equals the prefix_out row route_batch would report for
 * that request if it were routed next.  Prompts longer than the cache are
 * probed too (m_ij <= cache_blocks).  tokens_dev/offsets_dev as in
 * route_hash_blocks; prefix_out_dev int32 [n_req*W], caller-owned.  Reads
 * offsets_dev[n_req] (a synchronising copy), then asynchronous. */
rs_status route_probe(rs_ctx* ctx, int32_t instance, const int32_t* tokens_dev,
                      const int64_t* offsets_dev, int64_t n_req, int32_t* prefix_out_dev);

/* Completion of n requests of an instance: active blocks of worker_dev[i]
 * drop by blocks_dev[i] (int32 each); a counter never goes below zero.
 * Entries with a worker outside [0, W) are skipped and the call returns
 * RS_ERR_INVALID.  Synchronises. */
rs_status route_release(rs_ctx* ctx, int32_t instance, const int32_t* worker_dev,
                        const int32_t* blocks_dev, int32_t n);

/* Active blocks of an instance's W workers into active_host (int64 [W]).
 * Synchronises (reports pending device errors of route_batch). */
rs_status route_active(rs_ctx* ctx, int32_t instance, int64_t* active_host);

/* One request trace.  tokens: int32, 16-byte aligned, readable for
 * round_up(offsets[n_req], 4) entries; offsets: int64 [n_req + 1];
 * release: float64 [n_req] client release times (s, non-decreasing);
 * out_len: int32 [n_req] output tokens (>= 0).
 * hashes: used only when tokens is NULL.  A trace whose tokens are too many to
 * hold at once (the prompts enter the router only as the block hashes of
 * §2.2, which Eq. (1)'s cached-prefix term is computed from) is given by its
 * block hashes instead, as route_hash_blocks writes them for these offsets:
 * request i's k-th hash at floor(offsets[i]/16) + k, floor(offsets[n_req]/16)
 * entries, 8-byte aligned, in trace_mem like the other arrays.  Such a trace
 * skips the hashing step; everything else is the same.  route_hash_blocks
 * may produce the hashes chunk by chunk: hashing requests i0 .. i1-1 from a
 * token buffer that starts at token b = 16 * floor(offsets[i0] / 16), with
 * offsets rebased by b and the output pointer advanced by b / 16, writes
 * exactly their entries of this layout. */
typedef struct {
  const int32_t* tokens;
  const int64_t* offsets;
  const double* release;
  const int32_t* out_len;
  int64_t n_req;
  const uint64_t* hashes;
} rs_trace;

/* One replica of the closed-loop simulation (§7.4 client holding C requests
 * in flight) on trace `trace`, routing its first n_req requests. */
typedef struct {
  int32_t trace;        /* index into the traces array */
  int32_t C;            /* concurrency, 1 .. 65535 */
  int32_t policy;       /* RS_POLICY_* */
  int32_t controller;   /* 1: adaptive controller on (DYNAMO only) */
  float omega, tau;     /* Below-regime router parameters (>= 0) */
  uint64_t seed;        /* Philox key of this replica's sampling stream */
  int64_t n_req;        /* 0 .. trace n_req */
  /* Load-spike schedule (Experiment 3, §7.7): the client holds C requests in
   * flight before c_t1, c_mid on [c_t1, c_t2) and c_end from c_t2 on (s of
   * simulated time).  c_mid = 0: C throughout (the times are ignored). */
  double c_t1, c_t2;
  int32_t c_mid, c_end;
  /* Cache eviction (RS_EVICT_*).  RS_EVICT_FREQ is the KV Block Manager's
   * frequency rule (§2.2): a block's frequency is 1 when inserted, doubles
   * on a hit up to freq_max (1 .. 2^20) and drops by 1 per decay step of
   * decay_s seconds of simulated time (> 0, finite; step floor(a_i / decay_s)
   * at request i's arrival), never below 1.  Frequency 1 is cold, 2 and more
   * hot; the victim is the least recently used cold block, or the least
   * recently used block when all are hot.  freq_max = 1 is exact LRU.
   * Both fields are ignored under RS_EVICT_LRU. */
  int32_t eviction, freq_max;
  double decay_s;
} rs_replica_params;

typedef struct {
  int32_t status;           /* RS_OK or the replica's error */
  int32_t final_regime;     /* 0 Below, 1 Transition, 2 Saturated */
  int64_t n_routed;
  double sum_ttft, sum_e2e, makespan;     /* s */
  double poa_total;         /* Eq. (12): sum of window numerators / sum of OPTs */
  int64_t n_windows;        /* windows spanned (including empty ones) */
  int64_t near_ties;        /* top-two costs within 1e-6 relative */
  int64_t exact_ties;       /* top-two costs equal */
  int64_t sampled;          /* decisions drawn with tau > 0 */
  int64_t near_boundary;    /* draws within 1e-6 S of a cumulative boundary */
  int64_t hit_blocks;       /* sum of m_ij on the chosen worker */
  int64_t inserted_blocks, evicted_blocks;
  int64_t ticks, regime_switches;
  int32_t max_regime, reserved0;
  int64_t ticks_in_regime[3];
  double final_ewma;        /* -1 if no sample */
  int64_t probes;           /* hash-table lookups issued (work counter) */
  int64_t probe_blocks;     /* sum over decisions and workers of min(m_ij + 1, nb_i):
                               the lookups a first-miss probe needs */
  int64_t hashed_blocks;    /* sum of nb_i (full blocks) over routed requests */
  int64_t slow_path;        /* updates that needed the exact sequential path */
  int64_t rebuilds;         /* table/log compactions */
  double first_switch_t;    /* time of the first controller regime switch, -1 if none */
  double poa_static;        /* the realized assignment under the frozen cost model of
                               §6.4: sum over windows of sum_i c_{i, worker(i)} over
                               the sum of OPTs (the static counterfactual of §9) */
  /* KV-cache pressure (the regime-transition proposition of §5.3, rho =
   * resident blocks of every tier / (W cache_blocks)): arrival time of the
   * first request whose update pushed a block out of a G1 cache and rho just
   * after that update (-1, -1 if none); rho at the end */
  double first_evict_t, rho_first_evict, rho_end;
  /* Game 2 accounting (tiered, else 0): full blocks of routed requests found
   * in their worker's own G1 / G2 / G3, on another worker, nowhere; summed
   * Eq. kv-cost */
  int64_t kv_g1, kv_g2, kv_g3, kv_remote, kv_recompute;
  double kv_cost;
} rs_replica_result;

/* Per-request records, device memory, each pointer may be NULL.  Replica r's
 * requests start at row R_r = sum of n_req of replicas before r; per-worker
 * arrays hold W entries per row. */
typedef struct {
  int32_t* worker;        /* chosen worker sigma_i */
  double* arrival;        /* a_i */
  double* start;          /* service start */
  double* first_token;    /* start + Eq. (9) latency - w_c o */
  double* completion;     /* first token + O_i * itl */
  double* ttft;           /* first token - a_i */
  int32_t* nbt;           /* ceil(L_i / 16) */
  uint16_t* n_frozen;     /* [rows*W] min(in-service_j at a_i + 1, cap - 1) */
  uint16_t* prefix;       /* [rows*W] m_ij */
  float* cost;            /* [rows*W] Eq. (1) cost at the decision */
  double* kv_cost;        /* [rows] Eq. kv-cost of the request on its worker (tiered; optional) */
} rs_records;

enum { RS_SIM_NO_POA = 1 };   /* flags of simulate_replicas */

/* Runs n_replicas independent replicas (one per CTA) and, unless
 * RS_SIM_NO_POA, the Eq. (12) estimate per replica.  traces: host array of
 * n_traces descriptors whose pointers are in trace_mem (RS_MEM_DEVICE, or
 * RS_MEM_HOST: the library copies them to the device first).  params: host
 * array.  results_host: n_replicas entries, written before returning.
 * records: NULL or a host struct of device pointers (see rs_records).
 * Synchronises.  Per-replica failures are reported in results_host[r].status;
 * the call returns the first non-RS_OK replica status, or an argument error. */
rs_status simulate_replicas(rs_ctx* ctx, const rs_trace* traces, int32_t n_traces,
                            int32_t trace_mem, const rs_replica_params* params,
                            int32_t n_replicas, rs_replica_result* results_host,
                            const rs_records* records, int32_t flags);

/* Eq. (12) on caller records of one replica (device pointers, n rows,
 * cfg.W columns in the per-worker arrays; worker < 0 marks rows to skip).
 * Windows are [k w, (k+1) w) of completion time, w = cfg.poa_window; every
 * window up to the last routed completion is computed, however sparse the
 * records (the window scratch is sized from the records on the device first).
 * numer_host/opt_host/count_host: NULL or arrays of *n_windows_inout entries;
 * on return *n_windows_inout = windows spanned (if larger than the capacity
 * given, only that many are written).  poa_total_host: sum numer / sum OPT.
 * RS_ERR_INVALID when a routed row's completion is negative or not finite;
 * RS_ERR_CAPACITY beyond 2^31 - 2 windows.  Synchronises. */
rs_status poa_estimate(rs_ctx* ctx, const rs_records* records, int64_t n, double* numer_host,
                       double* opt_host, int64_t* count_host, int64_t* n_windows_inout,
                       double* poa_total_host);

/* Cache contents of one worker, least- to most-recently used, into keys_host
 * (capacity entries); *size = entries held.  source 0: live router instance
 * `index`; source 1: replica `index` of the last simulate_replicas call.
 * Synchronises. */
rs_status route_cache_dump(rs_ctx* ctx, int32_t source, int32_t index, int32_t worker,
                           uint64_t* keys_host, int64_t capacity, int64_t* size);

/* Device time of each kernel of the last simulate_replicas call, measured
 * with CUDA events on the context stream, and the kernel launches it made. */
typedef struct {
  float hash_ms, sim_ms, poa_ms, total_ms;
  int64_t launches;
  int64_t hashed_tokens;    /* tokens read by the block-hash kernel */
} rs_timing;
rs_status route_last_timing(const rs_ctx* ctx, rs_timing* out);

/* Saturation knee of load sweeps (§5.1, the PoA-growth proposition, item 3:
 * a second derivative of latency with respect to load above a threshold
 * marks the onset of saturation; Experiment 2 reads the difference quotients
 * of TTFT P99 across nine concurrency levels).
 *   records: device records as simulate_replicas wrote them; worker and ttft
 *     are read.  Replica r owns rows row_start[r] .. row_start[r+1] - 1
 *     (row_start: host, n_replicas + 1 nondecreasing entries, first >= 0).
 *   pct (1..100): stat[r] = the nearest-rank pct-th percentile of replica r's
 *     routed TTFTs (rows with worker >= 0), i.e. element ceil(pct n / 100) - 1
 *     of them in ascending order; NaN when it routed none.
 *   load: host, n_replicas entries, the load axis (normally C).
 *   sweep_start: host, n_sweeps + 1 nondecreasing replica indices <=
 *     n_replicas; sweep s = replicas sweep_start[s] .. sweep_start[s+1] - 1,
 *     meant in increasing load.
 * Outputs, host arrays, each may be NULL:
 *   stat, d1, d2 (n_replicas entries): d1[r] = (stat[r+1] - stat[r]) /
 *     (load[r+1] - load[r]) when r + 1 is in r's sweep; d2[r] = 2 (d1[r] -
 *     d1[r-1]) / (load[r+1] - load[r-1]) at interior points; NaN elsewhere and
 *     for replicas outside every sweep.
 *   knee_load, knee_index (n_sweeps entries): the first interior replica of
 *     the sweep with d2 > theta and its load; -1 / -1 if none; -2 / NaN (and
 *     no d1, d2) when the sweep's loads do not increase strictly.
 * Every value is computed on the device; returns after the outputs are
 * written.  RS_ERR_INVALID for NULL or inconsistent arguments. */
rs_status sweep_knee(rs_ctx* ctx, const rs_records* records, const int64_t* row_start,
                     int32_t n_replicas, const double* load, const int32_t* sweep_start,
                     int32_t n_sweeps, int32_t pct, double theta, double* stat, double* d1,
                     double* d2, double* knee_load, int32_t* knee_index);

/* Entry point that allocates nothing.  The paper has no counterpart: this
 * is a library service for callers that cannot allocate device memory when
 * they need an estimate -- a serving process whose GPU memory is owned up
 * front by another allocator, or a latency-critical path where cudaMalloc /
 * cudaFree would synchronise the device.
 *
 * Same result as poa_estimate for caller records of one replica (device
 * pointers, n rows, cfg->W <= 64 columns), computed in a fixed static device
 * array of RS_NOALLOC_POA_BYTES bytes that every GPU loading the library
 * holds until the process exits.  No context is needed; nothing is allocated
 * (no cudaMalloc, cudaFree or allocating library call) and nothing is read
 * back to the host: the work is enqueued on cuda_stream (NULL = legacy
 * default stream).
 *   cfg: host struct; poa_window, cap, the latency constants and W are used.
 *   numer_dev/opt_dev (double) and count_dev (int64), each NULL or
 *   max_windows entries: the first min(windows, max_windows) windows.
 *   poa_total_dev (double) and n_windows_dev (int64): one entry each.
 * Sizes: accepted when n (8 W + 60) + 4096 <= RS_NOALLOC_POA_BYTES, i.e. up to
 * 399 408 rows at W = 3 (171 175 at W = 17); larger calls return
 * RS_ERR_CAPACITY before any work.  The windows get the bytes the rows leave,
 * 48 per window and never fewer than n + 2 windows; records that span more
 * windows than that give *n_windows_dev = -1 (and no estimate).
 * The first call on a device takes the array's device address
 * (cudaGetSymbolAddress) for that device and keeps it for the life of the
 * process; make that first call before any stream capture.  The address is
 * not taken again, so the library cannot be used this way after a
 * cudaDeviceReset (which unloads the array) in the same process.  All calls
 * on a device share the one array and every call rewrites what it reads, so
 * calls that overlap on the GPU (other streams, other host threads) race and
 * must be serialised by the caller. */
#define RS_NOALLOC_POA_BYTES (32u * 1024u * 1024u)
rs_status poa_estimate_noalloc(const rs_config* cfg, const rs_records* records, int64_t n,
                               double* numer_dev, double* opt_dev, int64_t* count_dev,
                               int64_t max_windows, double* poa_total_dev,
                               int64_t* n_windows_dev, void* cuda_stream);

#ifdef __cplusplus
}
#endif
#endif
