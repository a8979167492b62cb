/*
 * CPU oracle for the KV-cache-aware routing simulation -- TEST INFRASTRUCTURE.
 *
 * Plain, slow, single-threaded C that computes what the paper's routing and
 * caching games define, step by step, so that the CUDA path can be checked
 * against it.  Only the test-suite, the smoke check and the CPU-baseline leg of
 * the benchmark may load it; the product path never does.  It shares no code,
 * header, table or helper with the CUDA library.
 *
 * Paper passages followed (section / equation numbers of the paper):
 *   router cost                 Eq. (1), §2.2
 *   softmax selection           Eq. (2), §2.2; tau -> 0 limit, §4.3
 *   routing-game cost           Eq. (7), Def. 3, §4.3
 *   superlinear latency         Eq. (9), §5.1; constants of §6.4
 *   saturation signal (EWMA)    Eq. (10), §6.2
 *   regime classification       Eq. (11), §6.2 (hysteresis paragraph)
 *   regime parameters           Table 2, §6.3; Algorithm 1, §6.4
 *   PoA estimate                Eq. (12), §6.4 (frozen-latency matrix,
 *                               replicated worker columns, Hungarian OPT)
 *   PoA of a one-shot game      Def. 7 (App. A), Nash equilibrium Def. 5
 *   closed-loop client          §7.4 (semaphore holding C requests in flight)
 *
 * Parity status: the block hash, the LRU cache and the Philox stream are the
 * readings this implementation fixes where the paper is silent (block size,
 * hash function, eviction order, RNG); they are pinned by properties, brute
 * force and published generator test vectors, not by the paper.
 */
#ifndef ROUTESIM_ORACLE_H
#define ROUTESIM_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum {
  ORC_OK = 0,
  ORC_ERR_INVALID = -1,
  ORC_ERR_OOM = -2,
  ORC_ERR_CAPACITY = -3,   /* a prompt has more full blocks than a cache holds */
  ORC_ERR_TIMEOUT = -5,    /* inconsistent event state (cannot happen) */
  ORC_ERR_COLLISION = -7   /* two blocks of one prompt share a chained hash */
};

enum { ORC_POLICY_DYNAMO = 0, ORC_POLICY_LOADBAL = 1,
       /* static counterfactual policies (§9, routing baselines) */
       ORC_POLICY_ROUNDROBIN = 2, ORC_POLICY_RANDOM = 3, ORC_POLICY_P2C = 4 };
/* eviction of the per-worker block caches: exact LRU, or the KV Block
 * Manager's frequency rule (§2.2) */
enum { ORC_EVICT_LRU = 0, ORC_EVICT_FREQ = 1 };

typedef struct {
  int32_t W;              /* decode workers (routing-game resources) */
  int32_t block;          /* tokens per KV block (even) */
  int64_t K;              /* cache capacity per worker, blocks */
  uint64_t hash_seed;     /* h_{-1} of the block-hash chain */
  double lat_a, lat_b, lat_d;  /* Eq. (9) a, b, d (beta = 2) */
  int32_t cap;            /* C_j: pole of Eq. (9); service slots = cap - 1 */
  double w_c;             /* cache weight of the §6.4 cost matrix */
  double itl;             /* seconds per output token */
  double dt;              /* controller polling interval Delta, s */
  double alpha;           /* EWMA weight of Eq. (10) */
  double theta1, theta2;  /* Eq. (11) thresholds, s */
  double eps_frac;        /* hysteresis margin epsilon = eps_frac * theta */
  int32_t hyst_k;         /* consecutive samples to change regime */
  float regime_tau[3];    /* Table 2; entry 0 replaced by the replica's own */
  float regime_omega[3];
  double poa_window;      /* window length of Eq. (12), s */
  /* Game 2 (§4.2, Eq. kv-cost): tiered = 1 gives every worker the exclusive
   * tiers G1 (K blocks), G2 (tier_k2) and G3 (tier_k3); an access brings a
   * block to G1, and each full tier hands its least recently used block to
   * the next (the last drops it).  Routing sees G1.  Each routed request is
   * charged, per full block on its worker i, alpha_t for its own tier t,
   * else d(i, j) + alpha_t for the cheapest copy on another worker j, else
   * gamma; d = tier_d_near within a node of tier_node workers, else
   * tier_d_far. */
  int32_t tiered, tier_node;
  int64_t tier_k2, tier_k3;
  double tier_alpha[3];
  double tier_gamma, tier_d_near, tier_d_far;
} orc_config;

typedef struct {
  int32_t C;              /* concurrency held by the client semaphore */
  int32_t policy;         /* ORC_POLICY_* */
  int32_t controller;     /* 1: adaptive controller (Algorithm 1) on */
  float omega, tau;       /* static router parameters (Below regime) */
  uint64_t seed;          /* Philox key of the sampling stream */
  int64_t n_req;          /* requests routed (prefix of the trace) */
  /* load-spike schedule (Experiment 3): C before c_t1, c_mid on [c_t1, c_t2),
   * c_end from c_t2 on; c_mid = 0 keeps C */
  double c_t1, c_t2;
  int32_t c_mid, c_end;
  /* cache eviction (ORC_EVICT_*); for FREQ the frequency cap (>= 1) and the
   * length of one decay step in s of simulated time (> 0) */
  int32_t eviction, freq_max;
  double decay_s;
} orc_replica;

typedef struct {
  int32_t status;
  int64_t n_routed;
  double sum_ttft, sum_e2e, makespan;
  int64_t near_ties, exact_ties, sampled, near_boundary;
  int64_t hit_blocks, inserted_blocks, evicted_blocks;
  int64_t ticks, regime_switches;
  int32_t final_regime, max_regime;
  int64_t ticks_in_regime[3];
  double final_ewma;
  double first_switch_t;   /* first regime switch, -1 if none */
  /* KV-cache pressure (the regime-transition proposition of §5.3): arrival
   * time of the first request whose update pushed a block out of a G1
   * cache, and rho = resident blocks (all tiers) over W K after that update
   * (-1, -1 if none); rho after the last request */
  double first_evict_t, rho_first_evict, rho_end;
  /* Game 2 accounting (tiered): blocks found in the own G1 / G2 / G3, on
   * another worker, nowhere; and the summed cost of Eq. kv-cost */
  int64_t kv_g1, kv_g2, kv_g3, kv_remote, kv_recompute;
  double kv_cost;
} orc_summary;

/* Per-request outputs; every pointer may be NULL.  Arrays of n (or n*W). */
typedef struct {
  int32_t* worker;        /* chosen worker sigma_i */
  double* arrival;        /* a_i */
  double* start;          /* service start s_i */
  double* first_token;    /* s_i + service TTFT */
  double* completion;     /* first token + O_i * itl */
  double* ttft;           /* first token - a_i (includes queueing) */
  int32_t* nbt;           /* ceil(L_i / block) */
  uint16_t* n_frozen;     /* [n*W] min(in-service_j(a_i) + 1, cap - 1) */
  uint16_t* prefix;       /* [n*W] m_ij: cached-prefix blocks on worker j */
  float* cost;            /* [n*W] router cost c_j used for the decision */
  double* kv_cost;        /* Eq. kv-cost of the request's blocks on its worker (tiered) */
} orc_records;

/* Block hashes of every full block.  Request i's hashes are written to
 * out[floor(offsets[i]/block) + k], k < floor(L_i/block). */
void orc_hash_blocks(const int32_t* tokens, const int64_t* offsets, int64_t n_req,
                     int32_t block, uint64_t seed, uint64_t* out);

/* SplitMix64 finalizer (exported for pins). */
uint64_t orc_mix64(uint64_t z);
/* Philox4x32-10 (exported for pins). */
void orc_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]);
/* exp for x <= 0 by Cody-Waite reduction + degree-7 Taylor (exported for pins). */
float orc_expf(float x);
/* orc_expf over an array (pins). */
void orc_expf_n(const float* x, float* y, int64_t n);
/* Worker choice of Eq. (2) (argmin when tau == 0); exported for pins.
 * u24: the 24-bit uniform draw (ignored when tau == 0). */
int32_t orc_select(const float* cost, int32_t W, float tau, uint32_t u24);

/* One replica of the closed-loop simulation.  Returns ORC_* status. */
int32_t orc_simulate(const orc_config* cfg, const int32_t* tokens, const int64_t* offsets,
                     const double* release, const int32_t* out_len, const orc_replica* rep,
                     orc_records* rec, orc_summary* sum,
                     uint64_t* cache_keys /* [W*K] LRU->MRU, nullable */,
                     int64_t* cache_sizes /* [W], nullable */,
                     double* tick_ewma /* [max_ticks], nullable */,
                     int32_t* tick_regime /* [max_ticks], nullable */, int64_t max_ticks);

/* Nearest-rank 99th percentile (the controller's TTFT P99 of §6.2). */
double orc_p99(const double* v, int64_t n);
/* Saturation knee of load sweeps (§5.1, PoA-growth proposition, item 3;
 * Experiment 2): per-replica nearest-rank percentile of routed TTFTs, first
 * and second divided differences over each sweep, first interior point with a
 * second difference above theta. */
int32_t orc_sweep_knee(int32_t n_rep, const int64_t* row_start, const int32_t* worker,
                       const double* ttft, const double* load, int32_t n_sweeps,
                       const int32_t* sweep_start, int32_t pct, double theta, double* stat,
                       double* d1, double* d2, double* knee_load, int32_t* knee_index);
/* The controller alone: one sample per entry of L (NaN = empty window);
 * writes the EWMA of Eq. (10) (-1 before the first sample) and the regime of
 * Eq. (11) after each sample. */
int32_t orc_controller_run(const orc_config* cfg, int64_t n, const double* L, double* ewma,
                           int32_t* regime);

/* PoA estimate of Eq. (12) over tumbling windows of completion time.
 * method: 0 auto, 1 Hungarian on the replicated square matrix, 2 min-cost flow.
 * numer/opt/count: [n_win_cap] per window id; returns windows used (or <0). */
int64_t orc_poa(const orc_config* cfg, int64_t n, const int32_t* worker, const double* completion,
                const double* ttft, const int32_t* nbt, const uint16_t* n_frozen,
                const uint16_t* prefix, int32_t method, double* numer, double* opt,
                int64_t* count, int64_t n_win_cap, double* poa_total);

/* Static counterfactual (§9): per window, sum of the frozen §6.4 costs of the
 * realized assignment, c_{i, worker(i)}.  Returns windows spanned. */
int64_t orc_static_numer(const orc_config* cfg, int64_t n, const int32_t* worker,
                         const double* completion, const int32_t* nbt, const uint16_t* n_frozen,
                         const uint16_t* prefix, double* numer_static, int64_t n_win_cap);

/* Min-cost assignment of n rows to W groups of `capw` identical columns;
 * cost is row-major [n*W].  method 1 Hungarian, 2 min-cost flow, 3 brute force
 * (n <= 9).  Returns the optimal total; assign[n] receives a minimiser. */
double orc_assign(const double* cost, int64_t n, int32_t W, int64_t capw, int32_t method,
                  int32_t* assign);

/* Exhaustive one-shot routing game (Def. 3 cost with Eq. (9) latency, Def. 7 PoA).
 * o: [n*W] overlaps in [0,1].  Outputs (nullable): opt, worst_ne, best_ne,
 * greedy (sequential best response in index order), n_ne, and
 * br_steps = improving moves of best-response dynamics started from greedy
 * (-1 if it did not reach an equilibrium within 10000 moves), and
 * max_ne_spread = the largest (max load - min load) over all equilibria.
 * A deviation counts as improving when it lowers the cost by more than 1e-12. */
int32_t orc_game_exhaustive(int32_t n, int32_t W, const double* o, double omega,
                            double lat_a, double lat_b, double lat_d, int32_t cap,
                            double* opt, double* worst_ne, double* best_ne, double* greedy,
                            int64_t* n_ne, int64_t* br_steps, int32_t* max_ne_spread);

/* Live router (route_batch semantics): n_instances independent routers. */
typedef struct orc_router orc_router;
orc_router* orc_router_new(const orc_config* cfg, float omega, float tau, uint64_t seed,
                           int32_t n_instances);
void orc_router_free(orc_router* r);
int32_t orc_router_route(orc_router* r, int32_t instance, const int32_t* tokens,
                         const int64_t* offsets, int64_t n_req, const int32_t* out_len,
                         int32_t* worker, float* cost, int32_t* prefix);
/* route_probe: m_ij of every request on every worker against the current
 * caches, nothing updated; prefix [n_req * W]. */
int32_t orc_router_probe(orc_router* r, int32_t instance, const int32_t* tokens,
                         const int64_t* offsets, int64_t n_req, int32_t* prefix);
int32_t orc_router_release(orc_router* r, int32_t instance, const int32_t* worker,
                           const int32_t* blocks, int64_t n);
int32_t orc_router_active(orc_router* r, int32_t instance, int64_t* active /* [W] */);
int32_t orc_router_cache(orc_router* r, int32_t instance, int32_t worker, uint64_t* keys,
                         int64_t* size);

#ifdef __cplusplus
}
#endif
#endif
