// Internal declarations of the routing library (host + device, not public).
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>

#include "routesim.h"

namespace rs {

constexpr int NT_SIM = 256;      // threads of a simulation / router CTA
constexpr int NT_POA = 256;      // threads of a PoA CTA (8 warps, one window each)
constexpr int POA_WMAX = 16;     // workers of the per-warp PoA solver (wider: k_poa_solve_wide)
constexpr int POA_WMAX_WIDE = 64;  // workers supported by the PoA estimate
constexpr int WMAX = 64;         // workers supported by the simulation

// Per-worker cache bookkeeping (shared memory while a kernel runs, global
// memory between calls).
struct CacheMeta {
  uint32_t size;    // live entries
  uint32_t T;       // next stamp
  uint32_t head;    // log position at or before the least-recent live entry
  uint32_t tombs;   // tombstoned slots
};

// Game 2 tiers of one simulated worker: the log positions from which the
// live entries are the top K_G1 (b1) and the top K_G1 + K_G2 (b2) of its
// recency stack, i.e. G1 = [b1, T), G2 = [b2, b1), G3 = [head, b2).
struct TierMeta {
  uint32_t b1;
  uint32_t b2;
};

// Kernel variants of the simulation: exact LRU, the frequency rule, Game 2 tiers.
constexpr int SIM_LRU = 0, SIM_FREQ = 1, SIM_TIER = 2;
constexpr int SIM_PROBE_CAP = 2048;   // W * nb up to which the probe captures every slot

// Frequency eviction's search state of one worker: while the decay step is
// below fmin, the log range [head, fscan) holds no live cold entry (fmin = 0:
// search from the head).
struct FreqMeta {
  uint32_t fscan;
  uint32_t fmin;
};

// Geometry of one worker's table: 8 * nbuckets slots (>= 4 K) and a log ring
// of R entries (>= 4 K).
struct TableGeom {
  uint32_t K;
  uint32_t bmask;      // nbuckets - 1
  uint32_t rmask;      // R - 1
  size_t slots;        // 8 * nbuckets
  size_t R;
};

TableGeom table_geom(int64_t K);

struct ModelConsts;
// The kernels' model constants from a configuration (every field set).
ModelConsts make_consts(const rs_config& c);

// One simulated replica as the kernel sees it.
struct SimDesc {
  const int64_t* offsets;
  const double* release;
  const int32_t* out_len;
  const uint64_t* hashes;   // block hashes of the replica's trace
  const uint8_t* dupflag;   // per request: 1 when two blocks share a chained hash
  int64_t n_req;
  int64_t rec_base;         // first record row
  int32_t C, policy, controller, eviction;   // eviction: RS_EVICT_*
  float omega, tau;
  uint64_t seed;
  double c_t1, c_t2;        // load-spike schedule: C, then c_mid on [c_t1, c_t2),
  int32_t c_mid, c_end;     // then c_end (c_mid = 0: C throughout)
  int32_t freq_max, reserved;   // frequency eviction: cap, and decay step length (s)
  double decay_s;
};

struct ModelConsts {
  double lat_a, lat_b, lat_d, w_c, itl, dt, alpha, theta1, theta2, eps_frac, poa_window;
  int32_t cap, hyst_k, W, write_cost;
  float regime_tau[3], regime_omega[3];
  double tier_alpha[3], tier_gamma, tier_dn, tier_df;   // Game 2 costs (Eq. kv-cost)
  int32_t tier_node, reserved;
};

struct SimBuffers {
  uint64_t* keys;           // [nsim][W][slots]
  uint32_t* stamp;          // [nsim][W][slots]
  uint32_t* log;            // [nsim][W][R]
  uint32_t* fexp;           // [nsim][W][slots] frequency eviction state, or NULL
  uint64_t* tmp;            // [nsim][K] rebuild scratch (and the frequency slow path's list)
  uint32_t* tmpe;           // [nsim][K] rebuild scratch of fexp, or NULL
  double* pend;             // [nsim][4][pend_cap]: 2 buffers x (first token, TTFT)
  int64_t pend_cap;
  CacheMeta* meta_out;      // [nsim][W]
  rs_replica_result* res;   // [nsim]
  rs_records rec;           // every field non-NULL except possibly cost and kv_cost
  float* dstat;             // [rows][6]: two lowest costs, draw position (see k_decision_stats)
  const double* wco_tab;    // [(nbmax+1)(nbmax+2)] w_c * (m / nbt), or NULL
  int wco_dim;              // nbmax + 2 (row length of wco_tab)
  unsigned char* slotmem;   // [nsim][sim_slot_bytes(cmax)] when SimLaunch::slots_global
};

struct SimLaunch {
  int nsim;
  int nbmax;                // max full blocks of any routed prompt
  int cmax;                 // max concurrency over replicas
  int slots_global;         // 1: per-request slot arrays in SimBuffers::slotmem
  int tiered;               // 1: Game 2 tiers (g.K = all tiers of a worker)
  int64_t k1, k12;          // G1 capacity, G1 + G2 capacity (k1 = g.K without tiers)
  TableGeom g;
  ModelConsts mc;
};

// Dynamic shared memory of one replica CTA; with slots_global the per-request
// slot arrays are in global memory instead (sim_slot_bytes per replica).
size_t sim_smem_bytes(int W, int nbmax, int cmax, int cap, bool slots_global,
                      bool tiered = false);
size_t sim_slot_bytes(int cmax);

// One trace for the block-hash kernels: requests req_base .. req_base+n_req-1
// of the launch's global request numbering.
struct HashJob {
  const int32_t* tokens;
  const int64_t* offsets;
  uint64_t* out;
  int64_t n_req;
  int64_t req_base;
};
constexpr int HASH_MAX_JOBS = 64;
cudaError_t launch_block_hash(const HashJob* jobs_dev, int njobs, int64_t total_req, uint64_t seed,
                              int64_t* nbmax_out, cudaStream_t st);
// *nbmax = max(*nbmax, the largest floor(L/16) over the jobs' requests).
cudaError_t launch_nbmax(const HashJob* jobs_dev, int njobs, int64_t total_req, int64_t* nbmax,
                         cudaStream_t st);
// flags[r] = 1 when two blocks of request r (numbered over the launch's jobs)
// share a chained hash, 0 when none do, 2 when it has more than nbmax blocks
// (not checked).  Fails with cudaErrorInvalidValue when one warp's set of
// 2^ceil(log2(2 nbmax)) hashes does not fit in shared memory.
cudaError_t launch_dup_flags(const HashJob* jobs_dev, int njobs, int64_t total_req, int64_t nbmax,
                             uint8_t* flags, cudaStream_t st);
cudaError_t launch_sim(const SimDesc* d_desc, const SimBuffers& b, const SimLaunch& L,
                       cudaStream_t st);
cudaError_t launch_wco_table(double* tab, int nbmax, double w_c, cudaStream_t st);
cudaError_t launch_decision_stats(const SimDesc* d_desc, const SimBuffers& b, const SimLaunch& L,
                                  cudaStream_t st);

// PoA of Eq. (12): one "problem" per replica.
struct PoaProblem {
  int64_t rec_base;         // first record row
  int64_t n;                // rows
  int64_t scratch_base;     // first row of this problem in the row-indexed scratch
  int64_t win_base;         // first window slot in the window-indexed scratch
  int64_t win_cap;          // window slots available
};

struct PoaBuffers {
  rs_records rec;
  double* cost;             // [rows][W]
  int32_t* order;           // [rows] row (relative) sorted by window, stable
  int32_t* asg;             // [rows]
  int32_t* wkey;            // [rows] window of each row (-1 skipped)
  int64_t* wstart;          // [win slots + problems]
  int64_t* wfill;           // [win slots]
  double* wnum;             // [win slots]
  double* wopt;             // [win slots]
  double* wstat;            // [win slots] frozen cost of the realized assignment
  int64_t* wcnt;            // [win slots]
  double* total;            // [problems]: PoA total
  double* total_static;     // [problems]: realized assignment's frozen cost / OPT
  int64_t* nwin;            // [problems]: windows spanned (or -1 on overflow)
  rs_replica_result* res;   // optional [problems] (poa_total, n_windows filled)
  // optional: the window slots (nslots of them) go to the solver warps of the
  // whole grid through the counter wnext, zeroed by launch_poa; wprob[slot]
  // = the problem owning the slot.  NULL: each problem's windows stay on its
  // own CTAs.
  int32_t* wprob;
  unsigned long long* wnext;
  int64_t nslots;
};

// Saturation knee of load sweeps: per-replica percentile, divided differences, knee.
cudaError_t launch_sweep_knee(const int32_t* worker, const double* ttft, const int64_t* row_start,
                              int n_rep, const double* load, const int32_t* sweep_start,
                              int n_sweeps, int pct, double theta, double* stat, double* d1,
                              double* d2, double* knee_load, int32_t* knee_index,
                              cudaStream_t st);
// maxw[p] = last window index of problem p's routed rows (-1 if none).
cudaError_t launch_poa_span(const PoaProblem* d_prob, int nprob, const rs_records& rec,
                            double window, long long* maxw, cudaStream_t st);
cudaError_t launch_poa(const PoaProblem* d_prob, int nprob, const PoaBuffers& b,
                       const ModelConsts& mc, cudaStream_t st);

// Live router kernels.
struct RouterState {
  uint64_t* keys;           // [W][slots]
  uint32_t* stamp;
  uint32_t* log;
  uint64_t* tmp;            // [K]
  CacheMeta* meta;          // [W]
  int64_t* active;          // [W]
  uint64_t* ordinal;        // [1]
  int32_t* status;          // [1] sticky device error
};

// m_ij of n_req requests (hashes in the route_hash_blocks layout) on every
// worker of one router instance, read-only; prefix_out [n_req * W].
cudaError_t launch_probe_batch(const RouterState& s, const int64_t* offsets, const uint64_t* hashes,
                               int64_t n_req, int W, const TableGeom& g, int32_t* prefix_out,
                               cudaStream_t st);
cudaError_t launch_route_batch(const RouterState& s, int32_t instance, const int64_t* offsets,
                               const uint64_t* hashes, int32_t n_req, const int32_t* out_len,
                               int32_t* worker_out, float* cost_out, int32_t* prefix_out,
                               int nbmax, const TableGeom& g, const ModelConsts& mc, float omega,
                               float tau, uint64_t seed, cudaStream_t st);
size_t router_smem(int W, int nbmax);
cudaError_t launch_route_release(const RouterState& s, const int32_t* worker, const int32_t* blocks,
                                 int32_t n, int32_t W, cudaStream_t st);
cudaError_t launch_clear_tables(uint64_t* keys, uint32_t* stamp, size_t nslots, CacheMeta* meta,
                                size_t nmeta, cudaStream_t st);

}  // namespace rs
