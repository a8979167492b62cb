// Host side of the C ABI declared in include/routesim.h: argument checks,
// library-owned device memory, kernel launches on the context stream, and
// per-kernel device timing with CUDA events.
#include <algorithm>
#include <cstdarg>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

#include "rs_internal.h"

using namespace rs;

namespace {

thread_local std::string g_init_error;

struct DevBuf {
  void* p = nullptr;
  size_t n = 0;
};

}  // namespace

struct rs_ctx {
  rs_config cfg;
  cudaStream_t st = nullptr;
  int device = 0;
  std::string err;
  TableGeom g;    // the live routers' caches (cache_blocks)
  TableGeom gs;   // the simulated workers' caches (all tiers)
  ModelConsts mc;
  // live router instances
  int32_t ninst = 0;
  DevBuf r_keys, r_stamp, r_log, r_tmp, r_meta, r_active, r_ord, r_status, r_hash, r_stats;
  // simulation scratch (grow-only)
  DevBuf keys, stamp, log, tmp, pend, meta_out, res, desc, hashes, stats, hjobs, dstat, wco, slots;
  DevBuf fexp, tmpe;   // frequency eviction state and its rebuild scratch
  DevBuf dupf;         // per request: a chained hash repeats within the prompt
  DevBuf djobs;        // every trace in use, for the block-count and flag kernels
  DevBuf h_hashes;     // staged block hashes of host traces given by their hashes
  DevBuf rec_worker, rec_arrival, rec_start, rec_first, rec_completion, rec_ttft, rec_nbt, rec_nfz,
      rec_prefix;
  DevBuf p_cost, p_order, p_asg, p_wkey, p_wstart, p_wfill, p_wnum, p_wopt, p_wcnt, p_total,
      p_nwin, p_prob, p_wstat, p_tstat, p_wprob, p_wnext;
  DevBuf k_rows, k_load, k_sweep, k_stat, k_d1, k_d2, k_kload, k_kidx;
  DevBuf h_tokens, h_offsets, h_release, h_outlen;
  int64_t* pinned = nullptr;   // small host staging for device -> host reads
  size_t pinned_n = 0;
  // last simulate_replicas call
  int32_t last_nsim = 0;
  cudaEvent_t ev[4] = {nullptr, nullptr, nullptr, nullptr};
  rs_timing timing;
};

namespace {

rs_status fail(rs_ctx* c, rs_status s, const char* fmt, ...) __attribute__((format(printf, 3, 4)));
rs_status fail(rs_ctx* c, rs_status s, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  if (c) c->err = buf; else g_init_error = buf;
  return s;
}

rs_status cuda_fail(rs_ctx* c, cudaError_t e, const char* what) {
  return fail(c, RS_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

#define CK(call, what)                                  \
  do {                                                  \
    cudaError_t e_ = (call);                            \
    if (e_ != cudaSuccess) return cuda_fail(ctx, e_, what); \
  } while (0)

rs_status ensure(rs_ctx* ctx, DevBuf& b, size_t bytes, const char* what) {
  if (bytes == 0) bytes = 16;
  if (b.n >= bytes) return RS_OK;
  if (b.p) {
    cudaError_t e = cudaFree(b.p);
    b.p = nullptr;
    b.n = 0;
    if (e != cudaSuccess) return cuda_fail(ctx, e, "cudaFree");
  }
  const size_t want = (bytes + 255) & ~(size_t)255;
  cudaError_t e = cudaMalloc(&b.p, want);
  if (e != cudaSuccess) {
    cudaGetLastError();
    b.p = nullptr;
    return fail(ctx, RS_ERR_OOM, "cudaMalloc of %zu bytes for %s failed: %s", want, what,
                cudaGetErrorString(e));
  }
  b.n = want;
  return RS_OK;
}

void release(DevBuf& b) {
  if (b.p) cudaFree(b.p);
  b.p = nullptr;
  b.n = 0;
}

rs_status ensure_pinned(rs_ctx* ctx, size_t n) {
  if (ctx->pinned_n >= n) return RS_OK;
  if (ctx->pinned) cudaFreeHost(ctx->pinned);
  ctx->pinned = nullptr;
  ctx->pinned_n = 0;
  CK(cudaMallocHost(reinterpret_cast<void**>(&ctx->pinned), n * sizeof(int64_t)), "cudaMallocHost");
  ctx->pinned_n = n;
  return RS_OK;
}

template <class T>
T* P(DevBuf& b) { return reinterpret_cast<T*>(b.p); }

rs_status check_config(const rs_config* cfg) {
  if (!cfg) return fail(nullptr, RS_ERR_INVALID, "cfg is NULL");
  if (cfg->W < 1 || cfg->W > WMAX) return fail(nullptr, RS_ERR_INVALID, "W must be in [1, %d]", WMAX);
  if (cfg->block_size != 16) return fail(nullptr, RS_ERR_INVALID, "block_size must be 16");
  if (cfg->cache_blocks < 1 || cfg->cache_blocks > (1ll << 24))
    return fail(nullptr, RS_ERR_INVALID, "cache_blocks must be in [1, 2^24]");
  if (cfg->cap < 2 || cfg->cap > 65535) return fail(nullptr, RS_ERR_INVALID, "cap must be in [2, 65535]");
  if (cfg->hyst_k < 1) return fail(nullptr, RS_ERR_INVALID, "hyst_k must be >= 1");
  if (!(cfg->dt > 0.0) || !(cfg->poa_window > 0.0) || !(cfg->alpha > 0.0 && cfg->alpha <= 1.0))
    return fail(nullptr, RS_ERR_INVALID, "dt, poa_window must be > 0 and alpha in (0, 1]");
  if (!(cfg->omega >= 0.0f) || !(cfg->tau >= 0.0f) || !std::isfinite(cfg->omega) ||
      !std::isfinite(cfg->tau))
    return fail(nullptr, RS_ERR_INVALID, "omega and tau must be finite and >= 0");
  for (int r = 0; r < 3; r++)
    if (!(cfg->regime_tau[r] >= 0.0f) || !(cfg->regime_omega[r] >= 0.0f))
      return fail(nullptr, RS_ERR_INVALID, "regime parameters must be >= 0");
  if (cfg->tiered != 0 && cfg->tiered != 1) return fail(nullptr, RS_ERR_INVALID, "tiered must be 0 or 1");
  if (cfg->tiered) {
    const double* a = cfg->tier_alpha;
    if (cfg->tier_k2 < 0 || cfg->tier_k3 < 0 ||
        cfg->cache_blocks + cfg->tier_k2 + cfg->tier_k3 > (1ll << 24))
      return fail(nullptr, RS_ERR_INVALID, "tier sizes must be >= 0, all tiers <= 2^24 blocks");
    if (!(a[0] >= 0.0 && a[0] < a[1] && a[1] < a[2] && a[2] < cfg->tier_gamma) ||
        !std::isfinite(cfg->tier_gamma))
      return fail(nullptr, RS_ERR_INVALID, "need 0 <= alpha_G1 < alpha_G2 < alpha_G3 < gamma < inf");
    if (!(cfg->tier_d_near >= 0.0) || !(cfg->tier_d_far >= 0.0) ||
        !std::isfinite(cfg->tier_d_near) || !std::isfinite(cfg->tier_d_far))
      return fail(nullptr, RS_ERR_INVALID, "tier_d_near and tier_d_far must be finite and >= 0");
    if (cfg->tier_node < 1) return fail(nullptr, RS_ERR_INVALID, "tier_node must be >= 1");
  }
  return RS_OK;
}

}  // namespace

namespace rs {
ModelConsts make_consts(const rs_config& c) {
  ModelConsts m;
  m.lat_a = c.lat_a; m.lat_b = c.lat_b; m.lat_d = c.lat_d; m.w_c = c.w_c; m.itl = c.itl;
  m.dt = c.dt; m.alpha = c.alpha; m.theta1 = c.theta1; m.theta2 = c.theta2;
  m.eps_frac = c.eps_frac; m.poa_window = c.poa_window; m.cap = c.cap; m.hyst_k = c.hyst_k;
  m.W = c.W; m.write_cost = 0;
  for (int r = 0; r < 3; r++) { m.regime_tau[r] = c.regime_tau[r]; m.regime_omega[r] = c.regime_omega[r]; }
  for (int t = 0; t < 3; t++) m.tier_alpha[t] = c.tier_alpha[t];
  m.tier_gamma = c.tier_gamma;
  m.tier_dn = c.tier_d_near;
  m.tier_df = c.tier_d_far;
  m.tier_node = c.tier_node > 0 ? c.tier_node : 1;
  m.reserved = 0;
  return m;
}
}  // namespace rs

namespace {

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

namespace rs {
TableGeom table_geom(int64_t K) {
  TableGeom g;
  g.K = (uint32_t)K;
  uint64_t nbk = 1;   // buckets of 8 keys, at least 4 K slots (live load <= 1/4)
  while (nbk * 8 < (uint64_t)(4 * K)) nbk <<= 1;
  uint64_t R = 1;
  while (R < (uint64_t)(4 * K)) R <<= 1;
  g.bmask = (uint32_t)(nbk - 1);
  g.slots = (size_t)(nbk * 8);
  g.R = (size_t)R;
  g.rmask = (uint32_t)(R - 1);
  return g;
}
}  // namespace rs

extern "C" {

void rs_config_default(rs_config* c) {
  if (!c) return;
  memset(c, 0, sizeof *c);
  c->W = 3;
  c->block_size = 16;
  c->cache_blocks = 65536;
  c->hash_seed = 0;
  c->omega = 1.0f;
  c->tau = 0.0f;
  c->seed = 0;
  c->lat_a = 0.005;
  c->lat_b = 0.020;
  c->lat_d = 0.010;
  c->cap = 64;
  c->hyst_k = 3;
  c->w_c = 0.015;
  c->itl = 0.012;
  c->dt = 5.0;
  c->alpha = 0.3;
  c->theta1 = 0.3;
  c->theta2 = 2.0;
  c->eps_frac = 0.1;
  c->regime_tau[0] = 0.0f; c->regime_tau[1] = 0.7f; c->regime_tau[2] = 0.8f;
  c->regime_omega[0] = 1.0f; c->regime_omega[1] = 1.0f; c->regime_omega[2] = 0.1f;
  c->poa_window = 5.0;
  c->tiered = 0;          // Game 2 tiers off; the paper gives no tier costs
  c->tier_node = 1;
  c->tier_k2 = 0;
  c->tier_k3 = 0;
  c->tier_alpha[0] = 1.0; c->tier_alpha[1] = 4.0; c->tier_alpha[2] = 20.0;
  c->tier_gamma = 100.0;
  c->tier_d_near = 2.0;
  c->tier_d_far = 10.0;
}

const char* route_last_error(const rs_ctx* ctx) {
  return ctx ? ctx->err.c_str() : g_init_error.c_str();
}

rs_status route_init(rs_ctx** out, const rs_config* cfg, int32_t n_instances, void* cuda_stream) {
  g_init_error.clear();
  if (!out) return fail(nullptr, RS_ERR_INVALID, "out is NULL");
  *out = nullptr;
  rs_status s = check_config(cfg);
  if (s != RS_OK) return s;
  if (n_instances < 0 || n_instances > 4096)
    return fail(nullptr, RS_ERR_INVALID, "n_instances must be in [0, 4096]");
  int ndev = 0;
  cudaError_t e = cudaGetDeviceCount(&ndev);
  if (e != cudaSuccess || ndev == 0) {
    cudaGetLastError();
    return fail(nullptr, RS_ERR_CUDA, "no CUDA device: %s", cudaGetErrorString(e));
  }
  rs_ctx* ctx = new rs_ctx();
  ctx->cfg = *cfg;
  ctx->st = reinterpret_cast<cudaStream_t>(cuda_stream);
  cudaGetDevice(&ctx->device);
  ctx->g = table_geom(cfg->cache_blocks);
  ctx->gs = cfg->tiered ? table_geom(cfg->cache_blocks + cfg->tier_k2 + cfg->tier_k3) : ctx->g;
  ctx->mc = make_consts(*cfg);
  memset(&ctx->timing, 0, sizeof ctx->timing);
  for (auto& ev : ctx->ev) {
    e = cudaEventCreate(&ev);
    if (e != cudaSuccess) {
      route_destroy(ctx);
      return fail(nullptr, RS_ERR_CUDA, "cudaEventCreate: %s", cudaGetErrorString(e));
    }
  }
  ctx->ninst = n_instances;
  if (n_instances > 0) {
    const size_t W = cfg->W, ni = n_instances;
    const size_t nsl = ni * W * ctx->g.slots;
    rs_status r = RS_OK;
    if ((r = ensure(ctx, ctx->r_keys, nsl * 8, "router keys")) ||
        (r = ensure(ctx, ctx->r_stamp, nsl * 4, "router stamps")) ||
        (r = ensure(ctx, ctx->r_log, ni * W * ctx->g.R * 4, "router log")) ||
        (r = ensure(ctx, ctx->r_tmp, ni * ctx->g.K * 8, "router rebuild scratch")) ||
        (r = ensure(ctx, ctx->r_meta, ni * W * sizeof(CacheMeta), "router meta")) ||
        (r = ensure(ctx, ctx->r_active, ni * W * 8, "router active")) ||
        (r = ensure(ctx, ctx->r_ord, ni * 8, "router ordinal")) ||
        (r = ensure(ctx, ctx->r_status, ni * 2 * 4, "router status")) ||
        (r = ensure(ctx, ctx->r_stats, 64, "router stats"))) {
      std::string m = ctx->err;
      route_destroy(ctx);
      return fail(nullptr, r, "%s", m.c_str());
    }
    e = launch_clear_tables(P<uint64_t>(ctx->r_keys), P<uint32_t>(ctx->r_stamp), nsl,
                            P<CacheMeta>(ctx->r_meta), ni * W, ctx->st);
    if (e == cudaSuccess) e = cudaMemsetAsync(ctx->r_active.p, 0, ni * W * 8, ctx->st);
    if (e == cudaSuccess) e = cudaMemsetAsync(ctx->r_ord.p, 0, ni * 8, ctx->st);
    if (e == cudaSuccess) e = cudaMemsetAsync(ctx->r_status.p, 0, ni * 2 * 4, ctx->st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(ctx->st);
    if (e != cudaSuccess) {
      route_destroy(ctx);
      return fail(nullptr, RS_ERR_CUDA, "router init: %s", cudaGetErrorString(e));
    }
  }
  *out = ctx;
  return RS_OK;
}

void route_destroy(rs_ctx* ctx) {
  if (!ctx) return;
  cudaStreamSynchronize(ctx->st);
  DevBuf* all[] = {&ctx->r_keys, &ctx->r_stamp, &ctx->r_log, &ctx->r_tmp, &ctx->r_meta,
                   &ctx->r_active, &ctx->r_ord, &ctx->r_status, &ctx->r_hash, &ctx->r_stats,
                   &ctx->keys, &ctx->stamp, &ctx->log, &ctx->tmp, &ctx->pend, &ctx->meta_out,
                   &ctx->res, &ctx->desc, &ctx->hashes, &ctx->stats, &ctx->hjobs, &ctx->dupf, &ctx->slots, &ctx->dstat, &ctx->wco, &ctx->rec_worker,
                   &ctx->rec_arrival, &ctx->rec_start, &ctx->rec_first, &ctx->rec_completion,
                   &ctx->rec_ttft, &ctx->rec_nbt, &ctx->rec_nfz, &ctx->rec_prefix, &ctx->p_cost,
                   &ctx->p_order, &ctx->p_asg, &ctx->p_wkey, &ctx->p_wstart, &ctx->p_wfill,
                   &ctx->p_wnum, &ctx->p_wopt, &ctx->p_wcnt, &ctx->p_total, &ctx->p_nwin,
                   &ctx->p_prob, &ctx->p_wstat, &ctx->p_tstat, &ctx->p_wprob, &ctx->p_wnext,
                   &ctx->h_tokens, &ctx->h_offsets,
                   &ctx->h_release, &ctx->h_outlen, &ctx->k_rows, &ctx->k_load, &ctx->k_sweep,
                   &ctx->k_stat, &ctx->k_d1, &ctx->k_d2, &ctx->k_kload, &ctx->k_kidx,
                   &ctx->fexp, &ctx->tmpe, &ctx->djobs, &ctx->h_hashes};
  for (DevBuf* b : all) release(*b);
  if (ctx->pinned) cudaFreeHost(ctx->pinned);
  for (auto& ev : ctx->ev)
    if (ev) cudaEventDestroy(ev);
  delete ctx;
}

static rs_status hash_jobs(rs_ctx* ctx, std::vector<HashJob>& jobs, int64_t* nbmax_dev);

rs_status route_hash_blocks(rs_ctx* ctx, const int32_t* tokens_dev, const int64_t* offsets_dev,
                            int64_t n_req, uint64_t* hashes_dev) {
  if (!ctx) return fail(nullptr, RS_ERR_INVALID, "ctx is NULL");
  ctx->err.clear();
  if (n_req < 0) return fail(ctx, RS_ERR_INVALID, "n_req < 0");
  if (n_req == 0) return RS_OK;
  if (!tokens_dev || !offsets_dev || !hashes_dev) return fail(ctx, RS_ERR_INVALID, "NULL pointer");
  if (!aligned16(tokens_dev)) return fail(ctx, RS_ERR_INVALID, "tokens must be 16-byte aligned");
  std::vector<HashJob> jobs(1);
  jobs[0] = HashJob{tokens_dev, offsets_dev, hashes_dev, n_req, 0};
  return hash_jobs(ctx, jobs, nullptr);
}

rs_status route_dup_flags(rs_ctx* ctx, const uint64_t* hashes_dev, const int64_t* offsets_dev,
                          int64_t n_req, int64_t max_blocks, uint8_t* flags_dev) {
  if (!ctx) return fail(nullptr, RS_ERR_INVALID, "ctx is NULL");
  ctx->err.clear();
  if (n_req < 0) return fail(ctx, RS_ERR_INVALID, "n_req < 0");
  if (max_blocks < 1 || max_blocks > 8192)
    return fail(ctx, RS_ERR_INVALID, "max_blocks must be in [1, 8192]");
  if (n_req == 0) return RS_OK;
  if (!hashes_dev || !offsets_dev || !flags_dev) return fail(ctx, RS_ERR_INVALID, "NULL pointer");
  HashJob job{nullptr, offsets_dev, const_cast<uint64_t*>(hashes_dev), n_req, 0};
  rs_status r = ensure(ctx, ctx->hjobs, sizeof(HashJob), "hash jobs");
  if (r != RS_OK) return r;
  CK(cudaMemcpyAsync(ctx->hjobs.p, &job, sizeof(HashJob), cudaMemcpyHostToDevice, ctx->st),
     "copy hash job");
  CK(launch_dup_flags(P<HashJob>(ctx->hjobs), 1, n_req, max_blocks, flags_dev, ctx->st),
     "duplicate flags launch");
  return RS_OK;   // (a copy from pageable memory has read its source when it returns)
}

// The jobs with their request numbers made relative to the first job of
// each launch group of HASH_MAX_JOBS (the kernels number requests from 0
// within a launch); jobs must number their requests contiguously.
static std::vector<HashJob> group_jobs(const std::vector<HashJob>& jobs) {
  std::vector<HashJob> out(jobs);
  for (size_t g0 = 0; g0 < out.size(); g0 += HASH_MAX_JOBS) {
    const size_t g1 = std::min(out.size(), g0 + HASH_MAX_JOBS);
    const int64_t base = jobs[g0].req_base;
    for (size_t k = g0; k < g1; k++) out[k].req_base -= base;
  }
  return out;
}

// Hashes every job (trace) in launches of up to HASH_MAX_JOBS traces.
static rs_status hash_jobs(rs_ctx* ctx, std::vector<HashJob>& jobs, int64_t* nbmax_dev) {
  if (jobs.empty()) return RS_OK;
  rs_status r = ensure(ctx, ctx->hjobs, sizeof(HashJob) * jobs.size(), "hash jobs");
  if (r != RS_OK) return r;
  const std::vector<HashJob> grp = group_jobs(jobs);
  CK(cudaMemcpyAsync(ctx->hjobs.p, grp.data(), sizeof(HashJob) * grp.size(),
                     cudaMemcpyHostToDevice, ctx->st),
     "copy hash jobs");
  for (size_t g0 = 0; g0 < jobs.size(); g0 += HASH_MAX_JOBS) {
    const size_t g1 = std::min(jobs.size(), g0 + HASH_MAX_JOBS);
    const int64_t total = jobs[g1 - 1].req_base + jobs[g1 - 1].n_req - jobs[g0].req_base;
    CK(launch_block_hash(P<HashJob>(ctx->hjobs) + g0, (int)(g1 - g0), total, ctx->cfg.hash_seed,
                         nbmax_dev, ctx->st),
       "block hash launch");
  }
  return RS_OK;
}

// Block hashes of one batch of a router instance into ctx->r_hash (sized from
// offsets_dev[n_req], read with a synchronising copy); nbmax_dev (nullable)
// receives the longest prompt's full blocks.
static rs_status hash_batch(rs_ctx* ctx, const int32_t* tokens_dev, const int64_t* offsets_dev,
                            int64_t n_req, int64_t* nbmax_dev) {
  rs_status r = ensure_pinned(ctx, 4);
  if (r != RS_OK) return r;
  CK(cudaMemcpyAsync(ctx->pinned, offsets_dev + n_req, 8, cudaMemcpyDeviceToHost, ctx->st),
     "read offsets");
  CK(cudaStreamSynchronize(ctx->st), "sync");
  const int64_t total = ctx->pinned[0];
  if (total < 0) return fail(ctx, RS_ERR_INVALID, "offsets[n_req] < 0");
  if ((r = ensure(ctx, ctx->r_hash, (size_t)(total / 16 + 1) * 8, "batch hashes")) != RS_OK) return r;
  std::vector<HashJob> jobs(1);
  jobs[0] = HashJob{tokens_dev, offsets_dev, P<uint64_t>(ctx->r_hash), n_req, 0};
  return hash_jobs(ctx, jobs, nbmax_dev);
}

// ---------------------------------------------------------------- live router

static rs_status router_state(rs_ctx* ctx, int32_t inst, RouterState* s) {
  if (inst < 0 || inst >= ctx->ninst) return fail(ctx, RS_ERR_INVALID, "instance out of range");
  const size_t W = ctx->cfg.W, i = inst;
  s->keys = P<uint64_t>(ctx->r_keys) + i * W * ctx->g.slots;
  s->stamp = P<uint32_t>(ctx->r_stamp) + i * W * ctx->g.slots;
  s->log = P<uint32_t>(ctx->r_log) + i * W * ctx->g.R;
  s->tmp = P<uint64_t>(ctx->r_tmp) + i * ctx->g.K;
  s->meta = P<CacheMeta>(ctx->r_meta) + i * W;
  s->active = P<int64_t>(ctx->r_active) + i * W;
  s->ordinal = P<uint64_t>(ctx->r_ord) + i;
  s->status = P<int32_t>(ctx->r_status) + 2 * i;
  return RS_OK;
}

rs_status route_batch(rs_ctx* ctx, int32_t instance, const int32_t* tokens_dev,
                      const int64_t* offsets_dev, int32_t n_req, const int32_t* out_len_dev,
                      int32_t* worker_out_dev, float* cost_out_dev, int32_t* prefix_out_dev) {
  if (!ctx) return fail(nullptr, RS_ERR_INVALID, "ctx is NULL");
  ctx->err.clear();
  RouterState s;
  rs_status r = router_state(ctx, instance, &s);
  if (r != RS_OK) return r;
  if (n_req < 0) return fail(ctx, RS_ERR_INVALID, "n_req < 0");
  if (n_req == 0) return RS_OK;
  if (!tokens_dev || !offsets_dev || !out_len_dev || !worker_out_dev)
    return fail(ctx, RS_ERR_INVALID, "NULL pointer");
  if (!aligned16(tokens_dev)) return fail(ctx, RS_ERR_INVALID, "tokens must be 16-byte aligned");
  CK(cudaMemsetAsync(ctx->r_stats.p, 0, 8, ctx->st), "memset");
  if ((r = hash_batch(ctx, tokens_dev, offsets_dev, n_req, P<int64_t>(ctx->r_stats))) != RS_OK)
    return r;
  CK(cudaMemcpyAsync(ctx->pinned, ctx->r_stats.p, 8, cudaMemcpyDeviceToHost, ctx->st), "read stats");
  CK(cudaStreamSynchronize(ctx->st), "sync");
  int64_t nbmax = ctx->pinned[0];
  if (nbmax > (int64_t)ctx->g.K) nbmax = ctx->g.K;   // longer prompts stop with RS_ERR_CAPACITY
  {
    int maxsmem = 0;
    cudaDeviceGetAttribute(&maxsmem, cudaDevAttrMaxSharedMemoryPerBlockOptin, ctx->device);
    if (router_smem(ctx->cfg.W, (int)std::max<int64_t>(nbmax, 1)) + 4096 > (size_t)maxsmem)
      return fail(ctx, RS_ERR_CAPACITY, "a prompt of %lld blocks needs too much shared memory",
                  (long long)nbmax);
  }
  ModelConsts mc = ctx->mc;
  CK(launch_route_batch(s, instance, offsets_dev, P<uint64_t>(ctx->r_hash), n_req, out_len_dev,
                        worker_out_dev, cost_out_dev, prefix_out_dev, (int)std::max<int64_t>(nbmax, 1),
                        ctx->g, mc, ctx->cfg.omega, ctx->cfg.tau, ctx->cfg.seed, ctx->st),
     "route_batch launch");
  return RS_OK;
}

rs_status route_probe(rs_ctx* ctx, int32_t instance, const int32_t* tokens_dev,
                      const int64_t* offsets_dev, int64_t n_req, int32_t* prefix_out_dev) {
  if (!ctx) return fail(nullptr, RS_ERR_INVALID, "ctx is NULL");
  ctx->err.clear();
  RouterState s;
  rs_status r = router_state(ctx, instance, &s);
  if (r != RS_OK) return r;
  if (n_req < 0) return fail(ctx, RS_ERR_INVALID, "n_req < 0");
  if (n_req == 0) return RS_OK;
  if (!tokens_dev || !offsets_dev || !prefix_out_dev) return fail(ctx, RS_ERR_INVALID, "NULL pointer");
  if (!aligned16(tokens_dev)) return fail(ctx, RS_ERR_INVALID, "tokens must be 16-byte aligned");
  if ((r = hash_batch(ctx, tokens_dev, offsets_dev, n_req, nullptr)) != RS_OK) return r;
  CK(launch_probe_batch(s, offsets_dev, P<uint64_t>(ctx->r_hash), n_req, ctx->cfg.W, ctx->g,
                        prefix_out_dev, ctx->st),
     "probe launch");
  return RS_OK;
}

static rs_status router_sync_status(rs_ctx* ctx, int32_t instance, int* bad) {
  rs_status r = ensure_pinned(ctx, 4);
  if (r != RS_OK) return r;
  CK(cudaMemcpyAsync(ctx->pinned, P<int32_t>(ctx->r_status) + 2 * instance, 8,
                     cudaMemcpyDeviceToHost, ctx->st),
     "read status");
  CK(cudaStreamSynchronize(ctx->st), "sync");
  const int32_t* st = reinterpret_cast<const int32_t*>(ctx->pinned);
  if (bad) *bad = st[1];
  if (st[0] != RS_OK)
    return fail(ctx, (rs_status)st[0], "router instance %d stopped on a device error (%d)", instance,
                st[0]);
  return RS_OK;
}

rs_status route_release(rs_ctx* ctx, int32_t instance, const int32_t* worker_dev,
                        const int32_t* blocks_dev, int32_t n) {
  if (!ctx) return fail(nullptr, RS_ERR_INVALID, "ctx is NULL");
  ctx->err.clear();
  RouterState s;
  rs_status r = router_state(ctx, instance, &s);
  if (r != RS_OK) return r;
  if (n < 0) return fail(ctx, RS_ERR_INVALID, "n < 0");
  if (n > 0 && (!worker_dev || !blocks_dev)) return fail(ctx, RS_ERR_INVALID, "NULL pointer");
  CK(launch_route_release(s, worker_dev, blocks_dev, n, ctx->cfg.W, ctx->st), "release launch");
  int bad = 0;
  r = router_sync_status(ctx, instance, &bad);
  if (r != RS_OK) return r;
  if (bad) {
    CK(cudaMemsetAsync(s.status + 1, 0, 4, ctx->st), "memset");
    CK(cudaStreamSynchronize(ctx->st), "sync");
    return fail(ctx, RS_ERR_INVALID, "release entries with a worker outside [0, W) were skipped");
  }
  return RS_OK;
}

rs_status route_active(rs_ctx* ctx, int32_t instance, int64_t* active_host) {
  if (!ctx) return fail(nullptr, RS_ERR_INVALID, "ctx is NULL");
  ctx->err.clear();
  RouterState s;
  rs_status r = router_state(ctx, instance, &s);
  if (r != RS_OK) return r;
  if (!active_host) return fail(ctx, RS_ERR_INVALID, "NULL pointer");
  CK(cudaMemcpyAsync(active_host, s.active, 8 * (size_t)ctx->cfg.W, cudaMemcpyDeviceToHost, ctx->st),
     "read active");
  return router_sync_status(ctx, instance, nullptr);
}

// ---------------------------------------------------------------- simulation

extern "C++" {
template <class T>
static rs_status pick_rec(rs_ctx* ctx, T* user, DevBuf& b, size_t bytes, T** dst) {
  if (user) {
    *dst = user;
    return RS_OK;
  }
  rs_status q = ensure(ctx, b, bytes, "records");
  *dst = reinterpret_cast<T*>(b.p);
  return q;
}
}

// Record arrays: the caller's where given, library scratch otherwise.
static rs_status records_effective(rs_ctx* ctx, const rs_records* user, int64_t rows, int W,
                                   bool want_cost, rs_records* eff) {
  memset(eff, 0, sizeof *eff);
  rs_records u;
  memset(&u, 0, sizeof u);
  if (user) u = *user;
  const size_t R = (size_t)std::max<int64_t>(rows, 1);
  rs_status r;
  if ((r = pick_rec(ctx, u.worker, ctx->rec_worker, R * 4, &eff->worker)) ||
      (r = pick_rec(ctx, u.arrival, ctx->rec_arrival, R * 8, &eff->arrival)) ||
      (r = pick_rec(ctx, u.start, ctx->rec_start, R * 8, &eff->start)) ||
      (r = pick_rec(ctx, u.first_token, ctx->rec_first, R * 8, &eff->first_token)) ||
      (r = pick_rec(ctx, u.completion, ctx->rec_completion, R * 8, &eff->completion)) ||
      (r = pick_rec(ctx, u.ttft, ctx->rec_ttft, R * 8, &eff->ttft)) ||
      (r = pick_rec(ctx, u.nbt, ctx->rec_nbt, R * 4, &eff->nbt)) ||
      (r = pick_rec(ctx, u.n_frozen, ctx->rec_nfz, R * 2 * W, &eff->n_frozen)) ||
      (r = pick_rec(ctx, u.prefix, ctx->rec_prefix, R * 2 * W, &eff->prefix)))
    return r;
  eff->cost = want_cost ? u.cost : nullptr;
  eff->kv_cost = u.kv_cost;   // optional
  return RS_OK;
}

// Eq. (12) for every problem in probs (rec_base, n, scratch_base set; the
// window slots are sized here): the last window of each problem is found on
// the device first, so that every window its records span gets a slot.
static rs_status run_poa(rs_ctx* ctx, const rs_records& rec, std::vector<PoaProblem>& probs,
                         int64_t rows, rs_replica_result* res_dev) {
  const int W = ctx->cfg.W;
  const int np = (int)probs.size();
  rs_status r;
  if ((r = ensure(ctx, ctx->p_cost, (size_t)rows * W * 8, "poa costs")) ||
      (r = ensure(ctx, ctx->p_order, (size_t)rows * 4, "poa order")) ||
      (r = ensure(ctx, ctx->p_asg, (size_t)rows * 4, "poa assignment")) ||
      (r = ensure(ctx, ctx->p_wkey, (size_t)rows * 4, "poa keys")) ||
      (r = ensure(ctx, ctx->p_tstat, (size_t)np * 8, "poa totals")) ||
      (r = ensure(ctx, ctx->p_total, (size_t)np * 8, "poa totals")) ||
      (r = ensure(ctx, ctx->p_nwin, (size_t)np * 8, "poa totals")) ||
      (r = ensure(ctx, ctx->p_prob, (size_t)np * sizeof(PoaProblem), "poa problems")) ||
      (r = ensure_pinned(ctx, (size_t)np)))
    return r;
  CK(cudaMemcpyAsync(ctx->p_prob.p, probs.data(), np * sizeof(PoaProblem), cudaMemcpyHostToDevice,
                     ctx->st),
     "copy poa problems");
  // last window of every problem (p_nwin serves as the span's output)
  CK(launch_poa_span(P<PoaProblem>(ctx->p_prob), np, rec, ctx->cfg.poa_window,
                     reinterpret_cast<long long*>(ctx->p_nwin.p), ctx->st),
     "poa span launch");
  CK(cudaMemcpyAsync(ctx->pinned, ctx->p_nwin.p, (size_t)np * 8, cudaMemcpyDeviceToHost, ctx->st),
     "read poa spans");
  CK(cudaStreamSynchronize(ctx->st), "sync");
  int64_t win_slots = 0;
  for (int k = 0; k < np; k++) {
    const int64_t last = ctx->pinned[k];   // -1: nothing routed
    if (last > (int64_t)INT32_MAX - 2)
      return fail(ctx, RS_ERR_CAPACITY,
                  "problem %d: completions span more than 2^31 - 2 PoA windows", k);
    probs[k].win_base = win_slots;
    probs[k].win_cap = last + 2;   // windows 0 .. last, and one to spare
    win_slots += probs[k].win_cap;
  }
  if ((r = ensure(ctx, ctx->p_wstart, (size_t)(win_slots + np) * 8, "poa windows")) ||
      (r = ensure(ctx, ctx->p_wfill, (size_t)win_slots * 8, "poa windows")) ||
      (r = ensure(ctx, ctx->p_wnum, (size_t)win_slots * 8, "poa windows")) ||
      (r = ensure(ctx, ctx->p_wopt, (size_t)win_slots * 8, "poa windows")) ||
      (r = ensure(ctx, ctx->p_wstat, (size_t)win_slots * 8, "poa windows")) ||
      (r = ensure(ctx, ctx->p_wcnt, (size_t)win_slots * 8, "poa windows")) ||
      (r = ensure(ctx, ctx->p_wprob, (size_t)win_slots * 4, "poa windows")) ||
      (r = ensure(ctx, ctx->p_wnext, 8, "poa work counter")))
    return r;
  CK(cudaMemcpyAsync(ctx->p_prob.p, probs.data(), np * sizeof(PoaProblem), cudaMemcpyHostToDevice,
                     ctx->st),
     "copy poa problems");
  PoaBuffers b;
  b.rec = rec;
  b.cost = P<double>(ctx->p_cost);
  b.order = P<int32_t>(ctx->p_order);
  b.asg = P<int32_t>(ctx->p_asg);
  b.wkey = P<int32_t>(ctx->p_wkey);
  b.wstart = P<int64_t>(ctx->p_wstart);
  b.wfill = P<int64_t>(ctx->p_wfill);
  b.wnum = P<double>(ctx->p_wnum);
  b.wstat = P<double>(ctx->p_wstat);
  b.wopt = P<double>(ctx->p_wopt);
  b.wcnt = P<int64_t>(ctx->p_wcnt);
  b.total = P<double>(ctx->p_total);
  b.total_static = P<double>(ctx->p_tstat);
  b.nwin = P<int64_t>(ctx->p_nwin);
  b.res = res_dev;
  b.wprob = P<int32_t>(ctx->p_wprob);
  b.wnext = P<unsigned long long>(ctx->p_wnext);
  b.nslots = win_slots;
  CK(launch_poa(P<PoaProblem>(ctx->p_prob), np, b, ctx->mc, ctx->st), "poa launch");
  return RS_OK;
}

rs_status simulate_replicas(rs_ctx* ctx, const rs_trace* traces, int32_t n_traces,
                            int32_t trace_mem, const rs_replica_params* params,
                            int32_t n_replicas, rs_replica_result* results_host,
                            const rs_records* records, int32_t flags) {
  if (!ctx) return fail(nullptr, RS_ERR_INVALID, "ctx is NULL");
  ctx->err.clear();
  if (n_replicas < 0 || n_traces < 0) return fail(ctx, RS_ERR_INVALID, "negative count");
  if (n_replicas == 0) return RS_OK;
  if (!traces || !params || !results_host) return fail(ctx, RS_ERR_INVALID, "NULL pointer");
  if (trace_mem != RS_MEM_DEVICE && trace_mem != RS_MEM_HOST)
    return fail(ctx, RS_ERR_INVALID, "trace_mem must be RS_MEM_DEVICE or RS_MEM_HOST");
  const int W = ctx->cfg.W;
  const TableGeom& g = ctx->gs;
  for (int t = 0; t < n_traces; t++) {
    const rs_trace& tr = traces[t];
    if (tr.n_req < 0) return fail(ctx, RS_ERR_INVALID, "trace %d: n_req < 0", t);
    if (tr.n_req > 0 && ((!tr.tokens && !tr.hashes) || !tr.offsets || !tr.release || !tr.out_len))
      return fail(ctx, RS_ERR_INVALID, "trace %d: NULL pointer", t);
    if (tr.n_req > 0 && tr.tokens && !aligned16(tr.tokens))
      return fail(ctx, RS_ERR_INVALID, "trace %d: tokens must be 16-byte aligned", t);
    if (tr.n_req > 0 && !tr.tokens && ((reinterpret_cast<uintptr_t>(tr.hashes) & 7u) != 0))
      return fail(ctx, RS_ERR_INVALID, "trace %d: hashes must be 8-byte aligned", t);
    if (tr.n_req > INT32_MAX) return fail(ctx, RS_ERR_CAPACITY, "trace %d: n_req > 2^31-1", t);
  }
  int64_t rows = 0, pend_cap = 0;
  int cmax = 1;
  bool any_freq = false;   // a replica evicts by frequency: its tables need fexp
  std::vector<char> used(n_traces, 0);
  for (int r = 0; r < n_replicas; r++) {
    const rs_replica_params& p = params[r];
    if (p.trace < 0 || p.trace >= n_traces) return fail(ctx, RS_ERR_INVALID, "replica %d: bad trace", r);
    if (p.C < 1 || p.C > 65535) return fail(ctx, RS_ERR_INVALID, "replica %d: C out of range", r);
    if (p.c_mid < 0 || p.c_mid > 65535 ||
        (p.c_mid > 0 && (p.c_end < 1 || p.c_end > 65535 || !(p.c_t1 >= 0.0) ||
                         !(p.c_t2 >= p.c_t1))))
      return fail(ctx, RS_ERR_INVALID, "replica %d: bad load-spike schedule", r);
    if (p.policy < RS_POLICY_DYNAMO || p.policy > RS_POLICY_P2C)
      return fail(ctx, RS_ERR_INVALID, "replica %d: bad policy", r);
    if (p.eviction != RS_EVICT_LRU && p.eviction != RS_EVICT_FREQ)
      return fail(ctx, RS_ERR_INVALID, "replica %d: bad eviction", r);
    if (p.eviction == RS_EVICT_FREQ) {
      if (p.freq_max < 1 || p.freq_max > (1 << 20))
        return fail(ctx, RS_ERR_INVALID, "replica %d: freq_max out of 1..2^20", r);
      if (!(p.decay_s > 0.0) || !std::isfinite(p.decay_s))
        return fail(ctx, RS_ERR_INVALID, "replica %d: decay_s must be finite and > 0", r);
      any_freq = true;
      if (ctx->cfg.tiered)
        return fail(ctx, RS_ERR_INVALID, "replica %d: frequency eviction with tiers", r);
    }
    if (!(p.omega >= 0.0f) || !(p.tau >= 0.0f) || !std::isfinite(p.omega) || !std::isfinite(p.tau))
      return fail(ctx, RS_ERR_INVALID, "replica %d: omega/tau must be finite and >= 0", r);
    if (p.n_req < 0 || p.n_req > traces[p.trace].n_req)
      return fail(ctx, RS_ERR_INVALID, "replica %d: n_req out of range", r);
    rows += p.n_req;
    cmax = std::max(cmax, p.C);
    if (p.c_mid > 0) cmax = std::max(cmax, std::max(p.c_mid, p.c_end));
    if (p.controller) pend_cap = std::max(pend_cap, p.n_req);
    used[p.trace] = 1;
  }
  const bool host = trace_mem == RS_MEM_HOST;
  rs_status r;
  // ---- trace geometry; host traces are staged on the device
  std::vector<int64_t> tot(n_traces, 0), hoff(n_traces, 0), rbase(n_traces, 0);
  std::vector<const int32_t*> dtok(n_traces);
  std::vector<const int64_t*> doff(n_traces);
  std::vector<const double*> drel(n_traces);
  std::vector<const int32_t*> dol(n_traces);
  // a trace given by its block hashes (tokens NULL) skips S1
  auto prehashed = [&](int t) { return traces[t].tokens == nullptr; };
  std::vector<const uint64_t*> dhash(n_traces, nullptr);
  if (host) {
    size_t tb = 0, ob = 0, nb = 0, hb = 0;
    for (int t = 0; t < n_traces; t++) {
      if (!used[t] || traces[t].n_req == 0) continue;
      const int64_t n = traces[t].n_req;
      tot[t] = traces[t].offsets[n];
      if (tot[t] < 0) return fail(ctx, RS_ERR_INVALID, "trace %d: offsets[n_req] < 0", t);
      if (prehashed(t))
        hb += (size_t)(tot[t] / 16 + 1) * 8;
      else
        tb += ((size_t)(tot[t] + 3) / 4 * 4) * 4 + 16;
      ob += (size_t)(n + 1) * 8;
      nb += (size_t)n;
    }
    if ((r = ensure(ctx, ctx->h_tokens, tb, "staged tokens")) ||
        (r = ensure(ctx, ctx->h_hashes, hb, "staged block hashes")) ||
        (r = ensure(ctx, ctx->h_offsets, ob, "staged offsets")) ||
        (r = ensure(ctx, ctx->h_release, nb * 8, "staged release")) ||
        (r = ensure(ctx, ctx->h_outlen, nb * 4, "staged out_len")))
      return r;
    size_t to = 0, ho = 0, oo = 0, no = 0;
    for (int t = 0; t < n_traces; t++) {
      if (!used[t] || traces[t].n_req == 0) continue;
      const int64_t n = traces[t].n_req;
      if (prehashed(t)) {
        const size_t hbytes = (size_t)(tot[t] / 16) * 8;
        uint64_t* hp = P<uint64_t>(ctx->h_hashes) + ho;
        if (hbytes)
          CK(cudaMemcpyAsync(hp, traces[t].hashes, hbytes, cudaMemcpyHostToDevice, ctx->st),
             "H2D hashes");
        dhash[t] = hp;
        ho += (size_t)(tot[t] / 16 + 1);
      } else {
        const size_t tbytes = (size_t)(tot[t] + 3) / 4 * 4 * 4;
        char* tp = static_cast<char*>(ctx->h_tokens.p) + to;
        CK(cudaMemcpyAsync(tp, traces[t].tokens, tbytes, cudaMemcpyHostToDevice, ctx->st),
           "H2D tokens");
        dtok[t] = reinterpret_cast<const int32_t*>(tp);
        to += (tbytes + 15) & ~(size_t)15;
      }
      CK(cudaMemcpyAsync(P<int64_t>(ctx->h_offsets) + oo, traces[t].offsets, (n + 1) * 8,
                         cudaMemcpyHostToDevice, ctx->st), "H2D offsets");
      CK(cudaMemcpyAsync(P<double>(ctx->h_release) + no, traces[t].release, n * 8,
                         cudaMemcpyHostToDevice, ctx->st), "H2D release");
      CK(cudaMemcpyAsync(P<int32_t>(ctx->h_outlen) + no, traces[t].out_len, n * 4,
                         cudaMemcpyHostToDevice, ctx->st), "H2D out_len");
      doff[t] = P<int64_t>(ctx->h_offsets) + oo;
      drel[t] = P<double>(ctx->h_release) + no;
      dol[t] = P<int32_t>(ctx->h_outlen) + no;
      oo += n + 1;
      no += n;
    }
  } else {
    if ((r = ensure_pinned(ctx, (size_t)n_traces + 1)) != RS_OK) return r;
    for (int t = 0; t < n_traces; t++) {
      dtok[t] = traces[t].tokens;
      dhash[t] = prehashed(t) ? traces[t].hashes : nullptr;
      doff[t] = traces[t].offsets;
      drel[t] = traces[t].release;
      dol[t] = traces[t].out_len;
      if (used[t] && traces[t].n_req > 0)
        CK(cudaMemcpyAsync(ctx->pinned + t, traces[t].offsets + traces[t].n_req, 8,
                           cudaMemcpyDeviceToHost, ctx->st), "read offsets");
    }
    CK(cudaStreamSynchronize(ctx->st), "sync");
    for (int t = 0; t < n_traces; t++)
      if (used[t] && traces[t].n_req > 0) tot[t] = ctx->pinned[t];
  }
  size_t hash_total = 0;
  for (int t = 0; t < n_traces; t++) {
    if (tot[t] < 0) return fail(ctx, RS_ERR_INVALID, "trace %d: offsets[n_req] < 0", t);
    hoff[t] = (int64_t)hash_total;
    if (used[t] && !dhash[t]) hash_total += (size_t)(tot[t] / 16 + 1);
  }
  if ((r = ensure(ctx, ctx->hashes, hash_total * 8, "block hashes")) ||
      (r = ensure(ctx, ctx->stats, (size_t)n_traces * 8, "trace stats")) ||
      (r = ensure_pinned(ctx, (size_t)n_traces + 1)))
    return r;
  // ---- K1: block hashes of every trace in use that comes as tokens.  The
  // hash jobs number their requests among themselves; the per-request flags
  // number the requests of every trace in use (rbase).
  int64_t launches = 0, hashed_tokens = 0;
  std::vector<HashJob> jobs, all;
  int64_t req_total = 0, hreq = 0;
  for (int t = 0; t < n_traces; t++) {
    if (!used[t] || traces[t].n_req == 0) continue;
    rbase[t] = req_total;
    uint64_t* hp = dhash[t] ? const_cast<uint64_t*>(dhash[t]) : P<uint64_t>(ctx->hashes) + hoff[t];
    all.push_back(HashJob{dtok[t], doff[t], hp, traces[t].n_req, req_total});
    if (!dhash[t]) {
      jobs.push_back(HashJob{dtok[t], doff[t], hp, traces[t].n_req, hreq});
      hreq += traces[t].n_req;
      hashed_tokens += tot[t];
    }
    req_total += traces[t].n_req;
  }
  if ((r = ensure(ctx, ctx->hjobs, sizeof(HashJob) * std::max<size_t>(jobs.size(), 1), "hash jobs")) ||
      (r = ensure(ctx, ctx->djobs, sizeof(HashJob) * std::max<size_t>(all.size(), 1), "trace jobs")))
    return r;
  std::vector<HashJob> hj = group_jobs(jobs);
  if (!jobs.empty())
    CK(cudaMemcpyAsync(ctx->hjobs.p, hj.data(), sizeof(HashJob) * hj.size(), cudaMemcpyHostToDevice,
                       ctx->st), "copy hash jobs");
  std::vector<HashJob> aj = group_jobs(all);
  CK(cudaMemcpyAsync(ctx->djobs.p, aj.data(), sizeof(HashJob) * aj.size(), cudaMemcpyHostToDevice,
                     ctx->st), "copy trace jobs");
  CK(cudaMemsetAsync(ctx->stats.p, 0, (size_t)n_traces * 8, ctx->st), "memset");
  // the events time the hash launches alone
  CK(cudaEventRecord(ctx->ev[0], ctx->st), "event");
  for (size_t g0 = 0; g0 < jobs.size(); g0 += HASH_MAX_JOBS) {
    const size_t g1 = std::min(jobs.size(), g0 + HASH_MAX_JOBS);
    const int64_t total = jobs[g1 - 1].req_base + jobs[g1 - 1].n_req - jobs[g0].req_base;
    CK(launch_block_hash(P<HashJob>(ctx->hjobs) + g0, (int)(g1 - g0), total, ctx->cfg.hash_seed,
                         nullptr, ctx->st),
       "block hash launch");
    launches++;
  }
  CK(cudaEventRecord(ctx->ev[1], ctx->st), "event");
  // the longest prompt's full blocks, over every trace in use
  for (size_t g0 = 0; g0 < all.size(); g0 += HASH_MAX_JOBS) {
    const size_t g1 = std::min(all.size(), g0 + HASH_MAX_JOBS);
    const int64_t total = all[g1 - 1].req_base + all[g1 - 1].n_req - all[g0].req_base;
    CK(launch_nbmax(P<HashJob>(ctx->djobs) + g0, (int)(g1 - g0), total, P<int64_t>(ctx->stats),
                    ctx->st),
       "block count launch");
    launches++;
  }
  CK(cudaMemcpyAsync(ctx->pinned, ctx->stats.p, 8, cudaMemcpyDeviceToHost, ctx->st), "read stats");
  CK(cudaStreamSynchronize(ctx->st), "sync");
  int64_t nbmax = std::max<int64_t>(1, ctx->pinned[0]);
  if (nbmax > (int64_t)g.K) nbmax = g.K;   // longer prompts stop their replica with RS_ERR_CAPACITY
  int maxsmem = 0;
  cudaDeviceGetAttribute(&maxsmem, cudaDevAttrMaxSharedMemoryPerBlockOptin, ctx->device);
  const size_t smem_room = (size_t)maxsmem > sizeof(int) * 2048 ? maxsmem - sizeof(int) * 2048 : 0;
  // per-request slot arrays in shared memory when they fit, else in global memory
  bool slots_global = false;
  const bool tiered = ctx->cfg.tiered != 0;
  if (tiered && (int64_t)W * nbmax > SIM_PROBE_CAP)
    return fail(ctx, RS_ERR_CAPACITY,
                "tiers need W * (longest prompt's full blocks) <= %d; have %d * %lld", SIM_PROBE_CAP,
                W, (long long)nbmax);
  size_t smem = sim_smem_bytes(W, (int)nbmax, cmax, ctx->cfg.cap, false, tiered);
  if (smem > smem_room) {
    slots_global = true;
    smem = sim_smem_bytes(W, (int)nbmax, cmax, ctx->cfg.cap, true, tiered);
  }
  if (smem > smem_room)
    return fail(ctx, RS_ERR_CAPACITY,
                "prompt of %lld blocks needs %zu bytes of shared memory per replica",
                (long long)nbmax, smem);
  // ---- scratch
  const size_t nsim = n_replicas;
  const size_t nsl = nsim * W * g.slots;
  if ((r = ensure(ctx, ctx->keys, nsl * 8, "cache keys")) ||
      (r = ensure(ctx, ctx->stamp, nsl * 4, "cache stamps")) ||
      (r = ensure(ctx, ctx->log, nsim * W * g.R * 4, "cache logs")) ||
      (r = ensure(ctx, ctx->tmp, nsim * g.K * 8, "rebuild scratch")) ||
      (r = ensure(ctx, ctx->pend, nsim * 5 * (size_t)std::max<int64_t>(pend_cap, 1) * 8, "controller windows")) ||
      (r = ensure(ctx, ctx->meta_out, nsim * W * sizeof(CacheMeta), "cache meta")) ||
      (r = ensure(ctx, ctx->res, nsim * sizeof(rs_replica_result), "results")) ||
      (r = ensure(ctx, ctx->desc, nsim * sizeof(SimDesc), "replica descriptors")) ||
      (r = ensure(ctx, ctx->dupf, (size_t)std::max<int64_t>(req_total, 1), "duplicate flags")) ||
      (r = ensure(ctx, ctx->dstat, (size_t)std::max<int64_t>(rows, 1) * 6 * sizeof(float),
                  "decision statistics")))
    return r;
  if (slots_global &&
      (r = ensure(ctx, ctx->slots, nsim * sim_slot_bytes(cmax), "request slots")) != RS_OK)
    return r;
  if (any_freq && ((r = ensure(ctx, ctx->fexp, nsl * 4, "frequency state")) ||
                   (r = ensure(ctx, ctx->tmpe, nsim * g.K * 4, "frequency rebuild scratch"))))
    return r;
  // w_c * (m / nbt) table for prompts up to nbmax blocks (none beyond 2048)
  const bool use_tab = nbmax <= 2048;
  if (use_tab &&
      (r = ensure(ctx, ctx->wco, (size_t)(nbmax + 1) * (nbmax + 2) * sizeof(double), "w_c o table")))
    return r;
  rs_records rec;
  const bool want_cost = records && records->cost;
  if ((r = records_effective(ctx, records, rows, W, want_cost, &rec)) != RS_OK) return r;
  std::vector<SimDesc> desc(nsim);
  std::vector<PoaProblem> probs(nsim);
  int64_t rb = 0;
  for (size_t k = 0; k < nsim; k++) {
    const rs_replica_params& p = params[k];
    SimDesc& d = desc[k];
    d.offsets = doff[p.trace];
    d.release = drel[p.trace];
    d.out_len = dol[p.trace];
    d.hashes = dhash[p.trace] ? dhash[p.trace] : P<uint64_t>(ctx->hashes) + hoff[p.trace];
    d.dupflag = P<uint8_t>(ctx->dupf) + rbase[p.trace];
    d.n_req = p.n_req;
    d.rec_base = rb;
    d.C = p.C;
    d.c_t1 = p.c_t1;
    d.c_t2 = p.c_t2;
    d.c_mid = p.c_mid > 0 ? p.c_mid : 0;
    d.c_end = p.c_mid > 0 ? p.c_end : 0;
    d.policy = p.policy;
    d.controller = p.controller ? 1 : 0;
    d.eviction = p.eviction;
    d.freq_max = p.eviction == RS_EVICT_FREQ ? p.freq_max : 1;
    d.reserved = 0;
    d.decay_s = p.eviction == RS_EVICT_FREQ ? p.decay_s : 1.0;
    d.omega = p.omega;
    d.tau = p.tau;
    d.seed = p.seed;
    probs[k].rec_base = rb;
    probs[k].n = p.n_req;
    probs[k].scratch_base = rb;
    rb += p.n_req;
  }
  CK(cudaMemcpyAsync(ctx->desc.p, desc.data(), nsim * sizeof(SimDesc), cudaMemcpyHostToDevice, ctx->st),
     "copy descriptors");
  SimBuffers sb;
  sb.keys = P<uint64_t>(ctx->keys);
  sb.stamp = P<uint32_t>(ctx->stamp);
  sb.log = P<uint32_t>(ctx->log);
  sb.tmp = P<uint64_t>(ctx->tmp);
  sb.fexp = any_freq ? P<uint32_t>(ctx->fexp) : nullptr;
  sb.tmpe = any_freq ? P<uint32_t>(ctx->tmpe) : nullptr;
  sb.pend = P<double>(ctx->pend);
  sb.pend_cap = std::max<int64_t>(pend_cap, 1);
  sb.meta_out = P<CacheMeta>(ctx->meta_out);
  sb.res = P<rs_replica_result>(ctx->res);
  sb.rec = rec;
  sb.dstat = P<float>(ctx->dstat);
  sb.wco_tab = use_tab ? P<double>(ctx->wco) : nullptr;
  sb.wco_dim = (int)nbmax + 2;
  sb.slotmem = slots_global ? P<unsigned char>(ctx->slots) : nullptr;
  SimLaunch L;
  L.nsim = (int)nsim;
  L.nbmax = (int)nbmax;
  L.tiered = tiered ? 1 : 0;
  L.k1 = ctx->cfg.cache_blocks;
  L.k12 = ctx->cfg.cache_blocks + (tiered ? ctx->cfg.tier_k2 : 0);
  L.cmax = cmax;
  L.slots_global = slots_global ? 1 : 0;
  L.g = g;
  L.mc = ctx->mc;
  L.mc.write_cost = want_cost ? 1 : 0;
  if (use_tab) {
    CK(launch_wco_table(P<double>(ctx->wco), (int)nbmax, ctx->cfg.w_c, ctx->st), "table launch");
    launches++;
  }
  // per-request duplicate-hash flags of every trace in use
  for (size_t g0 = 0; g0 < all.size(); g0 += HASH_MAX_JOBS) {
    const size_t g1 = std::min(all.size(), g0 + HASH_MAX_JOBS);
    const int64_t base = all[g0].req_base;
    const int64_t total = all[g1 - 1].req_base + all[g1 - 1].n_req - base;
    CK(launch_dup_flags(P<HashJob>(ctx->djobs) + g0, (int)(g1 - g0), total, nbmax,
                        P<uint8_t>(ctx->dupf) + base, ctx->st),
       "duplicate flags launch");
    launches++;
  }
  CK(launch_sim(P<SimDesc>(ctx->desc), sb, L, ctx->st), "simulation launch");
  CK(launch_decision_stats(P<SimDesc>(ctx->desc), sb, L, ctx->st), "statistics launch");
  launches += 2;
  CK(cudaEventRecord(ctx->ev[2], ctx->st), "event");
  if (!(flags & RS_SIM_NO_POA)) {
    if ((r = run_poa(ctx, rec, probs, rows, sb.res)) != RS_OK) return r;
    launches += 4;
  }
  CK(cudaEventRecord(ctx->ev[3], ctx->st), "event");
  CK(cudaMemcpyAsync(results_host, sb.res, nsim * sizeof(rs_replica_result), cudaMemcpyDeviceToHost,
                     ctx->st),
     "read results");
  CK(cudaStreamSynchronize(ctx->st), "sync");
  ctx->last_nsim = (int32_t)nsim;
  float ms[3] = {0, 0, 0};
  cudaEventElapsedTime(&ms[0], ctx->ev[0], ctx->ev[1]);
  cudaEventElapsedTime(&ms[1], ctx->ev[1], ctx->ev[2]);
  cudaEventElapsedTime(&ms[2], ctx->ev[2], ctx->ev[3]);
  ctx->timing.hash_ms = ms[0];
  ctx->timing.sim_ms = ms[1];
  ctx->timing.poa_ms = ms[2];
  ctx->timing.total_ms = ms[0] + ms[1] + ms[2];
  ctx->timing.launches = launches;
  ctx->timing.hashed_tokens = hashed_tokens;
  for (size_t k = 0; k < nsim; k++)
    if (results_host[k].status != RS_OK)
      return fail(ctx, (rs_status)results_host[k].status, "replica %zu stopped with status %d", k,
                  results_host[k].status);
  return RS_OK;
}

rs_status poa_estimate(rs_ctx* ctx, const rs_records* records, int64_t n, double* numer_host,
                       double* opt_host, int64_t* count_host, int64_t* n_windows_inout,
                       double* poa_total_host) {
  if (!ctx) return fail(nullptr, RS_ERR_INVALID, "ctx is NULL");
  ctx->err.clear();
  if (!records || !n_windows_inout || !poa_total_host) return fail(ctx, RS_ERR_INVALID, "NULL pointer");
  if (n < 0 || n > INT32_MAX) return fail(ctx, RS_ERR_INVALID, "n out of range");
  const rs_records& u = *records;
  if (n > 0 && (!u.worker || !u.completion || !u.ttft || !u.nbt || !u.n_frozen || !u.prefix))
    return fail(ctx, RS_ERR_INVALID, "records need worker, completion, ttft, nbt, n_frozen, prefix");
  if (ctx->cfg.W > POA_WMAX_WIDE)
    return fail(ctx, RS_ERR_INVALID, "the PoA estimator supports W <= %d", POA_WMAX_WIDE);
  std::vector<PoaProblem> probs(1);
  probs[0].rec_base = 0;
  probs[0].n = n;
  probs[0].scratch_base = 0;
  rs_status r = run_poa(ctx, u, probs, std::max<int64_t>(n, 1), nullptr);
  if (r != RS_OK) return r;
  const int64_t cap = *n_windows_inout;
  if ((r = ensure_pinned(ctx, 2)) != RS_OK) return r;
  CK(cudaMemcpyAsync(ctx->pinned, ctx->p_nwin.p, 8, cudaMemcpyDeviceToHost, ctx->st), "read");
  CK(cudaMemcpyAsync(ctx->pinned + 1, ctx->p_total.p, 8, cudaMemcpyDeviceToHost, ctx->st), "read");
  CK(cudaStreamSynchronize(ctx->st), "sync");
  const int64_t nw = ctx->pinned[0];
  double tot;
  memcpy(&tot, ctx->pinned + 1, 8);
  if (nw < 0)
    return fail(ctx, RS_ERR_INVALID, "a routed row has a negative or non-finite completion time");
  *n_windows_inout = nw;
  *poa_total_host = tot;
  const int64_t k = std::min(cap, nw);
  if (k > 0) {
    if (numer_host) CK(cudaMemcpyAsync(numer_host, ctx->p_wnum.p, k * 8, cudaMemcpyDeviceToHost, ctx->st), "read");
    if (opt_host) CK(cudaMemcpyAsync(opt_host, ctx->p_wopt.p, k * 8, cudaMemcpyDeviceToHost, ctx->st), "read");
    if (count_host) CK(cudaMemcpyAsync(count_host, ctx->p_wcnt.p, k * 8, cudaMemcpyDeviceToHost, ctx->st), "read");
    CK(cudaStreamSynchronize(ctx->st), "sync");
  }
  return RS_OK;
}

rs_status sweep_knee(rs_ctx* ctx, const rs_records* records, const int64_t* row_start,
                     int32_t n_replicas, const double* load, const int32_t* sweep_start,
                     int32_t n_sweeps, int32_t pct, double theta, double* stat_host,
                     double* d1_host, double* d2_host, double* knee_load_host,
                     int32_t* knee_index_host) {
  if (!ctx) return fail(nullptr, RS_ERR_INVALID, "ctx is NULL");
  ctx->err.clear();
  if (!records || !row_start || !sweep_start) return fail(ctx, RS_ERR_INVALID, "NULL pointer");
  if (n_replicas < 0 || n_sweeps < 0) return fail(ctx, RS_ERR_INVALID, "negative count");
  if (pct < 1 || pct > 100) return fail(ctx, RS_ERR_INVALID, "pct must be in 1..100");
  if (std::isnan(theta)) return fail(ctx, RS_ERR_INVALID, "theta is NaN");
  if (row_start[0] < 0) return fail(ctx, RS_ERR_INVALID, "row_start[0] < 0");
  for (int32_t r = 0; r < n_replicas; r++)
    if (row_start[r + 1] < row_start[r])
      return fail(ctx, RS_ERR_INVALID, "row_start decreases at replica %d", r);
  const int64_t rows = row_start[n_replicas];
  if (rows > 0 && (!records->worker || !records->ttft))
    return fail(ctx, RS_ERR_INVALID, "records need worker and ttft");
  if (n_replicas > 0 && !load) return fail(ctx, RS_ERR_INVALID, "load is NULL");
  if (sweep_start[0] < 0) return fail(ctx, RS_ERR_INVALID, "sweep_start[0] < 0");
  for (int32_t s = 0; s < n_sweeps; s++)
    if (sweep_start[s + 1] < sweep_start[s])
      return fail(ctx, RS_ERR_INVALID, "sweep_start decreases at sweep %d", s);
  if (sweep_start[n_sweeps] > n_replicas)
    return fail(ctx, RS_ERR_INVALID, "sweeps reach past the replicas");
  const size_t nr = (size_t)n_replicas, ns = (size_t)n_sweeps;
  rs_status r;
  if ((r = ensure(ctx, ctx->k_rows, (nr + 1) * 8, "knee rows")) != RS_OK) return r;
  if ((r = ensure(ctx, ctx->k_load, nr * 8, "knee load")) != RS_OK) return r;
  if ((r = ensure(ctx, ctx->k_sweep, (ns + 1) * 4, "knee sweeps")) != RS_OK) return r;
  if ((r = ensure(ctx, ctx->k_stat, nr * 8, "knee stat")) != RS_OK) return r;
  if ((r = ensure(ctx, ctx->k_d1, nr * 8, "knee d1")) != RS_OK) return r;
  if ((r = ensure(ctx, ctx->k_d2, nr * 8, "knee d2")) != RS_OK) return r;
  if ((r = ensure(ctx, ctx->k_kload, ns * 8, "knee load out")) != RS_OK) return r;
  if ((r = ensure(ctx, ctx->k_kidx, ns * 4, "knee index out")) != RS_OK) return r;
  CK(cudaMemcpyAsync(ctx->k_rows.p, row_start, (nr + 1) * 8, cudaMemcpyHostToDevice, ctx->st), "copy");
  if (nr) CK(cudaMemcpyAsync(ctx->k_load.p, load, nr * 8, cudaMemcpyHostToDevice, ctx->st), "copy");
  CK(cudaMemcpyAsync(ctx->k_sweep.p, sweep_start, (ns + 1) * 4, cudaMemcpyHostToDevice, ctx->st), "copy");
  CK(launch_sweep_knee(records->worker, records->ttft, P<int64_t>(ctx->k_rows), n_replicas,
                       P<double>(ctx->k_load), P<int32_t>(ctx->k_sweep), n_sweeps, pct, theta,
                       P<double>(ctx->k_stat), P<double>(ctx->k_d1), P<double>(ctx->k_d2),
                       P<double>(ctx->k_kload), P<int32_t>(ctx->k_kidx), ctx->st),
     "knee launch");
  if (nr) {
    if (stat_host) CK(cudaMemcpyAsync(stat_host, ctx->k_stat.p, nr * 8, cudaMemcpyDeviceToHost, ctx->st), "read");
    if (d1_host) CK(cudaMemcpyAsync(d1_host, ctx->k_d1.p, nr * 8, cudaMemcpyDeviceToHost, ctx->st), "read");
    if (d2_host) CK(cudaMemcpyAsync(d2_host, ctx->k_d2.p, nr * 8, cudaMemcpyDeviceToHost, ctx->st), "read");
  }
  if (ns) {
    if (knee_load_host) CK(cudaMemcpyAsync(knee_load_host, ctx->k_kload.p, ns * 8, cudaMemcpyDeviceToHost, ctx->st), "read");
    if (knee_index_host) CK(cudaMemcpyAsync(knee_index_host, ctx->k_kidx.p, ns * 4, cudaMemcpyDeviceToHost, ctx->st), "read");
  }
  CK(cudaStreamSynchronize(ctx->st), "sync");
  return RS_OK;
}

rs_status route_cache_dump(rs_ctx* ctx, int32_t source, int32_t index, int32_t worker,
                           uint64_t* keys_host, int64_t capacity, int64_t* size) {
  if (!ctx) return fail(nullptr, RS_ERR_INVALID, "ctx is NULL");
  ctx->err.clear();
  if (!size || (capacity > 0 && !keys_host)) return fail(ctx, RS_ERR_INVALID, "NULL pointer");
  const int W = ctx->cfg.W;
  if (worker < 0 || worker >= W) return fail(ctx, RS_ERR_INVALID, "worker out of range");
  const TableGeom& g = source == 1 ? ctx->gs : ctx->g;
  const uint64_t* kp;
  const uint32_t* sp;
  const uint32_t* lp;
  const CacheMeta* mp;
  if (source == 0) {
    RouterState s;
    rs_status r = router_state(ctx, index, &s);
    if (r != RS_OK) return r;
    kp = s.keys + (size_t)worker * g.slots;
    sp = s.stamp + (size_t)worker * g.slots;
    lp = s.log + (size_t)worker * g.R;
    mp = s.meta + worker;
  } else if (source == 1) {
    if (index < 0 || index >= ctx->last_nsim) return fail(ctx, RS_ERR_INVALID, "replica out of range");
    const size_t wi = (size_t)index * W + worker;
    kp = P<uint64_t>(ctx->keys) + wi * g.slots;
    sp = P<uint32_t>(ctx->stamp) + wi * g.slots;
    lp = P<uint32_t>(ctx->log) + wi * g.R;
    mp = P<CacheMeta>(ctx->meta_out) + wi;
  } else {
    return fail(ctx, RS_ERR_INVALID, "source must be 0 or 1");
  }
  std::vector<uint64_t> keys(g.slots);
  std::vector<uint32_t> stamps(g.slots), log(g.R);
  CacheMeta m;
  CK(cudaMemcpyAsync(keys.data(), kp, g.slots * 8, cudaMemcpyDeviceToHost, ctx->st), "read");
  CK(cudaMemcpyAsync(stamps.data(), sp, g.slots * 4, cudaMemcpyDeviceToHost, ctx->st), "read");
  CK(cudaMemcpyAsync(log.data(), lp, g.R * 4, cudaMemcpyDeviceToHost, ctx->st), "read");
  CK(cudaMemcpyAsync(&m, mp, sizeof m, cudaMemcpyDeviceToHost, ctx->st), "read");
  CK(cudaStreamSynchronize(ctx->st), "sync");
  int64_t k = 0;
  for (uint32_t t = m.head; t < m.T; t++) {
    const uint32_t x = log[t & g.rmask];
    if (x < g.slots && stamps[x] == t) {
      if (k < capacity) keys_host[k] = keys[x];
      k++;
    }
  }
  *size = k;
  if (k != (int64_t)m.size)
    return fail(ctx, RS_ERR_STATE, "cache of worker %d holds %lld live entries, size says %u", worker,
                (long long)k, m.size);
  return RS_OK;
}

rs_status route_last_timing(const rs_ctx* ctx, rs_timing* out) {
  if (!ctx || !out) return RS_ERR_INVALID;
  *out = ctx->timing;
  return RS_OK;
}

}  // extern "C"
