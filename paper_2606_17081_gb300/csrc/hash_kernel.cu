// KV block hashing of prompts (K1), in two passes over all traces of a call.
//
// Content pass (k_block_content): one warp per request, lane l takes blocks
// l and l + 32 of each 64-block span; a block's 64 bytes arrive as four
// 16-byte loads (five when the request does not start on a 16-byte boundary)
// and fold into the content hash g_k; the lane stores g_k ^ k at the block's
// output slot.  Fully parallel, coalesced, HBM-bound: 4 bytes per token in,
// 8 bytes per block out.
//
// Chain pass (k_block_chain): h_k = mix(h_{k-1} ^ g_k ^ k) is serial per
// request, so each lane owns one request at a time and each round moves every
// lane's request on by a chunk of 32 blocks: per request the warp reads the
// chunk's 32 values with one coalesced 256-byte load into shared memory,
// every lane folds its own row in order, and per request the warp writes the
// 32 hashes back with one coalesced store.  Lanes whose requests are done
// claim the next ones from a work counter (one atomic per warp for all of
// them), so the warps stay busy until the counter runs out.  The content pass
// lists the long prompts (HASH_LONG_NB blocks and more), and the counter hands
// those out first: their chains, serial and up to hundreds of blocks long,
// overlap the bulk instead of trailing it.  8 bytes per block in and out.
#include <climits>

#include "rs_device.cuh"

namespace rs {

constexpr int CONTENT_NT = 256;              // content pass: threads per CTA
constexpr int CHAIN_WARPS = 4;               // chain pass: warps per CTA
constexpr int CHAIN_NT = 32 * CHAIN_WARPS;
constexpr int CHAIN_ROW = 33;                // 32 staged blocks per request + 1 pad word
constexpr int CHAIN_ILP = 8;                 // requests whose chunks are loaded together
constexpr int64_t HASH_LONG_NB = 96;         // prompts of this many blocks are chained first

template <int S>
__device__ __forceinline__ void take16(const uint32_t (&a)[20], uint32_t (&w)[16]) {
#pragma unroll
  for (int j = 0; j < 16; j++) w[j] = a[j + S];
}

// The 64 bytes of one block starting `shift` int32 words into five int4.
struct BlockBytes {
  int4 v0, v1, v2, v3, v4;
};

__device__ __forceinline__ BlockBytes load_block(const int4* q, int shift) {
  BlockBytes b;
  b.v0 = __ldg(q);
  b.v1 = __ldg(q + 1);
  b.v2 = __ldg(q + 2);
  b.v3 = __ldg(q + 3);
  b.v4 = shift ? __ldg(q + 4) : make_int4(0, 0, 0, 0);
  return b;
}

__device__ __forceinline__ uint64_t content_of(const BlockBytes& b, int shift) {
  const uint32_t a[20] = {(uint32_t)b.v0.x, (uint32_t)b.v0.y, (uint32_t)b.v0.z, (uint32_t)b.v0.w,
                          (uint32_t)b.v1.x, (uint32_t)b.v1.y, (uint32_t)b.v1.z, (uint32_t)b.v1.w,
                          (uint32_t)b.v2.x, (uint32_t)b.v2.y, (uint32_t)b.v2.z, (uint32_t)b.v2.w,
                          (uint32_t)b.v3.x, (uint32_t)b.v3.y, (uint32_t)b.v3.z, (uint32_t)b.v3.w,
                          (uint32_t)b.v4.x, (uint32_t)b.v4.y, (uint32_t)b.v4.z, (uint32_t)b.v4.w};
  uint32_t w[16];
  switch (shift) {
    case 0: take16<0>(a, w); break;
    case 1: take16<1>(a, w); break;
    case 2: take16<2>(a, w); break;
    default: take16<3>(a, w); break;
  }
  return block_content16(w);
}

__device__ __forceinline__ int find_job(const HashJob* jobs, int njobs, int64_t r) {
  int j = 0;
  while (j + 1 < njobs && r >= jobs[j + 1].req_base) j++;
  return j;
}

__global__ void __launch_bounds__(CONTENT_NT) k_block_content(const HashJob* __restrict__ jobs,
                                                              int njobs, int64_t total_req,
                                                              HashSched* __restrict__ sched,
                                                              int64_t* __restrict__ long_list) {
  __shared__ HashJob s_jobs[HASH_MAX_JOBS];
  for (int j = threadIdx.x; j < njobs; j += CONTENT_NT) s_jobs[j] = jobs[j];
  __syncthreads();
  const int lane = threadIdx.x & 31;
  const int64_t warp0 = ((int64_t)blockIdx.x * CONTENT_NT + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * CONTENT_NT) >> 5;
  for (int64_t r = warp0; r < total_req; r += nwarps) {
    const HashJob& J = s_jobs[find_job(s_jobs, njobs, r)];
    const int64_t i = r - J.req_base;
    const int64_t o0 = __ldg(J.offsets + i);
    const int64_t nb = (__ldg(J.offsets + i + 1) - o0) >> 4;
    const int shift = (int)(o0 & 3);
    const int4* q = reinterpret_cast<const int4*>(J.tokens) + (o0 >> 2);
    uint64_t* out = J.out + (o0 >> 4);
    if (lane == 0 && nb >= HASH_LONG_NB)   // its chain goes first in the chain pass
      long_list[atomicAdd(&sched->nlong, 1ull)] = r;
    for (int64_t k0 = 0; k0 < nb; k0 += 64) {
      // both blocks' loads go out before either is folded
      const int64_t ka = k0 + lane, kb = ka + 32;
      const bool va = ka < nb, vb = kb < nb;
      BlockBytes ba, bb;
      if (va) ba = load_block(q + 4 * ka, shift);
      if (vb) bb = load_block(q + 4 * kb, shift);
      if (va) out[ka] = content_of(ba, shift) ^ (uint64_t)ka;
      if (vb) out[kb] = content_of(bb, shift) ^ (uint64_t)kb;
    }
  }
}

__global__ void __launch_bounds__(CHAIN_NT) k_block_chain(const HashJob* __restrict__ jobs,
                                                          int njobs, int64_t total_req,
                                                          uint64_t seed,
                                                          int64_t* __restrict__ nbmax,
                                                          HashSched* __restrict__ sched,
                                                          const int64_t* __restrict__ long_list) {
  __shared__ HashJob s_jobs[HASH_MAX_JOBS];
  __shared__ uint64_t s_stage[CHAIN_WARPS][32 * CHAIN_ROW];
  __shared__ int64_t s_max[CHAIN_WARPS];
  for (int j = threadIdx.x; j < njobs; j += CHAIN_NT) s_jobs[j] = jobs[j];
  __syncthreads();
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const unsigned lt_mask = (1u << lane) - 1u;
  uint64_t* stage = s_stage[wid];
  uint64_t* row = stage + lane * CHAIN_ROW;
  int64_t local_max = 0;
  // indices 0 .. nlong-1 of the work counter are the long prompts, then come
  // all requests in order (long ones skipped: they are chained already)
  const int64_t nlong = (int64_t)sched->nlong;
  const int64_t nidx = nlong + total_req;
  bool exhausted = false;   // the work counter has passed the last index (warp-uniform)
  // this lane's request: blocks [c0, nb) of the hashes at oaddr, chain value h
  bool has = false;
  unsigned long long oaddr = 0;
  int64_t nb = 0, c0 = 0;
  uint64_t h = seed;
  for (;;) {
    // ---- lanes without a request claim the next ones, one atomic per warp
    unsigned need = __ballot_sync(FULL_MASK, !has);
    while (need && !exhausted) {
      const int cnt = __popc(need);
      unsigned long long b = 0;
      if (lane == 0) b = atomicAdd(&sched->work, (unsigned long long)cnt);
      b = __shfl_sync(FULL_MASK, b, 0);
      if ((int64_t)b + cnt >= nidx) exhausted = true;
      const int64_t v = (int64_t)b + __popc(need & lt_mask);
      const bool listed = v < nlong;
      const int64_t r = listed ? long_list[v] : v - nlong;
      if (!has && v < nidx) {
        const HashJob& J = s_jobs[find_job(s_jobs, njobs, r)];
        const int64_t i = r - J.req_base;
        const int64_t o0 = __ldg(J.offsets + i);
        nb = (__ldg(J.offsets + i + 1) - o0) >> 4;
        oaddr = (unsigned long long)(J.out + (o0 >> 4));
        c0 = 0;
        h = seed;
        local_max = nb > local_max ? nb : local_max;
        // a prompt without a full block has nothing to chain; a long one
        // reached in order was chained from the list
        has = nb > 0 && (listed || nb < HASH_LONG_NB);
      }
      need = __ballot_sync(FULL_MASK, !has);
    }
    const unsigned busy = __ballot_sync(FULL_MASK, has);
    if (!busy) break;
    // ---- 1. every busy lane's chunk into its row, CHAIN_ILP requests at a time
    unsigned act = busy;
    while (act) {
      int rq[CHAIN_ILP];
      bool vq[CHAIN_ILP];
      uint64_t gq[CHAIN_ILP];
#pragma unroll
      for (int u = 0; u < CHAIN_ILP; u++) {
        rq[u] = act ? __ffs(act) - 1 : -1;
        act &= act - 1;   // no-op once empty
      }
#pragma unroll
      for (int u = 0; u < CHAIN_ILP; u++) {
        const int src = rq[u] < 0 ? 0 : rq[u];
        const int64_t nbu = __shfl_sync(FULL_MASK, nb, src);
        const int64_t k = __shfl_sync(FULL_MASK, c0, src) + lane;
        const uint64_t* ou = reinterpret_cast<const uint64_t*>(__shfl_sync(FULL_MASK, oaddr, src));
        vq[u] = rq[u] >= 0 && k < nbu;
        if (vq[u]) gq[u] = ou[k];
      }
#pragma unroll
      for (int u = 0; u < CHAIN_ILP; u++)
        if (vq[u]) stage[rq[u] * CHAIN_ROW + lane] = gq[u];
    }
    __syncwarp();
    // ---- 2. each lane chains its own request through the chunk
    const int64_t left = nb - c0;
    const int m = !has ? 0 : (left < 32 ? (int)left : 32);
#pragma unroll 4
    for (int j = 0; j < m; j++) {
      h = chain_step(h, row[j]);
      row[j] = h;
    }
    __syncwarp();
    // ---- 3. coalesced stores, one request at a time
    act = busy;
    while (act) {
      const int ra = __ffs(act) - 1;
      act &= act - 1;
      const int64_t nba = __shfl_sync(FULL_MASK, nb, ra);
      const int64_t k = __shfl_sync(FULL_MASK, c0, ra) + lane;
      uint64_t* oa = reinterpret_cast<uint64_t*>(__shfl_sync(FULL_MASK, oaddr, ra));
      if (k < nba) oa[k] = stage[ra * CHAIN_ROW + lane];
    }
    __syncwarp();
    if (has) {
      c0 += 32;
      if (c0 >= nb) has = false;
    }
  }
  if (nbmax) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const int64_t v = __shfl_xor_sync(FULL_MASK, local_max, o);
      local_max = v > local_max ? v : local_max;
    }
    if (lane == 0) s_max[wid] = local_max;
    __syncthreads();
    if (threadIdx.x == 0) {
      int64_t mx = 0;
      for (int w = 0; w < CHAIN_WARPS; w++) mx = s_max[w] > mx ? s_max[w] : mx;
      if (mx > 0) atomicMax(reinterpret_cast<unsigned long long*>(nbmax), (unsigned long long)mx);
    }
  }
}

cudaError_t launch_block_hash(const HashJob* jobs_dev, int njobs, int64_t total_req, uint64_t seed,
                              int64_t* nbmax_out, HashSched* sched, int64_t* long_list,
                              cudaStream_t st) {
  if (total_req <= 0) return cudaSuccess;
  if (njobs < 1 || njobs > HASH_MAX_JOBS || !sched || !long_list) return cudaErrorInvalidValue;
  int dev = 0, sms = 0, per_sm = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  // content: one warp per request, grid-strided
  int64_t cb = (total_req + CONTENT_NT / 32 - 1) / (CONTENT_NT / 32);
  if (cb > (int64_t)sms * 16) cb = (int64_t)sms * 16;
  k_block_content<<<(unsigned)cb, CONTENT_NT, 0, st>>>(jobs_dev, njobs, total_req, sched,
                                                       long_list);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  // chain: one wave of resident CTAs; the work counter hands out the requests
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_block_chain, CHAIN_NT, 0);
  if (e != cudaSuccess) return e;
  int64_t nblk = (int64_t)sms * (per_sm > 0 ? per_sm : 1);
  const int64_t need = (total_req + CHAIN_NT - 1) / CHAIN_NT;
  if (nblk > need) nblk = need;
  k_block_chain<<<(unsigned)nblk, CHAIN_NT, 0, st>>>(jobs_dev, njobs, total_req, seed, nbmax_out,
                                                     sched, long_list);
  return cudaGetLastError();
}

}  // namespace rs
