// KV block hashing of prompts (K1), in two passes over all traces of a call.
//
// Content pass: one warp per request, lane l takes block k0 + l of a
// 32-block chunk; the block's 64 bytes arrive as four 16-byte loads (five when
// the request does not start on a 16-byte boundary) and fold into the content
// hash g_k; the lane stores g_k ^ k at the block's output slot.  Fully
// parallel, coalesced, HBM-bound (4 bytes per token in, 8 per block out).
//
// Chain pass: one thread per request folds its slots in order,
// h_k = mix(h_{k-1} ^ g_k ^ k), in place; loads run four slots ahead.  One
// 64-bit mix per block; the serial dependence is per request only.
#include <climits>

#include "rs_device.cuh"

namespace rs {

template <int S>
__device__ __forceinline__ void take16(const uint32_t (&a)[20], uint32_t (&w)[16]) {
#pragma unroll
  for (int j = 0; j < 16; j++) w[j] = a[j + S];
}

__device__ __forceinline__ uint64_t hash_block(const int4* q, int shift) {
  const int4 v0 = __ldg(q), v1 = __ldg(q + 1), v2 = __ldg(q + 2), v3 = __ldg(q + 3);
  const int4 v4 = shift ? __ldg(q + 4) : make_int4(0, 0, 0, 0);
  const uint32_t a[20] = {(uint32_t)v0.x, (uint32_t)v0.y, (uint32_t)v0.z, (uint32_t)v0.w,
                          (uint32_t)v1.x, (uint32_t)v1.y, (uint32_t)v1.z, (uint32_t)v1.w,
                          (uint32_t)v2.x, (uint32_t)v2.y, (uint32_t)v2.z, (uint32_t)v2.w,
                          (uint32_t)v3.x, (uint32_t)v3.y, (uint32_t)v3.z, (uint32_t)v3.w,
                          (uint32_t)v4.x, (uint32_t)v4.y, (uint32_t)v4.z, (uint32_t)v4.w};
  uint32_t w[16];
  switch (shift) {
    case 0: take16<0>(a, w); break;
    case 1: take16<1>(a, w); break;
    case 2: take16<2>(a, w); break;
    default: take16<3>(a, w); break;
  }
  return block_content16(w);
}

constexpr int HASH_NT = 256;

__device__ __forceinline__ int find_job(const HashJob* jobs, int njobs, int64_t r) {
  int j = 0;
  while (j + 1 < njobs && r >= jobs[j + 1].req_base) j++;
  return j;
}

__global__ void __launch_bounds__(HASH_NT) k_block_content(const HashJob* __restrict__ jobs,
                                                           int njobs, int64_t total_req) {
  __shared__ HashJob s_jobs[HASH_MAX_JOBS];
  for (int j = threadIdx.x; j < njobs; j += HASH_NT) s_jobs[j] = jobs[j];
  __syncthreads();
  const int lane = threadIdx.x & 31;
  const int64_t warp0 = ((int64_t)blockIdx.x * HASH_NT + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * HASH_NT) >> 5;
  for (int64_t r = warp0; r < total_req; r += nwarps) {
    const HashJob& J = s_jobs[find_job(s_jobs, njobs, r)];
    const int64_t i = r - J.req_base;
    const int64_t o0 = __ldg(J.offsets + i);
    const int64_t nb = (__ldg(J.offsets + i + 1) - o0) >> 4;
    const int shift = (int)(o0 & 3);
    const int4* q = reinterpret_cast<const int4*>(J.tokens) + (o0 >> 2);
    uint64_t* out = J.out + (o0 >> 4);
    for (int64_t k = lane; k < nb; k += 32) out[k] = hash_block(q + 4 * k, shift) ^ (uint64_t)k;
  }
}

__global__ void __launch_bounds__(HASH_NT) k_block_chain(const HashJob* __restrict__ jobs,
                                                         int njobs, int64_t total_req,
                                                         uint64_t seed,
                                                         int64_t* __restrict__ nbmax) {
  __shared__ HashJob s_jobs[HASH_MAX_JOBS];
  __shared__ int64_t s_max[HASH_NT / 32];
  for (int j = threadIdx.x; j < njobs; j += HASH_NT) s_jobs[j] = jobs[j];
  __syncthreads();
  int64_t local_max = 0;
  const int64_t stride = (int64_t)gridDim.x * HASH_NT;
  for (int64_t r = (int64_t)blockIdx.x * HASH_NT + threadIdx.x; r < total_req; r += stride) {
    const HashJob& J = s_jobs[find_job(s_jobs, njobs, r)];
    const int64_t i = r - J.req_base;
    const int64_t o0 = J.offsets[i];
    const int64_t nb = (J.offsets[i + 1] - o0) >> 4;
    local_max = nb > local_max ? nb : local_max;
    uint64_t* out = J.out + (o0 >> 4);
    uint64_t h = seed;
    int64_t k = 0;
    for (; k + 4 <= nb; k += 4) {
      const uint64_t x0 = out[k], x1 = out[k + 1], x2 = out[k + 2], x3 = out[k + 3];
      h = chain_step(h, x0); out[k] = h;
      h = chain_step(h, x1); out[k + 1] = h;
      h = chain_step(h, x2); out[k + 2] = h;
      h = chain_step(h, x3); out[k + 3] = h;
    }
    for (; k < nb; k++) {
      h = chain_step(h, out[k]);
      out[k] = h;
    }
  }
  if (nbmax) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const int64_t v = __shfl_xor_sync(FULL_MASK, local_max, o);
      local_max = v > local_max ? v : local_max;
    }
    if ((threadIdx.x & 31) == 0) s_max[threadIdx.x >> 5] = local_max;
    __syncthreads();
    if (threadIdx.x == 0) {
      int64_t m = 0;
      for (int w = 0; w < HASH_NT / 32; w++) m = s_max[w] > m ? s_max[w] : m;
      if (m > 0) atomicMax(reinterpret_cast<unsigned long long*>(nbmax), (unsigned long long)m);
    }
  }
}

cudaError_t launch_block_hash(const HashJob* jobs_dev, int njobs, int64_t total_req, uint64_t seed,
                              int64_t* nbmax_out, cudaStream_t st) {
  if (total_req <= 0) return cudaSuccess;
  if (njobs < 1 || njobs > HASH_MAX_JOBS) return cudaErrorInvalidValue;
  int64_t wb = (total_req + 7) / 8;              // 8 warps per CTA, one request each
  if (wb > 152 * 16) wb = 152 * 16;
  k_block_content<<<(unsigned)wb, HASH_NT, 0, st>>>(jobs_dev, njobs, total_req);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  int64_t tb = (total_req + HASH_NT - 1) / HASH_NT;
  if (tb > 152 * 8) tb = 152 * 8;
  k_block_chain<<<(unsigned)tb, HASH_NT, 0, st>>>(jobs_dev, njobs, total_req, seed, nbmax_out);
  return cudaGetLastError();
}

}  // namespace rs
