// KV block hashing of prompts (K1): one fused pass over all traces of a call.
//
// One warp per request, lane l on block k0 + l of each 32-block chunk:
//  1. content: the block's 64 bytes arrive as four 16-byte loads (five when
//     the request does not start on a 16-byte boundary) and fold into g_k;
//  2. prefix: H_k = H_{k-1} P + g_k (mod 2^64) is an affine map per block, and
//     composing affine maps is associative, so the warp computes the chunk's
//     H values with a five-step shuffle scan (step s combines partials 2^s
//     blocks apart: a = a_prev P^(2^s) + a), then adds the carry H_{k0-1}
//     times P^(l+1);
//  3. the lane stores mix(H_k ^ k); lane 31's H carries to the next chunk.
// No serial chain per request remains: the pass streams tokens once (4 bytes
// per token in) and hashes once (8 bytes per block out), the HBM floor.
#include <climits>

#include "rs_device.cuh"

namespace rs {

constexpr int HASH_NT = 256;

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

// P^(2^s), s = 0..5, by repeated squaring (mod 2^64)
__host__ __device__ constexpr uint64_t p_pow2(int s) {
  uint64_t x = PREFIX_P;
  for (int i = 0; i < s; i++) x *= x;
  return x;
}

__global__ void __launch_bounds__(HASH_NT) k_block_hash(const HashJob* __restrict__ jobs,
                                                        int njobs, int64_t total_req,
                                                        uint64_t seed,
                                                        int64_t* __restrict__ nbmax) {
  __shared__ HashJob s_jobs[HASH_MAX_JOBS];
  __shared__ int64_t s_max[HASH_NT / 32];
  for (int j = threadIdx.x; j < njobs; j += HASH_NT) s_jobs[j] = jobs[j];
  __syncthreads();
  const int lane = threadIdx.x & 31;
  // P^(lane + 1): the factor of the carry H_{k0-1} at this lane's block
  uint64_t plane = 1;
#pragma unroll
  for (int s = 0; s < 6; s++)
    if (((lane + 1) >> s) & 1) plane *= p_pow2(s);
  int64_t local_max = 0;
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
    local_max = nb > local_max ? nb : local_max;
    uint64_t carry = seed;   // H_{k0 - 1}
    for (int64_t k0 = 0; k0 < nb; k0 += 32) {
      const int64_t k = k0 + lane;
      const bool valid = k < nb;
      uint64_t a = 0;   // g_k; blocks past the prompt add nothing to the ones before
      if (valid) a = content_of(load_block(q + 4 * k, shift), shift);
      // inclusive scan: a = sum over j <= l of g_(k0+j) P^(l - j)
#pragma unroll
      for (int s = 0; s < 5; s++) {
        const int o = 1 << s;
        const uint64_t ap = __shfl_up_sync(FULL_MASK, a, o);
        if (lane >= o) a = ap * p_pow2(s) + a;
      }
      const uint64_t H = carry * plane + a;
      if (valid) out[k] = prefix_output(H, (uint64_t)k);
      carry = __shfl_sync(FULL_MASK, H, 31);
    }
  }
  if (nbmax) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const int64_t v = __shfl_xor_sync(FULL_MASK, local_max, o);
      local_max = v > local_max ? v : local_max;
    }
    if (lane == 0) s_max[threadIdx.x >> 5] = local_max;
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
  int dev = 0, sms = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  int64_t nblk = (total_req + HASH_NT / 32 - 1) / (HASH_NT / 32);   // one warp per request
  if (nblk > (int64_t)sms * 16) nblk = (int64_t)sms * 16;
  k_block_hash<<<(unsigned)nblk, HASH_NT, 0, st>>>(jobs_dev, njobs, total_req, seed, nbmax_out);
  return cudaGetLastError();
}

}  // namespace rs
