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
#include <algorithm>
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
  // w[j] = a[j + shift] by two selects on the shift's bits (no branch)
  uint32_t c[19], w[16];
  const bool s1 = shift & 1, s2 = shift & 2;
#pragma unroll
  for (int j = 0; j < 19; j++) c[j] = s1 ? a[j + 1] : a[j];
#pragma unroll
  for (int j = 0; j < 16; j++) w[j] = s2 ? c[j + 2] : c[j];
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
  // one warp per request, up to 64 CTAs per SM (six are resident at a time):
  // prompt lengths vary, and short grid-stride runs per warp leave a shorter
  // tail than long ones (the cap was chosen by measurement)
  int64_t nblk = (total_req + HASH_NT / 32 - 1) / (HASH_NT / 32);
  if (nblk > (int64_t)sms * 64) nblk = (int64_t)sms * 64;
  k_block_hash<<<(unsigned)nblk, HASH_NT, 0, st>>>(jobs_dev, njobs, total_req, seed, nbmax_out);
  return cudaGetLastError();
}

// The largest number of full blocks of any request of the jobs (offsets
// only): atomicMax into *nbmax, which the caller clears.
__global__ void __launch_bounds__(256) k_nbmax(const HashJob* __restrict__ jobs, int njobs,
                                               int64_t total_req, int64_t* __restrict__ nbmax) {
  __shared__ HashJob s_jobs[HASH_MAX_JOBS];
  __shared__ int64_t s_max[8];
  for (int j = threadIdx.x; j < njobs; j += blockDim.x) s_jobs[j] = jobs[j];
  __syncthreads();
  int64_t m = 0;
  for (int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; r < total_req;
       r += (int64_t)gridDim.x * blockDim.x) {
    const HashJob& J = s_jobs[find_job(s_jobs, njobs, r)];
    const int64_t i = r - J.req_base;
    const int64_t nb = (__ldg(J.offsets + i + 1) - __ldg(J.offsets + i)) >> 4;
    m = nb > m ? nb : m;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const int64_t v = __shfl_xor_sync(FULL_MASK, m, o);
    m = v > m ? v : m;
  }
  if ((threadIdx.x & 31) == 0) s_max[threadIdx.x >> 5] = m;
  __syncthreads();
  if (threadIdx.x == 0) {
    int64_t x = 0;
    for (int w = 0; w < (int)(blockDim.x >> 5); w++) x = s_max[w] > x ? s_max[w] : x;
    if (x > 0) atomicMax(reinterpret_cast<unsigned long long*>(nbmax), (unsigned long long)x);
  }
}

cudaError_t launch_nbmax(const HashJob* jobs_dev, int njobs, int64_t total_req, int64_t* nbmax,
                         cudaStream_t st) {
  if (total_req <= 0) return cudaSuccess;
  if (njobs < 1 || njobs > HASH_MAX_JOBS) return cudaErrorInvalidValue;
  int dev = 0, sms = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  int64_t nblk = (total_req + 255) / 256;
  if (nblk > (int64_t)sms * 4) nblk = (int64_t)sms * 4;
  k_nbmax<<<(unsigned)nblk, 256, 0, st>>>(jobs_dev, njobs, total_req, nbmax);
  return cudaGetLastError();
}

// Duplicate block hashes within one prompt (a 64-bit collision, which the
// simulation reports as RS_ERR_COLLISION at that request): flags[r] = 1 when
// two blocks of request r share a chained hash, 0 when none do, 2 when the
// request has more than nbmax blocks (not checked; in the simulation such a
// prompt is longer than the cache and stops its replica for capacity before
// any update).  One warp per request, each warp with an open-addressing set
// of cap entries in shared memory (cap a power of two >= 2 nbmax; the set of
// a request uses the first power of two >= 2 nb of them).  Hashes are >= 2,
// so 0 marks an empty entry.
__global__ void __launch_bounds__(256) k_dup_flags(const HashJob* __restrict__ jobs, int njobs,
                                                   int64_t total_req, int64_t nbmax, uint32_t cap,
                                                   uint8_t* __restrict__ flags) {
  extern __shared__ unsigned long long dset[];
  __shared__ HashJob s_jobs[HASH_MAX_JOBS];
  for (int j = threadIdx.x; j < njobs; j += blockDim.x) s_jobs[j] = jobs[j];
  __syncthreads();
  const int lane = threadIdx.x & 31, wpc = (int)(blockDim.x >> 5);
  unsigned long long* set = dset + (size_t)(threadIdx.x >> 5) * cap;
  const int64_t nw = (int64_t)gridDim.x * wpc;
  for (int64_t r = (int64_t)blockIdx.x * wpc + (threadIdx.x >> 5); r < total_req; r += nw) {
    const HashJob& J = s_jobs[find_job(s_jobs, njobs, r)];
    const int64_t i = r - J.req_base;
    const int64_t o0 = __ldg(J.offsets + i);
    const int64_t nb = (__ldg(J.offsets + i + 1) - o0) >> 4;
    int dup = nb > nbmax ? 2 : 0;
    if (nb >= 2 && nb <= nbmax) {   // warp-uniform (2 nb <= cap)
      uint32_t m = 2;
      while (m < 2 * nb) m <<= 1;
      const uint32_t mask = m - 1;
      for (uint32_t e = lane; e < m; e += 32) set[e] = 0ull;
      __syncwarp();
      const uint64_t* h = J.out + (o0 >> 4);
      for (int64_t k = lane; k < nb; k += 32) {
        const unsigned long long x = __ldg(h + k);
        uint32_t d = (uint32_t)(x ^ (x >> 29)) & mask;
        for (uint32_t it = 0; it <= mask; it++) {
          const unsigned long long prev = atomicCAS(set + d, 0ull, x);
          if (prev == 0ull) break;
          if (prev == x) {
            dup = 1;
            break;
          }
          d = (d + 1) & mask;
        }
      }
      dup = __any_sync(FULL_MASK, dup);   // (every lane's claims are made before the next clear)
    }
    if (lane == 0) flags[r] = (uint8_t)dup;
  }
}

cudaError_t launch_dup_flags(const HashJob* jobs_dev, int njobs, int64_t total_req, int64_t nbmax,
                             uint8_t* flags, cudaStream_t st) {
  if (total_req <= 0) return cudaSuccess;
  if (njobs < 1 || njobs > HASH_MAX_JOBS || nbmax < 1) return cudaErrorInvalidValue;
  int dev = 0, sms = 0, maxsm = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e == cudaSuccess)
    e = cudaDeviceGetAttribute(&maxsm, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  if (e != cudaSuccess) return e;
  uint32_t cap = 2;
  while ((int64_t)cap < 2 * nbmax) cap <<= 1;
  // dynamic shared memory beside the static job table: up to the default
  // 48 KB per CTA without opting in, else one warp's set with the opt-in
  const size_t per_warp = (size_t)cap * 8;
  const size_t stat = sizeof(HashJob) * HASH_MAX_JOBS;
  const size_t room = (size_t)maxsm - stat, dflt = 48 * 1024 - stat;
  if (per_warp > room) return cudaErrorInvalidValue;
  int wpc = (int)std::min<size_t>(8, std::max<size_t>(1, dflt / per_warp));
  const size_t smem = per_warp * wpc;
  if (smem > dflt) {
    e = cudaFuncSetAttribute(k_dup_flags, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
  }
  int64_t nblk = (total_req + wpc - 1) / wpc;
  if (nblk > (int64_t)sms * 16) nblk = (int64_t)sms * 16;
  k_dup_flags<<<(unsigned)nblk, 32 * wpc, smem, st>>>(jobs_dev, njobs, total_req, nbmax, cap,
                                                     flags);
  return cudaGetLastError();
}

}  // namespace rs
