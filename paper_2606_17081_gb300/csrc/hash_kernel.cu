// KV block hashing of prompts (K1).
//
// One warp per request: lane l hashes block k0 + l of a 32-block chunk (its
// 64 bytes arrive as four 16-byte loads, five when the request does not start
// on a 16-byte boundary), then the warp folds the chunk into the hash chain
// h_k = mix(h_{k-1} ^ g_k ^ k) with register shuffles.  Reads 4 bytes per
// token and writes 8 bytes per full block: HBM-bound.
#include <climits>

#include "rs_device.cuh"

namespace rs {

template <int S>
__device__ __forceinline__ void take16(const uint32_t (&a)[20], uint32_t (&w)[16]) {
#pragma unroll
  for (int j = 0; j < 16; j++) w[j] = a[j + S];
}

__global__ void __launch_bounds__(256) k_block_hash(const int32_t* __restrict__ tokens,
                                                    const int64_t* __restrict__ offsets,
                                                    int64_t n_req, uint64_t seed,
                                                    uint64_t* __restrict__ out,
                                                    int64_t* __restrict__ nbmax) {
  const int lane = threadIdx.x & 31;
  const int64_t warp0 = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const int4* tok4 = reinterpret_cast<const int4*>(tokens);
  int64_t local_max = 0;
  for (int64_t i = warp0; i < n_req; i += nwarps) {
    const int64_t o0 = __ldg(offsets + i);
    const int64_t o1 = __ldg(offsets + i + 1);
    const int64_t nb = (o1 - o0) >> 4;
    local_max = nb > local_max ? nb : local_max;
    const int64_t base = o0 >> 4;
    const int shift = (int)(o0 & 3);
    const int4* q0 = tok4 + (o0 >> 2);
    uint64_t h = seed;
    for (int64_t k0 = 0; k0 < nb; k0 += 32) {
      const int64_t k = k0 + lane;
      uint64_t x = 0;
      if (k < nb) {
        const int4* q = q0 + 4 * k;
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
        x = block_content16(w) ^ (uint64_t)k;
      }
      const int lim = nb - k0 < 32 ? (int)(nb - k0) : 32;
      uint64_t mine = 0;
#pragma unroll
      for (int l = 0; l < 32; l++) {
        const uint64_t xl = __shfl_sync(FULL_MASK, x, l);
        if (l < lim) {
          h = chain_step(h, xl);
          if (lane == l) mine = h;
        }
      }
      if (k < nb) out[base + k] = mine;
    }
  }
  if (nbmax) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const int64_t v = __shfl_xor_sync(FULL_MASK, local_max, o);
      local_max = v > local_max ? v : local_max;
    }
    if (lane == 0 && local_max > 0)
      atomicMax(reinterpret_cast<unsigned long long*>(nbmax), (unsigned long long)local_max);
  }
}

cudaError_t launch_block_hash(const int32_t* tokens, const int64_t* offsets, int64_t n_req,
                              uint64_t seed, uint64_t* out, int64_t* nbmax_out, cudaStream_t st) {
  if (n_req <= 0) return cudaSuccess;
  int64_t blocks = (n_req + 7) / 8;
  const int64_t cap = 152 * 16;
  if (blocks > cap) blocks = cap;
  k_block_hash<<<(unsigned)blocks, 256, 0, st>>>(tokens, offsets, n_req, seed, out, nbmax_out);
  return cudaGetLastError();
}

}  // namespace rs
