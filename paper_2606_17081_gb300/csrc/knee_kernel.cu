// Saturation knee of load sweeps (§5.1, the PoA-growth proposition, item 3:
// the second derivative of latency with respect to load above a threshold
// marks the onset of saturation; Experiment 2 takes difference quotients of
// TTFT P99 across a sweep of concurrency levels).
//
// k_replica_pct (one CTA per replica): the nearest-rank percentile of the
// replica's routed TTFTs by an exact radix select on order-preserving 64-bit
// keys of the doubles, eight passes of 8-bit digits over the replica's rows
// (histograms in shared memory, warp-aggregated increments).  The result is
// an element of the input, so it is bit-exact.
//
// k_sweep_knee (one thread per sweep; a sweep is a handful of levels): the
// neighbour difference quotients, the three-point second divided difference
// and the first interior level above the threshold, each operation rounded
// once in the order written.
#include "rs_device.cuh"

namespace rs {

constexpr int NT_PCT = 256;

// ascending doubles <-> ascending unsigned keys (sign-magnitude to offset binary)
__device__ __forceinline__ uint64_t order_key(double v) {
  const uint64_t u = (uint64_t)__double_as_longlong(v);
  return (u >> 63) ? ~u : (u | 0x8000000000000000ull);
}

__device__ __forceinline__ double key_value(uint64_t k) {
  const uint64_t u = (k >> 63) ? (k & 0x7FFFFFFFFFFFFFFFull) : ~k;
  return __longlong_as_double((long long)u);
}

__global__ void __launch_bounds__(NT_PCT) k_replica_pct(const int32_t* __restrict__ worker,
                                                        const double* __restrict__ ttft,
                                                        const int64_t* __restrict__ row_start,
                                                        int pct, double* __restrict__ stat,
                                                        double* __restrict__ d1,
                                                        double* __restrict__ d2) {
  __shared__ unsigned hist[256];
  __shared__ unsigned long long s_cnt;
  __shared__ uint64_t s_prefix;
  __shared__ long long s_rank;
  const int r = blockIdx.x;
  const int64_t a = row_start[r], b = row_start[r + 1];
  const int lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    s_cnt = 0;
    s_prefix = 0;
    d1[r] = __longlong_as_double(0x7FF8000000000000ll);
    d2[r] = __longlong_as_double(0x7FF8000000000000ll);
  }
  __syncthreads();
  unsigned c = 0;
  for (int64_t i = a + threadIdx.x; i < b; i += NT_PCT) c += worker[i] >= 0;
  c = __reduce_add_sync(FULL_MASK, c);
  if (lane == 0 && c) atomicAdd(&s_cnt, (unsigned long long)c);
  __syncthreads();
  const long long n = (long long)s_cnt;
  if (n == 0) {
    if (threadIdx.x == 0) stat[r] = __longlong_as_double(0x7FF8000000000000ll);
    return;
  }
  if (threadIdx.x == 0) s_rank = ((long long)pct * n + 99) / 100 - 1;   // 0-based ascending
  uint64_t mask = 0;
  for (int shift = 56; shift >= 0; shift -= 8) {
    hist[threadIdx.x] = 0;   // NT_PCT == 256 bins
    __syncthreads();
    const uint64_t prefix = s_prefix;
    for (int64_t i0 = a; i0 < b; i0 += NT_PCT) {
      const int64_t i = i0 + threadIdx.x;
      int digit = -1;
      if (i < b && worker[i] >= 0) {
        const uint64_t k = order_key(ttft[i]);
        if ((k & mask) == prefix) digit = (int)((k >> shift) & 255u);
      }
      const unsigned peers = __match_any_sync(FULL_MASK, digit);
      if (digit >= 0 && (__ffs(peers) - 1) == lane) atomicAdd(&hist[digit], __popc(peers));
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      long long k = s_rank;
      int d = 0;
      for (; d < 255; d++) {
        if (k < (long long)hist[d]) break;
        k -= hist[d];
      }
      s_rank = k;
      s_prefix = prefix | ((uint64_t)d << shift);
    }
    mask |= 255ull << shift;
    __syncthreads();
  }
  if (threadIdx.x == 0) stat[r] = key_value(s_prefix);
}

__global__ void k_sweep_knee(const double* __restrict__ load, const double* __restrict__ stat,
                             const int32_t* __restrict__ sweep_start, int n_sweeps, double theta,
                             double* __restrict__ d1, double* __restrict__ d2,
                             double* __restrict__ knee_load, int32_t* __restrict__ knee_index) {
  const int s = blockIdx.x * blockDim.x + threadIdx.x;
  if (s >= n_sweeps) return;
  const int a = sweep_start[s], b = sweep_start[s + 1];
  bool inc = true;
  for (int r = a + 1; r < b; r++) inc &= load[r] > load[r - 1];
  if (!inc) {
    knee_load[s] = __longlong_as_double(0x7FF8000000000000ll);
    knee_index[s] = -2;
    return;
  }
  for (int r = a; r + 1 < b; r++)
    d1[r] = __ddiv_rn(__dsub_rn(stat[r + 1], stat[r]), __dsub_rn(load[r + 1], load[r]));
  double kl = -1.0;
  int ki = -1;
  for (int r = a + 1; r + 1 < b; r++) {
    const double v = __ddiv_rn(__dmul_rn(2.0, __dsub_rn(d1[r], d1[r - 1])),
                               __dsub_rn(load[r + 1], load[r - 1]));
    d2[r] = v;
    if (ki < 0 && v > theta) {
      ki = r;
      kl = load[r];
    }
  }
  knee_load[s] = kl;
  knee_index[s] = ki;
}

cudaError_t launch_sweep_knee(const int32_t* worker, const double* ttft, const int64_t* row_start,
                              int n_rep, const double* load, const int32_t* sweep_start,
                              int n_sweeps, int pct, double theta, double* stat, double* d1,
                              double* d2, double* knee_load, int32_t* knee_index,
                              cudaStream_t st) {
  static_assert(NT_PCT == 256, "one histogram bin per thread");
  if (n_rep > 0) {
    k_replica_pct<<<n_rep, NT_PCT, 0, st>>>(worker, ttft, row_start, pct, stat, d1, d2);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  if (n_sweeps > 0) {
    k_sweep_knee<<<(n_sweeps + 127) / 128, 128, 0, st>>>(load, stat, sweep_start, n_sweeps, theta,
                                                        d1, d2, knee_load, knee_index);
    return cudaGetLastError();
  }
  return cudaSuccess;
}

}  // namespace rs
