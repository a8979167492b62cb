// poa_estimate_noalloc: the windowed PoA estimate without any allocation.
//
// Some callers cannot allocate device memory at the moment they want an
// estimate: a serving process whose GPU memory is owned up front by another
// allocator (so a cudaMalloc would fail or fragment it), or a latency-critical
// path where cudaMalloc / cudaFree would synchronise the device.  This entry
// point runs the same two PoA kernels as poa_estimate, but their scratch lives
// in one fixed array of static device memory (RS_NOALLOC_POA_BYTES bytes)
// that every GPU loading the library holds until the process exits.  The
// caller passes inputs and outputs in device memory; nothing is allocated and
// nothing is copied to the host.
#include <mutex>

#include "rs_internal.h"

namespace rs {

static __device__ __align__(256) unsigned char g_poa_scratch[RS_NOALLOC_POA_BYTES];

namespace {

constexpr int kMaxDevices = 64;
std::mutex g_mu;
void* g_scratch_ptr[kMaxDevices] = {};   // device address of g_poa_scratch per device

size_t up256(size_t x) { return (x + 255) & ~(size_t)255; }

// Carve-up of the static array for n rows of W workers (byte offsets): the
// fixed entries and the row arrays first, then the window arrays, which get
// every byte that remains (win slots each).
struct NoallocLayout {
  size_t prob, total, nwin, tstat, cost, order, asg, wkey, wstart, wfill, wnum, wopt, wcnt, wstat,
      end;
  int64_t win;   // window slots (< 1: the rows leave no room)
};

// Accepted sizes: n (8 W + 60) + NOALLOC_SLACK <= RS_NOALLOC_POA_BYTES, i.e. per
// row its cost row (8 W), order, assignment and window key (12) and six
// window entries (48) for n of the windows; the slack covers the fixed
// entries, two more windows and the 256-byte alignment of 14 arrays.
constexpr size_t NOALLOC_SLACK = 4096;

bool noalloc_fits(int64_t n, int W) {
  const size_t rows = (size_t)(n > 0 ? n : 1);
  return rows <= ((size_t)RS_NOALLOC_POA_BYTES - NOALLOC_SLACK) / (size_t)(8 * W + 60);
}

NoallocLayout layout(int64_t n, int W) {
  NoallocLayout L;
  const size_t rows = (size_t)(n > 0 ? n : 1);
  size_t o = 0;
  L.prob = o; o = up256(o + sizeof(PoaProblem));
  L.total = o; o = up256(o + 8);
  L.nwin = o; o = up256(o + 8);
  L.tstat = o; o = up256(o + 8);
  L.cost = o; o = up256(o + rows * (size_t)W * 8);
  L.order = o; o = up256(o + rows * 4);
  L.asg = o; o = up256(o + rows * 4);
  L.wkey = o; o = up256(o + rows * 4);
  // six window arrays of win entries (wstart one more), each 256-aligned
  const size_t room = (size_t)RS_NOALLOC_POA_BYTES > o + 6 * 256 + 8
                          ? (size_t)RS_NOALLOC_POA_BYTES - o - 6 * 256 - 8 : 0;
  L.win = (int64_t)(room / 48);
  const size_t win = (size_t)(L.win > 0 ? L.win : 0);
  L.wstart = o; o = up256(o + (win + 1) * 8);
  L.wfill = o; o = up256(o + win * 8);
  L.wnum = o; o = up256(o + win * 8);
  L.wopt = o; o = up256(o + win * 8);
  L.wcnt = o; o = up256(o + win * 8);
  L.wstat = o; o = up256(o + win * 8);
  L.end = o;
  return L;
}

__global__ void k_noalloc_setup(PoaProblem pr, PoaProblem* dst) { *dst = pr; }

// Copies the per-window results (at most max_windows) and the totals out of
// the static scratch into the caller's buffers.
__global__ void k_noalloc_out(const double* wnum, const double* wopt, const int64_t* wcnt,
                              const double* total, const int64_t* nwin, int64_t max_windows,
                              double* numer, double* opt, int64_t* count, double* total_out,
                              int64_t* nwin_out) {
  const int64_t nw = *nwin;
  const int64_t k = nw < max_windows ? nw : max_windows;
  for (int64_t w = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; w < k;
       w += (int64_t)gridDim.x * blockDim.x) {
    if (numer) numer[w] = wnum[w];
    if (opt) opt[w] = wopt[w];
    if (count) count[w] = wcnt[w];
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    *total_out = *total;
    *nwin_out = nw;
  }
}

}  // namespace

}  // namespace rs

using namespace rs;

extern "C" rs_status poa_estimate_noalloc(const rs_config* cfg, const rs_records* records,
                                          int64_t n, double* numer_dev, double* opt_dev,
                                          int64_t* count_dev, int64_t max_windows,
                                          double* poa_total_dev, int64_t* n_windows_dev,
                                          void* cuda_stream) {
  if (!cfg || !records || !poa_total_dev || !n_windows_dev) return RS_ERR_INVALID;
  if (cfg->W < 1 || cfg->W > POA_WMAX_WIDE || cfg->cap < 2 || cfg->cap > 65535 ||
      !(cfg->poa_window > 0.0))
    return RS_ERR_INVALID;
  if (n < 0 || max_windows < 0) return RS_ERR_INVALID;
  const rs_records& u = *records;
  if (n > 0 && (!u.worker || !u.completion || !u.ttft || !u.nbt || !u.n_frozen || !u.prefix))
    return RS_ERR_INVALID;
  if (!noalloc_fits(n, cfg->W)) return RS_ERR_CAPACITY;
  const NoallocLayout L = layout(n, cfg->W);
  if (L.end > (size_t)RS_NOALLOC_POA_BYTES || L.win < (n > 0 ? n : 1) + 2) return RS_ERR_CAPACITY;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return RS_ERR_CUDA;
  void* base = nullptr;
  {
    // first call on a device: take the static array's device address
    std::lock_guard<std::mutex> lk(g_mu);
    if (!g_scratch_ptr[dev]) {
      void* p = nullptr;
      if (cudaGetSymbolAddress(&p, g_poa_scratch) != cudaSuccess || !p) {
        cudaGetLastError();
        return RS_ERR_CUDA;
      }
      g_scratch_ptr[dev] = p;
    }
    base = g_scratch_ptr[dev];
  }
  unsigned char* s = static_cast<unsigned char*>(base);
  cudaStream_t st = reinterpret_cast<cudaStream_t>(cuda_stream);
  PoaProblem pr;
  pr.rec_base = 0;
  pr.n = n;
  pr.scratch_base = 0;
  pr.win_base = 0;
  pr.win_cap = L.win;   // windows past this give *n_windows_dev = -1
  PoaProblem* dprob = reinterpret_cast<PoaProblem*>(s + L.prob);
  k_noalloc_setup<<<1, 1, 0, st>>>(pr, dprob);
  if (cudaGetLastError() != cudaSuccess) return RS_ERR_CUDA;
  const ModelConsts mc = make_consts(*cfg);
  PoaBuffers b;
  b.rec = u;
  b.cost = reinterpret_cast<double*>(s + L.cost);
  b.order = reinterpret_cast<int32_t*>(s + L.order);
  b.asg = reinterpret_cast<int32_t*>(s + L.asg);
  b.wkey = reinterpret_cast<int32_t*>(s + L.wkey);
  b.wstart = reinterpret_cast<int64_t*>(s + L.wstart);
  b.wfill = reinterpret_cast<int64_t*>(s + L.wfill);
  b.wnum = reinterpret_cast<double*>(s + L.wnum);
  b.wopt = reinterpret_cast<double*>(s + L.wopt);
  b.wcnt = reinterpret_cast<int64_t*>(s + L.wcnt);
  b.wstat = reinterpret_cast<double*>(s + L.wstat);
  b.total_static = reinterpret_cast<double*>(s + L.tstat);
  b.total = reinterpret_cast<double*>(s + L.total);
  b.nwin = reinterpret_cast<int64_t*>(s + L.nwin);
  b.res = nullptr;
  b.wprob = nullptr;   // one problem: its windows stay on its own CTAs
  b.wnext = nullptr;
  b.nslots = 0;
  if (launch_poa(dprob, 1, b, mc, st) != cudaSuccess) return RS_ERR_CUDA;
  k_noalloc_out<<<64, 256, 0, st>>>(b.wnum, b.wopt, b.wcnt, b.total, b.nwin, max_windows,
                                    numer_dev, opt_dev, count_dev, poa_total_dev, n_windows_dev);
  if (cudaGetLastError() != cudaSuccess) return RS_ERR_CUDA;
  return RS_OK;
}
