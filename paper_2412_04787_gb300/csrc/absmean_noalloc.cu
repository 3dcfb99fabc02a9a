// dqt_absmean_init_noalloc: the AbsMean initialisation (Eq. 2-4) for callers
// that cannot allocate device memory.
//
// dqt_absmean_init needs a small device workspace for its deterministic
// two-stage fp64 reduction (kAbsmeanBlocks partial sums plus the total).
// Some callers cannot provide one.  A framework that owns all device memory
// through its own pool may hand a plugin only the tensors it manages and
// forbid side allocations; code running inside a custom allocator's own
// set-up cannot call cudaMalloc without recursing into itself; a job that
// reserves its whole memory budget up front has no bytes left to ask for.
// This entry point keeps that workspace in a file-scope device array
// instead, so it allocates nothing.
//
// The array is g_absmean_scratch below: kAbsmeanBlocks + 1 = 1025 doubles
// (8200 bytes).  Every GPU that loads the library holds it until the process
// exits.  All calls on a device share it and it keeps the last call's
// contents; each call overwrites every slot it reads before reading it, so
// nothing needs clearing.  Calls whose kernels overlap on the GPU (different
// streams, or different host threads) race on the array: serialise them.
#include <stdint.h>

#include <atomic>

#include "../../include/dqt.h"
#include "dqt_internal.h"

namespace {

static __device__ __align__(256) double g_absmean_scratch[dqt::kAbsmeanBlocks + 1];

constexpr int kMaxDevices = 64;
// Per-device address cache.  Host threads may call concurrently: the cache
// is atomic (every thread that finds it empty stores the same address).
std::atomic<double*> g_scratch_ptr[kMaxDevices] = {};

// Largest element count whose mean divisor converts to fp64 exactly.
constexpr int64_t kMaxNumel = int64_t(1) << 53;

// Device address of the scratch array on the current device.  The host-side
// name g_absmean_scratch is only a stand-in for the device symbol, so the
// address is looked up once per device, with that device current.
double* scratch_on_current_device(int* status) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
    *status = DQT_ERR_CUDA;
    return nullptr;
  }
  double* cached = g_scratch_ptr[dev].load(std::memory_order_relaxed);
  if (!cached) {
    double* p = nullptr;
    if (cudaGetSymbolAddress(reinterpret_cast<void**>(&p), g_absmean_scratch) != cudaSuccess ||
        !p) {
      *status = DQT_ERR_CUDA;
      return nullptr;
    }
    cached = p;
    g_scratch_ptr[dev].store(cached, std::memory_order_relaxed);
  }
  *status = DQT_OK;
  return cached;
}

}  // namespace

extern "C" int dqt_absmean_init_noalloc(const float* W0, int64_t numel, dqt_grid_t grid,
                                        int8_t* codes, float* s_w, void* stream) {
  // the same argument rules as dqt_absmean_init (shared helpers)
  if (!W0 || !codes || !s_w || numel <= 0 || !dqt::grid_ok(grid) || grid.qmax <= 0)
    return DQT_ERR_ARG;
  if (numel > kMaxNumel) return DQT_ERR_RANGE;
  static_assert(sizeof(g_absmean_scratch) >= (dqt::kAbsmeanBlocks + 1) * sizeof(double),
                "scratch holds the partial sums and the total");
  int rc = DQT_OK;
  double* ws = scratch_on_current_device(&rc);
  if (!ws) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (dqt::launch_absmean_partial(W0, numel, ws, st)) return DQT_ERR_CUDA;
  double sum = 0.0;
  if (cudaMemcpyAsync(&sum, ws + dqt::kAbsmeanBlocks, sizeof(double), cudaMemcpyDeviceToHost,
                      st) != cudaSuccess)
    return DQT_ERR_CUDA;
  if (cudaStreamSynchronize(st) != cudaSuccess) return DQT_ERR_CUDA;
  const double absmean = sum / static_cast<double>(numel);
  if (!dqt::absmean_ok(absmean)) return DQT_ERR_ARG;
  const float s = static_cast<float>(static_cast<double>(grid.qmax) / absmean);
  *s_w = s;
  return dqt::launch_absmean_codes(W0, numel, s, grid.qmin, grid.qmax, codes, st) ? DQT_ERR_CUDA
                                                                                    : DQT_OK;
}
