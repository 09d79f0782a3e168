// Allocation-free variant of the bf16 linear entry point.
//
// Some callers cannot allocate device memory at the moment they run a linear: code
// that runs inside a host callback or a custom allocator, code that must not grow the
// device's memory footprint after start-up (a fixed memory budget per process), or a
// runtime whose device memory is owned by another allocator.  For them this entry
// point keeps the split-K scratch of the tensor-core linear in file-scope device
// arrays that exist for as long as the library is loaded, so a call allocates
// nothing: the caller passes inputs and outputs, the library owns the scratch.
//
// Limits: M <= 32 token rows; at most 4096 output tiles (N <= 4096 * 128 columns for
// M <= 32); the grid is capped at 160 CTAs (devices with more SMs use 160 of them).
// Every call shares the arrays (each GPU that loads the library holds 5.2 MB of them
// until the process exits), so calls that overlap on the GPU (two streams, or two
// host threads) race on the scratch and must be serialised by the caller.
#include <cstdio>
#include <cstring>
#include <mutex>

#include "../../include/chimera.h"
#include "common.cuh"
#include "kernels.h"

constexpr int NA_MAX_M = 32;
constexpr int NA_MAX_GRID = 160;
constexpr int NA_MAX_TILES = 4096;
constexpr size_t NA_WS_FLOATS = static_cast<size_t>(NA_MAX_GRID) * 2 * 128 * NA_MAX_M;

// The scratch: split-K partial tiles, one arrival counter per output tile (zero
// between launches), and the device error word.
static __device__ __align__(256) float g_na_ws[NA_WS_FLOATS];
static __device__ __align__(256) int g_na_counters[NA_MAX_TILES];
static __device__ __align__(256) int g_na_err[64];

namespace chimera {
namespace {

struct NaDevice {
  bool ready = false;
  float* ws = nullptr;
  int* counters = nullptr;
  int* err = nullptr;
};
constexpr int NA_MAX_DEVICES = 64;
std::mutex g_na_mu;
NaDevice g_na_dev[NA_MAX_DEVICES];

// Device addresses of the arrays, looked up once per device with that device current
// (in host code the array names are host-side stand-ins, not device addresses).
const NaDevice* na_setup(int dev) {
  std::lock_guard<std::mutex> lk(g_na_mu);
  NaDevice& d = g_na_dev[dev];
  if (d.ready) return &d;
  void* ws = nullptr;
  void* cnt = nullptr;
  void* err = nullptr;
  if (cudaGetSymbolAddress(&ws, g_na_ws) != cudaSuccess) return nullptr;
  if (cudaGetSymbolAddress(&cnt, g_na_counters) != cudaSuccess) return nullptr;
  if (cudaGetSymbolAddress(&err, g_na_err) != cudaSuccess) return nullptr;
  d.ws = static_cast<float*>(ws);
  d.counters = static_cast<int*>(cnt);
  d.err = static_cast<int*>(err);
  d.ready = true;
  return &d;
}

}  // namespace

// Read and clear the error word of the static scratch on the current device (0 when
// the device never ran the entry point).  Returns 0, or -1 when a CUDA call failed.
int noalloc_take_error(int* word) {
  *word = 0;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= NA_MAX_DEVICES) return -1;
  int* err = nullptr;
  {
    std::lock_guard<std::mutex> lk(g_na_mu);
    if (!g_na_dev[dev].ready) return 0;
    err = g_na_dev[dev].err;
  }
  int e = 0;
  if (cudaMemcpy(&e, err, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess) return -1;
  if (e && cudaMemset(err, 0, sizeof(int)) != cudaSuccess) return -1;
  *word = e;
  return 0;
}

}  // namespace chimera

using namespace chimera;

extern "C" chimera_status chimera_op_linear_noalloc(int epi, int out_f32, int M, int N, int K, const void* X,
                                                    const void* X_lo, int ldx, const void* W, void* Y, int ldy,
                                                    void* cuda_stream) {
  if (epi < 0 || epi > 2 || M < 1 || N < 1 || K < 1 || !X || !W || !Y || ldx < K || ldy < N) return CHIMERA_EINVAL;
  if (M > NA_MAX_M) {
    fprintf(stderr, "chimera_op_linear_noalloc: M = %d exceeds the static scratch limit of %d rows\n", M,
            NA_MAX_M);
    return CHIMERA_EINVAL;
  }
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= NA_MAX_DEVICES) return CHIMERA_ECUDA;
  const NaDevice* d = na_setup(dev);
  if (!d) return CHIMERA_ECUDA;
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  TcLinearPlan plan;
  char msg[256];
  if (tc_linear_plan(&plan, M, N, K, X, X_lo, ldx, W, Y, nullptr, ldy, epi, epi == EPI_RESID ? 1 : out_f32, d->ws,
                     d->counters, d->err, msg, sizeof(msg)) != 0) {
    fprintf(stderr, "chimera_op_linear_noalloc: %s\n", msg);
    return CHIMERA_EINVAL;
  }
  const int tiles = plan.p.feat_tiles * plan.p.tok_tiles;
  if (tiles > NA_MAX_TILES) {
    fprintf(stderr, "chimera_op_linear_noalloc: %d output tiles exceed the static limit of %d\n", tiles,
            NA_MAX_TILES);
    return CHIMERA_EINVAL;
  }
  if (plan.grid > NA_MAX_GRID) plan.grid = NA_MAX_GRID;  // the partition follows gridDim
  // The counters must start at zero; an aborted earlier call could have left some
  // raised.  The partial tiles are fully written before use.  The error word is left
  // alone: it collects what every call flags until chimera_op_sync reads and clears it.
  if (cudaMemsetAsync(d->counters, 0, static_cast<size_t>(tiles) * sizeof(int), s) != cudaSuccess)
    return CHIMERA_ECUDA;
  return tc_linear_launch(plan, s) == cudaSuccess ? CHIMERA_OK : CHIMERA_ECUDA;
}
