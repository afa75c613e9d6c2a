// noalloc.cu — ef_hard_threshold_noalloc: the hard-threshold step for callers
// that must not allocate device memory.
//
// The regular entry points keep a per-stream workspace that grows with
// cudaMalloc (and synchronises the stream when it does). Some callers cannot
// allow that: an application whose memory is entirely owned by its own
// allocator or a framework's caching pool, a latency-critical loop that must
// never block in cudaMalloc/cudaFree, or a process running with a fixed
// device-memory budget. This entry point runs the same ordered compaction
// (the look-back kernel of ht.cu, one tile per CTA) with its only scratch —
// one status word per 4096-coordinate tile plus an error word — in a
// file-scope __device__ array of fixed size: one status word per
// 4096-coordinate tile, then the error word and the kernel's tile dispenser.
// It calls no cudaMalloc, cudaFree or allocating library routine.
//
// The array is allocated when the library is loaded and stays on every device
// that loads it until the process exits (512 KiB + 256 bytes). All calls on a
// device share it, so calls that overlap on the GPU (different streams, or
// different host threads without ordering) race and must be avoided.
#include <cmath>
#include <cstdlib>
#include <map>
#include <mutex>

#include "efsparse.h"
#include "internal.h"

namespace efs {
namespace {

constexpr uint32_t kNoallocMaxTiles = 1u << 16;                 // d <= 2^28
constexpr uint64_t kNoallocMaxD = uint64_t(kNoallocMaxTiles) * kTileElems;
constexpr uint32_t kNoallocErrorWord = kNoallocMaxTiles;        // index of the error word
constexpr uint32_t kNoallocClaimWord = kNoallocMaxTiles + 1;    // the tile dispenser (2 x u32)

// [0, kNoallocMaxTiles): epoch-tagged tile status words; then the error word
// and the tile dispenser.
static __device__ __align__(256) uint64_t g_noalloc_scratch[kNoallocMaxTiles + 32];

// First epoch on a device. Testing aid: EF_NOALLOC_FIRST_EPOCH (decimal,
// below 2^30) starts the count near the wrap so that a test can cross it.
uint32_t first_epoch() {
  const char* v = std::getenv("EF_NOALLOC_FIRST_EPOCH");
  if (!v) return 0;
  const unsigned long long x = std::strtoull(v, nullptr, 10);
  return x < (1ull << 30) ? static_cast<uint32_t>(x) : 0u;
}

struct NoallocDevice {
  uint64_t* scratch = nullptr;  // device address of g_noalloc_scratch on this device
  uint32_t epoch = 0;           // last epoch used on this device
};
std::mutex g_noalloc_mu;
std::map<int, NoallocDevice> g_noalloc_devices;

}  // namespace
}  // namespace efs

extern "C" ef_status ef_hard_threshold_noalloc(const float* g, float* e, float gamma,
                                               float lambda, uint64_t d, uint32_t* idx_out,
                                               float* val_out, uint32_t* count_out,
                                               uint32_t* status_out, ef_stream_t stream) {
  using namespace efs;
  const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (d > kNoallocMaxD) return EF_ERR_INVALID_ARG;  // larger than the fixed scratch
  if (!count_out || reinterpret_cast<uintptr_t>(count_out) % 4) return EF_ERR_INVALID_ARG;
  if (status_out && reinterpret_cast<uintptr_t>(status_out) % 4) return EF_ERR_INVALID_ARG;
  if (!std::isfinite(gamma) || !(lambda >= 0.0f)) return EF_ERR_INVALID_ARG;
  if (d > 0) {
    if (!g || !e || !idx_out || !val_out) return EF_ERR_INVALID_ARG;
    const uintptr_t a[4] = {reinterpret_cast<uintptr_t>(g), reinterpret_cast<uintptr_t>(e),
                            reinterpret_cast<uintptr_t>(idx_out),
                            reinterpret_cast<uintptr_t>(val_out)};
    for (uintptr_t x : a)
      if (x % 4) return EF_ERR_INVALID_ARG;
  }
  {
    // no two of the buffers may overlap (the status word is written after
    // the kernel, so an overlap would silently replace an output word)
    const uintptr_t nb = static_cast<uintptr_t>(d) * 4;
    const uintptr_t lo[6] = {reinterpret_cast<uintptr_t>(g), reinterpret_cast<uintptr_t>(e),
                             reinterpret_cast<uintptr_t>(idx_out),
                             reinterpret_cast<uintptr_t>(val_out),
                             reinterpret_cast<uintptr_t>(count_out),
                             reinterpret_cast<uintptr_t>(status_out)};
    const uintptr_t len[6] = {nb, nb, nb, nb, 4, status_out ? 4u : 0u};
    for (int i = 0; i < 6; ++i)
      for (int j = i + 1; j < 6; ++j)
        if (len[i] && len[j] && lo[i] < lo[j] + len[j] && lo[j] < lo[i] + len[i])
          return EF_ERR_INVALID_ARG;
  }

  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return EF_ERR_CUDA;
  uint64_t* scratch = nullptr;
  uint32_t epoch = 0;
  bool wrap = false;
  {
    std::lock_guard<std::mutex> lk(g_noalloc_mu);
    NoallocDevice& nd = g_noalloc_devices[dev];
    if (!nd.scratch) {
      // once per device, with that device current: the device address of the
      // array (its name in host code is only a host-side stand-in)
      void* p = nullptr;
      if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) {
        cudaGetLastError();
        return EF_ERR_CUDA;
      }
      nd.scratch = static_cast<uint64_t*>(p);
      nd.epoch = first_epoch();
    }
    if (nd.epoch >= (1u << 30) - 1) {
      nd.epoch = 0;
      wrap = true;
    }
    epoch = ++nd.epoch;
    scratch = nd.scratch;
  }
  uint32_t* error = reinterpret_cast<uint32_t*>(scratch + kNoallocErrorWord);
  // the array keeps the previous call's contents: clear what must start at
  // zero (the error word and the tile dispenser, which sit side by side; all
  // status words after an epoch wrap)
  if (wrap && cudaMemsetAsync(scratch, 0, sizeof(uint64_t) * kNoallocMaxTiles, s) != cudaSuccess)
    return EF_ERR_CUDA;
  if (cudaMemsetAsync(error, 0, 2 * sizeof(uint64_t), s) != cudaSuccess) return EF_ERR_CUDA;
  if (d == 0) {
    if (cudaMemsetAsync(count_out, 0, sizeof(uint32_t), s) != cudaSuccess) return EF_ERR_CUDA;
  } else {
    ScanCtx ctx;
    ctx.status = scratch;
    ctx.error = error;
    ctx.epoch = epoch;
    ctx.num_tiles = tiles_for(d);
    ctx.withheld_tile = withheld_tile();
    ctx.wait_limit_ns = wait_limit_ns();
    ctx.tile_claim = reinterpret_cast<uint32_t*>(scratch + kNoallocClaimWord);
    if (launch_hard_threshold_lookback(g, e, gamma, lambda, static_cast<uint32_t>(d), idx_out,
                                       val_out, count_out, ctx, s) != cudaSuccess)
      return EF_ERR_CUDA;
  }
  if (status_out &&
      cudaMemcpyAsync(status_out, error, sizeof(uint32_t), cudaMemcpyDeviceToDevice, s) !=
          cudaSuccess)
    return EF_ERR_CUDA;
  return EF_OK;
}
