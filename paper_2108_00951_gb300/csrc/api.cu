// api.cu — the extern "C" boundary declared in include/efsparse.h: host-side
// argument checks, the per-(device, stream) workspaces, and status reporting.
// Every compute step runs in the kernels of ht.cu, topk.cu, topk_layerwise.cu
// and aggregate.cu.
#include <atomic>
#include <cmath>
#include <cstring>
#include <map>
#include <mutex>
#include <utility>

#include "efsparse.h"
#include "internal.h"

namespace efs {
namespace {

std::mutex g_mu;
std::map<std::pair<int, cudaStream_t>, Workspace*> g_workspaces;
std::map<int, DeviceInfo> g_devices;
std::atomic<uint64_t> g_launches{0};
std::atomic<int64_t> g_withheld_tile{-1};
std::atomic<uint64_t> g_wait_limit_ns{2000000000ull};  // 2 s per wait
std::atomic<int> g_stream_kernel_mode{0};  // 0: by size, 1: chunks, 2: groups, 3: shallow ring

constexpr uint64_t kMaxD = 0xffffffffull;

bool overlaps(const void* a, size_t na, const void* b, size_t nb) {
  if (!a || !b || na == 0 || nb == 0) return false;
  const uintptr_t x = reinterpret_cast<uintptr_t>(a), y = reinterpret_cast<uintptr_t>(b);
  return x < y + nb && y < x + na;
}

bool aligned(const void* p, size_t a) { return reinterpret_cast<uintptr_t>(p) % a == 0; }

ef_status device_info(int dev, DeviceInfo* out) {
  std::lock_guard<std::mutex> lk(g_mu);
  auto it = g_devices.find(dev);
  if (it == g_devices.end()) {
    DeviceInfo info;
    if (cudaDeviceGetAttribute(&info.sm_count, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return EF_ERR_CUDA;
    ht_init_device(info);
    topk_init_device(info);
    topk_layerwise_init_device(info);
    aggregate_init_device();
    if (info.refine_blocks <= 0 || info.finalize_blocks <= 0) return EF_ERR_CUDA;
    it = g_devices.emplace(dev, info).first;
  }
  *out = it->second;
  return EF_OK;
}

// Find or grow the workspace of (current device, stream). Growth
// synchronises the stream once; the new header and tile-status array start
// at zero.
ef_status acquire_workspace(cudaStream_t stream, uint32_t tiles, uint32_t cand_cap,
                            size_t offsets, size_t stage, Workspace** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return EF_ERR_CUDA;
  std::lock_guard<std::mutex> lk(g_mu);
  Workspace*& ws = g_workspaces[std::make_pair(dev, stream)];
  if (!ws) {
    ws = new Workspace;
    ws->device = dev;
    ws->stream = stream;
    // the density hint (no hint when mapped host memory is unavailable)
    void* h = nullptr;
    if (cudaHostAlloc(&h, sizeof(uint32_t), cudaHostAllocMapped) == cudaSuccess) {
      void* dp = nullptr;
      *static_cast<volatile uint32_t*>(h) = 0u;
      if (cudaHostGetDevicePointer(&dp, h, 0) == cudaSuccess) {
        ws->density_host = static_cast<uint32_t*>(h);
        ws->density_dev = static_cast<uint32_t*>(dp);
      } else {
        cudaFreeHost(h);
      }
    }
    cudaGetLastError();
  }
  if (!ws->base || tiles > ws->status_tiles || cand_cap > ws->cand_cap ||
      offsets > ws->offsets_cap || stage > ws->stage_cap) {
    Workspace grown = *ws;
    if (tiles > grown.status_tiles) grown.status_tiles = tiles;
    if (cand_cap > grown.cand_cap) grown.cand_cap = cand_cap;
    if (offsets > grown.offsets_cap) grown.offsets_cap = offsets;
    if (stage > grown.stage_cap) grown.stage_cap = stage;
    const size_t bytes = grown.total_bytes();
    if (ws->base) {
      if (cudaStreamSynchronize(stream) != cudaSuccess) return EF_ERR_CUDA;
      cudaFree(ws->base);
      ws->base = nullptr;
    }
    void* p = nullptr;
    if (cudaMalloc(&p, bytes) != cudaSuccess) {
      cudaGetLastError();
      ws->status_tiles = ws->cand_cap = 0;
      ws->offsets_cap = ws->stage_cap = 0;
      return EF_ERR_NO_MEMORY;
    }
    grown.base = static_cast<char*>(p);
    grown.bytes = bytes;
    grown.dirty = true;
    *ws = grown;
  }
  if (ws->dirty) {
    // everything tagged with an epoch restarts from zero with the epochs
    const size_t clear = kHeaderBytes + sizeof(uint64_t) * ws->status_tiles;
    if (cudaMemsetAsync(ws->base, 0, clear, stream) != cudaSuccess ||
        cudaMemsetAsync(ws->chunks(), 0, sizeof(uint64_t) * kMaxChunks, stream) != cudaSuccess ||
        cudaMemsetAsync(ws->ht_chunks(0), 0, 2 * sizeof(uint64_t) * kMaxChunks, stream) !=
            cudaSuccess)
      return EF_ERR_CUDA;
    ws->epoch = 0;
    ws->ht_part_ready = false;  // no boundaries written for the next call
    ws->ht_last_tiles = 0;
    ws->dirty = false;
    if (ws->lw) ws->lw->valid = false;  // re-upload the tables, re-zero their counters
  }
  *out = ws;
  return EF_OK;
}

ef_status finish_launch(cudaError_t err, Workspace* ws) {
  if (err == cudaSuccess) return EF_OK;
  ws->dirty = true;  // a partial launch may leave the dispenser or barrier mid-way
  return EF_ERR_CUDA;
}

ef_status write_zero_count(uint32_t* count_out, cudaStream_t stream) {
  return cudaMemsetAsync(count_out, 0, sizeof(uint32_t), stream) == cudaSuccess ? EF_OK
                                                                                 : EF_ERR_CUDA;
}

ef_status write_err_zero(double* err_out, cudaStream_t stream) {
  if (!err_out) return EF_OK;
  return cudaMemsetAsync(err_out, 0, sizeof(double), stream) == cudaSuccess ? EF_OK : EF_ERR_CUDA;
}

ef_status hard_threshold_entry(const void* g, bool bf16, float* e, float gamma, float lambda,
                               uint64_t d, uint32_t* idx_out, float* val_out,
                               uint32_t* count_out, double* err_out, uint32_t* tiles_out,
                               cudaStream_t stream) {
  const size_t gsz = bf16 ? 2 : 4;
  if (!count_out || !aligned(count_out, 4)) return EF_ERR_INVALID_ARG;
  if (!std::isfinite(gamma) || !(lambda >= 0.0f)) return EF_ERR_INVALID_ARG;
  if (d > kMaxD) return EF_ERR_INVALID_ARG;
  if (err_out && !aligned(err_out, 8)) return EF_ERR_INVALID_ARG;
  if (tiles_out && !aligned(tiles_out, 4)) return EF_ERR_INVALID_ARG;
  if (d == 0) {
    ef_status z = write_zero_count(count_out, stream);
    if (z == EF_OK && tiles_out) z = write_zero_count(tiles_out, stream);  // one entry: 0
    return z != EF_OK ? z : write_err_zero(err_out, stream);
  }
  if (!g || !e || !idx_out || !val_out) return EF_ERR_INVALID_ARG;
  if (!aligned(g, gsz) || !aligned(e, 4) || !aligned(idx_out, 4) || !aligned(val_out, 4))
    return EF_ERR_INVALID_ARG;
  const size_t nb = static_cast<size_t>(d) * 4;
  const void* outs[3] = {idx_out, val_out, count_out};
  const size_t out_n[3] = {nb, nb, 4};
  for (int o = 0; o < 3; ++o) {
    if (overlaps(outs[o], out_n[o], g, d * gsz) || overlaps(outs[o], out_n[o], e, nb))
      return EF_ERR_INVALID_ARG;
    for (int p = o + 1; p < 3; ++p)
      if (overlaps(outs[o], out_n[o], outs[p], out_n[p])) return EF_ERR_INVALID_ARG;
  }
  if (overlaps(g, d * gsz, e, nb)) return EF_ERR_INVALID_ARG;
  if (err_out && (overlaps(err_out, 8, e, nb) || overlaps(err_out, 8, g, d * gsz) ||
                  overlaps(err_out, 8, idx_out, nb) || overlaps(err_out, 8, val_out, nb) ||
                  overlaps(err_out, 8, count_out, 4)))
    return EF_ERR_INVALID_ARG;
  const size_t tb = (static_cast<size_t>(tiles_for(d)) + 1) * 4;
  if (tiles_out && (overlaps(tiles_out, tb, e, nb) || overlaps(tiles_out, tb, g, d * gsz) ||
                    overlaps(tiles_out, tb, idx_out, nb) || overlaps(tiles_out, tb, val_out, nb) ||
                    overlaps(tiles_out, tb, count_out, 4) ||
                    (err_out && overlaps(tiles_out, tb, err_out, 8))))
    return EF_ERR_INVALID_ARG;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return EF_ERR_CUDA;
  DeviceInfo info;
  ef_status st = device_info(dev, &info);
  if (st != EF_OK) return st;
  Workspace* ws = nullptr;
  st = acquire_workspace(stream, tiles_for(d), 0, 0,
                         static_cast<size_t>(tiles_for(d)) * kTileElems, &ws);
  if (st != EF_OK) return st;
  return finish_launch(launch_hard_threshold(g, bf16, e, gamma, lambda, static_cast<uint32_t>(d),
                                             idx_out, val_out, count_out, err_out, tiles_out, *ws,
                                             info),
                       ws);
}

ef_status topk_entry(const void* g, bool bf16, float* e, float gamma, uint64_t k, uint64_t d,
                     uint32_t* idx_out, float* val_out, uint32_t* count_out, double* err_out,
                     cudaStream_t stream) {
  const size_t gsz = bf16 ? 2 : 4;
  if (!count_out || !aligned(count_out, 4)) return EF_ERR_INVALID_ARG;
  if (!std::isfinite(gamma)) return EF_ERR_INVALID_ARG;
  if (d > kMaxD || k > d) return EF_ERR_INVALID_ARG;
  if (err_out && !aligned(err_out, 8)) return EF_ERR_INVALID_ARG;
  if (d == 0) {
    const ef_status z = write_zero_count(count_out, stream);
    return z != EF_OK ? z : write_err_zero(err_out, stream);
  }
  if (!g || !e || (k > 0 && (!idx_out || !val_out))) return EF_ERR_INVALID_ARG;
  if (!aligned(g, gsz) || !aligned(e, 4) || !aligned(idx_out, 4) || !aligned(val_out, 4))
    return EF_ERR_INVALID_ARG;
  const size_t nb = static_cast<size_t>(d) * 4, kb = static_cast<size_t>(k) * 4;
  const void* outs[3] = {idx_out, val_out, count_out};
  const size_t out_n[3] = {kb, kb, 4};
  for (int o = 0; o < 3; ++o) {
    if (overlaps(outs[o], out_n[o], g, d * gsz) || overlaps(outs[o], out_n[o], e, nb))
      return EF_ERR_INVALID_ARG;
    for (int p = o + 1; p < 3; ++p)
      if (overlaps(outs[o], out_n[o], outs[p], out_n[p])) return EF_ERR_INVALID_ARG;
  }
  if (overlaps(g, d * gsz, e, nb)) return EF_ERR_INVALID_ARG;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return EF_ERR_CUDA;
  DeviceInfo info;
  ef_status st = device_info(dev, &info);
  if (st != EF_OK) return st;
  Workspace* ws = nullptr;
  st = acquire_workspace(stream, tiles_for(d), topk_candidate_capacity(d), 0,
                         static_cast<size_t>(tiles_for(d)) * kTileElems, &ws);
  if (st != EF_OK) return st;
  if (err_out && (overlaps(err_out, 8, e, nb) || overlaps(err_out, 8, g, d * gsz) ||
                  overlaps(err_out, 8, idx_out, kb) || overlaps(err_out, 8, val_out, kb) ||
                  overlaps(err_out, 8, count_out, 4)))
    return EF_ERR_INVALID_ARG;
  return finish_launch(launch_topk(g, bf16, e, gamma, static_cast<uint32_t>(k),
                                   static_cast<uint32_t>(d), idx_out, val_out, count_out, err_out,
                                   *ws, info),
                       ws);
}

ef_status topk_layerwise_entry(const void* g, bool bf16, float* e, float gamma, uint32_t n_seg,
                               const uint64_t* seg_end, const uint64_t* seg_k, uint64_t d,
                               uint32_t* idx_out, float* val_out, uint32_t* count_out,
                               double* err_out, cudaStream_t stream) {
  const size_t gsz = bf16 ? 2 : 4;
  if (!count_out || !aligned(count_out, 4)) return EF_ERR_INVALID_ARG;
  if (!std::isfinite(gamma) || d > kMaxD) return EF_ERR_INVALID_ARG;
  if (n_seg == 0 || n_seg >= (1u << 31) || !seg_end || !seg_k) return EF_ERR_INVALID_ARG;
  uint64_t lo = 0, total_k = 0;
  for (uint32_t s = 0; s < n_seg; ++s) {
    if (seg_end[s] < lo || seg_end[s] > d || seg_k[s] > seg_end[s] - lo)
      return EF_ERR_INVALID_ARG;
    total_k += seg_k[s];
    lo = seg_end[s];
  }
  if (lo != d) return EF_ERR_INVALID_ARG;
  if (err_out && !aligned(err_out, 8)) return EF_ERR_INVALID_ARG;
  if (d == 0) {
    const ef_status z = write_zero_count(count_out, stream);
    return z != EF_OK ? z : write_err_zero(err_out, stream);
  }
  if (!g || !e || (total_k > 0 && (!idx_out || !val_out))) return EF_ERR_INVALID_ARG;
  if (!aligned(g, gsz) || !aligned(e, 4) || !aligned(idx_out, 4) || !aligned(val_out, 4))
    return EF_ERR_INVALID_ARG;
  const size_t nb = static_cast<size_t>(d) * 4, kb = static_cast<size_t>(total_k) * 4;
  const void* outs[3] = {idx_out, val_out, count_out};
  const size_t out_n[3] = {kb, kb, 4};
  for (int o = 0; o < 3; ++o) {
    if (overlaps(outs[o], out_n[o], g, d * gsz) || overlaps(outs[o], out_n[o], e, nb))
      return EF_ERR_INVALID_ARG;
    for (int p = o + 1; p < 3; ++p)
      if (overlaps(outs[o], out_n[o], outs[p], out_n[p])) return EF_ERR_INVALID_ARG;
  }
  if (overlaps(g, d * gsz, e, nb)) return EF_ERR_INVALID_ARG;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return EF_ERR_CUDA;
  DeviceInfo info;
  ef_status st = device_info(dev, &info);
  if (st != EF_OK) return st;
  Workspace* ws = nullptr;
  st = acquire_workspace(stream, tiles_for(d), topk_candidate_capacity(d), 0,
                         static_cast<size_t>(tiles_for(d)) * kTileElems, &ws);
  if (st != EF_OK) return st;
  if (err_out && (overlaps(err_out, 8, e, nb) || overlaps(err_out, 8, g, d * gsz) ||
                  overlaps(err_out, 8, idx_out, kb) || overlaps(err_out, 8, val_out, kb) ||
                  overlaps(err_out, 8, count_out, 4)))
    return EF_ERR_INVALID_ARG;
  const cudaError_t perr = lw_prepare(*ws, seg_end, seg_k, n_seg, d, info);
  if (perr == cudaErrorMemoryAllocation) return EF_ERR_NO_MEMORY;
  if (perr != cudaSuccess) return EF_ERR_CUDA;
  return finish_launch(launch_topk_layerwise(g, bf16, e, gamma, static_cast<uint32_t>(d),
                                             idx_out, val_out, count_out, err_out, *ws, info),
                       ws);
}

}  // namespace

// A launch that may begin while the previous kernel on the stream finishes
// (programmatic dependent launch; every kernel here waits for its
// predecessor before reading what it wrote), optionally cooperative.
cudaError_t launch_pdl(const void* fn, dim3 grid, uint32_t block, uint32_t smem,
                       cudaStream_t stream, void** params, bool cooperative) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = dim3(block);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeCooperative;
  attr[1].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = cooperative ? 2 : 1;
  return cudaLaunchKernelExC(&cfg, fn, params);
}

void count_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }
uint64_t wait_limit_ns() { return g_wait_limit_ns.load(); }
int64_t withheld_tile() { return g_withheld_tile.load(); }
int stream_kernel_mode() { return g_stream_kernel_mode.load(); }

ScanCtx next_scan_ctx(Workspace& ws, uint32_t num_tiles) {
  if (ws.epoch >= (1u << 30) - 1) {  // epoch wrap: old words must not match again
    cudaMemsetAsync(ws.status(), 0, sizeof(uint64_t) * ws.status_tiles, ws.stream);
    cudaMemsetAsync(ws.chunks(), 0, sizeof(uint64_t) * kMaxChunks, ws.stream);
    ws.epoch = 0;
  }
  ++ws.epoch;
  ScanCtx c;
  c.status = ws.status();
  c.error = ws.u32(kOffError);
  c.epoch = ws.epoch;
  c.num_tiles = num_tiles;
  c.withheld_tile = withheld_tile();
  c.wait_limit_ns = wait_limit_ns();
  c.tile_claim = ws.u32(kOffTileClaim);
  return c;
}

// The aggregate entries: the plain sum (dense_out set) or the fused update
// (x set); tiles optional.
ef_status aggregate_entry(uint32_t n, const uint32_t* const* idx, const float* const* val,
                          const uint32_t* const* tiles, const uint32_t* counts, uint64_t d,
                          float* dense_out, float alpha, float* x, float* m, float momentum,
                          float lr, cudaStream_t s) {
  if (n == 0 || n > kMaxWorkers || !idx || !val || !counts) return EF_ERR_INVALID_ARG;
  if (d > kMaxD) return EF_ERR_INVALID_ARG;
  const bool apply = x != nullptr;
  if (apply && (!std::isfinite(alpha) || !std::isfinite(momentum) || !std::isfinite(lr)))
    return EF_ERR_INVALID_ARG;
  if (d == 0) return EF_OK;
  const size_t nb = static_cast<size_t>(d) * 4;
  if (!aligned(counts, 4)) return EF_ERR_INVALID_ARG;
  if (apply) {
    if (!aligned(x, 4) || (m && !aligned(m, 4))) return EF_ERR_INVALID_ARG;
    if (m && overlaps(x, nb, m, nb)) return EF_ERR_INVALID_ARG;
  } else if (!dense_out || !aligned(dense_out, 4)) {
    return EF_ERR_INVALID_ARG;
  }
  for (uint32_t i = 0; i < n; ++i) {
    if (!idx[i] || !val[i] || !aligned(idx[i], 4) || !aligned(val[i], 4))
      return EF_ERR_INVALID_ARG;
    if (tiles && (!tiles[i] || !aligned(tiles[i], 4))) return EF_ERR_INVALID_ARG;
  }
  const uint32_t nt = agg_tiles_for(d);
  int dev = 0;  // the per-device set-up (kernel attributes) on first use
  DeviceInfo info;
  if (cudaGetDevice(&dev) != cudaSuccess) return EF_ERR_CUDA;
  if (device_info(dev, &info) != EF_OK) return EF_ERR_CUDA;
  Workspace* ws = nullptr;
  const size_t offsets = tiles ? 0 : static_cast<size_t>(n) * (static_cast<size_t>(nt) + 1);
  const ef_status st = acquire_workspace(s, 0, 0, offsets, 0, &ws);
  if (st != EF_OK) return st;
  const uint32_t d32 = static_cast<uint32_t>(d);
  if (apply)
    return finish_launch(
        launch_aggregate_apply(n, idx, val, tiles, counts, d32, alpha, x, m, momentum, lr, *ws),
        ws);
  return finish_launch(launch_aggregate(n, idx, val, tiles, counts, d32, dense_out, *ws), ws);
}

}  // namespace efs

using efs::Workspace;

extern "C" {

ef_status ef_hard_threshold(const float* g, float* e, float gamma, float lambda, uint64_t d,
                            uint32_t* idx_out, float* val_out, uint32_t* count_out,
                            ef_stream_t stream) {
  return efs::hard_threshold_entry(g, false, e, gamma, lambda, d, idx_out, val_out, count_out,
                                   nullptr, nullptr, reinterpret_cast<cudaStream_t>(stream));
}

ef_status ef_hard_threshold_bf16(const uint16_t* g, float* e, float gamma, float lambda,
                                 uint64_t d, uint32_t* idx_out, float* val_out,
                                 uint32_t* count_out, ef_stream_t stream) {
  return efs::hard_threshold_entry(g, true, e, gamma, lambda, d, idx_out, val_out, count_out,
                                   nullptr, nullptr, reinterpret_cast<cudaStream_t>(stream));
}

ef_status ef_topk(const float* g, float* e, float gamma, uint64_t k, uint64_t d,
                  uint32_t* idx_out, float* val_out, uint32_t* count_out, ef_stream_t stream) {
  return efs::topk_entry(g, false, e, gamma, k, d, idx_out, val_out, count_out, nullptr,
                         reinterpret_cast<cudaStream_t>(stream));
}

ef_status ef_topk_bf16(const uint16_t* g, float* e, float gamma, uint64_t k, uint64_t d,
                       uint32_t* idx_out, float* val_out, uint32_t* count_out,
                       ef_stream_t stream) {
  return efs::topk_entry(g, true, e, gamma, k, d, idx_out, val_out, count_out, nullptr,
                         reinterpret_cast<cudaStream_t>(stream));
}

ef_status ef_topk_layerwise(const float* g, float* e, float gamma, uint32_t n_seg,
                            const uint64_t* seg_end, const uint64_t* seg_k, uint64_t d,
                            uint32_t* idx_out, float* val_out, uint32_t* count_out,
                            ef_stream_t stream) {
  return efs::topk_layerwise_entry(g, false, e, gamma, n_seg, seg_end, seg_k, d, idx_out,
                                   val_out, count_out, nullptr,
                                   reinterpret_cast<cudaStream_t>(stream));
}

ef_status ef_topk_layerwise_bf16(const uint16_t* g, float* e, float gamma, uint32_t n_seg,
                                 const uint64_t* seg_end, const uint64_t* seg_k, uint64_t d,
                                 uint32_t* idx_out, float* val_out, uint32_t* count_out,
                                 ef_stream_t stream) {
  return efs::topk_layerwise_entry(g, true, e, gamma, n_seg, seg_end, seg_k, d, idx_out,
                                   val_out, count_out, nullptr,
                                   reinterpret_cast<cudaStream_t>(stream));
}

ef_status ef_hard_threshold_ex(const void* g, ef_grad_type g_type, float* e, float gamma,
                               float lambda, uint64_t d, uint32_t* idx_out, float* val_out,
                               uint32_t* count_out, double* err_sq_out, ef_stream_t stream) {
  if (g_type != EF_GRAD_F32 && g_type != EF_GRAD_BF16) return EF_ERR_INVALID_ARG;
  return efs::hard_threshold_entry(g, g_type == EF_GRAD_BF16, e, gamma, lambda, d, idx_out,
                                   val_out, count_out, err_sq_out, nullptr,
                                   reinterpret_cast<cudaStream_t>(stream));
}

ef_status ef_hard_threshold_tiled(const void* g, ef_grad_type g_type, float* e, float gamma,
                                  float lambda, uint64_t d, uint32_t* idx_out, float* val_out,
                                  uint32_t* count_out, uint32_t* tiles_out, double* err_sq_out,
                                  ef_stream_t stream) {
  if (g_type != EF_GRAD_F32 && g_type != EF_GRAD_BF16) return EF_ERR_INVALID_ARG;
  if (!tiles_out) return EF_ERR_INVALID_ARG;
  return efs::hard_threshold_entry(g, g_type == EF_GRAD_BF16, e, gamma, lambda, d, idx_out,
                                   val_out, count_out, err_sq_out, tiles_out,
                                   reinterpret_cast<cudaStream_t>(stream));
}

ef_status ef_topk_ex(const void* g, ef_grad_type g_type, float* e, float gamma, uint64_t k,
                     uint64_t d, uint32_t* idx_out, float* val_out, uint32_t* count_out,
                     double* err_sq_out, ef_stream_t stream) {
  if (g_type != EF_GRAD_F32 && g_type != EF_GRAD_BF16) return EF_ERR_INVALID_ARG;
  return efs::topk_entry(g, g_type == EF_GRAD_BF16, e, gamma, k, d, idx_out, val_out, count_out,
                         err_sq_out, reinterpret_cast<cudaStream_t>(stream));
}

ef_status ef_topk_layerwise_ex(const void* g, ef_grad_type g_type, float* e, float gamma,
                               uint32_t n_seg, const uint64_t* seg_end, const uint64_t* seg_k,
                               uint64_t d, uint32_t* idx_out, float* val_out,
                               uint32_t* count_out, double* err_sq_out, ef_stream_t stream) {
  if (g_type != EF_GRAD_F32 && g_type != EF_GRAD_BF16) return EF_ERR_INVALID_ARG;
  return efs::topk_layerwise_entry(g, g_type == EF_GRAD_BF16, e, gamma, n_seg, seg_end, seg_k,
                                   d, idx_out, val_out, count_out, err_sq_out,
                                   reinterpret_cast<cudaStream_t>(stream));
}

ef_status sparse_aggregate(uint32_t n, const uint32_t* const* idx, const float* const* val,
                           const uint32_t* counts, uint64_t d, float* dense_out,
                           ef_stream_t stream) {
  return efs::aggregate_entry(n, idx, val, nullptr, counts, d, dense_out, 0.0f, nullptr,
                              nullptr, 0.0f, 0.0f, reinterpret_cast<cudaStream_t>(stream));
}

ef_status sparse_aggregate_tiled(uint32_t n, const uint32_t* const* idx, const float* const* val,
                                 const uint32_t* const* tiles, const uint32_t* counts, uint64_t d,
                                 float* dense_out, ef_stream_t stream) {
  if (!tiles) return EF_ERR_INVALID_ARG;
  return efs::aggregate_entry(n, idx, val, tiles, counts, d, dense_out, 0.0f, nullptr, nullptr,
                              0.0f, 0.0f, reinterpret_cast<cudaStream_t>(stream));
}

ef_status sparse_aggregate_apply(uint32_t n, const uint32_t* const* idx, const float* const* val,
                                 const uint32_t* counts, uint64_t d, float alpha, float* x,
                                 float* m, float momentum, float lr, ef_stream_t stream) {
  if (!x) return EF_ERR_INVALID_ARG;
  return efs::aggregate_entry(n, idx, val, nullptr, counts, d, nullptr, alpha, x, m, momentum,
                              lr, reinterpret_cast<cudaStream_t>(stream));
}

ef_status sparse_aggregate_apply_tiled(uint32_t n, const uint32_t* const* idx,
                                       const float* const* val, const uint32_t* const* tiles,
                                       const uint32_t* counts, uint64_t d, float alpha, float* x,
                                       float* m, float momentum, float lr, ef_stream_t stream) {
  if (!tiles || !x) return EF_ERR_INVALID_ARG;
  return efs::aggregate_entry(n, idx, val, tiles, counts, d, nullptr, alpha, x, m, momentum, lr,
                              reinterpret_cast<cudaStream_t>(stream));
}

ef_status ef_scaled_round_ex(const void* g, ef_grad_type g_type, float* e, float gamma,
                             int32_t scale_log2, uint64_t d, int32_t* q_out,
                             uint32_t* unsent_out, double* err_sq_out, ef_stream_t stream) {
  using namespace efs;
  const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (g_type != EF_GRAD_F32 && g_type != EF_GRAD_BF16) return EF_ERR_INVALID_ARG;
  const bool bf16 = g_type == EF_GRAD_BF16;
  const size_t gsz = bf16 ? 2 : 4;
  if (!std::isfinite(gamma) || scale_log2 < -100 || scale_log2 > 100) return EF_ERR_INVALID_ARG;
  if (d > kMaxD || !unsent_out || !aligned(unsent_out, 4)) return EF_ERR_INVALID_ARG;
  if (err_sq_out && !aligned(err_sq_out, 8)) return EF_ERR_INVALID_ARG;
  if (d == 0) {
    if (cudaMemsetAsync(unsent_out, 0, sizeof(uint32_t), s) != cudaSuccess) return EF_ERR_CUDA;
    return write_err_zero(err_sq_out, s);
  }
  if (!g || !e || !q_out || !aligned(g, gsz) || !aligned(e, 4) || !aligned(q_out, 4))
    return EF_ERR_INVALID_ARG;
  const size_t nb = static_cast<size_t>(d) * 4;
  if (overlaps(g, d * gsz, e, nb) || overlaps(q_out, nb, g, d * gsz) || overlaps(q_out, nb, e, nb) ||
      overlaps(unsent_out, 4, g, d * gsz) || overlaps(unsent_out, 4, e, nb) ||
      overlaps(unsent_out, 4, q_out, nb))
    return EF_ERR_INVALID_ARG;
  if (err_sq_out && (overlaps(err_sq_out, 8, g, d * gsz) || overlaps(err_sq_out, 8, e, nb) ||
                     overlaps(err_sq_out, 8, q_out, nb) || overlaps(err_sq_out, 8, unsent_out, 4)))
    return EF_ERR_INVALID_ARG;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return EF_ERR_CUDA;
  DeviceInfo info;
  ef_status st = device_info(dev, &info);
  if (st != EF_OK) return st;
  Workspace* ws = nullptr;
  st = acquire_workspace(s, 0, 0, 0, 0, &ws);
  if (st != EF_OK) return st;
  return finish_launch(launch_scaled_round(g, bf16, e, gamma, scale_log2,
                                           static_cast<uint32_t>(d), q_out, unsent_out,
                                           err_sq_out, *ws, info),
                       ws);
}

ef_status int_aggregate(uint32_t n, const int32_t* const* q, uint64_t d, int32_t scale_log2,
                        float* dense_out, ef_stream_t stream) {
  using namespace efs;
  if (n == 0 || n > kMaxWorkers || !q) return EF_ERR_INVALID_ARG;
  if (d > kMaxD || scale_log2 < -100 || scale_log2 > 100) return EF_ERR_INVALID_ARG;
  if (d == 0) return EF_OK;
  if (!dense_out || !aligned(dense_out, 4)) return EF_ERR_INVALID_ARG;
  for (uint32_t i = 0; i < n; ++i) {
    if (!q[i] || !aligned(q[i], 4)) return EF_ERR_INVALID_ARG;
    if (overlaps(q[i], static_cast<size_t>(d) * 4, dense_out, static_cast<size_t>(d) * 4))
      return EF_ERR_INVALID_ARG;
  }
  const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return EF_ERR_CUDA;
  DeviceInfo info;
  ef_status st = device_info(dev, &info);
  if (st != EF_OK) return st;
  Workspace* ws = nullptr;
  st = acquire_workspace(s, 0, 0, 0, 0, &ws);
  if (st != EF_OK) return st;
  return finish_launch(
      launch_int_aggregate(n, q, static_cast<uint32_t>(d), scale_log2, dense_out, *ws, info), ws);
}

ef_status ef_check_status(ef_stream_t stream) {
  const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (cudaStreamSynchronize(s) != cudaSuccess) return EF_ERR_CUDA;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return EF_ERR_CUDA;
  Workspace* ws = nullptr;
  {
    std::lock_guard<std::mutex> lk(efs::g_mu);
    auto it = efs::g_workspaces.find(std::make_pair(dev, s));
    if (it == efs::g_workspaces.end() || !it->second->base) return EF_OK;
    ws = it->second;
  }
  uint32_t bits = 0;
  uint32_t* dev_err = ws->u32(efs::kOffError);
  if (cudaMemcpyAsync(&bits, dev_err, sizeof bits, cudaMemcpyDeviceToHost, s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess)
    return EF_ERR_CUDA;
  if (bits == 0) return EF_OK;
  if (cudaMemsetAsync(dev_err, 0, sizeof bits, s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess)
    return EF_ERR_CUDA;
  {
    // a wait that ran out, or a selection that stopped early, may leave
    // barrier counters or histograms mid-way: re-clear the workspace before
    // the next launch on this stream
    std::lock_guard<std::mutex> lk(efs::g_mu);
    ws->dirty = true;
  }
  return (bits & efs::kDevErrTimeout) ? EF_ERR_TIMEOUT : EF_ERR_BAD_INPUT;
}

const char* ef_status_string(ef_status status) {
  switch (status) {
    case EF_OK: return "EF_OK";
    case EF_ERR_INVALID_ARG: return "EF_ERR_INVALID_ARG";
    case EF_ERR_CUDA: return "EF_ERR_CUDA";
    case EF_ERR_TIMEOUT: return "EF_ERR_TIMEOUT";
    case EF_ERR_BAD_INPUT: return "EF_ERR_BAD_INPUT";
    case EF_ERR_NO_MEMORY: return "EF_ERR_NO_MEMORY";
  }
  return "EF_ERR_UNKNOWN";
}

ef_status ef_workspace_release(void) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return EF_ERR_CUDA;
  if (cudaDeviceSynchronize() != cudaSuccess) return EF_ERR_CUDA;
  std::lock_guard<std::mutex> lk(efs::g_mu);
  for (auto it = efs::g_workspaces.begin(); it != efs::g_workspaces.end();) {
    if (it->first.first == dev) {
      if (it->second->base) cudaFree(it->second->base);
      if (it->second->density_host) cudaFreeHost(it->second->density_host);
      if (it->second->lw) {
        if (it->second->lw->dev) cudaFree(it->second->lw->dev);
        delete it->second->lw;
      }
      delete it->second;
      it = efs::g_workspaces.erase(it);
    } else {
      ++it;
    }
  }
  return EF_OK;
}

uint64_t ef_kernel_launches(void) { return efs::g_launches.load(); }

void ef_test_set_lookback_fault(int64_t withheld_tile, uint32_t spin_limit_us) {
  efs::g_withheld_tile.store(withheld_tile < 0 ? -1 : withheld_tile);
  efs::g_wait_limit_ns.store(withheld_tile < 0 ? 2000000000ull
                                               : static_cast<uint64_t>(spin_limit_us) * 1000ull);
}

void ef_test_set_stream_kernel(int mode) {
  efs::g_stream_kernel_mode.store(mode >= 1 && mode <= 3 ? mode : 0);
}

}  // extern "C"
