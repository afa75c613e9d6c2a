// ht.cu — the fused error-feedback + hard-threshold + compaction kernel.
//
// One pass over the d coordinates performs, per coordinate j (Algorithm 1
// with the hard-threshold sparsifier of Sec. 1 / Sec. 4.2):
//   a_j  = fmaf(gamma, g_j, e_j)                 corrected update p = e + gamma g
//   s_j  = (|a_j| >= lambda) and (a_j != 0)      j in S_lambda(a)
//   e_j <- s_j ? +0 : a_j                        error update e <- p - C(p)
// and writes the selected (j, a_j) pairs in ascending j through the ordered
// compaction. HBM traffic per coordinate is the algorithmic minimum: read g
// (4 B, or 2 B for bf16) and e (4 B), write e (4 B); plus 8 B per sent pair.
#include "compact.cuh"
#include "gradient.cuh"
#include "internal.h"
#include "stream_lookback.cuh"

namespace efs {
namespace {

__device__ __forceinline__ uint32_t in_support(float a, float lambda) {
  return (fabsf(a) >= lambda && a != 0.0f) ? 1u : 0u;
}

template <typename GT, bool kVec>
__global__ void __launch_bounds__(kThreads)
    ht_kernel(const GT* __restrict__ g, float* __restrict__ e, float gamma, float lambda,
              uint32_t d, uint32_t* __restrict__ idx_out, float* __restrict__ val_out,
              uint32_t* __restrict__ count_out, ScanCtx ctx) {
  // The tile comes from the dispenser, in the order CTAs start, so every
  // lower tile this CTA's look-back waits for is held by a running CTA.
  __shared__ uint32_t s_tile;
  if (threadIdx.x == 0) s_tile = atomicAdd(ctx.tile_claim, 1u);
  __syncthreads();
  const uint32_t tile = s_tile;
  if (tile >= ctx.num_tiles) {
    // the dispenser did not start at zero (an earlier launch was cut short):
    // touch nothing, report it, and still count this CTA as finished
    if (threadIdx.x == 0) {
      atomicOr(ctx.error, kDevErrTimeout);
      if (atomicAdd(ctx.tile_claim + 1, 1u) == gridDim.x - 1) {
        ctx.tile_claim[0] = 0;
        ctx.tile_claim[1] = 0;
      }
    }
    return;
  }
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const uint64_t first = element_index(tile, warp, 0, lane, 0);

  float a[kUnits][4];
  uint32_t sel[kUnits];
  const bool full_tile = static_cast<uint64_t>(tile + 1) * kTileElems <= d;

  if (kVec && full_tile) {
    GradVec<GT> gv[kUnits];
    float4 ev[kUnits];
#pragma unroll
    for (int v = 0; v < kUnits; ++v) {  // all loads in flight before any use
      gv[v].load(g + first + v * 128);
      ev[v] = ld_stream_f4(e + first + v * 128);
    }
#pragma unroll
    for (int v = 0; v < kUnits; ++v) {
      a[v][0] = __fmaf_rn(gamma, gv[v][0], ev[v].x);
      a[v][1] = __fmaf_rn(gamma, gv[v][1], ev[v].y);
      a[v][2] = __fmaf_rn(gamma, gv[v][2], ev[v].z);
      a[v][3] = __fmaf_rn(gamma, gv[v][3], ev[v].w);
      sel[v] = in_support(a[v][0], lambda) | (in_support(a[v][1], lambda) << 1) |
               (in_support(a[v][2], lambda) << 2) | (in_support(a[v][3], lambda) << 3);
      const float4 r = make_float4((sel[v] & 1u) ? 0.0f : a[v][0], (sel[v] & 2u) ? 0.0f : a[v][1],
                                   (sel[v] & 4u) ? 0.0f : a[v][2], (sel[v] & 8u) ? 0.0f : a[v][3]);
      st_stream_f4(e + first + v * 128, r);
    }
  } else {
#pragma unroll
    for (int v = 0; v < kUnits; ++v) {
      sel[v] = 0;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const uint64_t i = first + v * 128 + j;
        a[v][j] = 0.0f;
        if (i < d) {
          const float x = __fmaf_rn(gamma, grad_scalar(g, i), e[i]);
          const uint32_t s = in_support(x, lambda);
          a[v][j] = x;
          sel[v] |= s << j;
          e[i] = s ? 0.0f : x;
        }
      }
    }
  }
  compact_tile(ctx, tile, sel, a, idx_out, val_out, count_out, d);
  if (threadIdx.x == 0) {
    // every CTA took its tile before it counts itself finished; the last one
    // leaves the dispenser at zero for the next launch
    __threadfence();
    if (atomicAdd(ctx.tile_claim + 1, 1u) == gridDim.x - 1) {
      ctx.tile_claim[0] = 0;
      ctx.tile_claim[1] = 0;
    }
  }
}

// The hard-threshold step as a streaming-compaction op: a stage holds a
// tile of g followed by the same tile of e; the residual is written to e from
// registers with streaming stores.
template <typename GT>
struct HtOp {
  const GT* g;
  float* e;
  float gamma, lambda;
  uint32_t d;
  static constexpr uint32_t kGBytes = kTileElems * sizeof(GT);
  static constexpr uint32_t kStageBytes = kGBytes + kTileElems * sizeof(float);
  static constexpr uint32_t kWarpStagePairs = 768;  // on-chip staged pairs per compute warp
  static constexpr bool kKeepPairs = false;  // the message: read by the exchange, much later
  __device__ void prologue() const {}
  __device__ uint64_t initial_aux() const { return 0; }

  // the chunk's first tiles of g and e toward L2 before the wait for the
  // previous kernel (its tail leaves DRAM mostly idle)
  static constexpr uint32_t kPrefetchTiles = 8;
  __device__ __forceinline__ void prefetch(uint32_t t) const {
    prefetch_l2_1d(g + static_cast<size_t>(t) * kTileElems, kGBytes);
    prefetch_l2_1d(e + static_cast<size_t>(t) * kTileElems, kTileElems * sizeof(float));
  }
  __device__ __forceinline__ void fill(unsigned char* stage, uint32_t t, uint64_t* bar,
                                       uint64_t policy) const {
    tma_load_1d(stage, g + static_cast<size_t>(t) * kTileElems, kGBytes, bar, policy);
    tma_load_1d(stage + kGBytes, e + static_cast<size_t>(t) * kTileElems,
                kTileElems * sizeof(float), bar, policy);
  }

  __device__ __forceinline__ void tile_smem(const unsigned char* stage, uint32_t t, int warp,
                                            int lane, float (&a)[kSUnits][4],
                                            uint32_t (&sel)[kSUnits], uint64_t) const {
    const GT* gs = reinterpret_cast<const GT*>(stage);
    const float* es = reinterpret_cast<const float*>(stage + kGBytes);
    const int local = warp * kSWarpElems + lane * 4;
    float* eg = e + stream_element_index(t, warp, 0, lane, 0);
    // with lambda > 0, |a| >= lambda already excludes a == 0 (and NaN): one
    // comparison a coordinate; lambda == 0 keeps the a != 0 test
    const bool pos = lambda > 0.0f;
#pragma unroll
    for (int v = 0; v < kSUnits; ++v) {
      GradVec<GT> gv;
      if constexpr (sizeof(GT) == 4)
        gv.v = *reinterpret_cast<const float4*>(gs + local + v * 128);
      else
        gv.v = *reinterpret_cast<const uint2*>(gs + local + v * 128);
      const float4 ev = *reinterpret_cast<const float4*>(es + local + v * 128);
      a[v][0] = __fmaf_rn(gamma, gv[0], ev.x);
      a[v][1] = __fmaf_rn(gamma, gv[1], ev.y);
      a[v][2] = __fmaf_rn(gamma, gv[2], ev.z);
      a[v][3] = __fmaf_rn(gamma, gv[3], ev.w);
      bool s[4];
#pragma unroll
      for (int j = 0; j < 4; ++j)
        s[j] = pos ? fabsf(a[v][j]) >= lambda : in_support(a[v][j], lambda) != 0u;
      sel[v] = (s[0] ? 1u : 0u) | (s[1] ? 2u : 0u) | (s[2] ? 4u : 0u) | (s[3] ? 8u : 0u);
      st_stream_f4(eg + v * 128, make_float4(s[0] ? 0.0f : a[v][0], s[1] ? 0.0f : a[v][1],
                                             s[2] ? 0.0f : a[v][2], s[3] ? 0.0f : a[v][3]));
    }
  }

  __device__ __forceinline__ void tile_global(uint32_t t, int warp, int lane,
                                              float (&a)[kSUnits][4],
                                              uint32_t (&sel)[kSUnits], uint64_t) const {
    const uint64_t first = stream_element_index(t, warp, 0, lane, 0);
#pragma unroll
    for (int v = 0; v < kSUnits; ++v) {
      sel[v] = 0;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const uint64_t i = first + v * 128 + j;
        a[v][j] = 0.0f;
        if (i < d) {
          const float x = __fmaf_rn(gamma, grad_scalar(g, i), e[i]);
          const uint32_t sj = in_support(x, lambda);
          a[v][j] = x;
          sel[v] |= sj << j;
          e[i] = sj ? 0.0f : x;
        }
      }
    }
  }
};

// ring stages: 4 of 32 KB (fp32 g); bf16 g makes a stage 24 KB, and a fifth
// stage keeps about as many bytes in flight within the same shared memory
template <typename GT>
constexpr int kHtStages = sizeof(GT) == 2 ? 5 : 4;

template <typename GT, int kStages = kHtStages<GT>>
using HtGroupKernel = LbLayout<HtOp<GT>, kStages>;
template <typename GT>
using HtChunkKernel = StreamLayout<HtOp<GT>, kHtStages<GT>>;

// Streaming hard-threshold over dynamically claimed groups of tiles: one CTA
// per SM. A group waits only for groups claimed before it, held by running
// CTAs, so the launch needs no co-residency. Programmatic: it may start while
// the previous kernel on the stream finishes (the kernel waits for it before
// its first read). kStages: the ring depth (one stage fewer for dense calls,
// whose pair buffers then take the freed shared memory).
template <typename GT, int kStages>
cudaError_t launch_groups(const GT* g, float* e, float gamma, float lambda, uint32_t d,
                          uint32_t* idx_out, float* val_out, uint32_t* count_out, double* err_out,
                          uint32_t* tiles_out, Workspace& ws, const DeviceInfo& dev,
                          const ScanCtx& ctx, int per_sm) {
  const uint32_t tiles = tiles_for(d);
  HtOp<GT> op{g, e, gamma, lambda, d};
  const uint32_t groups = (tiles + kLbGroupTiles - 1) / kLbGroupTiles;
  const uint32_t slots = static_cast<uint32_t>(per_sm * dev.sm_count);
  const uint32_t grid = groups < slots ? groups : slots;
  uint32_t cap = d;
  ScanCtx c = ctx;
  // the groups' shares of ||e'||^2 use the per-tile count area (16 words a tile)
  LbArgs la{tiles_out, err_out, reinterpret_cast<FF*>(ws.counts()), ws.stage_idx(),
            ws.stage_val(), ws.density_dev};
  void* params[] = {&op, &d, &idx_out, &val_out, &count_out, &cap, &c, &la};
  const cudaError_t err = launch_pdl(
      reinterpret_cast<const void*>(&lookback_stream_kernel<HtOp<GT>, kStages>), grid,
      kLbThreads, HtGroupKernel<GT, kStages>::kSmem, ws.stream, params, false);
  count_launch();
  ws.ht_part_ready = false;  // the chunk kernel's boundaries are not written by this kernel
  return err;
}

// Streaming hard-threshold over static chunks (stream_compact.cuh): one CTA
// per SM, CTA c waiting only on the chunk totals of lower-numbered CTAs. The
// grid fits the device at once and CTAs are dispatched in index order, so
// those CTAs are running; if other work holds SMs long enough that one cannot
// start, the bounded wait ends the call with EF_ERR_TIMEOUT (never a hang or a
// wrong result). Balanced chunks: the previous call of this size wrote this
// call's chunk boundaries from its chunk totals (dense regions get fewer
// tiles); any boundaries partition the tiles, so the result never depends on
// them.
template <typename GT>
cudaError_t launch_chunks(const GT* g, float* e, float gamma, float lambda, uint32_t d,
                          uint32_t* idx_out, float* val_out, uint32_t* count_out, double* err_out,
                          uint32_t* tiles_out, Workspace& ws, const DeviceInfo& dev,
                          const ScanCtx& ctx, int per_sm) {
  const uint32_t tiles = tiles_for(d);
  HtOp<GT> op{g, e, gamma, lambda, d};
  uint32_t slots = static_cast<uint32_t>(per_sm * dev.sm_count);
  if (slots > kMaxChunks) slots = kMaxChunks;
  const uint32_t grid = tiles < slots ? tiles : slots;
  uint32_t cap = d;
  ScanCtx c = ctx;
  StreamArgs sa{ws.stage_idx(), ws.stage_val(), ws.counts(), ws.ht_chunks(ws.ht_seq), tiles_out,
                err_out, ws.errparts()};
  const uint32_t seq = ws.ht_seq;
  const bool same = seq > 0 && ws.ht_last_tiles == tiles && ws.ht_last_grid == grid;
  // (a call that returns ||e'||^2 uses equal chunks: the norm's summation
  // order follows the chunks, and it is reproducible for an input)
  sa.part_in = same && ws.ht_part_ready && !err_out ? ws.ht_part(seq) : nullptr;
  sa.prev_sums = same ? ws.ht_chunks(seq + 1) : nullptr;   // the other parity: seq - 1
  sa.prev_part = same && ws.ht_prev_balanced ? ws.ht_part(seq + 2) : nullptr;  // seq - 1
  sa.prev_epoch = ws.ht_last_epoch;
  sa.part_out = ws.ht_part(seq + 1);
  void* params[] = {&op, &d, &idx_out, &val_out, &count_out, &cap, &c, &sa};
  const cudaError_t err = launch_pdl(
      reinterpret_cast<const void*>(&stream_compact_kernel<HtOp<GT>, kHtStages<GT>>), grid,
      kStreamThreads, HtChunkKernel<GT>::kSmem, ws.stream, params, false);
  count_launch();
  ws.ht_prev_balanced = sa.part_in != nullptr;
  ws.ht_part_ready = err == cudaSuccess;
  ws.ht_last_tiles = tiles;
  ws.ht_last_grid = grid;
  ws.ht_last_epoch = c.epoch;
  ++ws.ht_seq;
  return err;
}

template <typename GT>
cudaError_t launch_typed(const GT* g, float* e, float gamma, float lambda, uint32_t d,
                         uint32_t* idx_out, float* val_out, uint32_t* count_out, double* err_out,
                         uint32_t* tiles_out, Workspace& ws, const DeviceInfo& dev) {
  const uint32_t tiles = tiles_for(d);
  const ScanCtx ctx = next_scan_ctx(ws, tiles);
  const uintptr_t ga = reinterpret_cast<uintptr_t>(g), ea = reinterpret_cast<uintptr_t>(e);
  if (ga % 16 == 0 && ea % 16 == 0) {
    const int per_group = sizeof(GT) == 4 ? dev.ht_group_per_sm_f32 : dev.ht_group_per_sm_bf16;
    const int per_dense = sizeof(GT) == 4 ? dev.ht_dense_per_sm_f32 : dev.ht_dense_per_sm_bf16;
    const int per_chunk = sizeof(GT) == 4 ? dev.ht_stream_per_sm_f32 : dev.ht_stream_per_sm_bf16;
    if (use_group_kernel(tiles)) {
      const int mode = stream_kernel_mode();
      const bool dense =
          mode == 3 || (mode == 0 && ws.density_host &&
                        *static_cast<volatile uint32_t*>(ws.density_host) >= kDenseRingHint);
      if (dense && per_dense > 0)
        return launch_groups<GT, kHtStages<GT> - 1>(g, e, gamma, lambda, d, idx_out, val_out,
                                                    count_out, err_out, tiles_out, ws, dev, ctx,
                                                    per_dense);
      if (per_group > 0)
        return launch_groups<GT, kHtStages<GT>>(g, e, gamma, lambda, d, idx_out, val_out,
                                                count_out, err_out, tiles_out, ws, dev, ctx,
                                                per_group);
    }
    if (per_chunk > 0)
      return launch_chunks(g, e, gamma, lambda, d, idx_out, val_out, count_out, err_out,
                           tiles_out, ws, dev, ctx, per_chunk);
  }
  const bool vec = (ga % (4 * sizeof(GT)) == 0) && (ea % 16 == 0);
  if (vec) {
    ht_kernel<GT, true><<<tiles, kThreads, 0, ws.stream>>>(g, e, gamma, lambda, d, idx_out,
                                                           val_out, count_out, ctx);
  } else {
    ht_kernel<GT, false><<<tiles, kThreads, 0, ws.stream>>>(g, e, gamma, lambda, d, idx_out,
                                                            val_out, count_out, ctx);
  }
  count_launch();
  cudaError_t err = cudaGetLastError();
  if (err == cudaSuccess && err_out) err = launch_error_norm(e, d, err_out, ws, dev);
  if (err == cudaSuccess && tiles_out) err = launch_list_tiles(idx_out, count_out, d, tiles_out, ws);
  return err;
}

template <typename GT, typename Layout>
int blocks_per_sm(const void* fn, int threads) {
  int n = 0;
  if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, Layout::kSmem) !=
          cudaSuccess ||
      cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, fn, threads, Layout::kSmem) != cudaSuccess)
    n = 0;
  cudaGetLastError();
  return n;
}

template <typename GT, int kStages>
int group_blocks_per_sm() {
  return blocks_per_sm<GT, HtGroupKernel<GT, kStages>>(
      reinterpret_cast<const void*>(&lookback_stream_kernel<HtOp<GT>, kStages>), kLbThreads);
}
template <typename GT>
int chunk_blocks_per_sm() {
  return blocks_per_sm<GT, HtChunkKernel<GT>>(
      reinterpret_cast<const void*>(&stream_compact_kernel<HtOp<GT>, kHtStages<GT>>),
      kStreamThreads);
}

}  // namespace

void ht_init_device(DeviceInfo& info) {
  info.ht_stream_per_sm_f32 = chunk_blocks_per_sm<float>();
  info.ht_stream_per_sm_bf16 = chunk_blocks_per_sm<uint16_t>();
  info.ht_group_per_sm_f32 = group_blocks_per_sm<float, kHtStages<float>>();
  info.ht_group_per_sm_bf16 = group_blocks_per_sm<uint16_t, kHtStages<uint16_t>>();
  info.ht_dense_per_sm_f32 = group_blocks_per_sm<float, kHtStages<float> - 1>();
  info.ht_dense_per_sm_bf16 = group_blocks_per_sm<uint16_t, kHtStages<uint16_t> - 1>();
}

// Launch the look-back kernel over caller-provided scratch (the tile-status
// words and the error word named by ctx); used by the allocation-free entry.
cudaError_t launch_hard_threshold_lookback(const float* g, float* e, float gamma, float lambda,
                                           uint32_t d, uint32_t* idx_out, float* val_out,
                                           uint32_t* count_out, const ScanCtx& ctx,
                                           cudaStream_t stream) {
  const uint32_t tiles = tiles_for(d);
  const bool vec = reinterpret_cast<uintptr_t>(g) % 16 == 0 &&
                   reinterpret_cast<uintptr_t>(e) % 16 == 0;
  if (vec)
    ht_kernel<float, true><<<tiles, kThreads, 0, stream>>>(g, e, gamma, lambda, d, idx_out,
                                                           val_out, count_out, ctx);
  else
    ht_kernel<float, false><<<tiles, kThreads, 0, stream>>>(g, e, gamma, lambda, d, idx_out,
                                                            val_out, count_out, ctx);
  count_launch();
  return cudaGetLastError();
}

cudaError_t launch_hard_threshold(const void* g, bool g_bf16, float* e, float gamma,
                                  float lambda, uint32_t d, uint32_t* idx_out, float* val_out,
                                  uint32_t* count_out, double* err_out, uint32_t* tiles_out,
                                  Workspace& ws, const DeviceInfo& dev) {
  if (g_bf16)
    return launch_typed(static_cast<const uint16_t*>(g), e, gamma, lambda, d, idx_out, val_out,
                        count_out, err_out, tiles_out, ws, dev);
  return launch_typed(static_cast<const float*>(g), e, gamma, lambda, d, idx_out, val_out,
                      count_out, err_out, tiles_out, ws, dev);
}

}  // namespace efs
