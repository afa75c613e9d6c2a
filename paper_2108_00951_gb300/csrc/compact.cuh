// compact.cuh — tile-level ordered stream compaction (step a4 of the hot
// path): turns each thread's selection bits into output positions with warp
// ballots and a block scan over warp totals, obtains the tile's global offset
// from the decoupled look-back, and writes the (index, value) pairs.
//
// Element layout of a tile (kTileElems = 4096): warp w owns the contiguous
// range [w*512, (w+1)*512); inside it, unit v of lane l covers the 4
// elements starting at v*128 + l*4. Every warp instruction therefore touches
// one contiguous 512-byte (fp32) span, and the output order — warp, then
// unit, then lane, then element — is ascending index order.
#pragma once

#include "common.cuh"

namespace efs {

__device__ __forceinline__ uint64_t element_index(uint32_t tile, int warp, int v, int lane, int j) {
  return static_cast<uint64_t>(tile) * kTileElems + warp * kWarpElems + v * 128 + lane * 4 + j;
}

// sel[v] bit j: element j of unit v is selected; a[v][j] is its value.
// All threads of the CTA must call this exactly once per tile.
// cap bounds every pair position (positions >= cap are never written and
// latch kDevErrOverflow); the last tile writes min(total, cap) to *count_out.
__device__ __forceinline__ void compact_tile(const ScanCtx& ctx, uint32_t tile,
                                             const uint32_t (&sel)[kUnits],
                                             const float (&a)[kUnits][4],
                                             uint32_t* __restrict__ idx_out,
                                             float* __restrict__ val_out,
                                             uint32_t* __restrict__ count_out, uint32_t cap) {
  __shared__ uint32_t s_warp_total[kWarps];
  __shared__ uint32_t s_excl;
  __shared__ int s_ok;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const uint32_t lt = lanemask_lt();

  // Position of each unit's first selected element within the warp's span.
  uint32_t unit_off[kUnits];
  uint32_t warp_total = 0;
#pragma unroll
  for (int v = 0; v < kUnits; ++v) {
    const uint32_t b0 = __ballot_sync(0xffffffffu, sel[v] & 1u);
    const uint32_t b1 = __ballot_sync(0xffffffffu, sel[v] & 2u);
    const uint32_t b2 = __ballot_sync(0xffffffffu, sel[v] & 4u);
    const uint32_t b3 = __ballot_sync(0xffffffffu, sel[v] & 8u);
    unit_off[v] = warp_total + __popc(b0 & lt) + __popc(b1 & lt) + __popc(b2 & lt) +
                  __popc(b3 & lt);
    warp_total += __popc(b0) + __popc(b1) + __popc(b2) + __popc(b3);
  }
  if (lane == 0) s_warp_total[warp] = warp_total;
  __syncthreads();

  uint32_t warp_excl = 0, tile_total = 0;
#pragma unroll
  for (int w = 0; w < kWarps; ++w) {
    const uint32_t c = s_warp_total[w];
    warp_excl += (w < warp) ? c : 0u;
    tile_total += c;
  }

  if (warp == 0) {
    uint32_t excl = 0;
    bool timed_out = false;
    if (tile == 0) {
      if (lane == 0) publish(ctx, tile, kFlagPrefix, tile_total);
    } else {
      if (lane == 0) publish(ctx, tile, kFlagAggregate, tile_total);
      excl = lookback_exclusive(ctx, tile, timed_out);
      if (lane == 0) publish(ctx, tile, kFlagPrefix, excl + tile_total);
    }
    if (lane == 0) {
      s_excl = excl;
      s_ok = timed_out ? 0 : 1;
      if (timed_out) atomicOr(ctx.error, kDevErrTimeout);
      if (tile == ctx.num_tiles - 1) {
        const uint32_t total = excl + tile_total;
        *count_out = total < cap ? total : cap;
      }
    }
  }
  __syncthreads();
  if (tile_total == 0 || !s_ok) return;

  const uint32_t base = s_excl + warp_excl;
  bool overflow = false;
#pragma unroll
  for (int v = 0; v < kUnits; ++v) {
    uint32_t pos = base + unit_off[v];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      if (sel[v] & (1u << j)) {
        if (pos < cap) {
          idx_out[pos] = static_cast<uint32_t>(element_index(tile, warp, v, lane, j));
          val_out[pos] = a[v][j];
        } else {
          overflow = true;
        }
        ++pos;
      }
    }
  }
  if (overflow) atomicOr(ctx.error, kDevErrOverflow);
}

}  // namespace efs
