// stream_compact.cuh — ordered stream compaction at memory speed: one
// launch of persistent CTAs (one per SM), TMA-fed tiles, warp-independent
// streaming of contiguous chunks, then pair placement.
//
// Why not a decoupled look-back, one tile per CTA: each CTA holds its tile
// while its look-back waits on L2 round trips that, under a saturated memory
// system, take microseconds; throughput is then resident-bytes / CTA
// lifetime, about a third of HBM bandwidth on this GPU. Resolving offsets
// inside the streaming loop of persistent CTAs instead couples every CTA to
// the slowest one, and even one CTA-wide barrier per tile puts each tile's
// latency chain on the refill path. So while streaming, nothing waits for
// anything but its own data.
//
// Phase 1 (streaming). CTA c owns the contiguous chunk of tiles
// [c*T/G, (c+1)*T/G) of kTileElems coordinates each. A producer warp fills a
// kStages-deep ring of shared-memory stages with bulk copies (cp.async.bulk,
// completing on the stage's "full" mbarrier) and refills a stage once all 16
// compute warps have released it (its "empty" mbarrier). Compute warp w owns
// the segment [w*256, (w+1)*256) of every tile: it computes the selection and
// its side effects (the residual store), compacts its selected (index, value)
// pairs with ballots into the segment's own staging slot, records the
// segment's count, and releases the stage. No CTA-wide barrier.
//
// Phase 2 (placement). Segments are ordered (tile, warp), which is coordinate
// order. Each CTA publishes its chunk's total (tagged with the launch's epoch),
// loads and scans its own segments' counts in shared memory, and then sums
// the totals of all earlier chunks in one batched load, waiting (bounded) for
// any not yet published; no grid-wide barrier is needed. Each warp then
// copies whole segments from staging to their final, ascending positions.
//
// Before its wait for the previous kernel on the stream (programmatic
// launch: the CTA becomes resident while that kernel's last CTAs place their
// pairs) a CTA pulls the first Op::kPrefetchTiles tiles of its chunk toward
// L2 with bulk prefetches.
//
// Error norm (when sa.err_out is set): a coordinate that is neither selected
// nor deferred (selection bits 4..7 of an op mark coordinates whose residual
// a later kernel decides) keeps a as its residual, so a^2 is its share of
// ||e'||^2. Each warp sums the squares of a tile segment in fp32 (fmaf per
// lane over its 8 coordinates, then a warp tree) and adds that in
// float-float (common.cuh); the CTA's share is published with its chunk
// total, and the last CTA adds the shares in a fixed order.
//
// Traffic beyond the step itself: 16 bytes per selected pair (staging write
// and read) plus 4 bytes per segment. Every wait (stage arrival, stage
// release, an earlier chunk's total) is bounded and latches kDevErrTimeout;
// after a timeout the CTA places no pair.
//
// An Op supplies the per-segment work:
//   static constexpr uint32_t kStageBytes;            bytes of one stage
//   void fill(unsigned char* stage, uint32_t tile, uint64_t* bar, uint64_t pol)
//        issue the bulk copies of a full tile (after expect_tx)
//   void tile_smem(const unsigned char* stage, uint32_t tile, int warp, int lane,
//                  float (&a)[kSUnits][4], uint32_t (&sel)[kSUnits])
//   void tile_global(uint32_t tile, int warp, int lane, float (&a)[..], uint32_t (&sel)[..])
//        compute values and selection bits (and side effects) of the calling
//        warp's segment, from the stage of a full tile, or from global memory
//        for the partial last tile.
//   (tile_smem and tile_global also receive `aux`, from
//   uint64_t initial_aux()  (all threads, after the wait for the previous
//   kernel; uniform))
//   void prologue()                     every thread, once, at the start
//   static constexpr uint32_t kPrefetchTiles;  tiles of the chunk pulled toward
//   void prefetch(uint32_t tile)               L2 before the wait for the previous kernel
//   static constexpr bool kKeepPairs;  the pairs are written with the L2
//                                      evict-last policy (a later kernel of the call reads them)
// Element layout: unit v of lane l of warp w covers the 4 coordinates from
// tile * kTileElems + w * 256 + v * 128 + l * 4 (see stream_element_index).
#pragma once

#include "compact.cuh"
#include "tma.cuh"

namespace efs {

constexpr int kSWarps = 16;                          // compute warps (segments per tile)
constexpr int kSUnits = 2;                           // 4-coordinate units per lane per segment
constexpr int kSWarpElems = 32 * 4 * kSUnits;        // 256 coordinates per segment
static_assert(kSWarps * kSWarpElems == kTileElems, "tile geometry");
constexpr int kComputeThreads = 32 * kSWarps;        // 512
constexpr int kStreamThreads = kComputeThreads + 32; // + 1 producer warp
constexpr int kProducerWarp = kSWarps;

__device__ __forceinline__ uint64_t stream_element_index(uint32_t tile, int warp, int v, int lane,
                                                        int j) {
  return static_cast<uint64_t>(tile) * kTileElems + warp * kSWarpElems + v * 128 + lane * 4 + j;
}

// Workspace pieces of a launch.
struct StreamArgs {
  uint32_t* stage_idx;   // [num_tiles * kTileElems] staged indices, segment-slotted
  float* stage_val;      // [num_tiles * kTileElems] staged values
  uint32_t* counts;      // [num_tiles * kSWarps] selected per segment
  uint64_t* chunk_sums;  // [gridDim.x] (epoch << 32) | chunk total
  uint32_t* tile_base;   // optional [num_tiles + 1]: output position of each tile's first
                         // pair, and the total (untruncated), or null
  double* err_out;       // optional: sum of a^2 over the coordinates whose residual is final
                         // here (not selected, not deferred), or null
  FF* err_parts;         // [gridDim.x] the CTAs' shares of it
  // Chunk boundaries (all optional; null: equal chunks of tiles):
  const uint32_t* part_in;    // [gridDim.x + 1] this launch's boundaries (tiles)
  const uint64_t* prev_sums;  // the previous launch's chunk totals, (epoch << 32) | total
  const uint32_t* prev_part;  // the previous launch's boundaries (null: equal chunks)
  uint32_t prev_epoch;        // the previous launch's epoch
  uint32_t* part_out;         // [gridDim.x + 1] boundaries computed for the next launch
};

// Weight of a chunk when the next launch's chunks are balanced: a coordinate
// counts 2, a selected pair 5 (a staged pair costs about two and a half
// coordinates of a CTA's time, staging and placement together; 3 and 8 were
// measured slower on dense vectors).
constexpr uint64_t kBalCoord = 2, kBalPair = 5;

// The next launch's left boundary of chunk c, from the previous launch's
// chunk totals and boundaries, by lanes 1..31 of one warp (lane 0 is busy
// elsewhere). The chunks' weights are summed, the target c/G of the total
// is located in one chunk, and the boundary is interpolated inside it
// (uniform density within a chunk). Monotone in c for any inputs, so the
// boundaries always partition the tiles. Equal chunks when the previous
// totals are missing or from another launch.
__device__ __forceinline__ static uint32_t next_chunk_boundary(const StreamArgs& sa, uint32_t c, uint32_t G, uint32_t T,
                                        int lane) {
  constexpr uint32_t kMask = 0xfffffffeu;
  const uint32_t eq = static_cast<uint32_t>(static_cast<uint64_t>(c) * T / G);
  if (!sa.prev_sums || c == 0) return c == 0 ? 0u : eq;
  const uint32_t L = lane - 1;  // 0..30
  const uint32_t qa = static_cast<uint32_t>(static_cast<uint64_t>(L) * G / 31);
  const uint32_t qb = static_cast<uint32_t>(static_cast<uint64_t>(L + 1) * G / 31);
  auto bounds = [&](uint32_t q, uint32_t& lo, uint32_t& hi) {
    if (sa.prev_part) {
      lo = min(__ldcg(sa.prev_part + q), T);
      hi = min(max(__ldcg(sa.prev_part + q + 1), lo), T);
    } else {
      lo = static_cast<uint32_t>(static_cast<uint64_t>(q) * T / G);
      hi = static_cast<uint32_t>(static_cast<uint64_t>(q + 1) * T / G);
    }
  };
  uint64_t mine = 0;
  bool ok = true;
  for (uint32_t q = qa; q < qb; ++q) {
    const uint64_t w = __ldcg(sa.prev_sums + q);
    uint32_t lo, hi;
    bounds(q, lo, hi);
    if (static_cast<uint32_t>(w >> 32) != sa.prev_epoch) ok = false;
    mine += kBalCoord * kTileElems * (hi - lo) + kBalPair * static_cast<uint32_t>(w);
  }
  if (__any_sync(kMask, !ok)) return eq;
  uint64_t incl = mine;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint64_t v = __shfl_up_sync(kMask, incl, o);
    if (static_cast<int>(L) >= o) incl += v;
  }
  const uint64_t total = __shfl_sync(kMask, incl, 31);
  const uint64_t target = total / G * c + total % G * c / G;  // floor(total * c / G)
  const uint64_t excl = incl - mine;
  uint32_t b = 0;
  bool here = target >= excl && target < incl;
  if (here) {
    uint64_t acc = excl;
    for (uint32_t q = qa; q < qb; ++q) {
      const uint64_t w = __ldcg(sa.prev_sums + q);
      uint32_t lo, hi;
      bounds(q, lo, hi);
      const uint64_t wq = kBalCoord * kTileElems * (hi - lo) + kBalPair * static_cast<uint32_t>(w);
      if (acc + wq > target) {
        b = lo + static_cast<uint32_t>((target - acc) * (hi - lo) / wq);
        break;
      }
      acc += wq;
    }
  }
  const uint32_t who = __ballot_sync(kMask, here);
  if (!who) return eq;
  return min(__shfl_sync(kMask, b, __ffs(who) - 1), T);
}

// A segment's count (<= 256: 9 bits) and its warp's earlier pairs in the
// chunk, saturated to 23 bits, in one word.
__device__ __forceinline__ uint32_t pack_count(uint32_t before, uint32_t count) {
  return (before < (1u << 23) ? before : (1u << 23) - 1u) << 9 | count;
}

template <class Op, int kStages>
struct StreamLayout {
  static constexpr uint32_t kRing = kStages * Op::kStageBytes;
  // each compute warp stages its first kWarpPairs pairs on chip, the rest in
  // the global staging slots
  static constexpr uint32_t kWarpPairs = Op::kWarpStagePairs;
  static constexpr uint32_t kStaging = kSWarps * kWarpPairs * 8;
  static constexpr uint32_t kSmem = kRing + kStaging;  // dynamic shared memory
  // phase 2 reuses the ring: per segment of a window, its output offset and
  // its warp's count of earlier pairs in the chunk
  static constexpr uint32_t kChunkSegs = kRing / 8;
  static_assert(kChunkSegs % kSWarps == 0, "whole tiles per window");
};

template <class Op, int kStages>
__global__ void __launch_bounds__(kStreamThreads, 1)
    stream_compact_kernel(Op op, uint32_t d, uint32_t* __restrict__ idx_out,
                          float* __restrict__ val_out, uint32_t* __restrict__ count_out,
                          uint32_t cap, ScanCtx ctx, StreamArgs sa) {
  extern __shared__ __align__(128) unsigned char smem[];
  __shared__ __align__(8) uint64_t s_full[kStages];
  __shared__ __align__(8) uint64_t s_empty[kStages];
  __shared__ uint32_t s_scratch[kStreamThreads / 32];
  __shared__ FF s_err[kSWarps];
  __shared__ FF s_err_sum[32];
  using L = StreamLayout<Op, kStages>;
  uint32_t* s_pair_idx = reinterpret_cast<uint32_t*>(smem + L::kRing);
  float* s_pair_val = reinterpret_cast<float*>(smem + L::kRing + kSWarps * L::kWarpPairs * 4);

  const uint32_t T = ctx.num_tiles, G = gridDim.x, c = blockIdx.x;
  // the chunk: written boundaries (by the previous launch, before it let this
  // one start), else equal chunks
  uint32_t t_lo = static_cast<uint32_t>(static_cast<uint64_t>(c) * T / G);
  uint32_t t_hi = static_cast<uint32_t>(static_cast<uint64_t>(c + 1) * T / G);
  if (sa.part_in) {
    t_lo = min(__ldcg(sa.part_in + c), T);
    t_hi = min(max(__ldcg(sa.part_in + c + 1), t_lo), T);
  }
  const uint32_t rounds = t_hi - t_lo;
  const uint32_t full_tiles = d / kTileElems;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&s_full[s], 1);
      mbar_init(&s_empty[s], kSWarps);
    }
    mbar_init_fence();
  }
  __syncthreads();
  // A dependent launch starts while the previous kernel's last CTAs place
  // their pairs, a phase that leaves DRAM mostly idle: pull the chunk's first
  // tiles toward L2 meanwhile. A prefetch is not a read of the data: L2 is the
  // point of coherence, so the previous kernel's writes still land before the
  // bulk copies below read these lines.
  if (threadIdx.x == 0)
    for (uint32_t r = 0; r < rounds && r < Op::kPrefetchTiles; ++r)
      if (t_lo + r < full_tiles) op.prefetch(t_lo + r);
  // everything the previous kernels on the stream wrote is read only after this
  griddep_wait();
  op.prologue();

  // ------------------------------------------------------------- phase 1
  bool failed = false;    // a wait of this thread ran out
  bool withheld = false;  // test hook: this CTA owns the withheld tile
  uint32_t chunk_total = 0;  // compute warps: pairs selected by this warp
  FF warp_err{0.0f, 0.0f};   // compute warps: their share of ||e'||^2
  uint64_t policy = 0;       // producer lane
  auto fill = [&](uint32_t r) {  // producer lane
    const int s = static_cast<int>(r % kStages);
    const uint32_t t = t_lo + r;
    if (t < full_tiles) {
      mbar_arrive_expect_tx(&s_full[s], Op::kStageBytes);
      op.fill(smem + s * Op::kStageBytes, t, &s_full[s], policy);
    } else {
      mbar_arrive(&s_full[s]);  // the partial last tile is read from global memory
    }
  };
  const bool producer = warp == kProducerWarp && lane == 0;
  if (producer) {
    policy = l2_evict_normal_policy();
    for (uint32_t r = 0; r < rounds && r < static_cast<uint32_t>(kStages); ++r) fill(r);
  }

  const uint64_t aux = op.initial_aux();  // uniform

  if (warp == kProducerWarp) {
    if (lane != 0) {
      // lanes 1..31: the next launch's boundary of this chunk, while lane 0
      // keeps the ring filled; visible before this launch lets the next start
      if (sa.part_out) {
        const uint32_t b = next_chunk_boundary(sa, c, G, T, lane);
        if (lane == 1) {
          sa.part_out[c] = b;
          if (c == G - 1) sa.part_out[G] = T;
          __threadfence();
        }
      }
    } else {
      uint32_t r = rounds < static_cast<uint32_t>(kStages) ? rounds : kStages;
      for (; r < rounds; ++r) {
        const int s = static_cast<int>(r % kStages);
        const uint32_t k = r / kStages;
        // wait for the 16 compute warps to release this stage's previous use
        if (!mbar_wait(&s_empty[s], (k - 1) & 1u, ctx.wait_limit_ns)) {
          failed = true;
          break;
        }
        fill(r);
      }
      // no copy may land after the CTA exits: wait for the last fill of
      // every stage (a completed phase reports complete immediately)
      for (uint32_t q = r > kStages ? r - kStages : 0; q < r; ++q)
        if (!mbar_wait(&s_full[q % kStages], (q / kStages) & 1u, ctx.wait_limit_ns))
          failed = true;
    }
  } else {
    const uint32_t lt = lanemask_lt();
    for (uint32_t r = 0; r < rounds; ++r) {
      const int s = static_cast<int>(r % kStages);
      const uint32_t t = t_lo + r;
      const bool arrived = mbar_wait(&s_full[s], (r / kStages) & 1u, ctx.wait_limit_ns);
      if (!__all_sync(0xffffffffu, arrived)) {  // stop at the first failed wait
        failed = true;
        break;
      }
      float a[kSUnits][4];
      uint32_t sel[kSUnits];
      if (t < full_tiles) {
        op.tile_smem(smem + s * Op::kStageBytes, t, warp, lane, a, sel, aux);
      } else {
        op.tile_global(t, warp, lane, a, sel, aux);
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&s_empty[s]);  // this warp is done with the stage
      if (sa.err_out) {
        float sq = 0.0f;
#pragma unroll
        for (int v = 0; v < kSUnits; ++v)
#pragma unroll
          for (int j = 0; j < 4; ++j)
            if (!((sel[v] >> j) & 0x11u)) sq = __fmaf_rn(a[v][j], a[v][j], sq);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
        if (lane == 0) warp_err = ff_add(warp_err, FF{sq, 0.0f});
      }
      uint32_t off[kSUnits];
      uint32_t total = 0;
#pragma unroll
      for (int v = 0; v < kSUnits; ++v) {
        const uint32_t b0 = __ballot_sync(0xffffffffu, sel[v] & 1u);
        const uint32_t b1 = __ballot_sync(0xffffffffu, sel[v] & 2u);
        const uint32_t b2 = __ballot_sync(0xffffffffu, sel[v] & 4u);
        const uint32_t b3 = __ballot_sync(0xffffffffu, sel[v] & 8u);
        off[v] = total + __popc(b0 & lt) + __popc(b1 & lt) + __popc(b2 & lt) + __popc(b3 & lt);
        total += __popc(b0) + __popc(b1) + __popc(b2) + __popc(b3);
      }
      const size_t seg = static_cast<size_t>(t) * kSWarps + warp;
      const uint32_t before = chunk_total;  // this warp's earlier pairs in the chunk
      chunk_total += total;
      // the count with the warp's earlier pairs (saturated: only <= the
      // on-chip share matters), which tells phase 2 where the pairs are
      if (lane == 0) sa.counts[seg] = pack_count(before, total);
      if (total) {
        // on chip while the warp's pairs fit, else the segment's global slot
        const bool on_chip = chunk_total <= L::kWarpPairs;
        uint32_t* sidx = on_chip ? s_pair_idx + warp * L::kWarpPairs + before
                                 : sa.stage_idx + seg * kSWarpElems;
        float* sval = on_chip ? s_pair_val + warp * L::kWarpPairs + before
                              : sa.stage_val + seg * kSWarpElems;
#pragma unroll
        for (int v = 0; v < kSUnits; ++v) {
          uint32_t pos = off[v];
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            if (sel[v] & (1u << j)) {
              sidx[pos] = static_cast<uint32_t>(stream_element_index(t, warp, v, lane, j));
              sval[pos] = a[v][j];
              ++pos;
            }
          }
        }
      }
      if (static_cast<int64_t>(t) == ctx.withheld_tile) withheld = true;
    }
  }
  if (__syncthreads_or(failed)) {
    if (threadIdx.x == 0) atomicOr(ctx.error, kDevErrTimeout);
    return;
  }
  // A CTA that owns the withheld tile never arrives: the others' barrier
  // waits run out (the failure-detection test).
  if (__syncthreads_or(withheld)) return;
  griddep_launch_dependents();  // streaming is done: the next kernel may be scheduled

  // ------------------------------------------------------------- phase 2
  const uint64_t keep_policy = Op::kKeepPairs ? l2_evict_last_policy() : 0ull;
  // the chunk's total (each compute warp contributes its own)
  uint32_t mine = lane == 0 && warp < kSWarps ? chunk_total : 0u;
  if (lane == 0) s_scratch[warp] = mine;
  if (lane == 0 && warp < kSWarps) s_err[warp] = warp_err;
  __syncthreads();
  if (threadIdx.x == 0) {
    uint32_t sum = 0;
    for (int w = 0; w < kSWarps; ++w) sum += s_scratch[w];
    if (sa.err_out) {  // the CTA's share of ||e'||^2, visible before the chunk total
      FF err{0.0f, 0.0f};
      for (int w = 0; w < kSWarps; ++w) err = ff_add(err, s_err[w]);
      sa.err_parts[c] = err;
      __threadfence();
    }
    st_relaxed_u64(sa.chunk_sums + c, (static_cast<uint64_t>(ctx.epoch) << 32) | sum);
  }
  // The chunk's segments, a window at a time (the ring is free now): their
  // counts and their warps' earlier pairs (coalesced loads; a segment was
  // staged on chip iff the two add up to at most the warp's share), an
  // exclusive scan of the counts into offsets within the window, then, once
  // the chunk's base is known, the copy. The first window is prepared before
  // the wait for the earlier chunks' totals, which hides its loads.
  const uint32_t lo = t_lo * kSWarps, hi = t_hi * kSWarps;
  uint32_t* seg_off = reinterpret_cast<uint32_t*>(smem);
  uint32_t* seg_pos = seg_off + L::kChunkSegs;  // the warp's earlier pairs
  constexpr int kNumWarps = kStreamThreads / 32;
  constexpr int kCopySegs = 8;
  // per thread: its contiguous run [rb, re) of the window, the run's offset
  // within the window, and the window's total
  uint32_t rb = 0, re = 0, run_off = 0, window_total = 0;
  auto prepare = [&](uint32_t w0, uint32_t n) {
    __syncthreads();  // the previous window's copy is done with the arrays
    for (uint32_t i = threadIdx.x; i < n; i += kStreamThreads) {
      const uint32_t packed = __ldcg(sa.counts + w0 + i);
      seg_off[i] = packed & 0x1ffu;
      seg_pos[i] = packed >> 9;
    }
    __syncthreads();
    const uint32_t per = (n + kStreamThreads - 1) / kStreamThreads;
    rb = threadIdx.x * per < n ? threadIdx.x * per : n;
    re = rb + per < n ? rb + per : n;
    uint32_t run = 0;
    for (uint32_t i = rb; i < re; ++i) {
      const uint32_t cnt = seg_off[i];
      seg_off[i] = run;
      run += cnt;
    }
    uint32_t incl = run;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t v = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += v;
    }
    if (lane == 31) s_scratch[warp] = incl;
    __syncthreads();
    uint32_t warp_base = 0, total = 0;
    for (int w = 0; w < kNumWarps; ++w) {
      const uint32_t x = s_scratch[w];
      warp_base += w < warp ? x : 0u;
      total += x;
    }
    run_off = warp_base + incl - run;
    window_total = total;
  };
  prepare(lo, hi - lo < L::kChunkSegs ? hi - lo : L::kChunkSegs);

  // sum of the earlier chunks' totals, waiting (bounded) for missing ones
  uint32_t base = 0;
  {
    const uint64_t t0 = global_timer_ns();
    uint32_t it = 0;
    bool done = false;
    while (!done) {
      uint32_t part = 0;
      bool present = true;
      for (uint32_t q = threadIdx.x; q < c; q += kStreamThreads) {
        const uint64_t w = ld_relaxed_u64(sa.chunk_sums + q);
        if (static_cast<uint32_t>(w >> 32) == ctx.epoch)
          part += static_cast<uint32_t>(w);
        else
          present = false;
      }
      part = warp_sum(part);
      __syncthreads();
      if (lane == 0) s_scratch[warp] = part;
      const bool all_present = __syncthreads_and(present);
      if (all_present) {
        for (int w = 0; w < kStreamThreads / 32; ++w) base += s_scratch[w];
        done = true;
        if (sa.err_out && c == G - 1) {
          // every earlier CTA's share was written before its chunk total
          __threadfence();
          __syncthreads();
          const FF err = sum_parts_ff(sa.err_parts, G, s_err_sum);
          if (threadIdx.x == 0) *sa.err_out = ff_to_double(err);
        }
      } else {
        const uint64_t now = global_timer_ns();
        const bool out_of_time = ++it > (1u << 26) || now - t0 > ctx.wait_limit_ns;
        if (__syncthreads_or(out_of_time)) {
          if (threadIdx.x == 0) atomicOr(ctx.error, kDevErrTimeout);
          return;
        }
        __nanosleep(64);
      }
    }
  }
  bool overflow = false;
  for (uint32_t w0 = lo; w0 < hi; w0 += L::kChunkSegs) {
    const uint32_t n = hi - w0 < L::kChunkSegs ? hi - w0 : L::kChunkSegs;
    if (w0 != lo) prepare(w0, n);
    const uint32_t thread_base = base + run_off;
    for (uint32_t i = rb; i < re; ++i) {
      seg_off[i] += thread_base;
      // windows start at whole tiles, so a tile's first segment has i % kSWarps == 0
      if (sa.tile_base && i % kSWarps == 0) sa.tile_base[(w0 + i) / kSWarps] = seg_off[i];
    }
    __syncthreads();
    const uint32_t window_end = base + window_total;
    // each warp copies kCopySegs adjacent segments at once, all of their
    // loads (shared memory for segments staged on chip) before the stores
    for (uint32_t i0 = warp * kCopySegs; i0 < n; i0 += kNumWarps * kCopySegs) {
      uint32_t dst[kCopySegs], cnt[kCopySegs], maxc = 0;
      const uint32_t* src_i[kCopySegs];
      const float* src_v[kCopySegs];
#pragma unroll
      for (int u = 0; u < kCopySegs; ++u) {
        const uint32_t i = i0 + u;
        dst[u] = i < n ? seg_off[i] : 0u;
        const uint32_t next = i + 1 < n ? seg_off[i + 1] : window_end;
        cnt[u] = i < n ? next - dst[u] : 0u;
        maxc = cnt[u] > maxc ? cnt[u] : maxc;
        const uint32_t pos = i < n ? seg_pos[i] : 0u;
        if (pos + cnt[u] <= L::kWarpPairs) {
          const uint32_t w = i % kSWarps;  // the segment's warp
          src_i[u] = s_pair_idx + w * L::kWarpPairs + pos;
          src_v[u] = s_pair_val + w * L::kWarpPairs + pos;
        } else {
          src_i[u] = sa.stage_idx + static_cast<size_t>(w0 + i) * kSWarpElems;
          src_v[u] = sa.stage_val + static_cast<size_t>(w0 + i) * kSWarpElems;
        }
      }
      for (uint32_t p0 = 0; p0 < maxc; p0 += 32) {
        uint32_t xi[kCopySegs];
        float xv[kCopySegs];
#pragma unroll
        for (int u = 0; u < kCopySegs; ++u) {
          if (p0 + lane < cnt[u]) {
            xi[u] = src_i[u][p0 + lane];
            xv[u] = src_v[u][p0 + lane];
          }
        }
#pragma unroll
        for (int u = 0; u < kCopySegs; ++u) {
          if (p0 + lane < cnt[u]) {
            const uint32_t q = dst[u] + p0 + lane;
            if (q < cap) {
              if constexpr (Op::kKeepPairs) {
                st_pair_policy(idx_out + q, val_out + q, xi[u], xv[u], keep_policy);
              } else {
                idx_out[q] = xi[u];
                val_out[q] = xv[u];
              }
            } else {
              overflow = true;
            }
          }
        }
      }
    }
    base = window_end;
  }
  if (hi == T * kSWarps && threadIdx.x == 0) {
    *count_out = base < cap ? base : cap;
    if (sa.tile_base) sa.tile_base[T] = base;
  }
  if (__syncthreads_or(overflow) && threadIdx.x == 0) atomicOr(ctx.error, kDevErrOverflow);
}

}  // namespace efs
