// stream_compact.cuh — single-pass ordered stream compaction at memory speed:
// persistent co-resident CTAs, TMA-fed tiles, and a chained per-CTA scan.
//
// Why not a plain decoupled look-back with one tile per CTA: every CTA would
// hold its tile in registers while its look-back waits on L2 round trips that,
// under a saturated memory system, take microseconds; throughput is then
// resident-bytes / CTA lifetime, about a third of HBM bandwidth on this GPU.
//
// Design (one cooperative launch, grid G = all co-resident CTAs):
//  * Tiles of kTileElems coordinates are assigned round-robin: CTA c owns
//    tiles c, c + G, c + 2G, ...
//  * 8 compute warps stream the CTA's tiles through a kStages-deep ring of
//    shared-memory stages filled by bulk copies (cp.async.bulk + mbarrier).
//    Per tile they compute the selection, publish the tile's count, and stage
//    the selected (index, value) pairs, in order, in a shared-memory pair ring.
//  * One scan warp per CTA turns the staged tiles into output: the first
//    selected coordinate of tile t lands at
//        offset(t) = incl(t - G) + sum_{t - G < u < t} count(u),
//    where incl(t - G) is this same CTA's previous tile's inclusive count (its
//    own running total) and the counts in between are the other CTAs'
//    published tile counts; for the CTA's first tile it is the sum of all
//    counts before it. It never needs another CTA's inclusive prefix, so no
//    prefix has to propagate across CTAs and the compute warps never wait on
//    L2 round trips. It then copies the staged pairs to their final positions
//    with coalesced stores.
//  * Counts are published in the tile-status array tagged with the launch's
//    epoch. Every wait (stage arrival, ring space, a missing count) is bounded
//    and latches kDevErrTimeout; after a timeout both roles leave their loops,
//    the copies still in flight get a bounded wait, and the kernel returns.
//
// An Op supplies the per-tile work:
//   static constexpr uint32_t kStageBytes;            bytes of one stage
//   void fill(unsigned char* stage, uint32_t tile, uint64_t* bar, uint64_t pol)
//        issue the bulk copies of a full tile (thread 0; after expect_tx)
//   void tile_smem(const unsigned char* stage, uint32_t tile, int warp, int lane,
//                  float (&a)[kUnits][4], uint32_t (&sel)[kUnits])
//   void tile_global(uint32_t tile, int warp, int lane, float (&a)[..], uint32_t (&sel)[..])
//        compute values and selection bits (and side effects such as the
//        residual store) for a full tile from its stage, or for the partial
//        last tile from global memory.
#pragma once

#include "compact.cuh"
#include "tma.cuh"

namespace efs {

constexpr int kComputeThreads = kThreads;              // 8 compute warps
constexpr int kStreamThreads = kComputeThreads + 32;   // + 1 scan warp
constexpr uint32_t kPairRing = kTileElems;             // staged pairs (>= 1 full tile)
constexpr uint32_t kEntryRing = 32;                    // staged tiles
constexpr int kScanBatch = 4;                          // rounds resolved per batch
constexpr int kScanWordsPerLane = 10;                  // counts per round per lane
// The scan warp reads at most 32 * kScanWordsPerLane counts per round, i.e.
// the G - 1 tiles between two of its own: launchers must keep G <= this.
constexpr uint32_t kMaxStreamGrid = 32u * kScanWordsPerLane + 1u;

template <class Op, int kStages>
struct StreamLayout {
  static constexpr uint32_t kRingOff = kStages * Op::kStageBytes;
  static constexpr uint32_t kSmem = kRingOff + kPairRing * 8;
};

template <class Op, int kStages>
__global__ void __launch_bounds__(kStreamThreads, 1)
    stream_compact_kernel(Op op, uint32_t d, uint32_t* __restrict__ idx_out,
                          float* __restrict__ val_out, uint32_t* __restrict__ count_out,
                          uint32_t cap, ScanCtx ctx) {
  extern __shared__ __align__(128) unsigned char smem[];
  __shared__ __align__(8) uint64_t s_full[kStages];
  __shared__ uint32_t s_warp_total[kWarps];
  __shared__ uint32_t s_ring_start;
  __shared__ uint32_t s_entry_count[kEntryRing];
  __shared__ uint32_t s_entry_start[kEntryRing];
  __shared__ volatile uint32_t s_produced;  // tiles staged by the compute warps
  __shared__ volatile uint32_t s_consumed;  // tiles written out by the scan warp
  __shared__ volatile uint32_t s_tail;      // pair-ring slots released
  __shared__ volatile int s_abort;
  using L = StreamLayout<Op, kStages>;
  uint32_t* ring_idx = reinterpret_cast<uint32_t*>(smem + L::kRingOff);
  float* ring_val = reinterpret_cast<float*>(smem + L::kRingOff + kPairRing * 4);

  const uint32_t T = ctx.num_tiles, G = gridDim.x, c = blockIdx.x;
  const uint32_t rounds = c < T ? (T - c + G - 1) / G : 0;
  const uint32_t full_tiles = d / kTileElems;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) mbar_init(&s_full[s], 1);
    mbar_init_fence();
    s_produced = 0;
    s_consumed = 0;
    s_tail = 0;
    s_abort = 0;
  }
  __syncthreads();

  if (threadIdx.x < kComputeThreads) {
    // ------------------------------------------------------ compute warps
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const uint32_t lt = lanemask_lt();
    uint64_t policy = 0;
    uint32_t issued = 0;  // thread 0: rounds whose stage fill was issued
    uint32_t head = 0;    // thread 0: pair-ring slots reserved
    auto fill = [&](uint32_t r) {
      const int s = static_cast<int>(r % kStages);
      const uint32_t t = c + r * G;
      if (t < full_tiles) {
        mbar_arrive_expect_tx(&s_full[s], Op::kStageBytes);
        op.fill(smem + s * Op::kStageBytes, t, &s_full[s], policy);
      } else {
        mbar_arrive(&s_full[s]);  // the partial last tile is read from global memory
      }
      issued = r + 1;
    };
    if (threadIdx.x == 0) {
      policy = l2_evict_first_policy();
      for (uint32_t r = 0; r < rounds && r < static_cast<uint32_t>(kStages); ++r) fill(r);
    }
    for (uint32_t r = 0; r < rounds; ++r) {
      const int s = static_cast<int>(r % kStages);
      const bool arrived = mbar_wait(&s_full[s], (r / kStages) & 1u, ctx.wait_limit_ns);
      if (group_bar_or(kComputeThreads, !arrived || s_abort)) {
        if (threadIdx.x == 0) {
          if (!arrived) atomicOr(ctx.error, kDevErrTimeout);
          s_abort = 1;
          for (uint32_t q = r; q < issued; ++q)  // let copies in flight land
            mbar_wait(&s_full[q % kStages], (q / kStages) & 1u, ctx.wait_limit_ns);
        }
        break;
      }
      const uint32_t t = c + r * G;
      float a[kUnits][4];
      uint32_t sel[kUnits];
      if (t < full_tiles)
        op.tile_smem(smem + s * Op::kStageBytes, t, warp, lane, a, sel);
      else
        op.tile_global(t, warp, lane, a, sel);

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
      group_bar(kComputeThreads);
      uint32_t warp_excl = 0, tile_total = 0;
#pragma unroll
      for (int w = 0; w < kWarps; ++w) {
        const uint32_t cw = s_warp_total[w];
        warp_excl += (w < warp) ? cw : 0u;
        tile_total += cw;
      }
      if (threadIdx.x == 0) {
        publish(ctx, t, kFlagAggregate, tile_total);
        // room for this tile's pairs and a free entry slot (bounded wait)
        const uint64_t t0 = global_timer_ns();
        uint32_t it = 0;
        while ((head - s_tail) + tile_total > kPairRing || r >= s_consumed + kEntryRing) {
          if (s_abort || ++it > (1u << 26) || global_timer_ns() - t0 > ctx.wait_limit_ns) {
            if (!s_abort) atomicOr(ctx.error, kDevErrTimeout);
            s_abort = 1;
            break;
          }
          __nanosleep(64);
        }
        __threadfence_block();
        s_ring_start = head;
        head += tile_total;
      }
      const bool abort_now = group_bar_or(kComputeThreads, s_abort != 0);
      if (abort_now) {
        if (threadIdx.x == 0)
          for (uint32_t q = r + 1; q < issued; ++q)
            mbar_wait(&s_full[q % kStages], (q / kStages) & 1u, ctx.wait_limit_ns);
        break;
      }
      if (tile_total) {
        const uint32_t base = s_ring_start + warp_excl;
#pragma unroll
        for (int v = 0; v < kUnits; ++v) {
          uint32_t pos = base + unit_off[v];
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            if (sel[v] & (1u << j)) {
              const uint32_t slot = pos % kPairRing;
              ring_idx[slot] = static_cast<uint32_t>(element_index(t, warp, v, lane, j));
              ring_val[slot] = a[v][j];
              ++pos;
            }
          }
        }
      }
      group_bar(kComputeThreads);  // pairs staged; stage s fully read
      if (threadIdx.x == 0) {
        s_entry_count[r % kEntryRing] = tile_total;
        s_entry_start[r % kEntryRing] = s_ring_start;
        __threadfence_block();
        s_produced = r + 1;
        if (r + kStages < rounds) fill(r + kStages);
      }
    }
  } else {
    // ------------------------------------------------------------ scan warp
    // Resolves staged tiles in order. The published counts it needs for up to
    // kScanBatch staged rounds are loaded into registers together (one L2
    // round trip per batch, not one per word), then the rounds are resolved
    // in order as far as their counts are present.
    const int lane = threadIdx.x & 31;
    uint32_t incl = 0;  // this CTA's running inclusive count
    uint32_t tail = 0;
    bool overflow = false;
    uint32_t r = 0;
    uint64_t last_progress = __shfl_sync(0xffffffffu, global_timer_ns(), 0);
    uint32_t idle_iters = 0;
    while (r < rounds) {
      const uint32_t produced = __shfl_sync(0xffffffffu, s_produced, 0);
      const int aborted = __shfl_sync(0xffffffffu, s_abort, 0);
      if (aborted) break;
      uint32_t done = 0;
      if (produced > r) {
        __threadfence_block();
        const uint32_t batch = produced - r < kScanBatch ? produced - r : kScanBatch;
        uint64_t w[kScanBatch][kScanWordsPerLane];
#pragma unroll
        for (int b = 0; b < kScanBatch; ++b) {
          const uint32_t q = r + b;
          const uint32_t t = c + q * G;
          const uint32_t lo = q == 0 ? 0u : t - G + 1;
#pragma unroll
          for (int k = 0; k < kScanWordsPerLane; ++k) {
            const uint32_t u = lo + lane + 32u * k;
            w[b][k] = (static_cast<uint32_t>(b) < batch && u < t) ? ld_relaxed_u64(ctx.status + u)
                                                                 : (uint64_t(ctx.epoch) << 34);
          }
        }
#pragma unroll
        for (int b = 0; b < kScanBatch; ++b) {
          if (static_cast<uint32_t>(b) >= batch || done != static_cast<uint32_t>(b)) break;
          uint32_t sum = 0;
          bool ready = true;
#pragma unroll
          for (int k = 0; k < kScanWordsPerLane; ++k) {
            if (static_cast<uint32_t>(w[b][k] >> 34) == ctx.epoch)
              sum += static_cast<uint32_t>(w[b][k]);
            else
              ready = false;
          }
          if (!__all_sync(0xffffffffu, ready)) break;
          const uint32_t q = r + b;
          const uint32_t t = c + q * G;
          const uint32_t cnt = s_entry_count[q % kEntryRing];
          const uint32_t start = s_entry_start[q % kEntryRing];
          const uint32_t excl = (q == 0 ? 0u : incl) + warp_sum(sum);
          for (uint32_t p = lane; p < cnt; p += 32) {
            const uint32_t slot = (start + p) % kPairRing;
            const uint32_t dst = excl + p;
            if (dst < cap) {
              idx_out[dst] = ring_idx[slot];
              val_out[dst] = ring_val[slot];
            } else {
              overflow = true;
            }
          }
          incl = excl + cnt;
          if (t == T - 1 && lane == 0) *count_out = incl < cap ? incl : cap;
          tail += cnt;
          ++done;
        }
      }
      const uint64_t now = __shfl_sync(0xffffffffu, global_timer_ns(), 0);
      if (done) {
        __syncwarp();
        if (lane == 0) {
          __threadfence_block();
          s_tail = tail;
          s_consumed = r + done;
        }
        r += done;
        last_progress = now;
        idle_iters = 0;
      } else {
        if (++idle_iters > (1u << 26) || now - last_progress > ctx.wait_limit_ns) {
          if (lane == 0) {
            atomicOr(ctx.error, kDevErrTimeout);
            s_abort = 1;
          }
          break;
        }
        __nanosleep(32);
      }
    }
    if (__any_sync(0xffffffffu, overflow) && lane == 0) atomicOr(ctx.error, kDevErrOverflow);
  }
  __syncthreads();
}

}  // namespace efs
