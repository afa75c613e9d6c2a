// stream_lookback.cuh — ordered stream compaction at memory speed with
// dynamically claimed work: persistent CTAs (one per SM) take groups of
// tiles from a global counter, stream them through a TMA-fed ring, and place
// each group's selected pairs straight from shared memory once a decoupled
// look-back has given the group its output position.
//
// Why dynamic groups: on this GPU the DRAM bandwidth a single SM receives
// varies from call to call by about +-15 % (the same SM is among the fastest
// in one call and the slowest in the next), so any partition fixed at launch
// leaves the memory system partly idle while the slowest CTAs finish.
// Claiming small groups balances that automatically, and because a group
// only ever waits for groups claimed before it (held by CTAs that are
// already running), progress does not depend on which CTAs are resident.
//
// Roles (warps of a CTA):
//  - 16 compute warps. Warp w owns the 256-coordinate segment [w*256,
//    (w+1)*256) of every tile (the element layout of stream_compact.cuh). A
//    group's two tiles arrive in consecutive ring stages; the warp computes
//    each tile's values and selection bits and releases its stage at once,
//    then, once for the group: the positions of its selected pairs (one warp
//    scan of the four units' counts), the pairs appended to its own circular
//    buffer in shared memory — or, for a segment that finds no room, to the
//    segment's slot in global memory —, the counts recorded in the group's
//    entry. The warp that completes a group publishes its aggregate.
//  - a producer warp: lane 1 claims groups, up to kLbClaimAhead ahead; lane 0
//    takes a claimed group when an entry is free and issues the bulk copies
//    (cp.async.bulk, completing on the stage's "full" mbarrier) of its tiles
//    as ring stages are released; after the last group, an end marker.
//  - a look-back warp: for each group of the CTA in claim order, the
//    decoupled look-back over the published group totals (Merrill & Garland,
//    the routine of the one-tile-per-CTA kernel), the inclusive total
//    published, then the output position of each of the group's segments in
//    (tile, warp) order, which is coordinate order.
//  - kLbPlaceWarps placer warps: for each group, once its positions are
//    there, they copy its segments (placer p: segments p, p + kLbPlaceWarps,
//    ...; a warp's lanes on consecutive pairs, so loads and stores are
//    coalesced) from the buffers or slots to the output, then hand the
//    buffers' space back and free the entry.
//
// Deadlock freedom. Take the lowest group m that is claimed but whose
// aggregate is not published. Groups below m have published aggregates, so
// the look-back (and then the placement) of every group below m completes,
// which frees every entry and buffer space they hold. The CTA holding m waits
// for nothing else: a compute warp never waits for buffer space (a segment
// without room goes to its slot), the producer waits only for entries of
// older groups of its own CTA and for its ring, and the ring's stages are
// released by the compute warps as soon as they have read them. So m is
// completed and the argument repeats; no wait depends on which CTAs are
// resident. Every wait is nevertheless bounded in time; one that runs out
// latches kDevErrTimeout, and the CTA stops (after its bulk copies have
// landed).
//
// Traffic: the op's own bytes plus 8 bytes per selected pair, written once,
// plus 16 bytes per pair that goes through a slot; 8 bytes of look-back
// status per group. The error norm (when la.err_out is set) follows
// stream_compact.cuh's rule per coordinate; each group's share (its warps'
// float-float shares in warp order) is stored per group, and the last CTA to
// finish adds the groups' shares in group order, so the value does not
// depend on which CTA took which group.
#pragma once

#include "stream_compact.cuh"

namespace efs {

constexpr int kLbProducerWarp = kSWarps;       // 16
constexpr int kLbScanWarp = kSWarps + 1;       // 17
constexpr int kLbPlaceWarp = kSWarps + 2;      // 18: the first placer warp
constexpr int kLbPlaceWarps = 12;  // with 8, placement bounds calls that send ~a quarter of a
                                   // vector; 12 cost nothing on sparser ones
constexpr int kLbThreads = 32 * (kSWarps + 2 + kLbPlaceWarps);  // 960
static_assert(kLbThreads <= 1024, "one CTA of at most 1024 threads");
constexpr uint32_t kLbGroupTiles = 2;          // tiles per claimed group (the placement
                                               // assumes 2: 32 segments, one per lane)
constexpr uint32_t kLbGroupSegs = kLbGroupTiles * kSWarps;
constexpr uint32_t kLbClaimAhead = 2;          // groups claimed before the producer needs them
constexpr uint32_t kLbEntries = 8;             // groups of a CTA in flight or pending
constexpr uint32_t kLbStageEnd = 0xffffffffu;
constexpr uint32_t kLbSuspendNs = 1000;        // a suspended wait re-checks its flag and limit this often
constexpr uint32_t kLbSegsPerLane = kLbGroupSegs / 32;  // segments per lane in the offset scan
static_assert(kLbGroupSegs % 32 == 0 && kLbSegsPerLane <= 2, "segments per look-back lane");

// One group of a CTA, from the producer taking it until its pairs are placed.
struct LbEntry {
  uint32_t cnt[kLbGroupSegs];  // pairs of segment (q, w) at q * 16 + w
  uint32_t off[kLbGroupSegs];  // output position of each segment's first pair
  FF err[kSWarps];             // the warps' shares of ||e'||^2 in this group
  uint32_t tag;                // (claim number << 2) | state: 0 counting, 1 aggregate
                               // published, 2 offsets ready
  uint32_t group;              // group index
  uint32_t ntiles;             // tiles of the group (the last group may have fewer)
  uint32_t arrivals;           // segments counted so far (complete: ntiles * 16)
  uint32_t total;              // the group's aggregate (once complete)
  uint32_t placed;             // kSWarps: the entry is free (set by the placers)
  uint32_t spilled;            // bit l: segment l's pairs are in its global slot
  uint32_t pad;
};
__device__ __forceinline__ uint32_t lb_tag(uint32_t seq, uint32_t state) { return (seq << 2) | state; }

template <class Op, int kStages>
struct LbLayout {
  static constexpr uint32_t kRing = kStages * Op::kStageBytes;
  // pair buffer per compute warp: what is left of 227 KB (less 2 KB of static
  // shared memory), in whole warps of pairs
  static constexpr uint32_t kEntryBytes = kLbEntries * sizeof(LbEntry);
  static constexpr uint32_t kBudget = 227u * 1024u - 2048u;
  static constexpr uint32_t kFifo = ((kBudget - kRing - kEntryBytes) / (kSWarps * 8u)) / 32u * 32u;
  // (a segment that finds no room goes to its global slot, so nothing waits
  // for buffer space; a buffer smaller than a segment would only spill more)
  static_assert(kFifo >= kSWarpElems, "a whole segment fits a warp's buffer");
  static constexpr uint32_t kOffEntries = kRing + kSWarps * kFifo * 8u;
  static constexpr uint32_t kSmem = kOffEntries + kEntryBytes;  // dynamic shared memory
};

struct LbArgs {
  uint32_t* tile_base;  // optional [num_tiles + 1]: output position of each tile's first pair,
                        // and the total (untruncated), or null
  double* err_out;      // optional: sum of a^2 over the coordinates whose residual is final
                        // here (not selected, not deferred), or null
  FF* err_parts;        // [groups] the groups' shares of it (used when err_out is set)
  uint32_t* slot_idx;   // [num_tiles * 16 * 256] a segment's pairs when its warp's buffer is
  float* slot_val;      // full: segment (tile, warp) at (tile * 16 + warp) * 256
  uint32_t* density_out;  // optional (host-mapped): the call's pair count * 65536 / d, a hint
                          // the host reads for later calls' choice of ring depth, or null
};

__device__ __forceinline__ uint32_t vld(const uint32_t& x) {
  return *reinterpret_cast<const volatile uint32_t*>(&x);
}
__device__ __forceinline__ void vst(uint32_t& x, uint32_t v) {
  *reinterpret_cast<volatile uint32_t*>(&x) = v;
}

// Bounded spin of one thread until pred() holds; false (and the CTA's failed
// flag set, the timeout latched) when the limit passes, false at once when
// another thread of the CTA has failed.
template <class Pred>
__device__ __forceinline__ bool lb_spin(Pred pred, uint32_t* s_failed, const ScanCtx& ctx) {
  if (pred()) return true;
  const uint64_t t0 = global_timer_ns();
  for (uint32_t it = 0;; ++it) {
    if (pred()) return true;
    if (vld(*s_failed)) return false;
    if (it > (1u << 26) || global_timer_ns() - t0 > ctx.wait_limit_ns) {
      vst(*s_failed, 1u);
      atomicOr(ctx.error, kDevErrTimeout);
      return false;
    }
    __nanosleep(64);
  }
}

// Bounded wait for an mbarrier phase, giving up when the CTA has failed.
__device__ __forceinline__ bool lb_mbar_wait(uint64_t* bar, uint32_t parity, uint32_t* s_failed,
                                             const ScanCtx& ctx) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  for (uint32_t it = 0;; ++it) {
    if (mbar_try_wait_for(bar, parity, kLbSuspendNs)) return true;
    if (vld(*s_failed)) return false;
    if (it > (1u << 26) || global_timer_ns() - t0 > ctx.wait_limit_ns) {
      vst(*s_failed, 1u);
      atomicOr(ctx.error, kDevErrTimeout);
      return false;
    }
  }
}

// x[j] for a run-time j without an indexed (local-memory) access.
__device__ __forceinline__ float lb_pick(const float (&x)[4], int j) {
  const float lo = (j & 1) ? x[1] : x[0];
  const float hi = (j & 1) ? x[3] : x[2];
  return (j & 2) ? hi : lo;
}

// Named barrier of the placer warps (id 2; 0 is __syncthreads, 1 group_bar).
__device__ __forceinline__ void lb_place_bar(int count) {
  asm volatile("bar.sync 2, %0;" ::"r"(count) : "memory");
}

// The test hook withholds a tile; here the group holding it never publishes.
__device__ __forceinline__ bool lb_withheld(const ScanCtx& ctx, uint32_t group) {
  return ctx.withheld_tile >= 0 &&
         static_cast<int64_t>(group) == ctx.withheld_tile / static_cast<int64_t>(kLbGroupTiles);
}

template <class Op, int kStages>
__global__ void __launch_bounds__(kLbThreads, 1)
    lookback_stream_kernel(Op op, uint32_t d, uint32_t* __restrict__ idx_out,
                           float* __restrict__ val_out, uint32_t* __restrict__ count_out,
                           uint32_t cap, ScanCtx ctx, LbArgs la) {
  extern __shared__ __align__(128) unsigned char smem[];
  __shared__ __align__(8) uint64_t s_full[kStages];
  __shared__ __align__(8) uint64_t s_empty[kStages];
  __shared__ uint32_t s_stage_tile[kStages];  // tile of the stage's current use, or the end
  __shared__ uint32_t s_stage_info[kStages];  // its group's entry slot | (tile in the group << 8)
  __shared__ uint32_t s_claimed;              // groups the producer took so far
  __shared__ uint32_t s_claim_done;           // the producer takes no more
  __shared__ uint32_t s_failed;               // a wait of this CTA ran out
  __shared__ uint32_t s_resolved;             // groups the look-back warp resolved
  __shared__ uint32_t s_freed[kSWarps];       // pairs of each compute warp placed so far
  __shared__ uint32_t s_place_go;             // the placers' next group is ready (else: stop)
  __shared__ uint32_t s_cq[kLbClaimAhead];    // groups claimed ahead, with the queue counts
  __shared__ uint32_t s_cq_tail, s_cq_head;
  __shared__ uint32_t s_last;                 // this CTA finished last
  __shared__ FF s_err_sum[32];
  using L = LbLayout<Op, kStages>;
  uint32_t* const f_idx = reinterpret_cast<uint32_t*>(smem + L::kRing);
  float* const f_val = reinterpret_cast<float*>(smem + L::kRing + kSWarps * L::kFifo * 4u);
  LbEntry* const ent = reinterpret_cast<LbEntry*>(smem + L::kOffEntries);

  const uint32_t T = ctx.num_tiles;
  const uint32_t G = (T + kLbGroupTiles - 1) / kLbGroupTiles;
  const uint32_t full_tiles = d / kTileElems;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&s_full[s], 1);
      mbar_init(&s_empty[s], kSWarps);
    }
    mbar_init_fence();
    s_claimed = 0;
    s_claim_done = 0;
    s_failed = 0;
    s_resolved = 0;
    s_cq_tail = 0;
    s_cq_head = 0;
  }
  if (threadIdx.x < kSWarps) s_freed[threadIdx.x] = 0;
  if (threadIdx.x < kLbEntries) {
    ent[threadIdx.x].placed = kSWarps;  // free
    ent[threadIdx.x].tag = 0xffffffffu;
  }
  __syncthreads();
  // A dependent launch starts while the previous kernel's last groups are
  // placed, a phase that leaves DRAM mostly idle: pull the first groups the
  // CTAs will claim (about two each, claimed in CTA order) toward L2
  // meanwhile. A prefetch is not a read of the data: L2 is the point of
  // coherence, so the previous kernel's writes still land before the bulk
  // copies read these lines. Whole tiles only.
  if (threadIdx.x == 0 && Op::kPrefetchTiles > 0) {
    const uint32_t full_tiles = d / kTileElems;
    for (uint32_t r = 0; r < 2; ++r)
      for (uint32_t j = 0; j < kLbGroupTiles; ++j) {
        const uint32_t t = (blockIdx.x + r * gridDim.x) * kLbGroupTiles + j;
        if (t < full_tiles) op.prefetch(t);
      }
  }
  // everything the previous kernels on the stream wrote (and the reset
  // group counter) is read only after this
  griddep_wait();
  op.prologue();
  const uint64_t aux = op.initial_aux();  // uniform

  if (warp == kLbProducerWarp) {
    if (lane == 1) {
      // ---------------------------------------------------- claimer
      // Claims groups up to kLbClaimAhead ahead of the producer, so that a
      // claim's round trip never stalls the producer's refills (a fence or
      // an mbarrier arrival of the producer would wait for it).
      uint32_t tail = 0;
      while (true) {
        if (!lb_spin([&] { return tail - vld(s_cq_head) < kLbClaimAhead; }, &s_failed, ctx)) break;
        const uint32_t g = atomicAdd(ctx.tile_claim, 1u);
        s_cq[tail % kLbClaimAhead] = g;
        __threadfence_block();
        vst(s_cq_tail, ++tail);
        if (g >= G) break;
      }
    }
    // ------------------------------------------------------ producer
    if (lane == 0) {
      const uint64_t policy = l2_evict_normal_policy();
      uint32_t r = 0, seq = 0;
      bool ok = true;
      // the stage of use r is free once its previous use was released
      auto stage_free = [&](int s) {
        return r < static_cast<uint32_t>(kStages) ||
               lb_mbar_wait(&s_empty[s], ((r / kStages) - 1) & 1u, &s_failed, ctx);
      };
      uint32_t cq_head = 0;
      while (ok) {
        const uint32_t slot = seq % kLbEntries;
        LbEntry& en = ent[slot];
        if (!lb_spin([&] { return vld(en.placed) == kSWarps; }, &s_failed, ctx)) {
          ok = false;
          break;
        }
        if (!lb_spin([&] { return vld(s_cq_tail) > cq_head; }, &s_failed, ctx)) {
          ok = false;
          break;
        }
        __threadfence_block();  // the claimed number after the count
        const uint32_t g = vld(s_cq[cq_head % kLbClaimAhead]);
        vst(s_cq_head, ++cq_head);
        if (g >= G) break;
        const uint32_t nt = min(kLbGroupTiles, T - g * kLbGroupTiles);
        en.group = g;
        en.ntiles = nt;
        en.arrivals = 0;
        en.spilled = 0;
        en.placed = 0;
        __threadfence_block();
        vst(en.tag, lb_tag(seq, 0));
        vst(s_claimed, seq + 1);
        for (uint32_t q = 0; q < nt; ++q, ++r) {
          const int s = static_cast<int>(r % kStages);
          if (!stage_free(s)) {
            ok = false;
            break;
          }
          const uint32_t t = g * kLbGroupTiles + q;
          s_stage_tile[s] = t;
          s_stage_info[s] = slot | (q << 8);
          if (t < full_tiles) {
            mbar_arrive_expect_tx(&s_full[s], Op::kStageBytes);
            op.fill(smem + s * Op::kStageBytes, t, &s_full[s], policy);
          } else {
            mbar_arrive(&s_full[s]);  // the partial last tile is read from global memory
          }
        }
        ++seq;
      }
      if (ok) {  // the end marker
        const int s = static_cast<int>(r % kStages);
        if (stage_free(s)) {
          s_stage_tile[s] = kLbStageEnd;
          mbar_arrive(&s_full[s]);
          ++r;
        }
      }
      vst(s_claim_done, 1u);
      griddep_launch_dependents();  // this CTA reads nothing more: the next kernel may be scheduled
      // no copy may land after the CTA exits: wait for the last use of every
      // stage (a completed phase reports complete at once)
      for (uint32_t q = r > static_cast<uint32_t>(kStages) ? r - kStages : 0; q < r; ++q)
        if (!mbar_wait(&s_full[q % kStages], (q / kStages) & 1u, ctx.wait_limit_ns))
          atomicOr(ctx.error, kDevErrTimeout);
    }
  } else if (warp == kLbScanWarp) {
    // ------------------------------------------------------ look-back
    for (uint32_t seq = 0;; ++seq) {
      uint32_t go = 0;
      if (lane == 0) {
        lb_spin([&] { return vld(s_claimed) > seq || vld(s_claim_done) != 0; }, &s_failed, ctx);
        go = vld(s_claimed) > seq && !vld(s_failed);
        if (go) {
          LbEntry& en = ent[seq % kLbEntries];
          go = lb_spin([&] { return vld(en.tag) == lb_tag(seq, 1); }, &s_failed, ctx);
        }
        __threadfence_block();
      }
      if (!__shfl_sync(0xffffffffu, go, 0)) break;
      __syncwarp();
      LbEntry& en = ent[seq % kLbEntries];
      const uint32_t g = en.group, nt = en.ntiles, total = en.total;
      bool timed_out = false;
      const uint32_t excl = lookback_exclusive(ctx, g, timed_out);
      if (timed_out) {
        if (lane == 0) {
          vst(s_failed, 1u);
          atomicOr(ctx.error, kDevErrTimeout);
        }
        break;
      }
      if (lane == 0 && !lb_withheld(ctx, g))
        st_relaxed_u64(ctx.status + g, pack_status(ctx.epoch, kFlagPrefix, excl + total));
      // segment positions in (tile, warp) order: lane l holds segments
      // l * kLbSegsPerLane onwards
      const uint32_t nseg = nt * kSWarps;
      uint32_t cs[kLbSegsPerLane], mine = 0;
#pragma unroll
      for (uint32_t i = 0; i < kLbSegsPerLane; ++i) {
        const uint32_t sg = lane * kLbSegsPerLane + i;
        cs[i] = sg < nseg ? en.cnt[sg] : 0u;
        mine += cs[i];
      }
      uint32_t incl = mine;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t v = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += v;
      }
      const uint32_t first = excl + incl - mine;
      uint32_t run = first;
#pragma unroll
      for (uint32_t i = 0; i < kLbSegsPerLane; ++i) {
        en.off[lane * kLbSegsPerLane + i] = run;
        run += cs[i];
      }
      // a tile's first segment is segment q * 16, the first of lane q * 16 / kLbSegsPerLane
      const uint32_t tile_first =
          __shfl_sync(0xffffffffu, first, (lane * (kSWarps / kLbSegsPerLane)) & 31);
      if (la.tile_base && static_cast<uint32_t>(lane) < nt)
        la.tile_base[g * kLbGroupTiles + lane] = tile_first;
      if (lane == 0) {
        if (g == G - 1) {
          const uint32_t end = excl + total;
          *count_out = end < cap ? end : cap;
          if (la.tile_base) la.tile_base[T] = end;
          if (la.density_out)
            *la.density_out = static_cast<uint32_t>((static_cast<uint64_t>(end) << 16) / d);
        }
        if (la.err_out) {
          FF s{0.0f, 0.0f};
          for (int w = 0; w < kSWarps; ++w) s = ff_add(s, en.err[w]);
          la.err_parts[g] = s;
        }
      }
      __syncwarp();
      if (lane == 0) {
        __threadfence_block();
        vst(en.tag, lb_tag(seq, 2));
        ++s_resolved;
      }
    }
  } else if (warp >= kLbPlaceWarp) {
    // ------------------------------------------------------ placement
    // For each group in claim order, once its offsets are there: its pairs,
    // in (tile, warp) order, are the output positions [off[0], off[0] + n).
    // The kLbPlaceWarps warps copy them together, lane k of placer warp p
    // taking the positions = 32 p + k modulo 32 kLbPlaceWarps, each from its
    // compute warp's buffer (coalesced stores); then the buffers' space is
    // handed back and the entry freed. Every placer warp tracks the buffer
    // heads itself (lane w < 16: compute warp w's oldest unplaced pair).
    const int pw = warp - kLbPlaceWarp;
    constexpr int kPlaceThreads = 32 * kLbPlaceWarps;
    const uint64_t keep_policy = Op::kKeepPairs ? l2_evict_last_policy() : 0ull;
    uint32_t head = 0;
    bool overflow = false;
    for (uint32_t seq = 0;; ++seq) {
      if (pw == 0 && lane == 0) {
        lb_spin([&] { return vld(s_claimed) > seq || vld(s_claim_done) != 0; }, &s_failed, ctx);
        uint32_t go = vld(s_claimed) > seq && !vld(s_failed);
        if (go) {
          LbEntry& en = ent[seq % kLbEntries];
          go = lb_spin([&] { return vld(en.tag) == lb_tag(seq, 2); }, &s_failed, ctx);
        }
        s_place_go = go;
      }
      lb_place_bar(kPlaceThreads);  // the decision and the offsets are visible to every placer
      if (!s_place_go) break;
      LbEntry& en = ent[seq % kLbEntries];
      const uint32_t nseg = en.ntiles * kSWarps;
      // lane l describes segment l (l < nseg): start within the group, count,
      // and its first pair's buffer position
      const uint32_t c = static_cast<uint32_t>(lane) < nseg ? en.cnt[lane] : 0u;
      const uint32_t first = en.off[0];
      const uint32_t start = static_cast<uint32_t>(lane) < nseg ? en.off[lane] - first : 0xffffffffu;
      const uint32_t spilled = en.spilled;
      const bool in_slot = (spilled >> lane) & 1u;
      const uint32_t c_buf = in_slot ? 0u : c;  // pairs the segment holds in its warp's buffer
      const int w = lane & (kSWarps - 1);
      // a buffered segment's first pair: its warp's head, after the warp's
      // tile-0 segment when that one is buffered too (kLbGroupTiles == 2); a
      // slotted segment's: its slot
      uint32_t src = __shfl_sync(0xffffffffu, head, w);
      const uint32_t c_prev = __shfl_sync(0xffffffffu, c_buf, (lane - kSWarps) & 31);
      if (lane >= kSWarps) src += c_prev;
      if (src >= L::kFifo) src -= L::kFifo;
      if (in_slot)
        src = ((en.group * kLbGroupTiles + static_cast<uint32_t>(lane) / kSWarps) * kSWarps +
               static_cast<uint32_t>(w)) * static_cast<uint32_t>(kSWarpElems);
      // placer warp p copies the segments l = p, p + kLbPlaceWarps, ...: the
      // segment's pairs are consecutive in its source and in the output, so
      // the warp's lanes take consecutive pairs (coalesced loads and stores)
      for (int l = pw; l < static_cast<int>(nseg); l += kLbPlaceWarps) {
        const uint32_t cl = __shfl_sync(0xffffffffu, c, l);
        const uint32_t dl = first + __shfl_sync(0xffffffffu, start, l);
        const uint32_t sl = __shfl_sync(0xffffffffu, src, l);
        const bool slotted = (spilled >> l) & 1u;
        const uint32_t fbase = static_cast<uint32_t>(l & (kSWarps - 1)) * L::kFifo;
        for (uint32_t k = lane; k < cl; k += 32) {
          uint32_t xi;
          float xv;
          if (slotted) {
            const size_t b = static_cast<size_t>(sl) + k;
            xi = la.slot_idx[b];  // written by a warp of this CTA (ordered by the fences)
            xv = la.slot_val[b];
          } else {
            uint32_t b = sl + k;
            if (b >= L::kFifo) b -= L::kFifo;
            xi = f_idx[fbase + b];
            xv = f_val[fbase + b];
          }
          const uint32_t pos = dl + k;
          if (pos < cap) {
            if constexpr (Op::kKeepPairs) {
              st_pair_policy(idx_out + pos, val_out + pos, xi, xv, keep_policy);
            } else {
              idx_out[pos] = xi;
              val_out[pos] = xv;
            }
          } else {
            overflow = true;
          }
        }
      }
      // every compute warp's buffer head moves past its pairs of the group
      const uint32_t c_tile1 = __shfl_sync(0xffffffffu, c_buf, (lane + kSWarps) & 31);
      const uint32_t mine_total = c_buf + (lane < kSWarps ? c_tile1 : 0u);
      if (lane < kSWarps) {
        head += mine_total;
        if (head >= L::kFifo) head -= L::kFifo;
      }
      lb_place_bar(kPlaceThreads);  // every placer is done with the buffers and the entry
      if (pw == 0) {
        if (lane < kSWarps) atomicAdd(&s_freed[lane], mine_total);
        if (lane == 0) {
          __threadfence_block();
          vst(en.placed, kSWarps);  // the entry is free
        }
      }
    }
    if (__any_sync(0xffffffffu, overflow) && lane == 0) atomicOr(ctx.error, kDevErrOverflow);
  } else {
    // ------------------------------------------------------ compute warps
    uint32_t* const my_idx = f_idx + warp * L::kFifo;
    float* const my_val = f_val + warp * L::kFifo;
    uint32_t tail = 0;      // next buffer position this warp writes
    uint32_t appended = 0;  // pairs appended so far (the placer counts the freed ones)
    FF warp_err{0.0f, 0.0f};  // lane 0: share of ||e'||^2 in the current group

    // A group's tiles arrive in consecutive ring uses; each tile is computed
    // and its stage released at once, and the group's bookkeeping (positions,
    // buffer, counts, arrival) is done once for both tiles.
    auto compute_tile = [&](int s, uint32_t t, float (&a)[kSUnits][4],
                            uint32_t (&sel)[kSUnits]) {
      if (t < full_tiles) {
        op.tile_smem(smem + s * Op::kStageBytes, t, warp, lane, a, sel, aux);
      } else {
        op.tile_global(t, warp, lane, a, sel, aux);
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&s_empty[s]);  // this warp is done with the stage
      if (la.err_out) {
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
    };
    static_assert(kSUnits == 2 && kLbGroupTiles == 2, "four units of a group packed in one scan");
    for (uint32_t r = 0;;) {
      int s = static_cast<int>(r % kStages);
      bool arrived = lb_mbar_wait(&s_full[s], (r / kStages) & 1u, &s_failed, ctx);
      if (!__all_sync(0xffffffffu, arrived)) break;
      const uint32_t t0 = s_stage_tile[s];
      const uint32_t slot = s_stage_info[s] & 0xffu;
      if (t0 == kLbStageEnd) break;
      LbEntry& en = ent[slot];
      const uint32_t nt = en.ntiles;
      float a[kLbGroupTiles][kSUnits][4];
      uint32_t sel[kLbGroupTiles][kSUnits] = {{0u, 0u}, {0u, 0u}};
      compute_tile(s, t0, a[0], sel[0]);
      ++r;
      if (nt == 2) {
        s = static_cast<int>(r % kStages);
        arrived = lb_mbar_wait(&s_full[s], (r / kStages) & 1u, &s_failed, ctx);
        if (!__all_sync(0xffffffffu, arrived)) break;
        compute_tile(s, t0 + 1, a[1], sel[1]);
        ++r;
      }
      // positions in coordinate order: one warp scan of the four units'
      // per-lane counts (at most 4 each, 128 a warp) packed in bytes
      const uint32_t cnt4 = __popc(sel[0][0] & 0xfu) | (__popc(sel[0][1] & 0xfu) << 8) |
                            (__popc(sel[1][0] & 0xfu) << 16) | (__popc(sel[1][1] & 0xfu) << 24);
      uint32_t incl4 = cnt4;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t x = __shfl_up_sync(0xffffffffu, incl4, o);
        if (lane >= o) incl4 += x;
      }
      const uint32_t all4 = __shfl_sync(0xffffffffu, incl4, 31);
      const uint32_t excl4 = incl4 - cnt4;
      const uint32_t u0 = all4 & 0xffu, u1 = (all4 >> 8) & 0xffu;
      const uint32_t u2 = (all4 >> 16) & 0xffu, u3 = all4 >> 24;
      const uint32_t seg_total[kLbGroupTiles] = {u0 + u1, u2 + u3};
      // each unit's first position within its tile's segment
      const uint32_t off[kLbGroupTiles][kSUnits] = {
          {excl4 & 0xffu, u0 + ((excl4 >> 8) & 0xffu)},
          {(excl4 >> 16) & 0xffu, u2 + (excl4 >> 24)}};
      // each segment's pairs go to the warp's buffer when it has room (the
      // placer frees it group by group), else to the segment's global slot;
      // bit q of to_slot: segment q goes to its slot
      uint32_t to_slot = 0;
      if ((seg_total[0] | seg_total[1]) && lane == 0) {
        const uint32_t held = appended - vld(s_freed[warp]);
        if (held + seg_total[0] > L::kFifo) to_slot |= 1u;
        const uint32_t held1 = held + ((to_slot & 1u) ? 0u : seg_total[0]);
        if (held1 + seg_total[1] > L::kFifo) to_slot |= 2u;
        if (to_slot != 3u) __threadfence_block();  // the buffer writes after the placer's reads
      }
      to_slot = __shfl_sync(0xffffffffu, to_slot, 0);
      __syncwarp();
      const uint32_t buf_total = ((to_slot & 1u) ? 0u : seg_total[0]) +
                                 ((to_slot & 2u) ? 0u : seg_total[1]);
      // each lane writes its selected pairs in coordinate order, one set
      // selection bit at a time (at a few percent density most lanes have
      // none, and the warp takes as many rounds as its fullest lane)
#pragma unroll
      for (int q = 0; q < 2; ++q) {
        const uint32_t t = t0 + q;
        const uint32_t first_elem =
            static_cast<uint32_t>(stream_element_index(t, warp, 0, lane, 0));
        if ((to_slot >> q) & 1u) {
          const size_t sb = (static_cast<size_t>(t) * kSWarps + warp) * kSWarpElems;
#pragma unroll
          for (int v = 0; v < kSUnits; ++v) {
            uint32_t p = off[q][v];
            for (uint32_t bits = sel[q][v] & 0xfu; bits; bits &= bits - 1, ++p) {
              const int j = __ffs(bits) - 1;
              la.slot_idx[sb + p] = first_elem + v * 128 + j;
              la.slot_val[sb + p] = lb_pick(a[q][v], j);
            }
          }
        } else {
#pragma unroll
          for (int v = 0; v < kSUnits; ++v) {
            uint32_t p = tail + ((q && !(to_slot & 1u)) ? seg_total[0] : 0u) + off[q][v];
            if (p >= L::kFifo) p -= L::kFifo;
            for (uint32_t bits = sel[q][v] & 0xfu; bits; bits &= bits - 1) {
              const int j = __ffs(bits) - 1;
              my_idx[p] = first_elem + v * 128 + j;
              my_val[p] = lb_pick(a[q][v], j);
              if (++p == L::kFifo) p = 0;
            }
          }
        }
      }
      tail += buf_total;
      if (tail >= L::kFifo) tail -= L::kFifo;
      appended += buf_total;
      uint32_t before = 0;
      if (lane == 0) {
        en.cnt[warp] = seg_total[0];
        if (nt == 2) en.cnt[kSWarps + warp] = seg_total[1];
        if (to_slot)
          atomicOr(&en.spilled, ((to_slot & 1u) << warp) | ((to_slot >> 1) << (kSWarps + warp)));
        if (la.err_out) {
          en.err[warp] = warp_err;
          warp_err = FF{0.0f, 0.0f};
        }
        __threadfence_block();  // the pairs and the counts before the arrival
        before = atomicAdd(&en.arrivals, nt);
      }
      before = __shfl_sync(0xffffffffu, before, 0);
      if (before + nt == nt * kSWarps) {
        // this warp counted the group's last segments: its aggregate
        if (lane == 0) __threadfence_block();
        __syncwarp();
        const uint32_t nseg = nt * kSWarps;
        uint32_t part = 0;
#pragma unroll
        for (uint32_t i = 0; i < kLbSegsPerLane; ++i) {
          const uint32_t sg = lane + 32 * i;
          part += sg < nseg ? vld(en.cnt[sg]) : 0u;
        }
        const uint32_t agg = warp_sum(part);
        if (lane == 0) {
          if (!lb_withheld(ctx, en.group))
            st_relaxed_u64(ctx.status + en.group, pack_status(ctx.epoch, kFlagAggregate, agg));
          en.total = agg;
          __threadfence_block();
          vst(en.tag, vld(en.tag) | 1u);  // (claim number, 0) -> (claim number, 1)
        }
      }
    }
  }

  // every CTA counts itself finished (after its resolved groups); the last
  // one leaves the counters at zero for the next launch and, when every
  // group was resolved, adds the groups' error shares
  __syncthreads();
  uint32_t resolved_all = 0;
  if (threadIdx.x == 0) {
    atomicAdd(ctx.tile_claim + 2, s_resolved);
    __threadfence();
    const uint32_t done = atomicAdd(ctx.tile_claim + 1, 1u);
    s_last = done == gridDim.x - 1 ? 1u : 0u;
    if (s_last) {
      __threadfence();
      resolved_all = atomicAdd(ctx.tile_claim + 2, 0u);
      ctx.tile_claim[0] = 0;
      ctx.tile_claim[1] = 0;
      ctx.tile_claim[2] = 0;
      s_resolved = resolved_all;
    }
  }
  __syncthreads();
  if (s_last && la.err_out) {
    __threadfence();
    const bool ok = s_resolved == G;
    const FF err = sum_parts_ff(la.err_parts, ok ? G : 0u, s_err_sum);
    if (threadIdx.x == 0) *la.err_out = ok ? ff_to_double(err) : err_invalid();
  }
}

}  // namespace efs
