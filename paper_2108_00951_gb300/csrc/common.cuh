// common.cuh — device-side building blocks shared by the efsparse kernels:
// the tile geometry, the per-stream workspace view, bounded waits, and the
// decoupled-lookback prefix used by the ordered compaction.
//
// The ordered compaction is a single-pass prefix scan with decoupled
// look-back, implemented from the published method (Merrill & Garland,
// "Single-pass Parallel Prefix Scan with Decoupled Look-back", NVIDIA
// NVR-2016-002): every tile publishes its own count as soon as it is known,
// then reads its predecessors' published counts until it meets an inclusive
// prefix. In the one-tile-per-CTA kernel a CTA takes its tile id from a
// global counter when it starts (not from its block index), so every tile it
// waits for belongs to a CTA that is already running: the scan makes progress
// whatever order or concurrency the hardware schedules CTAs in. The streaming
// kernels' CTAs wait only for lower-numbered CTAs of their grid, which are
// dispatched first; kernels with grid-wide barriers are cooperative launches.
// Every wait is bounded in iterations and wall time and latches an error
// instead of hanging.
//
// Throughput of the scan: a tile can only finish once it sees an inclusive
// prefix, so the set of resolved tiles grows by at most one look-back window
// per L2 round trip. With a 32-tile window and 4096-element tiles that caps a
// 12-byte-per-element pass near 2 TB/s on this GPU; each lane therefore reads
// four status words, giving a 128-tile window.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

namespace efs {

// ---------------------------------------------------------------- geometry
constexpr int kThreads = 256;                 // threads per CTA
constexpr int kWarps = kThreads / 32;         // 8
constexpr int kUnits = 4;                     // 4-element units per thread per tile
constexpr int kWarpElems = 32 * 4 * kUnits;   // 512 contiguous elements per warp
constexpr int kTileElems = kWarps * kWarpElems;  // 4096 elements per tile

// Latched device error bits (mapped to ef_status on the host).
constexpr uint32_t kDevErrTimeout = 1u;
constexpr uint32_t kDevErrBadInput = 2u;
constexpr uint32_t kDevErrOverflow = 4u;  // a pair position fell outside the output

// Tile status word: [63:34] epoch | [33:32] flag | [31:0] count.
constexpr uint32_t kFlagNone = 0, kFlagAggregate = 1, kFlagPrefix = 2;

// Everything a compaction launch needs from the per-stream workspace.
struct ScanCtx {
  uint64_t* status;        // one word per tile
  uint32_t* error;         // latched kDevErr* bits
  uint32_t epoch;          // tags this launch's status words (1 .. 2^30-1)
  uint32_t num_tiles;
  int64_t withheld_tile;   // test hook: this tile never publishes (-1: none)
  uint64_t wait_limit_ns;  // bound on any single wait
  // Tile dispenser of the one-tile-per-CTA kernel: [0] tiles handed out,
  // [1] CTAs finished. Zero between launches: the last CTA to finish resets
  // both.
  uint32_t* tile_claim;
};

// --------------------------------------------------------- memory helpers
__device__ __forceinline__ void st_relaxed_u64(uint64_t* p, uint64_t v) {
  asm volatile("st.relaxed.gpu.global.b64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}
__device__ __forceinline__ uint64_t ld_relaxed_u64(const uint64_t* p) {
  uint64_t v;
  asm volatile("ld.relaxed.gpu.global.b64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ uint32_t ld_acquire_u32(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void st_release_u32(uint32_t* p, uint32_t v) {
  asm volatile("st.release.gpu.global.b32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ uint64_t global_timer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
__device__ __forceinline__ uint32_t lanemask_lt() {
  uint32_t m;
  asm("mov.u32 %0, %%lanemask_lt;" : "=r"(m));
  return m;
}

// Streaming loads/stores: data touched once per call should not evict the
// small hot structures (tile status, histograms) from L2.
__device__ __forceinline__ float4 ld_stream_f4(const float* p) {
  float4 v;
  asm volatile("ld.global.cs.v4.f32 {%0,%1,%2,%3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "l"(p));
  return v;
}
__device__ __forceinline__ uint2 ld_stream_u2(const void* p) {
  uint2 v;
  asm volatile("ld.global.cs.v2.u32 {%0,%1}, [%2];" : "=r"(v.x), "=r"(v.y) : "l"(p));
  return v;
}
__device__ __forceinline__ void st_stream_f4(float* p, float4 v) {
  asm volatile("st.global.cs.v4.f32 [%0], {%1,%2,%3,%4};" ::"l"(p), "f"(v.x), "f"(v.y),
               "f"(v.z), "f"(v.w)
               : "memory");
}

__device__ __forceinline__ float bf16_bits_to_f32(uint32_t bits16) {
  return __uint_as_float(bits16 << 16);
}

__device__ __forceinline__ uint64_t pack_status(uint32_t epoch, uint32_t flag, uint32_t value) {
  return (static_cast<uint64_t>(epoch) << 34) | (static_cast<uint64_t>(flag) << 32) | value;
}

__device__ __forceinline__ uint32_t warp_sum(uint32_t v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Publish this tile's status (one 64-bit store, so flag and count are seen
// together). Called by one thread.
__device__ __forceinline__ void publish(const ScanCtx& ctx, uint32_t tile, uint32_t flag,
                                        uint32_t value) {
  if (static_cast<int64_t>(tile) == ctx.withheld_tile) return;  // test hook
  st_relaxed_u64(ctx.status + tile, pack_status(ctx.epoch, flag, value));
}

// Decoupled look-back, executed by one full warp: returns the number of
// selected elements in all tiles before `tile`. The window holds the 128
// nearest unresolved predecessors: load j of lane l inspects tile
// base - 32j - l, so each load instruction of the warp reads 32 consecutive
// status words (coalesced) and the distance order is (j, lane). It slides
// back 128 tiles at a time until it contains an inclusive prefix; only the
// positions up to the nearest prefix must be ready. On a wait that runs out,
// `timed_out` is set (uniformly) and a partial sum is returned; the caller
// must not use it for addressing.
constexpr int kLookbackPerLane = 4;
constexpr int kLookbackWindow = 32 * kLookbackPerLane;

__device__ __forceinline__ uint32_t lookback_exclusive(const ScanCtx& ctx, uint32_t tile,
                                                      bool& timed_out) {
  const int lane = threadIdx.x & 31;
  uint32_t excl = 0;
  int64_t base = static_cast<int64_t>(tile) - 1;
  uint64_t t_start = 0;
  uint32_t iters = 0;
  timed_out = false;
  while (true) {
    uint64_t word[kLookbackPerLane];
#pragma unroll
    for (int j = 0; j < kLookbackPerLane; ++j) {  // all loads in flight together
      const int64_t t = base - (32 * j + lane);
      word[j] = t >= 0 ? ld_relaxed_u64(ctx.status + t)
                       : pack_status(ctx.epoch, kFlagPrefix, 0);  // before tile 0: prefix 0
    }
    uint32_t flag[kLookbackPerLane], value[kLookbackPerLane];
#pragma unroll
    for (int j = 0; j < kLookbackPerLane; ++j) {
      const bool current = static_cast<uint32_t>(word[j] >> 34) == ctx.epoch;
      flag[j] = current ? (static_cast<uint32_t>(word[j] >> 32) & 3u) : kFlagNone;
      value[j] = current ? static_cast<uint32_t>(word[j]) : 0u;
    }
    // the nearest prefix: the first load with one, its lowest lane
    int jp = kLookbackPerLane, lp = 32;
#pragma unroll
    for (int j = kLookbackPerLane - 1; j >= 0; --j) {
      const uint32_t b = __ballot_sync(0xffffffffu, flag[j] == kFlagPrefix);
      if (b) {
        jp = j;
        lp = __ffs(b) - 1;
      }
    }
    bool ready = true;
    uint32_t sum = 0, ready_sum = 0;
#pragma unroll
    for (int j = 0; j < kLookbackPerLane; ++j) {
      if (j < jp || (j == jp && lane <= lp)) {  // up to and including the nearest prefix
        ready = ready && flag[j] != kFlagNone;
        sum += value[j];
        if (flag[j] != kFlagNone) ready_sum += value[j];
      }
    }
    if (!__all_sync(0xffffffffu, ready)) {
      const uint64_t now = __shfl_sync(0xffffffffu, global_timer_ns(), 0);
      if (iters == 0) t_start = now;
      ++iters;
      if (iters > (1u << 26) || now - t_start > ctx.wait_limit_ns) {
        timed_out = true;
        return excl + warp_sum(ready_sum);
      }
      __nanosleep(64);
      continue;
    }
    excl += warp_sum(sum);
    if (jp < kLookbackPerLane) return excl;
    base -= kLookbackWindow;
  }
}

// ---------------------------------------------------------- error norm
// Squared error norm ||e'||^2 = sum_j e'_j^2, deterministic for a given
// launch shape: squares are accumulated with fmaf in fp32 in fixed groups of
// at most 8 terms (a warp tree of 32 such groups in the streaming kernels),
// and the groups are added in float-float arithmetic (an unevaluated pair
// hi + lo of fp32 values, added with the error-free TwoSum of Knuth, so each
// addition is exact up to about 2^-44 relatively) in a fixed order. Every
// fp32 group sum carries at most 13 roundings of nonnegative terms, so the
// result is within 13 * 2^-24 (< 1e-6) of the exact sum, relatively, plus
// the squares below the fp32 range (|e'_j| < 2^-75), which contribute 0; a
// sum beyond the fp32 range is +inf. Float-float instead of fp64: fp64
// arithmetic is slow on this GPU (a 32-step fp64 chain cost microseconds).

// Written as ||e'||^2 when a failed step has none.
__device__ __forceinline__ double err_invalid() { return __longlong_as_double(0x7ff8000000000000ll); }

struct FF {  // hi + lo, |lo| <= ulp(hi) / 2
  float hi, lo;
};

// Knuth's TwoSum: s + t == a + b exactly, s = RN(a + b).
__device__ __forceinline__ void two_sum(float a, float b, float& s, float& t) {
  s = __fadd_rn(a, b);
  const float bb = __fsub_rn(s, a);
  t = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
}

__device__ __forceinline__ FF ff_add(FF x, FF y) {
  float s, t;
  two_sum(x.hi, y.hi, s, t);
  t = __fadd_rn(t, __fadd_rn(x.lo, y.lo));
  const float hi = __fadd_rn(s, t);  // renormalise: |t| is small against s
  return FF{hi, __fsub_rn(t, __fsub_rn(hi, s))};
}

__device__ __forceinline__ double ff_to_double(FF x) {
  return static_cast<double>(x.hi) + static_cast<double>(x.lo);
}

struct ErrAcc {
  FF total{0.0f, 0.0f};
  float part = 0.0f;
  int terms = 0;
  __device__ __forceinline__ void add(float x) {
    part = __fmaf_rn(x, x, part);
    if (++terms == 8) flush();
  }
  __device__ __forceinline__ void flush() {
    total = ff_add(total, FF{part, 0.0f});
    part = 0.0f;
    terms = 0;
  }
};

__device__ __forceinline__ FF warp_sum_ff(FF v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const FF w{__shfl_xor_sync(0xffffffffu, v.hi, o), __shfl_xor_sync(0xffffffffu, v.lo, o)};
    v = ff_add(v, w);
  }
  return v;
}

// Sum of one value per thread over the CTA in a fixed order (a warp tree,
// then a tree over the warps); the result is valid in thread 0. s_ff holds
// 32 values.
__device__ __forceinline__ FF block_sum_ff(FF v, FF* s_ff) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int nw = static_cast<int>(blockDim.x >> 5);
  v = warp_sum_ff(v);
  __syncthreads();  // an earlier use of s_ff is complete
  if (lane == 0) s_ff[warp] = v;
  __syncthreads();
  FF r{0.0f, 0.0f};
  if (warp == 0) r = warp_sum_ff(lane < nw ? s_ff[lane] : FF{0.0f, 0.0f});
  return r;
}

// Sum of parts[0, n) by the whole CTA in a fixed order (one round of loads,
// then the fixed trees); valid in thread 0.
__device__ __forceinline__ FF sum_parts_ff(const FF* parts, uint32_t n, FF* s_ff) {
  FF v{0.0f, 0.0f};
  for (uint32_t q = threadIdx.x; q < n; q += blockDim.x) {
    const float2 p = __ldcg(reinterpret_cast<const float2*>(parts) + q);
    v = ff_add(v, FF{p.x, p.y});
  }
  return block_sum_ff(v, s_ff);
}

// Bounded grid-wide barrier for a cooperative launch (all CTAs co-resident).
// Returns false, latching kDevErrTimeout, if the wait ran out.
// Programmatic dependent launch: wait until the grids this one depends on
// have completed and their memory is visible (a no-op when the launch did
// not allow an early start), and let dependent grids be scheduled.
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void griddep_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Bounded barrier of `count` co-resident CTAs sharing the (arrive, gen) words.
__device__ __forceinline__ bool group_barrier(uint32_t* arrive, uint32_t* gen, uint32_t count,
                                              uint64_t limit_ns, uint32_t* error) {
  __shared__ int s_ok;
  __syncthreads();
  if (threadIdx.x == 0) {
    int ok = 1;
    const uint32_t my_gen = ld_acquire_u32(gen);
    __threadfence();  // this CTA's global writes before arriving
    const uint32_t ticket = atomicAdd(arrive, 1u);
    if (ticket == count - 1) {
      atomicExch(arrive, 0u);
      __threadfence();
      st_release_u32(gen, my_gen + 1);
    } else {
      const uint64_t t0 = global_timer_ns();
      uint32_t iters = 0;
      while (ld_acquire_u32(gen) == my_gen) {
        if (++iters > (1u << 26) || global_timer_ns() - t0 > limit_ns) {
          atomicOr(error, kDevErrTimeout);
          ok = 0;
          break;
        }
        __nanosleep(128);
      }
    }
    s_ok = ok;
  }
  __syncthreads();
  return s_ok != 0;
}

__device__ __forceinline__ bool grid_barrier(uint32_t* arrive, uint32_t* gen, uint64_t limit_ns,
                                             uint32_t* error) {
  return group_barrier(arrive, gen, gridDim.x, limit_ns, error);
}

}  // namespace efs
