// topk.cu — error-feedback + Top-k sparsifier (the paper's baseline, Lemma 2):
// one streaming pass over the coordinates, then an exact radix select and an
// ordered compaction on a small candidate list.
//
// Order. Every coordinate j gets the 63-bit composite key
//     K_j = (bits(|a_j|) << 32) | (~j & 0xffffffff),
// where bits(|a_j|) is the fp32 encoding with the sign cleared. For
// non-negative IEEE values the encoding orders like the value (NaN above
// +inf), and the low word makes a lower index rank higher among equal
// magnitudes. All K_j are distinct, so the Top-k set is exactly
// { j : K_j >= K_(k) } for the k-th largest key K_(k).
//
// Kernels of one call:
//  1 sample   every CTA histograms the top 13 key bits of 2048 coordinates
//             spread over its share of the tiles, the histograms are merged,
//             and the last CTA to arrive derives the lower bound B with about
//             1.5 times the needed mass above it (or, when the candidates
//             would not fit, the full-array mode).
//  2 stream   the streaming compaction (stream_compact.cuh, or from 4096
//             tiles on stream_lookback.cuh): a =
//             fmaf(γ,g,e) is written over e (12 B per coordinate, the
//             algorithmic bytes) and the coordinates with K_j >= B are
//             emitted as an ordered (index, value) candidate list. This
//             kernel also zeroes the other of the two per-call state blocks
//             for the next call.
//  3 select   the exact threshold K_(k) over the candidates — or over all of
//             a when the candidates are short of k, overflowed, or were not
//             gathered — then the ordered compaction of K_j >= K_(k), zeroing
//             e at the selected coordinates. Up to 48 K candidates CTA 0
//             finds the threshold in shared memory (digit levels over the
//             candidates' own magnitude range) and slice CTAs write the pairs
//             in parallel; beyond, the whole grid runs a radix select (merged
//             histograms with bounded grid barriers; chunk counts, then
//             positions).
// The candidate path moves about 12 B per coordinate plus small amounts; the
// full-array path adds a read of a per digit level and two for the output.
#include "gradient.cuh"
#include "internal.h"
#include "select.cuh"
#include "stream_lookback.cuh"

namespace efs {
namespace {

constexpr uint64_t kSelectNone = 1ull << 63;  // above every composite key

// LSB of each digit of the composite key; digit 0 is bits 62..52.
__device__ __forceinline__ int digit_shift(int level) {
  return level == 0 ? 52 : level == 1 ? 42 : level == 2 ? 32 : level == 3 ? 21 : level == 4 ? 10 : 0;
}

__device__ __forceinline__ uint64_t composite_key(float a, uint64_t j) {
  return (static_cast<uint64_t>(__float_as_uint(a) & 0x7fffffffu) << 32) |
         static_cast<uint64_t>(~static_cast<uint32_t>(j));
}

struct TopkArgs {
  uint32_t* hist;        // [kHistLevels + 1][kHistBins]
  uint64_t* cand0;       // key buffers of the refine levels
  uint64_t* cand1;
  uint32_t* list_idx;    // ordered candidates from the streaming pass
  float* list_val;
  uint32_t* cand_count;  // [kHistLevels]
  uint32_t cand_cap;
  uint64_t* lower_bound;
  uint32_t* mode;        // 0: candidates, 1: full array
  uint32_t* sel;         // short-list threshold: flag (1 found, 2 failed), B, ties, last
  uint32_t* list_count;
  uint32_t* list_flags;
  uint32_t* bar_arrive;
  uint32_t* bar_gen;
  uint32_t* error;
  uint64_t* chunk_sums;
  uint32_t epoch;        // tags the finalize kernel's chunk totals
  uint64_t wait_limit_ns;
  double* err_out;       // optional ||e'||^2 of the step
  const double* stream_err;  // the streaming pass's share (coordinates below the bound)
  FF* err_parts;         // [gridDim.x] the select CTAs' shares
};

// ------------------------------------------------------------- 1 stream
// The streaming pass as a stream_compact op, with the sampling of its bound
// (run by topk_sample_kernel): every sample CTA histograms the top 13 key
// bits of 2048 coordinates spread evenly over its share of the tiles, the
// histograms are merged, and the last CTA derives the lower bound B with about
// 1.5 times the needed mass above it — or, when the candidates would not fit,
// chooses the full-array mode (nothing gathered). Streaming: a = fmaf(γ,g,e)
// is written over e and the coordinates with K_j >= B are selected (ordered
// candidates).
template <typename GT>
struct TopkCandOp {
  const GT* g;
  float* e;
  float gamma;
  uint32_t d, k, cand_cap;
  uint32_t* hist;      // global sample histogram [kSampleBins]
  uint32_t* stream_arrive;  // arrivals of the sample kernel's CTAs (zero at the call's start)
  uint32_t* mode;      // published for the select kernel
  uint64_t* lower_bound;
  uint32_t* other_state;    // the other state block: zeroed here for the next call
  static constexpr uint32_t kGBytes = kTileElems * sizeof(GT);
  static constexpr uint32_t kStageBytes = kGBytes + kTileElems * sizeof(float);
  static constexpr uint32_t kWarpStagePairs = 512;  // on-chip staged pairs per compute warp
  static constexpr bool kKeepPairs = true;  // the candidate list: the select reads it next
  static constexpr int kSampleBins = efs::kSampleBins;
  static constexpr int kSampleShift = 31 - kSampleBits;  // key bits below the sampled ones

  // no L2 prefetch before the wait: measured 3 %% slower (the previous call's
  // select, still running, re-reads its candidate list from L2)
  static constexpr uint32_t kPrefetchTiles = 0;
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

  __device__ __forceinline__ void accumulate(const unsigned char* stage, int warp, int lane, int v,
                                             float (&x)[4]) const {
    const GT* gs = reinterpret_cast<const GT*>(stage);
    const float* es = reinterpret_cast<const float*>(stage + kGBytes);
    const int local = warp * kSWarpElems + lane * 4 + v * 128;
    GradVec<GT> gv;
    if constexpr (sizeof(GT) == 4)
      gv.v = *reinterpret_cast<const float4*>(gs + local);
    else
      gv.v = *reinterpret_cast<const uint2*>(gs + local);
    const float4 ev = *reinterpret_cast<const float4*>(es + local);
    x[0] = __fmaf_rn(gamma, gv[0], ev.x);
    x[1] = __fmaf_rn(gamma, gv[1], ev.y);
    x[2] = __fmaf_rn(gamma, gv[2], ev.z);
    x[3] = __fmaf_rn(gamma, gv[3], ev.w);
  }

  // The sample: each compute thread reads one aligned group of 4 coordinates
  // of g and e straight from global memory (issued together with the ring's
  // first fills), the groups spread evenly over the CTA's chunk.
  __device__ void sample(uint32_t t_lo, uint32_t t_hi, int tid, uint32_t* s_hist) const {
    const uint64_t lo = static_cast<uint64_t>(t_lo) * kTileElems;
    const uint64_t end = static_cast<uint64_t>(t_hi) * kTileElems;
    const uint64_t hi = end < d ? end : d;
    const uint64_t groups = (hi - lo) / 4;  // whole groups of 4 inside [lo, hi)
    const uint64_t grp = groups >= static_cast<uint64_t>(kComputeThreads)
                             ? static_cast<uint64_t>(tid) * groups / kComputeThreads
                             : static_cast<uint64_t>(tid);
    const bool in = grp < groups;
    GradVec<GT> gv;
    float4 ev = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
    if (in) {
      const uint64_t p = lo + grp * 4;
      if constexpr (sizeof(GT) == 4)
        gv.v = __ldg(reinterpret_cast<const float4*>(g + p));
      else
        gv.v = __ldg(reinterpret_cast<const uint2*>(g + p));
      ev = __ldg(reinterpret_cast<const float4*>(e + p));
    }
    float x[4] = {0.0f, 0.0f, 0.0f, 0.0f};
    if (in) {
      x[0] = __fmaf_rn(gamma, gv[0], ev.x);
      x[1] = __fmaf_rn(gamma, gv[1], ev.y);
      x[2] = __fmaf_rn(gamma, gv[2], ev.z);
      x[3] = __fmaf_rn(gamma, gv[3], ev.w);
    }
#pragma unroll
    for (int j = 0; j < 4; ++j)
      hist_add_warp(s_hist, (__float_as_uint(x[j]) & 0x7fffffffu) >> kSampleShift, in);
  }

  __device__ void merge(const uint32_t* s_hist) const {
    for (int b = threadIdx.x; b < kSampleBins; b += blockDim.x)
      if (s_hist[b]) atomicAdd(&hist[b], s_hist[b]);
  }

  // every CTA, first thing, whatever happens later in the launch
  __device__ void prologue() const { clear_state(other_state); }

  // The sample kernel's CTAs arrive once each, after a fence that publishes
  // their merged histogram (the arrival counter starts at zero in every call:
  // the per-call reset of the control block); the last to arrive sees every
  // sample. Nothing waits, so the grid needs no co-residency.
  __device__ bool arrive_last() const {
    __shared__ int s_last;
    __syncthreads();
    if (threadIdx.x == 0) {
      __threadfence();
      s_last = atomicAdd(stream_arrive, 1u) == gridDim.x - 1 ? 1 : 0;
      if (s_last) __threadfence();  // the other CTAs' merges before its reads
    }
    __syncthreads();
    return s_last != 0;
  }

  // the bound the sample kernel published (complete: the kernel before this)
  __device__ uint64_t initial_aux() const { return __ldcg(lower_bound); }

  // The bound, by the last sample CTA (every thread of it): each compute
  // thread loads 16 consecutive bins of the merged histogram (vector loads,
  // all in flight together), a block suffix scan gives the sampled mass above
  // each thread's bins, and the thread holding the target-th largest sample
  // finds its bin; the bound is published with the mode.
  __device__ uint64_t choose() const {
    constexpr int kPer = kSampleBins / kComputeThreads;
    static_assert(kPer % 4 == 0 && kPer * kComputeThreads == kSampleBins, "sample bins");
    __shared__ uint64_t s_bound;
    __shared__ uint32_t s_bin, s_mass;
    __shared__ uint32_t s_w[kStreamThreads / 32];
    const int t = threadIdx.x;
    uint32_t c[kPer];
    uint32_t mine = 0;
    if (t < kComputeThreads) {
      const uint4* src = reinterpret_cast<const uint4*>(hist) + t * (kPer / 4);
      uint4 v[kPer / 4];
#pragma unroll
      for (int q = 0; q < kPer / 4; ++q) v[q] = __ldcg(src + q);
#pragma unroll
      for (int q = 0; q < kPer / 4; ++q) {
        c[4 * q] = v[q].x;
        c[4 * q + 1] = v[q].y;
        c[4 * q + 2] = v[q].z;
        c[4 * q + 3] = v[q].w;
      }
    } else {
#pragma unroll
      for (int i = 0; i < kPer; ++i) c[i] = 0;
    }
#pragma unroll
    for (int i = 0; i < kPer; ++i) mine += c[i];
    if (t == 0) s_bin = 0xffffffffu;
    uint32_t sampled;
    const uint32_t above = block_suffix_exclusive(mine, sampled, s_w);  // orders the reset
    const bool everything = sampled == d;
    uint32_t target = k;
    if (!everything) {
      // 1.5x the expected sampled count above the k-th key, plus 32: many
      // standard deviations of sampling noise; a miss costs the exact
      // full-array fallback, never a wrong result
      // (integer arithmetic: the products stay below 2^56; FP64 is slow here)
      const uint64_t x = 3ull * k * sampled / (2ull * d) + 32ull;
      target = x >= sampled ? sampled + 1 : static_cast<uint32_t>(x);
    }
    // the bin holding the target-th largest sample, and the sampled mass at
    // or above it
    if (target <= sampled && above < target && target - above <= mine) {
      uint32_t run = above;
#pragma unroll
      for (int i = kPer - 1; i >= 0; --i) {
        run += c[i];
        if (run >= target && run - c[i] < target) {
          s_bin = t * kPer + i;
          s_mass = run;
        }
      }
    }
    __syncthreads();
    if (t == 0) {
      const bool found = s_bin != 0xffffffffu;
      uint64_t bound = found ? static_cast<uint64_t>(s_bin) << (32 + kSampleShift) : 0ull;
      // expected candidates (the sampled mass scaled to d) above half the
      // capacity: 2 * mass * d / sampled > cap, compared exactly
      const bool too_many =
          found ? (everything ? 2ull * s_mass > cand_cap
                              : 2ull * s_mass * d > static_cast<uint64_t>(cand_cap) * sampled)
                : 2ull * d > cand_cap;
      uint32_t m = 0;
      if (k == 0) {
        bound = kSelectNone;
      } else if (too_many) {
        m = 1;                // the candidates would not fit: full-array selection
        bound = kSelectNone;  // and none gathered while streaming
      }
      s_bound = bound;
      *mode = m;
      *lower_bound = bound;
    }
    __syncthreads();
    return s_bound;
  }

  __device__ __forceinline__ void tile_smem(const unsigned char* stage, uint32_t t, int warp,
                                            int lane, float (&a)[kSUnits][4],
                                            uint32_t (&sel)[kSUnits], uint64_t bound) const {
    const uint64_t first = stream_element_index(t, warp, 0, lane, 0);
#pragma unroll
    for (int v = 0; v < kSUnits; ++v) {
      accumulate(stage, warp, lane, v, a[v]);
      st_stream_f4(e + first + v * 128, make_float4(a[v][0], a[v][1], a[v][2], a[v][3]));
      sel[v] = 0;
#pragma unroll
      for (int j = 0; j < 4; ++j)
        sel[v] |= (composite_key(a[v][j], first + v * 128 + j) >= bound ? 1u : 0u) << j;
    }
  }

  __device__ __forceinline__ void tile_global(uint32_t t, int warp, int lane,
                                              float (&a)[kSUnits][4],
                                              uint32_t (&sel)[kSUnits], uint64_t bound) const {
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
          e[i] = x;
          a[v][j] = x;
          sel[v] |= (composite_key(x, i) >= bound ? 1u : 0u) << j;
        }
      }
    }
  }
};

constexpr int kTkStages = 4;

// The candidate bound of the streaming pass, in a kernel of its own before
// it: every CTA histograms the top 13 key bits of 2048 coordinates spread
// over its share of the tiles — loaded before the wait for the previous
// kernel, since a stale value only moves the bound, never the result (the
// select checks the candidates and falls back to the whole array) — merges
// its histogram into the call's global one, and the last CTA to arrive
// derives the bound and publishes it with the mode. No CTA waits for
// another, so the launch needs no co-residency; the streaming pass then has
// no grid barrier and is a plain programmatic launch.
// All of it runs before the wait for the previous kernel (the select of the
// previous call, still running): the histogram, the arrival counter, the
// bound and the mode live in this call's state block, which the previous
// call's streaming pass zeroed and which that select does not read, and that
// streaming pass completed before this grid could start (the select waited
// for it before letting this kernel start). Only the last CTA waits, so the
// grid completes after the previous kernel; the others leave their SMs to the
// streaming pass, which may be scheduled from the start.
template <typename GT>
__global__ void __launch_bounds__(kStreamThreads)
    topk_sample_kernel(TopkCandOp<GT> op, uint32_t num_tiles) {
  __shared__ uint32_t s_hist[TopkCandOp<GT>::kSampleBins];
  const uint32_t T = num_tiles, G = gridDim.x, c = blockIdx.x;
  const uint32_t t_lo = static_cast<uint32_t>(static_cast<uint64_t>(c) * T / G);
  const uint32_t t_hi = static_cast<uint32_t>(static_cast<uint64_t>(c + 1) * T / G);
  for (int b = threadIdx.x; b < TopkCandOp<GT>::kSampleBins; b += blockDim.x) s_hist[b] = 0;
  griddep_launch_dependents();  // the streaming pass waits for this whole grid
  __syncthreads();
  if (threadIdx.x < kComputeThreads && t_hi > t_lo) op.sample(t_lo, t_hi, threadIdx.x, s_hist);
  __syncthreads();
  op.merge(s_hist);
  if (!op.arrive_last()) return;
  op.choose();
  griddep_wait();  // this grid completes after the previous kernel
}

// Inputs the bulk copies cannot take (not 16-byte aligned): a = fmaf(γ,g,e)
// written over e with plain loads, and the selection switched to the
// full-array mode (block 0 runs after the sampling kernel on the stream).
template <typename GT>
__global__ void __launch_bounds__(kThreads)
    topk_accumulate_plain_kernel(const GT* __restrict__ g, float* __restrict__ e, float gamma,
                                 uint32_t d, TopkArgs args, uint32_t* other_state) {
  clear_state(other_state);
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    *args.mode = 1;
    *args.lower_bound = kSelectNone;
  }
  for (uint64_t i = static_cast<uint64_t>(blockIdx.x) * kThreads + threadIdx.x; i < d;
       i += static_cast<uint64_t>(gridDim.x) * kThreads)
    e[i] = __fmaf_rn(gamma, grad_scalar(g, i), e[i]);
}

// Reads the (mode, source length) a refine/finalize launch works on; the
// streaming pass's flags decide whether the candidates are usable.
struct SourceInfo {
  uint32_t mode;   // 0: candidate list, 1: full array
  uint32_t n;      // source length
  bool failed;     // the streaming pass timed out: select nothing
};

__device__ __forceinline__ SourceInfo read_source(const TopkArgs& args, uint32_t d, uint32_t k) {
  SourceInfo si;
  const uint32_t flags = __ldcg(args.list_flags);
  const uint32_t count = __ldcg(args.list_count);
  si.failed = (flags & kDevErrTimeout) != 0;
  si.mode = __ldcg(args.mode);
  if (si.mode == 0 && ((flags & kDevErrOverflow) || count < k)) si.mode = 1;
  si.n = si.mode == 0 ? count : d;
  return si;
}

// Key of source element i: a candidate (index, value) or a coordinate of a.
__device__ __forceinline__ uint64_t source_key(const TopkArgs& args, const float* a, uint32_t mode,
                                               uint64_t i) {
  if (mode == 0) return composite_key(__ldcg(args.list_val + i), __ldcg(args.list_idx + i));
  return composite_key(__ldcg(a + i), i);
}

// Warp-aggregated append of the keys of the lanes with pred set.
__device__ __forceinline__ void warp_append(bool pred, uint64_t key, uint64_t* dst,
                                            uint32_t* count, uint32_t cap) {
  const uint32_t m = __ballot_sync(0xffffffffu, pred);
  if (m == 0) return;
  const int lane = threadIdx.x & 31;
  const int leader = __ffs(m) - 1;
  uint32_t base = 0;
  if (lane == leader) base = atomicAdd(count, static_cast<uint32_t>(__popc(m)));
  base = __shfl_sync(0xffffffffu, base, leader);
  if (pred) {
    const uint32_t pos = base + __popc(m & lanemask_lt());
    if (pos < cap) dst[pos] = key;
  }
}

// ------------------------------------------------------------- 2 select
// Exact threshold by radix select, then the ordered compaction of K >= it.
constexpr int kSelThreads = 1024;
constexpr uint32_t kSmallCand = 48u * 1024u;  // magnitudes one CTA holds in shared memory
constexpr uint32_t kSelSmem = kSmallCand * sizeof(uint32_t);

// Writes the source elements [lo, hi) with key >= thr, in order, to the
// outputs from position `base`, 4 consecutive elements per thread per block,
// and zeroes the residual at each; returns the number written. Whole CTA.
__device__ uint32_t write_selected(const TopkArgs& args, float* e, uint32_t mode, uint32_t lo,
                                   uint32_t hi, uint64_t thr, uint32_t base, uint32_t k,
                                   uint32_t* idx_out, float* val_out, bool& overflow,
                                   uint32_t* s_w) {
  const uint32_t start = base;
  for (uint32_t b0 = lo; b0 < hi; b0 += 4 * kSelThreads) {
    const uint32_t i0 = b0 + 4 * threadIdx.x;
    uint32_t sel = 0, coord[4];
    float val[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {  // all loads in flight before the scan
      const bool in = i0 + j < hi;
      coord[j] = in ? (mode == 0 ? __ldcg(args.list_idx + i0 + j) : i0 + j) : 0u;
      val[j] = in ? (mode == 0 ? __ldcg(args.list_val + i0 + j) : __ldcg(e + i0 + j)) : 0.0f;
    }
#pragma unroll
    for (int j = 0; j < 4; ++j)
      if (i0 + j < hi && composite_key(val[j], coord[j]) >= thr) sel |= 1u << j;
    uint32_t block_total;
    uint32_t pos = base + block_exclusive<kSelThreads>(__popc(sel), block_total, s_w);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      if (sel & (1u << j)) {
        if (pos < k) {
          idx_out[pos] = coord[j];
          val_out[pos] = val[j];
          e[coord[j]] = 0.0f;  // residual of a sent coordinate
        } else {
          overflow = true;
        }
        ++pos;
      }
    }
    base += block_total;
  }
  return base - start;
}

// A short candidate list (n <= kSmallCand) is resolved in two parts.
// CTA 0 finds the threshold in shared memory. The magnitudes of every
// candidate are loaded once, with their minimum and maximum. Digit levels
// narrow a window [B, B + W) of magnitude bit patterns (monotone in |a|):
// level 0 splits [min, max] into at most 2048 bins, each later level splits
// the chosen bin into at most 2048 sub-bins. The levels stop when the window holds exactly the remaining rank, or is
// one magnitude T wide; then equal magnitudes are taken in list order, which
// is index order (the lowest-index tie rule), up to list position `last`.
// The selection is |a| > B, or |a| == B at a position <= last. CTA 0
// publishes (B, ties, last) behind a flag; every slice CTA, having loaded
// its slice of kSliceElems positions meanwhile, publishes its slice's count,
// sums the earlier slices' counts, and writes its selected pairs in order,
// zeroing the residual at each.
constexpr uint32_t kSliceElems = 4 * kSelThreads;  // list positions per slice CTA

// CTA 0: the threshold of the list; returns false when the histograms do
// not find the rank (never for a well-formed list).
__device__ bool small_threshold(const TopkArgs& args, uint32_t n, uint32_t k, uint32_t* s_mag,
                                uint32_t* s_hist, uint32_t* s_w, SmallSelection& out) {
  __shared__ uint32_t s_lo[32], s_hi[32];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  constexpr int kBatch = 8;  // loads in flight per thread
  uint32_t lo = 0xffffffffu, hi = 0;
  for (uint32_t i0 = tid; i0 < n; i0 += kBatch * kSelThreads) {
    uint32_t v[kBatch];
#pragma unroll
    for (int j = 0; j < kBatch; ++j) {
      const uint32_t i = i0 + j * kSelThreads;
      v[j] = i < n ? __float_as_uint(__ldcg(args.list_val + i)) : 0u;
    }
#pragma unroll
    for (int j = 0; j < kBatch; ++j) {
      const uint32_t i = i0 + j * kSelThreads;
      if (i < n) {
        const uint32_t m = v[j] & 0x7fffffffu;
        s_mag[i] = m;
        lo = m < lo ? m : lo;
        hi = m > hi ? m : hi;
      }
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    lo = min(lo, __shfl_xor_sync(0xffffffffu, lo, o));
    hi = max(hi, __shfl_xor_sync(0xffffffffu, hi, o));
  }
  if (lane == 0) {
    s_lo[warp] = lo;
    s_hi[warp] = hi;
  }
  __syncthreads();
  lo = s_lo[lane];  // 32 warps
  hi = s_hi[lane];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    lo = min(lo, __shfl_xor_sync(0xffffffffu, lo, o));
    hi = max(hi, __shfl_xor_sync(0xffffffffu, hi, o));
  }
  return threshold_levels<kSelThreads>(MagsShared{s_mag}, n, k, lo, hi, s_hist, s_w, out);
}

// Slice CTA c of Gs: the selected pairs of list positions [c, c+1) * n / Gs.
__device__ void small_emit(const TopkArgs& args, float* e, uint32_t n, uint32_t k, uint32_t Gs,
                           uint32_t* idx_out, float* val_out, uint32_t* count_out,
                           uint32_t* s_w) {
  constexpr int kJ = kSliceElems / kSelThreads;  // positions per thread
  constexpr int kWarps = kSelThreads / 32;
  __shared__ SmallSelection s_sel;
  __shared__ uint32_t s_cnt[kJ * kWarps];
  __shared__ uint32_t s_flag;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const uint32_t c = blockIdx.x;
  const uint32_t lo = static_cast<uint32_t>(static_cast<uint64_t>(c) * n / Gs);
  const uint32_t hi = static_cast<uint32_t>(static_cast<uint64_t>(c + 1) * n / Gs);
  // the slice's candidates (position lo + j * kSelThreads + tid), loaded
  // before the threshold is known
  uint32_t coord[kJ], vbits[kJ];
#pragma unroll
  for (int j = 0; j < kJ; ++j) {
    const uint32_t i = lo + j * kSelThreads + tid;
    coord[j] = i < hi ? __ldcg(args.list_idx + i) : 0u;
    vbits[j] = i < hi ? __float_as_uint(__ldcg(args.list_val + i)) : 0u;
  }
  // the threshold and slice bases CTA 0 published (bounded wait)
  if (tid == 0) {
    uint32_t f = ld_acquire_u32(args.sel);
    const uint64_t t0 = global_timer_ns();
    for (uint32_t it = 0; f == 0; ++it) {
      if (it > (1u << 26) || global_timer_ns() - t0 > args.wait_limit_ns) {
        atomicOr(args.error, kDevErrTimeout);
        f = 2;
        break;
      }
      f = ld_acquire_u32(args.sel);
    }
    s_flag = f;
    if (f == 1) s_sel = SmallSelection{args.sel[1], args.sel[2], args.sel[3]};
  }
  __syncthreads();
  if (s_flag != 1) {  // no threshold: nothing is written
    if (c == 0 && tid == 0) *count_out = 0;
    return;
  }
  const SmallSelection sel = s_sel;
  uint32_t bits = 0;
#pragma unroll
  for (int j = 0; j < kJ; ++j) {
    const uint32_t i = lo + j * kSelThreads + tid;
    const uint32_t m = vbits[j] & 0x7fffffffu;
    const bool take = i < hi && (m > sel.B || (m == sel.B && (!sel.ties || i <= sel.last)));
    bits |= (take ? 1u : 0u) << j;
  }
  // per-(j, warp) counts in list order, then one scan over them
#pragma unroll
  for (int j = 0; j < kJ; ++j) {
    const uint32_t bal = __ballot_sync(0xffffffffu, (bits >> j) & 1u);
    if (lane == 0) s_cnt[j * kWarps + warp] = __popc(bal);
  }
  __syncthreads();
  const uint32_t mine = tid < kJ * kWarps ? s_cnt[tid] : 0u;
  uint32_t slice_total;
  const uint32_t off = block_exclusive<kSelThreads>(mine, slice_total, s_w);
  if (tid < kJ * kWarps) s_cnt[tid] = off;
  // publish the slice's count; sum the earlier slices' counts (bounded wait)
  if (tid == 0)
    st_relaxed_u64(args.chunk_sums + c, (static_cast<uint64_t>(args.epoch) << 32) | slice_total);
  uint32_t base = 0;
  {
    const uint64_t t0 = global_timer_ns();
    uint32_t it = 0;
    while (true) {
      uint32_t part = 0;
      bool present = true;
      for (uint32_t q = tid; q < c; q += kSelThreads) {
        const uint64_t w = ld_relaxed_u64(args.chunk_sums + q);
        if (static_cast<uint32_t>(w >> 32) == args.epoch)
          part += static_cast<uint32_t>(w);
        else
          present = false;
      }
      const bool all_present = __syncthreads_and(present);
      uint32_t sum;
      block_exclusive<kSelThreads>(part, sum, s_w);
      if (all_present) {
        base = sum;
        break;
      }
      const bool out_of_time = ++it > (1u << 26) || global_timer_ns() - t0 > args.wait_limit_ns;
      if (__syncthreads_or(out_of_time)) {
        if (tid == 0) atomicOr(args.error, kDevErrTimeout);
        return;
      }
    }
  }
  const uint32_t lt = lanemask_lt();
  bool overflow = false;
#pragma unroll
  for (int j = 0; j < kJ; ++j) {
    const uint32_t bal = __ballot_sync(0xffffffffu, (bits >> j) & 1u);
    if ((bits >> j) & 1u) {
      const uint32_t pos = base + s_cnt[j * kWarps + warp] + __popc(bal & lt);
      if (pos < k) {
        idx_out[pos] = coord[j];
        val_out[pos] = __uint_as_float(vbits[j]);
        e[coord[j]] = 0.0f;  // residual of a sent coordinate
      } else {
        overflow = true;
      }
    }
  }
  if (c == Gs - 1 && tid == 0) {
    const uint32_t end = base + slice_total;
    *count_out = end < k ? end : k;
  }
  if (__syncthreads_or(overflow) && tid == 0) atomicOr(args.error, kDevErrOverflow);
}

// Radix select of the k-th largest composite key of the source across the
// grid: merged global histograms, bounded grid barriers, candidate compaction
// into key buffers once a bucket fits.
__device__ uint64_t radix_threshold_grid(const TopkArgs& args, const float* a,
                                         const SourceInfo& si, uint32_t k, uint32_t* s_hist,
                                         uint32_t* s_w, bool& ok) {
  ok = true;
  uint64_t prefix = 0;
  uint32_t k_rem = k, n_in = si.n;
  int level = -1;
  int src = -1;  // -1: the source; 0/1: key buffer 0/1
  uint32_t src_count = si.n;
  Selection s{};
  const uint64_t stride = static_cast<uint64_t>(gridDim.x) * kSelThreads;
  do {
    ++level;
    const int sh = digit_shift(level);
    const int sh_prev = level == 0 ? 63 : digit_shift(level - 1);
    const int bits = sh_prev - sh;
    const uint32_t nb = 1u << bits;
    const bool compact = level > 0 && n_in <= args.cand_cap;
    const int dst = (src == 0) ? 1 : 0;
    uint64_t* dst_buf = dst ? args.cand1 : args.cand0;
    uint32_t* dst_count = args.cand_count + level;
    for (uint32_t b = threadIdx.x; b < nb; b += kSelThreads) s_hist[b] = 0;
    __syncthreads();
    const uint64_t* keys = src == 0 ? args.cand0 : args.cand1;
    constexpr int kBatch = 4;  // keys in flight per thread
    for (uint64_t base = static_cast<uint64_t>(blockIdx.x) * kSelThreads; base < src_count;
         base += kBatch * stride) {
      uint64_t key[kBatch];
#pragma unroll
      for (int j = 0; j < kBatch; ++j) {
        const uint64_t i = base + j * stride + threadIdx.x;
        key[j] = 0;
        if (i < src_count) key[j] = src < 0 ? source_key(args, a, si.mode, i) : __ldcg(keys + i);
      }
#pragma unroll
      for (int j = 0; j < kBatch; ++j) {
        const uint64_t i = base + j * stride + threadIdx.x;
        const bool valid = i < src_count;
        const bool match = valid && (level == 0 || (key[j] >> sh_prev) == prefix);
        hist_add_warp(s_hist, static_cast<uint32_t>(key[j] >> sh) & (nb - 1), match);
        if (compact) warp_append(match, key[j], dst_buf, dst_count, args.cand_cap);
      }
    }
    __syncthreads();
    uint32_t* gh = args.hist + level * kHistBins;
    for (uint32_t b = threadIdx.x; b < nb; b += kSelThreads)
      if (s_hist[b]) atomicAdd(&gh[b], s_hist[b]);
    if (!grid_barrier(args.bar_arrive, args.bar_gen, args.wait_limit_ns, args.error)) {
      ok = false;
      break;
    }
    s = select_bin<kSelThreads, true>(gh, nb, k_rem, s_w);
    if (!s.found) {
      ok = false;
      break;
    }
    prefix = (prefix << bits) | s.bin;
    const uint32_t n_prev = n_in;
    k_rem = s.k_rem;
    n_in = s.n_in;
    if (compact) {
      src = dst;
      src_count = n_prev;
    }
  } while (n_in != k_rem && level < kHistLevels - 1);
  // an unfound bin or an unresolved rank means the histograms disagree with
  // the data; a grid barrier latches its own timeout
  if (!s.found || n_in != k_rem) {
    if (threadIdx.x == 0 && blockIdx.x == 0) atomicOr(args.error, kDevErrBadInput);
    ok = false;
  }
  return prefix << digit_shift(level);
}

__global__ void __launch_bounds__(kSelThreads, 1)
    topk_select_kernel(float* __restrict__ e, uint32_t d, uint32_t k,
                       uint32_t* __restrict__ idx_out, float* __restrict__ val_out,
                       uint32_t* __restrict__ count_out, TopkArgs args) {
  extern __shared__ __align__(16) uint32_t s_mag[];
  __shared__ uint32_t s_hist[kHistBins];
  __shared__ uint32_t s_w[kSelThreads / 32];
  griddep_wait();  // the streaming pass (and all before it) is complete
  const SourceInfo si = read_source(args, d, k);
  if (k == 0 || si.failed) {
    if (blockIdx.x == 0 && threadIdx.x == 0) {
      if (si.failed) atomicOr(args.error, kDevErrTimeout);
      *count_out = 0;
      // nothing sent: every residual is a, all counted by the streaming pass
      if (args.err_out) *args.err_out = si.failed ? err_invalid() : *args.stream_err;
    }
    return;
  }
  if (si.mode == 0 && si.n <= kSmallCand) {
    // a few CTAs do the work: let the next kernel be scheduled on the rest of
    // the device (every kernel of this library waits for this grid before it
    // reads what this one writes; the whole grid's barriers are not used here)
    griddep_launch_dependents();
    const uint32_t Gs = min(gridDim.x, (si.n + kSliceElems - 1) / kSliceElems);
    if (blockIdx.x >= Gs) return;
    if (blockIdx.x == 0) {
      SmallSelection sel;
      const bool found = small_threshold(args, si.n, k, s_mag, s_hist, s_w, sel);
      if (threadIdx.x == 0) {
        if (found) {
          args.sel[1] = sel.B;
          args.sel[2] = sel.ties;
          args.sel[3] = sel.last;
        } else {
          atomicOr(args.error, kDevErrBadInput);
        }
        __threadfence();
        st_release_u32(args.sel, found ? 1u : 2u);
      }
      if (args.err_out) {
        // the candidates not sent keep a: their squares, plus the streaming
        // pass's share (every coordinate below the bound)
        ErrAcc acc;
        if (found)
          for (uint32_t i = threadIdx.x; i < si.n; i += kSelThreads)
            if (!selected(sel, s_mag[i], i)) acc.add(__uint_as_float(s_mag[i]));
        acc.flush();
        __shared__ FF s_d[32];
        const FF rem = block_sum_ff(acc.total, s_d);
        if (threadIdx.x == 0)
          *args.err_out = found ? *args.stream_err + ff_to_double(rem) : err_invalid();
      }
    }
    small_emit(args, e, si.n, k, Gs, idx_out, val_out, count_out, s_w);
    return;
  }
  bool ok = true;
  const uint64_t thr = radix_threshold_grid(args, e, si, k, s_hist, s_w, ok);
  if (!ok) {
    if (blockIdx.x == 0 && threadIdx.x == 0) {
      *count_out = 0;
      if (args.err_out) *args.err_out = err_invalid();
    }
    return;
  }
  // ordered compaction across the grid: chunk counts, then positions
  const uint32_t G = gridDim.x, c = blockIdx.x;
  const uint32_t lo = static_cast<uint32_t>(static_cast<uint64_t>(c) * si.n / G);
  const uint32_t hi = static_cast<uint32_t>(static_cast<uint64_t>(c + 1) * si.n / G);
  uint32_t mine = 0;
  ErrAcc acc;  // squares of the source positions not sent (their residual is a)
  for (uint32_t i0 = lo + threadIdx.x; i0 < hi; i0 += 4 * kSelThreads) {
    uint64_t key[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {  // loads in flight together
      const uint32_t i = i0 + j * kSelThreads;
      key[j] = i < hi ? source_key(args, e, si.mode, i) : 0ull;
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const bool in = i0 + j * kSelThreads < hi;
      mine += (in && key[j] >= thr) ? 1u : 0u;
      if (args.err_out && in && key[j] < thr)
        acc.add(__uint_as_float(static_cast<uint32_t>(key[j] >> 32)));
    }
  }
  uint32_t total;
  block_exclusive<kSelThreads>(mine, total, s_w);
  if (args.err_out) {
    acc.flush();
    __shared__ FF s_d[32];
    const FF share = block_sum_ff(acc.total, s_d);
    if (threadIdx.x == 0) {
      args.err_parts[c] = share;  // visible before the chunk total
      __threadfence();
    }
  }
  if (threadIdx.x == 0)
    st_relaxed_u64(args.chunk_sums + c, (static_cast<uint64_t>(args.epoch) << 32) | total);
  uint32_t base = 0;
  {
    const uint64_t t0 = global_timer_ns();
    uint32_t it = 0;
    while (true) {
      uint32_t part = 0;
      bool present = true;
      for (uint32_t q = threadIdx.x; q < c; q += kSelThreads) {
        const uint64_t w = ld_relaxed_u64(args.chunk_sums + q);
        if (static_cast<uint32_t>(w >> 32) == args.epoch)
          part += static_cast<uint32_t>(w);
        else
          present = false;
      }
      const bool all_present = __syncthreads_and(present);
      uint32_t sum;
      block_exclusive<kSelThreads>(part, sum, s_w);
      if (all_present) {
        base = sum;
        if (args.err_out && c == G - 1) {
          // every earlier CTA's share was written before its chunk total;
          // with candidates, the coordinates below the bound are the
          // streaming pass's (a full-array source covers every coordinate)
          __threadfence();
          __syncthreads();
          __shared__ FF s_d2[32];
          const FF shares = sum_parts_ff(args.err_parts, G, s_d2);
          if (threadIdx.x == 0)
            *args.err_out = (si.mode == 0 ? *args.stream_err : 0.0) + ff_to_double(shares);
        }
        break;
      }
      const bool out_of_time = ++it > (1u << 26) || global_timer_ns() - t0 > args.wait_limit_ns;
      if (__syncthreads_or(out_of_time)) {
        if (threadIdx.x == 0) atomicOr(args.error, kDevErrTimeout);
        return;
      }
      __nanosleep(64);
    }
  }
  bool overflow = false;
  const uint32_t written =
      write_selected(args, e, si.mode, lo, hi, thr, base, k, idx_out, val_out, overflow, s_w);
  if (c == G - 1 && threadIdx.x == 0) {
    const uint32_t end = base + written;
    *count_out = end < k ? end : k;
  }
  if (__syncthreads_or(overflow) && threadIdx.x == 0) atomicOr(args.error, kDevErrOverflow);
}

template <typename GT>
int tk_group_blocks_per_sm() {
  const void* fn =
      reinterpret_cast<const void*>(&lookback_stream_kernel<TopkCandOp<GT>, kTkStages>);
  const uint32_t smem = LbLayout<TopkCandOp<GT>, kTkStages>::kSmem;
  int n = 0;
  if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess ||
      cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, fn, kLbThreads, smem) != cudaSuccess)
    n = 0;
  cudaGetLastError();
  return n;
}

template <typename GT>
int tk_stream_blocks_per_sm() {
  const void* fn = reinterpret_cast<const void*>(&stream_compact_kernel<TopkCandOp<GT>, kTkStages>);
  const uint32_t smem = StreamLayout<TopkCandOp<GT>, kTkStages>::kSmem;
  int n = 0;
  if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess ||
      cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, fn, kStreamThreads, smem) != cudaSuccess)
    n = 0;
  cudaGetLastError();
  return n;
}

template <typename GT>
cudaError_t launch_typed(const GT* g, float* e, float gamma, uint32_t k, uint32_t d,
                         uint32_t* idx_out, float* val_out, uint32_t* count_out, double* err_out,
                         Workspace& ws, const DeviceInfo& dev) {
  const uint32_t tiles = tiles_for(d);
  cudaError_t err = cudaSuccess;
  // this call's zeroed state block, and the other one, cleared for the next call
  uint32_t* state = ws.topk_state(ws.topk_calls);
  uint32_t* other = ws.topk_state(ws.topk_calls + 1);
  ++ws.topk_calls;

  TopkArgs args;
  args.hist = state + kStHist / 4;
  args.cand0 = ws.cand(1);
  args.cand1 = ws.cand(2);
  args.list_idx = reinterpret_cast<uint32_t*>(ws.cand(0));
  args.list_val = reinterpret_cast<float*>(args.list_idx + ws.cand_cap);
  args.cand_count = state + kStCandCount / 4;
  args.cand_cap = ws.cand_cap;
  args.lower_bound = reinterpret_cast<uint64_t*>(state + kStLowerBound / 4);
  args.mode = state + kStMode / 4;
  args.sel = state + kStSelect / 4;
  args.list_count = ws.u32(kOffTkListCount);
  args.list_flags = state + kStListFlags / 4;
  args.bar_arrive = ws.u32(kOffBarArrive);
  args.bar_gen = ws.u32(kOffBarGen);
  args.error = ws.u32(kOffError);
  args.chunk_sums = ws.chunks();
  args.wait_limit_ns = wait_limit_ns();
  args.err_out = err_out;
  args.stream_err = ws.stream_err();
  args.err_parts = ws.errparts();

  // 1 sample + 2 stream (candidates). The bulk copies need 16-byte
  // aligned g and e; otherwise a plain pass writes a and the selection runs in
  // the full-array mode.
  ScanCtx ctx = next_scan_ctx(ws, tiles);
  ctx.error = args.list_flags;
  const int per_sm = sizeof(GT) == 4 ? dev.tk_stream_per_sm_f32 : dev.tk_stream_per_sm_bf16;
  const int per_sm_groups =
      sizeof(GT) == 4 ? dev.tk_group_per_sm_f32 : dev.tk_group_per_sm_bf16;
  const bool streamable = reinterpret_cast<uintptr_t>(e) % 16 == 0 &&
                          reinterpret_cast<uintptr_t>(g) % 16 == 0 && per_sm > 0;
  if (streamable) {
    TopkCandOp<GT> op{g, e, gamma, d, k, ws.cand_cap, state + kStSampleHist / 4,
                      state + kStStreamArrive / 4, args.mode, args.lower_bound, other};
    uint32_t slots = static_cast<uint32_t>(per_sm * dev.sm_count);
    if (slots > kMaxChunks) slots = kMaxChunks;
    const uint32_t grid = tiles < slots ? tiles : slots;
    uint32_t cap = ws.cand_cap;
    StreamArgs sa{ws.stage_idx(), ws.stage_val(), ws.counts(), ws.chunks(), nullptr,
                  err_out ? ws.stream_err() : nullptr, ws.errparts()};
    void* params[] = {&op, &d, &args.list_idx, &args.list_val, &args.list_count, &cap, &ctx, &sa};
    // the bound first (a small kernel without waits), then the streaming
    // pass, whose CTAs only wait for lower-numbered ones: plain launches
    uint32_t tiles_arg = tiles;
    void* sp[] = {&op, &tiles_arg};
    err = launch_pdl(reinterpret_cast<const void*>(&topk_sample_kernel<GT>), grid, kStreamThreads,
                     0, ws.stream, sp, false);
    count_launch();
    if (err != cudaSuccess) return err;
    if (use_group_kernel(tiles) && per_sm_groups > 0) {
      // claimed groups of tiles with look-back (stream_lookback.cuh): no
      // wait depends on which CTAs are resident
      const uint32_t groups = (tiles + kLbGroupTiles - 1) / kLbGroupTiles;
      const uint32_t gslots = static_cast<uint32_t>(per_sm_groups * dev.sm_count);
      const uint32_t ggrid = groups < gslots ? groups : gslots;
      LbArgs la{nullptr, err_out ? ws.stream_err() : nullptr, reinterpret_cast<FF*>(ws.counts()),
                ws.stage_idx(), ws.stage_val()};
      void* gp[] = {&op, &d, &args.list_idx, &args.list_val, &args.list_count, &cap, &ctx, &la};
      err = launch_pdl(
          reinterpret_cast<const void*>(&lookback_stream_kernel<TopkCandOp<GT>, kTkStages>),
          ggrid, kLbThreads, LbLayout<TopkCandOp<GT>, kTkStages>::kSmem, ws.stream, gp, false);
    } else {
      err = launch_pdl(
          reinterpret_cast<const void*>(&stream_compact_kernel<TopkCandOp<GT>, kTkStages>), grid,
          kStreamThreads, StreamLayout<TopkCandOp<GT>, kTkStages>::kSmem, ws.stream, params,
          false);
    }
    count_launch();
    if (err != cudaSuccess) return err;
  } else {
    const uint32_t grid = tiles < static_cast<uint32_t>(dev.sm_count * 8)
                              ? tiles : static_cast<uint32_t>(dev.sm_count * 8);
    topk_accumulate_plain_kernel<GT><<<grid, kThreads, 0, ws.stream>>>(g, e, gamma, d, args,
                                                                       other);
    count_launch();
    if ((err = cudaGetLastError()) != cudaSuccess) return err;
  }
  // 3 select (inputs the streaming pass could not take: the norm by a plain pass after it)
  if (!streamable) args.err_out = nullptr;
  args.epoch = next_scan_ctx(ws, 1).epoch;
  void* params[] = {(void*)&e, (void*)&d, (void*)&k, (void*)&idx_out, (void*)&val_out,
                    (void*)&count_out, (void*)&args};
  uint32_t grid = static_cast<uint32_t>(dev.refine_blocks);
  if (grid > kMaxChunks) grid = kMaxChunks;
  // (cooperative, for the reason given for the stream: grid barriers)
  err = launch_pdl(reinterpret_cast<const void*>(&topk_select_kernel), grid, kSelThreads,
                   kSelSmem, ws.stream, params, true);
  count_launch();
  if (err == cudaSuccess && err_out && !streamable) err = launch_error_norm(e, d, err_out, ws, dev);
  return err;
}

}  // namespace

void topk_init_device(DeviceInfo& info) {
  int a = 0;
  cudaFuncSetAttribute(topk_select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSelSmem);
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&a, topk_select_kernel, kSelThreads, kSelSmem);
  info.refine_blocks = a * info.sm_count;
  info.finalize_blocks = info.refine_blocks;
  info.tk_stream_per_sm_f32 = tk_stream_blocks_per_sm<float>();
  info.tk_stream_per_sm_bf16 = tk_stream_blocks_per_sm<uint16_t>();
  info.tk_group_per_sm_f32 = tk_group_blocks_per_sm<float>();
  info.tk_group_per_sm_bf16 = tk_group_blocks_per_sm<uint16_t>();
  cudaGetLastError();
}

uint32_t topk_candidate_capacity(uint64_t d) {
  const uint64_t floor_cap = 1u << 20;
  uint64_t cap = d / 16 > floor_cap ? d / 16 : floor_cap;
  if (cap > d) cap = d;
  if (cap == 0) cap = 1;
  return static_cast<uint32_t>(cap);
}

cudaError_t launch_topk(const void* g, bool g_bf16, float* e, float gamma, uint32_t k,
                        uint32_t d, uint32_t* idx_out, float* val_out, uint32_t* count_out,
                        double* err_out, Workspace& ws, const DeviceInfo& dev) {
  if (g_bf16)
    return launch_typed(static_cast<const uint16_t*>(g), e, gamma, k, d, idx_out, val_out,
                        count_out, err_out, ws, dev);
  return launch_typed(static_cast<const float*>(g), e, gamma, k, d, idx_out, val_out, count_out,
                      err_out, ws, dev);
}

}  // namespace efs
