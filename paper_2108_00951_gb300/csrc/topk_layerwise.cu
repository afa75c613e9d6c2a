// topk_layerwise.cu — error feedback with layer-wise Top-k: the vector is a
// concatenation of tensors (segments), and the Top-k sparsifier runs on each
// segment separately with its own k_s (the paper's experiments compress
// layer by layer, Sec. 6 and the Appendix on layer-wise compression). The
// sent pairs of segment s fill output positions [K_s, K_s + k_s), with
// K_s = k_0 + ... + k_{s-1}, in ascending index; ties in magnitude go to the
// lower index, NaN ranks above +inf (the entire-vector Top-k rules applied
// within each segment).
//
// Three launches, whatever the number of segments:
//  1 sample   one CTA for each segment longer than kLwWholeMax with
//             0 < k_s < d_s (up to kLwMaxParts for a long one with a small
//             k_s, each over an equal run of it, their histograms merged)
//             reads up to 4096 groups of 4 consecutive coordinates spread
//             evenly over it (all of them when it holds no more), histograms
//             the top 15 magnitude bits of a = fmaf(γ,g,e) in shared memory
//             and picks the candidate bound: the bin holding k_s samples when
//             every group was read, else about 1.5 times the needed mass
//             above it.
//  2 stream   the streaming compaction (stream_compact.cuh, or from 4096
//             tiles on stream_lookback.cuh): a = fmaf(γ,g,e)
//             is written over e (12 B per coordinate, the algorithmic bytes)
//             and the coordinates at or above their segment's bound are
//             emitted as one ordered candidate list, with the list position
//             of each tile's first candidate.
//  3 select   CTAs own groups of segments (balanced on the host). For each:
//             a short segment is read into shared memory whole; a longer one
//             takes its candidates (located from the tile positions) into
//             shared memory, or reads them (or, if the bound missed, the
//             segment) from global memory level by level; the exact
//             threshold follows from digit levels over the magnitudes, and
//             the pairs are written in order with e zeroed at each.
// The bound is only a filter: a segment whose candidates are fewer than k_s,
// or were cut off at the list's capacity, is selected from e itself, so the
// result is exact whatever the sample saw.
#include <algorithm>
#include <cstring>
#include <functional>
#include <queue>

#include "gradient.cuh"
#include "internal.h"
#include "select.cuh"
#include "stream_lookback.cuh"

namespace efs {
namespace {

constexpr int kLwThreads = 1024;  // select CTAs
constexpr uint32_t kLwSelectSmem = kLwSmemElems * sizeof(uint32_t);
constexpr int kLwSampleShift = 31 - kLwSampleBits;  // magnitude bits below the sampled ones
constexpr uint32_t kLwSampleSmem = kLwSampleBins * sizeof(uint32_t);  // the CTA's histogram
constexpr int kLwStages = 4;

__device__ __forceinline__ uint32_t mag_bits(float x) { return __float_as_uint(x) & 0x7fffffffu; }

// ------------------------------------------------------------- 1 sample
// One CTA per sampled segment or part of one (a part: an equal run of the
// segment's aligned groups, sampled the same way; the parts' histograms are
// merged in global memory), one round of loads: thread t reads groups
// t, t + 1024, t + 2048, t + 3072 of the segment's G <= 4096 groups of 4
// consecutive coordinates starting at multiples of 4 (one 16-byte load each
// of e and of an fp32 g, 8 bytes of a bf16 g). Group q starts at
// a0 + 4 floor(q step), a0 the first aligned coordinate inside the segment,
// step = (A - 1) / (G - 1) rounded down in 32.32 fixed point and A the
// aligned groups the segment holds (so the last group stays inside it);
// G == A samples every one.
//
// Programmatic dependent launch: the loads, the histogram and the parts'
// merge may run while the previous kernel on the stream finishes (a sample
// read before that kernel's writes only changes the bound, which is a
// filter); the bound is written after the wait, so no earlier reader of it
// sees the new one.
constexpr int kSampleThreads = 1024;

template <typename GT>
__global__ void __launch_bounds__(kSampleThreads, 1)
    lw_sample_kernel(const GT* __restrict__ g, const float* __restrict__ e, float gamma,
                     const LwSeg* __restrict__ segs, const uint2* __restrict__ sampled,
                     uint32_t* mbound, uint32_t cand_cap, uint32_t* part_hist) {
  extern __shared__ uint32_t s_hist[];  // [kLwSampleBins]
  __shared__ uint32_t s_w[kSampleThreads / 32];
  __shared__ uint32_t s_bin, s_mass, s_last;
  const int tid = threadIdx.x;
  griddep_launch_dependents();  // the stream pass may be scheduled (it waits for this grid)
  // this CTA's part of the segment: part `part` of `parts` equal runs of its
  // aligned groups (one part: the host's sampling plan), with merge slot `slot`
  const uint2 rec = sampled[blockIdx.x];
  const uint32_t si = rec.x, part = rec.y & 0xffu, parts = (rec.y >> 8) & 0xffu,
                 slot = rec.y >> 16;
  LwSeg s = segs[si];
  for (uint32_t b = tid; b < kLwSampleBins; b += kSampleThreads) s_hist[b] = 0;
  uint64_t a0 = (static_cast<uint64_t>(s.lo) + 3u) & ~static_cast<uint64_t>(3);
  if (parts > 1) {
    const uint64_t avail = (static_cast<uint64_t>(s.hi) - a0) / 4;  // whole groups inside
    const uint64_t g0 = part * avail / parts, g1 = (part + 1) * avail / parts;
    const uint64_t n = g1 - g0;
    s.groups = static_cast<uint32_t>(n < kLwSampleGroups ? n : kLwSampleGroups);
    s.step = s.groups > 1 ? ((n - 1) << 32) / (s.groups - 1) : 0;
    s.exact = 0;
    a0 += 4 * g0;
  }
  constexpr int kG = static_cast<int>(kLwSampleGroups / kSampleThreads);
  GradVec<GT> gv[kG];
  float4 ev[kG];
  bool in[kG];
#pragma unroll
  for (int q = 0; q < kG; ++q) {  // every load in flight before any use
    const uint32_t qq = q * kSampleThreads + tid;
    in[q] = qq < s.groups;
    const uint64_t p = a0 + 4u * ((static_cast<uint64_t>(in[q] ? qq : 0u) * s.step) >> 32);
    if (in[q]) {
      if constexpr (sizeof(GT) == 4)
        gv[q].v = __ldg(reinterpret_cast<const float4*>(g + p));
      else
        gv[q].v = __ldg(reinterpret_cast<const uint2*>(g + p));
      ev[q] = __ldg(reinterpret_cast<const float4*>(e + p));
    }
  }
  __syncthreads();
#pragma unroll
  for (int q = 0; q < kG; ++q) {
    const float x[4] = {in[q] ? __fmaf_rn(gamma, gv[q][0], ev[q].x) : 0.0f,
                        in[q] ? __fmaf_rn(gamma, gv[q][1], ev[q].y) : 0.0f,
                        in[q] ? __fmaf_rn(gamma, gv[q][2], ev[q].z) : 0.0f,
                        in[q] ? __fmaf_rn(gamma, gv[q][3], ev[q].w) : 0.0f};
#pragma unroll
    for (int j = 0; j < 4; ++j)
      if (in[q]) atomicAdd(&s_hist[mag_bits(x[j]) >> kLwSampleShift], 1u);
  }
  __syncthreads();
  if (parts > 1) {
    // add the part's histogram to the segment's merged one; the last part to
    // arrive takes the merged histogram, leaves it at zero, and goes on. No
    // wait first (the merge stays off the call's critical path): the copy of
    // this call's parity (two alternate) was left at zero by the last
    // sampling that used it, an earlier call's, and that grid is complete
    // before this one starts: each call's select waits for its stream pass,
    // which waits for the call's sampling, before it lets a later kernel start
    uint32_t* gh = part_hist + static_cast<size_t>(slot) * kLwPartHistWords;
    for (uint32_t b = tid; b < kLwSampleBins; b += kSampleThreads)
      if (s_hist[b]) atomicAdd(&gh[b], s_hist[b]);
    __syncthreads();
    if (tid == 0) {
      __threadfence();
      s_last = atomicAdd(&gh[kLwSampleBins], 1u) == parts - 1 ? 1u : 0u;
      if (s_last) __threadfence();  // the other parts' adds before the reads
    }
    __syncthreads();
    if (!s_last) return;
    constexpr int kBatch = 8;  // loads in flight per thread
    for (uint32_t b0 = tid; b0 < kLwSampleBins; b0 += kBatch * kSampleThreads) {
      uint32_t v[kBatch];
#pragma unroll
      for (int j = 0; j < kBatch; ++j) v[j] = __ldcg(&gh[b0 + j * kSampleThreads]);
#pragma unroll
      for (int j = 0; j < kBatch; ++j) {
        s_hist[b0 + j * kSampleThreads] = v[j];
        gh[b0 + j * kSampleThreads] = 0;
      }
    }
    if (tid == 0) gh[kLwSampleBins] = 0;
    __syncthreads();
  }
  // kPer consecutive bins per thread, summed in a lane-rotated order (no
  // two lanes of a warp on one bank)
  constexpr int kPer = static_cast<int>(kLwSampleBins) / kSampleThreads;
  static_assert(kPer == 32, "bins per thread: one per bank");
  const int lane = tid & 31;
  uint32_t mine = 0;
#pragma unroll
  for (int i = 0; i < kPer; ++i) mine += s_hist[tid * kPer + ((i + lane) & (kPer - 1))];
  if (tid == 0) s_bin = 0xffffffffu;
  uint32_t m;  // sampled coordinates
  const uint32_t above = block_suffix_exclusive(mine, m, s_w);  // orders the reset
  const uint64_t ds = s.hi - s.lo;
  // Every sampled coordinate is a coordinate of the segment, so at least
  // `target` coordinates lie at or above the bin found. With every group
  // sampled, target = k_s is therefore enough; otherwise 1.5x the expected
  // sampled count above the k_s-th magnitude, plus 32 (integer arithmetic;
  // the products stay below 2^50).
  const uint64_t target = s.exact ? s.k : 3ull * s.k * m / (2ull * ds) + 32ull;
  if (target <= m && above < target && target - above <= mine) {
    // the one thread whose bins hold the target walks them from the top
    uint64_t run = above;
    for (int i = kPer - 1; i >= 0; --i) {
      const uint32_t c = s_hist[tid * kPer + i];
      run += c;
      if (run >= target) {
        s_bin = tid * kPer + i;
        s_mass = static_cast<uint32_t>(run);
        break;
      }
    }
  }
  __syncthreads();
  griddep_wait();  // the previous kernel (which may read the bounds) is complete
  if (tid == 0) {
    uint32_t bound = kLwDeferred;
    // expected candidates (the sampled mass scaled to d_s) at most half the
    // list's capacity, else the segment is selected from e itself
    if (s_bin != 0xffffffffu &&
        2ull * s_mass * ds <= static_cast<uint64_t>(cand_cap) * m)
      bound = s_bin << kLwSampleShift;
    mbound[si] = bound;
  }
}

// ------------------------------------------------------------- 2 stream
// The streaming pass as a stream_compact op: a stage holds a tile of g then
// the same tile of e; a is written over e from registers, and a coordinate
// is a candidate when its magnitude bits reach its segment's bound.
template <typename GT>
struct LwCandOp {
  const GT* g;
  float* e;
  float gamma;
  uint32_t d;
  const uint32_t* seg_end;    // [n_seg] exclusive segment ends
  const uint32_t* mbound;     // [n_seg] candidate bounds (kLwNoBound, kLwDeferred: none)
  const uint32_t* tile_info;  // [tiles] first segment of the tile | kLwTileUniform
  uint32_t* other_state;      // the other Top-k state block: zeroed here for the next call
  static constexpr uint32_t kGBytes = kTileElems * sizeof(GT);
  static constexpr uint32_t kStageBytes = kGBytes + kTileElems * sizeof(float);
  static constexpr uint32_t kWarpStagePairs = 512;  // on-chip staged pairs per compute warp
  static constexpr bool kKeepPairs = true;  // the candidate list: the select reads it next
  __device__ void prologue() const { clear_state(other_state); }
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

  // selection bits of the lane's coordinates from their segments' bounds
  // (bit j: candidate; bit 4 + j: residual decided by the select)
  __device__ __forceinline__ void select(uint32_t t, uint64_t first, const float (&a)[kSUnits][4],
                                         uint32_t (&sel)[kSUnits]) const {
    const uint32_t info = __ldg(tile_info + t);
    if (info & kLwTileUniform) {
      const uint32_t b = __ldg(mbound + (info & ~kLwTileUniform));
      const uint32_t defer = b == kLwDeferred ? 0xf0u : 0u;
#pragma unroll
      for (int v = 0; v < kSUnits; ++v) {
        sel[v] = defer;
#pragma unroll
        for (int j = 0; j < 4; ++j) sel[v] |= (mag_bits(a[v][j]) >= b ? 1u : 0u) << j;
      }
    } else {
      uint32_t s = info;  // the tile's first segment; coordinates ascend below
#pragma unroll
      for (int v = 0; v < kSUnits; ++v) {
        sel[v] = 0;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const uint64_t i = first + v * 128 + j;
          if (i < d) {
            while (__ldg(seg_end + s) <= i) ++s;
            const uint32_t b = __ldg(mbound + s);
            sel[v] |= (mag_bits(a[v][j]) >= b ? 1u : 0u) << j;
            sel[v] |= (b == kLwDeferred ? 1u : 0u) << (4 + j);
          }
        }
      }
    }
  }

  __device__ __forceinline__ void tile_smem(const unsigned char* stage, uint32_t t, int warp,
                                            int lane, float (&a)[kSUnits][4],
                                            uint32_t (&sel)[kSUnits], uint64_t) const {
    const GT* gs = reinterpret_cast<const GT*>(stage);
    const float* es = reinterpret_cast<const float*>(stage + kGBytes);
    const int local = warp * kSWarpElems + lane * 4;
    const uint64_t first = stream_element_index(t, warp, 0, lane, 0);
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
      st_stream_f4(e + first + v * 128, make_float4(a[v][0], a[v][1], a[v][2], a[v][3]));
    }
    select(t, first, a, sel);
  }

  __device__ __forceinline__ void tile_global(uint32_t t, int warp, int lane,
                                              float (&a)[kSUnits][4],
                                              uint32_t (&sel)[kSUnits], uint64_t) const {
    const uint64_t first = stream_element_index(t, warp, 0, lane, 0);
#pragma unroll
    for (int v = 0; v < kSUnits; ++v) {
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const uint64_t i = first + v * 128 + j;
        a[v][j] = 0.0f;
        if (i < d) {
          const float x = __fmaf_rn(gamma, grad_scalar(g, i), e[i]);
          e[i] = x;
          a[v][j] = x;
        }
      }
    }
    select(t, first, a, sel);
    // lanes past d select nothing (their a is 0 but their segment is unknown)
#pragma unroll
    for (int v = 0; v < kSUnits; ++v)
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (first + v * 128 + j >= d) sel[v] &= ~(0x11u << j);
  }
};

// Inputs the bulk copies cannot take (not 16-byte aligned): a = fmaf(γ,g,e)
// written over e with plain loads; every segment is then selected from e.
template <typename GT>
__global__ void __launch_bounds__(kThreads)
    lw_accumulate_plain_kernel(const GT* __restrict__ g, float* __restrict__ e, float gamma,
                               uint32_t d, uint32_t* other_state) {
  clear_state(other_state);
  for (uint64_t i = static_cast<uint64_t>(blockIdx.x) * kThreads + threadIdx.x; i < d;
       i += static_cast<uint64_t>(gridDim.x) * kThreads)
    e[i] = __fmaf_rn(gamma, grad_scalar(g, i), e[i]);
}

// ------------------------------------------------------------- 3 select
struct LwArgs {
  const LwSeg* segs;
  const uint32_t* mbound;
  const LwCta* ctas;          // [grid] what each CTA selects
  const uint32_t* work_seg;   // segment ids of the single CTAs, grouped by CTA
  LwTeamState* teams;
  const uint32_t* tile_base;  // [tiles + 1] list position of each tile's first candidate
  const uint32_t* list_idx;   // ordered candidates of the streaming pass
  const float* list_val;
  const uint32_t* list_flags; // that pass's latched bits
  uint32_t* error;
  uint32_t* count_out;
  uint64_t wait_limit_ns;
  uint32_t tiles, cap, use_list;
  uint32_t total_k;
  double* err_out;            // optional ||e'||^2 of the step
  const double* stream_err;   // the streaming pass's share (final residuals)
  FF* err_parts;              // [gridDim.x] the select CTAs' shares
  uint32_t* err_arrive;       // select CTAs that published their share (zero at the start)
};

// The source a segment is selected from: its candidates [c0, c1) of the
// list when they are complete and at least k_s, else its coordinates of a
// (held in e after the stream). The list positions of lo and hi are the
// positions of their tiles' first candidates plus those tiles' candidates
// below them; all four tile positions are loaded at once, then both tiles
// scanned together. Whole CTA; every CTA of a team decides alike.
struct Source {
  bool list;
  uint32_t c0, n;
};
__device__ Source segment_source(const LwArgs& a, const LwSeg& s, uint32_t si) {
  Source src{false, 0, s.hi - s.lo};
  if (!a.use_list || __ldcg(a.mbound + si) >= kLwDeferred) return src;
  const uint32_t tl = s.lo / kTileElems, th = s.hi / kTileElems;  // tl < tiles, th <= tiles
  const uint32_t p0 = __ldcg(a.tile_base + tl), p1 = __ldcg(a.tile_base + tl + 1);
  const uint32_t q0 = __ldcg(a.tile_base + th);
  const uint32_t q1 = th < a.tiles ? __ldcg(a.tile_base + th + 1) : q0;
  // candidates of the partial tiles that lie below lo / hi (none to scan
  // when lo / hi starts a tile); a tile cut off at the capacity disqualifies
  const uint32_t e0 = s.lo % kTileElems ? p1 : p0, e1 = s.hi % kTileElems ? q1 : q0;
  if (e0 > a.cap || e1 > a.cap) return src;
  const uint32_t n0 = e0 - p0, n1 = e1 - q0, span = n0 > n1 ? n0 : n1;
  uint32_t below0 = 0, below1 = 0;
  for (uint32_t b = 0; b < span; b += kLwThreads) {
    const uint32_t i = b + threadIdx.x;
    const bool x0 = i < n0 && __ldcg(a.list_idx + p0 + i) < s.lo;
    const bool x1 = i < n1 && __ldcg(a.list_idx + q0 + i) < s.hi;
    below0 += __syncthreads_count(x0);
    below1 += __syncthreads_count(x1);
  }
  const uint32_t c0 = p0 + below0, c1 = q0 + below1;
  if (c1 <= a.cap && c1 - c0 >= s.k) src = Source{true, c0, c1 - c0};
  return src;
}

// Reads n fp32 values (8 loads in flight per thread), keeps their bits in
// s_bits when it is given (and the coordinates idx[0, n) in s_idx when both
// are given), and returns the minimum and maximum magnitude.
__device__ void load_minmax(const float* src, uint32_t n, uint32_t* s_bits, uint32_t& lo,
                            uint32_t& hi, uint32_t* s_lo, uint32_t* s_hi,
                            const uint32_t* idx = nullptr, uint32_t* s_idx = nullptr) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  constexpr int kBatch = 8;
  lo = 0xffffffffu;
  hi = 0;
  const bool with_idx = idx && s_idx;
  for (uint32_t i0 = tid; i0 < n; i0 += kBatch * kLwThreads) {
    uint32_t v[kBatch], x[kBatch];
#pragma unroll
    for (int j = 0; j < kBatch; ++j) {
      const uint32_t i = i0 + j * kLwThreads;
      v[j] = i < n ? __float_as_uint(__ldcg(src + i)) : 0u;
      x[j] = with_idx && i < n ? __ldcg(idx + i) : 0u;
    }
#pragma unroll
    for (int j = 0; j < kBatch; ++j) {
      const uint32_t i = i0 + j * kLwThreads;
      if (i < n) {
        if (s_bits) s_bits[i] = v[j];
        if (with_idx) s_idx[i] = x[j];
        const uint32_t m = v[j] & 0x7fffffffu;
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
  __syncthreads();  // an earlier use of s_lo / s_hi is complete
  if (lane == 0) {
    s_lo[warp] = lo;
    s_hi[warp] = hi;
  }
  __syncthreads();
  lo = lane < kLwThreads / 32 ? s_lo[lane] : 0xffffffffu;
  hi = lane < kLwThreads / 32 ? s_hi[lane] : 0u;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    lo = min(lo, __shfl_xor_sync(0xffffffffu, lo, o));
    hi = max(hi, __shfl_xor_sync(0xffffffffu, hi, o));
  }
}

// Sources of a selection: source position i has value bits bits(i) and
// coordinate index(i).
struct SrcShared {  // values in shared memory; coordinates lo + i, or from a list
  const uint32_t* s_bits;
  const uint32_t* idx;    // null: coordinates lo + i (or from s_idx)
  const uint32_t* s_idx;  // the list's coordinates in shared memory, or null
  uint32_t lo;
  __device__ __forceinline__ uint32_t bits(uint32_t i) const { return s_bits[i]; }
  __device__ __forceinline__ uint32_t index(uint32_t i) const {
    return s_idx ? s_idx[i] : idx ? __ldcg(idx + i) : lo + i;
  }
};
struct SrcGlobal {  // values in global memory; coordinates lo + i, or from a list
  const float* val;
  const uint32_t* idx;
  uint32_t lo;
  __device__ __forceinline__ uint32_t bits(uint32_t i) const {
    return __float_as_uint(__ldcg(val + i));
  }
  __device__ __forceinline__ uint32_t index(uint32_t i) const {
    return idx ? __ldcg(idx + i) : lo + i;
  }
};

// Ordered write-out of the selected source positions of [s0, s1), in two
// passes (the first also adds the squares of the positions not sent, with
// magnitude bits >= err_from, to *err when it is given). Warp w owns the contiguous part [s0 + w (s1-s0)/32, ...): it counts
// its selected positions (coalesced loads, 4 in flight per lane); the CTA's
// counts are scanned (plus `base`, the pairs of earlier CTAs of a team, which
// `publish` supplies once it sees the CTA's total; 0xffffffff: none, write
// nothing); then each warp writes its
// pairs at ascending positions with ballots, zeroing e at each. Positions at
// or past k are not written (overflow). Returns the CTA's count. Whole CTA.
template <class Src, class Publish>
__device__ uint32_t write_out(const Src& src, uint32_t s0, uint32_t s1, const SmallSelection& sel,
                              uint32_t k, uint32_t* idx_out, float* val_out, float* e,
                              bool& overflow, uint32_t* s_w, const Publish& publish,
                              ErrAcc* err, uint32_t err_from) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  constexpr int kNumWarps = kLwThreads / 32;
  const uint32_t len = s1 - s0;
  const uint32_t w0 = s0 + static_cast<uint32_t>(static_cast<uint64_t>(warp) * len / kNumWarps);
  const uint32_t w1 =
      s0 + static_cast<uint32_t>(static_cast<uint64_t>(warp + 1) * len / kNumWarps);
  uint32_t cnt = 0;
  for (uint32_t i0 = w0; i0 < w1; i0 += 4 * 32) {
    uint32_t b[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const uint32_t i = i0 + j * 32 + lane;
      b[j] = i < w1 ? src.bits(i) : 0u;
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const uint32_t i = i0 + j * 32 + lane;
      const uint32_t mg = b[j] & 0x7fffffffu;
      const bool take = i < w1 && selected(sel, mg, i);
      cnt += take ? 1u : 0u;
      // a position not sent keeps a; those at or above err_from are this
      // kernel's share of ||e'||^2 (the rest were counted while streaming)
      if (err && i < w1 && !take && mg >= err_from) err->add(__uint_as_float(b[j]));
    }
  }
  cnt = warp_sum(cnt);
  __syncthreads();  // an earlier use of s_w is complete
  if (lane == 0) s_w[warp] = cnt;
  __syncthreads();
  uint32_t before = 0, total = 0;
  for (int w = 0; w < kNumWarps; ++w) {
    const uint32_t x = s_w[w];
    before += w < warp ? x : 0u;
    total += x;
  }
  const uint32_t base = publish(total);
  if (base == 0xffffffffu) return total;  // the team's counts are unknown: write nothing
  const uint32_t lt = lanemask_lt();
  uint32_t pos = base + before;
  for (uint32_t i0 = w0; i0 < w1; i0 += 4 * 32) {
    uint32_t b[4], ix[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {  // values and coordinates in flight together
      const uint32_t i = i0 + j * 32 + lane;
      b[j] = i < w1 ? src.bits(i) : 0u;
      ix[j] = i < w1 ? src.index(i) : 0u;
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const uint32_t i = i0 + j * 32 + lane;
      const bool take = i < w1 && selected(sel, b[j] & 0x7fffffffu, i);
      const uint32_t bal = __ballot_sync(0xffffffffu, take);
      if (take) {
        const uint32_t q = pos + __popc(bal & lt);
        if (q < k) {
          const uint32_t idx = ix[j];
          idx_out[q] = idx;
          val_out[q] = __uint_as_float(b[j]);
          e[idx] = 0.0f;  // residual of a sent coordinate
        } else {
          overflow = true;
        }
      }
      pos += __popc(bal);
    }
  }
  return total;
}

struct NoTeam {
  __device__ uint32_t operator()(uint32_t) const { return 0; }
};

// One CTA selects segment s on its own. Returns false when the threshold
// was not found or the count differs from k (never for well-formed data).
// Where the streaming pass left a segment's residuals to the select: every
// position of a list source (candidates), and of an e source those at or above
// the bound the stream used (all of them without one).
__device__ __forceinline__ uint32_t err_from_for(const LwArgs& a, const LwSeg& s, uint32_t si,
                                                 bool list) {
  if (list || s.kind != kLwSampled) return 0u;
  const uint32_t b = __ldcg(a.mbound + si);
  return b >= kLwDeferred ? 0u : b;
}

__device__ bool select_single(const LwArgs& a, const LwSeg& s, uint32_t si, float* e,
                              uint32_t* idx_out, float* val_out, bool& overflow,
                              uint32_t* s_bits, uint32_t* s_hist, uint32_t* s_w, uint32_t* s_lo,
                              uint32_t* s_hi, ErrAcc* err) {
  uint32_t* io = idx_out + s.out;
  float* vo = val_out + s.out;
  const uint32_t ds = s.hi - s.lo;
  if (s.kind == kLwAll) {
    for (uint32_t i = threadIdx.x; i < ds; i += kLwThreads) {
      io[i] = s.lo + i;
      vo[i] = __ldcg(e + s.lo + i);
      e[s.lo + i] = 0.0f;
    }
    return true;
  }
  const Source src = s.kind == kLwWhole ? Source{false, 0, ds} : segment_source(a, s, si);
  const uint32_t err_from = err_from_for(a, s, si, src.list);
  const float* vals = src.list ? a.list_val + src.c0 : e + s.lo;
  const uint32_t* idxs = src.list ? a.list_idx + src.c0 : nullptr;
  SmallSelection sel;
  uint32_t lo, hi, got = 0;
  bool found;
  if (src.n <= kLwSmemElems) {
    // a list of at most half the capacity keeps its coordinates on chip too
    uint32_t* s_idx = idxs && src.n <= kLwSmemElems / 2 ? s_bits + kLwSmemElems / 2 : nullptr;
    load_minmax(vals, src.n, s_bits, lo, hi, s_lo, s_hi, idxs, s_idx);
    found = threshold_levels<kLwThreads>(MagsShared{s_bits}, src.n, s.k, lo, hi, s_hist, s_w, sel);
    if (found)
      got = write_out(SrcShared{s_bits, idxs, s_idx, s.lo}, 0, src.n, sel, s.k, io, vo, e,
                      overflow, s_w, NoTeam{}, err, err_from);
  } else {
    load_minmax(vals, src.n, nullptr, lo, hi, s_lo, s_hi);
    found = threshold_levels<kLwThreads>(MagsGlobal{vals}, src.n, s.k, lo, hi, s_hist, s_w, sel);
    if (found)
      got = write_out(SrcGlobal{vals, idxs, s.lo}, 0, src.n, sel, s.k, io, vo, e, overflow, s_w,
                      NoTeam{}, err, err_from);
  }
  return found && got == s.k;
}

// A team of T co-resident CTAs selects segment s: CTA r owns the source
// positions [r n / T, (r+1) n / T). The threshold is found by three digit
// levels of the magnitude bits (30..20, 19..10, 9..0): each CTA histograms
// the positions matching the prefix chosen so far into shared memory and adds
// that into the team's level histogram; after a team barrier every CTA reads
// the merged histogram and picks the same bin. The levels stop once the bin
// holds exactly the remaining rank; otherwise equal magnitudes at the last
// level are taken in position order (per-rank counts, a barrier, and the rank
// holding the cut publishes its position). The write-out scans per-rank
// counts behind one more barrier. Returns false on a barrier that ran out
// (latched as a timeout) or an inconsistent histogram.
__device__ bool select_team(const LwArgs& a, const LwSeg& s, uint32_t si, uint32_t T, uint32_t r,
                            LwTeamState* st, float* e, uint32_t* idx_out, float* val_out,
                            bool& overflow, bool& bad, uint32_t* s_hist, uint32_t* s_w,
                            ErrAcc* err) {
  __shared__ uint32_t s_found, s_last;
  const int tid = threadIdx.x;
  const Source src = segment_source(a, s, si);
  const uint32_t err_from = err_from_for(a, s, si, src.list);
  const float* vals = src.list ? a.list_val + src.c0 : e + s.lo;
  const uint32_t* idxs = src.list ? a.list_idx + src.c0 : nullptr;
  const MagsGlobal mag{vals};
  const uint32_t n = src.n;
  const uint32_t s0 = static_cast<uint32_t>(static_cast<uint64_t>(r) * n / T);
  const uint32_t s1 = static_cast<uint32_t>(static_cast<uint64_t>(r + 1) * n / T);
  auto barrier = [&]() {
    return group_barrier(&st->arrive, &st->gen, T, a.wait_limit_ns, a.error);
  };
  uint32_t prefix = 0, k_rem = s.k, n_in = n;
  int sh = 0;
  for (int level = 0; level < 3; ++level) {
    sh = level == 0 ? 20 : level == 1 ? 10 : 0;
    const int width = level == 0 ? 11 : 10;
    const uint32_t nb = 1u << width;
    for (uint32_t b = tid; b < nb; b += kLwThreads) s_hist[b] = 0;
    __syncthreads();
    for (uint32_t b0 = s0; b0 < s1; b0 += 4 * kLwThreads) {
      uint32_t m[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const uint32_t i = b0 + j * kLwThreads + tid;
        m[j] = i < s1 ? mag(i) : 0u;
      }
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const uint32_t i = b0 + j * kLwThreads + tid;
        const bool match = i < s1 && (level == 0 || (m[j] >> (sh + width)) == prefix);
        hist_add_warp(s_hist, (m[j] >> sh) & (nb - 1), match);
      }
    }
    __syncthreads();
    for (uint32_t b = tid; b < nb; b += kLwThreads)
      if (s_hist[b]) atomicAdd(&st->hist[level][b], s_hist[b]);
    if (!barrier()) return false;
    const Selection sl = select_bin<kLwThreads, true>(st->hist[level], nb, k_rem, s_w);
    if (!sl.found) {
      bad = true;
      return false;
    }
    prefix = (prefix << width) | sl.bin;
    k_rem = sl.k_rem;
    n_in = sl.n_in;
    if (n_in == k_rem) break;
  }
  SmallSelection sel{prefix << sh, 0u, 0xffffffffu};
  if (n_in != k_rem) {
    // sh == 0: the magnitude is prefix itself; take its first k_rem
    // occurrences in position order
    sel.ties = 1u;
    uint32_t c = 0;
    for (uint32_t i = s0 + tid; i < s1; i += kLwThreads) c += mag(i) == sel.B ? 1u : 0u;
    uint32_t mine;
    block_exclusive<kLwThreads>(c, mine, s_w);
    if (tid == 0) st->tie_cnt[r] = mine;
    if (!barrier()) return false;
    uint32_t before = 0;
    for (uint32_t q = 0; q < r; ++q) before += __ldcg(&st->tie_cnt[q]);
    if (before < k_rem && k_rem <= before + mine) {
      // this rank holds the cut: find it in position order
      uint32_t run = before;
      if (tid == 0) s_found = 0;
      for (uint32_t b0 = s0; b0 < s1; b0 += 4 * kLwThreads) {
        const uint32_t i0 = b0 + 4 * tid;
        uint32_t eq = 0;
#pragma unroll
        for (int j = 0; j < 4; ++j)
          if (i0 + j < s1 && mag(i0 + j) == sel.B) eq |= 1u << j;
        uint32_t blk;
        uint32_t at = run + block_exclusive<kLwThreads>(__popc(eq), blk, s_w);
#pragma unroll
        for (int j = 0; j < 4; ++j)
          if (eq & (1u << j)) {
            if (++at == k_rem) {
              s_last = i0 + j;
              s_found = 1;
            }
          }
        run += blk;
        __syncthreads();
        if (s_found) break;
      }
      if (tid == 0) st->last = s_last;
    }
    if (!barrier()) return false;
    sel.last = __ldcg(&st->last);
  }
  uint32_t* io = idx_out + s.out;
  float* vo = val_out + s.out;
  __shared__ uint32_t s_base;
  auto publish = [&](uint32_t total) -> uint32_t {
    if (tid == 0) st->cnt[r] = total;
    if (!barrier()) {
      if (tid == 0) s_base = 0xffffffffu;
      __syncthreads();
      return 0xffffffffu;  // no position is below k: nothing is written
    }
    if (tid == 0) {
      uint32_t before = 0, all = 0;
      for (uint32_t q = 0; q < T; ++q) {
        const uint32_t x = __ldcg(&st->cnt[q]);
        before += q < r ? x : 0u;
        all += x;
      }
      if (all != s.k) atomicOr(a.error, kDevErrBadInput);
      s_base = before;
    }
    __syncthreads();
    return s_base;
  };
  const SrcGlobal sg{vals, idxs, s.lo};
  write_out(sg, s0, s1, sel, s.k, io, vo, e, overflow, s_w, publish, err, err_from);
  if (s_base == 0xffffffffu) return false;
  // every CTA has read the level histograms (before the write-out barrier):
  // clear them for the next call
  if (r == 0)
    for (uint32_t b = tid; b < 3 * 2048; b += kLwThreads) (&st->hist[0][0])[b] = 0;
  return true;
}

__global__ void __launch_bounds__(kLwThreads, 1)
    lw_select_kernel(float* __restrict__ e, uint32_t* __restrict__ idx_out,
                     float* __restrict__ val_out, LwArgs a) {
  extern __shared__ __align__(16) uint32_t s_bits[];
  __shared__ uint32_t s_hist[kHistBins];
  __shared__ uint32_t s_w[kLwThreads / 32];
  __shared__ uint32_t s_lo[32], s_hi[32];
  const int tid = threadIdx.x;
  // a dependent launch may start early: the stream pass's results are read
  // only after this; the next call's sampling may then be scheduled (it
  // writes nothing this kernel reads before waiting for it)
  griddep_wait();
  griddep_launch_dependents();
  const bool failed = (__ldcg(a.list_flags) & kDevErrTimeout) != 0;
  if (blockIdx.x == 0 && tid == 0) {
    *a.count_out = failed ? 0u : a.total_k;
    if (failed) atomicOr(a.error, kDevErrTimeout);
  }
  if (failed) {  // a is incomplete: nothing is selected
    if (blockIdx.x == 0 && tid == 0 && a.err_out) *a.err_out = err_invalid();
    return;
  }
  bool overflow = false, bad = false;
  ErrAcc acc;
  ErrAcc* err = a.err_out ? &acc : nullptr;
  const LwCta me = a.ctas[blockIdx.x];
  if (me.team == kLwNoTeam) {
    for (uint32_t w = me.a; w < me.b; ++w) {
      const uint32_t si = a.work_seg[w];
      const LwSeg s = a.segs[si];
      __syncthreads();  // the previous segment is done with shared memory
      if (!select_single(a, s, si, e, idx_out, val_out, overflow, s_bits, s_hist, s_w, s_lo,
                         s_hi, err))
        bad = true;
    }
  } else {
    const LwSeg s = a.segs[me.a];
    select_team(a, s, me.a, me.b, me.rank, a.teams + me.team, e, idx_out, val_out, overflow, bad,
                s_hist, s_w, err);
  }
  if (__syncthreads_or(overflow) && tid == 0) atomicOr(a.error, kDevErrOverflow);
  if (__syncthreads_or(bad) && tid == 0) atomicOr(a.error, kDevErrBadInput);
  if (a.err_out) {
    // this CTA's share; the last CTA to arrive adds the shares in CTA order
    // to the streaming pass's
    __shared__ FF s_d[32];
    __shared__ uint32_t s_last_cta;
    acc.flush();
    const FF share = block_sum_ff(acc.total, s_d);
    if (tid == 0) {
      a.err_parts[blockIdx.x] = share;
      __threadfence();
      s_last_cta = atomicAdd(a.err_arrive, 1u) == gridDim.x - 1 ? 1u : 0u;
    }
    __syncthreads();
    if (s_last_cta) {
      __threadfence();
      const FF shares = sum_parts_ff(a.err_parts, gridDim.x, s_d);
      if (tid == 0) *a.err_out = *a.stream_err + ff_to_double(shares);
    }
  }
}

// ------------------------------------------------------------- host side
template <typename GT>
int lw_group_blocks_per_sm() {
  const void* fn = reinterpret_cast<const void*>(&lookback_stream_kernel<LwCandOp<GT>, kLwStages>);
  const uint32_t smem = LbLayout<LwCandOp<GT>, kLwStages>::kSmem;
  int n = 0;
  if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess ||
      cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, fn, kLbThreads, smem) != cudaSuccess)
    n = 0;
  cudaGetLastError();
  return n;
}

template <typename GT>
int lw_stream_blocks_per_sm() {
  const void* fn = reinterpret_cast<const void*>(&stream_compact_kernel<LwCandOp<GT>, kLwStages>);
  const uint32_t smem = StreamLayout<LwCandOp<GT>, kLwStages>::kSmem;
  int n = 0;
  if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess ||
      cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, fn, kStreamThreads, smem) != cudaSuccess)
    n = 0;
  cudaGetLastError();
  return n;
}

size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

// Work estimate of a segment's selection by one CTA, in positions handled.
uint64_t select_cost(const LwSeg& s) {
  const uint64_t ds = s.hi - s.lo;
  if (s.kind == kLwAll) return ds / 2 + 1024;
  if (s.kind == kLwWhole) return ds / 4 + 2048;
  return 3ull * s.k + 4096;  // sampled: about 1.5 k_s candidates, a few passes
}

template <typename GT>
cudaError_t launch_typed(const GT* g, float* e, float gamma, uint32_t d, uint32_t* idx_out,
                         float* val_out, uint32_t* count_out, double* err_out, Workspace& ws,
                         const DeviceInfo& dev) {
  const LwPlan& p = *ws.lw;
  cudaError_t err = cudaSuccess;
  uint32_t* state = ws.topk_state(ws.topk_calls);
  uint32_t* other = ws.topk_state(ws.topk_calls + 1);
  const uint32_t lw_parity = ws.topk_calls;
  ++ws.topk_calls;
  uint32_t* list_flags = state + kStListFlags / 4;
  uint32_t* list_idx = reinterpret_cast<uint32_t*>(ws.cand(0));
  float* list_val = reinterpret_cast<float*>(list_idx + ws.cand_cap);
  const LwSeg* segs = reinterpret_cast<const LwSeg*>(p.dev + p.off_segs);
  uint32_t* mbound = reinterpret_cast<uint32_t*>(p.dev + p.off_mbound);
  uint32_t* tile_base = reinterpret_cast<uint32_t*>(p.dev + p.off_tile_base);

  const int per_sm = sizeof(GT) == 4 ? dev.lw_stream_per_sm_f32 : dev.lw_stream_per_sm_bf16;
  const bool streamable = reinterpret_cast<uintptr_t>(e) % 16 == 0 &&
                          reinterpret_cast<uintptr_t>(g) % 16 == 0 && per_sm > 0;
  if (streamable) {
    // 1 sample
    if (p.n_sampled > 0) {
      const uint2* sampled = reinterpret_cast<const uint2*>(p.dev + p.off_samples);
      uint32_t cap = ws.cand_cap;
      // the merged histograms of the multi-part segments: two copies, by call parity
      uint32_t* part_hist = reinterpret_cast<uint32_t*>(p.dev + p.off_part_hist) +
                            static_cast<size_t>(lw_parity & 1u) * p.n_part_hist * kLwPartHistWords;
      void* sp[] = {(void*)&g, (void*)&e, (void*)&gamma, (void*)&segs, (void*)&sampled,
                    (void*)&mbound, (void*)&cap, (void*)&part_hist};
      err = launch_pdl(reinterpret_cast<const void*>(&lw_sample_kernel<GT>), p.n_sampled,
                       kSampleThreads, kLwSampleSmem, ws.stream, sp, false);
      count_launch();
      if (err != cudaSuccess) return err;
    }
    // 2 stream
    ScanCtx ctx = next_scan_ctx(ws, p.tiles);
    ctx.error = list_flags;
    LwCandOp<GT> op{g, e, gamma, d,
                    reinterpret_cast<const uint32_t*>(p.dev + p.off_seg_end), mbound,
                    reinterpret_cast<const uint32_t*>(p.dev + p.off_tile_info), other};
    uint32_t slots = static_cast<uint32_t>(per_sm * dev.sm_count);
    if (slots > kMaxChunks) slots = kMaxChunks;
    const uint32_t grid = p.tiles < slots ? p.tiles : slots;
    uint32_t cap = ws.cand_cap;
    uint32_t* list_count = ws.u32(kOffTkListCount);
    const int per_sm_groups =
        sizeof(GT) == 4 ? dev.lw_group_per_sm_f32 : dev.lw_group_per_sm_bf16;
    if (use_group_kernel(p.tiles) && per_sm_groups > 0) {
      // claimed groups of tiles with look-back (stream_lookback.cuh): no
      // wait depends on which CTAs are resident
      const uint32_t groups = (p.tiles + kLbGroupTiles - 1) / kLbGroupTiles;
      const uint32_t gslots = static_cast<uint32_t>(per_sm_groups * dev.sm_count);
      const uint32_t ggrid = groups < gslots ? groups : gslots;
      LbArgs la{tile_base, err_out ? ws.stream_err() : nullptr, reinterpret_cast<FF*>(ws.counts()),
                ws.stage_idx(), ws.stage_val()};
      void* gp[] = {&op, &d, &list_idx, &list_val, &list_count, &cap, &ctx, &la};
      err = launch_pdl(
          reinterpret_cast<const void*>(&lookback_stream_kernel<LwCandOp<GT>, kLwStages>), ggrid,
          kLbThreads, LbLayout<LwCandOp<GT>, kLwStages>::kSmem, ws.stream, gp, false);
    } else {
      StreamArgs sa{ws.stage_idx(), ws.stage_val(), ws.counts(), ws.chunks(), tile_base,
                    err_out ? ws.stream_err() : nullptr, ws.errparts()};
      void* params[] = {&op, &d, &list_idx, &list_val, &list_count, &cap, &ctx, &sa};
      // not cooperative: the only cross-CTA wait is on lower-numbered CTAs,
      // which are scheduled first
      err = launch_pdl(
          reinterpret_cast<const void*>(&stream_compact_kernel<LwCandOp<GT>, kLwStages>), grid,
          kStreamThreads, StreamLayout<LwCandOp<GT>, kLwStages>::kSmem, ws.stream, params, false);
    }
    count_launch();
    if (err != cudaSuccess) return err;
  } else {
    const uint32_t grid = p.tiles < static_cast<uint32_t>(dev.sm_count * 8)
                              ? p.tiles : static_cast<uint32_t>(dev.sm_count * 8);
    lw_accumulate_plain_kernel<GT><<<grid, kThreads, 0, ws.stream>>>(g, e, gamma, d, other);
    count_launch();
    if ((err = cudaGetLastError()) != cudaSuccess) return err;
  }
  // 3 select: a cooperative launch when there are teams, so that every
  // team's CTAs are resident
  LwArgs a;
  a.segs = segs;
  a.mbound = mbound;
  a.ctas = reinterpret_cast<const LwCta*>(p.dev + p.off_ctas);
  a.work_seg = reinterpret_cast<const uint32_t*>(p.dev + p.off_work_seg);
  a.teams = reinterpret_cast<LwTeamState*>(p.dev + p.off_teams);
  a.tile_base = tile_base;
  a.list_idx = list_idx;
  a.list_val = list_val;
  a.list_flags = list_flags;
  a.error = ws.u32(kOffError);
  a.count_out = count_out;
  a.wait_limit_ns = wait_limit_ns();
  a.tiles = p.tiles;
  a.cap = ws.cand_cap;
  a.use_list = streamable ? 1u : 0u;
  a.total_k = static_cast<uint32_t>(p.total_k);
  // inputs the streaming pass could not take: the norm by a plain pass after
  a.err_out = streamable ? err_out : nullptr;
  a.stream_err = ws.stream_err();
  a.err_parts = ws.errparts();
  a.err_arrive = state + kStErrArrive / 4;
  void* params[] = {(void*)&e, (void*)&idx_out, (void*)&val_out, (void*)&a};
  // (cooperative only when there are teams: nothing else waits on another CTA)
  err = launch_pdl(reinterpret_cast<const void*>(&lw_select_kernel), p.n_select_ctas, kLwThreads,
                   kLwSelectSmem, ws.stream, params, p.n_teams > 0);
  count_launch();
  if (err == cudaSuccess && err_out && !streamable) err = launch_error_norm(e, d, err_out, ws, dev);
  return err;
}

}  // namespace

void topk_layerwise_init_device(DeviceInfo& info) {
  int n = 0;
  // the sampling kernel's histogram (dynamic shared memory); a failure here
  // makes its launches fail, which the calls report
  cudaFuncSetAttribute(lw_sample_kernel<float>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                       kLwSampleSmem);
  cudaFuncSetAttribute(lw_sample_kernel<uint16_t>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                       kLwSampleSmem);
  cudaGetLastError();
  if (cudaFuncSetAttribute(lw_select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           kLwSelectSmem) != cudaSuccess ||
      cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, lw_select_kernel, kLwThreads,
                                                    kLwSelectSmem) != cudaSuccess)
    n = 0;
  info.lw_select_per_sm = n;
  info.lw_stream_per_sm_f32 = lw_stream_blocks_per_sm<float>();
  info.lw_stream_per_sm_bf16 = lw_stream_blocks_per_sm<uint16_t>();
  info.lw_group_per_sm_f32 = lw_group_blocks_per_sm<float>();
  info.lw_group_per_sm_bf16 = lw_group_blocks_per_sm<uint16_t>();
  cudaGetLastError();
}

cudaError_t lw_prepare(Workspace& ws, const uint64_t* seg_end, const uint64_t* seg_k,
                       uint32_t n_seg, uint64_t d, const DeviceInfo& dev) {
  if (!ws.lw) ws.lw = new LwPlan;
  LwPlan& p = *ws.lw;
  if (p.valid && p.d == d && p.n_seg == n_seg &&
      std::equal(seg_end, seg_end + n_seg, p.seg_end.begin()) &&
      std::equal(seg_k, seg_k + n_seg, p.seg_k.begin()))
    return cudaSuccess;
  p.valid = false;
  const uint32_t tiles = tiles_for(d);
  // segments, sampling CTAs
  std::vector<LwSeg> segs(n_seg);
  std::vector<uint32_t> ends(n_seg), mbound(n_seg, kLwNoBound);
  // the sampling CTAs: (segment, part | parts << 8 | merge slot << 16)
  std::vector<uint2> sampled;
  std::vector<uint32_t> parts_of(n_seg, 1);
  uint32_t n_sampled = 0, n_part_hist = 0;
  uint64_t lo = 0, total_k = 0;
  for (uint32_t s = 0; s < n_seg; ++s) {
    const uint64_t hi = seg_end[s], ds = hi - lo, k = seg_k[s];
    LwSeg& x = segs[s];
    x = LwSeg{0, static_cast<uint32_t>(lo), static_cast<uint32_t>(hi), static_cast<uint32_t>(k),
              static_cast<uint32_t>(total_k), 0, kLwNone, 0};
    static_assert(sizeof(LwSeg) == 32, "segment record");
    if (k == 0 || ds == 0)
      x.kind = kLwNone;
    else if (k == ds)
      x.kind = kLwAll;
    else if (ds <= kLwWholeMax)
      x.kind = kLwWhole;
    else
      x.kind = kLwSampled;
    if (x.kind == kLwSampled) {
      // every aligned group of 4 while there are at most kLwSampleGroups,
      // else kLwSampleGroups of them spread evenly
      const uint64_t avail = (hi - 4) / 4 - (lo + 3) / 4 + 1;
      x.groups = static_cast<uint32_t>(std::min<uint64_t>(avail, kLwSampleGroups));
      x.exact = x.groups == avail ? 1u : 0u;
      x.step = ((avail - 1) << 32) / (x.groups - 1);  // a segment of > 4096 holds > 1000 groups
      // A long segment with a small k_s would admit far more candidates
      // than one CTA holds: the bound keeps 32 samples' slack, i.e.
      // 32 d_s / (4 groups) coordinates. Up to kLwMaxParts CTAs then sample
      // equal runs of it (kLwSampleGroups groups each) into one merged
      // histogram, shrinking that slack: toward 3/4 of what one select CTA
      // holds with the coordinates (half its shared memory) when the 1.5 k_s
      // themselves fit there, else of what it holds as values alone.
      uint32_t parts = 1;
      if (!x.exact) {
        const uint64_t need = 3ull * k / 2;
        const uint64_t fit = need < kLwSmemElems * 3ull / 8 ? kLwSmemElems * 3ull / 8
                                                            : kLwSmemElems * 3ull / 4;
        const uint64_t slack = 32ull * ds / (4ull * x.groups);
        if (need + slack > fit && need < fit) {
          const uint64_t want = (slack + (fit - need) - 1) / (fit - need);
          parts = static_cast<uint32_t>(std::min<uint64_t>(
              std::min<uint64_t>(want, kLwMaxParts), avail / kLwSampleGroups));
          if (parts < 1) parts = 1;
        }
      }
      parts_of[s] = parts;
      const uint32_t slot = parts > 1 ? n_part_hist++ : 0u;
      for (uint32_t j = 0; j < parts; ++j) sampled.push_back(make_uint2(s, j | (parts << 8) | (slot << 16)));
      n_sampled += parts;
    }
    ends[s] = static_cast<uint32_t>(hi);
    mbound[s] = x.kind == kLwNone ? kLwNoBound : kLwDeferred;  // sampled: the sampler's
    total_k += k;
    lo = hi;
  }
  // tiles: the first segment of each, and whether it lies in one segment
  std::vector<uint32_t> tile_info(tiles);
  {
    uint32_t s = 0;
    for (uint32_t t = 0; t < tiles; ++t) {
      const uint64_t t0 = static_cast<uint64_t>(t) * kTileElems;
      const uint64_t t1 = std::min<uint64_t>(d, t0 + kTileElems);
      while (ends[s] <= t0) ++s;  // skips empty segments; ends[n_seg-1] == d > t0
      tile_info[t] = s | (ends[s] >= t1 ? kLwTileUniform : 0u);
    }
  }
  // Select work. A segment whose candidates may exceed one CTA's shared
  // memory, or whose own length would make a selection from e slow for one
  // CTA, gets a team of co-resident CTAs; the others go, longest first, onto
  // the least loaded of the remaining CTAs. At most sm_count x (select CTAs
  // per SM) CTAs in all, so that the cooperative launch is resident.
  const uint32_t budget =
      static_cast<uint32_t>(std::max(1, dev.sm_count * std::max(1, dev.lw_select_per_sm)));
  std::vector<uint32_t> team_seg, team_size, singles;
  for (uint32_t s = 0; s < n_seg; ++s) {
    const LwSeg& x = segs[s];
    if (x.kind == kLwNone) continue;
    uint32_t t = 1;
    if (x.kind == kLwSampled) {
      // candidates the bound aims at: 1.5 k_s, plus 32 samples' worth
      const uint64_t ds = x.hi - x.lo;
      const uint64_t sampled_groups = static_cast<uint64_t>(x.groups) * parts_of[s];
      const uint64_t est =
          x.exact ? x.k + 2048 : 3ull * x.k / 2 + 32ull * ds / (4ull * sampled_groups);
      uint64_t want = est > kLwSmemElems * 3ull / 4 ? (est + 24575) / 24576 : 1;
      // a segment one CTA would select slowly from e if its bound missed
      // gets a team, unless its merged sample makes a miss implausible
      if (parts_of[s] == 1) want = std::max<uint64_t>(want, (ds + (1u << 24) - 1) >> 24);
      t = static_cast<uint32_t>(std::min<uint64_t>(want, kLwMaxTeam));
    }
    if (t > 1) {
      team_seg.push_back(s);
      team_size.push_back(t);
    } else {
      singles.push_back(s);
    }
  }
  {
    // shrink the teams until they leave at least one CTA for the singles
    const uint32_t reserve = singles.empty() ? 0u : 1u;
    uint64_t sum = 0;
    for (uint32_t t : team_size) sum += t;
    while (sum + reserve > budget) {
      auto it = std::max_element(team_size.begin(), team_size.end());
      if (*it <= 1) break;
      --*it;
      --sum;
    }
    for (size_t q = 0; q < team_seg.size();) {  // a team of one is a single
      if (team_size[q] <= 1) {
        singles.push_back(team_seg[q]);
        team_seg.erase(team_seg.begin() + q);
        team_size.erase(team_size.begin() + q);
      } else {
        ++q;
      }
    }
  }
  uint32_t team_ctas = 0;
  for (uint32_t t : team_size) team_ctas += t;
  std::stable_sort(singles.begin(), singles.end(), [&](uint32_t x, uint32_t y) {
    return select_cost(segs[x]) > select_cost(segs[y]);
  });
  const uint32_t room = budget > team_ctas ? budget - team_ctas : 1u;
  // at least one CTA in all: it also writes the count and reports a failed stream
  const uint32_t n_single = static_cast<uint32_t>(std::min<size_t>(
      singles.size(), room)) + (singles.empty() && team_ctas == 0 ? 1u : 0u);
  std::vector<std::vector<uint32_t>> per(n_single);
  {
    using Load = std::pair<uint64_t, uint32_t>;
    std::priority_queue<Load, std::vector<Load>, std::greater<Load>> heap;
    for (uint32_t c = 0; c < n_single; ++c) heap.push(Load{0, c});
    for (uint32_t s : singles) {
      Load l = heap.top();
      heap.pop();
      per[l.second].push_back(s);
      l.first += select_cost(segs[s]);
      heap.push(l);
    }
  }
  std::vector<LwCta> ctas;
  std::vector<uint32_t> work_seg;
  for (uint32_t q = 0; q < team_seg.size(); ++q)  // teams first: the longest work
    for (uint32_t r = 0; r < team_size[q]; ++r) ctas.push_back(LwCta{q, team_seg[q], team_size[q], r});
  for (uint32_t c = 0; c < n_single; ++c) {
    const uint32_t a = static_cast<uint32_t>(work_seg.size());
    work_seg.insert(work_seg.end(), per[c].begin(), per[c].end());
    ctas.push_back(LwCta{kLwNoTeam, a, static_cast<uint32_t>(work_seg.size()), 0});
  }
  const uint32_t n_teams = static_cast<uint32_t>(team_seg.size());

  // device layout
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t at = off;
    off = align256(off + (bytes ? bytes : 1));
    return at;
  };
  p.off_segs = take(sizeof(LwSeg) * n_seg);
  p.off_seg_end = take(sizeof(uint32_t) * n_seg);
  p.off_mbound = take(sizeof(uint32_t) * n_seg);
  p.off_tile_info = take(sizeof(uint32_t) * tiles);
  p.off_samples = take(sizeof(uint2) * sampled.size());
  p.off_ctas = take(sizeof(LwCta) * ctas.size());
  p.off_work_seg = take(sizeof(uint32_t) * work_seg.size());
  const size_t upload = off;
  p.off_teams = take(sizeof(LwTeamState) * n_teams);
  p.off_part_hist = take(2 * sizeof(uint32_t) * kLwPartHistWords * n_part_hist);
  const size_t zero_end = off;
  p.off_tile_base = take(sizeof(uint32_t) * (tiles + 1));
  p.total = off;

  p.image.assign(upload, 0);
  auto put = [&](size_t at, const void* src, size_t bytes) {
    if (bytes) std::memcpy(p.image.data() + at, src, bytes);
  };
  put(p.off_segs, segs.data(), sizeof(LwSeg) * n_seg);
  put(p.off_seg_end, ends.data(), sizeof(uint32_t) * n_seg);
  put(p.off_mbound, mbound.data(), sizeof(uint32_t) * n_seg);
  put(p.off_tile_info, tile_info.data(), sizeof(uint32_t) * tiles);
  put(p.off_samples, sampled.data(), sizeof(uint2) * sampled.size());
  put(p.off_ctas, ctas.data(), sizeof(LwCta) * ctas.size());
  put(p.off_work_seg, work_seg.data(), sizeof(uint32_t) * work_seg.size());

  cudaError_t err;
  if (p.total > p.dev_bytes) {
    if (p.dev) {  // earlier launches may still read the old tables
      if ((err = cudaStreamSynchronize(ws.stream)) != cudaSuccess) return err;
      cudaFree(p.dev);
      p.dev = nullptr;
      p.dev_bytes = 0;
    }
    void* ptr = nullptr;
    if ((err = cudaMalloc(&ptr, p.total)) != cudaSuccess) {
      cudaGetLastError();
      return err;
    }
    p.dev = static_cast<char*>(ptr);
    p.dev_bytes = p.total;
  }
  // stream-ordered after every earlier launch that read the old tables
  if ((err = cudaMemcpyAsync(p.dev, p.image.data(), upload, cudaMemcpyHostToDevice,
                             ws.stream)) != cudaSuccess)
    return err;
  if ((err = cudaMemsetAsync(p.dev + p.off_teams, 0, zero_end - p.off_teams, ws.stream)) !=
      cudaSuccess)
    return err;
  p.seg_end.assign(seg_end, seg_end + n_seg);
  p.seg_k.assign(seg_k, seg_k + n_seg);
  p.d = d;
  p.n_seg = n_seg;
  p.n_sampled = n_sampled;
  p.n_part_hist = n_part_hist;
  p.n_select_ctas = static_cast<uint32_t>(ctas.size());
  p.n_teams = n_teams;
  p.tiles = tiles;
  p.total_k = total_k;
  p.valid = true;
  return cudaSuccess;
}

cudaError_t launch_topk_layerwise(const void* g, bool g_bf16, float* e, float gamma, uint32_t d,
                                  uint32_t* idx_out, float* val_out, uint32_t* count_out,
                                  double* err_out, Workspace& ws, const DeviceInfo& dev) {
  if (g_bf16)
    return launch_typed(static_cast<const uint16_t*>(g), e, gamma, d, idx_out, val_out,
                        count_out, err_out, ws, dev);
  return launch_typed(static_cast<const float*>(g), e, gamma, d, idx_out, val_out, count_out,
                      err_out, ws, dev);
}

}  // namespace efs
