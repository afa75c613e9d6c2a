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
//  1 sample   for each large segment (more than kLwSmemElems coordinates,
//             0 < k_s < d_s), CTAs read groups of 4 consecutive coordinates
//             spread evenly over it, histogram the top 13 magnitude bits of
//             a = fmaf(γ,g,e), and merge into the segment's histogram; the
//             last CTA of the segment to finish (an arrival counter) picks
//             the candidate bound with about 1.5 times the needed mass above
//             it, then clears the histogram and counter for the next call.
//  2 stream   the streaming compaction of stream_compact.cuh: a = fmaf(γ,g,e)
//             is written over e (12 B per coordinate, the algorithmic bytes)
//             and the coordinates at or above their segment's bound are
//             emitted as one ordered candidate list, with the list position
//             of each tile's first candidate.
//  3 select   CTAs own groups of segments (balanced on the host). For each:
//             a small segment is read into shared memory whole; a large one
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
#include "stream_compact.cuh"

namespace efs {
namespace {

constexpr int kLwThreads = 1024;  // sample and select CTAs
constexpr uint32_t kLwSelectSmem = kLwSmemElems * sizeof(uint32_t);
constexpr int kLwSampleShift = 31 - kSampleBits;  // magnitude bits below the sampled ones
constexpr int kLwStages = 4;

__device__ __forceinline__ uint32_t mag_bits(float x) { return __float_as_uint(x) & 0x7fffffffu; }

// ------------------------------------------------------------- 1 sample
template <typename GT>
__global__ void __launch_bounds__(kLwThreads)
    lw_sample_kernel(const GT* __restrict__ g, const float* __restrict__ e, float gamma,
                     const LwSeg* __restrict__ segs, const LwSample* __restrict__ samples,
                     uint32_t* hist, uint32_t* done, uint32_t* mbound, uint32_t cand_cap) {
  __shared__ uint32_t s_hist[kSampleBins];
  __shared__ uint32_t s_w[kLwThreads / 32];
  __shared__ uint32_t s_last, s_bin, s_mass;
  const int tid = threadIdx.x;
  const LwSample sp = samples[blockIdx.x];
  const LwSeg s = segs[sp.seg];
  for (int b = tid; b < kSampleBins; b += kLwThreads) s_hist[b] = 0;
  __syncthreads();
  // group q starts at lo + q (d_s - 4) / (groups - 1): the groups spread
  // evenly from the first to the last 4 coordinates of the segment
  const uint64_t span = static_cast<uint64_t>(s.hi - s.lo) - 4u;
  const uint64_t den = s.groups - 1u;
  constexpr int kG = static_cast<int>(kLwSampleGroupsPerCta / kLwThreads);
  float gv[kG][4], ev[kG][4];
  bool in[kG];
#pragma unroll
  for (int q = 0; q < kG; ++q) {  // every load in flight before any use
    const uint32_t qq = sp.q0 + q * kLwThreads + tid;
    in[q] = qq < sp.q1;
    const uint64_t p = s.lo + (in[q] ? static_cast<uint64_t>(qq) * span / den : 0u);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      gv[q][j] = in[q] ? grad_scalar(g, p + j) : 0.0f;
      ev[q][j] = in[q] ? __ldg(e + p + j) : 0.0f;
    }
  }
#pragma unroll
  for (int q = 0; q < kG; ++q)
#pragma unroll
    for (int j = 0; j < 4; ++j)
      hist_add_warp(s_hist, mag_bits(__fmaf_rn(gamma, gv[q][j], ev[q][j])) >> kLwSampleShift,
                    in[q]);
  __syncthreads();
  uint32_t* h = hist + static_cast<size_t>(s.slot) * kSampleBins;
  for (int b = tid; b < kSampleBins; b += kLwThreads)
    if (s_hist[b]) atomicAdd(&h[b], s_hist[b]);
  __threadfence();  // this CTA's histogram adds before its arrival
  __syncthreads();
  if (tid == 0) s_last = atomicAdd(done + sp.seg, 1u) == s.nblk - 1u ? 1u : 0u;
  __syncthreads();
  if (!s_last) return;
  __threadfence();  // every arrival's adds are visible to the last CTA
  // the segment's merged histogram: 8 consecutive bins per thread
  constexpr int kPer = kSampleBins / kLwThreads;
  static_assert(kPer == 8, "sample bins per thread");
  uint32_t c[kPer];
  {
    const uint4 v0 = __ldcg(reinterpret_cast<const uint4*>(h) + 2 * tid);
    const uint4 v1 = __ldcg(reinterpret_cast<const uint4*>(h) + 2 * tid + 1);
    c[0] = v0.x; c[1] = v0.y; c[2] = v0.z; c[3] = v0.w;
    c[4] = v1.x; c[5] = v1.y; c[6] = v1.z; c[7] = v1.w;
  }
  uint32_t mine = 0;
#pragma unroll
  for (int i = 0; i < kPer; ++i) mine += c[i];
  if (tid == 0) s_bin = 0xffffffffu;
  uint32_t m;  // sampled coordinates
  const uint32_t above = block_suffix_exclusive(mine, m, s_w);  // orders the reset
  // 1.5x the expected sampled count above the k_s-th magnitude, plus 32
  // (integer arithmetic; the products stay below 2^56)
  const uint64_t ds = s.hi - s.lo;
  const uint64_t target = 3ull * s.k * m / (2ull * ds) + 32ull;
  if (target <= m && above < target && target - above <= mine) {
    uint64_t run = above;
#pragma unroll
    for (int i = kPer - 1; i >= 0; --i) {
      run += c[i];
      if (run >= target && run - c[i] < target) {
        s_bin = tid * kPer + i;
        s_mass = static_cast<uint32_t>(run);
      }
    }
  }
  __syncthreads();
  // clear the histogram for the next call: every read of it is complete
  reinterpret_cast<uint4*>(h)[2 * tid] = make_uint4(0u, 0u, 0u, 0u);
  reinterpret_cast<uint4*>(h)[2 * tid + 1] = make_uint4(0u, 0u, 0u, 0u);
  if (tid == 0) {
    uint32_t bound = kLwNoBound;
    // expected candidates (the sampled mass scaled to d_s) at most half the
    // list's capacity, else the segment is selected from e itself
    if (s_bin != 0xffffffffu &&
        2ull * s_mass * ds <= static_cast<uint64_t>(cand_cap) * m)
      bound = s_bin << kLwSampleShift;
    mbound[sp.seg] = bound;
    done[sp.seg] = 0;
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
  const uint32_t* mbound;     // [n_seg] candidate bounds (kLwNoBound: none)
  const uint32_t* tile_info;  // [tiles] first segment of the tile | kLwTileUniform
  uint32_t* other_state;      // the other Top-k state block: zeroed here for the next call
  static constexpr uint32_t kGBytes = kTileElems * sizeof(GT);
  static constexpr uint32_t kStageBytes = kGBytes + kTileElems * sizeof(float);
  static constexpr uint32_t kWarpStagePairs = 512;  // on-chip staged pairs per compute warp
  static constexpr bool kPrepass = false;
  static constexpr int kSampleBins = 1;
  __device__ void sample(uint32_t, uint32_t, int, uint32_t*) const {}
  __device__ void merge(const uint32_t*) const {}
  __device__ void prologue() const { clear_state(other_state); }
  __device__ bool barrier(uint64_t, uint32_t*) const { return true; }
  __device__ uint64_t choose() const { return 0; }

  __device__ __forceinline__ void fill(unsigned char* stage, uint32_t t, uint64_t* bar,
                                       uint64_t policy) const {
    tma_load_1d(stage, g + static_cast<size_t>(t) * kTileElems, kGBytes, bar, policy);
    tma_load_1d(stage + kGBytes, e + static_cast<size_t>(t) * kTileElems,
                kTileElems * sizeof(float), bar, policy);
  }

  // selection bits of the lane's coordinates from their segments' bounds
  __device__ __forceinline__ void select(uint32_t t, uint64_t first, const float (&a)[kSUnits][4],
                                         uint32_t (&sel)[kSUnits]) const {
    const uint32_t info = __ldg(tile_info + t);
    if (info & kLwTileUniform) {
      const uint32_t b = __ldg(mbound + (info & ~kLwTileUniform));
#pragma unroll
      for (int v = 0; v < kSUnits; ++v) {
        sel[v] = 0;
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
            sel[v] |= (mag_bits(a[v][j]) >= __ldg(mbound + s) ? 1u : 0u) << j;
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
        if (first + v * 128 + j >= d) sel[v] &= ~(1u << j);
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
  const uint32_t* work_ptr;   // [grid + 1] each CTA's range of work_seg
  const uint32_t* work_seg;   // segment ids, grouped by CTA
  const uint32_t* tile_base;  // [tiles + 1] list position of each tile's first candidate
  const uint32_t* list_idx;   // ordered candidates of the streaming pass
  const float* list_val;
  const uint32_t* list_flags; // that pass's latched bits
  uint32_t* error;
  uint32_t* count_out;
  uint32_t tiles, cap, use_list;
  uint32_t total_k;
};

// Number of list entries with index < x (x <= d): the list position of x's
// tile, plus that tile's entries below x. ok = false when those entries were
// cut off at the list's capacity. Whole CTA; uniform result.
__device__ uint32_t list_position(const LwArgs& a, uint32_t x, bool& ok) {
  const uint32_t t = x / kTileElems;
  if (t >= a.tiles) return __ldcg(a.tile_base + a.tiles);
  const uint32_t p0 = __ldcg(a.tile_base + t);
  if (x % kTileElems == 0) return p0;
  const uint32_t p1 = __ldcg(a.tile_base + t + 1);
  if (p1 > a.cap) {
    ok = false;
    return p0;
  }
  uint32_t below = 0;
  for (uint32_t b = p0; b < p1; b += kLwThreads) {
    const uint32_t p = b + threadIdx.x;
    below += __syncthreads_count(p < p1 && __ldcg(a.list_idx + p) < x);
  }
  return p0 + below;
}

// Reads n fp32 values (8 loads in flight per thread), keeps their bits in
// s_bits when it is given, and returns the minimum and maximum magnitude.
__device__ void load_minmax(const float* src, uint32_t n, uint32_t* s_bits, uint32_t& lo,
                            uint32_t& hi, uint32_t* s_lo, uint32_t* s_hi) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  constexpr int kBatch = 8;
  lo = 0xffffffffu;
  hi = 0;
  for (uint32_t i0 = tid; i0 < n; i0 += kBatch * kLwThreads) {
    uint32_t v[kBatch];
#pragma unroll
    for (int j = 0; j < kBatch; ++j) {
      const uint32_t i = i0 + j * kLwThreads;
      v[j] = i < n ? __float_as_uint(__ldcg(src + i)) : 0u;
    }
#pragma unroll
    for (int j = 0; j < kBatch; ++j) {
      const uint32_t i = i0 + j * kLwThreads;
      if (i < n) {
        if (s_bits) s_bits[i] = v[j];
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
  lo = s_lo[lane];  // 32 warps
  hi = s_hi[lane];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    lo = min(lo, __shfl_xor_sync(0xffffffffu, lo, o));
    hi = max(hi, __shfl_xor_sync(0xffffffffu, hi, o));
  }
}

// Sources of a selection: list position i has value bits bits(i) and
// coordinate index(i).
struct SrcSharedArray {  // a whole segment in shared memory
  const uint32_t* s_bits;
  uint32_t lo;
  __device__ __forceinline__ uint32_t bits(uint32_t i) const { return s_bits[i]; }
  __device__ __forceinline__ uint32_t index(uint32_t i) const { return lo + i; }
};
struct SrcSharedList {  // candidates' values in shared memory
  const uint32_t* s_bits;
  const uint32_t* idx;
  __device__ __forceinline__ uint32_t bits(uint32_t i) const { return s_bits[i]; }
  __device__ __forceinline__ uint32_t index(uint32_t i) const { return __ldcg(idx + i); }
};
struct SrcGlobalList {  // candidates in global memory
  const float* val;
  const uint32_t* idx;
  __device__ __forceinline__ uint32_t bits(uint32_t i) const {
    return __float_as_uint(__ldcg(val + i));
  }
  __device__ __forceinline__ uint32_t index(uint32_t i) const { return __ldcg(idx + i); }
};
struct SrcGlobalArray {  // a segment of a in global memory (e after the stream)
  const float* val;
  uint32_t lo;
  __device__ __forceinline__ uint32_t bits(uint32_t i) const {
    return __float_as_uint(__ldcg(val + i));
  }
  __device__ __forceinline__ uint32_t index(uint32_t i) const { return lo + i; }
};

// Writes the selected positions of [0, n), in order, as pairs at out[0, k)
// and zeroes e at each; returns the number selected. Whole CTA.
template <class Src>
__device__ uint32_t emit_selected(const Src& src, uint32_t n, const SmallSelection& sel,
                                  uint32_t k, uint32_t* idx_out, float* val_out, float* e,
                                  bool& overflow, uint32_t* s_w) {
  uint32_t base = 0;
  for (uint32_t b0 = 0; b0 < n; b0 += 4 * kLwThreads) {
    const uint32_t i0 = b0 + 4 * threadIdx.x;
    uint32_t bits[4], take = 0;
#pragma unroll
    for (int j = 0; j < 4; ++j) bits[j] = i0 + j < n ? src.bits(i0 + j) : 0u;
#pragma unroll
    for (int j = 0; j < 4; ++j)
      if (i0 + j < n && selected(sel, bits[j] & 0x7fffffffu, i0 + j)) take |= 1u << j;
    uint32_t total;
    uint32_t pos = base + block_exclusive<kLwThreads>(__popc(take), total, s_w);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      if (take & (1u << j)) {
        if (pos < k) {
          const uint32_t idx = src.index(i0 + j);
          idx_out[pos] = idx;
          val_out[pos] = __uint_as_float(bits[j]);
          e[idx] = 0.0f;  // residual of a sent coordinate
        } else {
          overflow = true;
        }
        ++pos;
      }
    }
    base += total;
  }
  return base;
}

__global__ void __launch_bounds__(kLwThreads, 1)
    lw_select_kernel(float* __restrict__ e, uint32_t* __restrict__ idx_out,
                     float* __restrict__ val_out, LwArgs a) {
  extern __shared__ __align__(16) uint32_t s_bits[];
  __shared__ uint32_t s_hist[kHistBins];
  __shared__ uint32_t s_w[kLwThreads / 32];
  __shared__ uint32_t s_lo[32], s_hi[32];
  const int tid = threadIdx.x;
  const bool failed = (__ldcg(a.list_flags) & kDevErrTimeout) != 0;
  if (blockIdx.x == 0 && tid == 0) {
    *a.count_out = failed ? 0u : a.total_k;
    if (failed) atomicOr(a.error, kDevErrTimeout);
  }
  if (failed) return;  // a is incomplete: nothing is selected
  bool overflow = false, bad = false;
  const uint32_t w_end = a.work_ptr[blockIdx.x + 1];
  for (uint32_t w = a.work_ptr[blockIdx.x]; w < w_end; ++w) {
    const uint32_t si = a.work_seg[w];
    const LwSeg s = a.segs[si];
    uint32_t* io = idx_out + s.out;
    float* vo = val_out + s.out;
    const uint32_t ds = s.hi - s.lo;
    __syncthreads();  // the previous segment is done with shared memory
    if (s.kind == kLwAll) {
      for (uint32_t i = tid; i < ds; i += kLwThreads) {
        io[i] = s.lo + i;
        vo[i] = __ldcg(e + s.lo + i);
        e[s.lo + i] = 0.0f;
      }
      continue;
    }
    SmallSelection sel;
    uint32_t lo, hi, got = 0;
    bool found = false;
    if (s.kind == kLwWhole) {
      load_minmax(e + s.lo, ds, s_bits, lo, hi, s_lo, s_hi);
      found = threshold_levels<kLwThreads>(MagsShared{s_bits}, ds, s.k, lo, hi, s_hist, s_w, sel);
      if (found)
        got = emit_selected(SrcSharedArray{s_bits, s.lo}, ds, sel, s.k, io, vo, e, overflow, s_w);
    } else {  // kLwSampled
      bool use = a.use_list && __ldcg(a.mbound + si) != kLwNoBound;
      uint32_t c0 = 0, c1 = 0;
      if (use) {
        bool ok = true;
        c0 = list_position(a, s.lo, ok);
        c1 = list_position(a, s.hi, ok);
        use = ok && c1 <= a.cap && c1 - c0 >= s.k;
      }
      if (use && c1 - c0 <= kLwSmemElems) {
        const uint32_t n = c1 - c0;
        load_minmax(a.list_val + c0, n, s_bits, lo, hi, s_lo, s_hi);
        found = threshold_levels<kLwThreads>(MagsShared{s_bits}, n, s.k, lo, hi, s_hist, s_w, sel);
        if (found)
          got = emit_selected(SrcSharedList{s_bits, a.list_idx + c0}, n, sel, s.k, io, vo, e,
                              overflow, s_w);
      } else if (use) {
        const uint32_t n = c1 - c0;
        load_minmax(a.list_val + c0, n, nullptr, lo, hi, s_lo, s_hi);
        found = threshold_levels<kLwThreads>(MagsGlobal{a.list_val + c0}, n, s.k, lo, hi, s_hist,
                                             s_w, sel);
        if (found)
          got = emit_selected(SrcGlobalList{a.list_val + c0, a.list_idx + c0}, n, sel, s.k, io,
                              vo, e, overflow, s_w);
      } else {
        load_minmax(e + s.lo, ds, nullptr, lo, hi, s_lo, s_hi);
        found = threshold_levels<kLwThreads>(MagsGlobal{e + s.lo}, ds, s.k, lo, hi, s_hist, s_w,
                                             sel);
        if (found)
          got = emit_selected(SrcGlobalArray{e + s.lo, s.lo}, ds, sel, s.k, io, vo, e, overflow,
                              s_w);
      }
    }
    if (!found || got != s.k) bad = true;
  }
  if (__syncthreads_or(overflow) && tid == 0) atomicOr(a.error, kDevErrOverflow);
  if (__syncthreads_or(bad) && tid == 0) atomicOr(a.error, kDevErrBadInput);
}

// ------------------------------------------------------------- host side
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

// Work estimate of a segment's selection, in list positions handled.
uint64_t select_cost(const LwSeg& s) {
  const uint64_t ds = s.hi - s.lo;
  if (s.kind == kLwAll) return ds / 2 + 1024;
  if (s.kind == kLwWhole) return ds / 4 + 2048;
  return 3ull * s.k + 4096;  // sampled: about 1.5 k_s candidates, a few passes
}

template <typename GT>
cudaError_t launch_typed(const GT* g, float* e, float gamma, uint32_t d, uint32_t* idx_out,
                         float* val_out, uint32_t* count_out, Workspace& ws,
                         const DeviceInfo& dev) {
  const LwPlan& p = *ws.lw;
  cudaError_t err = cudaSuccess;
  uint32_t* state = ws.topk_state(ws.topk_calls);
  uint32_t* other = ws.topk_state(ws.topk_calls + 1);
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
    if (p.n_sample_ctas > 0) {
      lw_sample_kernel<GT><<<p.n_sample_ctas, kLwThreads, 0, ws.stream>>>(
          g, e, gamma, segs, reinterpret_cast<const LwSample*>(p.dev + p.off_samples),
          reinterpret_cast<uint32_t*>(p.dev + p.off_hist),
          reinterpret_cast<uint32_t*>(p.dev + p.off_done), mbound, ws.cand_cap);
      count_launch();
      if ((err = cudaGetLastError()) != cudaSuccess) return err;
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
    StreamArgs sa{ws.stage_idx(), ws.stage_val(), ws.counts(), ws.chunks(), tile_base};
    void* params[] = {&op, &d, &list_idx, &list_val, &list_count, &cap, &ctx, &sa};
    // a plain launch: the only cross-CTA wait is on lower-numbered CTAs,
    // which are scheduled first
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kStreamThreads);
    cfg.dynamicSmemBytes = StreamLayout<LwCandOp<GT>, kLwStages>::kSmem;
    cfg.stream = ws.stream;
    err = cudaLaunchKernelExC(
        &cfg, reinterpret_cast<const void*>(&stream_compact_kernel<LwCandOp<GT>, kLwStages>),
        params);
    count_launch();
    if (err != cudaSuccess) return err;
  } else {
    const uint32_t grid = p.tiles < static_cast<uint32_t>(dev.sm_count * 8)
                              ? p.tiles : static_cast<uint32_t>(dev.sm_count * 8);
    lw_accumulate_plain_kernel<GT><<<grid, kThreads, 0, ws.stream>>>(g, e, gamma, d, other);
    count_launch();
    if ((err = cudaGetLastError()) != cudaSuccess) return err;
  }
  // 3 select
  LwArgs a;
  a.segs = segs;
  a.mbound = mbound;
  a.work_ptr = reinterpret_cast<const uint32_t*>(p.dev + p.off_work_ptr);
  a.work_seg = reinterpret_cast<const uint32_t*>(p.dev + p.off_work_seg);
  a.tile_base = tile_base;
  a.list_idx = list_idx;
  a.list_val = list_val;
  a.list_flags = list_flags;
  a.error = ws.u32(kOffError);
  a.count_out = count_out;
  a.tiles = p.tiles;
  a.cap = ws.cand_cap;
  a.use_list = streamable ? 1u : 0u;
  a.total_k = static_cast<uint32_t>(p.total_k);
  lw_select_kernel<<<p.n_select_ctas, kLwThreads, kLwSelectSmem, ws.stream>>>(e, idx_out,
                                                                              val_out, a);
  count_launch();
  return cudaGetLastError();
}

}  // namespace

void topk_layerwise_init_device(DeviceInfo& info) {
  cudaFuncSetAttribute(lw_select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                       kLwSelectSmem);
  info.lw_stream_per_sm_f32 = lw_stream_blocks_per_sm<float>();
  info.lw_stream_per_sm_bf16 = lw_stream_blocks_per_sm<uint16_t>();
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
  std::vector<LwSample> samples;
  uint32_t n_sampled = 0;
  uint64_t lo = 0, total_k = 0;
  for (uint32_t s = 0; s < n_seg; ++s) {
    const uint64_t hi = seg_end[s], ds = hi - lo, k = seg_k[s];
    LwSeg& x = segs[s];
    x = LwSeg{static_cast<uint32_t>(lo), static_cast<uint32_t>(hi), static_cast<uint32_t>(k),
              static_cast<uint32_t>(total_k), kLwNone, 0, 0, 0};
    if (k == 0 || ds == 0)
      x.kind = kLwNone;
    else if (k == ds)
      x.kind = kLwAll;
    else if (ds <= kLwSmemElems)
      x.kind = kLwWhole;
    else
      x.kind = kLwSampled;
    if (x.kind == kLwSampled) {
      // about one group of 4 per 256 coordinates, 512 .. 65536 groups
      const uint64_t gr = std::min<uint64_t>(std::max<uint64_t>(ds / 256, 512), 65536);
      x.groups = static_cast<uint32_t>(gr);
      x.slot = n_sampled++;
      x.nblk = static_cast<uint32_t>((gr + kLwSampleGroupsPerCta - 1) / kLwSampleGroupsPerCta);
      for (uint32_t b = 0; b < x.nblk; ++b) {
        const uint32_t q0 = b * kLwSampleGroupsPerCta;
        const uint32_t q1 = std::min<uint32_t>(x.groups, q0 + kLwSampleGroupsPerCta);
        samples.push_back(LwSample{s, q0, q1, 0});
      }
    }
    ends[s] = static_cast<uint32_t>(hi);
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
  // select work: the segments with pairs to write, longest first onto the
  // least loaded CTA
  std::vector<uint32_t> items;
  for (uint32_t s = 0; s < n_seg; ++s)
    if (segs[s].kind != kLwNone) items.push_back(s);
  std::stable_sort(items.begin(), items.end(), [&](uint32_t x, uint32_t y) {
    return select_cost(segs[x]) > select_cost(segs[y]);
  });
  // at least one CTA: it also writes the count and reports a failed stream
  const uint32_t n_ctas = static_cast<uint32_t>(std::max<size_t>(
      1, std::min<size_t>(items.size(), static_cast<size_t>(dev.sm_count))));
  std::vector<std::vector<uint32_t>> per(n_ctas);
  {
    using Load = std::pair<uint64_t, uint32_t>;
    std::priority_queue<Load, std::vector<Load>, std::greater<Load>> heap;
    for (uint32_t c = 0; c < n_ctas; ++c) heap.push(Load{0, c});
    for (uint32_t s : items) {
      Load l = heap.top();
      heap.pop();
      per[l.second].push_back(s);
      l.first += select_cost(segs[s]);
      heap.push(l);
    }
  }
  std::vector<uint32_t> work_ptr(n_ctas + 1, 0), work_seg;
  for (uint32_t c = 0; c < n_ctas; ++c) {
    work_ptr[c] = static_cast<uint32_t>(work_seg.size());
    work_seg.insert(work_seg.end(), per[c].begin(), per[c].end());
  }
  work_ptr[n_ctas] = static_cast<uint32_t>(work_seg.size());

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
  p.off_samples = take(sizeof(LwSample) * samples.size());
  p.off_work_ptr = take(sizeof(uint32_t) * work_ptr.size());
  p.off_work_seg = take(sizeof(uint32_t) * work_seg.size());
  const size_t upload = off;
  p.off_done = take(sizeof(uint32_t) * n_seg);
  p.off_hist = take(sizeof(uint32_t) * kSampleBins * n_sampled);
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
  put(p.off_samples, samples.data(), sizeof(LwSample) * samples.size());
  put(p.off_work_ptr, work_ptr.data(), sizeof(uint32_t) * work_ptr.size());
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
  if ((err = cudaMemsetAsync(p.dev + p.off_done, 0, zero_end - p.off_done, ws.stream)) !=
      cudaSuccess)
    return err;
  p.seg_end.assign(seg_end, seg_end + n_seg);
  p.seg_k.assign(seg_k, seg_k + n_seg);
  p.d = d;
  p.n_seg = n_seg;
  p.n_sampled = n_sampled;
  p.n_sample_ctas = static_cast<uint32_t>(samples.size());
  p.n_select_ctas = n_ctas;
  p.tiles = tiles;
  p.total_k = total_k;
  p.valid = true;
  return cudaSuccess;
}

cudaError_t launch_topk_layerwise(const void* g, bool g_bf16, float* e, float gamma, uint32_t d,
                                  uint32_t* idx_out, float* val_out, uint32_t* count_out,
                                  Workspace& ws, const DeviceInfo& dev) {
  if (g_bf16)
    return launch_typed(static_cast<const uint16_t*>(g), e, gamma, d, idx_out, val_out,
                        count_out, ws, dev);
  return launch_typed(static_cast<const float*>(g), e, gamma, d, idx_out, val_out, count_out,
                      ws, dev);
}

}  // namespace efs
