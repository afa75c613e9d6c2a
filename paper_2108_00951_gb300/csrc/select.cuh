// select.cuh — block-level building blocks of the exact Top-k selections:
// warp-aggregated histogram adds, block scans, the histogram bin holding a
// given rank, and the magnitude threshold of a list of fp32 values with the
// lowest-position tie rule.
//
// Order used throughout: the magnitude bits bits(|a|) (the fp32 encoding with
// the sign cleared) order like |a| for every non-negative IEEE value, NaN
// above +inf; among equal magnitudes the lower position ranks higher. In
// every list these routines see, position order is index order.
#pragma once

#include "internal.h"

namespace efs {

// Lanes holding equal bins add once, with the number of lanes.
__device__ __forceinline__ void hist_add_warp(uint32_t* h, uint32_t bin, bool valid) {
  const uint32_t key = valid ? bin : 0xffffffffu;
  const uint32_t peers = __match_any_sync(0xffffffffu, key);
  if (valid && (__ffs(peers) - 1) == static_cast<int>(threadIdx.x & 31))
    atomicAdd(&h[bin], static_cast<uint32_t>(__popc(peers)));
}

struct Selection {
  uint32_t bin, k_rem, n_in, found;
};

// Exclusive suffix sum over the threads of the CTA (the sum of v over every
// higher thread index) and the block total. Whole CTA; blockDim.x a multiple
// of 32; s_w holds blockDim.x / 32 words.
__device__ __forceinline__ uint32_t block_suffix_exclusive(uint32_t v, uint32_t& total,
                                                           uint32_t* s_w) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int nw = static_cast<int>(blockDim.x >> 5);
  uint32_t incl = v;  // v summed over this lane and the higher lanes
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t x = __shfl_down_sync(0xffffffffu, incl, o);
    if (lane + o < 32) incl += x;
  }
  __syncthreads();  // a previous use of s_w is complete
  if (lane == 0) s_w[warp] = incl;
  __syncthreads();
  uint32_t wsuf = lane < nw ? s_w[lane] : 0u;  // warp totals over warps >= lane
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t x = __shfl_down_sync(0xffffffffu, wsuf, o);
    if (lane + o < 32) wsuf += x;
  }
  total = __shfl_sync(0xffffffffu, wsuf, 0);
  const uint32_t higher = __shfl_sync(0xffffffffu, wsuf, (warp + 1) & 31);
  return (warp + 1 < 32 ? higher : 0u) + incl - v;
}

// Find the bin holding the k_rem-th largest key of a histogram of nbins
// (2048 or 1024) bins, scanning from the highest bin. Whole CTA of kBlock
// threads (kBlock <= nbins); uniform result. kGlobal: the histogram is in
// global memory (read through L2), else in shared memory. s_w holds
// kBlock / 32 words.
template <int kBlock, bool kGlobal>
__device__ Selection select_bin(const uint32_t* hist, uint32_t nbins, uint32_t k_rem,
                                uint32_t* s_w) {
  constexpr int kMaxPer = kHistBins / kBlock;
  __shared__ Selection s_sel;
  const int t = threadIdx.x;
  const uint32_t per = nbins / kBlock;
  uint32_t c[kMaxPer];
  uint32_t sum = 0;
#pragma unroll
  for (int i = 0; i < kMaxPer; ++i) {
    c[i] = (static_cast<uint32_t>(i) < per)
               ? (kGlobal ? __ldcg(hist + t * per + i) : hist[t * per + i]) : 0u;
    sum += c[i];
  }
  if (t == 0) s_sel = Selection{0, 0, 0, 0};
  uint32_t total;
  const uint32_t above = block_suffix_exclusive(sum, total, s_w);  // orders the reset
  if (above < k_rem && k_rem - above <= sum) {
    uint32_t r = k_rem - above;
    bool done = false;
#pragma unroll
    for (int i = kMaxPer - 1; i >= 0; --i) {
      if (!done && static_cast<uint32_t>(i) < per) {
        if (c[i] >= r) {
          s_sel = Selection{t * per + i, r, c[i], 1u};
          done = true;
        } else {
          r -= c[i];
        }
      }
    }
  }
  __syncthreads();
  const Selection s = s_sel;
  __syncthreads();
  return s;
}

// Exclusive block-wide prefix sum of one value per thread; also returns the
// block total. Whole CTA of kBlock threads; s_w holds kBlock/32 words.
template <int kBlock>
__device__ __forceinline__ uint32_t block_exclusive(uint32_t v, uint32_t& total, uint32_t* s_w) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t incl = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t x = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += x;
  }
  __syncthreads();
  if (lane == 31) s_w[warp] = incl;
  __syncthreads();
  uint32_t before = 0;
  total = 0;
  for (int w = 0; w < kBlock / 32; ++w) {
    const uint32_t x = s_w[w];
    before += w < warp ? x : 0u;
    total += x;
  }
  return before + incl - v;
}

// Zeroes a Top-k state block, the grid's threads striding over it (the
// block belongs to the previous call on the workspace, which is complete).
__device__ __forceinline__ void clear_state(uint32_t* block) {
  constexpr uint32_t kWords = static_cast<uint32_t>(kTkStateBytes / sizeof(uint4));
  uint4* b4 = reinterpret_cast<uint4*>(block);
  for (uint32_t w = blockIdx.x * blockDim.x + threadIdx.x; w < kWords; w += gridDim.x * blockDim.x)
    b4[w] = make_uint4(0u, 0u, 0u, 0u);
}


// Threshold of a magnitude selection: |a| > B is taken, and |a| == B too,
// except that with `ties` set only up to list position `last`.
struct SmallSelection {
  uint32_t B;       // threshold magnitude bits
  uint32_t ties;    // 1: magnitudes equal to B are taken only up to `last`
  uint32_t last;    // list position of the last taken magnitude equal to B
};

// Magnitude bits of list position i, from shared or global memory (the
// stored words may carry the sign; it is cleared here).
struct MagsShared {
  const uint32_t* bits;
  __device__ __forceinline__ uint32_t operator()(uint32_t i) const {
    return bits[i] & 0x7fffffffu;
  }
};
struct MagsGlobal {
  const float* val;
  __device__ __forceinline__ uint32_t operator()(uint32_t i) const {
    return __float_as_uint(__ldcg(val + i)) & 0x7fffffffu;
  }
};

// Histogram pass of a level over the `cnt` magnitudes: those in the window
// [B, B + W) (W == 0: all) add to bin (m - B) >> sh. Whole CTA of kBlock.
template <int kBlock, class Mags>
__device__ __forceinline__ void window_hist(const Mags& mag, uint32_t cnt, uint32_t B, uint32_t W,
                                            int sh, uint32_t* s_hist) {
  for (uint32_t b0 = threadIdx.x; b0 < cnt; b0 += 4 * kBlock) {
    uint32_t m[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const uint32_t i = b0 + j * kBlock;
      m[j] = i < cnt ? mag(i) : 0u;
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const uint32_t off = m[j] - B;
      if (b0 + j * kBlock < cnt && m[j] >= B && (W == 0 || off < W))
        atomicAdd(&s_hist[off >> sh], 1u);
    }
  }
}

// The threshold taking exactly k (1 <= k <= n) of the n magnitudes, whose
// minimum and maximum are lo and hi. Digit levels narrow a window [B, B + W)
// of magnitude bit patterns: level 0 splits [lo, hi] into at most 2048 bins,
// each later level splits the chosen bin into at most 2048 sub-bins. The
// levels stop when the window holds exactly the remaining rank, or is one
// magnitude wide; then equal magnitudes are taken in position order up to
// `last`. Whole CTA of kBlock threads; uniform result; false when the
// histograms do not find the rank (never for a well-formed list).
template <int kBlock, class Mags>
__device__ bool threshold_levels(const Mags& mag, uint32_t n, uint32_t k, uint32_t lo,
                                 uint32_t hi, uint32_t* s_hist, uint32_t* s_w,
                                 SmallSelection& out) {
  __shared__ uint32_t s_last;
  const int tid = threadIdx.x;
  uint32_t B = lo, W = 0, k_rem = k, n_in = n;
  int sh = 0;
  while (((hi - lo) >> sh) >= static_cast<uint32_t>(kHistBins)) ++sh;
  if (hi == lo) W = 1;  // every magnitude is the same
  while (W != 1 && n_in != k_rem) {
    for (uint32_t b = tid; b < static_cast<uint32_t>(kHistBins); b += kBlock) s_hist[b] = 0;
    __syncthreads();
    window_hist<kBlock>(mag, n, B, W, sh, s_hist);
    __syncthreads();
    const Selection s = select_bin<kBlock, false>(s_hist, kHistBins, k_rem, s_w);
    if (!s.found) return false;
    B += s.bin << sh;
    W = 1u << sh;
    k_rem = s.k_rem;
    n_in = s.n_in;
    int bits = 0;
    while ((1u << bits) < W) ++bits;
    sh = bits > 11 ? bits - 11 : 0;
  }
  // at a one-wide threshold with more equal magnitudes than are taken, only
  // the first k_rem of them in position order
  const bool ties = W == 1 && n_in != k_rem;
  if (tid == 0) s_last = 0xffffffffu;
  if (ties) {
    const uint32_t per = (n + kBlock - 1) / kBlock;
    const uint32_t a0 = tid * per < n ? tid * per : n, a1 = a0 + per < n ? a0 + per : n;
    uint32_t cnt = 0;
    for (uint32_t i = a0; i < a1; ++i) cnt += mag(i) == B ? 1u : 0u;
    uint32_t total;
    const uint32_t before = block_exclusive<kBlock>(cnt, total, s_w);
    if (before < k_rem && k_rem <= before + cnt) {
      uint32_t r = k_rem - before;
      for (uint32_t i = a0; i < a1; ++i)
        if (mag(i) == B && --r == 0) {
          s_last = i;
          break;
        }
    }
  }
  __syncthreads();
  const uint32_t last = ties ? s_last : 0xffffffffu;
  __syncthreads();  // s_last may be reset by the next call
  out = SmallSelection{B, ties ? 1u : 0u, last};
  return true;
}

// Whether list position i with magnitude bits m is taken by selection s.
__device__ __forceinline__ bool selected(const SmallSelection& s, uint32_t m, uint32_t i) {
  return m > s.B || (m == s.B && (!s.ties || i <= s.last));
}

}  // namespace efs
