// topk.cu — error-feedback + Top-k sparsifier (the paper's baseline, Lemma 2)
// as a radix select on the magnitude bits, followed by the same ordered
// compaction as the hard-threshold path.
//
// Order. Every coordinate j gets the 63-bit composite key
//     K_j = (bits(|a_j|) << 32) | (~j & 0xffffffff),
// where bits(|a_j|) is the fp32 encoding with the sign cleared. For
// non-negative IEEE values the encoding orders like the value (NaN above
// +inf), and the low word makes a lower index rank higher among equal
// magnitudes. All K_j are distinct, so the Top-k set is exactly
// { j : K_j >= K_(k) } for the k-th largest key K_(k).
//
// Passes (launches per call: one memset of the small control block + 3):
//   A  accumulate: a = fmaf(gamma, g, e) is written over e, and a histogram
//      of the top 11 key bits (62..52) is built in shared memory and merged
//      into global memory. 12 B/coordinate, the algorithmic traffic.
//   R  refine (one cooperative launch, all CTAs co-resident): digit by digit
//      (bits 51..42, 41..32, 31..21, 20..10, 9..0) histogram the coordinates
//      whose key shares the bits fixed so far, pick the digit that contains
//      the k-th key, until the remaining rank equals the bucket size. The
//      first refine digit reads a (4 B/coordinate) and compacts the bucket's
//      keys into a candidate buffer when it fits; later digits read only
//      candidates. Every CTA selects redundantly from the merged histogram
//      after a bounded grid barrier, so control flow is uniform.
//   Z  select: the ordered compaction with predicate K_j >= threshold; e is
//      zeroed at the selected coordinates (the residual a - C(a)).
#include "compact.cuh"
#include "gradient.cuh"
#include "internal.h"

namespace efs {
namespace {

// LSB of each digit of the composite key; digit 0 is bits 62..52.
__device__ __forceinline__ int digit_shift(int level) {
  return level == 0 ? 52 : level == 1 ? 42 : level == 2 ? 32 : level == 3 ? 21 : level == 4 ? 10 : 0;
}

__device__ __forceinline__ uint64_t composite_key(float a, uint64_t j) {
  return (static_cast<uint64_t>(__float_as_uint(a) & 0x7fffffffu) << 32) |
         static_cast<uint64_t>(~static_cast<uint32_t>(j));
}

struct TopkArgs {
  uint32_t* hist;        // [kHistLevels][kHistBins]
  uint64_t* cand0;
  uint64_t* cand1;
  uint32_t* cand_count;  // [kHistLevels]
  uint32_t cand_cap;
  uint64_t* threshold;
  uint32_t* bar_arrive;
  uint32_t* bar_gen;
  uint32_t* error;
  uint64_t wait_limit_ns;
};

// Lanes holding equal bins add once, with the number of lanes.
__device__ __forceinline__ void hist_add_warp(uint32_t* h, uint32_t bin, bool valid) {
  const uint32_t key = valid ? bin : 0xffffffffu;
  const uint32_t peers = __match_any_sync(0xffffffffu, key);
  if (valid && (__ffs(peers) - 1) == static_cast<int>(threadIdx.x & 31))
    atomicAdd(&h[bin], static_cast<uint32_t>(__popc(peers)));
}

// ------------------------------------------------------------------ pass A
template <typename GT, bool kVec>
__global__ void __launch_bounds__(kThreads)
    topk_accumulate_kernel(const GT* __restrict__ g, float* __restrict__ e, float gamma,
                           uint32_t d, uint32_t num_tiles, uint32_t* __restrict__ hist0) {
  __shared__ uint32_t s_hist[kHistBins];
  for (int b = threadIdx.x; b < kHistBins; b += kThreads) s_hist[b] = 0;
  __syncthreads();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (uint32_t tile = blockIdx.x; tile < num_tiles; tile += gridDim.x) {
    const uint64_t first = element_index(tile, warp, 0, lane, 0);
    const bool full_tile = static_cast<uint64_t>(tile + 1) * kTileElems <= d;
    if (kVec && full_tile) {
      GradVec<GT> gv[kUnits];
      float4 ev[kUnits];
#pragma unroll
      for (int v = 0; v < kUnits; ++v) {
        gv[v].load(g + first + v * 128);
        ev[v] = ld_stream_f4(e + first + v * 128);
      }
#pragma unroll
      for (int v = 0; v < kUnits; ++v) {
        float4 a;
        a.x = __fmaf_rn(gamma, gv[v][0], ev[v].x);
        a.y = __fmaf_rn(gamma, gv[v][1], ev[v].y);
        a.z = __fmaf_rn(gamma, gv[v][2], ev[v].z);
        a.w = __fmaf_rn(gamma, gv[v][3], ev[v].w);
        // default caching: the refine and select passes re-read a
        *reinterpret_cast<float4*>(e + first + v * 128) = a;
        hist_add_warp(s_hist, (__float_as_uint(a.x) & 0x7fffffffu) >> 20, true);
        hist_add_warp(s_hist, (__float_as_uint(a.y) & 0x7fffffffu) >> 20, true);
        hist_add_warp(s_hist, (__float_as_uint(a.z) & 0x7fffffffu) >> 20, true);
        hist_add_warp(s_hist, (__float_as_uint(a.w) & 0x7fffffffu) >> 20, true);
      }
    } else {
#pragma unroll
      for (int v = 0; v < kUnits; ++v) {
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const uint64_t i = first + v * 128 + j;
          const bool ok = i < d;
          float x = 0.0f;
          if (ok) {
            x = __fmaf_rn(gamma, grad_scalar(g, i), e[i]);
            e[i] = x;
          }
          hist_add_warp(s_hist, (__float_as_uint(x) & 0x7fffffffu) >> 20, ok);
        }
      }
    }
  }
  __syncthreads();
  for (int b = threadIdx.x; b < kHistBins; b += kThreads)
    if (s_hist[b]) atomicAdd(&hist0[b], s_hist[b]);
}

// ------------------------------------------------------------------ pass R
struct Selection {
  uint32_t bin, k_rem, n_in, found;
};

// Find the bin holding the k_rem-th largest key of a histogram of nbins
// (2048 or 1024) bins, scanning from the highest bin. Whole CTA; uniform.
__device__ Selection select_bin(const uint32_t* hist, uint32_t nbins, uint32_t k_rem) {
  __shared__ uint32_t s_part[kThreads];
  __shared__ Selection s_sel;
  const int t = threadIdx.x;
  const uint32_t per = nbins / kThreads;  // 8 or 4 bins per thread
  uint32_t c[8];
  uint32_t sum = 0;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    c[i] = (static_cast<uint32_t>(i) < per) ? __ldcg(hist + t * per + i) : 0u;
    sum += c[i];
  }
  if (t == 0) s_sel = Selection{0, 0, 0, 0};
  s_part[t] = sum;
  __syncthreads();
  if (t < 32) {  // exclusive suffix sums over the 256 per-thread totals
    uint32_t loc[8], tot = 0;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      loc[i] = s_part[t * 8 + i];
      tot += loc[i];
    }
    uint32_t incl = tot;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t n = __shfl_down_sync(0xffffffffu, incl, o);
      if (t + o < 32) incl += n;
    }
    uint32_t above = incl - tot;
#pragma unroll
    for (int i = 7; i >= 0; --i) {
      s_part[t * 8 + i] = above;
      above += loc[i];
    }
  }
  __syncthreads();
  const uint32_t above = s_part[t];
  if (above < k_rem && k_rem - above <= sum) {
    uint32_t r = k_rem - above;
    bool done = false;
#pragma unroll
    for (int i = 7; i >= 0; --i) {
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

__device__ __forceinline__ void refine_visit(uint64_t key, bool valid, uint64_t prefix,
                                             int sh_prev, int sh, uint32_t nb, bool compact,
                                             uint64_t* dst, uint32_t* dst_count,
                                             uint32_t cap, uint32_t* s_hist) {
  const bool match = valid && (key >> sh_prev) == prefix;
  if (match) atomicAdd(&s_hist[(key >> sh) & (nb - 1)], 1u);
  if (compact) warp_append(match, key, dst, dst_count, cap);
}

template <bool kVec>
__global__ void __launch_bounds__(kThreads)
    topk_refine_kernel(const float* __restrict__ a, uint32_t d, uint32_t k, TopkArgs args) {
  __shared__ uint32_t s_hist[kHistBins];
  if (k == 0) {
    if (blockIdx.x == 0 && threadIdx.x == 0) *args.threshold = 1ull << 63;  // selects nothing
    return;
  }
  Selection s = select_bin(args.hist, kHistBins, k);
  bool ok = s.found != 0;
  uint64_t prefix = s.bin;
  uint32_t k_rem = s.k_rem, n_in = s.n_in;
  int level = 0;
  int src = -1;  // -1: scan all of a; 0/1: scan candidate buffer 0/1
  uint32_t src_count = d;

  while (ok && n_in != k_rem && level < kHistLevels - 1) {
    ++level;
    const int sh_prev = digit_shift(level - 1), sh = digit_shift(level);
    const int bits = sh_prev - sh;
    const uint32_t nb = 1u << bits;
    const bool compact = n_in <= args.cand_cap;
    const int dst = (src == 0) ? 1 : 0;
    uint64_t* dst_buf = dst ? args.cand1 : args.cand0;
    uint32_t* dst_count = args.cand_count + level;
    for (uint32_t b = threadIdx.x; b < nb; b += kThreads) s_hist[b] = 0;
    __syncthreads();

    if (src < 0) {
      const uint64_t units = (static_cast<uint64_t>(d) + 3) / 4;
      const uint64_t full_units = d / 4;
      for (uint64_t base = static_cast<uint64_t>(blockIdx.x) * kThreads; base < units;
           base += static_cast<uint64_t>(gridDim.x) * kThreads) {
        const uint64_t u = base + threadIdx.x;
        float x[4];
        bool valid[4];
        if (kVec && u < full_units) {
          const float4 q = __ldcg(reinterpret_cast<const float4*>(a) + u);
          x[0] = q.x; x[1] = q.y; x[2] = q.z; x[3] = q.w;
          valid[0] = valid[1] = valid[2] = valid[3] = true;
        } else {
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const uint64_t i = u * 4 + j;
            valid[j] = i < d;
            x[j] = valid[j] ? __ldcg(a + i) : 0.0f;
          }
        }
#pragma unroll
        for (int j = 0; j < 4; ++j)
          refine_visit(composite_key(x[j], u * 4 + j), valid[j], prefix, sh_prev, sh, nb,
                       compact, dst_buf, dst_count, args.cand_cap, s_hist);
      }
    } else {
      const uint64_t* src_buf = src ? args.cand1 : args.cand0;
      for (uint64_t base = static_cast<uint64_t>(blockIdx.x) * kThreads; base < src_count;
           base += static_cast<uint64_t>(gridDim.x) * kThreads) {
        const uint64_t i = base + threadIdx.x;
        const bool valid = i < src_count;
        const uint64_t key = valid ? __ldcg(src_buf + i) : 0ull;
        refine_visit(key, valid, prefix, sh_prev, sh, nb, compact, dst_buf, dst_count,
                     args.cand_cap, s_hist);
      }
    }
    __syncthreads();
    uint32_t* gh = args.hist + level * kHistBins;
    for (uint32_t b = threadIdx.x; b < nb; b += kThreads)
      if (s_hist[b]) atomicAdd(&gh[b], s_hist[b]);
    if (!grid_barrier(args.bar_arrive, args.bar_gen, args.wait_limit_ns, args.error)) {
      ok = false;
      break;
    }
    s = select_bin(gh, nb, k_rem);
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
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    // an unfound bin or an unresolved rank means the histograms disagree
    // with the data (e changed during the call); the barrier latches its own
    if (!s.found || n_in != k_rem) atomicOr(args.error, kDevErrBadInput);
    ok = ok && n_in == k_rem;
    *args.threshold = ok ? (prefix << digit_shift(level)) : (1ull << 63);
  }
}

// ------------------------------------------------------------------ pass Z
template <bool kVec>
__global__ void __launch_bounds__(kThreads)
    topk_select_kernel(float* __restrict__ e, uint32_t d, const uint64_t* __restrict__ threshold,
                       uint32_t k, uint32_t* __restrict__ idx_out, float* __restrict__ val_out,
                       uint32_t* __restrict__ count_out, ScanCtx ctx) {
  const uint32_t tile = blockIdx.x;
  const uint64_t thr = __ldcg(threshold);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const uint64_t first = element_index(tile, warp, 0, lane, 0);
  float a[kUnits][4];
  uint32_t sel[kUnits];
  const bool full_tile = static_cast<uint64_t>(tile + 1) * kTileElems <= d;
  if (kVec && full_tile) {
    float4 q[kUnits];
#pragma unroll
    for (int v = 0; v < kUnits; ++v) q[v] = __ldcg(reinterpret_cast<const float4*>(e + first + v * 128));
#pragma unroll
    for (int v = 0; v < kUnits; ++v) {
      a[v][0] = q[v].x; a[v][1] = q[v].y; a[v][2] = q[v].z; a[v][3] = q[v].w;
    }
  } else {
#pragma unroll
    for (int v = 0; v < kUnits; ++v)
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const uint64_t i = first + v * 128 + j;
        a[v][j] = i < d ? __ldcg(e + i) : 0.0f;
      }
  }
#pragma unroll
  for (int v = 0; v < kUnits; ++v) {
    sel[v] = 0;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const uint64_t i = first + v * 128 + j;
      if (i < d && composite_key(a[v][j], i) >= thr) {
        sel[v] |= 1u << j;
        e[i] = 0.0f;  // residual of a sent coordinate
      }
    }
  }
  compact_tile(ctx, tile, sel, a, idx_out, val_out, count_out, k);
}

template <typename GT>
cudaError_t launch_typed(const GT* g, float* e, float gamma, uint32_t k, uint32_t d,
                         uint32_t* idx_out, float* val_out, uint32_t* count_out, Workspace& ws,
                         const DeviceInfo& dev) {
  const uint32_t tiles = tiles_for(d);
  cudaError_t err = cudaMemsetAsync(ws.base + kOffTopkReset, 0, kTopkResetBytes, ws.stream);
  if (err != cudaSuccess) return err;

  const bool e_vec = reinterpret_cast<uintptr_t>(e) % 16 == 0;
  const bool vec = e_vec && reinterpret_cast<uintptr_t>(g) % (4 * sizeof(GT)) == 0;
  const uint32_t grid_a = static_cast<uint32_t>(
      tiles < static_cast<uint32_t>(dev.sm_count * 4) ? tiles : dev.sm_count * 4);
  uint32_t* hist = ws.u32(kOffHist);
  if (vec)
    topk_accumulate_kernel<GT, true><<<grid_a, kThreads, 0, ws.stream>>>(g, e, gamma, d, tiles, hist);
  else
    topk_accumulate_kernel<GT, false><<<grid_a, kThreads, 0, ws.stream>>>(g, e, gamma, d, tiles, hist);
  count_launch();
  if ((err = cudaGetLastError()) != cudaSuccess) return err;

  TopkArgs args;
  args.hist = hist;
  args.cand0 = ws.cand(0);
  args.cand1 = ws.cand(1);
  args.cand_count = ws.u32(kOffCandCount);
  args.cand_cap = ws.cand_cap;
  args.threshold = ws.u64(kOffThreshold);
  args.bar_arrive = ws.u32(kOffBarArrive);
  args.bar_gen = ws.u32(kOffBarGen);
  args.error = ws.u32(kOffError);
  args.wait_limit_ns = wait_limit_ns();
  const float* a = e;
  void* params[] = {(void*)&a, (void*)&d, (void*)&k, (void*)&args};
  const void* fn = e_vec ? reinterpret_cast<const void*>(&topk_refine_kernel<true>)
                         : reinterpret_cast<const void*>(&topk_refine_kernel<false>);
  err = cudaLaunchCooperativeKernel(fn, dim3(dev.refine_blocks), dim3(kThreads), params, 0,
                                    ws.stream);
  count_launch();
  if (err != cudaSuccess) return err;

  const ScanCtx ctx = next_scan_ctx(ws, tiles);
  if (e_vec)
    topk_select_kernel<true><<<tiles, kThreads, 0, ws.stream>>>(e, d, args.threshold, k, idx_out,
                                                                val_out, count_out, ctx);
  else
    topk_select_kernel<false><<<tiles, kThreads, 0, ws.stream>>>(e, d, args.threshold, k, idx_out,
                                                                 val_out, count_out, ctx);
  count_launch();
  return cudaGetLastError();
}

}  // namespace

int topk_refine_blocks_per_sm() {
  int a = 0, b = 0;
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&a, topk_refine_kernel<true>, kThreads, 0);
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&b, topk_refine_kernel<false>, kThreads, 0);
  return a < b ? a : b;
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
                        Workspace& ws, const DeviceInfo& dev) {
  if (g_bf16)
    return launch_typed(static_cast<const uint16_t*>(g), e, gamma, k, d, idx_out, val_out,
                        count_out, ws, dev);
  return launch_typed(static_cast<const float*>(g), e, gamma, k, d, idx_out, val_out, count_out,
                      ws, dev);
}

}  // namespace efs
