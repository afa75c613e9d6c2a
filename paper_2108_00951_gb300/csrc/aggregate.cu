// aggregate.cu — decompress and sum n workers' sparse vectors (the exchange
// step of Algorithm 1, Delta_bar = (1/n) sum_i Delta_i, without the 1/n).
//
// Deterministic by construction: the dense range [0, d) is cut into tiles of
// kAggTile coordinates; one CTA owns a tile in shared memory, starts it at
// +0.0f and adds worker 0's pairs, then worker 1's, ..., with a CTA barrier
// between workers. Within one worker the indices are distinct (the lists are
// strictly ascending), so no two threads add to the same slot at once, and
// every coordinate receives its contributions in ascending worker order —
// the same fp32 sum as the plain sequential loop.
//
// Kernel 1 finds, by binary search, where each worker's sorted list crosses
// each tile boundary; kernel 2 does the reduction and writes each dense tile
// once with 16-byte stores. Traffic: 8 B per pair read + 4 B per coordinate
// written (+ the small offsets table).
//
// The same reduction can instead end in the model update that follows the
// exchange (sparse_aggregate_apply): Delta' = alpha * s rounded once, then
// x <- x - Delta' (Algorithm 1), or m <- fmaf(mu, m, Delta') and
// x <- fmaf(-lr, Delta' + m, x) (the Appendix's EF SGD with momentum by
// gradient compression). The dense sum then never reaches memory: 8 B per
// coordinate (read and write x), 16 B with momentum, instead of writing the
// sum and a second pass that reads it back.
#include "internal.h"

namespace efs {
namespace {

struct AggPtrs {
  const uint32_t* idx[kMaxWorkers];
  const float* val[kMaxWorkers];
  const uint32_t* tiles[kMaxWorkers];  // the lists' tile indexes, when the caller has them
};

// off[i * (tiles + 1) + t] = number of entries of list i below t * kAggTile;
// off[i * (tiles + 1) + tiles] = counts[i]. Grid: blockIdx.y = list, x over
// the tiles + 1 entries. Two ways to the same numbers, chosen per list:
//  - a list with at least (tiles + 1) / 16 and at most 8 (tiles + 1) entries
//    is scattered: entry p (p = 0..count, count standing for the end) owns the
//    tiles t with list[p - 1] < t * kAggTile <= list[p] and writes p there —
//    two loads per entry and no dependent chain; a run of more than 8 tiles
//    is written by the whole warp;
//  - other lists: one binary search per tile (14-23 dependent loads, but
//    independent of the list's length).
// Either way every entry lies in [0, count]; a list that is not strictly
// ascending is latched as bad input (scatter) and may leave entries the
// reduction clamps to the list.
__global__ void __launch_bounds__(kThreads)
    agg_offsets_kernel(AggPtrs p, const uint32_t* __restrict__ counts, uint32_t n,
                       uint32_t tiles, uint32_t* __restrict__ off, uint32_t* __restrict__ error) {
  griddep_wait();                // the lists and counts come from the kernels before
  griddep_launch_dependents();    // the reduction may be scheduled (it waits for this grid)
  const uint32_t per = tiles + 1;
  const uint32_t i = blockIdx.y;
  const uint32_t tx = blockIdx.x * kThreads + threadIdx.x;
  const uint32_t stride = gridDim.x * kThreads;  // >= per
  const int lane = threadIdx.x & 31;
  const uint32_t cnt = counts[i];
  const uint32_t* x = p.idx[i];
  uint32_t* o = off + static_cast<uint64_t>(i) * per;
  const bool scatter = cnt >= per / 16 && static_cast<uint64_t>(cnt) <= 8ull * per;
  if (!scatter) {
    if (tx >= per) return;
    uint32_t result = cnt;
    if (tx < tiles) {
      const uint64_t target = static_cast<uint64_t>(tx) * kAggTile;
      uint32_t lo = 0, hi = cnt;
      while (lo < hi) {
        const uint32_t mid = lo + (hi - lo) / 2;
        if (static_cast<uint64_t>(__ldg(x + mid)) < target)
          lo = mid + 1;
        else
          hi = mid;
      }
      result = lo;
    }
    o[tx] = result;
    return;
  }
  bool bad = false;
#pragma unroll 1
  for (uint32_t q = 0; q < 9; ++q) {  // positions tx + q * stride <= cnt (cnt <= 8 per)
    const uint32_t pos = tx + q * stride;
    const bool has = pos <= cnt;
    uint32_t t_lo = 1, t_hi = 0;  // empty
    if (has) {
      const uint32_t cur = pos < cnt ? __ldg(x + pos) : 0u;
      const uint32_t prev = pos > 0 ? __ldg(x + pos - 1) : 0u;
      if (pos > 0 && pos < cnt && prev >= cur) bad = true;  // not strictly ascending
      t_lo = pos == 0 ? 0u : min(prev / kAggTile + 1u, per);
      t_hi = pos == cnt ? tiles : min(cur / kAggTile, tiles - 1u);
      if (pos < cnt && t_hi < t_lo) t_lo = t_hi + 1;  // nothing (malformed, or a shared tile)
    }
    const bool mine = has && t_lo <= t_hi && t_hi - t_lo < 8;
    if (mine)
      for (uint32_t t = t_lo; t <= t_hi; ++t) o[t] = pos;
    // longer runs: the whole warp writes them, one run after another
    uint32_t m = __ballot_sync(0xffffffffu, has && t_lo <= t_hi && !mine);
    while (m) {
      const int l = __ffs(m) - 1;
      m &= m - 1;
      const uint32_t a = __shfl_sync(0xffffffffu, t_lo, l);
      const uint32_t b = __shfl_sync(0xffffffffu, t_hi, l);
      const uint32_t v = __shfl_sync(0xffffffffu, pos, l);
      for (uint32_t t = a + lane; t <= b; t += 32) o[t] = v;
    }
  }
  if (bad) atomicOr(error, kDevErrBadInput);
}

// What the reduction does with a finished tile.
enum AggMode { kAggDense = 0, kAggSgd = 1, kAggMomentum = 2 };
struct AggOut {
  float* out;  // kAggDense: the sum; otherwise x, updated in place
  float* m;    // kAggMomentum: the momentum, updated in place
  float alpha, mu, lr;
};

template <int kMode>
__device__ __forceinline__ void apply_update(const AggOut& o, float s, float& x, float& m) {
  const float delta = __fmul_rn(o.alpha, s);
  if constexpr (kMode == kAggSgd) {
    x = __fsub_rn(x, delta);
  } else {
    m = __fmaf_rn(o.mu, m, delta);
    x = __fmaf_rn(-o.lr, __fadd_rn(delta, m), x);
  }
}

// 4-byte asynchronous copy global -> shared (no register staging).
__device__ __forceinline__ void cp_async_4(void* dst, const void* src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(
                   static_cast<uint32_t>(__cvta_generic_to_shared(dst))),
               "l"(src)
               : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.wait_all;" ::: "memory");
}

// Bulk prefetch of [p, p + bytes) into L2 (16-byte aligned, bytes % 16 == 0).
__device__ __forceinline__ void prefetch_l2_bulk(const void* p, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}

template <bool kVec, int kMode>
__global__ void __launch_bounds__(kThreads)
    agg_reduce_kernel(AggPtrs p, uint32_t n, uint32_t d, uint32_t tiles,
                      const uint32_t* __restrict__ off, const uint32_t* __restrict__ counts,
                      AggOut o, uint32_t* __restrict__ error) {
  __shared__ __align__(16) float acc[kAggTile];
  __shared__ uint32_t s_lo[kMaxWorkers], s_pre[kMaxWorkers + 1];
  __shared__ uint32_t st_idx[kAggStage];
  __shared__ float st_val[kAggStage];
  const uint32_t t = blockIdx.x;
  const int lane = threadIdx.x & 31;
  const uint64_t j0 = static_cast<uint64_t>(t) * kAggTile;
  for (int q = threadIdx.x; q < kAggTile / 4; q += kThreads)
    reinterpret_cast<float4*>(acc)[q] = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
  if constexpr (kMode != kAggDense) {
    // the tile's x (and m), read by the epilogue, on their way to L2 while
    // the pairs are gathered (a prefetch: no data moves into the CTA)
    if (kVec && threadIdx.x == 0 && j0 + kAggTile <= d) {
      prefetch_l2_bulk(o.out + j0, kAggTile * sizeof(float));
      if constexpr (kMode == kAggMomentum) prefetch_l2_bulk(o.m + j0, kAggTile * sizeof(float));
    }
  }
  griddep_wait();  // the offsets (and everything before them) are complete
  griddep_launch_dependents();  // the next kernel waits for this grid before its reads
  for (uint32_t i = threadIdx.x; i < n; i += kThreads) {
    // the list's range in this tile: from the offsets kernel, or from the
    // caller's tile index, clamped to the list (never out of bounds)
    const uint32_t* r = off ? off + static_cast<uint64_t>(i) * (tiles + 1) : p.tiles[i];
    const uint32_t cnt = counts[i];
    uint32_t lo = min(r[t], cnt), hi = min(r[t + 1], cnt);
    s_lo[i] = lo;
    s_pre[i + 1] = hi > lo ? hi - lo : 0u;  // this tile's pairs of worker i
  }
  __syncthreads();
  if (threadIdx.x < 32) {  // s_pre: the tile's pairs of the workers before each one
    uint32_t carry = 0;
    for (uint32_t i0 = 0; i0 < n; i0 += 32) {
      const uint32_t i = i0 + lane;
      uint32_t v = i < n ? s_pre[i + 1] : 0u;
#pragma unroll
      for (int o2 = 1; o2 < 32; o2 <<= 1) {
        const uint32_t x = __shfl_up_sync(0xffffffffu, v, o2);
        if (lane >= o2) v += x;
      }
      if (i < n) s_pre[i + 1] = carry + v;
      carry += __shfl_sync(0xffffffffu, v, 31);
    }
    if (lane == 0) s_pre[0] = 0;
  }
  __syncthreads();
  bool bad = false;
  const uint32_t total = s_pre[n];
  // The tile's pairs of all workers, in worker order, a stage at a time:
  // every copy of a stage is in flight at once (one round trip), then the
  // stage is added worker by worker, with a barrier between workers so that
  // each coordinate receives its contributions in worker order.
  for (uint32_t b0 = 0; b0 < total; b0 += kAggStage) {
    const uint32_t bn = total - b0 < kAggStage ? total - b0 : kAggStage;
    {
      uint32_t i = 0;
      for (uint32_t q = threadIdx.x; q < bn; q += kThreads) {
        const uint32_t gp = b0 + q;
        while (s_pre[i + 1] <= gp) ++i;
        const uint32_t src = s_lo[i] + (gp - s_pre[i]);
        cp_async_4(st_idx + q, p.idx[i] + src);
        cp_async_4(st_val + q, p.val[i] + src);
      }
    }
    cp_async_wait_all();
    __syncthreads();
    uint32_t i = 0;
    while (s_pre[i + 1] <= b0) ++i;  // the stage's first worker (uniform)
    for (; i < n && s_pre[i] < b0 + bn; ++i) {
      const uint32_t a = (s_pre[i] > b0 ? s_pre[i] : b0) - b0;
      const uint32_t z = (s_pre[i + 1] < b0 + bn ? s_pre[i + 1] : b0 + bn) - b0;
      if (a >= z) continue;  // uniform: no pairs of worker i here
      for (uint32_t q = a + threadIdx.x; q < z; q += kThreads) {
        const uint32_t j = st_idx[q];
        const uint64_t r = static_cast<uint64_t>(j) - j0;  // wraps when j < j0
        if (r < kAggTile && j < d)
          acc[r] += st_val[q];
        else
          bad = true;  // unsorted or out-of-range input: skipped, latched
      }
      __syncthreads();
    }
  }
  if (bad) atomicOr(error, kDevErrBadInput);
  if (kVec && j0 + kAggTile <= d) {
    float4* out = reinterpret_cast<float4*>(o.out + j0);
    float4* mom = kMode == kAggMomentum ? reinterpret_cast<float4*>(o.m + j0) : nullptr;
    for (int q = threadIdx.x; q < kAggTile / 4; q += kThreads) {
      const float4 sv = reinterpret_cast<const float4*>(acc)[q];
      if constexpr (kMode == kAggDense) {
        out[q] = sv;
      } else {
        float4 xv = out[q];
        float4 mv = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
        if constexpr (kMode == kAggMomentum) mv = mom[q];
        apply_update<kMode>(o, sv.x, xv.x, mv.x);
        apply_update<kMode>(o, sv.y, xv.y, mv.y);
        apply_update<kMode>(o, sv.z, xv.z, mv.z);
        apply_update<kMode>(o, sv.w, xv.w, mv.w);
        out[q] = xv;
        if constexpr (kMode == kAggMomentum) mom[q] = mv;
      }
    }
  } else {
    for (int q = threadIdx.x; q < kAggTile; q += kThreads) {
      if (j0 + q >= d) continue;
      if constexpr (kMode == kAggDense) {
        o.out[j0 + q] = acc[q];
      } else {
        float xv = o.out[j0 + q], mv = 0.0f;
        if constexpr (kMode == kAggMomentum) mv = o.m[j0 + q];
        apply_update<kMode>(o, acc[q], xv, mv);
        o.out[j0 + q] = xv;
        if constexpr (kMode == kAggMomentum) o.m[j0 + q] = mv;
      }
    }
  }
}

template <int kMode>
cudaError_t launch_reduce(bool vec, AggPtrs p, uint32_t n, uint32_t d, uint32_t tiles,
                          const uint32_t* off, const uint32_t* counts, AggOut o, Workspace& ws) {
  uint32_t* error = ws.u32(kOffError);
  void* params[] = {&p, &n, &d, &tiles, &off, &counts, &o, &error};
  const void* fn = vec ? reinterpret_cast<const void*>(&agg_reduce_kernel<true, kMode>)
                       : reinterpret_cast<const void*>(&agg_reduce_kernel<false, kMode>);
  return launch_pdl(fn, tiles, kThreads, 0, ws.stream, params, false);
}

cudaError_t launch_common(uint32_t n, const uint32_t* const* idx, const float* const* val,
                          const uint32_t* const* tile_index, const uint32_t* counts, uint32_t d,
                          const AggOut& o, int mode, Workspace& ws) {
  AggPtrs p;
  for (uint32_t i = 0; i < kMaxWorkers; ++i) {
    p.idx[i] = i < n ? idx[i] : nullptr;
    p.val[i] = i < n ? val[i] : nullptr;
    p.tiles[i] = i < n && tile_index ? tile_index[i] : nullptr;
  }
  const uint32_t tiles = agg_tiles_for(d);
  cudaError_t err = cudaSuccess;
  uint32_t* off = nullptr;
  if (!tile_index) {  // locate each list's tile boundaries first
    const dim3 grid1((tiles + 1 + kThreads - 1) / kThreads, n);
    off = ws.offsets();
    const uint32_t* counts_arg = counts;
    uint32_t n_arg = n, tiles_arg = tiles;
    uint32_t* error = ws.u32(kOffError);
    void* params[] = {&p, &counts_arg, &n_arg, &tiles_arg, &off, &error};
    err = launch_pdl(reinterpret_cast<const void*>(&agg_offsets_kernel), grid1, kThreads, 0,
                     ws.stream, params, false);
    count_launch();
    if (err != cudaSuccess) return err;
  }
  const bool vec = reinterpret_cast<uintptr_t>(o.out) % 16 == 0 &&
                   reinterpret_cast<uintptr_t>(o.m) % 16 == 0;
  if (mode == kAggDense)
    err = launch_reduce<kAggDense>(vec, p, n, d, tiles, off, counts, o, ws);
  else if (mode == kAggSgd)
    err = launch_reduce<kAggSgd>(vec, p, n, d, tiles, off, counts, o, ws);
  else
    err = launch_reduce<kAggMomentum>(vec, p, n, d, tiles, off, counts, o, ws);
  count_launch();
  return err;
}
}  // namespace

void aggregate_init_device() {
  const void* fns[] = {
      reinterpret_cast<const void*>(&agg_reduce_kernel<true, kAggDense>),
      reinterpret_cast<const void*>(&agg_reduce_kernel<false, kAggDense>),
      reinterpret_cast<const void*>(&agg_reduce_kernel<true, kAggSgd>),
      reinterpret_cast<const void*>(&agg_reduce_kernel<false, kAggSgd>),
      reinterpret_cast<const void*>(&agg_reduce_kernel<true, kAggMomentum>),
      reinterpret_cast<const void*>(&agg_reduce_kernel<false, kAggMomentum>)};
  for (const void* f : fns)
    cudaFuncSetAttribute(f, cudaFuncAttributePreferredSharedMemoryCarveout,
                         cudaSharedmemCarveoutMaxShared);
  cudaGetLastError();
}

cudaError_t launch_aggregate(uint32_t n, const uint32_t* const* idx, const float* const* val,
                             const uint32_t* const* tiles, const uint32_t* counts, uint32_t d,
                             float* dense_out, Workspace& ws) {
  return launch_common(n, idx, val, tiles, counts, d,
                       AggOut{dense_out, nullptr, 1.0f, 0.0f, 0.0f}, kAggDense, ws);
}

cudaError_t launch_aggregate_apply(uint32_t n, const uint32_t* const* idx,
                                   const float* const* val, const uint32_t* const* tiles,
                                   const uint32_t* counts, uint32_t d, float alpha, float* x,
                                   float* m, float mu, float lr, Workspace& ws) {
  return launch_common(n, idx, val, tiles, counts, d, AggOut{x, m, alpha, mu, lr},
                       m ? kAggMomentum : kAggSgd, ws);
}

cudaError_t launch_list_tiles(const uint32_t* idx, const uint32_t* count, uint32_t d,
                              uint32_t* tiles_out, Workspace& ws) {
  AggPtrs p;
  for (uint32_t i = 0; i < kMaxWorkers; ++i) {
    p.idx[i] = i == 0 ? idx : nullptr;
    p.val[i] = nullptr;
    p.tiles[i] = nullptr;
  }
  uint32_t n = 1, tiles = agg_tiles_for(d);
  const dim3 grid((tiles + 1 + kThreads - 1) / kThreads, 1);
  uint32_t* error = ws.u32(kOffError);
  void* params[] = {&p, &count, &n, &tiles, &tiles_out, &error};
  const cudaError_t err = launch_pdl(reinterpret_cast<const void*>(&agg_offsets_kernel), grid,
                                     kThreads, 0, ws.stream, params, false);
  count_launch();
  return err;
}

}  // namespace efs
