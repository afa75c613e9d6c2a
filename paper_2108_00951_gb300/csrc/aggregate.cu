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
};

// off[i * (tiles + 1) + t] = number of entries of list i below t * kAggTile;
// off[i * (tiles + 1) + tiles] = counts[i].
__global__ void __launch_bounds__(kThreads)
    agg_offsets_kernel(AggPtrs p, const uint32_t* __restrict__ counts, uint32_t n,
                       uint32_t tiles, uint32_t* __restrict__ off) {
  const uint64_t per = static_cast<uint64_t>(tiles) + 1;
  const uint64_t gid = static_cast<uint64_t>(blockIdx.x) * kThreads + threadIdx.x;
  if (gid >= per * n) return;
  const uint32_t i = static_cast<uint32_t>(gid / per);
  const uint32_t t = static_cast<uint32_t>(gid % per);
  const uint32_t cnt = counts[i];
  uint32_t result = cnt;
  if (t < tiles) {
    const uint64_t target = static_cast<uint64_t>(t) * kAggTile;
    const uint32_t* x = p.idx[i];
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
  off[gid] = result;
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

template <bool kVec, int kMode>
__global__ void __launch_bounds__(kThreads)
    agg_reduce_kernel(AggPtrs p, uint32_t n, uint32_t d, uint32_t tiles,
                      const uint32_t* __restrict__ off, AggOut o,
                      uint32_t* __restrict__ error) {
  __shared__ __align__(16) float acc[kAggTile];
  __shared__ uint32_t s_lo[kMaxWorkers], s_hi[kMaxWorkers];
  const uint32_t t = blockIdx.x;
  const uint64_t j0 = static_cast<uint64_t>(t) * kAggTile;
  for (int q = threadIdx.x; q < kAggTile / 4; q += kThreads)
    reinterpret_cast<float4*>(acc)[q] = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
  for (uint32_t i = threadIdx.x; i < n; i += kThreads) {
    s_lo[i] = off[static_cast<uint64_t>(i) * (tiles + 1) + t];
    s_hi[i] = off[static_cast<uint64_t>(i) * (tiles + 1) + t + 1];
  }
  __syncthreads();
  bool bad = false;
  for (uint32_t i = 0; i < n; ++i) {
    const uint32_t lo = s_lo[i], hi = s_hi[i];
    if (lo >= hi) continue;  // uniform across the CTA
    const uint32_t* __restrict__ xi = p.idx[i];
    const float* __restrict__ vi = p.val[i];
    for (uint32_t q = lo + threadIdx.x; q < hi; q += kThreads) {
      const uint32_t j = __ldg(xi + q);
      const uint64_t r = static_cast<uint64_t>(j) - j0;  // wraps when j < j0
      if (r < kAggTile && j < d)
        acc[r] += __ldg(vi + q);
      else
        bad = true;  // unsorted or out-of-range input: skipped, latched
    }
    __syncthreads();
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
void launch_reduce(bool vec, const AggPtrs& p, uint32_t n, uint32_t d, uint32_t tiles,
                   const uint32_t* off, const AggOut& o, Workspace& ws) {
  if (vec)
    agg_reduce_kernel<true, kMode><<<tiles, kThreads, 0, ws.stream>>>(p, n, d, tiles, off, o,
                                                                      ws.u32(kOffError));
  else
    agg_reduce_kernel<false, kMode><<<tiles, kThreads, 0, ws.stream>>>(p, n, d, tiles, off, o,
                                                                       ws.u32(kOffError));
}

cudaError_t launch_common(uint32_t n, const uint32_t* const* idx, const float* const* val,
                          const uint32_t* counts, uint32_t d, const AggOut& o, int mode,
                          Workspace& ws) {
  AggPtrs p;
  for (uint32_t i = 0; i < kMaxWorkers; ++i) {
    p.idx[i] = i < n ? idx[i] : nullptr;
    p.val[i] = i < n ? val[i] : nullptr;
  }
  const uint32_t tiles = agg_tiles_for(d);
  const uint64_t entries = static_cast<uint64_t>(n) * (tiles + 1);
  const uint32_t grid1 = static_cast<uint32_t>((entries + kThreads - 1) / kThreads);
  uint32_t* off = ws.offsets();
  agg_offsets_kernel<<<grid1, kThreads, 0, ws.stream>>>(p, counts, n, tiles, off);
  count_launch();
  cudaError_t err = cudaGetLastError();
  if (err != cudaSuccess) return err;
  const bool vec = reinterpret_cast<uintptr_t>(o.out) % 16 == 0 &&
                   reinterpret_cast<uintptr_t>(o.m) % 16 == 0;
  if (mode == kAggDense)
    launch_reduce<kAggDense>(vec, p, n, d, tiles, off, o, ws);
  else if (mode == kAggSgd)
    launch_reduce<kAggSgd>(vec, p, n, d, tiles, off, o, ws);
  else
    launch_reduce<kAggMomentum>(vec, p, n, d, tiles, off, o, ws);
  count_launch();
  return cudaGetLastError();
}
}  // namespace

cudaError_t launch_aggregate(uint32_t n, const uint32_t* const* idx, const float* const* val,
                             const uint32_t* counts, uint32_t d, float* dense_out,
                             Workspace& ws) {
  return launch_common(n, idx, val, counts, d, AggOut{dense_out, nullptr, 1.0f, 0.0f, 0.0f},
                       kAggDense, ws);
}

cudaError_t launch_aggregate_apply(uint32_t n, const uint32_t* const* idx,
                                   const float* const* val, const uint32_t* counts, uint32_t d,
                                   float alpha, float* x, float* m, float mu, float lr,
                                   Workspace& ws) {
  return launch_common(n, idx, val, counts, d, AggOut{x, m, alpha, mu, lr},
                       m ? kAggMomentum : kAggSgd, ws);
}

}  // namespace efs
