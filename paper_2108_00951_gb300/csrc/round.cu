// round.cu — error feedback with scaled integer rounding, an absolute
// compressor (Sec. 5: a rounding with error bounded by eps has
// kappa^2 = d eps^2; the scaled integer rounding of in-network aggregation is
// one), and the exchange of its integer messages.
//
// Compression, per coordinate (Algorithm 1 with C = scaled rounding):
//   a_j = fmaf(gamma, g_j, e_j); s_j = a_j 2^m (exact: a power-of-two scale);
//   q_j = round-half-to-even(s_j) as int32; C(a)_j = q_j 2^-m; e'_j = a_j - C(a)_j.
// Both q_j 2^-m and a_j - C(a)_j are exact in fp32 (q_j is an fp32 integer
// and C(a)_j lies on a's grid or coarser), so a = C(a) + e' holds bit for bit
// and |e'_j| <= 2^(-m-1). A coordinate with |s_j| >= 2^31 (or NaN) does not
// fit an int32 message: q_j = 0, e'_j = a_j, and it is counted.
// One streaming pass: 16 bytes per coordinate (read g and e, write e' and q;
// 14 for a bf16 g), 4 coordinates per thread per iteration, 16-byte accesses
// when the arrays allow.
//
// Exchange: S_j = sum_i q_i[j] in int64 (exact: the order does not matter)
// and dense_j = RN(S_j) 2^-m, one rounding. 4 n + 4 bytes per coordinate.
#include "gradient.cuh"
#include "internal.h"

namespace efs {
namespace {

constexpr int kRoundThreads = 256;

__device__ __forceinline__ float pow2f(int m) {  // 2^m for -126 <= m <= 127
  return __int_as_float((127 + m) << 23);
}

// One coordinate: q, e', and whether it was sent.
__device__ __forceinline__ bool round_one(float a, float scale, float unscale, int32_t& q,
                                          float& e_new) {
  const float s = __fmul_rn(a, scale);
  if (!(fabsf(s) < 2147483648.0f)) {  // does not fit an int32 (or NaN): kept in e
    q = 0;
    e_new = a;
    return false;
  }
  q = __float2int_rn(s);
  e_new = __fsub_rn(a, __fmul_rn(static_cast<float>(q), unscale));
  return true;
}

// Each CTA publishes its count of coordinates not sent (and its share of
// ||e'||^2) and counts itself in; the last CTA to arrive writes the totals
// (shares added in a fixed order) and resets the counter. No CTA waits.
template <typename GT, bool kVec>
__global__ void __launch_bounds__(kRoundThreads)
    scaled_round_kernel(const GT* __restrict__ g, float* __restrict__ e, float gamma, int m,
                        uint32_t d, int32_t* __restrict__ q, uint32_t* __restrict__ unsent,
                        uint32_t* cnt_parts, FF* err_parts, uint32_t* arrive, double* err_out) {
  __shared__ FF s_ff[32];
  __shared__ uint32_t s_cnt[kRoundThreads / 32];
  __shared__ uint32_t s_last;
  const float scale = pow2f(m), unscale = pow2f(-m);
  const int lane = threadIdx.x & 31;
  const uint64_t groups = (static_cast<uint64_t>(d) + 3) / 4;
  const uint64_t stride = static_cast<uint64_t>(gridDim.x) * kRoundThreads;
  ErrAcc acc;
  uint32_t not_sent = 0;
  griddep_wait();  // g and e may come from the kernels before (programmatic launch)
  for (uint64_t gi = static_cast<uint64_t>(blockIdx.x) * kRoundThreads + threadIdx.x;
       gi < groups; gi += stride) {
    const uint64_t j0 = gi * 4;
    float a[4], en[4];
    int32_t qq[4];
    if (kVec && j0 + 4 <= d) {
      GradVec<GT> gv;
      gv.load(g + j0);
      const float4 ev = ld_stream_f4(e + j0);
      a[0] = __fmaf_rn(gamma, gv[0], ev.x);
      a[1] = __fmaf_rn(gamma, gv[1], ev.y);
      a[2] = __fmaf_rn(gamma, gv[2], ev.z);
      a[3] = __fmaf_rn(gamma, gv[3], ev.w);
#pragma unroll
      for (int j = 0; j < 4; ++j) not_sent += round_one(a[j], scale, unscale, qq[j], en[j]) ? 0u : 1u;
      st_stream_f4(e + j0, make_float4(en[0], en[1], en[2], en[3]));
      *reinterpret_cast<int4*>(q + j0) = make_int4(qq[0], qq[1], qq[2], qq[3]);
      if (err_out)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc.add(en[j]);
    } else {
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const uint64_t i = j0 + j;
        if (i < d) {
          const float x = __fmaf_rn(gamma, grad_scalar(g, i), e[i]);
          int32_t qi;
          float ei;
          not_sent += round_one(x, scale, unscale, qi, ei) ? 0u : 1u;
          e[i] = ei;
          q[i] = qi;
          if (err_out) acc.add(ei);
        }
      }
    }
  }
  griddep_launch_dependents();  // the next kernel may be scheduled (it waits for this grid)
  const uint32_t warp_total = warp_sum(not_sent);
  if (lane == 0) s_cnt[threadIdx.x >> 5] = warp_total;
  FF share{0.0f, 0.0f};
  if (err_out) {
    acc.flush();
    share = block_sum_ff(acc.total, s_ff);  // synchronises the CTA
  } else {
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    uint32_t c = 0;
    for (int w = 0; w < kRoundThreads / 32; ++w) c += s_cnt[w];
    cnt_parts[blockIdx.x] = c;
    if (err_out) err_parts[blockIdx.x] = share;
    __threadfence();
    s_last = atomicAdd(arrive, 1u) == gridDim.x - 1 ? 1u : 0u;
  }
  __syncthreads();
  if (s_last) {
    __threadfence();
    uint32_t c = 0;
    for (uint32_t b = threadIdx.x; b < gridDim.x; b += kRoundThreads) c += __ldcg(cnt_parts + b);
    c = warp_sum(c);
    __syncthreads();  // s_cnt is reused
    if (lane == 0) s_cnt[threadIdx.x >> 5] = c;
    FF t{0.0f, 0.0f};
    if (err_out) t = sum_parts_ff(err_parts, gridDim.x, s_ff);  // synchronises the CTA
    else __syncthreads();
    if (threadIdx.x == 0) {
      uint32_t total = 0;
      for (int w = 0; w < kRoundThreads / 32; ++w) total += s_cnt[w];
      *unsent = total;
      if (err_out) *err_out = ff_to_double(t);
      *arrive = 0;  // ready for the next call
    }
  }
}

struct IntPtrs {
  const int32_t* q[kMaxWorkers];
};

template <bool kVec>
__global__ void __launch_bounds__(kRoundThreads)
    int_aggregate_kernel(IntPtrs p, uint32_t n, uint32_t d, int m, float* __restrict__ dense) {
  const float unscale = pow2f(-m);
  const uint64_t groups = (static_cast<uint64_t>(d) + 3) / 4;
  const uint64_t stride = static_cast<uint64_t>(gridDim.x) * kRoundThreads;
  griddep_wait();  // the messages come from the kernels before (programmatic launch)
  griddep_launch_dependents();
  for (uint64_t gi = static_cast<uint64_t>(blockIdx.x) * kRoundThreads + threadIdx.x;
       gi < groups; gi += stride) {
    const uint64_t j0 = gi * 4;
    long long s[4] = {0, 0, 0, 0};
    if (kVec && j0 + 4 <= d) {
      for (uint32_t i = 0; i < n; ++i) {
        const int4 v = __ldcs(reinterpret_cast<const int4*>(p.q[i] + j0));
        s[0] += v.x;
        s[1] += v.y;
        s[2] += v.z;
        s[3] += v.w;
      }
      *reinterpret_cast<float4*>(dense + j0) =
          make_float4(__fmul_rn(__ll2float_rn(s[0]), unscale), __fmul_rn(__ll2float_rn(s[1]), unscale),
                      __fmul_rn(__ll2float_rn(s[2]), unscale), __fmul_rn(__ll2float_rn(s[3]), unscale));
    } else {
      for (uint32_t i = 0; i < n; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j)
          if (j0 + j < d) s[j] += p.q[i][j0 + j];
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (j0 + j < d) dense[j0 + j] = __fmul_rn(__ll2float_rn(s[j]), unscale);
    }
  }
}

uint32_t grid_for(uint32_t d, const DeviceInfo& dev) {
  const uint64_t groups = (static_cast<uint64_t>(d) + 3) / 4;
  uint64_t grid = (groups + kRoundThreads - 1) / kRoundThreads;
  // 4 CTAs of 256 threads per SM, the same number on every SM (a grid that
  // leaves some SMs one CTA more than others was measured 5 % slower)
  const uint64_t cap = static_cast<uint64_t>(dev.sm_count) * 4;
  if (grid > cap) grid = cap;
  if (grid > kMaxChunks) grid = kMaxChunks;
  return static_cast<uint32_t>(grid > 0 ? grid : 1);
}

template <typename GT>
cudaError_t launch_round_typed(const GT* g, float* e, float gamma, int m, uint32_t d, int32_t* q,
                               uint32_t* unsent, double* err_out, Workspace& ws,
                               const DeviceInfo& dev) {
  const bool vec = reinterpret_cast<uintptr_t>(g) % (4 * sizeof(GT)) == 0 &&
                   reinterpret_cast<uintptr_t>(e) % 16 == 0 &&
                   reinterpret_cast<uintptr_t>(q) % 16 == 0;
  const uint32_t grid = grid_for(d, dev);
  uint32_t* cnt_parts = ws.cntparts();
  FF* err_parts = ws.errparts();
  uint32_t* arrive = ws.u32(kOffErrArrive);
  void* params[] = {&g, &e, &gamma, &m, &d, &q, &unsent, &cnt_parts, &err_parts, &arrive, &err_out};
  const void* fn = vec ? reinterpret_cast<const void*>(&scaled_round_kernel<GT, true>)
                       : reinterpret_cast<const void*>(&scaled_round_kernel<GT, false>);
  const cudaError_t err = launch_pdl(fn, grid, kRoundThreads, 0, ws.stream, params, false);
  count_launch();
  return err;
}

}  // namespace

cudaError_t launch_scaled_round(const void* g, bool g_bf16, float* e, float gamma, int m,
                                uint32_t d, int32_t* q, uint32_t* unsent, double* err_out,
                                Workspace& ws, const DeviceInfo& dev) {
  if (g_bf16)
    return launch_round_typed(static_cast<const uint16_t*>(g), e, gamma, m, d, q, unsent,
                              err_out, ws, dev);
  return launch_round_typed(static_cast<const float*>(g), e, gamma, m, d, q, unsent, err_out, ws,
                            dev);
}

cudaError_t launch_int_aggregate(uint32_t n, const int32_t* const* q, uint32_t d, int m,
                                 float* dense_out, Workspace& ws, const DeviceInfo& dev) {
  IntPtrs p;
  bool vec = reinterpret_cast<uintptr_t>(dense_out) % 16 == 0;
  for (uint32_t i = 0; i < kMaxWorkers; ++i) {
    p.q[i] = i < n ? q[i] : nullptr;
    if (i < n && reinterpret_cast<uintptr_t>(q[i]) % 16 != 0) vec = false;
  }
  const uint32_t grid = grid_for(d, dev);
  void* params[] = {&p, &n, &d, &m, &dense_out};
  const void* fn = vec ? reinterpret_cast<const void*>(&int_aggregate_kernel<true>)
                       : reinterpret_cast<const void*>(&int_aggregate_kernel<false>);
  const cudaError_t err = launch_pdl(fn, grid, kRoundThreads, 0, ws.stream, params, false);
  count_launch();
  return err;
}

}  // namespace efs
