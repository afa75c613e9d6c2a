// errnorm.cu — the squared error norm ||e'||^2 of a finished step by one
// plain pass over e' (the total error's per-step term, Sec. 1 and the remark
// after the EF convergence theorem). The streaming kernels compute it on the
// fly; this pass serves the paths that do not stream (inputs the bulk copies
// cannot take).
//
// CTA c sums the contiguous range [c d / G, (c+1) d / G): per thread, the
// accumulator of common.cuh over coalesced positions; per CTA, a fixed-order
// sum of the threads. Each CTA stores its share, fences, and counts itself
// in; the last to arrive adds the G shares in a fixed order, writes the
// result and resets the counter. No CTA waits for another.
#include "internal.h"

namespace efs {
namespace {

constexpr int kErrThreads = 256;

__global__ void __launch_bounds__(kErrThreads)
    error_norm_kernel(const float* __restrict__ e, uint32_t d, FF* parts, uint32_t* arrive,
                      double* err_out) {
  __shared__ FF s_d[32];
  __shared__ uint32_t s_last;
  const uint32_t G = gridDim.x, c = blockIdx.x;
  const uint32_t lo = static_cast<uint32_t>(static_cast<uint64_t>(c) * d / G);
  const uint32_t hi = static_cast<uint32_t>(static_cast<uint64_t>(c + 1) * d / G);
  ErrAcc acc;
  for (uint32_t i0 = lo + threadIdx.x; i0 < hi; i0 += 4 * kErrThreads) {
    float v[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const uint32_t i = i0 + j * kErrThreads;
      v[j] = i < hi ? __ldcg(e + i) : 0.0f;
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) acc.add(v[j]);
  }
  acc.flush();
  const FF mine = block_sum_ff(acc.total, s_d);
  if (threadIdx.x == 0) {
    parts[c] = mine;
    __threadfence();
    s_last = atomicAdd(arrive, 1u) == G - 1 ? 1u : 0u;
  }
  __syncthreads();
  if (s_last) {
    __threadfence();
    const FF t = sum_parts_ff(parts, G, s_d);
    if (threadIdx.x == 0) {
      *err_out = ff_to_double(t);
      *arrive = 0;  // ready for the next pass
    }
  }
}

}  // namespace

cudaError_t launch_error_norm(const float* e, uint32_t d, double* err_out, Workspace& ws,
                              const DeviceInfo& dev) {
  uint32_t grid = static_cast<uint32_t>(dev.sm_count) * 4;
  if (grid > kMaxChunks) grid = kMaxChunks;
  const uint32_t need = (d + 4 * kErrThreads - 1) / (4 * kErrThreads);
  if (grid > need) grid = need > 0 ? need : 1;
  error_norm_kernel<<<grid, kErrThreads, 0, ws.stream>>>(e, d, ws.errparts(),
                                                         ws.u32(kOffErrArrive), err_out);
  count_launch();
  return cudaGetLastError();
}

}  // namespace efs
