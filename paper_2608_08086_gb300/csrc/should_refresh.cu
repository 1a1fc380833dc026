// Refresh rule for sm_103a (Sec. 4.2, Eq. archer-distance and
// Eq. archer-controller, with the cache-age cap of Sec. 6):
//   D_t = #{i : g_t[i] != g_r[i]},  refresh iff D_t >= K or age_t >= max_age,
// and on refresh g_r <- g_t, age <- 0.  One CTA per sequence; integer only.

#include "archer_device.cuh"
#include "archer_internal.h"

namespace archer {
namespace {

constexpr int kThreads = 256;

__global__ void __launch_bounds__(kThreads)
should_refresh_kernel(int G, const int32_t* __restrict__ g_cur, int32_t* __restrict__ g_anchor,
                      int32_t* __restrict__ age, int K, int max_age, int update_anchor,
                      int32_t* __restrict__ dist_out, uint8_t* __restrict__ flag_out) {
  __shared__ int warp_sum[kThreads / 32];
  __shared__ int s_flag;
  const int b = blockIdx.x;
  const int32_t* gc = g_cur + static_cast<size_t>(b) * G;
  int32_t* ga = g_anchor + static_cast<size_t>(b) * G;
  int d = 0;
  for (int i = threadIdx.x; i < G; i += kThreads) d += (gc[i] != ga[i]) ? 1 : 0;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) d += __shfl_xor_sync(0xffffffffu, d, o);
  if ((threadIdx.x & 31) == 0) warp_sum[threadIdx.x >> 5] = d;
  __syncthreads();   // also orders every read of g_anchor before the rewrite below
  if (threadIdx.x == 0) {
    int dist = 0;
    for (int w = 0; w < kThreads / 32; ++w) dist += warp_sum[w];
    const long long age_t = static_cast<long long>(age[b]) + 1;
    const bool f = (dist >= K) || (max_age > 0 && age_t >= max_age);
    if (dist_out) dist_out[b] = dist;
    flag_out[b] = f ? 1 : 0;
    if (update_anchor) age[b] = f ? 0 : static_cast<int32_t>(age_t);
    s_flag = f ? 1 : 0;
  }
  __syncthreads();
  if (update_anchor && s_flag)
    for (int i = threadIdx.x; i < G; i += kThreads) ga[i] = gc[i];
}

}  // namespace

int should_refresh_launch(int B, int G, const int32_t* g_cur, int32_t* g_anchor, int32_t* age, int K,
                          int max_age, int update_anchor, int32_t* dist, uint8_t* flag, cudaStream_t stream) {
  if (B == 0) return ARCHER_OK;
  should_refresh_kernel<<<B, kThreads, 0, stream>>>(G, g_cur, g_anchor, age, K, max_age, update_anchor, dist, flag);
  return cuda_status(cudaGetLastError(), "should_refresh launch");
}

}  // namespace archer
