// Synthetic stand-in for the rollback decoder D of Algorithm 1 (Sec. 4.2).
// The paper takes D as given (its confidence rule reads the scores of the
// decoder-control step, Sec. 6); this confidence-threshold rule lets the
// refresh decisions depend on the scoring kernel's outputs in tests and
// trajectories.  Per sequence, from the scores of the previous step:
//   * a masked position with max_prob >= tau_accept takes its top-1 token;
//   * an unmasked position whose token has cur_prob < tau_remask is masked
//     again (rolled back);
//   * if masked positions remain and none was accepted, the masked position
//     with the largest max_prob (lowest index on ties) takes its top-1.
// One CTA per sequence; decisions in fp32.

#include "archer_internal.h"

namespace archer {
namespace {

constexpr int kThreads = 256;

__global__ void __launch_bounds__(kThreads)
decoder_update_kernel(int G, float tau_accept, float tau_remask, int32_t mask_token,
                      const float* __restrict__ max_prob, const int32_t* __restrict__ top1,
                      const float* __restrict__ cur_prob, int32_t* __restrict__ g, uint8_t* __restrict__ changed) {
  __shared__ unsigned long long warp_best[kThreads / 32];
  const int b = blockIdx.x;
  const size_t base = static_cast<size_t>(b) * G;
  int accepted = 0;
  // best masked position: key = (max_prob bits, ~index): the largest key has
  // the largest probability (non-negative floats order like their bits) and,
  // among equals, the lowest index
  unsigned long long best = 0;
  for (int i = threadIdx.x; i < G; i += kThreads) {
    const int32_t cur = g[base + i];
    int32_t nxt = cur;
    if (cur == mask_token) {
      const float mp = max_prob[base + i];
      const unsigned long long key =
          (static_cast<unsigned long long>(__float_as_uint(mp)) << 32) | (0xFFFFFFFFu - static_cast<uint32_t>(i));
      best = key > best ? key : best;
      if (mp >= tau_accept) {
        nxt = top1[base + i];
        accepted = 1;
      }
    } else if (cur_prob[base + i] < tau_remask) {
      nxt = mask_token;
    }
    g[base + i] = nxt;
    changed[base + i] = nxt != cur ? 1 : 0;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const unsigned long long other = __shfl_xor_sync(0xffffffffu, best, o);
    best = other > best ? other : best;
  }
  if ((threadIdx.x & 31) == 0) warp_best[threadIdx.x >> 5] = best;
  accepted = __syncthreads_or(accepted);          // also publishes warp_best
  if (threadIdx.x == 0 && !accepted) {
    unsigned long long m = 0;
    for (int w = 0; w < kThreads / 32; ++w) m = warp_best[w] > m ? warp_best[w] : m;
    if (m != 0) {                                  // some position was masked
      const int i = static_cast<int>(0xFFFFFFFFu - static_cast<uint32_t>(m & 0xFFFFFFFFull));
      g[base + i] = top1[base + i];
      changed[base + i] = top1[base + i] != mask_token ? 1 : 0;
    }
  }
}

}  // namespace

int decoder_update_launch(int B, int G, float tau_accept, float tau_remask, int32_t mask_token,
                          const float* max_prob, const int32_t* top1, const float* cur_prob, int32_t* g,
                          uint8_t* changed, cudaStream_t stream) {
  if (B == 0 || G == 0) return ARCHER_OK;
  decoder_update_kernel<<<B, kThreads, 0, stream>>>(G, tau_accept, tau_remask, mask_token, max_prob, top1,
                                                    cur_prob, g, changed);
  return cuda_status(cudaGetLastError(), "decoder_update launch");
}

}  // namespace archer
