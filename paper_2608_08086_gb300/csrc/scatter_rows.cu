// Row scatter for staging a step's new response rows (the Q/K/V rows of the
// positions the decoder changed, in every layer) into the layer tensors: one
// CTA per source row, 16-byte vector copies, up to two destinations per row
// (a query row lives both in the response-query tensor and in the all-query
// tensor of the refresh pass).

#include "archer_internal.h"

namespace archer {
namespace {

constexpr int kThreads = 128;

__global__ void __launch_bounds__(kThreads)
scatter_rows_kernel(int batch, int n, int words, const uint4* __restrict__ src, const int64_t* __restrict__ pos,
                    uint4* __restrict__ dst0, int rows0, int row00, uint4* __restrict__ dst1, int rows1, int row01) {
  const long long row = blockIdx.x;                    // (outer, b, r) in that order
  const int r = static_cast<int>(row % n);
  const long long ob = row / n;                        // outer * batch + b
  const int b = static_cast<int>(ob % batch);
  const int64_t p = pos[static_cast<long long>(b) * n + r];
  const uint4* s = src + row * words;
  const bool ok0 = p >= 0 && p + row00 < rows0;
  const bool ok1 = dst1 && p >= 0 && p + row01 < rows1;
  uint4* d0 = dst0 + (ob * rows0 + row00 + p) * words;
  uint4* d1 = dst1 ? dst1 + (ob * rows1 + row01 + p) * words : nullptr;
  for (int w = threadIdx.x; w < words; w += kThreads) {
    const uint4 v = s[w];
    if (ok0) d0[w] = v;
    if (ok1) d1[w] = v;
  }
}

}  // namespace

int scatter_rows_launch(int n_outer, int batch, int n, size_t row_bytes, const void* src, const int64_t* pos,
                        void* dst0, int rows0, int row00, void* dst1, int rows1, int row01, cudaStream_t stream) {
  const long long blocks = static_cast<long long>(n_outer) * batch * n;
  if (blocks == 0 || row_bytes == 0) return ARCHER_OK;
  scatter_rows_kernel<<<static_cast<unsigned>(blocks), kThreads, 0, stream>>>(
      batch, n, static_cast<int>(row_bytes / 16), static_cast<const uint4*>(src), pos, static_cast<uint4*>(dst0),
      rows0, row00, static_cast<uint4*>(dst1), rows1, row01);
  return cuda_status(cudaGetLastError(), "scatter_rows launch");
}

}  // namespace archer
