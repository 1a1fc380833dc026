// Decoder scoring for sm_103a: per row of vocabulary logits, the fp32
// softmax's max probability, the top-1 id (lowest index on ties), the
// top-1/top-2 probability margin and optionally p(current token).  These are
// the inputs of the rollback decoder's confidence rule (Sec. 6; the decision
// margin of Eq. theory-margin is taken on them).
//
// HBM-streaming reduction, one pass over the logits:
//   * a row is cut into chunks of kThreads * kUnroll 16-byte words; one CTA
//     per (row, chunk) issues all its loads up front (coalesced, 16 B/thread);
//   * pass A over the registers: max and second value per thread (for bf16
//     with packed bf16x2 max/min, 1.5 ops per element), CTA-reduced;
//   * pass B: sum of 2^((z - m) log2 e) with the CTA max m -- exactly one ex2
//     per element; the lowest index of m is found by the threads holding it;
//   * chunk partials (m, sum, top-2 value, index) go to the workspace and the
//     CTA exits at once -- no CTA waits on another, so HBM reads stay in
//     flight; a combine kernel (one warp per row) then merges each row's
//     partials and writes the outputs.  A row of one chunk skips both.

#include <cfloat>
#include <cmath>
#include <mutex>

#include <cuda.h>

#include "archer_device.cuh"
#include "archer_internal.h"

namespace archer {
namespace {

constexpr int kThreads = 256;
constexpr int kUnroll = 8;                       // 16-byte words per thread per chunk
constexpr int kWordsPerChunk = kThreads * kUnroll;
constexpr float kLog2e = 1.4426950408889634f;

struct Partial {
  float m;      // chunk max
  float s;      // sum of 2^((z - m) log2 e) over the chunk
  float t2;     // chunk second value (multiset: equals m on a tie)
  int idx;      // lowest index attaining m
};

// Merge of (top1, top2) value pairs with multiset semantics.
__device__ __forceinline__ void merge_top2(float& a1, float& a2, float b1, float b2) {
  const float hi = fmaxf(a1, b1);
  const float lo = fminf(a1, b1);
  a2 = fmaxf(lo, fmaxf(a2, b2));
  a1 = hi;
}

template <typename T>
struct Vec;
template <>
struct Vec<__nv_bfloat16> {
  static constexpr int kElems = 8;
};
template <>
struct Vec<float> {
  static constexpr int kElems = 4;
};

__device__ __forceinline__ void unpack(const uint4& w, float (&v)[8], __nv_bfloat16*) {
  const uint32_t u[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    v[2 * i] = __uint_as_float(u[i] << 16);
    v[2 * i + 1] = __uint_as_float(u[i] & 0xFFFF0000u);
  }
}
__device__ __forceinline__ void unpack(const uint4& w, float (&v)[4], float*) {
  v[0] = __uint_as_float(w.x);
  v[1] = __uint_as_float(w.y);
  v[2] = __uint_as_float(w.z);
  v[3] = __uint_as_float(w.w);
}

// Block-wide reduction of (top1, top2) and, second, of (sum, min index).
struct Smem {
  float a[kThreads / 32];
  float b[kThreads / 32];
  int i[kThreads / 32];
  float m_block, t2_block;
  int last;
};

__device__ __forceinline__ void block_top2(float& t1, float& t2, Smem& sm) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float b1 = __shfl_xor_sync(0xffffffffu, t1, o);
    const float b2 = __shfl_xor_sync(0xffffffffu, t2, o);
    merge_top2(t1, t2, b1, b2);
  }
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  if (l == 0) { sm.a[w] = t1; sm.b[w] = t2; }
  __syncthreads();
  if (threadIdx.x == 0) {
    float x1 = sm.a[0], x2 = sm.b[0];
    for (int k = 1; k < kThreads / 32; ++k) merge_top2(x1, x2, sm.a[k], sm.b[k]);
    sm.m_block = x1;
    sm.t2_block = x2;
  }
  __syncthreads();
  t1 = sm.m_block;
  t2 = sm.t2_block;
}

__device__ __forceinline__ void block_sum_minidx(float& s, int& idx, Smem& sm) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    s += __shfl_xor_sync(0xffffffffu, s, o);
    idx = min(idx, __shfl_xor_sync(0xffffffffu, idx, o));
  }
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  __syncthreads();   // sm.a reused
  if (l == 0) { sm.a[w] = s; sm.i[w] = idx; }
  __syncthreads();
  if (threadIdx.x == 0) {
    float ss = 0.f;
    int ii = INT_MAX;
    for (int k = 0; k < kThreads / 32; ++k) { ss += sm.a[k]; ii = min(ii, sm.i[k]); }
    s = ss;
    idx = ii;
  }
}

__device__ __forceinline__ float load_logit(const void* row, int dtype, int j) {
  return dtype == ARCHER_DTYPE_BF16
             ? __bfloat162float(static_cast<const __nv_bfloat16*>(row)[j])
             : static_cast<const float*>(row)[j];
}

// Writes the outputs of one row from its merged (M, S, top2, idx).
__device__ __forceinline__ void write_row(int row, float M, float S, float t2, int idx, const void* zrow,
                                          int dtype, int vocab, const uint8_t* mask_state,
                                          const int32_t* cur_tokens, float* max_prob, int32_t* top1,
                                          float* margin, float* cur_prob) {
  const float inv = 1.0f / S;
  max_prob[row] = inv;
  top1[row] = idx;
  margin[row] = vocab > 1 ? (1.0f - ex2_approx((t2 - M) * kLog2e)) * inv : inv;
  if (cur_prob) {
    float c = 0.f;
    const bool masked = mask_state && mask_state[row] != 0;
    if (cur_tokens && !masked) {
      const int t = cur_tokens[row];
      if (t >= 0 && t < vocab) c = ex2_approx((load_logit(zrow, dtype, t) - M) * kLog2e) * inv;
    }
    cur_prob[row] = c;
  }
}

template <typename T>
__global__ void __launch_bounds__(kThreads)
decode_scores_kernel(const T* __restrict__ logits, int64_t row_stride, int vocab, int chunks,
                     const uint8_t* __restrict__ mask_state, const int32_t* __restrict__ cur_tokens,
                     float* __restrict__ max_prob, int32_t* __restrict__ top1, float* __restrict__ margin,
                     float* __restrict__ cur_prob, Partial* __restrict__ parts, int aligned) {
  constexpr int E = Vec<T>::kElems;              // elements per 16-byte word
  constexpr int dtype = sizeof(T) == 2 ? ARCHER_DTYPE_BF16 : ARCHER_DTYPE_F32;
  asm volatile("griddepcontrol.launch_dependents;");   // the merge may be scheduled (it waits for this grid)
  __shared__ Smem sm;
  const int row = blockIdx.x / chunks;
  const int chunk = blockIdx.x - row * chunks;
  const T* zrow = logits + row * row_stride;
  const int64_t chunk_elem0 = static_cast<int64_t>(chunk) * kWordsPerChunk * E;

  // ---- issue all loads (word u of this thread covers elements e0 .. e0+E-1)
  uint4 w[kUnroll];
  const uint4* zw = reinterpret_cast<const uint4*>(zrow);
#pragma unroll
  for (int u = 0; u < kUnroll; ++u) {
    const int64_t e0 = chunk_elem0 + (static_cast<int64_t>(u) * kThreads + threadIdx.x) * E;
    if (aligned && e0 + E <= vocab) {
      w[u] = __ldcs(zw + e0 / E);                 // streamed once: evict-first
    } else {
      // ragged tail or rows not 16-byte aligned: element-wise, -inf past the vocabulary
      float v[E];
#pragma unroll
      for (int e = 0; e < E; ++e) v[e] = (e0 + e < vocab) ? load_logit(zrow, dtype, (int)(e0 + e)) : -INFINITY;
      if constexpr (E == 8) {   // exact: every value is a bf16 value or -inf
        w[u] = make_uint4(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]), pack_bf16x2(v[4], v[5]),
                          pack_bf16x2(v[6], v[7]));
      } else {
        w[u] = make_uint4(__float_as_uint(v[0]), __float_as_uint(v[1]), __float_as_uint(v[2]),
                          __float_as_uint(v[3]));
      }
    }
  }

  // ---- pass A: per-thread top-2 values, then CTA-wide
  float t1 = -INFINITY, t2 = -INFINITY;
  if constexpr (E == 8) {
    __nv_bfloat162 M1 = __floats2bfloat162_rn(-INFINITY, -INFINITY);
    __nv_bfloat162 M2 = M1;
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const uint32_t q[4] = {w[u].x, w[u].y, w[u].z, w[u].w};
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const __nv_bfloat162 x = *reinterpret_cast<const __nv_bfloat162*>(&q[i]);
        M2 = __hmax2(M2, __hmin2(M1, x));
        M1 = __hmax2(M1, x);
      }
    }
    const float a = __low2float(M1), c = __high2float(M1);
    t1 = fmaxf(a, c);
    t2 = fmaxf(fminf(a, c), fmaxf(__low2float(M2), __high2float(M2)));
  } else {
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      float v[4];
      unpack(w[u], v, (float*)nullptr);
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        t2 = fmaxf(t2, fminf(t1, v[e]));
        t1 = fmaxf(t1, v[e]);
      }
    }
  }
  const float my_t1 = t1;
  float m_blk = t1, t2_blk = t2;
  block_top2(m_blk, t2_blk, sm);

  // ---- pass B: sum of exps relative to the CTA max; lowest index of the max
  // A chunk whose logits are all -inf contributes a zero sum (not NaN).
  const float neg_m = (m_blk == -INFINITY) ? 0.f : -m_blk * kLog2e;
  float s = 0.f;
#pragma unroll
  for (int u = 0; u < kUnroll; ++u) {
    float v[E];
    unpack(w[u], v, (T*)nullptr);
#pragma unroll
    for (int e = 0; e < E; ++e) s += ex2_approx(fmaf(v[e], kLog2e, neg_m));
  }
  int idx = INT_MAX;
  if (my_t1 == m_blk) {
    for (int u = 0; u < kUnroll && idx == INT_MAX; ++u) {
      float v[E];
      unpack(w[u], v, (T*)nullptr);
      const int64_t e0 = chunk_elem0 + (static_cast<int64_t>(u) * kThreads + threadIdx.x) * E;
#pragma unroll
      for (int e = E - 1; e >= 0; --e)
        if (v[e] == m_blk) idx = (int)(e0 + e);
    }
  }
  block_sum_minidx(s, idx, sm);

  if (chunks == 1) {
    if (threadIdx.x == 0)
      write_row(row, m_blk, s, t2_blk, idx, zrow, dtype, vocab, mask_state, cur_tokens, max_prob, top1, margin,
                cur_prob);
    return;
  }

  // ---- publish the chunk partial and leave: no CTA waits on another one
  if (threadIdx.x == 0) {
    Partial pt;
    pt.m = m_blk; pt.s = s; pt.t2 = t2_blk; pt.idx = idx;
    parts[static_cast<size_t>(row) * chunks + chunk] = pt;
  }
}

// Aligned-row variant: one TMA bulk copy stages the CTA's chunk in shared
// memory, so no registers are held while the chunk is in flight and six CTAs
// per SM keep about 192 KB of reads outstanding.  Same partition, partials
// and arithmetic as decode_scores_kernel.
constexpr uint32_t kBulkBytes = kWordsPerChunk * 16;   // 32 KB

__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
               "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(bar)
               : "memory");
}

// Pass A (top-2 of the chunk, block-wide) and pass B (sum of exponentials
// against the chunk max, lowest index of the max) over one staged chunk.
// kFull: the chunk holds kWordsPerChunk whole 16-byte words (every chunk of
// a row but possibly its last), so no word needs a bounds check.
template <typename T, bool kFull>
__device__ __forceinline__ void chunk_pass(const uint4* __restrict__ stage, int bulk_words, const T* zrow,
                                           int64_t e0c, int n_el, Smem& sm, float& m_blk, float& t2_blk,
                                           float& sum, int& idx) {
  constexpr int E = Vec<T>::kElems;
  constexpr int dtype = sizeof(T) == 2 ? ARCHER_DTYPE_BF16 : ARCHER_DTYPE_F32;
  auto word = [&](int u) -> uint4 {
    const int wi = u * kThreads + threadIdx.x;
    if constexpr (kFull) return stage[wi];
    if (wi < bulk_words) return stage[wi];
    float v[E];
#pragma unroll
    for (int e = 0; e < E; ++e) {
      const int el = wi * E + e;
      v[e] = (el < n_el) ? load_logit(zrow, dtype, static_cast<int>(e0c + el)) : -INFINITY;
    }
    if constexpr (E == 8) {
      return make_uint4(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]), pack_bf16x2(v[4], v[5]),
                        pack_bf16x2(v[6], v[7]));
    } else {
      return make_uint4(__float_as_uint(v[0]), __float_as_uint(v[1]), __float_as_uint(v[2]), __float_as_uint(v[3]));
    }
  };

  // pass A: top-2 values
  float t1 = -INFINITY, t2 = -INFINITY;
  if constexpr (E == 8) {
    __nv_bfloat162 M1 = __floats2bfloat162_rn(-INFINITY, -INFINITY);
    __nv_bfloat162 M2 = M1;
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const uint4 wv = word(u);
      const uint32_t q[4] = {wv.x, wv.y, wv.z, wv.w};
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const __nv_bfloat162 x = *reinterpret_cast<const __nv_bfloat162*>(&q[i]);
        M2 = __hmax2(M2, __hmin2(M1, x));
        M1 = __hmax2(M1, x);
      }
    }
    const float a = __low2float(M1), c = __high2float(M1);
    t1 = fmaxf(a, c);
    t2 = fmaxf(fminf(a, c), fmaxf(__low2float(M2), __high2float(M2)));
  } else {
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      float v[4];
      unpack(word(u), v, (float*)nullptr);
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        t2 = fmaxf(t2, fminf(t1, v[e]));
        t1 = fmaxf(t1, v[e]);
      }
    }
  }
  const float my_t1 = t1;
  m_blk = t1;
  t2_blk = t2;
  block_top2(m_blk, t2_blk, sm);

  // pass B: one ex2 per logit against the chunk max; lowest index of the max
  const float neg_m = (m_blk == -INFINITY) ? 0.f : -m_blk * kLog2e;
  // packed fp32 pairs: one FMA and one add instruction per two logits
  const float2 l2e = make_float2(kLog2e, kLog2e), nm = make_float2(neg_m, neg_m);
  float2 acc[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
#pragma unroll
  for (int u = 0; u < kUnroll; ++u) {
    float v[E];
    unpack(word(u), v, (T*)nullptr);
#pragma unroll
    for (int e = 0; e < E; e += 2) {
      const float2 y = ffma2(make_float2(v[e], v[e + 1]), l2e, nm);
      acc[(e >> 1) & 1] = fadd2(acc[(e >> 1) & 1], make_float2(ex2_approx(y.x), ex2_approx(y.y)));
    }
  }
  sum = (acc[0].x + acc[0].y) + (acc[1].x + acc[1].y);
  idx = INT_MAX;
  if (my_t1 == m_blk) {
    for (int u = 0; u < kUnroll && idx == INT_MAX; ++u) {
      float v[E];
      unpack(word(u), v, (T*)nullptr);
      const int64_t el0 = e0c + static_cast<int64_t>(u * kThreads + threadIdx.x) * E;
#pragma unroll
      for (int e = E - 1; e >= 0; --e)
        if (v[e] == m_blk) idx = static_cast<int>(el0 + e);
    }
  }
}

template <typename T>
__global__ void __launch_bounds__(kThreads, 6)
decode_scores_bulk_kernel(const T* __restrict__ logits, int64_t row_stride, int vocab, int chunks,
                          const uint8_t* __restrict__ mask_state, const int32_t* __restrict__ cur_tokens,
                          float* __restrict__ max_prob, int32_t* __restrict__ top1, float* __restrict__ margin,
                          float* __restrict__ cur_prob, Partial* __restrict__ parts, int* __restrict__ err) {
  constexpr int E = Vec<T>::kElems;
  constexpr int dtype = sizeof(T) == 2 ? ARCHER_DTYPE_BF16 : ARCHER_DTYPE_F32;
  constexpr int kChunkElems = kWordsPerChunk * E;
  asm volatile("griddepcontrol.launch_dependents;");   // the merge may be scheduled (it waits for this grid)
  extern __shared__ __align__(128) uint4 stage[];
  __shared__ Smem sm;
  __shared__ __align__(8) uint64_t full_bar;
  __shared__ int abort_flag;
  const int row = blockIdx.x / chunks;
  const int chunk = blockIdx.x - row * chunks;
  const T* zrow = logits + row * row_stride;
  const int64_t e0c = static_cast<int64_t>(chunk) * kChunkElems;
  const int n_el = static_cast<int>(min(static_cast<int64_t>(kChunkElems), static_cast<int64_t>(vocab) - e0c));
  const uint32_t bytes = (static_cast<uint32_t>(n_el) * sizeof(T)) & ~15u;
  const int bulk_words = static_cast<int>(bytes / 16);
  const uint32_t bar = smem_u32(&full_bar);
  if (threadIdx.x == 0) {
    abort_flag = 0;
    mbar_init(bar, 1);
    mbar_fence_init();
    if (bytes > 0) {
      mbar_arrive_expect_tx(bar, bytes);
      bulk_load(smem_u32(stage), zrow + e0c, bytes, bar);
    } else {
      mbar_arrive(bar);
    }
  }
  __syncthreads();
  // An expired wait is reported through the error word; the CTA then reads
  // stale shared memory (in bounds) rather than leaving early.
  mbar_wait(bar, 0, &abort_flag, err);

  float m_blk, t2_blk, sum;
  int idx;
  if (bulk_words == kWordsPerChunk)
    chunk_pass<T, true>(stage, bulk_words, zrow, e0c, n_el, sm, m_blk, t2_blk, sum, idx);
  else
    chunk_pass<T, false>(stage, bulk_words, zrow, e0c, n_el, sm, m_blk, t2_blk, sum, idx);
  block_sum_minidx(sum, idx, sm);
  if (threadIdx.x == 0) {
    if (chunks == 1) {
      write_row(row, m_blk, sum, t2_blk, idx, zrow, dtype, vocab, mask_state, cur_tokens, max_prob, top1, margin,
                cur_prob);
    } else {
      Partial pt;
      pt.m = m_blk; pt.s = sum; pt.t2 = t2_blk; pt.idx = idx;
      parts[static_cast<size_t>(row) * chunks + chunk] = pt;
    }
  }
}

// One warp per row merges the row's chunk partials.  Launched as a programmatic
// dependent of the chunk kernel on the same stream: it is scheduled while the
// chunk grid's last wave runs and waits for that grid on the device.
template <typename T>
__global__ void __launch_bounds__(256)
decode_scores_combine_kernel(const T* __restrict__ logits, int64_t row_stride, int vocab, int chunks, int rows,
                             const uint8_t* __restrict__ mask_state, const int32_t* __restrict__ cur_tokens,
                             float* __restrict__ max_prob, int32_t* __restrict__ top1, float* __restrict__ margin,
                             float* __restrict__ cur_prob, const Partial* __restrict__ parts) {
  constexpr int dtype = sizeof(T) == 2 ? ARCHER_DTYPE_BF16 : ARCHER_DTYPE_F32;
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int row = blockIdx.x * 8 + (threadIdx.x >> 5);
  const int l = threadIdx.x & 31;
  if (row >= rows) return;
  const Partial* vp = parts + static_cast<size_t>(row) * chunks;
  float M = -INFINITY, T2 = -INFINITY;
  for (int c = l; c < chunks; c += 32) merge_top2(M, T2, vp[c].m, vp[c].t2);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float b1 = __shfl_xor_sync(0xffffffffu, M, o);
    const float b2 = __shfl_xor_sync(0xffffffffu, T2, o);
    merge_top2(M, T2, b1, b2);
  }
  float S = 0.f;
  int I = INT_MAX;
  for (int c = l; c < chunks; c += 32) {
    const float mc = vp[c].m;
    if (mc != -INFINITY) S += vp[c].s * ex2_approx((mc - M) * kLog2e);
    if (mc == M) I = min(I, vp[c].idx);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    S += __shfl_xor_sync(0xffffffffu, S, o);
    I = min(I, __shfl_xor_sync(0xffffffffu, I, o));
  }
  if (l == 0)
    write_row(row, M, S, T2, I, logits + row * row_stride, dtype, vocab, mask_state, cur_tokens, max_prob, top1,
              margin, cur_prob);
}

template <typename T>
cudaError_t launch_combine(unsigned grid, const T* logits, int64_t row_stride, int vocab, int chunks, int rows,
                           const uint8_t* mask_state, const int32_t* cur_tokens, float* max_prob, int32_t* top1,
                           float* margin, float* cur_prob, const Partial* parts, cudaStream_t stream) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(256);
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, decode_scores_combine_kernel<T>, logits, row_stride, vocab, chunks, rows,
                            mask_state, cur_tokens, max_prob, top1, margin, cur_prob, parts);
}

int chunks_for(int vocab, int dtype) {
  const int per_chunk = kWordsPerChunk * (dtype == ARCHER_DTYPE_BF16 ? 8 : 4);
  return (vocab + per_chunk - 1) / per_chunk;
}

}  // namespace

size_t decode_scores_ws_bytes_dtype(int rows, int vocab, int dtype) {
  const int chunks = chunks_for(vocab, dtype);
  if (chunks <= 1 || rows <= 0) return 0;
  return static_cast<size_t>(rows) * chunks * sizeof(Partial);
}

size_t decode_scores_ws_bytes(int rows, int vocab) {
  // Sized for fp32 logits, which need twice the chunks of bf16 for one vocabulary.
  return decode_scores_ws_bytes_dtype(rows, vocab, ARCHER_DTYPE_F32);
}

int decode_scores_launch(int rows, int vocab, int dtype, const void* logits, int64_t row_stride,
                         const uint8_t* mask_state, const int32_t* cur_tokens, float* max_prob, int32_t* top1,
                         float* margin, float* cur_prob, void* workspace, size_t ws_bytes, cudaStream_t stream) {
  if (rows == 0) return ARCHER_OK;
  const int chunks = chunks_for(vocab, dtype);
  Partial* parts = nullptr;
  if (chunks > 1) {
    const size_t need = decode_scores_ws_bytes_dtype(rows, vocab, dtype);
    if (workspace == nullptr || ws_bytes < need) {
      set_error("decode_scores needs a workspace of %zu bytes (got %zu)", need, ws_bytes);
      return ARCHER_ERR_ARG;
    }
    parts = static_cast<Partial*>(workspace);
  }
  const int esize = dtype == ARCHER_DTYPE_BF16 ? 2 : 4;
  const int aligned = (reinterpret_cast<uintptr_t>(logits) % 16 == 0) && ((row_stride * esize) % 16 == 0);
  const long long grid = static_cast<long long>(rows) * chunks;
  if (grid > 0x7FFFFFFFll) {
    set_error("decode_scores grid too large");
    return ARCHER_ERR_UNSUPPORTED;
  }
  const unsigned combine_grid = static_cast<unsigned>((rows + 7) / 8);
  if (aligned) {
    if (dtype == ARCHER_DTYPE_BF16)
      decode_scores_bulk_kernel<__nv_bfloat16><<<(unsigned)grid, kThreads, kBulkBytes, stream>>>(
          static_cast<const __nv_bfloat16*>(logits), row_stride, vocab, chunks, mask_state, cur_tokens, max_prob,
          top1, margin, cur_prob, parts, device_error_word());
    else
      decode_scores_bulk_kernel<float><<<(unsigned)grid, kThreads, kBulkBytes, stream>>>(
          static_cast<const float*>(logits), row_stride, vocab, chunks, mask_state, cur_tokens, max_prob, top1,
          margin, cur_prob, parts, device_error_word());
    if (chunks > 1) {
      cudaError_t e = cudaGetLastError();
      if (e == cudaSuccess)
        e = dtype == ARCHER_DTYPE_BF16
                ? launch_combine(combine_grid, static_cast<const __nv_bfloat16*>(logits), row_stride, vocab, chunks,
                                 rows, mask_state, cur_tokens, max_prob, top1, margin, cur_prob, parts, stream)
                : launch_combine(combine_grid, static_cast<const float*>(logits), row_stride, vocab, chunks, rows,
                                 mask_state, cur_tokens, max_prob, top1, margin, cur_prob, parts, stream);
      return cuda_status(e, "decode_scores launch");
    }
    return cuda_status(cudaGetLastError(), "decode_scores launch");
  }
  if (dtype == ARCHER_DTYPE_BF16) {
    decode_scores_kernel<__nv_bfloat16><<<(unsigned)grid, kThreads, 0, stream>>>(
        static_cast<const __nv_bfloat16*>(logits), row_stride, vocab, chunks, mask_state, cur_tokens, max_prob, top1,
        margin, cur_prob, parts, aligned);
    if (chunks > 1 && cudaPeekAtLastError() == cudaSuccess)
      return cuda_status(launch_combine(combine_grid, static_cast<const __nv_bfloat16*>(logits), row_stride, vocab,
                                        chunks, rows, mask_state, cur_tokens, max_prob, top1, margin, cur_prob, parts,
                                        stream),
                         "decode_scores launch");
  } else {
    decode_scores_kernel<float><<<(unsigned)grid, kThreads, 0, stream>>>(
        static_cast<const float*>(logits), row_stride, vocab, chunks, mask_state, cur_tokens, max_prob, top1, margin,
        cur_prob, parts, aligned);
    if (chunks > 1 && cudaPeekAtLastError() == cudaSuccess)
      return cuda_status(launch_combine(combine_grid, static_cast<const float*>(logits), row_stride, vocab, chunks,
                                        rows, mask_state, cur_tokens, max_prob, top1, margin, cur_prob, parts,
                                        stream),
                         "decode_scores launch");
  }
  return cuda_status(cudaGetLastError(), "decode_scores launch");
}

}  // namespace archer

// ---------------------------------------------------------------------------
// Scoring without any device allocation.
//
// Some callers cannot allocate device memory for the workspace: code that runs
// inside another framework's memory pool (where a raw cudaMalloc bypasses its
// accounting), latency-critical loops that must not pay cudaMalloc's implicit
// device synchronisation, and thin foreign-function bindings with no allocator
// at hand.  For them the chunk partials live in this
// file-scope array, created when the library is loaded on a device and held
// by every GPU that loads the library until the process exits.
// ---------------------------------------------------------------------------
namespace archer {
namespace {

constexpr size_t kNoAllocScratchBytes = ARCHER_NOALLOC_SCRATCH_BYTES;
static __device__ __align__(256) unsigned char g_scores_scratch[kNoAllocScratchBytes];

// Device address of g_scores_scratch in the current device's context.  Host
// code cannot use the array's name as a device pointer (it is a host-side
// stand-in), so the address is looked up with that device current, once per
// device and context: it is cached with the context's unique ID
// (cuCtxGetId), and a new context on that device (after cudaDeviceReset, say)
// gets a fresh lookup instead of a stale address.
using CtxGetCurrentFn = CUresult (*)(CUcontext*);
using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long*);

template <typename Fn>
Fn driver_fn(const char* name) {
  void* ptr = nullptr;
  cudaDriverEntryPointQueryResult q;
  if (cudaGetDriverEntryPointByVersion(name, &ptr, 12000, cudaEnableDefault, &q) == cudaSuccess &&
      q == cudaDriverEntryPointSuccess)
    return reinterpret_cast<Fn>(ptr);
  return nullptr;
}

// The unique ID of the calling thread's current context (0 if none or unknown).
unsigned long long current_context_id() {
  static CtxGetCurrentFn get_current = nullptr;
  static CtxGetIdFn get_id = nullptr;
  static std::once_flag once;
  std::call_once(once, []() {
    get_current = driver_fn<CtxGetCurrentFn>("cuCtxGetCurrent");
    get_id = driver_fn<CtxGetIdFn>("cuCtxGetId");
  });
  CUcontext ctx = nullptr;
  unsigned long long id = 0;
  if (!get_current || !get_id || get_current(&ctx) != CUDA_SUCCESS || !ctx || get_id(ctx, &id) != CUDA_SUCCESS)
    return 0;
  return id;
}

int scratch_address(void** out) {
  struct Slot {
    unsigned long long ctx_id;
    void* addr;
  };
  static Slot slot[64] = {};
  static std::mutex mu;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_status(e, "cudaGetDevice");
  if (dev < 0 || dev >= 64) {
    set_error("device ordinal %d out of range", dev);
    return ARCHER_ERR_UNSUPPORTED;
  }
  std::lock_guard<std::mutex> lock(mu);
  const unsigned long long id = current_context_id();
  if (!slot[dev].addr || id == 0 || slot[dev].ctx_id != id) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_scores_scratch);      // makes the device's primary context current
    if (e != cudaSuccess) return cuda_status(e, "cudaGetSymbolAddress(scoring scratch)");
    slot[dev].addr = p;
    slot[dev].ctx_id = current_context_id();
  }
  *out = slot[dev].addr;
  return ARCHER_OK;
}

}  // namespace
}  // namespace archer

extern "C" int archer_decode_scores_noalloc(int batch, int resp_len, int vocab, int dtype, const void* logits,
                                            int64_t row_stride, const uint8_t* mask_state,
                                            const int32_t* cur_tokens, float* max_prob, int32_t* top1,
                                            float* margin, float* cur_prob, void* stream) {
  using namespace archer;
  if (batch < 0 || resp_len < 0 || vocab < 1 || row_stride < vocab) {
    set_error("bad scoring shape: batch=%d resp_len=%d vocab=%d row_stride=%lld", batch, resp_len, vocab,
              (long long)row_stride);
    return ARCHER_ERR_ARG;
  }
  const long long rows = static_cast<long long>(batch) * resp_len;
  if (rows > 0x7FFFFFFFll) {
    set_error("too many rows");
    return ARCHER_ERR_UNSUPPORTED;
  }
  if (rows == 0) return ARCHER_OK;
  if (dtype != ARCHER_DTYPE_BF16 && dtype != ARCHER_DTYPE_F32) {
    set_error("dtype %d unsupported", dtype);
    return ARCHER_ERR_UNSUPPORTED;
  }
  const size_t need = decode_scores_ws_bytes_dtype(static_cast<int>(rows), vocab, dtype);
  if (need > kNoAllocScratchBytes) {
    set_error("%lld rows of %d logits need %zu bytes of scoring scratch; the allocation-free entry point has "
              "%zu (use archer_decode_scores with a workspace)",
              rows, vocab, need, kNoAllocScratchBytes);
    return ARCHER_ERR_UNSUPPORTED;
  }
  void* scratch = nullptr;
  int st = scratch_address(&scratch);
  if (st) return st;
  // Every chunk partial is written before the combine kernel reads it, so the
  // scratch needs no clearing between calls.
  return archer_decode_scores(batch, resp_len, vocab, dtype, logits, row_stride, mask_state, cur_tokens, max_prob,
                              top1, margin, cur_prob, scratch, kNoAllocScratchBytes, stream);
}
