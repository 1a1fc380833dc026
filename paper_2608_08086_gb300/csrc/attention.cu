// Asymmetric cached attention and prompt-refresh attention for sm_103a.
//
// Computes, per (sequence b, query head h), Attn(Q, [K_p || K_g], [V_p || V_g])
// with no mask (Sec. 4.1, Eq. archer-attention): the cached step uses the G
// response queries and the anchored prompt cache K_p(g_r); the refresh pass
// (Sec. 4.2, Algorithm 1's FullForward) uses all N = P + G queries and the
// fresh prompt K/V.  The KV loop walks the prompt segment and then the
// response segment through two TMA tensor maps, so the concatenation is never
// formed in memory.  GQA: query head h reads KV head h / (Hq / Hkv).
//
// One CTA = one 128-row query tile of one (b, h); 6 warps:
//   warps 0-3  softmax: thread t owns query row t (TMEM lane t); online
//              softmax in the log2 domain with a lazily raised running max
//              (O and l are rescaled only when the tile max exceeds the max in
//              use by more than 2^8), P written to TMEM as bf16 pairs.
//   warp 4     TMA producer: Q once, then K and V tiles into 2-stage rings.
//   warp 5     MMA issuer (one thread): S = Q K^T (SS, K-major operands) into
//              a double-buffered TMEM S, then O += P V (P from TMEM, V as an
//              MN-major smem operand), fp32 accumulation in TMEM.
// TMEM (512 columns): S0 [0,128) S1 [128,256) O [256,256+D) P0 [384,448) P1 [448,512).
// Every hand-off is an mbarrier; every wait is bounded (archer_device.cuh).

#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <mutex>

#include <cudaTypedefs.h>

#include "archer_device.cuh"
#include "archer_internal.h"
#include "tmem_ldst.cuh"

namespace archer {
namespace {

constexpr int kBM = 128;          // query rows per CTA (tcgen05 M)
constexpr int kBN = 128;          // keys per KV tile (N of Q K^T, K of P V)
constexpr int kThreads = 192;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColS0 = 0, kColS1 = 128, kColO = 256, kColP0 = 384, kColP1 = 448;
constexpr uint32_t kChunkBytes = 128 * 128;   // 128 rows x 128 B (64 bf16) swizzle region

struct AttnParams {
  int P, G, Hq, Hkv, M;
  int q_begin_refresh, q_begin_cached, default_refresh;
  float scale_log2;           // softmax_scale * log2(e)
  long long wait_limit;       // SM clocks a bounded wait may take
  int debug_skip_last_pv;     // test hook: withhold the last PV and its commits
  const uint8_t* flags;
  __nv_bfloat16* out;
  float* lse;
  int* err;
};

template <int D>
struct Layout {
  static constexpr int kChunks = D / 64;                  // 128-byte column chunks
  static constexpr uint32_t kTile = kChunks * kChunkBytes;  // one 128-row tile of D bf16
  static constexpr int kKS = 2, kVS = 2;                  // K / V ring stages
  static constexpr uint32_t kOffQ = 0;
  static constexpr uint32_t kOffK = kOffQ + kTile;
  static constexpr uint32_t kOffV = kOffK + kKS * kTile;
  static constexpr uint32_t kOffBar = kOffV + kVS * kTile;
  // q_full, k_full[KS], k_empty[KS], v_full[VS], v_empty[VS], s_full[2], p_full[2], pv_done[2]
  static constexpr int kBars = 1 + 2 * kKS + 2 * kVS + 2 + 2 + 2;
  static constexpr uint32_t kOffHolder = kOffBar + 8 * kBars;
  static constexpr uint32_t kOffAbort = kOffHolder + 4;
  static constexpr uint32_t kUsed = kOffAbort + 4;
  // + 1 KB to align the base to 1024 B; at least 120 KB so that one CTA
  // holds an SM (the CTA allocates all 512 TMEM columns).
  static constexpr uint32_t kSmemBytes = (kUsed + 1024 > 120 * 1024) ? kUsed + 1024 : 120 * 1024;
};

// Warp-uniform bounded wait for the softmax warps (tcgen05.ld/st are
// .sync.aligned, so all 32 lanes must take the same path).
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, volatile int* abort,
                                          int* err, long long limit) {
  const long long t0 = clock64();
  while (true) {
    const bool done = mbar_try_wait(bar, parity);
    if (__all_sync(0xffffffffu, done)) return true;
    const bool give_up = (*abort != 0) || (clock64() - t0 > limit);
    if (__any_sync(0xffffffffu, give_up)) {
      if ((threadIdx.x & 31) == 0 && !*abort) {
        *abort = 1;
        if (err) atomicOr(err, kErrWaitTimeout);
      }
      return false;
    }
  }
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
attn_fwd_kernel(const __grid_constant__ CUtensorMap tmQ,
                const __grid_constant__ CUtensorMap tmKpR, const __grid_constant__ CUtensorMap tmVpR,
                const __grid_constant__ CUtensorMap tmKpC, const __grid_constant__ CUtensorMap tmVpC,
                const __grid_constant__ CUtensorMap tmKg, const __grid_constant__ CUtensorMap tmVg,
                const AttnParams p) {
  using L = Layout<D>;
  extern __shared__ uint8_t smem_raw[];

  const int qt = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const bool refresh = p.flags ? (p.flags[b] != 0) : (p.default_refresh != 0);
  const int q0 = (refresh ? p.q_begin_refresh : p.q_begin_cached) + qt * kBM;
  if (q0 >= p.M) return;  // uniform over the CTA, before any barrier or TMEM use

  const int kvh = h / (p.Hq / p.Hkv);
  const int n_p = (p.P + kBN - 1) / kBN;
  const int n_g = (p.G + kBN - 1) / kBN;
  const int T = n_p + n_g;

  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (base - raw);
  const uint32_t sQ = base + L::kOffQ;
  const uint32_t sK = base + L::kOffK;
  const uint32_t sV = base + L::kOffV;
  const uint32_t bars = base + L::kOffBar;
  const uint32_t bar_q_full = bars;
  const uint32_t bar_k_full = bars + 8;                         // + 8 * stage
  const uint32_t bar_k_empty = bar_k_full + 8 * L::kKS;
  const uint32_t bar_v_full = bar_k_empty + 8 * L::kKS;
  const uint32_t bar_v_empty = bar_v_full + 8 * L::kVS;
  const uint32_t bar_s_full = bar_v_empty + 8 * L::kVS;         // + 8 * buffer
  const uint32_t bar_p_full = bar_s_full + 16;
  const uint32_t bar_pv_done = bar_p_full + 16;                 // + 8 * (tile & 1)
  uint32_t* holder = reinterpret_cast<uint32_t*>(gbase + L::kOffHolder);
  volatile int* abort = reinterpret_cast<volatile int*>(gbase + L::kOffAbort);

  const int warp = threadIdx.x >> 5;
  if (threadIdx.x == 0) {
    mbar_init(bar_q_full, 1);
    for (int s = 0; s < L::kKS; ++s) {
      mbar_init(bar_k_full + 8 * s, 1);
      mbar_init(bar_k_empty + 8 * s, 1);
    }
    for (int s = 0; s < L::kVS; ++s) {
      mbar_init(bar_v_full + 8 * s, 1);
      mbar_init(bar_v_empty + 8 * s, 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(bar_s_full + 8 * i, 1);
      mbar_init(bar_p_full + 8 * i, kBM);
      mbar_init(bar_pv_done + 8 * i, 1);
    }
    *abort = 0;
    mbar_fence_init();
  }
  if (warp == 5) {
    tmem_alloc(smem_u32(holder), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *holder;

  if (warp == 4) {
    // ------------------------------------------------------------ producer
    if (elect_lane0()) {
      const CUtensorMap* mKp = refresh ? &tmKpR : &tmKpC;
      const CUtensorMap* mVp = refresh ? &tmVpR : &tmVpC;
      tma_prefetch_map(&tmQ);
      mbar_arrive_expect_tx(bar_q_full, L::kTile);
      for (int c = 0; c < L::kChunks; ++c)
        tma_load_4d(sQ + c * kChunkBytes, &tmQ, bar_q_full, c * 64, h, q0, b);
      for (int j = 0; j < T; ++j) {
        const bool in_prompt = j < n_p;
        const int row = in_prompt ? j * kBN : (j - n_p) * kBN;
        const int ks = j % L::kKS, kuse = j / L::kKS;
        if (kuse > 0 && !mbar_wait(bar_k_empty + 8 * ks, (kuse - 1) & 1, abort, p.err, p.wait_limit)) break;
        mbar_arrive_expect_tx(bar_k_full + 8 * ks, L::kTile);
        const CUtensorMap* mk = in_prompt ? mKp : &tmKg;
        for (int c = 0; c < L::kChunks; ++c)
          tma_load_4d(sK + ks * L::kTile + c * kChunkBytes, mk, bar_k_full + 8 * ks, c * 64, kvh,
                      row, b);
        const int vs = j % L::kVS, vuse = j / L::kVS;
        if (vuse > 0 && !mbar_wait(bar_v_empty + 8 * vs, (vuse - 1) & 1, abort, p.err, p.wait_limit)) break;
        mbar_arrive_expect_tx(bar_v_full + 8 * vs, L::kTile);
        const CUtensorMap* mv = in_prompt ? mVp : &tmVg;
        for (int c = 0; c < L::kChunks; ++c)
          tma_load_4d(sV + vs * L::kTile + c * kChunkBytes, mv, bar_v_full + 8 * vs, c * 64, kvh,
                      row, b);
      }
    }
    __syncwarp();
  } else if (warp == 5) {
    // ------------------------------------------------------------ MMA issuer
    if (elect_lane0()) {
      constexpr uint32_t idesc_qk = idesc_bf16_f32(kBM, kBN, 0, 0);
      constexpr uint32_t idesc_pv = idesc_bf16_f32(kBM, D, 0, 1);
      auto issue_qk = [&](uint32_t s_col, uint32_t k_tile) {
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t off = (kk >> 2) * kChunkBytes + (kk & 3) * 32;
          umma_ss(tmem + s_col, sdesc_sw128(sQ + off, 16, 1024), sdesc_sw128(k_tile + off, 16, 1024),
                  idesc_qk, kk > 0 ? 1u : 0u);
        }
      };
      auto issue_pv = [&](uint32_t p_col, uint32_t v_tile, bool acc) {
#pragma unroll
        for (int kk = 0; kk < kBN / 16; ++kk) {
          umma_ts(tmem + kColO, tmem + p_col + kk * 8, sdesc_sw128(v_tile + kk * 2048, kChunkBytes, 1024),
                  idesc_pv, (acc || kk > 0) ? 1u : 0u);
        }
      };
      bool ok = mbar_wait(bar_q_full, 0, abort, p.err, p.wait_limit) && mbar_wait(bar_k_full, 0, abort, p.err, p.wait_limit);
      if (ok) {
        tc_fence_after();
        issue_qk(kColS0, sK);
        umma_commit(bar_s_full);
        umma_commit(bar_k_empty);
      }
      for (int j = 0; ok && j < T; ++j) {
        if (j + 1 < T) {
          const int ks = (j + 1) % L::kKS;
          if (!mbar_wait(bar_k_full + 8 * ks, ((j + 1) / L::kKS) & 1, abort, p.err, p.wait_limit)) break;
          tc_fence_after();
          const int sb = (j + 1) & 1;
          issue_qk(sb ? kColS1 : kColS0, sK + ks * L::kTile);
          umma_commit(bar_s_full + 8 * sb);
          umma_commit(bar_k_empty + 8 * ks);
        }
        const int vs = j % L::kVS;
        if (!mbar_wait(bar_v_full + 8 * vs, (j / L::kVS) & 1, abort, p.err, p.wait_limit)) break;
        if (!mbar_wait(bar_p_full + 8 * (j & 1), (j >> 1) & 1, abort, p.err, p.wait_limit)) break;
        if (p.debug_skip_last_pv && j == T - 1) break;   // the softmax's last wait must now expire
        tc_fence_after();
        issue_pv((j & 1) ? kColP1 : kColP0, sV + vs * L::kTile, j > 0);
        umma_commit(bar_pv_done + 8 * (j & 1));
        umma_commit(bar_v_empty + 8 * vs);
      }
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ softmax
    const int r = threadIdx.x;                                    // query row in the tile
    const uint32_t t_lane = tmem + (static_cast<uint32_t>(warp * 32) << 16);
    const float sl2 = p.scale_log2;
    float m_used = -INFINITY;                                    // running max (log2 units)
    float l_sum = 0.f;
    bool ok = true;
    for (int j = 0; j < T; ++j) {
      const int sb = j & 1;
      if (!warp_wait(bar_s_full + 8 * sb, (j >> 1) & 1, abort, p.err, p.wait_limit)) { ok = false; break; }
      tc_fence_after();
      uint32_t sr[128];
      tmem_ld_128(t_lane + (sb ? kColS1 : kColS0), sr);
      float x[128];
#pragma unroll
      for (int c = 0; c < 128; ++c) x[c] = __uint_as_float(sr[c]);
      const int valid = j < n_p ? min(kBN, p.P - j * kBN) : min(kBN, p.G - (j - n_p) * kBN);
      if (valid < kBN) {
#pragma unroll
        for (int c = 0; c < 128; ++c)
          if (c >= valid) x[c] = -INFINITY;
      }
      float mx[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) mx[i] = x[i];
#pragma unroll
      for (int c = 8; c < 128; ++c) mx[c & 7] = fmaxf(mx[c & 7], x[c]);
      const float tmax = fmaxf(fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])),
                               fmaxf(fmaxf(mx[4], mx[5]), fmaxf(mx[6], mx[7])));
      const float mt2 = tmax * sl2;
      // PV_j commits to pv_done[j & 1], so each barrier's next phase belongs to
      // a PV that needs this thread's next P: no wait below can see its
      // barrier two phases ahead.
      if (j >= 2) {
        // P[sb] was last read by PV_{j-2}.
        if (!warp_wait(bar_pv_done + 8 * sb, ((j - 2) >> 1) & 1, abort, p.err, p.wait_limit)) { ok = false; break; }
        tc_fence_after();
      }
      if (j == 0) {
        m_used = mt2;
      } else if (__any_sync(0xffffffffu, mt2 > m_used + 8.0f)) {
        // Rescale O: wait until PV_{j-1} has finished accumulating into it.
        if (!warp_wait(bar_pv_done + 8 * (sb ^ 1), ((j - 1) >> 1) & 1, abort, p.err, p.wait_limit)) { ok = false; break; }
        tc_fence_after();
        const float m_new = fmaxf(m_used, mt2);
        const float alpha = ex2_approx(m_used - m_new);
        m_used = m_new;
        l_sum *= alpha;
#pragma unroll
        for (int c0 = 0; c0 < D; c0 += 32) {
          uint32_t o[32];
          tmem_ld_32(t_lane + kColO + c0, o);
#pragma unroll
          for (int c = 0; c < 32; ++c) o[c] = __float_as_uint(__uint_as_float(o[c]) * alpha);
          tmem_st_32(t_lane + kColO + c0, o);
        }
      }
      const float neg_m = -m_used;
      uint32_t pk[64];
      float ls[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int c = 0; c < 64; ++c) {
        const float p0 = ex2_approx(fmaf(x[2 * c], sl2, neg_m));
        const float p1 = ex2_approx(fmaf(x[2 * c + 1], sl2, neg_m));
        ls[c & 3] += p0 + p1;
        pk[c] = pack_bf16x2(p0, p1);
      }
      l_sum += (ls[0] + ls[1]) + (ls[2] + ls[3]);
      tmem_st_64(t_lane + (sb ? kColP1 : kColP0), pk);
      tc_fence_before();
      mbar_arrive(bar_p_full + 8 * sb);
    }
    if (ok && warp_wait(bar_pv_done + 8 * ((T - 1) & 1), ((T - 1) >> 1) & 1, abort, p.err, p.wait_limit)) {
      tc_fence_after();
      const float inv_l = 1.0f / l_sum;
      const int q = q0 + r;
      const bool live = q < p.M;
      __nv_bfloat16* orow = p.out + ((static_cast<size_t>(b) * p.M + q) * p.Hq + h) * D;
#pragma unroll
      for (int c0 = 0; c0 < D; c0 += 32) {
        uint32_t o[32];
        tmem_ld_32(t_lane + kColO + c0, o);
        uint32_t w[16];
#pragma unroll
        for (int c = 0; c < 16; ++c)
          w[c] = pack_bf16x2(__uint_as_float(o[2 * c]) * inv_l, __uint_as_float(o[2 * c + 1]) * inv_l);
        if (live) {
          uint4* dst = reinterpret_cast<uint4*>(orow + c0);
#pragma unroll
          for (int v = 0; v < 4; ++v) dst[v] = make_uint4(w[4 * v], w[4 * v + 1], w[4 * v + 2], w[4 * v + 3]);
        }
      }
      if (live && p.lse)
        p.lse[(static_cast<size_t>(b) * p.Hq + h) * p.M + q] = (m_used + log2f(l_sum)) * 0.69314718055994531f;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 5) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// ------------------------------------------------------------------ host side

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, []() {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  });
  return fn;
}

// [B, L, H, D] bf16 as a 4-D map (D, H, L, B) with a 64 x 1 x 128 x 1 box and
// 128-byte swizzle: one box = 128 rows of 128 bytes, a canonical SW128 region.
bool make_map(CUtensorMap* map, const void* ptr, int B, int L, int H, int D) {
  auto fn = encode_fn();
  if (!fn) return false;
  const cuuint64_t dims[4] = {(cuuint64_t)D, (cuuint64_t)H, (cuuint64_t)L, (cuuint64_t)B};
  const cuuint64_t strides[3] = {(cuuint64_t)D * 2, (cuuint64_t)H * D * 2, (cuuint64_t)L * H * D * 2};
  const cuuint32_t box[4] = {64, 1, 128, 1};
  const cuuint32_t estr[4] = {1, 1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(ptr), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int D>
int launch_d(const AttnCall& c, cudaStream_t stream) {
  using L = Layout<D>;
  static int configured_device = -1;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return cuda_status(cudaGetLastError(), "cudaGetDevice");
  if (configured_device != dev) {
    cudaError_t e = cudaFuncSetAttribute(attn_fwd_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)L::kSmemBytes);
    if (e != cudaSuccess) return cuda_status(e, "cudaFuncSetAttribute(attention)");
    configured_device = dev;
  }
  CUtensorMap mq, mkr, mvr, mkc, mvc, mkg, mvg;
  bool ok = make_map(&mq, c.q, c.B, c.M, c.Hq, D) && make_map(&mkg, c.kg, c.B, c.G, c.Hkv, D) &&
            make_map(&mvg, c.vg, c.B, c.G, c.Hkv, D);
  if (ok && c.P > 0) {
    ok = make_map(&mkr, c.kp_refresh, c.B, c.P, c.Hkv, D) && make_map(&mvr, c.vp_refresh, c.B, c.P, c.Hkv, D) &&
         make_map(&mkc, c.kp_cached, c.B, c.P, c.Hkv, D) && make_map(&mvc, c.vp_cached, c.B, c.P, c.Hkv, D);
  } else {
    mkr = mkg; mvr = mvg; mkc = mkg; mvc = mvg;   // never read when P == 0
  }
  if (!ok) {
    set_error("cuTensorMapEncodeTiled failed (pointer alignment or shape)");
    return ARCHER_ERR_CUDA;
  }
  AttnParams prm;
  prm.P = c.P; prm.G = c.G; prm.Hq = c.Hq; prm.Hkv = c.Hkv; prm.M = c.M;
  prm.q_begin_refresh = c.q_begin_refresh;
  prm.q_begin_cached = c.q_begin_cached;
  prm.default_refresh = c.default_refresh;
  prm.scale_log2 = c.scale * 1.4426950408889634f;
  // Test hook (host-set): ARCHER_DEBUG_STALL_ATTENTION=1 withholds the last PV
  // product, so a bounded wait expires after ~1e6 clocks and the call reports
  // ARCHER_ERR_TIMEOUT through archer_check_device; the context stays usable.
  const char* stall = std::getenv("ARCHER_DEBUG_STALL_ATTENTION");
  prm.debug_skip_last_pv = (stall && stall[0] == '1') ? 1 : 0;
  prm.wait_limit = prm.debug_skip_last_pv ? 1000000ll : kWaitLimitCycles;
  prm.flags = c.flags;
  prm.out = static_cast<__nv_bfloat16*>(c.out);
  prm.lse = c.lse;
  prm.err = device_error_word();
  // Query tiles needed by the longest query range (a refreshed sequence's).
  const int rows = c.M - (c.flags || c.default_refresh ? c.q_begin_refresh : c.q_begin_cached);
  const dim3 grid((rows + kBM - 1) / kBM, c.Hq, c.B);
  attn_fwd_kernel<D><<<grid, kThreads, L::kSmemBytes, stream>>>(mq, mkr, mvr, mkc, mvc, mkg, mvg, prm);
  return cuda_status(cudaGetLastError(), "attention launch");
}

// Bit-exact copy of each flagged sequence's prompt K/V (16-byte words); a
// NULL source skips that tensor.
__global__ void cache_rewrite_kernel(const uint4* __restrict__ k_src, const uint4* __restrict__ v_src,
                                     uint4* __restrict__ k_dst, uint4* __restrict__ v_dst,
                                     const uint8_t* __restrict__ flags, size_t words_per_seq) {
  const int b = blockIdx.y;
  if (flags && flags[b] == 0) return;
  const size_t off = static_cast<size_t>(b) * words_per_seq;
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < words_per_seq;
       i += (size_t)gridDim.x * blockDim.x) {
    if (k_src) k_dst[off + i] = k_src[off + i];
    if (v_src) v_dst[off + i] = v_src[off + i];
  }
}

}  // namespace

int attn_launch(const AttnCall& c, cudaStream_t stream) {
  if (c.B == 0) return ARCHER_OK;
  if (c.D == 128) return launch_d<128>(c, stream);
  if (c.D == 64) return launch_d<64>(c, stream);
  set_error("head_dim %d is not supported (64 or 128)", c.D);
  return ARCHER_ERR_UNSUPPORTED;
}

int cache_rewrite_launch(int B, size_t bytes_per_seq, const void* k_src, const void* v_src, void* k_dst,
                         void* v_dst, const uint8_t* flags, cudaStream_t stream) {
  if (B == 0 || bytes_per_seq == 0) return ARCHER_OK;
  const size_t words = bytes_per_seq / 16;
  int blocks_x = (int)std::min<size_t>((words + 255) / 256, 1024);
  const dim3 grid(blocks_x, B);
  cache_rewrite_kernel<<<grid, 256, 0, stream>>>(static_cast<const uint4*>(k_src), static_cast<const uint4*>(v_src),
                                                 static_cast<uint4*>(k_dst), static_cast<uint4*>(v_dst), flags,
                                                 words);
  return cuda_status(cudaGetLastError(), "cache rewrite launch");
}

}  // namespace archer
