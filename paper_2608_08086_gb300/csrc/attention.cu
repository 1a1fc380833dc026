// Attention launches (Sec. 4.1 Eq. archer-attention; Sec. 4.2 Algorithm 1's
// FullForward for the refresh): the launch plan (one or two query tiles per
// work item, key splits, the single-tile tail, the persistent grid), the TMA
// tensor maps, the kernel parameters, the split merge and the standalone
// cache copy.  The kernels themselves are in attention_kernels.cuh.

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdio>
#include <mutex>

#include "attention_kernels.cuh"

namespace archer {
namespace {

// ------------------------------------------------------------------ host side

std::atomic<int> g_debug_stall{0};   // set by archer_debug_stall_attention

constexpr int kMaxSplit = 16;
constexpr int kMinSplitTiles = 16;  // fewer key tiles: no split

// The current device's SM count, queried once per device (host threads may
// race on the first query; they store the same value).
int sm_count() {
  static std::atomic<int> count[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  int c = count[dev].load(std::memory_order_relaxed);
  if (c == 0 && cudaDeviceGetAttribute(&c, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess)
    count[dev].store(c, std::memory_order_relaxed);
  return c;
}

struct SplitPlan {
  int tiles_per_cta = 2, n_split = 1, per = 0;
  size_t bytes = 0;
};

// First, one query tile per CTA (the one-tile kernel, S double buffered) when
// a query range holds one tile anyway, or when two-tile CTAs would fill at
// most half the SMs (twice the CTAs, for latency-bound launches).  Then, when
// the grid still leaves SMs idle, the T key tiles are split across CTAs if
// they are many enough to pay for the merge: as many splits as whole grids
// fit on the SMs, none empty.  Measured on the GB300 with the one-tile kernel
// (B 1, 32 heads, G 256, launches replayed from a CUDA graph): P 2048 (T 18)
// 18.8 -> 17.4 us split in two, while P 1024 (T 10) is 12.3 us whole against
// 14.2 us split and T 6 9.3 us against 12.3 us.
SplitPlan split_plan(int B, int P, int G, int Hq, int D, int rows, int M, int sms) {
  SplitPlan sp;
  const int T = (P + kBN - 1) / kBN + (G + kBN - 1) / kBN;
  sp.per = T;
  const long long pairs = static_cast<long long>((rows + 2 * kBM - 1) / (2 * kBM)) * Hq * B;
  // One tile per CTA (the one-tile kernel) when a query range has one tile
  // anyway, or when two-tile CTAs would fill at most half the SMs.
  if (sms > 0 && (rows <= kBM || 2 * pairs <= sms)) sp.tiles_per_cta = 1;
  const int rows_per_cta = sp.tiles_per_cta * kBM;
  const long long ctas = static_cast<long long>((rows + rows_per_cta - 1) / rows_per_cta) * Hq * B;
  if (ctas <= 0 || sms <= 0 || ctas >= sms || T < kMinSplitTiles) return sp;
  int s = static_cast<int>(std::min<long long>(std::min(T, kMaxSplit), sms / ctas));
  if (s < 2) return sp;
  sp.per = (T + s - 1) / s;
  sp.n_split = (T + sp.per - 1) / sp.per;
  if (sp.n_split < 2) { sp.n_split = 1; sp.per = T; return sp; }
  sp.bytes = static_cast<size_t>(sp.n_split) * B * Hq * M * (static_cast<size_t>(D) * 4 + 8);
  return sp;
}

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
  CUtensorMap mq, mkr, mvr, mkc, mvc, mkg, mvg, mo;
  bool ok = make_map(&mq, c.q, c.B, c.M, c.Hq, D) && make_map(&mkg, c.kg, c.B, c.G, c.Hkv, D) &&
            make_map(&mvg, c.vg, c.B, c.G, c.Hkv, D) && make_map(&mo, c.out, c.B, c.M, c.Hq, D);
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
  // Test hook (archer_debug_stall_attention): the launch withholds the last
  // PV product, so a bounded wait expires after ~1e6 clocks and the call
  // reports ARCHER_ERR_TIMEOUT through archer_check_device; the context stays
  // usable.  One relaxed atomic load per launch.
  prm.debug_skip_last_pv = g_debug_stall.load(std::memory_order_relaxed);
  prm.wait_limit = prm.debug_skip_last_pv ? 1000000ll : kWaitLimitCycles;
  // The rewrite applies to launches that refresh some sequence.
  prm.rewrite = (c.P > 0 && (c.flags || c.default_refresh)) ? c.rewrite : 0;
  prm.kp_src = static_cast<const uint4*>(c.kp_refresh);
  prm.vp_src = static_cast<const uint4*>(c.vp_refresh);
  prm.kp_dst = static_cast<uint4*>(const_cast<void*>(c.kp_cached));
  prm.vp_dst = static_cast<uint4*>(const_cast<void*>(c.vp_cached));
  prm.flags = c.flags;
  prm.out = static_cast<__nv_bfloat16*>(c.out);
  prm.lse = c.lse;
  prm.err = device_error_word();
  const size_t usable_ws = (c.ws && !(reinterpret_cast<uintptr_t>(c.ws) & 15u)) ? c.ws_bytes : 0;
  AttnPlan pl;
  int st = attn_plan(c, usable_ws, 0, &pl);
  if (st) return st;
  prm.tiles_per_cta = pl.tiles_per_cta;
  prm.n_split = pl.n_split;
  prm.tiles_per_split = pl.per;
  prm.ws_o = nullptr;
  prm.ws_ml = nullptr;
  if (pl.n_split > 1) {
    prm.ws_o = static_cast<float*>(c.ws);
    prm.ws_ml = reinterpret_cast<float2*>(static_cast<char*>(c.ws) +
                                          static_cast<size_t>(pl.n_split) * c.B * c.Hq * c.M * D * 4);
  }
  prm.B = c.B;
  prm.tiles_x = pl.tiles_x;
  prm.n_unit_ctas = pl.n_unit_ctas;
  const bool persist = pl.kernel == kPlanPersistent;
  prm.n_lone = persist ? 2 * pl.tail : 0;
  // A programmatic dependent launch: its launch latency overlaps the previous
  // kernel on the stream, which every CTA waits for before its first read.
  // One query tile per CTA runs the one-tile kernel (S double buffered).
  cudaLaunchConfig_t lc = {};
  const bool rw = prm.rewrite != 0;
  // A refresh whose compute grid leaves SMs idle copies the cache there: up
  // to one copy CTA per idle SM, one warp per (sequence, KV head, prompt tile,
  // K or V) unit at most.
  prm.copy_ctas = 0;
  if (rw && !persist) {
    const int sms = sm_count();
    const long long units = static_cast<long long>(c.B) * c.Hkv * ((c.P + kBN - 1) / kBN) * 2;
    const long long want = (units + kThreadsRw / 32 - 1) / (kThreadsRw / 32);
    if (sms > pl.grid) prm.copy_ctas = static_cast<int>(std::min<long long>(sms - pl.grid, want));
  }
  lc.gridDim = dim3(static_cast<unsigned>(pl.grid + prm.copy_ctas));
  lc.stream = stream;
  cudaLaunchAttribute la[1];
  la[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  la[0].val.programmaticStreamSerializationAllowed = 1;
  lc.attrs = la;
  lc.numAttrs = 1;
  const CUtensorMap maps[8] = {mq, mkr, mvr, mkc, mvc, mkg, mvg, mo};
  st = rw ? launch_fwd_rewrite(D, pl.kernel, lc, maps, prm) : launch_fwd_plain(D, pl.kernel, lc, maps, prm);
  if (st || pl.n_split == 1) return st;
  // The merge is a programmatic dependent launch: it is scheduled while the
  // attention grid still runs and waits for it on the device.
  const long long threads = static_cast<long long>(c.B) * c.M * c.Hq * (D / 8);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>((threads + 255) / 256));
  cfg.blockDim = dim3(256);
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cuda_status(cudaLaunchKernelEx(&cfg, attn_combine_kernel<D>, static_cast<const float*>(prm.ws_o),
                                        static_cast<const float2*>(prm.ws_ml), pl.n_split, c.B, c.Hq, c.M, c.flags,
                                        c.default_refresh, c.q_begin_refresh, c.q_begin_cached, prm.out, prm.lse),
                     "attention combine launch");
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

size_t attn_workspace_bytes(int B, int P, int G, int Hq, int D, int M) {
  return split_plan(B, P, G, Hq, D, M, M, sm_count()).bytes;
}

int attn_plan(const AttnCall& c, size_t usable_ws, int sms, AttnPlan* pl) {
  *pl = AttnPlan{};
  if (sms <= 0) sms = sm_count();
  // Query tiles needed by the longest query range (a refreshed sequence's).
  const int rows = c.M - (c.flags || c.default_refresh ? c.q_begin_refresh : c.q_begin_cached);
  SplitPlan sp = split_plan(c.B, c.P, c.G, c.Hq, c.D, rows, c.M, sms);
  pl->split_bytes = sp.bytes;
  if (sp.n_split > 1 && usable_ws < sp.bytes) {
    sp.n_split = 1;                                 // no (usable) workspace: one CTA per tile pair
    sp.per = (c.P + kBN - 1) / kBN + (c.G + kBN - 1) / kBN;
  }
  pl->tiles_per_cta = sp.tiles_per_cta;
  pl->n_split = sp.n_split;
  pl->per = sp.per;
  const int rows_per_cta = sp.tiles_per_cta * kBM;
  pl->tiles_x = ((rows + rows_per_cta - 1) / rows_per_cta) * sp.n_split;
  const long long units = static_cast<long long>(pl->tiles_x) * c.Hq * c.B;
  if (units > 0x3FFFFFFFll) {
    set_error("too many attention work units (%lld)", units);
    return ARCHER_ERR_UNSUPPORTED;
  }
  pl->units = static_cast<int>(units);
  // A last wave of tile pairs at most half full runs as one wave of single
  // tiles instead: each of its SMs then finishes in about 0.7 of a pair's time.
  int tail = 0;
  if (sp.n_split == 1 && sp.tiles_per_cta == 2 && sms > 0 && units > sms) {
    const int r = static_cast<int>(units % sms);
    if (r > 0 && 2 * r <= sms) tail = r;
  }
  // The persistent two-tile kernel (one CTA per SM walking the items) when no
  // item is split or single: the query ranges in use are whole tile pairs,
  // and either no last wave would run as single tiles or every SM has three
  // items or more (measured: the 32-layer trajectory's 512 items, 3.4 per SM,
  // 93.3 -> 91.1 us against flat pairs with single-tile tails).
  bool persist = false;
  if (sp.tiles_per_cta == 2 && sp.n_split == 1 && sms > 0 && units > sms) {
    const bool uses_c = c.flags || !c.default_refresh, uses_r = c.flags || c.default_refresh;
    const bool whole = (!uses_c || (c.M - c.q_begin_cached) % (2 * kBM) == 0) &&
                       (!uses_r || (c.M - c.q_begin_refresh) % (2 * kBM) == 0);
    persist = whole && (tail == 0 || units >= 3LL * sms);
  }
  // A cached step's persistent walk, when its last wave is at most half full,
  // walks that wave as single tiles: CTA x < 2 tail takes one tile of item
  // units - tail + x / 2 after its items, on the one-tile kernel's schedule
  // (S double buffered: a lone tile's key step is about 0.56 of a pair's),
  // so that the busiest SMs take about half an item fewer.  Measured on the
  // 32-layer trajectory's cached step: 89.0 -> 85.2 us.  Refresh launches
  // walk their last wave in pairs: with the tail they measured slower
  // (trajectory refresh 253 -> 269 us, long-prompt refresh 2996 -> 3030 us).
  if (persist && (c.flags || c.default_refresh)) tail = 0;
  pl->tail = tail;
  pl->n_unit_ctas = static_cast<int>(units) - tail;
  pl->kernel = sp.tiles_per_cta == 1 ? kPlanOneTile : (persist ? kPlanPersistent : kPlanTwoTile);
  pl->grid = persist ? sms : static_cast<int>(units) + tail;
  return ARCHER_OK;
}

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

extern "C" int archer_debug_stall_attention(int on) {
  return archer::g_debug_stall.exchange(on ? 1 : 0, std::memory_order_relaxed);
}
