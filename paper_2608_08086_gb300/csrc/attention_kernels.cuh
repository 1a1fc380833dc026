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
// One CTA = two 128-row query tiles (A and B) of one (b, h) sharing every K/V
// tile; 10 warps:
//   warp 0     MMA issuer: lane 0 waits and issues alone.  Per K/V
//              tile j: PV_A(j), QK_A(j+1), PV_B(j), QK_B(j+1), so the tensor
//              pipe works on one tile while the other tile's softmax runs.  It
//              waits on two barriers (P_A(j), which also says that the pair
//              (V_j, K_{j+1}) has landed, and P_B(j)) and commits three times
//              per tile j: every wait or commit between two MMA batches idles
//              the tensor pipe.  tcgen05.mma executes in issue order, so QK_X(j+1)
//              overwrites S_X only after PV_X(j) has read P_X(j), and the
//              commit that announces S_X(j+1) also covers PV_X(j): when the
//              softmax sees S_X(j+1), O_X is stable and may be rescaled without
//              a wait.
//   warp 1     TMA producer: Q_A, Q_B once, then pairs (V_{u-1}, K_u) of
//              128-key tiles (u = 0 .. T; the first pair holds K_0 only, the
//              last V_{T-1} only) through two pair slots, one full barrier
//              per slot.  It waits for each pair to land itself and adds one
//              arrival to P_A of the key tile that reads it, and it takes a
//              slot as free from tile B's S barrier, whose commit after the
//              key tile that last read the slot covers those reads.
//   warps 2-9  softmax: one warpgroup per tile.  Warp w reaches TMEM lanes
//              32 (w % 4) .. 32 (w % 4) + 31, so lane i of warp w owns query
//              row 32 (w % 4) + i and all 128 key columns of its tile, read
//              from TMEM once per tile; exponentials use the running max in
//              use, raised lazily (only when the tile max exceeds it by more
//              than 2^8, rescaling l and O); P (bf16 pairs) is written over S
//              columns already read.  (Two warpgroups per tile, each with half
//              the columns and a shared-memory max exchange, measured 3 %
//              slower: the extra warps' waiting and exchange cost the MMA warp
//              more issue slots than the shorter rows saved.)
// TMEM (512 columns): S_A [0,128) S_B [128,256) O_A [256,256+D) O_B [384,384+D).
// Every hand-off is an mbarrier; every wait is bounded (archer_device.cuh).
//
// Launches whose grid would fill at most half the SMs take one query tile per
// CTA and run the one-tile instantiation (kSingle): the free TMEM columns
// double-buffer S (S(j) in [128 (j % 2), +128), O in [256, 256+D)), so the MMA
// warp computes S(j+2) while the softmax works on S(j+1) and the key step
// costs the longer of one tile's MMAs and one tile's softmax rather than their
// sum.  With one Q tile in shared memory there is room for three K/V pair
// slots.  The S barrier's commit after each P V also tells the softmax when O
// may be rescaled and, after the last one, that O is final.
//
// Two-tile launches with many CTAs' worth of work run attn_fwd_persist_kernel
// instead: one CTA per SM walks the work items, so the set-up happens once
// and the next item's Q tiles and first K/V pairs load while the current one
// finishes (its comment gives the barrier phases across items).
//
// This header holds the kernels and their parameters; attention_step.cu
// instantiates the kernels of launches without the cache rewrite,
// attention_rewrite.cu those with it (separate translation units, so that a
// change to one set leaves the other's code as it is), attention.cu the launch
// plan and the host side.
#pragma once

#include <atomic>
#include <cmath>

#include <cudaTypedefs.h>

#include "archer_device.cuh"
#include "archer_internal.h"
#include "tmem_ldst.cuh"

namespace archer {

constexpr int kBM = 128;          // query rows per tile (tcgen05 M)
constexpr int kBN = 128;          // keys per KV tile (N of Q K^T, K of P V)
constexpr int kThreads = 320;     // MMA warp + producer warp + 2 softmax warpgroups
constexpr int kThreadsRw = 352;   // + the copy warp of the kernels that rewrite the cache
constexpr int kWarpMma = 0, kWarpProducer = 1, kWarpSoftmax0 = 2, kWarpCopy = 10, kCopyWarps = 1;
constexpr uint32_t kTmemCols = 512;
// TMEM columns of tile t's S (P is written over its first 64 columns) and O.
__host__ __device__ constexpr uint32_t col_s(int t) { return 128u * static_cast<uint32_t>(t); }
__host__ __device__ constexpr uint32_t col_o(int t) { return 256u + 128u * static_cast<uint32_t>(t); }
constexpr uint32_t kChunkBytes = 128 * 128;   // 128 rows x 128 B (64 bf16) swizzle region

struct AttnParams {
  int P, G, Hq, Hkv, M;
  int q_begin_refresh, q_begin_cached, default_refresh;
  float scale_log2;           // softmax_scale * log2(e)
  long long wait_limit;       // SM clocks a bounded wait may take
  int debug_skip_last_pv;     // test hook: withhold the last PV and its commits
  // Fused cache rewrite (C_r <- C_p(g_t) of Algorithm 1): bit 0 copies K, bit
  // 1 V, from the fresh prompt tensors to the cache, for refreshed sequences.
  // The kernels built for it have an extra copy warp (see copy_prompt_share).
  int rewrite;
  int copy_ctas;              // > 0: the grid's last copy_ctas CTAs do the whole copy (idle SMs)
  const uint4* kp_src;        // [B, P, Hkv, D] fresh prompt K / V (16-byte words)
  const uint4* vp_src;
  uint4* kp_dst;              // the cache
  uint4* vp_dst;
  const uint8_t* flags;
  __nv_bfloat16* out;
  float* lse;
  int* err;
  // Split over the key tiles (grids smaller than the SM count): CTA x of a
  // launch is (query tile pair x / n_split, split x % n_split); split s takes
  // key tiles [s * tiles_per_split, (s + 1) * tiles_per_split) of the T tiles
  // and writes its unnormalised O, running max and row sum to the workspace
  // instead of out; attn_combine_kernel merges the splits.
  int n_split, tiles_per_split;
  int tiles_per_cta;          // query tiles per CTA: 2 (ping-pong), or 1 for grids far below the SM count
  // Flat grid: CTA x < n_unit_ctas is unit x, units numbered (tile pair x
  // split) fastest, then head, then sequence; the CTAs after them each take one
  // tile of the last n_tail_pairs tile pairs (a nearly empty last wave of pairs
  // becomes one wave of single tiles).
  int B, tiles_x, n_unit_ctas;
  float* ws_o;                // [n_split, B, Hq, M, D] fp32
  float2* ws_ml;              // [n_split, B, Hq, M] (max in log2 units, row sum)
  // Persistent kernel: it walks items 0 .. n_unit_ctas - 1 in pairs; with
  // n_lone > 0 the items after them run as n_lone single query tiles, CTA x <
  // n_lone taking tile x mod 2 of item n_unit_ctas + x / 2 after its items.
  int n_lone;
};

// kSingle: the one-tile kernel (one Q tile, three pair slots, S double
// buffered in TMEM).
template <int D, bool kSingle = false>
struct Layout {
  static constexpr int kChunks = D / 64;                    // 128-byte column chunks
  static constexpr uint32_t kTile = kChunks * kChunkBytes;  // one 128-row tile of D bf16
  static constexpr int kSlots = kSingle ? 3 : 2;            // pair slots: [V tile | K tile]
  static constexpr uint32_t kOffQ = 0;                      // Q_A, Q_B (Q only when kSingle)
  static constexpr uint32_t kOffKV = kOffQ + (kSingle ? 1 : 2) * kTile;
  static constexpr uint32_t kOffBar = kOffKV + kSlots * 2 * kTile;
  // q_full, full[slots], s_full[2], p_full[2] (a pair slot is known free from
  // the S barrier whose commit covers the pair's last reader)
  static constexpr int kBars = 1 + kSlots + 4;
  static constexpr uint32_t kOffHolder = kOffBar + 8 * kBars;
  static constexpr uint32_t kOffAbort = kOffHolder + 4;
  static constexpr uint32_t kOffDrain = kOffAbort + 4;        // abort path: the MMA warp's MMAs done
  static constexpr uint32_t kUsed = kOffDrain + 8;
  // + 1 KB to align the base to 1024 B; at least 120 KB so that one CTA
  // holds an SM (the CTA allocates all 512 TMEM columns).
  static constexpr uint32_t kSmemBytes = (kUsed + 1024 > 120 * 1024) ? kUsed + 1024 : 120 * 1024;
  static_assert(kUsed + 1024 <= 232448, "shared memory budget");
};

// Launches attn_fwd_kernel / attn_fwd_persist_kernel (kind = kPlanTwoTile,
// kPlanOneTile or kPlanPersistent) for head_dim D with the tensor maps
// m = {Q, K_p refresh, V_p refresh, K_p cached, V_p cached, K_g, V_g, out}; lc
// carries the grid, stream and attributes (block size and shared memory are
// set here).  Without the fused cache rewrite: attention_step.cu; with it:
// attention_rewrite.cu.
int launch_fwd_plain(int D, int kind, cudaLaunchConfig_t lc, const CUtensorMap* m, const AttnParams& prm);
int launch_fwd_rewrite(int D, int kind, cudaLaunchConfig_t lc, const CUtensorMap* m, const AttnParams& prm);

namespace {

// Warp-uniform wait bounded by the clock alone (the abort flag is already
// set when it runs): lets in-flight MMAs and copies land before the CTA frees
// TMEM or exits.  Returns whether the phase completed.
__device__ __forceinline__ bool drain_wait(uint32_t bar, uint32_t parity, long long limit) {
  const long long t0 = clock64();
  while (!__all_sync(0xffffffffu, mbar_try_wait(bar, parity)))
    if (__any_sync(0xffffffffu, clock64() - t0 > limit)) return false;
  return true;
}

// Warp-uniform bounded wait for the softmax warps (tcgen05.ld/st are
// .sync.aligned, so all 32 lanes must take the same path).
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, volatile int* abort,
                                          int* err, long long limit) {
  // The first poll reads no clock: an already complete phase costs one
  // try_wait and one vote.
  if (__all_sync(0xffffffffu, mbar_try_wait(bar, parity))) return true;
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

// v, as a value the compiler cannot see through: what is computed from it is
// recomputed there, not kept alive from an earlier computation of the same.
// A descriptor the compiler cannot see through: the MMA-issuing thread starts
// each batch from an opaque copy of its base descriptor, placed after the
// wait that precedes the batch, and steps to the next MMA's operand with one
// add after each MMA.  Otherwise the compiler computes a key step's
// descriptors ahead of that wait, on the issuing warp's critical path (the
// warp shares its SM sub-partition with two softmax warps, so every
// instruction there costs several cycles), instead of between MMAs, where
// they overlap the tensor core's work.
__device__ __forceinline__ uint64_t opaque_desc(uint64_t v) {
  uint64_t r;
  asm volatile("mov.b64 %0, %1;" : "=l"(r) : "l"(v));
  return r;
}
__device__ __forceinline__ int opaque_int(int v) {
  asm volatile("" : "+r"(v));
  return v;
}

__device__ __forceinline__ float max3f(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

__device__ __forceinline__ float max128(const float (&x)[128]) {
  float m[4] = {x[0], x[1], x[2], x[3]};
#pragma unroll
  for (int c = 4; c < 128; c += 2) m[(c >> 1) & 3] = max3f(m[(c >> 1) & 3], x[c], x[c + 1]);
  return max3f(m[0], m[1], fmaxf(m[2], m[3]));
}

// Loads this lane's 128 score columns and masks keys >= valid.
__device__ __forceinline__ void load_scores128(uint32_t taddr, int valid, float (&x)[128]) {
  uint32_t r[128];
  tmem_ld_128(taddr, r);
#pragma unroll
  for (int c = 0; c < 128; ++c) x[c] = __uint_as_float(r[c]);
  if (valid < 128) {                // only the last tile of a segment is ragged
#pragma unroll
    for (int c = 0; c < 128; ++c)
      if (c >= valid) x[c] = -INFINITY;
  }
}

// Fused cache rewrite: one unit = prompt tile `tile` (up to 128 rows of D
// bf16) of K or V of (sequence b, KV head kvh), copied global -> registers ->
// global by n_lanes threads (lane = 0 .. n_lanes - 1), 16 bytes per access,
// kCopyUnroll accesses in flight per thread.  Reads no shared memory (the
// tensor cores' operands use its bandwidth) and waits on no other thread.
constexpr int kCopyUnroll = 16;
template <int D>
__device__ __forceinline__ void copy_prompt_unit(const AttnParams& p, int b, int kvh, int tile, bool is_v, int lane,
                                                 int n_lanes) {
  constexpr int kRowWords = D * 2 / 16;
  if (!(p.rewrite & (is_v ? 2 : 1))) return;
  const uint4* src = is_v ? p.vp_src : p.kp_src;
  uint4* dst = is_v ? p.vp_dst : p.kp_dst;
  const int r0 = tile * kBN;
  const int words = min(kBN, p.P - r0) * kRowWords;
  // word w of the unit: row r0 + w / kRowWords, 16-byte column w % kRowWords
  const size_t base = (static_cast<size_t>(b) * p.P + r0) * p.Hkv + kvh;
  auto at = [&](int w) { return (base + static_cast<size_t>(w / kRowWords) * p.Hkv) * kRowWords + w % kRowWords; };
  for (int w0 = lane; w0 < words; w0 += n_lanes * kCopyUnroll) {
    uint4 v[kCopyUnroll];
#pragma unroll
    for (int i = 0; i < kCopyUnroll; ++i)
      if (w0 + n_lanes * i < words) v[i] = __ldg(src + at(w0 + n_lanes * i));
#pragma unroll
    for (int i = 0; i < kCopyUnroll; ++i)
      if (w0 + n_lanes * i < words) dst[at(w0 + n_lanes * i)] = v[i];
  }
}

// The copy warps of a refresh with the fused cache rewrite.  The work items
// that load the key tiles of one (sequence b, KV head kvh) -- the Hq / Hkv
// query heads of the group times the query-tile items of each, `n_writers` in
// all, this one `writer` -- share the copy: the prompt tiles t_lo .. t_hi - 1
// make 2 (t_hi - t_lo) units (tile, K or V), and unit i goes to writer
// i mod n_writers, copied by the CTA's kCopyWarps copy warps together.
template <int D>
__device__ __forceinline__ void copy_prompt_share(const AttnParams& p, int b, int kvh, int t_lo, int t_hi, int writer,
                                                  int n_writers) {
  const int lane = threadIdx.x - 32 * kWarpCopy;
  for (int unit = writer; unit < 2 * (t_hi - t_lo); unit += n_writers)
    copy_prompt_unit<D>(p, b, kvh, t_lo + (unit >> 1), unit & 1, lane, 32 * kCopyWarps);
}

// The copy CTAs of a refresh whose compute grid leaves SMs idle: every unit
// (sequence, KV head, prompt tile, K or V) of the refreshed sequences, one
// warp per unit, units dealt round-robin over the copy CTAs' warps.
template <int D>
__device__ __forceinline__ void copy_prompt_all(const AttnParams& p, int cta, int n_ctas) {
  constexpr int kWarps = kThreadsRw / 32;
  const int n_p = (p.P + kBN - 1) / kBN;
  const long long units = static_cast<long long>(p.B) * p.Hkv * n_p * 2;
  for (long long u = static_cast<long long>(cta) * kWarps + (threadIdx.x >> 5); u < units;
       u += static_cast<long long>(n_ctas) * kWarps) {
    const int is_v = static_cast<int>(u & 1);
    const long long t = u >> 1;                       // (b, kvh, tile), tile fastest
    const int tile = static_cast<int>(t % n_p);
    const int kvh = static_cast<int>((t / n_p) % p.Hkv);
    const int b = static_cast<int>(t / (static_cast<long long>(n_p) * p.Hkv));
    const bool refresh = p.flags ? (p.flags[b] != 0) : (p.default_refresh != 0);
    if (refresh) copy_prompt_unit<D>(p, b, kvh, tile, is_v, threadIdx.x & 31, 32);
  }
}

// The output epilogue: O (fp32 in TMEM, this thread's row r of the tile),
// scaled by inv_l, rounded to bf16 and written into shared memory at `stage`
// in the 128-byte-swizzled layout of the output tensor map (64-column chunks
// of kChunkBytes; row r's 16-byte unit u at (u ^ (r mod 8)) * 16 of its
// 128-byte row), for one TMA store of the tile.  Rows 16 bytes apart in the
// banks for every 8 consecutive rows: no bank conflicts.
template <int D>
__device__ __forceinline__ void stage_o_row(uint32_t t_lane_o, uint32_t stage, int r, float inv_l) {
#pragma unroll
  for (int c0 = 0; c0 < D; c0 += 32) {
    uint32_t o[32];
    tmem_ld_32(t_lane_o + c0, o);
    const uint32_t row = stage + (c0 / 64) * kChunkBytes + static_cast<uint32_t>(r) * 128u;
#pragma unroll
    for (int v = 0; v < 4; ++v) {
      const uint32_t unit = static_cast<uint32_t>((c0 % 64) / 8 + v) ^ static_cast<uint32_t>(r & 7);
      const uint32_t w0 = pack_bf16x2(__uint_as_float(o[8 * v]) * inv_l, __uint_as_float(o[8 * v + 1]) * inv_l);
      const uint32_t w1 = pack_bf16x2(__uint_as_float(o[8 * v + 2]) * inv_l, __uint_as_float(o[8 * v + 3]) * inv_l);
      const uint32_t w2 = pack_bf16x2(__uint_as_float(o[8 * v + 4]) * inv_l, __uint_as_float(o[8 * v + 5]) * inv_l);
      const uint32_t w3 = pack_bf16x2(__uint_as_float(o[8 * v + 6]) * inv_l, __uint_as_float(o[8 * v + 7]) * inv_l);
      asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(row + unit * 16u), "r"(w0), "r"(w1), "r"(w2),
                   "r"(w3)
                   : "memory");
    }
  }
}

// The tile's warpgroup (128 threads, named barrier bar_id) has staged its
// rows: one thread stores the 128 x D tile to rows q0 .. q0 + 127 of head h of
// sequence b (rows past the tensor's end are not written) and waits until the
// store has read shared memory (and, with `complete`, until it is done).
template <int D>
__device__ __forceinline__ void store_o_tile(const CUtensorMap* map, uint32_t stage, uint32_t bar_id, bool issuer,
                                             bool write, int h, int q0, int b, bool complete) {
  fence_proxy_async_smem();
  named_barrier(bar_id, kBM);
  if (issuer) {
    if (write) {
#pragma unroll
      for (int c = 0; c < D / 64; ++c) tma_store_4d(map, stage + c * kChunkBytes, c * 64, h, q0, b);
    }
    bulk_commit_group();
    if (complete) bulk_wait_group_all();
    else bulk_wait_group_read<0>();
  }
}

template <int D, bool kSingle, bool kRewrite>
__global__ void __launch_bounds__(kRewrite ? kThreadsRw : kThreads, 1)
attn_fwd_kernel(const __grid_constant__ CUtensorMap tmQ,
                const __grid_constant__ CUtensorMap tmKpR, const __grid_constant__ CUtensorMap tmVpR,
                const __grid_constant__ CUtensorMap tmKpC, const __grid_constant__ CUtensorMap tmVpC,
                const __grid_constant__ CUtensorMap tmKg, const __grid_constant__ CUtensorMap tmVg,
                const __grid_constant__ CUtensorMap tmO, const AttnParams p) {
  using L = Layout<D, kSingle>;
  if constexpr (kRewrite) {
    if (p.copy_ctas > 0 && static_cast<int>(blockIdx.x) >= static_cast<int>(gridDim.x) - p.copy_ctas) {
      asm volatile("griddepcontrol.wait;" ::: "memory");     // the flags and prompt K/V are written
      asm volatile("griddepcontrol.launch_dependents;");
      copy_prompt_all<D>(p, blockIdx.x - (gridDim.x - p.copy_ctas), p.copy_ctas);
      return;
    }
  }
  // pair u lives in slot u mod kSlots, that slot's use u div kSlots
  auto slot_of = [](int u) { return L::kSlots == 2 ? (u & 1) : (u % L::kSlots); };
  auto use_of = [](int u) { return L::kSlots == 2 ? (u >> 1) : (u / L::kSlots); };
  extern __shared__ uint8_t smem_raw[];

  int unit = blockIdx.x, tile_off = 0;
  const bool tail_single = unit >= p.n_unit_ctas;
  if (tail_single) {                      // one tile of a tail pair (no splits here)
    tile_off = (unit - p.n_unit_ctas) & 1;
    unit = p.n_unit_ctas + ((unit - p.n_unit_ctas) >> 1);
  }
  const int tpx = unit % p.tiles_x;
  const int h = (unit / p.tiles_x) % p.Hq, b = unit / (p.tiles_x * p.Hq);
  const int tp = tpx / p.n_split, split = tpx % p.n_split;
  // Launched as a programmatic dependent of the stream's previous kernel: wait
  // for it before reading anything it may have written (flags, Q/K/V).  With
  // no flags to read, the wait is deferred to just before the first load (and
  // taken by every thread after the set-up barrier), so the barrier set-up
  // and TMEM allocation overlap the previous kernel's tail.
  if (p.flags) asm volatile("griddepcontrol.wait;" ::: "memory");
  // Lets a programmatic dependent (the split merge, the next layer) be
  // scheduled once every CTA of this grid is resident; it still waits for
  // this grid's completion.
  asm volatile("griddepcontrol.launch_dependents;");
  const bool refresh = p.flags ? (p.flags[b] != 0) : (p.default_refresh != 0);
  const int q0 = (refresh ? p.q_begin_refresh : p.q_begin_cached) + (tp * p.tiles_per_cta + tile_off) * kBM;
  if (q0 >= p.M) return;  // uniform over the CTA, before any barrier or TMEM use
  const bool has_b = !tail_single && p.tiles_per_cta == 2 && q0 + kBM < p.M;

  const int kvh = h / (p.Hq / p.Hkv);
  const int n_p = (p.P + kBN - 1) / kBN;
  const int n_g = (p.G + kBN - 1) / kBN;
  const int j0 = split * p.tiles_per_split;                        // this CTA's first key tile
  const int T = min(n_p + n_g, j0 + p.tiles_per_split) - j0;      // and its number of tiles
  if (T <= 0) return;      // the host sizes splits so that none is empty; uniform anyway
  const bool partial = p.n_split > 1;

  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (base - raw);
  const uint32_t sQ = base + L::kOffQ;
  const uint32_t sKV = base + L::kOffKV;
  const uint32_t bars = base + L::kOffBar;
  const uint32_t bar_q_full = bars;
  const uint32_t bar_full = bars + 8;                           // + 8 * slot
  // S ready / P written, + 8 * tile (A = 0, B = 1); the one-tile kernel: + 8 * S buffer.
  // P_A (and the one-tile kernel's P) also count the producer's "pair landed".
  const uint32_t bar_s_full = bar_full + 8 * L::kSlots;
  const uint32_t bar_p_full = bar_s_full + 16;
  const uint32_t bar_drain = base + L::kOffDrain;
  uint32_t* holder = reinterpret_cast<uint32_t*>(gbase + L::kOffHolder);
  volatile int* abort = reinterpret_cast<volatile int*>(gbase + L::kOffAbort);

  const int warp = threadIdx.x >> 5;
  const bool lane0 = (threadIdx.x & 31) == 0;
  const CUtensorMap* mKp = refresh ? &tmKpR : &tmKpC;
  const CUtensorMap* mVp = refresh ? &tmVpR : &tmVpC;
  // Producer lane 0: pair u = (V_{u-1}, K_u) into its pair slot, [V tile | K tile].
  auto issue_pair = [&](int u) {
    const int slot = slot_of(u);
    const bool has_v = u >= 1, has_k = u < T;
    mbar_arrive_expect_tx(bar_full + 8 * slot, (has_v && has_k ? 2 : 1) * L::kTile);
    for (int part = has_v ? 0 : 1; part < (has_k ? 2 : 1); ++part) {
      const int j = j0 + (part == 0 ? u - 1 : u);             // global key tile
      const bool in_prompt = j < n_p;
      const int row = in_prompt ? j * kBN : (j - n_p) * kBN;
      const CUtensorMap* map = in_prompt ? (part == 0 ? mVp : mKp) : (part == 0 ? &tmVg : &tmKg);
      const uint32_t dst = sKV + (2 * slot + part) * L::kTile;
      for (int c = 0; c < L::kChunks; ++c)
        tma_load_4d(dst + c * kChunkBytes, map, bar_full + 8 * slot, c * 64, kvh, row, b);
    }
  };
  // The producer's lane 0 sets up the barriers and issues the Q tiles and
  // the pairs whose slots start free before the CTA-wide barrier, so those
  // loads overlap the TMEM allocation and the barrier itself.
  const int u_pre = min(L::kSlots, T + 1);
  if (warp == kWarpProducer && lane0) {
    mbar_init(bar_q_full, 1);
    for (int s = 0; s < L::kSlots; ++s) {
      mbar_init(bar_full + 8 * s, 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(bar_s_full + 8 * i, 1);
      mbar_init(bar_p_full + 8 * i, (kSingle || i == 0) ? kBM + 1 : kBM);   // + the producer's arrival
    }
    *abort = 0;
    mbar_fence_init();
    if (!p.flags) asm volatile("griddepcontrol.wait;" ::: "memory");
    tma_prefetch_map(&tmQ);
    mbar_arrive_expect_tx(bar_q_full, has_b ? 2 * L::kTile : L::kTile);
    for (int t = 0; t < (has_b ? 2 : 1); ++t)
      for (int c = 0; c < L::kChunks; ++c)
        tma_load_4d(sQ + t * L::kTile + c * kChunkBytes, &tmQ, bar_q_full, c * 64, h, q0 + t * kBM, b);
    for (int u = 0; u < u_pre; ++u) issue_pair(u);
  }
  if (warp == kWarpMma) {
    tmem_alloc(smem_u32(holder), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (!p.flags) asm volatile("griddepcontrol.wait;" ::: "memory");
  const uint32_t tmem = *holder;

  int last_pair = -1;          // producer: the last pair whose loads were issued
  bool mma_done = false;       // MMA warp: every MMA issued and committed to the S barriers
  if (warp == kWarpProducer) {
    // ------------------------------------------------------------ producer
    // The whole warp runs the loop and waits (warp-uniform); lane 0 issues.

    // Two-tile kernel: the MMA warp's wait for P_A(j) also covers "pair j+1
    // has landed" (the barrier counts kBM + 1 arrivals): once that pair has
    // landed and phase j-1 is over, so that this arrival cannot count towards
    // it, the producer adds its arrival to phase j.  The MMA warp then waits
    // once less per key tile.
    // In the loop, the slot poll just before (tile B's S commit of key step
    // v-2) already implies that phase v-2 is over; only the last arrival,
    // after the loop, waits for it explicitly.
    auto landed = [&](int v, bool wait_prev) {  // pair v landed -> phase v-1 of P_A
      if (!warp_wait(bar_full + 8 * slot_of(v), static_cast<uint32_t>(use_of(v)) & 1u, abort, p.err,
                     p.wait_limit))
        return false;
      if (wait_prev && v >= 2 &&
          !warp_wait(bar_p_full, static_cast<uint32_t>(v - 2) & 1u, abort, p.err, p.wait_limit))
        return false;
      if (lane0) mbar_arrive(bar_p_full);
      __syncwarp();
      return true;
    };
    // One-tile kernel: the same for P(j) (buffer j % 2) and pair min(j+2, T),
    // the pair the MMA warp reads next (K_{j+2}; for the last tiles V_{T-1}),
    // once the buffer's previous phase (tile j-2) is over.
    int next_j = 0;
    auto landed1 = [&](int j) {
      const int v = min(j + 2, T);
      if (!warp_wait(bar_full + 8 * slot_of(v), static_cast<uint32_t>(use_of(v)) & 1u, abort, p.err,
                     p.wait_limit))
        return false;
      if (j >= 2 &&
          !warp_wait(bar_p_full + 8 * (j & 1), static_cast<uint32_t>((j - 2) >> 1) & 1u, abort, p.err, p.wait_limit))
        return false;
      if (lane0) mbar_arrive(bar_p_full + 8 * (j & 1));
      __syncwarp();
      return true;
    };
    int u = u_pre;
    bool ok = true;
    for (; u <= T; ++u) {
      const int use = use_of(u);
      if constexpr (!kSingle) {
        // Slot of pair u free: its previous pair u-2 was read by the MMAs of
        // key step u-3 (or the prologue), which the last tile's S commit of
        // that step covers (completion u-2).  Polled before the arrival that
        // lets key step u-2 start, so that barrier cannot be two phases ahead.
        if (!warp_wait(bar_s_full + 8 * (has_b ? 1 : 0), static_cast<uint32_t>(u - 2) & 1u, abort, p.err,
                       p.wait_limit))
          break;
        if (!(ok = landed(u - 1, false))) break;   // u >= 2: pairs 0 .. u-1 are issued
      } else {
        // S(0) announced (buffer 0's first completion), polled before the
        // arrival that lets key step 0 complete that buffer again: the poll
        // for pair 4 below then waits on the completion right after one this
        // warp has seen, so its parity cannot alias.
        if (u == 3 && !(ok = warp_wait(bar_s_full, 0u, abort, p.err, p.wait_limit))) break;
        while (ok && next_j < T && min(next_j + 2, T) <= u - 1) ok = landed1(next_j++);
        if (!ok) break;
        // Slot of pair u free: its previous pair u-3 was last read by P V of
        // key step u-4 (or, for pair 0, by the prologue), which the commit
        // announcing S(u-2) covers.  S(u) needs this very pair, so that
        // buffer's barrier cannot be two phases ahead.
        if (use > 0 && !warp_wait(bar_s_full + 8 * ((u - 2) & 1), static_cast<uint32_t>((u - 2) >> 1) & 1u, abort,
                                  p.err, p.wait_limit))
          break;
      }
      if (lane0) issue_pair(u);
      __syncwarp();
    }
    last_pair = u - 1;         // the loop breaks before issuing pair u
    if (ok && u == T + 1) {                     // every pair is issued: the arrivals left
      if constexpr (!kSingle) landed(T, true);
      else
        while (ok && next_j < T) ok = landed1(next_j++);
    }
  } else if (warp >= kWarpCopy) {        // present only in the kRewrite kernels (11 warps)
    // ------------------------------------------------------------ cache copy
    // Items of one (sequence, KV head): the group's query heads times the
    // query-tile items of each (every key split copies its own tiles).
    if constexpr (kRewrite) {
      if (refresh && tile_off == 0 && p.copy_ctas == 0) {
        const int per_head = p.tiles_x / p.n_split;
        copy_prompt_share<D>(p, b, kvh, j0, min(j0 + T, n_p), (h % (p.Hq / p.Hkv)) * per_head + tp,
                             (p.Hq / p.Hkv) * per_head);
      }
    }
  } else if (warp == kWarpMma) {
    // ------------------------------------------------------------ MMA issuer
    // Lane 0 runs the schedule alone: its waits are single-thread bounded
    // waits, and it issues every MMA and commit (measured a little faster
    // than the whole warp waiting together and reconverging after each
    // batch).
    constexpr uint32_t idesc_qk = idesc_bf16_f32(kBM, kBN, 0, 0);
    constexpr uint32_t idesc_pv = idesc_bf16_f32(kBM, D, 0, 1);
    const int n_tiles = has_b ? 2 : 1;
    // Operand descriptors built once (Q tile 0; the K and V halves of pair
    // slot 0); an MMA's own descriptor is one of these plus its offset
    // (desc_add), so a key step's MMAs cost few instructions.
    const uint64_t qd0 = sdesc_sw128(sQ, 16, 1024);
    const uint64_t kd0 = sdesc_sw128(sKV + L::kTile, 16, 1024), vd0 = sdesc_sw128(sKV, kChunkBytes, 1024);
    auto issue_qk = [&](int t, uint64_t kd) {
      const uint64_t qd = desc_add(qd0, t * L::kTile);
#pragma unroll
      for (int kk = 0; kk < D / 16; ++kk) {
        const uint32_t off = (kk >> 2) * kChunkBytes + (kk & 3) * 32;
        umma_ss(tmem + col_s(t), desc_add(qd, off), desc_add(kd, off), idesc_qk, kk > 0 ? 1u : 0u);
      }
    };
    // P V over the tile's 128 keys (8 MMAs of K = 16); P of keys
    // [64 h, 64 h + 64) lives in S columns [64 h, 64 h + 32).
    auto issue_pv = [&](int t, uint64_t vd, bool acc) {
#pragma unroll
      for (int kk = 0; kk < 8; ++kk)
        umma_ts(tmem + col_o(t), tmem + col_s(t) + 64 * (kk >> 2) + (kk & 3) * 8, desc_add(vd, kk * 2048), idesc_pv,
                (acc || kk > 0) ? 1u : 0u);
    };
    auto v_tile_of = [&](int u) { return desc_add(vd0, slot_of(u) * 2 * L::kTile); };
    auto k_tile_of = [&](int u) { return desc_add(kd0, slot_of(u) * 2 * L::kTile); };
    auto phase_of = [&](int u) { return static_cast<uint32_t>(use_of(u)) & 1u; };
    if constexpr (kSingle) {
      // One query tile, S double buffered: S(j) in buffer j & 1 (columns
      // col_s(j & 1), P(j) written over it), O in col_o(0).  Per key tile j:
      // wait P(j) (with the producer's arrival it also says that pair
      // min(j + 2, T) has landed); O += P(j) V_j; S(j + 2) = Q K_{j+2}^T into
      // the buffer P(j) came from (issue order: P V reads P(j) first); one
      // commit.  That commit also covers P V of tile j, so it tells the
      // producer that pair j + 1 is read and, when no S(j + 2) is left (it is
      // issued all the same), says only "O holds P V up to tile j" (the last
      // one: O final).  The softmax of tile j + 1 runs meanwhile on the other
      // buffer, so the key step is the longer of one tile's MMAs and one
      // tile's softmax instead of their sum.
      auto issue_qk1 = [&](int bf, uint64_t kd) {
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t off = (kk >> 2) * kChunkBytes + (kk & 3) * 32;
          umma_ss(tmem + col_s(bf), desc_add(qd0, off), desc_add(kd, off), idesc_qk, kk > 0 ? 1u : 0u);
        }
      };
      auto issue_pv1 = [&](int bf, uint64_t vd, bool acc) {
#pragma unroll
        for (int kk = 0; kk < 8; ++kk)
          umma_ts(tmem + col_o(0), tmem + col_s(bf) + 64 * (kk >> 2) + (kk & 3) * 8, desc_add(vd, kk * 2048),
                  idesc_pv, (acc || kk > 0) ? 1u : 0u);
      };
      // pairs 0 (K_0) and 1 (V_0, K_1): S(0) and S(1).  Lane 0 alone runs
      // the schedule (single-thread bounded waits); the other lanes wait for
      // it at the end.
      bool ok = true;
      int j = 0;
      if (lane0) {
        ok = mbar_wait(bar_q_full, 0, abort, p.err, p.wait_limit) &&
             mbar_wait(bar_full, phase_of(0), abort, p.err, p.wait_limit);
        if (ok) {
          tc_fence_after();
          issue_qk1(0, k_tile_of(0));
          umma_commit(bar_s_full);
          ok = mbar_wait(bar_full + 8 * slot_of(1), phase_of(1), abort, p.err, p.wait_limit);
        }
        if (ok && T > 1) {
          tc_fence_after();
          issue_qk1(1, k_tile_of(1));
          umma_commit(bar_s_full + 8);
        }
        for (; ok && j < T; ++j) {
          const int u = j + 1;                // pair (V_j, K_{j+1})
          const bool more2 = j + 2 < T;       // S(j + 2) to compute
          // P(j) also says pair min(j + 2, T) has landed (the producer's arrival)
          if (!mbar_wait(bar_p_full + 8 * (j & 1), static_cast<uint32_t>(j >> 1) & 1u, abort, p.err, p.wait_limit)) {
            ok = false;
            break;
          }
          if (p.debug_skip_last_pv && j + 1 == T) { ok = false; break; }   // the softmax's final wait must expire
          tc_fence_after();
          issue_pv1(j & 1, v_tile_of(u), j > 0);
          if (more2) issue_qk1(j & 1, k_tile_of(u + 1));
          umma_commit(bar_s_full + 8 * (j & 1));   // S(j + 2), or only "P V of tile j done"
        }
      }
      __syncwarp();
      mma_done = __shfl_sync(0xffffffffu, (ok && j == T) ? 1 : 0, 0) != 0;
    } else {
      // Lane 0 alone runs the schedule (single-thread bounded waits); the
      // other lanes wait for it at the end.
      bool ok = true;
      int j = 0;
      if (lane0) {
        ok = mbar_wait(bar_q_full, 0, abort, p.err, p.wait_limit) &&
             mbar_wait(bar_full, phase_of(0), abort, p.err, p.wait_limit);
        if (ok) {
          tc_fence_after();
          for (int t = 0; t < n_tiles; ++t) {
            issue_qk(t, k_tile_of(0));
            umma_commit(bar_s_full + 8 * t);
          }
        }
        for (; ok && j < T; ++j) {
          const bool more = j + 1 < T;
          const int u = j + 1;                  // pair (V_j, K_{j+1}), landed: P_A(j) says so
          for (int t = 0; t < n_tiles; ++t) {
            if (!mbar_wait(bar_p_full + 8 * t, j & 1, abort, p.err, p.wait_limit)) { ok = false; break; }
            if (p.debug_skip_last_pv && !more) { ok = false; break; }   // the softmax's final wait must expire
            tc_fence_after();
            issue_pv(t, v_tile_of(u), j > 0);
            if (more) issue_qk(t, k_tile_of(u));
            umma_commit(bar_s_full + 8 * t);     // S_t(j+1) ready -- or, after the last tile, O_t final
          }
          if (!ok) break;
        }
      }
      __syncwarp();
      mma_done = __shfl_sync(0xffffffffu, (ok && j == T) ? 1 : 0, 0) != 0;
    }
  } else {
    // ------------------------------------------------------------ softmax
    const int t = (warp - kWarpSoftmax0) >> 2;                    // 0 = tile A, 1 = tile B
    if (t == 0 || has_b) {
      const int r = (warp & 3) * 32 + (threadIdx.x & 31);
      const uint32_t t_lane = tmem + (static_cast<uint32_t>((warp & 3) * 32) << 16);
      const uint32_t colS = col_s(t), colO = col_o(t);
      const uint32_t bar_s = bar_s_full + 8 * t;
      const uint32_t bar_ph = bar_p_full + 8 * t;
      const float sl2 = p.scale_log2;
      float m_used = -INFINITY;
      float2 l2 = make_float2(0.f, 0.f);
      // O *= a, 16 columns at a time (the row's scores stay in registers)
      auto rescale_o = [&](float a) {
#pragma unroll 1
        for (int c0 = 0; c0 < D; c0 += 16) {
          uint32_t o[16];
          tmem_ld_16(t_lane + colO + c0, o);
#pragma unroll
          for (int k = 0; k < 16; ++k) o[k] = __float_as_uint(__uint_as_float(o[k]) * a);
          tmem_st_16(t_lane + colO + c0, o);
        }
      };
      // An expired wait sets the abort flag; the warp then stops its key steps
      // (after a failed wait a parity poll of a later phase could pass on a
      // stale one, and an arrival on P without the producer's would drive
      // that barrier's pending count below zero) and goes to the epilogue
      // over stale TMEM (in bounds).
      bool failed = false;
      for (int j = 0; j < T; ++j) {
        // kSingle: S(j), P(j) in buffer j & 1 (its (j / 2)-th use)
        const uint32_t bar_sj = kSingle ? bar_s_full + 8 * (j & 1) : bar_s;
        const uint32_t bar_pj = kSingle ? bar_p_full + 8 * (j & 1) : bar_ph;
        const uint32_t col_sj = kSingle ? col_s(j & 1) : colS;
        if (!warp_wait(bar_sj, kSingle ? (j >> 1) & 1 : j & 1, abort, p.err, p.wait_limit)) {
          failed = true;
          break;
        }
        tc_fence_after();
        const int jg = j0 + j;
        const int valid = jg < n_p ? min(kBN, p.P - jg * kBN) : min(kBN, p.G - (jg - n_p) * kBN);
        // The row's 128 scores are read from TMEM once and kept in registers.
        float x[128];
        load_scores128(t_lane + col_sj, valid, x);
        const float tm = max128(x) * sl2;
        if (j == 0) {
          m_used = tm;
        } else if (__any_sync(0xffffffffu, tm > m_used + 8.0f)) {
          // O must hold P V up to tile j-1, complete: with two tiles S(j) was
          // announced after it; with one, S(j+1) is (its commit follows P V
          // of tile j-1; the barrier cannot be further ahead: S(j+3) needs
          // this P).
          if constexpr (kSingle)
            failed = !warp_wait(bar_s_full + 8 * ((j + 1) & 1), static_cast<uint32_t>((j + 1) >> 1) & 1u, abort,
                                p.err, p.wait_limit);
          const float m_new = fmaxf(m_used, tm);
          const float a = ex2_approx(m_used - m_new);
          m_used = m_new;
          l2.x *= a;
          l2.y *= a;
          rescale_o(a);
        }
        const float2 neg_m = make_float2(-m_used, -m_used);
        const float2 slv = make_float2(sl2, sl2);
        float2 acc[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          // P of keys [32q, 32q + 32) as bf16 pairs over S columns that were
          // already read: keys [64h, 64h + 64) go to columns [64h, 64h + 32),
          // the layout the MMA warp's P V reads; each store stays in flight
          // while the next chunk is computed.
          uint32_t pk[16];
#pragma unroll
          for (int k = 0; k < 16; ++k) {
            const float2 y = ffma2(make_float2(x[32 * q + 2 * k], x[32 * q + 2 * k + 1]), slv, neg_m);
            const float2 pr = make_float2(ex2_approx(y.x), ex2_approx(y.y));
            acc[k & 1] = fadd2(acc[k & 1], pr);
            pk[k] = pack_bf16x2(pr.x, pr.y);
          }
          tmem_st_16_async(t_lane + col_sj + 64 * (q >> 1) + 16 * (q & 1), pk);
        }
        tmem_wait_st();
        l2 = fadd2(l2, fadd2(acc[0], acc[1]));
        tc_fence_before();
        mbar_arrive(bar_pj);
        if (failed) break;                 // (the one-tile rescale wait expired)
      }
      bool ok = false;
      if (failed) {
      } else if constexpr (kSingle) {
        // O final: the commit after P V of tile T-1 (buffer (T+1) & 1, the
        // phase after S(T-1) on that buffer).
        ok = warp_wait(bar_s_full + 8 * ((T + 1) & 1), static_cast<uint32_t>((T + 1) >> 1) & 1u, abort, p.err,
                       p.wait_limit);
      } else {
        ok = warp_wait(bar_s, T & 1, abort, p.err, p.wait_limit);
      }
      tc_fence_after();
      const float l_sum = l2.x + l2.y;
      const int q = q0 + t * kBM + r;
      const bool live = ok && q < p.M;
      if (partial) {
        const size_t row = ((static_cast<size_t>(split) * p.B + b) * p.Hq + h) * p.M + q;
        float* orow_ws = p.ws_o + row * D;
#pragma unroll
        for (int c0 = 0; c0 < D; c0 += 32) {
          uint32_t o[32];
          tmem_ld_32(t_lane + colO + c0, o);
          if (live) {
            float4* dst = reinterpret_cast<float4*>(orow_ws + c0);
#pragma unroll
            for (int v = 0; v < 8; ++v)
              dst[v] = make_float4(__uint_as_float(o[4 * v]), __uint_as_float(o[4 * v + 1]),
                                   __uint_as_float(o[4 * v + 2]), __uint_as_float(o[4 * v + 3]));
          }
        }
        if (live) p.ws_ml[row] = make_float2(m_used, l_sum);
      } else {
        // The tile's Q region is free once O is final (its last reader, the
        // tile's last Q K^T, finished before): the bf16 tile is staged there
        // and written by one TMA store.
        stage_o_row<D>(t_lane + colO, sQ + t * L::kTile, r, 1.0f / l_sum);
        store_o_tile<D>(&tmO, sQ + t * L::kTile, 1u + t, threadIdx.x == 32 * (kWarpSoftmax0 + 4 * t), ok, h,
                        q0 + t * kBM, b, true);
        if (live && p.lse)
          p.lse[(static_cast<size_t>(b) * p.Hq + h) * p.M + q] = (m_used + log2f(l_sum)) * 0.69314718055994531f;
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  // After an expired wait no role may leave work in flight: the MMA warp
  // waits for its MMAs before TMEM is freed, and the producer for the loads
  // it issued before the CTA's shared memory is released (both bounded).
  const bool aborted = *abort != 0;
  if (warp == kWarpMma) {
    if (aborted || !mma_done) {
      if (lane0) {
        mbar_init(bar_drain, 1);
        mbar_fence_init();
        umma_commit(bar_drain);
      }
      __syncwarp();
      drain_wait(bar_drain, 0, p.wait_limit);
    }
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  } else if (warp == kWarpProducer && aborted) {
    drain_wait(bar_q_full, 0, p.wait_limit);
    for (int u = max(0, last_pair - (L::kSlots - 1)); u <= last_pair; ++u)
      drain_wait(bar_full + 8 * slot_of(u), static_cast<uint32_t>(use_of(u)) & 1u, p.wait_limit);
  }
}

// Persistent two-tile kernel: one CTA per SM walks work items x = blockIdx.x,
// blockIdx.x + gridDim.x, ... (a work item = two 128-query tiles of one
// (b, h), exactly as one CTA of the two-tile attn_fwd_kernel), so that the CTA's
// set-up happens once and the next item's Q tiles and first K/V pairs load
// while the current item finishes.  Barrier phases run on across items: with
// k the item's rank among this CTA's items and T key tiles per item, S_X and
// the K/V pairs share one running index k (T + 1) + u (the item's S commits:
// S(0) after the prologue, then one per key step; its pairs u = 0 .. T), and
// P_X completes k T + j times.  Two more barriers per tile: "O final"
// (committed after the item's last P V, with that step's S commit) and "O
// drained" (the tile's softmax warpgroup, after its epilogue has read O); the
// MMA warp waits for the latter before the next item's first P V.  Used for
// two-tile launches without splits whose items all hold two tiles.
// The persistent kernel's shared memory: the two-tile layout, then "O final"
// and "O drained" per tile and "staged" (40 bytes), the softmax warpgroups'
// stop decisions (16 bytes), the single-tile tail's barriers (64 bytes), then,
// 1024-byte aligned, the output staging buffer of one tile.
template <int D>
constexpr uint32_t kPersistStopOff = Layout<D, false>::kUsed + 40 + 8;   // 4 ints: stop decisions (tile, parity)
template <int D>
constexpr uint32_t kPersistLoneOff = kPersistStopOff<D> + 16;          // 8 barriers of the single-tile tail
template <int D>
constexpr uint32_t kPersistStageOff = (kPersistLoneOff<D> + 64 + 1023u) & ~1023u;
template <int D>
constexpr uint32_t kPersistSmemBytes = kPersistStageOff<D> + Layout<D, false>::kTile + 1024;
static_assert(kPersistSmemBytes<128> <= 232448 && kPersistSmemBytes<64> <= 232448, "shared memory budget");

template <int D, bool kRewrite, bool kLone>
__global__ void __launch_bounds__(kRewrite ? kThreadsRw : kThreads, 1)
attn_fwd_persist_kernel(const __grid_constant__ CUtensorMap tmQ,
                        const __grid_constant__ CUtensorMap tmKpR, const __grid_constant__ CUtensorMap tmVpR,
                        const __grid_constant__ CUtensorMap tmKpC, const __grid_constant__ CUtensorMap tmVpC,
                        const __grid_constant__ CUtensorMap tmKg, const __grid_constant__ CUtensorMap tmVg,
                        const __grid_constant__ CUtensorMap tmO, const AttnParams p) {
  using L = Layout<D, false>;
  static_assert(!(kRewrite && kLone), "the single-tile tail serves cached steps (no cache rewrite)");
  extern __shared__ uint8_t smem_raw[];
  if (p.flags) asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;");

  const int n_units = kLone ? p.n_unit_ctas : p.tiles_x * p.Hq * p.B;   // items walked in pairs
  const int n_p = (p.P + kBN - 1) / kBN;
  const int n_g = (p.G + kBN - 1) / kBN;
  const int T = n_p + n_g;                                       // key tiles per item (no splits)
  // Item x -> (b, h, first query row); q0 >= M: nothing to do for it.
  auto decode = [&](int x, int& b, int& h, bool& refresh) {
    const int tp = x % p.tiles_x;
    h = (x / p.tiles_x) % p.Hq;
    b = x / (p.tiles_x * p.Hq);
    refresh = p.flags ? (p.flags[b] != 0) : (p.default_refresh != 0);
    return (refresh ? p.q_begin_refresh : p.q_begin_cached) + tp * 2 * kBM;
  };

  // The loads an item starts with -- its two Q tiles and the K/V tiles of its
  // first two pairs (K_0; V_0, K_1) -- prefetched into L2 (a hint) two to five
  // key steps before the current item ends, the step staggered over the CTAs
  // (their items end together, so unstaggered prefetches arrive in one burst).
  // Without it the next item's Q and first pairs, loaded only once the current
  // item's last key steps are done, reach the SM after its last P V.
  auto prefetch_item = [&](int x) {
    if (x >= n_units) return;
    int b, h;
    bool refresh;
    const int q0 = decode(x, b, h, refresh);
    if (q0 >= p.M) return;
    const int kvh = h / (p.Hq / p.Hkv);
    for (int t = 0; t < 2; ++t)
      if (q0 + t * kBM < p.M)
        for (int c = 0; c < L::kChunks; ++c) tma_prefetch_4d(&tmQ, c * 64, h, q0 + t * kBM, b);
    for (int part = 0; part < 3; ++part) {             // K_0, V_0, K_1
      const int j = part == 2 ? 1 : 0;
      if (j >= T) break;
      const bool is_v = part == 1, in_prompt = j < n_p;
      const int row = in_prompt ? j * kBN : (j - n_p) * kBN;
      const CUtensorMap* map = in_prompt ? (is_v ? (refresh ? &tmVpR : &tmVpC) : (refresh ? &tmKpR : &tmKpC))
                                         : (is_v ? &tmVg : &tmKg);
      for (int c = 0; c < L::kChunks; ++c) tma_prefetch_4d(map, c * 64, kvh, row, b);
    }
  };

  // The CTA's single tail tile (kLone, blockIdx.x < n_lone): its first query
  // row (>= M: nothing to do), and the L2 prefetch of its Q tile, K_0, V_0, K_1.
  auto lone_q0 = [&](int& b, int& h, bool& refresh, int cta = static_cast<int>(blockIdx.x)) {
    return decode(n_units + cta / 2, b, h, refresh) + (cta & 1) * kBM;
  };
  auto prefetch_lone = [&]() {
    int b, h;
    bool refresh;
    const int q0 = lone_q0(b, h, refresh);
    if (q0 >= p.M) return;
    const int kvh = h / (p.Hq / p.Hkv);
    for (int c = 0; c < L::kChunks; ++c) tma_prefetch_4d(&tmQ, c * 64, h, q0, b);
    for (int part = 0; part < 3; ++part) {             // K_0, V_0, K_1
      const int j = part == 2 ? 1 : 0;
      if (j >= T) break;
      const bool is_v = part == 1, in_prompt = j < n_p;
      const int row = in_prompt ? j * kBN : (j - n_p) * kBN;
      const CUtensorMap* map = in_prompt ? (is_v ? (refresh ? &tmVpR : &tmVpC) : (refresh ? &tmKpR : &tmKpC))
                                         : (is_v ? &tmVg : &tmKg);
      for (int c = 0; c < L::kChunks; ++c) tma_prefetch_4d(map, c * 64, kvh, row, b);
    }
  };

  // A launch without refresh flags (a cached step) waits for the grid it
  // depends on only after its set-up.  Its loads all come after that wait;
  // an L2 prefetch is only a hint, and L2 stays coherent with whatever the
  // previous grid still writes (the first layer's inputs can be its
  // outputs).  So the producer lane prefetches the CTA's first item into L2
  // right away, while the previous launch ends: every launch of a step reads
  // a layer's K/V afresh from DRAM.
  if (!p.flags && threadIdx.x == 32 * kWarpProducer) prefetch_item(blockIdx.x);
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (base - raw);
  const uint32_t sQ = base + L::kOffQ;
  const uint32_t sKV = base + L::kOffKV;
  const uint32_t bars = base + L::kOffBar;
  const uint32_t bar_q_full = bars;
  const uint32_t bar_full = bars + 8;                            // + 8 * slot
  const uint32_t bar_s_full = bar_full + 8 * L::kSlots;          // + 8 * tile
  const uint32_t bar_p_full = bar_s_full + 16;                   // + 8 * tile; P_A also counts "pair landed"
  const uint32_t bar_drain = base + L::kOffDrain;
  const uint32_t bar_o_ready = bar_drain + 8;                    // + 8 * tile: O final for the item
  const uint32_t bar_o_free = bar_o_ready + 16;                  // + 8 * tile: O read by the epilogue
  // The output tile's staging buffer (the next item's Q is already loading
  // into the Q tiles when an item's epilogue runs), used by tile A and tile B
  // of every item in turn: use n = 2 k + t waits for completion n - 1 of
  // "staged" (the previous user's store has read it) and completes it once
  // its own store has.
  const uint32_t bar_staged = bar_o_free + 16;
  const uint32_t stage = base + kPersistStageOff<D>;
  // The single-tile tail (kLone): CTA x < n_lone, after its items, takes tile
  // x mod 2 of item n_units + x / 2 alone, on the one-tile kernel's schedule
  // with barriers of its own: Q, two pair slots (pair u = V_{u-2} and K_u in
  // slot u mod 2), one S barrier per S buffer (S(j) in TMEM buffer j mod 2 --
  // the S columns of tiles A and B -- committed after Q K_j^T; the commit
  // after key step j's P V announces S(j + 2) and says that P V is done), one
  // P barrier per S buffer (P(j) on barrier j mod 2: the warpgroup's 128
  // threads and the producer's "pair j + 2 landed"; a thread can read S(j + 1)
  // before P(j) is complete, never S(j + 2), so its arrivals never run two
  // steps ahead on one barrier) and O final.
  const uint32_t lone = base + kPersistLoneOff<D>;
  const uint32_t lq_full = lone, l_full = lone + 8, l_s = lone + 24, l_p = lone + 40, l_o = lone + 56;
  uint32_t* holder = reinterpret_cast<uint32_t*>(gbase + L::kOffHolder);
  volatile int* abort = reinterpret_cast<volatile int*>(gbase + L::kOffAbort);

  const int warp = threadIdx.x >> 5;
  const bool lane0 = (threadIdx.x & 31) == 0;
  auto slot_of = [](int g) { return g & 1; };
  auto phase_of = [](int g) { return static_cast<uint32_t>(g >> 1) & 1u; };
  if (warp == kWarpProducer && lane0) {
    mbar_init(bar_q_full, 2);                                    // the Q loads' arrival + the producer's gate
    for (int s = 0; s < L::kSlots; ++s) mbar_init(bar_full + 8 * s, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(bar_s_full + 8 * i, 1);
      mbar_init(bar_p_full + 8 * i, i == 0 ? kBM + 1 : kBM);
      mbar_init(bar_o_ready + 8 * i, 1);
      mbar_init(bar_o_free + 8 * i, kBM);
    }
    mbar_init(bar_staged, 1);
    if constexpr (kLone) {
      mbar_init(lq_full, 1);
      for (int i = 0; i < 2; ++i) {
        mbar_init(l_full + 8 * i, 1);
        mbar_init(l_s + 8 * i, 1);
        mbar_init(l_p + 8 * i, kBM + 1);
      }
      mbar_init(l_o, 1);
    }
    *abort = 0;
    mbar_fence_init();
  }
  if (warp == kWarpMma) {
    tmem_alloc(smem_u32(holder), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (!p.flags) asm volatile("griddepcontrol.wait;" ::: "memory");
  const uint32_t tmem = *holder;
  const int stride = static_cast<int>(gridDim.x);

  int last_pair = -1;          // producer: the last pair (running index) whose loads were issued
  int q_loads = 0;             // producer: Q loads issued
  int lone_use0 = -1, lone_use1 = -1;   // producer: the single tail tile's latest use of pair slot 0 / 1
  bool lone_q = false;         // producer: the single tail tile's Q load issued
  bool gate_pending = false;   // producer: the latest Q load still lacks its gate arrival
  bool mma_done = false;
  if (warp == kWarpProducer) {
    // ------------------------------------------------------------ producer
    // Pairs in running order g = k (T + 1) + u, pair g in slot g & 1 (after
    // pair g - 2).  The producer polls S_B for every completion in turn, each
    // poll before its own signal that the completion after the polled one
    // needs, so a parity poll can never see a phase two away from the one it
    // means.  With g0 = k (T + 1):
    //   u = 0   the item's Q tiles (Q full counts the loads' arrival and a
    //           gate) and pair g0 (K_0).  Q and the slot were last read by the
    //           previous item's key step T - 2 (its prologue when T = 1),
    //           which S_B completion g0 - 2, polled at that item's end, covers.
    //   u = 1   S_B completion g0 - 1 (the previous item's last key step: its
    //           P V read pair g0 - 1, whose slot pair g0 + 1 takes); then the
    //           gate, without which this item's prologue cannot complete S_B.
    //   u >= 2  S_B completion g - 2 (the prologue or key step u - 3, the last
    //           reads of pair g - 2); then pair g - 1's arrival on P_A (its
    //           landing seen before that poll), without which key step u - 2
    //           cannot complete S_B.
    //   end     S_B completion g0 + T - 1 (key step T - 2, or the prologue), then
    //           the arrival for the item's last pair (landed, seen before).
    // An arrival on P_A must fall in the phase it is meant for: each follows an
    // S_B completion that the MMA warp committed after waiting for the phase
    // before.
    bool ok = true;
    int k = 0;
    for (int x = blockIdx.x; ok && x < n_units; x += stride) {
      int b, h;
      bool refresh;
      const int q0 = decode(x, b, h, refresh);
      if (q0 >= p.M) continue;
      const int kvh = h / (p.Hq / p.Hkv);
      const CUtensorMap* mKp = refresh ? &tmKpR : &tmKpC;
      const CUtensorMap* mVp = refresh ? &tmVpR : &tmVpC;
      const int g0 = k * (T + 1);
      // deep L2 prefetch of the K/V stream (below): cached steps of
      // one-query-head-per-kv-head shapes, by the first item of the head, in
      // the single-tile-tail instantiation only (carrying the code, even
      // untaken, slowed the kernel that walks the long-prompt GQA step)
      const bool lead = kLone && p.Hq == p.Hkv && (x % p.tiles_x) == 0;
      // Pair v's landing is waited for before the S_B poll that its arrival
      // on P_A must follow, so that the arrival comes right after that poll
      // (key step j's softmax warps arrive on P_A soon after S_B's completion
      // for key step j - 1).
      auto landed = [&](int v) { return warp_wait(bar_full + 8 * slot_of(v), phase_of(v), abort, p.err, p.wait_limit); };
      auto arrive = [&]() {
        if (lane0) mbar_arrive(bar_p_full);
        __syncwarp();
        return true;
      };
      for (int u = 0; u <= T; ++u) {
        const int g = g0 + u;
        if (u == 1) {
          if (k >= 1 && !warp_wait(bar_s_full + 8, static_cast<uint32_t>(g0 - 1) & 1u, abort, p.err, p.wait_limit)) {
            ok = false;
            break;
          }
          if (lane0) mbar_arrive(bar_q_full);                  // the gate
          __syncwarp();
          gate_pending = false;
        } else if (u >= 2) {
          if (!landed(g - 1) ||
              !warp_wait(bar_s_full + 8, static_cast<uint32_t>(g - 2) & 1u, abort, p.err, p.wait_limit) || !arrive()) {
            ok = false;
            break;
          }
        }
        if (u == 0) {
          if (lane0) {
            if (k == 0) tma_prefetch_map(&tmQ);
            mbar_arrive_expect_tx(bar_q_full, 2 * L::kTile);
            for (int t = 0; t < 2; ++t)
              for (int c = 0; c < L::kChunks; ++c)
                tma_load_4d(sQ + t * L::kTile + c * kChunkBytes, &tmQ, bar_q_full, c * 64, h, q0 + t * kBM, b);
          }
          __syncwarp();
          ++q_loads;
          gate_pending = true;
        }
        if (lane0) {
          const int slot = slot_of(g);
          const bool has_v = u >= 1, has_k = u < T;
          mbar_arrive_expect_tx(bar_full + 8 * slot, (has_v && has_k ? 2 : 1) * L::kTile);
          for (int part = has_v ? 0 : 1; part < (has_k ? 2 : 1); ++part) {
            const int j = part == 0 ? u - 1 : u;                // key tile
            const bool in_prompt = j < n_p;
            const int row = in_prompt ? j * kBN : (j - n_p) * kBN;
            const CUtensorMap* map = in_prompt ? (part == 0 ? mVp : mKp) : (part == 0 ? &tmVg : &tmKg);
            const uint32_t dst = sKV + (2 * slot + part) * L::kTile;
            for (int c = 0; c < L::kChunks; ++c)
              tma_load_4d(dst + c * kChunkBytes, map, bar_full + 8 * slot, c * 64, kvh, row, b);
          }
          // the K/V tiles of pair g + 2 (V_{u+1}, K_{u+2}) into L2 now, two
          // key steps before their own load, where each kv head feeds a
          // single query head: its K/V stream then comes from DRAM for one
          // pair of items (with several query heads per kv head the tiles are
          // read by many items at once and mostly hit L2, and the prefetch
          // instructions only delay the producer's arrivals)
          if constexpr (kLone) {
            for (int part = 0; lead && part < 2; ++part) {
              const int j = part == 0 ? u + 1 : u + 2;
              if (j >= T) continue;
              const bool in_prompt = j < n_p;
              const int row = in_prompt ? j * kBN : (j - n_p) * kBN;
              const CUtensorMap* map = in_prompt ? (part == 0 ? mVp : mKp) : (part == 0 ? &tmVg : &tmKg);
              for (int c = 0; c < L::kChunks; ++c) tma_prefetch_4d(map, c * 64, kvh, row, b);
            }
          }
          if (u == max(0, T - 2 - (static_cast<int>(blockIdx.x) & 3))) {
            if constexpr (kLone) {
              if (x + stride < n_units) prefetch_item(x + stride);
              else if (static_cast<int>(blockIdx.x) < p.n_lone) prefetch_lone();
            } else {
              prefetch_item(x + stride);
            }
          }
        }
        __syncwarp();
        last_pair = g;
      }
      if (!ok) break;
      // the item's end: S_B completion g0 + T - 1, then the last pair's arrival
      if (!landed(g0 + T) ||
          !warp_wait(bar_s_full + 8, static_cast<uint32_t>(g0 + T - 1) & 1u, abort, p.err, p.wait_limit) || !arrive()) {
        ok = false;
        break;
      }
      ++k;
    }
    if constexpr (kLone) {
      // ------------------------------------------------ the single tail tile
      // Its Q tile and first pair wait for S_B completion k (T + 1) - 1, the
      // last item's last key step (its P V read both pair slots; Q was last
      // read by key step T - 2, polled at that item's end), the next S_B
      // completion in turn.  Pair u (V_{u-2}, K_u) goes into slot u mod 2 once
      // the commit announcing S(u - 2) -- completion u / 2 - 1 of that S
      // buffer's barrier, after the last reads of pair u - 2 -- is seen.  Once
      // the pair has landed the producer arrives on P(u - 2)'s barrier: the
      // commit it polled followed the MMA warp's wait for that barrier's
      // previous phase (P(u - 4)), so the arrival falls in its own phase.
      // Each poll comes before the producer's own arrival that the next
      // completion of its barrier needs.
      int b = 0, h = 0;
      bool refresh = false;
      const int q0 = static_cast<int>(blockIdx.x) < p.n_lone ? lone_q0(b, h, refresh) : p.M;   // decoded only if it exists
      if (ok && q0 < p.M) {
        const int kvh = h / (p.Hq / p.Hkv);
        const CUtensorMap* mKp = refresh ? &tmKpR : &tmKpC;
        const CUtensorMap* mVp = refresh ? &tmVpR : &tmVpC;
        ok = k == 0 ||
             warp_wait(bar_s_full + 8, static_cast<uint32_t>(k * (T + 1) - 1) & 1u, abort, p.err, p.wait_limit);
        if (ok) {
          if (lane0) {
            mbar_arrive_expect_tx(lq_full, L::kTile);
            for (int c = 0; c < L::kChunks; ++c) tma_load_4d(sQ + c * kChunkBytes, &tmQ, lq_full, c * 64, h, q0, b);
          }
          __syncwarp();
          lone_q = true;
        }
        for (int u = 0; ok && u <= T + 1; ++u) {
          if (u == 1 && T < 2) continue;                   // no K_1
          const int slot = u & 1;
          if (u >= 2 &&
              !warp_wait(l_s + 8 * slot, static_cast<uint32_t>(u / 2 - 1) & 1u, abort, p.err, p.wait_limit)) {
            ok = false;
            break;
          }
          if (lane0) {
            const bool has_v = u >= 2, has_k = u < T;
            mbar_arrive_expect_tx(l_full + 8 * slot, (has_v && has_k ? 2 : 1) * L::kTile);
            for (int part = has_v ? 0 : 1; part < (has_k ? 2 : 1); ++part) {
              const int j = part == 0 ? u - 2 : u;         // key tile
              const bool in_prompt = j < n_p;
              const int row = in_prompt ? j * kBN : (j - n_p) * kBN;
              const CUtensorMap* map = in_prompt ? (part == 0 ? mVp : mKp) : (part == 0 ? &tmVg : &tmKg);
              const uint32_t dst = sKV + (2 * slot + part) * L::kTile;
              for (int c = 0; c < L::kChunks; ++c)
                tma_load_4d(dst + c * kChunkBytes, map, l_full + 8 * slot, c * 64, kvh, row, b);
            }
          }
          __syncwarp();
          if (slot) lone_use1 = u >> 1;
          else lone_use0 = u >> 1;
          if (u >= 2) {
            if (!warp_wait(l_full + 8 * slot, static_cast<uint32_t>(u >> 1) & 1u, abort, p.err, p.wait_limit)) {
              ok = false;
              break;
            }
            if (lane0) mbar_arrive(l_p + 8 * slot);      // P(u - 2): barrier (u - 2) mod 2 = slot
            __syncwarp();
          }
        }
      }
    }
    __syncwarp();              // reconverged before the teardown
  } else if (warp >= kWarpCopy) {        // present only in the kRewrite kernels (11 warps)
    // ------------------------------------------------------------ cache copy
    // Its share of every refreshed item's prompt tiles, ahead of the walk:
    // nothing orders it against the other roles.
    if constexpr (kRewrite) {
      for (int x = blockIdx.x; x < n_units; x += stride) {
        int b, h;
        bool refresh;
        const int q0 = decode(x, b, h, refresh);
        if (q0 >= p.M || !refresh) continue;
        copy_prompt_share<D>(p, b, h / (p.Hq / p.Hkv), 0, n_p,
                             (h % (p.Hq / p.Hkv)) * p.tiles_x + (q0 - p.q_begin_refresh) / (2 * kBM),
                             (p.Hq / p.Hkv) * p.tiles_x);
      }
    }
  } else if (warp == kWarpMma) {
    // ------------------------------------------------------------ MMA issuer
    // Lane 0 alone.  Per item: wait for Q and pair k (T + 1) (K_0), S(0) of
    // both tiles; per key step j: wait P_X (k T + j; P_A also says the pair
    // landed), before the item's first P V also "O drained" of the previous
    // item, then P_X V_j and Q_X K_{j+1}^T, commit S_X; after the last step
    // also "O final".
    constexpr uint32_t idesc_qk = idesc_bf16_f32(kBM, kBN, 0, 0);
    constexpr uint32_t idesc_pv = idesc_bf16_f32(kBM, D, 0, 1);
    // Operand descriptors built once: the Q tiles, and the K and V halves of
    // both pair slots; an MMA's own descriptor is one of these plus its
    // offset (desc_add), so a key step's 32 MMAs cost few instructions.
    const uint64_t qd0 = sdesc_sw128(sQ, 16, 1024), qd1 = sdesc_sw128(sQ + L::kTile, 16, 1024);
    const uint64_t kd0 = sdesc_sw128(sKV + L::kTile, 16, 1024), kd1 = sdesc_sw128(sKV + 3 * L::kTile, 16, 1024);
    const uint64_t vd0 = sdesc_sw128(sKV, kChunkBytes, 1024), vd1 = sdesc_sw128(sKV + 2 * L::kTile, kChunkBytes, 1024);
    // Each batch's descriptors step from an opaque copy of its base, one add
    // after each MMA (see opaque_desc).
    auto issue_qk = [&](int t, uint64_t kd) {
      uint64_t qa = opaque_desc(t == 0 ? qd0 : qd1), ka = opaque_desc(kd);
#pragma unroll
      for (int kk = 0; kk < D / 16; ++kk) {
        umma_ss(tmem + col_s(t), qa, ka, idesc_qk, kk > 0 ? 1u : 0u);
        const uint32_t step = (kk & 3) == 3 ? kChunkBytes - 96 : 32;   // to (kk + 1): 32 B, or the next chunk
        qa = desc_add(qa, step);
        ka = desc_add(ka, step);
      }
    };
    auto issue_pv = [&](int t, uint64_t vd, bool acc) {
      uint64_t va = opaque_desc(vd);
#pragma unroll
      for (int kk = 0; kk < 8; ++kk) {
        umma_ts(tmem + col_o(t), tmem + col_s(t) + 64 * (kk >> 2) + (kk & 3) * 8, va, idesc_pv, (acc || kk > 0) ? 1u : 0u);
        va = desc_add(va, 2048);
      }
    };
    auto v_tile_of = [&](int g) { return slot_of(g) ? vd1 : vd0; };
    auto k_tile_of = [&](int g) { return slot_of(g) ? kd1 : kd0; };
    bool ok = true;
    if (lane0) {
      int k = 0;
      for (int x = blockIdx.x; ok && x < n_units; x += stride) {
        int b, h;
        bool refresh;
        if (decode(x, b, h, refresh) >= p.M) continue;
        const int g0 = k * (T + 1);
        ok = mbar_wait(bar_q_full, static_cast<uint32_t>(k) & 1u, abort, p.err, p.wait_limit) &&
             mbar_wait(bar_full + 8 * slot_of(g0), phase_of(g0), abort, p.err, p.wait_limit);
        if (!ok) break;
        tc_fence_after();
        for (int t = 0; t < 2; ++t) {
          issue_qk(t, k_tile_of(g0));
          umma_commit(bar_s_full + 8 * t);
        }
        for (int j = 0; ok && j < T; ++j) {
          const bool more = j + 1 < T;
          const int g = g0 + j + 1;                             // pair (V_j, K_{j+1})
          for (int t = 0; t < 2; ++t) {
            if (p.debug_skip_last_pv && !more) { ok = false; break; }   // the softmax's wait for O must expire
            if (!mbar_wait(bar_p_full + 8 * t, static_cast<uint32_t>(k * T + j) & 1u, abort, p.err,
                           p.wait_limit) ||
                (j == 0 && k >= 1 &&
                 !mbar_wait(bar_o_free + 8 * t, static_cast<uint32_t>(k - 1) & 1u, abort, p.err, p.wait_limit))) {
              ok = false;
              break;
            }
            tc_fence_after();
            issue_pv(t, v_tile_of(g), j > 0);
            if (more) issue_qk(t, k_tile_of(g));
            umma_commit(bar_s_full + 8 * t);
            if (!more) umma_commit(bar_o_ready + 8 * t);
          }
        }
        ++k;
      }
      if constexpr (kLone) {
        // ---------------------------------------------- the single tail tile
        // Prologue: S(0) = Q K_0^T into S buffer 0, S(1) into buffer 1.  Key
        // step j: P(j) (P also says pair j + 2 landed), before the first P V
        // "O drained" of tile A's previous item, then P(j) V_j from buffer
        // j mod 2 and, while tiles remain, S(j + 2) = Q K_{j+2}^T into that
        // buffer (after the P V that reads it: MMAs run in issue order), one
        // commit on the buffer's barrier; after the last step also O final.
        int b = 0, h = 0;
        bool refresh = false;
        const int q0 = static_cast<int>(blockIdx.x) < p.n_lone ? lone_q0(b, h, refresh) : p.M;
        if (ok && q0 < p.M) {
          auto qk_lone = [&](int buf, uint64_t kd) {
            uint64_t qa = opaque_desc(qd0), ka = opaque_desc(kd);
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk) {
              umma_ss(tmem + col_s(buf), qa, ka, idesc_qk, kk > 0 ? 1u : 0u);
              const uint32_t step = (kk & 3) == 3 ? kChunkBytes - 96 : 32;
              qa = desc_add(qa, step);
              ka = desc_add(ka, step);
            }
          };
          ok = mbar_wait(lq_full, 0, abort, p.err, p.wait_limit) && mbar_wait(l_full, 0, abort, p.err, p.wait_limit);
          if (ok) {
            tc_fence_after();
            qk_lone(0, kd0);                               // K_0: slot 0's K part
            umma_commit(l_s);
          }
          if (ok && T >= 2) {
            ok = mbar_wait(l_full + 8, 0, abort, p.err, p.wait_limit);
            if (ok) {
              tc_fence_after();
              qk_lone(1, kd1);                             // K_1: slot 1's K part
              umma_commit(l_s + 8);
            }
          }
          for (int j = 0; ok && j < T; ++j) {
            if (p.debug_skip_last_pv && j + 1 == T) { ok = false; break; }   // the softmax's wait for O must expire
            if (!mbar_wait(l_p + 8 * (j & 1), static_cast<uint32_t>(j >> 1) & 1u, abort, p.err, p.wait_limit) ||
                (j == 0 && k >= 1 &&
                 !mbar_wait(bar_o_free, static_cast<uint32_t>(k - 1) & 1u, abort, p.err, p.wait_limit))) {
              ok = false;
              break;
            }
            tc_fence_after();
            const int s = j & 1;                           // P(j)'s buffer and pair j + 2's slot
            uint64_t va = opaque_desc(s ? vd1 : vd0);
#pragma unroll
            for (int kk = 0; kk < 8; ++kk) {
              umma_ts(tmem + col_o(0), tmem + col_s(s) + 64 * (kk >> 2) + (kk & 3) * 8, va, idesc_pv,
                      (j > 0 || kk > 0) ? 1u : 0u);
              va = desc_add(va, 2048);
            }
            if (j + 2 < T) qk_lone(s, s ? kd1 : kd0);
            umma_commit(l_s + 8 * s);
            if (j + 1 == T) umma_commit(l_o);
          }
        }
      }
    }
    __syncwarp();
    mma_done = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
  } else {
    // ------------------------------------------------------------ softmax
    // As in the two-tile attn_fwd_kernel, per item: S_X(j) is S_X's completion
    // k (T + 1) + j; O final is "O final" k; after the epilogue the warpgroup
    // arrives on "O drained".
    const int t = (warp - kWarpSoftmax0) >> 2;
    const int r = (warp & 3) * 32 + (threadIdx.x & 31);
    const uint32_t t_lane = tmem + (static_cast<uint32_t>((warp & 3) * 32) << 16);
    const uint32_t colS = col_s(t), colO = col_o(t);
    const uint32_t bar_s = bar_s_full + 8 * t;
    const uint32_t bar_ph = bar_p_full + 8 * t;
    const float sl2 = p.scale_log2;
    auto rescale_o = [&](float a) {
#pragma unroll 1
      for (int c0 = 0; c0 < D; c0 += 16) {
        uint32_t o[16];
        tmem_ld_16(t_lane + colO + c0, o);
#pragma unroll
        for (int kq = 0; kq < 16; ++kq) o[kq] = __float_as_uint(__uint_as_float(o[kq]) * a);
        tmem_st_16(t_lane + colO + c0, o);
      }
    };
    // After an expired wait a warp stops its key steps (see attn_fwd_kernel)
    // and goes to the item's epilogue; whether the walk goes on is decided
    // once per item for the whole warpgroup (the epilogue's named barrier
    // needs all four warps): its first thread samples the abort flag into
    // shared memory before that barrier, every thread reads it after.
    volatile int* stop_flag = reinterpret_cast<volatile int*>(gbase + kPersistStopOff<D>);
    int k = 0;
    for (int x = blockIdx.x; x < n_units; x += stride) {
      int b, h;
      bool refresh;
      const int q0 = decode(x, b, h, refresh);
      if (q0 >= p.M) continue;
      float m_used = -INFINITY;
      float2 l2 = make_float2(0.f, 0.f);
      bool failed = false;
      for (int j = 0; j < T; ++j) {
        if (!warp_wait(bar_s, static_cast<uint32_t>(k * (T + 1) + j) & 1u, abort, p.err, p.wait_limit)) {
          failed = true;
          break;
        }
        tc_fence_after();
        const int valid = j < n_p ? min(kBN, p.P - j * kBN) : min(kBN, p.G - (j - n_p) * kBN);
        float xs[128];
        load_scores128(t_lane + colS, valid, xs);
        const float tm = max128(xs) * sl2;
        if (j == 0) {
          m_used = tm;
        } else if (__any_sync(0xffffffffu, tm > m_used + 8.0f)) {
          // O holds P V up to tile j-1, complete (S(j) was announced after it).
          const float m_new = fmaxf(m_used, tm);
          const float a = ex2_approx(m_used - m_new);
          m_used = m_new;
          l2.x *= a;
          l2.y *= a;
          rescale_o(a);
        }
        const float2 neg_m = make_float2(-m_used, -m_used);
        const float2 slv = make_float2(sl2, sl2);
        float2 acc[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          uint32_t pk[16];
#pragma unroll
          for (int kq = 0; kq < 16; ++kq) {
            const float2 y = ffma2(make_float2(xs[32 * q + 2 * kq], xs[32 * q + 2 * kq + 1]), slv, neg_m);
            const float2 pr = make_float2(ex2_approx(y.x), ex2_approx(y.y));
            acc[kq & 1] = fadd2(acc[kq & 1], pr);
            pk[kq] = pack_bf16x2(pr.x, pr.y);
          }
          tmem_st_16_async(t_lane + colS + 64 * (q >> 1) + 16 * (q & 1), pk);
        }
        tmem_wait_st();
        l2 = fadd2(l2, fadd2(acc[0], acc[1]));
        tc_fence_before();
        mbar_arrive(bar_ph);
      }
      const bool ok =
          !failed && warp_wait(bar_o_ready + 8 * t, static_cast<uint32_t>(k) & 1u, abort, p.err, p.wait_limit);
      tc_fence_after();
      const float l_sum = l2.x + l2.y;
      const int q = q0 + t * kBM + r;
      const bool live = ok && q < p.M;
      const int use = 2 * k + t;                       // this tile's turn on the staging buffer
      if (use > 0)
        warp_wait(bar_staged, static_cast<uint32_t>(use - 1) & 1u, abort, p.err, p.wait_limit);
      stage_o_row<D>(t_lane + colO, stage, r, 1.0f / l_sum);
      tc_fence_before();
      mbar_arrive(bar_o_free + 8 * t);                 // O has been read out of TMEM
      const bool issuer = threadIdx.x == 32 * (kWarpSoftmax0 + 4 * t);
      volatile int* stop = stop_flag + 2 * t + (k & 1);  // two slots: the next item's cannot overtake a reader
      if (issuer) *stop = *abort;
      store_o_tile<D>(&tmO, stage, 1u + t, issuer, ok, h, q0 + t * kBM, b, false);
      if (issuer) mbar_arrive(bar_staged);
      if (live && p.lse)
        p.lse[(static_cast<size_t>(b) * p.Hq + h) * p.M + q] = (m_used + log2f(l_sum)) * 0.69314718055994531f;
      ++k;
      if (*stop) break;
    }
    if constexpr (kLone) {
      // ------------------------------------------------ the single tail tile
      // Tile A's warpgroup, after its items: key step j reads S(j) from buffer
      // j mod 2 (completion j / 2 of that buffer's barrier: the prologue's,
      // then the commit after key step j - 2), writes P(j) over it and arrives
      // on P.  A rescale of O must see key step j - 1's P V done: the commit
      // after it is the next completion of the other buffer (the one that
      // announces S(j + 1)).  Then O final, and the epilogue in its turn on the
      // staging buffer.
      bool has_lone;
      {
        int b = 0, h = 0;
        bool refresh = false;
        // not after an abort (the walk stops only then; the flag stays set)
        has_lone = t == 0 && !*abort && static_cast<int>(blockIdx.x) < p.n_lone && lone_q0(b, h, refresh) < p.M;
      }
      if (has_lone) {
        float m_used = -INFINITY;
        float2 l2 = make_float2(0.f, 0.f);
        bool failed = false;
        for (int j = 0; j < T; ++j) {
          const int s = j & 1;
          if (!warp_wait(l_s + 8 * s, static_cast<uint32_t>(j >> 1) & 1u, abort, p.err, p.wait_limit)) {
            failed = true;
            break;
          }
          tc_fence_after();
          const int valid = j < n_p ? min(kBN, p.P - j * kBN) : min(kBN, p.G - (j - n_p) * kBN);
          float xs[128];
          load_scores128(t_lane + col_s(s), valid, xs);
          const float tm = max128(xs) * sl2;
          if (j == 0) {
            m_used = tm;
          } else if (__any_sync(0xffffffffu, tm > m_used + 8.0f)) {
            if (!warp_wait(l_s + 8 * (s ^ 1), static_cast<uint32_t>(((j - 1) >> 1) + 1) & 1u, abort, p.err,
                           p.wait_limit)) {
              failed = true;
              break;
            }
            tc_fence_after();
            const float m_new = fmaxf(m_used, tm);
            const float a = ex2_approx(m_used - m_new);
            m_used = m_new;
            l2.x *= a;
            l2.y *= a;
            rescale_o(a);
          }
          const float2 neg_m = make_float2(-m_used, -m_used);
          const float2 slv = make_float2(sl2, sl2);
          float2 acc[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            uint32_t pk[16];
#pragma unroll
            for (int kq = 0; kq < 16; ++kq) {
              const float2 y = ffma2(make_float2(xs[32 * q + 2 * kq], xs[32 * q + 2 * kq + 1]), slv, neg_m);
              const float2 pr = make_float2(ex2_approx(y.x), ex2_approx(y.y));
              acc[kq & 1] = fadd2(acc[kq & 1], pr);
              pk[kq] = pack_bf16x2(pr.x, pr.y);
            }
            tmem_st_16_async(t_lane + col_s(s) + 64 * (q >> 1) + 16 * (q & 1), pk);
          }
          tmem_wait_st();
          l2 = fadd2(l2, fadd2(acc[0], acc[1]));
          tc_fence_before();
          mbar_arrive(l_p + 8 * s);
        }
        const bool ok = !failed && warp_wait(l_o, 0, abort, p.err, p.wait_limit);
        tc_fence_after();
        // (b, h, q0) decoded again from an opaque copy of the CTA index: no
        // registers held across the key loop
        int b, h;
        bool refresh;
        const int q0 = lone_q0(b, h, refresh, opaque_int(static_cast<int>(blockIdx.x)));
        const float l_sum = l2.x + l2.y;
        const int q = q0 + r;
        const bool live = ok && q < p.M;
        const int use = 2 * k;                           // tile A's turn on the staging buffer
        if (use > 0) warp_wait(bar_staged, static_cast<uint32_t>(use - 1) & 1u, abort, p.err, p.wait_limit);
        stage_o_row<D>(t_lane + colO, stage, r, 1.0f / l_sum);
        tc_fence_before();
        mbar_arrive(bar_o_free);                         // O has been read out of TMEM
        const bool issuer = threadIdx.x == 32 * kWarpSoftmax0;
        store_o_tile<D>(&tmO, stage, 1u, issuer, ok, h, q0, b, false);
        if (issuer) mbar_arrive(bar_staged);
        if (live && p.lse)
          p.lse[(static_cast<size_t>(b) * p.Hq + h) * p.M + q] = (m_used + log2f(l_sum)) * 0.69314718055994531f;
      }
    }
    // the output stores are complete before the CTA exits (they wait on no other thread)
    if (threadIdx.x == 32 * (kWarpSoftmax0 + 4 * t)) bulk_wait_group_all();
    __syncwarp();
  }

  tc_fence_before();
  __syncthreads();
  const bool aborted = *abort != 0;
  if (warp == kWarpMma) {
    if (aborted || !mma_done) {
      if (lane0) {
        mbar_init(bar_drain, 1);
        mbar_fence_init();
        umma_commit(bar_drain);
      }
      __syncwarp();
      drain_wait(bar_drain, 0, p.wait_limit);
    }
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  } else if (warp == kWarpProducer && aborted) {
    if (gate_pending && lane0) mbar_arrive(bar_q_full);   // the last Q load's phase can then complete
    __syncwarp();
    if (q_loads > 0) drain_wait(bar_q_full, static_cast<uint32_t>(q_loads - 1) & 1u, p.wait_limit);
    for (int g = max(0, last_pair - 1); g <= last_pair; ++g) drain_wait(bar_full + 8 * slot_of(g), phase_of(g), p.wait_limit);
    if constexpr (kLone) {     // the single tail tile's Q load and its latest use of each pair slot
      if (lone_q) drain_wait(lq_full, 0, p.wait_limit);
      if (lone_use0 >= 0) drain_wait(l_full, static_cast<uint32_t>(lone_use0) & 1u, p.wait_limit);
      if (lone_use1 >= 0) drain_wait(l_full + 8, static_cast<uint32_t>(lone_use1) & 1u, p.wait_limit);
    }
  }
}

// Merges the key-range splits of one output row (b, q, h): with m_s the
// split's running max (log2 units), l_s its row sum and O_s its unnormalised
// output, out = sum_s 2^(m_s - m) O_s / sum_s 2^(m_s - m) l_s, m = max_s m_s.
// One thread per 8 output columns of a row; rows a launch did not compute
// (below q_begin) are left alone.  Launched as a programmatic dependent of the
// attention kernel: it waits for that grid before reading the workspace.
template <int D>
__global__ void __launch_bounds__(256)
attn_combine_kernel(const float* __restrict__ ws_o, const float2* __restrict__ ws_ml, int n_split, int B, int Hq,
                    int M, const uint8_t* __restrict__ flags, int default_refresh, int q_begin_refresh,
                    int q_begin_cached, __nv_bfloat16* __restrict__ out, float* __restrict__ lse) {
  constexpr int kChunks = D / 8;
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const long long idx = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
  const long long rows = static_cast<long long>(B) * M * Hq;
  if (idx >= rows * kChunks) return;
  const int ch = static_cast<int>(idx % kChunks);
  const long long r = idx / kChunks;                              // [b][q][h] order, as out
  const int h = static_cast<int>(r % Hq);
  const int q = static_cast<int>((r / Hq) % M);
  const int b = static_cast<int>(r / (static_cast<long long>(Hq) * M));
  const bool refresh = flags ? (flags[b] != 0) : (default_refresh != 0);
  if (q < (refresh ? q_begin_refresh : q_begin_cached)) return;
  const size_t row0 = (static_cast<size_t>(b) * Hq + h) * M + q;   // workspace [split][b][h][q]
  const size_t stride = static_cast<size_t>(B) * Hq * M;
  float m = -INFINITY;
  for (int sp = 0; sp < n_split; ++sp) m = fmaxf(m, ws_ml[sp * stride + row0].x);
  float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  float l = 0.f;
#pragma unroll 4
  for (int sp = 0; sp < n_split; ++sp) {
    const float2 ml = ws_ml[sp * stride + row0];
    const float w = ex2_approx(ml.x - m);
    l += w * ml.y;
    const float4* o = reinterpret_cast<const float4*>(ws_o + (sp * stride + row0) * D + ch * 8);
    const float4 a0 = o[0], a1 = o[1];
    acc[0] += w * a0.x; acc[1] += w * a0.y; acc[2] += w * a0.z; acc[3] += w * a0.w;
    acc[4] += w * a1.x; acc[5] += w * a1.y; acc[6] += w * a1.z; acc[7] += w * a1.w;
  }
  const float inv_l = 1.0f / l;
  *reinterpret_cast<uint4*>(out + ((static_cast<size_t>(b) * M + q) * Hq + h) * D + ch * 8) =
      make_uint4(pack_bf16x2(acc[0] * inv_l, acc[1] * inv_l), pack_bf16x2(acc[2] * inv_l, acc[3] * inv_l),
                 pack_bf16x2(acc[4] * inv_l, acc[5] * inv_l), pack_bf16x2(acc[6] * inv_l, acc[7] * inv_l));
  if (lse && ch == 0) lse[(static_cast<size_t>(b) * Hq + h) * M + q] = (m + log2f(l)) * 0.69314718055994531f;
}

template <int D, bool kRw>
int launch_fwd(int kind, cudaLaunchConfig_t lc, const CUtensorMap* m, const AttnParams& prm) {
  // Shared-memory limits are per device; setting them twice (two host threads
  // on a first call) is harmless.
  static std::atomic<bool> configured[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return cuda_status(cudaGetLastError(), "cudaGetDevice");
  if (dev < 0 || dev >= 64) {
    set_error("device ordinal %d out of range", dev);
    return ARCHER_ERR_UNSUPPORTED;
  }
  const int two = (int)Layout<D, false>::kSmemBytes, one = (int)Layout<D, true>::kSmemBytes,
            pers = (int)kPersistSmemBytes<D>;
  if (!configured[dev].load(std::memory_order_acquire)) {
    cudaError_t e = cudaFuncSetAttribute(attn_fwd_kernel<D, false, kRw>, cudaFuncAttributeMaxDynamicSharedMemorySize, two);
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(attn_fwd_kernel<D, true, kRw>, cudaFuncAttributeMaxDynamicSharedMemorySize, one);
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(attn_fwd_persist_kernel<D, kRw, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               pers);
    if constexpr (!kRw) {      // a single-tile tail only in cached steps (no rewrite)
      if (e == cudaSuccess)
        e = cudaFuncSetAttribute(attn_fwd_persist_kernel<D, false, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 pers);
    }
    if (e != cudaSuccess) return cuda_status(e, "cudaFuncSetAttribute(attention)");
    configured[dev].store(true, std::memory_order_release);
  }
  lc.blockDim = dim3(kRw ? kThreadsRw : kThreads);
  lc.dynamicSmemBytes = kind == kPlanOneTile ? one : (kind == kPlanPersistent ? pers : two);
  cudaError_t e;
  if (kind == kPlanOneTile)
    e = cudaLaunchKernelEx(&lc, attn_fwd_kernel<D, true, kRw>, m[0], m[1], m[2], m[3], m[4], m[5], m[6], m[7], prm);
  else if (kind == kPlanPersistent && prm.n_lone > 0) {
    if constexpr (!kRw)
      e = cudaLaunchKernelEx(&lc, attn_fwd_persist_kernel<D, false, true>, m[0], m[1], m[2], m[3], m[4], m[5], m[6],
                             m[7], prm);
    else
      e = cudaErrorInvalidValue;            // the plan gives refresh launches no single-tile tail
  } else if (kind == kPlanPersistent)
    e = cudaLaunchKernelEx(&lc, attn_fwd_persist_kernel<D, kRw, false>, m[0], m[1], m[2], m[3], m[4], m[5], m[6],
                           m[7], prm);
  else
    e = cudaLaunchKernelEx(&lc, attn_fwd_kernel<D, false, kRw>, m[0], m[1], m[2], m[3], m[4], m[5], m[6], m[7], prm);
  return cuda_status(e, "attention launch");
}

}  // namespace
}  // namespace archer
