// The C ABI of libarcher (include/archer.h): argument validation, scale
// defaults, status codes and the per-thread error text.  Every compute step is
// a kernel launched on the caller's stream; nothing here allocates, copies
// data or synchronises (archer_check_device excepted, by its contract).

#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>

#include "archer_internal.h"

namespace archer {

namespace {
thread_local char g_last_error[512] = "";
__device__ int g_device_error = 0;

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
}  // namespace

void set_error(const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_last_error, sizeof(g_last_error), fmt, ap);
  va_end(ap);
}

int cuda_status(cudaError_t e, const char* what) {
  if (e == cudaSuccess) return ARCHER_OK;
  set_error("%s: %s", what, cudaGetErrorString(e));
  return ARCHER_ERR_CUDA;
}

int* device_error_word() {
  // One address per device; looked up once per device.
  static int* addr[64] = {nullptr};
  static std::mutex mu;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
  std::lock_guard<std::mutex> lock(mu);
  if (!addr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_device_error) != cudaSuccess) return nullptr;
    addr[dev] = static_cast<int*>(p);
  }
  return addr[dev];
}

namespace {

int check_shape(const archer_shape* s, float* scale) {
  if (!s) { set_error("shape is NULL"); return ARCHER_ERR_ARG; }
  if (s->batch < 0 || s->prompt_len < 0 || s->resp_len < 1 || s->n_heads < 1 || s->n_kv_heads < 1) {
    set_error("bad shape: batch=%d prompt_len=%d resp_len=%d n_heads=%d n_kv_heads=%d", s->batch, s->prompt_len,
              s->resp_len, s->n_heads, s->n_kv_heads);
    return ARCHER_ERR_ARG;
  }
  if (s->n_heads % s->n_kv_heads != 0) {
    set_error("n_heads (%d) must be a multiple of n_kv_heads (%d)", s->n_heads, s->n_kv_heads);
    return ARCHER_ERR_ARG;
  }
  if (s->head_dim != 64 && s->head_dim != 128) {
    set_error("head_dim %d unsupported (64 or 128)", s->head_dim);
    return ARCHER_ERR_UNSUPPORTED;
  }
  if (s->batch > 65535 || s->n_heads > 65535 ||
      static_cast<long long>(s->prompt_len) + s->resp_len > (1ll << 30)) {
    set_error("shape too large for one launch");
    return ARCHER_ERR_UNSUPPORTED;
  }
  float sc = s->softmax_scale;
  if (!(sc == sc) || std::isinf(sc)) { set_error("softmax_scale is not finite"); return ARCHER_ERR_ARG; }
  if (sc <= 0.f) sc = 1.0f / std::sqrt(static_cast<float>(s->head_dim));
  *scale = sc;
  return ARCHER_OK;
}

int check_ptrs(const char* names, std::initializer_list<const void*> ptrs) {
  int i = 0;
  for (const void* p : ptrs) {
    if (!p) { set_error("pointer #%d of (%s) is NULL", i, names); return ARCHER_ERR_ARG; }
    if (!aligned16(p)) { set_error("pointer #%d of (%s) is not 16-byte aligned", i, names); return ARCHER_ERR_ARG; }
    ++i;
  }
  return ARCHER_OK;
}

static_assert(ARCHER_KERNEL_TWO_TILE == kPlanTwoTile && ARCHER_KERNEL_ONE_TILE == kPlanOneTile &&
                  ARCHER_KERNEL_PERSISTENT == kPlanPersistent,
              "public kernel ids follow the planner's");

// The fields of an archer_attn_step call that do not depend on its buffers.
AttnCall step_call(const archer_shape* s, float scale) {
  AttnCall c{};
  c.B = s->batch; c.P = s->prompt_len; c.G = s->resp_len;
  c.Hq = s->n_heads; c.Hkv = s->n_kv_heads; c.D = s->head_dim;
  c.scale = scale;
  c.M = c.G;
  c.flags = nullptr; c.default_refresh = 0;
  c.q_begin_refresh = 0; c.q_begin_cached = 0;
  return c;
}

// The same for archer_prompt_refresh: every position is a query of a
// refreshed sequence, rows P.. of a sequence whose flag is clear.
AttnCall refresh_call(const archer_shape* s, float scale, const uint8_t* flags) {
  AttnCall c = step_call(s, scale);
  c.M = c.P + c.G;
  c.flags = flags; c.default_refresh = 1;
  c.q_begin_refresh = 0; c.q_begin_cached = c.P;
  return c;
}

}  // namespace
}  // namespace archer

using namespace archer;

extern "C" {

int archer_attn_step(const archer_shape* shape, const void* q_resp, const void* k_cache, const void* v_cache,
                     const void* k_resp, const void* v_resp, void* out, float* lse, void* workspace,
                     size_t ws_bytes, void* stream) {
  float scale = 0.f;
  int st = check_shape(shape, &scale);
  if (st) return st;
  if ((st = check_ptrs("q_resp, k_resp, v_resp, out", {q_resp, k_resp, v_resp, out}))) return st;
  if (shape->prompt_len > 0 && (st = check_ptrs("k_cache, v_cache", {k_cache, v_cache}))) return st;
  if (lse && (reinterpret_cast<uintptr_t>(lse) & 3u)) { set_error("lse is not 4-byte aligned"); return ARCHER_ERR_ARG; }
  AttnCall c = step_call(shape, scale);
  c.q = q_resp;
  c.kp_refresh = k_cache; c.vp_refresh = v_cache;
  c.kp_cached = k_cache; c.vp_cached = v_cache;
  c.kg = k_resp; c.vg = v_resp;
  c.out = out; c.lse = lse;
  c.ws = workspace; c.ws_bytes = ws_bytes;
  return attn_launch(c, static_cast<cudaStream_t>(stream));
}

int archer_prompt_refresh(const archer_shape* shape, const void* q_all, const void* k_prompt_new,
                          const void* v_prompt_new, const void* k_resp, const void* v_resp, void* out, float* lse,
                          void* k_cache, void* v_cache, const uint8_t* refresh_flags, void* workspace,
                          size_t ws_bytes, void* stream) {
  float scale = 0.f;
  int st = check_shape(shape, &scale);
  if (st) return st;
  if ((st = check_ptrs("q_all, k_resp, v_resp, out", {q_all, k_resp, v_resp, out}))) return st;
  if (shape->prompt_len > 0 &&
      (st = check_ptrs("k_prompt_new, v_prompt_new, k_cache, v_cache", {k_prompt_new, v_prompt_new, k_cache, v_cache})))
    return st;
  if (lse && (reinterpret_cast<uintptr_t>(lse) & 3u)) { set_error("lse is not 4-byte aligned"); return ARCHER_ERR_ARG; }
  const cudaStream_t s = static_cast<cudaStream_t>(stream);
  AttnCall c = refresh_call(shape, scale, refresh_flags);
  c.q = q_all;
  c.kp_refresh = k_prompt_new; c.vp_refresh = v_prompt_new;
  c.kp_cached = k_cache; c.vp_cached = v_cache;
  c.kg = k_resp; c.vg = v_resp;
  c.out = out; c.lse = lse;
  c.ws = workspace; c.ws_bytes = ws_bytes;
  // The cache rewrite C_r <- C_p(g_t) happens inside the attention launch:
  // the kernel stores each fresh prompt K/V tile it loads for a refreshed
  // sequence back to the cache (nothing to do where the buffers coincide).
  c.rewrite = (k_prompt_new != k_cache ? 1 : 0) | (v_prompt_new != v_cache ? 2 : 0);
  return attn_launch(c, s);
}

int archer_attn_plan_query(const archer_shape* shape, int op, size_t ws_bytes, int sm_count,
                           archer_attn_plan* plan) {
  if (!plan) { set_error("plan is NULL"); return ARCHER_ERR_ARG; }
  *plan = archer_attn_plan{};
  float scale = 0.f;
  int st = check_shape(shape, &scale);
  if (st) return st;
  static const uint8_t some_flags = 1;     // never read: only "flags given" matters
  AttnCall c;
  if (op == ARCHER_PLAN_ATTN_STEP) c = step_call(shape, scale);
  else if (op == ARCHER_PLAN_REFRESH_ALL) c = refresh_call(shape, scale, nullptr);
  else if (op == ARCHER_PLAN_REFRESH_FLAGS) c = refresh_call(shape, scale, &some_flags);
  else { set_error("unknown plan op %d", op); return ARCHER_ERR_ARG; }
  if (c.B == 0) return ARCHER_OK;                 // the calls launch nothing
  AttnPlan pl;
  if ((st = attn_plan(c, ws_bytes, sm_count, &pl))) return st;
  plan->kernel = pl.kernel;
  plan->tiles_per_cta = pl.tiles_per_cta;
  plan->n_split = pl.n_split;
  plan->key_tiles_per_split = pl.per;
  plan->work_items = pl.units;
  plan->grid = pl.grid;
  plan->single_tail = pl.tail;
  plan->split_workspace = pl.split_bytes;
  return ARCHER_OK;
}

size_t archer_attn_workspace_size(const archer_shape* shape, int n_queries) {
  float scale = 0.f;
  if (check_shape(shape, &scale) != ARCHER_OK || n_queries < 1 || shape->batch == 0) return 0;
  return attn_workspace_bytes(shape->batch, shape->prompt_len, shape->resp_len, shape->n_heads, shape->head_dim,
                              n_queries);
}

int archer_cache_rewrite(const archer_shape* shape, const void* k_src, const void* v_src, void* k_dst, void* v_dst,
                         const uint8_t* refresh_flags, void* stream) {
  float scale = 0.f;
  int st = check_shape(shape, &scale);
  if (st) return st;
  if (shape->prompt_len == 0) return ARCHER_OK;
  if ((st = check_ptrs("k_src, v_src, k_dst, v_dst", {k_src, v_src, k_dst, v_dst}))) return st;
  const size_t per_seq = static_cast<size_t>(shape->prompt_len) * shape->n_kv_heads * shape->head_dim * 2;
  return cache_rewrite_launch(shape->batch, per_seq, k_src, v_src, k_dst, v_dst, refresh_flags,
                              static_cast<cudaStream_t>(stream));
}

int archer_decode_scores(int batch, int resp_len, int vocab, int dtype, const void* logits, int64_t row_stride,
                         const uint8_t* mask_state, const int32_t* cur_tokens, float* max_prob, int32_t* top1,
                         float* margin, float* cur_prob, void* workspace, size_t ws_bytes, void* stream) {
  if (batch < 0 || resp_len < 0 || vocab < 1 || row_stride < vocab) {
    set_error("bad scoring shape: batch=%d resp_len=%d vocab=%d row_stride=%lld", batch, resp_len, vocab,
              (long long)row_stride);
    return ARCHER_ERR_ARG;
  }
  if (dtype != ARCHER_DTYPE_BF16 && dtype != ARCHER_DTYPE_F32) {
    set_error("dtype %d unsupported", dtype);
    return ARCHER_ERR_UNSUPPORTED;
  }
  const long long rows = static_cast<long long>(batch) * resp_len;
  if (rows > 0x7FFFFFFFll) { set_error("too many rows"); return ARCHER_ERR_UNSUPPORTED; }
  if (rows == 0) return ARCHER_OK;
  const int esize = dtype == ARCHER_DTYPE_BF16 ? 2 : 4;
  if (!logits || (reinterpret_cast<uintptr_t>(logits) % esize) != 0) {
    set_error("logits is NULL or not aligned to its element size");
    return ARCHER_ERR_ARG;
  }
  if (!max_prob || !top1 || !margin) { set_error("max_prob, top1 and margin must not be NULL"); return ARCHER_ERR_ARG; }
  return decode_scores_launch(static_cast<int>(rows), vocab, dtype, logits, row_stride, mask_state, cur_tokens,
                              max_prob, top1, margin, cur_prob, workspace, ws_bytes,
                              static_cast<cudaStream_t>(stream));
}

size_t archer_decode_scores_workspace_size(int rows, int vocab) { return decode_scores_ws_bytes(rows, vocab); }

int archer_should_refresh(int batch, int resp_len, const int32_t* g_cur, int32_t* g_anchor, int32_t* age, int K,
                          int max_age, int update_anchor, int32_t* dist_out, uint8_t* flag_out, void* stream) {
  if (batch < 0 || resp_len < 0) { set_error("bad shape: batch=%d resp_len=%d", batch, resp_len); return ARCHER_ERR_ARG; }
  if (batch == 0) return ARCHER_OK;
  if ((resp_len > 0 && (!g_cur || !g_anchor)) || !age || !flag_out) {
    set_error("g_cur, g_anchor, age and flag_out must not be NULL");
    return ARCHER_ERR_ARG;
  }
  return should_refresh_launch(batch, resp_len, g_cur, g_anchor, age, K, max_age, update_anchor, dist_out, flag_out,
                               static_cast<cudaStream_t>(stream));
}

int archer_decoder_update(int batch, int resp_len, float tau_accept, float tau_remask, int32_t mask_token,
                          const float* max_prob, const int32_t* top1, const float* cur_prob, int32_t* g,
                          uint8_t* changed, void* stream) {
  if (batch < 0 || resp_len < 0) { set_error("bad shape: batch=%d resp_len=%d", batch, resp_len); return ARCHER_ERR_ARG; }
  if (batch == 0 || resp_len == 0) return ARCHER_OK;
  if (!max_prob || !top1 || !cur_prob || !g || !changed) {
    set_error("max_prob, top1, cur_prob, g and changed must not be NULL");
    return ARCHER_ERR_ARG;
  }
  if (!(tau_accept == tau_accept) || !(tau_remask == tau_remask)) { set_error("thresholds must not be NaN"); return ARCHER_ERR_ARG; }
  return decoder_update_launch(batch, resp_len, tau_accept, tau_remask, mask_token, max_prob, top1, cur_prob, g,
                               changed, static_cast<cudaStream_t>(stream));
}

int archer_scatter_rows(int n_outer, int batch, int n, size_t row_bytes, const void* src, const int64_t* pos,
                        void* dst0, int dst0_rows, int dst0_row0, void* dst1, int dst1_rows, int dst1_row0,
                        void* stream) {
  if (n_outer < 0 || batch < 0 || n < 0 || dst0_rows < 0 || dst0_row0 < 0 || dst1_rows < 0 || dst1_row0 < 0) {
    set_error("negative size");
    return ARCHER_ERR_ARG;
  }
  if (static_cast<long long>(n_outer) * batch * n == 0) return ARCHER_OK;
  if (row_bytes % 16 != 0 || row_bytes / 16 > 0x7FFFFFFF) { set_error("row_bytes must be a multiple of 16"); return ARCHER_ERR_ARG; }
  if (static_cast<long long>(n_outer) * batch * n > 0x7FFFFFFFll) { set_error("too many rows"); return ARCHER_ERR_UNSUPPORTED; }
  int st;
  if ((st = check_ptrs("src, pos, dst0", {src, pos, dst0}))) return st;
  if (dst1 && (st = check_ptrs("dst1", {dst1}))) return st;
  return scatter_rows_launch(n_outer, batch, n, row_bytes, src, pos, dst0, dst0_rows, dst0_row0, dst1, dst1_rows,
                             dst1_row0, static_cast<cudaStream_t>(stream));
}

int archer_check_device(void* stream) {
  cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_status(e, "cudaStreamSynchronize");
  int v = 0;
  if ((e = cudaMemcpyFromSymbol(&v, g_device_error, sizeof(int))) != cudaSuccess)
    return cuda_status(e, "reading the device error word");
  if (v == 0) return ARCHER_OK;
  const int zero = 0;
  if ((e = cudaMemcpyToSymbol(g_device_error, &zero, sizeof(int))) != cudaSuccess)
    return cuda_status(e, "clearing the device error word");
  set_error("a kernel's bounded wait expired (device error bits 0x%x)", v);
  return ARCHER_ERR_TIMEOUT;
}

const char* archer_status_string(int status) {
  switch (status) {
    case ARCHER_OK: return "ok";
    case ARCHER_ERR_ARG: return "invalid argument";
    case ARCHER_ERR_UNSUPPORTED: return "unsupported shape";
    case ARCHER_ERR_CUDA: return "CUDA error";
    case ARCHER_ERR_TIMEOUT: return "device wait timed out";
    default: return "unknown status";
  }
}

const char* archer_last_error(void) { return g_last_error; }

int archer_version(void) { return 200; }

}  // extern "C"
