/*
 * libarcher -- the per-step hot path of Archer's asymmetric-cache denoising
 * step (Adaptive Reuse of Cached Hidden States for Efficient Rollback,
 * arXiv 2608.08086) for one NVIDIA GB300 (sm_103a).
 *
 * Plain C ABI: device pointers, sizes and a CUDA stream.  No call allocates
 * device memory, synchronises the device or prints.  Every call is
 * asynchronous on `stream` (a cudaStream_t passed as void*; NULL = the legacy
 * default stream) and returns an archer_status.  A non-zero status means that
 * nothing was launched, except ARCHER_ERR_CUDA from a failed launch; the
 * reason is available from archer_last_error() on the calling thread.
 *
 * Layouts (all contiguous, row-major, bf16 = IEEE bfloat16 bit patterns):
 *   queries  [B, M, Hq,  D]     M = G (cached step) or N = P + G (refresh)
 *   prompt   [B, P, Hkv, D]     K and V separately (the cache C_p, Sec. 4.1)
 *   response [B, G, Hkv, D]     K and V separately
 *   output   [B, M, Hq,  D]     bf16;  lse [B, Hq, M] fp32 (natural log)
 * Every device pointer must be 16-byte aligned; D must be 64 or 128;
 * Hq % Hkv == 0 (GQA: query head h reads KV head h / (Hq / Hkv)).
 */
#ifndef ARCHER_H_
#define ARCHER_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum archer_status {
  ARCHER_OK = 0,
  ARCHER_ERR_ARG = -1,          /* null pointer, negative size, misalignment  */
  ARCHER_ERR_UNSUPPORTED = -2,  /* valid but unsupported shape (e.g. D = 96)   */
  ARCHER_ERR_CUDA = -3,         /* a CUDA runtime/driver call failed          */
  ARCHER_ERR_TIMEOUT = -4       /* a kernel's bounded wait expired            */
} archer_status;

typedef enum archer_dtype {
  ARCHER_DTYPE_BF16 = 0,
  ARCHER_DTYPE_F32 = 1
} archer_dtype;

/* Problem statement of one attention layer (Sec. 4.1: prompt p of length P,
 * response g of length G, N = P + G).  softmax_scale <= 0 selects
 * 1/sqrt(head_dim). */
typedef struct archer_shape {
  int batch;        /* B  >= 0                                */
  int prompt_len;   /* P  >= 0 (P = 0: response-only attention) */
  int resp_len;     /* G  >= 1                                */
  int n_heads;      /* Hq >= 1                                */
  int n_kv_heads;   /* Hkv >= 1, Hq % Hkv == 0                */
  int head_dim;     /* D in {64, 128}                         */
  float softmax_scale;
} archer_shape;

/*
 * Cached response step -- Sec. 4.1, Eq. archer-cached and Eq. archer-attention:
 *   out = Attn(Q_g(g_t), [K_p(g_r) || K_g(g_t)], [V_p(g_r) || V_g(g_t)])
 * Non-causal: each of the G response queries attends to all P cached prompt
 * keys and all G fresh response keys; the concatenation is never formed.
 *   q_resp  [B, G, Hq, D]  bf16     k_cache, v_cache [B, P, Hkv, D] bf16 (read)
 *   k_resp, v_resp [B, G, Hkv, D] bf16
 *   out     [B, G, Hq, D]  bf16 (written)
 *   lse     [B, Hq, G] fp32 (written; may be NULL)
 *   workspace / ws_bytes: 16-byte aligned scratch of at least
 *   archer_attn_workspace_size() bytes, any contents.  With it, a launch whose
 *   grid leaves SMs idle splits its key tiles across CTAs and merges the
 *   splits in a second kernel; with NULL (or too small) it runs unsplit, with
 *   the same result up to rounding.  Owned by the caller; must not be used by
 *   another call that can overlap on the GPU.
 * k_cache/v_cache may be NULL only when P == 0.
 */
int archer_attn_step(const archer_shape* shape, const void* q_resp, const void* k_cache,
                     const void* v_cache, const void* k_resp, const void* v_resp, void* out,
                     float* lse, void* workspace, size_t ws_bytes, void* stream);

/*
 * Prompt refresh -- Sec. 4.2 and Algorithm 1's FullForward: every position of
 * a refreshed sequence is a query over the fresh [K_p(g_t) || K_g(g_t)], and
 * the prompt cache is replaced by the fresh prompt K/V (C_r <- C_p(g_t)).
 *   q_all [B, N, Hq, D] bf16 (rows 0..P-1 prompt queries, P..N-1 response queries)
 *   k_prompt_new, v_prompt_new [B, P, Hkv, D] bf16: fresh prompt K/V
 *   k_resp, v_resp [B, G, Hkv, D] bf16
 *   out [B, N, Hq, D] bf16; lse [B, Hq, N] fp32 (may be NULL)
 *   k_cache, v_cache [B, P, Hkv, D] bf16: for a refreshed sequence overwritten
 *     with k_prompt_new / v_prompt_new (no copy when the pointers are equal;
 *     otherwise the two must not overlap); for a sequence whose flag is clear,
 *     read as the anchored cache.  The rewrite happens inside the attention
 *     launch: one kernel per call (plus the split merge, when it splits).
 *   refresh_flags [B] uint8 (device; may be NULL = refresh every sequence).
 *     A sequence whose flag is 0 takes the cached step instead: its rows
 *     P..N-1 of out/lse get Attn(Q_g, [K_cache || K_g], ...), its rows 0..P-1
 *     are left untouched and its cache is kept.  This serves a batch with
 *     per-sequence refresh decisions in one call.
 */
int archer_prompt_refresh(const archer_shape* shape, const void* q_all, const void* k_prompt_new,
                          const void* v_prompt_new, const void* k_resp, const void* v_resp,
                          void* out, float* lse, void* k_cache, void* v_cache,
                          const uint8_t* refresh_flags, void* workspace, size_t ws_bytes,
                          void* stream);

/* Launch plan of one attention call, for tests and capacity planning.
 * op: ARCHER_PLAN_ATTN_STEP (archer_attn_step), ARCHER_PLAN_REFRESH_ALL
 * (archer_prompt_refresh with refresh_flags NULL) or ARCHER_PLAN_REFRESH_FLAGS
 * (with flags).  ws_bytes: the 16-byte aligned workspace the call would get
 * (0: none).  sm_count: SMs of the GPU to plan for; <= 0 queries the current
 * device.  With sm_count > 0 the call is host arithmetic only (no CUDA call,
 * no GPU needed).  The attention calls launch exactly this plan: 128-row
 * query tiles, one or two per work item; the key range of an item split when
 * the grid leaves SMs idle and the workspace suffices (a merge kernel then
 * follows); a persistent grid of sm_count CTAs when items of two whole tiles
 * outnumber the SMs.  A last wave of items at most half full runs as single
 * tiles (in a persistent walk, one each on its first CTAs after their items).
 * Writes *plan (zeros for batch 0); returns ARCHER_OK, or
 * ARCHER_ERR_ARG / ARCHER_ERR_UNSUPPORTED for a shape the calls would reject.
 * Sec. 4.1 defines the attention this plans; the plan itself is this
 * library's. */
enum {
  ARCHER_PLAN_ATTN_STEP = 0,
  ARCHER_PLAN_REFRESH_ALL = 1,
  ARCHER_PLAN_REFRESH_FLAGS = 2
};
enum {
  ARCHER_KERNEL_TWO_TILE = 0,    /* one CTA per item of two query tiles */
  ARCHER_KERNEL_ONE_TILE = 1,    /* one CTA per query tile (S double buffered) */
  ARCHER_KERNEL_PERSISTENT = 2   /* one CTA per SM walking two-tile items */
};
typedef struct archer_attn_plan {
  int kernel;                /* ARCHER_KERNEL_*                                   */
  int tiles_per_cta;         /* query tiles per work item: 1 or 2                 */
  int n_split;               /* key-range splits per item (> 1: merge kernel)     */
  int key_tiles_per_split;   /* 128-key tiles one split walks                     */
  int work_items;            /* items over (sequence, head, query range, split)   */
  int grid;                  /* CTAs of the attention launch                      */
  int single_tail;           /* last-wave items run as single tiles (a two-tile  */
                             /* launch: appended one-tile CTAs; persistent: the  */
                             /* walk's first 2 x this CTAs take one tile each)   */
  size_t split_workspace;    /* workspace bytes a split wants (0: no split wanted) */
} archer_attn_plan;
int archer_attn_plan_query(const archer_shape* shape, int op, size_t ws_bytes, int sm_count,
                           archer_attn_plan* plan);

/* Scratch bytes that let archer_attn_step / archer_prompt_refresh split the
 * key tiles of a launch over n_queries (= G or N) query rows per sequence:
 * n_split * B * Hq * n_queries * (4 D + 8), n_split chosen from the SM count;
 * 0 when the launch's grid already fills the GPU (or the shape is invalid).
 * The paper defines no such scratch: this sizing query, like the workspace
 * arguments of the attention calls, is this library's own addition (the
 * split-KV merge needs fp32 partials, and no call allocates). */
size_t archer_attn_workspace_size(const archer_shape* shape, int n_queries);

/*
 * Decoder scoring -- the inputs of the rollback decoder's confidence rule
 * (Sec. 6 "confidence"; the decision margin of Eq. theory-margin is taken on
 * these probabilities).  For each of the batch * resp_len rows of logits z:
 *   p        = softmax(z) in fp32
 *   top1     = the lowest index attaining max_j z_j
 *   max_prob = p[top1]
 *   margin   = p[top1] - p[top2], top2 the next index in (value desc, index
 *              asc) order (margin 0 on a tie; = max_prob when vocab == 1)
 *   cur_prob = p[cur_tokens[r]] where mask_state[r] == 0 and
 *              0 <= cur_tokens[r] < vocab, else 0   (skipped when NULL)
 *   logits:   [batch * resp_len rows, row_stride elements], dtype bf16 or f32,
 *             row_stride >= vocab (rows whose start is not 16-byte aligned
 *             are read element-wise, which is slower).  -inf entries have
 *             probability 0; NaN gives undefined
 *             results.  A row with no finite entry is undefined.
 *   mask_state [rows] uint8 (may be NULL = unmasked); cur_tokens [rows] int32
 *   (may be NULL); outputs [rows] fp32 / int32 device arrays.
 *   workspace: at least archer_decode_scores_workspace_size(rows, vocab) bytes
 *   of scratch (chunk partials), any contents; 0 bytes when the vocabulary
 *   fits one chunk.  Two launches: a chunk kernel and, for multi-chunk rows,
 *   a combine kernel.
 */
int archer_decode_scores(int batch, int resp_len, int vocab, int dtype, const void* logits,
                         int64_t row_stride, const uint8_t* mask_state, const int32_t* cur_tokens,
                         float* max_prob, int32_t* top1, float* margin, float* cur_prob,
                         void* workspace, size_t ws_bytes, void* stream);

/* Workspace bytes archer_decode_scores needs for rows x vocab logits of
 * either dtype (sized for fp32, which needs the most).  The workspace pair of
 * archer_decode_scores and this query are this library's additions to the
 * scoring operation, so that no call allocates. */
size_t archer_decode_scores_workspace_size(int rows, int vocab);

/*
 * Decoder scoring without any device allocation.  The paper has no
 * counterpart: this serves callers that cannot allocate a workspace -- code
 * running inside another framework's memory pool, latency-critical loops that
 * must not pay cudaMalloc's device synchronisation, thin bindings with no
 * allocator at hand.  Same arguments and results as archer_decode_scores,
 * without workspace / ws_bytes.
 *   Scratch: a static device array of ARCHER_NOALLOC_SCRATCH_BYTES (4 MiB),
 *   created when the library is loaded on a device and held by that device
 *   until the process exits.  A call needs 16 bytes per 32 KB chunk of each
 *   row (rows * ceil(vocab * element size / 32768) * 16 bytes, none when a
 *   row is one chunk); one needing more than 4 MiB (for a 152,064-entry
 *   vocabulary: more than 26,214 rows of bf16 logits, or 13,797 rows of fp32)
 *   returns ARCHER_ERR_UNSUPPORTED and launches nothing.
 *   The first call on a device, and the first after that device's context was
 *   replaced (cudaDeviceReset), looks up the array's device address (this may
 *   load the library's device code on that device); make that first call
 *   before any stream capture.
 *   Every call shares the one array per device (which keeps the last call's
 *   partials; nothing in it needs clearing): calls that can overlap on the GPU
 *   (other streams, other host threads) race and must be serialised by the
 *   caller.
 *   Calls no cudaMalloc / cudaFree.
 */
#define ARCHER_NOALLOC_SCRATCH_BYTES (4u << 20)
int archer_decode_scores_noalloc(int batch, int resp_len, int vocab, int dtype, const void* logits,
                                 int64_t row_stride, const uint8_t* mask_state,
                                 const int32_t* cur_tokens, float* max_prob, int32_t* top1,
                                 float* margin, float* cur_prob, void* stream);

/*
 * Refresh rule -- Sec. 4.2, Eq. archer-distance and Eq. archer-controller,
 * with the cache-age signal A_t = t - r of Sec. 6 as an optional cap:
 *   age_t   = age[b] + 1           (denoising steps since the anchor, this one included)
 *   dist[b] = D_t = sum_i [g_cur[b, i] != g_anchor[b, i]]
 *   flag[b] = D_t >= K  or  (max_age > 0 and age_t >= max_age)
 * With update_anchor != 0 a flagged sequence gets g_anchor <- g_cur and
 * age <- 0 (g_r <- g_t in Algorithm 1), an unflagged one age <- age_t.
 * With update_anchor == 0 only dist_out and flag_out are written.
 *   g_cur, g_anchor [batch, resp_len] int32 (token ids; a mask id is just
 *   another value); age [batch] int32; dist_out [batch] int32 (may be NULL);
 *   flag_out [batch] uint8.  K = INT32_MAX never refreshes on distance.
 */
int archer_should_refresh(int batch, int resp_len, const int32_t* g_cur, int32_t* g_anchor,
                          int32_t* age, int K, int max_age, int update_anchor, int32_t* dist_out,
                          uint8_t* flag_out, void* stream);

/*
 * Synthetic rollback decoder (a stand-in for the decoder D that Algorithm 1
 * takes as given; the paper's method has no counterpart -- it is the
 * environment the refresh rule reacts to).  Per sequence, from the scores of
 * the previous step (archer_decode_scores with mask_state = (g == mask_token)
 * and cur_tokens = g):
 *   a masked position with max_prob >= tau_accept takes its top-1 token;
 *   an unmasked position with cur_prob < tau_remask is masked again;
 *   if masked positions remain and none was accepted, the masked position
 *   with the largest max_prob (lowest index on ties) takes its top-1.
 *   g [batch, resp_len] int32 (updated in place); max_prob, top1, cur_prob
 *   [batch * resp_len]; changed [batch, resp_len] uint8 (written: 1 where g
 *   changed).  Decisions in fp32.
 */
int archer_decoder_update(int batch, int resp_len, float tau_accept, float tau_remask,
                          int32_t mask_token, const float* max_prob, const int32_t* top1,
                          const float* cur_prob, int32_t* g, uint8_t* changed, void* stream);

/*
 * Row scatter (staging, no counterpart in the paper's method): puts a step's
 * new response rows -- the Q, K or V rows of the positions the decoder
 * changed, for every layer -- into the layer tensors.  For o < n_outer,
 * b < batch, r < n, the row_bytes bytes at
 *   src + ((o * batch + b) * n + r) * row_bytes
 * are copied to
 *   dst0 + ((o * batch + b) * dst0_rows + dst0_row0 + pos[b * n + r]) * row_bytes
 * and, when dst1 is not NULL, likewise to dst1 (dst1_rows, dst1_row0).
 * pos [batch, n] int64; a position outside [0, dst_rows - dst_row0) is
 * skipped.  row_bytes a multiple of 16; pointers 16-byte aligned.
 */
int archer_scatter_rows(int n_outer, int batch, int n, size_t row_bytes, const void* src,
                        const int64_t* pos, void* dst0, int dst0_rows, int dst0_row0, void* dst1,
                        int dst1_rows, int dst1_row0, void* stream);

/* Bit-exact copy of a refreshed sequence's prompt K/V into the cache
 * (the cache rewrite C_r <- C_p(g_t) of Algorithm 1) for sequences whose flag
 * is set (all when flags is NULL).  src/dst [B, P, Hkv, D] bf16.  A standalone
 * copy for callers that rebuild a cache outside a refresh:
 * archer_prompt_refresh already rewrites the cache inside its own launch. */
int archer_cache_rewrite(const archer_shape* shape, const void* k_src, const void* v_src,
                         void* k_dst, void* v_dst, const uint8_t* refresh_flags, void* stream);

/*
 * One denoising step of Algorithm 1 over an L-layer stack, captured once as a
 * CUDA graph and replayed with no host synchronisation (the refresh decision
 * stays on the device):
 *   1. the refresh rule (archer_should_refresh with update_anchor = 1);
 *   2. a one-CTA kernel reduces the flags and sets the graph's conditional
 *      value to "any sequence flagged" (and adds 1 to *refresh_count if so);
 *   3. an if/else conditional node: if any flag, every layer runs
 *      archer_prompt_refresh with the per-sequence flags (unflagged sequences
 *      take the cached step in the same launch; flagged ones get their cache
 *      rewritten), else every layer runs archer_attn_step;
 *   4. archer_decode_scores over the step's logits (skipped if logits NULL).
 * Every pointer below is captured into the graph: the buffers must stay
 * allocated and in place for the graph's lifetime, and each step's inputs
 * (token ids, Q/K/V rows, logits) are written into them before the launch.
 * One graph serves one stream at a time; launches on one stream serialise.
 */
typedef struct archer_layer_io {
  const void* q_all;          /* [B, N, Hq, D]  read by a refresh            */
  const void* q_resp;         /* [B, G, Hq, D]  read by a cached step        */
  const void* k_prompt_new;   /* [B, P, Hkv, D] fresh prompt K (refresh)      */
  const void* v_prompt_new;
  const void* k_resp;         /* [B, G, Hkv, D]                              */
  const void* v_resp;
  void* k_cache;              /* [B, P, Hkv, D] the prompt cache C_p          */
  void* v_cache;
  void* out_full;             /* [B, N, Hq, D]  written by a refresh          */
  void* out_step;             /* [B, G, Hq, D]  written by a cached step      */
} archer_layer_io;

typedef struct archer_step_desc {
  archer_shape shape;         /* the layers' common shape                     */
  int n_layers;               /* L >= 1                                       */
  const archer_layer_io* layers;   /* [L], copied at creation                 */
  /* refresh rule (see archer_should_refresh) */
  const int32_t* g_cur;       /* [B, G] */
  int32_t* g_anchor;          /* [B, G] */
  int32_t* age;               /* [B]    */
  int K;
  int max_age;
  int32_t* dist_out;          /* [B], may be NULL */
  uint8_t* flag_out;          /* [B]    */
  int32_t* refresh_count;     /* one int32, may be NULL: +1 per refreshing step */
  /* decoder scoring (see archer_decode_scores); logits NULL skips it */
  int vocab;
  int logits_dtype;
  const void* logits;         /* [B * G, row_stride] */
  int64_t row_stride;
  const uint8_t* mask_state;
  const int32_t* cur_tokens;
  float* max_prob;
  int32_t* top1;
  float* margin;
  float* cur_prob;
  void* scores_workspace;
  size_t scores_workspace_bytes;
  /* attention scratch shared by the layers (they run one after another):
   * archer_attn_workspace_size(shape, N) bytes let small launches split */
  void* attn_workspace;
  size_t attn_workspace_bytes;
} archer_step_desc;

typedef struct archer_step_graph archer_step_graph;

/* Validates desc, captures and instantiates the graph (host work, done once;
 * the capture runs on a private stream and launches nothing).  *out receives
 * the handle (NULL on failure).  Calls no cudaMalloc; the graph's own objects
 * are the CUDA runtime's.  Errors: ARCHER_ERR_ARG for a NULL desc/out, no
 * layers, batch < 1, missing rule buffers or scoring outputs, and whatever
 * status the captured calls return for their arguments (the same checks as
 * when called directly); ARCHER_ERR_CUDA if capture or instantiation fails.
 * Nothing is left half-built. */
int archer_step_graph_create(const archer_step_desc* desc, archer_step_graph** out);

/* Launches one step on `stream` (asynchronous; ARCHER_ERR_ARG for a NULL
 * graph, ARCHER_ERR_CUDA if the launch fails).  Device-side wait timeouts
 * inside the step surface through archer_check_device, as for direct calls. */
int archer_step_graph_launch(archer_step_graph* graph, void* stream);

/* Frees the graph; call it after the graph's last launch has completed.
 * NULL is a no-op. */
int archer_step_graph_destroy(archer_step_graph* graph);

/* Test hook for failure detection (the paper has no counterpart): with
 * on != 0, every attention launch that follows withholds its last P V product,
 * so the softmax warps' bounded wait expires (after about 1e6 SM clocks), the
 * kernel leaves cleanly with TMEM freed, and archer_check_device reports
 * ARCHER_ERR_TIMEOUT; the outputs of those launches are undefined.  on == 0
 * restores normal launches.  Process-wide; returns the previous setting.
 * No GPU fault, trap or hang is involved: every wait stays bounded. */
int archer_debug_stall_attention(int on);

/* Reads and clears the device-side error word that kernels set when a
 * bounded wait expires.  Synchronises `stream`.  Returns ARCHER_OK or
 * ARCHER_ERR_TIMEOUT (or ARCHER_ERR_CUDA). */
int archer_check_device(void* stream);

/* Human-readable text for a status code (static storage). */
const char* archer_status_string(int status);

/* Detail of the last failed call on this thread ("" if none). */
const char* archer_last_error(void);

/* Library version: major * 10000 + minor * 100 + patch. */
int archer_version(void);

#ifdef __cplusplus
}  /* extern "C" */
#endif

#endif  /* ARCHER_H_ */
