// Host-side declarations shared by the C-ABI layer (api.cu) and the kernel
// translation units.  Not part of the public interface (include/archer.h).
#pragma once

#include <cuda_runtime.h>

#include <cstddef>
#include <cstdint>

#include "../../include/archer.h"

namespace archer {

// Records a formatted message as this thread's archer_last_error().
void set_error(const char* fmt, ...);

// Maps a CUDA error to ARCHER_ERR_CUDA with a message naming `what`.
int cuda_status(cudaError_t e, const char* what);

// Device error word (kernels OR kErr* bits into it).
int* device_error_word();

struct AttnCall {
  int B, P, G, Hq, Hkv, D;
  float scale;            // > 0
  const void* q;          // [B, M, Hq, D]
  int M;                  // rows of q / out
  const void* kp_refresh; // prompt K/V used by refreshed sequences
  const void* vp_refresh;
  const void* kp_cached;  // prompt K/V used by sequences taking the cached step
  const void* vp_cached;
  const void* kg;
  const void* vg;
  void* out;
  float* lse;
  const uint8_t* flags;   // nullable
  int default_refresh;    // used when flags == nullptr
  int q_begin_refresh;    // first query row of a refreshed sequence
  int q_begin_cached;     // first query row of a cached sequence
  void* ws;               // nullable: split-KV workspace (see attn_workspace_bytes)
  size_t ws_bytes;
  // Fused cache rewrite of refreshed sequences: bit 0 stores the fresh prompt
  // K (kp_refresh) into kp_cached, bit 1 V into vp_cached.  The two buffers of a
  // pair must not overlap unless they are the same buffer (then no bit).
  int rewrite = 0;
};

int attn_launch(const AttnCall& c, cudaStream_t stream);

// Workspace a launch over M query rows needs to split its key tiles across
// CTAs (0 when the launch would not split: its grid already fills the GPU).
size_t attn_workspace_bytes(int B, int P, int G, int Hq, int D, int M);

// The launch an attention call makes on a GPU of `sms` SMs (<= 0: the
// current device's count) with `usable_ws` bytes of aligned workspace.  Host
// arithmetic only when sms > 0 (no CUDA call); the launch reads its kernel,
// grid and split from it.
constexpr int kPlanTwoTile = 0, kPlanOneTile = 1, kPlanPersistent = 2;
struct AttnPlan {
  int kernel = kPlanTwoTile;
  int tiles_per_cta = 2;     // 128-row query tiles per work item
  int n_split = 1;           // key-range splits per item (> 1: a merge kernel follows)
  int per = 0;               // key tiles per split
  int tiles_x = 0;           // items per (sequence, head), splits included
  int units = 0;             // items over the launch
  int tail = 0;              // trailing one-tile CTAs of a two-tile launch
  int n_unit_ctas = 0;       // CTAs that run whole items
  int grid = 0;              // CTAs launched
  size_t split_bytes = 0;    // workspace the split wants (0: no split wanted)
};
int attn_plan(const AttnCall& c, size_t usable_ws, int sms, AttnPlan* plan);

int cache_rewrite_launch(int B, size_t bytes_per_seq, const void* k_src, const void* v_src,
                         void* k_dst, void* v_dst, const uint8_t* flags, cudaStream_t stream);

int decode_scores_launch(int rows, int vocab, int dtype, const void* logits, int64_t row_stride,
                         const uint8_t* mask_state, const int32_t* cur_tokens, float* max_prob,
                         int32_t* top1, float* margin, float* cur_prob, void* workspace,
                         size_t ws_bytes, cudaStream_t stream);
size_t decode_scores_ws_bytes(int rows, int vocab);

int decoder_update_launch(int B, int G, float tau_accept, float tau_remask, int32_t mask_token,
                          const float* max_prob, const int32_t* top1, const float* cur_prob, int32_t* g,
                          uint8_t* changed, cudaStream_t stream);

int scatter_rows_launch(int n_outer, int batch, int n, size_t row_bytes, const void* src, const int64_t* pos,
                        void* dst0, int rows0, int row00, void* dst1, int rows1, int row01, cudaStream_t stream);

int should_refresh_launch(int B, int G, const int32_t* g_cur, int32_t* g_anchor, int32_t* age,
                          int K, int max_age, int update_anchor, int32_t* dist, uint8_t* flag,
                          cudaStream_t stream);

}  // namespace archer
