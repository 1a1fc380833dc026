// One denoising step of Algorithm 1 (state-anchored rollback decoding) over an
// L-layer stack, captured once as a CUDA graph whose refresh decision stays on
// the device (Sec. 4.2): the rule kernel writes the per-sequence flags, a
// one-CTA kernel reduces them into the value of an if/else conditional node,
// and the node runs either every layer's refresh pass (per-sequence flags,
// cache rewrite) or every layer's cached step.  Scoring follows.  The host
// launches one graph per step and never waits for the flags.

#include <cstring>
#include <vector>

#include "archer_internal.h"

struct archer_step_graph {
  cudaGraph_t graph = nullptr;
  cudaGraphExec_t exec = nullptr;
  int device = -1;
};

namespace archer {
namespace {

// any = OR over flags[0, B); the conditional takes `any`; *count += any.
__global__ void __launch_bounds__(256)
refresh_condition_kernel(const uint8_t* __restrict__ flags, int B, cudaGraphConditionalHandle handle,
                         int32_t* refresh_count) {
  int any = 0;
  for (int b = threadIdx.x; b < B; b += blockDim.x) any |= flags[b] != 0;
  any = __syncthreads_or(any);
  if (threadIdx.x == 0) {
    cudaGraphSetConditional(handle, any ? 1u : 0u);
    if (refresh_count && any) *refresh_count += 1;
  }
}

// Ends a capture left open by a failed step, dropping the partial graph.
void abandon_capture(cudaStream_t s) {
  cudaStreamCaptureStatus st = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(s, &st) == cudaSuccess && st != cudaStreamCaptureStatusNone) {
    cudaGraph_t g = nullptr;
    cudaStreamEndCapture(s, &g);
    if (g) cudaGraphDestroy(g);
  }
  cudaGetLastError();
}

int check_desc(const archer_step_desc* d) {
  if (!d) { set_error("step desc is NULL"); return ARCHER_ERR_ARG; }
  if (d->n_layers < 1 || !d->layers) { set_error("n_layers must be >= 1 with a layers array"); return ARCHER_ERR_ARG; }
  if (d->shape.batch < 1) { set_error("a step graph needs batch >= 1"); return ARCHER_ERR_ARG; }
  if (!d->g_cur || !d->g_anchor || !d->age || !d->flag_out) {
    set_error("g_cur, g_anchor, age and flag_out must not be NULL");
    return ARCHER_ERR_ARG;
  }
  if (d->logits && (!d->max_prob || !d->top1 || !d->margin)) {
    set_error("scoring needs max_prob, top1 and margin");
    return ARCHER_ERR_ARG;
  }
  return ARCHER_OK;
}

// Captures the L layers of one branch on `s` (already capturing into a body).
int capture_layers(const archer_step_desc& d, const std::vector<archer_layer_io>& io, bool refresh,
                   cudaStream_t s) {
  for (int l = 0; l < d.n_layers; ++l) {
    const archer_layer_io& x = io[l];
    int st = refresh
        ? archer_prompt_refresh(&d.shape, x.q_all, x.k_prompt_new, x.v_prompt_new, x.k_resp, x.v_resp, x.out_full,
                                nullptr, x.k_cache, x.v_cache, d.flag_out, d.attn_workspace,
                                d.attn_workspace_bytes, s)
        : archer_attn_step(&d.shape, x.q_resp, x.k_cache, x.v_cache, x.k_resp, x.v_resp, x.out_step, nullptr,
                           d.attn_workspace, d.attn_workspace_bytes, s);
    if (st) return st;
  }
  return ARCHER_OK;
}

int build(const archer_step_desc& d, archer_step_graph* g) {
  std::vector<archer_layer_io> io(d.layers, d.layers + d.n_layers);
  cudaStream_t cs = nullptr, bs = nullptr;
  int st = ARCHER_OK;
  cudaError_t e;
  auto fail = [&](int status) {
    if (cs) { abandon_capture(cs); cudaStreamDestroy(cs); }
    if (bs) { abandon_capture(bs); cudaStreamDestroy(bs); }
    return status;
  };
  if ((e = cudaStreamCreateWithFlags(&cs, cudaStreamNonBlocking)) != cudaSuccess) return fail(cuda_status(e, "stream"));
  if ((e = cudaStreamCreateWithFlags(&bs, cudaStreamNonBlocking)) != cudaSuccess) return fail(cuda_status(e, "stream"));
  if ((e = cudaStreamBeginCapture(cs, cudaStreamCaptureModeRelaxed)) != cudaSuccess)
    return fail(cuda_status(e, "cudaStreamBeginCapture"));
  const int B = d.shape.batch;
  if ((st = archer_should_refresh(B, d.shape.resp_len, d.g_cur, d.g_anchor, d.age, d.K, d.max_age, 1, d.dist_out,
                                  d.flag_out, cs)))
    return fail(st);
  cudaGraph_t graph = nullptr;
  const cudaGraphNode_t* deps = nullptr;
  size_t n_deps = 0;
  cudaStreamCaptureStatus cst;
  if ((e = cudaStreamGetCaptureInfo(cs, &cst, nullptr, &graph, &deps, nullptr, &n_deps)) != cudaSuccess)
    return fail(cuda_status(e, "cudaStreamGetCaptureInfo"));
  cudaGraphConditionalHandle handle;
  if ((e = cudaGraphConditionalHandleCreate(&handle, graph, 0, cudaGraphCondAssignDefault)) != cudaSuccess)
    return fail(cuda_status(e, "cudaGraphConditionalHandleCreate"));
  refresh_condition_kernel<<<1, 256, 0, cs>>>(d.flag_out, B, handle, d.refresh_count);
  if ((e = cudaGetLastError()) != cudaSuccess) return fail(cuda_status(e, "refresh condition launch"));
  if ((e = cudaStreamGetCaptureInfo(cs, &cst, nullptr, &graph, &deps, nullptr, &n_deps)) != cudaSuccess)
    return fail(cuda_status(e, "cudaStreamGetCaptureInfo"));
  cudaGraphNodeParams cp = {cudaGraphNodeTypeConditional};
  cp.conditional.handle = handle;
  cp.conditional.type = cudaGraphCondTypeIf;
  cp.conditional.size = 2;                        // [0] runs when any flag is set, [1] otherwise
  cudaGraphNode_t cond = nullptr;
  if ((e = cudaGraphAddNode(&cond, graph, deps, nullptr, n_deps, &cp)) != cudaSuccess)
    return fail(cuda_status(e, "adding the conditional node"));
  cudaGraph_t body_refresh = cp.conditional.phGraph_out[0], body_cached = cp.conditional.phGraph_out[1];
  for (int branch = 0; branch < 2; ++branch) {
    cudaGraph_t body = branch == 0 ? body_refresh : body_cached;
    if ((e = cudaStreamBeginCaptureToGraph(bs, body, nullptr, nullptr, 0, cudaStreamCaptureModeRelaxed)) !=
        cudaSuccess)
      return fail(cuda_status(e, "capturing a conditional body"));
    if ((st = capture_layers(d, io, branch == 0, bs))) return fail(st);
    cudaGraph_t got = nullptr;
    if ((e = cudaStreamEndCapture(bs, &got)) != cudaSuccess) return fail(cuda_status(e, "ending a body capture"));
  }
  if ((e = cudaStreamUpdateCaptureDependencies(cs, &cond, nullptr, 1, cudaStreamSetCaptureDependencies)) !=
      cudaSuccess)
    return fail(cuda_status(e, "cudaStreamUpdateCaptureDependencies"));
  if (d.logits) {
    const int rows_b = B, rows_g = d.shape.resp_len;
    if ((st = archer_decode_scores(rows_b, rows_g, d.vocab, d.logits_dtype, d.logits, d.row_stride, d.mask_state,
                                   d.cur_tokens, d.max_prob, d.top1, d.margin, d.cur_prob, d.scores_workspace,
                                   d.scores_workspace_bytes, cs)))
      return fail(st);
  }
  cudaGraph_t done = nullptr;
  if ((e = cudaStreamEndCapture(cs, &done)) != cudaSuccess) return fail(cuda_status(e, "cudaStreamEndCapture"));
  g->graph = done;
  if ((e = cudaGraphInstantiate(&g->exec, done, 0)) != cudaSuccess) return fail(cuda_status(e, "cudaGraphInstantiate"));
  cudaStreamDestroy(cs);
  cudaStreamDestroy(bs);
  return ARCHER_OK;
}

}  // namespace
}  // namespace archer

using namespace archer;

extern "C" {

int archer_step_graph_create(const archer_step_desc* desc, archer_step_graph** out) {
  if (!out) { set_error("out is NULL"); return ARCHER_ERR_ARG; }
  *out = nullptr;
  int st = check_desc(desc);
  if (st) return st;
  archer_step_graph* g = new archer_step_graph();
  cudaGetDevice(&g->device);
  if ((st = build(*desc, g))) {
    if (g->exec) cudaGraphExecDestroy(g->exec);
    if (g->graph) cudaGraphDestroy(g->graph);
    delete g;
    return st;
  }
  *out = g;
  return ARCHER_OK;
}

int archer_step_graph_launch(archer_step_graph* graph, void* stream) {
  if (!graph || !graph->exec) { set_error("graph is NULL"); return ARCHER_ERR_ARG; }
  return cuda_status(cudaGraphLaunch(graph->exec, static_cast<cudaStream_t>(stream)), "cudaGraphLaunch");
}

int archer_step_graph_destroy(archer_step_graph* graph) {
  if (!graph) return ARCHER_OK;
  if (graph->exec) cudaGraphExecDestroy(graph->exec);
  if (graph->graph) cudaGraphDestroy(graph->graph);
  delete graph;
  return ARCHER_OK;
}

}  // extern "C"
