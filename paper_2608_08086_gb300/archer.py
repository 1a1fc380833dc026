"""Python binding of libarcher's C ABI (include/archer.h), via ctypes.

Argument marshalling only: each function checks dtypes, shapes and devices of
the torch tensors it is given, passes their device pointers, sizes and the
current CUDA stream to the C function of the same name, and raises
ArcherError on a non-zero status.  Every step of the computation runs in
libarcher's CUDA kernels; there is no fallback path, and importing this
module fails loudly when libarcher.so is missing.
"""
from __future__ import annotations

import ctypes
import math
import os

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libarcher.so")

ARCHER_OK = 0
ARCHER_ERR_ARG = -1
ARCHER_ERR_UNSUPPORTED = -2
ARCHER_ERR_CUDA = -3
ARCHER_ERR_TIMEOUT = -4
ARCHER_DTYPE_BF16 = 0
ARCHER_DTYPE_F32 = 1
K_INFINITE = 2**31 - 1


class ArcherError(RuntimeError):
    def __init__(self, status: int, detail: str):
        super().__init__(f"archer status {status}: {detail}")
        self.status = status


class archer_shape(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int), ("prompt_len", ctypes.c_int), ("resp_len", ctypes.c_int),
                ("n_heads", ctypes.c_int), ("n_kv_heads", ctypes.c_int), ("head_dim", ctypes.c_int),
                ("softmax_scale", ctypes.c_float)]


class archer_layer_io(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in ("q_all", "q_resp", "k_prompt_new", "v_prompt_new", "k_resp",
                                               "v_resp", "k_cache", "v_cache", "out_full", "out_step")]


class archer_step_desc(ctypes.Structure):
    _fields_ = [("shape", archer_shape), ("n_layers", ctypes.c_int), ("layers", ctypes.POINTER(archer_layer_io)),
                ("g_cur", ctypes.c_void_p), ("g_anchor", ctypes.c_void_p), ("age", ctypes.c_void_p),
                ("K", ctypes.c_int), ("max_age", ctypes.c_int), ("dist_out", ctypes.c_void_p),
                ("flag_out", ctypes.c_void_p), ("refresh_count", ctypes.c_void_p),
                ("vocab", ctypes.c_int), ("logits_dtype", ctypes.c_int), ("logits", ctypes.c_void_p),
                ("row_stride", ctypes.c_int64), ("mask_state", ctypes.c_void_p), ("cur_tokens", ctypes.c_void_p),
                ("max_prob", ctypes.c_void_p), ("top1", ctypes.c_void_p), ("margin", ctypes.c_void_p),
                ("cur_prob", ctypes.c_void_p), ("scores_workspace", ctypes.c_void_p),
                ("scores_workspace_bytes", ctypes.c_size_t), ("attn_workspace", ctypes.c_void_p),
                ("attn_workspace_bytes", ctypes.c_size_t)]


class archer_attn_plan(ctypes.Structure):
    _fields_ = [("kernel", ctypes.c_int), ("tiles_per_cta", ctypes.c_int), ("n_split", ctypes.c_int),
                ("key_tiles_per_split", ctypes.c_int), ("work_items", ctypes.c_int), ("grid", ctypes.c_int),
                ("single_tail", ctypes.c_int), ("split_workspace", ctypes.c_size_t)]


ARCHER_PLAN_ATTN_STEP, ARCHER_PLAN_REFRESH_ALL, ARCHER_PLAN_REFRESH_FLAGS = 0, 1, 2
ARCHER_KERNEL_TWO_TILE, ARCHER_KERNEL_ONE_TILE, ARCHER_KERNEL_PERSISTENT = 0, 1, 2


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"{LIB_PATH} is missing: build it with paper_2608_08086_gb300.build.build() "
                          "(there is no CPU fallback)")
    L = ctypes.CDLL(LIB_PATH)
    vp, i, sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t
    sp = ctypes.POINTER(archer_shape)
    L.archer_attn_step.argtypes = [sp, vp, vp, vp, vp, vp, vp, vp, vp, sz, vp]
    L.archer_prompt_refresh.argtypes = [sp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, sz, vp]
    L.archer_attn_plan_query.argtypes = [sp, i, sz, i, ctypes.POINTER(archer_attn_plan)]
    L.archer_attn_workspace_size.argtypes = [sp, i]
    L.archer_attn_workspace_size.restype = sz
    L.archer_decode_scores.argtypes = [i, i, i, i, vp, ctypes.c_int64, vp, vp, vp, vp, vp, vp, vp, sz, vp]
    L.archer_decode_scores_workspace_size.argtypes = [i, i]
    L.archer_decode_scores_workspace_size.restype = sz
    L.archer_should_refresh.argtypes = [i, i, vp, vp, vp, i, i, i, vp, vp, vp]
    L.archer_cache_rewrite.argtypes = [sp, vp, vp, vp, vp, vp, vp]
    L.archer_scatter_rows.argtypes = [i, i, i, sz, vp, vp, vp, i, i, vp, i, i, vp]
    L.archer_decoder_update.argtypes = [i, i, ctypes.c_float, ctypes.c_float, ctypes.c_int32, vp, vp, vp, vp, vp,
                                        vp]
    L.archer_check_device.argtypes = [vp]
    L.archer_debug_stall_attention.argtypes = [i]
    L.archer_status_string.argtypes = [i]
    L.archer_status_string.restype = ctypes.c_char_p
    L.archer_last_error.argtypes = []
    L.archer_last_error.restype = ctypes.c_char_p
    L.archer_version.argtypes = []
    L.archer_step_graph_create.argtypes = [ctypes.POINTER(archer_step_desc), ctypes.POINTER(vp)]
    L.archer_step_graph_launch.argtypes = [vp, vp]
    L.archer_step_graph_destroy.argtypes = [vp]
    for name in ("archer_attn_step", "archer_prompt_refresh", "archer_decode_scores", "archer_should_refresh",
                 "archer_cache_rewrite", "archer_check_device", "archer_version", "archer_step_graph_create",
                 "archer_decoder_update", "archer_scatter_rows", "archer_attn_plan_query",
                 "archer_step_graph_launch", "archer_step_graph_destroy", "archer_debug_stall_attention"):
        getattr(L, name).restype = ctypes.c_int
    return L


lib = _load()


def _raise(status: int):
    if status != ARCHER_OK:
        raise ArcherError(status, f"{lib.archer_status_string(status).decode()}: {lib.archer_last_error().decode()}")


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream))


def _ptr(t, dtype=None, what=""):
    if t is None:
        return None
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{what} must be a CUDA tensor")
    if dtype is not None and t.dtype != dtype:
        raise TypeError(f"{what} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{what} must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


def make_shape(batch, prompt_len, resp_len, n_heads, n_kv_heads, head_dim, softmax_scale=None):
    s = archer_shape()
    s.batch, s.prompt_len, s.resp_len = int(batch), int(prompt_len), int(resp_len)
    s.n_heads, s.n_kv_heads, s.head_dim = int(n_heads), int(n_kv_heads), int(head_dim)
    s.softmax_scale = float(softmax_scale) if softmax_scale else 0.0
    return s


def _expect(t, shape, what):
    if tuple(t.shape) != tuple(shape):
        raise ValueError(f"{what} has shape {tuple(t.shape)}, expected {tuple(shape)}")


_attn_ws_cache: dict = {}


def attn_workspace(shape: archer_shape, n_queries: int, device=None) -> torch.Tensor | None:
    """A split-KV workspace for launches over n_queries rows, cached per
    (device, size); None when the launch would not split.  Calls that may
    overlap on the GPU must not share one."""
    n = int(lib.archer_attn_workspace_size(ctypes.byref(shape), int(n_queries)))
    if n == 0:
        return None
    dev = torch.device("cuda", torch.cuda.current_device()) if device is None else torch.device(device)
    key = (dev, n)
    if key not in _attn_ws_cache:
        _attn_ws_cache[key] = torch.empty(n, dtype=torch.uint8, device=dev)
    return _attn_ws_cache[key]


def archer_attn_step(shape: archer_shape, q_resp, k_cache, v_cache, k_resp, v_resp, out, lse=None,
                     workspace=None, stream=None):
    """Cached response step (Sec. 4.1, Eq. archer-attention); see include/archer.h."""
    B, P, G, Hq, Hkv, D = (shape.batch, shape.prompt_len, shape.resp_len, shape.n_heads, shape.n_kv_heads,
                           shape.head_dim)
    bf = torch.bfloat16
    _expect(q_resp, (B, G, Hq, D), "q_resp")
    _expect(k_resp, (B, G, Hkv, D), "k_resp")
    _expect(v_resp, (B, G, Hkv, D), "v_resp")
    _expect(out, (B, G, Hq, D), "out")
    if P > 0:
        _expect(k_cache, (B, P, Hkv, D), "k_cache")
        _expect(v_cache, (B, P, Hkv, D), "v_cache")
    if lse is not None:
        _expect(lse, (B, Hq, G), "lse")
    ws = attn_workspace(shape, G, q_resp.device) if workspace is None else workspace
    if ws is False:
        ws = None
    _raise(lib.archer_attn_step(ctypes.byref(shape), _ptr(q_resp, bf, "q_resp"), _ptr(k_cache, bf, "k_cache"),
                                _ptr(v_cache, bf, "v_cache"), _ptr(k_resp, bf, "k_resp"), _ptr(v_resp, bf, "v_resp"),
                                _ptr(out, bf, "out"), _ptr(lse, torch.float32, "lse"), _ptr(ws, None, "workspace"),
                                ctypes.c_size_t(0 if ws is None else ws.numel() * ws.element_size()),
                                _stream(stream)))


def archer_prompt_refresh(shape: archer_shape, q_all, k_prompt_new, v_prompt_new, k_resp, v_resp, out,
                          lse=None, k_cache=None, v_cache=None, refresh_flags=None, workspace=None, stream=None):
    """Prompt refresh (Sec. 4.2, Algorithm 1's FullForward); see include/archer.h."""
    B, P, G, Hq, Hkv, D = (shape.batch, shape.prompt_len, shape.resp_len, shape.n_heads, shape.n_kv_heads,
                           shape.head_dim)
    N = P + G
    bf = torch.bfloat16
    _expect(q_all, (B, N, Hq, D), "q_all")
    _expect(k_resp, (B, G, Hkv, D), "k_resp")
    _expect(v_resp, (B, G, Hkv, D), "v_resp")
    _expect(out, (B, N, Hq, D), "out")
    if k_cache is None:
        k_cache = k_prompt_new
    if v_cache is None:
        v_cache = v_prompt_new
    if P > 0:
        for t, n in ((k_prompt_new, "k_prompt_new"), (v_prompt_new, "v_prompt_new"), (k_cache, "k_cache"),
                     (v_cache, "v_cache")):
            _expect(t, (B, P, Hkv, D), n)
    if lse is not None:
        _expect(lse, (B, Hq, N), "lse")
    if refresh_flags is not None:
        _expect(refresh_flags, (B,), "refresh_flags")
    ws = attn_workspace(shape, N, q_all.device) if workspace is None else workspace
    if ws is False:
        ws = None
    _raise(lib.archer_prompt_refresh(
        ctypes.byref(shape), _ptr(q_all, bf, "q_all"), _ptr(k_prompt_new, bf, "k_prompt_new"),
        _ptr(v_prompt_new, bf, "v_prompt_new"), _ptr(k_resp, bf, "k_resp"), _ptr(v_resp, bf, "v_resp"),
        _ptr(out, bf, "out"), _ptr(lse, torch.float32, "lse"), _ptr(k_cache, bf, "k_cache"),
        _ptr(v_cache, bf, "v_cache"), _ptr(refresh_flags, torch.uint8, "refresh_flags"), _ptr(ws, None, "workspace"),
        ctypes.c_size_t(0 if ws is None else ws.numel() * ws.element_size()), _stream(stream)))


def archer_attn_plan_query(shape: archer_shape, op: int = ARCHER_PLAN_ATTN_STEP, ws_bytes: int = 0,
                           sm_count: int = 0) -> dict:
    """The launch an attention call makes (kernel, split, grid); with
    sm_count > 0 host arithmetic only, no GPU needed."""
    plan = archer_attn_plan()
    _raise(lib.archer_attn_plan_query(ctypes.byref(shape), int(op), ctypes.c_size_t(int(ws_bytes)), int(sm_count),
                                      ctypes.byref(plan)))
    return {name: int(getattr(plan, name)) for name, _ in archer_attn_plan._fields_}


def archer_attn_workspace_size(shape: archer_shape, n_queries: int) -> int:
    return int(lib.archer_attn_workspace_size(ctypes.byref(shape), int(n_queries)))


def archer_decode_scores_workspace_size(rows: int, vocab: int) -> int:
    return int(lib.archer_decode_scores_workspace_size(int(rows), int(vocab)))


_ws_cache: dict = {}


def scores_workspace(rows: int, vocab: int, device=None) -> torch.Tensor | None:
    """A zero-filled workspace for archer_decode_scores, cached per (device, size).
    Calls that may overlap on the GPU must not share one."""
    n = archer_decode_scores_workspace_size(rows, vocab)
    if n == 0:
        return None
    dev = torch.device("cuda", torch.cuda.current_device()) if device is None else torch.device(device)
    key = (dev, n)
    if key not in _ws_cache:
        _ws_cache[key] = torch.zeros(n, dtype=torch.uint8, device=dev)
    return _ws_cache[key]


def archer_decode_scores(logits, max_prob, top1, margin, mask_state=None, cur_tokens=None, cur_prob=None,
                         vocab=None, workspace=None, stream=None):
    """Decoder scoring; logits [B, G, row_stride] or [rows, row_stride] (bf16 or fp32).
    Outputs are flat [rows] tensors (fp32, int32, fp32, fp32)."""
    if logits.dtype == torch.bfloat16:
        dtype = ARCHER_DTYPE_BF16
    elif logits.dtype == torch.float32:
        dtype = ARCHER_DTYPE_F32
    else:
        raise TypeError("logits must be bf16 or fp32")
    if logits.dim() == 3:
        batch, resp_len, stride = logits.shape
    elif logits.dim() == 2:
        batch, (resp_len, stride) = 1, logits.shape
    else:
        raise ValueError("logits must be [B, G, V] or [rows, V]")
    vocab = stride if vocab is None else int(vocab)
    rows = batch * resp_len
    for t, n, dt in ((max_prob, "max_prob", torch.float32), (top1, "top1", torch.int32),
                     (margin, "margin", torch.float32)):
        if t.numel() != rows or t.dtype != dt:
            raise ValueError(f"{n} must hold {rows} {dt} values")
    if cur_prob is not None and (cur_prob.numel() != rows or cur_prob.dtype != torch.float32):
        raise ValueError("cur_prob must hold rows fp32 values")
    for t, n in ((mask_state, "mask_state"), (cur_tokens, "cur_tokens")):
        if t is not None and t.numel() != rows:
            raise ValueError(f"{n} must hold {rows} values")
    if workspace is None:
        workspace = scores_workspace(rows, vocab, logits.device)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _raise(lib.archer_decode_scores(
        batch, resp_len, vocab, dtype, _ptr(logits, None, "logits"), ctypes.c_int64(stride),
        _ptr(mask_state, torch.uint8, "mask_state"), _ptr(cur_tokens, torch.int32, "cur_tokens"),
        _ptr(max_prob, None, "max_prob"), _ptr(top1, None, "top1"), _ptr(margin, None, "margin"),
        _ptr(cur_prob, None, "cur_prob"), _ptr(workspace, None, "workspace"), ctypes.c_size_t(ws_bytes),
        _stream(stream)))


def archer_should_refresh(g_cur, g_anchor, age, K, max_age, update_anchor, dist_out, flag_out, stream=None):
    """Refresh rule (Sec. 4.2, Eq. archer-distance / archer-controller); see include/archer.h."""
    B, G = g_cur.shape
    _expect(g_anchor, (B, G), "g_anchor")
    _expect(age, (B,), "age")
    _expect(flag_out, (B,), "flag_out")
    if dist_out is not None:
        _expect(dist_out, (B,), "dist_out")
    i32 = torch.int32
    _raise(lib.archer_should_refresh(B, G, _ptr(g_cur, i32, "g_cur"), _ptr(g_anchor, i32, "g_anchor"),
                                     _ptr(age, i32, "age"), int(min(K, K_INFINITE)), int(max_age),
                                     int(bool(update_anchor)), _ptr(dist_out, i32, "dist_out"),
                                     _ptr(flag_out, torch.uint8, "flag_out"), _stream(stream)))


def archer_decoder_update(g, max_prob, top1, cur_prob, changed, tau_accept, tau_remask, mask_token=-1,
                          stream=None):
    """Synthetic rollback decoder (stand-in for D); see include/archer.h."""
    B, G = g.shape
    _expect(changed, (B, G), "changed")
    for t, n, dt in ((max_prob, "max_prob", torch.float32), (top1, "top1", torch.int32),
                     (cur_prob, "cur_prob", torch.float32)):
        if t.numel() != B * G or t.dtype != dt:
            raise ValueError(f"{n} must hold {B * G} {dt} values")
    _raise(lib.archer_decoder_update(B, G, float(tau_accept), float(tau_remask), int(mask_token),
                                     _ptr(max_prob, None, "max_prob"), _ptr(top1, None, "top1"),
                                     _ptr(cur_prob, None, "cur_prob"), _ptr(g, torch.int32, "g"),
                                     _ptr(changed, torch.uint8, "changed"), _stream(stream)))


def archer_scatter_rows(src, pos, dst0, dst0_row0=0, dst1=None, dst1_row0=0, stream=None):
    """Row scatter (see include/archer.h): src [O, B, n, *row], pos [B, n] int64,
    dst [O, B, rows, *row] (same row shape); rows of dst0 / dst1 start at
    dst*_row0."""
    O, B, n = src.shape[:3]
    row = src[0, 0, 0].numel() * src.element_size() if src.numel() else 0
    for d, name in ((dst0, "dst0"), (dst1, "dst1")):
        if d is not None and (tuple(d.shape[:2]) != (O, B) or d[0, 0, 0].numel() * d.element_size() != row):
            raise ValueError(f"{name} must be [O, B, rows, ...] with src's row size")
    _expect(pos, (B, n), "pos")
    _raise(lib.archer_scatter_rows(
        O, B, n, ctypes.c_size_t(row), _ptr(src, None, "src"), _ptr(pos, torch.int64, "pos"),
        _ptr(dst0, None, "dst0"), dst0.shape[2], int(dst0_row0), _ptr(dst1, None, "dst1"),
        0 if dst1 is None else dst1.shape[2], int(dst1_row0), _stream(stream)))


def archer_cache_rewrite(shape: archer_shape, k_src, v_src, k_dst, v_dst, refresh_flags=None, stream=None):
    """Copy each flagged sequence's prompt K/V [B, P, Hkv, D] (bf16) from src to
    dst (all four tensors required; flags None = every sequence); see
    include/archer.h."""
    want = (shape.batch, shape.prompt_len, shape.n_kv_heads, shape.head_dim)
    for t, n in ((k_src, "k_src"), (v_src, "v_src"), (k_dst, "k_dst"), (v_dst, "v_dst")):
        if t is not None:
            _expect(t, want, n)
    if refresh_flags is not None:
        _expect(refresh_flags, (shape.batch,), "refresh_flags")
    bf = torch.bfloat16
    _raise(lib.archer_cache_rewrite(ctypes.byref(shape), _ptr(k_src, bf, "k_src"), _ptr(v_src, bf, "v_src"),
                                    _ptr(k_dst, bf, "k_dst"), _ptr(v_dst, bf, "v_dst"),
                                    _ptr(refresh_flags, torch.uint8, "refresh_flags"), _stream(stream)))


def archer_check_device(stream=None):
    _raise(lib.archer_check_device(_stream(stream)))


def archer_debug_stall_attention(on: bool) -> bool:
    """Test hook: attention launches withhold their last P V product while on
    (their bounded wait expires; archer_check_device reports the timeout).
    Returns the previous setting."""
    return bool(lib.archer_debug_stall_attention(int(bool(on))))


def archer_version() -> int:
    return int(lib.archer_version())


def default_scale(head_dim: int) -> float:
    return 1.0 / math.sqrt(head_dim)


class StepGraph:
    """One denoising step of Algorithm 1 over an L-layer stack as a CUDA graph
    (archer_step_graph_create): rule, device-side refresh branch, L attention
    layers, scoring.  Every tensor given here is captured by address: keep
    them alive and write each step's inputs into them in place."""

    def __init__(self, shape: archer_shape, layers, g_cur, g_anchor, age, K, max_age, flag_out, dist_out=None,
                 refresh_count=None, logits=None, max_prob=None, top1=None, margin=None, vocab=None,
                 mask_state=None, cur_tokens=None, cur_prob=None, workspace=None):
        bf = torch.bfloat16
        B, G = g_cur.shape
        if B != shape.batch or G != shape.resp_len:
            raise ValueError("g_cur must be [batch, resp_len]")
        # the graph holds raw addresses: every size is checked here, before capture
        P, Hq, Hkv, D = shape.prompt_len, shape.n_heads, shape.n_kv_heads, shape.head_dim
        N = P + G
        want = {"q_all": (B, N, Hq, D), "q_resp": (B, G, Hq, D), "k_prompt_new": (B, P, Hkv, D),
                "v_prompt_new": (B, P, Hkv, D), "k_resp": (B, G, Hkv, D), "v_resp": (B, G, Hkv, D),
                "k_cache": (B, P, Hkv, D), "v_cache": (B, P, Hkv, D), "out_full": (B, N, Hq, D),
                "out_step": (B, G, Hq, D)}
        for i, l in enumerate(layers):
            for name, shp in want.items():
                _expect(l[name], shp, f"layers[{i}].{name}")
        for t, n in ((g_anchor, "g_anchor"), (age, "age"), (flag_out, "flag_out"), (dist_out, "dist_out"),
                     (refresh_count, "refresh_count")):
            if t is not None:
                _expect(t, (B, G) if n == "g_anchor" else ((1,) if n == "refresh_count" else (B,)), n)
        if logits is not None:
            for t, n in ((max_prob, "max_prob"), (top1, "top1"), (margin, "margin"), (cur_prob, "cur_prob"),
                         (mask_state, "mask_state"), (cur_tokens, "cur_tokens")):
                if t is not None and t.numel() != B * G:
                    raise ValueError(f"{n} must hold {B * G} values")
        self._keep = []            # tensors whose addresses the graph holds
        ios = (archer_layer_io * len(layers))()
        for i, l in enumerate(layers):
            for name in archer_layer_io._fields_:
                t = l[name[0]]
                self._keep.append(t)
                setattr(ios[i], name[0], _ptr(t, bf, name[0]))
        d = archer_step_desc()
        d.shape = shape
        d.n_layers = len(layers)
        d.layers = ios
        i32 = torch.int32
        d.g_cur, d.g_anchor, d.age = _ptr(g_cur, i32, "g_cur"), _ptr(g_anchor, i32, "g_anchor"), _ptr(age, i32, "age")
        d.K, d.max_age = int(min(K, K_INFINITE)), int(max_age)
        d.dist_out = _ptr(dist_out, i32, "dist_out")
        d.flag_out = _ptr(flag_out, torch.uint8, "flag_out")
        d.refresh_count = _ptr(refresh_count, i32, "refresh_count")
        self._keep += [g_cur, g_anchor, age, flag_out, dist_out, refresh_count]
        if logits is not None:
            if logits.dtype not in (torch.bfloat16, torch.float32):
                raise TypeError("logits must be bf16 or fp32")
            stride = logits.shape[-1]
            if logits.numel() != B * G * stride:
                raise ValueError("logits must hold batch * resp_len rows")
            d.vocab = stride if vocab is None else int(vocab)
            d.logits_dtype = ARCHER_DTYPE_BF16 if logits.dtype == torch.bfloat16 else ARCHER_DTYPE_F32
            d.logits, d.row_stride = _ptr(logits, None, "logits"), stride
            d.mask_state = _ptr(mask_state, torch.uint8, "mask_state")
            d.cur_tokens = _ptr(cur_tokens, i32, "cur_tokens")
            d.max_prob, d.top1 = _ptr(max_prob, torch.float32, "max_prob"), _ptr(top1, i32, "top1")
            d.margin, d.cur_prob = _ptr(margin, torch.float32, "margin"), _ptr(cur_prob, torch.float32, "cur_prob")
            if workspace is None:
                workspace = scores_workspace(B * G, d.vocab, logits.device)
            d.scores_workspace = _ptr(workspace, None, "workspace")
            d.scores_workspace_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
            self._keep += [logits, mask_state, cur_tokens, max_prob, top1, margin, cur_prob, workspace]
        # one scratch for every layer: the larger of the refresh and cached launches' needs
        sizes = [int(lib.archer_attn_workspace_size(ctypes.byref(shape), m))
                 for m in (shape.prompt_len + shape.resp_len, shape.resp_len)]
        aws = attn_workspace(shape, (shape.prompt_len + shape.resp_len, shape.resp_len)[sizes.index(max(sizes))],
                             g_cur.device)
        if aws is not None:
            d.attn_workspace, d.attn_workspace_bytes = _ptr(aws, None, "attn_workspace"), aws.numel()
            self._keep.append(aws)
        h = ctypes.c_void_p()
        _raise(lib.archer_step_graph_create(ctypes.byref(d), ctypes.byref(h)))
        self._h = h

    def launch(self, stream=None):
        _raise(lib.archer_step_graph_launch(self._h, _stream(stream)))

    def close(self):
        if getattr(self, "_h", None):
            torch.cuda.synchronize()
            lib.archer_step_graph_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
