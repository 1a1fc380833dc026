"""Algorithm 1 (state-anchored rollback decoding) driven through the C ABI.

The rollback decoder D is replaced by the seeded redraw of ``synth`` (a fixed
number of response positions per sequence get a new token and new Q/K/V rows
in every layer each step).  Per step t:

  1. stage the redraw (token ids and Q/K/V rows)           -- stands in for D
  2. archer_should_refresh: D_t = d_H(g_t, g_r), flag = D_t >= K or age_t >= max_age;
     flagged sequences take g_r <- g_t, age <- 0 (Sec. 4.2, Eq. archer-controller)
  3. the flags are read back to the host (one 1-byte-per-sequence copy)
  4. per layer: archer_prompt_refresh (if any flag; per-sequence flags, prompt
     cache rewritten) or archer_attn_step (Eq. archer-cached)
  5. archer_decode_scores over the step's logits.
Step 0 is the FullForward that builds every layer's prompt cache.
``mode="eager"`` refreshes every step (K = 0), the full-recomputation comparator.
``mode="graph"`` ("eager-graph") runs the same rule as "archer" ("eager") but each step after the build is
one replay of an archer_step_graph (rule, device-side refresh branch, layers,
scoring): the host never reads the flags to decide, so steps queue back to
back.

Per-layer buffers are slices of stacked tensors so that one indexed copy
stages a redraw for all layers.  With ``source="host"`` every input comes
from the host generator of ``synth`` (bit-identical to what the oracle sees);
with ``source="device"`` inputs are drawn on the GPU once, and redraw rows come
from a pre-drawn pool (cycled), so that all inputs are resident in HBM.
"""
from __future__ import annotations

import math

import numpy as np
import torch

from . import archer as A
from . import synth


def _dev_bits(bits, device):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).to(device)


class DeviceTrajectory:
    def __init__(self, wl: synth.Workload, seed: int = 0, mode: str = "archer", source: str = "host",
                 device="cuda", layers: int | None = None, score: bool = True, pool_steps: int = 8,
                 max_steps: int | None = None, record: bool = False, decoder: str = "redraw",
                 closed_loop: dict | None = None):
        self.wl, self.seed, self.mode, self.source = wl, seed, mode, source
        self.device = torch.device(device)
        sh = wl.shape
        self.B, self.P, self.G = sh.batch, sh.prompt_len, sh.resp_len
        self.Hq, self.Hkv, self.D = sh.n_heads, sh.n_kv_heads, sh.head_dim
        self.N = self.P + self.G
        self.L = wl.layers if layers is None else layers
        if mode not in ("archer", "eager", "graph", "eager-graph"):
            raise ValueError(f"unknown mode {mode}")
        self.graph_mode = mode in ("graph", "eager-graph")
        if decoder not in ("redraw", "closed") or (decoder == "closed" and source != "host"):
            raise ValueError("decoder is 'redraw' or 'closed' (closed: host source only)")
        self.closed = decoder == "closed"
        self.cl = dict(synth.CLOSED_LOOP, **(closed_loop or {}))
        eager = mode in ("eager", "eager-graph")
        self.K = 0 if eager else wl.radius_k
        self.max_age = 0 if eager else wl.max_age
        self.score = score and wl.logits_rows > 0
        self.record = record
        self.shape = A.make_shape(self.B, self.P, self.G, self.Hq, self.Hkv, self.D)
        self.pool_steps = pool_steps
        self.max_steps = wl.steps if max_steps is None else max_steps
        self._n_refresh_steps = 0
        self.graph = None
        self.t = -1
        self.attn_events = []          # (start, end, kind, launches): CUDA events around a step's layer loop
                                       # (its launches back to back, as in the untimed step) or a scoring call
        self.time_attention = False
        self.layer_ready = None        # optional per-layer CUDA events a refresh layer waits on
        self._alloc()

    # ------------------------------------------------------------------ setup
    def _alloc(self):
        B, P, G, N, Hq, Hkv, D, L = self.B, self.P, self.G, self.N, self.Hq, self.Hkv, self.D, self.L
        dev, bf = self.device, torch.bfloat16
        std = 1.0 / math.sqrt(D)
        if self.source == "host":
            g0 = synth.traj_initial_tokens(self.wl, self.seed)
            if self.closed:
                g0 = np.full((B, G), synth.MASK_TOKEN, dtype=np.int32)
            init = [synth.traj_layer_initial(self.wl, self.seed, layer) for layer in range(L)]
            self.q_all = torch.stack([_dev_bits(x["q_all"], dev) for x in init])
            self.k_resp = torch.stack([_dev_bits(x["k_resp"], dev) for x in init])
            self.v_resp = torch.stack([_dev_bits(x["v_resp"], dev) for x in init])
            self.k_new = torch.stack([_dev_bits(x["k_new"], dev) for x in init])
            self.v_new = torch.stack([_dev_bits(x["v_new"], dev) for x in init])
            self.g_host = g0.copy()
        else:
            tag = ("traj-dev", self.seed)
            self.q_all = synth.device_normal(tag + ("q",), (L, B, N, Hq, D), std, dev)
            self.k_resp = synth.device_normal(tag + ("kg",), (L, B, G, Hkv, D), std, dev)
            self.v_resp = synth.device_normal(tag + ("vg",), (L, B, G, Hkv, D), std, dev)
            self.k_new = synth.device_normal(tag + ("kp",), (L, B, P, Hkv, D), std, dev)
            self.v_new = synth.device_normal(tag + ("vp",), (L, B, P, Hkv, D), std, dev)
            self.g_host = synth.traj_initial_tokens(self.wl, self.seed)
            n = self.wl.redraws_per_step
            self.pool = {
                "q": synth.device_normal(tag + ("pool-q",), (self.pool_steps, L, B, n, Hq, D), std, dev),
                "k": synth.device_normal(tag + ("pool-k",), (self.pool_steps, L, B, n, Hkv, D), std, dev),
                "v": synth.device_normal(tag + ("pool-v",), (self.pool_steps, L, B, n, Hkv, D), std, dev),
            }
            # the token trajectory is cheap: plan it on the host for every step
            self.plan = []
            g = self.g_host.copy()
            for t in range(1, self.max_steps + 1):
                pos, new = synth.traj_redraw(self.wl, self.seed, t, g)
                g[np.arange(B)[:, None], pos] = new
                self.plan.append((torch.from_numpy(pos).to(dev), torch.from_numpy(new).to(dev)))
        self.q_resp = self.q_all[:, :, P:].contiguous()
        self.k_cache = torch.zeros_like(self.k_new)
        self.v_cache = torch.zeros_like(self.v_new)
        self.g = torch.from_numpy(self.g_host).to(dev)
        self.g_anchor = self.g.clone()
        self.age = torch.zeros(B, dtype=torch.int32, device=dev)
        self.dist = torch.zeros(B, dtype=torch.int32, device=dev)
        self.flag = torch.ones(B, dtype=torch.uint8, device=dev)
        self.flag_host = torch.ones(B, dtype=torch.uint8).pin_memory()
        self.out_step = torch.empty(B, G, Hq, D, dtype=bf, device=dev)
        self.out_full = torch.empty(B, N, Hq, D, dtype=bf, device=dev)
        self.refresh_count = torch.zeros(1, dtype=torch.int32, device=dev)
        if self.score:
            rows, V = B * G, self.wl.vocab
            if self.source == "host" and self.graph_mode:
                dt = torch.bfloat16 if self.wl.logits_dtype == "bf16" else torch.float32
                self.logits = torch.empty(rows, V, dtype=dt, device=dev)   # fixed: the graph holds its address
            elif self.source == "host":
                self.logits = None
            else:
                dt = torch.bfloat16 if self.wl.logits_dtype == "bf16" else torch.float32
                self.logits = synth.device_logits(rows, V, dev, seed=self.seed, std=self.wl.logits_std,
                                                  boost_max=self.wl.logits_boost, dtype=dt)
            self.max_prob = torch.empty(rows, dtype=torch.float32, device=dev)
            self.top1 = torch.empty(rows, dtype=torch.int32, device=dev)
            self.margin = torch.empty(rows, dtype=torch.float32, device=dev)
            if self.closed:
                self.cur_prob = torch.empty(rows, dtype=torch.float32, device=dev)
                self.mask_state = (self.g == synth.MASK_TOKEN).to(torch.uint8)
                self.changed = torch.zeros(B, G, dtype=torch.uint8, device=dev)
            self.ws = A.scores_workspace(rows, V, dev)

    # ------------------------------------------------------------------ pieces
    def _timed(self, kind, fn, launches=1):
        if not self.time_attention:
            fn()
            return
        s, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        s.record()
        fn()
        e.record()
        self.attn_events.append((s, e, kind, launches))

    def _forward(self, refresh: bool, flags):
        outs = []

        def layers():
            for layer in range(self.L):
                if refresh:
                    if self.layer_ready is not None:
                        torch.cuda.current_stream().wait_event(self.layer_ready[layer])
                    A.archer_prompt_refresh(
                        self.shape, self.q_all[layer], self.k_new[layer], self.v_new[layer], self.k_resp[layer],
                        self.v_resp[layer], self.out_full, None, self.k_cache[layer], self.v_cache[layer],
                        refresh_flags=flags)
                    if self.record:
                        outs.append(self.out_full.clone())
                else:
                    A.archer_attn_step(
                        self.shape, self.q_resp[layer], self.k_cache[layer], self.v_cache[layer], self.k_resp[layer],
                        self.v_resp[layer], self.out_step)
                    if self.record:
                        outs.append(self.out_step.clone())

        # one event pair around the step's L launches: an event between two
        # launches would keep the second from starting while the first ends
        self._timed("refresh" if refresh else "step", layers, self.L)
        return outs

    def _score(self, t):
        if not self.score:
            return None
        self._upload_logits(t)
        if self.closed:
            self._timed("score", lambda: A.archer_decode_scores(
                self.logits, self.max_prob, self.top1, self.margin, mask_state=self.mask_state, cur_tokens=self.g,
                cur_prob=self.cur_prob, workspace=self.ws))
        else:
            self._timed("score", lambda: A.archer_decode_scores(self.logits, self.max_prob, self.top1, self.margin,
                                                                workspace=self.ws))
        if self.record:
            sc = {"max_prob": self.max_prob.clone(), "top1": self.top1.clone(), "margin": self.margin.clone()}
            if self.closed:
                sc["cur_prob"] = self.cur_prob.clone()
            return sc
        return None

    def _upload_logits(self, t):
        if self.source != "host":
            return
        if self.closed:
            z = synth.closed_loop_logits(self.wl, self.seed, t, self.cl["boost_per_step"])
        else:
            z = synth.traj_logits(self.wl, self.seed, t)
        z = _dev_bits(z, self.device) if self.wl.logits_dtype == "bf16" else torch.from_numpy(z).to(self.device)
        if self.graph_mode:
            self.logits.copy_(z)
        else:
            self.logits = z

    def _closed_loop_decode(self, t):
        # D: the confidence rule on the previous step's scores, on the device;
        # every position's candidate rows are uploaded, the changed ones kept
        A.archer_decoder_update(self.g, self.max_prob, self.top1, self.cur_prob, self.changed,
                                self.cl["tau_accept"], self.cl["tau_remask"], synth.MASK_TOKEN)
        self.mask_state.copy_((self.g == synth.MASK_TOKEN).to(torch.uint8))
        ch = self.changed.bool()[:, :, None, None]
        P = self.P
        for layer in range(self.L):
            rows = synth.closed_loop_rows(self.wl, self.seed, t, layer)
            q, k, v = (_dev_bits(rows[c], self.device) for c in ("q", "k", "v"))
            self.q_resp[layer].copy_(torch.where(ch, q, self.q_resp[layer]))
            self.q_all[layer][:, P:] = torch.where(ch, q, self.q_all[layer][:, P:])
            self.k_resp[layer].copy_(torch.where(ch, k, self.k_resp[layer]))
            self.v_resp[layer].copy_(torch.where(ch, v, self.v_resp[layer]))

    def _stage_redraw(self, t):
        if self.closed:
            return self._closed_loop_decode(t)
        B, P = self.B, self.P
        if self.wl.redraws_per_step == 0:
            return
        bidx = torch.arange(B, device=self.device)[:, None]
        if self.source == "host":
            pos, new = synth.traj_redraw(self.wl, self.seed, t, self.g_host)
            self.g_host[np.arange(B)[:, None], pos] = new
            pos_d = torch.from_numpy(pos).to(self.device)
            self.g[bidx, pos_d] = torch.from_numpy(new).to(self.device)
            rows = [synth.traj_redraw_rows(self.wl, self.seed, t, layer) for layer in range(self.L)]
            q, k, v = (torch.stack([_dev_bits(r[c], self.device) for r in rows]) for c in ("q", "k", "v"))
        else:
            pos_d, new_d = self.plan[(t - 1) % len(self.plan)]
            self.g[bidx, pos_d] = new_d
            slot = (t - 1) % self.pool_steps
            q, k, v = self.pool["q"][slot], self.pool["k"][slot], self.pool["v"][slot]
        self._scatter(q, k, v, pos_d)

    def _scatter(self, q, k, v, pos_d):
        # new rows of the redrawn positions into every layer's tensors: Q into the
        # cached step's and the refresh pass's query tensors, K and V into the
        # response K/V (one native scatter launch each)
        A.archer_scatter_rows(q, pos_d, self.q_resp, 0, self.q_all, self.P)
        A.archer_scatter_rows(k, pos_d, self.k_resp)
        A.archer_scatter_rows(v, pos_d, self.v_resp)

    def _stage_fresh_prompt(self, t):
        # Fresh prompt Q/K/V for a refresh (the model's prompt states under g_t).
        if self.source != "host":
            return            # device source: the resident fresh-prompt tensors stand in
        for layer in range(self.L):
            fp = synth.traj_fresh_prompt(self.wl, self.seed, t, layer)
            self.q_all[layer][:, :self.P] = _dev_bits(fp["q_prompt"], self.device)
            self.k_new[layer].copy_(_dev_bits(fp["k_new"], self.device))
            self.v_new[layer].copy_(_dev_bits(fp["v_new"], self.device))

    # ------------------------------------------------------------------ steps
    def build(self):
        """Step 0: FullForward in every layer builds the prompt cache; then score."""
        self.t = 0
        self.flag.fill_(1)
        outs = self._forward(True, None)
        self.g_anchor.copy_(self.g)
        self.age.zero_()
        sc = self._score(0)
        self._n_refresh_steps = 1
        return {"t": 0, "flag": np.ones(self.B, np.uint8), "dist": np.zeros(self.B, np.int32), "out": outs,
                "scores": sc}

    @property
    def n_refresh_steps(self):
        """Steps that refreshed (the build included); a device read in graph mode."""
        if self.graph_mode and self.graph is not None:
            return 1 + int(self.refresh_count.item())
        return self._n_refresh_steps

    def _make_graph(self):
        layers = [{"q_all": self.q_all[l], "q_resp": self.q_resp[l], "k_prompt_new": self.k_new[l],
                   "v_prompt_new": self.v_new[l], "k_resp": self.k_resp[l], "v_resp": self.v_resp[l],
                   "k_cache": self.k_cache[l], "v_cache": self.v_cache[l], "out_full": self.out_full,
                   "out_step": self.out_step} for l in range(self.L)]
        sc = {}
        if self.score:
            sc = dict(logits=self.logits, max_prob=self.max_prob, top1=self.top1, margin=self.margin,
                      workspace=self.ws)
            if self.closed:
                sc.update(mask_state=self.mask_state, cur_tokens=self.g, cur_prob=self.cur_prob)
        self.refresh_count.zero_()
        self.graph = A.StepGraph(self.shape, layers, self.g, self.g_anchor, self.age, self.K, self.max_age,
                                 self.flag, dist_out=self.dist, refresh_count=self.refresh_count, **sc)

    def _graph_step(self, t):
        self._stage_redraw(t)
        self._stage_fresh_prompt(t)       # host source: the graph may refresh, so the fresh prompt is staged
        if self.score:
            self._upload_logits(t)
        if self.graph is None:
            self._make_graph()
        self.graph.launch()
        rec = {"t": t}
        if self.record:
            torch.cuda.synchronize()
            flags = self.flag.cpu().numpy()
            refreshed = bool(flags.any())
            # the layers share one output buffer: only the last layer's survives the replay
            outs = [None] * (self.L - 1) + [(self.out_full if refreshed else self.out_step).clone()]
            rec.update({"flag": flags, "out": outs, "dist": self.dist.cpu().numpy(), "g": self.g.cpu().numpy(),
                        "scores": ({"max_prob": self.max_prob.clone(), "top1": self.top1.clone(),
                                    "margin": self.margin.clone(),
                                    **({"cur_prob": self.cur_prob.clone()} if self.closed else {})}
                                   if self.score else None)})
        return rec

    def step(self):
        t = self.t = self.t + 1
        if self.graph_mode:
            return self._graph_step(t)
        self._stage_redraw(t)
        A.archer_should_refresh(self.g, self.g_anchor, self.age, self.K, self.max_age, True, self.dist, self.flag)
        self.flag_host.copy_(self.flag, non_blocking=True)
        torch.cuda.current_stream().synchronize()
        flags = self.flag_host.numpy()
        refresh = bool(flags.any())
        if refresh:
            self._n_refresh_steps += 1
            self._stage_fresh_prompt(t)
        outs = self._forward(refresh, self.flag if refresh else None)
        sc = self._score(t)
        rec = {"t": t, "flag": flags.copy(), "out": outs, "scores": sc}
        if self.record:
            rec["dist"] = self.dist.cpu().numpy()
            rec["g"] = self.g.cpu().numpy()
        return rec

    # ------------------------------------------------------------ checkpoint
    _STATE = ("q_all", "q_resp", "k_resp", "v_resp", "k_new", "v_new", "k_cache", "v_cache", "g", "g_anchor", "age",
              "dist", "flag", "refresh_count")
    _SCORES = ("max_prob", "top1", "margin", "cur_prob", "mask_state")

    def checkpoint(self) -> dict:
        """The trajectory's state in host memory: the step, the token state
        (g, the anchor g_r, the age), every layer's tensors -- the prompt cache
        C_p is the state Archer carries between steps (Sec. 4.2) -- and the last
        scores (the closed-loop decoder reads them).  restore() continues
        bit for bit."""
        torch.cuda.synchronize()
        st = {"t": self.t, "n_refresh": self._n_refresh_steps, "g_host": self.g_host.copy()}
        for name in self._STATE + self._SCORES:
            if hasattr(self, name):
                st[name] = getattr(self, name).detach().cpu().clone()
        return st

    def restore(self, st: dict):
        """Loads a checkpoint() into this trajectory's (same-shaped) tensors,
        in place: a step graph captured on them stays valid."""
        for name in self._STATE + self._SCORES:
            if name in st:
                getattr(self, name).copy_(st[name])
        self.t = st["t"]
        self._n_refresh_steps = st["n_refresh"]
        self.g_host = st["g_host"].copy()
        torch.cuda.synchronize()

    def attention_flops(self, refresh: bool) -> float:
        """Algorithmic attention FLOPs of one step over all layers: 4 B Hq M N D
        (Q K^T and P V, 2 flops per multiply-add), M = N on refresh, G cached."""
        M = self.N if refresh else self.G
        return 4.0 * self.B * self.Hq * M * self.N * self.D * self.L
